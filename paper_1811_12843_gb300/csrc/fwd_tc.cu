// Tensor-core forward of the evaluation phase (placeholder until the tcgen05 kernels land).
#include "fwd_tc.h"

namespace lipz {

struct TcPlan {
  int unused;
};

bool tc_supported(int, int, int, int) { return false; }

TcPlan* tc_plan_create(const TcShape&, void*, void*, int64_t, float*, const int*,
                       const __nv_bfloat16*, const float*, int64_t, const int64_t*,
                       const __nv_bfloat16*, const float*, int64_t, const int64_t*,
                       std::string* msg) {
  if (msg) *msg = "tensor-core forward not built";
  return nullptr;
}

int tc_run_g(TcPlan*, cudaStream_t, std::string* msg) {
  if (msg) *msg = "tensor-core forward not built";
  return 1;
}

int tc_run_d(TcPlan*, cudaStream_t, std::string* msg) {
  if (msg) *msg = "tensor-core forward not built";
  return 1;
}

void tc_plan_destroy(TcPlan* p) { delete p; }

}  // namespace lipz
