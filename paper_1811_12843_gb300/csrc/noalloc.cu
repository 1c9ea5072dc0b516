// Fitness from device-resident logits without any device allocation.
//
// The fitness kernel needs the per-pair losses L_G, L_D of every cell as intermediate storage.
// Here that storage is one file-scope __device__ array, so a call allocates nothing: it is for
// callers that cannot call cudaMalloc at the time they need the fitness (a serving loop whose
// device memory another allocator has fully reserved, or a latency-critical path that cannot
// take the implicit synchronisation of cudaMalloc / cudaFree).
#include <cstring>
#include <mutex>

#include "engine.h"
#include "lipz.h"

namespace {

constexpr int kMaxCells = LIPZ_NOALLOC_MAX_CELLS;
constexpr int kMaxDevices = 64;

// [0, 25 * max) pair L_G, [25 * max, 50 * max) pair L_D, then one int: the non-finite flag.
// Every GPU that loads the library holds this array (about 800 KB) until the process exits.
static __device__ __align__(256) float g_scratch[2 * 25 * kMaxCells + 64];

std::mutex g_mu;
float* g_scratch_addr[kMaxDevices] = {};

// Device address of g_scratch on the current device, looked up once per device (with that
// device current) and kept for the life of the process: the array moves if the device's
// primary context is torn down (cudaDeviceReset), so the call must not be used across one.
// The host symbol g_scratch is only a stand-in for the device array and must not reach a
// kernel.
cudaError_t scratch_address(float** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = static_cast<float*>(p);
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" LIPZ_API int lipz_fitness_from_logits_noalloc(const float* logits, int32_t cells,
                                                         int32_t batch, float* fit_g,
                                                         float* fit_d, void* stream) {
  if (!logits || !fit_g || !fit_d) return LIPZ_ERR_INVALID;
  if (cells < 1 || cells > kMaxCells || batch < 1) return LIPZ_ERR_INVALID;
  float* scratch = nullptr;
  if (scratch_address(&scratch) != cudaSuccess) {
    cudaGetLastError();
    return LIPZ_ERR_CUDA;
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  float* LG = scratch;
  float* LD = scratch + 25 * kMaxCells;
  int* flag = reinterpret_cast<int*>(scratch + 50 * kMaxCells);
  // the flag keeps the lowest cell with a non-finite loss: start above every cell index
  if (cudaMemsetAsync(flag, 0x7F, sizeof(int), st) != cudaSuccess) {
    cudaGetLastError();
    return LIPZ_ERR_CUDA;
  }
  // clear an error left by an unrelated earlier call, so that the check after the launch
  // reports this launch only
  cudaGetLastError();
  lipz::launch_fitness(logits, cells, batch, LG, LD, fit_g, fit_d, flag, st);
  if (cudaGetLastError() != cudaSuccess) return LIPZ_ERR_CUDA;
  return LIPZ_OK;
}
