// Shared device helpers of the grid-iteration engine: Philox4x32-10, Box-Muller, bf16
// conversions, the grouped-GEMM problem descriptor and launch helpers.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace lipz {

typedef __nv_bfloat16 bf16;

// ---- programmatic dependent launch: kernels of one grid iteration are launched with
// programmatic stream serialization, so a kernel is launched while the previous one retires;
// each waits for the previous kernel to complete and flush its memory (pdl_wait) before it
// touches global memory. Kernels signal no early completion: the next kernel starts only once
// every block of the previous one has exited. Without the launch attribute the wait is a no-op.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_kernel(bool pdl, void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                          cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  // only on an explicitly created stream: the legacy and per-thread default streams are
  // shared with other work and keep plain stream order
  const bool shared = st == nullptr || st == cudaStreamLegacy || st == cudaStreamPerThread;
  cfg.numAttrs = (pdl && !shared) ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t st, Args... args) {
  return launch_kernel(true, kernel, grid, block, smem, st, args...);
}

// ---- Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): ten rounds, key bumped by the Weyl
// constants between rounds; one round maps (c0, c1, c2, c3) to
// (hi(M1 c2) ^ c1 ^ k0, lo(M1 c2), hi(M0 c0) ^ c3 ^ k1, lo(M0 c0)).
struct U4 {
  uint32_t x, y, z, w;
};

__device__ __forceinline__ U4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                     uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t p0lo = 0xD2511F53u * c0, p0hi = __umulhi(0xD2511F53u, c0);
    const uint32_t p1lo = 0xCD9E8D57u * c2, p1hi = __umulhi(0xCD9E8D57u, c2);
    const uint32_t n0 = p1hi ^ c1 ^ k0, n2 = p0hi ^ c3 ^ k1;
    c0 = n0;
    c1 = p1lo;
    c2 = n2;
    c3 = p0lo;
  }
  return U4{c0, c1, c2, c3};
}

// Block `blk` of the (stream, t, cell) sequence of a grid with seed `seed`.
__device__ __forceinline__ U4 philox_block(uint64_t seed, uint32_t stream, uint32_t t,
                                           uint32_t cell, uint32_t blk) {
  return philox(blk, cell, t, stream, (uint32_t)seed, (uint32_t)(seed >> 32));
}

__device__ __forceinline__ uint32_t mulhi_u32(uint32_t w, uint32_t n) { return __umulhi(w, n); }

// Box-Muller: u1 = ((wa >> 8) + 1) / 2^24 in (0, 1], v = (wb >> 8) / 2^24; r = sqrt(-2 ln u1);
// returns (r cos 2 pi v, r sin 2 pi v).
__device__ __forceinline__ float2 box_muller(uint32_t wa, uint32_t wb) {
  const float u1 = (float)((wa >> 8) + 1u) * 5.9604644775390625e-8f;
  const float v = (float)(wb >> 8) * 5.9604644775390625e-8f;
  const float r = sqrtf(-2.0f * logf(u1));
  float s, c;
  sincospif(2.0f * v, &s, &c);
  return make_float2(r * c, r * s);
}

// ---- element conversions
template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<bf16>(bf16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// ---- activations (forward from the pre-activation, derivative from the stored output)
enum Act : int { ACT_NONE = 0, ACT_RELU = 1, ACT_LRELU = 2, ACT_TANH = 3 };

__device__ __forceinline__ float act_fwd(int act, float a, float slope) {
  switch (act) {
    case ACT_RELU: return a > 0.f ? a : 0.f;
    case ACT_LRELU: return a > 0.f ? a : slope * a;
    case ACT_TANH: return tanhf(a);
    default: return a;
  }
}

// Derivative expressed through the stored output y = act(a): ReLU: y > 0; LeakyReLU:
// y > 0 ? 1 : slope (the sign of y is the sign of a); tanh: 1 - y^2.
__device__ __forceinline__ float act_bwd(int act, float y, float slope) {
  switch (act) {
    case ACT_RELU: return y > 0.f ? 1.f : 0.f;
    case ACT_LRELU: return y > 0.f ? 1.f : slope;
    case ACT_TANH: return 1.f - y * y;
    default: return 1.f;
  }
}

// One Adam step (Kingma & Ba 2015, Algorithm 1) of one parameter, the bias corrections folded
// into ib1 = 1 / (1 - beta1^t) and ib2 = 1 / (1 - beta2^t). Every operation is spelled out (no
// contraction left to the compiler), so the stand-alone Adam kernel and the Adam fused into
// the tensor-core backward give the same bits for the same gradient. The square root and the
// division of the step use the hardware approximations (a few ulp): the step is about lr in
// size, so their error lies far below the fp32 rounding of the weight it is added to.
__device__ __forceinline__ float sqrt_approx(float x) {
  float r;
  asm("sqrt.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ void adam_elem(float& w, float& m, float& v, float g, float b1,
                                          float b2, float lr, float ib1, float ib2, float eps) {
  m = __fmaf_rn(b1, m, __fmul_rn(1.f - b1, g));
  v = __fmaf_rn(b2, v, __fmul_rn(__fmul_rn(1.f - b2, g), g));
  const float den = __fadd_rn(sqrt_approx(__fmul_rn(v, ib2)), eps);
  w = __fsub_rn(w, __fdividef(__fmul_rn(lr, __fmul_rn(m, ib1)), den));
}

// ---- grouped GEMM problem: C[m, n] = epi( sum_k A[m*sam + k*sak] * B[k*sbk + n*sbn] )
// Epilogues: EPI_BIAS_ACT: act(acc + bias[n]);  EPI_DACT: acc * act_bwd(aux[m*sxm + n*sxn]);
// EPI_STORE: acc. Element strides; pointers typed by the launch.
enum Epi : int { EPI_STORE = 0, EPI_BIAS_ACT = 1, EPI_DACT = 2 };

// A problem whose weight operand belongs to a selected individual sets wsel: the operand
// (wsel_op 1 = A, 2 = B) and the bias move by wsel[cell] * wsel_stride elements.
struct GemmDesc {
  const void* A;
  const void* B;
  void* C;
  const float* bias;
  const void* aux;
  const int* wsel;
  int64_t sam, sak, sbk, sbn, scm, scn, sxm, sxn;
  int64_t wsel_stride;
  int M, N, K;
  int wsel_op, cell, pad;
};

// Column sums: out[n] = sum_{r < rows} X[r * ld + n], n < cols (bias gradients).
struct ColSumDesc {
  const void* X;
  float* out;
  int64_t ld;
  int rows, cols;
};

// Dot of each row with a vector plus a bias (the discriminator's last layer):
// out[r] = sum_k X[r * ld + k] * w[k] + bias[0].
struct GemvDesc {
  const void* X;
  const void* w;
  const float* bias;
  float* out;
  const int* wsel;
  int64_t ld;
  int64_t wsel_stride;
  int rows, K, cell, pad;
};

}  // namespace lipz
