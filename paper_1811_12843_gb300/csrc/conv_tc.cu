// Tensor-core (tcgen05 / TMEM) implicit-GEMM convolution of the DCGAN discriminator's
// evaluation: y[m][o] = LeakyReLU(sum_k A[m][k] W[o][k]) for the 4x4 / stride 2 / pad 1
// convolutions, with m = (image, output row, output column) and k = (ky, kx, input channel).
// Activations are channel-last (NHWC), so the A operand of one 64-wide k chunk is, for a layer
// with at least 64 input channels, 128 contiguous bytes of one input pixel per row: four warps
// gather it with 16-byte loads straight into the 128-byte-swizzled K-major layout the MMA
// reads. The first layer reads the channel-major (CHW) images of the evaluation buffer with
// scalar loads (K = 48). Weights, re-laid out as [out][ky][kx][in], arrive by TMA. One CTA per
// SM over 128-row tiles; accumulators (up to 256 columns per job) alternate between two TMEM
// regions so that the epilogue of one job overlaps the MMAs of the next.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "common.cuh"
#include "conv_tc.h"
#include "tc_ptx.cuh"

namespace lipz {
namespace ctc {

using namespace ::lipz::tc;

constexpr int BM = 128, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = 256 * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int THREADS = 320;  // warp 0 TMA, 1 MMA, 2-5 gather, 6-9 epilogue
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 256;

__global__ void __launch_bounds__(THREADS, 1)
    k_conv_tc(const __grid_constant__ CUtensorMap mW, const __grid_constant__ CtcParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  uint8_t* misc = gbase + STAGES * STAGE_BYTES;
  const uint32_t bars = smem_u32(misc);
  const uint32_t bFullA = bars, bFullB = bars + 8 * STAGES, bEmpty = bars + 16 * STAGES;
  const uint32_t bAccF = bars + 24 * STAGES, bAccE = bAccF + 16, bFinal = bAccE + 16;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(misc + 240);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 244);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bFullA + 8 * s, 128);
      mbar_init(bFullB + 8 * s, 1);
      mbar_init(bEmpty + 8 * s, 1);
    }
    mbar_init(bAccF, 1);
    mbar_init(bAccF + 8, 1);
    mbar_init(bAccE, 128);
    mbar_init(bAccE + 8, 128);
    mbar_init(bFinal, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(
        smem_u32((const void*)tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  const int M = p.rows << (2 * p.lho);
  const int nbox = p.nbox;

  if (warp == 0) {
    // ---- weights by TMA
    if (lane == 0) {
      int stage = 0, issued[STAGES] = {0, 0, 0, 0};
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
        const ConvTcDesc d = p.descs[tile / p.mtiles];
        const int indiv = __ldg(&p.wsel[d.wsel_idx]);
        for (int j = 0; j < p.nj && ok; ++j)
          for (int kc = 0; kc < p.kchunks; ++kc) {
            if (!mbar_wait(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 21)) {
              ok = false;
              break;
            }
            mbar_expect_tx(bFullB + 8 * stage, (uint32_t)(nbox * BK * 2));
            tma_load_3d(base + stage * STAGE_BYTES + A_BYTES, &mW, bFullB + 8 * stage, kc * BK,
                        j * 256, indiv);
            issued[stage]++;
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
      }
      if (!ok) {
        for (int s = 0; s < STAGES; ++s)
          if (issued[s] > 0) {
            volatile int never = 0;
            mbar_wait(bFullB + 8 * s, (uint32_t)((issued[s] - 1) & 1), &never, p.err, 22);
          }
      }
    }
  } else if (warp == 1) {
    // ---- MMA issue
    if (lane == 0) {
      int stage = 0, uses[2] = {0, 0}, jobs = 0;
      uint32_t phase = 0;
      bool ok = true;
      const uint32_t idesc = idesc_bf16(BM, nbox);
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x)
        for (int j = 0; j < p.nj && ok; ++j, ++jobs) {
          const int R = jobs & 1;
          if (uses[R] > 0 &&
              !mbar_wait(bAccE + 8 * R, (uint32_t)((uses[R] - 1) & 1), abort_flag, p.err, 23)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t dt = tmem + (uint32_t)(R * 256);
          for (int kc = 0; kc < p.kchunks; ++kc) {
            if (!mbar_wait(bFullA + 8 * stage, phase, abort_flag, p.err, 24) ||
                !mbar_wait(bFullB + 8 * stage, phase, abort_flag, p.err, 25)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sA = base + stage * STAGE_BYTES, sB = sA + A_BYTES;
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              tc_mma(dt, sw128_desc(sA + kk * 32), sw128_desc(sB + kk * 32), idesc,
                     (kc | kk) != 0 ? 1u : 0u);
            tc_commit(bEmpty + 8 * stage);
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          tc_commit(bAccF + 8 * R);
          uses[R]++;
        }
      tc_commit(bFinal);
      volatile int never = 0;
      mbar_wait(bFinal, 0u, &never, p.err, 26);
    }
  } else if (warp < 6) {
    // ---- A operand: thread r gathers row r of every k chunk
    const int r = threadIdx.x - 64;
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    const int lhi = p.lhi, Hi = 1 << lhi;
    for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
      const ConvTcDesc d = p.descs[tile / p.mtiles];
      const int m = (tile % p.mtiles) * BM + r;
      const bool valid = m < M;
      const int nb = m >> (2 * p.lho), oy = (m >> p.lho) & ((1 << p.lho) - 1),
                ox = m & ((1 << p.lho) - 1);
      for (int j = 0; j < p.nj && ok; ++j)
        for (int kc = 0; kc < p.kchunks; ++kc) {
          if (!mbar_wait_warp(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 27)) {
            ok = false;
            break;
          }
          const uint32_t row = base + stage * STAGE_BYTES + (uint32_t)r * 128u;
          if (p.nchw_in) {
            // first layer: k = (ky * 4 + kx) * 3 + c over 48 values, CHW image input
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              uint32_t w[4];
#pragma unroll
              for (int e2 = 0; e2 < 4; ++e2) {
                float f[2];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                  const int k = u * 8 + e2 * 2 + h;
                  f[h] = 0.f;
                  if (valid && k < 48) {
                    const int tap = k / 3, c = k - 3 * tap;
                    const int iy = 2 * oy - 1 + (tap >> 2), ix = 2 * ox - 1 + (tap & 3);
                    if (iy >= 0 && iy < Hi && ix >= 0 && ix < Hi)
                      f[h] = __bfloat162float(
                          d.in[((int64_t)(nb * 3 + c) << (2 * lhi)) + (iy << lhi) + ix]);
                  }
                }
                w[e2] = pack_bf16(f[0], f[1]);
              }
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                               row + ((uint32_t)(u ^ (r & 7)) << 4)),
                           "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3])
                           : "memory");
            }
          } else {
            // channel-last input with ci a multiple of 64: one tap, 64 channels per chunk
            const int k0 = kc * BK;
            const int tap = k0 / p.ci, c0 = k0 - tap * p.ci;
            const int iy = 2 * oy - 1 + (tap >> 2), ix = 2 * ox - 1 + (tap & 3);
            const bool in = valid && iy >= 0 && iy < Hi && ix >= 0 && ix < Hi;
            const uint4* src = reinterpret_cast<const uint4*>(
                d.in + ((((int64_t)nb << (2 * lhi)) + (iy << lhi) + ix) * p.ci + c0));
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              const uint4 v = in ? __ldg(src + u) : make_uint4(0u, 0u, 0u, 0u);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                               row + ((uint32_t)(u ^ (r & 7)) << 4)),
                           "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                           : "memory");
            }
          }
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          mbar_arrive(bFullA + 8 * stage);
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
    }
  } else {
    // ---- epilogue: LeakyReLU, bf16, channel-last rows
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    int uses[2] = {0, 0}, jobs = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
      const ConvTcDesc d = p.descs[tile / p.mtiles];
      const int m = (tile % p.mtiles) * BM + row;
      const bool valid = m < M;
      for (int j = 0; j < p.nj && ok; ++j, ++jobs) {
        const int R = jobs & 1;
        if (!mbar_wait_warp(bAccF + 8 * R, (uint32_t)(uses[R] & 1), abort_flag, p.err, 28)) {
          ok = false;
          break;
        }
        tc_fence_after();
        for (int g = 0; g < nbox / 32; ++g) {
          uint32_t v[32];
          LIPZ_TMEM_LD32(tmem + lane_base + (uint32_t)(R * 256 + g * 32), v);
          tmem_wait_ld();
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 32; e += 2) {
            float a = __uint_as_float(v[e]), b = __uint_as_float(v[e + 1]);
            a = a > 0.f ? a : p.slope * a;
            b = b > 0.f ? b : p.slope * b;
            pk[e >> 1] = pack_bf16(a, b);
          }
          if (valid) {
            uint4* o = reinterpret_cast<uint4*>(d.out + (int64_t)m * p.co + j * 256 + g * 32);
#pragma unroll
            for (int u = 0; u < 4; ++u)
              o[u] = make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
          }
        }
        tc_fence_before();
        mbar_arrive(bAccE + 8 * R);
        uses[R]++;
      }
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
}

// [out][in][ky][kx] -> [out][ky][kx][in] for the five discriminator tensors of every
// individual (bf16 copies).
__global__ void k_relayout_d(const bf16* __restrict__ src, bf16* __restrict__ dst, int n_indiv,
                             int64_t Ps, RelayoutD r) {
  pdl_wait();
  const int64_t total = (int64_t)n_indiv * r.P;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    const int64_t ind = e / r.P, k = e - ind * r.P;
    int l = 0;
    while (l + 1 < 5 && k >= r.off[l + 1]) ++l;
    const int64_t i = k - r.off[l];
    const int ci = r.ci[l];
    // destination index i = (o * 16 + tap) * ci + c
    const int64_t c = i % ci, t = (i / ci) & 15, o = i / (16 * (int64_t)ci);
    dst[ind * Ps + k] = src[ind * Ps + r.off[l] + (o * ci + c) * 16 + t];
  }
}

}  // namespace ctc

namespace {
PFN_cuTensorMapEncodeTiled_v12000 g_encode_ctc = nullptr;
}

bool ctc_make_map(CUtensorMap* m, const void* base, uint64_t K, uint64_t rows, uint64_t depth,
                  uint64_t depth_elems, uint32_t box_rows, std::string* msg) {
  if (!g_encode_ctc) {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess || !fn) {
      if (msg) *msg = "cuTensorMapEncodeTiled is not available";
      return false;
    }
    g_encode_ctc = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  }
  cuuint64_t dims[3] = {K, rows, depth};
  cuuint64_t strides[2] = {K * 2, depth_elems * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_encode_ctc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled (convolution weights) failed: " + std::to_string((int)r);
    return false;
  }
  return true;
}

bool ctc_prepare(std::string* msg) {
  if (cudaFuncSetAttribute(ctc::k_conv_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           ctc::SMEM_BYTES) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cannot reserve shared memory for the tensor-core convolution";
    return false;
  }
  return true;
}

void launch_conv_tc(const CUtensorMap& mW, const CtcParams& p, int sms, cudaStream_t st) {
  const int grid = p.n_tiles < sms ? p.n_tiles : sms;
  launch_pdl(ctc::k_conv_tc, dim3(grid), dim3(ctc::THREADS), ctc::SMEM_BYTES, st, mW, p);
}

void launch_relayout_d(const bf16* src, bf16* dst, int n_indiv, int64_t Ps, const RelayoutD& r,
                       cudaStream_t st) {
  launch_pdl(ctc::k_relayout_d, dim3(1216), dim3(256), 0, st, src, dst, n_indiv, Ps, r);
}

}  // namespace lipz
