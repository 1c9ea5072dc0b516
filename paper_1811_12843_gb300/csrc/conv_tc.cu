// Tensor-core (tcgen05 / TMEM) implicit-GEMM convolutions of the DCGAN networks:
// y[m][o] = epilogue(sum_k A[m][k] W[o][k]) for the 4x4 / stride 2 / pad 1 convolutions, with
// m = (image, output row, output column) and k = (ky, kx, input channel), and for the stride-2
// transposed convolutions by output parity class (k = (tap of the class, input channel)).
// Activations are channel-last (NHWC), so the A operand of one 64-wide k chunk is one tap's 64
// channels of 128 input pixels: the TMA warp loads it through a 5-D activation map (channels,
// columns, rows, images, problems) whose traversal stride 2 picks the convolution's input
// pixels, or whose per-class row/column offset picks the transposed convolution's, straight
// into the 128-byte-swizzled K-major layout the MMA reads. The 3-channel first layer reads
// channel-major (CHW) images: four gather warps build its rows (K = 48) from input patches
// staged in shared memory one tile ahead. Weights, re-laid out as [out][tap][in], arrive by
// TMA. One CTA per SM over 128-row tiles; accumulators (up to 256 columns per job) alternate
// between two TMEM regions so that the epilogue of one job overlaps the MMAs of the next.
// The weight-gradient kernel (k_wgrad_tc) and the channel-last batch norm live here too.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
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
// first-layer input patches: 3 channels x 10 rows x 72 columns (64 interior at column 4)
constexpr int PATCH_BYTES = 4352;
// epilogue staging for coalesced row stores: 32 rows x 36 words per epilogue warp
constexpr int STG_WORDS = 32 * 36;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + 256 + 3 * PATCH_BYTES + 4 * STG_WORDS * 4;
constexpr int LAG = 2;  // copy groups a gather thread keeps in flight (< STAGES)

// 16-byte global -> shared copy; bytes = 0 writes zeros (src must still be a valid address)
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async8(uint32_t dst, const void* src, int bytes) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(src), "r"(bytes)
               : "memory");
}

// Barrier of the four epilogue warps (named barrier 2), plain and with an OR vote.
__device__ __forceinline__ void epi_bar() { asm volatile("bar.sync 2, 128;" ::: "memory"); }
__device__ __forceinline__ bool epi_bar_or(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 2, 128, p;\n"
      " selp.u32 %0, 1, 0, q;\n}"
      : "=r"(r)
      : "r"((uint32_t)pred)
      : "memory");
  return r != 0;
}

// Barrier of the four gather warps (named barrier 1) that returns whether any thread passed
// true.
__device__ __forceinline__ bool gather_bar_or(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, 128, p;\n"
      " selp.u32 %0, 1, 0, q;\n}"
      : "=r"(r)
      : "r"((uint32_t)pred)
      : "memory");
  return r != 0;
}

enum { AK_CONV = 0, AK_TRANS = 1, AK_SCATTER = 2, AK_NCHW = 3, AK_GATHER = 4,
       AK_NCHW_WIDE = 5, AK_TRANS_C = 6 };

// dynamic shared memory of a variant: the compact first layer (three 24 KB stages) and the
// compact parity classes (256-row tiles of weight tiles of at most 64 rows: two 40 KB stages,
// no patch buffers) fit two CTAs per SM
constexpr int conv_smem(int ak) {
  return ak == AK_NCHW
             ? 1024 + 3 * (A_BYTES + 64 * BK * 2) + 256 + 3 * PATCH_BYTES + 4 * STG_WORDS * 4
         : ak == AK_TRANS_C ? 1024 + 2 * (2 * A_BYTES + 64 * BK * 2) + 256 + 4 * STG_WORDS * 4
                            : SMEM_BYTES;
}

// AK: how the A tiles arrive (AK_CONV / AK_TRANS / AK_SCATTER: TMA through the activation map
// for the convolution, the parity classes, the scatter mode; AK_NCHW / AK_NCHW_WIDE: built
// from staged first-layer patches, the former for weight tiles of at most 64 rows in a compact
// layout that fits two CTAs per SM; AK_GATHER: gathered channel-last rows, convolution or
// parity classes as p.transposed says). OM: the out_mode. Each launch runs the instantiation
// its parameters name, so that a kernel holds only its own code paths.
template <int AK, int OM>
__global__ void __launch_bounds__(THREADS, AK == AK_NCHW || AK == AK_TRANS_C ? 2 : 1)
    k_conv_tc(const __grid_constant__ CUtensorMap mW, const __grid_constant__ CUtensorMap mA,
              const __grid_constant__ CtcParams p) {
  extern __shared__ uint8_t smem_raw[];
  constexpr bool kTma = AK == AK_CONV || AK == AK_TRANS || AK == AK_SCATTER || AK == AK_TRANS_C;
  constexpr bool kScatter = AK == AK_SCATTER, kNchw = AK == AK_NCHW || AK == AK_NCHW_WIDE;
  // AK_NCHW (weight tiles of at most 64 rows): three 24 KB stages and 256 TMEM columns, so
  // that two CTAs share an SM
  constexpr bool kCompact = AK == AK_NCHW || AK == AK_TRANS_C;
  constexpr int STAGES = AK == AK_NCHW ? 3 : AK == AK_TRANS_C ? 2 : ctc::STAGES;
  constexpr uint32_t STAGE_BYTES = AK == AK_NCHW     ? A_BYTES + 64 * BK * 2
                                   : AK == AK_TRANS_C ? 2 * A_BYTES + 64 * BK * 2
                                                      : ctc::STAGE_BYTES;
  // the first layer's patch buffers sit between the barriers and the epilogue staging
  constexpr int kPatchArea = AK == AK_TRANS_C ? 0 : 3 * PATCH_BYTES;
  constexpr uint32_t kTmemCols = kCompact ? 256 : 512, kAccStride = kCompact ? 128 : 256;
  const bool transposed = AK == AK_TRANS || AK == AK_TRANS_C || (AK == AK_GATHER && p.transposed);
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
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_u32((const void*)tmem_slot)),
                 "r"(kTmemCols));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  // output pixels per problem (per parity class when transposed)
  // rows of a problem: output pixels (class pixels when transposed; input pixels in scatter)
  const int lq = kScatter ? p.lhi : p.lho - (transposed ? 1 : 0);
  const int M = p.rows << (2 * lq);
  const int nbox = p.nbox;

  if (warp == 0) {
    // ---- weights by TMA
    if (lane == 0) {
      int stage = 0, issued[STAGES] = {};
      uint32_t phase = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
        const int pc = tile / p.mtiles;  // problem (x 4 parity classes when transposed)
        const ConvTcDesc d = p.descs[transposed ? pc >> 2 : pc];
        const int cls = transposed ? (pc & 3) : 0;
        const int indiv = __ldg(&p.wsel[d.wsel_idx]);
        // channel-last A rows by TMA (a_tma): the tile is 128 consecutive output pixels (class
        // pixels when transposed) of whole rows; its origin is image n0, row y0
        const int m0 = (tile % p.mtiles) * (p.m2 ? 2 * BM : BM);
        const int n0 = m0 >> (2 * lq), y0 = (m0 >> lq) & ((1 << lq) - 1);
        // m2: the second 128 rows of a 256-row tile
        const int n1 = (m0 + BM) >> (2 * lq), y1 = ((m0 + BM) >> lq) & ((1 << lq) - 1);
        for (int j = 0; j < p.nj && ok; ++j)
          for (int kc = 0; kc < p.kchunks; ++kc) {
            if (!mbar_wait(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 21)) {
              ok = false;
              break;
            }
            mbar_expect_tx(bFullB + 8 * stage,
                           (uint32_t)(nbox * BK * 2 + (kTma ? (p.m2 ? 2 : 1) * A_BYTES : 0)));
            if constexpr (kTma) {
              // Convolution: tap (ky, kx), input rows 2 y - 1 + ky, columns 2 x - 1 + kx (the
              // map's traversal stride 2). Transposed, class (a, b), tap (u, v): ky = (a + 1)
              // mod 2 + 2u, input row y + (a + 1 - ky) / 2, column x + (b + 1 - kx) / 2.
              const int k0 = kc * BK;
              const int tap = k0 / p.ci, c0 = k0 - tap * p.ci;
              // input row = ym * (tile row origin) + ya
              int x, ya, ym;
              if (kScatter) {
                ym = 1;
                ya = 0;
                x = 0;
              } else if (transposed) {
                const int a = cls >> 1, b = cls & 1;
                const int ky = ((a + 1) & 1) + 2 * (tap >> 1), kx = ((b + 1) & 1) + 2 * (tap & 1);
                ym = 1;
                ya = (a + 1 - ky) >> 1;
                x = (b + 1 - kx) >> 1;
              } else {
                ym = 2;
                ya = (tap >> 2) - 1;
                x = (tap & 3) - 1;
              }
              const int prob = transposed ? pc >> 2 : pc;
              tma_load_5d(base + stage * STAGE_BYTES, &mA, bFullB + 8 * stage, c0, x,
                          ym * y0 + ya, n0, prob);
              if (p.m2)
                tma_load_5d(base + stage * STAGE_BYTES + A_BYTES, &mA, bFullB + 8 * stage, c0, x,
                            ym * y1 + ya, n1, prob);
            }
            tma_load_3d(base + stage * STAGE_BYTES + (p.m2 ? 2 : 1) * A_BYTES, &mW,
                        bFullB + 8 * stage, kc * BK, cls * p.cls_rows + j * 256, indiv);
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
          const uint32_t dt = tmem + (uint32_t)(R * kAccStride);
          for (int kc = 0; kc < p.kchunks; ++kc) {
            if ((!kTma && !mbar_wait(bFullA + 8 * stage, phase, abort_flag, p.err, 24)) ||
                !mbar_wait(bFullB + 8 * stage, phase, abort_flag, p.err, 25)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sA = base + stage * STAGE_BYTES;
            const uint32_t sB = sA + (p.m2 ? 2 : 1) * A_BYTES;
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk) {
              tc_mma(dt, sw128_desc(sA + kk * 32), sw128_desc(sB + kk * 32), idesc,
                     (kc | kk) != 0 ? 1u : 0u);
              if (p.m2)
                tc_mma(dt + (uint32_t)nbox, sw128_desc(sA + A_BYTES + kk * 32),
                       sw128_desc(sB + kk * 32), idesc, (kc | kk) != 0 ? 1u : 0u);
            }
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
  } else if (warp < 6 && !kTma) {
    // ---- A operand: thread r gathers row r of every k chunk. Channel-last rows arrive by
    // 16-byte cp.async (zero fill outside the image), a stage marked full LAG chunks later once
    // its copy group has landed; the first layer's rows are built from staged input patches.
    const int r = threadIdx.x - 64;
    int stage = 0, arr_stage = 0, pending = 0;
    uint32_t phase = 0;
    bool ok = true;
    const int lhi = p.lhi, Hi = 1 << lhi;
    if constexpr (kNchw) {
      // first layer (3 channels, 64 x 64 CHW images, 32 x 32 outputs, one k chunk of
      // k = c * 16 + ky * 4 + kx over 48 values, the weights' own [out][c][ky][kx] order): a
      // tile's 128 rows are 4 output rows, fed by
      // a 3 x 10 x 64 input patch that the gather threads copy one tile ahead by 8-byte
      // cp.async into one of three shared buffers whose halo columns stay zero
      uint8_t* patches = misc + 256;
      const uint32_t patch0 = smem_u32(patches);
      for (int i = r; i < 3 * PATCH_BYTES / 16; i += 128)
        *reinterpret_cast<uint4*>(patches + 16 * i) = make_uint4(0u, 0u, 0u, 0u);
      gather_bar_or(false);
      auto prefetch = [&](int tile, int buf) {
        if (tile < p.n_tiles) {
          const ConvTcDesc d = p.descs[tile / p.mtiles];
          const int m0 = (tile % p.mtiles) * BM;
          const int nb = m0 >> 10, oy0 = (m0 >> 5) & 31;
          for (int u = r; u < 480; u += 128) {
            const int c = u / 160, rem = u - c * 160, pr = rem >> 4, q = rem & 15;
            const int iy = 2 * oy0 - 1 + pr;
            const bool in = iy >= 0 && iy < 64;
            const bf16* src = in ? d.in + ((int64_t)(nb * 3 + c) << 12) + (iy << 6) + 4 * q : d.in;
            cp_async8(patch0 + (uint32_t)(buf * PATCH_BYTES + ((c * 10 + pr) * 72 + 4 + 4 * q) * 2),
                      src, in ? 8 : 0);
          }
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
      };
      prefetch(blockIdx.x, 0);
      int buf = 0;
      const int ox = r & 31, oyl = r >> 5;
      for (int tile = blockIdx.x; tile < p.n_tiles; tile += gridDim.x) {
        prefetch(tile + gridDim.x, buf == 2 ? 0 : buf + 1);
        asm volatile("cp.async.wait_group 1;" ::: "memory");
        const bool okw = mbar_wait_warp(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 27);
        if (gather_bar_or(!okw)) {
          ok = false;
          break;
        }
        const bool valid = (tile % p.mtiles) * BM + r < M;
        const unsigned short* pb =
            reinterpret_cast<const unsigned short*>(patches + buf * PATCH_BYTES);
        const uint32_t row = base + stage * STAGE_BYTES + (uint32_t)r * 128u;
        // group (c, ky) = k / 4: the four kx values are patch columns 2 ox + 3 .. 2 ox + 6 of
        // patch row c * 10 + 2 oyl + ky, taken from the three aligned words at 2 ox + 2
        const uint32_t* pw = reinterpret_cast<const uint32_t*>(pb);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const int gidx = 2 * u + hh;  // c * 4 + ky
            if (gidx < 12 && valid) {
              const int c = gidx >> 2, ky = gidx & 3;
              const int e0 = (c * 10 + 2 * oyl + ky) * 72 + 2 * ox + 2;
              const uint32_t w0 = pw[e0 >> 1], w1 = pw[(e0 >> 1) + 1], w2 = pw[(e0 >> 1) + 2];
              w[2 * hh] = __byte_perm(w0, w1, 0x5432);
              w[2 * hh + 1] = __byte_perm(w1, w2, 0x5432);
            }
          }
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                           row + ((uint32_t)(u ^ (r & 7)) << 4)),
                       "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3])
                       : "memory");
        }
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        mbar_arrive(bFullA + 8 * stage);
        if (++stage == STAGES) {
          stage = 0;
          phase ^= 1u;
        }
        buf = buf == 2 ? 0 : buf + 1;
      }
    } else
    for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
      const int pc = tile / p.mtiles;
      const ConvTcDesc d = p.descs[transposed ? pc >> 2 : pc];
      const int cls = transposed ? (pc & 3) : 0;
      const int m = (tile % p.mtiles) * BM + r;
      const bool valid = m < M;
      const int nb = m >> (2 * lq);
      int oy = (m >> lq) & ((1 << lq) - 1), ox = m & ((1 << lq) - 1);
      if (transposed) {
        oy = 2 * oy + (cls >> 1);
        ox = 2 * ox + (cls & 1);
      }
      for (int j = 0; j < p.nj && ok; ++j)
        for (int kc = 0; kc < p.kchunks; ++kc) {
          if (!mbar_wait_warp(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 27)) {
            ok = false;
            break;
          }
          const uint32_t row = base + stage * STAGE_BYTES + (uint32_t)r * 128u;
          {
            // channel-last input with ci a multiple of 64: one tap, 64 channels per chunk.
            // Convolution: tap (ky, kx) of 16, input pixel (2 oy - 1 + ky, 2 ox - 1 + kx).
            // Transposed (stride 2, pad 1, by class): tap (u, v) of 4, ky = (oy + 1) mod 2 + 2u,
            // input pixel ((oy + 1 - ky) / 2, (ox + 1 - kx) / 2).
            const int k0 = kc * BK;
            const int tap = k0 / p.ci, c0 = k0 - tap * p.ci;
            int iy, ix, ty = 0, tx = 0;
            if (transposed) {
              const int ky = ((oy + 1) & 1) + 2 * (tap >> 1), kx = ((ox + 1) & 1) + 2 * (tap & 1);
              ty = oy + 1 - ky;
              tx = ox + 1 - kx;
              iy = ty >> 1;
              ix = tx >> 1;
            } else {
              iy = 2 * oy - 1 + (tap >> 2);
              ix = 2 * ox - 1 + (tap & 3);
            }
            const bool in = valid && ty >= 0 && tx >= 0 && iy >= 0 && iy < Hi && ix >= 0 &&
                            ix < Hi;
            const bf16* src =
                in ? d.in + ((((int64_t)nb << (2 * lhi)) + (iy << lhi) + ix) * p.ci + c0) : d.in;
#pragma unroll
            for (int u = 0; u < 8; ++u)
              cp_async16(row + ((uint32_t)(u ^ (r & 7)) << 4), src + (in ? 8 * u : 0),
                         in ? 16 : 0);
            asm volatile("cp.async.commit_group;" ::: "memory");
            if (++pending > LAG) {
              asm volatile("cp.async.wait_group %0;" ::"n"(LAG) : "memory");
              asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
              mbar_arrive(bFullA + 8 * arr_stage);
              arr_stage = arr_stage + 1 == STAGES ? 0 : arr_stage + 1;
              --pending;
            }
          }
          if (++stage == STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
    }
    // the last chunks (and, after an expired wait, every copy still in flight)
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    for (; pending > 0; --pending) {
      mbar_arrive(bFullA + 8 * arr_stage);
      arr_stage = arr_stage + 1 == STAGES ? 0 : arr_stage + 1;
    }
  } else if (warp >= 6) {
    // ---- epilogue: LeakyReLU, bf16, channel-last rows
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    uint32_t* stg = reinterpret_cast<uint32_t*>(misc + 256 + kPatchArea) + (warp - 6) * STG_WORDS;
    // tma_out (first layer, 64 channels): the tile's 128 rows x 128 bytes go to the staging area
    // (1024-byte aligned) in the 128-byte swizzle, and one thread stores them by TMA through the
    // output map (passed as mA, which the first layer's gather does not use)
    const bool kTmaOut = AK == AK_NCHW && OM == CTC_LRELU_HWC && p.tma_out;
    const uint32_t tileb = smem_u32(misc + 256 + kPatchArea);
    int uses[2] = {0, 0}, jobs = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
      const int pc = tile / p.mtiles;
      const ConvTcDesc d = p.descs[transposed ? pc >> 2 : pc];
      const int cls = transposed ? (pc & 3) : 0;
      const int m = (tile % p.mtiles) * (p.m2 ? 2 * BM : BM) + row;
      const bool valid = m < M;
      const int nb = m >> (2 * lq);
      int oy = (m >> lq) & ((1 << lq) - 1), ox = m & ((1 << lq) - 1);
      if (transposed) {
        oy = 2 * oy + (cls >> 1);
        ox = 2 * ox + (cls & 1);
      }
      // CTC_LRELU_LOGIT: this row's share of its image's logit (the 4 x 4 x C output layer on
      // the bf16 activations, pixel = row mod 16), summed over the jobs
      float dot = 0.f;
      const bf16* w5 = nullptr;
      if constexpr (OM == CTC_LRELU_LOGIT)
        w5 = p.logit_w + (int64_t)__ldg(&p.wsel[d.wsel_idx]) * p.logit_ws +
             (int64_t)(m & 15) * p.co;
      for (int j = 0; j < p.nj && ok; ++j, ++jobs) {
        const int R = jobs & 1;
        // the scatter epilogue synchronises the four warps: they leave together
        const bool okw =
            mbar_wait_warp(bAccF + 8 * R, (uint32_t)(uses[R] & 1), abort_flag, p.err, 28);
        if ((kScatter || kTmaOut) ? epi_bar_or(!okw) : !okw) {
          ok = false;
          break;
        }
        tc_fence_after();
        if constexpr (kScatter) {
          // input pixel (y0 + q, lane) holds Y[tap * 4 + o] (16 taps, 3 channels); the taps are
          // added one after the other into the tile's 10 x 66 output window in shared memory
          // (output row 2 y - 1 + ky, column 2 x - 1 + kx; window origin (2 y0 - 1, -1))
          float* acc = reinterpret_cast<float*>(stg - (warp - 6) * STG_WORDS);
          const int et = threadIdx.x - 192;
          const int m0t = m - row;  // the tile's first input pixel: image img, rows 4 blk ..
          const int img = m0t >> 10, blk = (m0t >> 7) & 7;
          for (int i = et; i < 1980; i += 128) acc[i] = 0.f;
          uint32_t v[32], w[32];  // columns 0..31 (taps 0..7) and 32..63 (taps 8..15)
          LIPZ_TMEM_LD32(tmem + lane_base + (uint32_t)(R * kAccStride), v);
          LIPZ_TMEM_LD32(tmem + lane_base + (uint32_t)(R * kAccStride + 32), w);
          tmem_wait_ld();
          tc_fence_before();
          mbar_arrive(bAccE + 8 * R);
          uses[R]++;
          epi_bar();
          // taps with ky < 2 first (warp q writes window rows 2q, 2q + 1: no two warps share a
          // row), then ky >= 2 (rows 2q + 2, 2q + 3); inside a warp the taps go in order
#pragma unroll
          for (int tap = 0; tap < 16; ++tap) {
            float* a = acc + ((2 * q + (tap >> 2)) * 66 + 2 * lane + (tap & 3)) * 3;
            const uint32_t* y = tap < 8 ? v + tap * 4 : w + (tap - 8) * 4;
            if (valid) {
              a[0] += __uint_as_float(y[0]);
              a[1] += __uint_as_float(y[1]);
              a[2] += __uint_as_float(y[2]);
            }
            if (tap == 7 || tap == 15)
              epi_bar();
            else
              __syncwarp();
          }
          // window rows 2..7 (output rows 8 blk + 1 .. 8 blk + 6) are complete; rows 0, 1, 8, 9
          // are shared with the blocks above and below and go to the halo buffer
          const bool tv = m0t < M;
          if (tv) {
            for (int i = et; i < 6 * 64 * 3; i += 128) {
              const int o = i / 384, rem = i - o * 384, lr = 2 + (rem >> 6), gx = rem & 63;
              const int64_t oi = (((int64_t)img * 3 + o) << 12) + ((8 * blk - 1 + lr) << 6) + gx;
              float x = acc[(lr * 66 + gx + 1) * 3 + o];
              if (OM == CTC_TANH_CHW) {
                x = tanhf(x);
              } else {
                const float f = __bfloat162float(d.aux[oi]);
                x = x * (1.f - f * f);
              }
              d.out[oi] = __float2bfloat16_rn(x);
            }
            float* h = p.halo + (((int64_t)pc * p.rows + img) * 8 + blk) * 768;
            for (int i = et; i < 768; i += 128) {
              const int pr = i / 192, rem = i - pr * 192, gx = rem / 3, o = rem - gx * 3;
              h[i] = acc[((pr < 2 ? pr : pr + 6) * 66 + gx + 1) * 3 + o];
            }
          }
          epi_bar();
          continue;
        }
        if (OM == CTC_TANH_CHW || OM == CTC_DTANH_CHW) {
          // a few output channels (the image's colours), channel-major images: tanh, or the
          // delta times tanh' = 1 - f^2 with f the stored tanh output
          uint32_t v[16];
          LIPZ_TMEM_LD16(tmem + lane_base + (uint32_t)(R * kAccStride), v);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 16; ++e)
            if (valid && e < p.co) {
              const int64_t o = (((int64_t)nb * p.co + e) << (2 * p.lho)) + (oy << p.lho) + ox;
              float x = __uint_as_float(v[e]);
              if (OM == CTC_TANH_CHW) {
                x = tanhf(x);
              } else {
                const float f = __bfloat162float(d.aux[o]);
                x = x * (1.f - f * f);
              }
              d.out[o] = __float2bfloat16_rn(x);
            }
        } else {
          for (int h = 0; h < (p.m2 ? 2 : 1); ++h) {
          // row m + 128 h of the tile (its accumulator columns start at h * nbox); valid and
          // pix shadow the first half's
          const int mh = m + h * BM;
          const bool valid = mh < M;
          int oyh = (mh >> lq) & ((1 << lq) - 1), oxh = mh & ((1 << lq) - 1);
          if (transposed) {
            oyh = 2 * oyh + (cls >> 1);
            oxh = 2 * oxh + (cls & 1);
          }
          const int64_t pix = ((int64_t)(mh >> (2 * lq)) << (2 * p.lho)) + (oyh << p.lho) + oxh;
          if (kTmaOut) {
            // the previous tile's store has read the staging area before anyone rewrites it
            if (threadIdx.x == 192) bulk_wait_read<0>();
            epi_bar();
          }
          for (int g = 0; g < nbox / 32; ++g) {
            uint32_t v[32];
            LIPZ_TMEM_LD32(tmem + lane_base + (uint32_t)(R * kAccStride + h * nbox + g * 32), v);
            tmem_wait_ld();
            // the row's 32 columns go to the warp's staging rows (fp32 words, or bf16 pairs),
            // then out in 16-byte pieces, lpr lanes per row, so that each store instruction
            // writes whole rows' contiguous bytes
            const bool f32 = OM == CTC_F32_HWC;
            if (f32) {
#pragma unroll
              for (int u = 0; u < 8; ++u)
                *reinterpret_cast<uint4*>(stg + lane * 36 + 4 * u) =
                    make_uint4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
            } else {
            uint32_t pk[16];
            if (OM == CTC_DLRELU_HWC) {
              // the LeakyReLU derivative at the stored activation (same sign as its input)
              uint4 au[4] = {make_uint4(0u, 0u, 0u, 0u), make_uint4(0u, 0u, 0u, 0u),
                             make_uint4(0u, 0u, 0u, 0u), make_uint4(0u, 0u, 0u, 0u)};
              if (valid) {
                const uint4* ap =
                    reinterpret_cast<const uint4*>(d.aux + pix * p.co + j * 256 + g * 32);
#pragma unroll
                for (int u = 0; u < 4; ++u) au[u] = __ldg(ap + u);
              }
              const __nv_bfloat16* ab = reinterpret_cast<const __nv_bfloat16*>(au);
#pragma unroll
              for (int e = 0; e < 32; e += 2) {
                float a = __uint_as_float(v[e]), b = __uint_as_float(v[e + 1]);
                a = __bfloat162float(ab[e]) > 0.f ? a : p.slope * a;
                b = __bfloat162float(ab[e + 1]) > 0.f ? b : p.slope * b;
                pk[e >> 1] = pack_bf16(a, b);
              }
            } else {
#pragma unroll
              for (int e = 0; e < 32; e += 2) {
                float a = __uint_as_float(v[e]), b = __uint_as_float(v[e + 1]);
                a = a > 0.f ? a : p.slope * a;
                b = b > 0.f ? b : p.slope * b;
                pk[e >> 1] = pack_bf16(a, b);
              }
            }
            if (kTmaOut) {
              // row `row`, 16-byte units 4 g + u of its 128 bytes, in the 128-byte swizzle
              const uint32_t rb = tileb + (uint32_t)row * 128u;
#pragma unroll
              for (int u = 0; u < 4; ++u)
                asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                                 rb + ((uint32_t)((4 * g + u) ^ (row & 7)) << 4)),
                             "r"(pk[4 * u]), "r"(pk[4 * u + 1]), "r"(pk[4 * u + 2]),
                             "r"(pk[4 * u + 3])
                             : "memory");
              continue;
            }
            if constexpr (OM == CTC_LRELU_LOGIT) {
              // the output layer instead of storing the activations
              const uint4* wp = reinterpret_cast<const uint4*>(w5 + j * 256 + g * 32);
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const uint4 wv = __ldg(wp + u);
                const uint32_t ww[4] = {wv.x, wv.y, wv.z, wv.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const float2 af =
                      __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&pk[4 * u + e]));
                  const float2 wf =
                      __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&ww[e]));
                  dot = fmaf(af.x, wf.x, dot);
                  dot = fmaf(af.y, wf.y, dot);
                }
              }
            } else {
#pragma unroll
              for (int u = 0; u < 4; ++u)
                *reinterpret_cast<uint4*>(stg + lane * 36 + 4 * u) =
                    make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2], pk[4 * u + 3]);
            }
            }
            if constexpr (OM == CTC_LRELU_LOGIT) continue;
            __syncwarp();
            if (f32 && p.bn_part) {
              // batch-norm statistics: sum and sum of squares of column `lane` over the warp's
              // valid rows, in row order, into this (tile, half, lane quarter)'s slot
              const unsigned vm = __ballot_sync(0xffffffffu, valid);
              float bs = 0.f, bq = 0.f;
#pragma unroll 8
              for (int rr = 0; rr < 32; ++rr) {
                const float x = __uint_as_float(stg[rr * 36 + lane]);
                if ((vm >> rr) & 1u) {
                  bs += x;
                  bq = fmaf(x, x, bq);
                }
              }
              const int64_t slot = ((int64_t)tile * (p.m2 ? 2 : 1) + h) * 4 + q;
              p.bn_part[slot * p.co + j * 256 + g * 32 + lane] = make_float2(bs, bq);
            }
            const int lpr = f32 ? 8 : 4, rpi = 32 / lpr;
            const int part = lane % lpr;
            for (int it = 0; it < lpr; ++it) {
              const int rr = it * rpi + lane / lpr;
              const int64_t pr = __shfl_sync(0xffffffffu, pix, rr);
              const int vr = __shfl_sync(0xffffffffu, valid ? 1 : 0, rr);
              const uint4 w = *reinterpret_cast<const uint4*>(stg + rr * 36 + 4 * part);
              if (vr) {
                const int64_t e = pr * p.co + j * 256 + g * 32;
                if (f32)
                  *reinterpret_cast<uint4*>(reinterpret_cast<float*>(d.out) + e + 4 * part) = w;
                else
                  *reinterpret_cast<uint4*>(d.out + e + 8 * part) = w;
              }
            }
            __syncwarp();
          }
          if (kTmaOut) {
            // the four warps' rows are written: one thread stores the tile
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            epi_bar();
            if (threadIdx.x == 192) {
              tma_store_3d(&mA, tileb, j * 256, mh - row, pc);
              bulk_commit();
            }
          }
          }
        }
        tc_fence_before();
        mbar_arrive(bAccE + 8 * R);
        uses[R]++;
      }
      if constexpr (OM == CTC_LRELU_LOGIT) {
        // an image's 16 pixels are 16 consecutive rows (lanes); fixed-order tree
#pragma unroll
        for (int off = 8; off > 0; off >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, off);
        if (ok && (lane & 15) == 0 && valid) d.logits[m >> 4] = dot;
      }
    }
  }
  // the last TMA stores of the output have finished before the CTA leaves
  if (AK == AK_NCHW && OM == CTC_LRELU_HWC && p.tma_out && threadIdx.x == 192) bulk_wait_all();
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                 "r"(kTmemCols));
}

// ---- weight gradients on tcgen05 -----------------------------------------------------------
// dW[m][c][tap] = sum over pixels q of A[q][m] * B[(s qy - p + ky, s qx - p + kx)][c], A and B
// channel-last (M and Cb multiples of 64), as a GEMM with M = channels of A, N = (tap, c) and
// K = the pixels of A, split into chunks of up to 64 x 64 pixels. Both operands are MN-major:
// each gather thread writes one pixel row (128 bytes = 64 channels) of one 64-channel atom in
// the 128-byte swizzle (atoms 8 KB apart). Tiles: (problem, split, M tile of 128, N tile of
// 256); fp32 partial sums per split go to part[problem][split][M][N] in (tap, c) order.
constexpr int WG_THREADS = 320;  // warp 1 MMA, warps 2-5 gather, warps 6-9 epilogue
constexpr int WG_STAGES = 4;
// the 3-channel B operand's input patches: 3 channels x 6 rows x 72 columns (64 interior at
// column 4), three buffers
constexpr int WG_PATCH_BYTES = 2688;
constexpr int WG_SMEM =
    1024 + WG_STAGES * STAGE_BYTES + 256 + 4 * STG_WORDS * 4 + 3 * WG_PATCH_BYTES;
constexpr int WG_LAG = 2;  // copy groups a gather thread keeps in flight (< WG_STAGES)

// BCHW: p.b_chw at compile time (the 3-channel channel-major B operand)
template <bool BCHW>
__global__ void __launch_bounds__(WG_THREADS, 1)
    k_wgrad_tc(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB,
               const __grid_constant__ WgtcParams p) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* misc = smem_raw + (base - raw) + WG_STAGES * STAGE_BYTES;
  const uint32_t bars = smem_u32(misc);
  const uint32_t bFull = bars, bEmpty = bars + 8 * WG_STAGES;
  const uint32_t bAccF = bars + 16 * WG_STAGES, bAccE = bAccF + 16, bFinal = bAccE + 16;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(misc + 240);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 244);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < WG_STAGES; ++s) {
      // a_tma: the producer's expect-tx arrival (+ the 128 gather threads that build the
      // 3-channel B operand)
      mbar_init(bFull + 8 * s, !p.a_tma ? 128 : (BCHW ? 129 : 1));
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
  // b_chw: b is a 3-channel channel-major image stack, N = 48 (tap, channel) columns in one
  // 64-wide tile; M (a multiple of 64) may leave the upper half of a 128-row tile empty
  const int mt_n = (p.M + 127) / 128, nt_n = BCHW ? 1 : p.N / 256;
  const int per_split = mt_n * nt_n;
  const int la = p.la, lb = p.lb;
  const int64_t Kp = (int64_t)p.rows << (2 * la);  // pixels of A per problem
  auto split_range = [&](int split, int64_t& k0, int64_t& k1) {
    k0 = (int64_t)split * p.kc;
    k1 = k0 + p.kc < Kp ? k0 + p.kc : Kp;
  };
  const bool tma = p.a_tma;
  if (warp == 0 && tma) {
    // a_tma: both operands by TMA, MN-major rows of 64 channels: A boxes of 64 pixels from the
    // [problem][pixel][M] map, B boxes of the chunk's 64 A pixels mapped to b's pixels (s y - p
    // + ky, s x - p + kx) by the 5-D map's traversal stride
    if (lane == 0) {
      int stage = 0, issued[WG_STAGES] = {};
      uint32_t phase = 0;
      bool ok = true;
      const int Wa = 1 << la, Ha = Wa;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
        const int prob = tile / (p.splits * per_split);
        const int split = (tile / per_split) % p.splits;
        const int mt = (tile % per_split) / nt_n, nt = tile % nt_n;
        int64_t k0, k1;
        split_range(split, k0, k1);
        for (int64_t kb = k0; kb < k1; kb += 64) {
          if (!mbar_wait(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 36)) {
            ok = false;
            break;
          }
          const uint32_t full = bFull + 8 * stage;
          mbar_expect_tx(full, (uint32_t)(BCHW ? A_BYTES : STAGE_BYTES));
          const uint32_t sA = base + stage * STAGE_BYTES, sB = sA + A_BYTES;
          tma_load_3d(sA, &mA, full, mt * 128, (int)kb, prob);
          tma_load_3d(sA + 8192, &mA, full, mt * 128 + 64, (int)kb, prob);
          if constexpr (BCHW) {
            issued[stage]++;
            if (++stage == WG_STAGES) {
              stage = 0;
              phase ^= 1u;
            }
            continue;
          }
          const int nb = (int)(kb >> (2 * la));
          const int ay0 = (int)((kb >> la) & (Ha - 1)), ax0 = (int)(kb & (Wa - 1));
#pragma unroll
          for (int atom = 0; atom < 4; ++atom) {
            const int n0 = nt * 256 + atom * 64;
            const int tap = n0 / p.Cb, c0 = n0 - tap * p.Cb;
            tma_load_5d(sB + atom * 8192, &mB, full, c0, p.s * ax0 - p.p + (tap & 3),
                        p.s * ay0 - p.p + (tap >> 2), nb, prob);
          }
          issued[stage]++;
          if (++stage == WG_STAGES) {
            stage = 0;
            phase ^= 1u;
          }
        }
      }
      if (!ok) {
        for (int st2 = 0; st2 < WG_STAGES; ++st2)
          if (issued[st2] > 0) {
            volatile int never = 0;
            mbar_wait(bFull + 8 * st2, (uint32_t)((issued[st2] - 1) & 1), &never, p.err, 37);
          }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int stage = 0, uses[2] = {0, 0}, jobs = 0;
      uint32_t phase = 0;
      bool ok = true;
      const uint32_t idesc = idesc_bf16_major(128, BCHW ? 64 : 256, 1, 1);
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x, ++jobs) {
        const int split = (tile / per_split) % p.splits;
        int64_t k0, k1;
        split_range(split, k0, k1);
        const int R = jobs & 1;
        if (uses[R] > 0 &&
            !mbar_wait(bAccE + 8 * R, (uint32_t)((uses[R] - 1) & 1), abort_flag, p.err, 31)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t dt = tmem + (uint32_t)(R * 256);
        bool first = true;
        for (int64_t kb = k0; kb < k1; kb += 64) {
          if (!mbar_wait(bFull + 8 * stage, phase, abort_flag, p.err, 32)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sA = base + stage * STAGE_BYTES, sB = sA + A_BYTES;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            tc_mma(dt, sw128_mn_desc(sA + kk * 2048, 8192), sw128_mn_desc(sB + kk * 2048, 8192),
                   idesc, first ? 0u : 1u);
            first = false;
          }
          tc_commit(bEmpty + 8 * stage);
          if (++stage == WG_STAGES) {
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
      mbar_wait(bFinal, 0u, &never, p.err, 33);
    }
  } else if (warp >= 2 && warp < 6 && tma && BCHW) {
    // the 3-channel B operand with A by TMA: a chunk's 64 A pixels are two rows of the 32-wide
    // A image (first-layer geometry: b is 3 x 64 x 64, s = 2, p = 1), fed by a 3 x 6 x 64
    // patch of b that the threads copy one chunk ahead by 8-byte cp.async into one of three
    // buffers (halo columns zero); thread t builds 16-byte units 4 (t >> 6) .. + 3 of row t & 63
    const int t = threadIdx.x - 64;
    const int row = t & 63, half = t >> 6;
    const uint32_t sw = (uint32_t)(row & 7);
    uint8_t* patches = misc + 256 + 4 * STG_WORDS * 4;
    const uint32_t patch0 = smem_u32(patches);
    for (int i = t; i < 3 * WG_PATCH_BYTES / 16; i += 128)
      *reinterpret_cast<uint4*>(patches + 16 * i) = make_uint4(0u, 0u, 0u, 0u);
    gather_bar_or(false);
    // the chunks this CTA builds, in order: (tile, kb) over its tiles and their splits' chunks
    // (every split holds at least one); the patch prefetch runs one chunk ahead
    struct Chunk {
      int tile;
      int64_t kb, k1;
    };
    auto start = [&](Chunk& c, int tile_x) {
      c.tile = tile_x;
      if (tile_x < p.n_tiles) {
        int64_t k0;
        split_range((tile_x / per_split) % p.splits, k0, c.k1);
        c.kb = k0;
      }
    };
    auto advance = [&](Chunk& c) {
      c.kb += 64;
      if (c.kb >= c.k1) start(c, c.tile + gridDim.x);
    };
    auto prefetch = [&](int tile_x, int64_t kb_x, int buf) {
      if (tile_x < p.n_tiles) {
        const WgtcDesc dx = p.descs[tile_x / (p.splits * per_split)];
        const int nb = (int)(kb_x >> 10), ay0 = (int)((kb_x >> 5) & 31);
        for (int u = t; u < 288; u += 128) {  // 3 channels x 6 rows x 16 pieces of 4
          const int c = u / 96, rem = u - c * 96, pr = rem >> 4, qq = rem & 15;
          const int iy = 2 * ay0 - 1 + pr;
          const bool in = iy >= 0 && iy < 64;
          const bf16* src = in ? dx.b + ((int64_t)(nb * 3 + c) << 12) + (iy << 6) + 4 * qq : dx.b;
          cp_async8(patch0 +
                        (uint32_t)(buf * WG_PATCH_BYTES + ((c * 6 + pr) * 72 + 4 + 4 * qq) * 2),
                    src, in ? 8 : 0);
        }
      }
      asm volatile("cp.async.commit_group;" ::: "memory");
    };
    Chunk cur, nxt;
    start(cur, blockIdx.x);
    nxt = cur;
    prefetch(cur.tile, cur.kb, 0);
    int buf = 0, stage = 0;
    uint32_t phase = 0;
    while (cur.tile < p.n_tiles) {
      advance(nxt);
      prefetch(nxt.tile, nxt.kb, buf == 2 ? 0 : buf + 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
      const bool okw = mbar_wait_warp(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 38);
      if (gather_bar_or(!okw)) break;
      const bool qv = cur.kb + row < cur.k1;
      const int ayl = row >> 5, ax = row & 31;
      const unsigned short* pb =
          reinterpret_cast<const unsigned short*>(patches + buf * WG_PATCH_BYTES);
      const uint32_t sB = base + stage * STAGE_BYTES + A_BYTES;
#pragma unroll
      for (int uu = 0; uu < 4; ++uu) {
        const int u = half * 4 + uu;
        uint32_t w[4];
#pragma unroll
        for (int e2 = 0; e2 < 4; ++e2) {
          uint32_t hv[2];
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int k = u * 8 + e2 * 2 + h;  // k = tap * 3 + c
            hv[h] = 0u;
            if (k < 48 && qv) {
              const int tap = k / 3, c = k - 3 * tap;
              hv[h] = pb[(c * 6 + 2 * ayl + (tap >> 2)) * 72 + 2 * ax + (tap & 3) + 3];
            }
          }
          w[e2] = hv[0] | (hv[1] << 16);
        }
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                         sB + (uint32_t)row * 128u + (((uint32_t)u ^ sw) << 4)),
                     "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3])
                     : "memory");
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_arrive(bFull + 8 * stage);
      if (++stage == WG_STAGES) {
        stage = 0;
        phase ^= 1u;
      }
      buf = buf == 2 ? 0 : buf + 1;
      cur = nxt;
    }
    asm volatile("cp.async.wait_group 0;" ::: "memory");
  } else if (warp >= 2 && warp < 6 && !tma) {
    // gather: thread t copies pixel row (t & 63) of A atom (t >> 6) and of B atoms 2 (t >> 6),
    // 2 (t >> 6) + 1 with 16-byte cp.async (zero fill outside the image); a stage is marked
    // full WG_LAG chunks later, once its copy group has landed
    const int t = threadIdx.x - 64;
    const int row = t & 63, half = t >> 6;
    const uint32_t sw = (uint32_t)(row & 7);
    int stage = 0, arr_stage = 0, pending = 0;
    uint32_t phase = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
      const int prob = tile / (p.splits * per_split);
      const int split = (tile / per_split) % p.splits;
      const int mt = (tile % per_split) / nt_n, nt = tile % nt_n;
      const WgtcDesc d = p.descs[prob];
      int64_t k0, k1;
      split_range(split, k0, k1);
      for (int64_t kb = k0; kb < k1; kb += 64) {
        if (!mbar_wait_warp(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 34)) {
          ok = false;
          break;
        }
        const uint32_t sA = base + stage * STAGE_BYTES, sB = sA + A_BYTES;
        const int64_t q = kb + row;  // pixel of A
        const bool qv = q < k1;
        const int nb = (int)(q >> (2 * la));
        const int ay = (int)((q >> la) & ((1 << la) - 1)), ax = (int)(q & ((1 << la) - 1));
        {
          const bool av = qv && mt * 128 + half * 64 < p.M;
          const bf16* src = av ? d.a + q * p.M + mt * 128 + half * 64 : d.a;
          const uint32_t dst = sA + (uint32_t)half * 8192u + (uint32_t)row * 128u;
#pragma unroll
          for (int u = 0; u < 8; ++u)
            cp_async16(dst + (((uint32_t)u ^ sw) << 4), src + (av ? 8 * u : 0), av ? 16 : 0);
        }
        if constexpr (BCHW) {
          // row `row` of the single B atom, columns k = tap * 3 + c (k < 48, zero above);
          // thread half h writes the 16-byte units 4h .. 4h + 3 (k = 32h .. 32h + 31)
#pragma unroll
          for (int uu = 0; uu < 4; ++uu) {
            const int u = half * 4 + uu;
            uint32_t w[4];
#pragma unroll
            for (int e2 = 0; e2 < 4; ++e2) {
              uint32_t hv[2];
#pragma unroll
              for (int h = 0; h < 2; ++h) {
                const int k = u * 8 + e2 * 2 + h;
                hv[h] = 0u;
                if (k < 48 && qv) {
                  const int tap = k / 3, c = k - 3 * tap;
                  const int by = ay * p.s - p.p + (tap >> 2), bx = ax * p.s - p.p + (tap & 3);
                  if (by >= 0 && by < (1 << lb) && bx >= 0 && bx < (1 << lb))
                    hv[h] = (uint32_t)__bfloat16_as_ushort(
                        d.b[((int64_t)(nb * 3 + c) << (2 * lb)) + (by << lb) + bx]);
                }
              }
              w[e2] = hv[0] | (hv[1] << 16);
            }
            asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                             sB + (uint32_t)row * 128u + (((uint32_t)u ^ sw) << 4)),
                         "r"(w[0]), "r"(w[1]), "r"(w[2]), "r"(w[3])
                         : "memory");
          }
        } else
#pragma unroll
        for (int aa = 0; aa < 2; ++aa) {
          const int atom = 2 * half + aa;
          const int n0 = nt * 256 + atom * 64;
          const int tap = n0 / p.Cb, c0 = n0 - tap * p.Cb;
          const int by = ay * p.s - p.p + (tap >> 2), bx = ax * p.s - p.p + (tap & 3);
          const bool in = qv && by >= 0 && by < (1 << lb) && bx >= 0 && bx < (1 << lb);
          const bf16* src =
              in ? d.b + ((((int64_t)nb << (2 * lb)) + (by << lb) + bx) * p.Cb + c0) : d.b;
          const uint32_t dst = sB + (uint32_t)atom * 8192u + (uint32_t)row * 128u;
#pragma unroll
          for (int u = 0; u < 8; ++u)
            cp_async16(dst + (((uint32_t)u ^ sw) << 4), src + (in ? 8 * u : 0), in ? 16 : 0);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
        if (++pending > WG_LAG) {
          asm volatile("cp.async.wait_group %0;" ::"n"(WG_LAG) : "memory");
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          mbar_arrive(bFull + 8 * arr_stage);
          arr_stage = arr_stage + 1 == WG_STAGES ? 0 : arr_stage + 1;
          --pending;
        }
        if (++stage == WG_STAGES) {
          stage = 0;
          phase ^= 1u;
        }
      }
    }
    // the last chunks (and, after an expired wait, every copy still in flight)
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    for (; pending > 0; --pending) {
      mbar_arrive(bFull + 8 * arr_stage);
      arr_stage = arr_stage + 1 == WG_STAGES ? 0 : arr_stage + 1;
    }
  } else if (warp >= 6) {
    // epilogue: row m of the tile, 256 columns in groups of 32, fp32 partial sums, staged in
    // shared memory and stored as whole rows (eight lanes per 128-byte row piece)
    const int q4 = warp & 3;
    const int r = q4 * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q4 * 32) << 16;
    uint32_t* stg = reinterpret_cast<uint32_t*>(misc + 256) + (warp - 6) * STG_WORDS;
    int uses[2] = {0, 0}, jobs = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x, ++jobs) {
      const int prob = tile / (p.splits * per_split);
      const int split = (tile / per_split) % p.splits;
      const int mt = (tile % per_split) / nt_n, nt = tile % nt_n;
      const int R = jobs & 1;
      if (!mbar_wait_warp(bAccF + 8 * R, (uint32_t)(uses[R] & 1), abort_flag, p.err, 35)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float* o = p.part + (((int64_t)prob * p.splits + split) * p.M + mt * 128 + r) * p.N +
                 nt * 256;
      constexpr int groups = BCHW ? 2 : 8;
      for (int g = 0; g < groups; ++g) {
        uint32_t v[32];
        LIPZ_TMEM_LD32(tmem + lane_base + (uint32_t)(R * 256 + g * 32), v);
        tmem_wait_ld();
#pragma unroll
        for (int u = 0; u < 8; ++u)
          *reinterpret_cast<uint4*>(stg + lane * 36 + 4 * u) =
              make_uint4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
        __syncwarp();
        for (int it = 0; it < 8; ++it) {
          const int rr = it * 4 + (lane >> 3), part = lane & 7;
          const uint4 w = *reinterpret_cast<const uint4*>(stg + rr * 36 + 4 * part);
          if (mt * 128 + q4 * 32 + rr < p.M)
            *reinterpret_cast<uint4*>(o + (int64_t)(rr - lane) * p.N + g * 32 + 4 * part) = w;
        }
        __syncwarp();
      }
      tc_fence_before();
      mbar_arrive(bAccE + 8 * R);
      uses[R]++;
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
}

// Scatter mode: the output rows 8k - 1 and 8k of every image are shared by row blocks k - 1
// and k (their halo rows 2, 3 and 0, 1); add them in that order and apply the epilogue (tanh,
// or the delta times 1 - f^2). Grid: (problem x image); 64 x 64 x 3 outputs per image.
__global__ void __launch_bounds__(256) k_scatter_fix(const ConvTcDesc* __restrict__ descs,
                                                     const float* __restrict__ halo, int rows,
                                                     int out_mode) {
  pdl_wait();
  const int pi = blockIdx.x;  // problem * rows + image
  const ConvTcDesc d = descs[pi / rows];
  const int img = pi % rows;
  const float* h = halo + (int64_t)pi * 8 * 768;
  // element i: column gx = i mod 64 (neighbouring threads write neighbouring columns), then
  // channel o, then halo row t and block boundary k
  for (int i = threadIdx.x; i < 9 * 2 * 64 * 3; i += 256) {
    const int gx = i & 63, r = i >> 6;  // r = (k * 2 + t) * 3 + o
    const int kt = r / 3, o = r - 3 * kt, k = kt >> 1, t = kt & 1;
    const int gy = 8 * k - 1 + t;
    if (gy < 0 || gy > 63) continue;
    float x = 0.f;
    if (k > 0) x += h[(k - 1) * 768 + (2 + t) * 192 + gx * 3 + o];
    if (k < 8) x += h[k * 768 + t * 192 + gx * 3 + o];
    const int64_t oi = (((int64_t)img * 3 + o) << 12) + (gy << 6) + gx;
    if (out_mode == CTC_TANH_CHW) {
      x = tanhf(x);
    } else {
      const float f = __bfloat162float(d.aux[oi]);
      x = x * (1.f - f * f);
    }
    d.out[oi] = __float2bfloat16_rn(x);
  }
}

// Scatter-mode weights of a 4x4 transposed convolution to 3 channels: src [k][3][16] (64
// input channels k, 3 outputs j, 16 taps) of every individual -> dst [tap * 4 + j][k] (64 x 64,
// row j = 3 zero).
__global__ void k_relayout_s(const bf16* __restrict__ src, int64_t src_ps, int64_t src_off,
                             bf16* __restrict__ dst) {
  pdl_wait();
  const int64_t ind = blockIdx.y;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < 4096; e += gridDim.x * blockDim.x) {
    const int n = e >> 6, k = e & 63, tap = n >> 2, j = n & 3;
    dst[ind * 4096 + e] =
        j < 3 ? src[ind * src_ps + src_off + (k * 3 + j) * 16 + tap] : __float2bfloat16_rn(0.f);
  }
}

// b_chw: part[problem][split][m][tap * 3 + c] (64 columns) -> dW[m][c][tap], summed over the
// splits in order.
__global__ void __launch_bounds__(256) k_wgrad_tc_reduce_chw(const __grid_constant__ WgtcParams p) {
  pdl_wait();
  const int prob = blockIdx.y;
  const int64_t MN = (int64_t)p.M * p.N;
  const float* part = p.part + (int64_t)prob * p.splits * MN;
  float* out = p.descs[prob].dw;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < p.M * 48; e += gridDim.x * blockDim.x) {
    const int m = e / 48, j = e - m * 48;  // j = c * 16 + tap
    const int64_t src = (int64_t)m * p.N + (j & 15) * 3 + (j >> 4);
    float acc = 0.f;
    for (int sp = 0; sp < p.splits; ++sp) acc += part[sp * MN + src];
    out[e] = acc;
  }
}

// part[problem][split][m][(tap, c)] -> dW[m][c][tap], summed over the splits in order; a
// block turns one row m and 64 channels through shared memory (grid: M * Cb / 64, problems).
__global__ void __launch_bounds__(256) k_wgrad_tc_reduce(const __grid_constant__ WgtcParams p) {
  __shared__ float tile[16][65];
  pdl_wait();
  const int prob = blockIdx.y;
  const int cchunks = p.Cb / 64;
  const int m = blockIdx.x / cchunks, c0 = (blockIdx.x - m * cchunks) * 64;
  const int64_t MN = (int64_t)p.M * p.N;
  const float* part = p.part + (int64_t)prob * p.splits * MN + (int64_t)m * p.N + c0;
  // the four outputs of a thread, each summed over the splits in split order, with all four
  // loads of a split issued together
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int sp = 0; sp < p.splits; ++sp) {
    float v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int i = threadIdx.x + 256 * u;
      v[u] = part[(int64_t)sp * MN + (int64_t)(i >> 6) * p.Cb + (i & 63)];
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) acc[u] += v[u];
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int i = threadIdx.x + 256 * u;
    tile[i >> 6][i & 63] = acc[u];
  }
  __syncthreads();
  float* out = p.descs[prob].dw + (int64_t)m * p.N + (int64_t)c0 * 16;
  for (int i = threadIdx.x; i < 1024; i += 256) out[i] = tile[i & 15][i >> 4];
}

// Weight re-layouts, one block per (output row of one tensor, individual); channels pass
// through shared memory in chunks of RL_CH so that reads and writes are contiguous runs.
constexpr int RL_CH = 256;
struct RelayoutRows {
  int n;
  int64_t src_off[5], dst_off[5];
  int o[5], c[5];
};

// [o][c][ky][kx] -> [o][ky][kx][c]
__global__ void __launch_bounds__(256) k_relayout_rows(const bf16* __restrict__ src, int64_t src_ps,
                                                       bf16* __restrict__ dst, int64_t dst_ps,
                                                       RelayoutRows r) {
  __shared__ bf16 sh[16][RL_CH + 2];
  pdl_wait();
  int row = blockIdx.x, l = 0;
  while (l + 1 < r.n && row >= r.o[l]) row -= r.o[l++];
  const int c = r.c[l];
  const bf16* sp = src + blockIdx.y * src_ps + r.src_off[l] + (int64_t)row * c * 16;
  bf16* dp = dst + blockIdx.y * dst_ps + r.dst_off[l] + (int64_t)row * c * 16;
  for (int cb = 0; cb < c; cb += RL_CH) {
    const int n = c - cb < RL_CH ? c - cb : RL_CH;
    for (int e = threadIdx.x; e < n * 16; e += 256) sh[e & 15][e >> 4] = sp[cb * 16 + e];
    __syncthreads();
    // (the channel counts are powers of two: a shift instead of a division where they are)
    const bool pow2 = (n & (n - 1)) == 0;
    const int ln = __ffs(n) - 1;
    for (int e = threadIdx.x; e < n * 16; e += 256) {
      const int t = pow2 ? e >> ln : e / n, cc = e - t * n;
      dp[t * c + cb + cc] = sh[t][cc];
    }
    __syncthreads();
  }
}

// Generator transposed-convolution weights [in][out][ky][kx] -> by output parity class
// [class][out][tap][in] (tap (u, v): ky = (py + 1) mod 2 + 2u, kx = (px + 1) mod 2 + 2v), rows
// of a class cls_rows apart (the padding rows are left as they are: zero). One block per
// (output channel o of one tensor, individual).
__global__ void __launch_bounds__(256) k_relayout_g(const bf16* __restrict__ src, int64_t src_ps,
                                                    bf16* __restrict__ dst, int64_t dst_ps,
                                                    RelayoutG r) {
  __shared__ bf16 sh[16][RL_CH + 2];
  pdl_wait();
  int o = blockIdx.x, l = 0;
  while (l + 1 < r.n && o >= r.co[l]) o -= r.co[l++];
  const int ci = r.ci[l], co = r.co[l];
  const bf16* sp = src + blockIdx.y * src_ps + r.src_off[l] + (int64_t)o * 16;
  bf16* dp = dst + blockIdx.y * dst_ps + r.dst_off[l];
  for (int cb = 0; cb < ci; cb += RL_CH) {
    const int n = ci - cb < RL_CH ? ci - cb : RL_CH;
    for (int e = threadIdx.x; e < n * 16; e += 256)
      sh[e & 15][e >> 4] = sp[(int64_t)(cb + (e >> 4)) * co * 16 + (e & 15)];
    __syncthreads();
    const bool pow2 = (n & (n - 1)) == 0;
    const int ln = __ffs(n) - 1;
    for (int e = threadIdx.x; e < n * 16; e += 256) {
      const int ct = pow2 ? e >> ln : e / n, cc = e - ct * n;  // (class, tap) = ct
      const int cls = ct >> 2, t = ct & 3;
      const int ky = (((cls >> 1) + 1) & 1) + 2 * (t >> 1);
      const int kx = (((cls & 1) + 1) & 1) + 2 * (t & 1);
      dp[(((int64_t)cls * r.cls_rows[l] + o) * 4 + t) * ci + cb + cc] = sh[ky * 4 + kx][cc];
    }
    __syncthreads();
  }
}

// Training-mode batch normalisation + ReLU on channel-last data, in two launches over blocks
// (group of 32 channels, problem, pixel chunk): each stats block sums its chunk's values and
// squares per channel (lane = channel, warps over pixels, fixed order) into
// part[problem][chunk]; the last block of a (channel group, problem) to finish combines the
// chunks' sums in float64 in chunk order (mean, and the variance as E[x^2] - mean^2) into the
// descriptor's mean and inverse deviation. The apply blocks normalise, add the shift, apply
// ReLU and round to bf16.
constexpr int BN_CHUNKS = 32;

__global__ void __launch_bounds__(256) k_bn_stats_hwc(const BnDesc* __restrict__ descs,
                                                      float2* __restrict__ part, int cmax,
                                                      unsigned* __restrict__ counters) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int lane = threadIdx.x & 31;
  const int ch = blockIdx.x * 32 + lane;
  const int w = threadIdx.x >> 5;
  const int64_t m = (int64_t)d.n << d.lhw;
  const int64_t p0 = m * blockIdx.z / BN_CHUNKS, p1 = m * (blockIdx.z + 1) / BN_CHUNKS;
  __shared__ float sh[8][32][2];
  __shared__ int is_last;
  float s = 0.f, q = 0.f;
  if (ch < d.C) {
    int64_t px = p0 + w;
    for (; px + 24 < p1; px += 32) {
      float v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = d.c[(px + 8 * u) * d.C + ch];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        s += v[u];
        q = fmaf(v[u], v[u], q);
      }
    }
    for (; px < p1; px += 8) {
      const float v = d.c[px * d.C + ch];
      s += v;
      q = fmaf(v, v, q);
    }
  }
  sh[w][lane][0] = s;
  sh[w][lane][1] = q;
  __syncthreads();
  float2* pp = part + (int64_t)blockIdx.y * BN_CHUNKS * cmax;
  if (w == 0 && ch < d.C) {
    float ts = 0.f, tq = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      ts += sh[i][lane][0];
      tq += sh[i][lane][1];
    }
    pp[(int64_t)blockIdx.z * cmax + ch] = make_float2(ts, tq);
  }
  __threadfence();
  __syncthreads();
  unsigned* cnt = counters + (int64_t)blockIdx.y * gridDim.x + blockIdx.x;
  if (threadIdx.x == 0) is_last = atomicAdd(cnt, 1u) == BN_CHUNKS - 1;
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  if (w == 0 && ch < d.C) {
    double ts = 0.0, tq = 0.0;
    for (int z = 0; z < BN_CHUNKS; ++z) {
      const float2 v = __ldcg(&pp[(int64_t)z * cmax + ch]);
      ts += v.x;
      tq += v.y;
    }
    const double mean_d = ts / (double)m;
    const double var_d = fmax(tq / (double)m - mean_d * mean_d, 0.0);
    d.mean[ch] = (float)mean_d;
    d.inv[ch] = rsqrtf((float)var_d + 1e-5f);
  }
  if (threadIdx.x == 0) *cnt = 0u;
}

// The statistics when the producing convolution summed them (CtcParams::bn_part): problem pr
// owns slots [pr T, (pr + 1) T) of part ([slot][C] float2: sum, sum of squares over one lane
// quarter's rows of one tile). Warp w of the 32 takes slots w, w + 32, ... (four loads in
// flight, float sums in slot order); warp 0 adds the 32 warp sums in float64 in warp order.
__global__ void __launch_bounds__(1024) k_bn_finalize_hwc(const BnDesc* __restrict__ descs,
                                                          const float2* __restrict__ part, int T) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int ch = blockIdx.x * 32 + lane;
  __shared__ float sh[32][32][2];
  float s = 0.f, q = 0.f;
  if (ch < d.C) {
    const float2* pp = part + (int64_t)blockIdx.y * T * d.C + ch;
    int t = w;
    for (; t + 96 < T; t += 128) {
      float2 v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = pp[(int64_t)(t + 32 * u) * d.C];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        s += v[u].x;
        q += v[u].y;
      }
    }
    for (; t < T; t += 32) {
      const float2 v = pp[(int64_t)t * d.C];
      s += v.x;
      q += v.y;
    }
  }
  sh[w][lane][0] = s;
  sh[w][lane][1] = q;
  __syncthreads();
  if (w == 0 && ch < d.C) {
    double ts = 0.0, tq = 0.0;
    for (int i = 0; i < 32; ++i) {
      ts += sh[i][lane][0];
      tq += sh[i][lane][1];
    }
    const double m = (double)((int64_t)d.n << d.lhw);
    const double mean_d = ts / m;
    const double var_d = fmax(tq / m - mean_d * mean_d, 0.0);
    d.mean[ch] = (float)mean_d;
    d.inv[ch] = rsqrtf((float)var_d + 1e-5f);
  }
}

__global__ void __launch_bounds__(256) k_bn_apply_hwc(const BnDesc* __restrict__ descs,
                                                      const int* __restrict__ wsel_override) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int ch = blockIdx.x * 32 + (threadIdx.x & 31);
  const int w = threadIdx.x >> 5;
  if (ch >= d.C) return;
  const int64_t m = (int64_t)d.n << d.lhw;
  const float mean = d.mean[ch], inv = d.inv[ch];
  const int* ws = wsel_override ? wsel_override : d.wsel;
  const float* P = d.params + (ws ? (int64_t)ws[d.wsel_idx] * d.wsel_stride : 0);
  const float sc = P[d.off_gamma + ch] * inv, b = P[d.off_beta + ch];
  bf16* h = (bf16*)d.h;
  const int64_t p0 = m * blockIdx.z / BN_CHUNKS, p1 = m * (blockIdx.z + 1) / BN_CHUNKS;
  int64_t px = p0 + w;
  for (; px + 24 < p1; px += 32) {
    float v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) v[u] = d.c[(px + 8 * u) * d.C + ch];
#pragma unroll
    for (int u = 0; u < 4; ++u)
      h[(px + 8 * u) * d.C + ch] = __float2bfloat16_rn(fmaxf(fmaf(sc, v[u] - mean, b), 0.f));
  }
  for (; px < p1; px += 8)
    h[px * d.C + ch] = __float2bfloat16_rn(fmaxf(fmaf(sc, d.c[px * d.C + ch] - mean, b), 0.f));
}

// The apply pass with four channels per thread (C a multiple of 4, at most 1024): 16-byte
// loads of the fp32 input and 8-byte stores of the bf16 output, whole rows per warp; block z
// of a problem takes elements [z E, (z + 1) E) with E = BN_APPLY_ELEMS. Same arithmetic as
// k_bn_apply_hwc.
constexpr int BN_APPLY_ELEMS = 32768;
__global__ void __launch_bounds__(256) k_bn_apply_hwc4(const BnDesc* __restrict__ descs,
                                                       const int* __restrict__ wsel_override) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int nq = d.C >> 2;
  const int64_t total = ((int64_t)d.n << d.lhw) * d.C;
  const int64_t e0 = (int64_t)blockIdx.x * BN_APPLY_ELEMS;
  if (e0 >= total) return;
  const int64_t e1 = min(total, e0 + (int64_t)BN_APPLY_ELEMS);
  // this thread's channel quad is fixed: the step (1024 elements) is a multiple of C
  const int64_t first = e0 + 4 * threadIdx.x;
  const int c0 = (int)((first >> 2) % nq) * 4;
  const int* ws = wsel_override ? wsel_override : d.wsel;
  const float* P = d.params + (ws ? (int64_t)ws[d.wsel_idx] * d.wsel_stride : 0);
  float mean[4], sc[4], b[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    mean[u] = d.mean[c0 + u];
    sc[u] = P[d.off_gamma + c0 + u] * d.inv[c0 + u];
    b[u] = P[d.off_beta + c0 + u];
  }
  const float4* x = reinterpret_cast<const float4*>(d.c);
  uint2* h = reinterpret_cast<uint2*>(d.h);
  int64_t e = first;
  for (; e + 3 * 1024 < e1; e += 4 * 1024) {
    float4 v[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) v[k] = x[(e + k * 1024) >> 2];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float a0 = fmaxf(fmaf(sc[0], v[k].x - mean[0], b[0]), 0.f);
      const float a1 = fmaxf(fmaf(sc[1], v[k].y - mean[1], b[1]), 0.f);
      const float a2 = fmaxf(fmaf(sc[2], v[k].z - mean[2], b[2]), 0.f);
      const float a3 = fmaxf(fmaf(sc[3], v[k].w - mean[3], b[3]), 0.f);
      h[(e + k * 1024) >> 2] = make_uint2(pack_bf16(a0, a1), pack_bf16(a2, a3));
    }
  }
  for (; e < e1; e += 1024) {
    const float4 v = x[e >> 2];
    const float a0 = fmaxf(fmaf(sc[0], v.x - mean[0], b[0]), 0.f);
    const float a1 = fmaxf(fmaf(sc[1], v.y - mean[1], b[1]), 0.f);
    const float a2 = fmaxf(fmaf(sc[2], v.z - mean[2], b[2]), 0.f);
    const float a3 = fmaxf(fmaf(sc[3], v.w - mean[3], b[3]), 0.f);
    h[e >> 2] = make_uint2(pack_bf16(a0, a1), pack_bf16(a2, a3));
  }
}

// Backward through ReLU and the batch normalisation on channel-last bf16 activations, same
// block layout as the forward: dy = dh where h > 0, xhat = (c - mean) inv; the stats blocks
// sum dy and dy xhat per channel and chunk, the last block of a (channel group, problem)
// combines the chunks in float64 in chunk order into dbeta and dgamma (the gradient slots);
// the apply blocks write dc = gamma inv (dy - dbeta / m - xhat dgamma / m) in bf16.
__global__ void __launch_bounds__(256) k_bn_back_stats_hwc(const BnDesc* __restrict__ descs,
                                                           float2* __restrict__ part, int cmax,
                                                           unsigned* __restrict__ counters) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int lane = threadIdx.x & 31;
  const int ch = blockIdx.x * 32 + lane;
  const int w = threadIdx.x >> 5;
  const int64_t m = (int64_t)d.n << d.lhw;
  const int64_t p0 = m * blockIdx.z / BN_CHUNKS, p1 = m * (blockIdx.z + 1) / BN_CHUNKS;
  __shared__ float sh[8][32][2];
  __shared__ int is_last;
  const bf16* h = (const bf16*)d.h;
  float sb = 0.f, sg = 0.f;
  if (ch < d.C) {
    const float mean = d.mean[ch], inv = d.inv[ch];
    int64_t px = p0 + w;
    for (; px + 24 < p1; px += 32) {
      float hv[4], dv[4], cv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int64_t o = (px + 8 * u) * d.C + ch;
        hv[u] = __bfloat162float(h[o]);
        dv[u] = d.dh[o];
        cv[u] = d.c[o];
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const float dy = hv[u] > 0.f ? dv[u] : 0.f;
        sb += dy;
        sg = fmaf(dy, (cv[u] - mean) * inv, sg);
      }
    }
    for (; px < p1; px += 8) {
      const int64_t o = px * d.C + ch;
      const float dy = __bfloat162float(h[o]) > 0.f ? d.dh[o] : 0.f;
      sb += dy;
      sg = fmaf(dy, (d.c[o] - mean) * inv, sg);
    }
  }
  sh[w][lane][0] = sb;
  sh[w][lane][1] = sg;
  __syncthreads();
  float2* pp = part + (int64_t)blockIdx.y * BN_CHUNKS * cmax;
  if (w == 0 && ch < d.C) {
    float tb = 0.f, tg = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      tb += sh[i][lane][0];
      tg += sh[i][lane][1];
    }
    pp[(int64_t)blockIdx.z * cmax + ch] = make_float2(tb, tg);
  }
  __threadfence();
  __syncthreads();
  unsigned* cnt = counters + (int64_t)blockIdx.y * gridDim.x + blockIdx.x;
  if (threadIdx.x == 0) is_last = atomicAdd(cnt, 1u) == BN_CHUNKS - 1;
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  if (w == 0 && ch < d.C) {
    double tb = 0.0, tg = 0.0;
    for (int z = 0; z < BN_CHUNKS; ++z) {
      const float2 v = __ldcg(&pp[(int64_t)z * cmax + ch]);
      tb += v.x;
      tg += v.y;
    }
    d.dparams[d.off_gamma + ch] = (float)tg;
    d.dparams[d.off_beta + ch] = (float)tb;
  }
  if (threadIdx.x == 0) *cnt = 0u;
}

__global__ void __launch_bounds__(256) k_bn_back_apply_hwc(const BnDesc* __restrict__ descs) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int ch = blockIdx.x * 32 + (threadIdx.x & 31);
  const int w = threadIdx.x >> 5;
  if (ch >= d.C) return;
  const int64_t m = (int64_t)d.n << d.lhw;
  const float mean = d.mean[ch], inv = d.inv[ch];
  const float* P = d.params + (d.wsel ? (int64_t)d.wsel[d.wsel_idx] * d.wsel_stride : 0);
  const float gi = P[d.off_gamma + ch] * inv;
  const float k1 = d.dparams[d.off_beta + ch] / (float)m;
  const float k2 = d.dparams[d.off_gamma + ch] / (float)m;
  const bf16* h = (const bf16*)d.h;
  bf16* dc = (bf16*)d.dc;
  const int64_t p0 = m * blockIdx.z / BN_CHUNKS, p1 = m * (blockIdx.z + 1) / BN_CHUNKS;
  int64_t px = p0 + w;
  for (; px + 24 < p1; px += 32) {
    float hv[4], dv[4], cv[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t o = (px + 8 * u) * d.C + ch;
      hv[u] = __bfloat162float(h[o]);
      dv[u] = d.dh[o];
      cv[u] = d.c[o];
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float dy = hv[u] > 0.f ? dv[u] : 0.f;
      dc[(px + 8 * u) * d.C + ch] = __float2bfloat16_rn(gi * (dy - k1 - (cv[u] - mean) * inv * k2));
    }
  }
  for (; px < p1; px += 8) {
    const int64_t o = px * d.C + ch;
    const float dy = __bfloat162float(h[o]) > 0.f ? d.dh[o] : 0.f;
    dc[o] = __float2bfloat16_rn(gi * (dy - k1 - (d.c[o] - mean) * inv * k2));
  }
}

// The backward passes with four channels per thread (C a multiple of 4 dividing 1024), 1024
// threads per block, blocks over 4096-element steps: the stats block z of a problem takes steps
// [S z / 32, S (z + 1) / 32) (S = steps of the problem; the last block also the tail), its
// threads of one channel quad are added in thread order into part[problem][z][C], and the
// problem's last block adds the 32 chunks in float64 in chunk order (one counter per problem).
constexpr int BN_B_THREADS = 1024;
__global__ void __launch_bounds__(BN_B_THREADS) k_bn_back_stats_hwc4(
    const BnDesc* __restrict__ descs, float2* __restrict__ part, int cmax,
    unsigned* __restrict__ counters) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int nq = d.C >> 2;
  const int64_t m = (int64_t)d.n << d.lhw;
  const int64_t total = m * d.C, steps = total / 4096;
  const int z = blockIdx.x;
  int64_t e = (steps * z / BN_CHUNKS) * 4096 + 4 * threadIdx.x;
  const int64_t e1 = z == BN_CHUNKS - 1 ? total : (steps * (z + 1) / BN_CHUNKS) * 4096;
  const int c0 = (4 * threadIdx.x) % d.C;
  float mean[4], inv[4], sb[4] = {0.f, 0.f, 0.f, 0.f}, sg[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    mean[u] = d.mean[c0 + u];
    inv[u] = d.inv[c0 + u];
  }
  const uint2* h = reinterpret_cast<const uint2*>(d.h);
  const float4* dh = reinterpret_cast<const float4*>(d.dh);
  const float4* cc = reinterpret_cast<const float4*>(d.c);
  for (; e < e1; e += 4096) {
    const uint2 hv = h[e >> 2];
    const float4 dv = dh[e >> 2], cv = cc[e >> 2];
    const float2 h01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&hv.x));
    const float2 h23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&hv.y));
    const float hq[4] = {h01.x, h01.y, h23.x, h23.y};
    const float dq[4] = {dv.x, dv.y, dv.z, dv.w}, cq[4] = {cv.x, cv.y, cv.z, cv.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float dy = hq[u] > 0.f ? dq[u] : 0.f;
      sb[u] += dy;
      sg[u] = fmaf(dy, (cq[u] - mean[u]) * inv[u], sg[u]);
    }
  }
  __shared__ float4 shb[BN_B_THREADS], shg[BN_B_THREADS];
  __shared__ int is_last;
  shb[threadIdx.x] = make_float4(sb[0], sb[1], sb[2], sb[3]);
  shg[threadIdx.x] = make_float4(sg[0], sg[1], sg[2], sg[3]);
  __syncthreads();
  float2* pp = part + (int64_t)blockIdx.y * BN_CHUNKS * cmax;
  if ((int)threadIdx.x < nq) {
    float4 tb = make_float4(0.f, 0.f, 0.f, 0.f), tg = tb;
    for (int t = threadIdx.x; t < BN_B_THREADS; t += nq) {
      const float4 b = shb[t], g = shg[t];
      tb.x += b.x; tb.y += b.y; tb.z += b.z; tb.w += b.w;
      tg.x += g.x; tg.y += g.y; tg.z += g.z; tg.w += g.w;
    }
    float2* o = pp + (int64_t)z * cmax + 4 * threadIdx.x;
    o[0] = make_float2(tb.x, tg.x);
    o[1] = make_float2(tb.y, tg.y);
    o[2] = make_float2(tb.z, tg.z);
    o[3] = make_float2(tb.w, tg.w);
  }
  __threadfence();
  __syncthreads();
  unsigned* cnt = counters + blockIdx.y;
  if (threadIdx.x == 0) is_last = atomicAdd(cnt, 1u) == BN_CHUNKS - 1;
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  for (int ch = threadIdx.x; ch < d.C; ch += BN_B_THREADS) {
    double tb = 0.0, tg = 0.0;
    for (int k = 0; k < BN_CHUNKS; ++k) {
      const float2 v = __ldcg(&pp[(int64_t)k * cmax + ch]);
      tb += v.x;
      tg += v.y;
    }
    d.dparams[d.off_gamma + ch] = (float)tg;
    d.dparams[d.off_beta + ch] = (float)tb;
  }
  if (threadIdx.x == 0) *cnt = 0u;
}

// dc = gamma inv (dy - dbeta / m - xhat dgamma / m), four channels per thread, as
// k_bn_back_apply_hwc; blocks over BN_APPLY_ELEMS elements as k_bn_apply_hwc4.
__global__ void __launch_bounds__(256) k_bn_back_apply_hwc4(const BnDesc* __restrict__ descs) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int64_t m = (int64_t)d.n << d.lhw;
  const int64_t total = m * d.C;
  const int64_t e0 = (int64_t)blockIdx.x * BN_APPLY_ELEMS;
  if (e0 >= total) return;
  const int64_t e1 = min(total, e0 + (int64_t)BN_APPLY_ELEMS);
  const int64_t first = e0 + 4 * threadIdx.x;
  const int c0 = (int)(first % d.C);
  const float* P = d.params + (d.wsel ? (int64_t)d.wsel[d.wsel_idx] * d.wsel_stride : 0);
  float mean[4], inv[4], gi[4], k1[4], k2[4];
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    mean[u] = d.mean[c0 + u];
    inv[u] = d.inv[c0 + u];
    gi[u] = P[d.off_gamma + c0 + u] * inv[u];
    k1[u] = d.dparams[d.off_beta + c0 + u] / (float)m;
    k2[u] = d.dparams[d.off_gamma + c0 + u] / (float)m;
  }
  const uint2* h = reinterpret_cast<const uint2*>(d.h);
  const float4* dh = reinterpret_cast<const float4*>(d.dh);
  const float4* cc = reinterpret_cast<const float4*>(d.c);
  uint2* dc = reinterpret_cast<uint2*>(d.dc);
  for (int64_t e = first; e < e1; e += 1024) {
    const uint2 hv = h[e >> 2];
    const float4 dv = dh[e >> 2], cv = cc[e >> 2];
    const float2 h01 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&hv.x));
    const float2 h23 = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&hv.y));
    const float hq[4] = {h01.x, h01.y, h23.x, h23.y};
    const float dq[4] = {dv.x, dv.y, dv.z, dv.w}, cq[4] = {cv.x, cv.y, cv.z, cv.w};
    float o[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float dy = hq[u] > 0.f ? dq[u] : 0.f;
      o[u] = gi[u] * (dy - k1[u] - (cq[u] - mean[u]) * inv[u] * k2[u]);
    }
    dc[e >> 2] = make_uint2(pack_bf16(o[0], o[1]), pack_bf16(o[2], o[3]));
  }
}

// ---- the generator's first layer on tcgen05 -------------------------------------------------
// A 4x4 transposed convolution of a 1x1 input is the plain product y[n][(tap, o)] =
// sum_c z[n][c] W[c][o][tap] (Table 1, CelebA column: z of 100 entries to 4 x 4 x 8 ngf). One
// CTA computes one problem's rows (B <= 128) against 256 consecutive (tap, o) columns: the
// noise rows are loaded into the 128-byte-swizzled K-major layout (K padded with zeros to 128),
// the weights arrive by TMA from a [individual][(tap, o)][128] copy (launch_relayout_g1), eight
// MMAs accumulate in TMEM, and each epilogue thread stores its row's 256 fp32 values
// channel-last (y[n][tap * co + o], the layout the channel-last batch norm reads).
constexpr int D1_THREADS = 128;
constexpr int D1_SMEM = 1024 + 2 * A_BYTES + 2 * B_BYTES + 64;

// Sum of v over the 32 lanes of a warp for 16 columns, reduce-scattered: lanes 2j and 2j + 1
// return the sum of column j (a fixed tree of lane exchanges).
__device__ __forceinline__ float colsum16(const float (&v)[16], int lane) {
  float a8[8], a4[4], a2[2];
  const bool b4 = lane & 16, b3 = lane & 8, b2 = lane & 4, b1 = lane & 2;
#pragma unroll
  for (int i = 0; i < 8; ++i)
    a8[i] = (b4 ? v[8 + i] : v[i]) + __shfl_xor_sync(0xffffffffu, b4 ? v[i] : v[8 + i], 16);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    a4[i] = (b3 ? a8[4 + i] : a8[i]) + __shfl_xor_sync(0xffffffffu, b3 ? a8[i] : a8[4 + i], 8);
#pragma unroll
  for (int i = 0; i < 2; ++i)
    a2[i] = (b2 ? a4[2 + i] : a4[i]) + __shfl_xor_sync(0xffffffffu, b2 ? a4[i] : a4[2 + i], 4);
  const float a1 = (b1 ? a2[1] : a2[0]) + __shfl_xor_sync(0xffffffffu, b1 ? a2[0] : a2[1], 2);
  return a1 + __shfl_xor_sync(0xffffffffu, a1, 1);
}

__global__ void __launch_bounds__(D1_THREADS) k_dense1_tc(const __grid_constant__ CUtensorMap mW,
                                                          const ConvDesc* __restrict__ descs,
                                                          const int* __restrict__ wsel_override,
                                                          int rows, int ca, int N, int* err,
                                                          float2* __restrict__ bn_part) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sA = base, sB = base + 2 * A_BYTES;
  uint8_t* misc = gbase + 2 * A_BYTES + 2 * B_BYTES;
  const uint32_t bFull = smem_u32(misc), bMma = bFull + 8;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(misc + 16);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 20);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * 256;
  if (threadIdx.x == 0) {
    mbar_init(bFull, 1);
    mbar_init(bMma, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 256;" ::"r"(
        smem_u32((const void*)tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  const ConvDesc d = descs[blockIdx.y];
  const int* ws = wsel_override ? wsel_override : d.wsel;
  const int indiv = ws ? __ldg(&ws[d.wsel_idx]) : 0;
  if (threadIdx.x == 0) {
    mbar_expect_tx(bFull, 2u * B_BYTES);
    tma_load_3d(sB, &mW, bFull, 0, n0, indiv);
    tma_load_3d(sB + B_BYTES, &mW, bFull, BK, n0, indiv);
  }
  // the noise rows, 8-byte loads (ca a multiple of 4, rows 8-byte aligned); 16-byte unit u of
  // row r (K elements 8u .. 8u + 7) goes to unit u ^ (r & 7) of its 128-byte row
  {
    const bf16* z = (const bf16*)d.a;
    const int r = threadIdx.x;
    const uint2* zr = reinterpret_cast<const uint2*>(z + (int64_t)r * ca);
#pragma unroll 4
    for (int u = 0; u < 16; ++u) {
      const int k = 8 * u;
      uint2 lo = make_uint2(0u, 0u), hi = make_uint2(0u, 0u);
      if (r < rows) {
        if (k < ca) lo = zr[k >> 2];
        if (k + 4 < ca) hi = zr[(k >> 2) + 1];
      }
      const uint32_t addr = sA + (uint32_t)((u >> 3) * A_BYTES) + (uint32_t)r * 128u +
                            ((uint32_t)((u & 7) ^ (r & 7)) << 4);
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(lo.x), "r"(lo.y),
                   "r"(hi.x), "r"(hi.y)
                   : "memory");
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (mbar_wait(bFull, 0u, abort_flag, err, 41)) {
      tc_fence_after();
      constexpr uint32_t idesc = idesc_bf16(BM, 256);
#pragma unroll
      for (int c = 0; c < 2; ++c)
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk)
          tc_mma(tmem, sw128_desc(sA + c * A_BYTES + kk * 32), sw128_desc(sB + c * B_BYTES + kk * 32),
                 idesc, (c | kk) != 0 ? 1u : 0u);
      tc_commit(bMma);
    }
  }
  // bn_part: the batch-norm sums of this tile's 256 channels of one tap over the problem's rows
  // (rows past `rows` are zero products): per warp by colsum16 into shared memory (the
  // operand buffers, free once the accumulator is ready), then the four warps in order
  float2* red = reinterpret_cast<float2*>(gbase);  // [4 warps][256]
  const bool mma_ok = mbar_wait_warp(bMma, 0u, abort_flag, err, 42);
  if (mma_ok) {
    tc_fence_after();
    const int row = warp * 32 + lane;
    float* out = (float*)d.out + (int64_t)row * N + n0;
#pragma unroll 1
    for (int g = 0; g < 16; ++g) {
      uint32_t r[16];
      LIPZ_TMEM_LD16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(g * 16), r);
      tmem_wait_ld();
      if (row < rows && n0 + g * 16 < N) {
        float4* o = reinterpret_cast<float4*>(out + g * 16);
#pragma unroll
        for (int q = 0; q < 4; ++q)
          o[q] = make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                             __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3]));
      }
      if (bn_part) {
        float v[16], v2[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          v[e] = __uint_as_float(r[e]);
          v2[e] = v[e] * v[e];
        }
        const float cs = colsum16(v, lane), cq = colsum16(v2, lane);
        if (!(lane & 1)) red[warp * 256 + g * 16 + (lane >> 1)] = make_float2(cs, cq);
      }
    }
  }
  if (bn_part) {
    __syncthreads();
    if (mma_ok) {
      const int co = N >> 4, tap = n0 / co, o0 = n0 - tap * co;
      float2* pp = bn_part + ((int64_t)blockIdx.y * 16 + tap) * co + o0;
      for (int c = threadIdx.x; c < 256; c += D1_THREADS) {
        float2 t = red[c];
#pragma unroll
        for (int w = 1; w < 4; ++w) {
          t.x += red[w * 256 + c].x;
          t.y += red[w * 256 + c].y;
        }
        pp[c] = t;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 256;" ::"r"(tmem));
}

// [individual][c][o][tap] (c < ca) -> [individual][(tap, o)][128], K padded with zeros
__global__ void k_relayout_g1(const bf16* __restrict__ src, int64_t src_ps, int64_t src_off,
                              bf16* __restrict__ dst, int64_t dst_ps, int ca, int co,
                              int n_indiv) {
  pdl_wait();
  const int N = 16 * co;
  const int64_t units = (int64_t)n_indiv * N * 16;  // 16-byte units of the copy
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < units;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int u = (int)(i & 15);
    const int64_t rn = i >> 4;
    const int n = (int)(rn % N);
    const int ind = (int)(rn / N);
    const int tap = n / co, o = n - tap * co;
    const bf16* w = src + (int64_t)ind * src_ps + src_off + (int64_t)o * 16 + tap;
    uint32_t v[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int k0 = 8 * u + 2 * e;
      const unsigned short a = k0 < ca ? __bfloat16_as_ushort(w[(int64_t)k0 * co * 16]) : 0;
      const unsigned short b =
          k0 + 1 < ca ? __bfloat16_as_ushort(w[(int64_t)(k0 + 1) * co * 16]) : 0;
      v[e] = (uint32_t)a | ((uint32_t)b << 16);
    }
    *reinterpret_cast<uint4*>(dst + (int64_t)ind * dst_ps + (int64_t)n * 128 + 8 * u) =
        make_uint4(v[0], v[1], v[2], v[3]);
  }
}


// ---- the generator's first-layer weight gradient on tcgen05 ---------------------------------
// dW1[c][o][tap] = sum_n z[n][c] dc1[n][tap][o], as the product of A = z^T (M = c, padded to
// 128 with zeros, K = n) and B = dc1 with its columns in (o, tap) order (k_relayout_dc1), both
// MN-major in the 128-byte swizzle: the noise rows are written into A's atoms by the CTA's
// threads, B arrives by TMA. One CTA per (256 columns, cell); K = B <= 128 in two chunks; each
// epilogue thread stores its row's 256 fp32 values, which are contiguous in dW1.
constexpr int D1W_SMEM = 1024 + 2 * 2 * 8192 + 2 * 4 * 8192 + 64;

__global__ void __launch_bounds__(128) k_dense1_wgrad_tc(const __grid_constant__ CUtensorMap mB,
                                                         const bf16* __restrict__ z,
                                                         int64_t z_cell, float* __restrict__ dw,
                                                         int64_t dw_cell, int rows, int ca, int N,
                                                         int* err) {
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sA = base, sB = base + 2 * 16384;  // [chunk][M box][64 k][128 B], [chunk][4][..]
  uint8_t* misc = gbase + 2 * 16384 + 2 * 32768;
  const uint32_t bFull = smem_u32(misc), bMma = bFull + 8;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(misc + 16);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 20);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n0 = blockIdx.x * 256, cell = blockIdx.y;
  if (threadIdx.x == 0) {
    mbar_init(bFull, 1);
    mbar_init(bMma, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 0) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], 256;" ::"r"(
        smem_u32((const void*)tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();
  if (threadIdx.x == 0) {
    mbar_expect_tx(bFull, 2u * 4u * 8192u);
    for (int kc = 0; kc < 2; ++kc)
      for (int i = 0; i < 4; ++i)
        tma_load_3d(sB + (uint32_t)(kc * 32768 + i * 8192), &mB, bFull, n0 + 64 * i, kc * 64,
                    cell);
  }
  // A: 16-byte unit u (channels 8u' .. 8u' + 7 of M box b) of k row kr of chunk kc sits at unit
  // u ^ (kr & 7) of that row; channels past ca and samples past rows are zero
  {
    const bf16* zc = z + (int64_t)cell * z_cell;
    for (int i = threadIdx.x; i < 2 * 2 * 64 * 8; i += 128) {
      const int u = i & 7, kr = (i >> 3) & 63, b = (i >> 9) & 1, kc = i >> 10;
      const int n = kc * 64 + kr, c = b * 64 + u * 8;
      uint2 lo = make_uint2(0u, 0u), hi = make_uint2(0u, 0u);
      if (n < rows) {
        const uint2* zr = reinterpret_cast<const uint2*>(zc + (int64_t)n * ca);
        if (c < ca) lo = zr[c >> 2];
        if (c + 4 < ca) hi = zr[(c >> 2) + 1];
      }
      const uint32_t addr = sA + (uint32_t)(kc * 16384 + b * 8192 + kr * 128) +
                            ((uint32_t)(u ^ (kr & 7)) << 4);
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(lo.x), "r"(lo.y),
                   "r"(hi.x), "r"(hi.y)
                   : "memory");
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    if (mbar_wait(bFull, 0u, abort_flag, err, 43)) {
      tc_fence_after();
      constexpr uint32_t idesc = idesc_bf16_major(BM, 256, 1, 1);
#pragma unroll
      for (int kc = 0; kc < 2; ++kc)
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk)
          tc_mma(tmem, sw128_mn_desc(sA + kc * 16384 + kk * 2048, 8192),
                 sw128_mn_desc(sB + kc * 32768 + kk * 2048, 8192), idesc, (kc | kk) != 0 ? 1u : 0u);
      tc_commit(bMma);
    }
  }
  if (mbar_wait_warp(bMma, 0u, abort_flag, err, 44)) {
    tc_fence_after();
    const int row = warp * 32 + lane;  // channel c of z
    float* out = dw + (int64_t)cell * dw_cell + (int64_t)row * N + n0;
#pragma unroll 1
    for (int g = 0; g < 16; ++g) {
      uint32_t r[16];
      LIPZ_TMEM_LD16(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)(g * 16), r);
      tmem_wait_ld();
      if (row < ca) {
        float4* o = reinterpret_cast<float4*>(out + g * 16);
#pragma unroll
        for (int q = 0; q < 4; ++q)
          o[q] = make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]),
                             __uint_as_float(r[4 * q + 2]), __uint_as_float(r[4 * q + 3]));
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 256;" ::"r"(tmem));
}

// dc1 [n][16 taps][co] -> [n][co][16 taps] (bf16), one block per (sample, cell) through shared
// memory
__global__ void __launch_bounds__(256) k_relayout_dc1(const bf16* __restrict__ src,
                                                      int64_t src_cell, bf16* __restrict__ dst,
                                                      int rows, int co) {
  extern __shared__ uint8_t smem_dc1[];
  bf16* sh = reinterpret_cast<bf16*>(smem_dc1);  // [16][co + 2]
  pdl_wait();
  const int n = blockIdx.x, cell = blockIdx.y;
  const bf16* sp = src + (int64_t)cell * src_cell + (int64_t)n * 16 * co;
  bf16* dp = dst + ((int64_t)cell * rows + n) * 16 * co;
  for (int i = threadIdx.x; i < 16 * co; i += 256) sh[(i / co) * (co + 2) + (i % co)] = sp[i];
  __syncthreads();
  for (int i = threadIdx.x; i < 16 * co; i += 256) dp[i] = sh[(i & 15) * (co + 2) + (i >> 4)];
}

}  // namespace ctc

bool wgtc_prepare(std::string* msg) {
  if (cudaFuncSetAttribute(ctc::k_wgrad_tc<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           ctc::WG_SMEM) != cudaSuccess ||
      cudaFuncSetAttribute(ctc::k_wgrad_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           ctc::WG_SMEM) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cannot reserve shared memory for the tensor-core weight gradients";
    return false;
  }
  return true;
}

void launch_wgrad_tc(const CUtensorMap& mA, const CUtensorMap& mB, const WgtcParams& p, int sms,
                     cudaStream_t st) {
  const int grid = p.n_tiles < sms ? p.n_tiles : sms;
  launch_pdl(p.b_chw ? ctc::k_wgrad_tc<true> : ctc::k_wgrad_tc<false>, dim3(grid),
             dim3(ctc::WG_THREADS), ctc::WG_SMEM, st, mA, mB, p);
  if (p.b_chw)
    launch_pdl(ctc::k_wgrad_tc_reduce_chw, dim3((p.M * 48 + 255) / 256, p.n_probs), dim3(256), 0,
               st, p);
  else
    launch_pdl(ctc::k_wgrad_tc_reduce, dim3(p.M * (p.Cb / 64), p.n_probs), dim3(256), 0, st, p);
}

void launch_relayout_c(const bf16* src, int64_t src_ps, bf16* dst, int64_t dst_ps, int n_indiv,
                       const RelayoutC& r, cudaStream_t st) {
  ctc::RelayoutRows q;
  memset(&q, 0, sizeof q);
  q.n = r.n;
  int rows = 0;
  for (int l = 0; l < r.n; ++l) {
    q.src_off[l] = r.src_off[l];
    q.dst_off[l] = r.dst_off[l];
    // a 3-channel tensor is read in its own [out][c][ky][kx] order by the first-layer gather,
    // straight from src: no rows
    q.o[l] = r.c[l] == 3 ? 0 : r.o[l];
    q.c[l] = r.c[l];
    rows += q.o[l];
  }
  launch_pdl(ctc::k_relayout_rows, dim3(rows, n_indiv), dim3(256), 0, st, src, src_ps, dst, dst_ps,
             q);
}

void launch_relayout_g(const bf16* src, int64_t src_ps, bf16* dst, int64_t dst_ps, int n_indiv,
                       const RelayoutG& r, cudaStream_t st) {
  int rows = 0;
  for (int l = 0; l < r.n; ++l) rows += r.co[l];
  launch_pdl(ctc::k_relayout_g, dim3(rows, n_indiv), dim3(256), 0, st, src, src_ps, dst, dst_ps, r);
}

namespace {
// the apply pass: four channels per thread where the layout allows it
void bn_apply(const BnDesc* descs, int n_problems, int channels, const int* wsel,
              int64_t elems, cudaStream_t st) {
  if (channels % 4 == 0 && channels <= 1024 && 1024 % channels == 0 && elems > 0) {
    const int64_t blocks = (elems + ctc::BN_APPLY_ELEMS - 1) / ctc::BN_APPLY_ELEMS;
    launch_pdl(ctc::k_bn_apply_hwc4, dim3((unsigned)blocks, n_problems), dim3(256), 0, st,
               descs, wsel);
  } else {
    const dim3 grid((channels + 31) / 32, n_problems, ctc::BN_CHUNKS);
    launch_pdl(ctc::k_bn_apply_hwc, grid, dim3(256), 0, st, descs, wsel);
  }
}
}  // namespace

void launch_bn_relu_hwc(const BnDesc* descs, int n_problems, int channels, const int* wsel,
                        float* part, unsigned* counters, int64_t elems, cudaStream_t st) {
  const dim3 grid((channels + 31) / 32, n_problems, ctc::BN_CHUNKS);
  launch_pdl(ctc::k_bn_stats_hwc, grid, dim3(256), 0, st, descs, (float2*)part, channels,
             counters);
  bn_apply(descs, n_problems, channels, wsel, elems, st);
}

void launch_bn_relu_hwc_part(const BnDesc* descs, int n_problems, int channels, const int* wsel,
                             const float2* part, int slots, int64_t elems, cudaStream_t st) {
  launch_pdl(ctc::k_bn_finalize_hwc, dim3((channels + 31) / 32, n_problems), dim3(1024), 0, st,
             descs, part, slots);
  bn_apply(descs, n_problems, channels, wsel, elems, st);
}

void launch_bn_relu_backward_hwc(const BnDesc* descs, int n_problems, int channels,
                                 float* part, unsigned* counters, int64_t elems, cudaStream_t st) {
  if (channels % 4 == 0 && channels <= 1024 && 1024 % channels == 0 && elems >= 4096) {
    launch_pdl(ctc::k_bn_back_stats_hwc4, dim3(ctc::BN_CHUNKS, n_problems),
               dim3(ctc::BN_B_THREADS), 0, st, descs, (float2*)part, channels, counters);
    const int64_t blocks = (elems + ctc::BN_APPLY_ELEMS - 1) / ctc::BN_APPLY_ELEMS;
    launch_pdl(ctc::k_bn_back_apply_hwc4, dim3((unsigned)blocks, n_problems), dim3(256), 0, st,
               descs);
    return;
  }
  const dim3 grid((channels + 31) / 32, n_problems, ctc::BN_CHUNKS);
  launch_pdl(ctc::k_bn_back_stats_hwc, grid, dim3(256), 0, st, descs, (float2*)part, channels,
             counters);
  launch_pdl(ctc::k_bn_back_apply_hwc, grid, dim3(256), 0, st, descs);
}

int64_t bn_hwc_part_floats(int n_problems, int channels) {
  return (int64_t)n_problems * ctc::BN_CHUNKS * channels * 2;
}

int64_t bn_hwc_counters(int n_problems, int channels) {
  return (int64_t)n_problems * ((channels + 31) / 32);
}

namespace {
PFN_cuTensorMapEncodeTiled_v12000 g_encode_ctc = nullptr;

bool ensure_encode(std::string* msg) {
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
  return true;
}
}  // namespace

bool ctc_make_map(CUtensorMap* m, const void* base, uint64_t K, uint64_t rows, uint64_t depth,
                  uint64_t depth_elems, uint32_t box_rows, std::string* msg) {
  if (!ensure_encode(msg)) return false;
  cuuint64_t dims[3] = {K, rows, depth};
  cuuint64_t strides[2] = {K * 2, depth_elems * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_encode_ctc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg)
      *msg = "cuTensorMapEncodeTiled (convolution weights) failed: " + std::to_string((int)r);
    return false;
  }
  return true;
}

bool ctc_make_out_map(CUtensorMap* m, CtcParams* q, const ConvTcDesc* descs, int n_probs,
                      std::string* msg) {
  q->tma_out = 0;
  if (!q->nchw_in || q->out_mode != CTC_LRELU_HWC || q->co != 64 || q->nj != 1 || q->m2 ||
      n_probs < 1)
    return true;
  const int64_t M = (int64_t)q->rows << (2 * q->lho);  // output pixels of a problem
  if (M % ctc::BM != 0) return true;
  const int64_t per = M * q->co;
  int64_t pstride = per;
  if (n_probs > 1) pstride = (int64_t)(descs[1].out - descs[0].out);
  if (pstride < per || pstride % 8 != 0 || ((uintptr_t)descs[0].out & 15) != 0) return true;
  for (int i = 2; i < n_probs; ++i)
    if ((int64_t)(descs[i].out - descs[0].out) != i * pstride) return true;
  if (!ensure_encode(msg)) return false;
  cuuint64_t dims[3] = {(cuuint64_t)q->co, (cuuint64_t)M, (cuuint64_t)n_probs};
  cuuint64_t strides[2] = {(cuuint64_t)q->co * 2, (cuuint64_t)(pstride * 2)};
  cuuint32_t box[3] = {64, (cuuint32_t)ctc::BM, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_encode_ctc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, (void*)descs[0].out, dims,
                            strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled (convolution output) failed: " + std::to_string((int)r);
    return false;
  }
  q->tma_out = 1;
  return true;
}

bool ctc_make_act_map(CUtensorMap* m, CtcParams* q, const ConvTcDesc* descs, int n_probs,
                      std::string* msg, bool use_tma) {
  q->a_tma = 0;
  q->m2 = 0;
  if (!use_tma || q->nchw_in || q->ci % 64 != 0 || n_probs < 1) return true;
  const int lq = q->scatter ? q->lhi : q->lho - q->transposed;
  if (lq > 7) return true;
  const int64_t Wi = (int64_t)1 << q->lhi;
  const int64_t per = (int64_t)q->rows * Wi * Wi * q->ci;  // elements of one problem's input
  int64_t pstride = per;
  if (n_probs > 1) pstride = (int64_t)(descs[1].in - descs[0].in);
  if (pstride < per || pstride % 8 != 0) return true;
  for (int k = 1; k < n_probs; ++k)
    if (descs[k].in != descs[0].in + (int64_t)k * pstride) return true;
  if (!ensure_encode(msg)) return false;
  const int stride = q->transposed || q->scatter ? 1 : 2;
  const int tw = 1 << lq, th = std::min(1 << lq, 128 / tw), tn = std::max(1, 128 / (tw * th));
  cuuint64_t dims[5] = {(cuuint64_t)q->ci, (cuuint64_t)Wi, (cuuint64_t)Wi, (cuuint64_t)q->rows,
                        (cuuint64_t)n_probs};
  cuuint64_t strides[4] = {(cuuint64_t)q->ci * 2, (cuuint64_t)(Wi * q->ci * 2),
                           (cuuint64_t)(Wi * Wi * q->ci * 2), (cuuint64_t)(pstride * 2)};
  cuuint32_t box[5] = {64, (cuuint32_t)(tw * stride), (cuuint32_t)(th * stride), (cuuint32_t)tn, 1};
  cuuint32_t es[5] = {1, (cuuint32_t)stride, (cuuint32_t)stride, 1, 1};
  CUresult r = g_encode_ctc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5,
                            const_cast<bf16*>(descs[0].in), dims, strides, box, es,
                            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg)
      *msg = "cuTensorMapEncodeTiled (convolution activations) failed: " +
             std::to_string((int)r);
    return false;
  }
  q->a_tma = 1;
  // 256-row tiles (two accumulators sharing each weight chunk) for narrow weight tiles
  if (!q->scatter && q->nbox <= 128 &&
      (q->out_mode == CTC_LRELU_HWC || q->out_mode == CTC_F32_HWC ||
       q->out_mode == CTC_DLRELU_HWC)) {
    const int M = q->rows << (2 * lq);
    const int mt2 = (M + 255) / 256;
    q->n_tiles = q->n_tiles / q->mtiles * mt2;
    q->mtiles = mt2;
    q->m2 = 1;
  }
  return true;
}

namespace {
using ConvKernel = void (*)(const CUtensorMap, const CUtensorMap, const CtcParams);
struct ConvVariant {
  int ak, om;
  ConvKernel k;
};
// the (A kind, out mode) pairs the DCGAN launches use; the gathered form takes them all
const ConvVariant kConvVariants[] = {
    {ctc::AK_CONV, CTC_LRELU_HWC, ctc::k_conv_tc<ctc::AK_CONV, CTC_LRELU_HWC>},
    {ctc::AK_CONV, CTC_F32_HWC, ctc::k_conv_tc<ctc::AK_CONV, CTC_F32_HWC>},
    {ctc::AK_CONV, CTC_LRELU_LOGIT, ctc::k_conv_tc<ctc::AK_CONV, CTC_LRELU_LOGIT>},
    {ctc::AK_TRANS, CTC_F32_HWC, ctc::k_conv_tc<ctc::AK_TRANS, CTC_F32_HWC>},
    {ctc::AK_TRANS, CTC_TANH_CHW, ctc::k_conv_tc<ctc::AK_TRANS, CTC_TANH_CHW>},
    {ctc::AK_TRANS, CTC_DLRELU_HWC, ctc::k_conv_tc<ctc::AK_TRANS, CTC_DLRELU_HWC>},
    {ctc::AK_TRANS, CTC_DTANH_CHW, ctc::k_conv_tc<ctc::AK_TRANS, CTC_DTANH_CHW>},
    {ctc::AK_TRANS_C, CTC_F32_HWC, ctc::k_conv_tc<ctc::AK_TRANS_C, CTC_F32_HWC>},
    {ctc::AK_TRANS_C, CTC_DLRELU_HWC, ctc::k_conv_tc<ctc::AK_TRANS_C, CTC_DLRELU_HWC>},
    {ctc::AK_SCATTER, CTC_TANH_CHW, ctc::k_conv_tc<ctc::AK_SCATTER, CTC_TANH_CHW>},
    {ctc::AK_SCATTER, CTC_DTANH_CHW, ctc::k_conv_tc<ctc::AK_SCATTER, CTC_DTANH_CHW>},
    {ctc::AK_NCHW, CTC_LRELU_HWC, ctc::k_conv_tc<ctc::AK_NCHW, CTC_LRELU_HWC>},
    {ctc::AK_NCHW, CTC_F32_HWC, ctc::k_conv_tc<ctc::AK_NCHW, CTC_F32_HWC>},
    {ctc::AK_NCHW_WIDE, CTC_LRELU_HWC, ctc::k_conv_tc<ctc::AK_NCHW_WIDE, CTC_LRELU_HWC>},
    {ctc::AK_NCHW_WIDE, CTC_F32_HWC, ctc::k_conv_tc<ctc::AK_NCHW_WIDE, CTC_F32_HWC>},
    {ctc::AK_GATHER, CTC_LRELU_HWC, ctc::k_conv_tc<ctc::AK_GATHER, CTC_LRELU_HWC>},
    {ctc::AK_GATHER, CTC_F32_HWC, ctc::k_conv_tc<ctc::AK_GATHER, CTC_F32_HWC>},
    {ctc::AK_GATHER, CTC_TANH_CHW, ctc::k_conv_tc<ctc::AK_GATHER, CTC_TANH_CHW>},
    {ctc::AK_GATHER, CTC_DLRELU_HWC, ctc::k_conv_tc<ctc::AK_GATHER, CTC_DLRELU_HWC>},
    {ctc::AK_GATHER, CTC_DTANH_CHW, ctc::k_conv_tc<ctc::AK_GATHER, CTC_DTANH_CHW>},
    {ctc::AK_GATHER, CTC_LRELU_LOGIT, ctc::k_conv_tc<ctc::AK_GATHER, CTC_LRELU_LOGIT>},
};

int conv_ak(const CtcParams& p) {
  return p.scatter   ? ctc::AK_SCATTER
         : p.nchw_in ? (p.nbox <= 64 ? ctc::AK_NCHW : ctc::AK_NCHW_WIDE)
         : p.a_tma   ? (p.transposed ? (p.m2 && p.nbox <= 64 ? ctc::AK_TRANS_C : ctc::AK_TRANS)
                                     : ctc::AK_CONV)
                     : ctc::AK_GATHER;
}

ConvKernel conv_kernel(const CtcParams& p) {
  const int ak = conv_ak(p);
  for (const ConvVariant& v : kConvVariants)
    if (v.ak == ak && v.om == p.out_mode) return v.k;
  return nullptr;
}
}  // namespace

bool wgtc_make_maps(CUtensorMap* mA, CUtensorMap* mB, WgtcParams* q, const WgtcDesc* descs,
                    int n_probs, std::string* msg) {
  q->a_tma = 0;
  if (n_probs < 1 || q->M % 64 != 0) return true;
  // b_chw: A by TMA only, B built from staged patches (first-layer geometry only)
  if (q->b_chw && (q->la != 5 || q->lb != 6 || q->s != 2 || q->p != 1)) return true;
  if (!q->b_chw && q->Cb % 64 != 0) return true;
  const int64_t Wa = (int64_t)1 << q->la, Wb = (int64_t)1 << q->lb;
  const int64_t Kp = (int64_t)q->rows * Wa * Wa;
  const int64_t per_a = Kp * q->M, per_b = (int64_t)q->rows * Wb * Wb * q->Cb;
  int64_t sa = per_a, sb = per_b;
  if (n_probs > 1) {
    sa = (int64_t)(descs[1].a - descs[0].a);
    sb = (int64_t)(descs[1].b - descs[0].b);
  }
  if (q->b_chw) sb = per_b;  // b is read through the descriptors
  if (sa < per_a || sb < per_b || sa % 8 != 0 || sb % 8 != 0) return true;
  for (int k = 1; k < n_probs; ++k)
    if (descs[k].a != descs[0].a + k * sa || (!q->b_chw && descs[k].b != descs[0].b + k * sb))
      return true;
  if (!ensure_encode(msg)) return false;
  {
    cuuint64_t dims[3] = {(cuuint64_t)q->M, (cuuint64_t)Kp, (cuuint64_t)n_probs};
    cuuint64_t strides[2] = {(cuuint64_t)q->M * 2, (cuuint64_t)sa * 2};
    cuuint32_t box[3] = {64, 64, 1};
    cuuint32_t es[3] = {1, 1, 1};
    if (g_encode_ctc(mA, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<bf16*>(descs[0].a), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
      if (msg) *msg = "cuTensorMapEncodeTiled (weight-gradient A) failed";
      return false;
    }
  }
  if (!q->b_chw) {
    // the 64 A pixels of a chunk: tw columns of th rows of tn images, in raster order
    const int tw = (int)std::min<int64_t>(Wa, 64), th = (int)std::min<int64_t>(Wa, 64 / tw);
    const int tn = std::max(1, 64 / (tw * th));
    cuuint64_t dims[5] = {(cuuint64_t)q->Cb, (cuuint64_t)Wb, (cuuint64_t)Wb, (cuuint64_t)q->rows,
                          (cuuint64_t)n_probs};
    cuuint64_t strides[4] = {(cuuint64_t)q->Cb * 2, (cuuint64_t)(Wb * q->Cb * 2),
                             (cuuint64_t)(Wb * Wb * q->Cb * 2), (cuuint64_t)sb * 2};
    cuuint32_t box[5] = {64, (cuuint32_t)(tw * q->s), (cuuint32_t)(th * q->s), (cuuint32_t)tn, 1};
    cuuint32_t es[5] = {1, (cuuint32_t)q->s, (cuuint32_t)q->s, 1, 1};
    if (g_encode_ctc(mB, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<bf16*>(descs[0].b), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS) {
      if (msg) *msg = "cuTensorMapEncodeTiled (weight-gradient B) failed";
      return false;
    }
  }
  q->a_tma = 1;
  return true;
}

bool ctc_prepare(std::string* msg) {
  for (const ConvVariant& v : kConvVariants)
    if (cudaFuncSetAttribute(v.k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             ctc::conv_smem(v.ak)) != cudaSuccess) {
      cudaGetLastError();
      if (msg) *msg = "cannot reserve shared memory for the tensor-core convolution";
      return false;
    }
  if (cudaFuncSetAttribute(ctc::k_dense1_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           ctc::D1_SMEM) != cudaSuccess ||
      cudaFuncSetAttribute(ctc::k_dense1_wgrad_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           ctc::D1W_SMEM) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cannot reserve shared memory for the generator's first layer";
    return false;
  }
  return true;
}

bool dense1_wgrad_make_map(CUtensorMap* m, const bf16* dc1t, int rows, int co, int cells,
                           std::string* msg) {
  if (!ensure_encode(msg)) return false;
  cuuint64_t dims[3] = {(cuuint64_t)16 * co, (cuuint64_t)rows, (cuuint64_t)cells};
  cuuint64_t strides[2] = {(cuuint64_t)16 * co * 2, (cuuint64_t)rows * 16 * co * 2};
  cuuint32_t box[3] = {64, 64, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_encode_ctc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, (void*)dc1t, dims, strides,
                            box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled (first-layer deltas) failed: " + std::to_string((int)r);
    return false;
  }
  return true;
}

void launch_dense1_wgrad_tc(const CUtensorMap& mB, const bf16* z, int64_t z_cell,
                            const bf16* dc1, int64_t dc1_cell, bf16* dc1t, float* dw,
                            int64_t dw_cell, int rows, int ca, int co, int cells, int* err,
                            cudaStream_t st) {
  launch_pdl(ctc::k_relayout_dc1, dim3(rows, cells), dim3(256), (size_t)16 * (co + 2) * 2, st,
             dc1, dc1_cell, dc1t, rows, co);
  launch_pdl(ctc::k_dense1_wgrad_tc, dim3(16 * co / 256, cells), dim3(128),
             (size_t)ctc::D1W_SMEM, st, mB, z, z_cell, dw, dw_cell, rows, ca, 16 * co, err);
}

bool dense1_tc_supported(int rows, int ca, int co) {
  return rows >= 1 && rows <= ctc::BM && ca >= 1 && ca <= 2 * ctc::BK && ca % 4 == 0 &&
         (16 * co) % 256 == 0;
}

void launch_dense1_tc(const CUtensorMap& mW, const ConvDesc* descs, int n_problems,
                      const int* wsel_override, int rows, int ca, int co, int* err,
                      cudaStream_t st, float2* bn_part) {
  if (n_problems <= 0) return;
  launch_pdl(ctc::k_dense1_tc, dim3(16 * co / 256, n_problems), dim3(ctc::D1_THREADS),
             (size_t)ctc::D1_SMEM, st, mW, descs, wsel_override, rows, ca, 16 * co, err,
             bn_part);
}

void launch_relayout_g1(const bf16* src, int64_t src_ps, int64_t src_off, bf16* dst,
                        int64_t dst_ps, int ca, int co, int n_indiv, cudaStream_t st) {
  const int64_t units = (int64_t)n_indiv * 16 * co * 16;
  const int blocks = (int)std::min<int64_t>((units + 255) / 256, 4096);
  launch_pdl(ctc::k_relayout_g1, dim3(blocks), dim3(256), 0, st, src, src_ps, src_off, dst,
             dst_ps, ca, co, n_indiv);
}

bool launch_conv_tc(const CUtensorMap& mW, const CUtensorMap& mA, const CtcParams& p, int sms,
                    cudaStream_t st) {
  const ConvKernel k = conv_kernel(p);
  if (!k) return false;
  const int ak = conv_ak(p);
  // the compact variants: two CTAs per SM
  const int ctas = ak == ctc::AK_NCHW || ak == ctc::AK_TRANS_C ? 2 * sms : sms;
  const int grid = p.n_tiles < ctas ? p.n_tiles : ctas;
  launch_pdl(k, dim3(grid), dim3(ctc::THREADS), ctc::conv_smem(ak), st, mW, mA, p);
  return true;
}

void launch_scatter_fix(const ConvTcDesc* descs, const float* halo, int n_problems, int rows,
                        int out_mode, cudaStream_t st) {
  launch_pdl(ctc::k_scatter_fix, dim3(n_problems * rows), dim3(256), 0, st, descs, halo, rows,
             out_mode);
}

void launch_relayout_s(const bf16* src, int64_t src_ps, int64_t src_off, bf16* dst, int n_indiv,
                       cudaStream_t st) {
  launch_pdl(ctc::k_relayout_s, dim3(4, n_indiv), dim3(256), 0, st, src, src_ps, src_off, dst);
}

void launch_relayout_d(const bf16* src, bf16* dst, int n_indiv, int64_t Ps, const RelayoutD& r,
                       cudaStream_t st) {
  ctc::RelayoutRows q;
  memset(&q, 0, sizeof q);
  q.n = 5;
  int rows = 0;
  for (int l = 0; l < 5; ++l) {
    q.src_off[l] = q.dst_off[l] = r.off[l];
    q.c[l] = r.ci[l];
    // the first layer is read in its own [out][c][ky][kx] order, straight from src: no rows
    q.o[l] = l == 0 ? 0 : (int)((r.off[l + 1] - r.off[l]) / (16 * (int64_t)r.ci[l]));
    rows += q.o[l];
  }
  launch_pdl(ctc::k_relayout_rows, dim3(rows, n_indiv), dim3(256), 0, st, src, Ps, dst, Ps, q);
}

}  // namespace lipz
