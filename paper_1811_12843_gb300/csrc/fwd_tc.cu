// Tensor-core forward of the evaluation phase (Section 3, step 2: every generator and every
// discriminator of each 5-cell neighbourhood on the cell's minibatch), bf16 operands, fp32
// accumulation in tensor memory.
//
// One persistent kernel per population: CTAs walk 128-row tiles of (cell, slot) problems.
//   generator  tile: z rows of cell c through G_{nbr[c][i]}: 64 -> 256 -> 256 -> x (tanh), the
//                    fakes land in E[c] rows B (1 + i) + r;
//   discriminator tile: rows of E[c] (x_c, then the five fake batches) through
//                    D_{nbr[c][j]}: x -> 256 -> 256 -> 1; the logit lands in logits[c][j][r].
// The layers of a tile are chained on chip: layer 1 streams A (activations) and B (weights)
// through a TMA ring in 128-byte-swizzled K-major chunks, tcgen05.mma accumulates into TMEM;
// the epilogue warps read TMEM, add the bias, apply the activation, round to bf16 and write
// the next layer's A operand into shared memory (same swizzled layout); the next layer's MMAs
// read it there while its weights stream through the ring. The discriminator's 256 -> 1 layer
// is a dot product in the epilogue of layer 2.
//
// Warp roles (320 threads): warp 0 = TMA producer, warp 1 = TMEM allocator + MMA issuer,
// warps 2..9 = epilogue (two warps per TMEM lane quarter, each owning half of the columns).
// Every wait on an mbarrier is bounded (about one second): on expiry the CTA records an error
// code, stops issuing work, drains what it issued, frees its tensor memory and exits.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>

#include "common.cuh"
#include "fwd_tc.h"

namespace lipz {
namespace tc {

constexpr int BM = 128;                      // rows per tile = TMEM lanes
constexpr int BK = 64;                       // K elements per stage: one 128-byte swizzle row
constexpr int HID = 256;                     // hidden width (one N = 256 MMA)
constexpr int STAGES = 3;
constexpr int A_BYTES = BM * BK * 2;         // 16 KB
constexpr int B_BYTES = HID * BK * 2;        // 32 KB
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int H_CHUNK = BM * BK * 2;         // one 64-column chunk of the on-chip activation
constexpr int H_BYTES = BM * HID * 2;        // 64 KB
constexpr int N3 = 112;                      // generator output columns per MMA block
constexpr int NUM_EPI_WARPS = 8;
constexpr int THREADS = 64 + 32 * NUM_EPI_WARPS;
constexpr int MISC_BYTES = 2048;
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + H_BYTES + MISC_BYTES;
constexpr unsigned long long WAIT_NS = 1000000000ull;  // bound on any single wait

enum { KIND_G = 0, KIND_D = 1 };
enum { EPI_TO_H = 0, EPI_LOGIT = 1, EPI_TO_E = 2 };

struct KParams {
  int kind;
  int cells, B, z, x;
  int rows;       // rows per problem: B (generator) or 6B (discriminator)
  int mtiles;     // 128-row tiles per problem
  int n_tiles;    // cells * 5 * mtiles
  int kc1;        // K chunks of layer 1
  int n3;         // generator output blocks of N3 columns
  const int* nbr;
  const float* wmaster;  // fp32 masters (biases)
  const bf16* wb;        // bf16 copies (the discriminator's output weights)
  int64_t pstride;
  int64_t off_b1, off_b2, off_b3, off_w3;
  bf16* E;
  int64_t e_cell;
  float* logits;
  float slope;
  int* err;
};

struct Job {
  int a_from_h;  // A operand: 0 = TMA stream, 1 = the on-chip activation
  int kchunks;
  int n;         // MMA N
  int region;    // TMEM accumulator region (256 columns each)
  int bmap;      // weight map 0, 1, 2
  int brow0;     // first weight row (output column) of this job
  int box_rows;  // rows of the weight box
  int epi;
};

__device__ __forceinline__ Job get_job(const KParams& p, int j) {
  Job J;
  if (j == 0) {
    J = Job{0, p.kc1, HID, 0, 0, 0, HID, EPI_TO_H};
  } else if (j == 1) {
    J = Job{1, HID / BK, HID, 1, 1, 0, HID, p.kind == KIND_D ? EPI_LOGIT : EPI_TO_H};
  } else {
    const int nb = j - 2;
    const int n = min(N3, p.x - nb * N3);
    J = Job{1, HID / BK, n, nb & 1, 2, nb * N3, N3, EPI_TO_E};
  }
  return J;
}

__device__ __forceinline__ int n_jobs(const KParams& p) { return p.kind == KIND_D ? 2 : 2 + p.n3; }

// ---- PTX wrappers ------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count));
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ unsigned long long globaltimer() {
  unsigned long long t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Bounded wait for the phase of `parity` to complete. Returns false (and raises the CTA's
// abort flag and the kernel's error code) if it does not complete within WAIT_NS, or if
// another role of the CTA has aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          int* err, int code) {
  if (mbar_try(bar, parity)) return true;
  const unsigned long long t0 = globaltimer();
  for (uint32_t it = 1;; ++it) {
    if (mbar_try(bar, parity)) return true;
    if ((it & 255u) == 0) {
      if (*abort_flag) return false;
      if (globaltimer() - t0 > WAIT_NS) {
        *abort_flag = 1;
        atomicExch(err, code);
        return false;
      }
    }
  }
}

__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* map, uint32_t bar,
                                            int x, int y, int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
      "l"((uint64_t)map), "r"(x), "r"(y), "r"(z), "r"(bar)
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   bar)
               : "memory");
}
__device__ __forceinline__ void tc_mma(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc,
                                       uint32_t acc) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d),
      "l"(a), "l"(b), "r"(idesc), "r"(acc)
      : "memory");
}

// Shared-memory matrix descriptor of a K-major operand in the 128-byte swizzle layout: rows of
// 128 bytes, 8-row groups 1024 bytes apart (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
  uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;            // leading byte offset (unused for swizzled K-major)
  d |= (uint64_t)(1024 >> 4) << 32;  // stride byte offset
  d |= (uint64_t)1 << 46;            // version
  d |= (uint64_t)2 << 61;            // 128-byte swizzle
  return d;
}

// Instruction descriptor, kind::f16: fp32 accumulator, bf16 A and B, both K-major, N, M.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) |
         ((uint32_t)(M >> 4) << 24);
}

#define LIPZ_TMEM_LD32(taddr, r)                                                                 \
  asm volatile(                                                                                  \
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14," \
      "%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"             \
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),      \
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),  \
        "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),            \
        "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),            \
        "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])             \
      : "r"(taddr))

#define LIPZ_TMEM_LD16(taddr, r)                                                                 \
  asm volatile(                                                                                  \
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14," \
      "%15}, [%16];"                                                                             \
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),      \
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),  \
        "=r"(r[14]), "=r"(r[15])                                                                 \
      : "r"(taddr))

__device__ __forceinline__ void tmem_wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// ---- the kernel ----------------------------------------------------------------------------
__global__ void __launch_bounds__(THREADS, 1)
    k_mlp_fwd(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB1,
              const __grid_constant__ CUtensorMap mB2, const __grid_constant__ CUtensorMap mB3,
              const KParams p) {
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte alignment for the swizzled tiles
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sStage = base;                                 // STAGES x (A | B)
  const uint32_t sH = base + STAGES * STAGE_BYTES;              // on-chip activation
  uint8_t* misc = gbase + STAGES * STAGE_BYTES + H_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(misc);           // 16 barriers
  const uint32_t bFull = smem_u32(bars), bEmpty = bFull + 8 * STAGES;
  const uint32_t bAcc = bEmpty + 8 * STAGES;                    // [2]
  const uint32_t bReg = bAcc + 16;                              // [2]
  const uint32_t bH = bReg + 16;
  const uint32_t bPart = bH + 8;
  const uint32_t bFinal = bPart + 8;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(misc + 256);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 260);
  float* part = reinterpret_cast<float*>(misc + 512);           // [128] partial logits

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bFull + 8 * s, 1);
      mbar_init(bEmpty + 8 * s, 1);
    }
    mbar_init(bAcc, 1);
    mbar_init(bAcc + 8, 1);
    mbar_init(bReg, 32 * NUM_EPI_WARPS);
    mbar_init(bReg + 8, 32 * NUM_EPI_WARPS);
    mbar_init(bH, 32 * NUM_EPI_WARPS);
    mbar_init(bPart, 32 * NUM_EPI_WARPS / 2);
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
  const int nj = n_jobs(p);

  if (warp == 0) {
    // ================================ TMA producer ================================
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued[STAGES] = {0, 0, 0};
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
        const int prob = tile / p.mtiles, m0 = (tile % p.mtiles) * BM;
        const int c = prob / 5;
        const int k = __ldg(&p.nbr[prob]);
        for (int j = 0; j < nj && ok; ++j) {
          const Job J = get_job(p, j);
          const CUtensorMap* mb = J.bmap == 0 ? &mB1 : (J.bmap == 1 ? &mB2 : &mB3);
          for (int kc = 0; kc < J.kchunks; ++kc) {
            if (!mbar_wait(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 1)) {
              ok = false;
              break;
            }
            const uint32_t bytes = (J.a_from_h ? 0u : (uint32_t)A_BYTES) +
                                   (uint32_t)(BK * J.box_rows * 2);
            const uint32_t full = bFull + 8 * stage;
            mbar_expect_tx(full, bytes);
            const uint32_t sA = sStage + stage * STAGE_BYTES;
            if (!J.a_from_h) tma_load_3d(sA, &mA, full, kc * BK, m0, c);
            tma_load_3d(sA + A_BYTES, mb, full, kc * BK, J.brow0, k);
            issued[stage]++;
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      if (!ok) {
        // drain: every load issued must land before the CTA exits
        for (int s = 0; s < STAGES; ++s)
          if (issued[s] > 0) {
            volatile int never = 0;
            mbar_wait(bFull + 8 * s, (uint32_t)((issued[s] - 1) & 1), &never, p.err, 1);
          }
      }
    }
  } else if (warp == 1) {
    // ================================ MMA issuer ================================
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int reg_uses[2] = {0, 0};
      int h_total = 0, h_seen = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
        for (int j = 0; j < nj && ok; ++j) {
          const Job J = get_job(p, j);
          const int R = J.region;
          if (reg_uses[R] > 0 &&
              !mbar_wait(bReg + 8 * R, (uint32_t)((reg_uses[R] - 1) & 1), abort_flag, p.err, 2)) {
            ok = false;
            break;
          }
          if (J.a_from_h) {
            while (h_seen < h_total) {
              if (!mbar_wait(bH, (uint32_t)(h_seen & 1), abort_flag, p.err, 3)) {
                ok = false;
                break;
              }
              ++h_seen;
            }
            if (!ok) break;
          }
          tc_fence_after();
          const uint32_t d = tmem + (uint32_t)(R * HID);
          const uint32_t idesc = idesc_bf16(BM, J.n);
          for (int kc = 0; kc < J.kchunks; ++kc) {
            if (!mbar_wait(bFull + 8 * stage, phase, abort_flag, p.err, 4)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sA = J.a_from_h ? sH + kc * H_CHUNK : sStage + stage * STAGE_BYTES;
            const uint32_t sB = sStage + stage * STAGE_BYTES + A_BYTES;
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              tc_mma(d, sw128_desc(sA + kk * 32), sw128_desc(sB + kk * 32), idesc,
                     (kc | kk) != 0 ? 1u : 0u);
            tc_commit(bEmpty + 8 * stage);
            if (++stage == STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          tc_commit(bAcc + 8 * R);
          reg_uses[R]++;
          if (J.epi == EPI_TO_H) ++h_total;
        }
      }
      // all MMAs issued by this thread complete before tensor memory is released
      tc_commit(bFinal);
      volatile int never = 0;
      mbar_wait(bFinal, 0u, &never, p.err, 5);
    }
  } else {
    // ================================ epilogue ================================
    const int ew = warp - 2;
    const int q = warp & 3;        // TMEM lane quarter this warp may access
    const int hf = ew >> 2;        // column half
    const int row = q * 32 + lane; // row of the tile
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    int reg_uses[2] = {0, 0};
    bool ok = true;
    for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
      const int prob = tile / p.mtiles, m0 = (tile % p.mtiles) * BM;
      const int c = prob / 5, slot = prob % 5;
      const int k = __ldg(&p.nbr[prob]);
      const float* wm = p.wmaster + (int64_t)k * p.pstride;
      for (int j = 0; j < nj && ok; ++j) {
        const Job J = get_job(p, j);
        const int R = J.region;
        if (!mbar_wait(bAcc + 8 * R, (uint32_t)(reg_uses[R] & 1), abort_flag, p.err, 6)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tbase = tmem + lane_base + (uint32_t)(R * HID);
        if (J.epi == EPI_TO_H) {
          const float* bias = wm + (j == 0 ? p.off_b1 : p.off_b2);
          const bool lrelu = p.kind == KIND_D;
#pragma unroll 1
          for (int cg = hf * 4; cg < hf * 4 + 4; ++cg) {
            uint32_t r[32];
            LIPZ_TMEM_LD32(tbase + cg * 32, r);
            tmem_wait_ld();
            uint32_t pk[16];
#pragma unroll
            for (int e = 0; e < 32; e += 2) {
              float a0 = __uint_as_float(r[e]) + __ldg(&bias[cg * 32 + e]);
              float a1 = __uint_as_float(r[e + 1]) + __ldg(&bias[cg * 32 + e + 1]);
              a0 = a0 > 0.f ? a0 : (lrelu ? p.slope * a0 : 0.f);
              a1 = a1 > 0.f ? a1 : (lrelu ? p.slope * a1 : 0.f);
              pk[e >> 1] = pack_bf16(a0, a1);
            }
            const uint32_t chunk = sH + (uint32_t)((cg >> 1) * H_CHUNK) + (uint32_t)row * 128u;
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const uint32_t unit = (uint32_t)((cg & 1) * 4 + u);
              const uint32_t addr = chunk + ((unit ^ (uint32_t)(row & 7)) << 4);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr),
                           "r"(pk[4 * u]), "r"(pk[4 * u + 1]), "r"(pk[4 * u + 2]),
                           "r"(pk[4 * u + 3])
                           : "memory");
            }
          }
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          tc_fence_before();
          mbar_arrive(bReg + 8 * R);
          mbar_arrive(bH);
        } else if (J.epi == EPI_LOGIT) {
          const float* bias = wm + p.off_b2;
          const bf16* w3 = p.wb + (int64_t)k * p.pstride + p.off_w3;
          float acc = 0.f;
#pragma unroll 1
          for (int cg = hf * 4; cg < hf * 4 + 4; ++cg) {
            uint32_t r[32];
            LIPZ_TMEM_LD32(tbase + cg * 32, r);
            tmem_wait_ld();
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              float a = __uint_as_float(r[e]) + __ldg(&bias[cg * 32 + e]);
              a = a > 0.f ? a : p.slope * a;
              a = __bfloat162float(__float2bfloat16_rn(a));
              acc = fmaf(a, __bfloat162float(w3[cg * 32 + e]), acc);
            }
          }
          tc_fence_before();
          if (hf == 1) {
            part[row] = acc;
            mbar_arrive(bPart);
            mbar_arrive(bReg + 8 * R);
          } else {
            if (!mbar_wait(bPart, (uint32_t)(reg_uses[R] & 1), abort_flag, p.err, 7)) {
              ok = false;
              break;
            }
            const float logit = acc + part[row] + __ldg(wm + p.off_b3);
            mbar_arrive(bReg + 8 * R);
            const int rr = m0 + row;
            if (rr < p.rows) p.logits[(int64_t)prob * p.rows + rr] = logit;
          }
        } else {
          // generator output block: bias + tanh, bf16, into the fake rows of E[c]
          const float* bias = wm + p.off_b3;
          const int ng = J.n / 16;
          const int g0 = hf ? 4 : 0, g1 = hf ? ng : min(4, ng);
          const int rr = m0 + row;
          bf16* dst = p.E + (int64_t)c * p.e_cell + (int64_t)((1 + slot) * p.B + rr) * p.x;
#pragma unroll 1
          for (int gi = g0; gi < g1; ++gi) {
            uint32_t r[16];
            LIPZ_TMEM_LD16(tbase + gi * 16, r);
            tmem_wait_ld();
            const int col0 = J.brow0 + gi * 16;
            uint32_t pk[8];
#pragma unroll
            for (int e = 0; e < 16; e += 2)
              pk[e >> 1] = pack_bf16(tanhf(__uint_as_float(r[e]) + __ldg(&bias[col0 + e])),
                                     tanhf(__uint_as_float(r[e + 1]) + __ldg(&bias[col0 + e + 1])));
            if (rr < p.B) {
              uint4* o = reinterpret_cast<uint4*>(dst + col0);
              o[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
              o[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
            }
          }
          tc_fence_before();
          mbar_arrive(bReg + 8 * R);
        }
        reg_uses[R]++;
      }
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, 512;" ::"r"(tmem));
  }
}

}  // namespace tc

// ---- host side -----------------------------------------------------------------------------
struct TcPlan {
  TcShape s;
  CUtensorMap mZ, mE, mG1, mG2, mG3, mD1, mD2;
  tc::KParams pg, pd;
  int grid_g, grid_d;
  int* err;
};

namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

bool get_encoder(std::string* msg) {
  if (g_encode) return true;
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                   cudaEnableDefault, &q);
  if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) {
    cudaGetLastError();
    if (msg) *msg = "cuTensorMapEncodeTiled is unavailable";
    return false;
  }
  g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  return true;
}

// 3-D bf16 map {inner, rows, depth} with a {64, box_rows, 1} box in the 128-byte swizzle.
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t depth,
              uint64_t row_bytes, uint64_t depth_bytes, uint32_t box_rows, std::string* msg) {
  cuuint64_t dims[3] = {inner, rows, depth};
  cuuint64_t strides[2] = {row_bytes, depth_bytes};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

}  // namespace

bool tc_supported(int z, int h, int x, int B) {
  return h == tc::HID && z % 16 == 0 && z >= 64 && z <= 256 && x % 16 == 0 && x >= 64 && B >= 1;
}

TcPlan* tc_plan_create(const TcShape& s, void* Z, void* E, int64_t e_cell, float* logits,
                       const int* nbr, const __nv_bfloat16* Gwb, const float* Gw, int64_t PGs,
                       const int64_t* goff, const __nv_bfloat16* Dwb, const float* Dw,
                       int64_t PDs, const int64_t* doff, std::string* msg) {
  if (!tc_supported(s.z, s.h, s.x, s.B)) {
    if (msg) *msg = "shape not supported by the tensor-core forward";
    return nullptr;
  }
  if (!get_encoder(msg)) return nullptr;
  TcPlan* p = new TcPlan();
  memset(p, 0, sizeof *p);
  p->s = s;
  const uint64_t C = s.cells, B = s.B, z = s.z, x = s.x, h = s.h;
  bool ok = make_map(&p->mZ, Z, z, B, C, z * 2, B * z * 2, 128, msg) &&
            make_map(&p->mE, E, x, 6 * B, C, x * 2, (uint64_t)e_cell * 2, 128, msg) &&
            make_map(&p->mG1, Gwb + goff[0], z, h, C, z * 2, PGs * 2, 256, msg) &&
            make_map(&p->mG2, Gwb + goff[2], h, h, C, h * 2, PGs * 2, 256, msg) &&
            make_map(&p->mG3, Gwb + goff[4], h, x, C, h * 2, PGs * 2, tc::N3, msg) &&
            make_map(&p->mD1, Dwb + doff[0], x, h, C, x * 2, PDs * 2, 256, msg) &&
            make_map(&p->mD2, Dwb + doff[2], h, h, C, h * 2, PDs * 2, 256, msg);
  if (!ok) {
    delete p;
    return nullptr;
  }
  if (cudaMalloc(&p->err, sizeof(int)) != cudaSuccess || cudaMemset(p->err, 0, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cudaMalloc for the error flag failed";
    delete p;
    return nullptr;
  }
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (cudaFuncSetAttribute(tc::k_mlp_fwd, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           tc::SMEM_BYTES) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cannot reserve shared memory for the tensor-core forward";
    cudaFree(p->err);
    delete p;
    return nullptr;
  }
  tc::KParams g{};
  g.kind = tc::KIND_G;
  g.cells = s.cells;
  g.B = s.B;
  g.z = s.z;
  g.x = s.x;
  g.rows = s.B;
  g.mtiles = (s.B + tc::BM - 1) / tc::BM;
  g.n_tiles = s.cells * 5 * g.mtiles;
  g.kc1 = (s.z + tc::BK - 1) / tc::BK;
  g.n3 = (s.x + tc::N3 - 1) / tc::N3;
  g.nbr = nbr;
  g.wmaster = Gw;
  g.wb = Gwb;
  g.pstride = PGs;
  g.off_b1 = goff[1];
  g.off_b2 = goff[3];
  g.off_b3 = goff[5];
  g.off_w3 = goff[4];
  g.E = (bf16*)E;
  g.e_cell = e_cell;
  g.logits = logits;
  g.slope = s.slope;
  g.err = p->err;
  tc::KParams d = g;
  d.kind = tc::KIND_D;
  d.rows = 6 * s.B;
  d.mtiles = (6 * s.B + tc::BM - 1) / tc::BM;
  d.n_tiles = s.cells * 5 * d.mtiles;
  d.kc1 = (s.x + tc::BK - 1) / tc::BK;
  d.n3 = 0;
  d.wmaster = Dw;
  d.wb = Dwb;
  d.pstride = PDs;
  d.off_b1 = doff[1];
  d.off_b2 = doff[3];
  d.off_b3 = doff[5];
  d.off_w3 = doff[4];
  p->pg = g;
  p->pd = d;
  p->grid_g = g.n_tiles < sms ? g.n_tiles : sms;
  p->grid_d = d.n_tiles < sms ? d.n_tiles : sms;
  return p;
}

int tc_run_g(TcPlan* p, cudaStream_t st, std::string* msg) {
  tc::k_mlp_fwd<<<p->grid_g, tc::THREADS, tc::SMEM_BYTES, st>>>(p->mZ, p->mG1, p->mG2, p->mG3,
                                                                p->pg);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    if (msg) *msg = std::string("generator forward launch: ") + cudaGetErrorString(e);
    return 1;
  }
  return 0;
}

int tc_run_d(TcPlan* p, cudaStream_t st, std::string* msg) {
  tc::k_mlp_fwd<<<p->grid_d, tc::THREADS, tc::SMEM_BYTES, st>>>(p->mE, p->mD1, p->mD2, p->mD2,
                                                                p->pd);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    if (msg) *msg = std::string("discriminator forward launch: ") + cudaGetErrorString(e);
    return 1;
  }
  return 0;
}

int* tc_error_flag(TcPlan* p) { return p ? p->err : nullptr; }

void tc_plan_destroy(TcPlan* p) {
  if (!p) return;
  if (p->err) cudaFree(p->err);
  delete p;
}

}  // namespace lipz
