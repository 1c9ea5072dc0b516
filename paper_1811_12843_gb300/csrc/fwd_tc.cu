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

#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <vector>

#include "common.cuh"
#include "fwd_tc.h"
#include "tc_ptx.cuh"

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
constexpr int N3 = 256;                      // generator output columns per MMA block
constexpr int NUM_EPI_WARPS = 8;
constexpr int THREADS = 64 + 32 * NUM_EPI_WARPS;
constexpr int MISC_BYTES = 2048;
constexpr int BIAS_MAX = 256 + 256 + 1024;  // floats per tile: b1, b2, then b3 (G) or w3, b3 (D)
constexpr int BIAS_BYTES = 2 * BIAS_MAX * 4;  // double-buffered by tile
constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + H_BYTES + MISC_BYTES + BIAS_BYTES;

enum { KIND_G = 0, KIND_D = 1, KIND_GRAM = 2 };
enum { EPI_TO_H = 0, EPI_LOGIT = 1, EPI_TO_E = 2, EPI_ACT_OUT = 3, EPI_GRAM = 4 };

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
  // training forward: one problem per cell, weights of individual wsel[cell], and the
  // activations of both hidden layers stored ([problem][rows][256] bf16) for the backward
  int train;
  const int* wsel;
  bf16* act1;
  bf16* act2;
  // two-part training problems (non-null): problem 2c + part of cell c takes B rows of E[c],
  // slot 0 (the real rows) or slot 1 + part_slot[c] (the selected generator's fakes), through
  // a 4-D map {x, B, 6, cells}
  const int* part_slot;
  // centre-only generator forward (non-zero): problem c is cell c's own generator on z_c,
  // written to E[c] as the fakes of slot 0
  int centre;
  int indiv_off;  // centre-only mode: individual index of cell 0's centre (snapshot * cells)
  // Gram kind (mixture score): problem c is the Gram matrix of E[c]'s rows with themselves,
  // reduced in the epilogue to per-row sums of exp(-||e_r - e_s||^2 / x) over the columns s of
  // each block of B rows. rnorm [cells][rows] holds ||e_r||^2; the sums go to
  // gram_out[cell][row][half][6], half = 2 * column block + column half of the tile.
  const float* rnorm;
  float* gram_out;
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

template <int KND>
__device__ __forceinline__ Job get_job(const KParams& p, int j) {
  Job J;
  if (KND == KIND_GRAM) {
    // column block j of the Gram matrix: MMA N rounded up to 16 (rows past 6B read as zero)
    const int n = min(HID, p.rows - j * HID);
    J = Job{0, p.kc1, (n + 15) & ~15, j & 1, 0, j * HID, HID, EPI_GRAM};
  } else if (j == 0) {
    J = Job{0, p.kc1, HID, 0, 0, 0, HID, EPI_TO_H};
  } else if (j == 1) {
    const int epi = KND == KIND_D ? EPI_LOGIT : (p.train ? EPI_ACT_OUT : EPI_TO_H);
    J = Job{1, HID / BK, HID, 1, 1, 0, HID, epi};
  } else {
    const int nb = j - 2;
    const int n = min(N3, p.x - nb * N3);
    // the last output block always lands in region 1, so the next tile's first layer
    // (region 0) need not wait for the tile's last epilogue
    J = Job{1, HID / BK, (n + 15) & ~15, (nb + p.n3) & 1, 2, nb * N3, N3, EPI_TO_E};
  }
  return J;
}

template <int KND>
__device__ __forceinline__ int n_jobs(const KParams& p) {
  if (KND == KIND_GRAM) return (p.rows + HID - 1) / HID;
  return (KND == KIND_D || p.train) ? 2 : 2 + p.n3;
}

// Problem -> (cell whose activations are the A operand, individual whose weights are B).
template <int KND>
__device__ __forceinline__ int prob_cell(const KParams& p, int prob) {
  return (p.train || p.centre || KND == KIND_GRAM) ? prob : prob / 5;
}
template <int KND>
__device__ __forceinline__ int prob_individual(const KParams& p, int prob) {
  if (p.train) return __ldg(&p.wsel[p.part_slot ? prob >> 1 : prob]);
  if (KND == KIND_GRAM) return prob;
  return p.centre ? p.indiv_off + prob : __ldg(&p.nbr[prob]);
}

// tanh from its definition, tanh(x) = 1 - 2 / (1 + e^(2x)), with e^(2x) by the hardware base-2
// exponential, for |x| >= 1/4; below that its Taylor series x - x^3/3 + 2x^5/15 - 17x^7/315 +
// 62x^9/2835 (truncation error under 1382 x^11 / 155925: relative below 1e-8). Relative error
// about 1e-6 at |x| = 1/4, where the cancellation in 1 - 2/(1 + e) is largest, and below it
// elsewhere; |x| is clamped at 16, where the fp32 value is 1.
__device__ __forceinline__ float tanh_fast(float x) {
  const float ax = fminf(fabsf(x), 16.f);
  const float e = ex2_approx(2.8853900817779268f * ax);  // e^(2|x|): 2 log2(e) |x|
  const float t = 1.f - __fdividef(2.f, 1.f + e);
  const float x2 = ax * ax;
  float q = fmaf(x2, 0.021869488536155203f, -0.053968253968253971f);
  q = fmaf(x2, q, 0.13333333333333333f);
  q = fmaf(x2, q, -0.33333333333333333f);
  const float s = ax * fmaf(x2, q, 1.f);
  return copysignf(ax < 0.25f ? s : t, x);
}

// ---- the kernel ----------------------------------------------------------------------------
// KND: p.kind at compile time (one variant per network kind, each with only its own paths)
template <int KND>
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
  const uint32_t bH = bReg + 16;      // [4]: 64-column chunk c of the activation is written
  const uint32_t bPart = bH + 32;
  const uint32_t bFinal = bPart + 8;
  const uint32_t bBias = bFinal + 8;  // [2]: the tile's biases are in shared memory
  float* s_bias = reinterpret_cast<float*>(misc + MISC_BYTES);  // [2][BIAS_MAX]
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
    for (int c = 0; c < HID / BK; ++c) mbar_init(bH + 8 * c, 32 * NUM_EPI_WARPS);
    mbar_init(bPart, 32 * NUM_EPI_WARPS / 2);
    mbar_init(bFinal, 1);
    mbar_init(bBias, 32 * NUM_EPI_WARPS);
    mbar_init(bBias + 8, 32 * NUM_EPI_WARPS);
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
  const int nj = n_jobs<KND>(p);
  // the set-up above touched no global memory: from here on the previous kernel's results
  // are needed (programmatic dependent launch)
  pdl_wait();

  if (warp == 0) {
    // ================================ TMA producer ================================
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int issued[STAGES] = {0, 0, 0};
      bool ok = true;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
        const int prob = tile / p.mtiles, m0 = (tile % p.mtiles) * BM;
        const int c = prob_cell<KND>(p, prob);
        const int k = prob_individual<KND>(p, prob);
        for (int j = 0; j < nj && ok; ++j) {
          const Job J = get_job<KND>(p, j);
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
            if (J.a_from_h) {
            } else if (p.part_slot) {
              const int cell = prob >> 1;
              const int slot = (prob & 1) ? 1 + __ldg(&p.part_slot[cell]) : 0;
              tma_load_4d(sA, &mA, full, kc * BK, m0, slot, cell);
            } else {
              tma_load_3d(sA, &mA, full, kc * BK, m0, c);
            }
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
      int h_total = 0;  // activations written to H so far (each chunk barrier: one phase each)
      bool ok = true;
      int jobs_done = 0;
      for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x) {
        for (int j = 0; j < nj && ok; ++j, ++jobs_done) {
          const Job J = get_job<KND>(p, j);
          // the Gram kind alternates the two accumulators over all its jobs (3 per tile)
          const int R = KND == KIND_GRAM ? (jobs_done & 1) : J.region;
          if (reg_uses[R] > 0 &&
              !mbar_wait(bReg + 8 * R, (uint32_t)((reg_uses[R] - 1) & 1), abort_flag, p.err, 2)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + (uint32_t)(R * HID);
          const uint32_t idesc = idesc_bf16(BM, J.n);
          for (int kc = 0; kc < J.kchunks; ++kc) {
            // a layer reading the on-chip activation starts on chunk kc as soon as the epilogue
            // has written that chunk (write number h_total - 1)
            if (J.a_from_h &&
                !mbar_wait(bH + 8 * kc, (uint32_t)((h_total - 1) & 1), abort_flag, p.err, 3)) {
              ok = false;
              break;
            }
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
    int ltile = 0, jobs_done = 0;
    const int et = threadIdx.x - 64;  // epilogue thread 0..255
    for (int tile = blockIdx.x; tile < p.n_tiles && ok; tile += gridDim.x, ++ltile) {
      const int prob = tile / p.mtiles, m0 = (tile % p.mtiles) * BM;
      const int c = prob_cell<KND>(p, prob), slot = p.centre ? 0 : prob % 5;
      const int k = prob_individual<KND>(p, prob);
      const float* wm = p.wmaster ? p.wmaster + (int64_t)k * p.pstride : nullptr;
      const int rr = m0 + row;
      const bool row_ok = rr < p.rows;
      const int64_t act_off = ((int64_t)prob * p.rows + rr) * HID;
      // The tile's biases (and D's output weights) go to shared memory once, while the MMAs
      // run, so that no epilogue waits on a global load. Buffer ltile & 1; a thread cannot
      // reach tile ltile + 2 before every thread has passed this tile's arrival.
      float* sb = s_bias + (ltile & 1) * BIAS_MAX;
      if (KND == KIND_GRAM) {
        // the squared norms of the cell's rows (the Gram tile's row and column terms)
        // -|e_s|^2 / x for the cell's rows s, zero for the 32 entries past the last row
        const float ix = 1.f / (float)p.x;
        for (int i = et; i < p.rows + 32; i += 32 * NUM_EPI_WARPS)
          sb[i] = i < p.rows ? -__ldg(&p.rnorm[(int64_t)c * p.rows + i]) * ix : 0.f;
        mbar_arrive(bBias + 8 * (ltile & 1));
        if (!mbar_wait_warp(bBias + 8 * (ltile & 1), (uint32_t)((ltile >> 1) & 1), abort_flag,
                            p.err, 8)) {
          ok = false;
          break;
        }
      } else {
        // every load is issued before the first is stored, so their latencies overlap
        const int nb3 = KND == KIND_D ? HID + 1 : p.x;
        constexpr int NV = (BIAS_MAX + 32 * NUM_EPI_WARPS - 1) / (32 * NUM_EPI_WARPS);
        float v[NV];
#pragma unroll
        for (int u = 0; u < NV; ++u) {
          const int i = et + u * 32 * NUM_EPI_WARPS;
          v[u] = 0.f;
          if (i >= 512 + nb3) continue;
          if (i < 256) v[u] = wm[p.off_b1 + i];
          else if (i < 512) v[u] = wm[p.off_b2 + i - 256];
          else if (KND == KIND_D)
            v[u] = i < 512 + HID
                       ? __bfloat162float(p.wb[(int64_t)k * p.pstride + p.off_w3 + i - 512])
                       : wm[p.off_b3];
          else v[u] = wm[p.off_b3 + i - 512];
        }
#pragma unroll
        for (int u = 0; u < NV; ++u) {
          const int i = et + u * 32 * NUM_EPI_WARPS;
          if (i < 512 + nb3) sb[i] = v[u];
        }
        mbar_arrive(bBias + 8 * (ltile & 1));
        if (!mbar_wait_warp(bBias + 8 * (ltile & 1), (uint32_t)((ltile >> 1) & 1), abort_flag,
                            p.err, 8)) {
          ok = false;
          break;
        }
      }
      for (int j = 0; j < nj && ok; ++j, ++jobs_done) {
        const Job J = get_job<KND>(p, j);
        const int R = KND == KIND_GRAM ? (jobs_done & 1) : J.region;
        if (!mbar_wait_warp(bAcc + 8 * R, (uint32_t)(reg_uses[R] & 1), abort_flag, p.err, 6)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tbase = tmem + lane_base + (uint32_t)(R * HID);
        if (J.epi == EPI_TO_H || J.epi == EPI_ACT_OUT) {
          const float* bias = sb + (j == 0 ? 0 : 256);
          const bool lrelu = KND == KIND_D;
          const bool to_h = J.epi == EPI_TO_H;
          bf16* gout = j == 0 ? p.act1 : p.act2;
          // chunk by chunk (64 columns, both column halves at once), so that the next layer's
          // MMAs can start on chunk 0 while the epilogue still writes chunks 1..3
#pragma unroll 1
          for (int ch = 0; ch < HID / BK; ++ch) {
            {
              const int cg = 2 * ch + hf;  // this warp's 32 columns of the chunk
              uint32_t r[32];
              LIPZ_TMEM_LD32(tbase + cg * 32, r);
              tmem_wait_ld();
              const float4* b4 = reinterpret_cast<const float4*>(bias + cg * 32);
              uint32_t pk[16];
#pragma unroll
              for (int e = 0; e < 32; e += 4) {
                const float4 bb = b4[e >> 2];
                float a0 = __uint_as_float(r[e]) + bb.x;
                float a1 = __uint_as_float(r[e + 1]) + bb.y;
                float a2 = __uint_as_float(r[e + 2]) + bb.z;
                float a3 = __uint_as_float(r[e + 3]) + bb.w;
                const float lo = lrelu ? p.slope : 0.f;
                a0 = a0 > 0.f ? a0 : lo * a0;
                a1 = a1 > 0.f ? a1 : lo * a1;
                a2 = a2 > 0.f ? a2 : lo * a2;
                a3 = a3 > 0.f ? a3 : lo * a3;
                pk[e >> 1] = pack_bf16(a0, a1);
                pk[(e >> 1) + 1] = pack_bf16(a2, a3);
              }
              if (to_h) {
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
              if (gout && row_ok) {
                bf16* o = gout + act_off + cg * 32;  // 256-bit stores: 32-byte aligned rows
#pragma unroll
                for (int u = 0; u < 4; u += 2)
                  st_global_v8(o + 8 * u, make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2],
                                                     pk[4 * u + 3]),
                               make_uint4(pk[4 * u + 4], pk[4 * u + 5], pk[4 * u + 6],
                                          pk[4 * u + 7]));
              }
            }
            if (to_h) {
              asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
              mbar_arrive(bH + 8 * ch);
            }
          }
          tc_fence_before();
          mbar_arrive(bReg + 8 * R);
        } else if (J.epi == EPI_LOGIT) {
          const float* bias = sb + 256;
          const float* w3 = sb + 512;
          float acc = 0.f;
#pragma unroll 1
          for (int cp = hf * 4; cp < hf * 4 + 4; cp += 2) {
            uint32_t r2[2][32];
            LIPZ_TMEM_LD32(tbase + cp * 32, r2[0]);
            LIPZ_TMEM_LD32(tbase + (cp + 1) * 32, r2[1]);
            tmem_wait_ld();
#pragma unroll
            for (int h2 = 0; h2 < 2; ++h2) {
              const int cg = cp + h2;
              const uint32_t(&r)[32] = r2[h2];
              const float4* b4 = reinterpret_cast<const float4*>(bias + cg * 32);
              const float4* w4 = reinterpret_cast<const float4*>(w3 + cg * 32);
              uint32_t pk[16];
#pragma unroll
              for (int e = 0; e < 32; e += 4) {
                const float4 bb = b4[e >> 2], ww = w4[e >> 2];
                float a0 = __uint_as_float(r[e]) + bb.x;
                float a1 = __uint_as_float(r[e + 1]) + bb.y;
                float a2 = __uint_as_float(r[e + 2]) + bb.z;
                float a3 = __uint_as_float(r[e + 3]) + bb.w;
                a0 = a0 > 0.f ? a0 : p.slope * a0;
                a1 = a1 > 0.f ? a1 : p.slope * a1;
                a2 = a2 > 0.f ? a2 : p.slope * a2;
                a3 = a3 > 0.f ? a3 : p.slope * a3;
                pk[e >> 1] = pack_bf16(a0, a1);
                pk[(e >> 1) + 1] = pack_bf16(a2, a3);
                const __nv_bfloat162 q01 = *reinterpret_cast<const __nv_bfloat162*>(&pk[e >> 1]);
                const __nv_bfloat162 q23 =
                    *reinterpret_cast<const __nv_bfloat162*>(&pk[(e >> 1) + 1]);
                acc = fmaf(__low2float(q01), ww.x, acc);
                acc = fmaf(__high2float(q01), ww.y, acc);
                acc = fmaf(__low2float(q23), ww.z, acc);
                acc = fmaf(__high2float(q23), ww.w, acc);
              }
              if (p.act2 && row_ok) {
                bf16* o = p.act2 + act_off + cg * 32;
#pragma unroll
                for (int u = 0; u < 4; u += 2)
                  st_global_v8(o + 8 * u, make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2],
                                                     pk[4 * u + 3]),
                               make_uint4(pk[4 * u + 4], pk[4 * u + 5], pk[4 * u + 6],
                                          pk[4 * u + 7]));
              }
            }
          }
          tc_fence_before();
          if (hf == 1) {
            part[row] = acc;
            mbar_arrive(bPart);
            mbar_arrive(bReg + 8 * R);
          } else {
            if (!mbar_wait_warp(bPart, (uint32_t)(reg_uses[R] & 1), abort_flag, p.err, 7)) {
              ok = false;
              break;
            }
            const float logit = acc + part[row] + sb[512 + HID];
            mbar_arrive(bReg + 8 * R);
            if (row_ok) p.logits[(int64_t)prob * p.rows + rr] = logit;
          }
        } else if (J.epi == EPI_GRAM) {
          // Gaussian kernel exp((2 e_r.e_s - |e_r|^2 - |e_s|^2) / x) of this thread's row r
          // against the warp's 128 columns s, summed per column block of B >= 32 rows: a group
          // of 32 columns meets at most one block boundary (at column sp of the group, the same
          // for every lane), columns past the last row count zero; two interleaved partial sums
          // per side, combined in a fixed order
          const float nr = row_ok ? sb[rr] : 0.f;
          const float two_ix = 2.f / (float)p.x;
          float acc[6] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll 1
          for (int cg = hf * 4; cg < hf * 4 + 4; ++cg) {
            const int col0 = J.brow0 + cg * 32;
            if (col0 >= p.rows) break;
            uint32_t r[32];
            LIPZ_TMEM_LD32(tbase + cg * 32, r);
            tmem_wait_ld();
            const int blk = col0 / p.B;
            const int sp = (blk + 1) * p.B - col0;
            const int nv = p.rows - col0;
            const float4* s4 = reinterpret_cast<const float4*>(sb + col0);
            float lo0 = 0.f, lo1 = 0.f, hi0 = 0.f, hi1 = 0.f;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const float4 ns = s4[q];
              const float nsv[4] = {ns.x, ns.y, ns.z, ns.w};
#pragma unroll
              for (int u = 0; u < 4; ++u) {
                const int e = 4 * q + u;
                float v = __expf(fmaf(__uint_as_float(r[e]), two_ix, nr + nsv[u]));
                v = e < nv ? v : 0.f;
                const float vl = e < sp ? v : 0.f, vh = e < sp ? 0.f : v;
                if (e & 1) {
                  lo1 += vl;
                  hi1 += vh;
                } else {
                  lo0 += vl;
                  hi0 += vh;
                }
              }
            }
            const float lo = lo0 + lo1, hi = hi0 + hi1;
#pragma unroll
            for (int t = 0; t < 6; ++t) acc[t] += t == blk ? lo : (t == blk + 1 ? hi : 0.f);
          }
          tc_fence_before();
          mbar_arrive(bReg + 8 * R);
          if (row_ok) {
            float* o = p.gram_out + (((int64_t)c * p.rows + rr) * (2 * nj) + 2 * j + hf) * 6;
#pragma unroll
            for (int t = 0; t < 6; ++t) o[t] = acc[t];
          }
        } else {
          // generator output block: bias + tanh, bf16, into the fake rows of E[c]
          const float* bias = sb + 512;
          const int ng = J.n / 16;
          const int split = (ng + 1) / 2;
          const int g0 = hf ? split : 0, g1 = hf ? ng : split;
          bf16* dst = p.E + (int64_t)c * p.e_cell + (int64_t)((1 + slot) * p.B + rr) * p.x;
#pragma unroll 1
          for (int gi = g0; gi < g1; ++gi) {
            uint32_t r[16];
            LIPZ_TMEM_LD16(tbase + gi * 16, r);
            tmem_wait_ld();
            const int col0 = J.brow0 + gi * 16;
            float bv[16];
            {
              const float4* b4 = reinterpret_cast<const float4*>(bias + col0);
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const float4 t = b4[q];
                bv[4 * q] = t.x;
                bv[4 * q + 1] = t.y;
                bv[4 * q + 2] = t.z;
                bv[4 * q + 3] = t.w;
              }
            }
            uint32_t pk[8];
#pragma unroll
            for (int e = 0; e < 16; e += 2)
              pk[e >> 1] = pack_bf16(tanh_fast(__uint_as_float(r[e]) + bv[e]),
                                     tanh_fast(__uint_as_float(r[e + 1]) + bv[e + 1]));
            if (rr < p.B && col0 < p.x)  // one 256-bit store per row and 16 columns
              st_global_v8(dst + col0, make_uint4(pk[0], pk[1], pk[2], pk[3]),
                           make_uint4(pk[4], pk[5], pk[6], pk[7]));
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


// ---- evaluation by CTA pairs (tcgen05 .cta_group::2) ----------------------------------------
// The two CTAs of a cluster share every weight chunk: each loads half of the chunk's rows
// (128 of the 256 output columns), holds its own 128 rows of the activations, and the pair's
// MMAs (M = 256, issued by rank 0) read both halves, so a weight byte brought from L2 serves
// 256 rows instead of 128. A pair works on one individual:
//   generator: the individual's 5B rows (the z rows of every cell whose neighbourhood holds it,
//              in the order of its (cell, slot) problems), two 128-row blocks per pair; the
//              noise rows are gathered into shared memory by a warp of their own;
//   discriminator: two 128-row tiles of (cell, slot) problems that share the individual (a
//              lone tile's partner computes zeros and stores nothing).
constexpr int HB_BYTES = (HID / 2) * BK * 2;  // 16 KB: half of a 256-row weight box

template <int KND>
struct PCfg;
// generator: rings of weight halves only (its first layer's A is the gathered noise tile);
// sixteen epilogue warps (its output epilogue, tanh and the fakes' stores, is the longest)
template <>
struct PCfg<KIND_G> {
  static constexpr int STAGES = 8, STAGE = HB_BYTES, A_IN = 0, ZBUF = A_BYTES, NE = 16;
};
// discriminator: each stage holds the A chunk and the weight half; eight epilogue warps (two
// column halves: the logit's two partial dot products are added in the one-CTA kernel's order)
template <>
struct PCfg<KIND_D> {
  static constexpr int STAGES = 4, STAGE = A_BYTES + HB_BYTES, A_IN = 1, ZBUF = 0, NE = 8;
};
// warps: producer, MMA issuer, NE epilogue warps, noise gather
template <int KND>
constexpr int pair_threads() {
  return 32 * (3 + PCfg<KND>::NE);
}
template <int KND>
constexpr int pair_smem_bytes() {
  return 1024 + PCfg<KND>::STAGES * PCfg<KND>::STAGE + PCfg<KND>::ZBUF + H_BYTES + MISC_BYTES +
         BIAS_BYTES;
}
static_assert(pair_smem_bytes<KIND_G>() <= 232448, "generator pair kernel: shared memory");
static_assert(pair_smem_bytes<KIND_D>() <= 232448, "discriminator pair kernel: shared memory");
static_assert(2 * PCfg<KIND_G>::STAGES + 14 <= 32, "barriers must fit below the TMEM slot");

struct PParams {
  int B, x, rows;  // rows per problem: B (generator) or 6B (discriminator)
  int kc1, n3;
  int n_pairs;
  // generator: {individual, first row of the pair's 256, offset into plist, rows of the
  // individual}; discriminator: {individual, problem of rank 0, problem of rank 1 (-1: none),
  // first row of rank 0's tile << 16 | first row of rank 1's tile}; problem = cell * 5 + slot
  const int4* pairs;
  const int2* plist;  // generator: (cell, slot) of each problem of an individual, in row order
  const bf16* Z;      // generator: noise [cells][B][64]
  const float* wmaster;
  const bf16* wb;
  int64_t pstride;
  int64_t off_b1, off_b2, off_b3, off_w3;
  bf16* E;
  int64_t e_cell;
  float* logits;
  float slope;
  int* err;
  // discriminator training forward (train != 0): pair job c * mt + t takes m-tile t of both
  // parts of cell c through discriminator wsel[c]: rank 0 the B real rows (slot 0 of E[c]),
  // rank 1 the selected generator's fakes (slot 1 + part_slot[c]); both hidden activations go
  // to act1 / act2 ([2c + part][B][256] bf16), the logits to logits[(2c + part) B + row]
  int train, mt;
  const int* wsel;
  const int* part_slot;
  bf16* act1;
  bf16* act2;
};

template <int KND>
__device__ __forceinline__ Job pair_job(const PParams& p, int j) {
  if (j == 0) return Job{0, p.kc1, HID, 0, 0, 0, HID, EPI_TO_H};
  if (j == 1) return Job{1, HID / BK, HID, 1, 1, 0, HID, KND == KIND_D ? EPI_LOGIT : EPI_TO_H};
  const int nb = j - 2;
  const int n = min(N3, p.x - nb * N3);
  return Job{1, HID / BK, (n + 15) & ~15, (nb + p.n3) & 1, 2, nb * N3, N3, EPI_TO_E};
}

template <int KND>
__global__ void __launch_bounds__(pair_threads<KND>(), 1)
    k_mlp_fwd_pair(const __grid_constant__ CUtensorMap mA, const __grid_constant__ CUtensorMap mB1,
                   const __grid_constant__ CUtensorMap mB2, const __grid_constant__ CUtensorMap mB3,
                   const PParams p) {
  using CF = PCfg<KND>;
  constexpr int NE = CF::NE;               // epilogue warps
  constexpr int CP = NE / 4;               // column parts (warps per TMEM lane quarter)
  constexpr int ARRIVALS = 2 * NE;         // one per epilogue warp of both CTAs
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sStage = base;                        // STAGES x ([A] | weight half)
  const uint32_t sZ = base + CF::STAGES * CF::STAGE;   // generator: the gathered noise rows
  const uint32_t sH = sZ + CF::ZBUF;                   // on-chip activation (own 128 rows)
  uint8_t* misc = gbase + CF::STAGES * CF::STAGE + CF::ZBUF + H_BYTES;
  uint64_t* bars = reinterpret_cast<uint64_t*>(misc);
  const uint32_t bFull = smem_u32(bars);               // [STAGES], used in rank 0
  const uint32_t bEmpty = bFull + 8 * CF::STAGES;      // [STAGES]
  const uint32_t bAcc = bEmpty + 8 * CF::STAGES;       // [2]
  const uint32_t bReg = bAcc + 16;                     // [2], rank 0
  const uint32_t bH = bReg + 16;                       // [4], rank 0
  const uint32_t bPart = bH + 32;
  const uint32_t bFinal = bPart + 8;
  const uint32_t bBias = bFinal + 8;                   // [2]
  const uint32_t bZfull = bBias + 16;                  // rank 0
  const uint32_t bZempty = bZfull + 8;
  float* s_bias = reinterpret_cast<float*>(misc + MISC_BYTES);
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(misc + 256);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 260);
  float* part_buf = reinterpret_cast<float*>(misc + 512);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < CF::STAGES; ++s) {
      mbar_init(bFull + 8 * s, 1);
      mbar_init(bEmpty + 8 * s, 1);
    }
    for (int r = 0; r < 2; ++r) {
      mbar_init(bAcc + 8 * r, 1);
      mbar_init(bReg + 8 * r, ARRIVALS);
      mbar_init(bBias + 8 * r, 32 * NE);
    }
    for (int c = 0; c < HID / BK; ++c) mbar_init(bH + 8 * c, ARRIVALS);
    mbar_init(bPart, 32 * NE / 2);
    mbar_init(bFinal, 1);
    mbar_init(bZfull, 2);
    mbar_init(bZempty, 1);
    *abort_flag = 0;
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  if (warp == 1) {
    // one warp of each CTA of the pair allocates together: the same columns in both
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], 512;" ::"r"(
        smem_u32((const void*)tmem_slot)));
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;");
  }
  tc_fence_before();
  cluster_sync_all();  // no remote arrival before the peer's barriers exist
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // rank 0's barriers that both CTAs arrive on
  const uint32_t lFull = mapa_shared(bFull, 0), lReg = mapa_shared(bReg, 0);
  const uint32_t lH = mapa_shared(bH, 0), lZfull = mapa_shared(bZfull, 0);
  const int nj = KND == KIND_D ? 2 : 2 + p.n3;
  const int cid = (int)cluster_id_x(), ncl = (int)nclusters_x();
  pdl_wait();

  if (warp == 0) {
    // ================================ TMA producer (both CTAs) ================================
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int pi = cid; pi < p.n_pairs && ok; pi += ncl) {
        const bool train = KND == KIND_D && p.train;
        const int4 pr = train ? make_int4(0, 0, 0, 0) : __ldg(&p.pairs[pi]);
        const int k = train ? __ldg(&p.wsel[pi / p.mt]) : pr.x;
        int a_cell = 0, a_row = p.rows;  // no problem: rows past the end read as zero
        if (train) {
          // (rows of the tile past the part's B read the next slot's rows: never stored)
          const int cell = pi / p.mt, t = pi - cell * p.mt;
          a_cell = cell;
          a_row = (rank ? 1 + __ldg(&p.part_slot[cell]) : 0) * p.B + t * BM;
        } else if (KND == KIND_D) {
          const int prob = rank ? pr.z : pr.y;
          if (prob >= 0) {
            a_cell = prob / 5;
            a_row = rank ? (pr.w & 0xFFFF) : (pr.w >> 16);
          }
        }
        for (int j = 0; j < nj && ok; ++j) {
          const Job J = pair_job<KND>(p, j);
          const CUtensorMap* mb = J.bmap == 0 ? &mB1 : (J.bmap == 1 ? &mB2 : &mB3);
          const bool a_ring = CF::A_IN && !J.a_from_h;
          const uint32_t bytes = (a_ring ? (uint32_t)A_BYTES : 0u) + (uint32_t)HB_BYTES;
          for (int kc = 0; kc < J.kchunks; ++kc) {
            if (!mbar_wait(bEmpty + 8 * stage, phase ^ 1u, abort_flag, p.err, 1)) {
              ok = false;
              break;
            }
            // rank 0 expects both CTAs' bytes; the peer's may land first
            if (leader) mbar_expect_tx(bFull + 8 * stage, 2 * bytes);
            const uint32_t sS = sStage + stage * CF::STAGE;
            const uint32_t full = lFull + 8 * stage;
            if (a_ring) tma_load_3d_cg2(sS, &mA, full, kc * BK, a_row, a_cell);
            tma_load_3d_cg2(sS + (CF::A_IN ? A_BYTES : 0), mb, full, kc * BK,
                            J.brow0 + (int)rank * (J.n / 2), k);
            if (++stage == CF::STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
        }
      }
      if (!ok) {
        // loads issued here complete on rank 0's barriers: give them time to land before the
        // CTA leaves
        const unsigned long long t0 = globaltimer();
        while (globaltimer() - t0 < 200000ull) {
        }
      }
    }
  } else if (warp == 1) {
    // ================================ MMA issuer (rank 0) ================================
    if (leader && lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      int reg_uses[2] = {0, 0};
      int h_total = 0, zuse = 0;
      int h_seen[HID / BK] = {0, 0, 0, 0};  // activation write each chunk was last waited for
      bool ok = true;
      for (int pi = cid; pi < p.n_pairs && ok; pi += ncl) {
        for (int j = 0; j < nj && ok; ++j) {
          const Job J = pair_job<KND>(p, j);
          const int R = J.region;
          if (reg_uses[R] > 0 &&
              !mbar_wait(bReg + 8 * R, (uint32_t)((reg_uses[R] - 1) & 1), abort_flag, p.err, 2)) {
            ok = false;
            break;
          }
          if (KND == KIND_G && j == 0 &&
              !mbar_wait(bZfull, (uint32_t)(zuse & 1), abort_flag, p.err, 9)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + (uint32_t)(R * HID);
          const uint32_t idesc = idesc_bf16(2 * BM, J.n);
          for (int kc = 0; kc < J.kchunks; ++kc) {
            // (the generator's output blocks read the same activation: wait for it once)
            if (J.a_from_h && h_seen[kc] != h_total) {
              if (!mbar_wait(bH + 8 * kc, (uint32_t)((h_total - 1) & 1), abort_flag, p.err, 3)) {
                ok = false;
                break;
              }
              h_seen[kc] = h_total;
            }
            if (!mbar_wait(bFull + 8 * stage, phase, abort_flag, p.err, 4)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sS = sStage + stage * CF::STAGE;
            const uint32_t sA = (KND == KIND_G && j == 0)
                                    ? sZ
                                    : (J.a_from_h ? sH + kc * H_CHUNK : sS);
            const uint32_t sB = sS + (CF::A_IN ? A_BYTES : 0);
            // a 16-element K step is 32 bytes: 2 in the descriptors' address field (a 1024-byte
            // aligned tile plus at most 96 bytes never carries out of it)
            const uint64_t dA = sw128_desc(sA), dB = sw128_desc(sB);
            tc_mma_cg2(d, dA, dB, idesc, kc != 0 ? 1u : 0u);
#pragma unroll
            for (int kk = 1; kk < BK / 16; ++kk)
              tc_mma_cg2_acc(d, dA + 2 * kk, dB + 2 * kk, idesc);
            tc_commit_cg2(bEmpty + 8 * stage, 3);
            if (++stage == CF::STAGES) {
              stage = 0;
              phase ^= 1u;
            }
          }
          if (!ok) break;
          if (KND == KIND_G && j == 0) {
            tc_commit_cg2(bZempty, 3);
            ++zuse;
          }
          tc_commit_cg2(bAcc + 8 * R, 3);
          reg_uses[R]++;
          if (J.epi == EPI_TO_H) ++h_total;
        }
      }
      // every MMA (they write both CTAs' tensor memory) completes before it is released
      tc_commit_cg2(bFinal, 3);
      volatile int never = 0;
      mbar_wait(bFinal, 0u, &never, p.err, 5);
    }
  } else if (warp < 2 + NE) {
    // ================================ epilogue (own 128 rows) ================================
    const int ew = warp - 2;
    const int q = warp & 3;          // TMEM lane quarter this warp may access
    const int part = ew >> 2;        // column part: HID / CP columns of every region
    const int row = q * 32 + lane;
    const uint32_t lane_base = (uint32_t)(q * 32) << 16;
    const int et = threadIdx.x - 64;
    int reg_uses[2] = {0, 0};
    bool ok = true;
    int ltile = 0;
    // a warp's share is done (tensor memory read; for H chunks the rows written and made
    // visible to the tensor cores by every lane's proxy fence): lane 0 arrives on rank 0's
    // barrier. The H chunk is this CTA's own shared memory, read by this SM's tensor core.
    auto warp_signal = [&](uint32_t bar_cluster) {
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(bar_cluster);
    };
    // a tile's biases (and the discriminator's output weights): this thread's share, loaded
    // from global memory one tile ahead, so that a tile's staging waits on no memory latency
    // (the generator's first layer, one K chunk, does not cover it)
    constexpr int NV = (BIAS_MAX + 32 * NE - 1) / (32 * NE);
    auto load_bias = [&](int kk, float (&v)[NV]) {
      const float* wm = p.wmaster + (int64_t)kk * p.pstride;
      const int nb3 = KND == KIND_D ? HID + 1 : p.x;
#pragma unroll
      for (int u = 0; u < NV; ++u) {
        const int i = et + u * 32 * NE;
        v[u] = 0.f;
        if (i >= 512 + nb3) continue;
        if (i < 256) v[u] = wm[p.off_b1 + i];
        else if (i < 512) v[u] = wm[p.off_b2 + i - 256];
        else if (KND == KIND_D)
          v[u] = i < 512 + HID
                     ? __bfloat162float(p.wb[(int64_t)kk * p.pstride + p.off_w3 + i - 512])
                     : wm[p.off_b3];
        else v[u] = wm[p.off_b3 + i - 512];
      }
    };
    auto tile_individual = [&](int q) {
      return (KND == KIND_D && p.train) ? __ldg(&p.wsel[q / p.mt]) : __ldg(&p.pairs[q]).x;
    };
    float vb[NV];
    if (cid < p.n_pairs) load_bias(tile_individual(cid), vb);
    for (int pi = cid; pi < p.n_pairs && ok; pi += ncl, ++ltile) {
      const bool train = KND == KIND_D && p.train;
      const int4 pr = train ? make_int4(0, 0, 0, 0) : __ldg(&p.pairs[pi]);
      const int k = train ? __ldg(&p.wsel[pi / p.mt]) : pr.x;
      bool row_ok;
      bf16* dst = nullptr;   // generator: this row of the fakes
      int64_t lidx = 0;      // discriminator: this row's logit (training: and activations)
      if (train) {
        const int cell = pi / p.mt, rr = (pi - cell * p.mt) * BM + row;
        row_ok = rr < p.B;
        lidx = (int64_t)(2 * cell + (int)rank) * p.B + rr;
      } else if (KND == KIND_G) {
        const int gr = pr.y + (int)rank * BM + row;
        row_ok = gr < pr.w;
        if (row_ok) {
          const int pp = gr / p.B, b = gr - pp * p.B;
          const int2 cs = __ldg(&p.plist[pr.z + pp]);
          dst = p.E + (int64_t)cs.x * p.e_cell + (int64_t)((1 + cs.y) * p.B + b) * p.x;
        }
      } else {
        const int prob = rank ? pr.z : pr.y;
        const int rr = (rank ? (pr.w & 0xFFFF) : (pr.w >> 16)) + row;
        row_ok = prob >= 0 && rr < p.rows;
        lidx = (int64_t)prob * p.rows + rr;
      }
      (void)k;
      float* sb = s_bias + (ltile & 1) * BIAS_MAX;
      {
        const int nb3 = KND == KIND_D ? HID + 1 : p.x;
#pragma unroll
        for (int u = 0; u < NV; ++u) {
          const int i = et + u * 32 * NE;
          if (i < 512 + nb3) sb[i] = vb[u];
        }
        // the next tile's, in flight while this one computes
        if (pi + ncl < p.n_pairs) load_bias(tile_individual(pi + ncl), vb);
        mbar_arrive(bBias + 8 * (ltile & 1));
        if (!mbar_wait_warp(bBias + 8 * (ltile & 1), (uint32_t)((ltile >> 1) & 1), abort_flag,
                            p.err, 8)) {
          ok = false;
          break;
        }
      }
      for (int j = 0; j < nj && ok; ++j) {
        const Job J = pair_job<KND>(p, j);
        const int R = J.region;
        if (!mbar_wait_warp(bAcc + 8 * R, (uint32_t)(reg_uses[R] & 1), abort_flag, p.err, 6)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tbase = tmem + lane_base + (uint32_t)(R * HID);
        if (J.epi == EPI_TO_H) {
          // chunk by chunk (64 columns; this warp's 64 / CP of each), so that the next layer
          // starts on chunk 0 while the others are written
          const float* bias = sb + (j == 0 ? 0 : 256);
          const float lo = KND == KIND_D ? p.slope : 0.f;
          constexpr int W = BK / CP;  // columns of a chunk per warp: 32 or 16
#pragma unroll 1
          for (int ch = 0; ch < HID / BK; ++ch) {
            const int col0 = ch * BK + part * W;
            uint32_t r[W];
            if (W == 32) {
              LIPZ_TMEM_LD32(tbase + col0, r);
            } else {
              LIPZ_TMEM_LD16(tbase + col0, r);
            }
            tmem_wait_ld();
            const float4* b4 = reinterpret_cast<const float4*>(bias + col0);
            uint32_t pk[W / 2];
#pragma unroll
            for (int e = 0; e < W; e += 4) {
              const float4 bb = b4[e >> 2];
              float a0 = __uint_as_float(r[e]) + bb.x;
              float a1 = __uint_as_float(r[e + 1]) + bb.y;
              float a2 = __uint_as_float(r[e + 2]) + bb.z;
              float a3 = __uint_as_float(r[e + 3]) + bb.w;
              a0 = a0 > 0.f ? a0 : lo * a0;
              a1 = a1 > 0.f ? a1 : lo * a1;
              a2 = a2 > 0.f ? a2 : lo * a2;
              a3 = a3 > 0.f ? a3 : lo * a3;
              pk[e >> 1] = pack_bf16(a0, a1);
              pk[(e >> 1) + 1] = pack_bf16(a2, a3);
            }
            const uint32_t chunk = sH + (uint32_t)(ch * H_CHUNK) + (uint32_t)row * 128u;
#pragma unroll
            for (int u = 0; u < W / 8; ++u) {
              const uint32_t unit = (uint32_t)(part * (W / 8) + u);
              const uint32_t addr = chunk + ((unit ^ (uint32_t)(row & 7)) << 4);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(pk[4 * u]),
                           "r"(pk[4 * u + 1]), "r"(pk[4 * u + 2]), "r"(pk[4 * u + 3])
                           : "memory");
            }
            if (train && j == 0 && row_ok) {
              bf16* o = p.act1 + lidx * HID + col0;  // 256-bit stores: 32-byte aligned rows
#pragma unroll
              for (int u = 0; u < W / 8; u += 2)
                st_global_v8(o + 8 * u, make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2],
                                                   pk[4 * u + 3]),
                             make_uint4(pk[4 * u + 4], pk[4 * u + 5], pk[4 * u + 6],
                                        pk[4 * u + 7]));
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            warp_signal(lH + 8 * ch);
          }
          tc_fence_before();
          warp_signal(lReg + 8 * R);
        } else if (KND == KIND_D && J.epi == EPI_LOGIT) {
          // LeakyReLU of layer 2, rounded to bf16, dotted with the output weights: each column
          // half's partial dot product, the halves added as in the one-CTA kernel
          const float* bias = sb + 256;
          const float* w3 = sb + 512;
          float acc = 0.f;
#pragma unroll 1
          for (int cp = part * 4; cp < part * 4 + 4; cp += 2) {
            uint32_t r2[2][32];
            LIPZ_TMEM_LD32(tbase + cp * 32, r2[0]);
            LIPZ_TMEM_LD32(tbase + (cp + 1) * 32, r2[1]);
            tmem_wait_ld();
#pragma unroll
            for (int h2 = 0; h2 < 2; ++h2) {
              const int cg = cp + h2;
              const uint32_t(&r)[32] = r2[h2];
              const float4* b4 = reinterpret_cast<const float4*>(bias + cg * 32);
              const float4* w4 = reinterpret_cast<const float4*>(w3 + cg * 32);
              uint32_t pk[16];
#pragma unroll
              for (int e = 0; e < 32; e += 4) {
                const float4 bb = b4[e >> 2], ww = w4[e >> 2];
                float a0 = __uint_as_float(r[e]) + bb.x;
                float a1 = __uint_as_float(r[e + 1]) + bb.y;
                float a2 = __uint_as_float(r[e + 2]) + bb.z;
                float a3 = __uint_as_float(r[e + 3]) + bb.w;
                a0 = a0 > 0.f ? a0 : p.slope * a0;
                a1 = a1 > 0.f ? a1 : p.slope * a1;
                a2 = a2 > 0.f ? a2 : p.slope * a2;
                a3 = a3 > 0.f ? a3 : p.slope * a3;
                const uint32_t q01 = pack_bf16(a0, a1), q23 = pack_bf16(a2, a3);
                pk[e >> 1] = q01;
                pk[(e >> 1) + 1] = q23;
                const __nv_bfloat162 v01 = *reinterpret_cast<const __nv_bfloat162*>(&q01);
                const __nv_bfloat162 v23 = *reinterpret_cast<const __nv_bfloat162*>(&q23);
                acc = fmaf(__low2float(v01), ww.x, acc);
                acc = fmaf(__high2float(v01), ww.y, acc);
                acc = fmaf(__low2float(v23), ww.z, acc);
                acc = fmaf(__high2float(v23), ww.w, acc);
              }
              if (train && row_ok) {
                bf16* o = p.act2 + lidx * HID + cg * 32;
#pragma unroll
                for (int u = 0; u < 4; u += 2)
                  st_global_v8(o + 8 * u, make_uint4(pk[4 * u], pk[4 * u + 1], pk[4 * u + 2],
                                                     pk[4 * u + 3]),
                               make_uint4(pk[4 * u + 4], pk[4 * u + 5], pk[4 * u + 6],
                                          pk[4 * u + 7]));
              }
            }
          }
          tc_fence_before();
          if (part == 1) {
            part_buf[row] = acc;
            mbar_arrive(bPart);
            warp_signal(lReg + 8 * R);
          } else {
            if (!mbar_wait_warp(bPart, (uint32_t)(reg_uses[R] & 1), abort_flag, p.err, 7)) {
              ok = false;
              break;
            }
            const float logit = acc + part_buf[row] + sb[512 + HID];
            warp_signal(lReg + 8 * R);
            if (row_ok) p.logits[lidx] = logit;
          }
        } else if (KND == KIND_G) {
          // generator output block: bias + tanh, bf16, into this row's fakes; this warp's
          // share of the block's 16-column groups
          const float* bias = sb + 512;
          const int ng = J.n / 16;
          const int per = (ng + CP - 1) / CP;
          const int g0 = part * per, g1 = min(ng, g0 + per);
#pragma unroll 1
          for (int gi = g0; gi < g1; ++gi) {
            uint32_t r[16];
            LIPZ_TMEM_LD16(tbase + gi * 16, r);
            tmem_wait_ld();
            const int col0 = J.brow0 + gi * 16;
            const float4* b4 = reinterpret_cast<const float4*>(bias + col0);
            uint32_t pk[8];
#pragma unroll
            for (int qq = 0; qq < 4; ++qq) {
              const float4 t = b4[qq];
              pk[2 * qq] = pack_bf16(tanh_fast(__uint_as_float(r[4 * qq]) + t.x),
                                     tanh_fast(__uint_as_float(r[4 * qq + 1]) + t.y));
              pk[2 * qq + 1] = pack_bf16(tanh_fast(__uint_as_float(r[4 * qq + 2]) + t.z),
                                         tanh_fast(__uint_as_float(r[4 * qq + 3]) + t.w));
            }
            if (row_ok && col0 < p.x)  // one 256-bit store per row and 16 columns (E's rows,
                                       // slots and cells are 32-byte aligned: x % 16 == 0)
              st_global_v8(dst + col0, make_uint4(pk[0], pk[1], pk[2], pk[3]),
                           make_uint4(pk[4], pk[5], pk[6], pk[7]));
          }
          tc_fence_before();
          warp_signal(lReg + 8 * R);
        }
        reg_uses[R]++;
      }
    }
  } else if (KND == KIND_G) {
    // ================================ noise gather (generator) ================================
    // this CTA's 128 rows of the individual's z rows, 16-byte units in the 128-byte swizzle
    int zuse = 0;
    for (int pi = cid; pi < p.n_pairs; pi += ncl, ++zuse) {
      const int4 pr = __ldg(&p.pairs[pi]);
      if (zuse > 0 &&
          !mbar_wait_warp(bZempty, (uint32_t)((zuse - 1) & 1), abort_flag, p.err, 10))
        break;
      const int row0 = pr.y + (int)rank * BM;
#pragma unroll 1
      for (int t0 = 0; t0 < 32; t0 += 8) {
        uint4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int idx = lane + 32 * (t0 + u);
          const int r = idx >> 3, c16 = idx & 7;
          const int gr = row0 + r;
          v[u] = make_uint4(0u, 0u, 0u, 0u);
          if (gr < pr.w) {
            const int pp = gr / p.B, b = gr - pp * p.B;
            const int2 cs = __ldg(&p.plist[pr.z + pp]);
            v[u] = __ldg(reinterpret_cast<const uint4*>(p.Z + ((int64_t)cs.x * p.B + b) * BK) +
                         c16);
          }
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int idx = lane + 32 * (t0 + u);
          const int r = idx >> 3, c16 = idx & 7;
          const uint32_t addr = sZ + (uint32_t)r * 128u + ((uint32_t)(c16 ^ (r & 7)) << 4);
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v[u].x),
                       "r"(v[u].y), "r"(v[u].z), "r"(v[u].w)
                       : "memory");
        }
      }
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0) mbar_arrive_remote(lZfull);
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // neither CTA leaves while the peer may still arrive on its barriers
  tc_fence_after();
  if (warp == 1) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, 512;" ::"r"(tmem));
  }
}

}  // namespace tc

// ---- host side -----------------------------------------------------------------------------
struct TcPlan {
  TcShape s;
  CUtensorMap mZ, mE, mG1, mG2, mG3, mD1, mD2, mE4, mEB;
  // weight maps of the CTA-pair kernels: boxes of half the output columns (128 rows)
  CUtensorMap mG1h, mG2h, mG3h, mD1h, mD2h;
  tc::KParams pg, pgc, pd, pgt, pdt, pgram;
  tc::PParams ppg, ppd, ppdt;
  int grid_g, grid_gc, grid_d, grid_gt, grid_dt, grid_gram;
  int ncl_g, ncl_d;        // co-resident clusters of the pair kernels (0: pair path off)
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

// bf16 4-D map {inner, rows, slots, depth}; box {64, 128, 1, 1}, 128-byte swizzle: rows past
// `rows` within a slot read as zero.
bool make_map4(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t slots,
               uint64_t depth, uint64_t row_bytes, uint64_t slot_bytes, uint64_t depth_bytes,
               std::string* msg) {
  cuuint64_t dims[4] = {inner, rows, slots, depth};
  cuuint64_t strides[3] = {row_bytes, slot_bytes, depth_bytes};
  cuuint32_t box[4] = {64, (cuuint32_t)tc::BM, 1, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims,
                        strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled (4-D) failed (" + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

// Launch on clusters of two CTAs (the pairs), with programmatic dependent launch on a created
// stream as launch_kernel does.
template <typename... KArgs, typename... Args>
cudaError_t launch_pairs(void (*kernel)(KArgs...), int clusters, int threads, size_t smem,
                         cudaStream_t st, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * clusters);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  const bool shared = st == nullptr || st == cudaStreamLegacy || st == cudaStreamPerThread;
  cfg.attrs = attr;
  cfg.numAttrs = shared ? 1 : 2;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Clusters of two that can be resident at once (one CTA per SM), 0 if the query fails.
template <typename K>
int max_pair_clusters(K kernel, int threads, size_t smem) {
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
      cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute a;
  a.id = cudaLaunchAttributeClusterDimension;
  a.val.clusterDim.x = 2;
  a.val.clusterDim.y = 1;
  a.val.clusterDim.z = 1;
  cfg.attrs = &a;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, (const void*)kernel, &cfg) != cudaSuccess) {
    cudaGetLastError();
    return 0;
  }
  return n;
}

}  // namespace

void tc_build_pairs(const int* nbr, int cells, int n_indiv, int B, std::vector<int4>* gpairs,
                    std::vector<int4>* dpairs, std::vector<int2>* plist) {
  std::vector<std::vector<int>> lists(n_indiv);  // problems (cell * 5 + slot) per individual
  for (int i = 0; i < cells * 5; ++i) lists[nbr[i]].push_back(i);
  gpairs->clear();
  dpairs->clear();
  plist->clear();
  const int mt = (6 * B + tc::BM - 1) / tc::BM;
  for (int k = 0; k < n_indiv; ++k) {
    const std::vector<int>& L = lists[k];
    if (L.empty()) continue;
    const int off = (int)plist->size();
    for (int pr : L) plist->push_back(make_int2(pr / 5, pr % 5));
    const int nr = (int)L.size() * B;
    for (int r0 = 0; r0 < nr; r0 += 2 * tc::BM) gpairs->push_back(make_int4(k, r0, off, nr));
    std::vector<int2> tiles;  // (problem, first row)
    for (int pr : L)
      for (int t = 0; t < mt; ++t) tiles.push_back(make_int2(pr, t * tc::BM));
    for (size_t i = 0; i < tiles.size(); i += 2) {
      const int2 a = tiles[i];
      const int2 b = i + 1 < tiles.size() ? tiles[i + 1] : make_int2(-1, 0);
      dpairs->push_back(make_int4(k, a.x, b.x, (a.y << 16) | b.y));
    }
  }
}

namespace {
bool env_flag(const char* name) {
  const char* v = getenv(name);
  return v && v[0] && v[0] != '0';
}
}  // namespace

bool tc_supported(int z, int h, int x, int B) {
  return h == tc::HID && z % 16 == 0 && z >= 64 && z <= 256 && x % 16 == 0 && x >= 64 &&
         x <= 1024 && B >= 1;
}

TcPlan* tc_plan_create(const TcShape& s, const TcBuffers& b, std::string* msg) {
  if (!tc_supported(s.z, s.h, s.x, s.B)) {
    if (msg) *msg = "shape not supported by the tensor-core forward";
    return nullptr;
  }
  if (!get_encoder(msg)) return nullptr;
  TcPlan* p = new TcPlan();
  memset(p, 0, sizeof *p);
  p->s = s;
  const uint64_t C = s.cells, B = s.B, z = s.z, x = s.x, h = s.h, NI = s.n_indiv;
  bool ok = make_map(&p->mZ, b.Z, z, B, C, z * 2, B * z * 2, 128, msg) &&
            make_map(&p->mE, b.E, x, 6 * B, C, x * 2, (uint64_t)b.e_cell * 2, 128, msg) &&
            make_map(&p->mEB, b.E, x, 6 * B, C, x * 2, (uint64_t)b.e_cell * 2, 256, msg) &&
            make_map4(&p->mE4, b.E, x, B, 6, C, x * 2, B * x * 2, (uint64_t)b.e_cell * 2, msg) &&
            make_map(&p->mG1, b.Gwb + b.goff[0], z, h, NI, z * 2, b.PGs * 2, 256, msg) &&
            make_map(&p->mG2, b.Gwb + b.goff[2], h, h, NI, h * 2, b.PGs * 2, 256, msg) &&
            make_map(&p->mG3, b.Gwb + b.goff[4], h, x, NI, h * 2, b.PGs * 2, tc::N3, msg) &&
            make_map(&p->mD1, b.Dwb + b.doff[0], x, h, NI, x * 2, b.PDs * 2, 256, msg) &&
            make_map(&p->mD2, b.Dwb + b.doff[2], h, h, NI, h * 2, b.PDs * 2, 256, msg) &&
            make_map(&p->mG1h, b.Gwb + b.goff[0], z, h, NI, z * 2, b.PGs * 2, 128, msg) &&
            make_map(&p->mG2h, b.Gwb + b.goff[2], h, h, NI, h * 2, b.PGs * 2, 128, msg) &&
            make_map(&p->mG3h, b.Gwb + b.goff[4], h, x, NI, h * 2, b.PGs * 2, 128, msg) &&
            make_map(&p->mD1h, b.Dwb + b.doff[0], x, h, NI, x * 2, b.PDs * 2, 128, msg) &&
            make_map(&p->mD2h, b.Dwb + b.doff[2], h, h, NI, h * 2, b.PDs * 2, 128, msg);
  if (!ok) {
    delete p;
    return nullptr;
  }
  if (cudaMalloc(&p->err, sizeof(int)) != cudaSuccess ||
      cudaMemset(p->err, 0, sizeof(int)) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cudaMalloc for the error flag failed";
    delete p;
    return nullptr;
  }
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (cudaFuncSetAttribute(tc::k_mlp_fwd<tc::KIND_G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           tc::SMEM_BYTES) != cudaSuccess ||
      cudaFuncSetAttribute(tc::k_mlp_fwd<tc::KIND_D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           tc::SMEM_BYTES) != cudaSuccess ||
      cudaFuncSetAttribute(tc::k_mlp_fwd<tc::KIND_GRAM>,
                           cudaFuncAttributeMaxDynamicSharedMemorySize,
                           tc::SMEM_BYTES) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cannot reserve shared memory for the tensor-core forward";
    cudaFree(p->err);
    delete p;
    return nullptr;
  }
  auto tiles = [](int rows) { return (rows + tc::BM - 1) / tc::BM; };
  tc::KParams g{};
  g.kind = tc::KIND_G;
  g.cells = s.cells;
  g.B = s.B;
  g.z = s.z;
  g.x = s.x;
  g.rows = s.B;
  g.mtiles = tiles(s.B);
  g.n_tiles = s.cells * 5 * g.mtiles;
  g.kc1 = (s.z + tc::BK - 1) / tc::BK;
  g.n3 = (s.x + tc::N3 - 1) / tc::N3;
  g.nbr = b.nbr;
  g.wmaster = b.Gw;
  g.wb = b.Gwb;
  g.pstride = b.PGs;
  g.off_b1 = b.goff[1];
  g.off_b2 = b.goff[3];
  g.off_b3 = b.goff[5];
  g.off_w3 = b.goff[4];
  g.E = (bf16*)b.E;
  g.e_cell = b.e_cell;
  g.logits = b.logits;
  g.slope = s.slope;
  g.err = p->err;
  tc::KParams gc = g;  // every cell's own generator only (later minibatch steps)
  gc.centre = 1;
  gc.indiv_off = b.indiv_off;
  gc.n_tiles = s.cells * g.mtiles;
  tc::KParams d = g;
  d.kind = tc::KIND_D;
  d.rows = 6 * s.B;
  d.mtiles = tiles(6 * s.B);
  d.n_tiles = s.cells * 5 * d.mtiles;
  d.kc1 = (s.x + tc::BK - 1) / tc::BK;
  d.n3 = 0;
  d.wmaster = b.Dw;
  d.wb = b.Dwb;
  d.pstride = b.PDs;
  d.off_b1 = b.doff[1];
  d.off_b2 = b.doff[3];
  d.off_b3 = b.doff[5];
  d.off_w3 = b.doff[4];
  tc::KParams gt = g;  // selected generator of each cell on its own z: both hidden layers
  gt.train = 1;
  gt.wsel = b.src_g;
  gt.n_tiles = s.cells * g.mtiles;
  gt.act1 = (bf16*)b.TH1;
  gt.act2 = (bf16*)b.TH2;
  tc::KParams dt = d;  // selected discriminator on [x_c; selected fakes], read from E
  dt.train = 1;
  dt.wsel = b.src_d;
  dt.part_slot = b.sel_g;
  dt.rows = s.B;
  dt.mtiles = tiles(s.B);
  dt.n_tiles = s.cells * 2 * dt.mtiles;
  dt.act1 = (bf16*)b.TG1;
  dt.act2 = (bf16*)b.TG2;
  dt.logits = b.TL;
  tc::KParams gm{};  // Gram matrix of every cell's evaluation rows (mixture score)
  gm.kind = tc::KIND_GRAM;
  gm.cells = s.cells;
  gm.B = s.B;
  gm.z = s.z;
  gm.x = s.x;
  gm.rows = 6 * s.B;
  gm.mtiles = tiles(6 * s.B);
  gm.n_tiles = s.cells * gm.mtiles;
  gm.kc1 = (s.x + tc::BK - 1) / tc::BK;
  gm.E = (bf16*)b.E;
  gm.e_cell = b.e_cell;
  gm.err = p->err;
  gm.rnorm = b.rnorm;
  gm.gram_out = b.gram_out;
  p->pg = g;
  p->pgc = gc;
  p->pgram = gm;
  p->pd = d;
  p->pgt = gt;
  p->pdt = dt;
  // the CTA-pair evaluation kernels (generator: z == 64, its one noise chunk gathered;
  // first rows of discriminator tiles packed in 16 bits); LIPZ_FWD_SINGLE=1 keeps the
  // one-CTA kernels (for comparisons)
  tc::PParams pp{};
  pp.B = s.B;
  pp.x = s.x;
  pp.n3 = g.n3;
  pp.Z = (const bf16*)b.Z;
  pp.E = (bf16*)b.E;
  pp.e_cell = b.e_cell;
  pp.logits = b.logits;
  pp.slope = s.slope;
  pp.err = p->err;
  tc::PParams ppg = pp, ppd = pp;
  ppg.rows = s.B;
  ppg.kc1 = g.kc1;
  ppg.wmaster = b.Gw;
  ppg.wb = b.Gwb;
  ppg.pstride = b.PGs;
  ppg.off_b1 = b.goff[1];
  ppg.off_b2 = b.goff[3];
  ppg.off_b3 = b.goff[5];
  ppg.off_w3 = b.goff[4];
  ppd.rows = 6 * s.B;
  ppd.kc1 = d.kc1;
  ppd.wmaster = b.Dw;
  ppd.wb = b.Dwb;
  ppd.pstride = b.PDs;
  ppd.off_b1 = b.doff[1];
  ppd.off_b2 = b.doff[3];
  ppd.off_b3 = b.doff[5];
  ppd.off_w3 = b.doff[4];
  p->ppg = ppg;
  p->ppd = ppd;
  tc::PParams ppdt = ppd;  // the training discriminators: both parts of a cell on one pair
  ppdt.train = 1;
  ppdt.mt = tiles(s.B);
  ppdt.n_pairs = s.cells * ppdt.mt;
  ppdt.rows = s.B;
  ppdt.wsel = b.src_d;
  ppdt.part_slot = b.sel_g;
  ppdt.act1 = (bf16*)b.TG1;
  ppdt.act2 = (bf16*)b.TG2;
  ppdt.logits = b.TL;
  p->ppdt = ppdt;
  const bool pairs_on = !env_flag("LIPZ_FWD_SINGLE");
  p->ncl_g = pairs_on && s.z == tc::BK
                 ? max_pair_clusters(tc::k_mlp_fwd_pair<tc::KIND_G>, tc::pair_threads<tc::KIND_G>(),
                                     tc::pair_smem_bytes<tc::KIND_G>())
                 : 0;
  p->ncl_d = pairs_on && 6 * s.B < 65536
                 ? max_pair_clusters(tc::k_mlp_fwd_pair<tc::KIND_D>, tc::pair_threads<tc::KIND_D>(),
                                     tc::pair_smem_bytes<tc::KIND_D>())
                 : 0;
  if (env_flag("LIPZ_VERBOSE"))
    fprintf(stderr, "lipz: tensor-core forward: %d SMs, CTA-pair clusters resident: generator %d, "
            "discriminator %d\n", sms, p->ncl_g, p->ncl_d);
  auto grid = [sms](int n) { return n < sms ? n : sms; };
  p->grid_g = grid(g.n_tiles);
  p->grid_gc = grid(gc.n_tiles);
  p->grid_gram = grid(gm.n_tiles);
  p->grid_d = grid(d.n_tiles);
  p->grid_gt = grid(gt.n_tiles);
  p->grid_dt = grid(dt.n_tiles);
  return p;
}

namespace {
int launch(int grid, const CUtensorMap& a, const CUtensorMap& b1, const CUtensorMap& b2,
           const CUtensorMap& b3, const tc::KParams& kp, cudaStream_t st, const char* what,
           std::string* msg) {
  auto k = kp.kind == tc::KIND_GRAM ? tc::k_mlp_fwd<tc::KIND_GRAM>
           : kp.kind == tc::KIND_D  ? tc::k_mlp_fwd<tc::KIND_D>
                                    : tc::k_mlp_fwd<tc::KIND_G>;
  launch_pdl(k, dim3(grid), dim3(tc::THREADS), tc::SMEM_BYTES, st, a, b1, b2, b3, kp);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    if (msg) *msg = std::string(what) + " launch: " + cudaGetErrorString(e);
    return 1;
  }
  return 0;
}
}  // namespace

namespace {
int launch_pair(int ncl, const CUtensorMap& a, const CUtensorMap& b1, const CUtensorMap& b2,
                const CUtensorMap& b3, const tc::PParams& pp, bool gen, cudaStream_t st,
                std::string* msg) {
  const int clusters = pp.n_pairs < ncl ? pp.n_pairs : ncl;
  if (clusters <= 0) return 0;
  cudaError_t e =
      gen ? launch_pairs(tc::k_mlp_fwd_pair<tc::KIND_G>, clusters, tc::pair_threads<tc::KIND_G>(),
                         (size_t)tc::pair_smem_bytes<tc::KIND_G>(), st, a, b1, b2, b3, pp)
          : launch_pairs(tc::k_mlp_fwd_pair<tc::KIND_D>, clusters, tc::pair_threads<tc::KIND_D>(),
                         (size_t)tc::pair_smem_bytes<tc::KIND_D>(), st, a, b1, b2, b3, pp);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) {
    cudaGetLastError();
    if (msg)
      *msg = std::string(gen ? "generator" : "discriminator") +
             " forward (CTA pairs) launch: " + cudaGetErrorString(e);
    return 1;
  }
  return 0;
}
}  // namespace

int tc_run_g(TcPlan* p, cudaStream_t st, std::string* msg) {
  if (p->ncl_g > 0 && p->ppg.pairs)
    return launch_pair(p->ncl_g, p->mZ, p->mG1h, p->mG2h, p->mG3h, p->ppg, true, st, msg);
  return launch(p->grid_g, p->mZ, p->mG1, p->mG2, p->mG3, p->pg, st, "generator forward", msg);
}

void tc_set_nbr(TcPlan* p, const int* nbr, const TcPairs* pairs) {
  p->pg.nbr = nbr;
  p->pd.nbr = nbr;
  p->ppg.pairs = pairs ? pairs->g : nullptr;
  p->ppg.n_pairs = pairs ? pairs->ng : 0;
  p->ppg.plist = pairs ? pairs->plist : nullptr;
  p->ppd.pairs = pairs ? pairs->d : nullptr;
  p->ppd.n_pairs = pairs ? pairs->nd : 0;
  p->ppd.plist = pairs ? pairs->plist : nullptr;
}

int tc_run_g_centre(TcPlan* p, cudaStream_t st, std::string* msg) {
  return launch(p->grid_gc, p->mZ, p->mG1, p->mG2, p->mG3, p->pgc, st, "centre generator forward",
                msg);
}

int tc_run_gram(TcPlan* p, cudaStream_t st, std::string* msg) {
  if (!p->pgram.rnorm || !p->pgram.gram_out || !tc_gram_supported(p->s.B)) {
    if (msg) *msg = "tensor-core Gram kernel: no buffers, or batch outside 32..250";
    return 1;
  }
  return launch(p->grid_gram, p->mE, p->mEB, p->mEB, p->mEB, p->pgram, st, "mixture Gram", msg);
}

int tc_gram_halves(int B) { return 2 * ((6 * B + tc::HID - 1) / tc::HID); }

// B >= 32: a 32-column group meets at most one block boundary; the norms and 32 zero entries
// past them fit one bias buffer
bool tc_gram_supported(int B) { return B >= 32 && 6 * B + 32 <= tc::BIAS_MAX; }

int tc_run_d(TcPlan* p, cudaStream_t st, std::string* msg) {
  if (p->ncl_d > 0 && p->ppd.pairs)
    return launch_pair(p->ncl_d, p->mE, p->mD1h, p->mD2h, p->mD2h, p->ppd, false, st, msg);
  return launch(p->grid_d, p->mE, p->mD1, p->mD2, p->mD2, p->pd, st, "discriminator forward",
                msg);
}

int tc_run_train_g(TcPlan* p, cudaStream_t st, std::string* msg) {
  return launch(p->grid_gt, p->mZ, p->mG1, p->mG2, p->mG3, p->pgt, st, "generator training forward",
                msg);
}

int tc_run_train_d(TcPlan* p, cudaStream_t st, std::string* msg) {
  if (p->ncl_d > 0)
    return launch_pair(p->ncl_d, p->mE, p->mD1h, p->mD2h, p->mD2h, p->ppdt, false, st, msg);
  return launch(p->grid_dt, p->mE4, p->mD1, p->mD2, p->mD2, p->pdt, st,
                "discriminator training forward", msg);
}

int* tc_error_flag(TcPlan* p) { return p ? p->err : nullptr; }

void tc_plan_destroy(TcPlan* p) {
  if (!p) return;
  if (p->err) cudaFree(p->err);
  delete p;
}

}  // namespace lipz
