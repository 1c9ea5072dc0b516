// Tensor-core backward of the training step (Section 3, step 3: the gradient update of every
// cell's selected generator and discriminator), bf16 operands and fp32 accumulation in TMEM.
//
// One grouped GEMM kernel serves every product of the backward: per cell, a 128 x BN output
// tile of C = A * B^T over K, where each operand is read by TMA either K-major (rows of K) or
// MN-major (rows of M or N, K in the outer dimension; used for the transposed products dW =
// delta^T X and delta W, so no transposed copy is ever written). Epilogues: fp32 store
// (weight gradients) or bf16 delta times the activation derivative read from the stored
// forward output. The z coordinate of a weight operand is the cell's selected individual.
// A weight-gradient tile can instead apply Adam on the spot (EPI_ADAM): the gradient never
// leaves the accumulator. A loader warp streams the selected individual's old weights and
// moments by TMA into shared memory, 32 columns at a time, while the epilogue turns the
// previous chunk into the cell's new weights, moments and bf16 copy.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <cstring>

#include "bwd_tc.h"
#include "common.cuh"
#include "tc_ptx.cuh"

namespace lipz {
namespace tcb {

using namespace lipz::tc;

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int A_BYTES = BM * BK * 2;        // 16 KB
constexpr int B_BYTES = 256 * BK * 2;       // 32 KB (BN <= 256)
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int MN_BOX_BYTES = 64 * BK * 2;   // one {64 MN, 64 K} box
constexpr int NUM_EPI_WARPS = 8;
constexpr int EPI_THREADS = 32 * NUM_EPI_WARPS;
// bias-gradient partial sums: [2 tiles][4 TMEM lane quarters][256 columns] fp32
constexpr int BIAS_PART_BYTES = 2 * 4 * 256 * 4;
// fused Adam: a chunk is 64 rows (one half of a tile) x 32 fp32 columns of each of w, m, v (one
// 128-byte row each, 128-byte swizzle), updated in place, plus the new bf16 copy (64-byte rows,
// no swizzle). Chunks alternate between the two row halves, so each half of the epilogue
// works through its own two of the four buffers. w, m and v lie a fixed distance apart in
// memory, so that one TMA box {32, 64, 1, 3} of a 4-D map moves the chunk's three arrays: a
// tiled TMA operation holds its issuing thread for about 0.2 us whatever its size up to 16 KB,
// so one box per array made the issuing thread, not the bytes, bound the stream.
constexpr int ADAM_COLS = 32;
constexpr int ADAM_ROWS = 64;
constexpr int ADAM_ARRAY_BYTES = ADAM_ROWS * ADAM_COLS * 4;            // 8 KB
constexpr int ADAM_WB_BYTES = ADAM_ROWS * ADAM_COLS * 2;               // 4 KB
constexpr int ADAM_BUF_BYTES = 3 * ADAM_ARRAY_BYTES + ADAM_WB_BYTES;   // 28 KB

// Without fused Adam: four operand stages. With it: two operand stages, four Adam chunk
// buffers and two more warps (the Adam stream's loader and storer). One CTA per SM either way.
template <bool FUSED>
struct Cfg {
  static constexpr int STAGES = FUSED ? 2 : 4;
  static constexpr int ADAM_BUFS = FUSED ? 4 : 0;
  static constexpr int THREADS = 64 + EPI_THREADS + (FUSED ? 64 : 0);
  static constexpr int SMEM =
      1024 + STAGES * STAGE_BYTES + ADAM_BUFS * ADAM_BUF_BYTES + 256 + BIAS_PART_BYTES;
};

enum { EPI_F32 = 0, EPI_DACT = 1, EPI_ADAM = 2 };

// Adam of one weight tensor fused into the tile that computes its gradient (Section 3, step 3:
// the selected individual of the cell takes one Adam step and becomes the cell's new centre).
// The old snapshot is read and the new one written through the stage's tensor maps.
struct AdamRef {
  const int* src;                  // individual each cell trains
  const float4* coef;              // per cell: lr, 1 / (1 - beta1^t), 1 / (1 - beta2^t), t
  float beta1, beta2, eps;
};

struct GParams {
  int cells;
  int M, N, K, BN;
  int mtiles, ntiles, kchunks;
  int a_mn, b_mn;       // operand layouts (1 = MN-major)
  int a_row0, b_row0;   // first row of a K-major operand
  const int* a_sel;     // z coordinate of A: a_sel[cell] (weights of the selected individual)
  const int* b_sel;     //   or the cell itself when null
  int epi, act;
  float slope;
  void* C;
  int64_t c_cell, scm, scn;  // C[cell * c_cell + m * scm + n * scn]
  const bf16* aux;
  int64_t aux_cell, sxm, sxn;
  int aux_wrap_at, aux_wrap_sub;  // aux row of m: m < wrap_at ? m : m - wrap_sub
  const int* aux_sel;             // non-null: aux also advances (1 + aux_sel[cell]) * aux_sel_stride
  int64_t aux_sel_stride;
  // split K (ksplit > 0): chunks [0, ksplit) read K rows kc * 64 of A and of B's slot 0;
  // chunks [ksplit, kchunks) read K rows (kc - ksplit) * 64 of A shifted by a_k_off1 and of B's
  // slot 1 + b_slot_sel[cell]; B is then a 4-D map {n, K rows, slots, cells}
  int ksplit, a_k_off1;
  const int* b_slot_sel;
  // EPI_DACT: column sums of the fp32 deltas over rows m < bias_rows go to
  // bias_out[cell * bias_cell + n] (a bias gradient); null = none
  float* bias_out;
  int64_t bias_cell;
  int bias_rows;
  AdamRef adam;
  int* err;
};

// OR of pred over the eight epilogue warps (named barrier 1, 256 threads); also orders their
// earlier global stores before their later loads.
__device__ __forceinline__ bool epi_any(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p, q;\n setp.ne.u32 p, %1, 0;\n bar.red.or.pred q, 1, 256, p;\n"
      " selp.u32 %0, 1, 0, q;\n}"
      : "=r"(r)
      : "r"((uint32_t)pred)
      : "memory");
  return r != 0;
}

__device__ __forceinline__ float dact(int act, float y, float slope) {
  switch (act) {
    case ACT_RELU: return y > 0.f ? 1.f : 0.f;
    case ACT_LRELU: return y > 0.f ? 1.f : slope;
    case ACT_TANH: return 1.f - y * y;
    default: return 1.f;
  }
}

// ---------------------------------------------------------------------------------------------
// The whole backward of one cell in one CTA: the nine products run as consecutive stages of a
// single tile stream (double-buffered TMEM, one TMA ring). A stage that reads an earlier
// stage's output waits until the epilogue has finished that stage's last tile: the epilogue
// threads fence their global stores into the async proxy, meet on an mbarrier, and one of
// them advances a tile counter in shared memory that the producer polls before loading.
// ---------------------------------------------------------------------------------------------
constexpr int MAX_STAGES = 9;

struct Stage {
  GParams p;
  int dep;      // stage whose output this one reads (-1: none)
  int tile0;    // tiles of the cell before this stage
  int publish;  // a later stage reads this one's output: its tiles are published and counted
};

struct CellPlan {
  Stage st[MAX_STAGES];
  int n_stages, tiles_per_cell, pub_per_cell, cells;
  int pub_end[MAX_STAGES];  // tiles of the cell published by the end of stage k
  int* err;
  // fused Adam: the biases' and D's output layer's step, applied by the epilogue warps to each
  // cell once its tiles are done (all of its gradients are then in gG / gD)
  int has_ranges;
  AdamRanges rg, rd;
  float beta1, beta2, eps;
};

struct StageMaps {
  CUtensorMap a[MAX_STAGES];
  CUtensorMap b[MAX_STAGES];
  CUtensorMap ao[MAX_STAGES];  // old w, m, v (EPI_ADAM stages): {in, out, individual, array}
  CUtensorMap an[MAX_STAGES];  // new w, m, v: {in, out, cell, array}
  CUtensorMap nb[MAX_STAGES];  // new bf16 copy
};

__device__ __forceinline__ void stage_tile(const GParams& p, int t, int& m0, int& n0, int& n) {
  m0 = (t / p.ntiles) * BM;
  n0 = (t % p.ntiles) * p.BN;
  n = min(p.BN, p.N - n0);
  n = p.b_mn ? (n + 63) & ~63 : (n + 15) & ~15;
}

// 16 accumulator columns of one row: fp32 store, or bf16 delta times the activation
// derivative (read from the stored forward output). `full` = all 16 columns lie inside N.
__device__ __forceinline__ void epi16(const GParams& p, const uint32_t (&r)[16], int cell, int m,
                                      int arow, int col0, bool full, float dlo, bool is_tanh,
                                      float (&vout)[16], const uint4* xpre = nullptr) {
  if (p.epi == EPI_F32) {
    float* C = reinterpret_cast<float*>(p.C) + (int64_t)cell * p.c_cell + (int64_t)m * p.scm;
    if (p.scn == 1) {
      if (full) {
        float4* o = reinterpret_cast<float4*>(C + col0);
#pragma unroll
        for (int u = 0; u < 4; ++u)
          o[u] = make_float4(__uint_as_float(r[4 * u]), __uint_as_float(r[4 * u + 1]),
                             __uint_as_float(r[4 * u + 2]), __uint_as_float(r[4 * u + 3]));
      } else {
        for (int e = 0; e < 16 && col0 + e < p.N; ++e) C[col0 + e] = __uint_as_float(r[e]);
      }
    } else {
      // transposed output: lanes hold consecutive rows, so each store is one coalesced line
      const int64_t sc = p.scn;
      float* o = C + (int64_t)col0 * sc;
      if (full) {
#pragma unroll
        for (int e = 0; e < 16; ++e) o[e * sc] = __uint_as_float(r[e]);
      } else {
        for (int e = 0; e < 16 && col0 + e < p.N; ++e) o[e * sc] = __uint_as_float(r[e]);
      }
    }
    return;
  }
  bf16* C = reinterpret_cast<bf16*>(p.C) + (int64_t)cell * p.c_cell + (int64_t)m * p.scm;
  const bf16* X = p.aux + (int64_t)cell * p.aux_cell + (int64_t)arow * p.sxm;
  if (p.aux_sel) X += (int64_t)(1 + __ldg(&p.aux_sel[cell])) * p.aux_sel_stride;
  if (p.sxn == 1 && p.scn == 1 && full) {
    // the caller may have loaded this group's forward output ahead (xpre)
    const uint4* x4 = xpre ? xpre : reinterpret_cast<const uint4*>(X + col0);
    const uint4 q0 = x4[0], q1 = x4[1];
    const uint32_t w[8] = {q0.x, q0.y, q0.z, q0.w, q1.x, q1.y, q1.z, q1.w};
    uint32_t pk[8];
#pragma unroll
    for (int e = 0; e < 16; e += 2) {
      const __nv_bfloat162 y2 = *reinterpret_cast<const __nv_bfloat162*>(&w[e >> 1]);
      const float y0 = __low2float(y2), y1 = __high2float(y2);
      const float d0 = is_tanh ? 1.f - y0 * y0 : (y0 > 0.f ? 1.f : dlo);
      const float d1 = is_tanh ? 1.f - y1 * y1 : (y1 > 0.f ? 1.f : dlo);
      vout[e] = __uint_as_float(r[e]) * d0;
      vout[e + 1] = __uint_as_float(r[e + 1]) * d1;
      __nv_bfloat162 b2 = __floats2bfloat162_rn(vout[e], vout[e + 1]);
      pk[e >> 1] = *reinterpret_cast<uint32_t*>(&b2);
    }
    // rows and column groups are 32-byte aligned here
    st_global_v8(C + col0, make_uint4(pk[0], pk[1], pk[2], pk[3]),
                 make_uint4(pk[4], pk[5], pk[6], pk[7]));
    return;
  }
  for (int e = 0; e < 16; ++e) {
    const int col = col0 + e;
    if (col >= p.N) break;
    const float y = __bfloat162float(X[(int64_t)col * p.sxn]);
    const float d = is_tanh ? 1.f - y * y : (y > 0.f ? 1.f : dlo);
    vout[e] = __uint_as_float(r[e]) * d;
    C[(int64_t)col * p.scn] = __float2bfloat16_rn(vout[e]);
  }
}

// Sum of v over the 32 lanes of a warp for 16 columns, reduce-scattered: lanes 2j and 2j + 1
// return the sum of column j. Each partial sum is formed by one lane, in a fixed order.
__device__ __forceinline__ float warp_colsum16(const float (&v)[16], int lane) {
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

// Epilogue of one tile: warp (q, hf) owns TMEM lane quarter q (rows 32q .. 32q + 31) and column
// half hf. With a bias output, the column sums of the tile's fp32 deltas over the counted rows
// go through warp_colsum16 and shared memory (one partial per lane quarter, double-buffered by
// bias tile) and are added in a fixed order into bias_out (stored by the first row tile).
__device__ __forceinline__ bool epilogue_tile(const GParams& p, int cell, int m0, int n0, int n,
                                              uint32_t tbase, int hf, int row, int q, int lane,
                                              float* bpart, int& btile, uint32_t bSum,
                                              volatile int* abort_flag, int* err) {
  const int m = m0 + row;
  const int ng = n / 16;
  const int half = (ng + 1) / 2;
  const int g0 = hf ? half : 0, g1 = hf ? ng : half;
  const bool row_ok = m < p.M;
  const int arow = m < p.aux_wrap_at ? m : m - p.aux_wrap_sub;
  const bool is_tanh = p.act == ACT_TANH;
  const float dlo = p.act == ACT_RELU ? 0.f : p.slope;
  const bool bias = p.epi == EPI_DACT && p.bias_out != nullptr;
  const bool brow = row_ok && m < p.bias_rows;
  float* bp = bpart + (btile & 1) * (4 * 256) + q * 256;
  int gi = g0;
  // EPI_DACT reads its row's stored forward output: the next pair of groups' values are loaded
  // while this pair is converted (one memory latency per tile instead of one per pair)
  const bool pre = p.epi == EPI_DACT && p.sxn == 1 && p.scn == 1 && row_ok;
  const bf16* X = nullptr;
  if (pre) {
    X = p.aux + (int64_t)cell * p.aux_cell + (int64_t)arow * p.sxm;
    if (p.aux_sel) X += (int64_t)(1 + __ldg(&p.aux_sel[cell])) * p.aux_sel_stride;
  }
  // (16 bf16 of a row per 256-bit load: the stored outputs' rows are 32-byte aligned)
  auto load_pair = [&](int g, uint4(&d)[4]) {
    const bf16* x = X + n0 + g * 16;
    if (n0 + g * 16 + 16 <= p.N) {
      const U8 v = ld_global_v8(x);
      d[0] = v.a;
      d[1] = v.b;
    }
    if (g + 1 < g1 && n0 + g * 16 + 32 <= p.N) {
      const U8 v = ld_global_v8(x + 16);
      d[2] = v.a;
      d[3] = v.b;
    }
  };
  uint4 xc[4], xn[4];
  if (pre && gi < g1) load_pair(gi, xc);
  // two 16-column groups per TMEM load where possible
  for (; gi + 1 < g1; gi += 2) {
    if (pre && gi + 2 < g1) load_pair(gi + 2, xn);
    uint32_t r[32];
    LIPZ_TMEM_LD32(tbase + gi * 16, r);
    tmem_wait_ld();
    const int col0 = n0 + gi * 16;
    const uint32_t(&ra)[16] = *reinterpret_cast<const uint32_t(*)[16]>(&r[0]);
    const uint32_t(&rb)[16] = *reinterpret_cast<const uint32_t(*)[16]>(&r[16]);
    float va[16], vb[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) va[e] = vb[e] = 0.f;
    if (row_ok) {
      epi16(p, ra, cell, m, arow, col0, col0 + 16 <= p.N, dlo, is_tanh, va, pre ? &xc[0] : nullptr);
      if (col0 + 16 < p.N)
        epi16(p, rb, cell, m, arow, col0 + 16, col0 + 32 <= p.N, dlo, is_tanh, vb,
              pre ? &xc[2] : nullptr);
    }
    if (pre) {
#pragma unroll
      for (int u = 0; u < 4; ++u) xc[u] = xn[u];
    }
    if (bias) {
      if (!brow) {
#pragma unroll
        for (int e = 0; e < 16; ++e) va[e] = vb[e] = 0.f;
      }
      const float s0 = warp_colsum16(va, lane), s1 = warp_colsum16(vb, lane);
      if (!(lane & 1)) {
        bp[gi * 16 + (lane >> 1)] = s0;
        bp[(gi + 1) * 16 + (lane >> 1)] = s1;
      }
    }
  }
  if (gi < g1) {
    uint32_t r[16];
    LIPZ_TMEM_LD16(tbase + gi * 16, r);
    tmem_wait_ld();
    const int col0 = n0 + gi * 16;
    float va[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) va[e] = 0.f;
    if (row_ok && col0 < p.N)
      epi16(p, r, cell, m, arow, col0, col0 + 16 <= p.N, dlo, is_tanh, va, pre ? &xc[0] : nullptr);
    if (bias) {
      if (!brow) {
#pragma unroll
        for (int e = 0; e < 16; ++e) va[e] = 0.f;
      }
      const float s0 = warp_colsum16(va, lane);
      if (!(lane & 1)) bp[gi * 16 + (lane >> 1)] = s0;
    }
  }
  if (bias) {
    // once every epilogue thread has written its partials (mbarrier bSum[btile & 1]), the
    // lane-quarter-0 warp of each column half adds the four quarters (fixed order) into the
    // running sum over row tiles. A buffer is rewritten two bias tiles later, which needs the
    // TMEM region that this tile's readers (those warps included) release after this.
    const uint32_t bar = bSum + 8 * (btile & 1);
    mbar_arrive(bar);
    if (q == 0) {
      if (!mbar_wait_warp(bar, (uint32_t)((btile >> 1) & 1), abort_flag, err, 20)) return false;
      const float* b0 = bpart + (btile & 1) * (4 * 256);
      for (int col = g0 * 16 + lane; col < g1 * 16; col += 32) {
        const int gc = n0 + col;
        if (gc < p.N) {
          const float t = ((b0[col] + b0[256 + col]) + b0[512 + col]) + b0[768 + col];
          float* o = p.bias_out + (int64_t)cell * p.bias_cell + gc;
          *o = m0 == 0 ? t : *o + t;
        }
      }
    }
    ++btile;
  }
  return true;
}

// Adam epilogue of one weight-gradient tile: for each 32-column chunk of the thread's row half
// h, the warp's 16 columns of its row. Chunk number cj of a half sits in buffer 2 (cj & 1) + h
// (its (cj >> 1)-th use) as three 64 x 128-byte boxes of old w, m, v in the 128-byte swizzle
// (16-byte unit u of box row r at unit u ^ (r & 7)); the new values go back to the same places,
// the bf16 copy to the buffer's 64-byte-row box, and the loader warp stores the four boxes once
// the half's 128 threads have arrived on aDone. Returns false on a timeout.
__device__ __forceinline__ bool adam_tile(const GParams& p, int cell, int m0, int n0,
                                          uint32_t tbase, int hf, int row, uint32_t sAdam,
                                          uint32_t aFull, uint32_t aDone, int& cj,
                                          volatile int* abort_flag, int* err) {
  const AdamRef& a = p.adam;
  const float4 cf = __ldg(&a.coef[cell]);
  const bool row_ok = m0 + row < p.M;
  const int h = row / ADAM_ROWS, rr = row % ADAM_ROWS;
  const int nch = (min(p.BN, p.N - n0) + ADAM_COLS - 1) / ADAM_COLS;
  for (int k = 0; k < nch; ++k, ++cj) {
    const int bi = 2 * (cj & 1) + h;
    if (!mbar_wait_warp(aFull + 8 * bi, (uint32_t)((cj >> 1) & 1), abort_flag, err, 18))
      return false;
    const int cl = k * ADAM_COLS + 16 * hf;  // first column of this thread, within the tile
    const uint32_t bb = sAdam + (uint32_t)(bi * ADAM_BUF_BYTES);
    const uint32_t rb = bb + (uint32_t)rr * 128u;
    // the TMEM load is warp-collective: every lane takes part, live row or not
    uint32_t r[16];
    LIPZ_TMEM_LD16(tbase + cl, r);
    tmem_wait_ld();
    if (row_ok && n0 + cl < p.N) {
      float w[16], mm[16], v[16];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t off = (uint32_t)(((4 * hf + u) ^ (rr & 7)) << 4);
        asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                     : "=f"(w[4 * u]), "=f"(w[4 * u + 1]), "=f"(w[4 * u + 2]), "=f"(w[4 * u + 3])
                     : "r"(rb + off)
                     : "memory");
        asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                     : "=f"(mm[4 * u]), "=f"(mm[4 * u + 1]), "=f"(mm[4 * u + 2]),
                       "=f"(mm[4 * u + 3])
                     : "r"(rb + ADAM_ARRAY_BYTES + off)
                     : "memory");
        asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                     : "=f"(v[4 * u]), "=f"(v[4 * u + 1]), "=f"(v[4 * u + 2]), "=f"(v[4 * u + 3])
                     : "r"(rb + 2 * ADAM_ARRAY_BYTES + off)
                     : "memory");
      }
#pragma unroll
      for (int e = 0; e < 16; ++e)
        adam_elem(w[e], mm[e], v[e], __uint_as_float(r[e]), a.beta1, a.beta2, cf.x, cf.y, cf.z,
                  a.eps);
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t off = (uint32_t)(((4 * hf + u) ^ (rr & 7)) << 4);
        asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(rb + off), "f"(w[4 * u]),
                     "f"(w[4 * u + 1]), "f"(w[4 * u + 2]), "f"(w[4 * u + 3])
                     : "memory");
        asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(rb + ADAM_ARRAY_BYTES + off),
                     "f"(mm[4 * u]), "f"(mm[4 * u + 1]), "f"(mm[4 * u + 2]), "f"(mm[4 * u + 3])
                     : "memory");
        asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(rb + 2 * ADAM_ARRAY_BYTES +
                                                                      off),
                     "f"(v[4 * u]), "f"(v[4 * u + 1]), "f"(v[4 * u + 2]), "f"(v[4 * u + 3])
                     : "memory");
      }
      const uint32_t wbr = bb + 3 * ADAM_ARRAY_BYTES + (uint32_t)rr * 64u + (uint32_t)hf * 32u;
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(wbr),
                   "r"(pack_bf16(w[0], w[1])), "r"(pack_bf16(w[2], w[3])),
                   "r"(pack_bf16(w[4], w[5])), "r"(pack_bf16(w[6], w[7]))
                   : "memory");
      asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(wbr + 16),
                   "r"(pack_bf16(w[8], w[9])), "r"(pack_bf16(w[10], w[11])),
                   "r"(pack_bf16(w[12], w[13])), "r"(pack_bf16(w[14], w[15]))
                   : "memory");
    }
    // make the new values visible to the TMA store, then hand the chunk to the loader warp
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    mbar_arrive(aDone + 8 * bi);
  }
  return true;
}

template <bool FUSED>
__global__ void __launch_bounds__(Cfg<FUSED>::THREADS, 1)
    k_bwd_cells(const __grid_constant__ StageMaps maps, const __grid_constant__ CellPlan cp) {
  constexpr int STAGES = Cfg<FUSED>::STAGES;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  uint8_t* gbase = smem_raw + (base - raw);
  const uint32_t sAdam = base + STAGES * STAGE_BYTES;  // [ADAM_BUFS][w | m | v] chunks
  uint8_t* misc = gbase + STAGES * STAGE_BYTES + Cfg<FUSED>::ADAM_BUFS * ADAM_BUF_BYTES;
  const uint32_t bFull = smem_u32(misc), bEmpty = bFull + 8 * STAGES;
  const uint32_t bAcc = bEmpty + 8 * STAGES, bReg = bAcc + 16, bFinal = bReg + 16;
  const uint32_t bEpi = bFinal + 8;    // [2], alternating by tile
  const uint32_t aFull = bEpi + 16;   // [4] Adam chunk buffers: old values landed
  const uint32_t aDone = aFull + 32;  // [4] new values written back by the epilogue half
  const uint32_t bSum = aDone + 32;   // [2] bias partial sums written, by bias tile
  const uint32_t aFree = bSum + 16;   // [4] the stores have read the buffer
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(misc + 224);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(misc + 228);
  volatile int* done_tiles = reinterpret_cast<volatile int*>(misc + 232);
  float* bpart = reinterpret_cast<float*>(misc + 256);  // bias partial sums

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bFull + 8 * s, 1);
      mbar_init(bEmpty + 8 * s, 1);
    }
    mbar_init(bAcc, 1);
    mbar_init(bAcc + 8, 1);
    mbar_init(bReg, EPI_THREADS);
    mbar_init(bReg + 8, EPI_THREADS);
    mbar_init(bFinal, 1);
    mbar_init(bEpi, EPI_THREADS);
    mbar_init(bEpi + 8, EPI_THREADS);
    for (int b = 0; b < Cfg<FUSED>::ADAM_BUFS; ++b) {
      mbar_init(aFull + 8 * b, 1);
      mbar_init(aDone + 8 * b, EPI_THREADS / 2);
      mbar_init(aFree + 8 * b, 1);
    }
    mbar_init(bSum, EPI_THREADS);
    mbar_init(bSum + 8, EPI_THREADS);
    *abort_flag = 0;
    *done_tiles = 0;
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
  int* err = cp.err;
  // the set-up above touched no global memory: from here on the previous kernel's results
  // are needed (programmatic dependent launch)
  pdl_wait();

  if (warp == 0) {
    if (lane == 0) {
      int issued[STAGES] = {};
      bool ok = true;
      int stage = 0;
      uint32_t phase = 0;
      int cells_done = 0;
      for (int cell = blockIdx.x; cell < cp.cells && ok; cell += gridDim.x, ++cells_done) {
        for (int si = 0; si < cp.n_stages && ok; ++si) {
          const GParams& p = cp.st[si].p;
          const int dep = cp.st[si].dep;
          if (dep >= 0) {
            // the stage reads the output of stage `dep` of this cell: wait for its last tile
            const int need = cells_done * cp.pub_per_cell + cp.pub_end[dep];
            const unsigned long long t0 = globaltimer();
            uint32_t it = 0;
            while (*done_tiles < need) {
              if ((++it & 255u) == 0) {
                if (*abort_flag) {
                  ok = false;
                  break;
                }
                if (globaltimer() - t0 > WAIT_NS) {
                  *abort_flag = 1;
                  atomicExch(err, 16);
                  ok = false;
                  break;
                }
              }
            }
            if (!ok) break;
            __threadfence_block();
          }
          const CUtensorMap* mA = &maps.a[si];
          const CUtensorMap* mB = &maps.b[si];
          const int za = p.a_sel ? __ldg(&p.a_sel[cell]) : cell;
          const int zb = p.b_sel ? __ldg(&p.b_sel[cell]) : cell;
          const uint32_t b_bytes =
              p.b_mn ? (uint32_t)((p.BN / 64) * MN_BOX_BYTES) : (uint32_t)(p.BN * 128);
          const int nt = p.mtiles * p.ntiles;
          for (int t = 0; t < nt && ok; ++t) {
            int m0, n0, n;
            stage_tile(p, t, m0, n0, n);
            for (int kc = 0; kc < p.kchunks; ++kc) {
              if (!mbar_wait(bEmpty + 8 * stage, phase ^ 1u, abort_flag, err, 11)) {
                ok = false;
                break;
              }
              const uint32_t full = bFull + 8 * stage;
              mbar_expect_tx(full, (uint32_t)A_BYTES + b_bytes);
              const uint32_t sA = base + stage * STAGE_BYTES, sB = sA + A_BYTES;
              const bool part1 = p.ksplit > 0 && kc >= p.ksplit;
              const int kk = part1 ? kc - p.ksplit : kc;
              const int ka = kk * BK + (part1 ? p.a_k_off1 : 0);
              if (p.a_mn) {
                tma_load_3d(sA, mA, full, m0, ka, za);
                tma_load_3d(sA + MN_BOX_BYTES, mA, full, m0 + 64, ka, za);
              } else {
                tma_load_3d(sA, mA, full, ka, p.a_row0 + m0, za);
              }
              if (p.ksplit > 0) {
                const int slot = part1 ? 1 + __ldg(&p.b_slot_sel[cell]) : 0;
                for (int i = 0; i < p.BN / 64; ++i)
                  tma_load_4d(sB + i * MN_BOX_BYTES, mB, full, n0 + 64 * i, kk * BK, slot, cell);
              } else if (p.b_mn) {
                for (int i = 0; i < p.BN / 64; ++i)
                  tma_load_3d(sB + i * MN_BOX_BYTES, mB, full, n0 + 64 * i, kc * BK, zb);
              } else {
                tma_load_3d(sB, mB, full, kc * BK, p.b_row0 + n0, zb);
              }
              issued[stage]++;
              if (++stage == STAGES) {
                stage = 0;
                phase ^= 1u;
              }
            }
          }
        }
      }
      if (!ok) {
        for (int s = 0; s < STAGES; ++s)
          if (issued[s] > 0) {
            volatile int never = 0;
            mbar_wait(bFull + 8 * s, (uint32_t)((issued[s] - 1) & 1), &never, err, 11);
          }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int lt = 0;
      for (int cell = blockIdx.x; cell < cp.cells && ok; cell += gridDim.x) {
        for (int si = 0; si < cp.n_stages && ok; ++si) {
          const GParams& p = cp.st[si].p;
          const int nt = p.mtiles * p.ntiles;
          for (int t = 0; t < nt && ok; ++t, ++lt) {
            int m0, n0, n;
            stage_tile(p, t, m0, n0, n);
            const int R = lt & 1, use = lt >> 1;
            if (use > 0 &&
                !mbar_wait(bReg + 8 * R, (uint32_t)((use - 1) & 1), abort_flag, err, 15)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t d = tmem + (uint32_t)(R * 256);
            const uint32_t idesc = idesc_bf16_major(BM, n, p.a_mn, p.b_mn);
            for (int kc = 0; kc < p.kchunks; ++kc) {
              if (!mbar_wait(bFull + 8 * stage, phase, abort_flag, err, 12)) {
                ok = false;
                break;
              }
              tc_fence_after();
              const uint32_t sA = base + stage * STAGE_BYTES, sB = sA + A_BYTES;
#pragma unroll
              for (int kk = 0; kk < BK / 16; ++kk) {
                const uint64_t ad = p.a_mn ? sw128_mn_desc(sA + kk * 2048, MN_BOX_BYTES)
                                           : sw128_desc(sA + kk * 32);
                const uint64_t bd = p.b_mn ? sw128_mn_desc(sB + kk * 2048, MN_BOX_BYTES)
                                           : sw128_desc(sB + kk * 32);
                tc_mma(d, ad, bd, idesc, (kc | kk) != 0 ? 1u : 0u);
              }
              tc_commit(bEmpty + 8 * stage);
              if (++stage == STAGES) {
                stage = 0;
                phase ^= 1u;
              }
            }
            if (!ok) break;
            tc_commit(bAcc + 8 * R);
          }
        }
      }
      tc_commit(bFinal);
      volatile int never = 0;
      mbar_wait(bFinal, 0u, &never, err, 14);
    }
  } else if (FUSED && warp >= 2 + NUM_EPI_WARPS) {
    // ===== Adam stream: the old w, m, v of every chunk of every EPI_ADAM tile, in tile order,
    // into the four buffers in turn, and the new w, m, v and bf16 copy back out. A tiled TMA
    // operation holds its issuing thread for about 0.2 us, so two warps share the work:
    //   loader: a chunk's load, once the storer has released the chunk's buffer;
    //   storer: a chunk's two stores once its epilogue half is done, then, when the stores
    //           have read the buffer, its release to the loader (releasing it one chunk later,
    //           to keep a store group in flight, was slower: the stream is bound by the
    //           latency of each buffer's round trip). =====
    const bool storer = warp == 3 + NUM_EPI_WARPS;
    if (lane == 0) {
      constexpr int NB = Cfg<FUSED>::ADAM_BUFS > 0 ? Cfg<FUSED>::ADAM_BUFS : 1;
      int buf = 0, uses[NB] = {};
      bool ok = true;
      for (int cell = blockIdx.x; cell < cp.cells && ok; cell += gridDim.x) {
        for (int si = 0; si < cp.n_stages && ok; ++si) {
          const GParams& p = cp.st[si].p;
          if (p.epi != EPI_ADAM) continue;
          const int zi = __ldg(&p.adam.src[cell]);
          const int nt = p.mtiles * p.ntiles;
          for (int t = 0; t < nt && ok; ++t) {
            const int m0 = (t / p.ntiles) * BM, n0 = (t % p.ntiles) * p.BN;
            const int nch = (min(p.BN, p.N - n0) + ADAM_COLS - 1) / ADAM_COLS;
            for (int k = 0; k < 2 * nch; ++k) {
              const int x0 = n0 + (k >> 1) * ADAM_COLS, y0 = m0 + (k & 1) * ADAM_ROWS;
              const uint32_t bb = sAdam + (uint32_t)(buf * ADAM_BUF_BYTES);
              if (storer) {
                // the (uses[buf] + 1)-th chunk of this buffer is written back
                if (!mbar_wait(aDone + 8 * buf, (uint32_t)(uses[buf] & 1), abort_flag, err, 19)) {
                  ok = false;
                  break;
                }
                tma_store_4d(&maps.an[si], bb, x0, y0, cell, 0);
                tma_store_3d(&maps.nb[si], bb + 3 * ADAM_ARRAY_BYTES, x0, y0, cell);
                bulk_commit();
                bulk_wait_read<0>();  // the stores have read the buffer: it may be refilled
                mbar_arrive(aFree + 8 * buf);
              } else {
                if (uses[buf] > 0 && !mbar_wait(aFree + 8 * buf, (uint32_t)((uses[buf] - 1) & 1),
                                                abort_flag, err, 21)) {
                  ok = false;
                  break;
                }
                const uint32_t full = aFull + 8 * buf;
                mbar_expect_tx(full, (uint32_t)(3 * ADAM_ARRAY_BYTES));
                tma_load_4d(bb, &maps.ao[si], full, x0, y0, zi, 0);
              }
              uses[buf]++;
              if (++buf == NB) buf = 0;
            }
          }
        }
      }
      if (storer) {
        bulk_wait_all();
      } else if (!ok) {
        // loads issued here land on this CTA's barriers: wait for them before it leaves
        for (int b = 0; b < NB; ++b)
          if (uses[b] > 0) {
            volatile int never = 0;
            mbar_wait(aFull + 8 * b, (uint32_t)((uses[b] - 1) & 1), &never, err, 19);
          }
      }
    }
  } else {
    const int ew = warp - 2, q = warp & 3, hf = ew >> 2;
    const int row = q * 32 + lane;
    bool ok = true;
    int lt = 0, pub = 0;
    int cj = 0;  // Adam chunks of this thread's row half so far
    int btile = 0;  // bias-summing tiles so far
    for (int cell = blockIdx.x; cell < cp.cells; cell += gridDim.x) {
      for (int si = 0; si < cp.n_stages && ok; ++si) {
        const GParams& p = cp.st[si].p;
        const bool publish = cp.st[si].publish != 0;
        const int nt = p.mtiles * p.ntiles;
        for (int t = 0; t < nt; ++t, ++lt) {
          int m0, n0, n;
          stage_tile(p, t, m0, n0, n);
          const int R = lt & 1, use = lt >> 1;
          if (!mbar_wait_warp(bAcc + 8 * R, (uint32_t)(use & 1), abort_flag, err, 13)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(R * 256);
          if constexpr (FUSED) {
            if (p.epi == EPI_ADAM) {
              if (!adam_tile(p, cell, m0, n0, tbase, hf, row, sAdam, aFull, aDone, cj,
                             abort_flag, err)) {
                ok = false;
                break;
              }
            } else if (!epilogue_tile(p, cell, m0, n0, n, tbase, hf, row, q, lane, bpart, btile,
                                      bSum, abort_flag, err)) {
              ok = false;
              break;
            }
          } else if (!epilogue_tile(p, cell, m0, n0, n, tbase, hf, row, q, lane, bpart, btile,
                                    bSum, abort_flag, err)) {
            ok = false;
            break;
          }
          if (publish) {
            // publish the tile's global stores to the async proxy (a later stage loads them by
            // TMA). The arrival on bEpi[pub & 1] comes before the arrival on bReg, so no thread
            // can reach the next-but-one published tile (same barrier) before every thread
            // has arrived here.
            asm volatile("fence.proxy.async;" ::: "memory");
            mbar_arrive(bEpi + 8 * (pub & 1));
          }
          tc_fence_before();
          mbar_arrive(bReg + 8 * R);
          if (publish) {
            if (warp == 2) {
              // one warp counts the tile once all epilogue threads have published their stores
              if (!mbar_wait_warp(bEpi + 8 * (pub & 1), (uint32_t)((pub >> 1) & 1), abort_flag,
                                  err, 17)) {
                ok = false;
                break;
              }
              if (lane == 0) {
                __threadfence_block();
                *done_tiles = pub + 1;
              }
              __syncwarp();
            }
            ++pub;
          }
        }
      }
      if (FUSED && cp.has_ranges) {
        // the cell's last tile is done by every epilogue thread (its bias sums are in gG / gD):
        // the remaining Adam ranges of the cell, the eight warps together (they leave
        // together when any of them gave up)
        if (epi_any(!ok)) {
          ok = false;
          break;
        }
        const int et = threadIdx.x - 64;
        for (int pp = 0; pp < 2; ++pp) {
          const AdamRanges& r = pp ? cp.rd : cp.rg;
          const int s = __ldg(&r.src[cell]);
          const float4 cf = __ldg(&r.coef[cell]);
          if (et == 0) {
            r.new_p.step[cell] = (int)cf.w;
            r.new_p.lr[cell] = cf.x;
          }
          const int64_t so = (int64_t)s * r.Ps, co = (int64_t)cell * r.Ps;
          for (int q = 0; q < r.n; ++q)
            for (int i = et; i < r.len[q]; i += EPI_THREADS) {
              const int64_t k = r.off[q] + i;
              float w = r.old_p.w[so + k], m = r.old_p.m[so + k], v = r.old_p.v[so + k];
              adam_elem(w, m, v, r.grad[co + k], cp.beta1, cp.beta2, cf.x, cf.y, cf.z, cp.eps);
              r.new_p.w[co + k] = w;
              r.new_p.m[co + k] = m;
              r.new_p.v[co + k] = v;
              if (r.new_p.wb) r.new_p.wb[co + k] = __float2bfloat16_rn(w);
            }
        }
      }
      if (!ok) break;
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

}  // namespace tcb

// ---- host side -----------------------------------------------------------------------------
namespace {

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;

bool encoder(std::string* msg) {
  if (g_enc) return true;
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                   cudaEnableDefault, &q);
  if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn) {
    cudaGetLastError();
    if (msg) *msg = "cuTensorMapEncodeTiled is unavailable";
    return false;
  }
  g_enc = (PFN_cuTensorMapEncodeTiled_v12000)fn;
  return true;
}

// bf16 3-D map {inner, rows, depth}; box {64, box_rows, 1}, 128-byte swizzle.
bool map3(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t depth,
          uint64_t depth_elems, uint32_t box_rows, std::string* msg) {
  cuuint64_t dims[3] = {inner, rows, depth};
  cuuint64_t strides[2] = {inner * 2, depth_elems * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                     box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled failed (" + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

// fp32 4-D map over one weight tensor [out][in] of w, m and v of every individual: {in, out,
// individuals, array}, the arrays `part` floats apart; box {32, 64, 1, 3} (the three arrays'
// 64 x 128-byte boxes one after another in shared memory), 128-byte swizzle.
bool map4f(CUtensorMap* m, const float* base, uint64_t inner, uint64_t rows, uint64_t depth,
           uint64_t depth_elems, uint64_t part, std::string* msg) {
  cuuint64_t dims[4] = {inner, rows, depth, 3};
  cuuint64_t strides[3] = {inner * 4, depth_elems * 4, part * 4};
  cuuint32_t box[4] = {(cuuint32_t)tcb::ADAM_COLS, (cuuint32_t)tcb::ADAM_ROWS, 1, 3};
  cuuint32_t es[4] = {1, 1, 1, 1};
  CUresult r = g_enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float*>(base), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled (fp32, 4-D) failed (" + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

// bf16 3-D map over one tensor's bf16 copy of every cell: {in, out, cells}, box {32, 64, 1},
// no swizzle (64-byte rows).
bool map3b_rows(CUtensorMap* m, const bf16* base, uint64_t inner, uint64_t rows, uint64_t depth,
                uint64_t depth_elems, std::string* msg) {
  cuuint64_t dims[3] = {inner, rows, depth};
  cuuint64_t strides[2] = {inner * 2, depth_elems * 2};
  cuuint32_t box[3] = {(cuuint32_t)tcb::ADAM_COLS, (cuuint32_t)tcb::ADAM_ROWS, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = g_enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<bf16*>(base), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled (bf16 rows) failed (" + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

// bf16 4-D map {inner, rows, slots, depth} (E seen as [cells][6][B][x]); box {64, 64, 1, 1},
// 128-byte swizzle: rows past `rows` within a slot read as zero.
bool map4(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t slots,
          uint64_t depth, uint64_t slot_elems, uint64_t depth_elems, std::string* msg) {
  cuuint64_t dims[4] = {inner, rows, slots, depth};
  cuuint64_t strides[3] = {inner * 2, slot_elems * 2, depth_elems * 2};
  cuuint32_t box[4] = {64, 64, 1, 1};
  cuuint32_t es[4] = {1, 1, 1, 1};
  CUresult r = g_enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims,
                     strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    if (msg) *msg = "cuTensorMapEncodeTiled (4-D) failed (" + std::to_string((int)r) + ")";
    return false;
  }
  return true;
}

struct Gemm {
  CUtensorMap a, b;
  CUtensorMap ao;      // old w, m, v of the tensor (fused Adam), by individual and array
  CUtensorMap an, nb;  // new w, m, v by cell and array; new bf16 copy by cell
  tcb::GParams p;
  int grid;
};

}  // namespace

struct TcbPlan {
  // order of execution: D1, dW2d, A3, dW1d, A2, dW3g, A1, dW2g, dW1g
  Gemm g[9];
  int n;
  int* err;
  tcb::StageMaps maps;  // the same nine products as one per-cell kernel
  tcb::CellPlan cells;
  int grid_cells;
  bool fused;  // weight tensors take their Adam step in the backward's epilogue
};

bool tcb_supported(int z, int h, int x, int B) {
  return h == 256 && z == 64 && x % 16 == 0 && x >= 64 && B >= 1 && B <= 256;
}

TcbPlan* tcb_plan_create(const TcbShape& s, const TcbBuffers& b, std::string* msg) {
  if (!tcb_supported(s.z, s.h, s.x, s.B)) {
    if (msg) *msg = "shape not supported by the tensor-core backward";
    return nullptr;
  }
  if (!encoder(msg)) return nullptr;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  TcbPlan* P = new TcbPlan();
  memset(P, 0, sizeof *P);
  if (cudaMalloc(&P->err, 4) != cudaSuccess || cudaMemset(P->err, 0, 4) != cudaSuccess) {
    cudaGetLastError();
    if (msg) *msg = "cudaMalloc for the error flag failed";
    delete P;
    return nullptr;
  }
  const int C = s.cells, B = s.B, h = s.h, x = s.x, z = s.z;
  const uint64_t NI = s.n_indiv;
  const bf16* Gw = b.Gwb;
  const bf16* Dw = b.Dwb;
  auto base_params = [&](int M, int N, int K, int BN) {
    tcb::GParams q;
    memset(&q, 0, sizeof q);
    q.M = M;
    q.N = N;
    q.K = K;
    q.BN = BN;
    q.mtiles = (M + 127) / 128;
    q.ntiles = (N + BN - 1) / BN;
    q.kchunks = (K + 63) / 64;
    q.slope = s.slope;
    q.aux_wrap_at = 1 << 30;
    q.err = P->err;
    q.cells = C;
    return q;
  };
  bool ok = true;
  int i = 0;
  auto finish = [&](Gemm& G) {
    const int tiles = C * G.p.mtiles * G.p.ntiles;
    G.grid = tiles < sms ? tiles : sms;
  };
  // weight-gradient stage of tensor `off` of a population: Adam in the epilogue when fused
  // weight-gradient stage of the tensor at `off` of a population, whose gradient tile is
  // [out = M][in = N] row-major (scm = N, scn = 1): Adam in the epilogue when fused
  auto fuse = [&](Gemm& G, const TcbBuffers::AdamPop& a, const int* src, int64_t off,
                  int64_t Ps) {
    if (!b.fuse_adam) return;
    if (G.p.scn != 1 || G.p.scm != G.p.N || G.p.N % 16 != 0 || off % 8 != 0 || Ps % 8 != 0) {
      if (msg) *msg = "fused Adam needs 16-column tensors at 8-element offsets";
      ok = false;
      return;
    }
    G.p.epi = tcb::EPI_ADAM;
    G.p.adam.src = src;
    G.p.adam.coef = a.coef;
    G.p.adam.beta1 = b.beta1;
    G.p.adam.beta2 = b.beta2;
    G.p.adam.eps = b.eps;
    // w, m, v are one allocation in three equal parts: the part size is the 4th dimension's
    // stride, the same for the old and the new snapshot
    const int64_t part = a.m - a.w;
    if (part <= 0 || a.v - a.m != part || a.m_new - a.w_new != part ||
        a.v_new - a.m_new != part) {
      if (msg) *msg = "fused Adam needs w, m, v at equal distances";
      ok = false;
      return;
    }
    ok = ok && map4f(&G.ao, a.w + off, G.p.N, G.p.M, NI, Ps, part, msg) &&
         map4f(&G.an, a.w_new + off, G.p.N, G.p.M, C, Ps, part, msg) &&
         map3b_rows(&G.nb, a.wb_new + off, G.p.N, G.p.M, C, Ps, msg);
  };

  // 1. D1 = (J2 @ W2d) * lrelu'(TG1 rows r or r - B): M = 3B rows, N = 256, K = 256
  {
    Gemm& G = P->g[i++];
    G.p = base_params(3 * B, h, h, 256);
    G.p.b_mn = 1;
    G.p.b_sel = b.src_d;
    G.p.epi = tcb::EPI_DACT;
    G.p.act = ACT_LRELU;
    G.p.C = b.D1;
    G.p.c_cell = (int64_t)3 * B * h;
    G.p.scm = h;
    G.p.scn = 1;
    G.p.aux = (const bf16*)b.TG1;
    G.p.aux_cell = (int64_t)2 * B * h;
    G.p.sxm = h;
    G.p.sxn = 1;
    G.p.aux_wrap_at = 2 * B;
    G.p.aux_wrap_sub = B;
    G.p.bias_out = b.gD + b.doff[1];  // D's b1: rows of the D loss
    G.p.bias_cell = b.PDs;
    G.p.bias_rows = 2 * B;
    ok = ok && map3(&G.a, b.J2, h, 3 * B, C, (uint64_t)3 * B * h, 128, msg) &&
         map3(&G.b, Dw + b.doff[2], h, h, NI, b.PDs, 64, msg);
    finish(G);
  }
  // 2. dW2d[o][i] = sum_{r < 2B} J2[r][o] TG1[r][i]: M = o, N = i, K = 2B (TG1 ends at 2B).
  //    An epilogue thread owns one output row o: 16 consecutive parameters per group.
  {
    Gemm& G = P->g[i++];
    G.p = base_params(h, h, 2 * B, 256);
    G.p.a_mn = 1;
    G.p.b_mn = 1;
    G.p.epi = tcb::EPI_F32;
    G.p.C = b.gD + b.doff[2];
    G.p.c_cell = b.PDs;
    G.p.scm = h;
    G.p.scn = 1;
    fuse(G, b.adam_d, b.src_d, b.doff[2], b.PDs);
    ok = ok && map3(&G.a, b.J2, h, 3 * B, C, (uint64_t)3 * B * h, 64, msg) &&
         map3(&G.b, b.TG1, h, 2 * B, C, (uint64_t)2 * B * h, 64, msg);
    finish(G);
  }
  // 3. A3 = (D1[2B + r] @ W1d) * (1 - F^2): M = B, N = x (tiles of 256), K = 256
  {
    Gemm& G = P->g[i++];
    G.p = base_params(B, x, h, 256);
    G.p.a_row0 = 2 * B;
    G.p.b_mn = 1;
    G.p.b_sel = b.src_d;
    G.p.epi = tcb::EPI_DACT;
    G.p.act = ACT_TANH;
    G.p.C = b.A3;
    G.p.c_cell = (int64_t)B * x;
    G.p.scm = x;
    G.p.scn = 1;
    G.p.aux = (const bf16*)b.E;  // the selected generator's fakes: E[c] slot 1 + sel_g[c]
    G.p.aux_cell = b.e_cell;
    G.p.aux_sel = b.sel_g;
    G.p.aux_sel_stride = (int64_t)B * x;
    G.p.bias_out = b.gG + b.goff[5];  // G's b3
    G.p.bias_cell = b.PGs;
    G.p.bias_rows = B;
    G.p.sxm = x;
    G.p.sxn = 1;
    ok = ok && map3(&G.a, b.D1, h, 3 * B, C, (uint64_t)3 * B * h, 128, msg) &&
         map3(&G.b, Dw + b.doff[0], x, h, NI, b.PDs, 64, msg);
    finish(G);
  }
  // 4. dW1d[o][i] = sum_{r < 2B} D1[r][o] X[r][i]: M = o = 256, N = i = x, K = 2B, where X =
  //    [E[c] rows 0..B-1 (real); E[c] fake rows of slot sel_g[c]] read in place: K splits into
  //    the two B-row parts (rows past B in a part read as zero), D1 rows shifted by B in the
  //    second part
  {
    Gemm& G = P->g[i++];
    G.p = base_params(h, x, 2 * B, 256);
    G.p.kchunks = 2 * ((B + 63) / 64);
    G.p.ksplit = (B + 63) / 64;
    G.p.a_k_off1 = B;
    G.p.b_slot_sel = b.sel_g;
    G.p.a_mn = 1;
    G.p.b_mn = 1;
    G.p.epi = tcb::EPI_F32;
    G.p.C = b.gD + b.doff[0];
    G.p.c_cell = b.PDs;
    G.p.scm = x;
    G.p.scn = 1;
    fuse(G, b.adam_d, b.src_d, b.doff[0], b.PDs);
    ok = ok && map3(&G.a, b.D1, h, 3 * B, C, (uint64_t)3 * B * h, 64, msg) &&
         map4(&G.b, b.E, x, B, 6, C, (uint64_t)B * x, (uint64_t)b.e_cell, msg);
    finish(G);
  }
  // 5. A2 = (A3 @ W3g) * relu'(TH2): M = B, N = 256, K = x
  {
    Gemm& G = P->g[i++];
    G.p = base_params(B, h, x, 256);
    G.p.b_mn = 1;
    G.p.b_sel = b.src_g;
    G.p.epi = tcb::EPI_DACT;
    G.p.act = ACT_RELU;
    G.p.C = b.A2;
    G.p.c_cell = (int64_t)B * h;
    G.p.scm = h;
    G.p.scn = 1;
    G.p.aux = (const bf16*)b.TH2;
    G.p.aux_cell = (int64_t)B * h;
    G.p.bias_out = b.gG + b.goff[3];  // G's b2
    G.p.bias_cell = b.PGs;
    G.p.bias_rows = B;
    G.p.sxm = h;
    G.p.sxn = 1;
    ok = ok && map3(&G.a, b.A3, x, B, C, (uint64_t)B * x, 128, msg) &&
         map3(&G.b, Gw + b.goff[4], h, x, NI, b.PGs, 64, msg);
    finish(G);
  }
  // 6. dW3g[o][i] = sum_r A3[r][o] TH2[r][i]: M = o = x, N = i = 256, K = B
  {
    Gemm& G = P->g[i++];
    G.p = base_params(x, h, B, 256);
    G.p.a_mn = 1;
    G.p.b_mn = 1;
    G.p.epi = tcb::EPI_F32;
    G.p.C = b.gG + b.goff[4];
    G.p.c_cell = b.PGs;
    G.p.scm = h;
    G.p.scn = 1;
    fuse(G, b.adam_g, b.src_g, b.goff[4], b.PGs);
    ok = ok && map3(&G.a, b.A3, x, B, C, (uint64_t)B * x, 64, msg) &&
         map3(&G.b, b.TH2, h, B, C, (uint64_t)B * h, 64, msg);
    finish(G);
  }
  // 7. A1 = (A2 @ W2g) * relu'(TH1): M = B, N = 256, K = 256
  {
    Gemm& G = P->g[i++];
    G.p = base_params(B, h, h, 256);
    G.p.b_mn = 1;
    G.p.b_sel = b.src_g;
    G.p.epi = tcb::EPI_DACT;
    G.p.act = ACT_RELU;
    G.p.C = b.A1;
    G.p.c_cell = (int64_t)B * h;
    G.p.scm = h;
    G.p.scn = 1;
    G.p.aux = (const bf16*)b.TH1;
    G.p.aux_cell = (int64_t)B * h;
    G.p.bias_out = b.gG + b.goff[1];  // G's b1
    G.p.bias_cell = b.PGs;
    G.p.bias_rows = B;
    G.p.sxm = h;
    G.p.sxn = 1;
    ok = ok && map3(&G.a, b.A2, h, B, C, (uint64_t)B * h, 128, msg) &&
         map3(&G.b, Gw + b.goff[2], h, h, NI, b.PGs, 64, msg);
    finish(G);
  }
  // 8. dW2g[o][i] = sum_r A2[r][o] TH1[r][i]: M = o = 256, N = i = 256, K = B
  {
    Gemm& G = P->g[i++];
    G.p = base_params(h, h, B, 256);
    G.p.a_mn = 1;
    G.p.b_mn = 1;
    G.p.epi = tcb::EPI_F32;
    G.p.C = b.gG + b.goff[2];
    G.p.c_cell = b.PGs;
    G.p.scm = h;
    G.p.scn = 1;
    fuse(G, b.adam_g, b.src_g, b.goff[2], b.PGs);
    ok = ok && map3(&G.a, b.A2, h, B, C, (uint64_t)B * h, 64, msg) &&
         map3(&G.b, b.TH1, h, B, C, (uint64_t)B * h, 64, msg);
    finish(G);
  }
  // 9. dW1g[o][i] = sum_r A1[r][o] Z[r][i]: M = 256 (o), N = z (i), K = B
  {
    Gemm& G = P->g[i++];
    G.p = base_params(h, z, B, z);
    G.p.a_mn = 1;
    G.p.b_mn = 1;
    G.p.epi = tcb::EPI_F32;
    G.p.C = b.gG + b.goff[0];
    G.p.c_cell = b.PGs;
    G.p.scm = z;
    G.p.scn = 1;
    fuse(G, b.adam_g, b.src_g, b.goff[0], b.PGs);
    ok = ok && map3(&G.a, b.A1, h, B, C, (uint64_t)B * h, 64, msg) &&
         map3(&G.b, b.Z, z, B, C, (uint64_t)B * z, 64, msg);
    finish(G);
  }
  P->n = i;
  if (ok) {
    // per-cell megakernel: stage order as above; each stage's dependency on an earlier output
    const int deps[9] = {-1, -1, 0, 0, 2, 2, 4, 4, 6};
    int tile0 = 0, pub = 0;
    for (int k = 0; k < i; ++k) {
      int publish = 0;
      for (int j = k + 1; j < i; ++j) publish |= deps[j] == k;
      const int nt = P->g[k].p.mtiles * P->g[k].p.ntiles;
      P->maps.a[k] = P->g[k].a;
      P->maps.b[k] = P->g[k].b;
      P->maps.ao[k] = P->g[k].ao;
      P->maps.an[k] = P->g[k].an;
      P->maps.nb[k] = P->g[k].nb;
      P->cells.st[k].p = P->g[k].p;
      P->cells.st[k].dep = deps[k];
      P->cells.st[k].tile0 = tile0;
      P->cells.st[k].publish = publish;
      tile0 += nt;
      if (publish) pub += nt;
      P->cells.pub_end[k] = pub;
    }
    P->cells.n_stages = i;
    P->cells.tiles_per_cell = tile0;
    P->cells.pub_per_cell = pub;
    P->cells.cells = C;
    P->cells.err = P->err;
    P->grid_cells = C < sms ? C : sms;
    P->fused = b.fuse_adam != 0;
    P->cells.has_ranges = P->fused && b.ranges ? 1 : 0;
    if (P->cells.has_ranges) {
      P->cells.rg = b.ranges[0];
      P->cells.rd = b.ranges[1];
      P->cells.beta1 = b.beta1;
      P->cells.beta2 = b.beta2;
      P->cells.eps = b.eps;
    }
    const cudaError_t e =
        P->fused ? cudaFuncSetAttribute(tcb::k_bwd_cells<true>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        tcb::Cfg<true>::SMEM)
                 : cudaFuncSetAttribute(tcb::k_bwd_cells<false>,
                                        cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        tcb::Cfg<false>::SMEM);
    if (e != cudaSuccess) {
      cudaGetLastError();
      if (msg) *msg = "cannot reserve shared memory for the per-cell backward";
      ok = false;
    }
  }
  if (!ok) {
    cudaFree(P->err);
    delete P;
    return nullptr;
  }
  return P;
}

int tcb_run_cells(TcbPlan* P, cudaStream_t st, std::string* msg) {
  if (P->fused)
    launch_pdl(tcb::k_bwd_cells<true>, dim3(P->grid_cells), dim3(tcb::Cfg<true>::THREADS),
               tcb::Cfg<true>::SMEM, st, P->maps, P->cells);
  else
    launch_pdl(tcb::k_bwd_cells<false>, dim3(P->grid_cells), dim3(tcb::Cfg<false>::THREADS),
               tcb::Cfg<false>::SMEM, st, P->maps, P->cells);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    if (msg) *msg = std::string("per-cell backward launch: ") + cudaGetErrorString(e);
    return 1;
  }
  return 0;
}

int* tcb_error_flag(TcbPlan* P) { return P ? P->err : nullptr; }

void tcb_plan_destroy(TcbPlan* P) {
  if (!P) return;
  if (P->err) cudaFree(P->err);
  delete P;
}

}  // namespace lipz
