// CUDA-core kernels of the grid iteration: initialisation, minibatch draw, grouped GEMM for
// every layer and its transposes, the discriminator's last layer, BCE fitness, tournament
// selection, the logit-delta epilogue, column sums and the fused Adam/replacement update.
#include "common.cuh"
#include "engine.h"

namespace lipz {

// ------------------------------------------------------------------------------------------
// Step 1: random weights. Element k of the flat vector takes word k of the
// (stream, 0, individual) sequence: Xavier-uniform tensors s = word >> 8,
// q = (2 s + 1 - 2^24) 2^-24, w = a q; normal tensors take normal k (Box-Muller on the two
// words of block k / 4 that pair with it), w = a n or 1 + a n.
// ------------------------------------------------------------------------------------------
__global__ void k_init_params(float* __restrict__ w, bf16* __restrict__ wb, int64_t P,
                              int64_t Ps, Layout lay, uint64_t seed, uint32_t stream) {
  const int cell = blockIdx.y;
  const int64_t k0 = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 4;
  if (k0 >= Ps) return;
  const U4 r = philox_block(seed, stream, 0u, (uint32_t)cell, (uint32_t)(k0 >> 2));
  const uint32_t words[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const int64_t k = k0 + e;
    if (k >= Ps) break;
    float v = 0.f;
    if (k < P) {
      int t = 0;
      while (t + 1 < lay.n && k >= lay.off[t + 1]) ++t;
      const float a = lay.bound[t];
      if (lay.init[t] == INIT_UNIFORM) {
        if (a != 0.f) {
          const float q =
              (float)(2 * (int32_t)(words[e] >> 8) + 1 - (1 << 24)) * 5.9604644775390625e-8f;
          v = a * q;
        }
      } else {
        const float2 nn = e < 2 ? box_muller(r.x, r.y) : box_muller(r.z, r.w);
        const float n = (e & 1) ? nn.y : nn.x;
        v = lay.init[t] == INIT_NORMAL ? a * n : 1.f + a * n;
      }
    }
    w[(int64_t)cell * Ps + k] = v;
    if (wb) wb[(int64_t)cell * Ps + k] = __float2bfloat16_rn(v);
  }
}

void launch_init_params(float* w, bf16* wb, int64_t P, int64_t Ps, const Layout& lay, int cells,
                        uint64_t seed, uint32_t stream, cudaStream_t st) {
  dim3 grid((unsigned)((Ps / 4 + 255) / 256), cells);
  k_init_params<<<grid, 256, 0, st>>>(w, wb, P, Ps, lay, seed, stream);
}

__global__ void k_to_bf16(const float* __restrict__ w, bf16* __restrict__ wb, int64_t n) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += (int64_t)gridDim.x * blockDim.x)
    wb[i] = __float2bfloat16_rn(w[i]);
}

void launch_to_bf16(const float* w, bf16* wb, int64_t n, cudaStream_t st) {
  k_to_bf16<<<1216, 256, 0, st>>>(w, wb, n);
}

// ------------------------------------------------------------------------------------------
// Minibatch of cell c at iteration t, minibatch step k: row b = pool row mulhi(word_b, n_pool)
// of stream BATCH + 256 k (or row b of the caller's batch), z[b][d] = normal b*z_dim + d of
// stream NOISE + 256 k.
// Rows go to E[c][b] (the first B rows of the cell's evaluation input).
// ------------------------------------------------------------------------------------------
template <typename T>
__device__ __forceinline__ void store4(T* dst, float4 v);
template <>
__device__ __forceinline__ void store4<float>(float* dst, float4 v) {
  *reinterpret_cast<float4*>(dst) = v;
}
template <>
__device__ __forceinline__ void store4<bf16>(bf16* dst, float4 v) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
  uint2 pk;
  pk.x = *reinterpret_cast<uint32_t*>(&lo);
  pk.y = *reinterpret_cast<uint32_t*>(&hi);
  *reinterpret_cast<uint2*>(dst) = pk;
}

// Four minibatch rows per warp: one Philox block gives the four rows' pool indices, and the
// rows' 16-byte-vector copies are issued together (every load, then every store), so a warp
// waits for memory once; then each row's normals, one Philox block (four normals) per lane at
// a time. The pool is held in the population's precision, so a drawn row is a plain copy;
// rows given by the caller (xin, fp32) are rounded here.
constexpr int DRAW_RPW = 4;

template <typename T>
__global__ void k_draw_batch(const T* __restrict__ pool, int64_t n_pool,
                             const float* __restrict__ xin, T* __restrict__ E, int64_t e_cell,
                             T* __restrict__ Z, int B, int x_dim, int z_dim, uint64_t seed,
                             uint32_t t, uint32_t step, int parts) {
  pdl_wait();
  const uint32_t s_batch = 3u + (step << 8), s_noise = 4u + (step << 8);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = blockIdx.x * (blockDim.x >> 5) + warp, c = blockIdx.y;
  const int b0 = q * DRAW_RPW;
  if (b0 >= B) return;
  const int nb = min(DRAW_RPW, B - b0);
  T* const dst0 = E + (int64_t)c * e_cell + (int64_t)b0 * x_dim;
  if (!(parts & DRAW_REAL)) {
  } else if (xin) {
    for (int i = 0; i < nb; ++i) {
      T* dst = dst0 + (int64_t)i * x_dim;
      const float* src = xin + ((int64_t)c * B + b0 + i) * x_dim;
      const bool vec = (x_dim & 3) == 0 && ((reinterpret_cast<uintptr_t>(src) & 15) == 0) &&
                       ((reinterpret_cast<uintptr_t>(dst) & (4 * sizeof(T) - 1)) == 0);
      if (vec && x_dim <= 1024) {
        // the row's (up to eight per lane) 16-byte loads issued before its stores
        float4 v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int k = lane * 4 + 128 * u;
          if (k < x_dim) v[u] = __ldg(reinterpret_cast<const float4*>(src + k));
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int k = lane * 4 + 128 * u;
          if (k < x_dim) store4<T>(dst + k, v[u]);
        }
      } else if (vec) {
        for (int k = lane * 4; k < x_dim; k += 128)
          store4<T>(dst + k, __ldg(reinterpret_cast<const float4*>(src + k)));
      } else {
        for (int k = lane; k < x_dim; k += 32) dst[k] = from_f<T>(src[k]);
      }
    }
  } else {
    // rows 4q .. 4q + 3 take the four words of Philox block q
    const U4 r = philox_block(seed, s_batch, t, (uint32_t)c, (uint32_t)q);
    const uint32_t wd[DRAW_RPW] = {r.x, r.y, r.z, r.w};
    const int bytes = x_dim * (int)sizeof(T);
    const int n4 = bytes >> 4;
    const bool vec = (bytes & 15) == 0 &&
                     ((reinterpret_cast<uintptr_t>(pool) | reinterpret_cast<uintptr_t>(E)) & 15) == 0 &&
                     ((e_cell * (int64_t)sizeof(T)) & 15) == 0;
    if (vec && n4 > 128) {
      // long rows (images): row by row, four vectors of a row in flight per lane
      for (int i = 0; i < nb; ++i) {
        const uint4* s4 = reinterpret_cast<const uint4*>(
            pool + (int64_t)mulhi_u32(wd[i], (uint32_t)n_pool) * x_dim);
        uint4* d4 = reinterpret_cast<uint4*>(dst0 + (int64_t)i * x_dim);
#pragma unroll 4
        for (int k = lane; k < n4; k += 32) d4[k] = __ldg(s4 + k);
      }
    } else if (vec) {
      uint4 v[DRAW_RPW][4];
#pragma unroll
      for (int i = 0; i < DRAW_RPW; ++i) {
        const uint4* s4 = reinterpret_cast<const uint4*>(
            pool + (int64_t)mulhi_u32(wd[i], (uint32_t)n_pool) * x_dim);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int k = lane + 32 * u;
          if (i < nb && k < n4) v[i][u] = __ldg(s4 + k);
        }
      }
#pragma unroll
      for (int i = 0; i < DRAW_RPW; ++i) {
        uint4* d4 = reinterpret_cast<uint4*>(dst0 + (int64_t)i * x_dim);
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int k = lane + 32 * u;
          if (i < nb && k < n4) d4[k] = v[i][u];
        }
      }
    } else {
      for (int i = 0; i < nb; ++i) {
        const T* src = pool + (int64_t)mulhi_u32(wd[i], (uint32_t)n_pool) * x_dim;
        T* dst = dst0 + (int64_t)i * x_dim;
        for (int k = lane; k < x_dim; k += 32) dst[k] = src[k];
      }
    }
  }
  if (!(parts & DRAW_NOISE)) return;
  for (int i = 0; i < nb; ++i) {
    const int b = b0 + i;
    T* zr = Z + ((int64_t)c * B + b) * z_dim;
    const uint32_t n0 = (uint32_t)b * (uint32_t)z_dim;
    // normals n0 .. n0 + z_dim - 1; Philox block i holds normals 4i .. 4i + 3
    if ((z_dim & 3) == 0 && ((reinterpret_cast<uintptr_t>(zr) & (4 * sizeof(T) - 1)) == 0)) {
      // every block lies inside the row and its four normals are one aligned vector
      for (int k = lane * 4; k < z_dim; k += 128) {
        const U4 rn = philox_block(seed, s_noise, t, (uint32_t)c, (n0 + (uint32_t)k) >> 2);
        const float2 g01 = box_muller(rn.x, rn.y), g23 = box_muller(rn.z, rn.w);
        store4<T>(zr + k, make_float4(g01.x, g01.y, g23.x, g23.y));
      }
      continue;
    }
    for (uint32_t blk = (n0 >> 2) + lane; blk * 4 < n0 + (uint32_t)z_dim; blk += 32) {
      const U4 rn = philox_block(seed, s_noise, t, (uint32_t)c, blk);
      const float2 g01 = box_muller(rn.x, rn.y), g23 = box_muller(rn.z, rn.w);
      const float vv[4] = {g01.x, g01.y, g23.x, g23.y};
#pragma unroll
      for (int qq = 0; qq < 4; ++qq) {
        const uint32_t n = blk * 4 + qq;
        if (n >= n0 && n < n0 + (uint32_t)z_dim) zr[n - n0] = from_f<T>(vv[qq]);
      }
    }
  }
}

template <typename T>
void launch_draw_batch(const T* pool, int64_t n_pool, const float* xin, T* E, int64_t e_cell,
                       T* Z, int cells, int B, int x_dim, int z_dim, uint64_t seed, uint32_t t,
                       uint32_t step, int parts, bool pdl, cudaStream_t st) {
  launch_kernel(pdl, k_draw_batch<T>, dim3((B + 8 * DRAW_RPW - 1) / (8 * DRAW_RPW), cells),
                dim3(256), 0, st, pool, n_pool,
                xin, E, e_cell, Z, B, x_dim, z_dim, seed, t, step, parts);
}
template void launch_draw_batch<float>(const float*, int64_t, const float*, float*, int64_t,
                                       float*, int, int, int, int, uint64_t, uint32_t, uint32_t,
                                       int, bool, cudaStream_t);
template void launch_draw_batch<bf16>(const bf16*, int64_t, const float*, bf16*, int64_t, bf16*,
                                      int, int, int, int, uint64_t, uint32_t, uint32_t, int, bool,
                                      cudaStream_t);

// ------------------------------------------------------------------------------------------
// Grouped GEMM on CUDA cores: 64x64 output tile per block, k-slices of 16 staged in shared
// memory as fp32, 4x4 outputs per thread, fp32 accumulation in k order.
// ------------------------------------------------------------------------------------------
template <typename TI, typename TO, int EPI>
__global__ void __launch_bounds__(256) k_gemm(const GemmDesc* __restrict__ descs, int act,
                                              float slope) {
  pdl_wait();
  const GemmDesc d = descs[blockIdx.z];
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  if (m0 >= d.M || n0 >= d.N) return;
  const TI* A = (const TI*)d.A;
  const TI* Bm = (const TI*)d.B;
  const float* bias = d.bias;
  if (d.wsel) {
    const int64_t off = (int64_t)d.wsel[d.cell] * d.wsel_stride;
    if (d.wsel_op == 1) A += off; else Bm += off;
    if (bias) bias += off;
  }
  __shared__ float As[16][64 + 4];
  __shared__ float Bs[16][64 + 4];
  const int tid = threadIdx.x;
  const int tm = (tid >> 4) * 4, tn = (tid & 15) * 4;
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
  const bool a_kfast = d.sak == 1, b_nfast = d.sbn == 1;
  for (int k0 = 0; k0 < d.K; k0 += 16) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int idx = tid + 256 * i;
      int m, k;
      if (a_kfast) { m = idx >> 4; k = idx & 15; } else { m = idx & 63; k = idx >> 6; }
      float v = 0.f;
      if (m0 + m < d.M && k0 + k < d.K)
        v = to_f<TI>(A[(int64_t)(m0 + m) * d.sam + (int64_t)(k0 + k) * d.sak]);
      As[k][m] = v;
      int n, kk;
      if (b_nfast) { n = idx & 63; kk = idx >> 6; } else { n = idx >> 4; kk = idx & 15; }
      float w = 0.f;
      if (n0 + n < d.N && k0 + kk < d.K)
        w = to_f<TI>(Bm[(int64_t)(k0 + kk) * d.sbk + (int64_t)(n0 + n) * d.sbn]);
      Bs[kk][n] = w;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < 16; ++k) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[k][tm + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[k][tn + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  TO* C = (TO*)d.C;
  const TI* aux = (const TI*)d.aux;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + tm + i;
    if (m >= d.M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tn + j;
      if (n >= d.N) continue;
      float v = acc[i][j];
      if (EPI == EPI_BIAS_ACT) {
        v = act_fwd(act, v + (bias ? bias[n] : 0.f), slope);
      } else if (EPI == EPI_DACT) {
        v *= act_bwd(act, to_f<TI>(aux[(int64_t)m * d.sxm + (int64_t)n * d.sxn]), slope);
      }
      C[(int64_t)m * d.scm + (int64_t)n * d.scn] = from_f<TO>(v);
    }
  }
}

template <typename TI, typename TO, int EPI>
void launch_gemm(const GemmDesc* descs, int n_problems, int max_m, int max_n, int act,
                 float slope, cudaStream_t st) {
  if (n_problems <= 0 || max_m <= 0 || max_n <= 0) return;
  dim3 grid((max_n + 63) / 64, (max_m + 63) / 64, n_problems);
  launch_pdl(k_gemm<TI, TO, EPI>, grid, dim3(256), 0, st, descs, act, slope);
}
#define LIPZ_INST_GEMM(TI, TO, EPI) \
  template void launch_gemm<TI, TO, EPI>(const GemmDesc*, int, int, int, int, float, cudaStream_t);
LIPZ_INST_GEMM(float, float, EPI_STORE)
LIPZ_INST_GEMM(float, float, EPI_BIAS_ACT)
LIPZ_INST_GEMM(float, float, EPI_DACT)
LIPZ_INST_GEMM(bf16, float, EPI_STORE)
LIPZ_INST_GEMM(bf16, bf16, EPI_BIAS_ACT)
LIPZ_INST_GEMM(bf16, bf16, EPI_DACT)

// ------------------------------------------------------------------------------------------
// Discriminator output layer: one warp per row, lanes stride over k, fixed shuffle tree.
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void k_gemv(const GemvDesc* __restrict__ descs) {
  pdl_wait();
  const GemvDesc d = descs[blockIdx.y];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= d.rows) return;
  const T* w = (const T*)d.w;
  const float* bias = d.bias;
  if (d.wsel) {
    const int64_t off = (int64_t)d.wsel[d.cell] * d.wsel_stride;
    w += off;
    bias += off;
  }
  const T* x = (const T*)d.X + (int64_t)r * d.ld;
  float s = 0.f;
  for (int k = lane; k < d.K; k += 32) s = fmaf(to_f<T>(x[k]), to_f<T>(w[k]), s);
#pragma unroll
  for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) d.out[r] = s + bias[0];
}

template <typename T>
void launch_gemv(const GemvDesc* descs, int n_problems, int max_rows, cudaStream_t st) {
  if (n_problems <= 0 || max_rows <= 0) return;
  launch_pdl(k_gemv<T>, dim3((max_rows + 7) / 8, n_problems), dim3(256), 0, st, descs);
}
template void launch_gemv<float>(const GemvDesc*, int, int, cudaStream_t);
template void launch_gemv<bf16>(const GemvDesc*, int, int, cudaStream_t);

// ------------------------------------------------------------------------------------------
// Column sums (bias gradients). A block takes 64 columns of one problem: 32 lanes own two
// adjacent columns each, 8 row groups stride over the rows, and the 8 partial sums are added
// in a fixed order (deterministic).
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(256) k_colsum(const ColSumDesc* __restrict__ descs) {
  pdl_wait();
  // A block takes 256 columns of one problem: lane l owns columns 8l .. 8l + 7, warp w the
  // rows w, w + 8, ...; the 8 partial sums of a column are added in a fixed order.
  const ColSumDesc d = descs[blockIdx.y];
  const int lane = threadIdx.x & 31, rg = threadIdx.x >> 5;
  const int n0 = blockIdx.x * 256 + lane * 8;
  __shared__ float part[8][256];
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (n0 < d.cols) {
    const T* x = (const T*)d.X;
    const bool vec = sizeof(T) == 2 && n0 + 8 <= d.cols && (d.ld & 7) == 0 &&
                     ((reinterpret_cast<uintptr_t>(x) & 15) == 0);
    for (int r = rg; r < d.rows; r += 8) {
      const T* p = x + (int64_t)r * d.ld + n0;
      if (vec) {
        const uint4 q = __ldg(reinterpret_cast<const uint4*>(p));
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162*>(&w[e]);
          acc[2 * e] += __low2float(v);
          acc[2 * e + 1] += __high2float(v);
        }
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (n0 + e < d.cols) acc[e] += to_f<T>(p[e]);
      }
    }
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) part[rg][lane * 8 + e] = acc[e];
  __syncthreads();
  const int col = blockIdx.x * 256 + threadIdx.x;
  if (col < d.cols) {
    float t = 0.f;
#pragma unroll
    for (int g = 0; g < 8; ++g) t += part[g][threadIdx.x];
    d.out[col] = t;
  }
}

template <typename T>
void launch_colsum(const ColSumDesc* descs, int n_problems, int max_cols, cudaStream_t st) {
  if (n_problems <= 0 || max_cols <= 0) return;
  launch_pdl(k_colsum<T>, dim3((max_cols + 255) / 256, n_problems), dim3(256), 0, st, descs);
}
template void launch_colsum<float>(const ColSumDesc*, int, int, cudaStream_t);
template void launch_colsum<bf16>(const ColSumDesc*, int, int, cudaStream_t);

// ------------------------------------------------------------------------------------------
// Pair losses and fitness of every cell (one block per cell). logits[c][j][6B]: rows [0, B)
// real, rows [B (1 + i), B (2 + i)) fakes of generator slot i.
//   L_D[c][i][j] = mean softplus(-real_j) + mean softplus(fake_ij)
//   L_G[c][i][j] = mean softplus(-fake_ij)
//   f_G[c][i] = mean_j L_G,  f_D[c][j] = mean_i L_D
// Each mean is one warp's fixed-order reduction: the result does not depend on scheduling.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ float softplusf(float x) { return fmaxf(x, 0.f) + log1pf(expf(-fabsf(x))); }

// ------------------------------------------------------------------------------------------
// Tournament selection, replacement and learning-rate mutation: one thread per cell.
// ------------------------------------------------------------------------------------------
__device__ int tournament_slot(const float* f5, const uint32_t* w, int size) {
  int remaining[5] = {0, 1, 2, 3, 4};
  int left = 5, best = -1;
  for (int m = 0; m < size; ++m) {
    const int r = (int)mulhi_u32(w[m], (uint32_t)(5 - m));
    const int e = remaining[r];
    for (int q = r; q + 1 < left; ++q) remaining[q] = remaining[q + 1];
    --left;
    if (best < 0 || f5[e] < f5[best] || (f5[e] == f5[best] && e < best)) best = e;
  }
  return best;
}

__device__ float mutate(float lr, uint64_t seed, uint32_t stream, uint32_t t, uint32_t c,
                        float std, uint64_t thr) {
  const U4 r = philox_block(seed, stream, t, c, 0u);
  if ((uint64_t)r.x >= thr) return lr;
  const float n = box_muller(r.y, r.z).x;
  return fmaxf(lr + std * n, 1e-8f);
}

// Records the choice of population `pop` (0 G, 1 D) for cell c: slot s, source individual src,
// the new lr and the Adam coefficients (lr, 1 / (1 - beta1^t), 1 / (1 - beta2^t), t) of the
// source's next step t.
__device__ void write_choice(int c, int pop, int s, int src, float lr, const SelectParams& p,
                             const SelectIO& io) {
  const int step1 = io.step_old[pop][src] + 1;
  // 1 - beta^t = -expm1(t * log1p(-(1 - beta))): 1 - beta is exact in fp32 for beta in
  // [0.5, 1), and the expm1 form keeps full relative precision for beta^t near 1
  const float bc1 = -expm1f((float)step1 * log1pf(-(1.f - p.beta1)));
  const float bc2 = -expm1f((float)step1 * log1pf(-(1.f - p.beta2)));
  io.coef[pop][c] = make_float4(lr, 1.f / bc1, 1.f / bc2, (float)step1);
  io.sel[pop][c] = s;
  io.src[pop][c] = src;
  io.lr_new[pop][c] = lr;
}

// Tournament, replacement and lr mutation of population `pop` (0 G, 1 D) of cell c, given the
// five fitnesses f5 of the cell's neighbourhood; writes the selection, the source individual,
// the new lr and the Adam coefficients (lr, 1 / (1 - beta1^t), 1 / (1 - beta2^t), t).
__device__ void select_one(int c, int pop, const float* f5, const int* __restrict__ nbr,
                           const SelectParams& p, const SelectIO& io) {
  const U4 a = philox_block(p.seed, pop ? 6u : 5u, p.t, (uint32_t)c, 0u);
  const U4 b = philox_block(p.seed, pop ? 6u : 5u, p.t, (uint32_t)c, 1u);
  const uint32_t w[5] = {a.x, a.y, a.z, a.w, b.x};
  const int win = tournament_slot(f5, w, p.tournament_size);
  const int s = p.replace_always ? win : (f5[win] < f5[0] ? win : 0);
  const int src = nbr[c * 5 + s];
  float lr = io.lr_old[pop][src];
  if (p.lr_mutation)
    lr = mutate(lr, p.seed, pop ? 8u : 7u, p.t, (uint32_t)c, p.lr_mut_std, p.lr_mut_thr);
  write_choice(c, pop, s, src, lr, p, io);
}

// Later minibatch steps of an iteration: every cell's centre trains again, in place of a
// selection (slot 0, source individual off + c, its own lr, no mutation).
__global__ void k_centre_select(int cells, int off, SelectParams p, SelectIO io) {
  pdl_wait();
  const int gid = blockIdx.x * blockDim.x + threadIdx.x;
  const int c = gid >> 1;
  if (c >= cells) return;
  const int pop = gid & 1;
  write_choice(c, pop, 0, off + c, io.lr_old[pop][off + c], p, io);
}

__global__ void k_select(const float* __restrict__ fG, const float* __restrict__ fD,
                         const int* __restrict__ nbr, int cells, SelectParams p, SelectIO io) {
  pdl_wait();
  const int gid = blockIdx.x * blockDim.x + threadIdx.x;
  const int c = gid >> 1;
  if (c >= cells) return;
  const int pop = gid & 1;
  select_one(c, pop, (pop ? fD : fG) + c * 5, nbr, p, io);
}

template <bool SELECT>
__global__ void k_fitness(const float* __restrict__ logits, int B, float* __restrict__ LG,
                          float* __restrict__ LD, float* __restrict__ fG, float* __restrict__ fD,
                          int* __restrict__ flag, const int* __restrict__ nbr, SelectParams sp,
                          SelectIO io) {
  pdl_wait();
  const int c = blockIdx.x;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  __shared__ float real_s[5], fake_d[25], fake_g[25], f_s[10];
  const float* lc = logits + (int64_t)c * 5 * 6 * B;
  for (int task = warp; task < 30; task += nw) {
    float s1 = 0.f, s2 = 0.f;
    const bool real = task < 5;
    const int i = real ? 0 : (task - 5) / 5, j = real ? task : (task - 5) % 5;
    const float* l = lc + (int64_t)j * 6 * B + (real ? 0 : (int64_t)(1 + i) * B);
    if (B <= 128) {
      // a lane's (up to four) logits loaded before any is used: one memory latency per mean;
      // the terms are still added in increasing row order
      float x[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) x[u] = lane + 32 * u < B ? l[lane + 32 * u] : 0.f;
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (lane + 32 * u >= B) break;
        if (real) {
          s1 += softplusf(-x[u]);
        } else {
          s1 += softplusf(x[u]);
          s2 += softplusf(-x[u]);
        }
      }
    } else if (real) {
      for (int b = lane; b < B; b += 32) s1 += softplusf(-l[b]);
    } else {
      for (int b = lane; b < B; b += 32) {
        s1 += softplusf(l[b]);
        s2 += softplusf(-l[b]);
      }
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      s1 += __shfl_xor_sync(0xffffffffu, s1, o);
      s2 += __shfl_xor_sync(0xffffffffu, s2, o);
    }
    if (lane == 0) {
      if (task < 5) real_s[task] = s1 / (float)B;
      else {
        fake_d[task - 5] = s1 / (float)B;
        fake_g[task - 5] = s2 / (float)B;
      }
    }
  }
  __syncthreads();
  if (threadIdx.x < 25) {
    const int i = threadIdx.x / 5, j = threadIdx.x % 5;
    const float ld = real_s[j] + fake_d[threadIdx.x];
    const float lg = fake_g[threadIdx.x];
    LD[c * 25 + threadIdx.x] = ld;
    LG[c * 25 + threadIdx.x] = lg;
    if (!isfinite(ld) || !isfinite(lg)) atomicMin(flag, c);
    (void)i;
  }
  __syncthreads();
  if (threadIdx.x < 5) {
    const int i = threadIdx.x;
    float sg = 0.f, sd = 0.f;
    for (int j = 0; j < 5; ++j) {
      sg += fake_g[i * 5 + j];
      sd += real_s[i] + fake_d[j * 5 + i];  // f_D of slot i: mean over generator slots j
    }
    fG[c * 5 + i] = sg / 5.f;
    fD[c * 5 + i] = sd / 5.f;
    f_s[i] = sg / 5.f;
    f_s[5 + i] = sd / 5.f;
  }
  if (SELECT) {
    // the cell's tournaments follow at once: G in thread 0, D in thread 1
    __syncthreads();
    if (threadIdx.x < 2) select_one(c, threadIdx.x, f_s + 5 * threadIdx.x, nbr, sp, io);
  }
}

void launch_fitness(const float* logits, int cells, int B, float* LG, float* LD, float* fG,
                    float* fD, int* flag, cudaStream_t st) {
  // one warp per mean
  launch_pdl(k_fitness<false>, dim3(cells), dim3(960), 0, st, logits, B, LG, LD, fG, fD, flag,
             (const int*)nullptr, SelectParams{}, SelectIO{});
}

void launch_fitness_select(const float* logits, int cells, int B, float* LG, float* LD,
                           float* fG, float* fD, int* flag, const int* nbr,
                           const SelectParams& p, const SelectIO& io, cudaStream_t st) {
  launch_pdl(k_fitness<true>, dim3(cells), dim3(960), 0, st, logits, B, LG, LD, fG, fD, flag, nbr,
             p, io);
}

void launch_select(const float* fG, const float* fD, const int* nbr, int cells,
                   const SelectParams& p, const SelectIO& io, cudaStream_t st) {
  launch_pdl(k_select, dim3((2 * cells + 127) / 128), dim3(128), 0, st, fG, fD, nbr, cells, p,
             io);
}

void launch_centre_select(int cells, int off, const SelectParams& p, const SelectIO& io,
                          cudaStream_t st) {
  launch_pdl(k_centre_select, dim3((2 * cells + 127) / 128), dim3(128), 0, st, cells, off, p, io);
}

// ------------------------------------------------------------------------------------------
// Training input of cell c: TX[c] = [E[c] rows [0, B); E[c] rows of generator slot sel_g[c]].
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void k_train_prep(const T* __restrict__ E, int64_t e_cell, const int* __restrict__ sel_g,
                             T* __restrict__ TX, int B, int x_dim) {
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp, c = blockIdx.y;
  if (r >= 2 * B) return;
  const int src_row = r < B ? r : B * (1 + sel_g[c]) + (r - B);
  const T* s = E + (int64_t)c * e_cell + (int64_t)src_row * x_dim;
  T* d = TX + ((int64_t)c * 2 * B + r) * x_dim;
  const int bytes = x_dim * (int)sizeof(T);
  if ((bytes & 15) == 0 && (((uintptr_t)s | (uintptr_t)d) & 15) == 0) {
    const uint4* s4 = reinterpret_cast<const uint4*>(s);
    uint4* d4 = reinterpret_cast<uint4*>(d);
    for (int k = lane; k < bytes / 16; k += 32) d4[k] = s4[k];
  } else {
    for (int k = lane; k < x_dim; k += 32) d[k] = s[k];
  }
}

template <typename T>
void launch_train_prep(const T* E, int64_t e_cell, const int* sel_g, T* TX, int cells, int B,
                       int x_dim, cudaStream_t st) {
  launch_pdl(k_train_prep<T>, dim3((2 * B + 7) / 8, cells), dim3(256), 0, st, E, e_cell, sel_g,
             TX, B, x_dim);
}
template void launch_train_prep<float>(const float*, int64_t, const int*, float*, int, int, int,
                                       cudaStream_t);
template void launch_train_prep<bf16>(const bf16*, int64_t, const int*, bf16*, int, int, int,
                                      cudaStream_t);

// ------------------------------------------------------------------------------------------
// Logit deltas of the selected pair of cell c, rows [real, fake (D loss), fake (G loss)]:
//   dl = (s - 1)/B (real), s/B (fake, D loss), (s - 1)/B (fake, G loss), s = sigmoid(logit);
//   J2[r][k] = dl_r * w3[k] * lrelu'(g2[r'][k])  (r' = r, or r - B for the G-loss rows);
//   dW3 = sum_{r < 2B} dl_r g2[r],  db3 = sum_{r < 2B} dl_r.
// One block per cell, one thread per hidden unit.
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void __launch_bounds__(512) k_dlogit(
    const float* __restrict__ TL, const T* __restrict__ TG2, const T* __restrict__ wD,
    int64_t wD_stride, int64_t off_w3, const int* __restrict__ src_d, int B, int H, float slope,
    T* __restrict__ J2, float* __restrict__ gD, int64_t gD_stride, int64_t off_gw3,
    int64_t off_gb3, int64_t off_gb2) {
  pdl_wait();
  // Lanes own column groups of 8 (threads of the block: H / 8 groups x RG row groups); the RG
  // partial sums of dW3 and of db2 (the column sums of J2 over the D-loss rows) are added in a
  // fixed order.
  extern __shared__ float dl[];  // [3B] deltas, then [RG][H] and [RG][H] partial sums
  const int c = blockIdx.x;
  const int ng = (H + 7) / 8;
  const int RG = blockDim.x / ng;
  float* part = dl + 3 * B;
  float* part2 = part + RG * H;
  const float* l = TL + (int64_t)c * 2 * B;
  for (int r = threadIdx.x; r < 3 * B; r += blockDim.x) {
    const float x = r < 2 * B ? l[r] : l[r - B];
    const float s = 1.f / (1.f + expf(-x));
    dl[r] = (r < B || r >= 2 * B) ? (s - 1.f) / (float)B : s / (float)B;
  }
  __syncthreads();
  const int gi = threadIdx.x % ng, rg = threadIdx.x / ng;
  const int k0 = gi * 8;
  const T* w3 = wD + (int64_t)src_d[c] * wD_stride + off_w3;
  const T* g2 = TG2 + (int64_t)c * 2 * B * H;
  T* j2 = J2 + (int64_t)c * 3 * B * H;
  float wk[8], acc[8], acc2[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    wk[e] = k0 + e < H ? to_f<T>(w3[k0 + e]) : 0.f;
    acc[e] = 0.f;
    acc2[e] = 0.f;
  }
  if (rg < RG) {
    const bool vec = sizeof(T) == 2 && (H & 7) == 0;
    // the rows of this thread in groups of eight, the eight loads issued before any is used (one
    // memory latency per group); rows are still taken in increasing order
    constexpr int U = 8;
    for (int r0 = rg; vec && r0 < 3 * B; r0 += U * RG) {
      uint4 qv[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int r = r0 + u * RG;
        const int rr = r < 2 * B ? r : r - B;
        if (r < 3 * B) qv[u] = *reinterpret_cast<const uint4*>(g2 + (int64_t)rr * H + k0);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int r = r0 + u * RG;
        if (r >= 3 * B) break;
        const float dr = dl[r];
        // eight bf16 columns in one 16-byte load and store
        const uint4 q = qv[u];
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
        uint32_t o[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162*>(&w[e]);
          const float g0 = __low2float(v), g1 = __high2float(v);
          const float y0 = dr * wk[2 * e] * (g0 > 0.f ? 1.f : slope);
          const float y1 = dr * wk[2 * e + 1] * (g1 > 0.f ? 1.f : slope);
          __nv_bfloat162 y = __floats2bfloat162_rn(y0, y1);
          o[e] = *reinterpret_cast<uint32_t*>(&y);
          if (r < 2 * B) {
            acc[2 * e] = fmaf(dr, g0, acc[2 * e]);
            acc[2 * e + 1] = fmaf(dr, g1, acc[2 * e + 1]);
            acc2[2 * e] += y0;
            acc2[2 * e + 1] += y1;
          }
        }
        *reinterpret_cast<uint4*>(j2 + (int64_t)r * H + k0) = make_uint4(o[0], o[1], o[2], o[3]);
      }
    }
    for (int r = rg; !vec && r < 3 * B; r += RG) {
      const int rr = r < 2 * B ? r : r - B;
      const float dr = dl[r];
      {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          if (k0 + e >= H) break;
          const float gv = to_f<T>(g2[(int64_t)rr * H + k0 + e]);
          const float yv = dr * wk[e] * (gv > 0.f ? 1.f : slope);
          j2[(int64_t)r * H + k0 + e] = from_f<T>(yv);
          if (r < 2 * B) {
            acc[e] = fmaf(dr, gv, acc[e]);
            acc2[e] += yv;
          }
        }
      }
    }
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (k0 + e < H) {
        part[rg * H + k0 + e] = acc[e];
        part2[rg * H + k0 + e] = acc2[e];
      }
  }
  __syncthreads();
  float* g = gD + (int64_t)c * gD_stride;
  for (int k = threadIdx.x; k < H; k += blockDim.x) {
    float t = 0.f, t2 = 0.f;
    for (int q = 0; q < RG; ++q) {
      t += part[q * H + k];
      t2 += part2[q * H + k];
    }
    g[off_gw3 + k] = t;
    g[off_gb2 + k] = t2;
  }
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int r = 0; r < 2 * B; ++r) t += dl[r];
    g[off_gb3] = t;
  }
}

template <typename T>
void launch_dlogit(const float* TL, const T* TG2, const T* wD, int64_t wD_stride, int64_t off_w3,
                   const int* src_d, int cells, int B, int H, float slope, T* J2, float* gD,
                   int64_t gD_stride, int64_t off_gw3, int64_t off_gb3, int64_t off_gb2,
                   cudaStream_t st) {
  const int ng = (H + 7) / 8;
  int rg = 512 / ng;
  if (rg < 1) rg = 1;
  if (rg > 16) rg = 16;
  const int threads = ((rg * ng + 31) / 32) * 32;
  const size_t smem = (3 * (size_t)B + 2 * (size_t)(threads / ng) * H) * sizeof(float);
  launch_pdl(k_dlogit<T>, dim3(cells), dim3(threads), smem, st, TL, TG2, wD, wD_stride, off_w3,
             src_d, B, H, slope, J2, gD, gD_stride, off_gw3, off_gb3, off_gb2);
}
template void launch_dlogit<float>(const float*, const float*, const float*, int64_t, int64_t,
                                   const int*, int, int, int, float, float*, float*, int64_t,
                                   int64_t, int64_t, int64_t, cudaStream_t);
template void launch_dlogit<bf16>(const float*, const bf16*, const bf16*, int64_t, int64_t,
                                  const int*, int, int, int, float, bf16*, float*, int64_t,
                                  int64_t, int64_t, int64_t, cudaStream_t);

// ------------------------------------------------------------------------------------------
// Adam (Kingma & Ba 2015, Algorithm 1) fused with the replacement copy: the new centre of
// cell c starts from individual src[c] of the old snapshot and is written to cell c of the
// new snapshot (fp32 master, m, v, bf16 copy, step, lr). HBM-bound: 16-byte loads/stores,
// each thread walks float4 groups of its cell with a grid stride.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void adam4(float4& w, float4& m, float4& v, const float4 g, float b1,
                                      float b2, float lr, float ib1, float ib2, float eps) {
  adam_elem(w.x, m.x, v.x, g.x, b1, b2, lr, ib1, ib2, eps);
  adam_elem(w.y, m.y, v.y, g.y, b1, b2, lr, ib1, ib2, eps);
  adam_elem(w.z, m.z, v.z, g.z, b1, b2, lr, ib1, ib2, eps);
  adam_elem(w.w, m.w, v.w, g.w, b1, b2, lr, ib1, ib2, eps);
}

__global__ void __launch_bounds__(256) k_adam(PopView old_p, PopView new_p,
                                              const float* __restrict__ grad,
                                              const int* __restrict__ src,
                                              const float4* __restrict__ coef, int64_t P,
                                              int64_t Ps, float beta1, float beta2, float eps) {
  pdl_wait();
  const int c = blockIdx.y;
  const int s = src[c];
  const float4 cf = coef[c];
  const float lr = cf.x, ib1 = cf.y, ib2 = cf.z;
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    new_p.step[c] = (int)cf.w;
    new_p.lr[c] = lr;
  }
  const int64_t so = (int64_t)s * Ps, co = (int64_t)c * Ps;
  const int64_t n4 = P >> 2;
  const float4* __restrict__ w_in = reinterpret_cast<const float4*>(old_p.w + so);
  const float4* __restrict__ m_in = reinterpret_cast<const float4*>(old_p.m + so);
  const float4* __restrict__ v_in = reinterpret_cast<const float4*>(old_p.v + so);
  const float4* __restrict__ g_in = reinterpret_cast<const float4*>(grad + co);
  float4* w_out = reinterpret_cast<float4*>(new_p.w + co);
  float4* m_out = reinterpret_cast<float4*>(new_p.m + co);
  float4* v_out = reinterpret_cast<float4*>(new_p.v + co);
  uint2* b_out = new_p.wb ? reinterpret_cast<uint2*>(new_p.wb + co) : nullptr;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
       i += (int64_t)gridDim.x * blockDim.x) {
    float4 w = __ldcs(w_in + i), m = __ldcs(m_in + i), v = __ldcs(v_in + i);
    const float4 g = __ldcs(g_in + i);
    adam4(w, m, v, g, beta1, beta2, lr, ib1, ib2, eps);
    __stcs(w_out + i, w);
    __stcs(m_out + i, m);
    __stcs(v_out + i, v);
    if (b_out) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(w.x, w.y);
      __nv_bfloat162 hi = __floats2bfloat162_rn(w.z, w.w);
      uint2 pk;
      pk.x = *reinterpret_cast<uint32_t*>(&lo);
      pk.y = *reinterpret_cast<uint32_t*>(&hi);
      b_out[i] = pk;
    }
  }
  // tail (P not a multiple of 4)
  if (blockIdx.x == 0 && threadIdx.x < (P & 3)) {
    const int64_t k = (n4 << 2) + threadIdx.x;
    float wk = old_p.w[so + k], mk = old_p.m[so + k], vk = old_p.v[so + k];
    adam_elem(wk, mk, vk, grad[co + k], beta1, beta2, lr, ib1, ib2, eps);
    new_p.w[co + k] = wk;
    new_p.m[co + k] = mk;
    new_p.v[co + k] = vk;
    if (new_p.wb) new_p.wb[co + k] = __float2bfloat16_rn(wk);
  }
}

void launch_adam(const PopView& old_p, const PopView& new_p, const float* grad, const int* src,
                 const float4* coef, int cells, int64_t P, int64_t Ps, float beta1, float beta2,
                 float eps, cudaStream_t st) {
  // about 8 resident 256-thread blocks per SM over the whole population
  int per_cell = (int)((P / 4 + 255) / 256);
  const int target = (152 * 8 + cells - 1) / cells;
  if (per_cell > target * 4) per_cell = target * 4;
  if (per_cell < 1) per_cell = 1;
  dim3 grid(per_cell, cells);
  launch_pdl(k_adam, grid, dim3(256), 0, st, old_p, new_p, grad, src, coef, P, Ps, beta1, beta2,
             eps);
}

// ------------------------------------------------------------------------------------------
// Generator-mixture score (Section 3 step 4): squared norms of the evaluation rows, the Gaussian
// kernel's block sums (from a stored Gram matrix on the CUDA-core path), and the ES-(1+1) step.
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void k_row_norms(const T* __restrict__ E, int64_t e_cell, int rows, int x,
                            float* __restrict__ out) {
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp, c = blockIdx.y;
  if (r >= rows) return;
  const T* e = E + (int64_t)c * e_cell + (int64_t)r * x;
  float s = 0.f;
  for (int k = lane; k < x; k += 32) {
    const float v = to_f<T>(e[k]);
    s = fmaf(v, v, s);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) out[(int64_t)c * rows + r] = s;
}

template <typename T>
void launch_row_norms(const T* E, int64_t e_cell, int cells, int rows, int x, float* out,
                      cudaStream_t st) {
  launch_pdl(k_row_norms<T>, dim3((rows + 7) / 8, cells), dim3(256), 0, st, E, e_cell, rows, x,
             out);
}
template void launch_row_norms<float>(const float*, int64_t, int, int, int, float*, cudaStream_t);
template void launch_row_norms<bf16>(const bf16*, int64_t, int, int, int, float*, cudaStream_t);

// One warp per row r of cell c: for each block b of B columns, the sum over its columns s (in
// lane-strided order, then a fixed shuffle tree) of exp(-(n_r + n_s - 2 gram[r][s]) / x).
__global__ void k_mix_partials(const float* __restrict__ gram, const float* __restrict__ rnorm,
                               int rows, int B, int x, float* __restrict__ out) {
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp, c = blockIdx.y;
  if (r >= rows) return;
  const float* gr = gram + ((int64_t)c * rows + r) * rows;
  const float* n = rnorm + (int64_t)c * rows;
  const float nr = n[r], inv_x = 1.f / (float)x;
  for (int b = 0; b < rows / B; ++b) {
    float s = 0.f;
    for (int q = b * B + lane; q < (b + 1) * B; q += 32)
      s += __expf(-(nr + n[q] - 2.f * gr[q]) * inv_x);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) out[((int64_t)c * rows + r) * 6 + b] = s;
  }
}

void launch_mix_partials(const float* gram, const float* rnorm, int cells, int rows, int B, int x,
                         float* out, cudaStream_t st) {
  launch_pdl(k_mix_partials, dim3((rows + 7) / 8, cells), dim3(256), 0, st, gram, rnorm, rows, B,
             x, out);
}

__device__ __forceinline__ float mix_mmd2(const float* w, const float* S) {
  // sum_ij w_i w_j S[1+i][1+j] - 2 sum_i w_i S[1+i][0] + S[0][0]
  float q = 0.f, l = 0.f;
#pragma unroll
  for (int i = 0; i < 5; ++i) {
    float row = 0.f;
#pragma unroll
    for (int j = 0; j < 5; ++j) row = fmaf(w[j], S[(1 + i) * 6 + 1 + j], row);
    q = fmaf(w[i], row, q);
    l = fmaf(w[i], S[(1 + i) * 6], l);
  }
  return q - 2.f * l + S[0];
}

// One block per cell: the 6x6 block means S[a][b] = (sum over the rows r of block a and the
// column ranges h of part[c][r][h][b]) / B^2, then the ES-(1+1) step of the cell's weights w:
// w' = max(w + sigma n, 0) / sum (n: the first five normals of stream MIX at iteration t; w kept
// if the sum is 0), kept iff its squared MMD is lower. Warp a sums block a's rows: lane l takes
// rows l, l + 32, ... (all h), then a fixed shuffle tree.
__global__ void __launch_bounds__(192) k_mix_es(const float* __restrict__ part, int nh, int rows,
                                                int B, float* mix, float* __restrict__ S_out,
                                                float* __restrict__ score_out, uint64_t seed,
                                                uint32_t t, float sigma) {
  pdl_wait();
  const int c = blockIdx.x;
  __shared__ float S[36];
  const int a = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float acc[6] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int r = a * B + lane; r < (a + 1) * B; r += 32) {
    const float* q = part + ((int64_t)c * rows + r) * nh * 6;
    for (int h = 0; h < nh; ++h) {
#pragma unroll
      for (int b = 0; b < 6; ++b) acc[b] += q[h * 6 + b];
    }
  }
#pragma unroll
  for (int b = 0; b < 6; ++b) {
    float v = acc[b];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (lane == 0) {
      S[a * 6 + b] = v / ((float)B * (float)B);
      S_out[(int64_t)c * 36 + a * 6 + b] = S[a * 6 + b];
    }
  }
  __syncthreads();
  if (threadIdx.x != 0) return;
  float w[5], cand[5], nrm[5];
  const U4 r0 = philox_block(seed, 9u, t, (uint32_t)c, 0u);
  const U4 r1 = philox_block(seed, 9u, t, (uint32_t)c, 1u);
  const float2 n01 = box_muller(r0.x, r0.y), n23 = box_muller(r0.z, r0.w),
               n4 = box_muller(r1.x, r1.y);
  nrm[0] = n01.x;
  nrm[1] = n01.y;
  nrm[2] = n23.x;
  nrm[3] = n23.y;
  nrm[4] = n4.x;
  float tot = 0.f;
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    w[k] = mix[c * 5 + k];
    cand[k] = fmaxf(fmaf(sigma, nrm[k], w[k]), 0.f);
    tot += cand[k];
  }
#pragma unroll
  for (int k = 0; k < 5; ++k) cand[k] = tot > 0.f ? cand[k] / tot : w[k];
  const float old = mix_mmd2(w, S), nw = mix_mmd2(cand, S);
  const bool acc_new = nw < old;
  if (acc_new)
#pragma unroll
    for (int k = 0; k < 5; ++k) mix[c * 5 + k] = cand[k];
  score_out[c] = acc_new ? nw : old;
}

void launch_mix_es(const float* part, int nh, int cells, int rows, int B, float* mix, float* S,
                   float* score, uint64_t seed, uint32_t t, float sigma, cudaStream_t st) {
  launch_pdl(k_mix_es, dim3(cells), dim3(192), 0, st, part, nh, rows, B, mix, S, score, seed, t,
             sigma);
}

// The iteration's results for one host copy: out[0, n) = fG, out[n, 2n) = fD (n = cells * 5),
// then the eight status words (a null flag reads as its all-clear value: 0 for the first
// seven, INT_MAX for the last).
__global__ void k_gather_status(const float* __restrict__ fG, const float* __restrict__ fD, int n,
                                StatusFlags fl, float* __restrict__ out) {
  pdl_wait();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < 2 * n; i += gridDim.x * blockDim.x)
    out[i] = i < n ? fG[i] : fD[i - n];
  if (blockIdx.x == 0 && threadIdx.x < 8) {
    const int* f = fl.p[threadIdx.x];
    reinterpret_cast<int*>(out + 2 * n)[threadIdx.x] =
        f ? *f : (threadIdx.x < 7 ? 0 : 0x7FFFFFFF);
  }
}

void launch_gather_status(const float* fG, const float* fD, int n, const StatusFlags& fl,
                          float* out, bool pdl, cudaStream_t st) {
  launch_kernel(pdl, k_gather_status, dim3(2), dim3(256), 0, st, fG, fD, n, fl, out);
}

}  // namespace lipz
