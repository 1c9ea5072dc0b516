// CUDA-core kernels of the DCGAN networks (Table 1, CelebA column): one grouped implicit-GEMM
// kernel for convolutions, transposed convolutions and their weight gradients, training-mode
// batch normalisation forward and backward, and the discriminator's 4x4 -> 1 output layer.
// Images and activations are NCHW per sample; all spatial sizes are powers of two and every
// kernel is 4 x 4.
#include "common.cuh"
#include "engine.h"

namespace lipz {

// ------------------------------------------------------------------------------------------
// Implicit GEMM, 64 x 64 output tile per block, k-slices of 16 gathered into shared memory,
// 4 x 4 outputs per thread, fp32 accumulation in k order.
//   CONV_FWD:  y[n][o][i][j] = sum_{c,ky,kx} a[n][c][s i - p + ky][s j - p + kx] w[o][c][ky][kx]
//   CONVT_FWD: y[n][o][i][j] = sum_{c,ky,kx} a[n][c][(i + p - ky) / s][(j + p - kx) / s]
//              w[c][o][ky][kx]   (terms whose index is fractional or outside the image vanish)
//   WGRAD:     y[m][c][ky][kx] = sum_{n,i,j} a[n][m][i][j] b[n][c][s i - p + ky][s j - p + kx]
//              (split over K = n * Ha * Wa; partial sums reduced in a fixed order)
//   DENSE1:    the generator's first layer (1x1 input, kernel 4x4, stride 1, pad 0) as the plain
//              product y[n][(tap, o)] = sum_c a[n][c] w[c][o][tap] (M = n, N = 16 co, K = ca),
//              stored channel-last (tap, o) or channel-major (o, tap)
//   CONVT2:    CONVT_FWD at stride 2 by output parity class (i mod 2, j mod 2), one class per
//              block (blockIdx.z = problem * 4 + class): only the taps ky = (i + p) mod 2 + 2 u,
//              kx = (j + p) mod 2 + 2 v (u, v in {0, 1}) reach a pixel of the class, so K is
//              4 per input channel instead of 16
// ------------------------------------------------------------------------------------------
enum { CONV_FWD = CONV_FWD_MODE, CONVT_FWD = CONVT_FWD_MODE, WGRAD = WGRAD_MODE,
       CONVT2 = CONVT2_MODE, DENSE1 = DENSE1_MODE };
enum { CEPI_NONE = CEPI_NONE_, CEPI_LRELU = CEPI_LRELU_, CEPI_TANH = CEPI_TANH_,
       CEPI_DLRELU = CEPI_DLRELU_, CEPI_DTANH = CEPI_DTANH_ };

__device__ __forceinline__ void conv_dims(const ConvDesc& d, int mode, int& M, int& N, int& K) {
  if (mode == WGRAD) {
    M = d.ca;
    N = d.co * 16;
    K = d.n << (d.lha + d.lwa);
  } else if (mode == CONVT2) {
    M = d.n << (d.lho + d.lwo - 2);
    N = d.co;
    K = d.ca * 4;
  } else if (mode == DENSE1) {
    M = d.n;
    N = d.co * 16;
    K = d.ca;
  } else {
    M = d.n << (d.lho + d.lwo);
    N = d.co;
    K = d.ca * 16;
  }
}

template <int MODE, typename TI, typename TO, int EPI>
__global__ void __launch_bounds__(256) k_conv(const ConvDesc* __restrict__ descs,
                                              const int* __restrict__ wsel_override, int splits,
                                              float* __restrict__ part, float slope) {
  pdl_wait();
  const int prob = blockIdx.z / splits, split = blockIdx.z % splits;
  const ConvDesc d = descs[prob];
  int M, N, K;
  conv_dims(d, MODE, M, N, K);
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  if (m0 >= M || n0 >= N) return;
  const TI* A = (const TI*)d.a;
  const TI* Bm = (const TI*)d.b;
  if (MODE != WGRAD) {
    const int* ws = wsel_override ? wsel_override : d.wsel;
    if (ws) Bm += (int64_t)ws[d.wsel_idx] * d.wsel_stride;
  }
  // this block's k range (WGRAD: one of `splits` equal chunks, multiples of 16)
  int kb = 0, ke = K;
  if (MODE == WGRAD) {
    const int kc = ((K + splits - 1) / splits + 15) & ~15;
    kb = split * kc;
    ke = min(K, kb + kc);
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
  const int Ha = 1 << d.lha, Wa = 1 << d.lwa;
  // CONVT2: this block's output class and its first taps
  const int py = (split >> 1) & 1, px = split & 1;
  const int ky0 = (py + d.p) & 1, kx0 = (px + d.p) & 1;
  const int lqy = d.lho - 1, lqx = d.lwo - 1;
  for (int k0 = kb; k0 < ke; k0 += 16) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int idx = tid + 256 * q;
      // A element (m, k): k fastest (channel-last weight-gradient deltas: m fastest)
      {
        const bool mfast = MODE == WGRAD && d.a_hwc;
        const int mm = mfast ? (idx & 63) : (idx >> 4), kk = mfast ? (idx >> 6) : (idx & 15);
        const int m = m0 + mm, k = k0 + kk;
        float v = 0.f;
        if (m < M && k < ke) {
          if (MODE == DENSE1) {
            v = to_f<TI>(A[(int64_t)m * d.ca + k]);
          } else if (MODE == WGRAD) {
            const int nb = k >> (d.lha + d.lwa), yx = k & ((1 << (d.lha + d.lwa)) - 1);
            v = to_f<TI>(A[d.a_hwc ? (((int64_t)nb << (d.lha + d.lwa)) + yx) * d.ca + m
                                   : (((int64_t)nb * d.ca + m) << (d.lha + d.lwa)) + yx]);
          } else if (MODE == CONVT2) {
            const int nb = m >> (lqy + lqx);
            const int oy = 2 * ((m >> lqx) & ((1 << lqy) - 1)) + py;
            const int ox = 2 * (m & ((1 << lqx) - 1)) + px;
            const int c = k >> 2, ky = ky0 + 2 * ((k >> 1) & 1), kx = kx0 + 2 * (k & 1);
            const int iy = (oy + d.p - ky) >> 1, ix = (ox + d.p - kx) >> 1;
            if (oy + d.p - ky >= 0 && ox + d.p - kx >= 0 && iy < Ha && ix < Wa)
              v = to_f<TI>(A[d.a_hwc ? ((((int64_t)nb << (d.lha + d.lwa)) + (iy << d.lwa) + ix) *
                                            d.ca + c)
                                     : (((int64_t)nb * d.ca + c) << (d.lha + d.lwa)) +
                                           (iy << d.lwa) + ix]);
          } else {
            const int nb = m >> (d.lho + d.lwo);
            const int oy = (m >> d.lwo) & ((1 << d.lho) - 1), ox = m & ((1 << d.lwo) - 1);
            const int c = k >> 4, ky = (k >> 2) & 3, kx = k & 3;
            int iy, ix;
            bool ok;
            if (MODE == CONV_FWD) {
              iy = oy * d.s - d.p + ky;
              ix = ox * d.s - d.p + kx;
              ok = true;
            } else {
              const int ty = oy + d.p - ky, tx = ox + d.p - kx;
              ok = ty >= 0 && tx >= 0 && (ty % d.s) == 0 && (tx % d.s) == 0;
              iy = ty / d.s;
              ix = tx / d.s;
            }
            if (ok && iy >= 0 && iy < Ha && ix >= 0 && ix < Wa)
              v = to_f<TI>(A[d.a_hwc ? ((((int64_t)nb << (d.lha + d.lwa)) + (iy << d.lwa) + ix) *
                                            d.ca + c)
                                     : (((int64_t)nb * d.ca + c) << (d.lha + d.lwa)) +
                                           (iy << d.lwa) + ix]);
          }
        }
        As[kk][mm] = v;
      }
      // B element (k, n): n fastest for WGRAD (gathered image), k fastest for the weights
      {
        int kk, nn;
        if (MODE == WGRAD) {
          nn = idx & 63;
          kk = idx >> 6;
        } else {
          nn = idx >> 4;
          kk = idx & 15;
        }
        const int k = k0 + kk, n = n0 + nn;
        float v = 0.f;
        if (n < N && k < ke) {
          if (MODE == DENSE1) {
            // n = tap * co + o
            const int tap = n / d.co, o = n - tap * d.co;
            v = to_f<TI>(Bm[((int64_t)k * d.co + o) * 16 + tap]);
          } else if (MODE == WGRAD) {
            const int nb = k >> (d.lha + d.lwa);
            const int ay = (k >> d.lwa) & (Ha - 1), ax = k & (Wa - 1);
            // channel-last b: n = (tap, c) so that neighbouring threads read neighbouring
            // channels; otherwise n = (c, tap)
            int c, tap;
            if (d.b_hwc) {
              tap = n / d.co;
              c = n - tap * d.co;
            } else {
              c = n >> 4;
              tap = n & 15;
            }
            const int ky = tap >> 2, kx = tap & 3;
            const int by = ay * d.s - d.p + ky, bx = ax * d.s - d.p + kx;
            if (by >= 0 && by < (1 << d.lho) && bx >= 0 && bx < (1 << d.lwo))
              v = to_f<TI>(Bm[d.b_hwc ? ((((int64_t)nb << (d.lho + d.lwo)) + (by << d.lwo) + bx) *
                                             d.co + c)
                                      : (((int64_t)nb * d.co + c) << (d.lho + d.lwo)) +
                                            (by << d.lwo) + bx]);
          } else if (MODE == CONV_FWD) {
            v = to_f<TI>(Bm[(int64_t)n * K + k]);
          } else if (MODE == CONVT2) {
            const int ky = ky0 + 2 * ((k >> 1) & 1), kx = kx0 + 2 * (k & 1);
            v = to_f<TI>(Bm[((int64_t)(k >> 2) * d.co + n) * 16 + ky * 4 + kx]);
          } else {
            v = to_f<TI>(Bm[((int64_t)(k >> 4) * d.co + n) * 16 + (k & 15)]);
          }
        }
        Bs[kk][nn] = v;
      }
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
  if (MODE == WGRAD) {
    float* o = part + ((int64_t)blockIdx.z * M) * N;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int m = m0 + tm + i;
      if (m >= M) continue;
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int n = n0 + tn + j;
        if (n < N) {
          const int e = d.b_hwc ? (n % d.co) * 16 + n / d.co : n;
          o[(int64_t)m * N + e] = acc[i][j];
        }
      }
    }
    return;
  }
  TO* Y = (TO*)d.out;
  const TI* aux = (const TI*)d.aux;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + tm + i;
    if (m >= M) continue;
    int nb, yx;
    if (MODE == DENSE1) {
      nb = m;
      yx = 0;
    } else if (MODE == CONVT2) {
      nb = m >> (lqy + lqx);
      const int oy = 2 * ((m >> lqx) & ((1 << lqy) - 1)) + py;
      const int ox = 2 * (m & ((1 << lqx) - 1)) + px;
      yx = (oy << d.lwo) + ox;
    } else {
      nb = m >> (d.lho + d.lwo);
      yx = m & ((1 << (d.lho + d.lwo)) - 1);
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tn + j;
      if (n >= N) continue;
      int64_t o;
      if (MODE == DENSE1) {
        const int tap = n / d.co, oc = n - tap * d.co;
        o = d.nhwc_out ? (int64_t)m * N + n : ((int64_t)m * d.co + oc) * 16 + tap;
      } else {
        o = d.nhwc_out ? ((((int64_t)nb << (d.lho + d.lwo)) + yx) * d.co + n)
                       : ((((int64_t)nb * d.co + n) << (d.lho + d.lwo)) + yx);
      }
      float v = acc[i][j];
      if (EPI == CEPI_LRELU) v = v > 0.f ? v : slope * v;
      if (EPI == CEPI_TANH) v = tanhf(v);
      if (EPI == CEPI_DLRELU) v = to_f<TI>(aux[o]) > 0.f ? v : slope * v;
      if (EPI == CEPI_DTANH) {
        const float f = to_f<TI>(aux[o]);
        v = v * (1.f - f * f);
      }
      Y[o] = from_f<TO>(v);
    }
  }
}

// WGRAD partials -> weight gradient: y[e] = sum over splits, in split order.
__global__ void k_wgrad_reduce(const ConvDesc* __restrict__ descs, int splits,
                               const float* __restrict__ part, int64_t part_stride) {
  pdl_wait();
  const ConvDesc d = descs[blockIdx.y];
  const int64_t total = (int64_t)d.ca * d.co * 16;
  const float* p = part + (int64_t)blockIdx.y * splits * part_stride;
  float* y = (float*)d.out;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total;
       e += (int64_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int q = 0; q < splits; ++q) s += p[(int64_t)q * part_stride + e];
    y[e] = s;
  }
}

template <int MODE, typename TI, typename TO, int EPI>
void launch_conv_t(const ConvDesc* descs, int n_problems, int max_m, int max_n, const int* wsel,
                   int splits, float* part, int64_t part_stride, float slope, cudaStream_t st) {
  if (n_problems <= 0) return;
  // CONVT2: max_m counts every output pixel; a class holds a quarter of them
  const int zs = MODE == WGRAD ? splits : (MODE == CONVT2 ? 4 : 1);
  if (MODE == CONVT2) max_m = (max_m + 3) / 4;
  dim3 grid((max_n + 63) / 64, (max_m + 63) / 64, n_problems * zs);
  launch_pdl(k_conv<MODE, TI, TO, EPI>, grid, dim3(256), 0, st, descs, wsel, zs, part, slope);
  if (MODE == WGRAD)
    launch_pdl(k_wgrad_reduce, dim3(64, n_problems), dim3(256), 0, st, descs, splits,
               (const float*)part, part_stride);
}

// One entry point over the instantiated combinations; the element type of the gathered
// operands is the population precision (bf16 selects it), outputs as `out_f32` says.
void launch_conv(int mode, int epi, bool bf, bool out_f32, const ConvDesc* descs,
                 int n_problems, int max_m, int max_n, const int* wsel, int splits, float* part,
                 int64_t part_stride, float slope, cudaStream_t st) {
#define LIPZ_CONV(MODE, TI, TO, EPI)                                                          \
  launch_conv_t<MODE, TI, TO, EPI>(descs, n_problems, max_m, max_n, wsel, splits, part,     \
                                   part_stride, slope, st)
  if (mode == WGRAD) {
    if (bf) LIPZ_CONV(WGRAD, bf16, float, CEPI_NONE);
    else LIPZ_CONV(WGRAD, float, float, CEPI_NONE);
    return;
  }
  if (mode == DENSE1) {
    if (bf) LIPZ_CONV(DENSE1, bf16, float, CEPI_NONE);
    else LIPZ_CONV(DENSE1, float, float, CEPI_NONE);
    return;
  }
  if (mode == CONVT2) {
    if (bf) {
      if (out_f32) LIPZ_CONV(CONVT2, bf16, float, CEPI_NONE);
      else if (epi == CEPI_TANH) LIPZ_CONV(CONVT2, bf16, bf16, CEPI_TANH);
      else if (epi == CEPI_DLRELU) LIPZ_CONV(CONVT2, bf16, bf16, CEPI_DLRELU);
      else if (epi == CEPI_DTANH) LIPZ_CONV(CONVT2, bf16, bf16, CEPI_DTANH);
      else LIPZ_CONV(CONVT2, bf16, bf16, CEPI_NONE);
    } else {
      if (epi == CEPI_TANH) LIPZ_CONV(CONVT2, float, float, CEPI_TANH);
      else if (epi == CEPI_DLRELU) LIPZ_CONV(CONVT2, float, float, CEPI_DLRELU);
      else if (epi == CEPI_DTANH) LIPZ_CONV(CONVT2, float, float, CEPI_DTANH);
      else LIPZ_CONV(CONVT2, float, float, CEPI_NONE);
    }
    return;
  }
  if (bf) {
    if (out_f32) {
      if (mode == CONV_FWD) LIPZ_CONV(CONV_FWD, bf16, float, CEPI_NONE);
      else LIPZ_CONV(CONVT_FWD, bf16, float, CEPI_NONE);
    } else if (mode == CONV_FWD) {
      if (epi == CEPI_LRELU) LIPZ_CONV(CONV_FWD, bf16, bf16, CEPI_LRELU);
      else LIPZ_CONV(CONV_FWD, bf16, bf16, CEPI_NONE);
    } else {
      if (epi == CEPI_TANH) LIPZ_CONV(CONVT_FWD, bf16, bf16, CEPI_TANH);
      else if (epi == CEPI_DLRELU) LIPZ_CONV(CONVT_FWD, bf16, bf16, CEPI_DLRELU);
      else if (epi == CEPI_DTANH) LIPZ_CONV(CONVT_FWD, bf16, bf16, CEPI_DTANH);
      else LIPZ_CONV(CONVT_FWD, bf16, bf16, CEPI_NONE);
    }
  } else {
    if (mode == CONV_FWD) {
      if (epi == CEPI_LRELU) LIPZ_CONV(CONV_FWD, float, float, CEPI_LRELU);
      else LIPZ_CONV(CONV_FWD, float, float, CEPI_NONE);
    } else {
      if (epi == CEPI_TANH) LIPZ_CONV(CONVT_FWD, float, float, CEPI_TANH);
      else if (epi == CEPI_DLRELU) LIPZ_CONV(CONVT_FWD, float, float, CEPI_DLRELU);
      else if (epi == CEPI_DTANH) LIPZ_CONV(CONVT_FWD, float, float, CEPI_DTANH);
      else LIPZ_CONV(CONVT_FWD, float, float, CEPI_NONE);
    }
  }
#undef LIPZ_CONV
}

// ------------------------------------------------------------------------------------------
// Batch normalisation in training mode, per (problem, channel) over the batch and the image
// (m = n * H * W values), eps 1e-5; statistics in two passes (mean, then the centred sum of
// squares), block reductions in a fixed order.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ float block_sum_256(float v, float* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) sh[w] = v;
  __syncthreads();
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) s += sh[i];
  return s;
}

__device__ __forceinline__ const float* bn_params(const BnDesc& d, const int* wsel_override) {
  const int* ws = wsel_override ? wsel_override : d.wsel;
  return d.params + (ws ? (int64_t)ws[d.wsel_idx] * d.wsel_stride : 0);
}

// Forward: statistics, then h = relu(gamma (c - mean) inv + beta) in the population precision.
template <typename TO>
__global__ void __launch_bounds__(256) k_bn_relu(const BnDesc* __restrict__ descs,
                                                 const int* __restrict__ wsel_override) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int ch = blockIdx.x;
  const int hw = 1 << d.lhw;
  const int64_t m = (int64_t)d.n * hw;
  __shared__ float sh[8];
  float s = 0.f;
  for (int64_t e = threadIdx.x; e < m; e += 256) {
    const int64_t nb = e >> d.lhw, q = e & (hw - 1);
    s += d.c[((nb * d.C + ch) << d.lhw) + q];
  }
  const float mean = block_sum_256(s, sh) / (float)m;
  float v = 0.f;
  for (int64_t e = threadIdx.x; e < m; e += 256) {
    const int64_t nb = e >> d.lhw, q = e & (hw - 1);
    const float t = d.c[((nb * d.C + ch) << d.lhw) + q] - mean;
    v = fmaf(t, t, v);
  }
  const float var = block_sum_256(v, sh) / (float)m;
  const float inv = rsqrtf(var + 1e-5f);
  if (threadIdx.x == 0) {
    d.mean[ch] = mean;
    d.inv[ch] = inv;
  }
  const float* P = bn_params(d, wsel_override);
  const float g = P[d.off_gamma + ch], b = P[d.off_beta + ch];
  TO* h = (TO*)d.h;
  for (int64_t e = threadIdx.x; e < m; e += 256) {
    const int64_t nb = e >> d.lhw, q = e & (hw - 1);
    const int64_t o = ((nb * d.C + ch) << d.lhw) + q;
    h[o] = from_f<TO>(fmaxf(fmaf(g * inv, d.c[o] - mean, b), 0.f));
  }
}

// Backward through ReLU and the batch normalisation: dy = dh (h > 0), xhat = (c - mean) inv;
// dbeta = sum dy, dgamma = sum dy xhat (written to the gradient slots), then
// dc = gamma inv (dy - dbeta / m - xhat dgamma / m) in the population precision.
template <typename TO>
__global__ void __launch_bounds__(256) k_bn_relu_backward(const BnDesc* __restrict__ descs) {
  pdl_wait();
  const BnDesc d = descs[blockIdx.y];
  const int ch = blockIdx.x;
  const int hw = 1 << d.lhw;
  const int64_t m = (int64_t)d.n * hw;
  const TO* h = (const TO*)d.h;
  const float mean = d.mean[ch], inv = d.inv[ch];
  __shared__ float sh[8];
  float sb = 0.f, sg = 0.f;
  for (int64_t e = threadIdx.x; e < m; e += 256) {
    const int64_t nb = e >> d.lhw, q = e & (hw - 1);
    const int64_t o = d.hwc ? e * d.C + ch : ((nb * d.C + ch) << d.lhw) + q;
    const float dy = to_f<TO>(h[o]) > 0.f ? d.dh[o] : 0.f;
    sb += dy;
    sg = fmaf(dy, (d.c[o] - mean) * inv, sg);
  }
  const float dbeta = block_sum_256(sb, sh);
  const float dgamma = block_sum_256(sg, sh);
  if (threadIdx.x == 0) {
    d.dparams[d.off_gamma + ch] = dgamma;
    d.dparams[d.off_beta + ch] = dbeta;
  }
  const float* P = bn_params(d, nullptr);
  const float g = P[d.off_gamma + ch];
  const float k1 = dbeta / (float)m, k2 = dgamma / (float)m;
  TO* dc = (TO*)d.dc;
  for (int64_t e = threadIdx.x; e < m; e += 256) {
    const int64_t nb = e >> d.lhw, q = e & (hw - 1);
    const int64_t o = d.hwc ? e * d.C + ch : ((nb * d.C + ch) << d.lhw) + q;
    const float dy = to_f<TO>(h[o]) > 0.f ? d.dh[o] : 0.f;
    const float xhat = (d.c[o] - mean) * inv;
    dc[o] = from_f<TO>(g * inv * (dy - k1 - xhat * k2));
  }
}

void launch_bn_relu(bool bf, const BnDesc* descs, int n_problems, int channels, const int* wsel,
                    cudaStream_t st) {
  if (bf) launch_pdl(k_bn_relu<bf16>, dim3(channels, n_problems), dim3(256), 0, st, descs, wsel);
  else launch_pdl(k_bn_relu<float>, dim3(channels, n_problems), dim3(256), 0, st, descs, wsel);
}

void launch_bn_relu_backward(bool bf, const BnDesc* descs, int n_problems, int channels,
                             cudaStream_t st) {
  if (bf)
    launch_pdl(k_bn_relu_backward<bf16>, dim3(channels, n_problems), dim3(256), 0, st, descs);
  else
    launch_pdl(k_bn_relu_backward<float>, dim3(channels, n_problems), dim3(256), 0, st, descs);
}

// ------------------------------------------------------------------------------------------
// Discriminator output layer (4 x 4 kernel over the 4 x 4 map: a dot product of K values).
// ------------------------------------------------------------------------------------------
template <typename T>
__global__ void k_logit_dot(const LogitDesc* __restrict__ descs,
                            const int* __restrict__ wsel_override) {
  pdl_wait();
  const LogitDesc d = descs[blockIdx.y];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * (blockDim.x >> 5) + warp;
  if (r >= d.rows) return;
  const int* ws = wsel_override ? wsel_override : d.wsel;
  const T* w = (const T*)d.w + (ws ? (int64_t)ws[d.wsel_idx] * d.wsel_stride : 0);
  const T* x = (const T*)d.a + (int64_t)r * d.K;
  float s = 0.f;
  if (sizeof(T) == 2 && (d.K & 255) == 0 && (((uintptr_t)x | (uintptr_t)w) & 15) == 0) {
    // bf16: eight consecutive k per lane and load (16 bytes), four loads of each operand in
    // flight; lane l takes k = 256 i + 8 l .. + 7 in order
    const uint4* x4 = reinterpret_cast<const uint4*>(x) + lane;
    const uint4* w4 = reinterpret_cast<const uint4*>(w) + lane;
    const int n = d.K >> 8;
    for (int i0 = 0; i0 < n; i0 += 4) {
      uint4 xv[4], wv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u)
        if (i0 + u < n) {
          xv[u] = x4[(i0 + u) * 32];
          wv[u] = w4[(i0 + u) * 32];
        }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        if (i0 + u >= n) break;
        const uint32_t xa[4] = {xv[u].x, xv[u].y, xv[u].z, xv[u].w};
        const uint32_t wa[4] = {wv[u].x, wv[u].y, wv[u].z, wv[u].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 xf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&xa[e]));
          const float2 wf = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&wa[e]));
          s = fmaf(xf.x, wf.x, s);
          s = fmaf(xf.y, wf.y, s);
        }
      }
    }
  } else {
    for (int k = lane; k < d.K; k += 32) s = fmaf(to_f<T>(x[k]), to_f<T>(w[k]), s);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) d.logits[r] = s;
}

void launch_logit_dot(bool bf, const LogitDesc* descs, int n_problems, int max_rows,
                      const int* wsel, cudaStream_t st) {
  dim3 grid((max_rows + 7) / 8, n_problems);
  if (bf) launch_pdl(k_logit_dot<bf16>, grid, dim3(256), 0, st, descs, wsel);
  else launch_pdl(k_logit_dot<float>, grid, dim3(256), 0, st, descs, wsel);
}

// Logit deltas of cell c (rows: B real, B fake): the discriminator loss's dL/dlogit over the
// 2B rows, (sigmoid - 1) / B and sigmoid / B, and the generator loss's over the fake rows,
// (sigmoid - 1) / B; rounded to the population precision (they enter the output layer's
// products).
template <typename T>
__global__ void k_dc_dlogit(const float* __restrict__ logits, int B, T* __restrict__ dl_d,
                            T* __restrict__ dl_g) {
  pdl_wait();
  const int c = blockIdx.x;
  for (int r = threadIdx.x; r < 2 * B; r += blockDim.x) {
    const float l = logits[(int64_t)c * 2 * B + r];
    const float sg = 1.f / (1.f + expf(-l));
    dl_d[(int64_t)c * 2 * B + r] = from_f<T>((r < B ? sg - 1.f : sg) / (float)B);
    if (r >= B) dl_g[(int64_t)c * B + r - B] = from_f<T>((sg - 1.f) / (float)B);
  }
}

// Back through the output layer: da[r][k] = dl[r] w[k] (LeakyReLU derivative from a[r][k]) in
// the population precision; with dw, also dw[k] = sum_r dl[r] a[r][k] in row order.
template <typename T>
__global__ void k_logit_back(const LogitDesc* __restrict__ descs, int with_dw, float slope) {
  pdl_wait();
  const LogitDesc d = descs[blockIdx.y];
  const T* w = (const T*)d.w + (d.wsel ? (int64_t)d.wsel[d.wsel_idx] * d.wsel_stride : 0);
  const T* a = (const T*)d.a;
  const T* dl = (const T*)d.dl;
  T* da = (T*)d.da;
  if (sizeof(T) == 2 && (d.K & 1) == 0 && (((uintptr_t)a | (uintptr_t)da) & 3) == 0) {
    // bf16: two neighbouring k per thread (4-byte loads and stores), eight rows' loads issued
    // together; each k's sum still runs over the rows in order
    const int kh = d.K >> 1;
    for (int k2 = blockIdx.x * blockDim.x + threadIdx.x; k2 < kh; k2 += gridDim.x * blockDim.x) {
      const int k = 2 * k2;
      const float w0 = to_f<T>(w[k]), w1 = to_f<T>(w[k + 1]);
      float s0 = 0.f, s1 = 0.f;
      const __nv_bfloat162* a2 = reinterpret_cast<const __nv_bfloat162*>(a) + k2;
      __nv_bfloat162* da2 = reinterpret_cast<__nv_bfloat162*>(da) + k2;
      for (int r0 = 0; r0 < d.rows; r0 += 8) {
        float2 av[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          av[u] = r0 + u < d.rows ? __bfloat1622float2(a2[(int64_t)(r0 + u) * kh])
                                  : make_float2(0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          if (r0 + u >= d.rows) break;
          const float g = to_f<T>(dl[r0 + u]);
          s0 = fmaf(g, av[u].x, s0);
          s1 = fmaf(g, av[u].y, s1);
          if (da)
            da2[(int64_t)(r0 + u) * kh] =
                __floats2bfloat162_rn(av[u].x > 0.f ? g * w0 : slope * g * w0,
                                      av[u].y > 0.f ? g * w1 : slope * g * w1);
        }
      }
      if (with_dw) {
        d.dw[d.hwc_c ? (k % d.hwc_c) * 16 + k / d.hwc_c : k] = s0;
        d.dw[d.hwc_c ? ((k + 1) % d.hwc_c) * 16 + (k + 1) / d.hwc_c : k + 1] = s1;
      }
    }
    return;
  }
  for (int k = blockIdx.x * blockDim.x + threadIdx.x; k < d.K; k += gridDim.x * blockDim.x) {
    const float wk = to_f<T>(w[k]);
    float s = 0.f;
    for (int r = 0; r < d.rows; ++r) {
      const float g = to_f<T>(dl[r]);
      const float av = to_f<T>(a[(int64_t)r * d.K + k]);
      s = fmaf(g, av, s);
      if (da) da[(int64_t)r * d.K + k] = from_f<T>(av > 0.f ? g * wk : slope * g * wk);
    }
    if (with_dw) d.dw[d.hwc_c ? (k % d.hwc_c) * 16 + k / d.hwc_c : k] = s;
  }
}

void launch_dc_dlogit(bool bf, const float* logits, int cells, int B, void* dl_d, void* dl_g,
                      cudaStream_t st) {
  if (bf)
    launch_pdl(k_dc_dlogit<bf16>, dim3(cells), dim3(256), 0, st, logits, B, (bf16*)dl_d,
               (bf16*)dl_g);
  else
    launch_pdl(k_dc_dlogit<float>, dim3(cells), dim3(256), 0, st, logits, B, (float*)dl_d,
               (float*)dl_g);
}

void launch_logit_back(bool bf, const LogitDesc* descs, int n_problems, int K, bool with_dw,
                       float slope, cudaStream_t st) {
  dim3 grid((K + 255) / 256, n_problems);
  if (bf) launch_pdl(k_logit_back<bf16>, grid, dim3(256), 0, st, descs, with_dw ? 1 : 0, slope);
  else launch_pdl(k_logit_back<float>, grid, dim3(256), 0, st, descs, with_dw ? 1 : 0, slope);
}

}  // namespace lipz
