// Internal interface between the host scheduler (api.cu) and the kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace lipz {

struct GemmDesc;
struct GemvDesc;
struct ColSumDesc;
typedef __nv_bfloat16 bf16;

// Flat parameter layout of one individual: tensor t occupies [off[t], off[t+1]). Its
// initialisation: init[t] = INIT_UNIFORM: U(-bound, bound) (Xavier; 0 when bound is 0),
// INIT_NORMAL: bound * N(0, 1), INIT_ONE_NORMAL: 1 + bound * N(0, 1).
enum { INIT_UNIFORM = 0, INIT_NORMAL = 1, INIT_ONE_NORMAL = 2 };
struct Layout {
  int n;
  int64_t off[17];
  float bound[16];
  int init[16];
};

// One population snapshot (all cells): fp32 master weights, Adam moments, bf16 copy (bf16
// mode, else null), per-individual step count and learning rate. Per-cell stride Ps elements.
struct PopView {
  float* w;
  float* m;
  float* v;
  bf16* wb;
  int* step;
  float* lr;
};

struct SelectParams {
  uint64_t seed;
  uint32_t t;
  int tournament_size;
  int replace_always;
  int lr_mutation;
  float lr_mut_std;
  uint64_t lr_mut_thr;  // mutate iff word < thr (= floor(prob * 2^32))
  float beta1, beta2;
};

// Where selection reads the old snapshot and writes its results; index 0 = generator, 1 =
// discriminator population.
struct SelectIO {
  const float* lr_old[2];
  const int* step_old[2];
  int* sel[2];
  int* src[2];
  float* lr_new[2];
  float4* coef[2];
};

void launch_init_params(float* w, bf16* wb, int64_t P, int64_t Ps, const Layout& lay, int cells,
                        uint64_t seed, uint32_t stream, cudaStream_t st);
void launch_to_bf16(const float* w, bf16* wb, int64_t n, cudaStream_t st);

// parts: DRAW_REAL (the B real rows into E[c]), DRAW_NOISE (z into Z[c]), or both; pdl = false
// keeps plain stream order (after an event wait).
enum { DRAW_REAL = 1, DRAW_NOISE = 2 };
template <typename T>
void launch_draw_batch(const T* pool, int64_t n_pool, const float* xin, T* E, int64_t e_cell,
                       T* Z, int cells, int B, int x_dim, int z_dim, uint64_t seed, uint32_t t,
                       uint32_t step, int parts, bool pdl, cudaStream_t st);

template <typename TI, typename TO, int EPI>
void launch_gemm(const GemmDesc* descs, int n_problems, int max_m, int max_n, int act,
                 float slope, cudaStream_t st);
template <typename T>
void launch_gemv(const GemvDesc* descs, int n_problems, int max_rows, cudaStream_t st);
template <typename T>
void launch_colsum(const ColSumDesc* descs, int n_problems, int max_cols, cudaStream_t st);

// device status words of one iteration (error flags of the kernels that can stop early, the
// non-finite-loss flag last), any of them null
struct StatusFlags {
  const int* p[8];
};
void launch_gather_status(const float* fG, const float* fD, int n, const StatusFlags& fl,
                          float* out, bool pdl, cudaStream_t st);
void launch_fitness(const float* logits, int cells, int B, float* LG, float* LD, float* fG,
                    float* fD, int* flag, cudaStream_t st);
// Also writes, per cell and population, the Adam coefficients of the new centre's next step:
// (lr, 1 / (1 - beta1^(step+1)), 1 / (1 - beta2^(step+1)), step + 1).
void launch_select(const float* fG, const float* fD, const int* nbr, int cells,
                   const SelectParams& p, const SelectIO& io, cudaStream_t st);
// ---- DCGAN (conv_kernels.cu) ---------------------------------------------------------------
// One grouped implicit-GEMM problem. CONV / CONVT forward: a = input [n][ca][2^lha][2^lwa],
// b = weights of individual 0 (+ wsel[wsel_idx] * wsel_stride; a launch may pass its own wsel
// table), out = [n][co][2^lho][2^lwo], aux = the activation whose derivative the epilogue
// applies (shaped like out). Weight gradient: a = [n][ca][2^lha][2^lwa], b = the gathered
// operand [n][co][2^lho][2^lwo], out = fp32 [ca][co * 16].
struct ConvDesc {
  const void* a;
  const void* b;
  const int* wsel;
  int64_t wsel_stride;
  int wsel_idx;
  void* out;
  const void* aux;
  int n, ca, lha, lwa, co, lho, lwo, s, p;
  int nhwc_out;  // CONV / CONVT: store (and read aux) channel-last [n][2^lho][2^lwo][co]
  int a_hwc;     // operand a is channel-last [n][2^lha][2^lwa][ca]
  int b_hwc;     // WGRAD: operand b is channel-last [n][2^lho][2^lwo][co]
};
// Training-mode batch normalisation + ReLU of one problem: c = fp32 conv output
// [n][C][2^lhw], h = activation out, mean / inv [C]; parameters (gamma at off_gamma, beta at
// off_beta) of individual wsel[wsel_idx] in params (fp32 masters, stride wsel_stride).
// Backward: dh = fp32 dL/dh, dc = dL/dc out, dparams = this cell's gradient vector.
struct BnDesc {
  const float* c;
  void* h;
  float* mean;
  float* inv;
  const float* params;
  const int* wsel;
  int64_t wsel_stride;
  int wsel_idx;
  int64_t off_gamma, off_beta;
  int n, C, lhw;
  const float* dh;
  void* dc;
  float* dparams;
  int hwc;  // c, h, dh, dc channel-last [n][2^lhw][C]
};
// Discriminator output layer: a [rows][K] activations, w the weights (individual 0 + wsel),
// logits [rows] out; backward: dl [rows] in, da [rows][K] out (or null), dw [K] out.
struct LogitDesc {
  const void* a;
  const void* w;
  const int* wsel;
  int64_t wsel_stride;
  int wsel_idx;
  float* logits;
  int rows, K;
  const void* dl;
  void* da;
  float* dw;
  int hwc_c;  // non-zero: a and w are in (tap, channel) order over hwc_c channels; dw is
              // written in the weights' (channel, tap) order
};
enum { CONV_FWD_MODE = 0, CONVT_FWD_MODE = 1, WGRAD_MODE = 2, CONVT2_MODE = 3,
       DENSE1_MODE = 4 };
enum { CEPI_NONE_ = 0, CEPI_LRELU_ = 1, CEPI_TANH_ = 2, CEPI_DLRELU_ = 3, CEPI_DTANH_ = 4 };
void launch_conv(int mode, int epi, bool bf, bool out_f32, const ConvDesc* descs,
                 int n_problems, int max_m, int max_n, const int* wsel, int splits, float* part,
                 int64_t part_stride, float slope, cudaStream_t st);
void launch_bn_relu(bool bf, const BnDesc* descs, int n_problems, int channels, const int* wsel,
                    cudaStream_t st);
void launch_bn_relu_backward(bool bf, const BnDesc* descs, int n_problems, int channels,
                             cudaStream_t st);
void launch_logit_dot(bool bf, const LogitDesc* descs, int n_problems, int max_rows,
                      const int* wsel, cudaStream_t st);
void launch_dc_dlogit(bool bf, const float* logits, int cells, int B, void* dl_d, void* dl_g,
                      cudaStream_t st);
void launch_logit_back(bool bf, const LogitDesc* descs, int n_problems, int K, bool with_dw,
                       float slope, cudaStream_t st);

// Generator-mixture score and ES-(1+1) step (rows = 6B evaluation rows per cell).
template <typename T>
void launch_row_norms(const T* E, int64_t e_cell, int cells, int rows, int x, float* out,
                      cudaStream_t st);
void launch_mix_partials(const float* gram, const float* rnorm, int cells, int rows, int B, int x,
                         float* out, cudaStream_t st);
void launch_mix_es(const float* part, int nh, int cells, int rows, int B, float* mix, float* S,
                   float* score, uint64_t seed, uint32_t t, float sigma, cudaStream_t st);
// Choice of every cell's own centre (slot 0), for the later minibatch steps of an iteration.
void launch_centre_select(int cells, int off, const SelectParams& p, const SelectIO& io,
                          cudaStream_t st);
// Fitness and, in the same kernel, the selection of every cell (when nothing is read back
// between the two).
void launch_fitness_select(const float* logits, int cells, int B, float* LG, float* LD,
                           float* fG, float* fD, int* flag, const int* nbr,
                           const SelectParams& p, const SelectIO& io, cudaStream_t st);
template <typename T>
void launch_train_prep(const T* E, int64_t e_cell, const int* sel_g, T* TX, int cells, int B,
                       int x_dim, cudaStream_t st);
template <typename T>
void launch_dlogit(const float* TL, const T* TG2, const T* wD, int64_t wD_stride, int64_t off_w3,
                   const int* src_d, int cells, int B, int H, float slope, T* J2, float* gD,
                   int64_t gD_stride, int64_t off_gw3, int64_t off_gb3, int64_t off_gb2,
                   cudaStream_t st);
void launch_adam(const PopView& old_p, const PopView& new_p, const float* grad, const int* src,
                 const float4* coef, int cells, int64_t P, int64_t Ps, float beta1, float beta2,
                 float eps, cudaStream_t st);

// Adam + replacement restricted to n parameter ranges [off[q], off[q] + len[q]) of every cell
// (applied by the tensor-core backward to each cell after its last tile).
struct AdamRanges {
  PopView old_p, new_p;
  const float* grad;
  const int* src;
  const float4* coef;
  int64_t Ps;
  int n;
  int64_t off[8];
  int len[8];
};


}  // namespace lipz
