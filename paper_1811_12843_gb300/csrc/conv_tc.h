// Tensor-core implicit-GEMM convolution (conv_tc.cu) of the DCGAN discriminator's evaluation
// and the weight re-layout it reads.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "engine.h"

namespace lipz {

// One problem of a launch: input activations (channel-last [n][H][W][ci], or for the first
// layer the channel-major images [n][3][64][64] of the evaluation buffer), output channel-last
// [n][Ho][Wo][co], and the index of its individual in the launch's table.
struct ConvTcDesc {
  const bf16* in;
  bf16* out;
  const bf16* aux;  // CTC_DLRELU_HWC / CTC_DTANH_CHW: the activation whose derivative applies
  int wsel_idx;
  int pad;
  float* logits;  // CTC_LRELU_LOGIT: one logit per image
};

// A launch: problems of `rows` images; 4x4 / stride 2 / pad 1 convolution from ci x 2^lhi
// squared to co x 2^lho squared; K = 16 ci in (ky, kx, ci) order (the 3-channel first layer:
// (ci, ky, kx)), kchunks = ceil(K / 64);
// jobs of nbox = min(co, 256) output channels (nj of them); tiles of 128 output pixels
// (mtiles per problem). The weight map spans [individual][co][K] bf16. nchw_in: the first
// layer, which takes only 3-channel channel-major 64 x 64 images (ci 3, lhi 6, lho 5).
// transposed: a stride-2 / pad-1 transposed convolution computed by output parity class (tiles
// over problem x 4 classes x mtiles; K = 4 ci in (tap, ci) order; the weights of class cls
// start at row cls * cls_rows of the map). out_mode: CTC_LRELU_HWC (bf16 LeakyReLU,
// channel-last), CTC_F32_HWC (fp32 raw, channel-last), CTC_TANH_CHW (bf16 tanh, channel-major
// images; co <= 16).
// CTC_DLRELU_HWC: bf16 delta times the LeakyReLU derivative at aux (channel-last);
// CTC_DTANH_CHW: bf16 delta times 1 - aux^2 (aux the tanh output), channel-major images.
// CTC_LRELU_LOGIT: LeakyReLU as CTC_LRELU_HWC, then the 4 x 4 output layer in the epilogue
// (4 x 4 outputs; logit_w / logit_ws the output layer's [16 pixels][co] weights of each
// individual): one logit per image into the descriptor's logits, the activations not stored.
enum { CTC_LRELU_HWC = 0, CTC_F32_HWC = 1, CTC_TANH_CHW = 2, CTC_DLRELU_HWC = 3,
       CTC_DTANH_CHW = 4, CTC_LRELU_LOGIT = 5 };
struct CtcParams {
  const ConvTcDesc* descs;
  int rows, ci, lhi, co, lho, nchw_in, kchunks, nj, nbox, mtiles, n_tiles;
  int transposed, out_mode, cls_rows;
  int a_tma;  // A rows by TMA through the activation map (set by ctc_make_act_map)
  // scatter: a stride-2 transposed convolution to 3 channels (CTC_TANH_CHW / CTC_DTANH_CHW,
  // ci 64, 32 x 32 -> 64 x 64) as one GEMM over input pixels (N = 16 taps x 4, weights from
  // launch_relayout_s), each tile of 4 input rows adding its taps into an output window in
  // shared memory in a fixed order; the rows it shares with the next tile go to halo
  // (problems x rows x 8 x 768 floats) and launch_scatter_fix completes them
  int scatter;
  float* halo;
  // m2: 256-row tiles (set by ctc_make_act_map for channel-last outputs with nbox <= 128): two
  // 128-row A boxes and two accumulators (columns h * nbox) share each weight chunk
  int m2;
  const bf16* logit_w;  // CTC_LRELU_LOGIT
  int64_t logit_ws;
  // first layer, CTC_LRELU_HWC, 64 output channels: the output tiles go out by TMA through
  // the map that ctc_make_out_map builds (passed in place of the activation map)
  int tma_out;
  const int* wsel;
  float slope;
  int* err;
  // CTC_F32_HWC: non-null = also the batch-norm statistics of the output: per (tile, 128-row
  // half, TMEM lane quarter) slot the per-channel sum and sum of squares over its valid rows,
  // bn_part[slot][co] (slot = (tile * (m2 ? 2 : 1) + half) * 4 + quarter), for
  // launch_bn_relu_hwc_part
  float2* bn_part;
};

// Generator layers 2..5 (n of them): source offsets and sizes [in = ci][out = co][4][4];
// destination offsets (per individual, stride dst_ps) of the class-major copies with
// cls_rows rows per class.
struct RelayoutG {
  int n;
  int64_t src_off[4], dst_off[4];
  int ci[4], co[4], cls_rows[4];
};

// Offsets and input channels of the five discriminator tensors inside one individual (P its
// parameter count): [out][in][ky][kx] -> [out][ky][kx][in] for all but the first (3-channel)
// layer, whose convolution reads its weights in their own order (K = (in, ky, kx)) from the
// population itself.
struct RelayoutD {
  int64_t off[6];
  int ci[5];
  int64_t P;
};

// Weight gradients on tcgen05: per problem a = [rows][2^la][2^la][M] and b = the gathered
// operand [rows][2^lb][2^lb][Cb] (both channel-last, M a multiple of 128, Cb of 64, N = 16 Cb
// a multiple of 256; or, with b_chw, b = [rows][3][2^lb][2^lb] channel-major, Cb 3, N 64, M a
// multiple of 64); dw = the problem's [M][Cb][4][4] fp32 gradient. b's pixel for tap
// (ky, kx) of a's pixel (y, x) is (s y - p + ky, s x - p + kx). part holds
// n_probs x splits x M x N floats; split s covers a's pixels [s kc, (s + 1) kc) of each problem
// (kc a multiple of 64, every split non-empty).
struct WgtcDesc {
  const bf16* a;
  const bf16* b;
  float* dw;
};
struct WgtcParams {
  const WgtcDesc* descs;
  int n_probs, rows, M, N, Cb, la, lb, s, p, splits, n_tiles;
  int64_t kc;
  int b_chw;  // b is 3 channel-major channels (Cb 3, N 64 with 48 used, M a multiple of 64)
  int a_tma;  // operands by TMA through the maps of wgtc_make_maps (set there; with b_chw A only)
  float* part;
  int* err;
};
bool wgtc_prepare(std::string* msg);
// Maps of a weight-gradient launch whose problems' a (and, without b_chw, b) sit at uniform
// strides: sets q->a_tma = 1 when they apply (else the gather warps load both operands; with
// b_chw, a_tma loads A by TMA and builds B from staged patches, for 32 x 32 A images over
// 64 x 64 b images only); false only when the driver refuses a map.
bool wgtc_make_maps(CUtensorMap* mA, CUtensorMap* mB, WgtcParams* q, const WgtcDesc* descs,
                    int n_probs, std::string* msg);
void launch_wgrad_tc(const CUtensorMap& mA, const CUtensorMap& mB, const WgtcParams& p, int sms,
                     cudaStream_t st);

bool ctc_make_map(CUtensorMap* m, const void* base, uint64_t K, uint64_t rows, uint64_t depth,
                  uint64_t depth_elems, uint32_t box_rows, std::string* msg);
// Activation map of a launch whose problems' channel-last inputs (ci a multiple of 64) sit at
// a uniform stride from descs[0].in: dims (ci, W, W, rows, problems), a box of 64 channels by
// the input pixels of 128 output pixels (traversal stride 2 for the convolution, 1 for the
// parity classes). Sets q->a_tma = 1 when it applies (else 0, and the gather warps load A;
// use_tma = false forces that), and then q->m2 and the 256-row tile count where they apply;
// q->mtiles and q->n_tiles must count 128-row tiles on entry. False only when the driver
// refuses the map.
bool ctc_make_act_map(CUtensorMap* m, CtcParams* q, const ConvTcDesc* descs, int n_probs,
                      std::string* msg, bool use_tma = true);
// Output map of a first-layer launch (nchw_in, CTC_LRELU_HWC, co 64) whose problems' outputs
// sit at a uniform stride from descs[0].out: dims (64 channels, output pixels, problems), boxes
// of 128 pixels in the 128-byte swizzle. Sets q->tma_out = 1 when it applies (else 0); false
// only when the driver refuses the map.
bool ctc_make_out_map(CUtensorMap* m, CtcParams* q, const ConvTcDesc* descs, int n_probs,
                      std::string* msg);
bool ctc_prepare(std::string* msg);
void launch_scatter_fix(const ConvTcDesc* descs, const float* halo, int n_problems, int rows,
                        int out_mode, cudaStream_t st);
// [individual][64 input channels][3][4][4] at src_off (stride src_ps) -> dst [individual][64
// rows tap * 4 + output][64], the scatter mode's weights.
void launch_relayout_s(const bf16* src, int64_t src_ps, int64_t src_off, bf16* dst, int n_indiv,
                       cudaStream_t st);
// False (and nothing launched) when no kernel variant serves p's A kind and out mode.
bool launch_conv_tc(const CUtensorMap& mW, const CUtensorMap& mA, const CtcParams& p, int sms,
                    cudaStream_t st);
void launch_relayout_d(const bf16* src, bf16* dst, int n_indiv, int64_t Ps, const RelayoutD& r,
                       cudaStream_t st);
void launch_relayout_g(const bf16* src, int64_t src_ps, bf16* dst, int64_t dst_ps, int n_indiv,
                       const RelayoutG& r, cudaStream_t st);
// [o][c][ky][kx] -> [o][ky][kx][c] for n weight tensors (o rows, c channels each) from
// src_off to dst_off of every individual; tensors of 3 channels are left out (the first-layer
// gather reads them in their own order).
struct RelayoutC {
  int n;
  int64_t src_off[4], dst_off[4];
  int o[4], c[4];
};
void launch_relayout_c(const bf16* src, int64_t src_ps, bf16* dst, int64_t dst_ps, int n_indiv,
                       const RelayoutC& r, cudaStream_t st);
// Batch normalisation (training mode) + ReLU on fp32 channel-last input into bf16 channel-last
// output (BnDesc: c, h, mean, inv, params; n images of 2^lhw pixels, C channels); part holds
// bn_hwc_part_floats(n_problems, channels) floats of per-chunk sums; counters holds
// bn_hwc_counters(n_problems, channels) zeroed unsigned ints (the launch leaves them zero);
// elems = the elements of one problem (images x pixels x channels).
void launch_bn_relu_hwc(const BnDesc* descs, int n_problems, int channels, const int* wsel,
                        float* part, unsigned* counters, int64_t elems, cudaStream_t st);
// The same from statistics that the producing convolution summed into part (bn_part, `slots`
// slots per problem, consecutive): a finalize launch, then the apply launch.
void launch_bn_relu_hwc_part(const BnDesc* descs, int n_problems, int channels, const int* wsel,
                             const float2* part, int slots, int64_t elems, cudaStream_t st);
// Backward of launch_bn_relu_hwc (BnDesc: c, h, mean, inv, params, dh fp32, dc bf16, dparams),
// with the same part and counters buffers; elems = the elements of one problem.
void launch_bn_relu_backward_hwc(const BnDesc* descs, int n_problems, int channels,
                                 float* part, unsigned* counters, int64_t elems, cudaStream_t st);
// The generator's first layer (a 4x4 transposed convolution of the 1x1 noise input) as the
// product y[n][(tap, o)] = sum_c z[n][c] W[c][o][tap] on tcgen05 (DENSE1 descriptors: a = noise
// rows [n][ca] bf16, 8-byte aligned; out = fp32 channel-last [n][16 co]; the individual from
// wsel_override or the descriptor's wsel). mW maps the [individual][16 co][128] copy of
// launch_relayout_g1 (ctc_make_map, K 128, box 256 rows). rows <= 128, ca <= 128 and a multiple
// of 4, 16 co a multiple of 256 (dense1_tc_supported). bn_part (nullable): the batch-norm sums
// of the output, [problem][16 taps][co] float2, for launch_bn_relu_hwc_part with 16 slots.
bool dense1_tc_supported(int rows, int ca, int co);
void launch_dense1_tc(const CUtensorMap& mW, const ConvDesc* descs, int n_problems,
                      const int* wsel_override, int rows, int ca, int co, int* err,
                      cudaStream_t st, float2* bn_part = nullptr);
// The generator's first-layer weight gradient on tcgen05 (the same shape conditions as
// dense1_tc_supported): dw (fp32 [ca][co][4][4] of each cell, stride dw_cell) = z^T dc1, with
// z the cells' noise rows [rows][ca] (stride z_cell) and dc1 the layer's batch-norm-backward
// deltas, channel-last [rows][16][co] (stride dc1_cell); dc1t is a [cells][rows][co][16]
// scratch that a re-layout launch fills first, and mB its map (dense1_wgrad_make_map).
bool dense1_wgrad_make_map(CUtensorMap* m, const bf16* dc1t, int rows, int co, int cells,
                           std::string* msg);
void launch_dense1_wgrad_tc(const CUtensorMap& mB, const bf16* z, int64_t z_cell,
                            const bf16* dc1, int64_t dc1_cell, bf16* dc1t, float* dw,
                            int64_t dw_cell, int rows, int ca, int co, int cells, int* err,
                            cudaStream_t st);
// [individual][ca][co][4][4] at src_off (stride src_ps) -> dst [individual][(tap, o)][128]
// (stride dst_ps), K padded with zeros.
void launch_relayout_g1(const bf16* src, int64_t src_ps, int64_t src_off, bf16* dst,
                        int64_t dst_ps, int ca, int co, int n_indiv, cudaStream_t st);
int64_t bn_hwc_part_floats(int n_problems, int channels);
int64_t bn_hwc_counters(int n_problems, int channels);

}  // namespace lipz
