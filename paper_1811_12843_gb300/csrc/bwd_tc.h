// Tensor-core backward of the training step: the chain of grouped products that turns the
// logit deltas of every cell's selected pair into weight gradients, bf16 operands with fp32
// accumulation.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "engine.h"

namespace lipz {

struct TcbShape {
  int cells, B, z, h, x;
  float slope;
  int n_indiv;  // individuals per population snapshot (= cells)
};

// Buffers (bf16 unless noted) of one population snapshot:
//   Z [cells][B][z]; E [cells][6B][x] (the discriminator's training input is E[c] rows
//   [0, B) and the fake rows of slot sel_g[c], read in place);
//   TH1, TH2 [cells][B][256] and TG1 [cells][2B][256]: stored forward activations;
//   J2 [cells][3B][256]: logit deltas through D's last layer (rows: real, fake for L_D, fake
//   for L_G); D1 [cells][3B][256], A3 [cells][B][x], A2, A1 [cells][B][256]: deltas written
//   here; gG, gD fp32 [cells][PGs / PDs]: weight gradients written here;
//   Gwb, Dwb: bf16 weight copies with tensor offsets goff / doff; src_g, src_d: the individual
//   each cell trains.
struct TcbBuffers {
  const void *Z, *TH1, *TH2, *TG1, *J2;
  const void* E;        // [cells][6B][x]: real rows, then the fakes of slots 0..4
  int64_t e_cell;
  const int* sel_g;     // slot of each cell's selected generator (its fakes in E)
  void *D1, *A3, *A2, *A1;
  float *gG, *gD;
  const __nv_bfloat16 *Gwb, *Dwb;
  int64_t PGs, PDs;
  const int64_t *goff, *doff;
  const int *src_g, *src_d;
  // fuse_adam != 0: the weight-gradient tiles apply Adam instead of storing the gradient (the
  // biases and D's output layer stay in gG / gD). Per population: the old snapshot (read at
  // src[cell]), the new one (written at the cell) and the per-cell coefficients.
  int fuse_adam;
  struct AdamPop {
    const float *w, *m, *v;
    float *w_new, *m_new, *v_new;
    __nv_bfloat16* wb_new;
    const float4* coef;
  } adam_g, adam_d;
  float beta1, beta2, eps;
  // with fuse_adam: the remaining ranges (biases, D's output layer) of G and D, [2]; each CTA
  // applies them to its cell after the cell's last tile
  const AdamRanges* ranges;
};

struct TcbPlan;

// hidden == 256, z == 64, x a multiple of 16, 1 <= batch <= 256.
bool tcb_supported(int z, int h, int x, int B);
TcbPlan* tcb_plan_create(const TcbShape& s, const TcbBuffers& b, std::string* msg);
// All nine products of every cell in one launch (one CTA per cell), as stages in the order
// 0 D1, 1 dW2(D), 2 A3, 3 dW1(D), 4 A2, 5 dW3(G), 6 A1, 7 dW2(G), 8 dW1(G).
int tcb_run_cells(TcbPlan* p, cudaStream_t st, std::string* msg);
int* tcb_error_flag(TcbPlan* p);
void tcb_plan_destroy(TcbPlan* p);

}  // namespace lipz
