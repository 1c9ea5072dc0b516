// Tensor-core (tcgen05 / TMEM / TMA) forward of the evaluation phase, bf16 operands with fp32
// accumulation: every generator slot's fakes and every discriminator slot's logits of every
// cell, for the MLP shapes it supports.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>
#include <vector>

namespace lipz {

struct TcShape {
  int cells, B, z, h, x;
  float slope;
  int n_indiv;  // individuals the weight maps span (both snapshots: 2 * cells)
};

struct TcPlan;

// hidden == 256, z and x multiples of 16, 16 <= z <= 256, 16 <= x, batch >= 1.
bool tc_supported(int z, int h, int x, int B);

// Device buffers of one population snapshot that the tensor-core forward reads and writes.
//   Z: [cells][B][z] bf16; E: [cells][6B][x] bf16 (rows [0, B) real, then the fakes of slots
//   0..4, which the generator kernel writes); logits [cells][5][6B] fp32; nbr [cells][5]
//   (individual indices). Weights: bf16 copies (Gwb, Dwb) and fp32 masters (biases) of both
//   snapshots, individual k = snapshot * cells + cell, per-individual strides PGs / PDs,
//   tensor offsets goff / doff (W1, b1, W2, b2, W3, b3).
//   Training forward of the selected pairs: the discriminator reads E[c] rows [0, B) and the
//   fakes of slot sel_g[c] in place, src_g / src_d [cells] (selected individuals), outputs
//   TH1, TH2 [cells][B][256], TG1, TG2 [cells][2B][256] bf16 and TL [cells][2B] fp32.
struct TcBuffers {
  void* Z;
  void* E;
  int64_t e_cell;
  float* logits;
  const int* nbr;
  const __nv_bfloat16* Gwb;
  const float* Gw;
  int64_t PGs;
  const int64_t* goff;
  const __nv_bfloat16* Dwb;
  const float* Dw;
  int64_t PDs;
  const int64_t* doff;
  // mixture score: squared norms of E's rows [cells][6B] fp32 (input) and the Gram kernel's
  // per-row block sums [cells][6B][tc_gram_halves(B)][6] fp32 (output); null without mixture
  const float* rnorm;
  float* gram_out;
  int indiv_off;     // individual index of this snapshot's cell 0 (snapshot * cells)
  const int* sel_g;  // slot of each cell's selected generator (training: its fakes in E)
  const int* src_g;
  const int* src_d;
  void *TH1, *TH2, *TG1, *TG2;
  float* TL;
};

// Builds the TMA descriptors and launch parameters for one population snapshot. Returns null
// and a message on failure.
TcPlan* tc_plan_create(const TcShape& s, const TcBuffers& b, std::string* msg);

// Enqueue the generator kernel (fakes of every (cell, slot)) / the discriminator kernel (logits
// of every (cell, slot)) on `st`. 0 on success.
int tc_run_g(TcPlan* p, cudaStream_t st, std::string* msg);
// Work lists of the CTA-pair evaluation kernels for one neighbour table (device arrays built
// by tc_build_pairs): generator pairs g[ng], discriminator pairs d[nd], and the (cell, slot)
// problems of every individual (plist) they index.
struct TcPairs {
  const int4* g;
  int ng;
  const int4* d;
  int nd;
  const int2* plist;
};
// Host side of TcPairs for the neighbour table nbr [cells][5] (individual indices < n_indiv):
// per individual its problems in table order; generator pairs {individual, first row of the
// pair's 256, plist offset, rows = problems x B}; discriminator pairs {individual, problem of
// the first CTA, problem of the second (-1: none), first rows packed (first << 16 | second)}.
void tc_build_pairs(const int* nbr, int cells, int n_indiv, int B, std::vector<int4>* gpairs,
                    std::vector<int4>* dpairs, std::vector<int2>* plist);
// Neighbour table [cells][5] (individual indices) that the next evaluation runs read, and its
// pair lists (null: the one-CTA kernels run).
void tc_set_nbr(TcPlan* p, const int* nbr, const TcPairs* pairs);
// Generator forward of every cell's own centre on its z, into E's slot-0 fakes.
int tc_run_g_centre(TcPlan* p, cudaStream_t st, std::string* msg);
int tc_run_d(TcPlan* p, cudaStream_t st, std::string* msg);
// Mixture score: for every cell c and row r of E[c], the sums over each block b of B columns
// s of exp(-||E[c][r] - E[c][s]||^2 / x), into gram_out[c][r][h][b] split over the
// tc_gram_halves(B) column ranges h (32 <= B <= 250, i.e. tc_gram_supported).
int tc_run_gram(TcPlan* p, cudaStream_t st, std::string* msg);
int tc_gram_halves(int B);
bool tc_gram_supported(int B);
// Training forward of every cell's selected generator (hidden activations into TH1, TH2) and
// selected discriminator (TG1, TG2 and the logits TL).
int tc_run_train_g(TcPlan* p, cudaStream_t st, std::string* msg);
int tc_run_train_d(TcPlan* p, cudaStream_t st, std::string* msg);

// Device int that a kernel of the plan sets to a non-zero code when one of its bounded waits
// expired (the kernel then stopped early); the host reads and clears it.
int* tc_error_flag(TcPlan* p);

void tc_plan_destroy(TcPlan* p);

}  // namespace lipz
