// DCGAN networks of the grid (Table 1, CelebA column) on the CUDA-core kernels of
// conv_kernels.cu: the evaluation of every (cell, slot) pair and the training step of every
// cell's selected pair. The grid (api.cu) owns the populations, minibatches and selection; a
// plan owns its work buffers and the grouped-problem descriptors.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include "engine.h"

namespace lipz {

struct DcShape {
  int cells, B, z, ngf, ndf;
  bool bf;      // bf16 operands (population precision), else fp32
  float slope;  // LeakyReLU slope of the discriminator
  int n_indiv;  // individuals the population arrays hold (snapshots x cells)
};

// Populations: fp32 masters and the operand copies (bf16, or the fp32 masters) of every
// snapshot, individual k at k * PGs / k * PDs; tensor offsets of the layouts.
// Minibatch: Z [cells][B][z], E [cells][6B][3 * 64 * 64] (real rows, then the fakes of slots
// 0..4, which the evaluation writes); logits [cells][5][6B]. Training: src_g / src_d [cells]
// (selected individuals), gradients gG [cells][PGs], gD [cells][PDs] (fp32, every element
// written).
struct DcBuffers {
  const float* Gw;
  const void* Gop;
  const float* Dw;
  const void* Dop;
  int64_t PGs, PDs;
  const int64_t* goff;  // W1, gamma1, beta1, ..., W4, gamma4, beta4, W5 (13 tensors)
  const int64_t* doff;  // W1 .. W5
  const void* Z;
  void* E;
  int64_t e_cell;
  float* logits;
  const int* src_g;
  const int* src_d;
  float* gG;
  float* gD;
};

struct DcPlan;

// Generator / discriminator layouts in storage order (the oracle's): offsets of `n` tensors in
// lay (off[n] = parameter count) and their initialisation (N(0, 0.02^2) weights, batch-norm
// scales 1 + N(0, 0.02^2), shifts 0).
void dc_layouts(int z, int ngf, int ndf, Layout* lg, Layout* ld);

DcPlan* dc_plan_create(const DcShape& s, const DcBuffers& b, std::string* msg);
void dc_plan_destroy(DcPlan* p);

// Evaluation forward: every slot's generator on its cell's noise into E's fakes (dc_eval_g),
// then every slot's discriminator on E[c] into logits (dc_eval_d). nbr [cells][5]: individual
// of each slot.
// The individuals [lo, lo + n) whose weights the following evaluation / training reads (the
// per-iteration weight re-layouts cover only those); n <= 0: all of them.
void dc_set_indiv_range(DcPlan* p, int lo, int n);
int dc_eval_g(DcPlan* p, const int* nbr, cudaStream_t st, std::string* msg);
int dc_eval_d(DcPlan* p, const int* nbr, cudaStream_t st, std::string* msg);

// Forward and backward of every cell's selected pair (src_g, src_d) on the cell's minibatch
// (real rows of E, noise Z): the gradients into gG and gD.
int dc_train(DcPlan* p, cudaStream_t st, std::string* msg);

// Device int that a tensor-core kernel of the plan sets when one of its bounded waits expired
// (null without them); the host reads and clears it.
int* dc_error_flag(DcPlan* p);

// Kernel launches of dc_eval_g (part 0), dc_eval_d (part 1) and dc_train.
int dc_eval_launches(const DcPlan* p, int part);
int dc_train_launches(const DcPlan* p);

}  // namespace lipz
