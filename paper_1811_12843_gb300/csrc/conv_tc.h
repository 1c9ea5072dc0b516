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
  int wsel_idx;
  int pad;
};

// A launch: problems of `rows` images; 4x4 / stride 2 / pad 1 convolution from ci x 2^lhi
// squared to co x 2^lho squared; K = 16 ci in (ky, kx, ci) order, kchunks = ceil(K / 64);
// jobs of nbox = min(co, 256) output channels (nj of them); tiles of 128 output pixels
// (mtiles per problem). The weight map spans [individual][co][K] bf16.
struct CtcParams {
  const ConvTcDesc* descs;
  int rows, ci, lhi, co, lho, nchw_in, kchunks, nj, nbox, mtiles, n_tiles;
  const int* wsel;
  float slope;
  int* err;
};

// Offsets and input channels of the five discriminator tensors inside one individual (P its
// parameter count): [out][in][ky][kx] -> [out][ky][kx][in].
struct RelayoutD {
  int64_t off[6];
  int ci[5];
  int64_t P;
};

bool ctc_make_map(CUtensorMap* m, const void* base, uint64_t K, uint64_t rows, uint64_t depth,
                  uint64_t depth_elems, uint32_t box_rows, std::string* msg);
bool ctc_prepare(std::string* msg);
void launch_conv_tc(const CUtensorMap& mW, const CtcParams& p, int sms, cudaStream_t st);
void launch_relayout_d(const bf16* src, bf16* dst, int n_indiv, int64_t Ps, const RelayoutD& r,
                       cudaStream_t st);

}  // namespace lipz
