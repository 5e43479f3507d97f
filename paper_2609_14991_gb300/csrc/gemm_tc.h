// Tensor-core GEMMs of the stateful Transducer form; see gemm_tc.cu.
#pragma once

#include <cuda.h>

#include "decoder.h"

namespace tsd {

enum GemmEpilogue { kEncProj = 0, kLstm = 1, kJointIn = 2 };

struct GemmArgs {
  int M;              // rows of A (and of the output) this launch covers
  int N;              // output columns (a multiple of 32; B's rows are padded to a multiple of 128)
  int K;              // inner size, a multiple of 64
  int ld;             // kEncProj: output row stride; kJointIn: P_enc row stride (floats)
  const float* bias;  // [N]
  float* out;         // kEncProj: [M][ld]
};

// TMA maps of a K-major bf16 operand: A (128-row boxes) and B (boxes of the
// epilogue's output-tile width; B's rows are padded to a multiple of 128).
bool gemm_tc_map_a(CUtensorMap* m, const uint16_t* A, int rows, int K);
bool gemm_tc_map_b(CUtensorMap* m, int epi, const uint16_t* B, int rows, int K);
cudaError_t gemm_tc_prepare();
void launch_gemm_tc(int epi, const DecView& d, const GemmArgs& g, const CUtensorMap& a, const CUtensorMap& b,
                    cudaStream_t s, bool pdl);

}  // namespace tsd
