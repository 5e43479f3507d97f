// Tensor-core joint GEMM (tcgen05 + TMA + TMEM) with the fused selection
// epilogue; see joint_tc.cu.
#pragma once

#include <cuda.h>

#include "decoder.h"

namespace tsd {

struct JointTc {
  CUtensorMap mapA;  // joint input A [M_pad][H], 128 x 64 boxes
  CUtensorMap mapB;  // W_out label-major [N_pad][H], bn x 64 boxes
  CUtensorMap mapBias;  // fusion bias fp32 [M_pad][N_pad], 32 x 128 boxes
  CUtensorMap mapLogits;  // logits fp32 [M_pad][N_pad], 32 x 32 boxes (the streaming epilogue's stores)
  int bn = 256;      // labels per CTA tile (one selection partial each)
};

// Tile width for a row count: the widest whose tile count still fills the SMs.
int joint_tc_pick_bn(int M_max, int N_pad, int sms);
cudaError_t joint_tc_prepare(JointTc* jt, const uint16_t* A, int M_pad, const uint16_t* Wt, int N_pad, int H, int bn,
                             const float* bias, const float* logits);
void launch_joint_tc(const JointTc& jt, const DecView& d, int M, int step, cudaStream_t s, bool pdl);
// Greedy decoding with at most one LM (dense or streaming epilogue): joint_greedy.cu.
cudaError_t joint_greedy_prepare(int bn);
void launch_joint_greedy(const JointTc& jt, const DecView& d, int M, int step, cudaStream_t s, bool pdl);
// The default limit of a bounded wait (1 s).
unsigned long long tc_wait_ns_default();

}  // namespace tsd
