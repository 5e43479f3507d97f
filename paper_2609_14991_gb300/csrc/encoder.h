// Internal declarations of the cache-aware encoder (see tsd.h for the
// computation and encoder.cu for the driver).
#pragma once

#include <cuda.h>

#include <map>
#include <utility>
#include <vector>

#include "internal.h"

namespace tsd {

// Epilogues of the encoder's tensor-core GEMM, out = A . B^T (+ bias):
enum EncEpilogue {
  kEInit = 0,   // x[r][c]  = acc + bias                (fp32 residual stream)
  kEResid = 1,  // x[r][c] += alpha (acc + bias)        (fp32 residual stream)
  kESwish = 2,  // y[r][c]  = bf16(Swish(acc + bias))
  kEPlain = 3,  // y[r][c]  = bf16(acc + bias)
  kEGlu = 4,    // y[r][j]  = bf16((a + b_a) sigmoid(g + b_g)); B rows interleaved in 32-row
                //            groups (value rows j, then their gate rows), N = 2 outputs
};

struct EGemm {
  int M, N, K;        // output rows, B rows (GLU: twice the outputs), inner size (multiple of 64)
  const float* bias;  // [N], in B's row order
  void* out;          // kEInit / kEResid: float [rows][ld]; otherwise bf16 [rows][ld]
  int ld;             // output row stride (elements)
  float alpha;        // kEResid
  unsigned int* err;  // device status word
  int m0;             // first output row (rows m0 .. m0+M-1 of A and out; tiles past m0+M
                      // may read further rows of A, but write nothing there)
};

constexpr int kEgBN = 128;  // output-tile width (B rows per tile)
constexpr int kEncBranches = 2;  // most parallel branches of the encoder's chunk graph

bool egemm_map_a(CUtensorMap* m, const uint16_t* A, int rows, int K);
bool egemm_map_b(CUtensorMap* m, const uint16_t* B, int rows, int K);
cudaError_t egemm_prepare();
void launch_egemm(int epi, const EGemm& g, const CUtensorMap& a, const CUtensorMap& b, cudaStream_t s);

// Device pointers of one block's weights (B operands repacked where noted).
struct EncLayerDev {
  const float *ln_ff1_g, *ln_ff1_b, *ln_att_g, *ln_att_b, *ln_conv_g, *ln_conv_b, *ln_ff2_g, *ln_ff2_b,
      *ln_out_g, *ln_out_b;
  uint16_t *ff1_w1, *ff1_w2, *qkv_w, *pos_w, *out_w, *pw1_w /*GLU-interleaved*/, *pw2_w, *ff2_w1, *ff2_w2;
  float *ff1_b1, *ff1_b2, *qkv_b, *pos_u, *pos_v, *out_b, *pw1_b /*interleaved*/, *dw_w, *dw_b, *bn_scale,
      *bn_shift, *pw2_b, *ff2_b1, *ff2_b2;
  uint16_t* pos_tab;  // [n_off][d] bf16: W_pos r(delta) for delta = -(max_chunk-1) .. left+max_chunk-1
  CUtensorMap m_ff1_w1, m_ff1_w2, m_qkv, m_out, m_pw1, m_pw2, m_ff2_w1, m_ff2_w2;
};

}  // namespace tsd

struct tsd_encoder {
  tsd_encoder_cfg cfg{};
  int device = 0;
  tsd::DevArena arena;
  int n_off = 0;  // rows of each position table
  int M_pad = 0;  // work-buffer rows (max_streams * max_chunk, padded to 128)
  uint16_t* sub_w = nullptr;
  float* sub_b = nullptr;
  CUtensorMap m_sub{};
  std::vector<tsd::EncLayerDev> L;
  // work buffers
  uint16_t *feat = nullptr, *nrm = nullptr, *hid = nullptr, *qkv = nullptr, *att = nullptr, *glu = nullptr,
           *convz = nullptr, *outb = nullptr;
  float* x = nullptr;
  CUtensorMap m_feat{}, m_nrm{}, m_hid{}, m_att{}, m_convz{};
  // per-slot state
  uint16_t *kc = nullptr, *vc = nullptr, *cc = nullptr;  // [slot][layer][head][left][dh] x2, [slot][layer][K-1][d]
  int32_t* seen = nullptr;
  int32_t* slots_dev = nullptr;
  unsigned int* err = nullptr;
  std::vector<uint8_t> slot_open;
  int32_t* slots_host = nullptr;  // pinned staging for the slot list
  cudaEvent_t slots_ev = nullptr;
  cudaStream_t last_stream = nullptr, cap_stream = nullptr;
  // further branches of a captured chunk step, their fork and joins
  cudaStream_t branch[tsd::kEncBranches - 1] = {};
  cudaEvent_t fork_ev = nullptr, join_ev[tsd::kEncBranches - 1] = {};
  // captured graphs per (n, C, timing)
  struct Graph {
    cudaGraphExec_t exec = nullptr;
    std::vector<cudaEvent_t> ev;
    std::vector<int8_t> cls;
    bool pending = false;
  };
  std::map<std::pair<std::pair<int, int>, int>, Graph> graphs;
  int timing = 0;
  double ms[3] = {0, 0, 0};
  int64_t launches[3] = {0, 0, 0};

  // releases everything the encoder holds (also after a failed create)
  ~tsd_encoder() {
    for (auto& kv : graphs) {
      if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
      for (cudaEvent_t ev : kv.second.ev) cudaEventDestroy(ev);
    }
    if (slots_host) cudaFreeHost(slots_host);
    if (slots_ev) cudaEventDestroy(slots_ev);
    if (cap_stream) cudaStreamDestroy(cap_stream);
    for (int i = 0; i < tsd::kEncBranches - 1; ++i) {
      if (branch[i]) cudaStreamDestroy(branch[i]);
      if (join_ev[i]) cudaEventDestroy(join_ev[i]);
    }
    if (fork_ev) cudaEventDestroy(fork_ev);
    arena.release();
    cudaGetLastError();
  }
};
