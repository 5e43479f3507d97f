// Decoder internals shared by the host driver and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>

#include <map>
#include <tuple>

#include "internal.h"

namespace tsd {
struct JointTc;

// Per-call parameters, copied to the device before each chunk so that one
// captured graph serves every call of the same shape.
struct Params {
  const uint16_t* enc;  // [n][T][H] bf16
  int32_t* out_tok;     // [n][T*max_sym]
  int32_t* out_frame;
  float* out_score;
  int32_t* out_count;  // [n]
  int32_t n, T;
  float lambda, beta;
  int32_t slots[1];  // [n], the struct is allocated with room for max_streams
};

// Everything a kernel needs; passed by value.
struct DecView {
  int32_t V, N, N_pad, H, max_sym, K, n_ptiles, V4;
  const Params* params;
  const uint16_t* E;   // [N][H] bf16
  const uint16_t* Wt;  // [N_pad][H] bf16, label-major (rows >= N are zero)
  uint16_t* A;         // [M_pad][H] bf16, joint input of the current step
  float* bias;         // [M_pad][N_pad] fp32, lambda*LM + beta*boost of the current step
  float4* part;        // [M_pad][n_ptiles] (max logit, sum exp, best fused, best label)
  int32_t* r_t;        // [M_pad] frame
  int32_t* r_sym;      // [M_pad] labels emitted in this frame
  int32_t* r_cnt;      // [M_pad] labels emitted in this chunk
  // per-slot (x K hypotheses) persistent state
  int32_t* s_last;      // previous label (V = blank / start)
  int32_t* s_lm_len;    // [LMs][slots] LM chain length (order of the LM state)
  int32_t* s_lm_chain;  // [LMs][slots][kLmChain]
  int32_t* s_tr_len;
  int32_t* s_tr_chain;  // [.][kTrChain]
  // greedy: the table records of each chain element, kept with the chain so
  // the next step's searches start without fetching them:
  int4* s_lm_rec;       // [slots][kLmChain] first LM: (first arc, arcs, cumulative backoff bits, 0)
  int4* s_tr_rec;       // [slots][kTrChain] trie: (first child, children, depth of the children, 0)
  // stateful form (pred_D > 0): prediction network state and its buffers
  int32_t pred_D;       // LSTM width (0: the stateless joint input enc + E[last])
  uint16_t* pred_emb;   // [V+1][D] label embedding
  uint16_t* pred_h;     // [slots][D] LSTM output (bf16, as the products read it)
  float* pred_c;        // [slots][D] LSTM cell
  int32_t* pred_fresh;  // [slots] 1 until the start-of-sequence step has run
  uint16_t* pred_x;     // [M_pad][2D] LSTM input of the step: (embedding of the label, h)
  uint16_t* pred_hin;   // [M_pad][D] h after the step, input of the projection
  int32_t* pflag;       // [M_pad] 1 if the row's LSTM steps (a label was emitted, or the sequence starts)
  uint16_t* pred_enc;   // [rows][Henc] the chunk's encoder frames (a fixed address for TMA)
  float* pred_penc;     // [rows][H] W_enc enc + b_enc of the chunk
  LmView lm;
  TrieView tr;
  int32_t has_lm, has_tr;
  float* cap_logits;
  int32_t* cap_rows;
  int32_t cap_steps;
  // beam search (K > 1), per slot x K hypotheses
  float2* bpart;        // [M_pad][n_ptiles][1 + K]: (max, sum exp), then top-K (value, label)
  double* h_score;      // hypothesis score
  int32_t* h_live;      // 1 if the hypothesis slot holds a live hypothesis
  int32_t* h_node;      // label-sequence node (-1 = empty sequence)
  int32_t* h_len;       // label-sequence length
  unsigned long long* h_hash;  // rolling hash of the label sequence
  int32_t* pool_parent; // [slots][pool_cap] label-sequence nodes: parent node
  int32_t* pool_tok;    // [slots][pool_cap] label of the node
  int32_t* pool_n;      // [slots] nodes used
  int32_t pool_cap;
  // beam search with several labels per frame: the frame-exit set (same
  // layout as the hypotheses, [slots][K]) and each stream's frame and
  // expansion within it
  double* f_score;
  int32_t *f_live, *f_node, *f_len, *f_last, *f_lml, *f_trl;
  int32_t* f_lmc;       // [slots][K][kLmChain]
  int32_t* f_trc;       // [slots][K][kTrChain]
  unsigned long long* f_hash;
  int32_t* b_frame;     // [slots] frame of the chunk the beam is in (T: done)
  int32_t* b_exp;       // [slots] expansions taken in that frame
  int32_t topk;       // entries per row and tile in bpart: beam width, or prune_k
  int32_t prune;      // prune_k (0: fusion over every label)
  int32_t n_lm;       // n-gram LMs fused (0: none; several: greedy only)
  int32_t sms;        // SMs of the device (launch shapes)
  int32_t lm_stride;  // hypothesis slots per LM in s_lm_len / s_lm_chain
  LmView lmx[kMaxLm]; // every LM; lmx[0] equals lm
  float lm_w[kMaxLm]; // relative weights: LM i enters Eq. 1 with lambda * lm_w[i]
  float* dflt;        // [V4] per-call LM bias default lambda*log p(v) (0 past V)
  uint32_t* droot;    // [ceil(V4/32)] bit v: the trie root has a child labelled v
  // Greedy decoding with at most one LM (fused = 1).  Per row the joint
  // kernel's epilogue evaluates Eq. 1 for every label up to the row's
  // constant c_r, from the call's defaults dvec and the dense LM row of the
  // row's unigram state (LmView::dense0): F[v] = logit[v] + dvec[v] +
  // lambda * dense0[u][v].  The labels whose term differs from that (those
  // that a deeper LM state or a trie node below the root continues with, and
  // blank) are the row's correction list, written by the row pass before
  // the joint runs: the joint leaves them out of its per-tile best and
  // stores their raw logits; the next row pass evaluates them from the list.
  // fusion_path 0 (fz_dense = 0): the streaming form: the joint kernel
  // writes logit + dvec for every label and the row pass (row_stream.cu)
  // adds the row's LM and trie terms before it takes the argmax.
  int32_t fused;
  int32_t fz_dense;     // 1: the dense epilogue with the correction list; 0: streaming
  float* logits;        // [M_pad][N_pad] fp32: the listed labels' raw logits (dense) or every label's logit + dvec
  float* dvec;          // [N_pad] per call: lambda*log p(v) + beta*bonus*[the root has a child v]; 0 from V on
  int32_t* c_lab;       // [M_pad][V4] the row's listed labels
  float* c_add;         // [M_pad][V4] their term: F[v] = logit[v] + c_add
  int4* c_info;         // [M_pad] (dense row of the row's unigram state or -1, list length, c_r bits, -)
  uint32_t* c_mask;     // [M_pad][mask_words] bit v: label v is listed (blank always)
  int32_t mask_words;   // N_pad / 32
  // the row's copy of its stream's state within a chunk (previous label,
  // chain lengths, chains and records), so that a label step reads it by
  // row in one round
  int32_t* m_last;      // [M_pad]
  int32_t* m_lm_len;    // [M_pad]
  int32_t* m_tr_len;    // [M_pad]
  int32_t* m_lm;        // [M_pad][kLmChain]
  int4* m_lmr;          // [M_pad][kLmChain]
  int32_t* m_tr;        // [M_pad][kTrChain]
  int4* m_trr;          // [M_pad][kTrChain]
  int32_t* err;  // device status word: nonzero after a bounded wait expired
  // limit of the joint kernel's progress waits (a wait that drains copies or
  // MMAs still in flight before an early exit keeps the 1 s limit)
  unsigned long long wait_ns;
  unsigned long long* ctr;  // algorithmic bytes counted by row passes (replayed or timed)
  int32_t count;            // 1: every row pass adds its algorithmic bytes to *ctr
};

constexpr int kRowThreads = 256;

void launch_repack(const uint16_t* W, uint16_t* Wt, int H, int N, int N_pad, cudaStream_t s);
void launch_open(const DecView& d, int slot, cudaStream_t s);
void launch_fix_records(const DecView& d, int slot, cudaStream_t s);
void launch_open_pred(const DecView& d, int slot, cudaStream_t s);
void launch_copy_enc(const DecView& d, int64_t elems, cudaStream_t s, bool pdl);
void launch_row(const DecView& d, int M, int step, int mode, size_t smem, cudaStream_t s, bool pdl);
void launch_row_fused(const DecView& d, int M, int step, int mode, size_t smem, cudaStream_t s, bool pdl);
cudaError_t prepare_fused_kernels(size_t smem);
void launch_row_stream(const DecView& d, int M, int step, int mode, size_t smem, cudaStream_t s, bool pdl);
cudaError_t prepare_stream_kernels(size_t smem);
size_t row_stream_smem_bytes(int V4);
void launch_joint(const DecView& d, int M, int step, cudaStream_t s);
void launch_defaults(const DecView& d, cudaStream_t s);
size_t row_smem_bytes(int V4, int n_lm);
size_t row_fused_smem_bytes(int V4, int N_pad);
cudaError_t prepare_kernels(size_t row_smem);
void launch_row_beam(const DecView& d, int n, int step, int mode, size_t smem, cudaStream_t s, bool pdl);
void launch_row_pruned(const DecView& d, int M, int step, int mode, cudaStream_t s, bool pdl);
void launch_open_beam(const DecView& d, int slot, cudaStream_t s);
cudaError_t prepare_beam_kernels(size_t row_smem);
constexpr int kPoolCap = 8192;  // label-sequence nodes per beam stream

}  // namespace tsd

struct tsd_decoder {
  tsd_decoder_cfg cfg{};
  int device = 0;
  int N = 0, N_pad = 0, M_max = 0, M_pad = 0, n_ptiles = 0, V4 = 0;
  tsd::DevArena arena;
  const tsd_ngram* lm = nullptr;  // the first LM
  int n_lm = 0;
  const tsd_boost* boost = nullptr;
  tsd::DecView view{};
  tsd::Params* params_dev = nullptr;
  size_t params_bytes = 0;
  static constexpr int kRing = 4;
  char* staging[kRing] = {};
  cudaEvent_t staging_ev[kRing] = {};
  int ring_pos = 0;
  cudaStream_t cap_stream = nullptr;
  cudaStream_t last_stream = nullptr;
  std::vector<uint8_t> slot_open;
  int use_graphs = 1, timing = 0;
  size_t row_smem = 0;

  struct EventSet {
    std::vector<cudaEvent_t> ev;
    std::vector<int8_t> cls;  // class of the interval that starts at ev[i]
    cudaGraphExec_t exec = nullptr;
    bool pending = false;
  };
  struct Entry {
    EventSet set[2];
    int next = 0;
  };
  std::map<std::tuple<int, int, int, int>, Entry> entries;  // (n, T, graphs, timing)
  tsd::JointTc* jtc = nullptr;  // tensor-core joint kernel state
  // stateful form: repacked weights (K-major), biases and the GEMMs' TMA maps
  struct Pred {
    int D = 0, Henc = 0, G_pad = 0, H_pad = 0, MT_pad = 0;
    uint16_t *Wg = nullptr, *Wp = nullptr, *We = nullptr;
    float *bg = nullptr, *bp = nullptr, *be = nullptr;
    CUtensorMap encA, encB, lstmA, lstmB, projA, projB;
  } pred;
  int joint_kind = 0;           // 0 tensor cores, 1 CUDA cores
  int pdl = 1;                  // programmatic dependent launch between kernels
  int sms = 0;
  int last_n = 0, last_T = 0;   // shape of the last decode_chunk (for replay)
  // per-kernel-class device time of timed chunks: 0 row pass, 1 joint,
  // 2 prediction network and projections (stateful form)
  double ms[3] = {0, 0, 0};
  int64_t launches[3] = {0, 0, 0};
};
