// Internal declarations of the tsd library (not part of the C ABI).
#pragma once

#include <cuda_runtime.h>

#include <cstdint>
#include <string>
#include <vector>

#include "tsd.h"

namespace tsd {

// Longest LM order and phrase supported; they size the per-hypothesis chain
// buffers below.
constexpr int kMaxOrder = 16;
constexpr int kLmChain = 16;    // LM suffix chain: one state per order 1..order-1
constexpr int kMaxPhrase = 32;
constexpr int kTrChain = 32;    // trie suffix chain: nodes of depth >= 1, deepest first
constexpr int kPartialCols = 128;  // columns covered by one selection partial
constexpr int kNPad = 256;         // the vocabulary axis is padded to this multiple
constexpr int kMPad = 128;         // the row axis is padded to this multiple
constexpr int kMaxLm = 4;          // n-gram LMs fused at once (Eq. 1, sum over i)

// An NVTX range for the lifetime of the object (header-only NVTX 3: the
// calls do nothing unless a profiler is attached).
struct NvtxRange {
  explicit NvtxRange(const char* name);
  ~NvtxRange();
};

// Records a message for tsd_last_error() and returns st.
tsd_status fail(tsd_status st, const char* fmt, ...);
void clear_error();
tsd_status cuda_fail(cudaError_t e, const char* what);

#define TSD_CUDA(call)                                       \
  do {                                                       \
    cudaError_t _e = (call);                                 \
    if (_e != cudaSuccess) return ::tsd::cuda_fail(_e, #call); \
  } while (0)

// True if the test hook (tsd_debug_fail_alloc) makes this allocation fail.
bool alloc_hook_fires();

// Device allocations owned by one object; freed together.
struct DevArena {
  std::vector<void*> ptrs;
  int64_t bytes = 0;
  template <class T>
  tsd_status alloc(T** p, size_t count) {
    void* q = nullptr;
    size_t nb = sizeof(T) * (count ? count : 1);
    if (alloc_hook_fires()) return fail(TSD_ENOMEM, "cudaMalloc(%zu bytes) failed: injected by the test hook", nb);
    cudaError_t e = cudaMalloc(&q, nb);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(TSD_ENOMEM, "cudaMalloc(%zu bytes) failed: %s", nb, cudaGetErrorString(e));
    }
    ptrs.push_back(q);
    bytes += (int64_t)nb;
    *p = static_cast<T*>(q);
    return TSD_OK;
  }
  template <class T>
  tsd_status upload(T** p, const std::vector<T>& h) {
    tsd_status st = alloc(p, h.size());
    if (st) return st;
    if (!h.empty()) TSD_CUDA(cudaMemcpy(*p, h.data(), sizeof(T) * h.size(), cudaMemcpyHostToDevice));
    return TSD_OK;
  }
  void release() {
    for (void* q : ptrs) cudaFree(q);
    ptrs.clear();
    bytes = 0;
  }
};

// Device view of the n-gram tables.
//  State 0 is the empty context; states 1..V are the unigrams (state of
//  label v is 1+v); then every n-gram of orders 2..order-1, grouped by order.
//  The arcs of a state are its continuations (n-grams one order up), sorted
//  by label.  Arcs out of the empty context are the dense unigram arrays.
struct LmView {
  int32_t V = 0, order = 0;
  int64_t n_states = 0, n_arcs = 0;
  const int32_t* st_begin = nullptr;  // [S] first arc
  const int32_t* st_count = nullptr;  // [S] arcs
  const float* st_cum = nullptr;      // [S] sum of backoff weights over the state and its suffixes
  const int32_t* arc_tok = nullptr;   // [A] label
  const float* arc_logp = nullptr;    // [A] log p(label | state)
  const int32_t* arc_tgt = nullptr;   // [A] state of (state . label), -1 at the top order
  const float* uni_logp = nullptr;    // [V] log p(v)
  const int32_t* uni_tgt = nullptr;   // [V] state of the unigram v (0 if order == 1)
  // target records, so that finding a label's arc also yields the next
  // state's table record in the same load: (state, first arc, arcs,
  // cumulative backoff bits), state -1 at the top order
  const int4* arc_rec = nullptr;      // [A] record of arc_tgt
  // [V] the unigram state of v: (its dense row or -1, first arc, arcs,
  // cumulative backoff bits); the state id itself is 1 + v
  const int4* uni_rec = nullptr;
  // Every unigram state u (order >= 2, V x V4 floats at most 1 GiB) also
  // has a dense row: per label log p(v | u) - log p(v) - cum(u), 0 where u
  // has no arc v (the LM term of a label whose deepest arc is u's, relative
  // to lambda*log p(v) and the row's summed backoff).
  const float* dense0 = nullptr;      // [rows][V4]
  const int32_t* uni_dense = nullptr; // [V] dense row of the unigram state of v, or -1
  int32_t V4 = 0;                     // row stride of dense0
  int32_t n_dense = 0;                // rows of dense0
};

// Device view of the phrase trie.  Node 0 is the root.
struct TrieView {
  int32_t V = 0, n_nodes = 0, max_depth = 0, n_children = 0;
  float bonus = 0.f;
  const int32_t* nd_begin = nullptr;    // [Q] first child
  const int32_t* nd_count = nullptr;    // [Q] children
  const int32_t* nd_depth = nullptr;    // [Q]
  const int32_t* nd_fail = nullptr;     // [Q] failure link
  const int32_t* ch_tok = nullptr;      // [C] label (sorted within a node)
  const int32_t* ch_node = nullptr;     // [C] child node
  const int32_t* ch_next = nullptr;     // [C] node after the label: child, or 0 if it ends a phrase
  const int32_t* root_child = nullptr;  // [V] child of the root by label (0 = none)
  const int32_t* root_next = nullptr;   // [V] node after the label from the root
  // child records: (child node, node after the label, child's first child,
  // child's children); a root entry with child 0 means no child
  const int4* ch_rec = nullptr;         // [C]
  const int4* root_rec = nullptr;       // [V]
};

}  // namespace tsd

struct tsd_ngram {
  tsd::LmView view;
  tsd::DevArena arena;
  // host copies for state -> tuple queries
  std::vector<int32_t> st_parent, st_tok;
};

struct tsd_boost {
  tsd::TrieView view;
  tsd::DevArena arena;
  std::vector<int32_t> nd_parent, nd_tok;
};
