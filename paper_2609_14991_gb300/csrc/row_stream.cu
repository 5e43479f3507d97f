// Row pass of the fused decode step in its streaming form (greedy decoding,
// at most one n-gram LM, decoder option fusion_path 0): one CTA per
// hypothesis row.  The joint kernel before it wrote, for every label v of
// the row, logit[v] + D[v] with the call's shared defaults
// D[v] = lambda*log p(v) + beta*bonus*[the trie root has a child v] (0 for
// blank), and per-tile softmax partials of the raw logits; this pass finishes
// Eq. 1 for the row, takes the greedy decision and advances the state.
//
// Eq. 1 for label v < V at the row's state is
//   fused[v] = logit[v] - lse + lambda*log p_LM(v | h) + beta*bonus*(g(v) - depth)
// where the LM state is kept as its whole suffix chain (one state per order):
// log p_LM(v | h) is the arc v of the deepest chain state s_l that has one
// plus the backoff weights of the deeper states, or log p(v) plus all of
// them; g(v) is the depth of v's goto node from the deepest trie chain node
// with a child v (the trie chain holds every trie node that is a suffix of
// the current match), else [the root has a child v].  So
//   fused[v] + lse = (logit[v] + D[v]) + c_r + delta[v],
//   c_r = lambda*(summed backoff of the state) - beta*bonus*depth,
//   delta[v] = lambda*(log p(v | s_l) - summed backoff of s_l - log p(v))
//            + beta*bonus*(g(v) - [the root has a child v]),
// delta[v] = 0 for a label no chain element continues with.  For row r at
// label step s the pass
//   1. (before waiting for the joint kernel) loads the row's state and chains
//      (after the chunk's first step from the row's own copy, indexed by
//      row) and builds delta[v] in shared memory.  Level 0 (the previous
//      label's continuations, up to every label) is streamed once and writes
//      every label's level-0 delta (for a state with many continuations from
//      its dense row: per label log p(v | u) - log p(v) - cum_0, 0 for no
//      arc); meanwhile every arc of the levels above 0 (few: they continue
//      longer contexts) sets its level's bit in its label's level mask.  The
//      model is suffix-closed (a deeper level's labels are a subset of a
//      shallower one's), so a label's deepest level is its mask's highest bit,
//      and after a barrier that level's arc (held in registers) overwrites the
//      label's delta.  The trie chain nodes are scattered shallowest first
//      (the deepest overwrites);
//   2. (after the wait) the argmax of logit + D + c_r + delta over the labels
//      (blank: its logit alone; ties to the lowest label), i.e. the greedy
//      decision, and (for an emitted label) the log-sum-exp from the tile
//      partials for its fused score;
//   3. blank (or the per-frame label limit) advances the frame; a label y is
//      emitted and advances the chains, assembled from independent searches
//      of y in every chain element, each hit carrying the next state's table
//      record (first arc, arcs, summed backoff) in the same 16-byte load;
//   4. writes the joint input of step s, bf16(ReLU(enc_t + E[last])).
#include <algorithm>

#include "row_common.cuh"

namespace tsd {

namespace {

using row::best_merge;
using row::checked;
using row::kNegInf;
using row::lse_merge;

constexpr int kFzThreads = 128;  // 4 warps: seven CTAs per SM at 72 registers
constexpr int kStream = 4;       // level-0 arc groups of four per thread whose loads are issued together
constexpr int kDense = 8;        // dense level-0 quads per thread whose loads are issued together
constexpr int kFzWarps = kFzThreads / 32;

// Aligned groups of four arcs a chain level's arcs [b, b + c) span.
__device__ __forceinline__ int level_groups(int b, int c) { return c > 0 ? (b + c - (b & ~3) + 3) >> 2 : 0; }

// Position of y in the sorted arr[0, n), or -1, by one warp: 32-ary probes
// narrow the range to at most 124 entries, then one 16-byte load per lane
// covers them, from the 16-byte boundary at or below arr + lo.  A window so
// reads at most three entries before and after the range, inside the table
// (its label arrays start 16-byte aligned and are padded by four).  At most
// two dependent loads for n <= 3968.
__device__ __forceinline__ int warp_find_wide(const int32_t* __restrict__ arr, int n, int y, int lane) {
  row::reconverge();
  int lo = 0, hi = n;
  while (hi - lo > 124) {
    const int step = (hi - lo + 31) >> 5;
    const int idx = lo + lane * step;
    const int v = (idx < hi) ? __ldg(arr + idx) : INT_MAX;
    const unsigned m = __ballot_sync(0xffffffffu, v <= y);
    if (m == 0) return -1;
    lo = lo + (31 - __clz((int)m)) * step;
    hi = min(hi, lo + step);
  }
  const uintptr_t at = reinterpret_cast<uintptr_t>(arr + lo);
  const int4* g = reinterpret_cast<const int4*>(at & ~uintptr_t(15));
  const int first = 4 * lane - (int)((at & 15u) >> 2);  // this lane's first entry, relative to lo
  int pos = -1;
  if (first < hi - lo) {
    const int4 t = __ldg(g + lane);
    const int tv[4] = {t.x, t.y, t.z, t.w};
#pragma unroll
    for (int j = 3; j >= 0; --j)
      if (first + j >= 0 && first + j < hi - lo && tv[j] == y) pos = lo + first + j;
  }
  const unsigned m = __ballot_sync(0xffffffffu, pos >= 0);
  return m ? __shfl_sync(0xffffffffu, pos, __ffs((int)m) - 1) : -1;
}

// mode: 0 = label step, 1 = final step (apply the last decision only),
// 2 = replay (redo the step's work without committing any state or output;
// used only to time the kernel in isolation).
// VAR bit 0: the stateful form (LSTM input rows instead of the joint input);
// bit 2: few rows (at most two CTAs per SM are needed, registers are free).
template <int VAR>
__global__ void __launch_bounds__(kFzThreads) __maxnreg__((VAR & 4) ? 128 : 72) k_row_fz(DecView d, int step, int mode) {
  constexpr bool PRED = (VAR & 1) != 0;
  constexpr int QB = 8;     // label quads per thread whose loads are issued together
  constexpr int kHeld = 1;  // arc groups of four of the levels above 0 a thread keeps in registers
  const Params* __restrict__ P = d.params;
  const int r = blockIdx.x;
  const int V = d.V;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool commit = (mode != 2);
  const bool counting = (mode == 2 || d.count);
  extern __shared__ __align__(16) unsigned char smem[];
  // per label: its LM delta (0: none); the LM chain levels above 0 with an
  // arc for it (bit l); its trie goto depth (0: none)
  float* dlm = reinterpret_cast<float*>(smem);              // [V4]
  uint16_t* lev = reinterpret_cast<uint16_t*>(dlm + d.V4);  // [V4]
  uint8_t* dep = reinterpret_cast<uint8_t*>(lev + d.V4);    // [V4]

  __shared__ int s_t, s_sym, s_cnt, s_y, s_last, s_slot, s_T, s_n;
  __shared__ int s_nl, s_nt;
  __shared__ int32_t* s_out_tok;
  __shared__ int32_t* s_out_frame;
  __shared__ float* s_out_score;
  __shared__ int32_t* s_out_count;
  __shared__ const uint16_t* s_enc;
  __shared__ float s_lam, s_beta, s_score, s_lse;
  __shared__ int s_lm[kLmChain], s_tr[kTrChain];
  __shared__ int4 s_lmr[kLmChain];    // LM chain records: (first arc, arcs, summed backoff bits, -)
  __shared__ int4 s_trr[kTrChain];    // trie chain records: (first child, children, depth of the children, -)
  __shared__ int4 s_lm_hit[kLmChain]; // target record of y's arc at each old level (x = -2: none)
  __shared__ int4 s_tr_hit[kTrChain]; // child record of y at each old trie node (x = -1: none)
  __shared__ int4 s_uni_hit, s_root_hit;
  __shared__ float s_bv[kFzWarps];
  __shared__ int s_bi[kFzWarps];
  __shared__ unsigned long long s_bytes;  // algorithmic bytes of the row-step (when counting)
  __shared__ int s_bad;                   // TSD_CHECKS: a range check failed; the row stops

  // 1. Row state.  It was written by the previous row pass; under
  // programmatic launch this grid may start before its own wait, so these
  // loads go through L2 only (ld.global.cg), never a possibly stale L1 line.
  // After the chunk's first step the row's own copy of its state is read,
  // indexed by row, together with the slot (the chains are read whole: their
  // arrays have room for the longest).
  if (tid == 0) {
    const int slot = __ldcg(P->slots + r);
    s_slot = slot;
    s_T = __ldcg(&P->T);
    s_out_tok = P->out_tok;
    s_out_frame = P->out_frame;
    s_out_score = P->out_score;
    s_out_count = P->out_count;
    s_enc = P->enc;
    s_lam = P->lambda;
    s_beta = P->beta;
    s_n = P->n;
    s_bytes = 0;
    s_bad = !checked(slot >= 0 && slot < d.lm_stride, d.err, 1);
    if (step > 0) {
      s_t = __ldcg(d.r_t + r); s_sym = __ldcg(d.r_sym + r); s_cnt = __ldcg(d.r_cnt + r);
      s_nl = __ldcg(d.m_lm_len + r);
      s_nt = __ldcg(d.m_tr_len + r);
      s_last = __ldcg(d.m_last + r);
    }
  } else if (step > 0 && tid >= 32 && tid < 32 + kLmChain) {
    const int l = tid - 32;
    s_lm[l] = __ldcg(d.m_lm + (size_t)r * kLmChain + l);
    s_lmr[l] = __ldcg(d.m_lmr + (size_t)r * kLmChain + l);
  } else if (step > 0 && tid >= 64 && tid < 64 + kTrChain) {
    const int k = tid - 64;
    s_tr[k] = __ldcg(d.m_tr + (size_t)r * kTrChain + k);
    s_trr[k] = __ldcg(d.m_trr + (size_t)r * kTrChain + k);
  }
  {  // per-label scratch reset (the deltas are reset once the state is known)
    uint2* v4 = reinterpret_cast<uint2*>(lev);
    uint32_t* e4 = reinterpret_cast<uint32_t*>(dep);
    for (int q = tid; q < d.V4 / 4; q += blockDim.x) {
      v4[q] = make_uint2(0u, 0u);
      e4[q] = 0u;
    }
  }
  row::block_sync();
  if (s_bad) return;
  const int slot = s_slot, T = s_T;
  if (step == 0) {
    // the chunk's first step: the stream's state by slot, and the row's copy
    if (tid == 0) {
      s_t = 0; s_sym = 0; s_cnt = 0;
      s_nl = d.has_lm ? __ldcg(d.s_lm_len + slot) : 0;
      s_nt = d.has_tr ? __ldcg(d.s_tr_len + slot) : 0;
      s_last = __ldcg(d.s_last + slot);
      if (commit) {
        d.m_lm_len[r] = s_nl;
        d.m_tr_len[r] = s_nt;
        d.m_last[r] = s_last;
      }
    } else if (tid >= 32 && tid < 32 + kLmChain) {
      const int l = tid - 32;
      if (d.has_lm) {
        s_lm[l] = __ldcg(d.s_lm_chain + (size_t)slot * kLmChain + l);
        s_lmr[l] = __ldcg(d.s_lm_rec + (size_t)slot * kLmChain + l);
        if (commit) {
          d.m_lm[(size_t)r * kLmChain + l] = s_lm[l];
          d.m_lmr[(size_t)r * kLmChain + l] = s_lmr[l];
        }
      }
    } else if (tid >= 64 && tid < 64 + kTrChain) {
      const int k = tid - 64;
      if (d.has_tr) {
        s_tr[k] = __ldcg(d.s_tr_chain + slot * kTrChain + k);
        s_trr[k] = __ldcg(d.s_tr_rec + (size_t)slot * kTrChain + k);
        if (commit) {
          d.m_tr[(size_t)r * kTrChain + k] = s_tr[k];
          d.m_trr[(size_t)r * kTrChain + k] = s_trr[k];
        }
      }
    }
    row::block_sync();
  }
#ifdef TSD_CHECKS
  if (tid == 0) {  // every index the row will follow is inside its table
    bool ok = checked(s_nl >= 0 && s_nl <= kLmChain && s_nt >= 0 && s_nt <= kTrChain, d.err, 2) &&
              checked(s_last >= 0 && s_last <= V, d.err, 3);
    for (int l = 0; ok && l < s_nl; ++l) {
      const int4 c = s_lmr[l];
      ok = checked(s_lm[l] >= 0 && s_lm[l] < d.lm.n_states, d.err, 4) &&
           checked(c.x >= 0 && c.y >= 0 && (int64_t)c.x + c.y <= d.lm.n_arcs, d.err, 5) &&
           checked(l > 0 || (c.w >= -1 && c.w < d.lm.n_dense), d.err, 6);
    }
    for (int k = 0; ok && k < s_nt; ++k) {
      const int4 c = s_trr[k];
      ok = checked(s_tr[k] > 0 && s_tr[k] < d.tr.n_nodes, d.err, 7) &&
           checked(c.x >= 0 && c.y >= 0 && c.x + c.y <= d.tr.n_children && c.z >= 1 && c.z <= 63, d.err, 8);
    }
    s_bad = !ok;
  }
  row::block_sync();
  if (s_bad) return;
#endif
  // the encoder frames this step can use (t, or t+1 after a frame advance)
  // go to L1: no kernel of the chunk writes them
  if (!PRED && s_t < T) {
    const size_t fb = (size_t)d.H * 2;
    const uint16_t* f0 = s_enc + ((size_t)r * T + s_t) * d.H;
    row::prefetch_span(f0, s_t + 1 < T ? 2 * fb : fb, 0);
  }
  // In replay mode every row redoes a full step even if it had finished.
  const bool evaluated = (step > 0) && (s_t < T || !commit);
  const int nl_old = s_nl, nt_old = s_nt;
  const float lam = s_lam;
  const float bscale = s_beta * (d.has_tr ? d.tr.bonus : 0.f);

  if (evaluated) {
    const int4* t4 = reinterpret_cast<const int4*>(d.lm.arc_tok);
    const float4* p4 = reinterpret_cast<const float4*>(d.lm.arc_logp);
    // the aligned arc groups of the levels above 0, in level order: group g's
    // level and first arc (g below their count G)
    int G = 0;
    for (int l = 1; l < nl_old; ++l) G += level_groups(s_lmr[l].x, s_lmr[l].y);
    auto locate = [&](int g, int& l) {
      for (l = 1;; ++l) {
        const int n = level_groups(s_lmr[l].x, s_lmr[l].y);
        if (g < n) break;
        g -= n;
      }
      return (s_lmr[l].x & ~3) + 4 * g;
    };
    auto delta_of = [&](int l, float lp, int v) {
      return lam * (lp - __int_as_float(s_lmr[l].z)) - lam * __ldg(d.lm.uni_logp + v);
    };
    // 1a. the levels above 0 (few arcs: they continue longer contexts): each
    //     thread loads its first arc groups, labels and log-probabilities,
    //     and keeps them in registers
    int4 ht[kHeld];
    float4 hp[kHeld];
    int hl[kHeld], hi[kHeld];
#pragma unroll
    for (int u = 0; u < kHeld; ++u) {
      const int g = tid + u * kFzThreads;
      hl[u] = -1;
      hi[u] = 0;
      if (g < G) {
        int l;
        hi[u] = locate(g, l);
        ht[u] = __ldg(t4 + (hi[u] >> 2));
        hp[u] = __ldg(p4 + (hi[u] >> 2));
        hl[u] = l;
      }
    }
    // 1b. level 0 (the previous label's continuations, up to all V labels),
    //     streamed once: every label's level-0 delta (0 for no arc), which
    //     the deepest level above overwrites below
    if (nl_old > 0 && s_lmr[0].w >= 0 && s_lmr[0].y >= max(32, V / 8)) {  // many continuations
      // the state's dense row: per label log p(v | u) - log p(v) - cum_0, 0
      // for no arc (whose delta is 0 as well), contiguous
      const float4* R = reinterpret_cast<const float4*>(d.lm.dense0 + (size_t)s_lmr[0].w * d.lm.V4);
      float4* k4 = reinterpret_cast<float4*>(dlm);
      const int nq4 = d.lm.V4 / 4;
      for (int q0 = tid; q0 < nq4; q0 += kDense * kFzThreads) {
        float4 rq[kDense];
#pragma unroll
        for (int u = 0; u < kDense; ++u) {
          const int q = q0 + u * kFzThreads;
          if (q < nq4) rq[u] = __ldg(R + q);
        }
#pragma unroll
        for (int u = 0; u < kDense; ++u) {
          const int q = q0 + u * kFzThreads;
          if (q < nq4) k4[q] = make_float4(lam * rq[u].x, lam * rq[u].y, lam * rq[u].z, lam * rq[u].w);
        }
      }
    } else {
      // every label's delta starts at 0 (a dense row above writes them all)
      float4* k4 = reinterpret_cast<float4*>(dlm);
      for (int q = tid; q < d.V4 / 4; q += blockDim.x) k4[q] = make_float4(0.f, 0.f, 0.f, 0.f);
      row::block_sync();
    }
    if (nl_old > 0 && !(s_lmr[0].w >= 0 && s_lmr[0].y >= max(32, V / 8))) {
      const int b0 = s_lmr[0].x, c0 = s_lmr[0].y;
      const int a0 = b0 & ~3, G0 = level_groups(b0, c0);
      for (int gb = 0; gb < G0; gb += kStream * kFzThreads) {
        int4 tk[kStream];
        float4 lp[kStream];
#pragma unroll
        for (int u = 0; u < kStream; ++u) {
          const int g = gb + u * kFzThreads + tid;
          if (g < G0) {
            tk[u] = __ldg(t4 + (a0 >> 2) + g);
            lp[u] = __ldg(p4 + (a0 >> 2) + g);
          }
        }
#pragma unroll
        for (int u = 0; u < kStream; ++u) {
          const int g = gb + u * kFzThreads + tid;
          if (g < G0) {
            const int i0 = a0 + 4 * g;
            const int tv[4] = {tk[u].x, tk[u].y, tk[u].z, tk[u].w};
            const float pv[4] = {lp[u].x, lp[u].y, lp[u].z, lp[u].w};
#pragma unroll
            for (int j = 0; j < 4; ++j)
              if (i0 + j >= b0 && i0 + j < b0 + c0 && checked(tv[j] >= 0 && tv[j] < V, d.err, 9))
                dlm[tv[j]] = delta_of(0, pv[j], tv[j]);
          }
        }
      }
    }
    // 1c. every arc of the levels above 0 sets its level's bit in its
    //     label's word (two labels per 32-bit word), so a label's deepest
    //     level with an arc is its highest bit
    uint32_t* lev2 = reinterpret_cast<uint32_t*>(lev);
    auto offer = [&](int l, int i0, int4 tk) {
      const int b = s_lmr[l].x, c = s_lmr[l].y;
      const int tv[4] = {tk.x, tk.y, tk.z, tk.w};
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i0 + j >= b && i0 + j < b + c && checked(tv[j] >= 0 && tv[j] < V, d.err, 9))
          atomicOr(lev2 + (tv[j] >> 1), 1u << (l + 16 * (tv[j] & 1)));
    };
#pragma unroll
    for (int u = 0; u < kHeld; ++u)
      if (hl[u] >= 0) offer(hl[u], hi[u], ht[u]);
    for (int g = tid + kHeld * kFzThreads; g < G; g += kFzThreads) {  // past what registers hold
      int l;
      const int i0 = locate(g, l);
      offer(l, i0, __ldg(t4 + (i0 >> 2)));
    }
    if (nt_old > 0) {  // the trie chain nodes, shallowest first (the deepest overwrites)
      const int k = nt_old - 1;
      row::scatter_trie_node(d.tr.ch_tok, s_trr[k].x, s_trr[k].x + s_trr[k].y, (uint8_t)s_trr[k].z, dep);
    }
    row::block_sync();
    // 1d. the arc of each label at its deepest level writes the label's delta
    //     (one writer per label: a level's arcs have distinct labels)
    auto deepest = [&](int v) { return 31 - __clz((int)lev[v]); };
#pragma unroll
    for (int u = 0; u < kHeld; ++u) {
      if (hl[u] >= 0) {
        const int l = hl[u], b = s_lmr[l].x, c = s_lmr[l].y;
        const int tv[4] = {ht[u].x, ht[u].y, ht[u].z, ht[u].w};
        const float pv[4] = {hp[u].x, hp[u].y, hp[u].z, hp[u].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int i = hi[u] + j;
          if (i >= b && i < b + c && checked(tv[j] >= 0 && tv[j] < V, d.err, 9) && deepest(tv[j]) == l)
            dlm[tv[j]] = delta_of(l, pv[j], tv[j]);
        }
      }
    }
    for (int g = tid + kHeld * kFzThreads; g < G; g += kFzThreads) {  // past what registers hold
      int l;
      const int i0 = locate(g, l);
      const int4 tk = __ldg(t4 + (i0 >> 2));
      const float4 lq = __ldg(p4 + (i0 >> 2));
      const int b = s_lmr[l].x, c = s_lmr[l].y;
      const int tv[4] = {tk.x, tk.y, tk.z, tk.w};
      const float pv[4] = {lq.x, lq.y, lq.z, lq.w};
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i0 + j >= b && i0 + j < b + c && checked(tv[j] >= 0 && tv[j] < V, d.err, 9) && deepest(tv[j]) == l)
          dlm[tv[j]] = delta_of(l, pv[j], tv[j]);
    }
    if (nt_old > 1) {
      const int k = nt_old - 2;
      row::scatter_trie_node(d.tr.ch_tok, s_trr[k].x, s_trr[k].x + s_trr[k].y, (uint8_t)s_trr[k].z, dep);
    }
    for (int k = nt_old - 3; k >= 0; --k) {
      row::block_sync();
      row::scatter_trie_node(d.tr.ch_tok, s_trr[k].x, s_trr[k].x + s_trr[k].y, (uint8_t)s_trr[k].z, dep);
    }
    row::block_sync();
  }
  // Programmatic dependent launch: everything above reads only state the
  // previous row pass wrote (complete before the joint kernel in between let
  // this grid launch) and constant tables; the logits need the wait.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (evaluated) {
    // 2. the argmax of logit + D + c_r + delta over the labels (blank takes
    //    its logit alone); the log-sum-exp of the raw logits (from the tile
    //    partials) is needed only for an emitted label's score
    const float* lg = d.logits + (size_t)r * d.N_pad;
    if (counting && tid == 0) {
      // Algorithmic bytes: the row's logits and partials read, the row state
      // read and written, every arc of every LM chain level (label +
      // log-probability) and every child of every trie chain node (label)
      // with its record; searches and the joint input are added where they
      // happen; the call's shared rows once per launch by the host.
      unsigned long long ab = 0;
      for (int l = 0; l < nl_old; ++l) ab += 16 + 8ull * s_lmr[l].y;
      for (int k = 0; k < nt_old; ++k) ab += 16 + 4ull * s_trr[k].y;
      s_bytes = ab + 4ull * (V + 1) + 16ull * d.n_ptiles + 2ull * (24 + 4 * (nl_old + nt_old));
    }
    float bv = kNegInf;
    int bi = INT_MAX;
    {
      // c_r = lambda*(summed backoff of the state) - beta*bonus*depth
      const float cum_top = nl_old ? __int_as_float(s_lmr[nl_old - 1].z) : 0.f;
      const int depth_cur = nt_old ? s_trr[0].z - 1 : 0;
      const float cr = lam * cum_top - bscale * (float)depth_cur;
      const int nq = (V + 3) >> 2;  // quads holding labels < V
      const float4* l4 = reinterpret_cast<const float4*>(lg);
      const float4* k4 = reinterpret_cast<const float4*>(dlm);
      const uint32_t* e4 = reinterpret_cast<const uint32_t*>(dep);
      for (int q0 = tid; q0 < nq; q0 += QB * kFzThreads) {
        float4 lq[QB];
#pragma unroll
        for (int u = 0; u < QB; ++u) {
          const int q = q0 + u * kFzThreads;
          if (q < nq) lq[u] = __ldcg(l4 + q);
        }
#pragma unroll
        for (int u = 0; u < QB; ++u) {
          const int q = q0 + u * kFzThreads;
          if (q < nq) {
            const float4 kq = k4[q];
            const uint32_t eq = e4[q];
            const float lv[4] = {lq[u].x, lq[u].y, lq[u].z, lq[u].w};
            float dl[4] = {kq.x, kq.y, kq.z, kq.w};
            if (eq) {  // a label of this quad has a trie goto node
              const uint32_t rb = __ldg(d.droot + (q >> 3)) >> ((4 * q) & 31);
#pragma unroll
              for (int j = 0; j < 4; ++j) {
                const uint32_t e = (eq >> (8 * j)) & 0xffu;
                if (e) dl[j] += bscale * (float)e - (((rb >> j) & 1u) ? bscale : 0.f);
              }
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) {
              const float fv = lv[j] + (cr + dl[j]);
              if (4 * q + j < V && fv > bv) { bv = fv; bi = 4 * q + j; }
            }
          }
        }
      }
      if (tid == 0) {
        const float fb = __ldcg(lg + V);  // blank: D[V] = 0, no fusion terms
        if (fb > bv) { bv = fb; bi = V; }
      }
    }
    row::reconverge();
    for (int o = 16; o > 0; o >>= 1) {
      const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
      best_merge(bv, bi, v2, i2);
    }
    if (lane == 0) {
      s_bv[warp] = bv;
      s_bi[warp] = bi;
    }
    row::block_sync();
    // every thread merges the warps' bests (no second barrier)
    float b = s_bv[0];
    int bix = s_bi[0];
#pragma unroll
    for (int w = 1; w < kFzWarps; ++w) best_merge(b, bix, s_bv[w], s_bi[w]);
    const int y = (bix >= 0 && bix <= V) ? bix : V;
    if (tid == 0) {
      s_y = y;
      s_score = b;  // the fused score less the log-sum-exp
    }
    if (!PRED) row::prefetch_span(d.E + (size_t)(y != V ? y : s_last) * d.H, (size_t)d.H * 2, 32);
    if (y != V) {
      // 3a. independent searches of y in every chain element; each hit's
      //     record is the next chain element's
      if (tid == kFzThreads - 1) {
        s_root_hit = d.has_tr ? __ldg(d.tr.root_rec + y) : make_int4(0, 0, 0, 0);
      } else if (tid == kFzThreads - 2) {
        s_uni_hit = (d.has_lm && d.lm.order >= 2) ? __ldg(d.lm.uni_rec + y) : make_int4(-1, 0, 0, 0);
      }
      // the last warp's first tile partials load while it searches
      const float4* pr = d.part + (size_t)r * d.n_ptiles;
      float4 p0 = make_float4(kNegInf, 0.f, 0.f, 0.f);
      if (warp == kFzWarps - 1 && lane < d.n_ptiles) p0 = __ldcg(pr + lane);  // written by the joint kernel
      for (int task = warp; task < nl_old + nt_old; task += kFzWarps) {
        if (task < nl_old) {
          const int b = s_lmr[task].x, c = s_lmr[task].y;
          const int i = warp_find_wide(d.lm.arc_tok + b, c, y, lane);
          if (lane == 0) s_lm_hit[task] = (i >= 0) ? __ldg(d.lm.arc_rec + b + i) : make_int4(-2, 0, 0, 0);
          if (counting && lane == 0) atomicAdd(&s_bytes, 4ull * (32 - __clz(c + 1)) + 16);
        } else {
          const int k = task - nl_old;
          const int b = s_trr[k].x, c = s_trr[k].y;
          const int i = warp_find_wide(d.tr.ch_tok + b, c, y, lane);
          if (lane == 0) s_tr_hit[k] = (i >= 0) ? __ldg(d.tr.ch_rec + b + i) : make_int4(-1, 0, 0, 0);
          if (counting && lane == 0) atomicAdd(&s_bytes, 4ull * (32 - __clz(c + 1)) + 16);
        }
      }
      if (warp == kFzWarps - 1) {  // the log-sum-exp of the raw logits
        float pm = kNegInf, ps = 0.f;
        lse_merge(pm, ps, p0.x, p0.y);
        for (int j = lane + 32; j < d.n_ptiles; j += 32) {
          const float4 p = __ldcg(pr + j);
          lse_merge(pm, ps, p.x, p.y);
        }
        row::reconverge();
        for (int o = 16; o > 0; o >>= 1) {
          const float m2 = __shfl_xor_sync(0xffffffffu, pm, o);
          const float s2 = __shfl_xor_sync(0xffffffffu, ps, o);
          lse_merge(pm, ps, m2, s2);
        }
        if (lane == 0) s_lse = pm + logf(ps);
      }
      row::block_sync();
      // 3b. assemble the new chains in place (shared memory) and commit them
      //     (by slot, and by row for the next step): warp 0 the LM chain
      //     (y's unigram state, then the targets of y's arcs at the old levels
      //     up to the first level without one), warp 1 the trie chain (y's
      //     children of the old chain nodes, deepest first, then the root's;
      //     completing a phrase resets it), warp 2 the outputs
      if (warp == 0) {
        int ln = 0;
        if (d.has_lm && d.lm.order >= 2) {
          const int4 h = lane < nl_old ? s_lm_hit[lane] : make_int4(-2, 0, 0, 0);
          const bool cont =
              h.x >= 0 && checked(h.x < d.lm.n_states && h.y >= 0 && h.z >= 0 && (int64_t)h.y + h.z <= d.lm.n_arcs,
                                  d.err, 10);
          const unsigned miss = __ballot_sync(0xffffffffu, !cont);
          ln = 1 + min(miss ? __ffs((int)miss) - 1 : 32, kLmChain - 1);
          const int4 u = s_uni_hit;  // u.x is y's dense row
          // lane l >= 1 takes the hit of old level l - 1
          const int px = __shfl_up_sync(0xffffffffu, h.x, 1), py = __shfl_up_sync(0xffffffffu, h.y, 1);
          const int pz = __shfl_up_sync(0xffffffffu, h.z, 1), pw = __shfl_up_sync(0xffffffffu, h.w, 1);
          const int nst = lane == 0 ? 1 + y : px;
          const int4 nrec = lane == 0 ? make_int4(u.y, u.z, u.w, u.x) : make_int4(py, pz, pw, 0);
          __syncwarp();
          if (lane < ln) {
            s_lm[lane] = nst;
            s_lmr[lane] = nrec;
            if (commit) {
              d.s_lm_chain[(size_t)slot * kLmChain + lane] = nst;
              d.s_lm_rec[(size_t)slot * kLmChain + lane] = nrec;
              d.m_lm[(size_t)r * kLmChain + lane] = nst;
              d.m_lmr[(size_t)r * kLmChain + lane] = nrec;
            }
          }
        }
        if (lane == 0) {
          s_nl = ln;
          if (commit) {
            if (d.has_lm) d.s_lm_len[slot] = ln;
            d.m_lm_len[r] = ln;
          }
        }
      } else if (warp == 1) {
        const int4 h = lane < nt_old ? s_tr_hit[lane] : make_int4(-1, 0, 0, 0);
        const int dd = lane < nt_old ? s_trr[lane].z + 1 : 0;  // the child's children sit one deeper
        const bool ok = h.x >= 0 && checked(h.x > 0 && h.x < d.tr.n_nodes && h.w >= 0 && h.z + h.w <= d.tr.n_children,
                                            d.err, 11);
        const unsigned vm = __ballot_sync(0xffffffffu, ok);
        const int nv = __popc(vm);
        const int4 rh = s_root_hit;
        const bool root = rh.x != 0;
        // the first element of the new chain ends a phrase: the chain resets
        const int f = __ffs((int)vm) - 1;
        const int fy = __shfl_sync(0xffffffffu, h.y, f < 0 ? 0 : f);
        const bool reset = nv > 0 ? fy == 0 : (root && rh.y == 0);
        const int tn = reset ? 0 : min(nv + (root ? 1 : 0), kTrChain);
        __syncwarp();
        const int pos = __popc(vm & ((1u << lane) - 1u));
        if (ok && pos < tn) {
          s_tr[pos] = h.x;
          s_trr[pos] = make_int4(h.z, h.w, dd, 0);
        }
        if (lane == 0 && root && nv < tn) {
          s_tr[nv] = rh.x;
          s_trr[nv] = make_int4(rh.z, rh.w, 2, 0);
        }
        __syncwarp();
        if (commit && lane < tn) {
          d.s_tr_chain[slot * kTrChain + lane] = s_tr[lane];
          d.s_tr_rec[(size_t)slot * kTrChain + lane] = s_trr[lane];
          d.m_tr[(size_t)r * kTrChain + lane] = s_tr[lane];
          d.m_trr[(size_t)r * kTrChain + lane] = s_trr[lane];
        }
        if (lane == 0) {
          s_nt = tn;
          if (commit) {
            if (d.has_tr) d.s_tr_len[slot] = tn;
            d.m_tr_len[r] = tn;
          }
        }
      } else if (tid == 64) {
        if (commit) {
          const int cap = T * d.max_sym;
          const int o = r * cap + s_cnt;
          s_out_tok[o] = y;
          s_out_frame[o] = s_t;
          s_out_score[o] = s_score - s_lse;
          d.s_last[slot] = y;
          d.m_last[r] = y;
        }
        s_cnt += 1;
        s_last = y;
        s_sym += 1;
        if (s_sym >= d.max_sym) { s_t += 1; s_sym = 0; }
      }
    } else if (tid == 0) {
      s_t += 1;
      s_sym = 0;
    }
    row::block_sync();
  }

  if (PRED) {
    // Stateful form: the prediction network reads the label just emitted
    // (or, at a stream's first step, the start of sequence) and the row's h
    // from before this step; the LSTM kernel after this one runs the cell.
    const bool fresh = step == 0 && __ldcg(d.pred_fresh + slot) != 0;
    const bool stepped = fresh || (evaluated && s_y != V);
    if (tid == 0) {
      d.pflag[r] = stepped ? 1 : 0;
      if (fresh && commit) d.pred_fresh[slot] = 0;
    }
    if (stepped) {
      const int D = d.pred_D;
      const int lab = fresh ? V : s_y;
      const uint4* src_x = reinterpret_cast<const uint4*>(d.pred_emb + (size_t)lab * D);
      const uint4* src_h = reinterpret_cast<const uint4*>(d.pred_h + (size_t)slot * D);
      uint4* dst = reinterpret_cast<uint4*>(d.pred_x + (size_t)r * 2 * D);
      for (int i = tid; i < D / 4; i += blockDim.x) dst[i] = (i < D / 8) ? __ldg(src_x + i) : __ldcg(src_h + i - D / 8);
    }
  }
  if (counting && tid == 0 && evaluated) atomicAdd(d.ctr, s_bytes);
  if (mode == 1) {
    if (tid == 0) s_out_count[r] = s_cnt;
    return;
  }
  if (tid == 0 && commit) {
    d.r_t[r] = s_t;
    d.r_sym[r] = s_sym;
    d.r_cnt[r] = s_cnt;
  }
  const int t = commit ? s_t : min(s_t, T - 1);
  const int nl = s_nl, nt = s_nt;
  if (d.cap_rows && step < d.cap_steps && tid == 0 && commit) {
    int* c = d.cap_rows + ((size_t)step * s_n + r) * 4;
    if (t < T) {
      c[0] = t;
      c[1] = s_last;
      c[2] = nl ? s_lm[nl - 1] : 0;
      c[3] = nt ? s_tr[0] : 0;
    } else {
      c[0] = -1; c[1] = -1; c[2] = -1; c[3] = -1;
    }
  }
  if (t >= T) return;

  // 4. joint input of this step
  if (!PRED) row::build_joint_input(d, s_enc + ((size_t)r * T + t) * d.H, s_last, r);
  if (counting && tid == 0 && !PRED) atomicAdd(d.ctr, 6ull * d.H);  // encoder frame, embedding row, A row
}

}  // namespace

size_t row_stream_smem_bytes(int V4) { return (size_t)V4 * (sizeof(float) + sizeof(uint16_t) + sizeof(uint8_t)); }

cudaError_t prepare_stream_kernels(size_t smem) {
  cudaError_t e = cudaFuncSetAttribute(k_row_fz<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_row_fz<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_row_fz<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_row_fz<5>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  return e;
}

void launch_row_stream(const DecView& d, int M, int step, int mode, size_t smem, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(M);
  cfg.blockDim = dim3(kFzThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  const bool few = M <= 2 * d.sms;
  if (d.pred_D) {
    if (few) cudaLaunchKernelEx(&cfg, k_row_fz<5>, d, step, mode);
    else cudaLaunchKernelEx(&cfg, k_row_fz<1>, d, step, mode);
  } else {
    if (few) cudaLaunchKernelEx(&cfg, k_row_fz<4>, d, step, mode);
    else cudaLaunchKernelEx(&cfg, k_row_fz<0>, d, step, mode);
  }
}

}  // namespace tsd
