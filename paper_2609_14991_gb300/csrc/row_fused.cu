// Row pass of the fused decode step (greedy decoding, at most one n-gram
// LM): one CTA per hypothesis row.
//
// Eq. 1 for label v < V at the row's state is
//   fused[v] = logit[v] - lse + lambda*log p_LM(v | h) + beta*bonus*(g(v) - depth)
// where the LM state is kept as its whole suffix chain s_0 (the unigram state
// of the previous label u), s_1, ..., s_{L-1} (one state per order):
// log p_LM(v | h) is the arc v of the deepest chain state s_l that has one
// plus the backoff weights of the deeper states, or log p(v) plus all of
// them; g(v) is the depth of v's goto node from the deepest trie chain node
// with a child v (the trie chain holds every trie node that is a suffix of
// the current match), else [the root has a child v].  With cum_l the summed
// backoff of s_0..s_l and
//   c_r = lambda*cum_{L-1} - beta*bonus*depth   (one constant per row),
//   F[v] = fused[v] + lse - c_r
//        = logit[v] + lambda*(log p(v | s_l) - cum_l) + beta*bonus*g(v),
// with log p(v) and cum_{-1} = 0 when no chain state has an arc v.  Blank
// (label V) has F = logit[V] - c_r.
//
// The deeper chain states' labels are nested: s_{l+1} has an arc v only if
// s_l has one (the model is suffix-closed), so every label whose deepest arc
// is not s_0's is a label of s_1, which has few arcs (a context of two
// labels).  The joint kernel therefore evaluates, for every label,
//   F0[v] = logit[v] + D[v] + lambda*dense0[u][v],
//   D[v] = lambda*log p(v) + beta*bonus*[the root has a child v],
//   dense0[u][v] = log p(v | u) - log p(v) - cum_0 (0 if u has no arc v),
// which is F[v] for every label except those of s_1's arcs, the children of
// the trie chain nodes, and blank: this pass lists those for the row (label
// and its term F[v] - logit[v]) and marks them in a bitmask; the joint
// leaves them out of its per-tile best and stores their raw logits.
//
// For row r at label step s the pass
//   1. loads the row's state, both chains with their table records, and the
//      length of the list its previous step wrote (for the state the joint
//      just evaluated);
//   2. after waiting for the joint kernel: the log-sum-exp and the best
//      unlisted label from the tile partials, every listed label's F from its
//      stored logit, blank's, and the argmax of them all (ties to the lowest
//      label): the greedy decision and its fused score;
//   3. blank (or the per-frame label limit) advances the frame; a label y is
//      emitted and advances the chains, assembled from independent searches
//      of y in every chain element, each hit carrying the next state's table
//      record (first arc, arcs, summed backoff) in the same 16-byte load;
//   4. lists the labels of the new state: s_1's arcs, each with the term of
//      its deepest chain level (found by a shared-memory atomicMax of
//      ((level + 1) << 24 | position) over levels 1..L-1) plus the trie
//      term; then the trie chain nodes' children that are not s_1 labels,
//      with the level-0 LM term; the bitmask; c_r;
//   5. writes the joint input of step s, bf16(ReLU(enc_t + E[last])).
#include <algorithm>

#include "row_common.cuh"

namespace tsd {

namespace {

using row::best_merge;
using row::checked;
using row::kNegInf;
using row::lse_merge;
using row::warp_find;

constexpr int kFzThreads = 128;  // 4 warps: seven CTAs per SM at 72 registers (1024 rows over 147 SMs)
constexpr int kFzWarps = kFzThreads / 32;
constexpr int kHeld = 1;      // arc groups of four of levels 1.. a thread keeps in registers
constexpr int kListPre = 32;  // list entries loaded (one per thread) before the list's length is known
constexpr int kTrHeld = 1;    // trie chain children a thread keeps in registers

// Aligned groups of four arcs a chain level's arcs [b, b + c) span.
__device__ __forceinline__ int level_groups(int b, int c) { return c > 0 ? (b + c - (b & ~3) + 3) >> 2 : 0; }

// mode: 0 = label step, 1 = final step (apply the last decision only),
// 2 = replay (redo the step's work without committing any state or output;
// used only to time the kernel in isolation).
// VAR bit 0: the stateful form (LSTM input rows instead of the joint input);
// bit 2: few rows (at most two CTAs per SM are needed, registers are free).
template <int VAR>
__global__ void __launch_bounds__(kFzThreads) __maxnreg__((VAR & 4) ? 128 : 72) k_row_ep(DecView d, int step, int mode) {
  constexpr bool PRED = (VAR & 1) != 0;
  const Params* __restrict__ P = d.params;
  const int r = blockIdx.x;
  const int V = d.V;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool commit = (mode != 2);
  const bool counting = (mode == 2 || d.count);
  extern __shared__ __align__(16) unsigned char smem[];
  // per label: the offer tag, then (for the winners) the LM term's bits; the
  // list bitmask; the root's children bitmask; 1 if the label has its LM
  // term; the trie goto depth (0: none)
  uint32_t* key = reinterpret_cast<uint32_t*>(smem);                // [V4]
  uint32_t* msk = key + d.V4;                                        // [mask_words]
  uint32_t* rootw = msk + d.mask_words;                              // [mask_words]
  uint8_t* lmf = reinterpret_cast<uint8_t*>(rootw + d.mask_words);  // [V4]
  uint8_t* dep = lmf + d.V4;                                       // [V4]

  __shared__ int s_t, s_sym, s_cnt, s_y, s_last, s_slot, s_T, s_n;
  __shared__ int s_nl, s_nt, s_ext;
  __shared__ int32_t* s_out_tok;
  __shared__ int32_t* s_out_frame;
  __shared__ float* s_out_score;
  __shared__ int32_t* s_out_count;
  __shared__ const uint16_t* s_enc;
  __shared__ float s_lam, s_beta, s_score, s_lse, s_cr;
  __shared__ int4 s_ci;               // the list the joint evaluated: (dense row, length, c_r bits, -)
  __shared__ int s_lm[kLmChain], s_tr[kTrChain];
  __shared__ int4 s_lmr[kLmChain];    // LM chain records: (first arc, arcs, summed backoff bits, dense row at level 0)
  __shared__ int4 s_trr[kTrChain];    // trie chain records: (first child, children, depth of the children, -)
  __shared__ int4 s_lm_hit[kLmChain]; // target record of y's arc at each old level (x = -2: none)
  __shared__ int4 s_tr_hit[kTrChain]; // child record of y at each old trie node (x = -1: none)
  __shared__ int4 s_uni_hit, s_root_hit;
  __shared__ int s_gbeg[kLmChain + 1];  // arc groups of the LM levels 1.. before level l
  __shared__ int s_tpre[kTrChain + 1];  // children of the trie chain nodes before node k
  __shared__ float s_bv[kFzWarps];
  __shared__ int s_bi[kFzWarps];
  __shared__ unsigned long long s_bytes;  // algorithmic bytes of the row-step (when counting)
  __shared__ int s_bad;                   // TSD_CHECKS: a range check failed; the row stops

  // 1. Row state.  It was written by the previous row pass; under
  // programmatic launch this grid may start before its own wait, so these
  // loads go through L2 only (ld.global.cg), never a possibly stale L1 line.
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
    s_ext = 0;
    s_ci = step > 0 ? __ldcg(d.c_info + r) : make_int4(-1, 0, 0, 0);
    s_bad = !checked(slot >= 0 && slot < d.lm_stride, d.err, 1);
    if (step > 0) {  // the row's copy of its state, written by the previous row pass
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
  // the list of the state the joint evaluated: its first kListPre entries,
  // one per thread (loaded whatever its length, which lists rarely exceed;
  // entries past it are dropped once the length is known)
  int hv = -1;
  float ha = 0.f;
  if (step > 0 && tid < kListPre && tid < d.V4) {
    hv = __ldcg(d.c_lab + (size_t)r * d.V4 + tid);
    ha = __ldcg(d.c_add + (size_t)r * d.V4 + tid);
  }
  {  // per-label scratch reset
    uint4* k4 = reinterpret_cast<uint4*>(key);
    uint32_t* f4 = reinterpret_cast<uint32_t*>(lmf);
    uint32_t* e4 = reinterpret_cast<uint32_t*>(dep);
    for (int q = tid; q < d.V4 / 4; q += blockDim.x) {
      k4[q] = make_uint4(0u, 0u, 0u, 0u);
      f4[q] = 0u;
      e4[q] = 0u;
    }
    for (int q = tid; q < d.mask_words; q += blockDim.x) {
      msk[q] = 0u;
      rootw[q] = q < (V + 31) / 32 ? __ldg(d.droot + q) : 0u;
    }
  }
  row::block_sync();
  if (s_bad) return;
  const int slot = s_slot, T = s_T;
  if (tid >= s_ci.y) hv = -1;
  if (step == 0) {
    // the chunk's first step: the stream's state by slot (the chains are
    // read whole: their arrays have room for the longest), and the row's copy
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
    if (ok && step > 0 && s_t < T) ok = checked(s_ci.y >= 0 && s_ci.y <= d.V4, d.err, 12);
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

  // Programmatic dependent launch: everything above reads only state the
  // previous row pass wrote (complete before the joint kernel in between let
  // this grid launch) and constant tables; the partials and logits need the
  // wait.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (evaluated) {
    // 2. the decision: the log-sum-exp and the best unlisted label from the
    //    tile partials (warp 0), every listed label from its stored logit
    const float* lg = d.logits + (size_t)r * d.N_pad;
    const int4 ci = s_ci;
    const float cr_prev = __int_as_float(ci.z);
    float bv = kNegInf;
    int bi = INT_MAX;
    if (warp == 0) {
      float m = kNegInf, s = 0.f;
      const float4* pr = d.part + (size_t)r * d.n_ptiles;
      for (int j = lane; j < d.n_ptiles; j += 32) {
        const float4 p = __ldcg(pr + j);  // written by the joint kernel just before
        lse_merge(m, s, p.x, p.y);
        best_merge(bv, bi, p.z, __float_as_int(p.w));
      }
      row::reconverge();
      for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
        lse_merge(m, s, m2, s2);
      }
      if (lane == 0) s_lse = m + logf(s);
    }
    {
      if (hv >= 0 && checked(hv < V, d.err, 13)) best_merge(bv, bi, __ldcg(lg + hv) + ha, hv);
      const int32_t* cl = d.c_lab + (size_t)r * d.V4;
      const float* ca = d.c_add + (size_t)r * d.V4;
      for (int k0 = kListPre + tid; k0 < ci.y; k0 += 4 * kFzThreads) {
        int v[4];
        float a[4], x[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int k = k0 + u * kFzThreads;
          v[u] = -1;
          a[u] = 0.f;
          x[u] = kNegInf;
          if (k < ci.y) {
            v[u] = __ldcg(cl + k);
            a[u] = __ldcg(ca + k);
          }
        }
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (v[u] >= 0 && checked(v[u] < V, d.err, 13)) x[u] = __ldcg(lg + v[u]);
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (v[u] >= 0 && v[u] < V) best_merge(bv, bi, x[u] + a[u], v[u]);
      }
    }
    if (tid == 0) {
      const float fb = __ldcg(lg + V) - cr_prev;  // blank: no fusion terms
      if (fb > bv) { bv = fb; bi = V; }
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
      s_score = (b + cr_prev) - s_lse;
      if (counting) {
        // algorithmic bytes of the decision: partials, the list and its
        // logits, blank's logit, the row state read and written, the chain
        // records read
        unsigned long long ab = 16ull * d.n_ptiles + 12ull * ci.y + 4 + 16;
        ab += 2ull * (24 + 4 * (nl_old + nt_old)) + 16ull * (nl_old + nt_old);
        atomicAdd(&s_bytes, ab);
      }
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
      for (int task = warp; task < nl_old + nt_old; task += kFzWarps) {
        if (task < nl_old) {
          const int b = s_lmr[task].x, c = s_lmr[task].y;
          const int i = warp_find(d.lm.arc_tok + b, c, y, lane);
          if (lane == 0) s_lm_hit[task] = (i >= 0) ? __ldg(d.lm.arc_rec + b + i) : make_int4(-2, 0, 0, 0);
          if (counting && lane == 0) atomicAdd(&s_bytes, 4ull * (32 - __clz(c + 1)) + 16);
        } else {
          const int k = task - nl_old;
          const int b = s_trr[k].x, c = s_trr[k].y;
          const int i = warp_find(d.tr.ch_tok + b, c, y, lane);
          if (lane == 0) s_tr_hit[k] = (i >= 0) ? __ldg(d.tr.ch_rec + b + i) : make_int4(-1, 0, 0, 0);
          if (counting && lane == 0) atomicAdd(&s_bytes, 4ull * (32 - __clz(c + 1)) + 16);
        }
      }
      row::block_sync();
      // 3b. assemble the new chains in place (shared memory) and commit them:
      //     warp 0 the LM chain (y's unigram state, then the targets of y's
      //     arcs at the old levels up to the first level without one), warp 1
      //     the trie chain (y's children of the old chain nodes, deepest
      //     first, then the root's; a completed phrase resets it), warp 2
      //     the outputs
      if (warp == 0) {
        int ln = 0;
        if (d.has_lm && d.lm.order >= 2) {
          const int4 h = lane < nl_old ? s_lm_hit[lane] : make_int4(-2, 0, 0, 0);
          const bool cont =
              h.x >= 0 && checked(h.x < d.lm.n_states && h.y >= 0 && h.z >= 0 && (int64_t)h.y + h.z <= d.lm.n_arcs,
                                  d.err, 10);
          const unsigned miss = __ballot_sync(0xffffffffu, !cont);
          ln = 1 + min(miss ? __ffs((int)miss) - 1 : 32, kLmChain - 1);
          const int4 u = s_uni_hit;
          const int st = lane == 0 ? 1 + y : h.x;  // new level `lane`: y's unigram state, then targets
          const int4 rec = lane == 0 ? make_int4(u.y, u.z, u.w, u.x) : make_int4(0, 0, 0, 0);
          // lane l >= 1 takes the hit of old level l - 1
          const int px = __shfl_up_sync(0xffffffffu, h.x, 1), py = __shfl_up_sync(0xffffffffu, h.y, 1);
          const int pz = __shfl_up_sync(0xffffffffu, h.z, 1), pw = __shfl_up_sync(0xffffffffu, h.w, 1);
          const int4 nrec = lane == 0 ? rec : make_int4(py, pz, pw, 0);
          const int nst = lane == 0 ? st : px;
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
          if (commit && d.has_lm) {
            d.s_lm_len[slot] = ln;
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
          if (commit && d.has_tr) {
            d.s_tr_len[slot] = tn;
            d.m_tr_len[r] = tn;
          }
        }
      } else if (tid == 64) {
        if (commit) {
          const int cap = T * d.max_sym;
          const int o = r * cap + s_cnt;
          s_out_tok[o] = y;
          s_out_frame[o] = s_t;
          s_out_score[o] = s_score;
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
  if (mode == 1) {
    if (counting && tid == 0 && evaluated) atomicAdd(d.ctr, s_bytes);
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
  if (t >= T) {  // no joint input this step: the row's list is not read
    if (counting && tid == 0 && evaluated) atomicAdd(d.ctr, s_bytes);
    return;
  }

  // 4. the correction list of the row's (new) state, for the joint kernel
  //    of this step and the decision of the next.  Warp 0: the arc groups
  //    of levels 1.. before each level (a prefix sum over its lanes), c_r
  if (warp == 0) {
    const int l = lane + 1;
    const int4 rc = l < nl ? s_lmr[l] : make_int4(0, 0, 0, 0);
    const int g = l < nl ? level_groups(rc.x, rc.y) : 0;
    int incl = g;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (l <= max(nl, 1)) s_gbeg[l] = incl - g;
    if (counting) {  // every arc of levels 1.. (label + log-probability), every child label of the trie chain
      unsigned long long ab = (l < nl ? 8ull * rc.y : 0ull) + (lane < nt ? 4ull * s_trr[lane].y : 0ull);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) ab += __shfl_xor_sync(0xffffffffu, ab, o);
      if (lane == 0) s_bytes += ab;
    }
    if (lane == 0) {
      const float cum_top = nl ? __int_as_float(s_lmr[nl - 1].z) : 0.f;
      const int depth_cur = nt ? s_trr[0].z - 1 : 0;
      s_cr = lam * cum_top - bscale * (float)depth_cur;
    }
  } else if (warp == 1) {  // the trie chain's children before each node
    const int c = lane < nt ? s_trr[lane].y : 0;
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    s_tpre[lane + 1] = incl;
    if (lane == 0) s_tpre[0] = 0;
  }
  row::block_sync();
  // the trie chain's children, one per thread while they fit (label, node,
  // and later its level-0 LM term); otherwise every phase reads them again
  const int TC = s_tpre[nt];
  const bool tr_held = TC <= kTrHeld * kFzThreads;
  const int drow = (d.has_lm && nl >= 1) ? s_lmr[0].w : -1;
  const float* dense = drow >= 0 ? d.lm.dense0 + (size_t)drow * d.V4 : nullptr;
  int trv[kTrHeld], trk[kTrHeld];
  float trl[kTrHeld];
#pragma unroll
  for (int u = 0; u < kTrHeld; ++u) {
    const int f = tid + u * kFzThreads;
    trv[u] = -1;
    trk[u] = -1;
    trl[u] = 0.f;
    if (tr_held && f < TC) {
      int k = 0;
      while (f >= s_tpre[k + 1]) ++k;
      trk[u] = k;
      trv[u] = __ldg(d.tr.ch_tok + s_trr[k].x + (f - s_tpre[k]));
    }
  }
  // node k's children write their goto depth (phases run shallowest first)
  auto trie_phase = [&](int k) {
    if (!tr_held) {
      row::scatter_trie_node(d.tr.ch_tok, s_trr[k].x, s_trr[k].x + s_trr[k].y, (uint8_t)s_trr[k].z, dep);
      return;
    }
#pragma unroll
    for (int u = 0; u < kTrHeld; ++u)
      if (trk[u] == k && checked(trv[u] >= 0 && trv[u] < V, d.err, 15)) dep[trv[u]] = (uint8_t)s_trr[k].z;
  };
  const int4* t4 = reinterpret_cast<const int4*>(d.lm.arc_tok);
  const float4* p4 = reinterpret_cast<const float4*>(d.lm.arc_logp);
  // the group g of levels 1..: its level and first arc
  auto locate = [&](int g, int& l) {
    l = 1;
    while (g >= s_gbeg[l + 1]) ++l;
    return (s_lmr[l].x & ~3) + 4 * (g - s_gbeg[l]);
  };
  auto lm_term = [&](int l, float lp) { return lam * (lp - __int_as_float(s_lmr[l].z)); };
  // 4a. levels 1.. offer ((l + 1) << 24 | position) to their labels, so the
  //     deepest wins; the trie chain nodes scatter their goto depths,
  //     shallowest first (the deepest overwrites), one node per phase
  const int G = nl >= 2 ? s_gbeg[nl] : 0;
  int4 ht[kHeld];
  float4 hp[kHeld];
  int hl[kHeld], hi[kHeld];
#pragma unroll
  for (int u = 0; u < kHeld; ++u) {
    const int g = tid + u * kFzThreads;
    hl[u] = -1;
    hi[u] = 0;
    ht[u] = make_int4(0, 0, 0, 0);
    hp[u] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (g < G) {
      int l;
      hi[u] = locate(g, l);
      ht[u] = __ldg(t4 + (hi[u] >> 2));
      hp[u] = __ldg(p4 + (hi[u] >> 2));
      hl[u] = l;
    }
  }
  auto offer = [&](int l, int i0, int4 tk) {
    const int b = s_lmr[l].x, c = s_lmr[l].y;
    const uint32_t tag = (uint32_t)(l + 1) << 24;
    const int tv[4] = {tk.x, tk.y, tk.z, tk.w};
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if (i0 + j >= b && i0 + j < b + c && checked(tv[j] >= 0 && tv[j] < V, d.err, 9))
        atomicMax(key + tv[j], tag | (uint32_t)(i0 + j - b));
  };
#pragma unroll
  for (int u = 0; u < kHeld; ++u)
    if (hl[u] >= 0) offer(hl[u], hi[u], ht[u]);
  for (int g = tid + kHeld * kFzThreads; g < G; g += kFzThreads) {  // past what registers hold
    int l;
    const int i0 = locate(g, l);
    offer(l, i0, __ldg(t4 + (i0 >> 2)));
  }
  if (nt > 0) trie_phase(nt - 1);
  // the held children's level-0 LM terms (used if a child is not a level-1 label)
#pragma unroll
  for (int u = 0; u < kTrHeld; ++u)
    if (d.has_lm && trv[u] >= 0 && trv[u] < V)
      trl[u] = lam * ((dense ? __ldg(dense + trv[u]) : 0.f) + __ldg(d.lm.uni_logp + trv[u]));
  row::block_sync();
  // 4b. the winners among the held offers (one per label) compute their LM
  //     term; it is written once every offer is judged
  uint32_t won = 0;  // bit 4u + j: arc j of held group u won
  float wv[kHeld][4];
#pragma unroll
  for (int u = 0; u < kHeld; ++u) {
    const int tv[4] = {ht[u].x, ht[u].y, ht[u].z, ht[u].w};
    const float pv[4] = {hp[u].x, hp[u].y, hp[u].z, hp[u].w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      wv[u][j] = 0.f;
      if (hl[u] >= 0) {
        const int l = hl[u], b = s_lmr[l].x, c = s_lmr[l].y;
        const int i = hi[u] + j;
        if (i >= b && i < b + c && checked(tv[j] >= 0 && tv[j] < V, d.err, 9) &&
            key[tv[j]] == (((uint32_t)(l + 1) << 24) | (uint32_t)(i - b))) {
          won |= 1u << (4 * u + j);
          wv[u][j] = lm_term(l, pv[j]);
        }
      }
    }
  }
  if (nt > 1) trie_phase(nt - 2);
  row::block_sync();
#pragma unroll
  for (int u = 0; u < kHeld; ++u) {
    const int tv[4] = {ht[u].x, ht[u].y, ht[u].z, ht[u].w};
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if ((won >> (4 * u + j)) & 1u) {
        key[tv[j]] = __float_as_uint(wv[u][j]);
        lmf[tv[j]] = 1;
      }
  }
  // offers past what registers hold (states with very many continuations):
  // judged a round at a time, a barrier between the judging and the
  // writing; a label already written is skipped by its flag
  for (int g0 = kHeld * kFzThreads; g0 < G; g0 += kFzThreads) {
    row::block_sync();
    const int g = g0 + tid;
    int4 tk = make_int4(0, 0, 0, 0);
    float xv[4] = {0.f, 0.f, 0.f, 0.f};
    uint32_t xw = 0;
    if (g < G) {
      int l;
      const int i0 = locate(g, l);
      tk = __ldg(t4 + (i0 >> 2));
      const float4 lq = __ldg(p4 + (i0 >> 2));
      const int b = s_lmr[l].x, c = s_lmr[l].y;
      const uint32_t tag = (uint32_t)(l + 1) << 24;
      const int tv[4] = {tk.x, tk.y, tk.z, tk.w};
      const float pv[4] = {lq.x, lq.y, lq.z, lq.w};
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i0 + j >= b && i0 + j < b + c && checked(tv[j] >= 0 && tv[j] < V, d.err, 9) && lmf[tv[j]] == 0 &&
            key[tv[j]] == (tag | (uint32_t)(i0 + j - b))) {
          xw |= 1u << j;
          xv[j] = lm_term(l, pv[j]);
        }
    }
    row::block_sync();
    const int tv[4] = {tk.x, tk.y, tk.z, tk.w};
#pragma unroll
    for (int j = 0; j < 4; ++j)
      if ((xw >> j) & 1u) {
        key[tv[j]] = __float_as_uint(xv[j]);
        lmf[tv[j]] = 1;
      }
  }
  for (int k = nt - 3; k >= 0; --k) {
    row::block_sync();
    trie_phase(k);
  }
  row::block_sync();
  // 4c. the list: level 1's arcs in order (every label of a deeper level is
  //     one of them), then the trie chain's children that are not
  {
    int32_t* cl = d.c_lab + (size_t)r * d.V4;
    float* ca = d.c_add + (size_t)r * d.V4;
    const int b1 = nl >= 2 ? s_lmr[1].x : 0, c1 = nl >= 2 ? s_lmr[1].y : 0;
    auto emit1 = [&](int j, int v) {  // level-1 arc j, label v
      if (!checked(v >= 0 && v < V && lmf[v] != 0, d.err, 14)) return;
      const uint32_t e = dep[v];
      const float tr = e ? bscale * (float)e : (((rootw[v >> 5] >> (v & 31)) & 1u) ? bscale : 0.f);
      cl[j] = v;
      ca[j] = __uint_as_float(key[v]) + tr;
      atomicOr(msk + (v >> 5), 1u << (v & 31));
    };
    // level 1's arcs: the groups held in registers since the offers, then
    // the rest (groups 0 .. G1-1 of levels 1.. are level 1's)
#pragma unroll
    for (int u = 0; u < kHeld; ++u) {
      if (hl[u] == 1) {
        const int tv[4] = {ht[u].x, ht[u].y, ht[u].z, ht[u].w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int i = hi[u] + j;
          if (i >= b1 && i < b1 + c1) emit1(i - b1, tv[j]);
        }
      }
    }
    const int G1 = nl >= 2 ? s_gbeg[2] : 0;
    for (int g = tid + kHeld * kFzThreads; g < G1; g += kFzThreads) {
      const int i0 = (b1 & ~3) + 4 * g;
      const int4 tk = __ldg(t4 + (i0 >> 2));
      const int tv[4] = {tk.x, tk.y, tk.z, tk.w};
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (i0 + j >= b1 && i0 + j < b1 + c1) emit1(i0 + j - b1, tv[j]);
    }
    auto emit_tr = [&](int v, uint32_t dd, float lmv) {  // a child that is not a level-1 label
      const int j = c1 + atomicAdd(&s_ext, 1);
      cl[j] = v;
      ca[j] = lmv + bscale * (float)dd;
      atomicOr(msk + (v >> 5), 1u << (v & 31));
    };
#pragma unroll
    for (int u = 0; u < kTrHeld; ++u) {
      if (trk[u] >= 0 && trv[u] >= 0 && trv[u] < V) {
        const uint32_t dd = (uint32_t)s_trr[trk[u]].z;
        if (dep[trv[u]] == dd && lmf[trv[u]] == 0) emit_tr(trv[u], dd, trl[u]);
      }
    }
    for (int k = 0; !tr_held && k < nt; ++k) {
      const int b = s_trr[k].x, c = s_trr[k].y;
      const uint32_t dd = (uint32_t)s_trr[k].z;
      for (int i = tid; i < c; i += kFzThreads) {
        const int v = __ldg(d.tr.ch_tok + b + i);
        if (!checked(v >= 0 && v < V, d.err, 15) || dep[v] != dd || lmf[v] != 0) continue;
        float lmv = 0.f;  // the LM term when the deepest arc is level 0's, or none
        if (d.has_lm) lmv = lam * ((dense ? __ldg(dense + v) : 0.f) + __ldg(d.lm.uni_logp + v));
        emit_tr(v, dd, lmv);
      }
    }
    if (tid == 0) atomicOr(msk + (V >> 5), 1u << (V & 31));  // blank is always evaluated by the row pass
    row::block_sync();
    uint32_t* mo = d.c_mask + (size_t)r * d.mask_words;
    for (int q = tid; q < d.mask_words; q += kFzThreads) mo[q] = msk[q];
    if (tid == 0) {
      const int n = c1 + s_ext;
      d.c_info[r] = make_int4(drow, n, __float_as_int(s_cr), 0);
      if (counting) s_bytes += 8ull * n + 4ull * d.mask_words + 16 + 8ull * s_ext;
    }
  }

  // 5. joint input of this step
  if (!PRED) row::build_joint_input(d, s_enc + ((size_t)r * T + t) * d.H, s_last, r);
  if (counting && tid == 0) atomicAdd(d.ctr, s_bytes + (PRED ? 0ull : 6ull * d.H));  // + frame, embedding row, A row
}

}  // namespace

size_t row_fused_smem_bytes(int V4, int N_pad) {
  return (size_t)V4 * (sizeof(uint32_t) + 2 * sizeof(uint8_t)) + 2 * sizeof(uint32_t) * (size_t)(N_pad / 32);
}

cudaError_t prepare_fused_kernels(size_t smem) {
  cudaError_t e = cudaFuncSetAttribute(k_row_ep<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_row_ep<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_row_ep<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(k_row_ep<5>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  return e;
}

void launch_row_fused(const DecView& d, int M, int step, int mode, size_t smem, cudaStream_t s, bool pdl) {
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
    if (few) cudaLaunchKernelEx(&cfg, k_row_ep<5>, d, step, mode);
    else cudaLaunchKernelEx(&cfg, k_row_ep<1>, d, step, mode);
  } else {
    if (few) cudaLaunchKernelEx(&cfg, k_row_ep<4>, d, step, mode);
    else cudaLaunchKernelEx(&cfg, k_row_ep<0>, d, step, mode);
  }
}

}  // namespace tsd
