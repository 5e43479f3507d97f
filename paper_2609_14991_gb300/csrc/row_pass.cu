// Row pass of the fused decode step with several n-gram LMs (Eq. 1, the sum
// over LMs): one CTA per hypothesis row.  (Greedy decoding with at most one
// LM runs row_fused.cu instead.)
//
// For row r at label step s it
//   1. combines the joint kernel's per-tile partials of step s-1 into the
//      log-sum-exp of the row and its best fused label (Eq. 1 argmax);
//   2. applies the greedy decision: blank (or the per-frame label limit)
//      advances the frame, a label is emitted and advances the LM state and
//      the phrase-trie state;
//   3. writes the joint input of step s, bf16(ReLU(enc_t + E[last])), and
//   4. the dense fusion bias of step s, lambda*log p_LM(v|state) +
//      beta*boost(v|trie state) for every label v (Eq. 1, terms 2 and 3).
//
// LM state and phrase state are both kept as their whole suffix chain (one
// LM state per order; every trie node that is a suffix of the current one),
// so the next chain after label y is assembled from independent searches of
// y in each chain element -- no dependent pointer chase.
#include <algorithm>

#include "row_common.cuh"

namespace tsd {

namespace {

using row::best_merge;
using row::kNegInf;
using row::lse_merge;
using row::warp_find;

// Algorithmic bytes of a row's LM chain levels: each level's state record
// and arcs, and (when a label was emitted) its search: one probe per halving
// plus the arc found.
__device__ unsigned long long lm_level_bytes(const row::ChainRecs& rc, int nl, bool searched) {
  unsigned long long b = 0;
  for (int l = 0; l < nl; ++l) {
    b += 12 + 8ull * rc.lc[l];
    if (searched) b += 8 + 4ull * (32 - __clz(rc.lc[l] + 1)) + 4;
  }
  return b;
}

// The fusion bias row with several LMs (Eq. 1, the sum over LMs): per LM its
// chain levels deepest first into the scratch (a label keeps the first value
// it gets), then acc[v] += alpha_i * (that value, or the backoff to the
// unigram: the chain's summed backoff weights + log p_i(v)); the trie as in
// the single-LM pass; brow[v] = acc[v] + beta * boost(v).  All threads of
// the block call it; it returns thread 0's count of LM bytes (if counting).
__device__ unsigned long long bias_multi(const DecView& d, int L, const int (*lm_chain)[kLmChain], const int* nl,
                                         const int* tr_chain, int nt, row::ChainRecs& rc, float lam, float beta,
                                         float* brow, float* lmv, float* acc, uint8_t* dep, bool counting,
                                         bool searched) {
  const int tid = threadIdx.x, step = blockDim.x, V = d.V, nq = d.V4 / 4;
  unsigned long long bytes = 0;
  if (tid >= 32 && tid - 32 < nt) {
    const int q = tr_chain[tid - 32];
    rc.tb[tid - 32] = __ldg(d.tr.nd_begin + q);
    rc.tc[tid - 32] = __ldg(d.tr.nd_count + q);
    rc.td[tid - 32] = __ldg(d.tr.nd_depth + q) + 1;
  }
  uint32_t* d4 = reinterpret_cast<uint32_t*>(dep);
  float4* l4 = reinterpret_cast<float4*>(lmv);
  float4* a4 = reinterpret_cast<float4*>(acc);
  for (int q = tid; q < nq; q += step) d4[q] = 0u;
  const float unset = row::unset_value();
  for (int m = 0; m < L; ++m) {
    const int n = nl[m];
    if (tid < n) {
      const int st = lm_chain[m][tid];
      rc.lb[tid] = __ldg(TSD_LMX(d, m, st_begin) + st);
      rc.lc[tid] = __ldg(TSD_LMX(d, m, st_count) + st);
      rc.lo[tid] = __ldg(TSD_LMX(d, m, st_cum) + st);
    }
    for (int q = tid; q < nq; q += step) l4[q] = make_float4(unset, unset, unset, unset);
    row::block_sync();
    const float cum_top = n ? rc.lo[n - 1] : 0.f;
    const int32_t* arc_tok = TSD_LMX(d, m, arc_tok);
    const float* arc_logp = TSD_LMX(d, m, arc_logp);
    for (int p = 0; p < n; ++p) {
      const int l = n - 1 - p;
      row::scatter_lm_level(arc_tok, arc_logp, rc.lb[l], rc.lb[l] + rc.lc[l], cum_top - rc.lo[l], lmv);
      row::block_sync();
    }
    if (counting && tid == 0) bytes += lm_level_bytes(rc, n, searched);
    const float alpha = lam * row::lm_pick(m, d.lm_w[0], d.lm_w[1], d.lm_w[2], d.lm_w[3]);
    const float4* u4 = reinterpret_cast<const float4*>(TSD_LMX(d, m, uni_logp));  // padded past V
    for (int q = tid; q < nq; q += step) {
      const float4 l = l4[q];
      const float4 u = __ldg(u4 + q);
      float4 a = (m == 0) ? make_float4(0.f, 0.f, 0.f, 0.f) : a4[q];
      a.x += alpha * (isnan(l.x) ? u.x + cum_top : l.x);
      a.y += alpha * (isnan(l.y) ? u.y + cum_top : l.y);
      a.z += alpha * (isnan(l.z) ? u.z + cum_top : l.z);
      a.w += alpha * (isnan(l.w) ? u.w + cum_top : l.w);
      a4[q] = a;
    }
    row::block_sync();  // the scratch and the records are reused by the next LM
  }
  for (int p = 0; p < nt; ++p) {
    const int k = nt - 1 - p;
    row::scatter_trie_node(d.tr.ch_tok, rc.tb[k], rc.tb[k] + rc.tc[k], (uint8_t)rc.td[k], dep);
    row::block_sync();
  }
  const int depth_cur = nt ? rc.td[0] - 1 : 0;
  const float bscale = beta * (d.has_tr ? d.tr.bonus : 0.f);
  const float tr_base = -bscale * (float)depth_cur;
  float4* b4 = reinterpret_cast<float4*>(brow);
  for (int q = tid; q < nq; q += step) {
    const float4 a = a4[q];
    const uint32_t dd = d4[q];
    const uint32_t rb = __ldg(d.droot + (q >> 3)) >> ((4 * q) & 31);
    const float av[4] = {a.x, a.y, a.z, a.w};
    float o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int dj = (dd >> (8 * j)) & 0xff;
      const float btr = dj ? bscale * (float)(dj - depth_cur) : (((rb >> j) & 1u) ? bscale : 0.f) + tr_base;
      o[j] = (4 * q + j < V) ? av[j] + btr : 0.f;
    }
    b4[q] = make_float4(o[0], o[1], o[2], o[3]);
  }
  if (tid == 0) brow[V] = 0.f;
  return bytes;
}

// mode: 0 = label step, 1 = final step (apply the last decision only),
// 2 = replay (redo the step's work without committing any state or output;
// used only to time the kernel in isolation).
// VAR bit 0: the stateful form (LSTM input rows instead of the joint input);
// bit 1: several LMs; bit 2: few rows (at most two CTAs per SM are needed,
// so the kernel may use registers freely instead of fitting seven per SM).
// Each combination is its own instantiation, so the common ones carry none
// of the other paths' code or registers.
template <int VAR>
__global__ void __launch_bounds__(kRowThreads, (VAR & 4) ? 2 : 7) k_row(DecView d, int step, int mode) {
  constexpr bool PRED = (VAR & 1) != 0, MULTI = (VAR & 2) != 0;
  const Params* __restrict__ P = d.params;
  const int r = blockIdx.x;
  const int V = d.V;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool commit = (mode != 2);
  extern __shared__ __align__(16) unsigned char smem[];
  // per-label scratch: LM value from the chain (NaN unset), with several LMs
  // also their weighted sum, then the trie depth of the goto
  const int L = (MULTI && d.n_lm > 1) ? d.n_lm : 1;  // LM state blocks (1 without an LM)
  float* lmv = reinterpret_cast<float*>(smem);
  float* acc = lmv + d.V4;
  uint8_t* dep = reinterpret_cast<uint8_t*>(lmv + (L > 1 ? 2 : 1) * d.V4);

  __shared__ int s_t, s_sym, s_cnt, s_y, s_tr_len, s_last, s_slot, s_T;
  __shared__ int s_lm_len[kMaxLm];
  // the call's parameters, read once before the dependency wait
  __shared__ int32_t* s_out_tok;
  __shared__ int32_t* s_out_frame;
  __shared__ float* s_out_score;
  __shared__ int32_t* s_out_count;
  __shared__ const uint16_t* s_enc;
  __shared__ float s_lam, s_beta;
  __shared__ int s_n;
  __shared__ float s_score;
  __shared__ int s_lm[kMaxLm][kLmChain], s_tr[kTrChain];
  __shared__ int s_lm_tgt[kMaxLm][kLmChain];    // target state of y's arc at each LM level (-2 none)
  __shared__ int s_tr_node[kTrChain], s_tr_nxt[kTrChain];  // child by y of each trie chain node (-1 none)
  __shared__ int s_uni_tgt[kMaxLm], s_root_child, s_root_next;
  __shared__ row::ChainRecs rc;   // records of the chains the bias row is built from
  __shared__ row::ChainRecs rco;  // one LM: records of the current chains, kept with the state

  // The row state below was written by the previous row pass; under
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
    if (step == 0) {
      s_t = 0; s_sym = 0; s_cnt = 0;
    } else {
      s_t = __ldcg(d.r_t + r); s_sym = __ldcg(d.r_sym + r); s_cnt = __ldcg(d.r_cnt + r);
    }
    for (int i = 0; i < L; ++i) s_lm_len[i] = d.has_lm ? __ldcg(d.s_lm_len + i * d.lm_stride + slot) : 0;
    s_tr_len = d.has_tr ? __ldcg(d.s_tr_len + slot) : 0;
    s_last = __ldcg(d.s_last + slot);
  }
  row::block_sync();
  const int slot = s_slot, T = s_T;
  if (tid < L * kLmChain) {
    const int i = tid / kLmChain, l = tid % kLmChain;
    if (l < s_lm_len[i]) {
      s_lm[i][l] = __ldcg(d.s_lm_chain + ((size_t)i * d.lm_stride + slot) * kLmChain + l);
      if (L == 1) {
        const int4 q = __ldcg(d.s_lm_rec + (size_t)slot * kLmChain + l);
        rco.lb[l] = q.x;
        rco.lc[l] = q.y;
      }
    }
  }
  if (tid >= 64 && tid - 64 < s_tr_len) {
    const int k = tid - 64;
    s_tr[k] = __ldcg(d.s_tr_chain + slot * kTrChain + k);
    if (L == 1) {
      const int4 q = __ldcg(d.s_tr_rec + (size_t)slot * kTrChain + k);
      rco.tb[k] = q.x;
      rco.tc[k] = q.y;
    }
  }
  // The encoder frames this step can use (t, or t+1 after a frame advance)
  // go to L1 now, while the previous kernel still runs: no kernel of the
  // chunk writes them.  (The call's bias defaults are not prefetched: every
  // row would ask the same L2 lines for them at once.)
  if (s_t < T) {
    const size_t fb = (size_t)d.H * 2;
    const uint16_t* f0 = s_enc + ((size_t)r * T + s_t) * d.H;
    row::prefetch_span(f0, s_t + 1 < T ? 2 * fb : fb, 0);
  }
  row::block_sync();
  // In replay mode every row redoes a full step (decision, advance, joint
  // input, bias) even if it had finished the chunk, so the timing is that of
  // a mid-chunk step.
  const bool evaluated = (step > 0) && (s_t < T || !commit);
  // Programmatic dependent launch: everything above reads only state the
  // previous row pass wrote, which had completed before the joint kernel in
  // between let this grid launch; the joint's partials need the wait.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (evaluated) {
    // 1. combine the partials of the previous joint step
    if (warp == 0) {
      float m = kNegInf, s = 0.f, bv = kNegInf;
      int bi = INT_MAX;
      const float4* pr = d.part + (size_t)r * d.n_ptiles;
      for (int j = lane; j < d.n_ptiles; j += 32) {
        float4 p = __ldcg(pr + j);  // written by the joint kernel just before
        lse_merge(m, s, p.x, p.y);
        best_merge(bv, bi, p.z, __float_as_int(p.w));
      }
      row::reconverge();
      for (int o = 16; o > 0; o >>= 1) {
        float m2 = __shfl_xor_sync(0xffffffffu, m, o);
        float s2 = __shfl_xor_sync(0xffffffffu, s, o);
        float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
        int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
        lse_merge(m, s, m2, s2);
        best_merge(bv, bi, v2, i2);
      }
      if (lane == 0) {
        s_y = (bi >= 0 && bi <= V) ? bi : V;
        s_score = bv - (m + logf(s));
      }
    }
    row::block_sync();
    const int y = s_y;
    row::prefetch_span(d.E + (size_t)(y != V ? y : s_last) * d.H, (size_t)d.H * 2, 32);  // this step's E row
    if (y != V) {
      // 2a. independent searches of y in every chain element, each warp
      //     also fetching what the new chain needs from the arc it found
      int nl = 0;  // chain elements over all LMs
      for (int i = 0; i < L; ++i) nl += s_lm_len[i];
      const int nt = s_tr_len;
      if (tid == kRowThreads - 1) {
        s_root_child = d.has_tr ? __ldg(d.tr.root_child + y) : 0;
        s_root_next = d.has_tr ? __ldg(d.tr.root_next + y) : 0;
      } else if (tid >= kRowThreads - 1 - L) {
        const int i = tid - (kRowThreads - 1 - L);
        s_uni_tgt[i] = (d.has_lm && TSD_LMX(d, i, order) >= 2) ? __ldg(TSD_LMX(d, i, uni_tgt) + y) : -1;
      }
      for (int task = warp; task < nl + nt; task += kRowThreads / 32) {
        if (task < nl) {
          int m = 0, l = task;  // LM m, level l
          while (l >= s_lm_len[m]) l -= s_lm_len[m++];
          const int32_t* st_begin = TSD_LMX(d, m, st_begin);
          const int32_t* st_count = TSD_LMX(d, m, st_count);
          const int32_t* arc_tgt = TSD_LMX(d, m, arc_tgt);
          int b, c;
          if (L == 1) {  // records kept with the chain
            b = rco.lb[l];
            c = rco.lc[l];
          } else {
            const int st = s_lm[m][l];
            b = __ldg(st_begin + st);
            c = __ldg(st_count + st);
          }
          int i = warp_find(TSD_LMX(d, m, arc_tok) + b, c, y, lane);
          if (lane == 0) {
            const int tg = (i >= 0) ? __ldg(arc_tgt + b + i) : -2;
            s_lm_tgt[m][l] = tg;
            if (tg >= 0) {  // the new chain's state records
              row::prefetch_l1(st_begin + tg);
              row::prefetch_l1(st_count + tg);
              row::prefetch_l1(TSD_LMX(d, m, st_cum) + tg);
            }
          }
        } else {
          int k = task - nl;
          int b, c;
          if (L == 1) {
            b = rco.tb[k];
            c = rco.tc[k];
          } else {
            const int q = s_tr[k];
            b = __ldg(d.tr.nd_begin + q);
            c = __ldg(d.tr.nd_count + q);
          }
          int i = warp_find(d.tr.ch_tok + b, c, y, lane);
          if (lane == 0) {
            s_tr_node[k] = (i >= 0) ? __ldg(d.tr.ch_node + b + i) : -1;
            if (i >= 0) {
              const int nd = s_tr_node[k];
              row::prefetch_l1(d.tr.nd_begin + nd);
              row::prefetch_l1(d.tr.nd_count + nd);
              row::prefetch_l1(d.tr.nd_depth + nd);
            }
            s_tr_nxt[k] = (i >= 0) ? __ldg(d.tr.ch_next + b + i) : -1;
          }
        }
      }
      row::block_sync();
      // 2b. assemble the new chains (shared memory only) and emit
      if (tid == 0) {
        // each LM: y's unigram state, then the target of y's arc at every
        // level of the old chain up to the first level without one (the old
        // chain's arc targets are in s_lm_tgt, so the new chain is written
        // over the old one in place)
        for (int m = 0; m < L; ++m) {
          const int nold = s_lm_len[m];
          int ln = 0;
          if (s_uni_tgt[m] >= 0) {
            s_lm[m][ln++] = s_uni_tgt[m];
            for (int l = 0; l < nold && ln < kLmChain; ++l) {
              const int tgt = s_lm_tgt[m][l];
              if (tgt < 0) break;  // no arc at this level (-2) or the top order (-1)
              s_lm[m][ln++] = tgt;
            }
          }
          s_lm_len[m] = ln;
          if (commit) {
            int32_t* ch = d.s_lm_chain + ((size_t)m * d.lm_stride + slot) * kLmChain;
            for (int l = 0; l < ln; ++l) ch[l] = s_lm[m][l];
            if (d.has_lm) d.s_lm_len[m * d.lm_stride + slot] = ln;
          }
        }
        int tn = 0;
        bool reset = false;
        for (int i = 0; i < nt; ++i) {
          if (s_tr_node[i] < 0) continue;
          if (tn == 0 && s_tr_nxt[i] == 0) reset = true;
          if (tn < kTrChain) s_tr[tn++] = s_tr_node[i];
        }
        if (s_root_child != 0) {
          if (tn == 0 && s_root_next == 0) reset = true;
          if (tn < kTrChain) s_tr[tn++] = s_root_child;
        }
        if (reset) tn = 0;
        s_tr_len = tn;
        if (commit) {
          for (int l = 0; l < tn; ++l) d.s_tr_chain[slot * kTrChain + l] = s_tr[l];
          if (d.has_tr) d.s_tr_len[slot] = tn;
          const int cap = T * d.max_sym;
          const int o = r * cap + s_cnt;
          s_out_tok[o] = y;
          s_out_frame[o] = s_t;
          s_out_score[o] = s_score;
          d.s_last[slot] = y;
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
    // the chunk's last decision: the new chains' records for the next chunk
    if (L == 1 && commit) {
      if (tid < s_lm_len[0]) {
        const int st = s_lm[0][tid];
        d.s_lm_rec[(size_t)slot * kLmChain + tid] =
            make_int4(__ldg(d.lm.st_begin + st), __ldg(d.lm.st_count + st), __float_as_int(__ldg(d.lm.st_cum + st)), 0);
      }
      if (tid >= 64 && tid - 64 < s_tr_len) {
        const int q = s_tr[tid - 64];
        d.s_tr_rec[(size_t)slot * kTrChain + tid - 64] =
            make_int4(__ldg(d.tr.nd_begin + q), __ldg(d.tr.nd_count + q), __ldg(d.tr.nd_depth + q) + 1, 0);
      }
    }
    if (tid == 0) s_out_count[r] = s_cnt;
    return;
  }
  if (tid == 0 && commit) {
    d.r_t[r] = s_t;
    d.r_sym[r] = s_sym;
    d.r_cnt[r] = s_cnt;
  }
  const int t = commit ? s_t : min(s_t, T - 1);
  if (d.cap_rows && step < d.cap_steps && tid == 0 && commit) {
    int* c = d.cap_rows + ((size_t)step * s_n + r) * 4;
    if (t < T) {
      c[0] = t;
      c[1] = s_last;
      c[2] = s_lm_len[0] ? s_lm[0][s_lm_len[0] - 1] : 0;
      c[3] = s_tr_len ? s_tr[0] : 0;
    } else {
      c[0] = -1; c[1] = -1; c[2] = -1; c[3] = -1;
    }
  }
  if (t >= T) return;

  // 3. records of the new chains, scratch reset; 4. joint input of this
  // step (its loads overlap the records); 5. the fusion bias row
  const int nt = s_tr_len;
  const bool counting = (mode == 2 || d.count);
  unsigned long long lm_bytes = 0;  // thread 0: LM levels' records, arcs and searches
  int nl = s_lm_len[0];
  if (L == 1) {
    row::bias_prepare(d, s_lm[0], nl, s_tr, nt, rc, lmv, dep);
    if (commit) {  // the records stay with the chains for the next step's searches
      if (tid < nl) d.s_lm_rec[(size_t)slot * kLmChain + tid] = make_int4(rc.lb[tid], rc.lc[tid], __float_as_int(rc.lo[tid]), 0);
      if (tid >= 32 && tid - 32 < nt)
        d.s_tr_rec[(size_t)slot * kTrChain + tid - 32] = make_int4(rc.tb[tid - 32], rc.tc[tid - 32], rc.td[tid - 32], 0);
    }
    if (!PRED) row::build_joint_input(d, s_enc + ((size_t)r * T + t) * d.H, s_last, r);
    row::bias_finish(d, nl, nt, rc, s_lam, s_beta, d.bias + (size_t)r * d.N_pad, lmv, dep);
    if (counting && tid == 0) lm_bytes = lm_level_bytes(rc, nl, s_y != V && evaluated);
  } else if (MULTI) {
    if (!PRED) row::build_joint_input(d, s_enc + ((size_t)r * T + t) * d.H, s_last, r);
    lm_bytes = bias_multi(d, L, s_lm, s_lm_len, s_tr, nt, rc, s_lam, s_beta, d.bias + (size_t)r * d.N_pad, lmv,
                          acc, dep, counting, s_y != V && evaluated);
    nl = 0;
    for (int i = 0; i < L; ++i) nl += s_lm_len[i];
  }
  if (counting && tid == 0) {
    // Algorithmic bytes of this row-step: selection partials, row state,
    // the searches of the emitted label (one probe per halving plus the arc
    // it found), the joint input (encoder frame and embedding row read, A
    // row written), and every arc of every chain level and trie chain node
    // with its state record.  The dense bias row written for the GEMM
    // epilogue and the shared unigram/root rows are not counted here.
    unsigned long long bytes = (unsigned long long)d.n_ptiles * 16 + 2ull * (24 + 4 * (nl + nt));
    bytes += 6ull * d.H + lm_bytes;
    for (int k = 0; k < nt; ++k) bytes += 12 + 4ull * rc.tc[k];
    if (s_y != V && evaluated)
      for (int k = 0; k < nt; ++k) bytes += 8 + 4ull * (32 - __clz(rc.tc[k] + 1)) + 8;
    atomicAdd(d.ctr, bytes);
  }
}

// After a chain is written from the host: its elements' table records.
__global__ void k_fix_records(DecView d, int slot) {
  const int l = threadIdx.x;
  if (d.has_lm && l < kLmChain && l < d.s_lm_len[slot]) {
    const int st = d.s_lm_chain[(size_t)slot * kLmChain + l];
    // the fourth field of the first (unigram) level: its dense row, if any
    const int dense = (l == 0 && d.lm.order >= 2 && st >= 1 && st <= d.V) ? d.lm.uni_dense[st - 1] : -1;
    d.s_lm_rec[(size_t)slot * kLmChain + l] =
        make_int4(d.lm.st_begin[st], d.lm.st_count[st], __float_as_int(d.lm.st_cum[st]), dense);
  }
  if (d.has_tr && l < kTrChain && l < d.s_tr_len[slot]) {
    const int q = d.s_tr_chain[(size_t)slot * kTrChain + l];
    d.s_tr_rec[(size_t)slot * kTrChain + l] = make_int4(d.tr.nd_begin[q], d.tr.nd_count[q], d.tr.nd_depth[q] + 1, 0);
  }
}

__global__ void k_open(DecView d, int slot) {
  if (threadIdx.x == 0) {
    d.s_last[slot] = d.V;
    for (int i = 0; i < (d.n_lm > 1 ? d.n_lm : 1); ++i) d.s_lm_len[i * d.lm_stride + slot] = 0;
    d.s_tr_len[slot] = 0;
  }
}

__global__ void k_repack(const uint16_t* __restrict__ W, uint16_t* __restrict__ Wt, int H, int N, int N_pad) {
  __shared__ uint16_t tile[32][33];
  int k0 = blockIdx.y * 32, v0 = blockIdx.x * 32;
  int tx = threadIdx.x, ty = threadIdx.y;  // 32 x 8
  for (int i = ty; i < 32; i += 8) {
    int k = k0 + i, v = v0 + tx;
    tile[i][tx] = (k < H && v < N) ? W[(size_t)k * N + v] : (uint16_t)0;
  }
  row::block_sync();
  for (int i = ty; i < 32; i += 8) {
    int v = v0 + i, k = k0 + tx;
    if (v < N_pad && k < H) Wt[(size_t)v * H + k] = tile[tx][i];
  }
}

}  // namespace

size_t row_smem_bytes(int V4, int n_lm) {
  return (size_t)V4 * ((n_lm > 1 ? 2 : 1) * sizeof(float) + sizeof(uint8_t));
}


namespace {
// Per-call defaults of the fusion bias, which the row pass combines with
// the row's own terms: lambda * log p(v) for every label (0 past V), and a
// bitmask of the labels the trie root has a child for.  One small launch at
// the start of every chunk.
__global__ void k_defaults(DecView d) {
  const Params* P = d.params;
  const float lam = P->lambda;
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < d.V4) d.dflt[i] = (d.has_lm && i < d.V) ? lam * __ldg(d.lm.uni_logp + i) : 0.f;
  if (d.fused && i < d.N_pad) {
    // the defaults the joint kernel adds to its logits (0 from blank on)
    float x = 0.f;
    if (i < d.V) {
      if (d.has_lm) x = lam * __ldg(d.lm.uni_logp + i);
      if (d.has_tr && __ldg(d.tr.root_child + i) != 0) x += P->beta * d.tr.bonus;
    }
    d.dvec[i] = x;
  }

  if (i < (d.V4 + 31) / 32) {
    uint32_t m = 0;
    if (d.has_tr)
      for (int b = 0; b < 32; ++b) {
        const int v = i * 32 + b;
        if (v < d.V && __ldg(d.tr.root_child + v) != 0) m |= 1u << b;
      }
    d.droot[i] = m;
  }
}
}  // namespace

void launch_defaults(const DecView& d, cudaStream_t s) {
  k_defaults<<<(std::max(d.V4, d.N_pad) + 255) / 256, 256, 0, s>>>(d);
}

cudaError_t prepare_kernels(size_t row_smem) {
  // dynamic scratch plus the kernel's static shared memory may pass the
  // 48 KB default even when the scratch alone does not
  return cudaFuncSetAttribute(k_row<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)row_smem);
}

void launch_repack(const uint16_t* W, uint16_t* Wt, int H, int N, int N_pad, cudaStream_t s) {
  dim3 grid((N_pad + 31) / 32, (H + 31) / 32), block(32, 8);
  k_repack<<<grid, block, 0, s>>>(W, Wt, H, N, N_pad);
}

void launch_open(const DecView& d, int slot, cudaStream_t s) { k_open<<<1, 32, 0, s>>>(d, slot); }

void launch_fix_records(const DecView& d, int slot, cudaStream_t s) { k_fix_records<<<1, 32, 0, s>>>(d, slot); }

namespace {
// Stateful form, stream open: zero LSTM state, the start-of-sequence step pending.
__global__ void k_open_pred(DecView d, int slot) {
  const int D = d.pred_D;
  for (int u = threadIdx.x; u < D; u += blockDim.x) {
    d.pred_h[(size_t)slot * D + u] = 0;
    d.pred_c[(size_t)slot * D + u] = 0.f;
  }
  if (threadIdx.x == 0) d.pred_fresh[slot] = 1;
}

// Stateful form: the chunk's encoder frames (from the call's parameter
// block) to the fixed buffer the projection GEMM reads by TMA.
__global__ void k_copy_enc(DecView d, int64_t n16) {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const uint4* src = reinterpret_cast<const uint4*>(d.params->enc);
  uint4* dst = reinterpret_cast<uint4*>(d.pred_enc);
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += (int64_t)gridDim.x * blockDim.x)
    dst[i] = __ldg(src + i);
}
}  // namespace

void launch_open_pred(const DecView& d, int slot, cudaStream_t s) { k_open_pred<<<1, 256, 0, s>>>(d, slot); }

void launch_copy_enc(const DecView& d, int64_t elems, cudaStream_t s, bool pdl) {
  const int64_t n16 = elems / 8;  // H_enc is a multiple of 64
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)std::min<int64_t>((n16 + 255) / 256, 152 * 8));
  cfg.blockDim = dim3(256);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  cudaLaunchKernelEx(&cfg, k_copy_enc, d, n16);
}

void launch_row(const DecView& d, int M, int step, int mode, size_t smem, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(M);
  cfg.blockDim = dim3(kRowThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  // greedy decoding with at most one LM runs k_row_fz (row_fused.cu); this
  // pass serves several LMs (the stateful form takes one LM)
  cudaLaunchKernelEx(&cfg, k_row<2>, d, step, mode);
}

}  // namespace tsd
