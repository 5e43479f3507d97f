// Beam-search row pass: one cluster of K CTAs per stream, K hypotheses per
// stream.  The cluster's first CTA does steps 1-5; then every CTA k of the
// cluster builds step 6 for beam member k, reading its chains from the
// first CTA's shared memory.
//
// The search is frame-synchronous with at most S = max_symbols labels per
// frame: each label step is one expansion of the hypotheses still in their
// frame (set A).  At a step the first CTA
//   1. turns the joint kernel's per-tile partials into each hypothesis of A's
//      log-sum-exp and its K best extensions (blank keeps the labels, label v
//      appends v), scored hypothesis score + fused value - log-sum-exp (Eq. 1
//      summed along the hypothesis);
//   2. keeps the top K of those candidates by (score desc, hypothesis asc,
//      label asc) and sends each, in that order, to the frame-exit set F
//      (the blank, or a label at the frame's S-th expansion) or to the next A,
//      merging equal label sequences within a set by log-sum-exp of their
//      scores (F also holds the earlier expansions' exits);
//   3. searches each new label in its parent's LM and phrase-trie suffix
//      chains (independent per-level searches, as in the greedy pass);
//   4. builds the new hypotheses' chains;
//   5. keeps F's K best in insertion order; when A is empty or the S-th
//      expansion is done the frame ends and F is the beam of the next frame;
//      commits the beam, F and the stream's frame and expansion counters.
// With S = 1 every kept candidate leaves the frame: one label or blank per
// frame, the top K of the K (V+1) extensions merged.
// Label sequences live in a per-stream pool of (parent, label) nodes; two
// candidates are the same sequence when their lengths and rolling hashes
// agree and their node chains compare equal label by label.
#include <cooperative_groups.h>

#include "row_common.cuh"

namespace tsd {

namespace {

using row::kNegInf;
using row::lse_merge;
using row::warp_find;

constexpr int kMaxK = 8;
constexpr int kCandPerLane = 16;  // per-hypothesis candidates: n_tiles * K <= 512

__device__ __forceinline__ unsigned long long hash_push(unsigned long long h, int v) {
  return h * 0x100000001B3ull + (unsigned long long)(v + 1);
}

// The label sequences of pool nodes x and y are equal (-1 = empty sequence).
__device__ bool nodes_equal(const int32_t* par, const int32_t* tok, int x, int y, int cap) {
  for (int i = 0; i <= cap && x != y; ++i) {
    if (x < 0 || y < 0) return false;
    if (__ldcg(tok + x) != __ldcg(tok + y)) return false;
    x = __ldcg(par + x);
    y = __ldcg(par + y);
  }
  return x == y;
}

// seq(a) [+ label ea if ea >= 0] equals seq(b) [+ eb].
__device__ bool seq_equal(const int32_t* par, const int32_t* tok, int a, int ea, int b, int eb, int cap) {
  if (ea >= 0 && eb >= 0) return ea == eb && nodes_equal(par, tok, a, b, cap);
  if (ea < 0 && eb < 0) return nodes_equal(par, tok, a, b, cap);
  if (ea < 0) {
    if (a < 0 || __ldcg(tok + a) != eb) return false;
    return nodes_equal(par, tok, __ldcg(par + a), b, cap);
  }
  if (b < 0 || __ldcg(tok + b) != ea) return false;
  return nodes_equal(par, tok, a, __ldcg(par + b), cap);
}

__device__ __forceinline__ double log_add(double a, double b) {
  const double m = fmax(a, b);
  return m + log(exp(a - m) + exp(b - m));
}

// candidate order: score desc, hypothesis asc, label asc
__device__ __forceinline__ bool cand_before(double s1, int h1, int t1, double s2, int h2, int t2) {
  if (s1 != s2) return s1 > s2;
  if (h1 != h2) return h1 < h2;
  return t1 < t2;
}

// mode: 0 = label step, 1 = final step (apply the last frame's selection),
// 2 = replay (redo the step without committing anything; for timing).
// MS: several labels per frame (max_symbols > 1); without it the frame-exit
// set and the expansion counter fold away at compile time.
template <bool MS>
__global__ void __launch_bounds__(kRowThreads) k_row_beam(DecView d, int step, int mode) {
  const Params* __restrict__ P = d.params;
  cooperative_groups::cluster_group cluster = cooperative_groups::this_cluster();
  const int K = d.K, V = d.V;
  const int b = blockIdx.x / K;                 // stream of this cluster
  const int crank = (int)cluster.block_rank();  // survivor this CTA builds (step 4)
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool commit = (mode != 2);
  extern __shared__ __align__(16) unsigned char smem[];
  float* lmv = reinterpret_cast<float*>(smem);
  uint8_t* dep = reinterpret_cast<uint8_t*>(lmv + d.V4);

  __shared__ int s_slot, s_T;
  __shared__ int o_live[kMaxK], o_last[kMaxK], o_node[kMaxK], o_len[kMaxK], o_lml[kMaxK], o_trl[kMaxK];
  __shared__ double o_score[kMaxK];
  __shared__ unsigned long long o_hash[kMaxK];
  __shared__ int o_lm[kMaxK][kLmChain], o_tr[kMaxK][kTrChain];
  __shared__ int n_cnt;
  __shared__ int n_par[kMaxK], n_tok[kMaxK], n_node[kMaxK], n_len[kMaxK], n_lml[kMaxK], n_trl[kMaxK], n_last[kMaxK];
  __shared__ double n_score[kMaxK];
  __shared__ unsigned long long n_hash[kMaxK];
  __shared__ int n_lm[kMaxK][kLmChain], n_tr[kMaxK][kTrChain];
  __shared__ double c_score[kMaxK * kMaxK];
  __shared__ float c_inc[kMaxK * kMaxK];
  __shared__ int c_tok[kMaxK * kMaxK];
  __shared__ int s_sel[kMaxK], s_into[kMaxK];
  __shared__ int s_task0[kMaxK + 1];
  __shared__ int sr_lm[kMaxK][kLmChain];
  __shared__ int sr_trn[kMaxK][kTrChain], sr_trx[kMaxK][kTrChain];
  __shared__ int sr_uni[kMaxK], sr_rc[kMaxK], sr_rn[kMaxK];
  __shared__ row::ChainRecs rc;

  // frame-exit set F as loaded (entries of earlier expansions of this frame)
  __shared__ int e_cnt, e_node[kMaxK], e_len[kMaxK], e_last[kMaxK], e_lml[kMaxK], e_trl[kMaxK];
  __shared__ double e_score[kMaxK];
  __shared__ unsigned long long e_hash[kMaxK];
  __shared__ int e_lm[kMaxK][kLmChain], e_tr[kMaxK][kTrChain];
  __shared__ int n_dst[kMaxK];  // new record goes to F (1) or stays in the frame (0)
  // the beam after this step (its members' joint inputs and bias rows are built)
  __shared__ int a_cnt, a_build, a_frame;
  __shared__ int a_node[kMaxK], a_len[kMaxK], a_last[kMaxK], a_lml[kMaxK], a_trl[kMaxK];
  __shared__ double a_score[kMaxK];
  __shared__ unsigned long long a_hash[kMaxK];
  __shared__ int a_lm[kMaxK][kLmChain], a_tr[kMaxK][kTrChain];
  __shared__ int f_cnt, f_src[kMaxK];  // F after this step: entry (>= 0 new record j, <= -2 loaded entry -2-j)
  __shared__ int q_src[2 * kMaxK];     // F before pruning, in insertion order
  __shared__ double q_score[2 * kMaxK];
  __shared__ int s_bt, s_be, s_done;

  __shared__ int m_cnt, m_lml, m_trl, m_last, m_frame;  // member crank, copied from the first CTA
  __shared__ int m_lm[kLmChain], m_tr[kTrChain];
  if (crank == 0) {
  // previous state of this stream's hypotheses (written by the previous row
  // pass; L2-only loads, see the greedy pass)
  if (tid == 0) {
    s_slot = __ldcg(P->slots + b);
    s_T = __ldcg(&P->T);
  }
  row::block_sync();
  const int slot = s_slot, T = s_T;
  const int hb = slot * K;
  const int cap = d.pool_cap;
  const int32_t* pool_par = d.pool_parent + (size_t)slot * cap;
  const int32_t* pool_tok = d.pool_tok + (size_t)slot * cap;
  if (tid < K) {
    const int h = hb + tid;
    o_live[tid] = __ldcg(d.h_live + h);
    o_last[tid] = __ldcg(d.s_last + h);
    o_node[tid] = __ldcg(d.h_node + h);
    o_len[tid] = __ldcg(d.h_len + h);
    o_score[tid] = __ldcg(d.h_score + h);
    o_hash[tid] = __ldcg(d.h_hash + h);
    o_lml[tid] = d.has_lm ? __ldcg(d.s_lm_len + h) : 0;
    o_trl[tid] = d.has_tr ? __ldcg(d.s_tr_len + h) : 0;
  }
  if (tid == K) {
    // frame and expansion of this stream (reset at the chunk's first step;
    // a replay redoes one expansion of the final beam)
    s_bt = (step == 0 || mode == 2) ? 0 : __ldcg(d.b_frame + slot);
    s_be = (step == 0 || mode == 2) ? 0 : __ldcg(d.b_exp + slot);
    s_done = (step > 0 && mode != 2 && s_bt >= T) ? 1 : 0;
    e_cnt = 0;
  }
  row::block_sync();
  for (int i = tid; i < K * kLmChain; i += kRowThreads) {
    const int k = i / kLmChain, l = i % kLmChain;
    if (l < o_lml[k]) o_lm[k][l] = __ldcg(d.s_lm_chain + (size_t)(hb + k) * kLmChain + l);
  }
  for (int i = tid; i < K * kTrChain; i += kRowThreads) {
    const int k = i / kTrChain, l = i % kTrChain;
    if (l < o_trl[k]) o_tr[k][l] = __ldcg(d.s_tr_chain + (size_t)(hb + k) * kTrChain + l);
  }
  const int S = MS ? d.max_sym : 1;
  if (S > 1 && step > 0 && !s_done && s_be > 0) {
    // F holds the exits of this frame's earlier expansions
    if (tid < K) {
      const int h = hb + tid;
      const int live = __ldcg(d.f_live + h);
      if (live) {
        e_node[tid] = __ldcg(d.f_node + h);
        e_len[tid] = __ldcg(d.f_len + h);
        e_last[tid] = __ldcg(d.f_last + h);
        e_score[tid] = __ldcg(d.f_score + h);
        e_hash[tid] = __ldcg(d.f_hash + h);
        e_lml[tid] = __ldcg(d.f_lml + h);
        e_trl[tid] = __ldcg(d.f_trl + h);
      }
      if (live) atomicAdd(&e_cnt, 1);  // F is stored compact: live entries first
    }
    row::block_sync();
    for (int i = tid; i < K * kLmChain; i += kRowThreads) {
      const int k = i / kLmChain, l = i % kLmChain;
      if (k < e_cnt && l < e_lml[k]) e_lm[k][l] = __ldcg(d.f_lmc + (size_t)(hb + k) * kLmChain + l);
    }
    for (int i = tid; i < K * kTrChain; i += kRowThreads) {
      const int k = i / kTrChain, l = i % kTrChain;
      if (k < e_cnt && l < e_trl[k]) e_tr[k][l] = __ldcg(d.f_trc + (size_t)(hb + k) * kTrChain + l);
    }
  }
  row::block_sync();
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (step > 0 && !s_done) {
    // 1. per live hypothesis (warp k): log-sum-exp and its K best extensions
    if (warp < K) {
      const int k = warp;
      const bool live = o_live[k] != 0;
      const int r = b * K + k;
      const float2* bp = d.bpart + (size_t)r * d.n_ptiles * (1 + K);
      float m = kNegInf, s = 0.f;
      if (live) {
        for (int j = lane; j < d.n_ptiles; j += 32) {
          const float2 p = __ldcg(bp + (size_t)j * (1 + K));
          lse_merge(m, s, p.x, p.y);
        }
      }
      row::reconverge();
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
        lse_merge(m, s, m2, s2);
      }
      const float lse = m + logf(s);
      float cv[kCandPerLane];
      int ct[kCandPerLane];
      const int nc = live ? d.n_ptiles * K : 0;
#pragma unroll
      for (int q = 0; q < kCandPerLane; ++q) {
        const int i = lane + 32 * q;
        cv[q] = kNegInf;
        ct[q] = INT_MAX;
        if (i < nc) {
          const float2 p = __ldcg(bp + (size_t)(i / K) * (1 + K) + 1 + (i % K));
          cv[q] = p.x;
          ct[q] = __float_as_int(p.y);
        }
      }
      for (int round = 0; round < K; ++round) {
        row::reconverge();
        // this lane's best remaining (value desc, label asc)
        float bv = kNegInf;
        int bt = INT_MAX, bq = -1;
#pragma unroll
        for (int q = 0; q < kCandPerLane; ++q)
          if (cv[q] > bv || (cv[q] == bv && cv[q] != kNegInf && ct[q] < bt)) { bv = cv[q]; bt = ct[q]; bq = q; }
        float wv = bv;
        int wt = bt, wl = lane;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          const float v2 = __shfl_xor_sync(0xffffffffu, wv, o);
          const int t2 = __shfl_xor_sync(0xffffffffu, wt, o), l2 = __shfl_xor_sync(0xffffffffu, wl, o);
          if (v2 > wv || (v2 == wv && (t2 < wt || (t2 == wt && l2 < wl)))) { wv = v2; wt = t2; wl = l2; }
        }
        if (lane == wl && bq >= 0) {
#pragma unroll
          for (int q = 0; q < kCandPerLane; ++q)
            if (q == bq) cv[q] = kNegInf;
        }
        if (lane == 0) {
          const int c = k * K + round;
          const bool valid = wv != kNegInf && wt >= 0 && wt <= V;
          c_tok[c] = valid ? wt : -1;
          c_inc[c] = valid ? wv - lse : 0.f;
          c_score[c] = valid ? o_score[k] + (double)(wv - lse) : -1e300;
        }
      }
    }
    row::block_sync();
    // 2. global top K, then merge equal label sequences
    if (tid == 0) {
      bool used[kMaxK * kMaxK];
      for (int c = 0; c < K * K; ++c) used[c] = false;
      int nsel = 0;
      for (int round = 0; round < K; ++round) {
        int best = -1;
        for (int c = 0; c < K * K; ++c) {
          if (used[c] || c_tok[c] < 0) continue;
          if (best < 0 || cand_before(c_score[c], c / K, c_tok[c], c_score[best], best / K, c_tok[best])) best = c;
        }
        if (best < 0) break;
        used[best] = true;
        s_sel[nsel++] = best;
      }
      const bool last_exp = s_be >= S - 1;
      int cnt = 0;
      int pool_used = __ldcg(d.pool_n + slot);
      for (int i = 0; i < nsel; ++i) {
        const int c = s_sel[i], p = c / K, y = c_tok[c];
        const int dst = (y == V || last_exp) ? 1 : 0;
        const int len = o_len[p] + (y != V ? 1 : 0);
        const unsigned long long hsh = (y != V) ? hash_push(o_hash[p], y) : o_hash[p];
        int into = -1;
        if (dst == 1) {
          for (int j = 0; j < e_cnt; ++j) {
            if (e_len[j] != len || e_hash[j] != hsh) continue;
            if (seq_equal(pool_par, pool_tok, o_node[p], y != V ? y : -1, e_node[j], -1, cap)) {
              into = -2 - j;
              break;
            }
          }
        }
        if (into == -1) {
          for (int j = 0; j < cnt; ++j) {
            if (n_dst[j] != dst || n_len[j] != len || n_hash[j] != hsh) continue;
            const int pj = n_par[j];
            if (seq_equal(pool_par, pool_tok, o_node[p], y != V ? y : -1, o_node[pj], n_tok[j] != V ? n_tok[j] : -1,
                          cap)) {
              into = j;
              break;
            }
          }
        }
        if (into <= -2) {
          e_score[-2 - into] = log_add(e_score[-2 - into], c_score[c]);
        } else if (into >= 0) {
          n_score[into] = log_add(n_score[into], c_score[c]);
        } else {
          into = cnt++;
          n_par[into] = p;
          n_tok[into] = y;
          n_score[into] = c_score[c];
          n_len[into] = len;
          n_hash[into] = hsh;
          n_dst[into] = dst;
        }
        s_into[i] = into;
      }
      // label-sequence nodes of the survivors that appended a label
      for (int j = 0; j < cnt; ++j) {
        const int p = n_par[j];
        if (n_tok[j] == V) {
          n_node[j] = o_node[p];
        } else if (pool_used < cap) {
          n_node[j] = pool_used;
          if (commit) {
            d.pool_parent[(size_t)slot * cap + pool_used] = o_node[p];
            d.pool_tok[(size_t)slot * cap + pool_used] = n_tok[j];
          }
          ++pool_used;
        } else {
          n_node[j] = o_node[p];  // pool full: the label is not recorded
          if (commit) atomicOr(d.err, 8);
        }
      }
      if (commit) d.pool_n[slot] = pool_used;
      n_cnt = cnt;
      int tasks = 0;
      for (int j = 0; j < cnt; ++j) {
        s_task0[j] = tasks;
        if (n_tok[j] != V) tasks += o_lml[n_par[j]] + o_trl[n_par[j]];
      }
      s_task0[cnt] = tasks;
      if (d.cap_rows && step - 1 < d.cap_steps && commit) {
        for (int i = 0; i < K; ++i) {
          int* cr = d.cap_rows + ((size_t)(step - 1) * P->n * K + (size_t)b * K + i) * 4;
          if (i < nsel) {
            cr[0] = s_sel[i] / K;
            cr[1] = c_tok[s_sel[i]];
            cr[2] = __float_as_int(c_inc[s_sel[i]]);
            cr[3] = s_into[i];
          } else {
            cr[0] = -1; cr[1] = -1; cr[2] = 0; cr[3] = -1;
          }
        }
      }
    }
    row::block_sync();
    // 3. searches of each survivor's label in its parent's chains
    const int cnt = n_cnt;
    if (tid >= kRowThreads - kMaxK) {
      const int j = tid - (kRowThreads - kMaxK);
      if (j < cnt && n_tok[j] != V) {
        const int y = n_tok[j];
        sr_uni[j] = (d.has_lm && d.lm.order >= 2) ? __ldg(d.lm.uni_tgt + y) : -1;
        sr_rc[j] = d.has_tr ? __ldg(d.tr.root_child + y) : 0;
        sr_rn[j] = d.has_tr ? __ldg(d.tr.root_next + y) : 0;
      }
    }
    for (int task = warp; task < s_task0[cnt]; task += kRowThreads / 32) {
      int j = 0;
      while (j + 1 < cnt && s_task0[j + 1] <= task) ++j;
      const int p = n_par[j], y = n_tok[j];
      const int l = task - s_task0[j];
      if (l < o_lml[p]) {
        const int st = o_lm[p][l];
        const int bb = __ldg(d.lm.st_begin + st), c = __ldg(d.lm.st_count + st);
        const int i = warp_find(d.lm.arc_tok + bb, c, y, lane);
        if (lane == 0) sr_lm[j][l] = (i >= 0) ? __ldg(d.lm.arc_tgt + bb + i) : -2;
      } else {
        const int k = l - o_lml[p];
        const int q = o_tr[p][k];
        const int bb = __ldg(d.tr.nd_begin + q), c = __ldg(d.tr.nd_count + q);
        const int i = warp_find(d.tr.ch_tok + bb, c, y, lane);
        if (lane == 0) {
          sr_trn[j][k] = (i >= 0) ? __ldg(d.tr.ch_node + bb + i) : -1;
          sr_trx[j][k] = (i >= 0) ? __ldg(d.tr.ch_next + bb + i) : -1;
        }
      }
    }
    row::block_sync();
    // 4. survivors' chains (thread j for survivor j)
    if (tid < cnt) {
      const int j = tid, p = n_par[j], y = n_tok[j];
      if (y == V) {
        n_last[j] = o_last[p];
        n_lml[j] = o_lml[p];
        n_trl[j] = o_trl[p];
        for (int l = 0; l < o_lml[p]; ++l) n_lm[j][l] = o_lm[p][l];
        for (int l = 0; l < o_trl[p]; ++l) n_tr[j][l] = o_tr[p][l];
      } else {
        n_last[j] = y;
        int ln = 0;
        if (sr_uni[j] >= 0) {
          n_lm[j][ln++] = sr_uni[j];
          for (int l = 0; l < o_lml[p] && ln < kLmChain; ++l) {
            const int tgt = sr_lm[j][l];
            if (tgt < 0) break;
            n_lm[j][ln++] = tgt;
          }
        }
        n_lml[j] = ln;
        int tn = 0;
        bool reset = false;
        if (d.has_tr) {
          for (int k = 0; k < o_trl[p]; ++k) {
            if (sr_trn[j][k] < 0) continue;
            if (tn == 0 && sr_trx[j][k] == 0) reset = true;
            if (tn < kTrChain) n_tr[j][tn++] = sr_trn[j][k];
          }
          if (sr_rc[j] != 0) {
            if (tn == 0 && sr_rn[j] == 0) reset = true;
            if (tn < kTrChain) n_tr[j][tn++] = sr_rc[j];
          }
          if (reset) tn = 0;
        }
        n_trl[j] = tn;
      }
    }
    row::block_sync();
    // 5. F keeps its K best (score desc, earlier first) in insertion order:
    //    loaded entries, then this step's exits.  The frame ends when nothing
    //    stays in it or after its S-th expansion; F is then the beam.
    if (tid == 0) {
      const bool last_exp = s_be >= S - 1;
      int nf = 0;
      for (int j = 0; j < e_cnt; ++j) { q_src[nf] = -2 - j; q_score[nf++] = e_score[j]; }
      for (int j = 0; j < cnt; ++j)
        if (n_dst[j] == 1) { q_src[nf] = j; q_score[nf++] = n_score[j]; }
      int fc = 0;
      if (nf <= K) {
        for (int x = 0; x < nf; ++x) f_src[fc++] = q_src[x];
      } else {
        for (int x = 0; x < nf; ++x) {
          int rank = 0;
          for (int y = 0; y < nf; ++y)
            if (q_score[y] > q_score[x] || (q_score[y] == q_score[x] && y < x)) ++rank;
          if (rank < K) f_src[fc++] = q_src[x];
        }
      }
      f_cnt = fc;
      int na = 0;
      for (int j = 0; j < cnt; ++j) na += n_dst[j] == 0 ? 1 : 0;
      const bool frame_end = na == 0 || last_exp;
      if (frame_end) {
        for (int k = 0; k < fc; ++k) s_into[k] = f_src[k];  // the beam's sources
        a_cnt = fc;
        f_cnt = 0;
        s_bt = s_bt + 1;
        s_be = 0;
      } else {
        int k = 0;
        for (int j = 0; j < cnt; ++j)
          if (n_dst[j] == 0) s_into[k++] = j;
        a_cnt = k;
        s_be = s_be + 1;
      }
      a_frame = s_bt;
      a_build = s_bt < T ? a_cnt : 0;  // a finished stream evaluates nothing more
    }
    row::block_sync();
    // the beam's records from this step's new records (>= 0) or loaded F
    // entries; chains copied by the whole block
    if (tid < a_cnt) {
      const int k = tid, sidx = s_into[k];
      if (sidx >= 0) {
        a_node[k] = n_node[sidx]; a_len[k] = n_len[sidx]; a_last[k] = n_last[sidx]; a_score[k] = n_score[sidx];
        a_hash[k] = n_hash[sidx]; a_lml[k] = n_lml[sidx]; a_trl[k] = n_trl[sidx];
      } else {
        const int j = -2 - sidx;
        a_node[k] = e_node[j]; a_len[k] = e_len[j]; a_last[k] = e_last[j]; a_score[k] = e_score[j];
        a_hash[k] = e_hash[j]; a_lml[k] = e_lml[j]; a_trl[k] = e_trl[j];
      }
    }
    for (int i = tid; i < a_cnt * (kLmChain + kTrChain); i += kRowThreads) {
      const int k = i / (kLmChain + kTrChain), l = i % (kLmChain + kTrChain), sidx = s_into[k];
      const int j = sidx >= 0 ? sidx : -2 - sidx;
      if (l < kLmChain) a_lm[k][l] = sidx >= 0 ? n_lm[j][l] : e_lm[j][l];
      else a_tr[k][l - kLmChain] = sidx >= 0 ? n_tr[j][l - kLmChain] : e_tr[j][l - kLmChain];
    }
    row::block_sync();
  } else {
    // the chunk's first step, or a stream that finished its frames: the beam
    // as stored (at the first step, the hypotheses carried over)
    if (tid == 0) {
      int cnt = 0;
      for (int k = 0; k < K; ++k) cnt += o_live[k] ? 1 : 0;
      a_cnt = cnt;
      f_cnt = 0;
      a_frame = s_bt;
      a_build = s_done ? 0 : cnt;
    }
    if (tid < K) {
      const int k = tid;
      a_node[k] = o_node[k];
      a_len[k] = o_len[k];
      a_last[k] = o_last[k];
      a_score[k] = o_score[k];
      a_hash[k] = o_hash[k];
      a_lml[k] = o_lml[k];
      a_trl[k] = o_trl[k];
    }
    for (int i = tid; i < K * (kLmChain + kTrChain); i += kRowThreads) {
      const int k = i / (kLmChain + kTrChain), l = i % (kLmChain + kTrChain);
      if (l < kLmChain) a_lm[k][l] = o_lm[k][l];
      else a_tr[k][l - kLmChain] = o_tr[k][l - kLmChain];
    }
    if (d.cap_rows && step > 0 && step - 1 < d.cap_steps && commit && tid < K) {
      int* cr = d.cap_rows + ((size_t)(step - 1) * P->n * K + (size_t)b * K + tid) * 4;
      cr[0] = -1; cr[1] = -1; cr[2] = 0; cr[3] = -1;
    }
    row::block_sync();
  }
  const int cnt = a_cnt;

  // commit: the beam (compact, first cnt slots), F, and the counters
  if (commit && !(step > 0 && s_done)) {
    if (step > 0 && tid < K) {
      const int h = hb + tid;
      const bool live = tid < cnt;
      d.h_live[h] = live ? 1 : 0;
      if (live) {
        d.h_score[h] = a_score[tid];
        d.h_node[h] = a_node[tid];
        d.h_len[h] = a_len[tid];
        d.h_hash[h] = a_hash[tid];
        d.s_last[h] = a_last[tid];
        if (d.has_lm) d.s_lm_len[h] = a_lml[tid];
        if (d.has_tr) d.s_tr_len[h] = a_trl[tid];
      }
    }
    if (step > 0) {
      for (int i = tid; i < cnt * kLmChain; i += kRowThreads) {
        const int k = i / kLmChain, l = i % kLmChain;
        if (l < a_lml[k]) d.s_lm_chain[(size_t)(hb + k) * kLmChain + l] = a_lm[k][l];
      }
      for (int i = tid; i < cnt * kTrChain; i += kRowThreads) {
        const int k = i / kTrChain, l = i % kTrChain;
        if (l < a_trl[k]) d.s_tr_chain[(size_t)(hb + k) * kTrChain + l] = a_tr[k][l];
      }
    }
    if (S > 1) {
      // F (compact) for the frame's next expansion
      if (tid < K) {
        const int h = hb + tid, k = tid;
        const bool live = k < f_cnt;
        d.f_live[h] = live ? 1 : 0;
        if (live) {
          const int sidx = f_src[k];
          const bool nw = sidx >= 0;
          const int j = nw ? sidx : -2 - sidx;
          d.f_score[h] = nw ? n_score[j] : e_score[j];
          d.f_node[h] = nw ? n_node[j] : e_node[j];
          d.f_len[h] = nw ? n_len[j] : e_len[j];
          d.f_hash[h] = nw ? n_hash[j] : e_hash[j];
          d.f_last[h] = nw ? n_last[j] : e_last[j];
          d.f_lml[h] = nw ? n_lml[j] : e_lml[j];
          d.f_trl[h] = nw ? n_trl[j] : e_trl[j];
        }
      }
      for (int i = tid; i < f_cnt * (kLmChain + kTrChain); i += kRowThreads) {
        const int k = i / (kLmChain + kTrChain), l = i % (kLmChain + kTrChain);
        const int sidx = f_src[k];
        const bool nw = sidx >= 0;
        const int j = nw ? sidx : -2 - sidx;
        if (l < kLmChain) {
          if (l < (nw ? n_lml[j] : e_lml[j]))
            d.f_lmc[(size_t)(hb + k) * kLmChain + l] = nw ? n_lm[j][l] : e_lm[j][l];
        } else {
          const int q = l - kLmChain;
          if (q < (nw ? n_trl[j] : e_trl[j]))
            d.f_trc[(size_t)(hb + k) * kTrChain + q] = nw ? n_tr[j][q] : e_tr[j][q];
        }
      }
    }
    if (tid == 0) {
      d.b_frame[slot] = s_bt;
      d.b_exp[slot] = s_be;
    }
  }
  if (mode == 1) {
    if (tid == 0) {
      int best = 0;
      for (int j = 1; j < cnt; ++j)
        if (a_score[j] > a_score[best]) best = j;
      P->out_count[b] = cnt ? a_len[best] : 0;
      P->out_score[(size_t)b * T * d.max_sym] = cnt ? (float)a_score[best] : 0.f;
    }
  }
  // Algorithmic bytes (counted when timing): the K hypotheses' partials and state
  if (mode == 2 || d.count)
    if (tid == 0) atomicAdd(d.ctr, (unsigned long long)K * (d.n_ptiles * (1 + K) * 8 + 64));
  } else {
    // the joint input and bias rows written below are read by the previous
    // joint kernel: wait for it as the first CTA does
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  }
  if (mode == 1) return;  // the same for every CTA: no cluster barrier below is left waiting

  // 6. survivor crank's joint input and fusion bias for frame `step`.  Its
  //    chains come from the first CTA's shared memory (the cluster barrier
  //    makes them visible); a second barrier keeps the first CTA resident
  //    until every CTA has its copy.
  cluster.sync();
  {
    const int* rcnt = cluster.map_shared_rank(&a_build, 0);
    const int* rframe = cluster.map_shared_rank(&a_frame, 0);
    const int* rlml = cluster.map_shared_rank(&a_lml[0], 0);
    const int* rtrl = cluster.map_shared_rank(&a_trl[0], 0);
    const int* rlast = cluster.map_shared_rank(&a_last[0], 0);
    const int* rlm = cluster.map_shared_rank(&a_lm[0][0], 0);
    const int* rtr = cluster.map_shared_rank(&a_tr[0][0], 0);
    if (tid == 0) {
      m_cnt = *rcnt;
      m_frame = *rframe;
      m_lml = rlml[crank];
      m_trl = rtrl[crank];
      m_last = rlast[crank];
    }
    if (tid < kLmChain) m_lm[tid] = rlm[crank * kLmChain + tid];
    if (tid >= 32 && tid - 32 < kTrChain) m_tr[tid - 32] = rtr[crank * kTrChain + tid - 32];
  }
  cluster.sync();
  if (crank >= m_cnt) return;
  const int r = b * K + crank;
  const int Tn = __ldcg(&P->T);
  const uint16_t* enc_row = P->enc + ((size_t)b * Tn + min(m_frame, Tn - 1)) * d.H;
  row::bias_prepare(d, m_lm, m_lml, m_tr, m_trl, rc, lmv, dep);
  row::build_joint_input(d, enc_row, m_last, r);
  row::bias_finish(d, m_lml, m_trl, rc, P->lambda, P->beta, d.bias + (size_t)r * d.N_pad, lmv, dep);
  if ((mode == 2 || d.count) && tid == 0) {
    // per survivor: its joint input and every arc of its LM chain levels and
    // trie chain nodes with their records
    unsigned long long bytes = 6ull * d.H;
    for (int l = 0; l < m_lml; ++l) bytes += 12 + 8ull * rc.lc[l];
    for (int k = 0; k < m_trl; ++k) bytes += 12 + 4ull * rc.tc[k];
    atomicAdd(d.ctr, bytes);
  }
}

__global__ void k_open_beam(DecView d, int slot) {
  const int k = threadIdx.x;
  if (k < d.K) {
    const int h = slot * d.K + k;
    d.h_live[h] = (k == 0) ? 1 : 0;
    d.h_score[h] = 0.0;
    d.h_node[h] = -1;
    d.h_len[h] = 0;
    d.h_hash[h] = 0ull;
    d.s_last[h] = d.V;
    d.s_lm_len[h] = 0;
    d.s_tr_len[h] = 0;
  }
  if (k == 0) d.pool_n[slot] = 0;
}

}  // namespace

void launch_row_beam(const DecView& d, int n, int step, int mode, size_t smem, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n * d.K);
  cfg.blockDim = dim3(kRowThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;  // one cluster of K CTAs per stream
  attr[0].val.clusterDim.x = d.K;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  if (d.max_sym > 1) cudaLaunchKernelEx(&cfg, k_row_beam<true>, d, step, mode);
  else cudaLaunchKernelEx(&cfg, k_row_beam<false>, d, step, mode);
}

void launch_open_beam(const DecView& d, int slot, cudaStream_t s) { k_open_beam<<<1, 32, 0, s>>>(d, slot); }

cudaError_t prepare_beam_kernels(size_t row_smem) {
  // dynamic scratch plus the kernel's static shared memory may pass the
  // 48 KB default even when the scratch alone does not
  cudaError_t e = cudaFuncSetAttribute(k_row_beam<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)row_smem);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(k_row_beam<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)row_smem);
  return e;
}

}  // namespace tsd
