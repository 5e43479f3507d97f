// Row pass of pruned fusion: one CTA per row, no per-label work.
//
// The LM and boost terms of Eq. 1 re-rank only the acoustic model's k best
// outputs (the reading of Sec. III-C's remark that fusion only re-ranks the
// candidates the model proposes).  The joint kernel's epilogue keeps, per
// tile, the softmax partial and the k largest logits; this pass
//   1. merges them into the row's log-sum-exp and its k best outputs;
//   2. scores each candidate: its log-probability, lambda * log p_LM from the
//      deepest chain level that continues with it (else the backoff to the
//      unigram), beta * bonus from the deepest trie chain node that has it as
//      a child (else the root) -- one warp search per (candidate, chain
//      element), all independent;
//   3. takes the best (ties to the lower label) and advances the frame, LM
//      and trie state exactly as the full pass does, reusing the arcs the
//      searches found;
//   4. writes the joint input of the next step.  No bias row is needed.
#include "row_common.cuh"

namespace tsd {

namespace {

using row::kNegInf;
using row::lse_merge;
using row::warp_find;

constexpr int kMaxCand = 8;
constexpr int kCandPerLane = 16;  // tile candidates per lane: n_tiles * k <= 512

__global__ void __launch_bounds__(kRowThreads) k_row_pruned(DecView d, int step, int mode) {
  const Params* __restrict__ P = d.params;
  const int r = blockIdx.x;
  const int V = d.V, K = d.topk;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const bool commit = (mode != 2);

  __shared__ int s_t, s_sym, s_cnt, s_y, s_lm_len, s_tr_len, s_last, s_slot, s_T, s_nc;
  __shared__ int s_lm[kLmChain], s_tr[kTrChain];
  __shared__ row::ChainRecs rc;
  __shared__ float c_logit[kMaxCand], c_fused[kMaxCand];
  __shared__ int c_lab[kMaxCand];
  __shared__ int c_arc[kMaxCand][kLmChain];   // arc index of the candidate at each LM level (-1 none)
  __shared__ int c_child[kMaxCand][kTrChain]; // child index of the candidate at each trie node (-1 none)
  __shared__ int c_uni_tgt[kMaxCand], c_root_child[kMaxCand], c_root_next[kMaxCand];
  __shared__ float c_uni[kMaxCand];

  // Row state and the current chains' records: written by the previous row
  // pass, read before the dependency wait through L2 (see the full pass).
  if (tid == 0) {
    const int slot = __ldcg(P->slots + r);
    s_slot = slot;
    s_T = __ldcg(&P->T);
    if (step == 0) {
      s_t = 0; s_sym = 0; s_cnt = 0;
    } else {
      s_t = __ldcg(d.r_t + r); s_sym = __ldcg(d.r_sym + r); s_cnt = __ldcg(d.r_cnt + r);
    }
    s_lm_len = d.has_lm ? __ldcg(d.s_lm_len + slot) : 0;
    s_tr_len = d.has_tr ? __ldcg(d.s_tr_len + slot) : 0;
    s_last = __ldcg(d.s_last + slot);
  }
  row::block_sync();
  const int slot = s_slot, T = s_T;
  if (tid < s_lm_len) {
    const int st = __ldcg(d.s_lm_chain + slot * kLmChain + tid);
    s_lm[tid] = st;
    rc.lb[tid] = __ldg(d.lm.st_begin + st);
    rc.lc[tid] = __ldg(d.lm.st_count + st);
    rc.lo[tid] = __ldg(d.lm.st_cum + st);
  }
  if (tid >= 64 && tid - 64 < s_tr_len) {
    const int k = tid - 64;
    const int q = __ldcg(d.s_tr_chain + slot * kTrChain + k);
    s_tr[k] = q;
    rc.tb[k] = __ldg(d.tr.nd_begin + q);
    rc.tc[k] = __ldg(d.tr.nd_count + q);
    rc.td[k] = __ldg(d.tr.nd_depth + q) + 1;
  }
  row::block_sync();
  const bool evaluated = (step > 0) && (s_t < T || !commit);
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

  if (evaluated) {
    // 1. log-sum-exp and the k best outputs of the row (warp 0)
    if (warp == 0) {
      const float2* bp = d.bpart + (size_t)r * d.n_ptiles * (1 + K);
      float m = kNegInf, s = 0.f;
      for (int j = lane; j < d.n_ptiles; j += 32) {
        const float2 p = __ldcg(bp + (size_t)j * (1 + K));
        lse_merge(m, s, p.x, p.y);
      }
      float cv[kCandPerLane];
      int ct[kCandPerLane];
      const int nc = d.n_ptiles * K;
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
      row::reconverge();
      for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o), s2 = __shfl_xor_sync(0xffffffffu, s, o);
        lse_merge(m, s, m2, s2);
      }
      const float lse = m + logf(s);
      int got = 0;
      for (int round = 0; round < K; ++round) {
        row::reconverge();
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
        if (wv == kNegInf || wt < 0 || wt > V) break;  // warp-uniform
        if (lane == 0) {
          c_logit[got] = wv - lse;  // log p_AM of the candidate
          c_lab[got] = wt;
        }
        ++got;
      }
      if (lane == 0) s_nc = got;
    }
    row::block_sync();
    const int nc = s_nc, nl = s_lm_len, nt = s_tr_len;
    // 2. per candidate: unigram record and root child (one thread each), and
    //    one warp search per (candidate, chain element)
    if (tid >= kRowThreads - kMaxCand && tid - (kRowThreads - kMaxCand) < nc) {
      const int j = tid - (kRowThreads - kMaxCand), c = c_lab[j];
      const bool lab = c != V;
      c_uni[j] = (lab && d.has_lm) ? __ldg(d.lm.uni_logp + c) : 0.f;
      c_uni_tgt[j] = (lab && d.has_lm && d.lm.order >= 2) ? __ldg(d.lm.uni_tgt + c) : -1;
      c_root_child[j] = (lab && d.has_tr) ? __ldg(d.tr.root_child + c) : 0;
      c_root_next[j] = (lab && d.has_tr) ? __ldg(d.tr.root_next + c) : 0;
    }
    const int per = nl + nt;
    for (int task = warp; task < nc * per; task += kRowThreads / 32) {
      const int j = task / per, e = task % per, c = c_lab[j];
      if (e < nl) {
        const int i = (c == V) ? -1 : warp_find(d.lm.arc_tok + rc.lb[e], rc.lc[e], c, lane);
        if (lane == 0) c_arc[j][e] = i < 0 ? -1 : rc.lb[e] + i;
      } else {
        const int k = e - nl;
        const int i = (c == V) ? -1 : warp_find(d.tr.ch_tok + rc.tb[k], rc.tc[k], c, lane);
        if (lane == 0) c_child[j][k] = i < 0 ? -1 : rc.tb[k] + i;
      }
    }
    row::block_sync();
    // 3. fused value of each candidate, then the best (thread 0)
    if (tid < nc) {
      const int j = tid, c = c_lab[j];
      float f = c_logit[j];
      if (c != V) {
        const float lam = P->lambda, beta = P->beta;
        if (d.has_lm) {
          const float cum_top = nl ? rc.lo[nl - 1] : 0.f;
          float lm = c_uni[j] + cum_top;  // backoff to the unigram
          for (int l = nl - 1; l >= 0; --l)
            if (c_arc[j][l] >= 0) {
              lm = (cum_top - rc.lo[l]) + __ldg(d.lm.arc_logp + c_arc[j][l]);
              break;
            }
          f += lam * lm;
        }
        if (d.has_tr) {
          const int depth_cur = nt ? rc.td[0] - 1 : 0;
          int go = c_root_child[j] != 0 ? 1 : 0;  // deepest chain node with child c, else the root
          for (int k = 0; k < nt; ++k)
            if (c_child[j][k] >= 0) {
              go = rc.td[k];
              break;
            }
          f += beta * d.tr.bonus * (float)(go - depth_cur);
        }
      }
      c_fused[j] = f;
    }
    row::block_sync();
    if (tid == 0) {
      int b = 0;
      for (int j = 1; j < nc; ++j)
        if (c_fused[j] > c_fused[b] || (c_fused[j] == c_fused[b] && c_lab[j] < c_lab[b])) b = j;
      s_y = nc ? b : -1;  // the chosen candidate (its label in c_lab)
    }
    row::block_sync();
    const int jb = s_y;
    const int y = jb >= 0 ? c_lab[jb] : V;
    if (y != V) {
      // 4. new chains from the arcs the chosen candidate's searches found
      if (tid == 0) {
        int ln = 0;
        if (c_uni_tgt[jb] >= 0) {
          int nw[kLmChain];
          nw[ln++] = c_uni_tgt[jb];
          for (int l = 0; l < nl && ln < kLmChain; ++l) {
            if (c_arc[jb][l] < 0) break;
            const int tgt = __ldg(d.lm.arc_tgt + c_arc[jb][l]);
            if (tgt < 0) break;  // the top order
            nw[ln++] = tgt;
          }
          for (int l = 0; l < ln; ++l) s_lm[l] = nw[l];
        }
        int tn = 0, nwt[kTrChain];
        bool reset = false;
        for (int k = 0; k < nt; ++k) {
          if (c_child[jb][k] < 0) continue;
          const int nd = __ldg(d.tr.ch_node + c_child[jb][k]);
          if (tn == 0 && __ldg(d.tr.ch_next + c_child[jb][k]) == 0) reset = true;
          if (tn < kTrChain) nwt[tn++] = nd;
        }
        if (c_root_child[jb] != 0) {
          if (tn == 0 && c_root_next[jb] == 0) reset = true;
          if (tn < kTrChain) nwt[tn++] = c_root_child[jb];
        }
        if (reset) tn = 0;
        for (int l = 0; l < tn; ++l) s_tr[l] = nwt[l];
        s_lm_len = ln;
        s_tr_len = tn;
        if (commit) {
          for (int l = 0; l < ln; ++l) d.s_lm_chain[slot * kLmChain + l] = s_lm[l];
          for (int l = 0; l < tn; ++l) d.s_tr_chain[slot * kTrChain + l] = s_tr[l];
          if (d.has_lm) d.s_lm_len[slot] = ln;
          if (d.has_tr) d.s_tr_len[slot] = tn;
          const int cap = T * d.max_sym;
          const int o = r * cap + s_cnt;
          P->out_tok[o] = y;
          P->out_frame[o] = s_t;
          P->out_score[o] = c_fused[jb];
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
    if ((mode == 2 || d.count) && tid == 0) {
      // Algorithmic bytes: partials, row state and chain records, the
      // searches of every candidate in every chain element (one probe per
      // halving), the chosen arc's targets.
      unsigned long long bytes = (unsigned long long)d.n_ptiles * (1 + K) * 8 + 2ull * (24 + 4 * (nl + nt));
      bytes += 12ull * (nl + nt) + (unsigned long long)nc * 20;
      for (int l = 0; l < nl; ++l) bytes += (unsigned long long)nc * 4 * (32 - __clz(rc.lc[l] + 1)) + 8;
      for (int k = 0; k < nt; ++k) bytes += (unsigned long long)nc * 4 * (32 - __clz(rc.tc[k] + 1)) + 8;
      bytes += 6ull * d.H;
      atomicAdd(d.ctr, bytes);
    }
  }

  if (mode == 1) {
    if (tid == 0) P->out_count[r] = s_cnt;
    return;
  }
  if (tid == 0 && commit) {
    d.r_t[r] = s_t;
    d.r_sym[r] = s_sym;
    d.r_cnt[r] = s_cnt;
  }
  const int t = commit ? s_t : min(s_t, T - 1);
  if (d.cap_rows && step < d.cap_steps && tid == 0 && commit) {
    int* cr = d.cap_rows + ((size_t)step * P->n + r) * 4;
    if (t < T) {
      cr[0] = t;
      cr[1] = s_last;
      cr[2] = s_lm_len ? s_lm[s_lm_len - 1] : 0;
      cr[3] = s_tr_len ? s_tr[0] : 0;
    } else {
      cr[0] = -1; cr[1] = -1; cr[2] = -1; cr[3] = -1;
    }
  }
  if (t >= T) return;
  row::build_joint_input(d, P->enc + ((size_t)r * T + t) * d.H, s_last, r);
}

}  // namespace

void launch_row_pruned(const DecView& d, int M, int step, int mode, cudaStream_t s, bool pdl) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(M);
  cfg.blockDim = dim3(kRowThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  cudaLaunchKernelEx(&cfg, k_row_pruned, d, step, mode);
}

}  // namespace tsd
