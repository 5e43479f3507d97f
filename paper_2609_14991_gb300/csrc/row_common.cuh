// Device building blocks shared by the greedy and the beam row passes.
#pragma once

#include "decoder.h"

namespace tsd {
namespace row {

constexpr float kNegInf = -__builtin_huge_valf();

// Position of y in the sorted arr[0, n), or -1: a 32-ary search by one warp.
__device__ __forceinline__ int warp_find(const int32_t* __restrict__ arr, int n, int y, int lane) {
  int lo = 0, hi = n;
  while (hi - lo > 32) {
    int step = (hi - lo + 31) >> 5;
    int idx = lo + lane * step;
    int v = (idx < hi) ? __ldg(arr + idx) : INT_MAX;
    unsigned m = __ballot_sync(0xffffffffu, v <= y);
    if (m == 0) return -1;
    int last = 31 - __clz((int)m);
    lo = lo + last * step;
    hi = min(hi, lo + step);
  }
  int idx = lo + lane;
  bool hit = (idx < hi) && (__ldg(arr + idx) == y);
  unsigned m = __ballot_sync(0xffffffffu, hit);
  return m ? lo + __ffs((int)m) - 1 : -1;
}

// Merges two softmax partials (max, sum of exp(x - max)).
__device__ __forceinline__ void lse_merge(float& m, float& s, float m2, float s2) {
  if (m2 == kNegInf) return;
  if (m == kNegInf) { m = m2; s = s2; return; }
  float mx = fmaxf(m, m2);
  s = s * expf(m - mx) + s2 * expf(m2 - mx);
  m = mx;
}

__device__ __forceinline__ void best_merge(float& v, int& i, float v2, int i2) {
  if (v2 > v || (v2 == v && i2 < i)) { v = v2; i = i2; }
}

// Joint input of one row: A[r] = bf16(ReLU(enc_row + E[last])), block-strided.
__device__ __forceinline__ void build_joint_input(const DecView& d, const uint16_t* enc_row, int last, int r) {
  const int H = d.H;
  const uint4* e = reinterpret_cast<const uint4*>(enc_row);
  const uint4* g = reinterpret_cast<const uint4*>(d.E + (size_t)last * H);
  uint4* a = reinterpret_cast<uint4*>(d.A + (size_t)r * H);
  for (int i = threadIdx.x; i < H / 8; i += blockDim.x) {
    uint4 x = __ldg(e + i), z = __ldg(g + i);
    const __nv_bfloat162* xa = reinterpret_cast<const __nv_bfloat162*>(&x);
    const __nv_bfloat162* za = reinterpret_cast<const __nv_bfloat162*>(&z);
    uint4 out;
    __nv_bfloat162* oa = reinterpret_cast<__nv_bfloat162*>(&out);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      float2 xf = __bfloat1622float2(xa[q]);
      float2 zf = __bfloat1622float2(za[q]);
      float lo = fmaxf(xf.x + zf.x, 0.f), hi = fmaxf(xf.y + zf.y, 0.f);
      oa[q] = __floats2bfloat162_rn(lo, hi);
    }
    a[i] = out;
  }
}

// Shared-memory records of the chains a bias row is built from.
struct ChainRecs {
  int lb[kLmChain], lc[kLmChain];  // LM level: first arc, arcs
  float lo[kLmChain];              // LM level: cumulative backoff weight
  int tb[kTrChain], tc[kTrChain];  // trie chain node: first child, children
  int td[kTrChain];                // trie chain node: depth of its children
};

// Step 1 of a bias row (no barrier): fetch the chains' records, clear the
// per-label scratch.  All threads of the block call it.
__device__ __forceinline__ void bias_prepare(const DecView& d, const int* lm_chain, int nl, const int* tr_chain,
                                             int nt, ChainRecs& rc, unsigned long long* lmkey, int* dep) {
  const int tid = threadIdx.x;
  if (tid < nl) {
    const int st = lm_chain[tid];
    rc.lb[tid] = __ldg(d.lm.st_begin + st);
    rc.lc[tid] = __ldg(d.lm.st_count + st);
    rc.lo[tid] = __ldg(d.lm.st_cum + st);
  } else if (tid >= 32 && tid - 32 < nt) {
    const int q = tr_chain[tid - 32];
    rc.tb[tid - 32] = __ldg(d.tr.nd_begin + q);
    rc.tc[tid - 32] = __ldg(d.tr.nd_count + q);
    rc.td[tid - 32] = __ldg(d.tr.nd_depth + q) + 1;
  }
  for (int v = tid; v < d.V; v += blockDim.x) {
    lmkey[v] = 0ull;
    dep[v] = 0;
  }
}

// Step 2: the dense fusion bias row lambda*log p_LM(v|state) +
// beta*bonus*(goto depth - current depth) for every label v (blank: 0).
// Every chain level is merged at once: a label's LM score comes from the
// deepest level that continues with it (max of level << 32 | value bits),
// its goto depth from the deepest trie node that has it as a child.
__device__ __forceinline__ void bias_finish(const DecView& d, int nl, int nt, const ChainRecs& rc, float lam,
                                            float beta, float* brow, unsigned long long* lmkey, int* dep) {
  const int tid = threadIdx.x;
  const int V = d.V;
  __syncthreads();
  const float cum_top = nl ? rc.lo[nl - 1] : 0.f;
  for (int l = 0; l < nl; ++l) {
    const int b = rc.lb[l], c = rc.lc[l];
    const float off = cum_top - rc.lo[l];
    const unsigned long long lev = (unsigned long long)(l + 1) << 32;
    for (int j = tid; j < c; j += blockDim.x) {
      const int w = __ldg(d.lm.arc_tok + b + j);
      const float val = off + __ldg(d.lm.arc_logp + b + j);
      atomicMax(lmkey + w, lev | (unsigned long long)__float_as_uint(val));
    }
  }
  for (int k = 0; k < nt; ++k) {
    const int b = rc.tb[k], c = rc.tc[k], dd = rc.td[k];
    for (int j = tid; j < c; j += blockDim.x) atomicMax(dep + __ldg(d.tr.ch_tok + b + j), dd);
  }
  __syncthreads();
  const int depth_cur = nt ? rc.td[0] - 1 : 0;
  const float bscale = beta * (d.has_tr ? d.tr.bonus : 0.f);
  for (int v = tid; v < V; v += blockDim.x) {
    float b = 0.f;
    if (d.has_lm) {
      const unsigned long long k = lmkey[v];
      const float l = k ? __uint_as_float((unsigned)k) : cum_top + __ldg(d.lm.uni_logp + v);
      b = lam * l;
    }
    if (d.has_tr) {
      int dd = dep[v];
      if (dd == 0) dd = (__ldg(d.tr.root_child + v) != 0) ? 1 : 0;
      b += bscale * (float)(dd - depth_cur);
    }
    brow[v] = b;
  }
  if (tid == 0) brow[V] = 0.f;
}

}  // namespace row
}  // namespace tsd
