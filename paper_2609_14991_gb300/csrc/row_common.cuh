// Device building blocks shared by the greedy and the beam row passes.
#pragma once

#include "decoder.h"

namespace tsd {
namespace row {

constexpr float kNegInf = -__builtin_huge_valf();

// Range checks of the TSD_CHECKS build: a failed check records its code in
// the decoder's status word (the first one wins; tsd_decoder_check reports
// TSD_EDEVICE) and the caller skips the access.  In the ordinary build the
// condition is not evaluated.
#ifdef TSD_CHECKS
__device__ __forceinline__ bool checked(bool cond, int32_t* err, int code) {
  if (!cond) atomicCAS(err, 0, 0x100 + code);
  return cond;
}
#else
__device__ __forceinline__ constexpr bool checked(bool, int32_t*, int) { return true; }
#endif

// After divergent code (a single-thread section, a lane-strided loop) the
// lanes of a warp can keep running apart past the point where they could
// rejoin, and every warp-synchronous step after it (shuffle, ballot) then
// costs about ten times as much.  These force the warp back together.
__device__ __forceinline__ void reconverge() { __syncwarp(); }
__device__ __forceinline__ void block_sync() {
  __syncthreads();
  __syncwarp();
}

// Field f of LM i's tables (i < kMaxLm): a select over the kernel
// parameter's per-LM views, so no copy of the parameter block is made.
template <class T>
__device__ __forceinline__ T lm_pick(int i, T a0, T a1, T a2, T a3) {
  return i == 0 ? a0 : i == 1 ? a1 : i == 2 ? a2 : a3;
}
#define TSD_LMX(d, i, f) ::tsd::row::lm_pick((i), (d).lmx[0].f, (d).lmx[1].f, (d).lmx[2].f, (d).lmx[3].f)

// Requests the 128-byte line holding p into L1 (no result, no fault on a
// valid address); later loads of it then wait for L1 rather than L2.
__device__ __forceinline__ void prefetch_l1(const void* p) {
  asm volatile("prefetch.global.L1 [%0];" ::"l"(p));
}

// Lines [0, bytes) from base, one line per thread of the block from `first`.
__device__ __forceinline__ void prefetch_span(const void* base, size_t bytes, int first) {
  const int i = (int)threadIdx.x - first;
  if (i >= 0 && (size_t)i * 128 < bytes) prefetch_l1(static_cast<const char*>(base) + (size_t)i * 128);
}

// Position of y in the sorted arr[0, n), or -1: a 32-ary search by one warp.
__device__ __forceinline__ int warp_find(const int32_t* __restrict__ arr, int n, int y, int lane) {
  reconverge();
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

// Per-label scratch of a bias row in shared memory (5 bytes per label):
//   lmv[v] = log p_LM(v | state) from the deepest LM chain level that
//            continues with v, NaN if none does;
//   dep[v] = depth of v's trie goto node from the chain, 0 if none.
__device__ __forceinline__ float unset_value() { return __int_as_float(0x7fc00000); }

// Step 1 of a bias row (no barrier): fetch the chains' records, clear the
// per-label scratch.  All threads of the block call it.
__device__ __forceinline__ void bias_prepare(const DecView& d, const int* lm_chain, int nl, const int* tr_chain,
                                             int nt, ChainRecs& rc, float* lmv, uint8_t* dep) {
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
  const float unset = unset_value();
  float4* l4 = reinterpret_cast<float4*>(lmv);
  uint32_t* d4 = reinterpret_cast<uint32_t*>(dep);
  for (int q = tid; q < d.V4 / 4; q += blockDim.x) {  // V4 is a multiple of 16
    l4[q] = make_float4(unset, unset, unset, unset);
    d4[q] = 0u;
  }
}

// LM arcs [b, e) of one chain level into the scratch, in 16-byte groups of
// four from the aligned index below b (the arc arrays are padded past their
// last group); a label keeps the first value it gets.  Block-strided.
__device__ __forceinline__ void scatter_lm_level(const int32_t* arc_tok, const float* arc_logp, int b, int e,
                                                 float off, float* lmv) {
  const int a0 = b & ~3;
  const int ng = (e - a0 + 3) >> 2;
  const int4* t4 = reinterpret_cast<const int4*>(arc_tok + a0);
  const float4* p4 = reinterpret_cast<const float4*>(arc_logp + a0);
  for (int g = threadIdx.x; g < ng; g += blockDim.x) {
    const int4 t = __ldg(t4 + g);
    const float4 v = __ldg(p4 + g);
    const int i0 = a0 + 4 * g;
    if (i0 >= b && i0 < e && isnan(lmv[t.x])) lmv[t.x] = off + v.x;
    if (i0 + 1 >= b && i0 + 1 < e && isnan(lmv[t.y])) lmv[t.y] = off + v.y;
    if (i0 + 2 >= b && i0 + 2 < e && isnan(lmv[t.z])) lmv[t.z] = off + v.z;
    if (i0 + 3 >= b && i0 + 3 < e && isnan(lmv[t.w])) lmv[t.w] = off + v.w;
  }
}

// Trie children [b, e) of one chain node: their labels get goto depth dd.
__device__ __forceinline__ void scatter_trie_node(const int32_t* ch_tok, int b, int e, uint8_t dd, uint8_t* dep) {
  const int a0 = b & ~3;
  const int ng = (e - a0 + 3) >> 2;
  const int4* t4 = reinterpret_cast<const int4*>(ch_tok + a0);
  for (int g = threadIdx.x; g < ng; g += blockDim.x) {
    const int4 t = __ldg(t4 + g);
    const int i0 = a0 + 4 * g;
    if (i0 >= b && i0 < e) dep[t.x] = dd;
    if (i0 + 1 >= b && i0 + 1 < e) dep[t.y] = dd;
    if (i0 + 2 >= b && i0 + 2 < e) dep[t.z] = dd;
    if (i0 + 3 >= b && i0 + 3 < e) dep[t.w] = dd;
  }
}

// Step 1 when the chains' records are already in rc: the scratch reset only.
__device__ __forceinline__ void bias_init(const DecView& d, float* lmv, uint8_t* dep) {
  const float unset = unset_value();
  float4* l4 = reinterpret_cast<float4*>(lmv);
  uint32_t* d4 = reinterpret_cast<uint32_t*>(dep);
  for (int q = threadIdx.x; q < d.V4 / 4; q += blockDim.x) {
    l4[q] = make_float4(unset, unset, unset, unset);
    d4[q] = 0u;
  }
}

// Step 2: the dense fusion bias row lambda*log p_LM(v|state) +
// beta*bonus*(goto depth - current depth) for every label v (blank: 0).
// LM chain levels are applied deepest first, each label keeping the first
// value it gets; trie chain nodes shallowest first, the deepest node's child
// depth overwriting.  One barrier per level.  Labels no level touches take
// the call's defaults lambda*log p(v) and beta*bonus*[the root has a child v].
__device__ __forceinline__ void bias_finish(const DecView& d, int nl, int nt, const ChainRecs& rc, float lam,
                                            float beta, float* brow, float* lmv, uint8_t* dep) {
  const int tid = threadIdx.x;
  const int V = d.V;
  const int step = blockDim.x;
  block_sync();
  const float cum_top = nl ? rc.lo[nl - 1] : 0.f;
  const int phases = max(nl, nt);
  for (int p = 0; p < phases; ++p) {
    if (p < nl) {
      const int l = nl - 1 - p;
      scatter_lm_level(d.lm.arc_tok, d.lm.arc_logp, rc.lb[l], rc.lb[l] + rc.lc[l], cum_top - rc.lo[l], lmv);
    }
    if (p < nt) {
      const int k = nt - 1 - p;
      scatter_trie_node(d.tr.ch_tok, rc.tb[k], rc.tb[k] + rc.tc[k], (uint8_t)rc.td[k], dep);
    }
    block_sync();
  }
  const int depth_cur = nt ? rc.td[0] - 1 : 0;
  const float bscale = beta * (d.has_tr ? d.tr.bonus : 0.f);
  const float lm_base = lam * cum_top;
  const float tr_base = -bscale * (float)depth_cur;
  // four consecutive labels per thread: one 16-byte load of the defaults and
  // of the LM scratch, one 4-byte load of the trie scratch, one 16-byte store
  const float4* df4 = reinterpret_cast<const float4*>(d.dflt);
  const float4* l4 = reinterpret_cast<const float4*>(lmv);
  const uint32_t* d4 = reinterpret_cast<const uint32_t*>(dep);
  float4* b4 = reinterpret_cast<float4*>(brow);
  const int nq = d.V4 / 4;
  auto quad = [&](int q, float4 df, uint32_t rootw) {
    const float4 l = l4[q];
    const uint32_t dd = d4[q];
    const uint32_t rb = rootw >> ((4 * q) & 31);
    const float lv[4] = {l.x, l.y, l.z, l.w};
    const float dv[4] = {df.x, df.y, df.z, df.w};
    float o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int dj = (dd >> (8 * j)) & 0xff;
      const float blm = isnan(lv[j]) ? dv[j] + lm_base : lam * lv[j];
      const float btr = dj ? bscale * (float)(dj - depth_cur) : (((rb >> j) & 1u) ? bscale : 0.f) + tr_base;
      o[j] = (4 * q + j < V) ? blm + btr : 0.f;
    }
    b4[q] = make_float4(o[0], o[1], o[2], o[3]);
  };
  int q = tid;
  for (; q + step < nq; q += 2 * step) {  // two quads' loads in flight
    float4 df[2];
    uint32_t rw[2];
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      df[k] = __ldg(df4 + q + k * step);
      rw[k] = __ldg(d.droot + ((q + k * step) >> 3));
    }
#pragma unroll
    for (int k = 0; k < 2; ++k) quad(q + k * step, df[k], rw[k]);
  }
  for (; q < nq; q += step) quad(q, __ldg(df4 + q), __ldg(d.droot + (q >> 3)));
  if (tid == 0) brow[V] = 0.f;
}

}  // namespace row
}  // namespace tsd
