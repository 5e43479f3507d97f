// Host builders for the device tables: the backoff n-gram model (Eq. 1,
// second term) and the phrase-boosting trie (Eq. 1, third term).
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <atomic>
#include <map>
#include <memory>
#include <numeric>
#include <thread>

#include <nvtx3/nvToolsExt.h>

#include "internal.h"

namespace tsd {

NvtxRange::NvtxRange(const char* name) { nvtxRangePushA(name); }
NvtxRange::~NvtxRange() { nvtxRangePop(); }

namespace {
thread_local std::string g_err;

// Runs f(begin, end) over [0, n) on up to hardware_concurrency threads.
template <class F>
void parallel_for(int64_t n, F f) {
  int64_t nt = (int64_t)std::max(1u, std::min(32u, std::thread::hardware_concurrency()));
  if (n < 65536 || nt == 1) {
    f((int64_t)0, n);
    return;
  }
  std::vector<std::thread> th;
  int64_t chunk = (n + nt - 1) / nt;
  for (int64_t t = 0; t < nt; ++t) {
    int64_t b = t * chunk, e = std::min(n, b + chunk);
    if (b >= e) break;
    th.emplace_back([=] { f(b, e); });
  }
  for (auto& x : th) x.join();
}
}  // namespace

tsd_status fail(tsd_status st, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return st;
}

void clear_error() { g_err.clear(); }

tsd_status cuda_fail(cudaError_t e, const char* what) {
  cudaGetLastError();
  return fail(TSD_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

const char* last_error() { return g_err.c_str(); }

namespace {
std::atomic<int32_t> g_fail_alloc{0};  // allocations left before the injected failure (0: off)
}  // namespace

bool alloc_hook_fires() {
  int32_t n = g_fail_alloc.load();
  while (n > 0) {
    if (g_fail_alloc.compare_exchange_weak(n, n - 1)) return n == 1;
  }
  return false;
}

}  // namespace tsd

using namespace tsd;

extern "C" const char* tsd_last_error(void) { return tsd::last_error(); }

extern "C" const char* tsd_version(void) { return "tsd 0.1 sm_103a"; }

extern "C" tsd_status tsd_debug_fail_alloc(int32_t n) {
  clear_error();
  if (n < 0) return fail(TSD_EINVAL, "tsd_debug_fail_alloc: n=%d < 0", n);
  g_fail_alloc.store(n);
  return TSD_OK;
}

// ---------------------------------------------------------------------------
// n-gram tables
// ---------------------------------------------------------------------------
namespace {

struct OrderIn {
  int64_t n = 0;
  const int32_t* tok = nullptr;  // [n][k]
  const float* logp = nullptr;
  const float* bow = nullptr;
  std::vector<int64_t> perm;  // sorted position -> input index (empty = identity)
  int64_t at(int64_t j) const { return perm.empty() ? j : perm[(size_t)j]; }
};

bool tuple_less(const int32_t* a, const int32_t* b, int k) {
  return std::lexicographical_compare(a, a + k, b, b + k);
}

}  // namespace

extern "C" tsd_status tsd_ngram_build(int32_t V, int32_t order, const int64_t* count,
                                      const int32_t* const* ngrams, const float* const* logp,
                                      const float* const* bow, tsd_ngram** out) {
  clear_error();
  if (!out) return fail(TSD_EINVAL, "tsd_ngram_build: out is NULL");
  *out = nullptr;
  if (V < 1 || V > 32767) return fail(TSD_EINVAL, "tsd_ngram_build: V=%d out of range [1, 32767]", V);
  if (order < 1 || order > kMaxOrder)
    return fail(TSD_EINVAL, "tsd_ngram_build: order=%d out of range [1, %d]", order, kMaxOrder);
  if (!count || !ngrams || !logp) return fail(TSD_EINVAL, "tsd_ngram_build: NULL array");
  std::vector<OrderIn> in((size_t)order + 1);
  int64_t total_arcs = 0;
  for (int k = 1; k <= order; ++k) {
    OrderIn& o = in[(size_t)k];
    o.n = count[k - 1];
    if (o.n < 0) return fail(TSD_EINVAL, "tsd_ngram_build: negative count at order %d", k);
    if (o.n > 0 && (!ngrams[k - 1] || !logp[k - 1]))
      return fail(TSD_EINVAL, "tsd_ngram_build: NULL arrays for order %d", k);
    o.tok = ngrams[k - 1];
    o.logp = logp[k - 1];
    o.bow = (bow && k < order) ? bow[k - 1] : nullptr;
    if (k >= 2) total_arcs += o.n;
  }
  if (in[1].n != V) return fail(TSD_EINVAL, "tsd_ngram_build: %lld unigrams, need all %d", (long long)in[1].n, V);
  // the row pass tags arc indices with their level in 32-bit keys
  if (total_arcs >= (int64_t)1 << 28) return fail(TSD_EINVAL, "tsd_ngram_build: more than 2^28 n-grams above order 1");

  // range and value checks, then sort each order
  for (int k = 1; k <= order; ++k) {
    OrderIn& o = in[(size_t)k];
    bool bad_tok = false, bad_val = false;
    for (int64_t i = 0; i < o.n * k; ++i)
      if (o.tok[i] < 0 || o.tok[i] >= V) { bad_tok = true; break; }
    for (int64_t i = 0; i < o.n; ++i)
      if (!std::isfinite(o.logp[i]) || (o.bow && !std::isfinite(o.bow[i]))) { bad_val = true; break; }
    if (bad_tok) return fail(TSD_EINVAL, "tsd_ngram_build: token out of [0, %d) at order %d", V, k);
    if (bad_val) return fail(TSD_EINVAL, "tsd_ngram_build: non-finite logp/bow at order %d", k);
    bool sorted = true;
    for (int64_t i = 1; i < o.n && sorted; ++i)
      if (!tuple_less(o.tok + (i - 1) * k, o.tok + i * k, k)) sorted = false;
    if (!sorted) {
      o.perm.resize((size_t)o.n);
      std::iota(o.perm.begin(), o.perm.end(), 0);
      const int32_t* t = o.tok;
      std::sort(o.perm.begin(), o.perm.end(),
                [&](int64_t a, int64_t b) { return tuple_less(t + a * k, t + b * k, k); });
      for (int64_t j = 1; j < o.n; ++j)
        if (!tuple_less(t + o.at(j - 1) * k, t + o.at(j) * k, k))
          return fail(TSD_EINVAL, "tsd_ngram_build: duplicate n-gram at order %d", k);
    }
  }
  // unigrams are exactly 0..V-1 after sorting
  for (int64_t j = 0; j < V; ++j)
    if (in[1].tok[in[1].at(j)] != (int32_t)j) return fail(TSD_EINVAL, "tsd_ngram_build: unigram %lld missing", (long long)j);

  // state ids: 0 root, then orders 1..order-1
  std::vector<int64_t> base((size_t)order + 2, 0);
  base[1] = 1;
  for (int k = 1; k < order; ++k) base[(size_t)k + 1] = base[(size_t)k] + in[(size_t)k].n;
  const int64_t S = (order >= 2) ? base[(size_t)order] : 1;
  if (S > INT32_MAX) return fail(TSD_EINVAL, "tsd_ngram_build: too many states");

  std::unique_ptr<tsd_ngram> lm(new tsd_ngram());
  std::vector<int32_t> st_begin((size_t)S, 0), st_count((size_t)S, 0);
  std::vector<double> cum((size_t)S, 0.0);
  lm->st_parent.assign((size_t)S, 0);
  lm->st_tok.assign((size_t)S, -1);
  std::vector<int32_t> arc_tok((size_t)total_arcs), arc_tgt((size_t)total_arcs);
  std::vector<float> arc_logp((size_t)total_arcs);
  std::vector<float> uni_logp((size_t)V + 16, 0.f);  // padded: read in 16-byte groups
  std::vector<int32_t> uni_tgt((size_t)V);

  // per sorted position: context and suffix index in the order below, and
  // the child range in the order above
  std::vector<std::vector<int32_t>> ctx((size_t)order + 1), sfx((size_t)order + 1);
  std::vector<std::vector<int32_t>> chb((size_t)order + 1), chn((size_t)order + 1);
  for (int k = 1; k <= order; ++k) {
    chb[(size_t)k].assign((size_t)in[(size_t)k].n, 0);
    chn[(size_t)k].assign((size_t)in[(size_t)k].n, 0);
  }
  for (int64_t v = 0; v < V; ++v) {
    uni_logp[(size_t)v] = in[1].logp[in[1].at(v)];
    uni_tgt[(size_t)v] = (order >= 2) ? (int32_t)(base[1] + v) : 0;
    if (order >= 2) {
      int64_t s = base[1] + v;
      cum[(size_t)s] = in[1].bow ? (double)in[1].bow[in[1].at(v)] : 0.0;
      lm->st_tok[(size_t)s] = (int32_t)v;
    }
  }
  int64_t arc_off = 0;
  for (int k = 2; k <= order; ++k) {
    const OrderIn& o = in[(size_t)k];
    const OrderIn& lo = in[(size_t)k - 1];
    ctx[(size_t)k].assign((size_t)o.n, 0);
    sfx[(size_t)k].assign((size_t)o.n, 0);
    // contexts: prefixes are non-decreasing in sorted order -> merge
    int64_t p = 0;
    for (int64_t j = 0; j < o.n; ++j) {
      const int32_t* g = o.tok + o.at(j) * k;
      while (p < lo.n && tuple_less(lo.tok + lo.at(p) * (k - 1), g, k - 1)) ++p;
      if (p >= lo.n || !std::equal(g, g + k - 1, lo.tok + lo.at(p) * (k - 1)))
        return fail(TSD_EINVAL, "tsd_ngram_build: n-gram of order %d without its prefix (not prefix-closed)", k);
      ctx[(size_t)k][(size_t)j] = (int32_t)p;
      if (chn[(size_t)k - 1][(size_t)p] == 0) chb[(size_t)k - 1][(size_t)p] = (int32_t)j;
      chn[(size_t)k - 1][(size_t)p] += 1;
    }
    // suffixes: suffix(c.w) = suffix(c).w, searched among suffix(c)'s children
    std::vector<int32_t>& sf = sfx[(size_t)k];
    const std::vector<int32_t>& cx = ctx[(size_t)k];
    std::atomic<int> bad{0};
    const std::vector<int32_t>* lo_sfx = (k >= 3) ? &sfx[(size_t)k - 1] : nullptr;
    const std::vector<int32_t>& b2 = chb[(size_t)k - 2 >= 1 ? (size_t)k - 2 : 1];
    const std::vector<int32_t>& n2 = chn[(size_t)k - 2 >= 1 ? (size_t)k - 2 : 1];
    parallel_for(o.n, [&](int64_t b, int64_t e) {
      int local_bad = 0;
      for (int64_t j = b; j < e; ++j) {
        const int32_t* g = o.tok + o.at(j) * k;
        int32_t w = g[k - 1];
        if (k == 2) {
          sf[(size_t)j] = w;  // unigram w sits at sorted position w
          continue;
        }
        int32_t cs = (*lo_sfx)[(size_t)cx[(size_t)j]];  // suffix of the context, order k-2
        int32_t cb = b2[(size_t)cs], cn = n2[(size_t)cs];
        // children of cs in order k-1 are sorted by their last label
        int32_t l = 0, h = cn;
        while (l < h) {
          int32_t m = (l + h) / 2;
          int32_t t = lo.tok[lo.at(cb + m) * (k - 1) + (k - 2)];
          if (t < w) l = m + 1; else h = m;
        }
        if (l >= cn || lo.tok[lo.at(cb + l) * (k - 1) + (k - 2)] != w) {
          local_bad = 1;
          sf[(size_t)j] = -1;
        } else {
          sf[(size_t)j] = cb + l;
        }
      }
      if (local_bad) bad.store(1);
    });
    if (bad.load()) return fail(TSD_EINVAL, "tsd_ngram_build: n-gram of order %d without its suffix (not suffix-closed)", k);
    // arcs of order k, and states of order k (if below the top order)
    for (int64_t j = 0; j < o.n; ++j) {
      int64_t a = arc_off + j;
      int64_t i = o.at(j);
      arc_tok[(size_t)a] = o.tok[i * k + (k - 1)];
      arc_logp[(size_t)a] = o.logp[i];
      arc_tgt[(size_t)a] = (k < order) ? (int32_t)(base[(size_t)k] + j) : -1;
    }
    for (int64_t p2 = 0; p2 < lo.n; ++p2) {
      int64_t s = base[(size_t)k - 1] + p2;
      st_begin[(size_t)s] = (int32_t)(arc_off + chb[(size_t)k - 1][(size_t)p2]);
      st_count[(size_t)s] = chn[(size_t)k - 1][(size_t)p2];
    }
    if (k < order) {
      for (int64_t j = 0; j < o.n; ++j) {
        int64_t s = base[(size_t)k] + j;
        int64_t i = o.at(j);
        double bw = o.bow ? (double)o.bow[i] : 0.0;
        cum[(size_t)s] = bw + cum[(size_t)(base[(size_t)k - 1] + sf[(size_t)j])];
        lm->st_parent[(size_t)s] = (int32_t)(base[(size_t)k - 1] + cx[(size_t)j]);
        lm->st_tok[(size_t)s] = o.tok[i * k + (k - 1)];
      }
    }
    arc_off += o.n;
  }
  std::vector<float> st_cum((size_t)S);
  for (int64_t s = 0; s < S; ++s) st_cum[(size_t)s] = (float)cum[(size_t)s];
  // each arc's target record, and each unigram state's
  auto rec_of = [&](int64_t s) {
    int32_t cb;
    std::memcpy(&cb, &st_cum[(size_t)s], 4);
    return make_int4((int32_t)s, st_begin[(size_t)s], st_count[(size_t)s], cb);
  };
  std::vector<int4> arc_rec((size_t)total_arcs + 1), uni_rec((size_t)V);
  parallel_for(total_arcs, [&](int64_t b, int64_t e) {
    for (int64_t a = b; a < e; ++a) {
      const int32_t t = arc_tgt[(size_t)a];
      arc_rec[(size_t)a] = t >= 0 ? rec_of(t) : make_int4(-1, 0, 0, 0);
    }
  });
  arc_rec[(size_t)total_arcs] = make_int4(-1, 0, 0, 0);
  // a dense row for every unigram state u (V x V4 floats; left out above
  // 1 GiB): per label v the LM term of a row whose deepest state with an arc
  // v is u, relative to the call's defaults and the row's summed backoff:
  // log p(v | u) - log p(v) - cum(u), and 0 where u has no arc v
  const int64_t V4 = ((int64_t)V + 15) / 16 * 16;
  std::vector<int32_t> uni_dense((size_t)V, -1);
  int64_t n_dense = 0;
  if (order >= 2 && V * V4 * 4 <= (1ll << 30))
    for (int64_t u = 0; u < V; ++u) uni_dense[(size_t)u] = (int32_t)n_dense++;
  std::vector<float> dense0((size_t)std::max<int64_t>(1, n_dense) * V4, 0.f);
  parallel_for(n_dense > 0 ? V : 0, [&](int64_t b, int64_t e) {
    for (int64_t u = b; u < e; ++u) {
      const int32_t row = uni_dense[(size_t)u];
      const int64_t s = base[1] + u;
      for (int32_t a = st_begin[(size_t)s]; a < st_begin[(size_t)s] + st_count[(size_t)s]; ++a) {
        const int32_t t = arc_tok[(size_t)a];
        dense0[(size_t)row * V4 + t] =
            (float)((double)arc_logp[(size_t)a] - (double)uni_logp[(size_t)t] - cum[(size_t)s]);
      }
    }
  });
  for (int64_t u = 0; u < V; ++u) {
    if (order >= 2) {
      uni_rec[(size_t)u] = rec_of(uni_tgt[(size_t)u]);
      uni_rec[(size_t)u].x = uni_dense[(size_t)u];
    } else {
      uni_rec[(size_t)u] = make_int4(-1, 0, 0, 0);
    }
  }

  LmView& v = lm->view;
  v.V = V;
  v.order = order;
  v.n_states = S;
  v.n_arcs = total_arcs;
  int32_t *d_b, *d_c, *d_at, *d_ag, *d_ut;
  float *d_cum, *d_al, *d_ul;
  int4 *d_ar, *d_ur;
  float* d_dense;
  int32_t* d_ud;
  tsd_status st;
  // the row pass reads arcs in aligned groups of four: room for the last group
  arc_tok.resize((size_t)total_arcs + 4, 0);
  arc_logp.resize((size_t)total_arcs + 4, 0.f);
  if ((st = lm->arena.upload(&d_b, st_begin)) || (st = lm->arena.upload(&d_c, st_count)) ||
      (st = lm->arena.upload(&d_cum, st_cum)) || (st = lm->arena.upload(&d_at, arc_tok)) ||
      (st = lm->arena.upload(&d_al, arc_logp)) || (st = lm->arena.upload(&d_ag, arc_tgt)) ||
      (st = lm->arena.upload(&d_ul, uni_logp)) || (st = lm->arena.upload(&d_ut, uni_tgt)) ||
      (st = lm->arena.upload(&d_ar, arc_rec)) || (st = lm->arena.upload(&d_ur, uni_rec)) ||
      (st = lm->arena.upload(&d_dense, dense0)) || (st = lm->arena.upload(&d_ud, uni_dense))) {
    lm->arena.release();
    return st;
  }
  v.arc_rec = d_ar;
  v.uni_rec = d_ur;
  v.dense0 = d_dense;
  v.uni_dense = d_ud;
  v.V4 = (int32_t)V4;
  v.n_dense = (int32_t)n_dense;
  v.st_begin = d_b;
  v.st_count = d_c;
  v.st_cum = d_cum;
  v.arc_tok = d_at;
  v.arc_logp = d_al;
  v.arc_tgt = d_ag;
  v.uni_logp = d_ul;
  v.uni_tgt = d_ut;
  *out = lm.release();
  return TSD_OK;
}

extern "C" void tsd_ngram_free(tsd_ngram* lm) {
  if (!lm) return;
  lm->arena.release();
  delete lm;
}

extern "C" tsd_status tsd_ngram_info(const tsd_ngram* lm, int64_t* n_states, int64_t* n_arcs,
                                     int64_t* device_bytes) {
  clear_error();
  if (!lm) return fail(TSD_EINVAL, "tsd_ngram_info: NULL handle");
  if (n_states) *n_states = lm->view.n_states;
  if (n_arcs) *n_arcs = lm->view.n_arcs;
  if (device_bytes) *device_bytes = lm->arena.bytes;
  return TSD_OK;
}

extern "C" tsd_status tsd_ngram_state_tuple(const tsd_ngram* lm, int32_t state, int32_t* buf,
                                            int32_t cap, int32_t* len) {
  clear_error();
  if (!lm || !len) return fail(TSD_EINVAL, "tsd_ngram_state_tuple: NULL argument");
  if (state < 0 || state >= lm->view.n_states)
    return fail(TSD_EINVAL, "tsd_ngram_state_tuple: state %d out of range", state);
  int32_t tmp[kMaxOrder];
  int n = 0;
  for (int32_t s = state; s != 0 && n < kMaxOrder; s = lm->st_parent[(size_t)s]) tmp[n++] = lm->st_tok[(size_t)s];
  *len = n;
  for (int i = 0; i < n && i < cap; ++i) buf[i] = tmp[n - 1 - i];
  return TSD_OK;
}

// ---------------------------------------------------------------------------
// phrase trie
// ---------------------------------------------------------------------------
extern "C" tsd_status tsd_boost_build(int32_t V, int32_t n_phr, const int32_t* offsets,
                                      const int32_t* tokens, float token_bonus, tsd_boost** out) {
  clear_error();
  if (!out) return fail(TSD_EINVAL, "tsd_boost_build: out is NULL");
  *out = nullptr;
  if (V < 1 || V > 32767) return fail(TSD_EINVAL, "tsd_boost_build: V=%d out of range", V);
  if (n_phr < 0 || (n_phr > 0 && (!offsets || !tokens)))
    return fail(TSD_EINVAL, "tsd_boost_build: bad phrase arrays");
  if (!std::isfinite(token_bonus)) return fail(TSD_EINVAL, "tsd_boost_build: non-finite bonus");
  // trie with ordered children
  std::vector<std::map<int32_t, int32_t>> kids(1);
  std::vector<int32_t> depth(1, 0), parent(1, 0), tok(1, -1);
  std::vector<uint8_t> term(1, 0);
  for (int32_t i = 0; i < n_phr; ++i) {
    int32_t b = offsets[i], e = offsets[i + 1];
    if (b < 0 || e <= b) return fail(TSD_EINVAL, "tsd_boost_build: phrase %d is empty or has bad offsets", i);
    if (e - b > kMaxPhrase) return fail(TSD_EINVAL, "tsd_boost_build: phrase %d longer than %d", i, kMaxPhrase);
    int32_t node = 0;
    for (int32_t j = b; j < e; ++j) {
      int32_t t = tokens[j];
      if (t < 0 || t >= V) return fail(TSD_EINVAL, "tsd_boost_build: label %d out of [0, %d)", t, V);
      auto it = kids[(size_t)node].find(t);
      if (it == kids[(size_t)node].end()) {
        int32_t c = (int32_t)kids.size();
        kids[(size_t)node][t] = c;
        kids.emplace_back();
        depth.push_back(depth[(size_t)node] + 1);
        parent.push_back(node);
        tok.push_back(t);
        term.push_back(0);
        node = c;
      } else {
        node = it->second;
      }
    }
    term[(size_t)node] = 1;
  }
  const int32_t Q = (int32_t)kids.size();
  std::vector<int32_t> nd_begin((size_t)Q), nd_count((size_t)Q), nd_fail((size_t)Q, 0);
  std::vector<int32_t> ch_tok, ch_node, ch_next;
  int32_t max_depth = 0;
  for (int32_t q = 0; q < Q; ++q) {
    nd_begin[(size_t)q] = (int32_t)ch_tok.size();
    nd_count[(size_t)q] = (int32_t)kids[(size_t)q].size();
    for (auto& kv : kids[(size_t)q]) {
      ch_tok.push_back(kv.first);
      ch_node.push_back(kv.second);
      ch_next.push_back(term[(size_t)kv.second] ? 0 : kv.second);
    }
    max_depth = std::max(max_depth, depth[(size_t)q]);
  }
  // failure links in breadth-first order: fail(child(q, a)) = goto(fail(q), a)
  {
    std::vector<int32_t> queue;
    for (auto& kv : kids[0]) queue.push_back(kv.second);
    for (size_t h = 0; h < queue.size(); ++h) {
      int32_t q = queue[h];
      for (auto& kv : kids[(size_t)q]) {
        int32_t a = kv.first, c = kv.second;
        int32_t f = nd_fail[(size_t)q];
        if (q == 0) f = 0;
        int32_t g = 0;
        for (;;) {
          auto it = kids[(size_t)f].find(a);
          if (it != kids[(size_t)f].end() && it->second != c) { g = it->second; break; }
          if (f == 0) break;
          f = nd_fail[(size_t)f];
        }
        nd_fail[(size_t)c] = g;
        queue.push_back(c);
      }
    }
  }
  std::vector<int32_t> root_child((size_t)V, 0), root_next((size_t)V, 0);
  for (auto& kv : kids[0]) {
    root_child[(size_t)kv.first] = kv.second;
    root_next[(size_t)kv.first] = term[(size_t)kv.second] ? 0 : kv.second;
  }
  std::unique_ptr<tsd_boost> b(new tsd_boost());
  b->nd_parent = parent;
  b->nd_tok = tok;
  TrieView& v = b->view;
  v.V = V;
  v.n_nodes = Q;
  v.max_depth = max_depth;
  v.bonus = token_bonus;
  int32_t *a0 = nullptr, *a1 = nullptr, *a2 = nullptr, *a3 = nullptr, *a4 = nullptr, *a5 = nullptr, *a6 = nullptr,
          *a7 = nullptr, *a8 = nullptr;
  tsd_status st;
  std::vector<int4> ch_rec(ch_tok.size() + 1, make_int4(-1, 0, 0, 0)), root_rec((size_t)V, make_int4(0, 0, 0, 0));
  for (size_t c = 0; c < ch_tok.size(); ++c) {
    const int32_t q = ch_node[c];
    ch_rec[c] = make_int4(q, ch_next[c], nd_begin[(size_t)q], nd_count[(size_t)q]);
  }
  for (int32_t u = 0; u < V; ++u) {
    const int32_t q = root_child[(size_t)u];
    if (q) root_rec[(size_t)u] = make_int4(q, root_next[(size_t)u], nd_begin[(size_t)q], nd_count[(size_t)q]);
  }
  ch_tok.resize(ch_tok.size() + 4, 0);  // aligned groups of four in the row pass
  if ((st = b->arena.upload(&a0, nd_begin)) || (st = b->arena.upload(&a1, nd_count)) ||
      (st = b->arena.upload(&a2, depth)) || (st = b->arena.upload(&a3, nd_fail)) ||
      (st = b->arena.upload(&a4, ch_tok)) || (st = b->arena.upload(&a5, ch_node)) ||
      (st = b->arena.upload(&a6, ch_next)) || (st = b->arena.upload(&a7, root_child)) ||
      (st = b->arena.upload(&a8, root_next))) {
    b->arena.release();
    return st;
  }
  int4 *r0 = nullptr, *r1 = nullptr;
  if ((st = b->arena.upload(&r0, ch_rec)) || (st = b->arena.upload(&r1, root_rec))) {
    b->arena.release();
    return st;
  }
  v.ch_rec = r0;
  v.root_rec = r1;
  v.n_children = (int32_t)ch_node.size();
  v.nd_begin = a0;
  v.nd_count = a1;
  v.nd_depth = a2;
  v.nd_fail = a3;
  v.ch_tok = a4;
  v.ch_node = a5;
  v.ch_next = a6;
  v.root_child = a7;
  v.root_next = a8;
  *out = b.release();
  return TSD_OK;
}

extern "C" void tsd_boost_free(tsd_boost* b) {
  if (!b) return;
  b->arena.release();
  delete b;
}

extern "C" tsd_status tsd_boost_info(const tsd_boost* b, int32_t* n_nodes, int32_t* max_depth,
                                     int64_t* device_bytes) {
  clear_error();
  if (!b) return fail(TSD_EINVAL, "tsd_boost_info: NULL handle");
  if (n_nodes) *n_nodes = b->view.n_nodes;
  if (max_depth) *max_depth = b->view.max_depth;
  if (device_bytes) *device_bytes = b->arena.bytes;
  return TSD_OK;
}

extern "C" tsd_status tsd_boost_node_tuple(const tsd_boost* b, int32_t node, int32_t* buf,
                                           int32_t cap, int32_t* len) {
  clear_error();
  if (!b || !len) return fail(TSD_EINVAL, "tsd_boost_node_tuple: NULL argument");
  if (node < 0 || node >= b->view.n_nodes) return fail(TSD_EINVAL, "tsd_boost_node_tuple: node %d out of range", node);
  int32_t tmp[kMaxPhrase];
  int n = 0;
  for (int32_t q = node; q != 0 && n < kMaxPhrase; q = b->nd_parent[(size_t)q]) tmp[n++] = b->nd_tok[(size_t)q];
  *len = n;
  for (int i = 0; i < n && i < cap; ++i) buf[i] = tmp[n - 1 - i];
  return TSD_OK;
}
