// ORACLE -- test infrastructure, not part of the product.
//
// A plain, slow, obviously correct CPU implementation of the batched
// Transducer decode step with shallow fusion (Sec. III-C, Eq. 1 of the
// paper): joint logits, log-softmax, a weighted backoff n-gram score and a
// weighted phrase-boost bonus for every non-blank token, greedy (or beam)
// selection, and the advance of each hypothesis's history.  Floating point is
// double throughout, on the same bf16 inputs the GPU path receives.
//
// It shares no code with the CUDA library (no common headers, helpers or
// tables) and neither imports the other.  Only the test suite, the smoke
// check and the benchmark's CPU-baseline leg may load it.
//
// Functions and the passage each follows:
//   * joint logits:     x = bf16(ReLU(enc_t + E[last])), logits = W_out^T x
//                       (the workload's joint definition; Fig. 1 of the paper:
//                       prediction + joint networks propose candidates)
//   * log-softmax:      log p_AM(y|x) over all V+1 outputs (Eq. 1, term 1)
//   * n-gram score:     textbook backoff over a dictionary of n-grams
//                       (Eq. 1, term 2: a weighted sum over one or more LMs,
//                       sum_i alpha_i log p_LM_i; "n-gram language models
//                       over sub-word tokens", Sec. III-C).  Natural log.
//   * boost bonus:      naive suffix matching against the phrase list
//                       (Eq. 1, term 3; "phrase-boosting tree from a user word
//                       list", Sec. III-C).  Reading: bonus per token times the
//                       change of the longest matched phrase prefix; a
//                       completed phrase is banked and matching restarts.
//   * greedy decoding:  argmax of the fused score, lowest id on ties; blank
//                       (id V) or max_sym emissions end the frame (Sec. III:
//                       "greedy decoding emits text").  Pruned variant (the
//                       reading of Sec. III-C's remark that fusion only
//                       re-ranks the candidates the acoustic model proposes):
//                       the argmax runs over the acoustic model's k best
//                       outputs only (blank included, ties to the lower id).
//   * prediction network (the Transducer's stateful form, Fig. 1's
//                       prediction + joint networks): a one-layer LSTM over the
//                       previous label (blank = start of sequence) and joint
//                       projections, joint input = bf16(ReLU(W_enc enc_t + b_enc
//                       + W_pred h + b_pred)); the LSTM advances on every
//                       emitted label.
//   * beam search:      per frame up to S expansions, each the top-K of the
//                       extensions of the hypotheses still in the frame;
//                       identical label sequences merged by log-sum-exp.
//                       (Not in the paper; the beam workload defines it.)
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <set>
#include <vector>

#define ORACLE_API extern "C" __attribute__((visibility("default")))

namespace {

// bf16 bit pattern -> float (exact)
float bf16_bits_to_float(uint16_t b) {
  uint32_t x = (uint32_t)b << 16;
  float f;
  std::memcpy(&f, &x, 4);
  return f;
}

// float -> bf16 bit pattern, round to nearest even (inputs are finite)
uint16_t float_to_bf16_bits(float f) {
  uint32_t x;
  std::memcpy(&x, &f, 4);
  uint32_t keep = x >> 16;
  uint32_t rest = x & 0xFFFFu;
  if (rest > 0x8000u || (rest == 0x8000u && (keep & 1u))) keep += 1;
  return (uint16_t)keep;
}

// ---------------------------------------------------------------------------
// Dictionary of n-grams.  Order k holds its n-grams as sorted k-tuples; a
// lookup is a binary search for the exact tuple.
// ---------------------------------------------------------------------------
struct NGramDict {
  int32_t V = 0, N = 0;
  std::vector<std::vector<int32_t>> toks;  // [k-1]: n_k * k tokens, sorted
  std::vector<std::vector<double>> logp;   // [k-1]
  std::vector<std::vector<double>> bow;    // [k-1]

  // index of the tuple g (length k) in order k, or -1
  int64_t find(const int32_t* g, int k) const {
    if (k < 1 || k > N) return -1;
    const std::vector<int32_t>& t = toks[k - 1];
    int64_t lo = 0, hi = (int64_t)logp[k - 1].size();
    while (lo < hi) {
      int64_t mid = lo + (hi - lo) / 2;
      const int32_t* x = &t[(size_t)mid * k];
      if (std::lexicographical_compare(x, x + k, g, g + k)) lo = mid + 1;
      else hi = mid;
    }
    if (lo < (int64_t)logp[k - 1].size() && std::equal(g, g + k, &t[(size_t)lo * k])) return lo;
    return -1;
  }

  // log p(v | h) by backoff:
  //   p(h.v) if the n-gram h.v exists, else bow(h) + score(v | h[1:]),
  //   bow(h) = 0 if h is not in the dictionary; the empty context gives the
  //   unigram.  h holds at most N-1 tokens here.
  double score_ctx(const int32_t* h, int len, int32_t v) const {
    std::vector<int32_t> hv(h, h + len);
    hv.push_back(v);
    int64_t i = find(hv.data(), len + 1);
    if (i >= 0) return logp[len][(size_t)i];
    if (len == 0) return -std::numeric_limits<double>::infinity();
    int64_t j = find(h, len);
    double b = (j >= 0) ? bow[len - 1][(size_t)j] : 0.0;
    return b + score_ctx(h + 1, len - 1, v);
  }

  double score(const int32_t* hist, int64_t len, int32_t v) const {
    int64_t n = std::min<int64_t>(len, N - 1);
    return score_ctx(hist + (len - n), (int)n, v);
  }

  // The LM state of a history: its longest suffix of at most N-1 tokens that
  // is an n-gram of the model (the empty tuple if none).
  int state(const int32_t* hist, int64_t len, int32_t* out) const {
    int64_t n = std::min<int64_t>(len, N - 1);
    for (int64_t l = n; l >= 1; --l) {
      if (find(hist + (len - l), (int)l) >= 0) {
        std::memcpy(out, hist + (len - l), sizeof(int32_t) * (size_t)l);
        return (int)l;
      }
    }
    return 0;
  }
};

// ---------------------------------------------------------------------------
// Phrase list, matched naively: P = all non-empty phrase prefixes, F = the
// phrases.  m(g) = the largest l <= |g| with the last l tokens of g in P.
// ---------------------------------------------------------------------------
struct PhraseSet {
  int32_t V = 0;
  double bonus = 0;
  int max_len = 0;
  std::set<std::vector<int32_t>> prefixes, full;

  int match(const int32_t* g, int64_t len) const {
    int64_t top = std::min<int64_t>(len, max_len);
    for (int64_t l = top; l >= 1; --l) {
      std::vector<int32_t> s(g + (len - l), g + len);
      if (prefixes.count(s)) return (int)l;
    }
    return 0;
  }
  bool is_phrase(const int32_t* g, int64_t len) const {
    return full.count(std::vector<int32_t>(g, g + len)) > 0;
  }
  // bonus for emitting v after the unmatched-history g
  double score(const int32_t* g, int64_t len, int32_t v) const {
    std::vector<int32_t> gv(g, g + len);
    gv.push_back(v);
    return bonus * (double)(match(gv.data(), len + 1) - match(g, len));
  }
};

// One stream (greedy) or one hypothesis (beam): emitted labels and the index
// where phrase matching restarts.
struct Hyp {
  std::vector<int32_t> y;
  int64_t rho = 0;
  double score = 0;
  int32_t last(int32_t V) const { return y.empty() ? V : y.back(); }
};

// Prediction network weights (bf16 bit patterns, fp32 biases).
struct PredNet {
  int32_t V, D, Henc, H;
  const uint16_t* Ep;  // [V+1][D] label embedding; row V starts a sequence
  const uint16_t* Wg;  // [2D][4D]: rows x (embedding) then h; column 4u+q is gate q (i, f, g, o) of unit u
  const float* bg;     // [4D]
  const uint16_t* Wp;  // [D][H]
  const float* bp;     // [H]
  const uint16_t* We;  // [Henc][H]
  const float* be;     // [H]
};

// LSTM state: h as the bf16 the next products read, c in double.
struct PredState {
  std::vector<uint16_t> h;
  std::vector<double> c;
  bool ready = false;
};

struct Stream {
  int32_t V = 0;
  Hyp greedy;
  std::vector<Hyp> beam;  // empty until the first beam chunk
  PredState pred;
};

// After v was appended to h.y: restart matching if the longest matched
// prefix is a complete phrase.
void advance_rho(const PhraseSet* b, Hyp& h) {
  if (!b) return;
  const int32_t* g = h.y.data() + h.rho;
  int64_t len = (int64_t)h.y.size() - h.rho;
  int l = b->match(g, len);
  if (l > 0 && b->is_phrase(g + (len - l), l)) h.rho = (int64_t)h.y.size();
}

struct Model {
  int32_t V, H;
  const uint16_t* E;  // [V+1][H]
  const uint16_t* W;  // [H][V+1]
};

double sigmoid(double x) { return 1.0 / (1.0 + std::exp(-x)); }

// One LSTM step on label y: gates = bg + x W_g[0:D] + h W_g[D:2D] with
// x = Ep[y]; c' = s(f) c + s(i) tanh(g); h' = s(o) tanh(c'); h' is kept as
// the bf16 (through fp32) the next products read.
void lstm_step(const PredNet& p, int32_t y, PredState& st) {
  const int32_t D = p.D;
  if (!st.ready) {
    st.h.assign((size_t)D, 0);
    st.c.assign((size_t)D, 0.0);
    st.ready = true;
  }
  std::vector<double> g((size_t)4 * D);
  for (int32_t j = 0; j < 4 * D; ++j) g[(size_t)j] = (double)p.bg[j];
  for (int32_t k = 0; k < D; ++k) {
    const double xk = (double)bf16_bits_to_float(p.Ep[(size_t)y * D + k]);
    const double hk = (double)bf16_bits_to_float(st.h[(size_t)k]);
    const uint16_t* wx = p.Wg + (size_t)k * 4 * D;
    const uint16_t* wh = p.Wg + (size_t)(D + k) * 4 * D;
    for (int32_t j = 0; j < 4 * D; ++j)
      g[(size_t)j] += xk * (double)bf16_bits_to_float(wx[j]) + hk * (double)bf16_bits_to_float(wh[j]);
  }
  for (int32_t u = 0; u < D; ++u) {
    const double i = sigmoid(g[(size_t)4 * u]), f = sigmoid(g[(size_t)4 * u + 1]);
    const double gg = std::tanh(g[(size_t)4 * u + 2]), o = sigmoid(g[(size_t)4 * u + 3]);
    const double c = f * st.c[(size_t)u] + i * gg;
    st.c[(size_t)u] = c;
    st.h[(size_t)u] = float_to_bf16_bits((float)(o * std::tanh(c)));
  }
}

// Joint input of the stateful form: bf16(ReLU(W_enc enc_t + b_enc + W_pred h + b_pred)),
// the sum taken to fp32 before the rounding to bf16 (as the kernels store it).
void pred_joint_input(const PredNet& p, const uint16_t* enc_t, const PredState& st, std::vector<float>& x) {
  const int32_t H = p.H;
  std::vector<double> a((size_t)H);
  for (int32_t j = 0; j < H; ++j) a[(size_t)j] = (double)p.be[j] + (double)p.bp[j];
  for (int32_t k = 0; k < p.Henc; ++k) {
    const double ek = (double)bf16_bits_to_float(enc_t[k]);
    const uint16_t* w = p.We + (size_t)k * H;
    for (int32_t j = 0; j < H; ++j) a[(size_t)j] += ek * (double)bf16_bits_to_float(w[j]);
  }
  for (int32_t k = 0; k < p.D; ++k) {
    const double hk = (double)bf16_bits_to_float(st.h[(size_t)k]);
    const uint16_t* w = p.Wp + (size_t)k * H;
    for (int32_t j = 0; j < H; ++j) a[(size_t)j] += hk * (double)bf16_bits_to_float(w[j]);
  }
  x.resize((size_t)H);
  for (int32_t j = 0; j < H; ++j) {
    float v = (float)a[(size_t)j];
    if (v < 0.0f) v = 0.0f;
    x[(size_t)j] = bf16_bits_to_float(float_to_bf16_bits(v));
  }
}

// The LM term of Eq. 1: sum over the LMs of alpha_i * log p_LM_i(v | y),
// summed in the LMs' order.
struct LmTerm {
  static constexpr int kMax = 8;
  int n = 0;
  const NGramDict* lm[kMax] = {};
  double alpha[kMax] = {};
  double score(const int32_t* y, int64_t len, int32_t v) const {
    double t = alpha[0] * lm[0]->score(y, len, v);
    for (int i = 1; i < n; ++i) t += alpha[i] * lm[i]->score(y, len, v);
    return t;
  }
};

LmTerm one_lm(const void* lmp, double lambda) {
  LmTerm t;
  if (lmp) {
    t.n = 1;
    t.lm[0] = static_cast<const NGramDict*>(lmp);
    t.alpha[0] = lambda;
  }
  return t;
}

// fused[v] = log_softmax(logits)[v] + sum_i alpha_i*lm_i(v|y) + beta*boost(v|y[rho:]),
// fused[V] = log_softmax(logits)[V]
void fused_scores(const Model& m, const uint16_t* enc_t, const Hyp& h, const LmTerm& lms,
                  const PhraseSet* boost, double beta, std::vector<float>& x,
                  std::vector<double>& logits, std::vector<double>& fused, bool x_given = false) {
  const int32_t V = m.V, H = m.H, N = V + 1;
  const int32_t last = h.last(V);
  if (!x_given) x.resize((size_t)H);
  for (int32_t k = 0; k < H && !x_given; ++k) {
    float s = bf16_bits_to_float(enc_t[k]) + bf16_bits_to_float(m.E[(size_t)last * H + k]);
    if (s < 0.0f) s = 0.0f;
    x[(size_t)k] = bf16_bits_to_float(float_to_bf16_bits(s));
  }
  logits.assign((size_t)N, 0.0);
  for (int32_t k = 0; k < H; ++k) {
    const double xk = (double)x[(size_t)k];
    const uint16_t* wk = m.W + (size_t)k * N;
    for (int32_t v = 0; v < N; ++v) logits[(size_t)v] += xk * (double)bf16_bits_to_float(wk[v]);
  }
  double mx = -std::numeric_limits<double>::infinity();
  for (int32_t v = 0; v < N; ++v) mx = std::max(mx, logits[(size_t)v]);
  double se = 0;
  for (int32_t v = 0; v < N; ++v) se += std::exp(logits[(size_t)v] - mx);
  const double lse = mx + std::log(se);
  fused.assign((size_t)N, 0.0);
  const int32_t* y = h.y.data();
  const int64_t ylen = (int64_t)h.y.size();
  for (int32_t v = 0; v < V; ++v) {
    double f = logits[(size_t)v] - lse;
    if (lms.n) f += lms.score(y, ylen, v);
    if (boost) f += beta * boost->score(y + h.rho, ylen - h.rho, v);
    fused[(size_t)v] = f;
  }
  fused[(size_t)V] = logits[(size_t)V] - lse;
}

double logaddexp(double a, double b) {
  if (a == -std::numeric_limits<double>::infinity()) return b;
  if (b == -std::numeric_limits<double>::infinity()) return a;
  double m = std::max(a, b);
  return m + std::log(std::exp(a - m) + std::exp(b - m));
}

}  // namespace

// ===========================================================================
// C ABI
// ===========================================================================

// Builds the n-gram dictionary from per-order arrays: count[k-1] n-grams of
// order k, tokens[k-1] row-major [count][k], natural-log logp and bow (bow of
// the top order is ignored).  Returns NULL if a token is out of range, a
// unigram is missing or an n-gram repeats.
ORACLE_API void* oracle_lm_new(int32_t V, int32_t order, const int64_t* count,
                               const int32_t* const* tokens, const float* const* logp,
                               const float* const* bow) {
  if (V < 1 || order < 1) return nullptr;
  NGramDict* d = new NGramDict();
  d->V = V;
  d->N = order;
  d->toks.resize((size_t)order);
  d->logp.resize((size_t)order);
  d->bow.resize((size_t)order);
  for (int k = 1; k <= order; ++k) {
    int64_t n = count[k - 1];
    const int32_t* t = tokens[k - 1];
    // sort the tuples (unless they already come sorted)
    bool sorted = true;
    for (int64_t i = 1; i < n && sorted; ++i)
      sorted = std::lexicographical_compare(t + (i - 1) * k, t + i * k, t + i * k, t + i * k + k);
    std::vector<int64_t> idx;
    if (!sorted) {
      idx.resize((size_t)n);
      for (int64_t i = 0; i < n; ++i) idx[(size_t)i] = i;
      std::sort(idx.begin(), idx.end(), [&](int64_t a, int64_t b) {
        return std::lexicographical_compare(t + a * k, t + a * k + k, t + b * k, t + b * k + k);
      });
    }
    std::vector<int32_t>& dt = d->toks[(size_t)k - 1];
    dt.resize((size_t)n * k);
    d->logp[(size_t)k - 1].resize((size_t)n);
    d->bow[(size_t)k - 1].resize((size_t)n);
    for (int64_t j = 0; j < n; ++j) {
      int64_t i = sorted ? j : idx[(size_t)j];
      for (int q = 0; q < k; ++q) {
        int32_t tok = t[i * k + q];
        if (tok < 0 || tok >= V) { delete d; return nullptr; }
        dt[(size_t)j * k + q] = tok;
      }
      d->logp[(size_t)k - 1][(size_t)j] = (double)logp[k - 1][i];
      d->bow[(size_t)k - 1][(size_t)j] = (k < order && bow && bow[k - 1]) ? (double)bow[k - 1][i] : 0.0;
      if (j > 0 && std::equal(&dt[(size_t)(j - 1) * k], &dt[(size_t)(j - 1) * k] + k, &dt[(size_t)j * k])) {
        delete d;
        return nullptr;
      }
    }
  }
  if ((int64_t)d->logp[0].size() != V) { delete d; return nullptr; }
  return d;
}

ORACLE_API void oracle_lm_free(void* p) { delete static_cast<NGramDict*>(p); }

ORACLE_API double oracle_lm_score(const void* p, const int32_t* hist, int64_t len, int32_t v) {
  return static_cast<const NGramDict*>(p)->score(hist, len, v);
}

ORACLE_API int32_t oracle_lm_state(const void* p, const int32_t* hist, int64_t len, int32_t* out) {
  return static_cast<const NGramDict*>(p)->state(hist, len, out);
}

// Bow of an explicit context tuple (0 when absent) and logp of an explicit
// n-gram (NaN when absent): raw dictionary lookups for tests.
ORACLE_API double oracle_lm_lookup(const void* p, const int32_t* g, int32_t k, int32_t want_bow) {
  const NGramDict* d = static_cast<const NGramDict*>(p);
  int64_t i = d->find(g, k);
  if (i < 0) return want_bow ? 0.0 : std::numeric_limits<double>::quiet_NaN();
  return want_bow ? d->bow[(size_t)k - 1][(size_t)i] : d->logp[(size_t)k - 1][(size_t)i];
}

ORACLE_API void* oracle_boost_new(int32_t V, int32_t n_phr, const int32_t* offsets,
                                  const int32_t* tokens, double bonus) {
  PhraseSet* b = new PhraseSet();
  b->V = V;
  b->bonus = bonus;
  for (int32_t i = 0; i < n_phr; ++i) {
    int32_t len = offsets[i + 1] - offsets[i];
    if (len < 1) continue;
    std::vector<int32_t> p(tokens + offsets[i], tokens + offsets[i + 1]);
    for (int32_t tok : p)
      if (tok < 0 || tok >= V) { delete b; return nullptr; }
    for (int32_t l = 1; l <= len; ++l) b->prefixes.insert(std::vector<int32_t>(p.begin(), p.begin() + l));
    b->full.insert(p);
    b->max_len = std::max(b->max_len, (int)len);
  }
  return b;
}

ORACLE_API void oracle_boost_free(void* p) { delete static_cast<PhraseSet*>(p); }

ORACLE_API int32_t oracle_boost_match(const void* p, const int32_t* g, int64_t len) {
  return static_cast<const PhraseSet*>(p)->match(g, len);
}

ORACLE_API int32_t oracle_boost_is_phrase(const void* p, const int32_t* g, int64_t len) {
  return static_cast<const PhraseSet*>(p)->is_phrase(g, len) ? 1 : 0;
}

ORACLE_API double oracle_boost_score(const void* p, const int32_t* g, int64_t len, int32_t v) {
  return static_cast<const PhraseSet*>(p)->score(g, len, v);
}

ORACLE_API void* oracle_stream_new(int32_t V) {
  Stream* s = new Stream();
  s->V = V;
  return s;
}

ORACLE_API void oracle_stream_free(void* p) { delete static_cast<Stream*>(p); }

// Greedy history: copies up to cap labels, returns the full length.
ORACLE_API int64_t oracle_stream_history(const void* p, int32_t* buf, int64_t cap) {
  const Stream* s = static_cast<const Stream*>(p);
  int64_t n = (int64_t)s->greedy.y.size();
  for (int64_t i = 0; i < n && i < cap; ++i) buf[i] = s->greedy.y[(size_t)i];
  return n;
}

ORACLE_API int64_t oracle_stream_rho(const void* p) { return static_cast<const Stream*>(p)->greedy.rho; }

// Replaces the greedy history (e.g. to start from a given state).
ORACLE_API void oracle_stream_set_history(void* p, const int32_t* y, int64_t len, int64_t rho) {
  Stream* s = static_cast<Stream*>(p);
  s->greedy.y.assign(y, y + len);
  s->greedy.rho = rho;
}

// Report layout for oracle_decode_chunk / oracle_beam_chunk.
enum {
  REP_STEPS = 0,        // joint evaluations
  REP_MISMATCH = 1,     // followed decisions that lose to the oracle's argmax by more than gap_tol
  REP_NEAR_TIE = 2,     // followed decisions that differ from the argmax within gap_tol
  REP_MAX_SCORE_DIFF = 3,
  REP_MIN_GAP = 4,      // smallest top-2 gap seen
  REP_FIRST_BAD = 5,    // step of the first mismatch (-1 if none)
  REP_INCONSISTENT = 6, // followed sequence impossible under the decode rules
  REP_N = 8
};

// Greedy decode of one chunk of T frames for one stream (Sec. III; the
// frame loop of a Transducer with at most max_sym labels per frame).
//
// Free-running when follow_tok is NULL.  Otherwise the decisions under test
// are followed (follow_tok/frame/score, follow_count entries: the emitted
// labels and the frame each was emitted at, in order); at every evaluation
// the oracle checks that the followed decision is its own argmax or within
// gap_tol of it, and that the followed label's fused score is within
// score tolerance of its own (the largest difference is reported).
// Returns the number of labels emitted (written to out_* up to out_cap).
namespace {
// The acoustic model's k best outputs by logit (ties to the lower id).
std::vector<int32_t> am_top(const std::vector<double>& logits, int32_t k) {
  std::vector<int32_t> idx(logits.size());
  for (size_t v = 0; v < idx.size(); ++v) idx[v] = (int32_t)v;
  std::stable_sort(idx.begin(), idx.end(),
                   [&](int32_t a, int32_t b) { return logits[(size_t)a] > logits[(size_t)b]; });
  idx.resize((size_t)std::min<int64_t>(k, (int64_t)idx.size()));
  return idx;
}

// prune_k > 0: the decision is the best fused value among the acoustic
// model's prune_k best outputs.  In follow mode a followed label at the
// edge of that set (its logit within am_tol of the k-th) is accepted, and it
// is compared with the best fused value among the outputs that are in the
// set by more than am_tol.
int32_t decode_chunk_impl(Stream* s, const LmTerm& lm, const PhraseSet* boost, int32_t V, int32_t H,
                          const uint16_t* E, const uint16_t* W, const uint16_t* enc, int32_t T, double beta,
                          int32_t max_sym, const int32_t* follow_tok, const int32_t* follow_frame,
                          const float* follow_score, int32_t follow_count, double gap_tol, int32_t* out_tok,
                          int32_t* out_frame, double* out_score, int32_t out_cap, double* report,
                          int32_t prune_k = 0, double am_tol = 0.0, const PredNet* pn = nullptr) {
  Model m{V, H, E, W};
  std::vector<float> x;
  std::vector<double> logits, fused;
  double rep[REP_N] = {0, 0, 0, 0, std::numeric_limits<double>::infinity(), -1, 0, 0};
  int32_t emitted = 0, fpos = 0;
  Hyp& h = s->greedy;
  for (int32_t t = 0; t < T; ++t) {
    for (int32_t sym = 0; sym < max_sym;) {
      if (pn) {
        if (!s->pred.ready) lstm_step(*pn, V, s->pred);  // start of sequence
        pred_joint_input(*pn, enc + (size_t)t * pn->Henc, s->pred, x);
      }
      fused_scores(m, pn ? nullptr : enc + (size_t)t * H, h, lm, boost, beta, x, logits, fused, pn != nullptr);
      std::vector<uint8_t> cand((size_t)V + 1, prune_k > 0 ? 0 : 1);
      double kth = -std::numeric_limits<double>::infinity();
      if (prune_k > 0) {
        const std::vector<int32_t> top = am_top(logits, prune_k);
        for (int32_t c : top) cand[(size_t)c] = 1;
        kth = logits[(size_t)top.back()];
      }
      int32_t best = -1;
      for (int32_t v = 0; v <= V; ++v)
        if (cand[(size_t)v] && (best < 0 || fused[(size_t)v] > fused[(size_t)best])) best = v;
      double second = -std::numeric_limits<double>::infinity();
      for (int32_t v = 0; v <= V; ++v)
        if (cand[(size_t)v] && v != best) second = std::max(second, fused[(size_t)v]);
      rep[REP_MIN_GAP] = std::min(rep[REP_MIN_GAP], fused[(size_t)best] - second);
      int32_t y = best;
      if (follow_tok) {
        int32_t fy = (fpos < follow_count && follow_frame[fpos] == t) ? follow_tok[fpos] : V;
        if (fpos < follow_count && follow_frame[fpos] < t) rep[REP_INCONSISTENT] = 1;
        if (fy < 0 || fy > V) { rep[REP_INCONSISTENT] = 1; fy = V; }
        if (fy != best) {
          double gap = fused[(size_t)best] - fused[(size_t)fy];
          if (prune_k > 0) {
            // the best among the outputs surely in both candidate sets
            int32_t sure = -1;
            for (int32_t v = 0; v <= V; ++v)
              if (logits[(size_t)v] > kth + am_tol && (sure < 0 || fused[(size_t)v] > fused[(size_t)sure])) sure = v;
            gap = sure >= 0 ? fused[(size_t)sure] - fused[(size_t)fy] : 0.0;
            if (logits[(size_t)fy] < kth - am_tol) gap = std::numeric_limits<double>::infinity();
          }
          if (gap > gap_tol) {
            rep[REP_MISMATCH] += 1;
            if (rep[REP_FIRST_BAD] < 0) rep[REP_FIRST_BAD] = rep[REP_STEPS];
          } else {
            rep[REP_NEAR_TIE] += 1;
          }
        }
        if (fy != V) {
          double d = std::fabs((double)follow_score[fpos] - fused[(size_t)fy]);
          rep[REP_MAX_SCORE_DIFF] = std::max(rep[REP_MAX_SCORE_DIFF], d);
          ++fpos;
        }
        y = fy;
      }
      rep[REP_STEPS] += 1;
      if (y == V) break;
      if (emitted < out_cap) {
        out_tok[emitted] = y;
        out_frame[emitted] = t;
        out_score[emitted] = fused[(size_t)y];
      }
      ++emitted;
      h.y.push_back(y);
      advance_rho(boost, h);
      if (pn) lstm_step(*pn, y, s->pred);  // the prediction network reads the emitted label
      ++sym;
    }
  }
  if (follow_tok && fpos != follow_count) rep[REP_INCONSISTENT] = 1;
  if (report)
    for (int i = 0; i < REP_N; ++i) report[i] = rep[i];
  return emitted;
}
}  // namespace

ORACLE_API int32_t oracle_decode_chunk(void* sp, const void* lmp, const void* boostp, int32_t V,
                                       int32_t H, const uint16_t* E, const uint16_t* W,
                                       const uint16_t* enc, int32_t T, double lambda, double beta,
                                       int32_t max_sym, const int32_t* follow_tok,
                                       const int32_t* follow_frame, const float* follow_score,
                                       int32_t follow_count, double gap_tol, int32_t* out_tok,
                                       int32_t* out_frame, double* out_score, int32_t out_cap,
                                       double* report) {
  return decode_chunk_impl(static_cast<Stream*>(sp), one_lm(lmp, lambda), static_cast<const PhraseSet*>(boostp),
                           V, H, E, W, enc, T, beta, max_sym, follow_tok, follow_frame, follow_score, follow_count,
                           gap_tol, out_tok, out_frame, out_score, out_cap, report);
}

// The pruned variant: fusion re-ranks only the acoustic model's prune_k
// best outputs (see decode_chunk_impl); am_tol is the logit tolerance at the
// edge of that set in follow mode.
ORACLE_API int32_t oracle_decode_chunk_pruned(void* sp, const void* lmp, const void* boostp, int32_t V, int32_t H,
                                              const uint16_t* E, const uint16_t* W, const uint16_t* enc, int32_t T,
                                              double lambda, double beta, int32_t max_sym, int32_t prune_k,
                                              double am_tol, const int32_t* follow_tok, const int32_t* follow_frame,
                                              const float* follow_score, int32_t follow_count, double gap_tol,
                                              int32_t* out_tok, int32_t* out_frame, double* out_score,
                                              int32_t out_cap, double* report) {
  if (prune_k < 1) return -1;
  return decode_chunk_impl(static_cast<Stream*>(sp), one_lm(lmp, lambda), static_cast<const PhraseSet*>(boostp),
                           V, H, E, W, enc, T, beta, max_sym, follow_tok, follow_frame, follow_score, follow_count,
                           gap_tol, out_tok, out_frame, out_score, out_cap, report, prune_k, am_tol);
}

// The stateful form: joint input from the prediction network and the
// joint projections (enc rows have Henc entries); see PredNet.
ORACLE_API int32_t oracle_decode_chunk_pred(void* sp, const void* lmp, const void* boostp, int32_t V, int32_t H,
                                            int32_t Henc, int32_t D, const uint16_t* Ep, const uint16_t* Wg,
                                            const float* bg, const uint16_t* Wp, const float* bp,
                                            const uint16_t* We, const float* be, const uint16_t* W,
                                            const uint16_t* enc, int32_t T, double lambda, double beta,
                                            int32_t max_sym, const int32_t* follow_tok, const int32_t* follow_frame,
                                            const float* follow_score, int32_t follow_count, double gap_tol,
                                            int32_t* out_tok, int32_t* out_frame, double* out_score,
                                            int32_t out_cap, double* report) {
  PredNet pn{V, D, Henc, H, Ep, Wg, bg, Wp, bp, We, be};
  return decode_chunk_impl(static_cast<Stream*>(sp), one_lm(lmp, lambda), static_cast<const PhraseSet*>(boostp),
                           V, H, nullptr, W, enc, T, beta, max_sym, follow_tok, follow_frame, follow_score,
                           follow_count, gap_tol, out_tok, out_frame, out_score, out_cap, report, 0, 0.0, &pn);
}

// A stream's prediction-network state: h (bf16 bits) and c, D entries each;
// returns 0 before the first step.
ORACLE_API int32_t oracle_pred_state(const void* sp, uint16_t* h, double* c) {
  const Stream* s = static_cast<const Stream*>(sp);
  if (!s->pred.ready) return 0;
  for (size_t u = 0; u < s->pred.h.size(); ++u) {
    h[u] = s->pred.h[u];
    c[u] = s->pred.c[u];
  }
  return 1;
}

// The same with several LMs (Eq. 1, term 2 summed over i): n_lm LMs with
// weights alpha_i = lambda * weight[i].
ORACLE_API int32_t oracle_decode_chunk_lms(void* sp, int32_t n_lm, const void* const* lms, const double* weight,
                                           const void* boostp, int32_t V, int32_t H, const uint16_t* E,
                                           const uint16_t* W, const uint16_t* enc, int32_t T, double lambda,
                                           double beta, int32_t max_sym, const int32_t* follow_tok,
                                           const int32_t* follow_frame, const float* follow_score,
                                           int32_t follow_count, double gap_tol, int32_t* out_tok,
                                           int32_t* out_frame, double* out_score, int32_t out_cap,
                                           double* report) {
  LmTerm t;
  if (n_lm < 0 || n_lm > LmTerm::kMax) return -1;
  t.n = n_lm;
  for (int i = 0; i < n_lm; ++i) {
    if (!lms[i]) return -1;
    t.lm[i] = static_cast<const NGramDict*>(lms[i]);
    t.alpha[i] = lambda * weight[i];
  }
  return decode_chunk_impl(static_cast<Stream*>(sp), t, static_cast<const PhraseSet*>(boostp), V, H, E, W, enc, T,
                           beta, max_sym, follow_tok, follow_frame, follow_score, follow_count, gap_tol, out_tok,
                           out_frame, out_score, out_cap, report);
}

// Beam search, one frame-synchronous expansion (beam workload; several
// labels per frame).  A frame starts with the beam as its set A of
// hypotheses still in the frame and an empty set F of hypotheses that have
// left it.  One expansion takes, over every hypothesis of A and every
// output, the top K candidates by (score desc, hypothesis index in A asc,
// label asc); in that order a candidate goes to F if it is the blank (labels
// kept) or a label at the frame's S-th expansion (the frame then advances
// without another evaluation, as in greedy decoding), else to the next A;
// in either set equal label sequences merge by log-sum-exp in order of first
// appearance.  F then keeps its K best (score desc, earlier first), in
// insertion order.  The frame ends when A is empty or after S expansions,
// and F is the next frame's beam.  With S = 1 every kept candidate lands in
// F: the top K of the K (V+1) extensions, merged -- one label per frame.
namespace {
struct Kept {
  int32_t hyp, tok;
  double score;
};

void merge_into(std::vector<Hyp>& set, Hyp&& h) {
  for (Hyp& o : set) {
    if (o.y == h.y) {
      o.score = logaddexp(o.score, h.score);
      return;
    }
  }
  set.push_back(std::move(h));
}

void beam_expand(const PhraseSet* boost, int32_t V, int32_t S, int32_t K, int32_t e, std::vector<Hyp>& A,
                 std::vector<Hyp>& F, const std::vector<Kept>& kept) {
  std::vector<Hyp> A2;
  for (const Kept& c : kept) {
    Hyp h = A[(size_t)c.hyp];
    if (c.tok != V) {
      h.y.push_back(c.tok);
      advance_rho(boost, h);
    }
    h.score = c.score;
    merge_into((c.tok == V || e == S - 1) ? F : A2, std::move(h));
  }
  if ((int32_t)F.size() > K) {
    std::vector<size_t> order(F.size());
    for (size_t i = 0; i < order.size(); ++i) order[i] = i;
    std::stable_sort(order.begin(), order.end(), [&](size_t x, size_t y) { return F[x].score > F[y].score; });
    std::vector<char> keep(F.size(), 0);
    for (int32_t r = 0; r < K; ++r) keep[order[(size_t)r]] = 1;
    std::vector<Hyp> F2;
    for (size_t i = 0; i < F.size(); ++i)
      if (keep[i]) F2.push_back(std::move(F[i]));
    F = std::move(F2);
  }
  A = std::move(A2);
}
}  // namespace

// Beam search over one chunk with at most S labels per frame (see above).
// Returns the number of live hypotheses after the chunk.
ORACLE_API int32_t oracle_beam_chunk(void* sp, const void* lmp, const void* boostp, int32_t V,
                                     int32_t H, const uint16_t* E, const uint16_t* W,
                                     const uint16_t* enc, int32_t T, double lambda, double beta,
                                     int32_t K, int32_t S) {
  Stream* s = static_cast<Stream*>(sp);
  const NGramDict* lm = static_cast<const NGramDict*>(lmp);
  const PhraseSet* boost = static_cast<const PhraseSet*>(boostp);
  Model m{V, H, E, W};
  if (s->beam.empty()) s->beam.push_back(Hyp());
  std::vector<float> x;
  std::vector<double> logits, fused;
  for (int32_t t = 0; t < T; ++t) {
    std::vector<Hyp> A = std::move(s->beam), F;
    for (int32_t e = 0; e < S && !A.empty(); ++e) {
      std::vector<Kept> cands;
      for (int32_t i = 0; i < (int32_t)A.size(); ++i) {
        fused_scores(m, enc + (size_t)t * H, A[(size_t)i], one_lm(lm, lambda), boost, beta, x, logits, fused);
        for (int32_t v = 0; v <= V; ++v) cands.push_back({i, v, A[(size_t)i].score + fused[(size_t)v]});
      }
      std::sort(cands.begin(), cands.end(), [](const Kept& a, const Kept& b) {
        if (a.score != b.score) return a.score > b.score;
        if (a.hyp != b.hyp) return a.hyp < b.hyp;
        return a.tok < b.tok;
      });
      if ((int32_t)cands.size() > K) cands.resize((size_t)K);
      beam_expand(boost, V, S, K, e, A, F, cands);
    }
    s->beam = std::move(F);
  }
  return (int32_t)s->beam.size();
}

// Beam hypothesis i: copies up to cap labels to buf, writes its score and
// restart index, returns the label count (-1 if i is out of range).
ORACLE_API int64_t oracle_beam_hyp(const void* sp, int32_t i, int32_t* buf, int64_t cap,
                                   double* score, int64_t* rho) {
  const Stream* s = static_cast<const Stream*>(sp);
  if (i < 0 || i >= (int32_t)s->beam.size()) return -1;
  const Hyp& h = s->beam[(size_t)i];
  for (int64_t j = 0; j < (int64_t)h.y.size() && j < cap; ++j) buf[j] = h.y[(size_t)j];
  if (score) *score = h.score;
  if (rho) *rho = h.rho;
  return (int64_t)h.y.size();
}

// Beam search over one chunk following the selections under test.  Step s
// (an expansion; a stream's frames may take different numbers of them) kept
// sel_hyp/sel_tok/sel_inc[s*K + i] (i < K), in their order (hypothesis -1
// = none; hypothesis = index in the frame's set A): the hypothesis, the
// label (V = blank) and the score increment that was used.  After the last
// frame every remaining step must be empty.  The oracle scores every
// candidate itself and checks that
//   * each kept candidate's increment is its own fused value (largest
//     difference reported),
//   * no candidate left out beats a kept one by more than gap_tol, and the
//     kept ones are in non-increasing order up to gap_tol,
// then applies the expansion with its own scores (merges by log-sum-exp).
ORACLE_API int32_t oracle_beam_chunk_follow(void* sp, const void* lmp, const void* boostp, int32_t V,
                                            int32_t H, const uint16_t* E, const uint16_t* W,
                                            const uint16_t* enc, int32_t T, double lambda, double beta,
                                            int32_t K, const int32_t* sel_hyp, const int32_t* sel_tok,
                                            const float* sel_inc, double gap_tol, double* report, int32_t S,
                                            int32_t n_steps) {
  Stream* s = static_cast<Stream*>(sp);
  const NGramDict* lm = static_cast<const NGramDict*>(lmp);
  const PhraseSet* boost = static_cast<const PhraseSet*>(boostp);
  Model m{V, H, E, W};
  if (s->beam.empty()) s->beam.push_back(Hyp());
  double rep[REP_N] = {0, 0, 0, 0, std::numeric_limits<double>::infinity(), -1, 0, 0};
  std::vector<float> x;
  std::vector<double> logits, fused;
  int32_t step = 0;
  for (int32_t t = 0; t < T; ++t) {
    std::vector<Hyp> A = std::move(s->beam), F;
    for (int32_t e = 0; e < S && !A.empty(); ++e, ++step) {
      if (step >= n_steps) { rep[REP_INCONSISTENT] = 1; break; }
      const size_t nh = A.size();
      std::vector<std::vector<double>> f(nh);
      for (size_t i = 0; i < nh; ++i) {
        fused_scores(m, enc + (size_t)t * H, A[i], one_lm(lm, lambda), boost, beta, x, logits, fused);
        f[i] = fused;
      }
      std::vector<Kept> kept;
      std::vector<char> is_kept(nh * (size_t)(V + 1), 0);
      double min_kept = std::numeric_limits<double>::infinity(), prev = std::numeric_limits<double>::infinity();
      for (int32_t i = 0; i < K; ++i) {
        const int32_t h = sel_hyp[(size_t)step * K + i], v = sel_tok[(size_t)step * K + i];
        if (h < 0) continue;
        if (h >= (int32_t)nh || v < 0 || v > V) { rep[REP_INCONSISTENT] = 1; continue; }
        const double sc = A[(size_t)h].score + f[(size_t)h][(size_t)v];
        rep[REP_MAX_SCORE_DIFF] = std::max(rep[REP_MAX_SCORE_DIFF],
                                           std::fabs((double)sel_inc[(size_t)step * K + i] - f[(size_t)h][(size_t)v]));
        if (sc > prev + gap_tol) rep[REP_MISMATCH] += 1;  // out of order
        prev = sc;
        min_kept = std::min(min_kept, sc);
        is_kept[(size_t)h * (V + 1) + (size_t)v] = 1;
        kept.push_back({h, v, sc});
      }
      const size_t want = std::min((size_t)K, nh * (size_t)(V + 1));
      if (kept.size() != want) rep[REP_INCONSISTENT] = 1;
      double best_out = -std::numeric_limits<double>::infinity();
      for (size_t h = 0; h < nh; ++h)
        for (int32_t v = 0; v <= V; ++v)
          if (!is_kept[h * (V + 1) + (size_t)v]) best_out = std::max(best_out, A[h].score + f[h][(size_t)v]);
      if (best_out > min_kept + gap_tol) {
        rep[REP_MISMATCH] += 1;
        if (rep[REP_FIRST_BAD] < 0) rep[REP_FIRST_BAD] = step;
      } else if (best_out > min_kept) {
        rep[REP_NEAR_TIE] += 1;
      }
      rep[REP_MIN_GAP] = std::min(rep[REP_MIN_GAP], min_kept - best_out);
      beam_expand(boost, V, S, K, e, A, F, kept);
      rep[REP_STEPS] += 1;
    }
    s->beam = std::move(F);
  }
  for (; step < n_steps; ++step)
    for (int32_t i = 0; i < K; ++i)
      if (sel_hyp[(size_t)step * K + i] >= 0) rep[REP_INCONSISTENT] = 1;
  if (report)
    for (int i = 0; i < REP_N; ++i) report[i] = rep[i];
  return (int32_t)s->beam.size();
}

// Joint logits of one frame for a given previous label, in double, for the
// GEMM parity check (x = bf16(ReLU(enc + E[last])), logits = W_out^T x).
ORACLE_API void oracle_joint_logits(int32_t V, int32_t H, const uint16_t* E, const uint16_t* W,
                                    const uint16_t* enc_t, int32_t last, double* out) {
  Model m{V, H, E, W};
  Hyp h;
  if (last != V) h.y.push_back(last);
  std::vector<float> x;
  std::vector<double> logits, fused;
  fused_scores(m, enc_t, h, LmTerm(), nullptr, 0.0, x, logits, fused);
  for (int32_t v = 0; v <= V; ++v) out[v] = logits[(size_t)v];
}

// The full fused row (V+1 entries) for the greedy hypothesis of a stream at
// one frame: log-softmax of the joint plus the weighted LM and boost terms.
ORACLE_API void oracle_fused_row(const void* sp, const void* lmp, const void* boostp, int32_t V,
                                 int32_t H, const uint16_t* E, const uint16_t* W,
                                 const uint16_t* enc_t, double lambda, double beta, double* out) {
  const Stream* s = static_cast<const Stream*>(sp);
  Model m{V, H, E, W};
  std::vector<float> x;
  std::vector<double> logits, fused;
  fused_scores(m, enc_t, s->greedy, one_lm(lmp, lambda), static_cast<const PhraseSet*>(boostp), beta, x, logits,
               fused);
  for (int32_t v = 0; v <= V; ++v) out[v] = fused[(size_t)v];
}

// Emits the labels y[0..len) one by one from an empty history and records,
// for each, the boost bonus it earned (before the weight beta) and the
// restart index rho after it.
ORACLE_API void oracle_boost_trajectory(const void* boostp, const int32_t* y, int64_t len,
                                        double* bonus, int64_t* rho) {
  const PhraseSet* b = static_cast<const PhraseSet*>(boostp);
  Hyp h;
  for (int64_t i = 0; i < len; ++i) {
    bonus[i] = b->score(h.y.data() + h.rho, (int64_t)h.y.size() - h.rho, y[i]);
    h.y.push_back(y[i]);
    advance_rho(b, h);
    rho[i] = h.rho;
  }
}
