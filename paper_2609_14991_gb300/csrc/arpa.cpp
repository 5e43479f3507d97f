// Reader of ARPA back-off n-gram files (host only).
//
// The format: a "\data\" header with one "ngram k=count" line per order,
// then per order k a "\k-grams:" section of lines
//   log10 p <TAB> w1 ... wk [<TAB> log10 backoff]
// and "\end\".  Words map to label ids through a vocabulary (word i -> id i)
// or, without one, are the decimal ids themselves.  N-grams that hold a word
// outside the vocabulary (the sentence markers, <unk>) are dropped: the
// decoder scores no sentence boundaries (a stream has no start or end
// symbol).  log10 values become natural log, the unit of the fusion score
// (Eq. 1 adds LM log-probabilities to the acoustic model's natural-log
// posteriors).
#include <cerrno>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <memory>
#include <string>
#include <unordered_map>
#include <vector>

#include "internal.h"

struct tsd_arpa {
  int32_t V = 0, order = 0;
  int64_t skipped = 0;
  std::vector<int64_t> count;                // per order, kept n-grams
  std::vector<std::vector<int32_t>> tokens;  // per order, [count][k]
  std::vector<std::vector<float>> logp, bow;
};

namespace {

using tsd::fail;

// One line of the text: [b, e) without the line break.
struct Lines {
  const char* p;
  const char* end;
  bool next(const char*& b, const char*& e) {
    if (p >= end) return false;
    b = p;
    const char* q = static_cast<const char*>(std::memchr(p, '\n', (size_t)(end - p)));
    e = q ? q : end;
    p = q ? q + 1 : end;
    if (e > b && e[-1] == '\r') --e;
    return true;
  }
};

bool is_space(char c) { return c == ' ' || c == '\t'; }

// Splits [b, e) at blanks and tabs into at most `cap` fields.
int split(const char* b, const char* e, std::string* f, int cap) {
  int n = 0;
  while (b < e) {
    while (b < e && is_space(*b)) ++b;
    if (b >= e) break;
    const char* s = b;
    while (b < e && !is_space(*b)) ++b;
    if (n < cap) f[n] = std::string(s, (size_t)(b - s));
    ++n;
  }
  return n;
}

std::string trim(const char* b, const char* e) {
  while (b < e && is_space(*b)) ++b;
  while (e > b && is_space(e[-1])) --e;
  return std::string(b, (size_t)(e - b));
}

bool to_double(const std::string& s, double* v) {
  if (s.empty()) return false;
  char* end = nullptr;
  errno = 0;
  *v = std::strtod(s.c_str(), &end);
  return errno == 0 && end == s.c_str() + s.size();
}

}  // namespace

extern "C" tsd_status tsd_arpa_parse(const char* text, int64_t len, int32_t V, const char* const* vocab,
                                     tsd_arpa** out) {
  tsd::clear_error();
  if (!out) return fail(TSD_EINVAL, "tsd_arpa_parse: out is NULL");
  *out = nullptr;
  if (!text || len < 0) return fail(TSD_EINVAL, "tsd_arpa_parse: NULL text");
  if (V < 1 || V > 32767) return fail(TSD_EINVAL, "tsd_arpa_parse: V=%d out of range [1, 32767]", V);
  std::unordered_map<std::string, int32_t> ids;
  if (vocab) {
    ids.reserve((size_t)V * 2);
    for (int32_t i = 0; i < V; ++i) {
      if (!vocab[i]) return fail(TSD_EINVAL, "tsd_arpa_parse: vocabulary entry %d is NULL", i);
      if (!ids.emplace(vocab[i], i).second) return fail(TSD_EINVAL, "tsd_arpa_parse: word '%s' repeats", vocab[i]);
    }
  }
  auto word_id = [&](const std::string& w) -> int32_t {
    if (vocab) {
      auto it = ids.find(w);
      return it == ids.end() ? -1 : it->second;
    }
    if (w.empty() || w.size() > 6) return -1;
    int32_t v = 0;
    for (char c : w) {
      if (c < '0' || c > '9') return -1;
      v = v * 10 + (c - '0');
    }
    return v < V ? v : -1;
  };

  std::unique_ptr<tsd_arpa> a(new tsd_arpa());
  a->V = V;
  Lines L{text, text + len};
  const char *b, *e;
  // header
  bool in_data = false;
  std::vector<int64_t> declared;
  while (L.next(b, e)) {
    const std::string t = trim(b, e);
    if (!in_data) {
      if (t == "\\data\\") in_data = true;
      continue;
    }
    if (t.empty()) {
      if (!declared.empty()) break;
      continue;
    }
    if (t.compare(0, 6, "ngram ") != 0) break;
    const size_t eq = t.find('=');
    if (eq == std::string::npos) return fail(TSD_EINVAL, "tsd_arpa_parse: bad header line '%s'", t.c_str());
    const long k = std::strtol(t.c_str() + 6, nullptr, 10);
    const long long n = std::strtoll(t.c_str() + eq + 1, nullptr, 10);
    if (k != (long)declared.size() + 1 || n < 0)
      return fail(TSD_EINVAL, "tsd_arpa_parse: bad header line '%s'", t.c_str());
    declared.push_back((int64_t)n);
  }
  if (!in_data || declared.empty()) return fail(TSD_EINVAL, "tsd_arpa_parse: no \\data\\ header");
  const int order = (int)declared.size();
  if (order > tsd::kMaxOrder) return fail(TSD_EINVAL, "tsd_arpa_parse: order %d above %d", order, tsd::kMaxOrder);
  a->order = order;
  a->count.assign((size_t)order, 0);
  a->tokens.resize((size_t)order);
  a->logp.resize((size_t)order);
  a->bow.resize((size_t)order);
  std::string f[tsd::kMaxOrder + 3];
  for (int k = 1; k <= order; ++k) {
    const std::string head = "\\" + std::to_string(k) + "-grams:";
    bool found = false;
    while (L.next(b, e))
      if (trim(b, e) == head) {
        found = true;
        break;
      }
    if (!found) return fail(TSD_EINVAL, "tsd_arpa_parse: section %s missing", head.c_str());
    auto& tok = a->tokens[(size_t)k - 1];
    auto& lp = a->logp[(size_t)k - 1];
    auto& bw = a->bow[(size_t)k - 1];
    tok.reserve((size_t)declared[(size_t)k - 1] * k);
    lp.reserve((size_t)declared[(size_t)k - 1]);
    bw.reserve((size_t)declared[(size_t)k - 1]);
    int64_t seen = 0;
    const double ln10 = std::log(10.0);
    while (L.next(b, e)) {
      const char* s = b;
      while (s < e && is_space(*s)) ++s;
      if (s >= e || *s == '\\') break;
      const int nf = split(b, e, f, tsd::kMaxOrder + 3);
      if (nf != k + 1 && nf != k + 2)
        return fail(TSD_EINVAL, "tsd_arpa_parse: order %d line %lld has %d fields", k, (long long)seen + 1, nf);
      double p10 = 0, b10 = 0;
      if (!to_double(f[0], &p10) || (nf == k + 2 && !to_double(f[k + 1], &b10)))
        return fail(TSD_EINVAL, "tsd_arpa_parse: order %d line %lld: bad number", k, (long long)seen + 1);
      ++seen;
      int32_t w[tsd::kMaxOrder];
      bool known = true;
      for (int i = 0; i < k; ++i) {
        w[i] = word_id(f[1 + i]);
        if (w[i] < 0) known = false;
      }
      if (!known) {
        ++a->skipped;
        continue;
      }
      tok.insert(tok.end(), w, w + k);
      lp.push_back((float)(p10 * ln10));
      bw.push_back((float)(b10 * ln10));
    }
    if (seen != declared[(size_t)k - 1])
      return fail(TSD_EINVAL, "tsd_arpa_parse: order %d: header says %lld n-grams, found %lld", k,
                  (long long)declared[(size_t)k - 1], (long long)seen);
    a->count[(size_t)k - 1] = (int64_t)lp.size();
  }
  *out = a.release();
  return TSD_OK;
}

extern "C" tsd_status tsd_arpa_info(const tsd_arpa* a, int32_t* order, int64_t* counts, int32_t cap,
                                    int64_t* skipped) {
  tsd::clear_error();
  if (!a) return fail(TSD_EINVAL, "tsd_arpa_info: NULL handle");
  if (order) *order = a->order;
  if (counts)
    for (int32_t k = 0; k < cap && k < a->order; ++k) counts[k] = a->count[(size_t)k];
  if (skipped) *skipped = a->skipped;
  return TSD_OK;
}

extern "C" tsd_status tsd_arpa_arrays(const tsd_arpa* a, int32_t k, const int32_t** tokens, const float** logp,
                                      const float** bow) {
  tsd::clear_error();
  if (!a) return fail(TSD_EINVAL, "tsd_arpa_arrays: NULL handle");
  if (k < 1 || k > a->order) return fail(TSD_EINVAL, "tsd_arpa_arrays: order %d outside [1, %d]", k, a->order);
  if (tokens) *tokens = a->tokens[(size_t)k - 1].data();
  if (logp) *logp = a->logp[(size_t)k - 1].data();
  if (bow) *bow = a->bow[(size_t)k - 1].data();
  return TSD_OK;
}

extern "C" void tsd_arpa_free(tsd_arpa* a) { delete a; }

extern "C" tsd_status tsd_ngram_build_arpa(const char* text, int64_t len, int32_t V, const char* const* vocab,
                                           tsd_ngram** out) {
  tsd_arpa* a = nullptr;
  tsd_status st = tsd_arpa_parse(text, len, V, vocab, &a);
  if (st) return st;
  std::unique_ptr<tsd_arpa> hold(a);
  const int32_t* tk[tsd::kMaxOrder];
  const float* lp[tsd::kMaxOrder];
  const float* bw[tsd::kMaxOrder];
  for (int k = 0; k < a->order; ++k) {
    tk[k] = a->tokens[(size_t)k].data();
    lp[k] = a->logp[(size_t)k].data();
    bw[k] = a->bow[(size_t)k].data();
  }
  return tsd_ngram_build(V, a->order, a->count.data(), tk, lp, bw, out);
}
