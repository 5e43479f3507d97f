/*
 * Seeded synthetic inputs for the fused Transducer decode step.
 *
 * This module only draws data: Gaussian bf16 tensors (encoder frames,
 * predictor embedding table, joint output weights), a normalized backoff
 * n-gram model in ARPA-like arrays, and a phrase list for boosting.  It holds
 * none of the decode step's arithmetic (no joint product, no softmax, no
 * backoff walk, no phrase matching) and is used identically by the CPU oracle
 * and the CUDA path, which both receive its arrays as plain inputs.
 *
 * Random numbers come from Philox4x32-10 (Salmon, Moraes, Dror and Shaw,
 * "Parallel random numbers: as easy as 1, 2, 3", SC'11), a counter-based
 * generator: every value is addressed by (seed, tensor, stream, index), so any
 * subset of streams sees exactly the data it sees inside a larger batch, and
 * the output does not depend on how the work is split.
 *
 * Plain C99, integer-exact RNG; floating point only in Box-Muller and the LM
 * probabilities.  Builds the same on x86_64 and aarch64.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define SYNTH_API __attribute__((visibility("default")))

/* ------------------------------------------------------------------------ */
/* Philox4x32-10                                                             */
/* ------------------------------------------------------------------------ */
static void philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4]) {
  uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
  uint32_t k0 = key_in[0], k1 = key_in[1];
  for (int r = 0; r < 10; ++r) {
    uint64_t p0 = (uint64_t)0xD2511F53u * c0;
    uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t n0 = hi1 ^ c1 ^ k0, n1 = lo1, n2 = hi0 ^ c3 ^ k1, n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

SYNTH_API void synth_philox(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  philox4x32_10(ctr, key, out);
}

/* A stream of draws addressed by (seed, a, b, c); draw i uses counter
 * {i, a, b, c} and returns four 32-bit words. */
typedef struct {
  uint32_t key[2];
  uint32_t a, b, c;
} rng_t;

static rng_t rng_make(uint64_t seed, uint32_t a, uint32_t b, uint32_t c) {
  rng_t r;
  r.key[0] = (uint32_t)seed;
  r.key[1] = (uint32_t)(seed >> 32);
  r.a = a; r.b = b; r.c = c;
  return r;
}

static void rng_draw(const rng_t* r, uint32_t i, uint32_t out[4]) {
  uint32_t ctr[4] = {i, r->a, r->b, r->c};
  philox4x32_10(ctr, r->key, out);
}

/* uniform in the open interval (0, 1) */
static double u01(uint32_t w) { return ((double)w + 0.5) * (1.0 / 4294967296.0); }

static uint16_t f32_to_bf16_rne(float f) {
  uint32_t x;
  memcpy(&x, &f, 4);
  uint32_t lsb = (x >> 16) & 1u;
  x += 0x7FFFu + lsb;
  return (uint16_t)(x >> 16);
}

/* ------------------------------------------------------------------------ */
/* Gaussian bf16 tensors                                                     */
/* ------------------------------------------------------------------------ */
/* out[i] = bf16_RNE((float)(std * z_i)), z_i ~ N(0,1) by Box-Muller, for
 * i in [first, first + n) of the stream (seed, tensor_id, stream_id). */
SYNTH_API void synth_normal_bf16(uint64_t seed, uint32_t tensor_id, uint32_t stream_id,
                                 uint64_t first, uint64_t n, double std, uint16_t* out) {
  rng_t r = rng_make(seed, tensor_id, stream_id, 0x6E6F726Du /* "norm" */);
  const double two_pi = 6.283185307179586476925286766559;
  uint64_t i = first, end = first + n;
  while (i < end) {
    uint64_t block = i >> 2;
    uint32_t w[4];
    /* counter word 0 carries the low 32 bits of the block index, word 3 the
     * high bits folded into the constant lane */
    uint32_t ctr[4] = {(uint32_t)block, r.a, r.b, r.c ^ (uint32_t)(block >> 32)};
    philox4x32_10(ctr, r.key, w);
    double z[4];
    for (int p = 0; p < 2; ++p) {
      double ua = u01(w[2 * p]), ub = u01(w[2 * p + 1]);
      double rad = sqrt(-2.0 * log(ua));
      z[2 * p] = rad * cos(two_pi * ub);
      z[2 * p + 1] = rad * sin(two_pi * ub);
    }
    for (uint32_t lane = (uint32_t)(i & 3); lane < 4 && i < end; ++lane, ++i)
      out[i - first] = f32_to_bf16_rne((float)(std * z[lane]));
  }
}

/* ------------------------------------------------------------------------ */
/* Phrase list                                                               */
/* ------------------------------------------------------------------------ */
/* A small trie used only to reject duplicates and prefix relations while
 * drawing phrases. */
typedef struct {
  int32_t* tok;   /* token on the edge into the node */
  int32_t* first; /* first child */
  int32_t* next;  /* next sibling */
  uint8_t* term;  /* node ends a phrase */
  int32_t n, cap;
} ptrie_t;

static int ptrie_grow(ptrie_t* t) {
  int32_t cap = t->cap ? t->cap * 2 : 1024;
  int32_t* a = realloc(t->tok, sizeof(int32_t) * cap);
  if (!a) return -1;
  t->tok = a;
  a = realloc(t->first, sizeof(int32_t) * cap);
  if (!a) return -1;
  t->first = a;
  a = realloc(t->next, sizeof(int32_t) * cap);
  if (!a) return -1;
  t->next = a;
  uint8_t* b = realloc(t->term, cap);
  if (!b) return -1;
  t->term = b;
  t->cap = cap;
  return 0;
}

static int32_t ptrie_child(const ptrie_t* t, int32_t node, int32_t tok) {
  for (int32_t c = t->first[node]; c >= 0; c = t->next[c])
    if (t->tok[c] == tok) return c;
  return -1;
}

/* 1 if inserted; 0 if the phrase duplicates, extends or is extended by an
 * existing one; -1 on allocation failure. */
static int ptrie_try_insert(ptrie_t* t, const int32_t* p, int32_t len) {
  int32_t node = 0, i = 0;
  for (; i < len; ++i) {
    int32_t c = ptrie_child(t, node, p[i]);
    if (c < 0) break;
    node = c;
    if (t->term[node]) return 0; /* an existing phrase is a prefix */
  }
  if (i == len) return 0; /* duplicate or prefix of an existing phrase */
  for (; i < len; ++i) {
    if (t->n == t->cap && ptrie_grow(t)) return -1;
    int32_t c = t->n++;
    t->tok[c] = p[i];
    t->first[c] = -1;
    t->next[c] = t->first[node];
    t->term[c] = 0;
    t->first[node] = c;
    node = c;
  }
  t->term[node] = 1;
  return 1;
}

/* Draws n_phr phrases with lengths uniform in [len_min, len_max] and tokens
 * uniform over [0, V).  With probability share_frac a phrase starts with a
 * prefix (1 .. len-1 tokens) of an earlier phrase.  No phrase duplicates
 * another or is a prefix of another.  offsets has n_phr+1 entries; tokens has
 * room for n_phr*len_max.  Returns the number of phrases drawn (n_phr unless
 * the space is exhausted) or -1 on allocation failure. */
SYNTH_API int32_t synth_phrases(uint64_t seed, int32_t V, int32_t n_phr, int32_t len_min,
                                int32_t len_max, double share_frac, int32_t* offsets,
                                int32_t* tokens) {
  ptrie_t t = {0};
  if (ptrie_grow(&t)) return -1;
  t.n = 1;
  t.first[0] = -1; t.next[0] = -1; t.term[0] = 0; t.tok[0] = -1;
  rng_t r = rng_make(seed, 0x70687273u /* "phrs" */, 0, 0);
  int32_t* cand = malloc(sizeof(int32_t) * (size_t)(len_max > 0 ? len_max : 1));
  if (!cand) return -1;
  int32_t done = 0;
  offsets[0] = 0;
  uint32_t draw = 0;
  const uint32_t max_draws = (uint32_t)n_phr * 64u + 1024u;
  while (done < n_phr && draw < max_draws) {
    uint32_t w[4];
    rng_draw(&r, draw++, w);
    int32_t len = len_min + (int32_t)(w[0] % (uint32_t)(len_max - len_min + 1));
    int32_t start = 0;
    if (done > 0 && u01(w[1]) < share_frac && len > 1) {
      int32_t j = (int32_t)(w[2] % (uint32_t)done);
      int32_t plen = offsets[j + 1] - offsets[j];
      int32_t maxp = plen - 1 < len - 1 ? plen - 1 : len - 1;
      if (maxp >= 1) {
        start = 1 + (int32_t)(w[3] % (uint32_t)maxp);
        memcpy(cand, tokens + offsets[j], sizeof(int32_t) * start);
      }
    }
    for (int32_t i = start; i < len; i += 4) {
      uint32_t v[4];
      rng_draw(&r, draw++, v);
      for (int q = 0; q < 4 && i + q < len; ++q) cand[i + q] = (int32_t)(v[q] % (uint32_t)V);
    }
    int rc = ptrie_try_insert(&t, cand, len);
    if (rc < 0) { done = -1; break; }
    if (rc == 1) {
      memcpy(tokens + offsets[done], cand, sizeof(int32_t) * len);
      offsets[done + 1] = offsets[done] + len;
      ++done;
    }
  }
  free(cand);
  free(t.tok); free(t.first); free(t.next); free(t.term);
  return done;
}

/* ------------------------------------------------------------------------ */
/* Normalized backoff n-gram model                                           */
/* ------------------------------------------------------------------------ */
/*
 * Construction (absolute discounting with backoff, normalized by design):
 *  - unigram p(v) proportional to (v+1)^(-s) over all V tokens;
 *  - the budget of n-grams above order 1 is split equally over orders 2..N
 *    and water-filled upward under caps n_2 <= V^2/4 and n_k <= 8 n_{k-1};
 *  - each order-(k-1) n-gram g is a context with
 *    n(g) = min(cap(g), round(c * pi(g))) continuations, pi(g) being g's own
 *    sequence probability and c bisected to meet the order's budget;
 *    continuations are drawn without replacement from the continuations of
 *    g's suffix g[1:] (all tokens at order 2), weighted by their probability,
 *    which makes the model prefix- and suffix-closed;
 *  - counts are c(g,w) = 1 + Geometric(1/2); stored probability
 *    (c - D) / sum c, and the backoff weight of g spreads the discounted mass
 *    D n(g) / sum c over the tokens g does not continue, in proportion to
 *    their probability under g[1:].  Because of suffix closure the lower-order
 *    probability of every continuation is an explicit entry of the table, so
 *    the weight needs no backoff walk.
 * Per-order output: tokens (row-major, k per n-gram, lexicographic order),
 * natural-log probabilities, natural-log backoff weights (0 where the n-gram
 * continues nothing, and for the top order) and the raw counts.
 */

typedef struct {
  int64_t n;
  int32_t* tok;     /* last token */
  int64_t* ctx;     /* index of the context at order k-1 (unused at k=1) */
  int64_t* sfx;     /* index of the suffix n-gram at order k-1 (unused at k=1) */
  double* p;        /* conditional probability (as stored: exp of the fp32 log) */
  float* logp;
  float* bow;
  int32_t* count;
  double* pi;       /* sequence probability */
  double* cum;      /* prefix sum of p within the context's children */
  double* Z;        /* total mass the stored model gives this context */
  int64_t* ch_begin; /* children at order k+1 */
  int64_t* ch_count;
} order_t;

typedef struct {
  int32_t V, N;
  order_t* ord; /* ord[0] = order 1 */
  int32_t** tuples;
} synth_lm_t;

static void order_free(order_t* o) {
  free(o->tok); free(o->ctx); free(o->sfx); free(o->p); free(o->logp); free(o->bow);
  free(o->count); free(o->pi); free(o->cum); free(o->Z); free(o->ch_begin); free(o->ch_count);
  memset(o, 0, sizeof(*o));
}

SYNTH_API void synth_lm_free(synth_lm_t* m) {
  if (!m) return;
  if (m->ord)
    for (int k = 0; k < m->N; ++k) order_free(&m->ord[k]);
  if (m->tuples)
    for (int k = 0; k < m->N; ++k) free(m->tuples[k]);
  free(m->ord);
  free(m->tuples);
  free(m);
}

static int order_alloc(order_t* o, int64_t n) {
  o->n = n;
  size_t nn = (size_t)(n > 0 ? n : 1);
  o->tok = malloc(sizeof(int32_t) * nn);
  o->ctx = malloc(sizeof(int64_t) * nn);
  o->sfx = malloc(sizeof(int64_t) * nn);
  o->p = malloc(sizeof(double) * nn);
  o->logp = malloc(sizeof(float) * nn);
  o->bow = calloc(nn, sizeof(float));
  o->count = malloc(sizeof(int32_t) * nn);
  o->pi = malloc(sizeof(double) * nn);
  o->cum = malloc(sizeof(double) * nn);
  o->Z = malloc(sizeof(double) * nn);
  o->ch_begin = calloc(nn, sizeof(int64_t));
  o->ch_count = calloc(nn, sizeof(int64_t));
  return (o->tok && o->ctx && o->sfx && o->p && o->logp && o->bow && o->count && o->pi &&
          o->cum && o->Z && o->ch_begin && o->ch_count)
             ? 0
             : -1;
}

#include <pthread.h>
#include <unistd.h>

typedef void (*range_fn)(void* arg, int64_t b, int64_t e);
typedef struct {
  range_fn fn;
  void* arg;
  int64_t b, e;
} range_task_t;

static void* range_thread(void* p) {
  range_task_t* t = (range_task_t*)p;
  t->fn(t->arg, t->b, t->e);
  return NULL;
}

/* fn over [0, n) split across the online cores (at most 32 threads). */
static void run_parallel(int64_t n, range_fn fn, void* arg) {
  long nt = sysconf(_SC_NPROCESSORS_ONLN);
  if (nt < 1) nt = 1;
  if (nt > 32) nt = 32;
  if (n < 4096 || nt == 1) {
    fn(arg, 0, n);
    return;
  }
  pthread_t th[32];
  range_task_t tk[32];
  int64_t chunk = (n + nt - 1) / nt;
  int started = 0;
  for (long t = 0; t < nt; ++t) {
    int64_t b = t * chunk, e = b + chunk < n ? b + chunk : n;
    if (b >= e) break;
    tk[t].fn = fn; tk[t].arg = arg; tk[t].b = b; tk[t].e = e;
    if (pthread_create(&th[t], NULL, range_thread, &tk[t]) != 0) {
      fn(arg, b, e);
      tk[t].fn = NULL;
    }
    started = (int)t + 1;
  }
  for (int t = 0; t < started; ++t)
    if (tk[t].fn) pthread_join(th[t], NULL);
}

/* candidate range of context i at order k (k>=2): the continuations of its
 * suffix g[1:], which live in the order-(k-1) list (all V unigrams at k=2) */
static void cand_range(const synth_lm_t* m, int k, int64_t i, int64_t* b, int64_t* e) {
  if (k == 2) {
    *b = 0;
    *e = m->V;
  } else {
    const order_t* prev = &m->ord[k - 2]; /* order k-1, the contexts */
    const order_t* pp = &m->ord[k - 3];   /* order k-2, holds their suffixes' child ranges */
    int64_t s = prev->sfx[i];
    *b = pp->ch_begin[s];
    *e = pp->ch_begin[s] + pp->ch_count[s];
  }
}

static int64_t n_for(double c, double pi, int64_t cap) {
  double x = floor(c * pi + 0.5);
  if (x <= 0) return 0;
  if (x >= (double)cap) return cap;
  return (int64_t)x;
}

static int cmp_i64(const void* a, const void* b) {
  int64_t x = *(const int64_t*)a, y = *(const int64_t*)b;
  return (x > y) - (x < y);
}

typedef struct {
  double key;
  int64_t idx;
} es_t;

static int cmp_es_desc(const void* a, const void* b) {
  double x = ((const es_t*)a)->key, y = ((const es_t*)b)->key;
  if (x > y) return -1;
  if (x < y) return 1;
  int64_t i = ((const es_t*)a)->idx, j = ((const es_t*)b)->idx;
  return (i > j) - (i < j);
}

static int64_t total_for(double c, const double* pi, const int64_t* cap, int64_t nctx) {
  int64_t s = 0;
  for (int64_t i = 0; i < nctx; ++i) s += n_for(c, pi[i], cap[i]);
  return s;
}

typedef struct {
  double c;
  const double* pi;
  const int64_t* cap;
  int64_t part[64];
  int64_t chunk;
} total_job_t;

static void total_range(void* arg, int64_t b, int64_t e) {
  total_job_t* J = (total_job_t*)arg;
  J->part[b / J->chunk] = total_for(J->c, J->pi + b, J->cap + b, e - b);
}

static int64_t total_par(double c, const double* pi, const int64_t* cap, int64_t nctx) {
  if (nctx < 4096) return total_for(c, pi, cap, nctx);
  long nt = sysconf(_SC_NPROCESSORS_ONLN);
  if (nt < 1) nt = 1;
  if (nt > 32) nt = 32;
  total_job_t J;
  memset(&J, 0, sizeof(J));
  J.c = c; J.pi = pi; J.cap = cap;
  J.chunk = (nctx + nt - 1) / nt;
  run_parallel(nctx, total_range, &J);
  int64_t s = 0;
  for (int t = 0; t < 64; ++t) s += J.part[t];
  return s;
}

/* Efraimidis-Spirakis weighted sampling without replacement: keys
 * ln(u)/w, keep the n largest.  Writes the chosen indices to out. */
static void draw_es(const rng_t* r, uint32_t draw0, const double* p, int64_t b, int64_t e, int64_t n,
                    es_t* es, int64_t* out) {
  int64_t range = e - b;
  uint32_t w4[4];
  for (int64_t j = 0; j < range; ++j) {
    if ((j & 3) == 0) rng_draw(r, draw0 + (uint32_t)(j >> 2), w4);
    es[j].key = log(u01(w4[j & 3])) / p[b + j];
    es[j].idx = b + j;
  }
  qsort(es, (size_t)range, sizeof(es_t), cmp_es_desc);
  for (int64_t j = 0; j < n; ++j) out[j] = es[j].idx;
}

typedef struct {
  synth_lm_t* m;
  int k;
} tuple_job_t;

static void tuple_range(void* arg, int64_t x0, int64_t x1) {
  tuple_job_t* J = (tuple_job_t*)arg;
  const int k = J->k;
  const order_t* o = &J->m->ord[k - 1];
  for (int64_t x = x0; x < x1; ++x) {
    int32_t* dst = J->m->tuples[k - 1] + (size_t)x * k;
    if (k > 1) memcpy(dst, J->m->tuples[k - 2] + (size_t)o->ctx[x] * (k - 1), sizeof(int32_t) * (k - 1));
    dst[k - 1] = o->tok[x];
  }
}

typedef struct {
  synth_lm_t* m;
  int k;
  uint64_t seed;
  double discount, c;
  const int64_t* caps;
  const int64_t* start;
  double z_root;
  int failed;
} gen_job_t;

/* Draws the continuations of contexts [i0, i1) of order k-1. */
static void gen_contexts(void* arg, int64_t i0, int64_t i1) {
  gen_job_t* J = (gen_job_t*)arg;
  synth_lm_t* m = J->m;
  const int k = J->k;
  const double discount = J->discount, c = J->c, z_root = J->z_root;
  const uint64_t seed = J->seed;
  const int32_t V = m->V;
  order_t* ctxo = &m->ord[k - 2];
  const order_t* lower = &m->ord[k - 2];
  order_t* o = &m->ord[k - 1];
  const int64_t* caps = J->caps;
  int64_t* chosen = NULL;
  es_t* es = NULL;
  size_t chosen_cap = 0;
  (void)V;
  for (int64_t i = i0; i < i1; ++i) {
    const int64_t pos = J->start[i];
        int64_t b, e;
        cand_range(m, k, i, &b, &e);
        int64_t n = n_for(c, ctxo->pi[i], caps[i]);
        ctxo->ch_begin[i] = pos;
        ctxo->ch_count[i] = n;
        /* total stored mass of the suffix context g[1:] */
        double z_sfx = (k == 2) ? z_root : m->ord[k - 3].Z[ctxo->sfx[i]];
        if (n == 0) {
          ctxo->Z[i] = z_sfx; /* no continuations, no backoff weight */
          continue;
        }
        int64_t range = e - b;
        if ((size_t)range > chosen_cap) {
          chosen_cap = (size_t)range;
          free(chosen); free(es);
          chosen = malloc(sizeof(int64_t) * chosen_cap);
          es = malloc(sizeof(es_t) * chosen_cap);
          if (!chosen || !es) { J->failed = 1; free(chosen); free(es); return; }
        }
        rng_t r = rng_make(seed, 0x6C6D0000u | (uint32_t)k, (uint32_t)i, (uint32_t)((uint64_t)i >> 32));
        if (n == range) {
          for (int64_t j = 0; j < range; ++j) chosen[j] = b + j;
        } else if (n * 8 >= range) {
          draw_es(&r, 0, lower->p, b, e, n, es, chosen);
        } else {
          /* successive sampling by inverse CDF over the candidates' running
           * sum (which restarts at b), rejecting repeats */
          const double* cum = lower->cum;
          double tot = cum[e - 1];
          uint32_t d = 0x10000u;
          uint32_t tries = 0;
          int64_t got = 0;
          while (got < n && tries < (uint32_t)(n * 64 + 64)) {
            uint32_t w4[4];
            rng_draw(&r, d++, w4);
            for (int q = 0; q < 4 && got < n; ++q) {
              ++tries;
              double tgt = u01(w4[q]) * tot;
              int64_t lo = b, hi = e - 1;
              while (lo < hi) {
                int64_t mid = lo + (hi - lo) / 2;
                if (cum[mid] < tgt) lo = mid + 1; else hi = mid;
              }
              int dup = 0;
              for (int64_t j = 0; j < got; ++j)
                if (chosen[j] == lo) { dup = 1; break; }
              if (!dup) chosen[got++] = lo;
            }
          }
          if (got < n) draw_es(&r, 0x20000u, lower->p, b, e, n, es, chosen);
        }
        qsort(chosen, (size_t)n, sizeof(int64_t), cmp_i64);
        /* counts 1 + Geometric(1/2): trailing ones of a 64-bit word */
        int64_t csum = 0;
        uint32_t w4[4];
        for (int64_t j = 0; j < n; ++j) {
          if ((j & 1) == 0) rng_draw(&r, 0x40000u + (uint32_t)(j >> 1), w4);
          uint64_t bits = ((uint64_t)w4[(j & 1) * 2] << 32) | w4[(j & 1) * 2 + 1];
          int32_t g = 0;
          while ((bits & 1u) && g < 63) { ++g; bits >>= 1; }
          o->count[pos + j] = 1 + g;
          csum += 1 + g;
        }
        double lower_mass = 0, kept = 0;
        for (int64_t j = 0; j < n; ++j) {
          int64_t cidx = chosen[j];
          int64_t x = pos + j;
          o->tok[x] = lower->tok[cidx];
          o->ctx[x] = i;
          o->sfx[x] = cidx; /* the suffix g[1:]·w is the candidate itself */
          double p = ((double)o->count[x] - discount) / (double)csum;
          o->logp[x] = (float)log(p);
          o->p[x] = exp((double)o->logp[x]);
          o->pi[x] = ctxo->pi[i] * o->p[x];
          kept += o->p[x];
          lower_mass += lower->p[cidx];
        }
        /* the backoff weight spreads 1 - kept over the tokens g does not
         * continue, whose stored mass under g[1:] is z_sfx - lower_mass; the
         * context's resulting total is recorded for the next order */
        ctxo->bow[i] = (float)log((1.0 - kept) / (z_sfx - lower_mass));
        ctxo->Z[i] = kept + exp((double)ctxo->bow[i]) * (z_sfx - lower_mass);
        double acc = 0;
        for (int64_t j = 0; j < n; ++j) { acc += o->p[pos + j]; o->cum[pos + j] = acc; }
  }
  free(chosen);
  free(es);
}

SYNTH_API synth_lm_t* synth_lm_new(uint64_t seed, int32_t V, int32_t N, int64_t total,
                                   double zipf_s, double discount) {
  if (V < 2 || N < 1 || N > 16 || discount <= 0 || discount >= 1) return NULL;
  synth_lm_t* m = calloc(1, sizeof(synth_lm_t));
  if (!m) return NULL;
  m->V = V;
  m->N = N;
  m->ord = calloc((size_t)N, sizeof(order_t));
  m->tuples = calloc((size_t)N, sizeof(int32_t*));
  if (!m->ord || !m->tuples) { synth_lm_free(m); return NULL; }

  /* order budgets: equal split over orders 2..N, water-filled upward under
   * n_2 <= V^2/4 and n_k <= 8 n_{k-1} */
  int64_t target[17] = {0};
  {
    int64_t rest = total - V;
    if (rest < 0) rest = 0;
    int64_t fixed = 0;
    int lo_k = 2;
    while (lo_k <= N) {
      int64_t share = (rest - fixed) / (N - lo_k + 1);
      double cap = (lo_k == 2) ? 0.25 * (double)V * (double)V : 8.0 * (double)target[lo_k - 1];
      if ((double)share > cap) {
        target[lo_k] = (int64_t)cap;
        fixed += target[lo_k];
        ++lo_k;
        continue;
      }
      for (int k = lo_k; k <= N; ++k) target[k] = share;
      break;
    }
  }

  /* order 1: Zipf unigrams */
  order_t* o1 = &m->ord[0];
  if (order_alloc(o1, V)) { synth_lm_free(m); return NULL; }
  {
    double z = 0;
    for (int32_t v = 0; v < V; ++v) z += pow((double)v + 1.0, -zipf_s);
    double acc = 0;
    for (int32_t v = 0; v < V; ++v) {
      double p = pow((double)v + 1.0, -zipf_s) / z;
      o1->tok[v] = v;
      o1->ctx[v] = 0;
      o1->sfx[v] = 0;
      o1->logp[v] = (float)log(p);
      o1->p[v] = exp((double)o1->logp[v]);
      o1->pi[v] = o1->p[v];
      o1->count[v] = 0;
      acc += o1->p[v];
      o1->cum[v] = acc;
    }
  }

  /* Z of the empty context: the stored unigram mass */
  double z_root = o1->cum[V - 1];

  int64_t* caps = NULL;

  for (int k = 2; k <= N; ++k) {
    order_t* ctxo = &m->ord[k - 2];      /* contexts: order k-1 */
    int64_t nctx = ctxo->n;
    free(caps);
    caps = malloc(sizeof(int64_t) * (size_t)(nctx > 0 ? nctx : 1));
    if (!caps) { synth_lm_free(m); return NULL; }
    int64_t maxn = 0;
    for (int64_t i = 0; i < nctx; ++i) {
      int64_t b, e;
      cand_range(m, k, i, &b, &e);
      caps[i] = (k == 2) ? V - 1 : e - b;
      maxn += caps[i];
    }
    int64_t want = target[k] < maxn ? target[k] : maxn;
    /* bracket, then bisect the scale c so the order meets its budget (1%) */
    double lo_c = 0, hi_c = 1;
    for (int it = 0; it < 200 && total_par(hi_c, ctxo->pi, caps, nctx) < want; ++it) {
      lo_c = hi_c;
      hi_c *= 2;
    }
    double c = hi_c;
    for (int it = 0; it < 100; ++it) {
      double mid = 0.5 * (lo_c + hi_c);
      int64_t s = total_par(mid, ctxo->pi, caps, nctx);
      c = mid;
      if ((double)llabs(s - want) <= 0.01 * (double)want) break;
      if (s < want) lo_c = mid; else hi_c = mid;
    }
    int64_t nk = total_par(c, ctxo->pi, caps, nctx);
    order_t* o = &m->ord[k - 1];
    if (order_alloc(o, nk)) { free(caps); synth_lm_free(m); return NULL; }
    /* output positions, then every context in parallel (each context's
     * draws come from its own counter-based stream, so the result does not
     * depend on the thread count) */
    int64_t* start = malloc(sizeof(int64_t) * (size_t)(nctx + 1));
    if (!start) { free(caps); synth_lm_free(m); return NULL; }
    start[0] = 0;
    for (int64_t i = 0; i < nctx; ++i) start[i + 1] = start[i] + n_for(c, ctxo->pi[i], caps[i]);
    gen_job_t job = {m, k, seed, discount, c, caps, start, z_root, 0};
    run_parallel(nctx, gen_contexts, &job);
    free(start);
    if (job.failed) { free(caps); synth_lm_free(m); return NULL; }
  }
  free(caps);

  /* materialize the tuples in lexicographic order */
  for (int k = 1; k <= N; ++k) {
    order_t* o = &m->ord[k - 1];
    size_t nn = (size_t)(o->n > 0 ? o->n : 1);
    m->tuples[k - 1] = malloc(sizeof(int32_t) * nn * (size_t)k);
    if (!m->tuples[k - 1]) { synth_lm_free(m); return NULL; }
    tuple_job_t tj = {m, k};
    run_parallel(o->n, tuple_range, &tj);
  }
  return m;
}

SYNTH_API int64_t synth_lm_count(const synth_lm_t* m, int32_t k) {
  return (k >= 1 && k <= m->N) ? m->ord[k - 1].n : -1;
}

/* Copies order k (1-based) out: tokens [n*k], logp [n], bow [n], counts [n].
 * Any output pointer may be NULL. */
SYNTH_API void synth_lm_get(const synth_lm_t* m, int32_t k, int32_t* tokens, float* logp,
                            float* bow, int32_t* counts) {
  const order_t* o = &m->ord[k - 1];
  if (tokens) memcpy(tokens, m->tuples[k - 1], sizeof(int32_t) * (size_t)o->n * k);
  if (logp) memcpy(logp, o->logp, sizeof(float) * (size_t)o->n);
  if (bow) {
    if (k == m->N) memset(bow, 0, sizeof(float) * (size_t)o->n);
    else memcpy(bow, o->bow, sizeof(float) * (size_t)o->n);
  }
  if (counts) memcpy(counts, o->count, sizeof(int32_t) * (size_t)o->n);
}
