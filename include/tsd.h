/*
 * tsd.h -- fused streaming Transducer decode step with shallow fusion, for
 * one NVIDIA GB300 (sm_103a).
 *
 * The operation (paper Sec. III-C, Eq. 1): at every decoding step each
 * hypothesis's next-label candidates are re-ranked by
 *
 *     score(y) = log p_AM(y | x) + lambda * log p_LM(y) + beta * boost(y)
 *
 * where p_AM is the Transducer's joint output after log-softmax over the V
 * labels and blank, p_LM a backoff n-gram model over the same sub-word
 * labels, and boost(y) the bonus of a phrase-boosting tree built from a user
 * phrase list.  The LM and boost terms apply to the V non-blank labels only;
 * blank (id V) keeps its acoustic score.  The decoder consumes one encoder
 * chunk at a time and carries its state across chunks (Sec. III-B, the
 * cache-aware streaming loop of Fig. 1), emitting labels greedily (Sec. III)
 * or by beam search.
 *
 * The joint network is  logits = W_out^T ReLU(enc_t + E[last]),  with
 * W_out [H][V+1] and E [V+1][H] in bf16, the hidden sum in fp32 rounded once
 * to bf16, and an fp32-accumulated product; E[V] (the blank row) is the
 * start-of-sequence input.
 *
 * Conventions for every call:
 *   - Return TSD_OK (0) or a negative status; tsd_last_error() then gives a
 *     message for the calling thread.  No call throws or aborts.
 *   - NULL handles, NULL required pointers and out-of-range sizes return
 *     TSD_EINVAL before any device work.
 *   - "device" pointers are CUDA global memory of the current device;
 *     "host" pointers are ordinary (pageable or pinned) host memory.
 *   - A decoder has no internal locking: drive each decoder from one host
 *     thread, and issue all of its calls on one CUDA stream (or order them).
 */
#ifndef TSD_H
#define TSD_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define TSD_API __attribute__((visibility("default")))
#else
#define TSD_API
#endif

typedef int32_t tsd_status;

#define TSD_OK 0
#define TSD_EINVAL (-1)  /* bad argument: NULL pointer, size, token or table inconsistency */
#define TSD_ENOMEM (-2)  /* host or device allocation failed */
#define TSD_ECUDA (-3)   /* a CUDA runtime call failed (message has the CUDA error) */
#define TSD_ESTATE (-4)  /* slot closed, unknown or already in use; no free slot */
#define TSD_EDEVICE (-5) /* a device-side range check tripped (see tsd_last_error) */

typedef struct tsd_ngram tsd_ngram;
typedef struct tsd_boost tsd_boost;
typedef struct tsd_decoder tsd_decoder;

/* Message of the last failing call on this thread ("" if none). The pointer
 * stays valid until the next call on this thread. */
TSD_API const char* tsd_last_error(void);

/* Library version string, e.g. "tsd 0.1 sm_103a". */
TSD_API const char* tsd_version(void);

/* ------------------------------------------------------------------------
 * n-gram LM (Eq. 1, second term; Sec. III-C "GPU n-gram language models ...
 * over sub-word tokens").
 *
 * Builds the device tables of an order-`order` backoff model over labels
 * [0, V) from ARPA-like arrays, per order k = 1..order (index k-1):
 *   count[k-1]   number of n-grams of order k;
 *   ngrams[k-1]  host int32 [count][k], the tokens of each n-gram, any order;
 *   logp[k-1]    host float [count], natural-log conditional probability
 *                (an ARPA log10 source must be scaled by ln 10 first);
 *   bow[k-1]     host float [count], natural-log backoff weight, 0 = none
 *                (ignored for the top order; bow itself may be NULL).
 * The score of label v after history h is
 *   log p(v | h) = logp(h v)                 if h v is an n-gram,
 *                = bow(h) + log p(v | h[1:])  otherwise (bow = 0 if h is
 *                  not an n-gram), with only the last order-1 labels of h
 *                  used and log p(v | empty) = logp of the unigram v.
 * Requirements (else TSD_EINVAL): 1 <= order <= 16; every unigram [0, V)
 * present exactly once; fewer than 2^28 n-grams above order 1; tokens in
 * range; no duplicate n-gram; the set is
 * prefix- and suffix-closed (every prefix and every suffix of an n-gram is an
 * n-gram), as in any ARPA model estimated from counts; finite values.
 * The inputs are copied (the caller keeps ownership) and uploaded
 * synchronously to the current device. *out owns the device tables. */
TSD_API tsd_status tsd_ngram_build(int32_t V, int32_t order, const int64_t* count,
                           const int32_t* const* ngrams, const float* const* logp,
                           const float* const* bow, tsd_ngram** out);
TSD_API void tsd_ngram_free(tsd_ngram* lm);

/* Sizes of the built tables: LM states (root + every n-gram below the top
 * order), arcs (every n-gram above order 1), and device bytes held. */
TSD_API tsd_status tsd_ngram_info(const tsd_ngram* lm, int64_t* n_states, int64_t* n_arcs,
                          int64_t* device_bytes);

/* The label tuple an LM state id stands for (host call, no device work).
 * Writes up to cap labels, sets *len to the tuple length (0 for the root). */
TSD_API tsd_status tsd_ngram_state_tuple(const tsd_ngram* lm, int32_t state, int32_t* buf, int32_t cap,
                                 int32_t* len);

/* ------------------------------------------------------------------------
 * ARPA back-off n-gram files (the usual interchange format of n-gram
 * toolkits; the paper's n-gram LMs over sub-word tokens, Sec. III-C, come
 * as such files).  Host only: no device work.
 *
 * text[0, len): the file's contents: a "\data\" header with one
 * "ngram k=count" line per order, then per order k a "\k-grams:" section of
 * lines "log10 p  w1 .. wk  [log10 backoff]" separated by blanks or tabs.
 * vocab: NULL (each word is its decimal label id in [0, V)) or V strings
 * (word vocab[i] is label i; the strings are only read during the call).
 * N-grams holding any other word (<s>, </s>, <unk>) are dropped and counted
 * in *skipped: streams have no sentence start or end.  Values are converted
 * to natural log.  Errors (TSD_EINVAL): no header, a section missing, a line
 * with the wrong number of fields or a malformed number, a section whose
 * line count differs from its header, order above 16, a repeated vocabulary
 * word.  *out is owned by the caller (tsd_arpa_free). */
typedef struct tsd_arpa tsd_arpa;
TSD_API tsd_status tsd_arpa_parse(const char* text, int64_t len, int32_t V, const char* const* vocab,
                                  tsd_arpa** out);
/* The parsed order, the kept n-grams per order (counts[0 .. min(cap,
 * order)) ) and the dropped lines. */
TSD_API tsd_status tsd_arpa_info(const tsd_arpa* a, int32_t* order, int64_t* counts, int32_t cap,
                                 int64_t* skipped);
/* Order k's arrays in file order, valid until tsd_arpa_free: tokens
 * [count][k] int32, logp and bow (natural log; bow 0 where the file has
 * none) [count] float. */
TSD_API tsd_status tsd_arpa_arrays(const tsd_arpa* a, int32_t k, const int32_t** tokens, const float** logp,
                                   const float** bow);
TSD_API void tsd_arpa_free(tsd_arpa* a);
/* tsd_arpa_parse followed by tsd_ngram_build (same requirements: every
 * unigram of [0, V) present, prefix- and suffix-closed after the dropped
 * lines are removed). */
TSD_API tsd_status tsd_ngram_build_arpa(const char* text, int64_t len, int32_t V, const char* const* vocab,
                                        tsd_ngram** out);

/* ------------------------------------------------------------------------
 * Phrase boosting tree (Eq. 1, third term; Sec. III-C "a phrase-boosting
 * tree from a user word list", Fig. 1).
 *
 * Compiles n_phr phrases (host int32: phrase i is tokens[offsets[i] ..
 * offsets[i+1]), 1 <= length <= 32, labels in [0, V)) into an Aho-Corasick
 * trie with failure links.  boost(v) = token_bonus * (d(h v) - d(h)), where
 * d(g) is the length of the longest suffix of g that is a prefix of some
 * phrase, and g runs over the labels emitted since the last completed
 * phrase: when the longest match after an emission is a whole phrase, its
 * bonus is kept and matching restarts empty.  A partial match that fails
 * gives back what it earned.  Duplicate phrases are merged; a phrase that is
 * a prefix of another makes the longer one unreachable.
 * Inputs are copied; tables are uploaded synchronously to the current device. */
TSD_API tsd_status tsd_boost_build(int32_t V, int32_t n_phr, const int32_t* offsets,
                           const int32_t* tokens, float token_bonus, tsd_boost** out);
TSD_API void tsd_boost_free(tsd_boost* b);

/* Trie nodes (root included), the longest phrase, and device bytes held. */
TSD_API tsd_status tsd_boost_info(const tsd_boost* b, int32_t* n_nodes, int32_t* max_depth,
                          int64_t* device_bytes);

/* The label tuple (phrase prefix) a trie node stands for (host call). */
TSD_API tsd_status tsd_boost_node_tuple(const tsd_boost* b, int32_t node, int32_t* buf, int32_t cap,
                                int32_t* len);

/* ------------------------------------------------------------------------
 * Decoder.
 */
typedef struct {
  int32_t V;           /* non-blank labels; blank = V; 1 <= V <= 16384 */
  int32_t H;           /* joint hidden size; multiple of 64, 64 <= H <= 8192 */
  int32_t max_symbols; /* labels per frame, 1..64 (greedy: Sec. III; beam: expansions per frame) */
  int32_t beam_k;      /* 1 = greedy; 2..8 = beam search */
  int32_t max_streams; /* stream slots; max_streams * beam_k <= 4096 */
  int32_t max_T;       /* frames per chunk, 1 <= max_T <= 4096 */
  int32_t prune_k;     /* 0: fusion over every label (Eq. 1 as written).  1..8: pruned
                          fusion: the LM and boost terms re-rank only the acoustic
                          model's prune_k best outputs (blank included, ties to the
                          lower id), the reading of Sec. III-C's remark that fusion
                          only re-ranks the candidates the model proposes.  Needs
                          greedy decoding and at most one LM. */
} tsd_decoder_cfg;

/* Creates a decoder for one joint network and optional LM / phrase tree.
 *   W_out_bf16: device bf16 [H][V+1] (row-major), E_bf16: device bf16
 *   [V+1][H].  Both are copied (W_out repacked label-major, padded) on
 *   cuda_stream and may be freed once the stream reaches this point.
 *   lm, boost: may be NULL (then that term is 0); they must outlive the
 *   decoder and have the same V.
 * Allocates all device work memory up front; no later call allocates. */
TSD_API tsd_status tsd_decoder_create(const tsd_decoder_cfg* cfg, const void* W_out_bf16,
                              const void* E_bf16, const tsd_ngram* lm, const tsd_boost* boost,
                              void* cuda_stream, tsd_decoder** out);

/* The stateful Transducer form: the joint input is
 *   bf16(ReLU(W_enc enc_t + b_enc + W_pred h + b_pred))
 * where h is the output of a one-layer LSTM prediction network over the
 * previous label (Fig. 1: prediction and joint networks): on every emitted
 * label y it reads x = emb[y] (emb[V] starts a sequence) and updates
 *   gates = b_gates + (x, h) W_gates,   c' = s(f) c + s(i) tanh(g),
 *   h' = s(o) tanh(c')   (h kept as bf16, c as fp32).
 * Encoder frames passed to decode_chunk are then H_enc wide.  All weights
 * are device arrays, copied (and repacked) at create. */
typedef struct {
  int32_t D;             /* LSTM width: multiple of 64, 64 <= D <= 2048 */
  int32_t H_enc;         /* encoder frame width: multiple of 64, 64 <= H_enc <= 8192 */
  const void* emb;       /* bf16 [V+1][D] */
  const void* W_gates;   /* bf16 [2D][4D]: rows (x, then h); column 4u+q is gate q (i, f, g, o) of unit u */
  const float* b_gates;  /* fp32 [4D] */
  const void* W_pred;    /* bf16 [D][H] */
  const float* b_pred;   /* fp32 [H] */
  const void* W_enc;     /* bf16 [H_enc][H] */
  const float* b_enc;    /* fp32 [H] */
} tsd_pred_weights;

/* A decoder of the stateful form (greedy; prune_k 0; one LM or none).  E is
 * not used.  Stream export/import is not available for it. */
TSD_API tsd_status tsd_decoder_create_pred(const tsd_decoder_cfg* cfg, const tsd_pred_weights* pred,
                                           const void* W_out_bf16, const tsd_ngram* lm, const tsd_boost* boost,
                                           void* cuda_stream, tsd_decoder** out);
/* A stateful-form stream's prediction-network state: h (bf16 bits) and c,
 * D entries each (synchronizes). */
TSD_API tsd_status tsd_stream_pred_state(tsd_decoder* dec, int32_t slot, uint16_t* h, float* c);

/* The same with several n-gram LMs fused at once (Eq. 1, the sum over LMs
 * i of alpha_i log p_LM_i): LM i (host handle lms[i], same V, outliving the
 * decoder) enters with alpha_i = lambda * lm_weights[i], lambda being
 * decode_chunk's argument; lm_weights NULL means all 1.  0 <= n_lms <= 4;
 * n_lms > 1 needs greedy decoding (beam_k 1), else TSD_EINVAL.  Each stream
 * keeps one state per LM.  With n_lms 1 and weight 1 this is
 * tsd_decoder_create. */
TSD_API tsd_status tsd_decoder_create_multi(const tsd_decoder_cfg* cfg, const void* W_out_bf16,
                                            const void* E_bf16, const tsd_ngram* const* lms,
                                            const float* lm_weights, int32_t n_lms, const tsd_boost* boost,
                                            void* cuda_stream, tsd_decoder** out);
TSD_API void tsd_decoder_free(tsd_decoder* dec);

/* Opens a stream slot and resets its state on the decoder's stream: no
 * labels, previous label = blank (start of sequence), LM at the empty
 * context, phrase matching empty; beam: one empty hypothesis.
 * TSD_ESTATE if all slots are in use. */
TSD_API tsd_status tsd_stream_open(tsd_decoder* dec, int32_t* slot_out);
/* Frees a slot (TSD_ESTATE if it is not open). */
TSD_API tsd_status tsd_stream_close(tsd_decoder* dec, int32_t slot);

/* Decodes one encoder chunk of T frames for n open streams (the hot path).
 *   slots:  host int32 [n], distinct open slots; row i of every array below
 *           belongs to slots[i].
 *   enc_bf16: device bf16 [n][T][H], the chunk's encoder frames.
 *   lambda, beta: fusion weights of Eq. 1.
 *   Greedy (beam_k = 1): for each stream, labels are emitted frame by frame,
 *   at most max_symbols per frame, a blank or the limit ending the frame:
 *     out_tokens  device int32 [n][T*max_symbols]: emitted labels in order;
 *     out_frames  device int32 [n][T*max_symbols]: frame (0..T-1) of each;
 *     out_scores  device float [n][T*max_symbols]: its fused score (Eq. 1);
 *     out_counts  device int32 [n]: labels emitted this chunk.
 *   Beam (beam_k > 1), frame-synchronous with up to S = max_symbols labels
 *   per frame: each label step expands the hypotheses still in their frame
 *   by blank or a label; the top beam_k extensions are kept and, in order, a
 *   blank (or a label at the frame's S-th expansion) leaves the frame, the
 *   rest stay in it; within each set equal label sequences merge by
 *   log-sum-exp; the set that left keeps its beam_k best (in order of
 *   arrival) and becomes the next frame's beam when no hypothesis stays or
 *   after S expansions.  S = 1: one label or blank per frame.
 *   out_counts[i] = length of the best hypothesis, out_scores[i*T*max_symbols]
 *   = its score, out_tokens/out_frames are not written; read the labels with
 *   tsd_stream_result.  Each stream holds up to 8192 label-sequence nodes
 *   (at most beam_k per label step are added); a stream that outgrows them
 *   stops recording labels and tsd_decoder_check reports TSD_EDEVICE.
 * Asynchronous on cuda_stream (must be the decoder's stream order, see
 * above); the device arrays are borrowed until the stream passes this call.
 * T <= max_T and n <= max_streams, else TSD_EINVAL. */
TSD_API tsd_status tsd_decode_chunk(tsd_decoder* dec, int32_t n, const int32_t* slots,
                            const void* enc_bf16, int32_t T, float lambda, float beta,
                            int32_t* out_tokens, int32_t* out_frames, float* out_scores,
                            int32_t* out_counts, void* cuda_stream);

/* Reads a stream's state (synchronizes the decoder's stream; for a beam
 * decoder, that of the stream's first live hypothesis): the LM
 * state id (see tsd_ngram_state_tuple; 0 = empty context), the trie node
 * (tsd_boost_node_tuple; 0 = root) and the previous label (V = blank/SOS).
 * Any output pointer may be NULL. */
TSD_API tsd_status tsd_stream_state(tsd_decoder* dec, int32_t slot, int32_t* lm_state,
                            int32_t* trie_node, int32_t* last);

/* A stream's whole decoding state as a byte blob (synchronizes the
 * decoder's stream): previous label, every LM's and the trie's suffix
 * chains, and for beam decoders the hypotheses with their label sequences.
 * buf NULL: only *len (the bytes needed) is set; else cap must be >= *len
 * (TSD_EINVAL otherwise).  The blob is plain host memory owned by the
 * caller; importing it into an open slot of a decoder with the same V, beam
 * width, LMs and phrase tree (same tables) continues the stream there, so a
 * stream can move between decoders or devices, or be checkpointed.  Import
 * checks the blob's header, length and every id against the decoder's
 * tables before writing (TSD_EINVAL) and synchronizes. (No paper
 * counterpart: the paper's decoder keeps its state in the serving process.) */
TSD_API tsd_status tsd_stream_export(tsd_decoder* dec, int32_t slot, void* buf, int64_t cap, int64_t* len);
TSD_API tsd_status tsd_stream_import(tsd_decoder* dec, int32_t slot, const void* buf, int64_t len);

/* The state of LM lm_index (0 <= lm_index < number of LMs) for a slot
 * (beam: its first hypothesis), as tsd_stream_state reports the first LM's;
 * synchronizes with the decoder's last stream. */
TSD_API tsd_status tsd_stream_lm_state(tsd_decoder* dec, int32_t slot, int32_t lm_index, int32_t* lm_state);

/* Beam: the best live hypothesis of a slot (synchronizes): up to cap labels
 * into buf (host), *len = its length, *score = its score (may be NULL).
 * Greedy: not available (TSD_EINVAL); use the chunk outputs. */
TSD_API tsd_status tsd_stream_result(tsd_decoder* dec, int32_t slot, int32_t* buf, int32_t cap,
                             int32_t* len, float* score);

/* Beam: all live hypotheses of a slot (synchronizes).  Writes up to cap_hyps
 * entries: lengths[i], scores[i], and labels into buf at offsets i*cap_len
 * (up to cap_len each).  *n_hyps = live hypotheses. */
TSD_API tsd_status tsd_stream_hyps(tsd_decoder* dec, int32_t slot, int32_t* buf, int32_t cap_len,
                           int32_t* lengths, float* scores, int32_t cap_hyps, int32_t* n_hyps);

/* ------------------------------------------------------------------------
 * Execution control and instrumentation (no counterpart in the paper).
 */

/* 1 (default): each (n, T) shape of decode_chunk is captured once into a
 * CUDA graph and replayed; 0: kernels are launched one by one. */
TSD_API tsd_status tsd_decoder_set_graphs(tsd_decoder* dec, int32_t enable);

/* 1: record CUDA events around every kernel of later decode_chunk calls and
 * accumulate per-kernel device time; 0 (default): no events. */
TSD_API tsd_status tsd_decoder_set_timing(tsd_decoder* dec, int32_t enable);

/* Accumulated device time (ms) and launch counts since the last reset, per
 * kernel class: [0] row pass (state advance, LM + boost bias, joint input),
 * [1] joint GEMM with the fused log-softmax/selection epilogue, [2] the
 * stateful form's prediction network and projections (the chunk's encoder
 * copy and projection, each step's LSTM and joint-input GEMMs; 0 for a
 * stateless decoder).  n_classes (1..3) entries are written.  Waits for
 * outstanding timed work.  reset != 0 clears the totals after reading. */
TSD_API tsd_status tsd_decoder_timing(tsd_decoder* dec, double* ms, int64_t* launches, int32_t n_classes,
                              int32_t reset);

/* Algorithmic bytes counted by the row passes of timed decode_chunk calls
 * (set_timing(1)) since the last reset: per evaluated row, its partials, row
 * state, label searches, joint input and every arc of its LM chain levels and
 * trie chain nodes (the quantity the row pass's bandwidth roofline divides by
 * its time).  Waits for the device.  reset != 0 clears the total after reading. */
TSD_API tsd_status tsd_decoder_timed_bytes(tsd_decoder* dec, int64_t* row_bytes, int32_t reset);

/* Selects the joint GEMM kernel of later decode_chunk calls: 0 (default)
 * the tcgen05 tensor-core kernel, 1 the CUDA-core kernel (a cross-check of
 * the same contraction and epilogue).  Drops captured graphs. */
TSD_API tsd_status tsd_decoder_set_joint_kernel(tsd_decoder* dec, int32_t kind);

/* Waits for the decoder's stream and reports a device-side failure: every
 * wait inside the kernels is bounded, and one that expires records a code
 * that makes this call return TSD_EDEVICE (and clears it). */
TSD_API tsd_status tsd_decoder_check(tsd_decoder* dec);

/* Tuning knobs, by name (drops captured graphs):
 *   "pdl"      1 (default) / 0: programmatic dependent launch between the
 *              row pass and the joint kernel, so each kernel's set-up
 *              overlaps the tail of the one before;
 *   "joint_bn" 64, 128 or 256: labels per tensor-core CTA tile (default:
 *              chosen at create from the row count and the SM count);
 *   "fusion_path" 0 or 1, greedy decoding with at most one LM (default 0;
 *              1 keeps the V-wide logits out of memory):
 *              1 applies Eq. 1's level-0 LM term (a dense row per unigram
 *              state) in the joint kernel's epilogue and evaluates the other
 *              labels of the row's state (its longer contexts' continuations,
 *              the trie chain's children, blank) in the row pass; 0 is the
 *              streaming form, in which the joint kernel writes every logit
 *              and the row pass applies the whole LM and trie terms.  Both
 *              give the same decisions; TSD_EINVAL for other decoders;
 *   "wait_ns"  0 .. 1e10: the limit, in nanoseconds, of the joint kernel's
 *              waits for its operands and accumulator (default 1e9).  A wait
 *              that expires ends the kernel early -- after it has waited,
 *              with the 1 s limit, for every copy and MMA it started -- and
 *              the next tsd_decoder_check returns TSD_EDEVICE; that chunk's
 *              results are then undefined (but every index stays in range).
 *              A test hook for the failure path.
 * Unknown names return TSD_EINVAL. */
TSD_API tsd_status tsd_decoder_set_option(tsd_decoder* dec, const char* name, int64_t value);

/* Test hook: the n-th device allocation the library makes from now on
 * (n >= 1) fails as cudaMalloc would, and the call that makes it returns
 * TSD_ENOMEM after releasing what it had allocated; n = 0 turns the hook
 * off.  The hook is process-wide and fires once. */
TSD_API tsd_status tsd_debug_fail_alloc(int32_t n);

/* Measurement hook: launches one kernel of the last decode_chunk's final
 * label step reps times back to back on cuda_stream -- kernel 0 the row
 * pass (in a mode that redoes the step's work but commits no state or
 * output), kernel 1 the joint GEMM (idempotent) -- so a caller can time it
 * with CUDA events in isolation.  Later decode_chunk calls are unaffected.
 * If algo_bytes is non-NULL the call waits for the stream and stores the
 * algorithmic bytes of one launch: for the row pass, counted by the kernel
 * (partials, row state, label searches, joint input, every LM arc and trie
 * child of the chains, plus the shared unigram/root rows once; not the
 * dense bias it writes); for the joint kernel, its operands, bias rows and
 * partials.  TSD_ESTATE before the first decode_chunk. */
TSD_API tsd_status tsd_decoder_replay(tsd_decoder* dec, int32_t kernel, int32_t reps, void* cuda_stream,
                                      int64_t* algo_bytes);

/* ------------------------------------------------------------------------
 * Allocation-free joint selection (the paper has no counterpart; this is a
 * service for callers that cannot allocate device memory: code that runs
 * inside a memory pool or arena that owns all of the device's memory,
 * plugins handed pre-allocated buffers by their host framework, and
 * real-time paths that cannot afford cudaMalloc's implicit synchronization).
 *
 * For each of n rows: logits = A[r] . Wt^T (bf16 in, fp32 accumulate), the
 * log-softmax over the V+1 labels, and the label maximizing the fused value
 * logit + bias (bias 0 for blank = label V; ties to the lowest label):
 *   A_bf16   device bf16 [n][H], the joint input rows (16-byte aligned);
 *   Wt_bf16  device bf16 [V+1][H], W_out label-major (16-byte aligned);
 *   bias     device fp32 [n][V] (lambda*LM + beta*boost), or NULL for 0;
 *   out_label device int32 [n]; out_score device fp32 [n] = the fused value
 *   of out_label minus the row's log-sum-exp.
 * Limits: 1 <= n <= 1024, V + 1 <= 8192, H a multiple of 64 in [64, 8192];
 * larger sizes return TSD_EINVAL.  The call allocates nothing: its working
 * memory is a 1 MiB array compiled into the library, which every GPU that
 * loads the library keeps until the process exits.  The first call on a
 * device looks up that array's device address (cudaGetSymbolAddress); make
 * that first call before any stream capture.  The address is cached per
 * device for the life of the process: after cudaDeviceReset on a device the
 * cached address is stale, so do not call this entry point again on that
 * device in the same process.  All calls share the array:
 * calls that overlap on the GPU (different streams, or host threads on one
 * device without ordering) race and must be serialized by the caller.
 * Asynchronous on cuda_stream. */
TSD_API tsd_status tsd_joint_select_noalloc(int32_t n, int32_t H, int32_t V, const void* A_bf16,
                                            const void* Wt_bf16, const float* bias, int32_t* out_label,
                                            float* out_score, void* cuda_stream);

/* Kernel launches one decode_chunk(n, T) issues (for launch accounting). */
TSD_API tsd_status tsd_decoder_launches_per_chunk(const tsd_decoder* dec, int32_t n, int32_t T,
                                          int64_t* launches);

/* Test hook: when logits is non-NULL, later decode_chunk calls also write the
 * fp32 joint logits of every evaluation step s < max_steps into logits
 * (device float [max_steps][n*beam_k][V+1]) and, when rows is non-NULL, per
 * step and row the int32 quadruple (frame, previous label, LM state, trie
 * node) the step was evaluated at into rows (device [max_steps][n*beam_k][4]).
 * Pass NULLs to turn capture off.  Capture is slow; it is for parity tests. */
TSD_API tsd_status tsd_decoder_debug_capture(tsd_decoder* dec, float* logits, int32_t* rows,
                                     int32_t max_steps);

/* ------------------------------------------------------------------------
 * The cache-aware encoder chunk step (Sec. III-B: a FastConformer encoder
 * made streamable by chunked, limited-context attention and causal
 * convolutions, with a cache carried across chunks; Sec. IV-A: one encoder
 * frame is 80 ms and the look-ahead is the chunk).  Its output frames are
 * the enc input of tsd_decode_chunk (decoder H = d).
 *
 * Per stream and chunk of C encoder frames (C*stack feature frames):
 *   x = W_sub stack(features) + b_sub, then per block:
 *   x += 1/2 FF1(x);  x += MHSA(x);  x += Conv(x);  x += 1/2 FF2(x);
 *   x = LN_out(x)
 *   FF(x)   = W2 bf16(Swish(W1 bf16(LN(x)) + b1)) + b2
 *   MHSA(x) = W_o bf16(attn) + b_o with (q, k, v) = bf16(W_qkv bf16(LN(x))
 *             + b_qkv); per head a query frame sees the last `left` frames
 *             before its chunk (cached k, v) and every frame of its chunk,
 *             score = ((q + u).k + (q + v).p(delta)) / sqrt(dh), p(delta) =
 *             W_pos r(delta), r(delta) sinusoidal (sin at 2k, cos at 2k+1 of
 *             delta / 10000^(2k/d)), delta = query - key frame position
 *   Conv(x) = W_pw2 bf16(Swish(bn_scale (dw * g) + bn_shift)) + b_pw2 with
 *             g = bf16(a * sigmoid(b)), (a, b) = W_pw1 bf16(LN(x)) + b_pw1,
 *             dw * g the causal depthwise convolution over the last K
 *             frames of g (K-1 of them cached; zeros before the stream's
 *             first frame) plus b_dw
 * The chunk's output is bf16(x).  Matrix products take bf16 operands and
 * accumulate in fp32 on the tensor cores; the rest is fp32. */
typedef struct tsd_encoder tsd_encoder;

typedef struct {
  int32_t d;           /* model width: multiple of 128, 128 <= d <= 2048 */
  int32_t layers;      /* blocks, 1..64 */
  int32_t heads;       /* attention heads; d / heads is 64 or 128 */
  int32_t ff;          /* feed-forward width: multiple of 128, <= 8192 */
  int32_t kernel;      /* depthwise kernel K, 1..32 */
  int32_t left;        /* cached frames a query sees before its chunk, 0..128 */
  int32_t max_chunk;   /* largest C a call may pass, 1..32 */
  int32_t feat;        /* feature bins per 10 ms frame */
  int32_t stack;       /* feature frames per encoder frame; stack*feat a multiple of 64, <= 8192 */
  int32_t max_streams; /* slots, 1..4096 */
} tsd_encoder_cfg;

/* One block's weights, all device arrays (copied at create).  Matrices are
 * bf16 [out][in] row-major (y = W x); vectors fp32. */
typedef struct {
  const float *ln_ff1_g, *ln_ff1_b;
  const void* ff1_w1;  const float* ff1_b1;   /* [ff][d], [ff] */
  const void* ff1_w2;  const float* ff1_b2;   /* [d][ff], [d] */
  const float *ln_att_g, *ln_att_b;
  const void* qkv_w;   const float* qkv_b;    /* [3d][d] (rows q, k, v; head h owns columns h*dh..), [3d] */
  const void* pos_w;                          /* [d][d] */
  const float *pos_u, *pos_v;                 /* [d] each (head h: entries h*dh..) */
  const void* out_w;   const float* out_b;    /* [d][d], [d] */
  const float *ln_conv_g, *ln_conv_b;
  const void* pw1_w;   const float* pw1_b;    /* [2d][d] (rows 0..d-1 the GLU value, d..2d-1 its gate), [2d] */
  const float *dw_w, *dw_b;                   /* [d][K] (tap K-1 is the current frame), [d] */
  const float *bn_scale, *bn_shift;           /* [d] each */
  const void* pw2_w;   const float* pw2_b;    /* [d][d], [d] */
  const float *ln_ff2_g, *ln_ff2_b;
  const void* ff2_w1;  const float* ff2_b1;
  const void* ff2_w2;  const float* ff2_b2;
  const float *ln_out_g, *ln_out_b;
} tsd_encoder_layer;

/* Creates an encoder: sub_w bf16 [d][stack*feat] and sub_b fp32 [d] (device),
 * layers[cfg.layers].  Allocates all device memory up front (weights,
 * position tables, every slot's cache, work buffers for max_streams *
 * max_chunk frames).  TSD_EINVAL on a shape outside the limits above. */
TSD_API tsd_status tsd_encoder_create(const tsd_encoder_cfg* cfg, const void* sub_w, const float* sub_b,
                                      const tsd_encoder_layer* layers, void* cuda_stream, tsd_encoder** out);
TSD_API void tsd_encoder_free(tsd_encoder* enc);

/* Opens a stream slot with an empty cache (its first chunk sees no
 * history); TSD_ESTATE when every slot is open.  Asynchronous on the
 * encoder's last stream. */
TSD_API tsd_status tsd_encoder_open(tsd_encoder* enc, int32_t* slot_out);
TSD_API tsd_status tsd_encoder_close(tsd_encoder* enc, int32_t slot);

/* Encodes one chunk of C encoder frames for n open slots (host array
 * slots[n], distinct).  feats: device bf16 [n][C*stack][feat] (stream i's
 * feature frames, oldest first); out: device bf16 [n][C][d].  Each slot's
 * cache advances by C frames.  Asynchronous on cuda_stream; the first call
 * for an (n, C) captures a CUDA graph.  TSD_EINVAL on n, C outside
 * [1, max_streams] x [1, max_chunk]; TSD_ESTATE on a slot that is not open. */
TSD_API tsd_status tsd_encode_chunk(tsd_encoder* enc, int32_t n, const int32_t* slots, const void* feats_bf16,
                                    int32_t C, void* out_bf16, void* cuda_stream);

/* Waits for the encoder's stream; TSD_EDEVICE if a bounded wait inside a
 * kernel expired (the code is cleared). */
TSD_API tsd_status tsd_encoder_check(tsd_encoder* enc);

/* 1: later encode_chunk calls record CUDA events around every kernel and
 * accumulate device time per class: [0] tensor-core GEMMs, [1] attention,
 * [2] the rest (layer norms, depthwise convolution, cache bookkeeping). */
TSD_API tsd_status tsd_encoder_set_timing(tsd_encoder* enc, int32_t enable);
TSD_API tsd_status tsd_encoder_timing(tsd_encoder* enc, double* ms, int64_t* launches, int32_t n_classes,
                                      int32_t reset);
/* Tensor-core FLOPs of one encode_chunk(n, C) (2 M N K summed over its GEMMs). */
TSD_API tsd_status tsd_encoder_gemm_flops(const tsd_encoder* enc, int32_t n, int32_t C, double* flops);
/* Kernel launches of one encode_chunk(n, C) with timing off (for launch
 * accounting): the call's streams run as up to two parallel graph branches
 * of at least 256 frame rows each, each branch the subsampling GEMM, the
 * first block's first layer norm and 14 kernels per block (a block's
 * closing layer norm also computes the next block's first one), then one
 * kernel that advances the frame counts.  TSD_EINVAL on n, C outside
 * [1, max_streams] x [1, max_chunk]. */
TSD_API tsd_status tsd_encoder_launches_per_chunk(const tsd_encoder* enc, int32_t n, int32_t C, int64_t* launches);

#ifdef __cplusplus
}
#endif

#endif /* TSD_H */
