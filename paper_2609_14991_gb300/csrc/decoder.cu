// Decoder host driver: creation, stream slots and the per-chunk label loop.
//
// One decode_chunk(n, T) is T*max_sym label steps (the most any stream can
// need); each step is a row pass (decide, advance, joint input, fusion bias)
// followed by the joint GEMM with its fused selection epilogue, and a final
// row pass applies the last decision.  Every launch reads the call's
// arguments from a small device block written just before, so the whole
// chunk is captured once per (n, T) as a CUDA graph and replayed.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <memory>
#include <new>
#include <string>
#include <type_traits>

#include "decoder.h"
#include "gemm_tc.h"
#include "joint_tc.h"

using namespace tsd;

namespace {

int round_up(int x, int m) { return (x + m - 1) / m * m; }

tsd_status set_device(const tsd_decoder* d) {
  int cur = -1;
  TSD_CUDA(cudaGetDevice(&cur));
  if (cur != d->device) TSD_CUDA(cudaSetDevice(d->device));
  return TSD_OK;
}

int steps_per_chunk(const tsd_decoder* d, int T) { return T * d->cfg.max_symbols; }

// Events enqueue_chunk records with timing on: a mark before every row pass
// and joint launch (and, for the stateful form, before the chunk's encoder
// projection and each step's prediction-network GEMMs), and one at the end.
int n_marks(const tsd_decoder* d, int S) { return d->pred.D ? 3 * S + 4 : 2 * S + 2; }

// Enqueues one chunk's launches; with events, records one at each kernel
// boundary (external records, so they survive graph capture).
void enqueue_chunk(tsd_decoder* d, int M, int T, cudaStream_t s, const std::vector<cudaEvent_t>* ev,
                   std::vector<int8_t>* cls_out) {
  const int S = steps_per_chunk(d, T);
  int e = 0;
  // timed chunks also count the row passes' algorithmic bytes (second counter)
  DecView v = d->view;
  if (ev) {
    v.count = 1;
    v.ctr = d->view.ctr + 1;
  }
  auto mark = [&](int cls) {
    if (!ev) return;
    cudaEventRecordWithFlags((*ev)[(size_t)e], s, cudaEventRecordExternal);
    if (cls_out) (*cls_out)[(size_t)e] = (int8_t)cls;
    ++e;
  };
  const tsd_decoder::Pred& pr = d->pred;
  launch_defaults(v, s);
  if (pr.D) {
    // the chunk's encoder frames to a fixed buffer, then their projection
    mark(2);
    launch_copy_enc(v, (int64_t)M * T * pr.Henc, s, false);
    GemmArgs ge{M * T, d->cfg.H, pr.Henc, d->cfg.H, pr.be, v.pred_penc};
    launch_gemm_tc(kEncProj, v, ge, pr.encA, pr.encB, s, d->pdl && !ev);
  }
  for (int step = 0; step <= S; ++step) {
    const bool pdl = d->pdl && !ev && step > 0;  // the first launch follows the parameter copy
    NvtxRange nvtx_step("label step");  // host-side enqueue (captured once into the chunk's graph)
    mark(0);
    if (d->cfg.beam_k > 1) launch_row_beam(v, M / d->cfg.beam_k, step, step == S ? 1 : 0, d->row_smem, s, pdl);
    else if (d->cfg.prune_k > 0) launch_row_pruned(v, M, step, step == S ? 1 : 0, s, pdl);
    else if (v.fused && v.fz_dense) launch_row_fused(v, M, step, step == S ? 1 : 0, row_fused_smem_bytes(d->V4, d->N_pad), s, pdl);
    else if (v.fused) launch_row_stream(v, M, step, step == S ? 1 : 0, row_stream_smem_bytes(d->V4), s, pdl);
    else launch_row(v, M, step, step == S ? 1 : 0, d->row_smem, s, pdl);
    if (pr.D) {
      // the prediction network reads the labels just emitted; after the last
      // decision of the chunk only its state matters
      mark(2);
      GemmArgs gl{M, 4 * pr.D, 2 * pr.D, 0, pr.bg, nullptr};
      launch_gemm_tc(kLstm, v, gl, pr.lstmA, pr.lstmB, s, d->pdl && !ev);
      if (step < S) {
        GemmArgs gp{M, d->cfg.H, pr.D, d->cfg.H, pr.bp, nullptr};
        launch_gemm_tc(kJointIn, v, gp, pr.projA, pr.projB, s, d->pdl && !ev);
      }
    }
    if (step < S) {
      mark(1);
      if (d->joint_kind == 0) launch_joint_tc(*d->jtc, v, M, step, s, d->pdl && !ev);
      else launch_joint(v, M, step, s);
    }
  }
  mark(-1);
}

void harvest(tsd_decoder* d, tsd_decoder::EventSet& es) {
  if (!es.pending) return;
  cudaEventSynchronize(es.ev.back());
  for (size_t i = 0; i + 1 < es.ev.size(); ++i) {
    float ms = 0.f;
    const int c = es.cls[i];
    if (c >= 0 && c < 3 && cudaEventElapsedTime(&ms, es.ev[i], es.ev[i + 1]) == cudaSuccess) {
      d->ms[c] += ms;
      d->launches[c] += 1;
    }
  }
  cudaGetLastError();
  es.pending = false;
}

void destroy_set(tsd_decoder::EventSet& es) {
  if (es.exec) cudaGraphExecDestroy(es.exec);
  for (cudaEvent_t e : es.ev) cudaEventDestroy(e);
  es.ev.clear();
  es.exec = nullptr;
}

}  // namespace

namespace {
tsd_status create_impl(const tsd_decoder_cfg* cfg, const void* W_out_bf16, const void* E_bf16,
                       const tsd_ngram* const* lms, const float* lm_weights, int32_t n_lms, const tsd_boost* boost,
                       void* cuda_stream, tsd_decoder** out, const tsd_pred_weights* pw = nullptr) {
  if (!out) return fail(TSD_EINVAL, "tsd_decoder_create: out is NULL");
  *out = nullptr;
  if (!cfg || !W_out_bf16 || (!E_bf16 && !pw)) return fail(TSD_EINVAL, "tsd_decoder_create: NULL argument");
  if (pw) {
    if (pw->D < 64 || pw->D > 2048 || pw->D % 64)
      return fail(TSD_EINVAL, "tsd_decoder_create_pred: D=%d must be a multiple of 64 in [64, 2048]", pw->D);
    if (pw->H_enc < 64 || pw->H_enc > 8192 || pw->H_enc % 64)
      return fail(TSD_EINVAL, "tsd_decoder_create_pred: H_enc=%d must be a multiple of 64 in [64, 8192]", pw->H_enc);
    if (!pw->emb || !pw->W_gates || !pw->b_gates || !pw->W_pred || !pw->b_pred || !pw->W_enc || !pw->b_enc)
      return fail(TSD_EINVAL, "tsd_decoder_create_pred: NULL weight");
    if (cfg->beam_k != 1 || cfg->prune_k != 0)
      return fail(TSD_EINVAL, "tsd_decoder_create_pred: greedy decoding without pruning only");
  }
  const tsd_decoder_cfg c = *cfg;
  if (n_lms < 0 || n_lms > kMaxLm) return fail(TSD_EINVAL, "tsd_decoder_create: %d LMs, at most %d", n_lms, kMaxLm);
  if (n_lms > 0 && !lms) return fail(TSD_EINVAL, "tsd_decoder_create: NULL LM list");
  for (int i = 0; i < n_lms; ++i) {
    if (!lms[i]) return fail(TSD_EINVAL, "tsd_decoder_create: LM %d is NULL", i);
    if (lm_weights && !std::isfinite(lm_weights[i])) return fail(TSD_EINVAL, "tsd_decoder_create: LM weight %d not finite", i);
    if (lms[i]->view.V != c.V) return fail(TSD_EINVAL, "tsd_decoder_create: LM %d has V=%d, decoder V=%d", i, lms[i]->view.V, c.V);
  }
  if (n_lms > 1 && c.beam_k > 1) return fail(TSD_EINVAL, "tsd_decoder_create: several LMs need greedy decoding (beam_k 1)");
  if (c.prune_k < 0 || c.prune_k > 8) return fail(TSD_EINVAL, "tsd_decoder_create: prune_k=%d outside [0, 8]", c.prune_k);
  if (c.prune_k > 0 && (c.beam_k > 1 || n_lms > 1))
    return fail(TSD_EINVAL, "tsd_decoder_create: pruned fusion needs greedy decoding and at most one LM");
  if (c.prune_k > 0 && ((c.V + 1 + kNPad - 1) / kNPad * kNPad / 64) * c.prune_k > 512)
    return fail(TSD_EINVAL, "tsd_decoder_create: prune_k * (V+1)/64 must be <= 512");
  const tsd_ngram* lm = n_lms > 0 ? lms[0] : nullptr;
  if (c.V < 1 || c.V > 16384) return fail(TSD_EINVAL, "tsd_decoder_create: V=%d out of range [1, 16384]", c.V);
  if (c.H < 64 || c.H > 8192 || c.H % 64) return fail(TSD_EINVAL, "tsd_decoder_create: H=%d must be a multiple of 64 in [64, 8192]", c.H);
  if (c.beam_k < 1 || c.beam_k > 8) return fail(TSD_EINVAL, "tsd_decoder_create: beam_k=%d outside [1, 8]", c.beam_k);
  if (c.beam_k > 1 && ((c.V + 1 + kNPad - 1) / kNPad * kNPad / 64) * c.beam_k > 512)
    return fail(TSD_EINVAL, "tsd_decoder_create: beam_k * (V+1)/64 must be <= 512");
  if (c.max_symbols < 1 || c.max_symbols > 64) return fail(TSD_EINVAL, "tsd_decoder_create: max_symbols=%d out of range", c.max_symbols);
  if (c.max_streams < 1 || (int64_t)c.max_streams * c.beam_k > 4096)
    return fail(TSD_EINVAL, "tsd_decoder_create: max_streams=%d out of range", c.max_streams);
  if (c.max_T < 1 || c.max_T > 4096) return fail(TSD_EINVAL, "tsd_decoder_create: max_T=%d out of range", c.max_T);
  if (lm && lm->view.V != c.V) return fail(TSD_EINVAL, "tsd_decoder_create: LM has V=%d, decoder V=%d", lm->view.V, c.V);
  if (boost && boost->view.V != c.V) return fail(TSD_EINVAL, "tsd_decoder_create: boost has V=%d, decoder V=%d", boost->view.V, c.V);

  std::unique_ptr<tsd_decoder> d(new (std::nothrow) tsd_decoder());
  if (!d) return fail(TSD_ENOMEM, "tsd_decoder_create: host allocation failed");
  d->cfg = c;
  TSD_CUDA(cudaGetDevice(&d->device));
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  d->lm = lm;
  d->n_lm = n_lms;
  d->boost = boost;
  d->N = c.V + 1;
  d->N_pad = round_up(d->N, kNPad);
  d->M_max = c.max_streams * c.beam_k;
  d->M_pad = round_up(d->M_max, kMPad);
  d->n_ptiles = d->N_pad / kPartialCols;
  d->V4 = round_up(c.V, 16);
  // greedy decoding with at most one LM (whose unigram states have their
  // dense rows): the joint kernel's epilogue applies Eq. 1 up to the row's
  // correction list; several LMs and beam search keep the dense bias row
  const bool fused = c.beam_k == 1 && c.prune_k == 0 && n_lms <= 1 &&
                     (n_lms == 0 || !lm_weights || lm_weights[0] == 1.f) &&
                     (!lm || lm->view.order < 2 || lm->view.n_dense == lm->view.V);
  d->row_smem = fused ? std::max(row_fused_smem_bytes(d->V4, d->N_pad), row_stream_smem_bytes(d->V4))
                      : row_smem_bytes(d->V4, n_lms);
  if (d->row_smem > 200 * 1024) return fail(TSD_EINVAL, "tsd_decoder_create: V too large for the row pass");

  DevArena& A = d->arena;
  DecView& v = d->view;
  uint16_t *Wt = nullptr, *E = nullptr, *Abuf = nullptr;
  float* bias = nullptr;
  float4* part = nullptr;
  int32_t *rt = nullptr, *rs = nullptr, *rc = nullptr, *sl = nullptr, *sll = nullptr, *slc = nullptr, *stl = nullptr,
          *stc = nullptr, *err = nullptr;
  int4 *slr = nullptr, *strc = nullptr;
  unsigned long long* ctr = nullptr;
  float2* bpart = nullptr;
  float* dflt = nullptr;
  uint32_t* droot = nullptr;
  double* hscore = nullptr;
  int32_t *hlive = nullptr, *hnode = nullptr, *hlen = nullptr, *ppar = nullptr, *ptok = nullptr, *pn = nullptr;
  unsigned long long* hhash = nullptr;
  const size_t SK = (size_t)c.max_streams * c.beam_k;
  const size_t NL = (size_t)std::max(1, n_lms);  // LM state blocks
  d->params_bytes = sizeof(Params) + sizeof(int32_t) * (size_t)c.max_streams;
  char* pdev = nullptr;
  tsd_status st;
  if ((st = A.alloc(&Wt, (size_t)d->N_pad * c.H)) || (st = A.alloc(&E, (size_t)d->N * c.H)) ||
      (st = A.alloc(&Abuf, (size_t)d->M_pad * c.H)) || (st = A.alloc(&bias, (size_t)d->M_pad * d->N_pad)) ||
      (st = A.alloc(&part, (size_t)d->M_pad * (d->N_pad / 64))) || (st = A.alloc(&err, 1)) || (st = A.alloc(&ctr, 2)) || (st = A.alloc(&dflt, (size_t)d->V4)) || (st = A.alloc(&droot, (size_t)(d->V4 + 31) / 32)) || (st = A.alloc(&rt, (size_t)d->M_pad)) ||
      (st = A.alloc(&rs, (size_t)d->M_pad)) || (st = A.alloc(&rc, (size_t)d->M_pad)) ||
      (st = A.alloc(&sl, SK)) || (st = A.alloc(&sll, SK * NL)) || (st = A.alloc(&slc, SK * NL * kLmChain)) ||
      (st = A.alloc(&stl, SK)) || (st = A.alloc(&stc, SK * kTrChain)) || (st = A.alloc(&pdev, d->params_bytes)) ||
      (st = A.alloc(&slr, SK * kLmChain)) || (st = A.alloc(&strc, SK * kTrChain))) {
    A.release();
    return st;
  }
  if (fused) {
    v.mask_words = d->N_pad / 32;
    if ((st = A.alloc(&v.logits, (size_t)d->M_pad * d->N_pad)) || (st = A.alloc(&v.dvec, (size_t)d->N_pad)) ||
        (st = A.alloc(&v.c_lab, (size_t)d->M_pad * d->V4)) || (st = A.alloc(&v.c_add, (size_t)d->M_pad * d->V4)) ||
        (st = A.alloc(&v.c_info, (size_t)d->M_pad)) ||
        (st = A.alloc(&v.c_mask, (size_t)d->M_pad * v.mask_words)) || (st = A.alloc(&v.m_last, (size_t)d->M_pad)) ||
        (st = A.alloc(&v.m_lm_len, (size_t)d->M_pad)) || (st = A.alloc(&v.m_tr_len, (size_t)d->M_pad)) ||
        (st = A.alloc(&v.m_lm, (size_t)d->M_pad * kLmChain)) || (st = A.alloc(&v.m_lmr, (size_t)d->M_pad * kLmChain)) ||
        (st = A.alloc(&v.m_tr, (size_t)d->M_pad * kTrChain)) || (st = A.alloc(&v.m_trr, (size_t)d->M_pad * kTrChain))) {
      A.release();
      return st;
    }
    TSD_CUDA(cudaMemsetAsync(v.dvec, 0, sizeof(float) * (size_t)d->N_pad, s));
    TSD_CUDA(cudaMemsetAsync(v.logits, 0, sizeof(float) * (size_t)d->M_pad * d->N_pad, s));
    // no dense row and an empty list until a row pass has written the row's
    TSD_CUDA(cudaMemsetAsync(v.c_info, 0xff, sizeof(int4) * (size_t)d->M_pad, s));
    TSD_CUDA(cudaMemsetAsync(v.c_mask, 0, sizeof(uint32_t) * (size_t)d->M_pad * v.mask_words, s));
  }
  v.fused = fused ? 1 : 0;
  // the streaming form by default; the dense epilogue (fusion_path 1) keeps
  // the V-wide logits out of memory and runs within a few percent of it with
  // a wide vocabulary and many rows
  v.fz_dense = 0;
  const int topk = c.beam_k > 1 ? c.beam_k : c.prune_k;
  if (c.beam_k == 1 && c.prune_k > 0) {
    if ((st = A.alloc(&bpart, (size_t)d->M_pad * (d->N_pad / 64) * (1 + topk)))) {
      A.release();
      return st;
    }
  }
  if (c.beam_k > 1) {
    const size_t pool = (size_t)c.max_streams * kPoolCap;
    if ((st = A.alloc(&bpart, (size_t)d->M_pad * (d->N_pad / 64) * (1 + c.beam_k))) || (st = A.alloc(&hscore, SK)) ||
        (st = A.alloc(&hlive, SK)) || (st = A.alloc(&hnode, SK)) || (st = A.alloc(&hlen, SK)) ||
        (st = A.alloc(&hhash, SK)) || (st = A.alloc(&ppar, pool)) || (st = A.alloc(&ptok, pool)) ||
        (st = A.alloc(&pn, (size_t)c.max_streams)) || (st = A.alloc(&v.f_score, SK)) ||
        (st = A.alloc(&v.f_live, SK)) || (st = A.alloc(&v.f_node, SK)) || (st = A.alloc(&v.f_len, SK)) ||
        (st = A.alloc(&v.f_last, SK)) || (st = A.alloc(&v.f_lml, SK)) || (st = A.alloc(&v.f_trl, SK)) ||
        (st = A.alloc(&v.f_lmc, SK * kLmChain)) || (st = A.alloc(&v.f_trc, SK * kTrChain)) ||
        (st = A.alloc(&v.f_hash, SK)) || (st = A.alloc(&v.b_frame, (size_t)c.max_streams)) ||
        (st = A.alloc(&v.b_exp, (size_t)c.max_streams))) {
      A.release();
      return st;
    }
    TSD_CUDA(cudaMemsetAsync(v.f_live, 0, SK * sizeof(int32_t), s));
    TSD_CUDA(cudaMemsetAsync(v.b_frame, 0, (size_t)c.max_streams * sizeof(int32_t), s));
    TSD_CUDA(cudaMemsetAsync(v.b_exp, 0, (size_t)c.max_streams * sizeof(int32_t), s));
    if (!bpart || !hscore || !hlive || !hnode || !hlen || !hhash || !ppar || !ptok || !pn) {
      A.release();
      return fail(TSD_ENOMEM, "tsd_decoder_create: beam state not allocated");
    }
  }
  // stateful form: weights (repacked K-major), state and step buffers
  uint16_t *p_emb = nullptr, *p_h = nullptr, *p_x = nullptr, *p_hin = nullptr, *p_enc = nullptr;
  float *p_c = nullptr, *p_penc = nullptr;
  int32_t *p_fresh = nullptr, *p_flag = nullptr;
  if (pw) {
    tsd_decoder::Pred& pr = d->pred;
    pr.D = pw->D;
    pr.Henc = pw->H_enc;
    pr.G_pad = round_up(4 * pw->D, 128);
    pr.H_pad = round_up(c.H, 128);
    pr.MT_pad = round_up(c.max_streams * c.max_T, 128);
    const size_t D = (size_t)pw->D;
    if ((st = A.alloc(&p_emb, (size_t)d->N * D)) || (st = A.alloc(&pr.Wg, (size_t)pr.G_pad * 2 * D)) ||
        (st = A.alloc(&pr.bg, 4 * D)) || (st = A.alloc(&pr.Wp, (size_t)pr.H_pad * D)) ||
        (st = A.alloc(&pr.bp, (size_t)c.H)) || (st = A.alloc(&pr.We, (size_t)pr.H_pad * pr.Henc)) ||
        (st = A.alloc(&pr.be, (size_t)c.H)) || (st = A.alloc(&p_h, SK * D)) || (st = A.alloc(&p_c, SK * D)) ||
        (st = A.alloc(&p_fresh, SK)) || (st = A.alloc(&p_x, (size_t)d->M_pad * 2 * D)) ||
        (st = A.alloc(&p_hin, (size_t)d->M_pad * D)) || (st = A.alloc(&p_flag, (size_t)d->M_pad)) ||
        (st = A.alloc(&p_enc, (size_t)pr.MT_pad * pr.Henc)) || (st = A.alloc(&p_penc, (size_t)pr.MT_pad * c.H))) {
      A.release();
      return st;
    }
  }
  auto cleanup = [&](tsd_status e) {
    delete d->jtc;
    d->jtc = nullptr;
    for (int i = 0; i < tsd_decoder::kRing; ++i) {
      if (d->staging[i]) cudaFreeHost(d->staging[i]);
      if (d->staging_ev[i]) cudaEventDestroy(d->staging_ev[i]);
    }
    if (d->cap_stream) cudaStreamDestroy(d->cap_stream);
    A.release();
    return e;
  };
  cudaError_t ce;
  if ((ce = cudaMemsetAsync(Abuf, 0, sizeof(uint16_t) * (size_t)d->M_pad * c.H, s)) != cudaSuccess ||
      (ce = cudaMemsetAsync(bias, 0, sizeof(float) * (size_t)d->M_pad * d->N_pad, s)) != cudaSuccess ||
      (ce = cudaMemsetAsync(sll, 0, sizeof(int32_t) * SK * NL, s)) != cudaSuccess ||
      (ce = cudaMemsetAsync(stl, 0, sizeof(int32_t) * SK, s)) != cudaSuccess ||
      (ce = cudaMemsetAsync(err, 0, sizeof(int32_t), s)) != cudaSuccess ||
      (ce = cudaMemsetAsync(ctr, 0, 2 * sizeof(unsigned long long), s)) != cudaSuccess ||
      (ce = E_bf16 ? cudaMemcpyAsync(E, E_bf16, sizeof(uint16_t) * (size_t)d->N * c.H, cudaMemcpyDeviceToDevice, s)
                   : cudaMemsetAsync(E, 0, sizeof(uint16_t) * (size_t)d->N * c.H, s)) != cudaSuccess)
    return cleanup(cuda_fail(ce, "tsd_decoder_create: initial copies"));
  launch_repack(static_cast<const uint16_t*>(W_out_bf16), Wt, c.H, d->N, d->N_pad, s);
  if ((ce = cudaGetLastError()) != cudaSuccess) return cleanup(cuda_fail(ce, "tsd_decoder_create: repack"));
  if (pw) {
    tsd_decoder::Pred& pr = d->pred;
    const size_t D = (size_t)pr.D;
    if ((ce = cudaMemcpyAsync(p_emb, pw->emb, 2 * (size_t)d->N * D, cudaMemcpyDeviceToDevice, s)) != cudaSuccess ||
        (ce = cudaMemcpyAsync(pr.bg, pw->b_gates, 16 * D, cudaMemcpyDeviceToDevice, s)) != cudaSuccess ||
        (ce = cudaMemcpyAsync(pr.bp, pw->b_pred, 4 * (size_t)c.H, cudaMemcpyDeviceToDevice, s)) != cudaSuccess ||
        (ce = cudaMemcpyAsync(pr.be, pw->b_enc, 4 * (size_t)c.H, cudaMemcpyDeviceToDevice, s)) != cudaSuccess ||
        (ce = cudaMemsetAsync(p_h, 0, 2 * SK * D, s)) != cudaSuccess ||
        (ce = cudaMemsetAsync(p_c, 0, 4 * SK * D, s)) != cudaSuccess ||
        (ce = cudaMemsetAsync(p_fresh, 0, 4 * SK, s)) != cudaSuccess ||
        (ce = cudaMemsetAsync(p_flag, 0, 4 * (size_t)d->M_pad, s)) != cudaSuccess ||
        (ce = cudaMemsetAsync(p_x, 0, 4 * (size_t)d->M_pad * D, s)) != cudaSuccess ||
        (ce = cudaMemsetAsync(p_hin, 0, 2 * (size_t)d->M_pad * D, s)) != cudaSuccess ||
        (ce = cudaMemsetAsync(p_enc, 0, 2 * (size_t)pr.MT_pad * pr.Henc, s)) != cudaSuccess)
      return cleanup(cuda_fail(ce, "tsd_decoder_create_pred: weights"));
    // K-major copies of the three weight matrices (rows past N are zero)
    launch_repack(static_cast<const uint16_t*>(pw->W_gates), pr.Wg, 2 * pr.D, 4 * pr.D, pr.G_pad, s);
    launch_repack(static_cast<const uint16_t*>(pw->W_pred), pr.Wp, pr.D, c.H, pr.H_pad, s);
    launch_repack(static_cast<const uint16_t*>(pw->W_enc), pr.We, pr.Henc, c.H, pr.H_pad, s);
    if ((ce = cudaGetLastError()) != cudaSuccess) return cleanup(cuda_fail(ce, "tsd_decoder_create_pred: repack"));
    if (!gemm_tc_map_a(&pr.encA, p_enc, pr.MT_pad, pr.Henc) || !gemm_tc_map_b(&pr.encB, kEncProj, pr.We, pr.H_pad, pr.Henc) ||
        !gemm_tc_map_a(&pr.lstmA, p_x, d->M_pad, 2 * pr.D) || !gemm_tc_map_b(&pr.lstmB, kLstm, pr.Wg, pr.G_pad, 2 * pr.D) ||
        !gemm_tc_map_a(&pr.projA, p_hin, d->M_pad, pr.D) || !gemm_tc_map_b(&pr.projB, kJointIn, pr.Wp, pr.H_pad, pr.D))
      return cleanup(fail(TSD_ECUDA, "tsd_decoder_create_pred: TMA descriptors"));
    if ((ce = gemm_tc_prepare()) != cudaSuccess) return cleanup(cuda_fail(ce, "tsd_decoder_create_pred: kernel attributes"));
  }
  if ((ce = prepare_kernels(row_smem_bytes(d->V4, n_lms))) != cudaSuccess)
    return cleanup(cuda_fail(ce, "tsd_decoder_create: kernel attributes"));
  if (fused && ((ce = prepare_fused_kernels(d->row_smem)) != cudaSuccess ||
                (ce = prepare_stream_kernels(d->row_smem)) != cudaSuccess))
    return cleanup(cuda_fail(ce, "tsd_decoder_create: kernel attributes"));
  if ((ce = prepare_beam_kernels(d->row_smem)) != cudaSuccess) return cleanup(cuda_fail(ce, "tsd_decoder_create: kernel attributes"));
  if (hlive && (ce = cudaMemsetAsync(hlive, 0, sizeof(int32_t) * SK, s)) != cudaSuccess)
    return cleanup(cuda_fail(ce, "tsd_decoder_create: initial copies"));
  {
    int sms = 0;
    if ((ce = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, d->device)) != cudaSuccess)
      return cleanup(cuda_fail(ce, "tsd_decoder_create: SM count"));
    d->jtc = new (std::nothrow) JointTc();
    if (!d->jtc) return cleanup(fail(TSD_ENOMEM, "tsd_decoder_create: host allocation failed"));
    d->sms = sms;
    d->view.sms = sms;
    const int bn = joint_tc_pick_bn(d->M_max, d->N_pad, sms);
    if ((ce = joint_tc_prepare(d->jtc, Abuf, d->M_pad, Wt, d->N_pad, c.H, bn, bias, v.logits)) != cudaSuccess)
      return cleanup(cuda_fail(ce, "tsd_decoder_create: tensor-core GEMM setup (TMA descriptors)"));
  }
  for (int i = 0; i < tsd_decoder::kRing; ++i) {
    if ((ce = cudaHostAlloc(reinterpret_cast<void**>(&d->staging[i]), d->params_bytes, cudaHostAllocDefault)) != cudaSuccess)
      return cleanup(fail(TSD_ENOMEM, "tsd_decoder_create: pinned staging: %s", cudaGetErrorString(ce)));
    if ((ce = cudaEventCreateWithFlags(&d->staging_ev[i], cudaEventDisableTiming)) != cudaSuccess)
      return cleanup(cuda_fail(ce, "tsd_decoder_create: event"));
  }
  if ((ce = cudaStreamCreateWithFlags(&d->cap_stream, cudaStreamNonBlocking)) != cudaSuccess)
    return cleanup(cuda_fail(ce, "tsd_decoder_create: capture stream"));

  v.V = c.V;
  v.N = d->N;
  v.N_pad = d->N_pad;
  v.H = c.H;
  v.max_sym = c.max_symbols;
  v.K = c.beam_k;
  v.topk = topk;
  v.prune = c.prune_k;
  d->n_ptiles = d->N_pad / d->jtc->bn;
  v.n_ptiles = d->n_ptiles;
  v.V4 = d->V4;
  v.params = reinterpret_cast<const Params*>(pdev);
  d->params_dev = reinterpret_cast<Params*>(pdev);
  v.E = E;
  v.Wt = Wt;
  v.A = Abuf;
  v.bias = bias;
  v.part = part;
  v.r_t = rt;
  v.r_sym = rs;
  v.r_cnt = rc;
  v.s_last = sl;
  v.s_lm_len = sll;
  v.s_lm_chain = slc;
  v.s_tr_len = stl;
  v.s_tr_chain = stc;
  v.s_lm_rec = slr;
  v.s_tr_rec = strc;
  v.pred_D = pw ? pw->D : 0;
  v.pred_emb = p_emb;
  v.pred_h = p_h;
  v.pred_c = p_c;
  v.pred_fresh = p_fresh;
  v.pred_x = p_x;
  v.pred_hin = p_hin;
  v.pflag = p_flag;
  v.pred_enc = p_enc;
  v.pred_penc = p_penc;
  v.has_lm = lm ? 1 : 0;
  v.has_tr = boost ? 1 : 0;
  if (lm) v.lm = lm->view;
  v.n_lm = n_lms;
  v.lm_stride = (int32_t)SK;
  for (int i = 0; i < kMaxLm; ++i) {
    v.lmx[i] = i < n_lms ? lms[i]->view : LmView();
    v.lm_w[i] = i < n_lms ? (lm_weights ? lm_weights[i] : 1.f) : 0.f;
  }
  if (boost) v.tr = boost->view;
  v.cap_logits = nullptr;
  v.cap_rows = nullptr;
  v.cap_steps = 0;
  v.err = err;
  v.wait_ns = tc_wait_ns_default();
  v.ctr = ctr;
  v.count = 0;
  v.dflt = dflt;
  v.droot = droot;
  v.bpart = bpart;
  v.h_score = hscore;
  v.h_live = hlive;
  v.h_node = hnode;
  v.h_len = hlen;
  v.h_hash = hhash;
  v.pool_parent = ppar;
  v.pool_tok = ptok;
  v.pool_n = pn;
  v.pool_cap = kPoolCap;
  d->slot_open.assign((size_t)c.max_streams, 0);
  d->last_stream = s;
  *out = d.release();
  return TSD_OK;
}
}  // namespace

extern "C" tsd_status tsd_decoder_create(const tsd_decoder_cfg* cfg, const void* W_out_bf16,
                                         const void* E_bf16, const tsd_ngram* lm,
                                         const tsd_boost* boost, void* cuda_stream,
                                         tsd_decoder** out) {
  clear_error();
  const tsd_ngram* one[1] = {lm};
  return create_impl(cfg, W_out_bf16, E_bf16, one, nullptr, lm ? 1 : 0, boost, cuda_stream, out);
}

extern "C" tsd_status tsd_decoder_create_pred(const tsd_decoder_cfg* cfg, const tsd_pred_weights* pred,
                                              const void* W_out_bf16, const tsd_ngram* lm, const tsd_boost* boost,
                                              void* cuda_stream, tsd_decoder** out) {
  clear_error();
  if (!pred) return fail(TSD_EINVAL, "tsd_decoder_create_pred: NULL weights");
  const tsd_ngram* one[1] = {lm};
  return create_impl(cfg, W_out_bf16, nullptr, one, nullptr, lm ? 1 : 0, boost, cuda_stream, out, pred);
}

extern "C" tsd_status tsd_stream_pred_state(tsd_decoder* d, int32_t slot, uint16_t* h, float* c) {
  clear_error();
  if (!d || !h || !c) return fail(TSD_EINVAL, "tsd_stream_pred_state: NULL argument");
  if (!d->pred.D) return fail(TSD_EINVAL, "tsd_stream_pred_state: not a stateful-form decoder");
  if (slot < 0 || slot >= d->cfg.max_streams || !d->slot_open[(size_t)slot])
    return fail(TSD_ESTATE, "tsd_stream_pred_state: slot %d is not open", slot);
  tsd_status st = set_device(d);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  const size_t D = (size_t)d->pred.D;
  TSD_CUDA(cudaMemcpy(h, d->view.pred_h + (size_t)slot * D, 2 * D, cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(c, d->view.pred_c + (size_t)slot * D, 4 * D, cudaMemcpyDeviceToHost));
  return TSD_OK;
}

extern "C" tsd_status tsd_decoder_create_multi(const tsd_decoder_cfg* cfg, const void* W_out_bf16,
                                               const void* E_bf16, const tsd_ngram* const* lms,
                                               const float* lm_weights, int32_t n_lms, const tsd_boost* boost,
                                               void* cuda_stream, tsd_decoder** out) {
  clear_error();
  return create_impl(cfg, W_out_bf16, E_bf16, lms, lm_weights, n_lms, boost, cuda_stream, out);
}

extern "C" void tsd_decoder_free(tsd_decoder* d) {
  if (!d) return;
  set_device(d);
  cudaDeviceSynchronize();
  for (auto& kv : d->entries) {
    destroy_set(kv.second.set[0]);
    destroy_set(kv.second.set[1]);
  }
  for (int i = 0; i < tsd_decoder::kRing; ++i) {
    if (d->staging[i]) cudaFreeHost(d->staging[i]);
    if (d->staging_ev[i]) cudaEventDestroy(d->staging_ev[i]);
  }
  if (d->cap_stream) cudaStreamDestroy(d->cap_stream);
  d->arena.release();
  delete d->jtc;
  cudaGetLastError();
  delete d;
}

extern "C" tsd_status tsd_stream_open(tsd_decoder* d, int32_t* slot_out) {
  clear_error();
  if (!d || !slot_out) return fail(TSD_EINVAL, "tsd_stream_open: NULL argument");
  auto it = std::find(d->slot_open.begin(), d->slot_open.end(), 0);
  if (it == d->slot_open.end()) return fail(TSD_ESTATE, "tsd_stream_open: all %d slots are open", d->cfg.max_streams);
  tsd_status st = set_device(d);
  if (st) return st;
  int slot = (int)(it - d->slot_open.begin());
  if (d->cfg.beam_k > 1 && (!d->view.h_live || !d->view.pool_n))
    return fail(TSD_ESTATE, "tsd_stream_open: beam state missing");
  if (d->cfg.beam_k > 1) launch_open_beam(d->view, slot, d->last_stream);
  else launch_open(d->view, slot, d->last_stream);
  if (d->pred.D) launch_open_pred(d->view, slot, d->last_stream);
  TSD_CUDA(cudaGetLastError());
  *it = 1;
  *slot_out = slot;
  return TSD_OK;
}

extern "C" tsd_status tsd_stream_close(tsd_decoder* d, int32_t slot) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_stream_close: NULL decoder");
  if (slot < 0 || slot >= d->cfg.max_streams || !d->slot_open[(size_t)slot])
    return fail(TSD_ESTATE, "tsd_stream_close: slot %d is not open", slot);
  d->slot_open[(size_t)slot] = 0;
  return TSD_OK;
}

extern "C" tsd_status tsd_decode_chunk(tsd_decoder* d, int32_t n, const int32_t* slots,
                                       const void* enc_bf16, int32_t T, float lambda, float beta,
                                       int32_t* out_tokens, int32_t* out_frames, float* out_scores,
                                       int32_t* out_counts, void* cuda_stream) {
  clear_error();
  NvtxRange nvtx("tsd_decode_chunk");
  if (!d || !slots || !enc_bf16 || !out_counts) return fail(TSD_EINVAL, "tsd_decode_chunk: NULL argument");
  if (d->cfg.beam_k == 1 && (!out_tokens || !out_frames || !out_scores))
    return fail(TSD_EINVAL, "tsd_decode_chunk: NULL output array");
  if (d->cfg.beam_k > 1 && !out_scores) return fail(TSD_EINVAL, "tsd_decode_chunk: NULL out_scores");
  if (n < 1 || n > d->cfg.max_streams) return fail(TSD_EINVAL, "tsd_decode_chunk: n=%d out of [1, %d]", n, d->cfg.max_streams);
  if (T < 1 || T > d->cfg.max_T) return fail(TSD_EINVAL, "tsd_decode_chunk: T=%d out of [1, %d]", T, d->cfg.max_T);
  if (!std::isfinite(lambda) || !std::isfinite(beta)) return fail(TSD_EINVAL, "tsd_decode_chunk: non-finite weight");
  {
    std::vector<uint8_t> seen((size_t)d->cfg.max_streams, 0);
    for (int i = 0; i < n; ++i) {
      int s = slots[i];
      if (s < 0 || s >= d->cfg.max_streams || !d->slot_open[(size_t)s])
        return fail(TSD_ESTATE, "tsd_decode_chunk: slot %d is not open", s);
      if (seen[(size_t)s]) return fail(TSD_EINVAL, "tsd_decode_chunk: slot %d listed twice", s);
      seen[(size_t)s] = 1;
    }
  }
  tsd_status st = set_device(d);
  if (st) return st;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  d->last_stream = s;

  // call parameters -> pinned staging -> device
  const int slot_i = d->ring_pos;
  d->ring_pos = (d->ring_pos + 1) % tsd_decoder::kRing;
  TSD_CUDA(cudaEventSynchronize(d->staging_ev[slot_i]));
  Params* hp = reinterpret_cast<Params*>(d->staging[slot_i]);
  hp->enc = static_cast<const uint16_t*>(enc_bf16);
  hp->out_tok = out_tokens;
  hp->out_frame = out_frames;
  hp->out_score = out_scores;
  hp->out_count = out_counts;
  hp->n = n;
  hp->T = T;
  hp->lambda = lambda;
  hp->beta = beta;
  std::memcpy(hp->slots, slots, sizeof(int32_t) * (size_t)n);
  const size_t bytes = sizeof(Params) + sizeof(int32_t) * (size_t)n;
  TSD_CUDA(cudaMemcpyAsync(d->params_dev, hp, bytes, cudaMemcpyHostToDevice, s));
  TSD_CUDA(cudaEventRecord(d->staging_ev[slot_i], s));

  const int M = n * d->cfg.beam_k;
  const int S = steps_per_chunk(d, T);
  d->last_n = n;
  d->last_T = T;
  const int n_events = n_marks(d, S);
  auto key = std::make_tuple(n, T, d->use_graphs, d->timing);
  tsd_decoder::Entry& ent = d->entries[key];
  tsd_decoder::EventSet& es = ent.set[ent.next];
  if (d->timing) {
    ent.next ^= 1;
    harvest(d, es);
    if (es.ev.empty()) {
      es.ev.resize((size_t)n_events);
      es.cls.assign((size_t)n_events, -1);
      for (auto& e : es.ev) TSD_CUDA(cudaEventCreate(&e));
    }
  }
  const std::vector<cudaEvent_t>* evp = d->timing ? &es.ev : nullptr;
  if (d->use_graphs) {
    if (!es.exec) {
      cudaGraph_t g = nullptr;
      TSD_CUDA(cudaStreamBeginCapture(d->cap_stream, cudaStreamCaptureModeThreadLocal));
      enqueue_chunk(d, M, T, d->cap_stream, evp, d->timing ? &es.cls : nullptr);
      cudaError_t ce = cudaStreamEndCapture(d->cap_stream, &g);
      if (ce != cudaSuccess) return cuda_fail(ce, "tsd_decode_chunk: graph capture");
      ce = cudaGraphInstantiate(&es.exec, g, 0);
      cudaGraphDestroy(g);
      if (ce != cudaSuccess) {
        es.exec = nullptr;
        return cuda_fail(ce, "tsd_decode_chunk: graph instantiate");
      }
    }
    NvtxRange nvtx_launch("chunk graph launch");
    TSD_CUDA(cudaGraphLaunch(es.exec, s));
  } else {
    enqueue_chunk(d, M, T, s, evp, d->timing ? &es.cls : nullptr);
    TSD_CUDA(cudaGetLastError());
  }
  if (d->timing) es.pending = true;
  return TSD_OK;
}

extern "C" tsd_status tsd_stream_state(tsd_decoder* d, int32_t slot, int32_t* lm_state,
                                       int32_t* trie_node, int32_t* last) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_stream_state: NULL decoder");
  if (slot < 0 || slot >= d->cfg.max_streams || !d->slot_open[(size_t)slot])
    return fail(TSD_ESTATE, "tsd_stream_state: slot %d is not open", slot);
  tsd_status st = set_device(d);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  int32_t ll = 0, tl = 0, ls = 0, chain_lm[kLmChain], chain_tr[kTrChain];
  const DecView& v = d->view;
  const size_t h = (size_t)slot * d->cfg.beam_k;  // beam: the slot's first hypothesis
  TSD_CUDA(cudaMemcpy(&ls, v.s_last + h, 4, cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(&ll, v.s_lm_len + h, 4, cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(&tl, v.s_tr_len + h, 4, cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(chain_lm, v.s_lm_chain + h * kLmChain, sizeof(chain_lm), cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(chain_tr, v.s_tr_chain + h * kTrChain, sizeof(chain_tr), cudaMemcpyDeviceToHost));
  if (lm_state) *lm_state = ll > 0 ? chain_lm[ll - 1] : 0;
  if (trie_node) *trie_node = tl > 0 ? chain_tr[0] : 0;
  if (last) *last = ls;
  return TSD_OK;
}

extern "C" tsd_status tsd_stream_lm_state(tsd_decoder* d, int32_t slot, int32_t lm_index, int32_t* lm_state) {
  clear_error();
  if (!d || !lm_state) return fail(TSD_EINVAL, "tsd_stream_lm_state: NULL argument");
  if (slot < 0 || slot >= d->cfg.max_streams || !d->slot_open[(size_t)slot])
    return fail(TSD_ESTATE, "tsd_stream_lm_state: slot %d is not open", slot);
  if (lm_index < 0 || lm_index >= d->n_lm)
    return fail(TSD_EINVAL, "tsd_stream_lm_state: LM %d outside [0, %d)", lm_index, d->n_lm);
  tsd_status st = set_device(d);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  const DecView& v = d->view;
  const size_t h = (size_t)lm_index * (size_t)v.lm_stride + (size_t)slot * d->cfg.beam_k;
  int32_t ll = 0, chain[kLmChain];
  TSD_CUDA(cudaMemcpy(&ll, v.s_lm_len + h, 4, cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(chain, v.s_lm_chain + h * kLmChain, sizeof(chain), cudaMemcpyDeviceToHost));
  *lm_state = ll > 0 ? chain[ll - 1] : 0;
  return TSD_OK;
}

namespace {
// Stream state blob: a header, then per hypothesis (K = beam width) the
// previous label, each LM's chain (length + kLmChain ids), the trie chain
// (length + kTrChain ids), and for beam decoders the hypothesis record
// (live, node, length, score, hash); then the beam's label-sequence nodes.
struct BlobHeader {
  uint32_t magic, version;
  int32_t V, beam_k, n_lm, has_tr, pool_used, reserved;
};
constexpr uint32_t kBlobMagic = 0x53445354u;  // "TSDS"

int64_t blob_bytes(const tsd_decoder* d, int32_t pool_used) {
  const int K = d->cfg.beam_k, L = std::max(1, d->n_lm);
  int64_t per = 4 + (int64_t)L * 4 * (1 + kLmChain) + 4 * (1 + kTrChain);
  if (K > 1) per += 4 + 4 + 4 + 8 + 8;
  return (int64_t)sizeof(BlobHeader) + per * K + (K > 1 ? 8ll * pool_used : 0);
}

template <class T>
tsd_status copy_dev(T* dst, const T* src, size_t n, cudaMemcpyKind kind) {
  TSD_CUDA(cudaMemcpy(dst, src, sizeof(T) * n, kind));
  return TSD_OK;
}
}  // namespace

extern "C" tsd_status tsd_stream_export(tsd_decoder* d, int32_t slot, void* buf, int64_t cap, int64_t* len) {
  clear_error();
  if (!d || !len) return fail(TSD_EINVAL, "tsd_stream_export: NULL argument");
  if (d->pred.D) return fail(TSD_EINVAL, "tsd_stream_export: not available for the stateful form");
  if (slot < 0 || slot >= d->cfg.max_streams || !d->slot_open[(size_t)slot])
    return fail(TSD_ESTATE, "tsd_stream_export: slot %d is not open", slot);
  tsd_status st = set_device(d);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  const DecView& v = d->view;
  const int K = d->cfg.beam_k, L = std::max(1, d->n_lm);
  int32_t pool_used = 0;
  if (K > 1) TSD_CUDA(cudaMemcpy(&pool_used, v.pool_n + slot, 4, cudaMemcpyDeviceToHost));
  *len = blob_bytes(d, pool_used);
  if (!buf) return TSD_OK;
  if (cap < *len) return fail(TSD_EINVAL, "tsd_stream_export: %lld bytes needed, cap %lld", (long long)*len, (long long)cap);
  char* p = static_cast<char*>(buf);
  BlobHeader hd{kBlobMagic, 1u, d->cfg.V, K, d->n_lm, v.has_tr, pool_used, 0};
  std::memcpy(p, &hd, sizeof(hd));
  p += sizeof(hd);
  auto put = [&](const auto* src, size_t n) -> tsd_status {
    tsd_status s2 = copy_dev(reinterpret_cast<std::remove_const_t<std::remove_pointer_t<decltype(src)>>*>(p), src, n,
                             cudaMemcpyDeviceToHost);
    p += sizeof(*src) * n;
    return s2;
  };
  for (int k = 0; k < K; ++k) {
    const size_t h = (size_t)slot * K + k;
    if ((st = put(v.s_last + h, 1))) return st;
    for (int m = 0; m < L; ++m) {
      const size_t hm = (size_t)m * v.lm_stride + h;
      if ((st = put(v.s_lm_len + hm, 1)) || (st = put(v.s_lm_chain + hm * kLmChain, kLmChain))) return st;
    }
    if ((st = put(v.s_tr_len + h, 1)) || (st = put(v.s_tr_chain + h * kTrChain, kTrChain))) return st;
    if (K > 1 && ((st = put(v.h_live + h, 1)) || (st = put(v.h_node + h, 1)) || (st = put(v.h_len + h, 1)) ||
                  (st = put(v.h_score + h, 1)) || (st = put(v.h_hash + h, 1))))
      return st;
  }
  if (K > 1 && pool_used > 0) {
    if ((st = put(v.pool_parent + (size_t)slot * v.pool_cap, (size_t)pool_used)) ||
        (st = put(v.pool_tok + (size_t)slot * v.pool_cap, (size_t)pool_used)))
      return st;
  }
  return TSD_OK;
}

extern "C" tsd_status tsd_stream_import(tsd_decoder* d, int32_t slot, const void* buf, int64_t len) {
  clear_error();
  if (!d || !buf) return fail(TSD_EINVAL, "tsd_stream_import: NULL argument");
  if (d->pred.D) return fail(TSD_EINVAL, "tsd_stream_import: not available for the stateful form");
  if (slot < 0 || slot >= d->cfg.max_streams || !d->slot_open[(size_t)slot])
    return fail(TSD_ESTATE, "tsd_stream_import: slot %d is not open", slot);
  if (len < (int64_t)sizeof(BlobHeader)) return fail(TSD_EINVAL, "tsd_stream_import: blob too short");
  BlobHeader hd;
  std::memcpy(&hd, buf, sizeof(hd));
  const DecView& v = d->view;
  const int K = d->cfg.beam_k, L = std::max(1, d->n_lm);
  if (hd.magic != kBlobMagic || hd.version != 1u) return fail(TSD_EINVAL, "tsd_stream_import: not a stream state blob");
  if (hd.V != d->cfg.V || hd.beam_k != K || hd.n_lm != d->n_lm || hd.has_tr != v.has_tr)
    return fail(TSD_EINVAL, "tsd_stream_import: blob is for V=%d beam %d, %d LMs, boost %d; decoder has V=%d beam %d, %d LMs, boost %d",
                hd.V, hd.beam_k, hd.n_lm, hd.has_tr, d->cfg.V, K, d->n_lm, v.has_tr);
  if (hd.pool_used < 0 || hd.pool_used > v.pool_cap || len != blob_bytes(d, hd.pool_used))
    return fail(TSD_EINVAL, "tsd_stream_import: blob length %lld does not match its header", (long long)len);
  // check the contents before anything reaches the device
  {
    const char* q = static_cast<const char*>(buf) + sizeof(hd);
    auto rd = [&](size_t bytes) { const char* r = q; q += bytes; return r; };
    for (int k = 0; k < K; ++k) {
      int32_t last;
      std::memcpy(&last, rd(4), 4);
      if (last < 0 || last > d->cfg.V) return fail(TSD_EINVAL, "tsd_stream_import: previous label %d out of range", last);
      for (int m = 0; m < L; ++m) {
        int32_t n;
        std::memcpy(&n, rd(4), 4);
        const char* ch = rd(4 * kLmChain);
        if (n < 0 || n > kLmChain) return fail(TSD_EINVAL, "tsd_stream_import: LM chain length %d", n);
        const int64_t S = m < d->n_lm ? v.lmx[m].n_states : 1;
        for (int l = 0; l < n; ++l) {
          int32_t sid;
          std::memcpy(&sid, ch + 4 * l, 4);
          if (sid < 0 || sid >= S) return fail(TSD_EINVAL, "tsd_stream_import: LM state %d out of range", sid);
        }
      }
      int32_t tn;
      std::memcpy(&tn, rd(4), 4);
      const char* tch = rd(4 * kTrChain);
      if (tn < 0 || tn > kTrChain) return fail(TSD_EINVAL, "tsd_stream_import: trie chain length %d", tn);
      for (int l = 0; l < tn; ++l) {
        int32_t nd;
        std::memcpy(&nd, tch + 4 * l, 4);
        if (nd < 0 || nd >= v.tr.n_nodes) return fail(TSD_EINVAL, "tsd_stream_import: trie node %d out of range", nd);
      }
      if (K > 1) {
        int32_t node;
        rd(4);
        std::memcpy(&node, rd(4), 4);
        rd(4 + 8 + 8);
        if (node < -1 || node >= hd.pool_used) return fail(TSD_EINVAL, "tsd_stream_import: sequence node %d out of range", node);
      }
    }
    for (int32_t i = 0; K > 1 && i < hd.pool_used; ++i) {
      int32_t par, tok;
      std::memcpy(&par, q + 4 * (size_t)i, 4);
      std::memcpy(&tok, q + 4 * ((size_t)hd.pool_used + i), 4);
      if (par < -1 || par >= i) return fail(TSD_EINVAL, "tsd_stream_import: sequence node %d has parent %d", i, par);
      if (tok < 0 || tok >= d->cfg.V) return fail(TSD_EINVAL, "tsd_stream_import: sequence node %d has label %d", i, tok);
    }
  }
  tsd_status st = set_device(d);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  const char* p = static_cast<const char*>(buf) + sizeof(hd);
  auto get = [&](auto* dst, size_t n) -> tsd_status {
    tsd_status s2 = copy_dev(dst, reinterpret_cast<const std::remove_pointer_t<decltype(dst)>*>(p), n,
                             cudaMemcpyHostToDevice);
    p += sizeof(*dst) * n;
    return s2;
  };
  for (int k = 0; k < K; ++k) {
    const size_t h = (size_t)slot * K + k;
    if ((st = get(v.s_last + h, 1))) return st;
    for (int m = 0; m < L; ++m) {
      const size_t hm = (size_t)m * v.lm_stride + h;
      if ((st = get(v.s_lm_len + hm, 1)) || (st = get(v.s_lm_chain + hm * kLmChain, kLmChain))) return st;
    }
    if ((st = get(v.s_tr_len + h, 1)) || (st = get(v.s_tr_chain + h * kTrChain, kTrChain))) return st;
    if (K > 1 && ((st = get(v.h_live + h, 1)) || (st = get(v.h_node + h, 1)) || (st = get(v.h_len + h, 1)) ||
                  (st = get(v.h_score + h, 1)) || (st = get(v.h_hash + h, 1))))
      return st;
  }
  if (K > 1) {
    if (hd.pool_used > 0 && ((st = get(v.pool_parent + (size_t)slot * v.pool_cap, (size_t)hd.pool_used)) ||
                             (st = get(v.pool_tok + (size_t)slot * v.pool_cap, (size_t)hd.pool_used))))
      return st;
    TSD_CUDA(cudaMemcpy(v.pool_n + slot, &hd.pool_used, 4, cudaMemcpyHostToDevice));
  } else {
    // the greedy pass keeps each chain element's table records: derive them
    launch_fix_records(v, slot, d->last_stream);
    TSD_CUDA(cudaGetLastError());
    TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  }
  return TSD_OK;
}

namespace {
// Live hypotheses of a beam slot, read back from the device (synchronizes).
struct HostHyp {
  std::vector<int32_t> y;
  double score;
};

tsd_status read_hyps(tsd_decoder* d, int32_t slot, std::vector<HostHyp>& out) {
  const int K = d->cfg.beam_k;
  tsd_status st = set_device(d);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  const DecView& v = d->view;
  std::vector<int32_t> live(K), node(K), len(K);
  std::vector<double> score(K);
  const size_t h = (size_t)slot * K;
  TSD_CUDA(cudaMemcpy(live.data(), v.h_live + h, sizeof(int32_t) * K, cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(node.data(), v.h_node + h, sizeof(int32_t) * K, cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(len.data(), v.h_len + h, sizeof(int32_t) * K, cudaMemcpyDeviceToHost));
  TSD_CUDA(cudaMemcpy(score.data(), v.h_score + h, sizeof(double) * K, cudaMemcpyDeviceToHost));
  int32_t used = 0;
  TSD_CUDA(cudaMemcpy(&used, v.pool_n + slot, sizeof(int32_t), cudaMemcpyDeviceToHost));
  std::vector<int32_t> par((size_t)std::max(used, 1)), tok((size_t)std::max(used, 1));
  if (used > 0) {
    TSD_CUDA(cudaMemcpy(par.data(), v.pool_parent + (size_t)slot * v.pool_cap, sizeof(int32_t) * used, cudaMemcpyDeviceToHost));
    TSD_CUDA(cudaMemcpy(tok.data(), v.pool_tok + (size_t)slot * v.pool_cap, sizeof(int32_t) * used, cudaMemcpyDeviceToHost));
  }
  out.clear();
  for (int k = 0; k < K; ++k) {
    if (!live[k]) continue;
    HostHyp hy;
    hy.score = score[k];
    for (int x = node[k], i = 0; x >= 0 && x < used && i <= used; x = par[x], ++i) hy.y.push_back(tok[x]);
    std::reverse(hy.y.begin(), hy.y.end());
    out.push_back(std::move(hy));
  }
  return TSD_OK;
}

tsd_status check_beam_slot(tsd_decoder* d, int32_t slot, const char* fn) {
  if (!d) return fail(TSD_EINVAL, "%s: NULL decoder", fn);
  if (d->cfg.beam_k < 2) return fail(TSD_EINVAL, "%s: only beam decoders keep hypotheses", fn);
  if (slot < 0 || slot >= d->cfg.max_streams || !d->slot_open[(size_t)slot])
    return fail(TSD_ESTATE, "%s: slot %d is not open", fn, slot);
  return TSD_OK;
}
}  // namespace

extern "C" tsd_status tsd_stream_result(tsd_decoder* d, int32_t slot, int32_t* buf, int32_t cap, int32_t* len,
                                        float* score) {
  clear_error();
  tsd_status st = check_beam_slot(d, slot, "tsd_stream_result");
  if (st) return st;
  if (!len || (cap > 0 && !buf)) return fail(TSD_EINVAL, "tsd_stream_result: NULL output");
  std::vector<HostHyp> hy;
  if ((st = read_hyps(d, slot, hy))) return st;
  size_t best = 0;
  for (size_t i = 1; i < hy.size(); ++i)
    if (hy[i].score > hy[best].score) best = i;
  if (hy.empty()) {
    *len = 0;
    if (score) *score = 0.f;
    return TSD_OK;
  }
  *len = (int32_t)hy[best].y.size();
  for (int32_t i = 0; i < *len && i < cap; ++i) buf[i] = hy[best].y[(size_t)i];
  if (score) *score = (float)hy[best].score;
  return TSD_OK;
}

extern "C" tsd_status tsd_stream_hyps(tsd_decoder* d, int32_t slot, int32_t* buf, int32_t cap_len, int32_t* lengths,
                                      float* scores, int32_t cap_hyps, int32_t* n_hyps) {
  clear_error();
  tsd_status st = check_beam_slot(d, slot, "tsd_stream_hyps");
  if (st) return st;
  if (!n_hyps) return fail(TSD_EINVAL, "tsd_stream_hyps: NULL output");
  std::vector<HostHyp> hy;
  if ((st = read_hyps(d, slot, hy))) return st;
  *n_hyps = (int32_t)hy.size();
  for (int32_t i = 0; i < (int32_t)hy.size() && i < cap_hyps; ++i) {
    if (lengths) lengths[i] = (int32_t)hy[(size_t)i].y.size();
    if (scores) scores[i] = (float)hy[(size_t)i].score;
    if (buf)
      for (int32_t j = 0; j < (int32_t)hy[(size_t)i].y.size() && j < cap_len; ++j)
        buf[(size_t)i * cap_len + j] = hy[(size_t)i].y[(size_t)j];
  }
  return TSD_OK;
}

extern "C" tsd_status tsd_decoder_set_graphs(tsd_decoder* d, int32_t enable) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_decoder_set_graphs: NULL decoder");
  d->use_graphs = enable ? 1 : 0;
  return TSD_OK;
}

extern "C" tsd_status tsd_decoder_set_timing(tsd_decoder* d, int32_t enable) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_decoder_set_timing: NULL decoder");
  d->timing = enable ? 1 : 0;
  return TSD_OK;
}

extern "C" tsd_status tsd_decoder_timing(tsd_decoder* d, double* ms, int64_t* launches,
                                         int32_t n_classes, int32_t reset) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_decoder_timing: NULL decoder");
  tsd_status st = set_device(d);
  if (st) return st;
  for (auto& kv : d->entries) {
    harvest(d, kv.second.set[0]);
    harvest(d, kv.second.set[1]);
  }
  for (int i = 0; i < n_classes && i < 3; ++i) {
    if (ms) ms[i] = d->ms[i];
    if (launches) launches[i] = d->launches[i];
  }
  if (reset) {
    for (int i = 0; i < 3; ++i) {
      d->ms[i] = 0;
      d->launches[i] = 0;
    }
  }
  return TSD_OK;
}

extern "C" tsd_status tsd_decoder_timed_bytes(tsd_decoder* d, int64_t* row_bytes, int32_t reset) {
  clear_error();
  if (!d || !row_bytes) return fail(TSD_EINVAL, "tsd_decoder_timed_bytes: NULL argument");
  tsd_status st = set_device(d);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  unsigned long long b = 0;
  TSD_CUDA(cudaMemcpy(&b, d->view.ctr + 1, sizeof(b), cudaMemcpyDeviceToHost));
  *row_bytes = (int64_t)b;
  if (reset) TSD_CUDA(cudaMemset(d->view.ctr + 1, 0, sizeof(b)));
  return TSD_OK;
}

extern "C" tsd_status tsd_decoder_launches_per_chunk(const tsd_decoder* d, int32_t n, int32_t T,
                                                     int64_t* launches) {
  clear_error();
  if (!d || !launches) return fail(TSD_EINVAL, "tsd_decoder_launches_per_chunk: NULL argument");
  (void)n;
  const int64_t S = steps_per_chunk(d, T);
  *launches = d->pred.D ? 4 * S + 4 : 2 * S + 2;  // stateful form: + copy, projection, LSTM and joint input
  return TSD_OK;
}

namespace {
tsd_status drop_graphs(tsd_decoder* d) {
  tsd_status st = set_device(d);
  if (st) return st;
  cudaDeviceSynchronize();
  for (auto& kv : d->entries) {
    harvest(d, kv.second.set[0]);
    harvest(d, kv.second.set[1]);
    destroy_set(kv.second.set[0]);
    destroy_set(kv.second.set[1]);
  }
  d->entries.clear();
  return TSD_OK;
}
}  // namespace

extern "C" tsd_status tsd_decoder_set_joint_kernel(tsd_decoder* d, int32_t kind) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_decoder_set_joint_kernel: NULL decoder");
  if (kind != 0 && kind != 1) return fail(TSD_EINVAL, "tsd_decoder_set_joint_kernel: kind must be 0 or 1");
  if (kind == 1 && d->cfg.prune_k > 0)
    return fail(TSD_EINVAL, "tsd_decoder_set_joint_kernel: the CUDA-core kernel has no pruned-fusion epilogue");
  d->joint_kind = kind;
  d->n_ptiles = kind == 0 ? d->N_pad / d->jtc->bn : d->N_pad / kPartialCols;
  d->view.n_ptiles = d->n_ptiles;
  return drop_graphs(d);
}

extern "C" tsd_status tsd_decoder_set_option(tsd_decoder* d, const char* name, int64_t value) {
  clear_error();
  if (!d || !name) return fail(TSD_EINVAL, "tsd_decoder_set_option: NULL argument");
  const std::string n(name);
  if (n == "pdl") {
    d->pdl = value ? 1 : 0;
    return drop_graphs(d);
  }
  if (n == "wait_ns") {
    // limit of the joint kernel's progress waits; an expired wait ends the
    // kernel early (after draining its copies) and tsd_decoder_check reports it
    if (value < 0 || value > 10000000000ll)
      return fail(TSD_EINVAL, "tsd_decoder_set_option: wait_ns must be in [0, 1e10]");
    d->view.wait_ns = (unsigned long long)value;
    return drop_graphs(d);
  }
  if (n == "fusion_path") {
    // greedy decoding with at most one LM: 1 = Eq. 1's level-0 LM term in the
    // joint kernel's epilogue with a per-row correction list, 0 = the
    // streaming form (the row pass applies the LM and trie terms)
    if (value != 0 && value != 1) return fail(TSD_EINVAL, "tsd_decoder_set_option: fusion_path must be 0 or 1");
    if (!d->view.fused) return fail(TSD_EINVAL, "tsd_decoder_set_option: fusion_path applies to greedy decoding with at most one LM");
    d->view.fz_dense = (int32_t)value;
    return drop_graphs(d);
  }
  if (n == "joint_bn") {
    if (value != 64 && value != 128 && value != 256) return fail(TSD_EINVAL, "tsd_decoder_set_option: joint_bn must be 64, 128 or 256");
    tsd_status st = drop_graphs(d);
    if (st) return st;
    cudaError_t ce = joint_tc_prepare(d->jtc, d->view.A, d->M_pad, d->view.Wt, d->N_pad, d->cfg.H, (int)value,
                                      d->view.bias, d->view.logits);
    if (ce != cudaSuccess) return cuda_fail(ce, "tsd_decoder_set_option: joint_bn");
    if (d->joint_kind == 0) {
      d->n_ptiles = d->N_pad / d->jtc->bn;
      d->view.n_ptiles = d->n_ptiles;
    }
    return TSD_OK;
  }
  return fail(TSD_EINVAL, "tsd_decoder_set_option: unknown option '%s'", name);
}

extern "C" tsd_status tsd_decoder_replay(tsd_decoder* d, int32_t kernel, int32_t reps, void* cuda_stream,
                                         int64_t* algo_bytes) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_decoder_replay: NULL decoder");
  if (kernel != 0 && kernel != 1) return fail(TSD_EINVAL, "tsd_decoder_replay: kernel must be 0 (row pass) or 1 (joint)");
  if (reps < 1) return fail(TSD_EINVAL, "tsd_decoder_replay: reps < 1");
  if (d->last_n < 1) return fail(TSD_ESTATE, "tsd_decoder_replay: no chunk decoded yet");
  tsd_status st = set_device(d);
  if (st) return st;
  cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
  const int M = d->last_n * d->cfg.beam_k;
  const int S = steps_per_chunk(d, d->last_T);
  if (algo_bytes) TSD_CUDA(cudaMemsetAsync(d->view.ctr, 0, sizeof(unsigned long long), s));
  for (int i = 0; i < reps; ++i) {
    if (kernel == 0 && d->cfg.beam_k > 1) launch_row_beam(d->view, d->last_n, S - 1, 2, d->row_smem, s, false);
    else if (kernel == 0 && d->cfg.prune_k > 0) launch_row_pruned(d->view, M, S - 1, 2, s, false);
    else if (kernel == 0 && d->view.fused && d->view.fz_dense) launch_row_fused(d->view, M, S - 1, 2, row_fused_smem_bytes(d->V4, d->N_pad), s, false);
    else if (kernel == 0 && d->view.fused) launch_row_stream(d->view, M, S - 1, 2, row_stream_smem_bytes(d->V4), s, false);
    else if (kernel == 0) launch_row(d->view, M, S - 1, 2, d->row_smem, s, false);
    else if (d->joint_kind == 0) launch_joint_tc(*d->jtc, d->view, M, 1 << 30, s, false);
    else launch_joint(d->view, M, 1 << 30, s);
  }
  TSD_CUDA(cudaGetLastError());
  if (algo_bytes) {
    unsigned long long b = 0;
    TSD_CUDA(cudaMemcpyAsync(&b, d->view.ctr, sizeof(b), cudaMemcpyDeviceToHost, s));
    TSD_CUDA(cudaStreamSynchronize(s));
    if (kernel == 0) {
      // per launch, plus the dense unigram and root rows every launch reads once
      const int64_t shared = (int64_t)d->cfg.V * ((d->lm ? 4 : 0) + (d->boost ? 4 : 0));
      *algo_bytes = (int64_t)(b / (unsigned long long)reps) + shared;
    } else if (d->view.fused && !d->view.fz_dense) {
      // joint, streaming epilogue: the operands once (A rows, W_out), the
      // logits written and the softmax partials
      *algo_bytes = (int64_t)M * d->cfg.H * 2 + (int64_t)d->N * d->cfg.H * 2 + (int64_t)M * d->N * 4 +
                    (int64_t)M * d->n_ptiles * 8;
    } else if (d->view.fused) {
      // joint, dense epilogue: the operands once (A rows, W_out), each row's
      // dense LM row and mask, the defaults, the partials written (the
      // listed labels' logits are not counted)
      *algo_bytes = (int64_t)M * d->cfg.H * 2 + (int64_t)d->N * d->cfg.H * 2 + (int64_t)M * d->V4 * 4 +
                    (int64_t)M * d->view.mask_words * 4 + (int64_t)d->N_pad * 4 + (int64_t)M * d->n_ptiles * 16;
    } else {
      // joint: the operands once (A rows, W_out) and the bias rows read by the epilogue
      *algo_bytes = (int64_t)M * d->cfg.H * 2 + (int64_t)d->N * d->cfg.H * 2 + (int64_t)M * d->N * 4 +
                    (int64_t)M * d->n_ptiles * 16;
    }
  }
  return TSD_OK;
}

extern "C" tsd_status tsd_decoder_check(tsd_decoder* d) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_decoder_check: NULL decoder");
  tsd_status st = set_device(d);
  if (st) return st;
  TSD_CUDA(cudaStreamSynchronize(d->last_stream));
  int32_t e = 0;
  TSD_CUDA(cudaMemcpy(&e, d->view.err, sizeof(e), cudaMemcpyDeviceToHost));
  if (e) {
    TSD_CUDA(cudaMemset(d->view.err, 0, sizeof(e)));
    return fail(TSD_EDEVICE, "tsd_decoder_check: device status 0x%x (%s)", e,
                e >= 0x100 ? "a range check of the checked build failed" : "a bounded device wait expired");
  }
  return TSD_OK;
}

extern "C" tsd_status tsd_decoder_debug_capture(tsd_decoder* d, float* logits, int32_t* rows,
                                                int32_t max_steps) {
  clear_error();
  if (!d) return fail(TSD_EINVAL, "tsd_decoder_debug_capture: NULL decoder");
  if ((logits || rows) && max_steps < 1) return fail(TSD_EINVAL, "tsd_decoder_debug_capture: max_steps < 1");
  d->view.cap_logits = logits;
  d->view.cap_rows = rows;
  d->view.cap_steps = (logits || rows) ? max_steps : 0;
  return drop_graphs(d);  // captured graphs bake the view in
}
