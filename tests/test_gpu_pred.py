"""The stateful Transducer form on the GPU (LSTM prediction network and joint
projections on tcgen05 GEMMs) against the oracle."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu


def _decoder(w, p, lmA, ph, E, W, **kw):
    import torch

    import paper_2609_14991_gb300 as tsd

    dev = torch.device("cuda", 0)
    lm = tsd.NGram.from_arrays(lmA) if lmA is not None else None
    bo = tsd.Boost.from_phrases(w.V, ph, w.bonus) if ph is not None else None
    dec = tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev),
                      lm=lm, boost=bo, max_symbols=w.max_sym, max_streams=w.B, max_T=w.T, pred=p, **kw)
    return dec, lm, bo


def _f32(h):
    return (h.astype(np.uint32) << 16).view(np.float32)


def _chunk(dec, w, enc):
    import torch

    out = dec.decode_chunk(dec._slots, torch.from_numpy(enc.view(np.int16)).to(torch.device("cuda", 0)), w.lam, w.beta)
    torch.cuda.synchronize()
    t, f, s, n = (x.cpu().numpy() for x in (out.tokens, out.frames, out.scores, out.counts))
    return [(t[i, :n[i]], f[i, :n[i]], s[i, :n[i]]) for i in range(len(n))]


@pytest.mark.parametrize("V,H,D,Henc", [(256, 256, 128, 192), (1024, 512, 256, 512)])
def test_stateful_form_matches_oracle(V, H, D, Henc):
    """Follow mode over two chunks.  The prediction network's h is bf16 on
    both sides, rounded from gate sums taken in fp32 (GPU) and fp64 (oracle),
    so logits and fused scores are held to the GEMM tolerance (2e-2) and LM
    and trie states stay bit-exact.  h feeds back through W_g: a one-step
    rounding flip in one unit moves every gate of the next step by ~1e-4,
    which flips a few per cent of the next h roundings; the forget gates
    (< 1) keep that drift bounded, so after ~60 LSTM steps h and c are held
    to 1e-2 (absolute: near zero one drift is many bf16 steps) with under 15%
    of the h units differing."""
    w = synth.scaled(synth.WORKLOADS[0], V=V, H=H, B=5, T=16, n_phr=20, phr_len=(2, 5))
    p = synth.pred_weights(w, D=D, Henc=Henc)
    lmA = synth.ngram_lm(w.lm_seed, V, 3, 6000, w.zipf)
    ph = synth.phrases(w.boost_seed, V, w.n_phr, 2, 5, 0.2)
    E, W = synth.joint_weights(w)
    dec, lm, bo = _decoder(w, p, lmA, ph, E, W)
    dec._slots = [dec.open() for _ in range(w.B)]
    olm, obo = oracle.LM.from_arrays(lmA), oracle.Boost.from_phrases(V, ph, w.bonus)
    model, pn = oracle.Model(V, H, E, W), oracle.PredNet(V, H, p)
    streams = [oracle.Stream(V) for _ in range(w.B)]
    emitted = 0
    for c in range(2):
        enc = synth.enc_chunk_wide(w, range(w.B), c, Henc)
        got = _chunk(dec, w, enc)
        for i in range(w.B):
            tok, fr, sc = got[i]
            emitted += len(tok)
            _, _, _, rep = oracle.decode_chunk(streams[i], model, olm, obo, enc[i], w.lam, w.beta, w.max_sym,
                                               follow=(tok, fr, sc), gap_tol=pu.LOGIT_TOL, pred=pn)
            assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, (c, i, rep)
            assert rep[oracle.REP_MAX_SCORE_DIFF] <= pu.LOGIT_TOL, (c, i, rep)
            hist = streams[i].history()
            lm_state, trie_node, last = dec.state(dec._slots[i])
            assert lm.state_tuple(lm_state) == olm.state(hist)
            assert bo.node_tuple(trie_node) == pu.trie_tuple(obo, hist, streams[i].rho())
            hg, cg = dec.pred_state(dec._slots[i])
            ho, co = streams[i].pred_state(D)
            dh = np.abs(_f32(hg) - _f32(ho))
            assert dh.max() <= 1e-2 and (dh > 0).mean() < 0.15, (c, i, dh.max(), (dh > 0).mean())
            assert np.abs(cg - co).max() <= 1e-2, (c, i, np.abs(cg - co).max())
    assert emitted > w.B * w.T


def test_first_lstm_steps_round_like_the_oracle():
    """One frame, one label at most, from fresh streams: the start-of-sequence
    step (blank embedding, zero state) and at most one emission step.  With
    no drift to compound, h rounds as the oracle's does except where the fp32
    gate sum lands within ~1e-6 of a bf16 rounding boundary."""
    V, H, D = 512, 256, 256
    w = synth.scaled(synth.WORKLOADS[0], V=V, H=H, B=16, T=1, max_sym=1)
    p = synth.pred_weights(w, D=D, Henc=H)
    E, W = synth.joint_weights(w)
    dec, _, _ = _decoder(w, p, None, None, E, W)
    dec._slots = [dec.open() for _ in range(w.B)]
    model, pn = oracle.Model(V, H, E, W), oracle.PredNet(V, H, p)
    enc = synth.enc_chunk_wide(w, range(w.B), 0, H)
    got = _chunk(dec, w, enc)
    flips = 0
    for i in range(w.B):
        st = oracle.Stream(V)
        _, _, _, rep = oracle.decode_chunk(st, model, None, None, enc[i], 0.0, 0.0, 1, follow=got[i],
                                           gap_tol=pu.LOGIT_TOL, pred=pn)
        assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, (i, rep)
        hg, cg = dec.pred_state(dec._slots[i])
        ho, co = st.pred_state(D)
        steps = np.abs(hg.astype(np.int32) - ho.astype(np.int32))
        assert steps.max() <= 1, (i, steps.max())
        flips += int((steps > 0).sum())
        assert np.allclose(cg, co, rtol=1e-5, atol=1e-5), (i, np.abs(cg - co).max())
    assert flips <= w.B * D // 100, flips


def test_identity_projection_silent_predictor_is_the_stateless_decoder():
    """W_enc = I, b_enc = 0, W_pred = 0, b_pred = 0: the projection GEMM and
    the joint-input epilogue reproduce bf16(ReLU(enc)), so the decode is bit
    for bit that of the stateless decoder with a zero embedding table."""
    import torch

    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[0], V=512, H=256, B=6, T=12)
    p = synth.pred_weights(w, D=64, Henc=w.H)
    p.We = np.eye(w.H, dtype=np.float32).view(np.uint32).__rshift__(16).astype(np.uint16)
    p.be = np.zeros(w.H, dtype=np.float32)
    p.Wp = np.zeros_like(p.Wp)
    p.bp = np.zeros(w.H, dtype=np.float32)
    lmA = synth.ngram_lm(w.lm_seed, w.V, 3, 8000, w.zipf)
    ph = synth.phrases(w.boost_seed, w.V, 20, 2, 4, 0.0)
    E, W = synth.joint_weights(w)
    dec, _, _ = _decoder(w, p, lmA, ph, E, W)
    dec._slots = [dec.open() for _ in range(w.B)]
    dev = torch.device("cuda", 0)
    plain = tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.zeros((w.N, w.H), dtype=torch.int16,
                        device=dev), lm=tsd.NGram.from_arrays(lmA), boost=tsd.Boost.from_phrases(w.V, ph, w.bonus),
                        max_symbols=w.max_sym, max_streams=w.B, max_T=w.T)
    plain._slots = [plain.open() for _ in range(w.B)]
    for c in range(2):
        enc = synth.enc_chunk(w, range(w.B), c)
        a, b = _chunk(dec, w, enc), _chunk(plain, w, enc)
        for x, y in zip(a, b):
            for u, v in zip(x, y):
                assert np.array_equal(u, v)


def test_stateful_form_rejections():
    import torch

    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[0], V=64, H=128, B=2, T=4)
    p = synth.pred_weights(w, D=64, Henc=128)
    E, W = synth.joint_weights(w)
    with pytest.raises(tsd.TsdError):
        _decoder(synth.scaled(w, max_sym=1), p, None, None, E, W, beam_k=2)
    with pytest.raises(tsd.TsdError):
        _decoder(w, p, None, None, E, W, prune_k=2)
    bad = synth.pred_weights(w, D=64, Henc=128)
    bad.D = 96  # not a multiple of 64
    with pytest.raises((tsd.TsdError, AssertionError, ValueError)):
        _decoder(w, bad, None, None, E, W)
    dec, _, _ = _decoder(w, p, None, None, E, W)
    s = dec.open()
    with pytest.raises(tsd.TsdError):
        dec.export_state(s)
