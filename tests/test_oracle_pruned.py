"""Pins of the oracle's pruned fusion (fusion re-ranks only the acoustic
model's k best outputs), against what its definition fixes."""
from __future__ import annotations

import numpy as np

import oracle
import synth


def _setup(T=14, V=48):
    w = synth.scaled(synth.WORKLOADS[0], V=V, H=64, B=1, T=T)
    lm = oracle.LM.from_arrays(synth.ngram_lm(41, V, 3, 1200, 1.1))
    bo = oracle.Boost.from_phrases(V, synth.phrases(42, V, 8, 2, 4, 0.0), 1.0)
    E, W = synth.joint_weights(w)
    return w, lm, bo, oracle.Model(V, w.H, E, W), synth.enc_chunk(w, [0], 0)[0]


def test_k_covering_every_output_is_full_fusion():
    w, lm, bo, model, enc = _setup()
    a = oracle.decode_chunk(oracle.Stream(w.V), model, lm, bo, enc, 0.6, 1.5, 4)
    b = oracle.decode_chunk(oracle.Stream(w.V), model, lm, bo, enc, 0.6, 1.5, 4, prune_k=w.V + 1)
    for x, y in zip(a[:3], b[:3]):
        assert np.array_equal(x, y)


def test_k_one_is_acoustic_greedy():
    """With one candidate fusion cannot change a decision: the labels are
    those of plain greedy decoding on the logits (lambda = beta = 0)."""
    w, lm, bo, model, enc = _setup()
    a = oracle.decode_chunk(oracle.Stream(w.V), model, lm, bo, enc, 0.0, 0.0, 4)
    b = oracle.decode_chunk(oracle.Stream(w.V), model, lm, bo, enc, 0.9, 2.0, 4, prune_k=1)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_decisions_are_best_fused_among_acoustic_top_k():
    w, lm, bo, model, enc = _setup(T=20)
    k, lam, beta = 4, 0.8, 1.5
    toks, frames, scores, _ = oracle.decode_chunk(oracle.Stream(w.V), model, lm, bo, enc, lam, beta, 4, prune_k=k)
    assert len(toks) > 5
    hist, rho = [], 0
    for y, t, sc in zip(toks, frames, scores):
        lg = model.joint_logits(enc[t], hist[-1] if hist else w.V)
        order = sorted(range(w.V + 1), key=lambda v: (-lg[v], v))
        top = order[:k]
        assert y in top
        lse = np.max(lg) + np.log(np.sum(np.exp(lg - np.max(lg))))
        fused = {c: (lg[c] - lse) + (lam * lm.score(hist, c) + beta * bo.score(hist[rho:], c) if c != w.V else 0.0)
                 for c in top}
        best = max(top, key=lambda c: (fused[c], -c))
        assert y == best and abs(sc - fused[y]) < 1e-9
        hist.append(int(y))
        rho = int(bo.trajectory(hist)[1][-1])


def test_follow_accepts_a_label_at_the_edge_of_the_set():
    """In follow mode a label whose logit is within am_tol of the k-th best
    is not a mismatch, one far outside is."""
    w, lm, bo, model, enc = _setup(T=1)
    lg = model.joint_logits(enc[0], w.V)
    order = sorted(range(w.V + 1), key=lambda v: (-lg[v], v))
    k = 3
    outside = order[k]  # the (k+1)-th output
    gap = lg[order[k - 1]] - lg[outside]
    for tol, want_bad in ((gap + 1e-6, 0), (gap / 2 if gap > 0 else -1.0, 1)):
        if outside == w.V:
            return  # blank needs no follow entry; nothing to test here
        rep = oracle.decode_chunk(oracle.Stream(w.V), model, lm, bo, enc, 0.0, 0.0, 1,
                                  follow=([outside], [0], [0.0]), prune_k=k, am_tol=tol, gap_tol=1e9)[3]
        assert (rep[oracle.REP_MISMATCH] > 0) == bool(want_bad), (tol, rep)
