"""Pins of the oracle's several-LM fusion (Eq. 1, term 2 as a weighted sum
over LMs) and of its ARPA reader, against what the definitions fix."""
from __future__ import annotations

import math

import numpy as np
import pytest

import oracle
import synth
from tests.arpa_util import write_arpa


def _setup(T=12):
    w = synth.scaled(synth.WORKLOADS[0], V=40, H=64, B=1, T=T, lm_total=900, n_phr=6, phr_len=(2, 4))
    a = synth.ngram_lm(11, w.V, 3, 900, 1.1)
    b = synth.ngram_lm(12, w.V, 2, 400, 1.05)
    ph = synth.phrases(13, w.V, 6, 2, 4, 0.0)
    E, W = synth.joint_weights(w)
    model = oracle.Model(w.V, w.H, E, W)
    enc = synth.enc_chunk(w, [0], 0)[0]
    return w, oracle.LM.from_arrays(a), oracle.LM.from_arrays(b), oracle.Boost.from_phrases(w.V, ph, 1.0), model, enc


def test_zero_weight_lm_changes_nothing():
    """A second LM with weight 0 reduces to the single-LM decode exactly."""
    w, A, B, bo, model, enc = _setup()
    s1, s2 = oracle.Stream(w.V), oracle.Stream(w.V)
    t1, f1, sc1, _ = oracle.decode_chunk(s1, model, A, bo, enc, 0.4, 1.0, 3)
    t2, f2, sc2, _ = oracle.decode_chunk(s2, model, [(A, 1.0), (B, 0.0)], bo, enc, 0.4, 1.0, 3)
    assert np.array_equal(t1, t2) and np.array_equal(f1, f2)
    assert np.array_equal(sc1, sc2)


def test_same_lm_twice_is_the_summed_weight():
    """One LM listed twice with weights w1, w2 scores as that LM with w1 + w2."""
    w, A, B, bo, model, enc = _setup()
    s1, s2 = oracle.Stream(w.V), oracle.Stream(w.V)
    t1, _, sc1, _ = oracle.decode_chunk(s1, model, [(A, 0.25), (A, 0.5)], bo, enc, 0.8, 1.0, 3)
    t2, _, sc2, _ = oracle.decode_chunk(s2, model, A, bo, enc, 0.8 * 0.75, 1.0, 3)
    assert np.array_equal(t1, t2)
    assert np.allclose(sc1, sc2, rtol=0, atol=1e-12)


def test_fused_score_is_the_weighted_sum_of_the_terms():
    """Every emitted label's fused score equals log p_AM + lam * sum_i w_i *
    log p_LM_i + beta * boost, each term computed on its own (joint logits
    by the oracle's matmul, log-softmax here, LM and boost scores from the
    oracle's dictionary and suffix matcher)."""
    w, A, B, bo, model, enc = _setup(T=10)
    lam, wa, wb, beta = 0.7, 0.6, 0.3, 1.2
    st = oracle.Stream(w.V)
    toks, frames, scores, _ = oracle.decode_chunk(st, model, [(A, wa), (B, wb)], bo, enc, lam, beta, 3)
    assert len(toks) > 5
    hist = []
    rho = 0
    for y, t, sc in zip(toks, frames, scores):
        last = hist[-1] if hist else w.V
        lg = model.joint_logits(enc[t], last)
        lse = np.max(lg) + np.log(np.sum(np.exp(lg - np.max(lg))))
        expect = (lg[y] - lse) + lam * (wa * A.score(hist, y) + wb * B.score(hist, y)) + beta * bo.score(hist[rho:], y)
        assert sc == pytest.approx(expect, abs=1e-9)
        hist.append(int(y))
        _, restart = bo.trajectory(hist)
        rho = int(restart[-1])


def _arrays(seed=21, V=30, order=3, total=600):
    return synth.ngram_lm(seed, V, order, total, 1.1)


def test_arpa_round_trip_numeric_ids():
    a = _arrays()
    r = oracle.read_arpa(write_arpa(a), a.V)
    assert r.order == a.order and r.skipped == 0
    for k in range(a.order):
        assert np.array_equal(r.tokens[k], a.tokens[k])
        assert np.allclose(r.logp[k], a.logp[k], rtol=1e-6, atol=1e-6)
        assert np.allclose(r.bow[k], a.bow[k], rtol=1e-6, atol=1e-6)


def test_arpa_vocab_and_sentence_markers_skipped():
    a = _arrays(V=12, order=2, total=80)
    vocab = ["w%d" % i for i in range(a.V)]
    extra = {1: [(-1.5, "</s>", None), (-99.0, "<s>", -0.2)], 2: [(-0.7, "<s> w3", None), (-0.4, "w5 </s>", None)]}
    r = oracle.read_arpa(write_arpa(a, vocab=vocab, extra=extra), a.V, vocab=vocab)
    assert r.skipped == 4
    for k in range(a.order):
        assert np.array_equal(r.tokens[k], a.tokens[k])
    lm_a, lm_r = oracle.LM.from_arrays(a), oracle.LM(r.V, r.tokens, r.logp, r.bow)
    for h in ([], [3], [5, 7], [1, 2]):
        for v in range(a.V):
            assert lm_r.score(h, v) == pytest.approx(lm_a.score(h, v), abs=1e-5)


def test_arpa_is_log10():
    """A one-word LM with p = 1/10 in the file scores ln(1/10)."""
    text = "\\data\\\nngram 1=1\n\n\\1-grams:\n-1\t0\n\n\\end\\\n"
    r = oracle.read_arpa(text, 1)
    assert r.logp[0][0] == pytest.approx(math.log(0.1), rel=1e-7)


def test_arpa_count_mismatch_rejected():
    text = "\\data\\\nngram 1=2\n\n\\1-grams:\n-1\t0\n\n\\end\\\n"
    with pytest.raises(ValueError):
        oracle.read_arpa(text, 1)
