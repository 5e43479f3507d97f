"""Pins of the oracle's stateful Transducer form (prediction network +
joint projections) against what its definition fixes."""
from __future__ import annotations

import math

import numpy as np

import oracle
import synth


def _bf16(x):
    """float32 -> bf16 bit patterns, round to nearest even."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    keep = u >> 16
    rest = u & 0xFFFF
    keep = keep + ((rest > 0x8000) | ((rest == 0x8000) & (keep & 1 == 1)))
    return keep.astype(np.uint16)


def _setup(V=24, H=64, D=8, Henc=64, T=12):
    w = synth.scaled(synth.WORKLOADS[0], V=V, H=H, B=1, T=T)
    p = synth.pred_weights(w, D=D, Henc=Henc)
    E, W = synth.joint_weights(w)
    lm = oracle.LM.from_arrays(synth.ngram_lm(51, V, 3, 400, 1.1))
    bo = oracle.Boost.from_phrases(V, synth.phrases(52, V, 5, 2, 3, 0.0), 1.0)
    return w, p, E, W, lm, bo


def test_identity_projection_and_silent_predictor_is_the_stateless_form():
    """W_enc = I, b_enc = 0, W_pred = 0, b_pred = 0: the joint input is
    bf16(ReLU(enc)), the stateless form with a zero embedding table."""
    w, p, E, W, lm, bo = _setup()
    p.We = _bf16(np.eye(w.H, dtype=np.float32))
    p.be = np.zeros(w.H, dtype=np.float32)
    p.Wp = np.zeros_like(p.Wp)
    p.bp = np.zeros(w.H, dtype=np.float32)
    enc = synth.enc_chunk(w, [0], 0)[0]
    a = oracle.decode_chunk(oracle.Stream(w.V), oracle.Model(w.V, w.H, np.zeros_like(E), W), lm, bo, enc,
                            0.5, 1.0, 4)
    b = oracle.decode_chunk(oracle.Stream(w.V), oracle.Model(w.V, w.H, E, W), lm, bo, enc, 0.5, 1.0, 4,
                            pred=oracle.PredNet(w.V, w.H, p))
    for x, y in zip(a[:3], b[:3]):
        assert np.array_equal(x, y)


def test_constant_gates_follow_the_closed_form_recurrence():
    """With W_g = 0 the gates are the biases: after the start-of-sequence
    step and n emissions, c = s(i) tanh(g) (1 - s(f)^(n+1)) / (1 - s(f)) and
    h = bf16(s(o) tanh(c)) in every unit."""
    w, p, E, W, lm, bo = _setup(D=6)
    p.Wg = np.zeros_like(p.Wg)
    rng = np.random.default_rng(3)
    p.bg = rng.normal(0, 1, 4 * p.D).astype(np.float32)
    st = oracle.Stream(w.V)
    toks, _, _, _ = oracle.decode_chunk(st, oracle.Model(w.V, w.H, E, W), lm, bo, synth.enc_chunk(w, [0], 0)[0],
                                        0.5, 1.0, 4, pred=oracle.PredNet(w.V, w.H, p))
    n = len(toks)
    assert n > 3
    h, c = st.pred_state(p.D)
    sg = lambda x: 1.0 / (1.0 + math.exp(-x))
    for u in range(p.D):
        i, f, g, o = sg(p.bg[4 * u]), sg(p.bg[4 * u + 1]), math.tanh(p.bg[4 * u + 2]), sg(p.bg[4 * u + 3])
        want_c = i * g * (1 - f ** (n + 1)) / (1 - f)
        assert abs(c[u] - want_c) < 1e-12 * max(1.0, abs(want_c)) + 1e-12
        assert h[u] == _bf16(np.float32(o * math.tanh(want_c)))


def test_blank_does_not_advance_the_predictor():
    """A joint whose blank logit always wins emits nothing; the predictor
    then holds exactly its start-of-sequence state (one step on blank from
    zero state)."""
    w, p, E, W, lm, bo = _setup(D=5)
    W = W.copy()
    W[:, w.V] = _bf16(np.full(w.H, 60.0 / w.H, dtype=np.float32))  # blank column: a large logit
    st = oracle.Stream(w.V)
    toks, _, _, _ = oracle.decode_chunk(st, oracle.Model(w.V, w.H, E, W), None, None, synth.enc_chunk(w, [0], 0)[0],
                                        0.0, 0.0, 4, pred=oracle.PredNet(w.V, w.H, p))
    assert len(toks) == 0
    ref = oracle.Stream(w.V)
    # a one-frame chunk from a fresh stream: the same start-of-sequence state
    oracle.decode_chunk(ref, oracle.Model(w.V, w.H, E, W), None, None, synth.enc_chunk(w, [0], 0)[0][:1], 0.0, 0.0,
                        4, pred=oracle.PredNet(w.V, w.H, p))
    h1, c1 = st.pred_state(p.D)
    h2, c2 = ref.pred_state(p.D)
    assert np.array_equal(h1, h2) and np.array_equal(c1, c2)
    # and it is the LSTM step on the blank embedding from zeros
    sg = lambda x: 1.0 / (1.0 + np.exp(-x))
    x = (p.Ep[w.V].astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    Wg = (p.Wg.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    gates = p.bg.astype(np.float64) + x @ Wg[: p.D]
    cc = sg(gates[1::4]) * 0 + sg(gates[0::4]) * np.tanh(gates[2::4])
    assert np.allclose(c1, cc, rtol=0, atol=1e-12)
