"""Pins of the oracle's beam search with several labels per frame (the
frame-synchronous search: per frame up to S expansions of the hypotheses
still in the frame, blank or an S-th label leaves the frame)."""
from __future__ import annotations

import itertools

import numpy as np

import oracle
import synth


def oracle_bf16(x):
    """float -> bf16 bit patterns, round to nearest even."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    keep, rest = u >> 16, u & 0xFFFF
    keep = keep + ((rest > 0x8000) | ((rest == 0x8000) & (keep & 1 == 1)))
    return keep.astype(np.uint16)


def _tiny(V, H, seed):
    E = synth.normal_bf16(seed, 2, 0, 0, (V + 1) * H, 1.0).reshape(V + 1, H)
    W = synth.normal_bf16(seed, 3, 0, 0, H * (V + 1), 3.0 / np.sqrt(H)).reshape(H, V + 1)
    return oracle.Model(V, H, E, W)


def _fused(model, lm, bo, enc_t, y, lam, beta):
    st = oracle.Stream(model.V)
    rho = int(bo.trajectory(y)[1][-1]) if (y and bo is not None) else 0
    st.set_history(y, rho)
    return oracle.fused_row(st, model, lm, bo, enc_t, lam, beta)


def test_k1_is_greedy_with_s_labels_per_frame():
    """One hypothesis: the best extension each expansion, blank or the S-th
    label ends the frame -- greedy decoding with max_symbols = S."""
    w = synth.scaled(synth.WORKLOADS[0], H=48, T=30)
    E, W = synth.joint_weights(w)
    lm = oracle.LM.from_arrays(synth.ngram_lm(4, w.V, 3, 3000, 1.1))
    bo = oracle.Boost.from_phrases(w.V, synth.phrases(4, w.V, 8, 2, 4, 0.0), 1.0)
    enc = synth.enc_chunk(w, [2], 0)[0]
    W2 = W.copy()
    W2[:, w.V] = oracle_bf16(np.full(w.H, 2.0 / np.sqrt(w.H)))  # a stronger blank: some frames end early
    blanks = 0
    for Wx in (W, W2):
        model = oracle.Model(w.V, w.H, E, Wx)
        for S in (2, 3, 5):
            g = oracle.Stream(w.V)
            tok, fr, _, _ = oracle.decode_chunk(g, model, lm, bo, enc, 0.4, 1.0, S)
            b = oracle.Stream(w.V)
            oracle.beam_chunk(b, model, lm, bo, enc, 0.4, 1.0, 1, S)
            hyps = b.beam_hyps()
            assert len(hyps) == 1 and hyps[0][0] == tok.tolist(), S
            # the greedy path's score, blanks included: labels of frame t, then
            # the blank if fewer than S were emitted
            y, score = [], 0.0
            for t in range(w.T):
                for v in tok[fr == t]:
                    score += _fused(model, lm, bo, enc[t], y, 0.4, 1.0)[v]
                    y.append(int(v))
                if np.sum(fr == t) < S:
                    score += _fused(model, lm, bo, enc[t], y, 0.4, 1.0)[w.V]
                    blanks += 1
            assert abs(hyps[0][1] - score) < 1e-9, (S, hyps[0][1], score)
    assert blanks > 10


def test_wide_beam_sums_every_alignment():
    """K large enough to keep everything: each surviving label sequence
    scores the log-sum-exp over all its alignments, enumerated by brute force
    (per frame 0..S labels; fewer than S then a blank, exactly S then the
    next frame without a blank)."""
    V, H, T, S = 2, 16, 2, 2
    model = _tiny(V, H, 9)
    lm = oracle.LM.from_arrays(synth.ngram_lm(9, V, 2, 5, 1.1))
    bo = oracle.Boost(V, np.array([0, 2]), np.array([1, 0]), 1.0)
    enc = synth.normal_bf16(9, 1, 0, 0, T * H, 1.0).reshape(T, H)
    lam, beta = 0.5, 0.75
    b = oracle.Stream(V)
    oracle.beam_chunk(b, model, lm, bo, enc, lam, beta, 64, S)
    got = {tuple(y): s for y, s in b.beam_hyps()}
    want = {}

    def frames(t, y, score):
        if t == T:
            k = tuple(y)
            want[k] = np.logaddexp(want[k], score) if k in want else score
            return
        for n in range(S + 1):  # labels emitted in frame t
            for labels in itertools.product(range(V), repeat=n):
                yy, sc = list(y), score
                for v in labels:
                    sc += _fused(model, lm, bo, enc[t], yy, lam, beta)[v]
                    yy.append(v)
                if n < S:
                    sc += _fused(model, lm, bo, enc[t], yy, lam, beta)[V]
                frames(t + 1, yy, sc)

    frames(0, [], 0.0)
    assert set(got) == set(want)
    for k in want:
        assert abs(got[k] - want[k]) < 1e-9, k


def _driver(model, lm, bo, enc, lam, beta, K, S):
    """The search written out directly over fused rows: kept candidates per
    expansion and the final beam."""
    V = model.V
    beam = [([], 0.0)]
    sels = []
    for t in range(enc.shape[0]):
        A, F = beam, []
        for e in range(S):
            if not A:
                break
            cands = []
            for i, (y, sc) in enumerate(A):
                f = _fused(model, lm, bo, enc[t], y, lam, beta)
                cands += [(sc + f[v], i, v) for v in range(V + 1)]
            cands.sort(key=lambda c: (-c[0], c[1], c[2]))
            kept = cands[:K]
            sels.append(kept)
            A2 = []
            for sc, i, v in kept:
                y2 = A[i][0] + ([v] if v != V else [])
                dst = F if (v == V or e == S - 1) else A2
                for j, (yy, ss) in enumerate(dst):
                    if yy == y2:
                        dst[j] = (yy, float(np.logaddexp(ss, sc)))
                        break
                else:
                    dst.append((y2, sc))
            if len(F) > K:
                order = sorted(range(len(F)), key=lambda j: (-F[j][1], j))[:K]
                F = [F[j] for j in sorted(order)]
            A = A2
        beam = F
    return sels, beam


def test_free_running_and_follow_mode_agree_with_the_direct_search():
    V, H, T, K, S = 5, 16, 4, 3, 3
    model = _tiny(V, H, 13)
    lm = oracle.LM.from_arrays(synth.ngram_lm(13, V, 3, 40, 1.1))
    bo = oracle.Boost(V, np.array([0, 2, 3]), np.array([1, 2, 4]), 1.0)
    enc = synth.normal_bf16(13, 1, 0, 0, T * H, 1.0).reshape(T, H)
    sels, beam = _driver(model, lm, bo, enc, 0.4, 0.8, K, S)
    assert len(sels) > T  # some frames took more than one expansion
    free = oracle.Stream(V)
    oracle.beam_chunk(free, model, lm, bo, enc, 0.4, 0.8, K, S)
    got = free.beam_hyps()
    assert [h[0] for h in got] == [h[0] for h in beam]
    for (ya, sa), (yb, sb) in zip(got, beam):
        assert abs(sa - sb) < 1e-9
    n = T * S
    sh = np.full((n, K), -1, np.int32)
    stok = np.full((n, K), -1, np.int32)
    for s, kept in enumerate(sels):
        for i, (_, h, v) in enumerate(kept):
            sh[s, i], stok[s, i] = h, v
    sinc = np.zeros((n, K), np.float32)
    fol = oracle.Stream(V)
    rep = oracle.beam_chunk_follow(fol, model, lm, bo, enc, 0.4, 0.8, K, sh, stok, sinc, S=S)
    assert rep[oracle.REP_MISMATCH] == 0 and rep[oracle.REP_INCONSISTENT] == 0
    assert int(rep[oracle.REP_STEPS]) == len(sels)
    assert [h[0] for h in fol.beam_hyps()] == [h[0] for h in got]
    # a step after the last frame that still keeps candidates is inconsistent
    extra = sh.copy()
    extra[len(sels):, 0] = 0
    if len(sels) < n:
        rep = oracle.beam_chunk_follow(oracle.Stream(V), model, lm, bo, enc, 0.4, 0.8, K, extra, stok, sinc, S=S)
        assert rep[oracle.REP_INCONSISTENT] == 1
    # dropping the best candidate of the first expansion is flagged
    bad = stok.copy()
    f0 = _fused(model, lm, bo, enc[0], [], 0.4, 0.8)
    bad[0, 0] = int(np.argmin(f0))
    rep = oracle.beam_chunk_follow(oracle.Stream(V), model, lm, bo, enc, 0.4, 0.8, K, sh, bad, sinc, S=S)
    assert rep[oracle.REP_MISMATCH] >= 1
