"""Pins of the oracle to facts outside itself.

Each test checks the oracle against something the paper or the mathematics
fixes -- a hand-worked example, a closed form, a textbook special case, a
library routine on the same rounded inputs, or brute force on tiny inputs --
so that a dropped term, a wrong sign or index or a transposed operand in the
oracle fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _bf16_round_torch(x: np.ndarray) -> np.ndarray:
    """bf16 round-to-nearest-even by torch (a library routine), back to f32."""
    return torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).to(torch.float32).numpy()


def _tiny_model(V=11, H=24, seed=3):
    rng = np.random.default_rng(seed)
    E = synth.normal_bf16(seed, 2, 0, 0, (V + 1) * H, 1.0).reshape(V + 1, H)
    W = synth.normal_bf16(seed, 3, 0, 0, H * (V + 1), 3 / math.sqrt(H)).reshape(H, V + 1)
    return oracle.Model(V, H, E, W), rng


# ---------------------------------------------------------------------------
# joint logits and log-softmax (Eq. 1, first term)
# ---------------------------------------------------------------------------
def test_joint_input_rounding_matches_torch_bf16():
    """With W_out = identity the logits are the joint input itself:
    x = bf16_RNE(ReLU(f32(enc) + f32(E[last]))), checked against torch."""
    V, H = 15, 16
    E = synth.normal_bf16(1, 2, 0, 0, (V + 1) * H, 1.0).reshape(V + 1, H)
    I = np.zeros((H, V + 1), dtype=np.float32)
    I[np.arange(H), np.arange(H)] = 1.0
    W = (I.view(np.uint32) >> 16).astype(np.uint16)
    m = oracle.Model(V, H, E, W)
    for last in [V, 0, 7]:
        enc = synth.normal_bf16(9, 1, last, 0, H, 1.7)
        got = m.joint_logits(enc, last)[:H]
        s = synth.bf16_to_f32(enc) + synth.bf16_to_f32(E[last])
        want = _bf16_round_torch(np.maximum(s, 0))
        assert np.array_equal(got, want.astype(np.float64))


def test_joint_logits_match_float64_matmul():
    """logits = W_out^T x (W_out stored [H][V+1]); a transposed operand or a
    wrong embedding row fails this."""
    m, _ = _tiny_model()
    Wf = synth.bf16_to_f32(m.W).astype(np.float64)
    for last in [m.V, 2, 5]:
        enc = synth.normal_bf16(4, 1, last, 0, m.H, 1.0)
        x = _bf16_round_torch(np.maximum(synth.bf16_to_f32(enc) + synth.bf16_to_f32(m.E[last]), 0))
        want = x.astype(np.float64) @ Wf
        np.testing.assert_allclose(m.joint_logits(enc, last), want, rtol=0, atol=1e-12)


def test_log_softmax_sums_to_one_and_fusion_terms():
    """With lambda = beta = 0 the fused row is a log-softmax: sum exp = 1.
    With weights, every non-blank entry moves by exactly lambda*LM + beta*boost
    and the blank entry does not move (blank is not an LM token)."""
    m, _ = _tiny_model()
    lmA = synth.ngram_lm(2, m.V, 3, 200, 1.1)
    lm = oracle.LM.from_arrays(lmA)
    ph = synth.phrases(3, m.V, 4, 2, 3, 0.0)
    bo = oracle.Boost.from_phrases(m.V, ph, 1.0)
    st = oracle.Stream(m.V)
    st.set_history([1, 4, 2], 1)
    enc = synth.normal_bf16(5, 1, 0, 0, m.H, 1.0)
    f0 = oracle.fused_row(st, m, lm, bo, enc, 0.0, 0.0)
    assert abs(np.exp(f0).sum() - 1.0) < 1e-12
    lam, beta = 0.7, 1.3
    f = oracle.fused_row(st, m, lm, bo, enc, lam, beta)
    assert f[m.V] == f0[m.V]
    for v in range(m.V):
        want = f0[v] + lam * lm.score([1, 4, 2], v) + beta * bo.score([4, 2], v)
        assert abs(f[v] - want) < 1e-12


def _plain_greedy(model, enc, max_sym, last):
    """Textbook greedy Transducer decoding on raw joint logits (numpy/torch
    only): at each frame emit argmax labels until blank or max_sym."""
    Ef = synth.bf16_to_f32(model.E)
    Wf = synth.bf16_to_f32(model.W).astype(np.float64)
    out = []
    for t in range(enc.shape[0]):
        for _ in range(max_sym):
            x = _bf16_round_torch(np.maximum(synth.bf16_to_f32(enc[t]) + Ef[last], 0))
            y = int(np.argmax(x.astype(np.float64) @ Wf))
            if y == model.V:
                break
            out.append((y, t))
            last = y
    return out


def test_zero_weights_reduce_to_plain_greedy():
    """lambda = beta = 0: the fused decoder is plain greedy Transducer
    decoding (the argmax of the log-softmax is the argmax of the logits)."""
    w = synth.scaled(synth.WORKLOADS[0], H=64, T=30)
    E, W = synth.joint_weights(w)
    model = oracle.Model(w.V, w.H, E, W)
    lm = oracle.LM.from_arrays(synth.ngram_lm(9, w.V, 3, 3000, 1.1))
    bo = oracle.Boost.from_phrases(w.V, synth.phrases(9, w.V, 8, 2, 4, 0.0), 1.0)
    for s in range(2):
        enc = synth.enc_chunk(w, [s], 0)[0]
        st = oracle.Stream(w.V)
        tok, fr, _, rep = oracle.decode_chunk(st, model, lm, bo, enc, 0.0, 0.0, 5)
        assert list(zip(tok.tolist(), fr.tolist())) == _plain_greedy(model, enc, 5, w.V)


# ---------------------------------------------------------------------------
# n-gram backoff (Eq. 1, second term)
# ---------------------------------------------------------------------------
def _golden_lm():
    g = _golden("lm_tiny.json")
    V, N = g["V"], g["order"]
    toks = [[] for _ in range(N)]
    lps = [[] for _ in range(N)]
    bws = [[] for _ in range(N)]
    for e in g["ngrams"]:
        k = len(e["tokens"])
        toks[k - 1].append(e["tokens"])
        lps[k - 1].append(math.log(e["p"]))
        bws[k - 1].append(math.log(e["bow"]))
    lm = oracle.LM(V, [np.array(t, dtype=np.int32).reshape(-1, k + 1) for k, t in enumerate(toks)],
                   [np.array(x, dtype=np.float32) for x in lps], [np.array(x, dtype=np.float32) for x in bws])
    return g, lm


def test_lm_hand_worked_backoff():
    g, lm = _golden_lm()
    for c in g["scores"]:
        assert abs(lm.score(c["hist"], c["v"]) - math.log(c["p"])) < 1e-6, c["why"]


def test_lm_hand_worked_states():
    g, lm = _golden_lm()
    for c in g["states"]:
        assert list(lm.state(c["hist"])) == c["state"]


def test_lm_normalized_for_every_context():
    """The synthetic LM is built normalized, so sum_v exp(score(v|c)) = 1 for
    every context c, including contexts that are not n-grams; a dropped
    backoff weight or a wrong suffix breaks this."""
    V = 40
    lmA = synth.ngram_lm(21, V, 4, 4000, 1.1)
    lm = oracle.LM.from_arrays(lmA)
    rng = np.random.default_rng(1)
    ctxs = [[]]
    for k in range(lmA.order):
        for i in rng.choice(len(lmA.logp[k]), size=min(25, len(lmA.logp[k])), replace=False):
            ctxs.append(lmA.tokens[k][i].tolist())
    for _ in range(25):
        ctxs.append(rng.integers(0, V, rng.integers(1, 6)).tolist())
    for c in ctxs:
        s = sum(math.exp(lm.score(c, v)) for v in range(V))
        assert abs(s - 1.0) < 1e-5, c


def _katz_from_counts(lmA):
    """Absolute-discount backoff computed directly from the raw counts (the
    textbook estimator), independent of the stored backoff weights:
      p(w|h) = (c(h,w) - D) / sum c(h,.)                     if c(h,w) > 0
             = D n(h) / sum c(h,.) * p(w|h[1:]) / sum_{w': c(h,w')=0} p(w'|h[1:])
      p(w|h) = p(w|h[1:])                       if h continues nothing
      p(w|()) = the stored unigram."""
    D = lmA.discount
    V = lmA.V
    cont = {}
    for k in range(1, lmA.order):
        for t, c in zip(lmA.tokens[k].tolist(), lmA.counts[k].tolist()):
            cont.setdefault(tuple(t[:-1]), {})[t[-1]] = c
    uni = np.exp(lmA.logp[0].astype(np.float64))
    memo = {}

    def p(w, h):
        key = (w, h)
        if key in memo:
            return memo[key]
        if len(h) == 0:
            r = uni[w]
        elif h not in cont:
            r = p(w, h[1:])
        else:
            cs = cont[h]
            S = sum(cs.values())
            if w in cs:
                r = (cs[w] - D) / S
            else:
                rest = sum(p(u, h[1:]) for u in range(V) if u not in cs)
                r = D * len(cs) / S * p(w, h[1:]) / rest
        memo[key] = r
        return r

    return p


def test_lm_matches_counts_exhaustively_order3():
    """For every history of up to 2 tokens (and some longer ones, which the
    model truncates) and every token, the oracle's table lookup equals the
    counts-level estimator."""
    V = 7
    lmA = synth.ngram_lm(17, V, 3, 80, 1.1)
    lm = oracle.LM.from_arrays(lmA)
    p = _katz_from_counts(lmA)
    hists = [()] + [tuple(h) for L in (1, 2) for h in itertools.product(range(V), repeat=L)]
    for h in hists:
        for w in range(V):
            assert abs(lm.score(list(h), w) - math.log(p(w, h))) < 1e-5, (h, w)
    for h in itertools.product(range(V), repeat=3):
        for w in range(0, V, 3):
            assert lm.score(list(h), w) == lm.score(list(h[1:]), w)


def test_lm_state_carries_all_of_the_score():
    """score(v | h) depends on h only through its state: replacing the history
    by the state tuple changes no score; and the state is an n-gram while no
    longer suffix (within order-1 tokens) is one."""
    V = 12
    lmA = synth.ngram_lm(23, V, 4, 1500, 1.1)
    lm = oracle.LM.from_arrays(lmA)
    grams = set()
    for t in lmA.tokens:
        grams |= set(map(tuple, t.tolist()))
    rng = np.random.default_rng(5)
    for _ in range(60):
        h = rng.integers(0, V, rng.integers(0, 8)).tolist()
        s = lm.state(h)
        assert s == () or s in grams
        for L in range(len(s) + 1, min(len(h), lmA.order - 1) + 1):
            assert tuple(h[-L:]) not in grams
        for v in range(V):
            assert lm.score(h, v) == lm.score(list(s), v)


# ---------------------------------------------------------------------------
# phrase boosting (Eq. 1, third term)
# ---------------------------------------------------------------------------
def test_boost_hand_worked():
    g = _golden("boost_tiny.json")
    off = np.cumsum([0] + [len(p) for p in g["phrases"]])
    bo = oracle.Boost(g["V"], off, np.concatenate(g["phrases"]), g["bonus"])
    for tr in g["trajectories"]:
        b, r = bo.trajectory(tr["labels"])
        assert b.tolist() == tr["bonus"], tr["why"]
        assert r.tolist() == tr["rho"], tr["why"]
    for c in g["candidates"]:
        assert bo.score(c["g"], c["v"]) == c["bonus"]


def _automaton_bonus(phrases, seq, bonus):
    """An independent formulation: track only the currently matched phrase
    prefix; on a label take the longest suffix of (prefix + label) that is a
    phrase prefix, earn the change in its length, and bank + restart when it
    is a whole phrase.  Returns per-label bonuses and the completed length."""
    P = {tuple(p[:i]) for p in phrases for i in range(1, len(p) + 1)}
    F = {tuple(p) for p in phrases}
    cur, out, banked = (), [], 0
    for v in seq:
        s = cur + (v,)
        nxt = ()
        for i in range(len(s)):
            if s[i:] in P:
                nxt = s[i:]
                break
        out.append(bonus * (len(nxt) - len(cur)))
        if nxt in F:
            banked += len(nxt)
            nxt = ()
        cur = nxt
    return out, banked, len(cur)


def test_boost_brute_force_all_short_sequences():
    """Every label sequence of length <= 6 over V = 4 with several phrase
    sets: the oracle's per-label bonuses equal the prefix-tracking automaton,
    and they telescope to bonus * (completed lengths + current match)."""
    V = 4
    sets = [[[0, 1], [1, 2, 3]], [[0, 0, 1], [0, 1, 0]], [[2], [3, 3, 3]], [[1, 2], [2, 1], [0, 1, 2, 3]]]
    for ph in sets:
        off = np.cumsum([0] + [len(p) for p in ph])
        bo = oracle.Boost(V, off, np.concatenate(ph), 1.5)
        for L in range(1, 7):
            for seq in itertools.product(range(V), repeat=L):
                b, _ = bo.trajectory(list(seq))
                want, banked, part = _automaton_bonus(ph, seq, 1.5)
                assert b.tolist() == want, (ph, seq)
                assert abs(sum(b) - 1.5 * (banked + part)) < 1e-12


# ---------------------------------------------------------------------------
# beam search
# ---------------------------------------------------------------------------
def test_beam_k1_equals_greedy_one_symbol():
    """K = 1 keeps only the best extension each frame: the greedy decoder with
    at most one label per frame."""
    w = synth.scaled(synth.WORKLOADS[0], H=48, T=25)
    E, W = synth.joint_weights(w)
    model = oracle.Model(w.V, w.H, E, W)
    lm = oracle.LM.from_arrays(synth.ngram_lm(4, w.V, 3, 3000, 1.1))
    bo = oracle.Boost.from_phrases(w.V, synth.phrases(4, w.V, 8, 2, 4, 0.0), 1.0)
    enc = synth.enc_chunk(w, [1], 0)[0]
    g = oracle.Stream(w.V)
    tok, _, _, _ = oracle.decode_chunk(g, model, lm, bo, enc, 0.4, 1.0, 1)
    b = oracle.Stream(w.V)
    oracle.beam_chunk(b, model, lm, bo, enc, 0.4, 1.0, 1)
    hyps = b.beam_hyps()
    assert len(hyps) == 1 and hyps[0][0] == tok.tolist()


def test_beam_sums_alignments_exhaustively():
    """V = 2, T = 3 and K large enough to keep every candidate: each surviving
    label sequence scores the log-sum-exp over all its alignments (one label
    or blank per frame), enumerated by brute force."""
    V, H, T = 2, 16, 3
    model, _ = _tiny_model(V=V, H=H, seed=8)
    lm = oracle.LM.from_arrays(synth.ngram_lm(8, V, 2, 5, 1.1))
    bo = oracle.Boost(V, np.array([0, 2]), np.array([1, 0]), 1.0)
    enc = synth.normal_bf16(8, 1, 0, 0, T * H, 1.0).reshape(T, H)
    lam, beta = 0.5, 0.75
    b = oracle.Stream(V)
    oracle.beam_chunk(b, model, lm, bo, enc, lam, beta, 27)
    got = {tuple(y): s for y, s in b.beam_hyps()}
    want = {}
    for align in itertools.product(range(V + 1), repeat=T):
        y, score = [], 0.0
        for t, a in enumerate(align):
            st = oracle.Stream(V)
            rho = int(bo.trajectory(y)[1][-1]) if y else 0
            st.set_history(y, rho)
            score += oracle.fused_row(st, model, lm, bo, enc[t], lam, beta)[a]
            if a != V:
                y = y + [a]
        k = tuple(y)
        want[k] = np.logaddexp(want[k], score) if k in want else score
    assert set(got) == set(want)
    for k in want:
        assert abs(got[k] - want[k]) < 1e-9, k


def _brute_selections(model, lm, bo, enc, lam, beta, K):
    """Top-K kept candidates per frame by (score desc, hypothesis, label),
    from fused rows of each hypothesis: an independent driver of the beam."""
    V = model.V
    hyps = [([], 0.0, 0)]
    sels = []
    for t in range(enc.shape[0]):
        cands = []
        for i, (y, sc, rho) in enumerate(hyps):
            st = oracle.Stream(V)
            st.set_history(y, rho)
            f = oracle.fused_row(st, model, lm, bo, enc[t], lam, beta)
            cands += [(sc + f[v], i, v) for v in range(V + 1)]
        cands.sort(key=lambda c: (-c[0], c[1], c[2]))
        kept = cands[:K]
        sels.append(kept)
        nxt = []
        for sc, i, v in kept:
            y, _, rho = hyps[i]
            y2 = y + ([v] if v != V else [])
            rho2 = int(bo.trajectory(y2)[1][-1]) if y2 else 0
            for j, (yy, ss, rr) in enumerate(nxt):
                if yy == y2:
                    nxt[j] = (yy, float(np.logaddexp(ss, sc)), rr)
                    break
            else:
                nxt.append((y2, sc, rho2))
        hyps = nxt
    return sels, hyps


def test_beam_follow_mode():
    """Following the brute-force selections reproduces the free-running beam
    with no flagged frame; a selection that drops a clearly better candidate
    is flagged."""
    V, H, T, K = 6, 16, 5, 3
    model, _ = _tiny_model(V=V, H=H, seed=12)
    lm = oracle.LM.from_arrays(synth.ngram_lm(12, V, 3, 40, 1.1))
    bo = oracle.Boost(V, np.array([0, 2, 3]), np.array([1, 2, 4]), 1.0)
    enc = synth.normal_bf16(12, 1, 0, 0, T * H, 1.0).reshape(T, H)
    sels, hyps = _brute_selections(model, lm, bo, enc, 0.4, 0.8, K)
    free = oracle.Stream(V)
    oracle.beam_chunk(free, model, lm, bo, enc, 0.4, 0.8, K)
    got = free.beam_hyps()
    assert [h[0] for h in got] == [h[0] for h in hyps]
    for (ya, sa), (yb, sb, _) in zip(got, hyps):
        assert abs(sa - sb) < 1e-9
    sh = np.array([[c[1] for c in s] for s in sels], dtype=np.int32)
    stok = np.array([[c[2] for c in s] for s in sels], dtype=np.int32)
    sinc = np.zeros_like(sh, dtype=np.float32)
    fol = oracle.Stream(V)
    rep = oracle.beam_chunk_follow(fol, model, lm, bo, enc, 0.4, 0.8, K, sh, stok, sinc)
    assert rep[oracle.REP_MISMATCH] == 0 and rep[oracle.REP_INCONSISTENT] == 0
    assert [h[0] for h in fol.beam_hyps()] == [h[0] for h in got]
    # keep the worst candidate of hypothesis 0 instead of the best one at frame 0
    bad_tok = stok.copy()
    st0 = oracle.Stream(V)
    f0 = oracle.fused_row(st0, model, lm, bo, enc[0], 0.4, 0.8)
    bad_tok[0, 0] = int(np.argmin(f0))
    rep = oracle.beam_chunk_follow(oracle.Stream(V), model, lm, bo, enc, 0.4, 0.8, K, sh, bad_tok, sinc)
    assert rep[oracle.REP_MISMATCH] >= 1


def test_lm_order_of_input_does_not_matter():
    """The dictionary is the same whether the n-grams arrive sorted or not."""
    V = 9
    lmA = synth.ngram_lm(41, V, 3, 120, 1.1)
    a = oracle.LM.from_arrays(lmA)
    rng = np.random.default_rng(3)
    perms = [rng.permutation(len(x)) for x in lmA.logp]
    b = oracle.LM(V, [t[p] for t, p in zip(lmA.tokens, perms)], [x[p] for x, p in zip(lmA.logp, perms)],
                  [x[p] for x, p in zip(lmA.bow, perms)])
    for h in [[], [1], [2, 3], [4, 0, 7]]:
        for v in range(V):
            assert a.score(h, v) == b.score(h, v)
        assert a.state(h) == b.state(h)
