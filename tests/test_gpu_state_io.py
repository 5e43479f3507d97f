"""Stream state export and import: a stream exported after one chunk and
imported into another decoder (other slot ids) continues exactly as it
would have in the first, and the oracle, following the first decoder's
chunk and then the second's, finds every decision, fused score and state
of the migrated stream correct."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu


def _make(w, E, W, lms, ph, beam_k=1):
    import torch

    import paper_2609_14991_gb300 as tsd

    dev = torch.device("cuda", 0)
    bo = tsd.Boost.from_phrases(w.V, ph, w.bonus) if ph is not None else None
    kw = dict(boost=bo, max_symbols=w.max_sym, beam_k=beam_k, max_streams=2 * w.B, max_T=w.T)
    g = [(tsd.NGram.from_arrays(a), wt) for a, wt in lms]
    if len(g) == 1:
        kw["lm"] = g[0][0]
    else:
        kw["lms"] = g
    return tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev),
                       **kw)


def _chunk(dec, slots, w, c):
    import torch

    enc = torch.from_numpy(synth.enc_chunk(w, range(w.B), c).view(np.int16)).to(torch.device("cuda", 0))
    o = dec.decode_chunk(slots, enc, w.lam, w.beta)
    torch.cuda.synchronize()
    t, f, s, n = (x.cpu().numpy() for x in (o.tokens, o.frames, o.scores, o.counts))
    return [(t[i, :n[i]].tolist(), f[i, :n[i]].tolist(), s[i, :n[i]].tolist()) for i in range(len(slots))]


@pytest.mark.parametrize("n_lm", [1, 2])
def test_greedy_stream_moves_between_decoders(n_lm):
    w = synth.scaled(synth.WORKLOADS[0], V=128, H=128, B=4, T=16, n_phr=10, phr_len=(2, 4))
    lms = [(synth.ngram_lm(w.lm_seed + i, w.V, 3, 3000, 1.1), 1.0 - 0.4 * i) for i in range(n_lm)]
    ph = synth.phrases(w.boost_seed, w.V, 10, 2, 4, 0.0)
    E, W = synth.joint_weights(w)
    a, b = _make(w, E, W, lms, ph), _make(w, E, W, lms, ph)
    sa = [a.open() for _ in range(w.B)]
    _ = [b.open() for _ in range(w.B)]  # occupy other slot ids first
    sb = [b.open() for _ in range(w.B)]
    first = _chunk(a, sa, w, 0)
    for x, y in zip(sa, sb):
        b.import_state(y, a.export_state(x))
    second = _chunk(b, sb, w, 1)
    assert _chunk(a, sa, w, 1) == second
    for x, y in zip(sa, sb):
        assert a.state(x) == b.state(y)
    # the oracle follows chunk 0 as decoded by a, then chunk 1 as decoded by b
    olms = [(oracle.LM.from_arrays(x), wt) for x, wt in lms]
    obo = oracle.Boost.from_phrases(w.V, ph, w.bonus)
    model = oracle.Model(w.V, w.H, E, W)
    gl = b.lm if isinstance(b.lm, list) else [b.lm]
    for i in range(w.B):
        st = oracle.Stream(w.V)
        for c, res in ((0, first), (1, second)):
            tok, fr, sc = res[i]
            _, _, _, rep = oracle.decode_chunk(st, model, olms if n_lm > 1 else olms[0][0], obo,
                                               synth.enc_chunk(w, [i], c)[0], w.lam, w.beta, w.max_sym,
                                               follow=(tok, fr, sc), gap_tol=pu.GAP_TOL)
            assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, (i, c, rep)
            assert rep[oracle.REP_MAX_SCORE_DIFF] <= pu.SCORE_TOL, (i, c, rep)
        hist = st.history()
        lm_state, node, last = b.state(sb[i])
        assert last == (hist[-1] if hist else w.V)
        for m, g in enumerate(gl):
            got = b.lm_state(sb[i], m) if n_lm > 1 else lm_state
            assert g.state_tuple(got) == olms[m][0].state(hist), (i, m)
        assert b.boost.node_tuple(node) == pu.trie_tuple(obo, hist, st.rho()), i


def test_beam_stream_moves_between_decoders():
    w = synth.scaled(synth.WORKLOADS[3], V=96, H=128, B=3, T=10)
    lms = [(synth.ngram_lm(w.lm_seed, w.V, 3, 2000, 1.1), 1.0)]
    ph = synth.phrases(w.boost_seed, w.V, 8, 2, 4, 0.0)
    E, W = synth.joint_weights(w)
    a, b = _make(w, E, W, lms, ph, beam_k=3), _make(w, E, W, lms, ph, beam_k=3)
    sa = [a.open() for _ in range(w.B)]
    _ = [b.open() for _ in range(2)]
    sb = [b.open() for _ in range(w.B)]
    import torch

    caps = []
    for d in (a, b):
        rows = torch.full((w.T, w.B * 3, 4), -7, dtype=torch.int32, device="cuda")
        logits = torch.zeros((w.T, w.B * 3, w.N), dtype=torch.float32, device="cuda")
        d.debug_capture(logits, rows, w.T)
        caps.append(rows)
    _chunk(a, sa, w, 0)
    sel0 = caps[0].cpu().numpy().copy()
    for x, y in zip(sa, sb):
        b.import_state(y, a.export_state(x))
    _chunk(a, sa, w, 1)
    _chunk(b, sb, w, 1)
    sel1 = caps[1].cpu().numpy().copy()
    for x, y in zip(sa, sb):
        assert a.hyps(x) == b.hyps(y)
    # the oracle follows a's kept candidates over chunk 0 and b's over chunk 1
    olm = oracle.LM.from_arrays(lms[0][0])
    obo = oracle.Boost.from_phrases(w.V, ph, w.bonus)
    model = oracle.Model(w.V, w.H, E, W)
    K = 3
    for i in range(w.B):
        st = oracle.Stream(w.V)
        for c, sel in ((0, sel0), (1, sel1)):
            s_i = sel[:, i * K:(i + 1) * K, :]
            rep = oracle.beam_chunk_follow(st, model, olm, obo, synth.enc_chunk(w, [i], c)[0], w.lam, w.beta, K,
                                           s_i[:, :, 0], s_i[:, :, 1], s_i[:, :, 2].view(np.float32), pu.GAP_TOL,
                                           S=w.max_sym)
            assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, (i, c, rep)
            assert rep[oracle.REP_MAX_SCORE_DIFF] <= pu.SCORE_TOL, (i, c, rep)
        want = st.beam_hyps()
        got = b.hyps(sb[i])
        assert [g[0] for g in got] == [h[0] for h in want], i
        for (_, gs), h in zip(got, want):
            assert abs(gs - h[1]) <= pu.SCORE_TOL * 2 * w.T, i


def test_import_rejects_mismatched_or_damaged_blobs():
    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[0], V=64, H=128, B=2, T=8)
    lm = [(synth.ngram_lm(w.lm_seed, w.V, 3, 900, 1.1), 1.0)]
    ph = synth.phrases(w.boost_seed, w.V, 6, 2, 3, 0.0)
    E, W = synth.joint_weights(w)
    a = _make(w, E, W, lm, ph)
    s = [a.open() for _ in range(w.B)]
    _chunk(a, s, w, 0)
    blob = a.export_state(s[0])
    with pytest.raises(tsd.TsdError):  # truncated
        a.import_state(s[1], blob[:-4])
    bad = bytearray(blob)
    # after the 32-byte header: previous label (4 bytes), the LM chain length
    # (4) and its ids; claim one state with an id past the LM's states
    bad[36:40] = (1).to_bytes(4, "little")
    bad[40:44] = (1 << 30).to_bytes(4, "little")
    with pytest.raises(tsd.TsdError):
        a.import_state(s[1], bytes(bad))
    w2 = synth.scaled(w, V=65)
    E2, W2 = synth.joint_weights(w2)
    c = _make(w2, E2, W2, [(synth.ngram_lm(1, 65, 2, 200, 1.1), 1.0)], None)
    sc = c.open()
    with pytest.raises(tsd.TsdError):  # another vocabulary
        c.import_state(sc, blob)
    a.import_state(s[1], blob)  # the intact blob still imports
    assert a.state(s[1]) == a.state(s[0])
