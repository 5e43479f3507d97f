"""Stream state export and import: a stream exported after one chunk and
imported into another decoder (other slot ids) continues exactly as it
would have in the first."""
from __future__ import annotations

import numpy as np
import pytest

import synth

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
    _chunk(a, sa, w, 0)
    for x, y in zip(sa, sb):
        b.import_state(y, a.export_state(x))
    assert _chunk(a, sa, w, 1) == _chunk(b, sb, w, 1)
    for x, y in zip(sa, sb):
        assert a.state(x) == b.state(y)


def test_beam_stream_moves_between_decoders():
    w = synth.scaled(synth.WORKLOADS[3], V=96, H=128, B=3, T=10)
    lms = [(synth.ngram_lm(w.lm_seed, w.V, 3, 2000, 1.1), 1.0)]
    ph = synth.phrases(w.boost_seed, w.V, 8, 2, 4, 0.0)
    E, W = synth.joint_weights(w)
    a, b = _make(w, E, W, lms, ph, beam_k=3), _make(w, E, W, lms, ph, beam_k=3)
    sa = [a.open() for _ in range(w.B)]
    _ = [b.open() for _ in range(2)]
    sb = [b.open() for _ in range(w.B)]
    _chunk(a, sa, w, 0)
    for x, y in zip(sa, sb):
        b.import_state(y, a.export_state(x))
    _chunk(a, sa, w, 1)
    _chunk(b, sb, w, 1)
    for x, y in zip(sa, sb):
        assert a.hyps(x) == b.hyps(y)


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
