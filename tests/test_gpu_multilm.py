"""Several n-gram LMs fused at once (Eq. 1: the LM term is the sum over LMs
of alpha_i log p_LM_i) on the GPU, against the oracle on the same inputs."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu


def _decoder(w, lms, ph, E, W, beam_k=1):
    import torch

    import paper_2609_14991_gb300 as tsd

    dev = torch.device("cuda", 0)
    gl = [(tsd.NGram.from_arrays(a), wt) for a, wt in lms]
    bo = tsd.Boost.from_phrases(w.V, ph, w.bonus) if ph is not None else None
    dec = tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev),
                      lms=gl, boost=bo, max_symbols=w.max_sym, beam_k=beam_k, max_streams=w.B, max_T=w.T)
    return dec, gl, bo


@pytest.mark.parametrize("V,n_lm", [(256, 2), (1024, 3), (200, 4)])
def test_several_lms_match_oracle(V, n_lm):
    """Follow mode over two chunks: every LM's state bit-exact after each
    chunk, labels equal wherever the oracle's top-2 gap exceeds 1e-3, fused
    scores within 1e-4."""
    import torch

    w = synth.scaled(synth.WORKLOADS[0], V=V, H=256, B=5, T=24, n_phr=20, phr_len=(2, 5))
    specs = [(3, 6000, 1.1), (2, 2500, 1.05), (4, 9000, 1.2), (2, 800, 1.3)][:n_lm]
    arrays = [synth.ngram_lm(w.lm_seed + 17 * i, V, o, tot, z) for i, (o, tot, z) in enumerate(specs)]
    weights = [1.0, 0.5, 0.25, -0.2][:n_lm]
    ph = synth.phrases(w.boost_seed, V, w.n_phr, 2, 5, 0.2)
    E, W = synth.joint_weights(w)
    dec, gl, _ = _decoder(w, list(zip(arrays, weights)), ph, E, W)
    slots = [dec.open() for _ in range(w.B)]
    olms = [(oracle.LM.from_arrays(a), wt) for a, wt in zip(arrays, weights)]
    obo = oracle.Boost.from_phrases(V, ph, w.bonus)
    model = oracle.Model(V, w.H, E, W)
    streams = [oracle.Stream(V) for _ in range(w.B)]
    dev = torch.device("cuda", 0)
    for chunk in range(2):
        enc = synth.enc_chunk(w, range(w.B), chunk)
        out = dec.decode_chunk(slots, torch.from_numpy(enc.view(np.int16)).to(dev), w.lam, w.beta)
        torch.cuda.synchronize()
        toks, frames, scores, counts = (x.cpu().numpy() for x in (out.tokens, out.frames, out.scores, out.counts))
        for i in range(w.B):
            n = int(counts[i])
            _, _, _, rep = oracle.decode_chunk(streams[i], model, olms, obo, enc[i], w.lam, w.beta, w.max_sym,
                                               follow=(toks[i, :n], frames[i, :n], scores[i, :n]))
            assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, rep
            assert rep[oracle.REP_MAX_SCORE_DIFF] <= pu.SCORE_TOL, rep
            hist = streams[i].history()
            for m, (g, _) in enumerate(gl):
                assert g.state_tuple(dec.lm_state(slots[i], m)) == olms[m][0].state(hist), (chunk, i, m)


def test_one_lm_through_the_several_lm_entry_is_the_plain_decoder():
    """create_multi with one LM of weight 1 decodes exactly as create."""
    import torch

    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[0], V=300, H=192, B=3, T=20)
    a = synth.ngram_lm(w.lm_seed, w.V, 3, 5000, 1.1)
    ph = synth.phrases(w.boost_seed, w.V, 12, 2, 4, 0.0)
    E, W = synth.joint_weights(w)
    dev = torch.device("cuda", 0)
    enc = torch.from_numpy(synth.enc_chunk(w, range(w.B), 0).view(np.int16)).to(dev)
    multi, _, _ = _decoder(w, [(a, 1.0)], ph, E, W)
    plain = tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev),
                        lm=tsd.NGram.from_arrays(a), boost=tsd.Boost.from_phrases(w.V, ph, w.bonus),
                        max_symbols=w.max_sym, max_streams=w.B, max_T=w.T)
    outs = []
    for dec in (multi, plain):
        slots = [dec.open() for _ in range(w.B)]
        o = dec.decode_chunk(slots, enc, w.lam, w.beta)
        torch.cuda.synchronize()
        outs.append([x.cpu().numpy() for x in (o.tokens, o.frames, o.scores, o.counts)])
    (t1, f1, s1, c1), (t2, f2, s2, c2) = outs
    assert np.array_equal(c1, c2)
    for i in range(w.B):  # entries past a stream's count are not written
        n = int(c1[i])
        assert np.array_equal(t1[i, :n], t2[i, :n]) and np.array_equal(f1[i, :n], f2[i, :n])
        assert np.array_equal(s1[i, :n], s2[i, :n])


def test_several_lm_rejections():
    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[0], V=64, H=128, B=2, T=8, max_sym=1)
    a = synth.ngram_lm(5, w.V, 2, 300, 1.1)
    E, W = synth.joint_weights(w)
    with pytest.raises(tsd.TsdError):  # beam search takes one LM
        _decoder(w, [(a, 1.0), (a, 1.0)], None, E, W, beam_k=2)
    with pytest.raises(tsd.TsdError):  # at most four LMs
        _decoder(w, [(a, 1.0)] * 5, None, E, W)
    b = synth.ngram_lm(6, w.V + 1, 2, 300, 1.1)
    with pytest.raises(tsd.TsdError):  # vocabulary sizes must agree
        import torch

        dev = torch.device("cuda", 0)
        tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev),
                    lms=[(tsd.NGram.from_arrays(a), 1.0), (tsd.NGram.from_arrays(b), 1.0)], max_streams=2, max_T=8)
