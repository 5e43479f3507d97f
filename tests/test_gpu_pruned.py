"""Pruned fusion on the GPU (the LM and boost terms re-rank only the acoustic
model's k best outputs) against the oracle's pruned decode."""
from __future__ import annotations

import numpy as np
import pytest

import oracle
import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu


def _run(V, k, B=6, T=20, chunks=2, H=256, lm_order=3, lm_total=8000, n_phr=30, bn=None):
    import torch

    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[0], V=V, H=H, B=B, T=T, n_phr=n_phr, phr_len=(2, 5))
    a = synth.ngram_lm(w.lm_seed, V, lm_order, lm_total, w.zipf)
    ph = synth.phrases(w.boost_seed, V, n_phr, 2, 5, 0.2)
    E, W = synth.joint_weights(w)
    dev = torch.device("cuda", 0)
    lm, bo = tsd.NGram.from_arrays(a), tsd.Boost.from_phrases(V, ph, w.bonus)
    dec = tsd.Decoder(V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev),
                      lm=lm, boost=bo, max_symbols=w.max_sym, max_streams=B, max_T=T, prune_k=k)
    if bn:
        dec.set_option("joint_bn", bn)
    slots = [dec.open() for _ in range(B)]
    olm, obo = oracle.LM.from_arrays(a), oracle.Boost.from_phrases(V, ph, w.bonus)
    model = oracle.Model(V, w.H, E, W)
    streams = [oracle.Stream(V) for _ in range(B)]
    steps = 0
    for c in range(chunks):
        enc = synth.enc_chunk(w, range(B), c)
        out = dec.decode_chunk(slots, torch.from_numpy(enc.view(np.int16)).to(dev), w.lam, w.beta)
        torch.cuda.synchronize()
        toks, frames, scores, counts = (x.cpu().numpy() for x in (out.tokens, out.frames, out.scores, out.counts))
        for i in range(B):
            n = int(counts[i])
            _, _, _, rep = oracle.decode_chunk(streams[i], model, olm, obo, enc[i], w.lam, w.beta, w.max_sym,
                                               follow=(toks[i, :n], frames[i, :n], scores[i, :n]), prune_k=k,
                                               am_tol=pu.LOGIT_TOL, gap_tol=pu.GAP_TOL)
            assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, (c, i, rep)
            assert rep[oracle.REP_MAX_SCORE_DIFF] <= pu.SCORE_TOL, (c, i, rep)
            steps += int(rep[oracle.REP_STEPS])
            hist = streams[i].history()
            lm_state, trie_node, last = dec.state(slots[i])
            assert last == (hist[-1] if hist else V)
            assert lm.state_tuple(lm_state) == olm.state(hist)
            assert bo.node_tuple(trie_node) == pu.trie_tuple(obo, hist, streams[i].rho())
    assert steps > B * T


@pytest.mark.parametrize("V,k", [(256, 1), (256, 4), (1024, 8), (1024, 3)])
def test_pruned_matches_oracle(V, k):
    _run(V, k)


def test_pruned_large_vocabulary_wide_tiles():
    _run(4096, 6, B=4, T=12, H=512, lm_order=4, lm_total=40000, bn=256)


def test_pruned_rejections():
    import torch

    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[0], V=64, H=128, B=2, T=8, max_sym=1)
    E, W = synth.joint_weights(w)
    dev = torch.device("cuda", 0)
    args = (w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev))
    with pytest.raises(tsd.TsdError):
        tsd.Decoder(*args, max_symbols=1, beam_k=2, max_streams=2, max_T=8, prune_k=4)  # beam and pruning
    with pytest.raises(tsd.TsdError):
        tsd.Decoder(*args, max_streams=2, max_T=8, prune_k=9)  # at most 8 candidates
    dec = tsd.Decoder(*args, max_streams=2, max_T=8, prune_k=2)
    with pytest.raises(tsd.TsdError):
        dec.set_joint_kernel(1)  # the CUDA-core kernel has no pruned epilogue
