"""The allocation-free joint selection, tsd_joint_select_noalloc.

It exists for callers that cannot allocate device memory when they decode
(code inside a memory pool that owns the whole device, plugins given
pre-allocated buffers, real-time paths that cannot take cudaMalloc's
synchronization).  Its working memory is a fixed array inside the library.

The check: one label step from the start of a stream, computed two ways --
by the ordinary decoder (tsd_decode_chunk with one frame and one symbol per
frame, fresh streams) and by two consecutive calls of the allocation-free
entry point on the same joint input, weights and fusion bias -- must agree
within the tolerances of the parity tests; the selection is also checked
against the oracle's fused row for a fresh stream.  This file is collected
last.
"""
import numpy as np
import pytest

import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def test_noalloc_selection_matches_decoder_two_calls():
    assert torch.cuda.is_available(), "GPU test needs a CUDA device"
    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[1], B=200, T=1, chunks=1, max_sym=1, beta=1.5)
    lmA = synth.ngram_lm(31, w.V, 3, 60_000, 1.1)
    ph = synth.phrases(31, w.V, 400, 1, 4, 0.2)
    E, W = synth.joint_weights(w)
    dev = torch.device("cuda", 0)
    Wd = torch.from_numpy(W.view(np.int16)).to(dev)
    Ed = torch.from_numpy(E.view(np.int16)).to(dev)
    lm = tsd.NGram.from_arrays(lmA)
    bo = tsd.Boost.from_phrases(w.V, ph, w.bonus)
    dec = tsd.Decoder(w.V, w.H, Wd, Ed, lm=lm, boost=bo, max_symbols=1, max_streams=w.B, max_T=1)
    slots = [dec.open() for _ in range(w.B)]
    enc = synth.enc_chunk(w, range(w.B), 0)  # [B, 1, H]
    encd = torch.from_numpy(enc.view(np.int16)).to(dev)
    out = dec.decode_chunk(slots, encd, w.lam, w.beta)
    torch.cuda.synchronize()
    cnt = out.counts.cpu().numpy()
    tok = out.tokens.cpu().numpy()[:, 0]
    sc = out.scores.cpu().numpy()[:, 0]

    # the same step for the allocation-free entry point: joint input from the
    # start-of-sequence row E[V], W_out label-major, and the start state's
    # fusion bias (unigram LM score, bonus of labels that start a phrase)
    enc_f = torch.from_numpy(synth.bf16_to_f32(enc[:, 0])).to(dev)
    A = torch.relu(enc_f + torch.from_numpy(synth.bf16_to_f32(E[w.V])).to(dev)).to(torch.bfloat16).contiguous()
    Wt = torch.from_numpy(W.view(np.int16)).to(dev).t().contiguous()  # [V+1, H]
    starts = np.zeros(w.V, dtype=np.float32)
    for i in range(ph.n):
        starts[ph.phrase(i)[0]] = 1.0
    row = w.lam * lmA.logp[0].astype(np.float32) + np.float32(w.beta * w.bonus) * starts
    bias = torch.from_numpy(np.tile(row, (w.B, 1))).to(dev).contiguous()

    # fused values by torch on the same inputs, for the near-tie rule
    logits = A.float() @ torch.from_numpy(synth.bf16_to_f32(W)).to(dev)
    fused = logits.clone()
    fused[:, : w.V] += bias
    top2 = torch.topk(fused, 2, dim=1).values
    gap = (top2[:, 0] - top2[:, 1]).cpu().numpy()

    first = None
    for call in range(2):
        lab = torch.full((w.B,), -1, dtype=torch.int32, device=dev)
        score = torch.full((w.B,), float("nan"), dtype=torch.float32, device=dev)
        tsd.joint_select_noalloc(A, Wt.view(torch.int16), bias, lab, score)
        torch.cuda.synchronize()
        lab, score = lab.cpu().numpy(), score.cpu().numpy()
        want = np.where(cnt > 0, tok, w.V)
        clear = gap > pu.GAP_TOL
        assert clear.sum() > 0.9 * w.B
        assert np.array_equal(lab[clear], want[clear]), call
        emitted = clear & (cnt > 0)
        assert np.abs(score[emitted] - sc[emitted]).max() <= pu.SCORE_TOL, call
        assert np.isfinite(score).all()
        if first is None:
            first = (lab, score)
        else:
            assert np.array_equal(first[0], lab) and np.array_equal(first[1], score)

    # and against the oracle: the fused row of a fresh stream (empty history,
    # previous label = blank) in double precision, for a sample of rows
    import oracle

    olm = oracle.LM.from_arrays(lmA)
    obo = oracle.Boost.from_phrases(w.V, ph, w.bonus)
    model = oracle.Model(w.V, w.H, E, W)
    lab, score = first
    checked = 0
    for r in range(0, w.B, 7):
        f = oracle.fused_row(oracle.Stream(w.V), model, olm, obo, enc[r, 0], w.lam, w.beta)
        best = int(np.argmax(f))
        top2 = np.sort(f)[-2:]
        if top2[1] - top2[0] > pu.GAP_TOL:
            assert lab[r] == best, r
            checked += 1
        assert abs(float(score[r]) - f[lab[r]]) <= pu.SCORE_TOL, r
    assert checked > 20


def test_noalloc_rejects_sizes_beyond_its_array():
    assert torch.cuda.is_available(), "GPU test needs a CUDA device"
    import paper_2609_14991_gb300 as tsd

    dev = torch.device("cuda", 0)
    A = torch.zeros((1025, 64), dtype=torch.bfloat16, device=dev)
    Wt = torch.zeros((16, 64), dtype=torch.int16, device=dev)
    lab = torch.zeros(1025, dtype=torch.int32, device=dev)
    score = torch.zeros(1025, dtype=torch.float32, device=dev)
    with pytest.raises(tsd.TsdError) as e:
        tsd.joint_select_noalloc(A, Wt, None, lab, score)
    assert e.value.status == tsd.TSD_EINVAL
    Wbig = torch.zeros((8193, 64), dtype=torch.int16, device=dev)
    with pytest.raises(tsd.TsdError) as e:
        tsd.joint_select_noalloc(A[:4], Wbig, None, lab, score)
    assert e.value.status == tsd.TSD_EINVAL
