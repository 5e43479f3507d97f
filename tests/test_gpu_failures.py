"""Failure paths, made to happen without faulting the GPU.

* An allocation that fails (injected on the host by tsd_debug_fail_alloc,
  at every allocation point in turn) makes the call return TSD_ENOMEM,
  releases what the call had allocated, and leaves the library usable: the
  next build and create succeed and decode with parity.
* A bounded device wait that expires (the joint kernel's wait limit set to
  0 ns through the decoder option "wait_ns") ends the kernel early, after it
  has waited for every copy and MMA it started; tsd_decoder_check then
  returns TSD_EDEVICE, and new streams of the same decoder as well as a
  fresh decoder decode with parity against the oracle.
"""
import numpy as np
import pytest

import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


def _small():
    return synth.scaled(synth.WORKLOADS[0], V=200, H=128, B=5, T=16, lm_total=4000, n_phr=12, phr_len=(2, 4))


def _free_bytes():
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0]


def test_injected_allocation_failures_return_enomem_and_recover():
    import paper_2609_14991_gb300 as tsd

    w = _small()
    inp = pu.Inputs(w)
    dev = torch.device("cuda", 0)
    Wd = torch.from_numpy(inp.W.view(np.int16)).to(dev)
    Ed = torch.from_numpy(inp.E.view(np.int16)).to(dev)
    # table builders: every allocation point fails in turn
    points = {}
    for name, build in (("ngram", lambda: tsd.NGram.from_arrays(inp.lmA)),
                        ("boost", lambda: tsd.Boost.from_phrases(w.V, inp.ph, w.bonus))):
        before = _free_bytes()
        n = 0
        while True:
            n += 1
            tsd.debug_fail_alloc(n)
            try:
                obj = build()
            except tsd.TsdError as e:
                assert e.status == tsd.TSD_ENOMEM, (name, n, str(e))
                continue
            tsd.debug_fail_alloc(0)
            del obj
            break
        points[name] = n - 1
        assert before - _free_bytes() < (32 << 20), name  # nothing of the failed builds stays allocated
    lm = tsd.NGram.from_arrays(inp.lmA)
    bo = tsd.Boost.from_phrases(w.V, inp.ph, w.bonus)
    before = _free_bytes()
    n = 0
    while True:
        n += 1
        tsd.debug_fail_alloc(n)
        try:
            dec = tsd.Decoder(w.V, w.H, Wd, Ed, lm=lm, boost=bo, max_symbols=w.max_sym, max_streams=w.B, max_T=w.T)
        except tsd.TsdError as e:
            assert e.status == tsd.TSD_ENOMEM, (n, str(e))
            continue
        tsd.debug_fail_alloc(0)
        break
    points["decoder"] = n - 1
    assert points["ngram"] >= 8 and points["boost"] >= 8 and points["decoder"] >= 15, points
    del dec
    assert before - _free_bytes() < (64 << 20)
    # the library still works: a decode with parity
    run = pu.GpuRun(inp, range(w.B), 2)
    pu.assert_reports(pu.replay(inp, run, range(w.B)))


def test_expired_wait_reports_edevice_and_recovers():
    import paper_2609_14991_gb300 as tsd

    w = _small()
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(w.B), 1)  # a decoder that has decoded normally
    dec = run.dec
    dec.set_option("wait_ns", 0)
    enc = torch.from_numpy(synth.enc_chunk(w, range(w.B), 1).view(np.int16)).to(torch.device("cuda", 0))
    dec.decode_chunk(run.slots, enc, inp.lam, inp.beta)
    torch.cuda.synchronize()
    with pytest.raises(tsd.TsdError) as e:
        dec.check()
    assert e.value.status == tsd.TSD_EDEVICE
    dec.check()  # the code was cleared
    # the context and the decoder are usable: restore the limit, new streams
    dec.set_option("wait_ns", 1_000_000_000)
    for s in run.slots:
        dec.close(s)
    slots = [dec.open() for _ in range(w.B)]
    olm, obo, model = pu.oracle_models(inp)
    enc0 = synth.enc_chunk(w, range(w.B), 0)
    out = dec.decode_chunk(slots, torch.from_numpy(enc0.view(np.int16)).to(torch.device("cuda", 0)), inp.lam,
                           inp.beta)
    torch.cuda.synchronize()
    dec.check()
    import oracle

    toks, frames, scores, counts = (x.cpu().numpy() for x in (out.tokens, out.frames, out.scores, out.counts))
    for i in range(w.B):
        st = oracle.Stream(w.V)
        k = int(counts[i])
        _, _, _, rep = oracle.decode_chunk(st, model, olm, obo, enc0[i], inp.lam, inp.beta, w.max_sym,
                                           follow=(toks[i, :k], frames[i, :k], scores[i, :k]), gap_tol=pu.GAP_TOL)
        assert rep[oracle.REP_INCONSISTENT] == 0 and rep[oracle.REP_MISMATCH] == 0, (i, rep)
        assert rep[oracle.REP_MAX_SCORE_DIFF] <= pu.SCORE_TOL, (i, rep)
    # and a fresh decoder
    fresh = pu.GpuRun(inp, range(w.B), 2)
    pu.assert_reports(pu.replay(inp, fresh, range(w.B)))
