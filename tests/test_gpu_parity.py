"""GPU parity: the CUDA decode path against the oracle on the same seeded
inputs, through the C ABI.

Rules (fixed here, derived from the fp32 arithmetic of the kernels):
  * label sequences match wherever the oracle's top-2 gap exceeds 1e-3;
    at nearer ties either choice is valid and the oracle follows the GPU;
  * fused scores of emitted labels within 1e-4 absolute;
  * joint logits within 2e-2 of the oracle's double product of the same
    bf16-rounded inputs;
  * LM state and trie node bit-exact (as label tuples) after every chunk,
    and at every step where steps are captured.
"""
import numpy as np
import pytest

import oracle
import synth
from tests import parity_util as pu

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    import paper_2609_14991_gb300 as tsd

    tsd.lib()  # fails loudly if the library is missing


def _evaluations(tok, fr, T, max_sym):
    """(frame, labels emitted before) of every joint evaluation of one chunk,
    reconstructed from the emitted labels: a frame with j < max_sym labels
    had j + 1 evaluations (the last chose blank), one with max_sym had j."""
    ev = []
    hist = []
    p = 0
    for t in range(T):
        j = 0
        while True:
            ev.append((t, list(hist)))
            if p < len(tok) and fr[p] == t:
                hist.append(int(tok[p]))
                p += 1
                j += 1
                if j == max_sym:
                    break
            else:
                break
    return ev


def test_cfg0_full_parity_with_step_capture():
    w = synth.WORKLOADS[0]
    inp = pu.Inputs(w)
    S = w.T * w.max_sym
    run = pu.GpuRun(inp, range(w.B), 1, capture_steps=S)
    reps = pu.replay(inp, run, range(w.B))
    pu.assert_reports(reps)
    olm, obo, model = pu.oracle_models(inp)
    rows = run.cap_rows.cpu().numpy()
    logits = run.cap_logits.cpu().numpy()
    worst = 0.0
    for i in range(w.B):
        tok, fr, _ = run.emitted(i, 0)
        ev = _evaluations(tok, fr, w.T, w.max_sym)
        assert len(ev) <= S
        for s, (t, hist) in enumerate(ev):
            ft, last, lm_state, node = rows[s, i]
            assert ft == t
            assert last == (hist[-1] if hist else w.V)
            assert run.lm.state_tuple(lm_state) == olm.state(hist), (i, s)
            rho = int(obo.trajectory(hist)[1][-1]) if hist else 0
            assert run.bo.node_tuple(node) == pu.trie_tuple(obo, hist, rho), (i, s)
            if s % 9 == 0:
                want = model.joint_logits(run.enc[0][i][t], last)
                worst = max(worst, float(np.abs(logits[s, i] - want).max()))
        assert (rows[len(ev):, i, 0] == -1).all()  # finished rows stay idle
    assert worst < pu.LOGIT_TOL, worst
    print(f"cfg0: max |logit - oracle| = {worst:.2e}")


def test_cfg1_sampled_parity_full_length():
    w = synth.WORKLOADS[1]
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(w.B), w.chunks)
    reps = pu.replay(inp, run, [0, 21, 42, 63])
    pu.assert_reports(reps)


def test_cfg2_sampled_parity_full_size():
    w = synth.WORKLOADS[2]
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(w.B), w.chunks)
    reps = pu.replay(inp, run, [0, 129, 255])
    pu.assert_reports(reps)
    # the boost trie was exercised
    assert any(run.states[c][i][1] != 0 for c in range(w.chunks) for i in range(w.B))


def test_cfg4_full_size_parity():
    """The stress configuration at full size: V+1 = 4097, 1024 streams, a
    10-gram LM with ~100M n-grams, 50,000 phrases.  Every one of the 1024
    streams is replayed by the oracle over chunk 0 (LM and trie states of all
    streams compared), 64 streams over all 20 chunks; the last chunk's first
    label steps are captured and the joint logits of 32 rows compared label
    by label with the oracle's product."""
    w = synth.WORKLOADS[4]
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(w.B), w.chunks, capture_steps=3)
    models = pu.oracle_models(inp)
    long_sample = list(range(0, w.B, 16))
    pu.assert_reports(pu.replay(inp, run, long_sample, models=models))
    rest = [i for i in range(w.B) if i % 16]
    pu.assert_reports(pu.replay(inp, run, rest, chunks=1, models=models))
    assert max(len(run.lm.state_tuple(run.states[-1][i][0])) for i in range(w.B)) >= 3
    err, n = pu.captured_logit_error(run, models[2], 3, list(range(0, w.B, 32)))
    assert n >= 32 and err < pu.LOGIT_TOL, (err, n)


@pytest.mark.parametrize("path", [0, 1])
def test_fusion_paths_match_oracle(path):
    """Both forms of the greedy one-LM step (fusion_path 1: the level-0 LM
    term in the joint epilogue with a per-row correction list; 0: the
    streaming form) against the oracle, at the stress vocabulary (V+1 =
    4097) with a 6-gram LM and phrases: 48 streams replayed over both chunks,
    and the tiny workload in full."""
    w = synth.scaled(synth.WORKLOADS[4], B=160, chunks=2, lm_order=6, lm_total=400_000, n_phr=2000)
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(w.B), 2, options={"fusion_path": path})
    models = pu.oracle_models(inp)
    pu.assert_reports(pu.replay(inp, run, list(range(0, w.B, 10)) + [127, 128, 159], models=models))
    assert max(len(run.lm.state_tuple(run.states[-1][i][0])) for i in range(w.B)) >= 3
    w0 = synth.WORKLOADS[0]
    inp0 = pu.Inputs(w0)
    run0 = pu.GpuRun(inp0, range(w0.B), 1, options={"fusion_path": path})
    pu.assert_reports(pu.replay(inp0, run0, range(w0.B)))


@pytest.mark.parametrize("shape", ["cfg2", "cfg4"])
@pytest.mark.parametrize("bn", [64, 128, 256])
def test_joint_logits_elementwise(shape, bn):
    """Joint logits label by label against the oracle's double product of the
    same bf16 inputs, at the 0.6B-sized joint (H = 1024, V+1 = 1025) and the
    stress vocabulary (V+1 = 4097), for every tensor-core tile width: 200
    streams (the second 128-row tile is partial), every label including the
    last partial label tile and blank, the first 4 label steps of 2 chunks."""
    base = synth.WORKLOADS[2] if shape == "cfg2" else synth.WORKLOADS[4]
    w = synth.scaled(base, B=200, chunks=2, lm_order=4, lm_total=150_000, n_phr=400)
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(w.B), 2, capture_steps=4, options={"joint_bn": bn})
    models = pu.oracle_models(inp)
    err, n = pu.captured_logit_error(run, models[2], 4, range(w.B))
    assert n >= 4 * 190 and err < pu.LOGIT_TOL, (err, n)
    pu.assert_reports(pu.replay(inp, run, [0, 127, 128, 199], models=models))
    print(f"{shape} bn={bn}: max |logit - oracle| = {err:.2e} over {n} rows")


def test_cfg3_beam_parity():
    """Beam search, K=4, one label per frame: every frame's kept candidates
    are the oracle's top K (up to near ties), each candidate's score
    increment is within 1e-4, merges and surviving label sequences are the
    oracle's, in order, over all 40 chunks of 3 sampled streams."""
    w = synth.WORKLOADS[3]
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(w.B), w.chunks, capture_steps=w.T)
    reps = pu.replay_beam(inp, run, [0, 63, 127])
    pu.assert_reports(reps)
    assert all(len(run.beam_hyps[-1][i]) >= 1 for i in range(w.B))
    # merges happen: some frame keeps fewer than K hypotheses
    assert any(len(h) < w.beam for c in run.beam_hyps for h in c)


def test_beam_small_exhaustive_against_free_oracle():
    """Tiny beam (V=15, H=64, K=3..8) against the free-running oracle's beam,
    including the K = 8 limit and a stream with no LM or boost."""
    for K in (3, 8):
        w = synth.scaled(synth.WORKLOADS[0], V=15, H=64, B=5, T=9, beam=K, max_sym=1, lm_total=60)
        inp = pu.Inputs(w, lmA=synth.ngram_lm(7, 15, 3, 60, 1.1), ph=synth.phrases(7, 15, 3, 1, 3, 0.0))
        run = pu.GpuRun(inp, range(w.B), 3, capture_steps=w.T)
        pu.assert_reports(pu.replay_beam(inp, run, range(w.B)))
    w = synth.scaled(synth.WORKLOADS[0], V=15, H=64, B=2, T=6, beam=4, max_sym=1)
    inp = pu.Inputs(w, with_lm=False, with_boost=False)
    run = pu.GpuRun(inp, range(w.B), 2, capture_steps=w.T)
    pu.assert_reports(pu.replay_beam(inp, run, range(w.B)))


@pytest.mark.parametrize("S", [2, 5])
def test_beam_several_labels_per_frame(S):
    """Beam search with up to S labels per frame (frame-synchronous): every
    expansion's kept candidates checked and followed by the oracle, the
    surviving label sequences and scores compared after every chunk."""
    for K in (2, 4):
        w = synth.scaled(synth.WORKLOADS[0], V=15, H=64, B=4, T=7, beam=K, max_sym=S, lm_total=60)
        inp = pu.Inputs(w, lmA=synth.ngram_lm(7, 15, 3, 60, 1.1), ph=synth.phrases(7, 15, 3, 1, 3, 0.0))
        run = pu.GpuRun(inp, range(w.B), 3, capture_steps=w.T * S)
        pu.assert_reports(pu.replay_beam(inp, run, range(w.B)))
    # a stronger blank: frames end after fewer than S expansions
    w = synth.scaled(synth.WORKLOADS[0], V=15, H=64, B=3, T=8, beam=3, max_sym=S, lm_total=60)
    inp = pu.Inputs(w, lmA=synth.ngram_lm(7, 15, 3, 60, 1.1), ph=synth.phrases(7, 15, 3, 1, 3, 0.0))
    inp.W = inp.W.copy()
    inp.W[:, w.V] = pu.bf16_bits(np.full(w.H, 2.5 / np.sqrt(w.H), dtype=np.float32))
    run = pu.GpuRun(inp, range(w.B), 2, capture_steps=w.T * S)
    reps = pu.replay_beam(inp, run, range(w.B))
    pu.assert_reports(reps)
    assert sum(r["steps"] for r in reps) < w.B * 2 * w.T * S  # some frames ended early


def test_beam_several_labels_cfg3_shape():
    """The beam workload's shapes (V+1 = 1025, H = 1024, 6-gram 20M LM, 5,000
    phrases, K = 4) with up to 3 labels per frame, two chunks, three streams
    checked."""
    w = synth.scaled(synth.WORKLOADS[3], B=32, max_sym=3)
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(w.B), 2, capture_steps=w.T * 3)
    pu.assert_reports(pu.replay_beam(inp, run, [0, 15, 31]))


def _tokens(run, i):
    return np.concatenate([run.emitted(i, c)[0] for c in range(len(run.chunks))])


def test_chunking_stream_independence_determinism():
    w = synth.scaled(synth.WORKLOADS[0], B=6, T=120)
    inp = pu.Inputs(w)
    whole = pu.GpuRun(inp, range(6), 1)
    # the same frames in 4 chunks of 30 carry the state across calls
    split = pu.GpuRun(pu.Inputs(synth.scaled(w, T=30), inp.lmA, inp.ph), range(6), 4)
    for i in range(6):
        a = whole.emitted(i, 0)
        b = [split.emitted(i, c) for c in range(4)]
        assert np.array_equal(a[0], np.concatenate([x[0] for x in b]))
        assert np.array_equal(a[1], np.concatenate([x[1] + 30 * c for c, x in enumerate(b)]))
        assert np.array_equal(a[2], np.concatenate([x[2] for x in b]))
    # a subset decoded alone matches the same streams inside the batch
    sub = pu.GpuRun(inp, [4, 1], 1)
    for j, s in enumerate([4, 1]):
        for x, y in zip(sub.emitted(j, 0), whole.emitted(s, 0)):
            assert np.array_equal(x, y)
    # run to run and graph vs direct launches: bit identical
    again = pu.GpuRun(inp, range(6), 1, graphs=False)
    for i in range(6):
        for x, y in zip(again.emitted(i, 0), whole.emitted(i, 0)):
            assert np.array_equal(x, y)


@pytest.mark.parametrize("case", ["no_lm_no_boost", "zero_weights", "unigram_lm", "one_token_phrases",
                                  "one_symbol", "tiny"])
def test_edge_cases(case):
    base = synth.scaled(synth.WORKLOADS[0], B=3, T=40)
    kw = {}
    if case == "no_lm_no_boost":
        inp = pu.Inputs(base, with_lm=False, with_boost=False)
    elif case == "zero_weights":
        inp = pu.Inputs(synth.scaled(base, lam=0.0, beta=0.0))
    elif case == "unigram_lm":
        inp = pu.Inputs(base, lmA=synth.ngram_lm(3, base.V, 1, base.V, 1.1))
    elif case == "one_token_phrases":
        inp = pu.Inputs(base, ph=synth.phrases(5, base.V, 60, 1, 2, 0.0))
    elif case == "one_symbol":
        inp = pu.Inputs(synth.scaled(base, max_sym=1))
    else:  # odd vocabulary (V+1 = 16), smallest hidden size, a single stream and frame
        w = synth.scaled(base, V=15, H=64, B=1, T=1, lm_total=60)
        inp = pu.Inputs(w, lmA=synth.ngram_lm(7, 15, 3, 60, 1.1), ph=synth.phrases(7, 15, 3, 1, 3, 0.0))
    run = pu.GpuRun(inp, range(inp.w.B), 2)
    pu.assert_reports(pu.replay(inp, run, range(inp.w.B)))


def test_zero_weights_is_plain_greedy_on_gpu():
    """lambda = beta = 0: the GPU labels are the argmax of the raw logits
    (checked with torch's own bf16 matmul reference on the GPU's inputs)."""
    w = synth.scaled(synth.WORKLOADS[1], B=4, T=13, lam=0.0, beta=0.0)
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(4), 2, capture_steps=13 * 5)
    rows = run.cap_rows.cpu().numpy()
    Ef = torch.from_numpy(synth.bf16_to_f32(inp.E)).double()
    Wf = torch.from_numpy(synth.bf16_to_f32(inp.W)).double()
    for i in range(4):
        tok, fr, _ = run.emitted(i, 0)
        ev = _evaluations(tok, fr, w.T, w.max_sym)
        enc = torch.from_numpy(synth.bf16_to_f32(run.enc[0][i]))
        for s, (t, hist) in enumerate(ev):
            last = hist[-1] if hist else w.V
            x = torch.relu(enc[t] + Ef[last].float()).to(torch.bfloat16).double()
            lg = x @ Wf
            top2 = torch.topk(lg, 2).values
            y = int(torch.argmax(lg))
            chosen = int(tok[len(hist)]) if len(hist) < len(tok) and fr[len(hist)] == t else w.V
            if float(top2[0] - top2[1]) > pu.GAP_TOL:
                assert chosen == y, (i, s)


def test_tensor_core_and_cuda_core_kernels_agree():
    """The tcgen05 joint kernel and the CUDA-core kernel compute the same
    logits (to fp32 accumulation order) and the same decisions."""
    w = synth.scaled(synth.WORKLOADS[2], B=130, T=13, chunks=2)
    inp = pu.Inputs(w, lmA=synth.ngram_lm(11, w.V, 4, 200_000, 1.1))
    S = w.T * w.max_sym
    a = pu.GpuRun(inp, range(w.B), 1, capture_steps=S)
    b = pu.GpuRun(inp, range(w.B), 1, capture_steps=S, joint_kind=1)
    la, lb = a.cap_logits.cpu().numpy(), b.cap_logits.cpu().numpy()
    ra, rb = a.cap_rows.cpu().numpy(), b.cap_rows.cpu().numpy()
    same = (ra == rb).all(axis=2)  # rows evaluated at the same state
    assert same[0].all()
    diff = np.abs(la - lb)[same]
    assert diff.max() < 1e-3, diff.max()
    agree = sum(np.array_equal(a.emitted(i, 0)[0], b.emitted(i, 0)[0]) for i in range(w.B))
    assert agree >= w.B - 2  # sequences may part only at near ties
    pu.assert_reports(pu.replay(inp, a, [0, 64, 129]))


def test_launch_options_and_replay_do_not_change_results():
    """Programmatic dependent launch on/off and timing replays between chunks
    give bit-identical decodes; every tensor-core tile width passes parity
    (a different tile split only reorders the fp32 log-sum-exp)."""
    w = synth.scaled(synth.WORKLOADS[1], B=150, chunks=3)
    inp = pu.Inputs(w, lmA=synth.ngram_lm(13, w.V, 4, 300_000, 1.1), ph=synth.phrases(13, w.V, 300, 2, 6, 0.2))
    base = pu.GpuRun(inp, range(w.B), 3)
    exact = {"pdl off": pu.GpuRun(inp, range(w.B), 3, options={"pdl": 0}),
             "replays": pu.GpuRun(inp, range(w.B), 3, between_chunks=lambda d: (d.replay(0, 3), d.replay(1, 3)))}
    for name, r in exact.items():
        for c in range(3):
            for i in range(w.B):
                for x, y in zip(r.emitted(i, c), base.emitted(i, c)):
                    assert np.array_equal(x, y), (name, c, i)
    for bn in (64, 128, 256):
        r = pu.GpuRun(inp, range(w.B), 3, options={"joint_bn": bn})
        pu.assert_reports(pu.replay(inp, r, [0, 77, 149]))
        for c in range(3):
            for i in range(0, w.B, 7):
                np.testing.assert_allclose(r.emitted(i, c)[2][:5], base.emitted(i, c)[2][:5], atol=1e-5)
    assert base.dec.replay(0, 1, count_bytes=True) > 0


def test_status_errors_leave_decoder_usable():
    import paper_2609_14991_gb300 as tsd

    w = synth.scaled(synth.WORKLOADS[0], B=2, T=8)
    inp = pu.Inputs(w)
    run = pu.GpuRun(inp, range(2), 1)
    dec = run.dec
    enc = torch.zeros((2, 8, w.H), dtype=torch.int16, device="cuda")
    with pytest.raises(tsd.TsdError) as e:
        dec.open()  # both slots in use
    assert e.value.status == tsd.TSD_ESTATE
    with pytest.raises(tsd.TsdError) as e:
        dec.decode_chunk([0, 0], enc, 0.1, 0.1)
    assert e.value.status == tsd.TSD_EINVAL
    with pytest.raises(tsd.TsdError) as e:
        dec.decode_chunk([0, 1], torch.zeros((2, 9, w.H), dtype=torch.int16, device="cuda"), 0.1, 0.1)
    assert e.value.status == tsd.TSD_EINVAL
    dec.close(1)
    with pytest.raises(tsd.TsdError) as e:
        dec.decode_chunk([0, 1], enc, 0.1, 0.1)
    assert e.value.status == tsd.TSD_ESTATE
    with pytest.raises(tsd.TsdError):
        dec.close(1)
    s = dec.open()
    out = dec.decode_chunk([0, s], enc, 0.1, 0.1)
    torch.cuda.synchronize()
    assert out.counts.cpu().numpy().min() >= 0
