"""Parity harness: the CUDA decoder against the oracle on the same seeded
inputs (test infrastructure; imports the oracle).

The GPU decodes every stream; the oracle then walks a sample of the streams
through the same chunks, checking at every evaluation that the GPU's choice
is the oracle's argmax or within GAP_TOL of it (near ties may go either way),
that the fused score of each emitted label is within SCORE_TOL, and it
follows the GPU's choice.  After every chunk the GPU's LM state and trie node
must stand for exactly the tuples the oracle derives from the emitted labels.
"""
from __future__ import annotations

import concurrent.futures
import os
import sys
from typing import Dict, List, Optional, Sequence

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import oracle  # noqa: E402
import synth  # noqa: E402

GAP_TOL = 1e-3  # a choice that loses by less than this to the oracle's argmax is a near tie
SCORE_TOL = 1e-4  # fused scores, fp32 on the GPU vs double in the oracle
LOGIT_TOL = 2e-2  # joint logits vs the oracle's double product of the same bf16 inputs


def bf16_bits(x) -> np.ndarray:
    """float32 -> bf16 bit patterns, round to nearest even."""
    u = np.asarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    keep, rest = u >> 16, u & 0xFFFF
    keep = keep + ((rest > 0x8000) | ((rest == 0x8000) & (keep & 1 == 1)))
    return keep.astype(np.uint16)


class Inputs:
    def __init__(self, w: synth.Workload, lmA=None, ph=None, with_lm=True, with_boost=True):
        self.w = w
        self.E, self.W = synth.joint_weights(w)
        self.lmA = lmA if lmA is not None else (synth.lm_for(w) if with_lm else None)
        self.ph = ph if ph is not None else (synth.phrases_for(w) if with_boost else None)
        self.lam = w.lam if self.lmA is not None else 0.0
        self.beta = w.beta if self.ph is not None else 0.0


def trie_tuple(bo: oracle.Boost, hist: Sequence[int], rho: int):
    g = list(hist[rho:])
    m = bo.match(g) if g else 0
    return tuple(g[len(g) - m:]) if m else ()


class GpuRun:
    """Decodes `streams` (stream ids of the workload) for `chunks` chunks."""

    def __init__(self, inp: Inputs, streams: Sequence[int], chunks: int, T: Optional[int] = None,
                 capture_steps: int = 0, graphs: bool = True, joint_kind: int = 0, options=None,
                 between_chunks=None):
        import torch

        import paper_2609_14991_gb300 as tsd

        w = inp.w
        self.T = T or w.T
        self.streams = list(streams)
        dev = torch.device("cuda", 0)
        Wt = torch.from_numpy(inp.W.view(np.int16)).to(dev)
        Et = torch.from_numpy(inp.E.view(np.int16)).to(dev)
        self.lm = tsd.NGram.from_arrays(inp.lmA) if inp.lmA is not None else None
        self.bo = tsd.Boost.from_phrases(w.V, inp.ph, w.bonus) if inp.ph is not None else None
        n = len(self.streams)
        self.K = w.beam
        self.dec = tsd.Decoder(w.V, w.H, Wt, Et, lm=self.lm, boost=self.bo, max_symbols=w.max_sym, beam_k=w.beam,
                               max_streams=n, max_T=self.T)
        self.dec.set_graphs(graphs)
        if joint_kind:
            self.dec.set_joint_kernel(joint_kind)
        for k, v in (options or {}).items():
            self.dec.set_option(k, v)
        self.slots = [self.dec.open() for _ in range(n)]
        self.cap_logits = self.cap_rows = None
        M = n * self.K
        if capture_steps:
            self.cap_logits = torch.zeros((capture_steps, M, w.N), dtype=torch.float32, device=dev)
            self.cap_rows = torch.full((capture_steps, M, 4), -7, dtype=torch.int32, device=dev)
            self.dec.debug_capture(self.cap_logits, self.cap_rows, capture_steps)
        self.beam_sel: List[np.ndarray] = []   # per chunk: kept candidates [T, M, 4]
        self.beam_hyps: List[List] = []        # per chunk: per stream [(labels, score)]
        self.chunks: List[Dict] = []
        self.enc: List[np.ndarray] = []
        self.states: List[List] = []
        for c in range(chunks):
            enc = synth.enc_chunk(w, self.streams, c, self.T)
            et = torch.from_numpy(enc.view(np.int16)).to(dev)
            out = self.dec.decode_chunk(self.slots, et, inp.lam, inp.beta)
            torch.cuda.synchronize()
            cnt = out.counts.cpu().numpy()
            tok, fr, sc = out.tokens.cpu().numpy(), out.frames.cpu().numpy(), out.scores.cpu().numpy()
            self.chunks.append({"count": cnt, "tok": tok, "frame": fr, "score": sc})
            self.enc.append(enc)
            self.states.append([self.dec.state(s) for s in self.slots])
            if self.K > 1:
                if capture_steps:
                    self.beam_sel.append(self.cap_rows.cpu().numpy().copy())
                self.beam_hyps.append([self.dec.hyps(s) for s in self.slots])
            if between_chunks is not None:
                between_chunks(self.dec)
        self.dec.check()  # no bounded device wait expired

    def emitted(self, i: int, c: int):
        d = self.chunks[c]
        k = int(d["count"][i])
        return d["tok"][i, :k], d["frame"][i, :k], d["score"][i, :k]


def replay_stream(inp: Inputs, run: GpuRun, i: int, olm, obo, model, chunks: Optional[int] = None) -> Dict:
    """Oracle replay of the i-th stream of a GPU run over its first `chunks`
    chunks (all by default)."""
    w = inp.w
    st = oracle.Stream(w.V)
    rep_all = {"steps": 0, "mismatch": 0, "near_tie": 0, "max_score_diff": 0.0, "min_gap": np.inf,
               "inconsistent": 0, "state_errors": []}
    for c in range(len(run.chunks) if chunks is None else min(chunks, len(run.chunks))):
        tok, fr, sc = run.emitted(i, c)
        _, _, _, rep = oracle.decode_chunk(st, model, olm, obo, run.enc[c][i], inp.lam, inp.beta, w.max_sym,
                                           follow=(tok, fr, sc), gap_tol=GAP_TOL)
        rep_all["steps"] += int(rep[oracle.REP_STEPS])
        rep_all["mismatch"] += int(rep[oracle.REP_MISMATCH])
        rep_all["near_tie"] += int(rep[oracle.REP_NEAR_TIE])
        rep_all["max_score_diff"] = max(rep_all["max_score_diff"], float(rep[oracle.REP_MAX_SCORE_DIFF]))
        rep_all["min_gap"] = min(rep_all["min_gap"], float(rep[oracle.REP_MIN_GAP]))
        rep_all["inconsistent"] += int(rep[oracle.REP_INCONSISTENT])
        hist = st.history()
        lm_state, trie_node, last = run.states[c][i]
        want_last = hist[-1] if hist else w.V
        if last != want_last:
            rep_all["state_errors"].append((c, "last", last, want_last))
        if olm is not None:
            got = run.lm.state_tuple(lm_state)
            want = olm.state(hist)
            if got != want:
                rep_all["state_errors"].append((c, "lm", got, want))
        if obo is not None:
            got = run.bo.node_tuple(trie_node)
            want = trie_tuple(obo, hist, st.rho())
            if got != want:
                rep_all["state_errors"].append((c, "trie", got, want))
    return rep_all


def oracle_models(inp: Inputs):
    w = inp.w
    olm = oracle.LM.from_arrays(inp.lmA) if inp.lmA is not None else None
    obo = oracle.Boost.from_phrases(w.V, inp.ph, w.bonus) if inp.ph is not None else None
    model = oracle.Model(w.V, w.H, inp.E, inp.W)
    return olm, obo, model


def replay(inp: Inputs, run: GpuRun, sample: Sequence[int], threads: Optional[int] = None,
           chunks: Optional[int] = None, models=None) -> List[Dict]:
    olm, obo, model = models or oracle_models(inp)
    threads = threads or min(len(sample), os.cpu_count() or 4)
    with concurrent.futures.ThreadPoolExecutor(max_workers=threads) as ex:
        return list(ex.map(lambda i: replay_stream(inp, run, i, olm, obo, model, chunks), sample))


def captured_logit_error(run: GpuRun, model, steps: int, rows: Sequence[int], threads: Optional[int] = None):
    """Largest |GPU logit - oracle logit| over the captured steps and rows of
    the run's last chunk (capture keeps the last decode call's steps): every
    label of every (step, row) the row was evaluated at, against the oracle's
    double product of the same bf16 inputs (joint_logits of the captured
    frame and previous label).  Returns (max error, rows checked)."""
    caps = run.cap_rows.cpu().numpy()
    logits = run.cap_logits.cpu().numpy()
    K = run.K
    jobs = [(s, r) for s in range(min(steps, caps.shape[0])) for r in rows if caps[s, r, 0] >= 0]

    def one(job):
        s, r = job
        t, last = int(caps[s, r, 0]), int(caps[s, r, 1])
        want = model.joint_logits(run.enc[-1][r // K][t], last)
        return float(np.abs(logits[s, r] - want).max())

    threads = threads or (os.cpu_count() or 4)
    with concurrent.futures.ThreadPoolExecutor(max_workers=threads) as ex:
        errs = list(ex.map(one, jobs))
    return (max(errs) if errs else 0.0), len(jobs)


def assert_reports(reps: List[Dict]):
    for r in reps:
        assert r["inconsistent"] == 0, r
        assert r["mismatch"] == 0, r
        assert r["max_score_diff"] <= SCORE_TOL, r
        assert not r["state_errors"], r["state_errors"][:5]
        assert r["steps"] > 0


def replay_beam_stream(inp: Inputs, run: GpuRun, i: int, olm, obo, model) -> Dict:
    """Oracle replay of the i-th stream of a beam run: every frame's kept
    candidates are checked and followed; after every chunk the surviving
    label sequences must be the oracle's, in the same order, with scores
    within SCORE_TOL per frame decoded so far."""
    w = inp.w
    K = w.beam
    st = oracle.Stream(w.V)
    out = {"steps": 0, "mismatch": 0, "near_tie": 0, "max_score_diff": 0.0, "inconsistent": 0, "state_errors": []}
    frames = 0
    for c in range(len(run.chunks)):
        sel = run.beam_sel[c][:, i * K:(i + 1) * K, :]  # [steps, K, 4]: one row per expansion
        rep = oracle.beam_chunk_follow(st, model, olm, obo, run.enc[c][i], inp.lam, inp.beta, K,
                                       sel[:, :, 0], sel[:, :, 1], sel[:, :, 2].view(np.float32), GAP_TOL,
                                       S=w.max_sym)
        frames += run.T
        out["steps"] += int(rep[oracle.REP_STEPS])
        out["mismatch"] += int(rep[oracle.REP_MISMATCH])
        out["near_tie"] += int(rep[oracle.REP_NEAR_TIE])
        out["inconsistent"] += int(rep[oracle.REP_INCONSISTENT])
        out["max_score_diff"] = max(out["max_score_diff"], float(rep[oracle.REP_MAX_SCORE_DIFF]))
        want = st.beam_hyps(with_rho=True)
        got = run.beam_hyps[c][i]
        if [g[0] for g in got] != [h[0] for h in want]:
            out["state_errors"].append((c, "hyp sequences", len(got), len(want)))
            continue
        for (gy, gs), (wy, ws, _) in zip(got, want):
            if abs(gs - ws) > SCORE_TOL * frames:
                out["state_errors"].append((c, "hyp score", gs, ws))
        # the first hypothesis's LM state and trie node
        lm_state, trie_node, last = run.states[c][i]
        wy, _, wrho = want[0]
        if last != (wy[-1] if wy else w.V):
            out["state_errors"].append((c, "last", last))
        if olm is not None and run.lm.state_tuple(lm_state) != olm.state(wy):
            out["state_errors"].append((c, "lm"))
        if obo is not None and run.bo.node_tuple(trie_node) != trie_tuple(obo, wy, wrho):
            out["state_errors"].append((c, "trie"))
    return out


def replay_beam(inp: Inputs, run: GpuRun, sample: Sequence[int], threads: Optional[int] = None) -> List[Dict]:
    olm, obo, model = oracle_models(inp)
    threads = threads or min(len(sample), os.cpu_count() or 4)
    with concurrent.futures.ThreadPoolExecutor(max_workers=threads) as ex:
        return list(ex.map(lambda i: replay_beam_stream(inp, run, i, olm, obo, model), sample))
