"""Benchmark of the fused streaming decode step (one JSON line on stdout).

A step is one decode_chunk call: a 13-frame encoder chunk (the paper's
1040 ms look-ahead at 80 ms frames) for all B streams, through the whole hot
path -- joint GEMM, log-softmax, LM and phrase-boost fusion, greedy
selection and state advance, T*max_symbols label steps.

Workload (default, the largest configuration that fits one GPU): B=1024
streams, H=1024, V=4096+blank, a 10-gram LM with ~100M n-grams over Zipf(1.05)
unigrams, 50,000 boost phrases, lambda=0.6, beta=1.5, greedy with at most 5
labels per frame; synthetic seeded data.  The same run also times the
workload at B = 1, 16 and 128 streams (latency against throughput).
--config 0..3 selects the smaller workloads.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config C]

The reference arm (--impl reference) times the CPU oracle on this host's
cores on a bounded sample of the same workload and reports the same metric.
Under torchrun each rank decodes its own B streams (streams are independent:
weak scaling, no collective on the data path); rank 0 prints.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "fused decode encoder-frames/sec over B streams"
UNIT = "frames/s"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(PEAKS_FALLBACK), "fallback"


# DRAM traffic per launch (dram__bytes_read.sum + dram__bytes_write.sum) from
# one ncu capture of the kernel inside this bench's graph, keyed by (config,
# streams, kernel), with the hash of the kernel's sources (comments and blank
# space aside) at capture time: a changed kernel reports null until it is
# captured again.  The captures and
# their commands are summarised under profiles/.
KERNEL_SOURCES = {
    "joint": ["joint_greedy.cu", "joint_tc.h", "tc_common.cuh", "decoder.h", "internal.h"],
    "row_ep": ["row_fused.cu", "row_common.cuh", "decoder.h", "internal.h"],  # fusion_path 1
    "row_fz": ["row_stream.cu", "row_common.cuh", "decoder.h", "internal.h"],  # fusion_path 0
    "egemm": ["encoder_gemm.cu", "encoder.cu", "encoder.h", "tc_common.cuh", "internal.h"],
}
# keyed by (config, streams, kernel, fusion_path)
TRAFFIC = {
    (4, 1024, "row", 1): (10575616, "cadf021270fce30e"),
    (4, 1024, "joint", 0): (11052032, "b67360efb4e1a0ff"),
    (4, 1024, "row", 0): (29132544, "c491ab3e394847c6"),
}


def kernel_source_hash(kernel: str) -> str:
    """Hash of the kernel's sources without comments and blank space, so that
    only a change of code voids a recorded capture."""
    import hashlib
    import re

    h = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2609_14991_gb300", "csrc", f), encoding="utf-8") as fh:
            src = fh.read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)  # block comments
        src = re.sub(r"//[^\n]*", " ", src)  # line comments
        h.update(" ".join(src.split()).encode())
    return h.hexdigest()[:16]


# The encoder GEMMs' DRAM traffic per chunk (every k_egemm launch of one
# chunk step, summed), keyed by (encoder shape, streams, frames per chunk).
ENC_TRAFFIC = {}  # none recorded for the current encoder GEMM build


def recorded_traffic(w: synth.Workload, kernel: str, key=None, path=None):
    rec = (ENC_TRAFFIC if key else TRAFFIC).get(key or (w.cfg, w.B, kernel, path))
    if kernel == "row":
        kernel = "row_ep" if path == 1 else "row_fz"
    if rec is None or rec[1] != kernel_source_hash(kernel):
        return None
    return rec[0]


def workload_config(w: synth.Workload, lm_total: int, n_phr: int):
    return {"workload": f"cfg{w.cfg} {w.name}", "B_per_gpu": w.B, "T": w.T, "H": w.H, "V": w.V,
            "lm_order": w.lm_order, "lm_ngrams": lm_total, "boost_phrases": n_phr, "lambda": w.lam,
            "beta": w.beta, "max_symbols": w.max_sym, "beam": w.beam,
            "data": "synthetic seeded (Philox4x32-10): enc, E ~ N(0,1), W_out ~ N(0, 3/sqrt(H)); "
                    "normalized absolute-discount backoff LM over Zipf unigrams; random phrases"}


class Clocks:
    """Samples SM clocks and throttle reasons with nvidia-smi during a region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower() in ("active", "0x1", "1", "yes"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def rank_streams(rank: int, B: int):
    """The global stream ids rank `rank` decodes: its own block of B (streams
    are independent, so ranks share no data and exchange nothing)."""
    return list(range(rank * B, (rank + 1) * B))


def max_over_ranks(values, ws: int, device=None):
    """Element-wise maximum of a list of floats over all ranks (identity at
    ws == 1): the job's time is that of its slowest rank."""
    if ws <= 1:
        return [float(v) for v in values]
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t.cpu().tolist()]


def latency_stats(step_ms):
    a = np.asarray(step_ms, dtype=np.float64)
    return {"p50_ms": float(np.percentile(a, 50)), "p99_ms": float(np.percentile(a, 99)),
            "max_ms": float(a.max()), "steps": int(a.size)}


def workload(cfg: int, streams=None) -> synth.Workload:
    """The workload of a config, optionally with another stream count B."""
    w = synth.WORKLOADS[cfg]
    if streams and streams != w.B:
        w = synth.scaled(w, B=int(streams), name=w.name.replace(f"B={w.B}", f"B={int(streams)}"))
    return w


def extra_lms(w: synth.Workload, k: int):
    """k further LMs for the several-LM workload: the config's recipe at half
    its n-gram budget with other seeds, each entering Eq. 1 with weight
    lambda * 0.5 (the config's own LM keeps weight lambda)."""
    return [(synth.ngram_lm(w.lm_seed + 1000 * (i + 1), w.V, w.lm_order, w.lm_total // 2, w.zipf), 0.5)
            for i in range(k)]


def pred_weights(w: synth.Workload, D: int):
    """The stateful form's prediction network (D LSTM units) and joint
    projections; encoder frames stay H wide (H_enc = H)."""
    return synth.pred_weights(w, D=D, Henc=w.H) if D else None


def variant_config(args, w, extra):
    """The config keys that name a variant of the workload."""
    out, names = {}, []
    if extra:
        out.update(lms=1 + len(extra), lm_weights=[1.0] + [wt for _, wt in extra])
        names.append(f"+ {len(extra)} more LMs (half size, weight 0.5)")
    if args.prune_k:
        out["prune_k"] = args.prune_k
        names.append(f"fusion pruned to the acoustic top {args.prune_k}")
    if w.beam == 1 and not args.prune_k and not extra:
        out["fusion_path"] = 1 if args.fusion_path == 1 else 0  # the decoder's default: 0
    if args.pred:
        out["prediction_network"] = {"kind": "1-layer LSTM over the previous label", "D": args.pred, "H_enc": w.H}
        names.append(f"stateful form: LSTM prediction network D={args.pred} + joint projections")
    if args.encoder:
        e = synth.ENCODERS[args.encoder]
        out["encoder"] = {"shape": e.name, "d": e.d, "blocks": e.layers, "heads": e.heads, "ff": e.ff,
                          "kernel": e.kernel, "left_context_frames": e.left, "chunk_frames": w.T,
                          "features": f"{e.stack} x {e.feat} log-mel-like bins per 80 ms frame"}
        names.append(f"with the cache-aware encoder chunk step ({e.name}-shaped)")
    if names:
        out["workload"] = f"cfg{w.cfg} {w.name}, " + "; ".join(names)
    return out


def oracle_models(w, inp_lm, inp_ph, E, W, extra=(), pred=None):
    import oracle

    olm = oracle.LM.from_arrays(inp_lm) if inp_lm is not None else None
    if extra:
        olm = [(olm, 1.0)] + [(oracle.LM.from_arrays(a), wt) for a, wt in extra]
    obo = oracle.Boost.from_phrases(w.V, inp_ph, w.bonus) if inp_ph is not None else None
    pn = oracle.PredNet(w.V, w.H, pred) if pred is not None else None
    return olm, obo, oracle.Model(w.V, w.H, E, W), pn


def oracle_baseline(w, models, streams, chunks, threads=None, prune_k=0, encoder=None):
    """Times the oracle (as it stands) decoding `streams` x `chunks` of the
    workload on this host's cores; returns (frames/s, cores, sample, seconds).
    encoder: (oracle Encoder, its cfg) to run the encoder chunk step first."""
    import concurrent.futures

    import oracle

    threads = threads or len(os.sched_getaffinity(0))
    olm, obo, model, pn = models
    if encoder is None:
        encs = {c: synth.enc_chunk(w, streams, c) for c in range(chunks)}
    else:
        from oracle import encoder as oe

        ecfg = encoder[1]
        feats = {c: synth.features(ecfg, streams, c * w.T, w.T) for c in range(chunks)}

    def one(i):
        st = oracle.Stream(w.V)
        est = oe.EncoderStream(ecfg) if encoder is not None else None
        for c in range(chunks):
            frames = encs[c][i] if encoder is None else oe.encode_chunk(encoder[0], est, feats[c][i])
            oracle.decode_chunk(st, model, olm, obo, frames, w.lam, w.beta, w.max_sym, prune_k=prune_k,
                                pred=pn)

    t0 = time.perf_counter()
    with concurrent.futures.ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(one, range(len(streams))))
    dt = time.perf_counter() - t0
    frames = len(streams) * chunks * w.T
    used = min(threads, len(streams))
    sample = f"{len(streams)} streams x {chunks} chunks x {w.T} frames of the same workload ({frames} frames)"
    return frames / dt, used, sample, dt


def oracle_encoder(args):
    """(oracle encoder, its cfg) for --encoder, else None."""
    if not args.encoder:
        return None
    from oracle import encoder as oe

    cfg = synth.ENCODERS[args.encoder]
    return oe.Encoder(synth.encoder_weights(cfg)), cfg


def run_reference(args, w):
    """The reference arm: the CPU oracle on this host's cores."""
    ws, rank, _ = _dist()
    if rank != 0:
        return
    lmA = synth.lm_for(w)
    ph = synth.phrases_for(w)
    E, W = synth.joint_weights(w)
    n_str = args.ref_streams
    extra = extra_lms(w, args.extra_lms) if args.extra_lms else []
    models = oracle_models(w, lmA, ph, E, W, extra, pred_weights(w, args.pred))
    enc_o = oracle_encoder(args)
    if enc_o is not None:
        n_str = min(n_str, 16)  # the encoder step dominates the oracle's time
    # warm-up steps, then K timed steps; each step decodes a bounded sample
    for _ in range(args.warmup):
        oracle_baseline(w, models, list(range(2)), 1, prune_k=args.prune_k, encoder=enc_o)
    vals, dts = [], []
    for k in range(args.steps):
        v, cores, sample, dt = oracle_baseline(w, models, list(range(k * n_str, (k + 1) * n_str)), 1,
                                               prune_k=args.prune_k, encoder=enc_o)
        vals.append(v)
        dts.append(dt)
    value = float(np.mean(vals))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * float(np.mean(dts)),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": dict(workload_config(w, lmA.total + sum(a.total for a, _ in extra), ph.n if ph else 0),
                           **variant_config(args, w, extra)),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"per step: {sample}"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def stream_sweep(args, w, tsd, dev, stream, W, E, lm, lms, bo, pw, flush):
    """Frames/s and chunk latency of the same workload at the stream counts in
    args.sweep (one decoder each, same tables), K timed chunks after W
    warm-up chunks, L2 flushed before every timed chunk."""
    import torch

    out = []
    for B in args.sweep:
        if B == w.B or B < 1:
            continue
        d = tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev),
                        torch.from_numpy(E.view(np.int16)).to(dev), lm=None if lms else lm, lms=lms, boost=bo,
                        max_symbols=w.max_sym, beam_k=w.beam, max_streams=B, max_T=w.T, prune_k=args.prune_k,
                        pred=pw)
        if w.beam == 1 and not args.prune_k and not lms and getattr(args, "fusion_path_given", False):
            d.set_option("fusion_path", args.fusion_path)  # else the decoder's default for B streams
        sl = np.array([d.open() for _ in range(B)], dtype=np.int32)
        encs = [torch.from_numpy(synth.enc_chunk(w, range(B), c % w.chunks).view(np.int16)).to(dev)
                for c in range(args.warmup + args.steps)]
        o = d.alloc_out(B, w.T)
        op = (o.tokens.data_ptr(), o.frames.data_ptr(), o.scores.data_ptr(), o.counts.data_ptr())
        for c in range(args.warmup):
            d.decode_chunk_raw(sl, encs[c].data_ptr(), w.T, w.lam, w.beta, op, stream.cuda_stream)
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        for k, (a, b) in enumerate(ev):
            flush.zero_()
            a.record(stream)
            d.decode_chunk_raw(sl, encs[args.warmup + k].data_ptr(), w.T, w.lam, w.beta, op, stream.cuda_stream)
            b.record(stream)
        torch.cuda.synchronize()
        d.check()
        per = [a.elapsed_time(b) for a, b in ev]
        out.append({"B": B, "value": B * w.T * args.steps / (sum(per) / 1000.0), "ms_per_chunk": sum(per) / len(per),
                    **{k: v for k, v in latency_stats(per).items() if k != "steps"}})
        del d
    return out


def run_ours(args, w):
    import torch

    import paper_2609_14991_gb300 as tsd

    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    if ws > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream()

    lmA = synth.lm_for(w)
    ph = synth.phrases_for(w)
    E, W = synth.joint_weights(w)
    streams = rank_streams(rank, w.B)
    lm = tsd.NGram.from_arrays(lmA) if lmA is not None else None
    extra = extra_lms(w, args.extra_lms) if args.extra_lms else []
    lms = [(lm, 1.0)] + [(tsd.NGram.from_arrays(a), wt) for a, wt in extra] if extra else None
    bo = tsd.Boost.from_phrases(w.V, ph, w.bonus) if ph is not None else None
    pw = pred_weights(w, args.pred)
    dec = tsd.Decoder(w.V, w.H, torch.from_numpy(W.view(np.int16)).to(dev), torch.from_numpy(E.view(np.int16)).to(dev),
                      lm=None if lms else lm, lms=lms, boost=bo, max_symbols=w.max_sym, beam_k=w.beam,
                      max_streams=w.B, max_T=w.T, prune_k=args.prune_k, pred=pw)
    greedy1 = w.beam == 1 and not args.prune_k and not extra  # greedy decoding with at most one LM
    if greedy1:
        args.fusion_path_given = args.fusion_path is not None
        if args.fusion_path is None:  # the decoder's default: the streaming form
            args.fusion_path = 0
        dec.set_option("fusion_path", args.fusion_path)
    for kv in args.set or []:
        k, v = kv.split("=")
        dec.set_option(k, int(v))
    slots = [dec.open() for _ in range(w.B)]
    slots_np = np.array(slots, dtype=np.int32)
    n_chunks = args.warmup + args.steps + 1
    encoder = None
    if args.encoder:
        # the cache-aware encoder chunk step runs first in every step; its
        # frames are the decoder's input
        ecfg = synth.ENCODERS[args.encoder]
        need = pw.Henc if pw is not None else w.H
        if ecfg.d != need or w.T > 32:
            raise SystemExit(f"--encoder {args.encoder}: d={ecfg.d} must equal the decoder's input width {need} "
                             f"and chunks must be <= 32 frames")
        encoder = tsd.Encoder(synth.encoder_weights(ecfg), max_streams=w.B, max_chunk=w.T)
        eslots = np.array([encoder.open() for _ in range(w.B)], dtype=np.int32)
        encs = [torch.from_numpy(synth.features(ecfg, streams, (c % w.chunks) * w.T, w.T).view(np.int16)).to(dev)
                for c in range(n_chunks)]
        enc_frames = torch.empty((w.B, w.T, ecfg.d), dtype=torch.int16, device=dev)
    else:
        encs = [torch.from_numpy(synth.enc_chunk(w, streams, c % w.chunks).view(np.int16)).to(dev)
                for c in range(n_chunks)]
    out = dec.alloc_out(w.B, w.T)
    outp = (out.tokens.data_ptr(), out.frames.data_ptr(), out.scores.data_ptr(), out.counts.data_ptr())
    sh = stream.cuda_stream
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev)  # > 129 MB L2

    def step(c, src=None):
        src = encs[c] if src is None else src
        if encoder is not None:
            encoder.encode_chunk_raw(eslots, src.data_ptr(), w.T, enc_frames.data_ptr(), sh)
            dec.decode_chunk_raw(slots_np, enc_frames.data_ptr(), w.T, w.lam, w.beta, outp, sh)
        else:
            dec.decode_chunk_raw(slots_np, src.data_ptr(), w.T, w.lam, w.beta, outp, sh)

    def barrier():
        torch.cuda.synchronize()
        if ws > 1:
            import torch.distributed as dist

            dist.barrier()
        torch.cuda.synchronize()

    def timed_loop(first_chunk):
        starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        barrier()
        t0 = time.perf_counter()
        for k in range(args.steps):
            flush.zero_()  # L2 flush, outside the step's events
            starts[k].record(stream)
            step(first_chunk + k)
            ends[k].record(stream)
        barrier()
        wall = time.perf_counter() - t0
        per = [s.elapsed_time(e) for s, e in zip(starts, ends)]
        return float(sum(per)), wall, per

    # clocks and throttle reasons are sampled from here to the end of the GPU
    # work (the timed steps, their instrumented replay, the end-to-end steps
    # and the stream sweep), so the sample spans more than the short timed region
    clk = Clocks(local).__enter__()
    # warm-up (captures the chunk graph)
    for c in range(args.warmup):
        step(c)
    barrier()
    # timed region: K steps through the captured graph, no instrumentation
    t_ms, wall, step_ms = timed_loop(args.warmup)
    # the same K steps again with a CUDA event recorded at every kernel
    # boundary inside the graph: per-kernel device time for the roofline
    dec.set_timing(True)
    if encoder is not None:
        encoder.set_timing(True)
    for c in range(2):
        step(args.warmup + c)  # captures the two event-carrying graphs
    barrier()
    dec.timing(reset=True)
    dec.timed_bytes(reset=True)
    if encoder is not None:
        encoder.timing(reset=True)
    t_inst_ms, _, _ = timed_loop(args.warmup)
    kernel_ms, kernel_n = dec.timing(reset=True)
    row_timed_bytes = dec.timed_bytes(reset=True)
    dec.set_timing(False)
    enc_ms, enc_n = encoder.timing(reset=True) if encoder is not None else ({}, {})
    if encoder is not None:
        encoder.set_timing(False)
    t_ms, t_inst_ms = max_over_ranks([t_ms, t_inst_ms], ws, dev)
    frames = ws * w.B * w.T * args.steps
    value = frames / (t_ms / 1000.0)

    # end to end through the public API with host buffers: every step's H2D
    # copy of its chunk from pinned memory, the decode and the D2H of every
    # output are inside the region.  The inputs are double-buffered: chunk
    # k+1's copy runs on a copy stream while chunk k is decoded.
    host_enc = [e.cpu().pin_memory() for e in encs[-min(len(encs), 8):]]
    dev_enc = [torch.empty_like(encs[0]) for _ in range(2)]
    host_out = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in
                (out.tokens, out.frames, out.scores, out.counts)]
    e2e_steps = args.steps  # the same K steps as the headline
    copy_stream = torch.cuda.Stream()
    copied = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)

    def issue_copy(k):
        b = k % 2
        copy_stream.wait_event(e0 if k < 2 else consumed[b])  # buffer b's previous chunk is decoded
        with torch.cuda.stream(copy_stream):
            dev_enc[b].copy_(host_enc[k % len(host_enc)], non_blocking=True)
        copied[b].record(copy_stream)

    issue_copy(0)
    for k in range(e2e_steps):
        if k + 1 < e2e_steps:
            issue_copy(k + 1)
        stream.wait_event(copied[k % 2])
        step(0, dev_enc[k % 2])
        consumed[k % 2].record(stream)
        for h, d in zip(host_out, (out.tokens, out.frames, out.scores, out.counts)):
            h.copy_(d, non_blocking=True)
    e1.record(stream)
    barrier()
    e2e_ms = e0.elapsed_time(e1)
    h2d = int(dev_enc[0].numel() * dev_enc[0].element_size())
    d2h = int(sum(h.numel() * h.element_size() for h in host_out))
    e2e_val = ws * w.B * w.T * e2e_steps / (e2e_ms / 1000.0)

    # isolated kernel timings: the last chunk's final label step replayed
    # with CUDA events on the launching stream; "cold" flushes L2 before
    # every launch, "warm" launches back to back
    def replay_times(kind, reps=20):
        dec.replay(kind, 3)
        barrier()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for a, b in ev:
            flush.zero_()
            a.record(stream)
            dec.replay(kind, 1)
            b.record(stream)
        w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        w0.record(stream)
        dec.replay(kind, reps)
        w1.record(stream)
        barrier()
        cold = float(np.median([a.elapsed_time(b) for a, b in ev]))
        return cold, w0.elapsed_time(w1) / reps

    row_cold, row_warm = replay_times(0)
    joint_cold, joint_warm = replay_times(1)
    row_bytes = dec.replay(0, 1, count_bytes=True)
    joint_bytes = dec.replay(1, 1, count_bytes=True)

    sweep = None
    if args.sweep and ws == 1:
        sweep = stream_sweep(args, w, tsd, dev, stream, W, E, lm, lms, bo, pw, flush)
        sweep.append({"B": w.B, "value": value, "ms_per_chunk": t_ms / args.steps,
                      **{k: v for k, v in latency_stats(step_ms).items() if k != "steps"}})
        sweep.sort(key=lambda x: x["B"])

    # the other form of the greedy one-LM step on the same decoder and inputs
    # (fusion_path switched, graphs recaptured): its throughput and its two
    # kernels' production-graph figures
    alt = None
    if greedy1 and ws == 1 and not args.no_alt_path:
        alt_path = 1 - args.fusion_path
        dec.set_option("fusion_path", alt_path)
        for c in range(args.warmup):
            step(c)
        barrier()
        a_ms, _, _ = timed_loop(args.warmup)
        dec.set_timing(True)
        for c in range(2):
            step(args.warmup + c)
        barrier()
        dec.timing(reset=True)
        dec.timed_bytes(reset=True)
        timed_loop(args.warmup)
        a_kms, a_kn = dec.timing(reset=True)
        a_bytes = dec.timed_bytes(reset=True)
        dec.set_timing(False)
        a_tot = max(1e-9, sum(a_kms.values()))
        a_step = a_ms / args.steps
        a_shared = 0 if alt_path == 1 else w.V * ((4 if lmA is not None else 0) + (4 if ph is not None else 0))
        a_row_bytes = (a_bytes + a_shared * max(0, a_kn["row"] - args.steps)) / max(1, a_kn["row"])
        pk_a, pk_a_kind = peaks()
        a_joint_ms = a_step * (a_kms["joint"] / a_tot) / max(1e-9, a_kn["joint"] / args.steps)
        a_row_ms = a_step * (a_kms["row"] / a_tot) / max(1e-9, a_kn["row"] / args.steps)
        a_flop = 2.0 * w.B * w.H * (w.V + 1)
        alt = {"fusion_path": alt_path,
               "what": ("the same workload and decoder with the other form of the greedy one-LM step: "
                        + ("the LM level-0 term in the joint epilogue with a per-row correction list" if alt_path
                           else "the streaming form (the joint writes every logit + defaults, the row pass "
                                "applies the LM and trie terms)")),
               "value": w.B * w.T * args.steps / (a_ms / 1000.0), "unit": "frames/s", "ms_per_step": a_step,
               "joint": {"kernel": "k_joint_greedy<dense>" if alt_path else "k_joint_greedy<streaming>",
                         "avg_launch_ms": a_joint_ms, "achieved_tflops": a_flop / (a_joint_ms / 1000.0) / 1e12,
                         "frac": a_flop / (a_joint_ms / 1000.0) / 1e12 / pk_a["bf16_tflops_sustained"],
                         "peak_kind": f"{pk_a_kind} bf16 sustained"},
               "row": {"kernel": "k_row_ep" if alt_path else "k_row_fz", "avg_launch_ms": a_row_ms,
                       "bytes_per_launch": a_row_bytes, "achieved_gbs": a_row_bytes / (a_row_ms / 1000.0) / 1e9,
                       "frac": a_row_bytes / (a_row_ms / 1000.0) / 1e9 / pk_a["hbm_gbs"],
                       "peak_kind": f"{pk_a_kind} HBM copy"},
               "timing": "as the headline kernels: uninstrumented step time x device-time share / launches per step"}
    clk.__exit__(None, None, None)
    if rank != 0:
        return
    pk, pk_kind = peaks()
    M = w.B * w.beam
    flop_per_launch = 2.0 * M * w.H * (w.V + 1)
    total_ms = max(1e-9, sum(kernel_ms.values()) + sum(enc_ms.values()))
    share_joint = kernel_ms["joint"] / total_ms
    share_row = kernel_ms["row"] / total_ms
    share_pred = kernel_ms["pred"] / total_ms
    # In-graph figures: CUDA events at every kernel boundary on the launching
    # stream over the instrumented pass of the K timed steps.  A kernel timed
    # inside a long step takes the sustained bf16 peak.
    joint_ms = kernel_ms["joint"] / max(1, kernel_n["joint"])
    row_ms = kernel_ms["row"] / max(1, kernel_n["row"])
    # the greedy one-LM pass with the correction list (k_row_ep) reads no
    # shared V-wide row; the others read the call's unigram and root rows once
    # per launch
    ep = greedy1 and args.fusion_path != 0
    fz_stream = greedy1 and args.fusion_path == 0
    shared_rows = 0 if ep else w.V * ((4 * (1 + len(extra)) if lmA is not None else 0) + (4 if ph is not None else 0))
    row_launches_with_bias = kernel_n["row"] - args.steps  # the final row pass of a chunk builds no bias
    row_bytes_graph = row_timed_bytes + shared_rows * max(0, row_launches_with_bias)
    joint_roof = {"kernel": ("k_joint_greedy<dense>: joint GEMM (tcgen05) + epilogue applying Eq. 1 with the dense "
                             "LM row, log-softmax and selection partials") if ep else
                            ("k_joint_greedy<streaming>: joint GEMM (tcgen05) + epilogue writing logit + defaults "
                             "(TMA stores) and log-softmax partials") if fz_stream else
                            "k_joint_tc: joint GEMM (tcgen05) + fused log-softmax/selection epilogue",
                  "bound": "tensor", "unit": "TFLOP/s",
                  "achieved": flop_per_launch / (joint_ms / 1000.0) / 1e12,
                  "peak": pk["bf16_tflops_sustained"],
                  "peak_kind": f"{pk_kind} bf16 sustained (kernel timed inside the decode step)",
                  "algorithmic": f"2*M*H*(V+1) = {flop_per_launch:.4g} FLOP per launch (M={M} rows)",
                  "avg_launch_ms": joint_ms, "launches": kernel_n["joint"],
                  "traffic": recorded_traffic(w, "joint", path=args.fusion_path if greedy1 else None),
                  "bytes_per_launch": joint_bytes,
                  "share_of_device_time": share_joint,
                  "isolated": {"cold_l2_ms": joint_cold, "warm_l2_ms": joint_warm,
                               "achieved_cold": flop_per_launch / (joint_cold / 1000.0) / 1e12,
                               "achieved_warm": flop_per_launch / (joint_warm / 1000.0) / 1e12,
                               "peak": pk["bf16_tflops"], "peak_kind": f"{pk_kind} bf16 burst"}}
    joint_roof["frac"] = joint_roof["achieved"] / joint_roof["peak"]
    row_roof = {"kernel": "k_row_beam" if w.beam > 1 else ("k_row_ep" if ep else ("k_row_fz" if fz_stream else "k_row")),
                "what": ("decision from the tile partials and the correction list, LM/trie state advance, "
                         "the new state's correction list and mask, joint input") if ep else
                        ("the row's LM and trie deltas (every arc of its LM chain levels, its dense level-0 row, "
                         "the trie chain's children), argmax over the fused logits, state advance, joint input")
                        if fz_stream else
                        "selection merge, LM/trie state advance, joint input, fusion bias",
                "bound": "hbm", "unit": "GB/s",
                "achieved": row_bytes_graph / (kernel_ms["row"] / 1000.0) / 1e9,
                "peak": pk["hbm_gbs"], "peak_kind": f"{pk_kind} HBM copy",
                "algorithmic": (f"{row_bytes_graph / max(1, kernel_n['row']):.0f} B per launch on average, "
                                f"counted by the kernel per row (partials, the correction list read with its "
                                f"logits and written, the mask, row state, label searches, every arc of the LM "
                                f"chain levels 1.. and every child of the trie chain nodes, joint input)") if ep else
                               (f"{row_bytes_graph / max(1, kernel_n['row']):.0f} B per launch on average, "
                                f"counted by the kernel per evaluated row (the fused logits read back, partials, "
                                f"row state, label searches, joint input, every arc of the LM chain levels above "
                                f"0, the dense level-0 row, every child of the trie chain nodes) plus the shared "
                                f"unigram/root rows once per launch") if fz_stream else
                               (f"{row_bytes_graph / max(1, kernel_n['row']):.0f} B per launch on average, "
                                f"counted by the kernel per evaluated row (partials, row state, label searches, "
                                f"joint input, every arc of the LM chain levels and trie chain nodes) plus the "
                                f"shared unigram/root rows once per launch; the dense bias row is not counted"),
                "avg_launch_ms": row_ms, "launches": kernel_n["row"],
                "traffic": recorded_traffic(w, "row", path=args.fusion_path if greedy1 else None),
                "share_of_device_time": share_row,
                "isolated": {"what": "the chunk's last label step replayed with every row evaluated",
                             "bytes_per_launch": row_bytes, "cold_l2_ms": row_cold, "warm_l2_ms": row_warm,
                             "achieved_cold": row_bytes / (row_cold / 1000.0) / 1e9,
                             "achieved_warm": row_bytes / (row_warm / 1000.0) / 1e9}}
    row_roof["frac"] = row_roof["achieved"] / row_roof["peak"]
    # The instrumented pass serializes the kernels (an event between two
    # kernels ends their programmatic overlap) and adds the events' own cost,
    # so its per-launch times are upper bounds.  The same K steps without
    # instrumentation split by those device-time shares give each kernel's
    # time inside the production graph.
    mean_step_ms = t_ms / args.steps
    for roof_k, share, n_per_step, work in (
            (joint_roof, share_joint, kernel_n["joint"] / args.steps, flop_per_launch / 1e12),
            (row_roof, share_row, kernel_n["row"] / args.steps,
             row_bytes_graph / max(1, kernel_n["row"]) / 1e9)):
        ms_in_graph = mean_step_ms * share / max(1e-9, n_per_step)
        # the headline figures are the production graph's: the timed steps'
        # CUDA-event time (no instrumentation) apportioned by this kernel's
        # device-time share; the instrumented pass's own per-launch times stay
        # beside them (they are upper bounds: events between kernels end the
        # programmatic overlap and add their own cost)
        roof_k["serialized_with_kernel_events"] = {
            "what": "CUDA events at every kernel boundary inside the graph (second pass of the K steps, "
                    "programmatic launch off): per-launch device time",
            "avg_launch_ms": roof_k["avg_launch_ms"], "achieved": roof_k["achieved"], "frac": roof_k["frac"]}
        roof_k["avg_launch_ms"] = ms_in_graph
        roof_k["achieved"] = work / (ms_in_graph / 1000.0)
        roof_k["frac"] = roof_k["achieved"] / roof_k["peak"]
        roof_k["timing"] = ("avg_launch_ms = uninstrumented step time (CUDA events on the launching stream over the "
                            "K timed steps) x this kernel's share of device time (CUDA events at every kernel "
                            "boundary over a second pass of the same steps) / its launches per step")
    pred_roof = None
    if args.pred:
        # the stateful form's GEMMs per chunk: the encoder projection, an LSTM
        # gate GEMM per label step and after the last, a joint-input GEMM per step
        S = w.T * w.max_sym
        D = args.pred
        pred_flop = 2.0 * M * w.T * w.H * w.H + (S + 1) * 2.0 * M * (2 * D) * (4 * D) + S * 2.0 * M * D * w.H
        pred_chunk_ms = kernel_ms["pred"] / args.steps
        pred_roof = {"kernel": "k_gemm_tc: encoder projection, LSTM cell and joint-input GEMMs (tcgen05)",
                     "bound": "tensor", "unit": "TFLOP/s",
                     "achieved": pred_flop / (pred_chunk_ms / 1000.0) / 1e12,
                     "peak": pk["bf16_tflops_sustained"],
                     "peak_kind": f"{pk_kind} bf16 sustained (kernels timed inside the decode step)",
                     "algorithmic": f"{pred_flop:.4g} FLOP per chunk (M={M} rows, D={D}, S={S} label steps)",
                     "ms_per_chunk": pred_chunk_ms, "launches": kernel_n["pred"],
                     "traffic": None, "share_of_device_time": share_pred}
        pred_roof["frac"] = pred_roof["achieved"] / pred_roof["peak"]
        pred_roof["serialized_with_kernel_events"] = {
            "what": "CUDA events at every kernel boundary inside the graph (second pass, programmatic launch off)",
            "ms_per_chunk": pred_roof["ms_per_chunk"], "achieved": pred_roof["achieved"], "frac": pred_roof["frac"]}
        pred_roof["ms_per_chunk"] = mean_step_ms * share_pred
        pred_roof["achieved"] = pred_flop / (mean_step_ms * share_pred / 1000.0) / 1e12
        pred_roof["frac"] = pred_roof["achieved"] / pred_roof["peak"]
        pred_roof["timing"] = "uninstrumented step time x this class's share of device time (CUDA events)"
    enc_roof = None
    if encoder is not None:
        # the encoder's tensor-core GEMMs (subsampling, q/k/v, attention
        # output, the convolution module's pointwise maps, feed-forward)
        enc_flop = encoder.gemm_flops(w.B, w.T)
        share_enc = enc_ms["gemm"] / total_ms
        gemm_chunk_ms = enc_ms["gemm"] / args.steps
        enc_roof = {"kernel": "k_egemm: encoder GEMMs with fused bias/Swish/GLU/residual epilogues (tcgen05)",
                    "bound": "tensor", "unit": "TFLOP/s",
                    "achieved": enc_flop / (gemm_chunk_ms / 1000.0) / 1e12,
                    "peak": pk["bf16_tflops_sustained"],
                    "peak_kind": f"{pk_kind} bf16 sustained (kernels timed inside the step)",
                    "algorithmic": f"{enc_flop:.4g} FLOP per chunk (M={w.B * w.T} frame rows, 2 M N K per GEMM)",
                    "ms_per_chunk": gemm_chunk_ms, "launches": enc_n["gemm"],
                    "traffic": recorded_traffic(w, "egemm", (args.encoder, w.B, w.T)),
                    "traffic_unit": "DRAM bytes per chunk (all encoder GEMM launches of one chunk step)",
                    "share_of_device_time": share_enc,
                    "encoder_other_kernels": {
                        "attention_ms_per_chunk": enc_ms["attention"] / args.steps,
                        "attention_share": enc_ms["attention"] / total_ms,
                        "layer_norm_conv_cache_ms_per_chunk": enc_ms["other"] / args.steps,
                        "layer_norm_conv_cache_share": enc_ms["other"] / total_ms}}
        enc_roof["frac"] = enc_roof["achieved"] / enc_roof["peak"]
        enc_roof["serialized_with_kernel_events"] = {
            "what": "CUDA events at every kernel boundary (second pass, one sequence of kernels)",
            "ms_per_chunk": enc_roof["ms_per_chunk"], "achieved": enc_roof["achieved"], "frac": enc_roof["frac"]}
        enc_roof["in_production_graph"] = {
            "what": "uninstrumented step time x this class's share of device time (the instrumented pass runs "
                    "the encoder's kernels in one sequence; the production graph runs two branches of streams "
                    "whose kernels overlap, so this apportions the overlapped step by the serial shares)",
            "ms_per_chunk": mean_step_ms * share_enc,
            "achieved": enc_flop / (mean_step_ms * share_enc / 1000.0) / 1e12}
        enc_roof["in_production_graph"]["frac"] = enc_roof["in_production_graph"]["achieved"] / enc_roof["peak"]
        for k in ("ms_per_chunk", "achieved", "frac"):
            enc_roof[k] = enc_roof["in_production_graph"][k]
        del enc_roof["in_production_graph"]
        enc_roof["timing"] = ("uninstrumented step time x this class's share of device time (CUDA events); the "
                              "production graph runs two branches of streams whose kernels overlap, so this "
                              "apportions the overlapped step by the serial shares")
    # the dominant kernel is the one with the largest device time in the graph
    ranked = sorted([(share_joint, joint_roof), (share_row, row_roof)] + ([(share_pred, pred_roof)] if pred_roof else [])
                    + ([(share_enc, enc_roof)] if enc_roof else []), key=lambda x: -x[0])
    roof, other = ranked[0][1], ranked[1][1]
    launches = dec.launches_per_chunk(w.B, w.T)
    if encoder is not None:
        launches += encoder.launches_per_chunk(w.B, w.T)
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": t_ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": dict(workload_config(w, lmA.total + sum(a.total for a, _ in extra), ph.n if ph else 0),
                           **variant_config(args, w, extra),
                           **({"options": args.set} if args.set else {}),
                           l2="flushed (256 MB write) before every timed step, outside the step's events",
                           parallelism=f"dp{ws} (independent streams per GPU)"),
            "e2e": {"value": e2e_val, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "steps": e2e_steps,
                    "copies": "each step's chunk copied from pinned host memory and every output read back, "
                              "inside the timed region; chunk k+1's copy overlaps chunk k's decode"},
            "gpu_launches": int(launches * args.steps),
            "roofline": roof,
            "roofline_other_kernel": other,
            **({"roofline_third_kernel": ranked[2][1]} if len(ranked) > 2 else {}),
            "latency_per_chunk": latency_stats(step_ms),
            **({"alt_fusion_path": alt} if alt else {}),
            **({"stream_sweep": {"what": "the same workload (tables, weights, lambda, beta) decoded at other stream "
                                         "counts B in this run (each with the decoder's default fusion_path for "
                                         "its stream count): frames/s over K timed chunks (L2 flushed before "
                                         "each) and chunk latency; 1 chunk = T x 80 ms of audio",
                                 "points": sweep}} if sweep else {}),
            **({"first_token_latency_s": {
                "value": w.T * 0.080 + float(np.median(step_ms)) / 1000.0,
                "what": "a chunk's audio (T x 80 ms) arrives before it is encoded, then the chunk's encoder and "
                        "decoder compute (median timed step at this batch)"}} if encoder is not None else {}),
            "wall_s_timed_region": wall,
            "value_with_kernel_events": frames / (t_inst_ms / 1000.0),
            "kernel_timing": "per-kernel device time from CUDA events at every kernel boundary inside the "
                             "graph, over a second pass of the same K steps (value_with_kernel_events)",
            "clocks": clk.summary()}
    if not args.no_cpu_baseline and ws == 1:
        models = oracle_models(w, lmA, ph, E, W, extra, pw)
        enc_o = oracle_encoder(args)
        n_cpu = min(args.cpu_streams, 16) if enc_o is not None else args.cpu_streams
        v, cores, sample, dt = oracle_baseline(w, models, list(range(n_cpu)), 1 if enc_o else args.cpu_chunks,
                                               prune_k=args.prune_k, encoder=enc_o)
        # the same oracle on one host thread, on a smaller sample of the same streams
        n_one = max(1, min(n_cpu, args.cpu_streams_single))
        v1, _, sample1, dt1 = oracle_baseline(w, models, list(range(n_one)), 1, threads=1, prune_k=args.prune_k,
                                              encoder=enc_o)
        line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                                "sample": sample, "seconds": dt,
                                "single_thread": {"value": v1, "unit": UNIT, "cores": 1, "sample": sample1,
                                                  "seconds": dt1}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=4)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-streams", type=int, default=None)
    ap.add_argument("--cpu-chunks", type=int, default=None)
    ap.add_argument("--ref-streams", type=int, default=None, help="streams per step of the reference arm")
    ap.add_argument("--sweep", default=None,
                    help="comma-separated stream counts also timed in this run (config 4 default: 1,16,128)")
    ap.add_argument("--streams", type=int, default=None, help="streams B per GPU (default: the config's)")
    ap.add_argument("--extra-lms", type=int, default=0, help="fuse this many further LMs (several-LM workload)")
    ap.add_argument("--prune-k", type=int, default=0,
                    help="pruned fusion over the acoustic model's k best outputs (0: every label)")
    ap.add_argument("--pred", type=int, default=0,
                    help="stateful form: an LSTM prediction network of this many units (0: stateless)")
    ap.add_argument("--fusion-path", type=int, default=None, choices=(0, 1),
                    help="greedy decoding with at most one LM: 0 = the streaming form (the decoder's default), "
                         "1 = the LM level-0 term in the joint epilogue with a per-row correction list")
    ap.add_argument("--no-alt-path", action="store_true",
                    help="skip timing the other form of the greedy one-LM step (fusion_path)")
    ap.add_argument("--set", action="append", metavar="NAME=VALUE",
                    help="a decoder tuning option (tsd_decoder_set_option), e.g. pdl=0 or joint_bn=128")
    ap.add_argument("--encoder", default=None, choices=sorted(synth.ENCODERS),
                    help="run the cache-aware encoder chunk step before the decode in every step")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    w = workload(args.config, args.streams)
    # bounded CPU samples (about 10-30 s of oracle work on 16 cores)
    cpu_default = {0: (4, 1), 1: (64, 12), 2: (256, 6), 3: (64, 2), 4: (64, 1)}[args.config]
    args.cpu_streams = args.cpu_streams or min(cpu_default[0], w.B)
    args.cpu_chunks = args.cpu_chunks or cpu_default[1]
    args.cpu_streams_single = {0: 4, 1: 8, 2: 8, 3: 4, 4: 4}[args.config]
    args.ref_streams = args.ref_streams or {4: 32}.get(args.config, 64)
    if args.sweep is None:
        args.sweep = "1,16,128" if args.config == 4 and not args.streams else ""
    args.sweep = [int(x) for x in args.sweep.split(",") if x.strip()]
    if args.impl == "reference":
        run_reference(args, w)
    else:
        run_ours(args, w)


if __name__ == "__main__":
    main()
