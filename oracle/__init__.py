"""ORACLE -- test infrastructure, not part of the product.

Python handle on ``oracle.cpp``: a plain, slow, double-precision CPU
implementation of the fused Transducer decode step (Eq. 1 of the paper with
one or more weighted n-gram LMs and one phrase list), and a plain reader of
ARPA-format n-gram files (``read_arpa``).  Only the test suite, the smoke check and
the benchmark's CPU-baseline leg may import this package; the product library
never does, and this package never loads the product library.

Every function here marshals arguments only; the arithmetic is in
``oracle.cpp``.  Calls release the GIL (ctypes), so streams can be decoded on
several host threads at once.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import List, Optional, Sequence, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.environ.get("TSD_ORACLE_LIB") or os.path.join(_HERE, "liboracle.so")

REP_STEPS, REP_MISMATCH, REP_NEAR_TIE, REP_MAX_SCORE_DIFF, REP_MIN_GAP, REP_FIRST_BAD, REP_INCONSISTENT = range(7)


def build(force: bool = False) -> str:
    """Compile oracle.cpp with g++ (no fast-math, no FMA contraction, so the
    result is the same on x86_64 and aarch64)."""
    src = os.path.join(_HERE, "oracle.cpp")
    if os.environ.get("TSD_ORACLE_LIB"):
        return _LIB_PATH  # a prebuilt variant (used by the mutation tests)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(src):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["g++", "-O2", "-std=c++17", "-ffp-contract=off", "-shared", "-fPIC", src,
                               "-o", tmp])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB_PATH)
        vp, i32, i64, dbl = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        sig = {
            "oracle_lm_new": ([i32, i32, vp, vp, vp, vp], vp),
            "oracle_lm_free": ([vp], None),
            "oracle_lm_score": ([vp, vp, i64, i32], dbl),
            "oracle_lm_state": ([vp, vp, i64, vp], i32),
            "oracle_lm_lookup": ([vp, vp, i32, i32], dbl),
            "oracle_boost_new": ([i32, i32, vp, vp, dbl], vp),
            "oracle_boost_free": ([vp], None),
            "oracle_boost_match": ([vp, vp, i64], i32),
            "oracle_boost_is_phrase": ([vp, vp, i64], i32),
            "oracle_boost_score": ([vp, vp, i64, i32], dbl),
            "oracle_stream_new": ([i32], vp),
            "oracle_stream_free": ([vp], None),
            "oracle_stream_history": ([vp, vp, i64], i64),
            "oracle_stream_rho": ([vp], i64),
            "oracle_stream_set_history": ([vp, vp, i64, i64], None),
            "oracle_decode_chunk": ([vp, vp, vp, i32, i32, vp, vp, vp, i32, dbl, dbl, i32, vp, vp, vp, i32, dbl,
                                     vp, vp, vp, i32, vp], i32),
            "oracle_decode_chunk_lms": ([vp, i32, vp, vp, vp, i32, i32, vp, vp, vp, i32, dbl, dbl, i32, vp, vp, vp,
                                         i32, dbl, vp, vp, vp, i32, vp], i32),
            "oracle_decode_chunk_pruned": ([vp, vp, vp, i32, i32, vp, vp, vp, i32, dbl, dbl, i32, i32, dbl, vp, vp,
                                            vp, i32, dbl, vp, vp, vp, i32, vp], i32),
            "oracle_decode_chunk_pred": ([vp, vp, vp, i32, i32, i32, i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, i32,
                                          dbl, dbl, i32, vp, vp, vp, i32, dbl, vp, vp, vp, i32, vp], i32),
            "oracle_pred_state": ([vp, vp, vp], i32),
            "oracle_beam_chunk": ([vp, vp, vp, i32, i32, vp, vp, vp, i32, dbl, dbl, i32, i32], i32),
            "oracle_beam_hyp": ([vp, i32, vp, i64, vp, vp], i64),
            "oracle_beam_chunk_follow": ([vp, vp, vp, i32, i32, vp, vp, vp, i32, dbl, dbl, i32, vp, vp, vp, dbl,
                                          vp, i32, i32], i32),
            "oracle_joint_logits": ([i32, i32, vp, vp, vp, i32, vp], None),
            "oracle_fused_row": ([vp, vp, vp, i32, i32, vp, vp, vp, dbl, dbl, vp], None),
            "oracle_boost_trajectory": ([vp, vp, i64, vp, vp], None),
        }
        for name, (args, res) in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def _i32(seq) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(seq, dtype=np.int32))


class LM:
    """Dictionary-of-n-grams backoff LM (natural log)."""

    def __init__(self, V: int, tokens: Sequence[np.ndarray], logp: Sequence[np.ndarray],
                 bow: Sequence[np.ndarray]):
        self.V, self.order = V, len(tokens)
        self._keep = [np.ascontiguousarray(t, dtype=np.int32) for t in tokens]
        self._keep_lp = [np.ascontiguousarray(x, dtype=np.float32) for x in logp]
        self._keep_bw = [np.ascontiguousarray(x, dtype=np.float32) for x in bow]
        cnt = np.array([len(x) for x in self._keep_lp], dtype=np.int64)
        tp = (ctypes.c_void_p * self.order)(*[t.ctypes.data for t in self._keep])
        lp = (ctypes.c_void_p * self.order)(*[t.ctypes.data for t in self._keep_lp])
        bw = (ctypes.c_void_p * self.order)(*[t.ctypes.data for t in self._keep_bw])
        self.h = lib().oracle_lm_new(V, self.order, _p(cnt), tp, lp, bw)
        if not self.h:
            raise ValueError("oracle_lm_new rejected the n-gram arrays")

    @classmethod
    def from_arrays(cls, a) -> "LM":
        return cls(a.V, a.tokens, a.logp, a.bow)

    def __del__(self):
        if getattr(self, "h", None):
            lib().oracle_lm_free(self.h)
            self.h = None

    def score(self, hist: Sequence[int], v: int) -> float:
        h = _i32(hist)
        return lib().oracle_lm_score(self.h, _p(h), len(h), int(v))

    def state(self, hist: Sequence[int]) -> Tuple[int, ...]:
        h = _i32(hist)
        out = np.zeros(max(1, self.order), dtype=np.int32)
        n = lib().oracle_lm_state(self.h, _p(h), len(h), _p(out))
        return tuple(int(x) for x in out[:n])

    def lookup_logp(self, g: Sequence[int]) -> float:
        g = _i32(g)
        return lib().oracle_lm_lookup(self.h, _p(g), len(g), 0)

    def lookup_bow(self, g: Sequence[int]) -> float:
        g = _i32(g)
        return lib().oracle_lm_lookup(self.h, _p(g), len(g), 1)


class Boost:
    """Phrase list matched by naive suffix search."""

    def __init__(self, V: int, offsets: np.ndarray, tokens: np.ndarray, bonus: float):
        self.V = V
        self._off = _i32(offsets)
        self._tok = _i32(tokens) if len(tokens) else np.zeros(1, dtype=np.int32)
        self.h = lib().oracle_boost_new(V, len(self._off) - 1, _p(self._off), _p(self._tok), float(bonus))
        if not self.h:
            raise ValueError("oracle_boost_new rejected the phrase list")

    @classmethod
    def from_phrases(cls, V: int, p, bonus: float) -> "Boost":
        return cls(V, p.offsets, p.tokens, bonus)

    def __del__(self):
        if getattr(self, "h", None):
            lib().oracle_boost_free(self.h)
            self.h = None

    def match(self, g: Sequence[int]) -> int:
        g = _i32(g)
        return lib().oracle_boost_match(self.h, _p(g), len(g))

    def is_phrase(self, g: Sequence[int]) -> bool:
        g = _i32(g)
        return bool(lib().oracle_boost_is_phrase(self.h, _p(g), len(g)))

    def score(self, g: Sequence[int], v: int) -> float:
        g = _i32(g)
        return lib().oracle_boost_score(self.h, _p(g), len(g), int(v))

    def trajectory(self, y: Sequence[int]):
        """(bonus per emitted label, restart index after it) from an empty history."""
        y = _i32(y)
        b = np.zeros(max(1, len(y)), dtype=np.float64)
        r = np.zeros(max(1, len(y)), dtype=np.int64)
        lib().oracle_boost_trajectory(self.h, _p(y), len(y), _p(b), _p(r))
        return b[: len(y)].copy(), r[: len(y)].copy()


class Stream:
    def __init__(self, V: int):
        self.V = V
        self.h = lib().oracle_stream_new(V)

    def __del__(self):
        if getattr(self, "h", None):
            lib().oracle_stream_free(self.h)
            self.h = None

    def history(self) -> List[int]:
        n = lib().oracle_stream_history(self.h, None, 0)
        buf = np.zeros(max(1, n), dtype=np.int32)
        lib().oracle_stream_history(self.h, _p(buf), n)
        return [int(x) for x in buf[:n]]

    def rho(self) -> int:
        return int(lib().oracle_stream_rho(self.h))

    def set_history(self, y: Sequence[int], rho: int = 0):
        y = _i32(y)
        lib().oracle_stream_set_history(self.h, _p(y), len(y), int(rho))

    def pred_state(self, D: int):
        """(h as bf16 bits [D], c [D]) of the prediction network, or None
        before its first step."""
        h = np.zeros(D, dtype=np.uint16)
        c = np.zeros(D, dtype=np.float64)
        ok = lib().oracle_pred_state(self.h, _p(h), _p(c))
        return (h, c) if ok else None

    def beam_hyps(self, with_rho: bool = False):
        """[(labels, score)] or, with_rho, [(labels, score, restart index)]."""
        out = []
        i = 0
        while True:
            n = lib().oracle_beam_hyp(self.h, i, None, 0, None, None)
            if n < 0:
                return out
            buf = np.zeros(max(1, n), dtype=np.int32)
            sc = ctypes.c_double()
            rho = ctypes.c_int64()
            lib().oracle_beam_hyp(self.h, i, _p(buf), n, ctypes.byref(sc), ctypes.byref(rho))
            labels = [int(x) for x in buf[:n]]
            out.append((labels, sc.value, int(rho.value)) if with_rho else (labels, sc.value))
            i += 1


class Model:
    """The joint network's inputs (bf16 bit patterns as uint16)."""

    def __init__(self, V: int, H: int, E: np.ndarray, W: np.ndarray):
        assert E.dtype == np.uint16 and E.shape == (V + 1, H)
        assert W.dtype == np.uint16 and W.shape == (H, V + 1)
        self.V, self.H = V, H
        self.E = np.ascontiguousarray(E)
        self.W = np.ascontiguousarray(W)

    def joint_logits(self, enc_t: np.ndarray, last: int) -> np.ndarray:
        enc_t = np.ascontiguousarray(enc_t, dtype=np.uint16)
        out = np.zeros(self.V + 1, dtype=np.float64)
        lib().oracle_joint_logits(self.V, self.H, _p(self.E), _p(self.W), _p(enc_t), int(last), _p(out))
        return out


def fused_row(stream: Stream, model: Model, lm: Optional[LM], boost: Optional[Boost], enc_t: np.ndarray,
              lam: float, beta: float) -> np.ndarray:
    enc_t = np.ascontiguousarray(enc_t, dtype=np.uint16)
    out = np.zeros(model.V + 1, dtype=np.float64)
    lib().oracle_fused_row(stream.h, lm.h if lm else None, boost.h if boost else None, model.V, model.H,
                           _p(model.E), _p(model.W), _p(enc_t), float(lam), float(beta), _p(out))
    return out


class PredNet:
    """Prediction network and joint projections (synth.PredWeights layout)."""

    def __init__(self, V: int, H: int, p):
        self.V, self.H, self.D, self.Henc = V, H, p.D, p.Henc
        self.Ep = np.ascontiguousarray(p.Ep, dtype=np.uint16)
        self.Wg = np.ascontiguousarray(p.Wg, dtype=np.uint16)
        self.bg = np.ascontiguousarray(p.bg, dtype=np.float32)
        self.Wp = np.ascontiguousarray(p.Wp, dtype=np.uint16)
        self.bp = np.ascontiguousarray(p.bp, dtype=np.float32)
        self.We = np.ascontiguousarray(p.We, dtype=np.uint16)
        self.be = np.ascontiguousarray(p.be, dtype=np.float32)
        assert self.Ep.shape == (V + 1, self.D) and self.Wg.shape == (2 * self.D, 4 * self.D)
        assert self.Wp.shape == (self.D, H) and self.We.shape == (self.Henc, H)


def decode_chunk(stream: Stream, model: Model, lm: Optional[LM], boost: Optional[Boost], enc: np.ndarray,
                 lam: float, beta: float, max_sym: int, follow=None, gap_tol: float = 1e-3, prune_k: int = 0,
                 am_tol: float = 2e-2, pred: Optional[PredNet] = None):
    """Greedy decode of one chunk enc [T, H] for one stream.

    lm: None, one LM (weight lam), or a list of (LM, w) pairs: LM i enters
    Eq. 1 with weight alpha_i = lam * w.
    follow: None (free-running) or (tokens, frames, scores) of the decisions
    under test, which the oracle checks and then follows.
    prune_k > 0: pruned fusion over the acoustic model's prune_k best outputs
    (one LM); am_tol is the logit tolerance at the edge of that set.
    pred: the stateful form (prediction network + joint projections); enc
    rows are then pred.Henc wide and model.E is not used.
    Returns (tokens, frames, scores, report[8])."""
    enc = np.ascontiguousarray(enc, dtype=np.uint16)
    T = enc.shape[0]
    cap = T * max_sym
    ot = np.zeros(max(1, cap), dtype=np.int32)
    of = np.zeros(max(1, cap), dtype=np.int32)
    osc = np.zeros(max(1, cap), dtype=np.float64)
    rep = np.zeros(8, dtype=np.float64)
    if follow is not None:
        ft, ff, fs = (_i32(follow[0]), _i32(follow[1]), np.ascontiguousarray(follow[2], dtype=np.float32))
        fargs = (_p(ft), _p(ff), _p(fs), len(ft))
    else:
        fargs = (None, None, None, 0)
    if pred is not None:
        assert not isinstance(lm, (list, tuple)) and prune_k == 0
        n = lib().oracle_decode_chunk_pred(stream.h, lm.h if lm else None, boost.h if boost else None, model.V,
                                           model.H, pred.Henc, pred.D, _p(pred.Ep), _p(pred.Wg), _p(pred.bg),
                                           _p(pred.Wp), _p(pred.bp), _p(pred.We), _p(pred.be), _p(model.W), _p(enc),
                                           T, float(lam), float(beta), int(max_sym), *fargs, float(gap_tol),
                                           _p(ot), _p(of), _p(osc), cap, _p(rep))
    elif prune_k > 0:
        assert not isinstance(lm, (list, tuple)), "pruned fusion takes one LM"
        n = lib().oracle_decode_chunk_pruned(stream.h, lm.h if lm else None, boost.h if boost else None, model.V,
                                             model.H, _p(model.E), _p(model.W), _p(enc), T, float(lam), float(beta),
                                             int(max_sym), int(prune_k), float(am_tol), *fargs, float(gap_tol),
                                             _p(ot), _p(of), _p(osc), cap, _p(rep))
    elif isinstance(lm, (list, tuple)):
        hs = (ctypes.c_void_p * max(1, len(lm)))(*[m.h for m, _ in lm])
        ws = np.array([w for _, w in lm] or [0.0], dtype=np.float64)
        n = lib().oracle_decode_chunk_lms(stream.h, len(lm), hs, _p(ws), boost.h if boost else None, model.V,
                                          model.H, _p(model.E), _p(model.W), _p(enc), T, float(lam), float(beta),
                                          int(max_sym), *fargs, float(gap_tol), _p(ot), _p(of), _p(osc), cap,
                                          _p(rep))
        if n < 0:
            raise ValueError("oracle_decode_chunk_lms rejected the LM list")
    else:
        n = lib().oracle_decode_chunk(stream.h, lm.h if lm else None, boost.h if boost else None, model.V,
                                      model.H, _p(model.E), _p(model.W), _p(enc), T, float(lam), float(beta),
                                      int(max_sym), *fargs, float(gap_tol), _p(ot), _p(of), _p(osc), cap, _p(rep))
    n = min(n, cap)
    return ot[:n].copy(), of[:n].copy(), osc[:n].copy(), rep


def beam_chunk(stream: Stream, model: Model, lm: Optional[LM], boost: Optional[Boost], enc: np.ndarray,
               lam: float, beta: float, K: int, S: int = 1) -> int:
    """Beam search over one chunk, at most S labels per frame."""
    enc = np.ascontiguousarray(enc, dtype=np.uint16)
    return lib().oracle_beam_chunk(stream.h, lm.h if lm else None, boost.h if boost else None, model.V, model.H,
                                   _p(model.E), _p(model.W), _p(enc), enc.shape[0], float(lam), float(beta),
                                   int(K), int(S))


def beam_chunk_follow(stream: Stream, model: Model, lm: Optional[LM], boost: Optional[Boost], enc: np.ndarray,
                      lam: float, beta: float, K: int, sel_hyp: np.ndarray, sel_tok: np.ndarray,
                      sel_inc: np.ndarray, gap_tol: float = 1e-3, S: int = 1) -> np.ndarray:
    """Beam search over one chunk following kept candidates [steps, K] under
    test (one row per expansion); returns the report (see
    oracle_beam_chunk_follow)."""
    enc = np.ascontiguousarray(enc, dtype=np.uint16)
    n_steps = np.asarray(sel_hyp).shape[0]
    sh, st = _i32(sel_hyp).reshape(-1), _i32(sel_tok).reshape(-1)
    si = np.ascontiguousarray(sel_inc, dtype=np.float32).reshape(-1)
    rep = np.zeros(8, dtype=np.float64)
    lib().oracle_beam_chunk_follow(stream.h, lm.h if lm else None, boost.h if boost else None, model.V, model.H,
                                   _p(model.E), _p(model.W), _p(enc), enc.shape[0], float(lam), float(beta), int(K),
                                   _p(sh), _p(st), _p(si), float(gap_tol), _p(rep), int(S), int(n_steps))
    return rep


class ArpaArrays:
    """Per-order n-gram arrays read from an ARPA file (natural log)."""

    def __init__(self, V, tokens, logp, bow, skipped):
        self.V, self.order = V, len(tokens)
        self.tokens, self.logp, self.bow, self.skipped = tokens, logp, bow, skipped


def read_arpa(text: str, V: int, vocab: Optional[Sequence[str]] = None) -> ArpaArrays:
    """Reads an ARPA back-off n-gram file: the data header, then per order k a
    section of lines 'log10 p <k words> [log10 backoff]'.  Words map to ids
    through vocab (word i -> id i) or, without one, are decimal ids.  N-grams
    holding a word outside the vocabulary (sentence markers, <unk>) are
    skipped: the decoder scores no sentence boundaries.  log10 values are
    turned into natural log."""
    ln10 = float(np.log(10.0))
    ids = {w: i for i, w in enumerate(vocab)} if vocab is not None else None

    def word_id(w):
        if ids is not None:
            return ids.get(w)
        try:
            i = int(w)
        except ValueError:
            return None
        return i if 0 <= i < V else None

    lines = text.splitlines()
    counts, pos = {}, 0
    while pos < len(lines) and lines[pos].strip() != "\\data\\":
        pos += 1
    pos += 1
    while pos < len(lines) and lines[pos].strip().startswith("ngram "):
        k, n = lines[pos].strip()[len("ngram "):].split("=")
        counts[int(k)] = int(n)
        pos += 1
    order = max(counts) if counts else 0
    toks, lps, bws, skipped = [], [], [], 0
    for k in range(1, order + 1):
        while pos < len(lines) and lines[pos].strip() != "\\%d-grams:" % k:
            pos += 1
        pos += 1
        t, lp, bw, seen = [], [], [], 0
        while pos < len(lines) and lines[pos].strip() and not lines[pos].startswith("\\"):
            f = lines[pos].split()
            pos += 1
            seen += 1
            words = f[1:1 + k]
            w_ids = [word_id(w) for w in words]
            if any(i is None for i in w_ids):
                skipped += 1
                continue
            t.append(w_ids)
            lp.append(float(f[0]) * ln10)
            bw.append(float(f[1 + k]) * ln10 if len(f) > 1 + k else 0.0)
        if seen != counts.get(k, seen):
            raise ValueError("ARPA order %d: header says %d n-grams, found %d" % (k, counts[k], seen))
        toks.append(np.array(t, dtype=np.int32).reshape(-1, k))
        lps.append(np.array(lp, dtype=np.float32))
        bws.append(np.array(bw, dtype=np.float32))
    return ArpaArrays(V, toks, lps, bws, skipped)
