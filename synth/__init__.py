"""Seeded synthetic inputs shaped like the paper's decode workloads.

The paper (Sec. III-B, III-C; Table III) runs a FastConformer-Transducer with
n-gram shallow fusion and phrase boosting on real Thai audio with trained
weights; none of that data is available, so every input here is synthetic and
seeded.  This module draws data only: it contains none of the decode step's
arithmetic, and both the CPU oracle and the CUDA path consume its arrays as
plain inputs.  All random numbers come from the Philox4x32-10 counter-based
generator in ``synth.c``; each value is addressed by (seed, tensor, stream,
index) so a subset of streams sees the same data it sees inside a larger batch.

Workloads (sizes of the 115M and 0.6B joint networks, 13-frame chunks of
80 ms frames = the paper's 1040 ms look-ahead, Sec. IV-A and Table III):

====  ======  ====  =====  ==========  ===============================  =============================
cfg   B x K   H     V+1    T x chunks  LM                               boost list
====  ======  ====  =====  ==========  ===============================  =============================
0     4       320   257    200 x 1     3-gram ~20k, Zipf 1.1            16 phrases, len 2-6
1     64      640   1025   13 x 40     4-gram ~2M, Zipf 1.1             none
2     256     1024  1025   13 x 40     6-gram ~20M, Zipf 1.1            5k phrases, len 2-12, 20% shared
3     128x4   1024  1025   13 x 40     as cfg 2                         as cfg 2
4     1024    1024  4097   13 x 20     10-gram ~100M, Zipf 1.05         50k phrases, len 2-16, 20% shared
====  ======  ====  =====  ==========  ===============================  =============================
"""
from __future__ import annotations

import ctypes
import dataclasses
import math
import os
from typing import Dict, List, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libsynth.so")

TENSOR_ENC = 1
TENSOR_EMB = 2
TENSOR_WOUT = 3
TENSOR_PRED_EMB = 4
TENSOR_PRED_GATES = 5
TENSOR_PRED_GBIAS = 6
TENSOR_PRED_PROJ = 7
TENSOR_ENC_PROJ = 8
TENSOR_PROJ_BIAS = 9


def build(force: bool = False) -> str:
    """Compile synth.c into libsynth.so next to it (plain gcc, no GPU)."""
    src = os.path.join(_HERE, "synth.c")
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(src):
        import subprocess

        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c99", "-D_POSIX_C_SOURCE=200809L", "-shared", "-fPIC", src, "-o", tmp,
                               "-lm", "-lpthread"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB_PATH)
        u64, u32, i32, i64, dbl = ctypes.c_uint64, ctypes.c_uint32, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        vp = ctypes.c_void_p
        L.synth_philox.argtypes = [vp, vp, vp]
        L.synth_philox.restype = None
        L.synth_normal_bf16.argtypes = [u64, u32, u32, u64, u64, dbl, vp]
        L.synth_normal_bf16.restype = None
        L.synth_phrases.argtypes = [u64, i32, i32, i32, i32, dbl, vp, vp]
        L.synth_phrases.restype = i32
        L.synth_lm_new.argtypes = [u64, i32, i32, i64, dbl, dbl]
        L.synth_lm_new.restype = vp
        L.synth_lm_free.argtypes = [vp]
        L.synth_lm_free.restype = None
        L.synth_lm_count.argtypes = [vp, i32]
        L.synth_lm_count.restype = i64
        L.synth_lm_get.argtypes = [vp, i32, vp, vp, vp, vp]
        L.synth_lm_get.restype = None
        _lib = L
    return _lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def philox4x32_10(ctr, key) -> List[int]:
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().synth_philox(_ptr(c), _ptr(k), _ptr(out))
    return [int(x) for x in out]


def normal_bf16(seed: int, tensor_id: int, stream_id: int, first: int, n: int, std: float) -> np.ndarray:
    """n bf16 values (as uint16 bit patterns) of N(0, std^2)."""
    out = np.empty(n, dtype=np.uint16)
    lib().synth_normal_bf16(seed, tensor_id, stream_id, first, n, float(std), _ptr(out))
    return out


def bf16_to_f32(a: np.ndarray) -> np.ndarray:
    return (a.astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass
class NGramArrays:
    """ARPA-like backoff tables: per order k (1-based), tokens [n_k, k] in
    lexicographic order, natural-log probabilities, natural-log backoff
    weights (0 = none) and the raw counts they were estimated from."""

    V: int
    order: int
    tokens: List[np.ndarray]
    logp: List[np.ndarray]
    bow: List[np.ndarray]
    counts: List[np.ndarray]
    discount: float

    @property
    def total(self) -> int:
        return int(sum(len(x) for x in self.logp))


def ngram_lm(seed: int, V: int, order: int, total: int, zipf_s: float, discount: float = 0.7) -> NGramArrays:
    """The seeded LM (see _ngram_lm).  If TSD_SYNTH_CACHE names a directory,
    large models are kept there as .npz files and read back on later calls
    (the arrays are a pure function of the arguments)."""
    cache = os.environ.get("TSD_SYNTH_CACHE")
    if not cache or total < 1_000_000:
        return _ngram_lm(seed, V, order, total, zipf_s, discount)
    path = os.path.join(cache, f"lm_{seed}_{V}_{order}_{total}_{zipf_s}_{discount}.npz")
    if os.path.exists(path):
        z = np.load(path)
        return NGramArrays(V, order, [z[f"t{k}"] for k in range(order)], [z[f"l{k}"] for k in range(order)],
                           [z[f"b{k}"] for k in range(order)], [z[f"c{k}"] for k in range(order)], discount)
    a = _ngram_lm(seed, V, order, total, zipf_s, discount)
    os.makedirs(cache, exist_ok=True)
    tmp = path + f".tmp{os.getpid()}.npz"
    arrs = {}
    for k in range(order):
        arrs.update({f"t{k}": a.tokens[k], f"l{k}": a.logp[k], f"b{k}": a.bow[k], f"c{k}": a.counts[k]})
    np.savez(tmp, **arrs)
    os.replace(tmp, path)
    return a


def _ngram_lm(seed: int, V: int, order: int, total: int, zipf_s: float, discount: float = 0.7) -> NGramArrays:
    L = lib()
    h = L.synth_lm_new(seed, V, order, total, zipf_s, discount)
    if not h:
        raise MemoryError("synth_lm_new failed")
    try:
        toks, lps, bows, cnts = [], [], [], []
        for k in range(1, order + 1):
            n = L.synth_lm_count(h, k)
            t = np.empty((n, k), dtype=np.int32)
            lp = np.empty(n, dtype=np.float32)
            bw = np.empty(n, dtype=np.float32)
            ct = np.empty(n, dtype=np.int32)
            L.synth_lm_get(h, k, _ptr(t), _ptr(lp), _ptr(bw), _ptr(ct))
            toks.append(t)
            lps.append(lp)
            bows.append(bw)
            cnts.append(ct)
    finally:
        L.synth_lm_free(h)
    return NGramArrays(V, order, toks, lps, bows, cnts, discount)


@dataclasses.dataclass
class Phrases:
    offsets: np.ndarray  # int32 [n+1]
    tokens: np.ndarray  # int32 [offsets[-1]]

    @property
    def n(self) -> int:
        return len(self.offsets) - 1

    def phrase(self, i: int) -> List[int]:
        return [int(x) for x in self.tokens[self.offsets[i] : self.offsets[i + 1]]]


def phrases(seed: int, V: int, n: int, len_min: int, len_max: int, share_frac: float) -> Phrases:
    off = np.zeros(n + 1, dtype=np.int32)
    tok = np.zeros(max(1, n * len_max), dtype=np.int32)
    got = lib().synth_phrases(seed, V, n, len_min, len_max, share_frac, _ptr(off), _ptr(tok))
    if got < 0:
        raise MemoryError("synth_phrases failed")
    off = off[: got + 1].copy()
    return Phrases(off, tok[: off[-1]].copy())


@dataclasses.dataclass(frozen=True)
class Workload:
    cfg: int
    name: str
    V: int  # non-blank tokens; blank id = V
    H: int
    B: int
    T: int
    chunks: int
    lm_order: int
    lm_total: int
    zipf: float
    n_phr: int
    phr_len: tuple
    share: float
    bonus: float
    lam: float
    beta: float
    max_sym: int
    beam: int
    seed: int
    lm_seed: int
    boost_seed: int

    @property
    def N(self) -> int:
        return self.V + 1


def _w(cfg, name, V, H, B, T, chunks, lm_order, lm_total, zipf, n_phr, phr_len, share, bonus, lam, beta,
       max_sym, beam, data_cfg=None):
    seed = 1234 + cfg
    tseed = 1234 + (cfg if data_cfg is None else data_cfg)
    return Workload(cfg, name, V, H, B, T, chunks, lm_order, lm_total, zipf, n_phr, phr_len, share, bonus, lam,
                    beta, max_sym, beam, seed, tseed * 7919 + 1, tseed * 104729 + 3)


WORKLOADS: Dict[int, Workload] = {
    0: _w(0, "tiny-greedy-fusion V=256 H=320 B=4 T=200", 256, 320, 4, 200, 1, 3, 20_000, 1.1, 16, (2, 6), 0.0,
          1.0, 0.3, 1.0, 5, 1),
    1: _w(1, "small-model-streaming-greedy V=1024 H=640 B=64 T=13x40", 1024, 640, 64, 13, 40, 4, 2_000_000, 1.1,
          0, (2, 2), 0.0, 1.0, 0.5, 0.0, 5, 1),
    2: _w(2, "large-model-streaming-greedy-boost V=1024 H=1024 B=256 T=13x40", 1024, 1024, 256, 13, 40, 6,
          20_000_000, 1.1, 5000, (2, 12), 0.2, 1.0, 0.5, 1.5, 5, 1),
    3: _w(3, "beam-search-fusion K=4 V=1024 H=1024 B=128 T=13x40", 1024, 1024, 128, 13, 40, 6, 20_000_000, 1.1,
          5000, (2, 12), 0.2, 1.0, 0.5, 1.5, 1, 4, data_cfg=2),
    4: _w(4, "stress-roofline V=4096 H=1024 B=1024 T=13x20", 4096, 1024, 1024, 13, 20, 10, 100_000_000, 1.05,
          50000, (2, 16), 0.2, 1.0, 0.6, 1.5, 5, 1),
}


def scaled(w: Workload, **kw) -> Workload:
    """A copy of a workload with some fields replaced (smaller test cases)."""
    return dataclasses.replace(w, **kw)


def joint_weights(w: Workload):
    """(E [V+1, H], W_out [H, V+1]) as bf16 bit patterns.

    E ~ N(0, 1); W_out ~ N(0, std = 3/sqrt(H)) (the second parameter of the
    workload's N(0, 3/sqrt(H)) is read as a standard deviation)."""
    E = normal_bf16(w.seed, TENSOR_EMB, 0, 0, w.N * w.H, 1.0).reshape(w.N, w.H)
    W = normal_bf16(w.seed, TENSOR_WOUT, 0, 0, w.H * w.N, 3.0 / math.sqrt(w.H)).reshape(w.H, w.N)
    return E, W


def enc_chunk(w: Workload, streams, chunk: int, T: Optional[int] = None) -> np.ndarray:
    """Encoder frames [len(streams), T, H] (bf16 bits) of one chunk; stream s
    sees frames [chunk*T, (chunk+1)*T) of its own sequence."""
    T = w.T if T is None else T
    out = np.empty((len(streams), T, w.H), dtype=np.uint16)
    for i, s in enumerate(streams):
        out[i] = normal_bf16(w.seed, TENSOR_ENC, int(s), chunk * T * w.H, T * w.H, 1.0).reshape(T, w.H)
    return out


def lm_for(w: Workload) -> Optional[NGramArrays]:
    if w.lm_order <= 0:
        return None
    return ngram_lm(w.lm_seed, w.V, w.lm_order, w.lm_total, w.zipf, 0.7)


def phrases_for(w: Workload) -> Optional[Phrases]:
    if w.n_phr <= 0:
        return None
    return phrases(w.boost_seed, w.V, w.n_phr, w.phr_len[0], w.phr_len[1], w.share)


@dataclasses.dataclass
class PredWeights:
    """Prediction network and joint projections of the stateful Transducer
    form (bf16 bit patterns, fp32 biases): a one-layer LSTM of width D over
    the previous label, then joint input = ReLU(enc We + be + h Wp + bp)."""

    D: int
    Henc: int
    Ep: np.ndarray  # [V+1, D] label embedding (row V starts a sequence)
    Wg: np.ndarray  # [2D, 4D] gates; column 4u+q is gate q (i, f, g, o) of unit u; rows x then h
    bg: np.ndarray  # [4D] float32
    Wp: np.ndarray  # [D, H]
    bp: np.ndarray  # [H] float32
    We: np.ndarray  # [Henc, H]
    be: np.ndarray  # [H] float32


def pred_weights(w: Workload, D: int = 640, Henc: int = None) -> PredWeights:
    """Seeded prediction-network weights: Ep ~ N(0, 1); Wg ~ N(0, 1/sqrt(2D));
    gate biases ~ N(0, 0.1) plus 1 on the forget gates; Wp ~ N(0, 3/sqrt(D));
    We ~ N(0, 1/sqrt(Henc)); projection biases ~ N(0, 0.1).  The joint input
    then has about the spread of the stateless form's enc + E[last]."""
    Henc = Henc or w.H
    N, H = w.N, w.H
    bf = lambda t, n, std: normal_bf16(w.seed, t, 0, 0, n, std)
    Ep = bf(TENSOR_PRED_EMB, N * D, 1.0).reshape(N, D)
    Wg = bf(TENSOR_PRED_GATES, 2 * D * 4 * D, 1.0 / math.sqrt(2 * D)).reshape(2 * D, 4 * D)
    bg = bf16_to_f32(bf(TENSOR_PRED_GBIAS, 4 * D, 0.1)).copy()
    bg[1::4] += 1.0
    Wp = bf(TENSOR_PRED_PROJ, D * H, 3.0 / math.sqrt(D)).reshape(D, H)
    We = bf(TENSOR_ENC_PROJ, Henc * H, 1.0 / math.sqrt(Henc)).reshape(Henc, H)
    pb = bf16_to_f32(normal_bf16(w.seed, TENSOR_PROJ_BIAS, 0, 0, 2 * H, 0.1))
    return PredWeights(D, Henc, Ep, Wg, bg.astype(np.float32), Wp, pb[:H].copy(), We, pb[H:].copy())


def enc_chunk_wide(w: Workload, streams, chunk: int, Henc: int, T: Optional[int] = None) -> np.ndarray:
    """Encoder frames of width Henc (the stateful form projects them to H)."""
    T = w.T if T is None else T
    out = np.empty((len(streams), T, Henc), dtype=np.uint16)
    for i, s in enumerate(streams):
        out[i] = normal_bf16(w.seed, TENSOR_ENC, int(s), chunk * T * Henc, T * Henc, 1.0).reshape(T, Henc)
    return out


# --------------------------------------------------------------------------
# The cache-aware encoder (Sec. III-B): synthetic weights and features.

TENSOR_FEAT = 10
TENSOR_SUB_W = 11
TENSOR_SUB_B = 12
_TENSOR_LAYER0 = 1000  # layer l, tensor j -> 1000 + 64 l + j


@dataclasses.dataclass(frozen=True)
class EncoderCfg:
    """Shape of a cache-aware Conformer encoder: d model width, `layers`
    blocks of `heads` attention heads, feed-forward width ff, depthwise kernel
    K; attention sees `left` cached frames plus the whole current chunk of
    `chunk` frames; each encoder frame stacks `stack` feature frames of
    `feat` log-mel bins (80 ms from 10 ms features)."""

    name: str
    d: int
    layers: int
    heads: int
    ff: int
    kernel: int = 9
    left: int = 70
    chunk: int = 13
    feat: int = 80
    stack: int = 8
    seed: int = 777

    @property
    def dh(self) -> int:
        return self.d // self.heads

    @property
    def n_off(self) -> int:
        """Relative offsets query - key in a window: -(chunk-1) .. left+chunk-1."""
        return self.left + 2 * self.chunk - 1


# FastConformer-L-like (the 115M model) and FastConformer-XL-like (0.6B) shapes.
ENCODERS: Dict[str, EncoderCfg] = {
    "115m": EncoderCfg("115m", d=512, layers=17, heads=8, ff=2048),
    "0.6b": EncoderCfg("0.6b", d=1024, layers=24, heads=8, ff=4096),
}


@dataclasses.dataclass
class EncoderLayer:
    """One Conformer block.  Matrices are bf16 bit patterns stored
    [out][in] (y = W x); vectors are float32."""

    ln_ff1: tuple  # (gamma [d], beta [d])
    ff1_w1: np.ndarray  # [ff][d]
    ff1_b1: np.ndarray
    ff1_w2: np.ndarray  # [d][ff]
    ff1_b2: np.ndarray
    ln_att: tuple
    qkv_w: np.ndarray  # [3d][d]: rows q, then k, then v; head h owns columns h*dh .. (h+1)*dh-1 of each
    qkv_b: np.ndarray
    pos_w: np.ndarray  # [d][d], no bias: P = pos_w r(delta)
    pos_u: np.ndarray  # [d]: per head, the content bias added to the query
    pos_v: np.ndarray  # [d]: per head, the position bias added to the query
    out_w: np.ndarray  # [d][d]
    out_b: np.ndarray
    ln_conv: tuple
    pw1_w: np.ndarray  # [2d][d]: rows 0..d-1 the GLU value, d..2d-1 its gate
    pw1_b: np.ndarray
    dw_w: np.ndarray  # [d][K] float32 (bf16 values): tap K-1 is the current frame
    dw_b: np.ndarray
    bn_scale: np.ndarray  # [d]: batch norm at inference, an affine map per channel
    bn_shift: np.ndarray
    pw2_w: np.ndarray  # [d][d]
    pw2_b: np.ndarray
    ln_ff2: tuple
    ff2_w1: np.ndarray
    ff2_b1: np.ndarray
    ff2_w2: np.ndarray
    ff2_b2: np.ndarray
    ln_out: tuple


@dataclasses.dataclass
class EncoderWeights:
    cfg: EncoderCfg
    sub_w: np.ndarray  # [d][stack*feat]: the stacked feature frames -> d
    sub_b: np.ndarray
    layers: List[EncoderLayer]


def encoder_weights(cfg: EncoderCfg, layers: Optional[int] = None) -> EncoderWeights:
    """Seeded weights: matrices ~ N(0, 1/sqrt(fan_in)); biases ~ N(0, 0.02);
    layer-norm gains 1 + N(0, 0.1) and shifts N(0, 0.05); position biases
    u, v ~ N(0, 0.1); depthwise taps ~ N(0, 1/sqrt(K)); batch-norm scale
    1 + N(0, 0.1), shift N(0, 0.05)."""
    d, ff, K, s = cfg.d, cfg.ff, cfg.kernel, cfg.seed
    n_layers = cfg.layers if layers is None else layers

    def mat(t, rows, cols):
        return normal_bf16(s, t, 0, 0, rows * cols, 1.0 / math.sqrt(cols)).reshape(rows, cols)

    def vec(t, n, std, mean=0.0):
        return (bf16_to_f32(normal_bf16(s, t, 0, 0, n, std)) + np.float32(mean)).astype(np.float32)

    layers_out = []
    for l in range(n_layers):
        base = _TENSOR_LAYER0 + 64 * l
        j = iter(range(64))
        t = lambda: base + next(j)
        ln = lambda: (vec(t(), d, 0.1, 1.0), vec(t(), d, 0.05))
        L = EncoderLayer(
            ln_ff1=ln(), ff1_w1=mat(t(), ff, d), ff1_b1=vec(t(), ff, 0.02), ff1_w2=mat(t(), d, ff),
            ff1_b2=vec(t(), d, 0.02),
            ln_att=ln(), qkv_w=mat(t(), 3 * d, d), qkv_b=vec(t(), 3 * d, 0.02), pos_w=mat(t(), d, d),
            pos_u=vec(t(), d, 0.1), pos_v=vec(t(), d, 0.1), out_w=mat(t(), d, d), out_b=vec(t(), d, 0.02),
            ln_conv=ln(), pw1_w=mat(t(), 2 * d, d), pw1_b=vec(t(), 2 * d, 0.02),
            dw_w=bf16_to_f32(normal_bf16(s, t(), 0, 0, d * K, 1.0 / math.sqrt(K))).reshape(d, K).copy(),
            dw_b=vec(t(), d, 0.02), bn_scale=vec(t(), d, 0.1, 1.0), bn_shift=vec(t(), d, 0.05),
            pw2_w=mat(t(), d, d), pw2_b=vec(t(), d, 0.02),
            ln_ff2=ln(), ff2_w1=mat(t(), ff, d), ff2_b1=vec(t(), ff, 0.02), ff2_w2=mat(t(), d, ff),
            ff2_b2=vec(t(), d, 0.02),
            ln_out=ln())
        layers_out.append(L)
    sub_w = normal_bf16(s, TENSOR_SUB_W, 0, 0, d * cfg.stack * cfg.feat,
                        1.0 / math.sqrt(cfg.stack * cfg.feat)).reshape(d, cfg.stack * cfg.feat)
    sub_b = bf16_to_f32(normal_bf16(s, TENSOR_SUB_B, 0, 0, d, 0.02)).copy()
    return EncoderWeights(cfg, sub_w, sub_b, layers_out)


def features(cfg: EncoderCfg, streams, first: int, C: Optional[int] = None) -> np.ndarray:
    """Log-mel-like features of encoder frames first .. first+C-1 (C*stack
    feature frames) of each stream: N(0, 1) as bf16, [n][C*stack][feat].
    Frame f of a stream is the same whatever the chunking."""
    C = cfg.chunk if C is None else C
    per = cfg.stack * cfg.feat
    out = np.empty((len(streams), C * cfg.stack, cfg.feat), dtype=np.uint16)
    for i, st in enumerate(streams):
        out[i] = normal_bf16(cfg.seed, TENSOR_FEAT, int(st), first * per, C * per, 1.0).reshape(C * cfg.stack,
                                                                                             cfg.feat)
    return out
