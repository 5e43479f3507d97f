"""ORACLE -- test infrastructure, not part of the product.

A plain float64 numpy implementation of the cache-aware encoder chunk step.
Only the test suite, the smoke check and the benchmark's CPU legs may import
it; the product library never does, and this module never loads it.

What it computes (Sec. III-B; Sec. IV-A): a FastConformer encoder made
streamable by chunked, limited-context attention, causal convolutions and a
cache carried from chunk to chunk, so every chunk costs the same; one
encoder frame is 80 ms and the look-ahead is the chunk.  The paper fixes no
more than that.  The block follows the Conformer the paper builds on
(macaron feed-forward halves around self-attention and a convolution module,
a final layer norm), with these readings:

* subsampling: each encoder frame stacks `stack` consecutive feature frames
  and projects them linearly to d;
* attention: a query frame of the current chunk sees the `left` most recent
  frames before the chunk (the cache) and every frame of its chunk; scores
  add a relative-position term, ((q + u).k + (q + v).p(delta)) / sqrt(dh),
  with p(delta) = W_pos r(delta), r the sinusoidal code of the offset
  delta = query position - key position;
* convolution module: pointwise to 2d, GLU, a causal depthwise convolution
  over the last K frames (the K-1 previous ones come from the cache; zeros
  before the stream starts), batch norm as its inference-time affine map,
  Swish, pointwise back to d.

Rounding contract (the CUDA path computes in fp32 and rounds at the same
points): the operands of every matrix product are bf16 (each module's
layer-normed input, the feed-forward hidden layer after Swish, q/k/v and
the cached k/v, q + u and q + v, the position rows p(delta), the softmax
probabilities, the attention output, the GLU output and the cached GLU
output, the convolution module's Swish output) and the chunk's output is
bf16; everything else is float64 here.  With bf16_points=False nothing is
rounded (used by the pins, which compare exact arithmetic).
"""
from __future__ import annotations

import math
from typing import List

import numpy as np

LN_EPS = 1e-5


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Nearest bf16 value (8 significant bits, ties to even) of float64 x,
    returned as float64.  Magnitudes stay far inside bf16's range here."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)  # x = m 2^e, 0.5 <= |m| < 1
    return np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)


def bits_to_f64(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def f64_to_bits(x: np.ndarray) -> np.ndarray:
    """bf16 bit patterns of values that are already bf16 (exact)."""
    return (np.asarray(x, dtype=np.float64).astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)


def layer_norm(x: np.ndarray, gamma: np.ndarray, beta: np.ndarray) -> np.ndarray:
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS) * gamma + beta


def sigmoid(x: np.ndarray) -> np.ndarray:
    return 1.0 / (1.0 + np.exp(-x))


def swish(x: np.ndarray) -> np.ndarray:
    return x * sigmoid(x)


def sinusoid(delta: np.ndarray, d: int) -> np.ndarray:
    """r(delta): entries 2k and 2k+1 are sin and cos of delta / 10000^(2k/d)."""
    k = np.arange(d // 2, dtype=np.float64)
    w = np.power(10000.0, -2.0 * k / d)
    ang = np.asarray(delta, dtype=np.float64)[:, None] * w[None, :]
    r = np.empty((len(ang), d), dtype=np.float64)
    r[:, 0::2] = np.sin(ang)
    r[:, 1::2] = np.cos(ang)
    return r


class EncoderStream:
    """One stream's encoder cache: per block the k and v of the last `left`
    frames (oldest first) and the last K-1 GLU outputs, and the number of
    encoder frames seen."""

    def __init__(self, cfg):
        self.cfg = cfg
        self.seen = 0
        self.k: List[np.ndarray] = []
        self.v: List[np.ndarray] = []
        self.conv: List[np.ndarray] = []

    def _layer(self, l):
        while len(self.k) <= l:
            self.k.append(np.zeros((0, self.cfg.d)))
            self.v.append(np.zeros((0, self.cfg.d)))
            self.conv.append(np.zeros((self.cfg.kernel - 1, self.cfg.d)))


class Encoder:
    """The weights of `synth.EncoderWeights` as float64 arrays."""

    def __init__(self, w):
        self.cfg = w.cfg
        f = lambda a: bits_to_f64(a) if a.dtype == np.uint16 else np.asarray(a, dtype=np.float64)
        self.sub_w, self.sub_b = f(w.sub_w), f(w.sub_b)
        self.layers = []
        for L in w.layers:
            self.layers.append({k: (tuple(f(t) for t in v) if isinstance(v, tuple) else f(v))
                                for k, v in L.__dict__.items()})


def _feed_forward(x, gamma, beta, w1, b1, w2, b2, rnd):
    n = rnd(layer_norm(x, gamma, beta))
    h = rnd(swish(n @ w1.T + b1))
    return h @ w2.T + b2


def _attention(cfg, P, st, l, x, rnd):
    """Chunked, limited-context self-attention (Sec. III-B) with the
    relative-position term; appends the chunk's k and v to the cache."""
    C, d, H, dh = x.shape[0], cfg.d, cfg.heads, cfg.dh
    n = rnd(layer_norm(x, *P["ln_att"]))
    qkv = rnd(n @ P["qkv_w"].T + P["qkv_b"])
    q, k, v = qkv[:, :d], qkv[:, d:2 * d], qkv[:, 2 * d:]
    K = np.concatenate([st.k[l], k])  # window: cached frames, then the chunk
    V = np.concatenate([st.v[l], v])
    nv = st.k[l].shape[0]
    pos_q = st.seen + np.arange(C)
    pos_k = st.seen - nv + np.arange(nv + C)
    delta = pos_q[:, None] - pos_k[None, :]
    p = rnd(sinusoid(delta.reshape(-1), d) @ P["pos_w"].T)  # [C*(nv+C)][d]
    p = p.reshape(C, nv + C, d)
    out = np.zeros((C, d))
    for h in range(H):
        c = slice(h * dh, (h + 1) * dh)
        qu = rnd(q[:, c] + P["pos_u"][c])
        qv = rnd(q[:, c] + P["pos_v"][c])
        s = (qu @ K[:, c].T + np.einsum("ie,ije->ij", qv, p[:, :, c])) / math.sqrt(dh)
        s = s - s.max(axis=1, keepdims=True)
        a = np.exp(s)
        a = rnd(a / a.sum(axis=1, keepdims=True))
        out[:, c] = a @ V[:, c]
    o = rnd(out)
    st.k[l] = K[-cfg.left:] if cfg.left > 0 else K[:0]
    st.v[l] = V[-cfg.left:] if cfg.left > 0 else V[:0]
    return o @ P["out_w"].T + P["out_b"]


def _convolution(cfg, P, st, l, x, rnd):
    """The convolution module with a causal convolution (Sec. III-B):
    pointwise -> GLU -> causal depthwise convolution (cache of K-1 GLU
    outputs) -> batch-norm affine -> Swish -> pointwise."""
    C, d, K = x.shape[0], cfg.d, cfg.kernel
    n = rnd(layer_norm(x, *P["ln_conv"]))
    y = n @ P["pw1_w"].T + P["pw1_b"]
    glu = rnd(y[:, :d] * sigmoid(y[:, d:]))
    seq = np.concatenate([st.conv[l], glu])  # K-1 previous frames, then the chunk
    dw = np.empty((C, d))
    for t in range(C):
        dw[t] = (P["dw_w"] * seq[t:t + K].T).sum(axis=1) + P["dw_b"]
    z = rnd(swish(dw * P["bn_scale"] + P["bn_shift"]))
    st.conv[l] = seq[seq.shape[0] - (K - 1):]
    return z @ P["pw2_w"].T + P["pw2_b"]


def encode_chunk(enc: Encoder, st: EncoderStream, feats: np.ndarray, bf16_points: bool = True,
                 return_f64: bool = False):
    """One chunk of one stream (Sec. III-B: constant work per chunk, the
    cache carried across chunks; Sec. IV-A: 80 ms encoder frames): feats
    [C*stack][feat] (bf16 bit patterns) -> encoder frames [C][d] (bf16 bit
    patterns; with return_f64 the unrounded float64 values too).  Advances
    the stream's cache."""
    cfg = enc.cfg
    rnd = bf16_round if bf16_points else (lambda a: a)
    C = feats.shape[0] // cfg.stack
    z = bits_to_f64(feats).reshape(C, cfg.stack * cfg.feat)
    x = z @ enc.sub_w.T + enc.sub_b
    for l, P in enumerate(enc.layers):
        st._layer(l)
        x = x + 0.5 * _feed_forward(x, *P["ln_ff1"], P["ff1_w1"], P["ff1_b1"], P["ff1_w2"], P["ff1_b2"], rnd)
        x = x + _attention(cfg, P, st, l, x, rnd)
        x = x + _convolution(cfg, P, st, l, x, rnd)
        x = x + 0.5 * _feed_forward(x, *P["ln_ff2"], P["ff2_w1"], P["ff2_b1"], P["ff2_w2"], P["ff2_b2"], rnd)
        x = layer_norm(x, *P["ln_out"])
    st.seen += C
    out = bf16_round(x)
    return (f64_to_bits(out), x) if return_f64 else f64_to_bits(out)
