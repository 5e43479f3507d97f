"""Pins of the encoder oracle (oracle/encoder.py) against what its definition
fixes, from outside it: the bf16 rounding against torch's float32 -> bf16
conversion, and the chunked, cached computation against a full-sequence
formulation written here independently (whole-sequence tensors, a block
attention mask instead of a cache, torch's layer norm, GLU, Swish and
grouped 1-D convolution with left padding instead of a carried window)."""
from __future__ import annotations

import importlib.util
import math
import os

import numpy as np
import pytest

import synth


def _oracle_module():
    # the mutation tests point this at a copy with a planted mistake
    path = os.environ.get("TSD_ORACLE_ENCODER")
    if not path:
        from oracle import encoder
        return encoder
    spec = importlib.util.spec_from_file_location("oracle_encoder_variant", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


oe = _oracle_module()

torch = pytest.importorskip("torch")
F = torch.nn.functional


def _small(left=7, chunk=3, layers=2, d=64, heads=4, ff=128, K=5):
    cfg = synth.EncoderCfg("pin", d=d, layers=layers, heads=heads, ff=ff, kernel=K, left=left, chunk=chunk,
                           feat=16, stack=2, seed=4242)
    return cfg, synth.encoder_weights(cfg)


def _t(a):
    a = oe.bits_to_f64(a) if getattr(a, "dtype", None) == np.uint16 else np.asarray(a, dtype=np.float64)
    return torch.from_numpy(np.ascontiguousarray(a))


def full_sequence(w, feats, chunk, left):
    """The whole stream at once.  Frame p (in chunk p // chunk) attends to
    frames q with chunk_start(p) - left <= q < chunk_end(p); the depthwise
    convolution is causal with zero history.  No rounding."""
    cfg = w.cfg
    N = feats.shape[0] // cfg.stack
    d, H, dh, K = cfg.d, cfg.heads, cfg.dh, cfg.kernel
    x = F.linear(_t(feats).reshape(N, cfg.stack * cfg.feat), _t(w.sub_w), _t(w.sub_b))
    p = torch.arange(N)
    start = (p // chunk) * chunk
    allowed = (p[None, :] >= (start[:, None] - left)) & (p[None, :] < (start[:, None] + chunk))
    rel = (p[:, None] - p[None, :]).double()  # query position - key position
    k_idx = torch.arange(d // 2).double()
    freq = torch.pow(torch.tensor(10000.0, dtype=torch.float64), -2.0 * k_idx / d)
    ang = rel[:, :, None] * freq
    r = torch.stack([torch.sin(ang), torch.cos(ang)], dim=-1).reshape(N, N, d)  # sin at 2k, cos at 2k+1

    def ff(x, ln, w1, b1, w2, b2):
        n = F.layer_norm(x, (d,), _t(ln[0]), _t(ln[1]), eps=oe.LN_EPS)
        return F.linear(F.silu(F.linear(n, _t(w1), _t(b1))), _t(w2), _t(b2))

    for L in w.layers:
        x = x + 0.5 * ff(x, L.ln_ff1, L.ff1_w1, L.ff1_b1, L.ff1_w2, L.ff1_b2)
        n = F.layer_norm(x, (d,), _t(L.ln_att[0]), _t(L.ln_att[1]), eps=oe.LN_EPS)
        q, k, v = F.linear(n, _t(L.qkv_w), _t(L.qkv_b)).split(d, dim=1)
        pe = F.linear(r, _t(L.pos_w))  # [N][N][d]
        heads = []
        for h in range(H):
            c = slice(h * dh, (h + 1) * dh)
            content = (q[:, c] + _t(L.pos_u)[c]) @ k[:, c].T
            position = torch.einsum("pe,pqe->pq", q[:, c] + _t(L.pos_v)[c], pe[:, :, c])
            s = ((content + position) / math.sqrt(dh)).masked_fill(~allowed, float("-inf"))
            heads.append(torch.softmax(s, dim=1) @ v[:, c])
        x = x + F.linear(torch.cat(heads, dim=1), _t(L.out_w), _t(L.out_b))
        n = F.layer_norm(x, (d,), _t(L.ln_conv[0]), _t(L.ln_conv[1]), eps=oe.LN_EPS)
        g = F.glu(F.linear(n, _t(L.pw1_w), _t(L.pw1_b)), dim=1)  # first half * sigmoid(second half)
        y = F.conv1d(g.T[None], _t(L.dw_w)[:, None, :], _t(L.dw_b), padding=K - 1, groups=d)[0, :, :N].T
        z = F.silu(y * _t(L.bn_scale) + _t(L.bn_shift))
        x = x + F.linear(z, _t(L.pw2_w), _t(L.pw2_b))
        x = x + 0.5 * ff(x, L.ln_ff2, L.ff2_w1, L.ff2_b1, L.ff2_w2, L.ff2_b2)
        x = F.layer_norm(x, (d,), _t(L.ln_out[0]), _t(L.ln_out[1]), eps=oe.LN_EPS)
    return x.numpy()


def _chunked(w, feats, chunk, bf16_points=False):
    cfg = w.cfg
    enc, st = oe.Encoder(w), oe.EncoderStream(cfg)
    N = feats.shape[0] // cfg.stack
    outs = []
    for c0 in range(0, N, chunk):
        n = min(chunk, N - c0)
        _, x = oe.encode_chunk(enc, st, feats[c0 * cfg.stack:(c0 + n) * cfg.stack], bf16_points=bf16_points,
                               return_f64=True)
        outs.append(x)
    return np.concatenate(outs)


def test_bf16_rounding_is_torchs_conversion():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.normal(0, 1, 20000), rng.normal(0, 1e-3, 2000), rng.normal(0, 300, 2000)])
    x = x.astype(np.float32)
    # exact ties: bf16 values plus half an ulp, both parities
    ties = (oe.bits_to_f64(rng.integers(0x3000, 0x4800, 4000).astype(np.uint16)) *
            (1 + np.ldexp(1.0, -8))).astype(np.float32)
    x = np.concatenate([x, ties, -ties])
    want = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(oe.bf16_round(x.astype(np.float64)), want)


@pytest.mark.parametrize("left,chunk", [(7, 3), (4, 4), (0, 2), (10, 1)])
def test_chunked_cache_equals_full_sequence_with_a_block_mask(left, chunk):
    """Five or more chunks: the attention cache fills, then slides; the
    convolution cache carries K-1 frames across every chunk boundary."""
    cfg, w = _small(left=left, chunk=chunk)
    N = 5 * chunk + 2  # a ragged last chunk
    feats = synth.features(cfg, [3], 0, N)[0]
    a = _chunked(w, feats, chunk)
    b = full_sequence(w, feats, chunk, left)
    assert np.abs(a - b).max() < 1e-9, np.abs(a - b).max()


def test_rounded_path_stays_near_the_exact_one():
    """The bf16 rounding points move the output by about bf16 precision,
    not more: the rounding contract does not change what is computed."""
    cfg, w = _small()
    feats = synth.features(cfg, [1], 0, 12)[0]
    a = _chunked(w, feats, cfg.chunk, bf16_points=True)
    b = _chunked(w, feats, cfg.chunk, bf16_points=False)
    err = np.abs(a - b)
    assert 0 < err.max() < 0.15 and err.mean() < 0.02, (err.max(), err.mean())


def test_first_chunk_has_no_history():
    """A fresh stream's first chunk depends only on its own frames: features
    of other streams or earlier frames change nothing, and a stream with a
    different past gives a different first-chunk-after output."""
    cfg, w = _small()
    enc = oe.Encoder(w)
    f = synth.features(cfg, [5], 0, cfg.chunk)[0]
    a = oe.encode_chunk(enc, oe.EncoderStream(cfg), f)
    b = oe.encode_chunk(enc, oe.EncoderStream(cfg), f)
    assert np.array_equal(a, b)
    st = oe.EncoderStream(cfg)
    oe.encode_chunk(enc, st, synth.features(cfg, [6], 0, cfg.chunk)[0])
    c = oe.encode_chunk(enc, st, f)
    assert not np.array_equal(a, c)
