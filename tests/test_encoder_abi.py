"""The encoder's C entry points reject bad shapes and NULL weights with
TSD_EINVAL before any device work (no GPU needed)."""
from __future__ import annotations

import ctypes

import pytest

import paper_2609_14991_gb300 as tsd


def _cfg(**kw):
    base = dict(d=256, layers=2, heads=4, ff=512, kernel=5, left=12, max_chunk=13, feat=16, stack=4, max_streams=8)
    base.update(kw)
    return tsd.EncoderCfgC(*[base[n] for n, _ in tsd.EncoderCfgC._fields_])


def _layers(n, null_field=None):
    arr = (tsd.EncoderLayerC * n)()
    for i in range(n):
        for name, _ in tsd.EncoderLayerC._fields_:
            setattr(arr[i], name, 0 if name == null_field and i == n - 1 else 0x1000)
    return arr


def _create(cfg, layers, sub_w=0x1000, sub_b=0x1000):
    h = ctypes.c_void_p()
    return tsd.lib().tsd_encoder_create(ctypes.byref(cfg), sub_w, sub_b, ctypes.cast(layers, ctypes.c_void_p), None,
                                        ctypes.byref(h))


@pytest.mark.parametrize("kw,word", [
    (dict(d=192), "d="),
    (dict(d=256, heads=8), "d/heads"),     # 32-wide heads
    (dict(ff=500), "ff="),
    (dict(layers=0), "layers="),
    (dict(layers=65), "layers="),
    (dict(kernel=0), "kernel="),
    (dict(left=129), "left="),
    (dict(max_chunk=0), "max_chunk="),
    (dict(max_chunk=33), "max_chunk="),
    (dict(stack=3), "stack*feat"),
    (dict(max_streams=0), "max_streams="),
])
def test_bad_shapes_are_rejected(kw, word):
    cfg = _cfg(**kw)
    st = _create(cfg, _layers(max(1, min(cfg.layers, 64))))
    assert st == tsd.TSD_EINVAL
    assert word in tsd.lib().tsd_last_error().decode()


def test_null_weights_are_rejected():
    cfg = _cfg()
    st = _create(cfg, _layers(2, null_field="pos_w"))
    assert st == tsd.TSD_EINVAL and "NULL" in tsd.lib().tsd_last_error().decode()
    assert _create(cfg, _layers(2), sub_w=None) == tsd.TSD_EINVAL


def test_null_handles_are_rejected():
    assert tsd.lib().tsd_encode_chunk(None, 1, None, None, 1, None, None) == tsd.TSD_EINVAL
    assert tsd.lib().tsd_encoder_open(None, None) == tsd.TSD_EINVAL
    assert tsd.lib().tsd_encoder_check(None) == tsd.TSD_EINVAL
    x = ctypes.c_int64()
    assert tsd.lib().tsd_encoder_launches_per_chunk(None, 1, 1, ctypes.byref(x)) == tsd.TSD_EINVAL
    tsd.lib().tsd_encoder_free(None)  # no-op
