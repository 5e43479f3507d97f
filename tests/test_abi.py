"""The C-ABI library: it builds, loads, exports every entry point the header
declares, and rejects bad arguments with a status before any device work
(these run without a GPU)."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2609_14991_gb300 as tsd
from paper_2609_14991_gb300 import _build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    _build.build()
    return tsd.lib()


def declared_entry_points():
    src = open(os.path.join(ROOT, "include", "tsd.h")).read()
    return set(re.findall(r"^TSD_API\s+[\w\s\*]*?\b(tsd_\w+)\s*\(", src, flags=re.M))


def test_every_declared_symbol_is_exported_and_bound(L):
    names = declared_entry_points()
    assert len(names) >= 20
    for n in sorted(names):
        assert hasattr(L, n), n  # dlsym succeeds
        assert n in tsd.SIGNATURES, f"binding lacks {n}"
    assert set(tsd.SIGNATURES) == names


def test_version(L):
    assert "sm_103a" in tsd.version()


def _status(L, fn, *args):
    st = fn(*args)
    return st, L.tsd_last_error().decode()


def test_ngram_build_rejects_bad_tables(L):
    h = ctypes.c_void_p()
    st, msg = _status(L, L.tsd_ngram_build, 4, 2, None, None, None, None, ctypes.byref(h))
    assert st == tsd.TSD_EINVAL and "NULL" in msg

    def build(order_tokens, order=2, V=4):
        toks = [np.ascontiguousarray(t, dtype=np.int32) for t in order_tokens]
        lps = [np.full(len(t), -1.0, dtype=np.float32) for t in toks]
        cnt = np.array([len(t) for t in toks], dtype=np.int64)
        tp = (ctypes.c_void_p * order)(*[t.ctypes.data for t in toks])
        lp = (ctypes.c_void_p * order)(*[t.ctypes.data for t in lps])
        return _status(L, L.tsd_ngram_build, V, order, cnt.ctypes.data, tp, lp, None, ctypes.byref(h))

    uni = [[0], [1], [2], [3]]
    st, msg = build([[[0], [1], [2]], [[0, 1]]])  # a unigram missing
    assert st == tsd.TSD_EINVAL and "unigram" in msg
    st, msg = build([uni, [[0, 9]]])  # label out of range
    assert st == tsd.TSD_EINVAL and "out of" in msg
    st, msg = build([uni, [[0, 1], [0, 1]]])  # duplicate
    assert st == tsd.TSD_EINVAL and "duplicate" in msg
    st, msg = build([uni, [[0, 1]], [[2, 0, 1]]], order=3)  # (2,0) missing: not prefix-closed
    assert st == tsd.TSD_EINVAL and "prefix" in msg
    st, msg = build([uni, [[2, 0], [0, 3]], [[2, 0, 1]]], order=3)  # (0,1) missing: not suffix-closed
    assert st == tsd.TSD_EINVAL and "suffix" in msg
    st, msg = _status(L, L.tsd_ngram_build, 4, 17, np.zeros(17, np.int64).ctypes.data, None, None, None,
                      ctypes.byref(h))
    assert st == tsd.TSD_EINVAL


def test_boost_build_rejects_bad_phrases(L):
    h = ctypes.c_void_p()

    def build(phrases, V=8):
        off = np.cumsum([0] + [len(p) for p in phrases]).astype(np.int32)
        tok = np.array([x for p in phrases for x in p] or [0], dtype=np.int32)
        return _status(L, L.tsd_boost_build, V, len(phrases), off.ctypes.data, tok.ctypes.data,
                       ctypes.c_float(1.0), ctypes.byref(h))

    st, msg = build([[1, 2], [3, 8]])
    assert st == tsd.TSD_EINVAL and "label" in msg
    st, msg = build([[1] * 33])
    assert st == tsd.TSD_EINVAL and "longer" in msg
    st, msg = build([[1, 2], []])
    assert st == tsd.TSD_EINVAL and "empty" in msg


def test_decoder_create_rejects_bad_config(L):
    h = ctypes.c_void_p()
    dummy = ctypes.c_void_p(16)  # never dereferenced: validation fails first
    for cfg, word in [((0, 64, 5, 1, 4, 13), "V="), ((16, 100, 5, 1, 4, 13), "H="), ((16, 64, 0, 1, 4, 13), "max_symbols"),
                      ((16, 64, 5, 1, 0, 13), "max_streams"), ((16, 64, 5, 1, 4, 0), "max_T")]:
        c = tsd.DecoderCfg(*cfg)
        st, msg = _status(L, L.tsd_decoder_create, ctypes.byref(c), dummy, dummy, None, None, None, ctypes.byref(h))
        assert st == tsd.TSD_EINVAL and word in msg, (cfg, msg)
    st, msg = _status(L, L.tsd_decoder_create, None, dummy, dummy, None, None, None, ctypes.byref(h))
    assert st == tsd.TSD_EINVAL


def test_null_handles(L):
    assert L.tsd_stream_open(None, None) == tsd.TSD_EINVAL
    assert L.tsd_stream_close(None, 0) == tsd.TSD_EINVAL
    assert L.tsd_decode_chunk(None, 1, None, None, 1, 0.0, 0.0, None, None, None, None, None) == tsd.TSD_EINVAL
    assert L.tsd_ngram_info(None, None, None, None) == tsd.TSD_EINVAL
    assert L.tsd_boost_info(None, None, None, None) == tsd.TSD_EINVAL
    L.tsd_ngram_free(None)
    L.tsd_boost_free(None)
    L.tsd_decoder_free(None)


def test_noalloc_binding_rejects_bad_tensors_before_the_call(L):
    """The allocation-free entry point's binding checks its tensors (types,
    shapes, dtypes, device) before anything reaches the library: a mismatched
    hidden size and host tensors both raise."""
    torch = pytest.importorskip("torch")
    A = torch.zeros((4, 64), dtype=torch.bfloat16)
    Wt = torch.zeros((17, 64), dtype=torch.int16)
    lab = torch.zeros(4, dtype=torch.int32)
    sc = torch.zeros(4, dtype=torch.float32)
    with pytest.raises(ValueError, match="H = 64"):
        tsd.joint_select_noalloc(A, torch.zeros((17, 128), dtype=torch.int16), None, lab, sc)
    with pytest.raises(ValueError, match="bias"):
        tsd.joint_select_noalloc(A, Wt, torch.zeros((4, 15), dtype=torch.float32), lab, sc)
    with pytest.raises(ValueError, match="out_label"):
        tsd.joint_select_noalloc(A, Wt, None, torch.zeros(3, dtype=torch.int32), sc)
    with pytest.raises(ValueError, match="A must be bf16"):
        tsd.joint_select_noalloc(A.float(), Wt, None, lab, sc)
    with pytest.raises(ValueError, match="CUDA tensor"):
        tsd.joint_select_noalloc(A, Wt, None, lab, sc)
    with pytest.raises(TypeError):
        tsd.joint_select_noalloc(np.zeros((4, 64)), Wt, None, lab, sc)


def test_checked_build_compiles():
    """The range-checked variant (-DTSD_CHECKS) of the fused row pass builds."""
    import subprocess

    src = os.path.join(ROOT, "paper_2609_14991_gb300", "csrc", "row_fused.cu")
    out = os.path.join(ROOT, "paper_2609_14991_gb300", "_build_checks")
    os.makedirs(out, exist_ok=True)
    cmd = [_build.nvcc()] + _build._flags() + ["-DTSD_CHECKS", "-x", "cu", "-c", src, "-o",
                                                os.path.join(out, "row_fused_check_probe.o")]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr[-2000:]


def test_debug_fail_alloc_rejects_negative(L):
    assert L.tsd_debug_fail_alloc(-1) == tsd.TSD_EINVAL
    assert L.tsd_debug_fail_alloc(0) == tsd.TSD_OK
