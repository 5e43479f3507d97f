"""Fused streaming Transducer decode with n-gram shallow fusion and phrase
boosting on one GB300 (sm_103a).

A thin ctypes binding over the C ABI in ``include/tsd.h`` (``libtsd.so``):
the functions below only marshal arguments.  Every step of the decode path
runs in the library's CUDA kernels; PyTorch is used for device memory and
streams.  There is no CPU fallback: if the library is not built, importing
the binding's entry points raises.

Typical use::

    lm = NGram(V, tokens_per_order, logp_per_order, bow_per_order)
    boost = Boost(V, offsets, tokens, bonus)
    dec = Decoder(V, H, W_out, E, lm=lm, boost=boost, max_streams=B, max_T=13)
    slots = [dec.open() for _ in range(B)]
    out = dec.decode_chunk(slots, enc, lam=0.5, beta=1.5)   # enc: cuda bf16 [B, T, H]
"""
from __future__ import annotations

import ctypes
import os
from typing import List, Optional, Sequence, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
# TSD_LIBRARY selects another build of the library (the range-checked
# libtsd_checks.so); by default the in-tree libtsd.so
LIB_PATH = os.environ.get("TSD_LIBRARY") or os.path.join(_HERE, "libtsd.so")

TSD_OK, TSD_EINVAL, TSD_ENOMEM, TSD_ECUDA, TSD_ESTATE, TSD_EDEVICE = 0, -1, -2, -3, -4, -5
_STATUS = {-1: "EINVAL", -2: "ENOMEM", -3: "ECUDA", -4: "ESTATE", -5: "EDEVICE"}

# every entry point declared in include/tsd.h: name -> (argtypes, restype)
_vp, _i32, _i64, _f32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float
_P = ctypes.POINTER


class PredWeightsC(ctypes.Structure):
    _fields_ = [("D", _i32), ("H_enc", _i32), ("emb", _vp), ("W_gates", _vp), ("b_gates", _vp), ("W_pred", _vp),
                ("b_pred", _vp), ("W_enc", _vp), ("b_enc", _vp)]


class DecoderCfg(ctypes.Structure):
    _fields_ = [("V", _i32), ("H", _i32), ("max_symbols", _i32), ("beam_k", _i32), ("max_streams", _i32),
                ("max_T", _i32), ("prune_k", _i32)]


class EncoderCfgC(ctypes.Structure):
    _fields_ = [(n, _i32) for n in ("d", "layers", "heads", "ff", "kernel", "left", "max_chunk", "feat", "stack",
                                    "max_streams")]


# field order of tsd_encoder_layer
_ENC_LAYER_FIELDS = ["ln_ff1_g", "ln_ff1_b", "ff1_w1", "ff1_b1", "ff1_w2", "ff1_b2", "ln_att_g", "ln_att_b", "qkv_w",
                     "qkv_b", "pos_w", "pos_u", "pos_v", "out_w", "out_b", "ln_conv_g", "ln_conv_b", "pw1_w", "pw1_b",
                     "dw_w", "dw_b", "bn_scale", "bn_shift", "pw2_w", "pw2_b", "ln_ff2_g", "ln_ff2_b", "ff2_w1",
                     "ff2_b1", "ff2_w2", "ff2_b2", "ln_out_g", "ln_out_b"]


class EncoderLayerC(ctypes.Structure):
    _fields_ = [(n, _vp) for n in _ENC_LAYER_FIELDS]


SIGNATURES = {
    "tsd_last_error": ([], ctypes.c_char_p),
    "tsd_version": ([], ctypes.c_char_p),
    "tsd_ngram_build": ([_i32, _i32, _vp, _vp, _vp, _vp, _P(_vp)], _i32),
    "tsd_ngram_free": ([_vp], None),
    "tsd_ngram_info": ([_vp, _P(_i64), _P(_i64), _P(_i64)], _i32),
    "tsd_ngram_state_tuple": ([_vp, _i32, _vp, _i32, _P(_i32)], _i32),
    "tsd_boost_build": ([_i32, _i32, _vp, _vp, _f32, _P(_vp)], _i32),
    "tsd_boost_free": ([_vp], None),
    "tsd_boost_info": ([_vp, _P(_i32), _P(_i32), _P(_i64)], _i32),
    "tsd_boost_node_tuple": ([_vp, _i32, _vp, _i32, _P(_i32)], _i32),
    "tsd_decoder_create": ([_P(DecoderCfg), _vp, _vp, _vp, _vp, _vp, _P(_vp)], _i32),
    "tsd_decoder_create_multi": ([_P(DecoderCfg), _vp, _vp, _vp, _vp, _i32, _vp, _vp, _P(_vp)], _i32),
    "tsd_stream_lm_state": ([_vp, _i32, _i32, _P(_i32)], _i32),
    "tsd_decoder_create_pred": ([_P(DecoderCfg), _P(PredWeightsC), _vp, _vp, _vp, _vp, _P(_vp)], _i32),
    "tsd_stream_pred_state": ([_vp, _i32, _vp, _vp], _i32),
    "tsd_stream_export": ([_vp, _i32, _vp, _i64, _P(_i64)], _i32),
    "tsd_stream_import": ([_vp, _i32, _vp, _i64], _i32),
    "tsd_decoder_free": ([_vp], None),
    "tsd_stream_open": ([_vp, _P(_i32)], _i32),
    "tsd_stream_close": ([_vp, _i32], _i32),
    "tsd_decode_chunk": ([_vp, _i32, _vp, _vp, _i32, _f32, _f32, _vp, _vp, _vp, _vp, _vp], _i32),
    "tsd_stream_state": ([_vp, _i32, _P(_i32), _P(_i32), _P(_i32)], _i32),
    "tsd_stream_result": ([_vp, _i32, _vp, _i32, _P(_i32), _P(_f32)], _i32),
    "tsd_stream_hyps": ([_vp, _i32, _vp, _i32, _vp, _vp, _i32, _P(_i32)], _i32),
    "tsd_decoder_set_graphs": ([_vp, _i32], _i32),
    "tsd_decoder_set_timing": ([_vp, _i32], _i32),
    "tsd_decoder_timing": ([_vp, _vp, _vp, _i32, _i32], _i32),
    "tsd_decoder_launches_per_chunk": ([_vp, _i32, _i32, _P(_i64)], _i32),
    "tsd_arpa_parse": ([ctypes.c_char_p, _i64, _i32, _vp, _P(_vp)], _i32),
    "tsd_arpa_info": ([_vp, _P(_i32), _vp, _i32, _P(_i64)], _i32),
    "tsd_arpa_arrays": ([_vp, _i32, _P(_vp), _P(_vp), _P(_vp)], _i32),
    "tsd_arpa_free": ([_vp], None),
    "tsd_ngram_build_arpa": ([ctypes.c_char_p, _i64, _i32, _vp, _P(_vp)], _i32),
    "tsd_decoder_timed_bytes": ([_vp, _P(_i64), _i32], _i32),
    "tsd_decoder_debug_capture": ([_vp, _vp, _vp, _i32], _i32),
    "tsd_decoder_set_joint_kernel": ([_vp, _i32], _i32),
    "tsd_decoder_check": ([_vp], _i32),
    "tsd_decoder_set_option": ([_vp, ctypes.c_char_p, _i64], _i32),
    "tsd_decoder_replay": ([_vp, _i32, _i32, _vp, _P(_i64)], _i32),
    "tsd_joint_select_noalloc": ([_i32, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp], _i32),
    "tsd_debug_fail_alloc": ([_i32], _i32),
    "tsd_encoder_create": ([_P(EncoderCfgC), _vp, _vp, _vp, _vp, _P(_vp)], _i32),
    "tsd_encoder_free": ([_vp], None),
    "tsd_encoder_open": ([_vp, _P(_i32)], _i32),
    "tsd_encoder_close": ([_vp, _i32], _i32),
    "tsd_encode_chunk": ([_vp, _i32, _vp, _vp, _i32, _vp, _vp], _i32),
    "tsd_encoder_check": ([_vp], _i32),
    "tsd_encoder_set_timing": ([_vp, _i32], _i32),
    "tsd_encoder_timing": ([_vp, _vp, _vp, _i32, _i32], _i32),
    "tsd_encoder_gemm_flops": ([_vp, _i32, _i32, _P(ctypes.c_double)], _i32),
    "tsd_encoder_launches_per_chunk": ([_vp, _i32, _i32, _P(_i64)], _i32),
}

_lib = None


class TsdError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"tsd {_STATUS.get(status, status)}: {msg}")
        self.status = status


def lib() -> ctypes.CDLL:
    """The loaded library.  Raises if it has not been built: there is no
    fallback implementation."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it first (python -c 'import __graft_entry__ as g; "
                               "g.build()')")
        L = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in SIGNATURES.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _check(st: int):
    if st != TSD_OK:
        raise TsdError(st, lib().tsd_last_error().decode())


def version() -> str:
    return lib().tsd_version().decode()


def _i32arr(x) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(x, dtype=np.int32))


def _ptr(t) -> int:
    """Device or host address of a torch tensor / numpy array."""
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> int:
    import torch

    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


class NGram:
    """Backoff n-gram tables on the device (``tsd_ngram_build``)."""

    def __init__(self, V: int, tokens: Sequence[np.ndarray], logp: Sequence[np.ndarray],
                 bow: Optional[Sequence[np.ndarray]] = None):
        order = len(tokens)
        toks = [np.ascontiguousarray(t, dtype=np.int32) for t in tokens]
        lps = [np.ascontiguousarray(x, dtype=np.float32) for x in logp]
        bws = [np.ascontiguousarray(x, dtype=np.float32) for x in bow] if bow is not None else None
        cnt = np.array([len(x) for x in lps], dtype=np.int64)
        tp = (_vp * order)(*[t.ctypes.data for t in toks])
        lp = (_vp * order)(*[t.ctypes.data for t in lps])
        bp = (_vp * order)(*[t.ctypes.data for t in bws]) if bws is not None else None
        h = _vp()
        _check(lib().tsd_ngram_build(V, order, cnt.ctypes.data, tp, lp, bp, ctypes.byref(h)))
        self.h, self.V, self.order = h, V, order

    @classmethod
    def from_arrays(cls, a) -> "NGram":
        return cls(a.V, a.tokens, a.logp, a.bow)

    @classmethod
    def from_arpa(cls, text, V: int, vocab: Optional[Sequence[str]] = None) -> "NGram":
        """Tables from ARPA text (``tsd_ngram_build_arpa``)."""
        data = text.encode() if isinstance(text, str) else bytes(text)
        keep, vp = _vocab(vocab, V)
        h = _vp()
        _check(lib().tsd_ngram_build_arpa(data, len(data), V, vp, ctypes.byref(h)))
        obj = cls.__new__(cls)
        obj.h, obj.V = h, V
        obj.order = 0
        return obj

    def info(self) -> Tuple[int, int, int]:
        s, a, b = _i64(), _i64(), _i64()
        _check(lib().tsd_ngram_info(self.h, ctypes.byref(s), ctypes.byref(a), ctypes.byref(b)))
        return s.value, a.value, b.value

    def state_tuple(self, state: int) -> Tuple[int, ...]:
        buf = np.zeros(16, dtype=np.int32)
        n = _i32()
        _check(lib().tsd_ngram_state_tuple(self.h, int(state), buf.ctypes.data, 16, ctypes.byref(n)))
        return tuple(int(x) for x in buf[: n.value])

    def __del__(self):
        if getattr(self, "h", None):
            lib().tsd_ngram_free(self.h)
            self.h = None


class Boost:
    """Phrase-boosting trie on the device (``tsd_boost_build``)."""

    def __init__(self, V: int, offsets, tokens, bonus: float):
        off = _i32arr(offsets)
        tok = _i32arr(tokens) if len(tokens) else np.zeros(1, dtype=np.int32)
        h = _vp()
        _check(lib().tsd_boost_build(V, len(off) - 1, off.ctypes.data, tok.ctypes.data, float(bonus),
                                     ctypes.byref(h)))
        self.h, self.V = h, V

    @classmethod
    def from_phrases(cls, V: int, p, bonus: float) -> "Boost":
        return cls(V, p.offsets, p.tokens, bonus)

    def info(self) -> Tuple[int, int, int]:
        q, d, b = _i32(), _i32(), _i64()
        _check(lib().tsd_boost_info(self.h, ctypes.byref(q), ctypes.byref(d), ctypes.byref(b)))
        return q.value, d.value, b.value

    def node_tuple(self, node: int) -> Tuple[int, ...]:
        buf = np.zeros(32, dtype=np.int32)
        n = _i32()
        _check(lib().tsd_boost_node_tuple(self.h, int(node), buf.ctypes.data, 32, ctypes.byref(n)))
        return tuple(int(x) for x in buf[: n.value])

    def __del__(self):
        if getattr(self, "h", None):
            lib().tsd_boost_free(self.h)
            self.h = None


def debug_fail_alloc(n: int):
    """Test hook: the n-th device allocation from now on fails (0: off)."""
    _check(lib().tsd_debug_fail_alloc(int(n)))


def joint_select_noalloc(A, Wt, bias, out_label, out_score, stream=None):
    """Allocation-free joint selection (tsd_joint_select_noalloc): for callers
    that cannot allocate device memory.  A: cuda bf16 [n, H]; Wt: cuda bf16
    [V+1, H]; bias: cuda fp32 [n, V] or None; out_label: cuda int32 [n];
    out_score: cuda fp32 [n].  Nothing is allocated by this call."""
    import torch

    named = {"A": A, "Wt": Wt, "out_label": out_label, "out_score": out_score}
    if bias is not None:
        named["bias"] = bias
    for name, t in named.items():
        if not isinstance(t, torch.Tensor):
            raise TypeError(f"joint_select_noalloc: {name} must be a torch tensor")
    if A.dim() != 2 or A.dtype != torch.bfloat16:
        raise ValueError("joint_select_noalloc: A must be bf16 [n, H]")
    n, H = A.shape
    if Wt.dim() != 2 or Wt.element_size() != 2 or Wt.shape[1] != H:
        raise ValueError(f"joint_select_noalloc: Wt must be 2-byte [V+1, H] with H = {H}")
    V = Wt.shape[0] - 1
    if bias is not None and (bias.dtype != torch.float32 or tuple(bias.shape) != (n, V)):
        raise ValueError(f"joint_select_noalloc: bias must be float32 [{n}, {V}]")
    if out_label.dtype != torch.int32 or out_label.numel() < n:
        raise ValueError(f"joint_select_noalloc: out_label must be int32 with at least {n} elements")
    if out_score.dtype != torch.float32 or out_score.numel() < n:
        raise ValueError(f"joint_select_noalloc: out_score must be float32 with at least {n} elements")
    dev = torch.cuda.current_device() if torch.cuda.is_available() else None
    for name, t in named.items():
        if not t.is_cuda or t.device.index != dev:
            raise ValueError(f"joint_select_noalloc: {name} must be a CUDA tensor on the current device")
        if not t.is_contiguous():
            raise ValueError(f"joint_select_noalloc: {name} must be contiguous")
    _check(lib().tsd_joint_select_noalloc(n, H, V, _ptr(A), _ptr(Wt), _ptr(bias) if bias is not None else None,
                                          _ptr(out_label), _ptr(out_score), _stream(stream)))


class ChunkOut:
    """Device outputs of one decode_chunk call (torch tensors)."""

    def __init__(self, tokens, frames, scores, counts):
        self.tokens, self.frames, self.scores, self.counts = tokens, frames, scores, counts


class Decoder:
    """A decoder on the current CUDA device (``tsd_decoder_create``)."""

    def __init__(self, V: int, H: int, W_out, E, lm: Optional[NGram] = None, boost: Optional[Boost] = None,
                 max_symbols: int = 5, beam_k: int = 1, max_streams: int = 64, max_T: int = 64, stream=None,
                 lms: Optional[Sequence[Tuple[NGram, float]]] = None, prune_k: int = 0, pred=None):
        """lms: several LMs as (NGram, w) pairs instead of lm (LM i enters Eq. 1
        with weight lambda * w; ``tsd_decoder_create_multi``).  prune_k > 0:
        pruned fusion over the acoustic model's prune_k best outputs.  pred:
        the stateful form's weights (fields D, Henc, Ep, Wg, bg, Wp, bp, We, be
        as numpy arrays, bf16 bit patterns and fp32 biases;
        ``tsd_decoder_create_pred``); E is then ignored."""
        import torch

        assert W_out.is_cuda and E.is_cuda and W_out.element_size() == 2 and E.element_size() == 2
        assert tuple(W_out.shape) == (H, V + 1) and tuple(E.shape) == (V + 1, H)
        self.cfg = DecoderCfg(V, H, max_symbols, beam_k, max_streams, max_T, prune_k)
        self.V, self.H, self.max_symbols, self.beam_k = V, H, max_symbols, beam_k
        self.lm, self.boost = lm, boost  # kept alive: the decoder borrows them
        W_out = W_out.contiguous()
        E = E.contiguous()
        h = _vp()
        if pred is not None:
            dev = W_out.device
            up16 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev)
            up32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)
            t = dict(emb=up16(pred.Ep), Wg=up16(pred.Wg), bg=up32(pred.bg), Wp=up16(pred.Wp), bp=up32(pred.bp),
                     We=up16(pred.We), be=up32(pred.be))
            self._pred_keep = t
            self.pred_D = pred.D
            self.pred_Henc = pred.Henc
            pw = PredWeightsC(pred.D, pred.Henc, _ptr(t["emb"]), _ptr(t["Wg"]), _ptr(t["bg"]), _ptr(t["Wp"]),
                              _ptr(t["bp"]), _ptr(t["We"]), _ptr(t["be"]))
            _check(lib().tsd_decoder_create_pred(ctypes.byref(self.cfg), ctypes.byref(pw), _ptr(W_out),
                                                 lm.h if lm else None, boost.h if boost else None, _stream(stream),
                                                 ctypes.byref(h)))
        elif lms is not None:
            assert lm is None, "give lm or lms, not both"
            self.lm = [m for m, _ in lms]
            hs = (_vp * max(1, len(lms)))(*[m.h for m, _ in lms])
            ws = np.array([w for _, w in lms] or [0.0], dtype=np.float32)
            _check(lib().tsd_decoder_create_multi(ctypes.byref(self.cfg), _ptr(W_out), _ptr(E), hs, ws.ctypes.data,
                                                  len(lms), boost.h if boost else None, _stream(stream),
                                                  ctypes.byref(h)))
        else:
            _check(lib().tsd_decoder_create(ctypes.byref(self.cfg), _ptr(W_out), _ptr(E), lm.h if lm else None,
                                            boost.h if boost else None, _stream(stream), ctypes.byref(h)))
        self.h = h
        self._keep = []

    def __del__(self):
        if getattr(self, "h", None):
            lib().tsd_decoder_free(self.h)
            self.h = None

    def open(self) -> int:
        s = _i32()
        _check(lib().tsd_stream_open(self.h, ctypes.byref(s)))
        return s.value

    def close(self, slot: int):
        _check(lib().tsd_stream_close(self.h, int(slot)))

    def alloc_out(self, n: int, T: int) -> ChunkOut:
        import torch

        cap = T * self.max_symbols
        dev = torch.device("cuda", torch.cuda.current_device())
        return ChunkOut(torch.empty((n, cap), dtype=torch.int32, device=dev),
                        torch.empty((n, cap), dtype=torch.int32, device=dev),
                        torch.empty((n, cap), dtype=torch.float32, device=dev),
                        torch.empty((n,), dtype=torch.int32, device=dev))

    def decode_chunk(self, slots: Sequence[int], enc, lam: float, beta: float, out: Optional[ChunkOut] = None,
                     stream=None) -> ChunkOut:
        """enc: cuda bf16 (or int16/uint16 bit patterns) [n, T, H]."""
        n, T, H = enc.shape
        assert n == len(slots) and H == getattr(self, "pred_Henc", self.H) and enc.is_cuda and enc.is_contiguous()
        if out is None:
            out = self.alloc_out(n, T)
        sl = _i32arr(slots)
        _check(lib().tsd_decode_chunk(self.h, n, sl.ctypes.data, _ptr(enc), T, float(lam), float(beta),
                                      _ptr(out.tokens), _ptr(out.frames), _ptr(out.scores), _ptr(out.counts),
                                      _stream(stream)))
        return out

    def decode_chunk_raw(self, slots_np: np.ndarray, enc_ptr: int, T: int, lam: float, beta: float,
                         out_ptrs: Tuple[int, int, int, int], stream_handle: int):
        """Pointer-level call (for timing loops)."""
        _check(lib().tsd_decode_chunk(self.h, len(slots_np), slots_np.ctypes.data, enc_ptr, T, float(lam),
                                      float(beta), out_ptrs[0], out_ptrs[1], out_ptrs[2], out_ptrs[3],
                                      stream_handle))

    def state(self, slot: int) -> Tuple[int, int, int]:
        a, b, c = _i32(), _i32(), _i32()
        _check(lib().tsd_stream_state(self.h, int(slot), ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)))
        return a.value, b.value, c.value

    def export_state(self, slot: int) -> bytes:
        """The slot's decoding state as bytes (``tsd_stream_export``)."""
        n = _i64()
        _check(lib().tsd_stream_export(self.h, int(slot), None, 0, ctypes.byref(n)))
        buf = ctypes.create_string_buffer(max(1, n.value))
        _check(lib().tsd_stream_export(self.h, int(slot), buf, n.value, ctypes.byref(n)))
        return buf.raw[: n.value]

    def import_state(self, slot: int, blob: bytes):
        """Continues an exported stream in an open slot (``tsd_stream_import``)."""
        buf = ctypes.create_string_buffer(bytes(blob), len(blob))
        _check(lib().tsd_stream_import(self.h, int(slot), buf, len(blob)))

    def pred_state(self, slot: int):
        """(h as bf16 bits [D], c [D]) of a stateful-form stream."""
        h = np.zeros(self.pred_D, dtype=np.uint16)
        c = np.zeros(self.pred_D, dtype=np.float32)
        _check(lib().tsd_stream_pred_state(self.h, int(slot), h.ctypes.data, c.ctypes.data))
        return h, c

    def lm_state(self, slot: int, lm_index: int) -> int:
        """State id of LM lm_index for a slot (``tsd_stream_lm_state``)."""
        x = _i32()
        _check(lib().tsd_stream_lm_state(self.h, int(slot), int(lm_index), ctypes.byref(x)))
        return x.value

    def result(self, slot: int, cap: int = 1 << 16) -> Tuple[List[int], float]:
        buf = np.zeros(cap, dtype=np.int32)
        n, sc = _i32(), _f32()
        _check(lib().tsd_stream_result(self.h, int(slot), buf.ctypes.data, cap, ctypes.byref(n), ctypes.byref(sc)))
        return [int(x) for x in buf[: min(n.value, cap)]], sc.value

    def hyps(self, slot: int, cap_len: int = 4096) -> List[Tuple[List[int], float]]:
        K = self.beam_k
        buf = np.zeros(K * cap_len, dtype=np.int32)
        lens = np.zeros(K, dtype=np.int32)
        scs = np.zeros(K, dtype=np.float32)
        nh = _i32()
        _check(lib().tsd_stream_hyps(self.h, int(slot), buf.ctypes.data, cap_len, lens.ctypes.data,
                                     scs.ctypes.data, K, ctypes.byref(nh)))
        return [([int(x) for x in buf[i * cap_len: i * cap_len + min(lens[i], cap_len)]], float(scs[i]))
                for i in range(nh.value)]

    def set_graphs(self, enable: bool):
        _check(lib().tsd_decoder_set_graphs(self.h, 1 if enable else 0))

    def set_joint_kernel(self, kind: int):
        """0 = tcgen05 tensor-core GEMM (default), 1 = CUDA-core cross-check kernel."""
        _check(lib().tsd_decoder_set_joint_kernel(self.h, int(kind)))

    def set_option(self, name: str, value: int):
        _check(lib().tsd_decoder_set_option(self.h, name.encode(), int(value)))

    def replay(self, kernel: int, reps: int, stream=None, count_bytes: bool = False) -> int:
        """Re-launch one kernel (0 row pass, 1 joint) of the last chunk's final
        step reps times, for timing; with count_bytes, returns the algorithmic
        bytes of one launch (and waits for the stream)."""
        b = _i64(0)
        _check(lib().tsd_decoder_replay(self.h, int(kernel), int(reps), _stream(stream),
                                        ctypes.byref(b) if count_bytes else None))
        return b.value

    def check(self):
        """Raises TsdError(EDEVICE) if a bounded device wait expired."""
        _check(lib().tsd_decoder_check(self.h))

    def set_timing(self, enable: bool):
        _check(lib().tsd_decoder_set_timing(self.h, 1 if enable else 0))

    def timing(self, reset: bool = False):
        """({'row': ms, 'joint': ms, 'pred': ms}, {... launches}): device time
        of timed chunks per kernel class; 'pred' is the stateful form's
        prediction network and projections."""
        ms = np.zeros(3, dtype=np.float64)
        ln = np.zeros(3, dtype=np.int64)
        _check(lib().tsd_decoder_timing(self.h, ms.ctypes.data, ln.ctypes.data, 3, 1 if reset else 0))
        keys = ("row", "joint", "pred")
        return {k: float(ms[i]) for i, k in enumerate(keys)}, {k: int(ln[i]) for i, k in enumerate(keys)}

    def timed_bytes(self, reset: bool = False) -> int:
        """Algorithmic bytes counted by the row passes of timed chunks."""
        x = _i64()
        _check(lib().tsd_decoder_timed_bytes(self.h, ctypes.byref(x), 1 if reset else 0))
        return x.value

    def launches_per_chunk(self, n: int, T: int) -> int:
        x = _i64()
        _check(lib().tsd_decoder_launches_per_chunk(self.h, n, T, ctypes.byref(x)))
        return x.value

    def debug_capture(self, logits=None, rows=None, max_steps: int = 0):
        self._keep = [logits, rows]
        _check(lib().tsd_decoder_debug_capture(self.h, _ptr(logits) if logits is not None else None,
                                               _ptr(rows) if rows is not None else None, int(max_steps)))


def _vocab(vocab, V):
    if vocab is None:
        return None, None
    if len(vocab) != V:
        raise ValueError("vocabulary has %d words, V=%d" % (len(vocab), V))
    keep = [w.encode() if isinstance(w, str) else bytes(w) for w in vocab]
    arr = (ctypes.c_char_p * V)(*keep)
    return (keep, arr), ctypes.cast(arr, ctypes.c_void_p)


def parse_arpa(text, V: int, vocab: Optional[Sequence[str]] = None):
    """(tokens per order, logp per order, bow per order, dropped lines) of
    ARPA text, read by the library's host parser (``tsd_arpa_parse``)."""
    data = text.encode() if isinstance(text, str) else bytes(text)
    keep, vp = _vocab(vocab, V)
    h = _vp()
    _check(lib().tsd_arpa_parse(data, len(data), V, vp, ctypes.byref(h)))
    try:
        order = _i32()
        skipped = _i64()
        counts = np.zeros(16, dtype=np.int64)
        _check(lib().tsd_arpa_info(h, ctypes.byref(order), counts.ctypes.data, 16, ctypes.byref(skipped)))
        toks, lps, bws = [], [], []
        for k in range(1, order.value + 1):
            tp, lp, bp = _vp(), _vp(), _vp()
            _check(lib().tsd_arpa_arrays(h, k, ctypes.byref(tp), ctypes.byref(lp), ctypes.byref(bp)))
            n = int(counts[k - 1])
            if n:
                toks.append(np.ctypeslib.as_array(ctypes.cast(tp, ctypes.POINTER(ctypes.c_int32)), (n * k,))
                            .reshape(n, k).copy())
                lps.append(np.ctypeslib.as_array(ctypes.cast(lp, ctypes.POINTER(ctypes.c_float)), (n,)).copy())
                bws.append(np.ctypeslib.as_array(ctypes.cast(bp, ctypes.POINTER(ctypes.c_float)), (n,)).copy())
            else:
                toks.append(np.zeros((0, k), dtype=np.int32))
                lps.append(np.zeros(0, dtype=np.float32))
                bws.append(np.zeros(0, dtype=np.float32))
        return toks, lps, bws, int(skipped.value)
    finally:
        lib().tsd_arpa_free(h)


class Encoder:
    """The cache-aware encoder chunk step on the current CUDA device
    (``tsd_encoder_create``).  weights: an object with fields cfg (d, layers,
    heads, ff, kernel, left, chunk, feat, stack), sub_w, sub_b and layers (each
    with the fields of ``tsd_encoder_layer``; a layer norm as a (gamma, beta)
    pair named ln_ff1, ln_att, ln_conv, ln_ff2, ln_out), numpy arrays of bf16
    bit patterns (matrices) and float32 (vectors)."""

    def __init__(self, weights, max_streams: int = 64, max_chunk: Optional[int] = None, stream=None):
        import torch

        c = weights.cfg
        self.d, self.stack, self.feat = c.d, c.stack, c.feat
        self.max_chunk = max_chunk or c.chunk
        self.cfg = EncoderCfgC(c.d, len(weights.layers), c.heads, c.ff, c.kernel, c.left, self.max_chunk, c.feat,
                               c.stack, max_streams)
        dev = torch.device("cuda", torch.cuda.current_device())

        def up(a):
            a = np.ascontiguousarray(a)
            if a.dtype == np.uint16:
                return torch.from_numpy(a.view(np.int16)).to(dev)
            return torch.from_numpy(a.astype(np.float32)).to(dev)

        keep = [up(weights.sub_w), up(weights.sub_b)]
        layers = (EncoderLayerC * len(weights.layers))()
        for i, L in enumerate(weights.layers):
            vals = {}
            for name in ("ln_ff1", "ln_att", "ln_conv", "ln_ff2", "ln_out"):
                g, b = getattr(L, name)
                vals[name + "_g"], vals[name + "_b"] = up(g), up(b)
            for name in _ENC_LAYER_FIELDS:
                if name not in vals:
                    vals[name] = up(getattr(L, name))
            keep.extend(vals.values())
            for name in _ENC_LAYER_FIELDS:
                setattr(layers[i], name, _ptr(vals[name]))
        h = _vp()
        _check(lib().tsd_encoder_create(ctypes.byref(self.cfg), _ptr(keep[0]), _ptr(keep[1]), ctypes.cast(layers, _vp),
                                        _stream(stream), ctypes.byref(h)))
        self.h = h  # the encoder copied every weight; the uploads can go

    def __del__(self):
        if getattr(self, "h", None):
            lib().tsd_encoder_free(self.h)
            self.h = None

    def open(self) -> int:
        s = _i32()
        _check(lib().tsd_encoder_open(self.h, ctypes.byref(s)))
        return s.value

    def close(self, slot: int):
        _check(lib().tsd_encoder_close(self.h, int(slot)))

    def encode_chunk(self, slots: Sequence[int], feats, out=None, stream=None):
        """feats: cuda bf16 (or int16 bit patterns) [n, C*stack, feat] ->
        out: cuda int16 (bf16 bit patterns) [n, C, d]."""
        import torch

        n = len(slots)
        assert feats.is_cuda and feats.element_size() == 2 and feats.shape[0] == n
        assert feats.shape[2] == self.feat and feats.shape[1] % self.stack == 0
        C = feats.shape[1] // self.stack
        feats = feats.contiguous()
        if out is None:
            out = torch.empty((n, C, self.d), dtype=torch.int16, device=feats.device)
        sl = _i32arr(slots)
        _check(lib().tsd_encode_chunk(self.h, n, sl.ctypes.data, _ptr(feats), C, _ptr(out), _stream(stream)))
        return out

    def encode_chunk_raw(self, slots_np: np.ndarray, feats_ptr: int, C: int, out_ptr: int, stream_handle: int):
        _check(lib().tsd_encode_chunk(self.h, len(slots_np), slots_np.ctypes.data, feats_ptr, C, out_ptr,
                                      stream_handle))

    def check(self):
        _check(lib().tsd_encoder_check(self.h))

    def set_timing(self, on: bool):
        _check(lib().tsd_encoder_set_timing(self.h, 1 if on else 0))

    def timing(self, reset: bool = False):
        """({'gemm': ms, 'attention': ms, 'other': ms}, {... launches})"""
        ms = np.zeros(3, dtype=np.float64)
        ln = np.zeros(3, dtype=np.int64)
        _check(lib().tsd_encoder_timing(self.h, ms.ctypes.data, ln.ctypes.data, 3, 1 if reset else 0))
        keys = ("gemm", "attention", "other")
        return {k: float(ms[i]) for i, k in enumerate(keys)}, {k: int(ln[i]) for i, k in enumerate(keys)}

    def gemm_flops(self, n: int, C: int) -> float:
        x = ctypes.c_double()
        _check(lib().tsd_encoder_gemm_flops(self.h, n, C, ctypes.byref(x)))
        return x.value

    def launches_per_chunk(self, n: int, C: int) -> int:
        """Kernel launches of one encode_chunk(n, C) with timing off."""
        x = _i64()
        _check(lib().tsd_encoder_launches_per_chunk(self.h, int(n), int(C), ctypes.byref(x)))
        return x.value
