"""Incremental ViT encoding on GB300: Python binding of the C ABI in ``include/ivit.h``.

The functions below carry the C entry points' names and only marshal arguments
(torch tensors -> raw pointers, torch streams -> cudaStream_t); every step of the
encode runs in the CUDA library ``_build/libivit.so``.  There is no fallback: if the
library is missing, loading fails with an error that says how to build it.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional, Tuple

import numpy as np

from . import synth

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libivit.so")

IVIT_OK = 0
IVIT_ERR_ARG = -1
IVIT_ERR_SHAPE = -2
IVIT_ERR_OOM = -3
IVIT_ERR_CUDA = -4
IVIT_ERR_DEVICE = -5

EXPORTED = [
    "ivit_weights_size", "ivit_create", "ivit_encode_full", "ivit_encode_incremental",
    "ivit_get_changed", "ivit_get_cache", "ivit_reset", "ivit_timeline",
    "ivit_timeline_read", "ivit_device_status", "ivit_last_launch_count", "ivit_destroy",
    "ivit_last_error", "ivit_select_noalloc", "ivit_action_combine",
]
IVIT_NOALLOC_MAX_TOKENS = 65536


class IvitConfig(C.Structure):
    _fields_ = [
        ("img_h", C.c_int32), ("img_w", C.c_int32), ("patch", C.c_int32),
        ("dim", C.c_int32), ("depth", C.c_int32), ("heads", C.c_int32),
        ("mlp_dim", C.c_int32), ("n_streams", C.c_int32), ("n_views", C.c_int32),
        ("ln_eps", C.c_float), ("gelu", C.c_int32), ("select_mode", C.c_int32),
        ("threshold", C.c_float), ("topk", C.c_int32), ("ref_mode", C.c_int32),
        ("score_source", C.c_int32), ("schedule", C.c_int32), ("mlp_tokens", C.c_int32),
    ]


class IvitError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"ivit error {code}: {msg}")
        self.code = code


_lib: Optional[C.CDLL] = None


def load(path: str = LIB_PATH) -> C.CDLL:
    """Loads the CUDA library (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    L = C.CDLL(path)
    P, I, I64 = C.c_void_p, C.c_int, C.c_int64
    L.ivit_weights_size.restype = C.c_size_t
    L.ivit_weights_size.argtypes = [C.POINTER(IvitConfig)]
    L.ivit_create.argtypes = [C.POINTER(IvitConfig), P, C.POINTER(P)]
    L.ivit_encode_full.argtypes = [P, P, P, P]
    L.ivit_encode_incremental.argtypes = [P, P, P, P, P]
    L.ivit_get_changed.argtypes = [P, I, P, P, P]
    L.ivit_get_cache.argtypes = [P, I, I, P, P]
    L.ivit_reset.argtypes = [P, I]
    L.ivit_timeline.argtypes = [P, I]
    L.ivit_timeline_read.argtypes = [P, P, C.POINTER(C.c_double), C.POINTER(I64), C.POINTER(C.c_double),
                                     C.POINTER(C.c_double)]
    L.ivit_device_status.argtypes = [P, P]
    L.ivit_last_launch_count.restype = I64
    L.ivit_last_launch_count.argtypes = [P]
    L.ivit_destroy.argtypes = [P]
    L.ivit_destroy.restype = None
    L.ivit_last_error.restype = C.c_char_p
    L.ivit_last_error.argtypes = [P]
    L.ivit_action_combine.argtypes = [P, P, P, P, P, P, C.c_int32, C.c_int32, P, P]
    L.ivit_select_noalloc.argtypes = [P, P, C.c_int32, C.c_int32, C.c_int32, C.c_int32,
                                      C.c_float, C.c_int32, P, P, P]
    _lib = L
    return L


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _require(t, name: str, dtype_name: str, numel: int) -> None:
    """Rejects a tensor that the kernels would misread or index out of bounds: one in host
    memory, of another dtype (``dtype_name`` is the torch dtype's name, e.g. "uint8"), a
    non-contiguous view, or one with fewer than ``numel`` elements.  ``None`` (an optional
    output) and raw integer pointers pass unchecked: the caller vouches for those."""
    if t is None or isinstance(t, int):
        return
    if isinstance(t, np.ndarray):
        raise TypeError(f"{name}: a numpy array (host memory); a CUDA tensor is required")
    if t.device.type != "cuda":
        raise ValueError(f"{name}: tensor on {t.device}; a CUDA tensor is required")
    if str(t.dtype) != "torch." + dtype_name:
        raise TypeError(f"{name}: dtype {t.dtype}, expected torch.{dtype_name}")
    if not t.is_contiguous():
        raise ValueError(f"{name}: not contiguous")
    if t.numel() < numel:
        raise ValueError(f"{name}: {t.numel()} elements, the call needs {numel}")


# handle -> (views, frame bytes per view, tokens per view, width), registered at create so
# that the entry points can check the tensors they are given against the encoder's sizes
_dims = {}


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def make_config(shape: "synth.EncoderShape", n_streams: int = 1, n_views: int = 1,
                select_mode: int = synth.SEL_THRESHOLD, threshold: float = 0.98, topk: int = 0,
                ref_mode: int = synth.REF_PREV_FRAME, score_source: int = synth.SCORE_EMBED,
                schedule: int = synth.SCHED_INCREMENTAL, mlp_tokens: int = 0) -> IvitConfig:
    return IvitConfig(shape.img_h, shape.img_w, shape.patch, shape.dim, shape.depth, shape.heads,
                      shape.mlp_dim, n_streams, n_views, shape.ln_eps, shape.gelu, select_mode,
                      threshold, topk, ref_mode, score_source, schedule, mlp_tokens)


# ------------------------------------------------------------- C entry points

def ivit_weights_size(cfg: IvitConfig) -> int:
    return int(load().ivit_weights_size(C.byref(cfg)))


def ivit_last_error(handle: Optional[int] = None) -> str:
    return load().ivit_last_error(handle).decode(errors="replace")


def _check(code: int, handle: Optional[int]) -> int:
    if code < 0:
        raise IvitError(code, ivit_last_error(handle))
    return code


def ivit_create(cfg: IvitConfig, weights_u16: np.ndarray) -> int:
    w = np.ascontiguousarray(weights_u16, dtype=np.uint16)
    h = C.c_void_p()
    _check(load().ivit_create(C.byref(cfg), w.ctypes.data, C.byref(h)), None)
    n_tok = (cfg.img_h // cfg.patch) * (cfg.img_w // cfg.patch)
    _dims[h.value] = (cfg.n_streams * cfg.n_views, cfg.img_h * cfg.img_w * 3, n_tok, cfg.dim)
    return h.value


def _check_call(h: int, frames, tokens_out, changed_count=None) -> None:
    if h not in _dims:
        return  # a handle created outside this module: sizes unknown here
    sv, fbytes, n_tok, dim = _dims[h]
    _require(frames, "frames", "uint8", sv * fbytes)
    _require(tokens_out, "tokens_out", "bfloat16", sv * n_tok * dim)
    _require(changed_count, "changed_count", "int32", sv)


def ivit_encode_full(h: int, frames, tokens_out=None, stream=None) -> None:
    _check_call(h, frames, tokens_out)
    _check(load().ivit_encode_full(h, _ptr(frames), _ptr(tokens_out), _stream(stream)), h)


def ivit_encode_incremental(h: int, frames, tokens_out=None, changed_count=None,
                            stream=None) -> None:
    _check_call(h, frames, tokens_out, changed_count)
    _check(load().ivit_encode_incremental(h, _ptr(frames), _ptr(tokens_out),
                                          _ptr(changed_count), _stream(stream)), h)


def ivit_get_changed(h: int, sv: int, idx_out=None, count_out=None, stream=None) -> None:
    _check(load().ivit_get_changed(h, sv, _ptr(idx_out), _ptr(count_out), _stream(stream)), h)


def ivit_get_cache(h: int, which: int, layer: int, dst, stream=None) -> None:
    _check(load().ivit_get_cache(h, which, layer, _ptr(dst), _stream(stream)), h)


def ivit_reset(h: int, stream_index: int = -1) -> None:
    _check(load().ivit_reset(h, stream_index), h)


def ivit_timeline(h: int, enable: bool) -> None:
    """Timeline mode on or off (the encoder's CUDA graphs are captured again)."""
    _check(load().ivit_timeline(h, int(bool(enable))), h)


TIMELINE_FAMILIES = ("gemm", "attention", "layernorm", "other")


def ivit_timeline_read(h: int, stream=None) -> dict:
    """Per-family kernel time (ms) and launches of the last call, the GEMM launches'
    algorithmic bytes and the call's kernel span (ms); synchronises the stream."""
    ms = (C.c_double * 4)()
    n = (C.c_int64 * 4)()
    b = C.c_double()
    span = C.c_double()
    _check(load().ivit_timeline_read(h, _stream(stream), ms, n, C.byref(b), C.byref(span)), h)
    return {"ms": dict(zip(TIMELINE_FAMILIES, list(ms))), "launches": dict(zip(TIMELINE_FAMILIES, list(n))),
            "gemm_bytes": b.value, "span_ms": span.value}


def ivit_device_status(h: int, stream=None) -> int:
    return _check(load().ivit_device_status(h, _stream(stream)), h)


def ivit_last_launch_count(h: int) -> int:
    return int(load().ivit_last_launch_count(h))


def ivit_destroy(h: int) -> None:
    _dims.pop(h, None)
    load().ivit_destroy(h)


def ivit_select_noalloc(e_cur, e_ref, n_views: int, n_tok: int, dim: int, select_mode: int,
                        threshold: float, topk: int, idx_out, counts_out, stream=None) -> None:
    """Selection without device allocation (scratch in a fixed device array); for callers
    that cannot allocate, e.g. while a stream is being captured into a CUDA graph."""
    if 0 < n_views * n_tok <= IVIT_NOALLOC_MAX_TOKENS and dim > 0:
        # (other sizes are rejected by the library before any device work)
        _require(e_cur, "e_cur", "float32", n_views * n_tok * dim)
        _require(e_ref, "e_ref", "float32", n_views * n_tok * dim)
        _require(idx_out, "idx_out", "int32", n_views * n_tok)
        _require(counts_out, "counts_out", "int32", n_views)
    _check(load().ivit_select_noalloc(_ptr(e_cur), _ptr(e_ref), n_views, n_tok, dim, select_mode,
                                      threshold, topk, _ptr(idx_out), _ptr(counts_out),
                                      _stream(stream)), None)


def ivit_action_combine(x0, v0, v7, alpha, beta, b, xT, stream=None) -> None:
    """Eq. 9 action combine on device tensors: x0, v0, v7, b (or None), xT fp32 [B, A];
    alpha, beta fp32 [B]."""
    if x0.dim() != 2:
        raise ValueError(f"x0: shape {tuple(x0.shape)}, expected [batch, action width]")
    B, A = int(x0.shape[0]), int(x0.shape[1])
    for t, name in ((x0, "x0"), (v0, "v0"), (v7, "v7"), (b, "b"), (xT, "xT")):
        _require(t, name, "float32", B * A)
    _require(alpha, "alpha", "float32", B)
    _require(beta, "beta", "float32", B)
    _check(load().ivit_action_combine(_ptr(x0), _ptr(v0), _ptr(v7), _ptr(alpha), _ptr(beta),
                                      _ptr(b) if b is not None else None, B, A, _ptr(xT),
                                      _stream(stream)), None)


# ------------------------------------------------------------ convenience

class IncrementalViT:
    """Owns one library handle; torch tensors in and out (device memory, torch streams)."""

    def __init__(self, shape: "synth.EncoderShape", weights_u16: np.ndarray, n_streams: int = 1,
                 n_views: int = 1, select_mode: int = synth.SEL_THRESHOLD,
                 threshold: float = 0.98, topk: int = 0, ref_mode: int = synth.REF_PREV_FRAME,
                 score_source: int = synth.SCORE_EMBED, schedule: int = synth.SCHED_INCREMENTAL,
                 mlp_tokens: int = 0):
        import torch
        self.torch = torch
        self.shape = shape
        self.sv = n_streams * n_views
        self.cfg = make_config(shape, n_streams, n_views, select_mode, threshold, topk, ref_mode,
                               score_source, schedule, mlp_tokens)
        self.h = ivit_create(self.cfg, weights_u16)
        self.device = torch.device("cuda", torch.cuda.current_device())

    @classmethod
    def for_workload(cls, wl, weights_u16):
        return cls(wl.shape, weights_u16, wl.n_streams, wl.n_views, wl.select_mode, wl.threshold,
                   wl.topk, wl.ref_mode, wl.score_source, wl.schedule, wl.mlp_tokens)

    def close(self):
        if getattr(self, "h", None):
            ivit_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def tokens_buffer(self):
        return self.torch.empty((self.sv, self.shape.n_tokens, self.shape.dim),
                                dtype=self.torch.bfloat16, device=self.device)

    def encode_full(self, frames, out=None, stream=None):
        out = self.tokens_buffer() if out is None else out
        ivit_encode_full(self.h, frames, out, stream)
        return out

    def encode_incremental(self, frames, out=None, counts=None, stream=None):
        out = self.tokens_buffer() if out is None else out
        counts = (self.torch.empty(self.sv, dtype=self.torch.int32, device=self.device)
                  if counts is None else counts)
        ivit_encode_incremental(self.h, frames, out, counts, stream)
        return out, counts

    def changed(self, sv: int, stream=None):
        idx = self.torch.empty(self.shape.n_tokens, dtype=self.torch.int32, device=self.device)
        cnt = self.torch.empty(1, dtype=self.torch.int32, device=self.device)
        ivit_get_changed(self.h, sv, idx, cnt, stream)
        return idx[: int(cnt.item())]

    def cache(self, which: str, layer: int = 0, stream=None):
        code = {"K": 0, "V": 1, "tokens": 2, "ref": 3, "A": 4}[which]
        dt = self.torch.float32 if code in (3, 4) else self.torch.bfloat16
        dst = self.torch.empty((self.sv, self.shape.n_tokens, self.shape.dim), dtype=dt,
                               device=self.device)
        ivit_get_cache(self.h, code, layer, dst, stream)
        return dst

    def reset(self, stream_index: int = -1):
        ivit_reset(self.h, stream_index)

    def device_status(self, stream=None) -> int:
        return ivit_device_status(self.h, stream)
