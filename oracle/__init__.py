"""ctypes wrapper of the C oracle (``ivit_oracle.c``).

TEST INFRASTRUCTURE ONLY: the oracle is a plain, slow CPU restatement of temporal
token reuse (Sec. III-B) that the CUDA library is checked against.  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg and reference arm (both
time it on the host cores) may import it.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ivit_oracle.c")
_HDR = os.path.join(_HERE, "ivit_oracle.h")
_LIB = os.path.join(_HERE, "_build", "liboracle.so")

GELU_TANH, GELU_ERF = 0, 1
SCORE_EMBED, SCORE_KEY0 = 0, 1
SCHED_INCREMENTAL, SCHED_ODD_EVEN = 0, 1
MLP_UPDATED, MLP_ALL = 0, 1
SEL_THRESHOLD, SEL_TOPK = 0, 1
REF_PREV_FRAME, REF_LAST_REFRESH = 0, 1


class OrcConfig(C.Structure):
    _fields_ = [
        ("img_h", C.c_int32), ("img_w", C.c_int32), ("patch", C.c_int32),
        ("dim", C.c_int32), ("depth", C.c_int32), ("heads", C.c_int32),
        ("mlp_dim", C.c_int32), ("n_streams", C.c_int32), ("n_views", C.c_int32),
        ("ln_eps", C.c_float), ("gelu", C.c_int32), ("select_mode", C.c_int32),
        ("threshold", C.c_float), ("topk", C.c_int32), ("ref_mode", C.c_int32),
        ("score_source", C.c_int32), ("schedule", C.c_int32), ("mlp_tokens", C.c_int32),
    ]


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C, OpenMP) into ``_build/liboracle.so``."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    stale = (not os.path.exists(_LIB)
             or os.path.getmtime(_LIB) < max(os.path.getmtime(_SRC), os.path.getmtime(_HDR)))
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-D_GNU_SOURCE", "-fPIC", "-shared",
                               "-fopenmp", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib: Optional[C.CDLL] = None


def lib() -> C.CDLL:
    global _lib
    if _lib is None:
        L = C.CDLL(build())
        P = C.c_void_p
        L.orc_create.restype = P
        L.orc_create.argtypes = [C.POINTER(OrcConfig), P]
        L.orc_destroy.argtypes = [P]
        L.orc_set_threads.argtypes = [C.c_int]
        L.orc_encode_full.argtypes = [P, P, P]
        L.orc_encode_incremental.argtypes = [P, P, P, P, P, P]
        L.orc_reset.argtypes = [P, C.c_int]
        L.orc_get_cache.argtypes = [P, C.c_int, C.c_int, P]
        L.orc_patch_embed.argtypes = [C.POINTER(OrcConfig), P, P, P, P]
        L.orc_cosine.restype = C.c_float
        L.orc_cosine.argtypes = [P, P, C.c_int]
        L.orc_select_threshold.argtypes = [P, C.c_int, C.c_float, P]
        L.orc_select_topk.argtypes = [P, C.c_int, C.c_int, P]
        L.orc_layernorm.argtypes = [P, P, P, C.c_int, C.c_float, P]
        L.orc_linear.argtypes = [P, P, P, C.c_int, C.c_int, P]
        L.orc_gelu.restype = C.c_float
        L.orc_gelu.argtypes = [C.c_float, C.c_int]
        L.orc_attention.argtypes = [P, C.c_int, P, P, C.c_int, C.c_int, C.c_int, C.c_int,
                                    P, C.c_int]
        L.orc_layer0_keys.argtypes = [P, P, P, P, P, P, C.c_int, C.c_int, C.c_float, P]
        L.orc_action_combine.argtypes = [P, P, P, P, P, P, C.c_int, C.c_int, P]
        L.orc_euler.argtypes = [P, P, C.c_int, C.c_float, C.c_int, C.c_int, P]
        _lib = L
    return _lib


def _p(a: np.ndarray) -> int:
    return a.ctypes.data


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


def set_threads(n: int) -> None:
    lib().orc_set_threads(int(n))


def make_config(shape, n_streams=1, n_views=1, select_mode=SEL_THRESHOLD, threshold=0.98,
                topk=0, ref_mode=REF_PREV_FRAME, score_source=SCORE_EMBED,
                schedule=SCHED_INCREMENTAL, mlp_tokens=MLP_UPDATED) -> OrcConfig:
    return OrcConfig(shape.img_h, shape.img_w, shape.patch, shape.dim, shape.depth,
                     shape.heads, shape.mlp_dim, n_streams, n_views, shape.ln_eps,
                     shape.gelu, select_mode, threshold, topk, ref_mode, score_source, schedule,
                     mlp_tokens)


class Oracle:
    """Stateful oracle encoder over S*V views (mirrors the library's handle)."""

    def __init__(self, shape, weights_u16: np.ndarray, n_streams=1, n_views=1,
                 select_mode=SEL_THRESHOLD, threshold=0.98, topk=0,
                 ref_mode=REF_PREV_FRAME, score_source=SCORE_EMBED, schedule=SCHED_INCREMENTAL,
                 mlp_tokens=MLP_UPDATED):
        self.shape = shape
        self.cfg = make_config(shape, n_streams, n_views, select_mode, threshold, topk,
                               ref_mode, score_source, schedule, mlp_tokens)
        self.sv = n_streams * n_views
        self._w = np.ascontiguousarray(weights_u16, dtype=np.uint16)
        self._h = lib().orc_create(C.byref(self.cfg), _p(self._w))
        if not self._h:
            raise ValueError("oracle rejected the configuration")

    @classmethod
    def for_workload(cls, wl, weights_u16):
        return cls(wl.shape, weights_u16, wl.n_streams, wl.n_views, wl.select_mode,
                   wl.threshold, wl.topk, wl.ref_mode, wl.score_source, wl.schedule,
                   wl.mlp_tokens)

    def close(self):
        if self._h:
            lib().orc_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _tok(self) -> np.ndarray:
        return np.empty((self.sv, self.shape.n_tokens, self.shape.dim), np.float32)

    def encode_full(self, frames: np.ndarray) -> np.ndarray:
        fr = np.ascontiguousarray(frames, dtype=np.uint8)
        out = self._tok()
        if lib().orc_encode_full(self._h, _p(fr), _p(out)) != 0:
            raise RuntimeError("orc_encode_full failed")
        return out

    def encode_incremental(self, frames: np.ndarray):
        """Returns (tokens [SV,N,D], counts [SV], idx [SV,N] (-1 padded), sims [SV,N])."""
        fr = np.ascontiguousarray(frames, dtype=np.uint8)
        N = self.shape.n_tokens
        out = self._tok()
        counts = np.empty(self.sv, np.int32)
        idx = np.empty((self.sv, N), np.int32)
        sims = np.empty((self.sv, N), np.float32)
        if lib().orc_encode_incremental(self._h, _p(fr), _p(out), _p(counts), _p(idx),
                                        _p(sims)) != 0:
            raise RuntimeError("orc_encode_incremental failed")
        return out, counts, idx, sims

    def reset(self, stream: int = -1) -> None:
        if lib().orc_reset(self._h, int(stream)) != 0:
            raise ValueError("bad stream index")

    def cache(self, which: str, layer: int = 0) -> np.ndarray:
        code = {"K": 0, "V": 1, "tokens": 2, "ref": 3, "A": 4}[which]
        out = self._tok()
        if lib().orc_get_cache(self._h, code, int(layer), _p(out)) != 0:
            raise ValueError("bad cache request")
        return out


# ------------------------------------------------------------ building blocks

def patch_embed(shape, W_pe: np.ndarray, b_pe: np.ndarray, frame: np.ndarray) -> np.ndarray:
    cfg = make_config(shape)
    W, b = _f32(W_pe), _f32(b_pe)
    fr = np.ascontiguousarray(frame, dtype=np.uint8)
    e = np.empty((shape.n_tokens, shape.dim), np.float32)
    lib().orc_patch_embed(C.byref(cfg), _p(W), _p(b), _p(fr), _p(e))
    return e


def cosine(a, b) -> float:
    a, b = _f32(a), _f32(b)
    return float(lib().orc_cosine(_p(a), _p(b), a.size))


def select_threshold(sims, tau: float) -> np.ndarray:
    s = _f32(sims)
    idx = np.empty(s.size, np.int32)
    m = lib().orc_select_threshold(_p(s), s.size, float(tau), _p(idx))
    return idx[:m].copy()


def select_topk(sims, k: int) -> np.ndarray:
    s = _f32(sims)
    idx = np.empty(s.size, np.int32)
    m = lib().orc_select_topk(_p(s), s.size, int(k), _p(idx))
    return idx[:m].copy()


def layernorm(x, g, b, eps: float = 1e-6) -> np.ndarray:
    x, g, b = _f32(x), _f32(g), _f32(b)
    y = np.empty_like(x)
    lib().orc_layernorm(_p(x), _p(g), _p(b), x.size, float(eps), _p(y))
    return y


def linear(x, W, b) -> np.ndarray:
    x, W, b = _f32(x), _f32(W), _f32(b)
    y = np.empty(W.shape[0], np.float32)
    lib().orc_linear(_p(x), _p(W), _p(b), W.shape[1], W.shape[0], _p(y))
    return y


def gelu(x: float, mode: int) -> float:
    return float(lib().orc_gelu(float(x), int(mode)))


def layer0_keys(e, pos, ln_g, ln_b, W_K, b_K, eps: float = 1e-6) -> np.ndarray:
    e, pos, g, b, W, bk = (_f32(a) for a in (e, pos, ln_g, ln_b, W_K, b_K))
    n, D = e.shape
    k = np.empty((n, D), np.float32)
    lib().orc_layer0_keys(_p(e), _p(pos), _p(g), _p(b), _p(W), _p(bk), n, D, float(eps), _p(k))
    return k


def attention(q, k, v) -> np.ndarray:
    """One head: q [m, dh], k/v [n, dh] -> o [m, dh]."""
    q, k, v = _f32(q), _f32(k), _f32(v)
    m, dh = q.shape
    n = k.shape[0]
    o = np.empty((m, dh), np.float32)
    lib().orc_attention(_p(q), dh, _p(k), _p(v), dh, m, n, dh, _p(o), dh)
    return o


def action_combine(x0, v0, v7, alpha, beta, b=None) -> np.ndarray:
    """Eq. 9: x_T = x_0 + alpha v_0 + beta v_7 + b; x0, v0, v7, b [B, A], alpha, beta [B]."""
    x0, v0, v7, al, be = (_f32(a) for a in (x0, v0, v7, alpha, beta))
    bb = _f32(b) if b is not None else None
    B, A = x0.shape
    out = np.empty((B, A), np.float32)
    lib().orc_action_combine(_p(x0), _p(v0), _p(v7), _p(al), _p(be), _p(bb) if bb is not None else None,
                             B, A, _p(out))
    return out


def euler(x0, v, dt: float) -> np.ndarray:
    """x_T = x_0 + sum_t dt v_t; x0 [B, A], v [T, B, A]."""
    x0, v = _f32(x0), _f32(v)
    B, A = x0.shape
    out = np.empty((B, A), np.float32)
    lib().orc_euler(_p(x0), _p(v), v.shape[0], float(dt), B, A, _p(out))
    return out
