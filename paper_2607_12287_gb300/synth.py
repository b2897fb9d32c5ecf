"""Seeded synthetic inputs: encoder weights and camera streams.

Both the CUDA path (its tests and the bench) and the oracle's tests draw their inputs
from here.  The module holds none of the method's arithmetic -- no patch embedding,
no similarity score, no token selection, no encoder math -- only random draws, the
round-to-nearest-even conversion of the drawn weights to bf16, and pixel painting.

Weight buffer layout (bf16 elements, tensors back to back in this order, each stored
row-major; the same layout is documented in ``include/ivit.h``)::

    W_pe [D, P*P*3]   patch-embedding matrix; column k = (ky*P + kx)*3 + c
    b_pe [D]
    pos  [N, D]       learned absolute position embedding (N = (H/P)*(W/P))
    for each of the L layers:
        ln1_g [D], ln1_b [D]
        W_qkv [3D, D]  rows 0..D-1 = query, D..2D-1 = key, 2D..3D-1 = value;
                       head h owns rows h*dh..(h+1)*dh-1 of each block
        b_qkv [3D]
        W_o [D, D], b_o [D]
        ln2_g [D], ln2_b [D]
        W_1 [F, D], b_1 [F]
        W_2 [D, F], b_2 [D]
    lnf_g [D], lnf_b [D]

Frames are uint8 ``[S*V, H, W, 3]`` (HWC, row-major), view index ``s*V + v``.

The scene recipes stand in for the paper's robot camera feeds (224x224 RGB frames
from LIBERO/RoboTwin and up to three cameras, Sec. IV and Appendix A); those feeds
and the trained SigLIP/ViT weights are not available, so every input is drawn from a
seeded PCG64 generator.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Iterator, List, Optional, Sequence, Tuple

import numpy as np

GELU_TANH = 0
GELU_ERF = 1
SCORE_EMBED = 0
SCORE_KEY0 = 1
SCHED_INCREMENTAL = 0
SCHED_ODD_EVEN = 1
SEL_THRESHOLD = 0
SEL_TOPK = 1
REF_PREV_FRAME = 0
REF_LAST_REFRESH = 1


@dataclass(frozen=True)
class EncoderShape:
    """Shape of a pre-LN ViT encoder without CLS token (Sec. III-A: image -> tokens)."""

    img_h: int
    img_w: int
    patch: int
    dim: int
    depth: int
    heads: int
    mlp_dim: int
    gelu: int = GELU_TANH
    ln_eps: float = 1e-6

    @property
    def grid_h(self) -> int:
        return self.img_h // self.patch

    @property
    def grid_w(self) -> int:
        return self.img_w // self.patch

    @property
    def n_tokens(self) -> int:
        return self.grid_h * self.grid_w

    @property
    def patch_k(self) -> int:
        return self.patch * self.patch * 3

    @property
    def head_dim(self) -> int:
        return self.dim // self.heads


VIT_TINY_224 = EncoderShape(224, 224, 16, 192, 12, 3, 768, GELU_ERF)
SO400M_224 = EncoderShape(224, 224, 14, 1152, 27, 16, 4304, GELU_TANH)
SO400M_448 = EncoderShape(448, 448, 14, 1152, 27, 16, 4304, GELU_TANH)


def weight_layout(shape: EncoderShape) -> List[Tuple[str, Tuple[int, ...]]]:
    """Ordered (name, shape) list of the flat weight buffer (see module docstring)."""
    D, F, N, K = shape.dim, shape.mlp_dim, shape.n_tokens, shape.patch_k
    out: List[Tuple[str, Tuple[int, ...]]] = [
        ("W_pe", (D, K)), ("b_pe", (D,)), ("pos", (N, D))]
    for l in range(shape.depth):
        out += [
            (f"l{l}.ln1_g", (D,)), (f"l{l}.ln1_b", (D,)),
            (f"l{l}.W_qkv", (3 * D, D)), (f"l{l}.b_qkv", (3 * D,)),
            (f"l{l}.W_o", (D, D)), (f"l{l}.b_o", (D,)),
            (f"l{l}.ln2_g", (D,)), (f"l{l}.ln2_b", (D,)),
            (f"l{l}.W_1", (F, D)), (f"l{l}.b_1", (F,)),
            (f"l{l}.W_2", (D, F)), (f"l{l}.b_2", (D,)),
        ]
    out += [("lnf_g", (D,)), ("lnf_b", (D,))]
    return out


def weight_count(shape: EncoderShape) -> int:
    return int(sum(int(np.prod(s)) for _, s in weight_layout(shape)))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (round to nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to float32 (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _trunc_normal(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    """Normal(0, std) truncated at +-2 std by redrawing the tails."""
    x = rng.standard_normal(shape)
    bad = np.abs(x) > 2.0
    while bad.any():
        x[bad] = rng.standard_normal(int(bad.sum()))
        bad = np.abs(x) > 2.0
    return (x * std).astype(np.float32)


def make_weights(shape: EncoderShape, seed: int = 0) -> np.ndarray:
    """Seeded random-init weights as a flat uint16 (bf16 bits) buffer.

    Scales: W_pe std 1/(64*sqrt(P*P*3)) so a patch of uniform pixels embeds to
    roughly unit-scale values; W_q and W_k std sqrt(2/D) so attention logits have a
    standard deviation near 2 (attention that is neither uniform nor one-hot);
    W_v, W_o, W_1, W_2 std 0.02; biases and LN shifts N(0, 0.02); LN gains 1+N(0, 0.1);
    position embedding N(0, 0.1).  Every draw is truncated at 2 std and rounded to bf16.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    D = shape.dim
    parts = []
    for name, shp in weight_layout(shape):
        base = name.split(".")[-1]
        if base == "W_pe":
            w = _trunc_normal(rng, shp, 1.0 / (64.0 * np.sqrt(shape.patch_k)))
        elif base == "pos":
            w = _trunc_normal(rng, shp, 0.1)
        elif base == "W_qkv":
            w = np.concatenate([
                _trunc_normal(rng, (D, D), float(np.sqrt(2.0 / D))),
                _trunc_normal(rng, (D, D), float(np.sqrt(2.0 / D))),
                _trunc_normal(rng, (D, D), 0.02)], axis=0)
        elif base in ("W_o", "W_1", "W_2"):
            w = _trunc_normal(rng, shp, 0.02)
        elif base.endswith("_g"):
            w = 1.0 + _trunc_normal(rng, shp, 0.1)
        else:  # biases and LN shifts
            w = _trunc_normal(rng, shp, 0.02)
        parts.append(f32_to_bf16_bits(w.reshape(-1)))
    out = np.concatenate(parts)
    assert out.size == weight_count(shape)
    return out


def split_weights(shape: EncoderShape, flat: np.ndarray) -> dict:
    """Views of the flat buffer by tensor name (same dtype as ``flat``)."""
    out, off = {}, 0
    for name, shp in weight_layout(shape):
        n = int(np.prod(shp))
        out[name] = flat[off:off + n].reshape(shp)
        off += n
    return out


# --------------------------------------------------------------------------- scenes

def _smooth_texture(rng: np.random.Generator, h: int, w: int, cell: int = 16,
                    amp: float = 60.0, grain: float = 40.0) -> np.ndarray:
    """Static background: bilinear value noise plus uniform grain, uint8 [h, w, 3]."""
    gh, gw = h // cell + 2, w // cell + 2
    coarse = rng.uniform(-amp, amp, size=(gh, gw, 3))
    ys = np.arange(h) / cell
    xs = np.arange(w) / cell
    y0 = np.floor(ys).astype(int)
    x0 = np.floor(xs).astype(int)
    fy = (ys - y0)[:, None, None]
    fx = (xs - x0)[None, :, None]
    c00 = coarse[y0][:, x0]
    c01 = coarse[y0][:, x0 + 1]
    c10 = coarse[y0 + 1][:, x0]
    c11 = coarse[y0 + 1][:, x0 + 1]
    smooth = (c00 * (1 - fy) * (1 - fx) + c01 * (1 - fy) * fx
              + c10 * fy * (1 - fx) + c11 * fy * fx)
    img = 128.0 + smooth + rng.uniform(-grain, grain, size=(h, w, 3))
    # (fancy indexing above leaves the axes in another memory order: frames are row-major)
    return np.ascontiguousarray(np.clip(np.rint(img), 0, 255).astype(np.uint8))


def _pm1_noise(rng: np.random.Generator, img: np.ndarray) -> np.ndarray:
    """Add fresh noise in {-1, 0, +1} to every pixel, clipped to [0, 255]."""
    noise = rng.integers(0, 3, size=img.shape, dtype=np.uint8)
    out = img.astype(np.int16)
    out += noise
    out -= 1
    np.clip(out, 0, 255, out=out)
    return out.astype(np.uint8)


@dataclass
class _Rect:
    y: int
    x: int
    vy: int
    vx: int
    tex: np.ndarray  # uint8 [h, w, 3], moves with the rectangle


def _new_rect(rng, h_img, w_img, sizes, speeds, snap) -> _Rect:
    hh = int(rng.choice(sizes))
    ww = int(rng.choice(sizes))
    y = int(rng.integers(0, (h_img - hh) // snap + 1)) * snap
    x = int(rng.integers(0, (w_img - ww) // snap + 1)) * snap
    vy = int(rng.choice(speeds)) * int(rng.choice([-1, 1]))
    vx = int(rng.choice(speeds)) * int(rng.choice([-1, 1]))
    if rng.random() < 0.3:
        vy = 0  # some objects slide horizontally only
    tex = rng.integers(0, 256, size=(hh, ww, 3), dtype=np.uint8)
    return _Rect(y, x, vy, vx, tex)


def _step_rect(r: _Rect, h_img: int, w_img: int) -> None:
    hh, ww = r.tex.shape[:2]
    ny, nx = r.y + r.vy, r.x + r.vx
    if ny < 0 or ny + hh > h_img:
        r.vy = -r.vy
        ny = r.y + r.vy
    if nx < 0 or nx + ww > w_img:
        r.vx = -r.vx
        nx = r.x + r.vx
    r.y, r.x = ny, nx


def _paint(img: np.ndarray, r: _Rect) -> None:
    hh, ww = r.tex.shape[:2]
    img[r.y:r.y + hh, r.x:r.x + ww] = r.tex


@dataclass
class ViewScene:
    """Per-view recipe for the moving-rectangle scenes."""

    n_objects: Tuple[int, int]        # inclusive range of the object count
    sizes: Sequence[int]              # rectangle edge lengths in pixels
    speeds: Sequence[int]             # |velocity| per axis in pixels/frame
    count_walk_p: float = 0.0         # per-step probability of a +-1 object-count change


def stream_rects(shape: EncoderShape, views: Sequence[ViewScene], n_frames: int,
                 seed: int, noise: bool = True) -> Iterator[np.ndarray]:
    """Static textured background per view plus textured rectangles that move.

    Positions and velocities are multiples of half a patch, so every patch a
    rectangle touches has at least a quarter of its pixels replaced; with the
    uniform-noise textures this makes moving content clearly distinct from the
    +-1 pixel noise applied everywhere else.  Yields uint8 [len(views), H, W, 3].
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    H, W, snap = shape.img_h, shape.img_w, shape.patch // 2
    bgs = [_smooth_texture(rng, H, W) for _ in views]
    objs: List[List[_Rect]] = []
    for vs in views:
        k = int(rng.integers(vs.n_objects[0], vs.n_objects[1] + 1))
        objs.append([_new_rect(rng, H, W, vs.sizes, vs.speeds, snap) for _ in range(k)])
    for t in range(n_frames):
        frame = np.empty((len(views), H, W, 3), dtype=np.uint8)
        for vi, vs in enumerate(views):
            if t > 0:
                for r in objs[vi]:
                    _step_rect(r, H, W)
                if vs.count_walk_p > 0 and rng.random() < vs.count_walk_p:
                    if rng.random() < 0.5 and len(objs[vi]) > vs.n_objects[0]:
                        objs[vi].pop()
                    elif len(objs[vi]) < vs.n_objects[1]:
                        objs[vi].append(_new_rect(rng, H, W, vs.sizes, vs.speeds, snap))
            img = _pm1_noise(rng, bgs[vi]) if noise else bgs[vi].copy()
            for r in objs[vi]:
                _paint(img, r)
            frame[vi] = img
        yield frame


def stream_moving_square(shape: EncoderShape, n_frames: int, seed: int,
                         size: int = 48, y0: int = 88, x0: int = 8,
                         step: int = 16) -> Iterator[np.ndarray]:
    """Uniform-noise background fixed; a solid square moves ``step`` px/frame in x and
    turns back at the image's right edge (and again at ``x0``), so every frame of an
    arbitrarily long stream has motion.

    The square's colour has every channel in [0, 63] or [192, 255] (far from the
    background mean).  Every pixel outside the square gets fresh +-1 noise per frame.
    Yields uint8 [1, H, W, 3].
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    H, W = shape.img_h, shape.img_w
    bg = rng.integers(0, 256, size=(H, W, 3), dtype=np.uint8)
    lo = rng.integers(0, 64, size=3)
    colour = np.where(rng.random(3) < 0.5, lo, 192 + lo).astype(np.uint8)
    n_pos = max(1, (W - size - x0) // step + 1)  # left edges with the whole square inside
    period = max(1, 2 * (n_pos - 1))
    for t in range(n_frames):
        img = _pm1_noise(rng, bg)
        k = t % period
        x = x0 + step * (k if k < n_pos else period - k)
        img[y0:y0 + size, max(x, 0):min(x + size, W)] = colour
        yield img[None]


def stream_repaint(shape: EncoderShape, n_views: int, n_frames: int, k: int,
                   seed: int) -> Iterator[np.ndarray]:
    """Frame t = frame t-1 with ``k`` distinct patch-aligned blocks per view repainted
    with fresh uniform noise (no other pixel changes).  Yields uint8 [V, H, W, 3]."""
    rng = np.random.Generator(np.random.PCG64(seed))
    H, W, P = shape.img_h, shape.img_w, shape.patch
    gw, n = shape.grid_w, shape.n_tokens
    cur = np.stack([_smooth_texture(rng, H, W) for _ in range(n_views)])
    for t in range(n_frames):
        if t > 0:
            cur = cur.copy()
            for v in range(n_views):
                for tok in rng.choice(n, size=k, replace=False):
                    py, px = divmod(int(tok), gw)
                    cur[v, py * P:(py + 1) * P, px * P:(px + 1) * P] = rng.integers(
                        0, 256, size=(P, P, 3), dtype=np.uint8)
        yield cur


def stream_random(shape: EncoderShape, n_views: int, n_frames: int, seed: int,
                  change_p: float = 0.3) -> Iterator[np.ndarray]:
    """Small-case stream: uniform frame 0, then each patch is independently repainted
    with probability ``change_p`` per frame (other pixels untouched)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    H, W, P = shape.img_h, shape.img_w, shape.patch
    gw, n = shape.grid_w, shape.n_tokens
    cur = rng.integers(0, 256, size=(n_views, H, W, 3), dtype=np.uint8)
    for t in range(n_frames):
        if t > 0:
            cur = cur.copy()
            for v in range(n_views):
                for tok in np.nonzero(rng.random(n) < change_p)[0]:
                    py, px = divmod(int(tok), gw)
                    cur[v, py * P:(py + 1) * P, px * P:(px + 1) * P] = rng.integers(
                        0, 256, size=(P, P, 3), dtype=np.uint8)
        yield cur


def pixel_changed_patches(prev: np.ndarray, cur: np.ndarray, patch: int,
                          tol: int = 2) -> np.ndarray:
    """Ground truth of the scene recipe: bool [V, N], patches with a pixel that moved
    by more than ``tol`` grey levels between the two frames."""
    d = np.abs(cur.astype(np.int16) - prev.astype(np.int16)).max(axis=-1) > tol
    V, H, W = d.shape
    d = d.reshape(V, H // patch, patch, W // patch, patch).any(axis=(2, 4))
    return d.reshape(V, -1)


# ------------------------------------------------------------------------ workloads

@dataclass
class Workload:
    """A named stream workload: encoder shape, view layout, selection rule, scene."""

    name: str
    shape: EncoderShape
    n_streams: int
    n_views: int
    n_frames: int
    select_mode: int = SEL_THRESHOLD
    threshold: float = 0.98
    topk: int = 0
    ref_mode: int = REF_PREV_FRAME
    score_source: int = SCORE_EMBED
    schedule: int = SCHED_INCREMENTAL
    mlp_tokens: int = 0  # 0: blocks on the updated tokens only; 1: MLP on every token
    scene: str = "rects"
    views: Tuple[ViewScene, ...] = field(default_factory=tuple)
    repaint_k: int = 0
    seed: int = 1

    @property
    def sv(self) -> int:
        return self.n_streams * self.n_views

    def frames(self, n_frames: Optional[int] = None) -> Iterator[np.ndarray]:
        n = self.n_frames if n_frames is None else n_frames
        if self.scene == "square":
            return stream_moving_square(self.shape, n, self.seed)
        if self.scene == "repaint":
            return stream_repaint(self.shape, self.sv, n, self.repaint_k, self.seed)
        if self.scene == "random":
            return stream_random(self.shape, self.sv, n, self.seed)
        return stream_rects(self.shape, list(self.views), n, self.seed)


# About 10% of the 256 patches change per frame with three 21-35 px objects.
_VIEW_10 = ViewScene((3, 3), (21, 28, 35), (7, 14))
_VIEW_05 = ViewScene((2, 2), (21, 28), (7,))
_VIEW_15 = ViewScene((3, 4), (28, 35, 42), (7, 14))
_VIEW_30 = ViewScene((5, 5), (35, 42, 49), (7, 14))
# 448 px views (1024 patches): one to five 49-91 px objects, count random walk.
_VIEW_448 = ViewScene((1, 5), (49, 63, 77, 91), (7, 14), count_walk_p=0.1)

SWEEP_FRACTIONS = (0.0, 0.01, 0.05, 0.10, 0.25, 0.50, 1.0)


def sweep_workload(fraction: float, n_frames: int = 128) -> Workload:
    k = int(round(fraction * SO400M_224.n_tokens))
    return Workload(f"so400m_224_sweep_{int(round(fraction * 100))}pct", SO400M_224,
                    1, 1, n_frames, select_mode=SEL_TOPK, topk=k, scene="repaint",
                    repaint_k=k, seed=4)


WORKLOADS = {
    "vit_tiny_224_square": Workload(
        "vit_tiny_224_square", VIT_TINY_224, 1, 1, 8, scene="square", seed=1),
    "so400m_224_1view": Workload(
        "so400m_224_1view", SO400M_224, 1, 1, 64, views=(_VIEW_10,), seed=2),
    "so400m_224_3view": Workload(
        "so400m_224_3view", SO400M_224, 1, 3, 64,
        views=(_VIEW_05, _VIEW_15, _VIEW_30), seed=3),
    "so400m_448_16x2": Workload(
        "so400m_448_16x2", SO400M_448, 16, 2, 256, views=(_VIEW_448,) * 32, seed=5),
}
