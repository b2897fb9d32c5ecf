"""Pins of the oracle's building blocks against closed forms, brute force and
independent library routines (CPU only)."""
import math

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch
import torch.nn.functional as F

from paper_2607_12287_gb300 import synth

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")

SHAPE = synth.EncoderShape(32, 48, 8, 32, 2, 2, 64)  # 4x6 grid, ragged-free tiny


def _w(shape=SHAPE, seed=0):
    return synth.split_weights(shape, synth.bf16_bits_to_f32(synth.make_weights(shape, seed)))


# ------------------------------------------------------------------ patch embed

def test_patch_embed_constant_frame_closed_form(oracle_mod):
    # a frame of one grey level c embeds every patch to (c-128) * rowsum(W_pe) + b_pe
    w = _w()
    for c in (0, 77, 128, 255):
        frame = np.full((SHAPE.img_h, SHAPE.img_w, 3), c, np.uint8)
        e = oracle_mod.patch_embed(SHAPE, w["W_pe"], w["b_pe"], frame)
        want = (c - 128) * w["W_pe"].astype(np.float64).sum(1) + w["b_pe"]
        np.testing.assert_allclose(e, np.broadcast_to(want, e.shape), rtol=1e-6, atol=1e-6)


def test_patch_embed_single_pixel_picks_one_column(oracle_mod):
    # one pixel at (y, x, ch) = 129 over a 128 frame selects column (ky*P+kx)*3+ch of
    # W_pe for token (y//P)*gw + x//P, every other token is b_pe
    w = _w()
    P, gw = SHAPE.patch, SHAPE.grid_w
    y, x, ch = 13, 42, 2
    frame = np.full((SHAPE.img_h, SHAPE.img_w, 3), 128, np.uint8)
    frame[y, x, ch] = 129
    e = oracle_mod.patch_embed(SHAPE, w["W_pe"], w["b_pe"], frame)
    tok = (y // P) * gw + x // P
    col = ((y % P) * P + (x % P)) * 3 + ch
    want = np.broadcast_to(w["b_pe"], e.shape).copy()
    want[tok] += w["W_pe"][:, col]
    np.testing.assert_allclose(e, want, rtol=1e-6, atol=1e-7)


def test_patch_embed_random_vs_numpy_brute_force(oracle_mod):
    w = _w()
    rng = np.random.default_rng(3)
    frame = rng.integers(0, 256, (SHAPE.img_h, SHAPE.img_w, 3), dtype=np.uint8)
    e = oracle_mod.patch_embed(SHAPE, w["W_pe"], w["b_pe"], frame)
    P = SHAPE.patch
    want = np.zeros_like(e, dtype=np.float64)
    for i in range(SHAPE.n_tokens):
        py, px = divmod(i, SHAPE.grid_w)
        patch = frame[py * P:(py + 1) * P, px * P:(px + 1) * P, :].astype(np.float64) - 128
        want[i] = w["W_pe"].astype(np.float64) @ patch.reshape(-1) + w["b_pe"]
    np.testing.assert_allclose(e, want, rtol=1e-5, atol=1e-6)


# --------------------------------------------------------------------- cosine

def test_cosine_closed_forms(oracle_mod):
    rng = np.random.default_rng(0)
    a = rng.standard_normal(1152).astype(np.float32)
    assert abs(oracle_mod.cosine(a, a) - 1.0) < 1e-6
    assert abs(oracle_mod.cosine(a, -a) + 1.0) < 1e-6
    assert abs(oracle_mod.cosine(a, 3 * a) - 1.0) < 1e-6
    assert abs(oracle_mod.cosine([1, 0], [1, 1]) - 1 / math.sqrt(2)) < 1e-7
    assert oracle_mod.cosine([1, 0, 0], [0, 5, 0]) == 0.0
    assert oracle_mod.cosine(np.zeros(8), np.ones(8)) == 0.0  # clamped denominator


def test_cosine_vs_scipy_distance(oracle_mod):
    import scipy.spatial.distance as dist
    rng = np.random.default_rng(1)
    for _ in range(20):
        a, b = rng.standard_normal((2, 192)).astype(np.float32)
        assert abs(oracle_mod.cosine(a, b) - (1 - dist.cosine(a, b))) < 1e-5


# ------------------------------------------------------------------ selection

def test_select_threshold_brute_force(oracle_mod):
    rng = np.random.default_rng(2)
    s = rng.uniform(0.9, 1.0, 300).astype(np.float32)
    s[7] = np.float32(0.98)  # exactly tau: not selected (strict <)
    got = oracle_mod.select_threshold(s, 0.98)
    np.testing.assert_array_equal(got, np.nonzero(s < np.float32(0.98))[0])
    assert 7 not in got
    assert oracle_mod.select_threshold(np.ones(10), 0.98).size == 0
    np.testing.assert_array_equal(oracle_mod.select_threshold(np.zeros(10), 0.98), np.arange(10))


@pytest.mark.parametrize("k", [0, 1, 5, 17, 64, 100, 150])
def test_select_topk_brute_force_with_ties(oracle_mod, k):
    rng = np.random.default_rng(k)
    s = rng.choice(np.float32([0.1, 0.5, 0.5, 0.7, 0.99]), 100).astype(np.float32)
    got = oracle_mod.select_topk(s, k)
    order = np.lexsort((np.arange(100), s))  # sim ascending, then index ascending
    want = np.sort(order[:min(k, 100)])
    np.testing.assert_array_equal(got, want)


# ------------------------------------------------------------------ layernorm

def test_layernorm_closed_forms(oracle_mod):
    g = np.array([2.0, 2.0, 2.0, 2.0], np.float32)
    b = np.array([0.5, -0.5, 0.0, 1.0], np.float32)
    # constant row: zero variance -> output is the shift
    np.testing.assert_allclose(oracle_mod.layernorm([3, 3, 3, 3], g, b, 1e-6), b, atol=1e-6)
    # [1,2,3,4]: mean 2.5, biased var 1.25
    x = np.array([1, 2, 3, 4], np.float32)
    want = 2.0 * (x - 2.5) / math.sqrt(1.25 + 1e-6) + b
    np.testing.assert_allclose(oracle_mod.layernorm(x, g, b, 1e-6), want, rtol=1e-6)


def test_layernorm_vs_torch(oracle_mod):
    rng = np.random.default_rng(4)
    x, g, b = rng.standard_normal((3, 1152)).astype(np.float32)
    want = F.layer_norm(torch.from_numpy(x).double(), (1152,), torch.from_numpy(g).double(),
                        torch.from_numpy(b).double(), 1e-6).numpy()
    np.testing.assert_allclose(oracle_mod.layernorm(x, g, b, 1e-6), want, rtol=1e-5, atol=1e-6)


def test_linear_vs_numpy(oracle_mod):
    rng = np.random.default_rng(5)
    W = rng.standard_normal((37, 53)).astype(np.float32)
    x = rng.standard_normal(53).astype(np.float32)
    b = rng.standard_normal(37).astype(np.float32)
    want = W.astype(np.float64) @ x + b
    np.testing.assert_allclose(oracle_mod.linear(x, W, b), want, rtol=1e-6, atol=1e-6)


# ----------------------------------------------------------------------- gelu

def test_gelu_identities(oracle_mod):
    for mode in (synth.GELU_TANH, synth.GELU_ERF):
        assert oracle_mod.gelu(0.0, mode) == 0.0
        for x in (0.1, 0.7, 1.3, 2.9, 5.0):
            # gelu(x) - gelu(-x) = x for both forms (Phi(x) + Phi(-x) = 1)
            assert abs(oracle_mod.gelu(x, mode) - oracle_mod.gelu(-x, mode) - x) < 1e-6
        assert abs(oracle_mod.gelu(12.0, mode) - 12.0) < 1e-6
        assert abs(oracle_mod.gelu(-12.0, mode)) < 1e-6


def test_gelu_vs_library(oracle_mod):
    xs = np.linspace(-6, 6, 241).astype(np.float32)
    erf_form = [oracle_mod.gelu(x, synth.GELU_ERF) for x in xs]
    np.testing.assert_allclose(erf_form, xs * scipy.stats.norm.cdf(xs.astype(np.float64)),
                               rtol=1e-6, atol=1e-7)
    tanh_form = [oracle_mod.gelu(x, synth.GELU_TANH) for x in xs]
    want = F.gelu(torch.from_numpy(xs).double(), approximate="tanh").numpy()
    np.testing.assert_allclose(tanh_form, want, rtol=1e-6, atol=1e-7)
    # the two forms are different functions (a swapped mode would show up here)
    assert np.max(np.abs(np.array(tanh_form) - np.array(erf_form))) > 1e-4


# ------------------------------------------------------------------ attention

def test_attention_vs_naive_softmax(oracle_mod):
    rng = np.random.default_rng(6)
    m, n, dh = 5, 37, 72
    q, k, v = (rng.standard_normal((r, dh)).astype(np.float32) * 2 for r in (m, n, n))
    o = oracle_mod.attention(q, k, v)
    logits = q.astype(np.float64) @ k.astype(np.float64).T / math.sqrt(dh)
    want = scipy.special.softmax(logits, axis=1) @ v.astype(np.float64)
    np.testing.assert_allclose(o, want, rtol=1e-5, atol=1e-6)


def test_attention_special_cases(oracle_mod):
    rng = np.random.default_rng(7)
    dh = 64
    q = rng.standard_normal((3, dh)).astype(np.float32)
    v = rng.standard_normal((9, dh)).astype(np.float32)
    # one key: output is that value row
    np.testing.assert_allclose(oracle_mod.attention(q, v[:1], v[:1]), np.repeat(v[:1], 3, 0),
                               rtol=1e-6)
    # identical keys: uniform weights, output is the mean of the values
    k = np.repeat(rng.standard_normal((1, dh)).astype(np.float32), 9, 0)
    np.testing.assert_allclose(oracle_mod.attention(q, k, v), np.repeat(v.mean(0, keepdims=True), 3, 0),
                               rtol=1e-5, atol=1e-6)
    # one key aligned with a large query dominates
    k = rng.standard_normal((9, dh)).astype(np.float32) * 0.01
    k[4] = q[0] * 10
    o = oracle_mod.attention(q[:1], k, v)
    np.testing.assert_allclose(o[0], v[4], rtol=1e-4, atol=1e-4)
