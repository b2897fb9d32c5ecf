"""Pins of the oracle's encoder and incremental step (CPU only).

- full encode and caches == an fp64 ``torch.nn.functional`` restatement;
- incremental step == a masked fp64 restatement (Eq. 4-5, Sec. III-B);
- all-changed incremental == full encode (bitwise, same frames);
- identical consecutive frames select nothing and leave every cache byte unchanged;
- reset / cold views, top-k count, reference-update modes, pixel ground truth.
"""
import numpy as np
import pytest
import torch

from paper_2607_12287_gb300 import synth
from tests import restate

SHAPES = [
    synth.EncoderShape(32, 48, 8, 32, 2, 2, 64, synth.GELU_TANH),
    synth.EncoderShape(28, 28, 7, 48, 3, 3, 80, synth.GELU_ERF),
    # degenerate shapes: one token per view (attention over a single key returns its
    # value), and one-pixel patches (K = 3) with single-pixel-wide heads of 6
    synth.EncoderShape(8, 8, 8, 16, 2, 1, 32, synth.GELU_TANH),
    synth.EncoderShape(4, 6, 1, 24, 2, 4, 40, synth.GELU_ERF),
]


def rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-30))


@pytest.mark.parametrize("shape", SHAPES)
def test_full_encode_vs_restatement(oracle_mod, shape):
    w = synth.make_weights(shape, 11)
    W = restate.weights64(shape, w)
    frames = next(synth.stream_random(shape, 2, 1, 12))
    orc = oracle_mod.Oracle(shape, w, 1, 2)
    tok = orc.encode_full(frames)
    for v in range(2):
        t64, K64, V64, _ = restate.full(shape, W, frames[v])
        assert rel(tok[v], t64) < 1e-5
        for l in range(shape.depth):
            assert rel(orc.cache("K", l)[v], K64[l]) < 1e-5
            assert rel(orc.cache("V", l)[v], V64[l]) < 1e-5


@pytest.mark.parametrize("shape", SHAPES)
def test_incremental_vs_masked_restatement(oracle_mod, shape):
    w = synth.make_weights(shape, 21)
    W = restate.weights64(shape, w)
    frames = list(synth.stream_random(shape, 2, 4, 22, change_p=0.3))
    orc = oracle_mod.Oracle(shape, w, 2, 1)
    orc.encode_full(frames[0])
    state = []
    updated = 0
    for v in range(2):
        t64, K64, V64, e64 = restate.full(shape, W, frames[0][v])
        state.append([t64, K64, V64, e64])
    for f in frames[1:]:
        tok, counts, idx, sims = orc.encode_incremental(f)
        for v in range(2):
            t64, K64, V64, eref = state[v]
            e = restate.embed(shape, W, f[v])
            s64 = torch.nn.functional.cosine_similarity(e, eref, dim=1).numpy()
            np.testing.assert_allclose(sims[v], s64, atol=1e-5)
            mask = s64 < 0.98
            assert np.all(np.abs(s64 - 0.98) > 1e-3), "stream too close to the threshold"
            np.testing.assert_array_equal(idx[v, :counts[v]], np.nonzero(mask)[0])
            K64, V64, t64 = restate.run_rows(shape, W, e, mask, K64, V64, t64)
            state[v] = [t64, K64, V64, e]
            assert rel(tok[v], t64) < 1e-5
            for l in range(shape.depth):
                assert rel(orc.cache("K", l)[v], K64[l]) < 1e-5
        updated += int(counts.sum())
    assert updated > 0  # the stream exercised the incremental path


def test_all_changed_incremental_equals_full_bitwise(oracle_mod):
    shape = SHAPES[0]
    w = synth.make_weights(shape, 31)
    f0, f1 = synth.stream_random(shape, 3, 2, 32)
    a = oracle_mod.Oracle(shape, w, 1, 3, threshold=2.0)  # every sim < 2: all change
    a.encode_full(f0)
    tok_a, counts, _, _ = a.encode_incremental(f1)
    assert np.all(counts == shape.n_tokens)
    b = oracle_mod.Oracle(shape, w, 1, 3)
    tok_b = b.encode_full(f1)
    assert np.array_equal(tok_a, tok_b)
    for l in range(shape.depth):
        assert np.array_equal(a.cache("K", l), b.cache("K", l))
        assert np.array_equal(a.cache("V", l), b.cache("V", l))


def test_identical_frames_change_nothing(oracle_mod):
    shape = SHAPES[1]
    w = synth.make_weights(shape, 41)
    f0, f1 = synth.stream_random(shape, 2, 2, 42)
    orc = oracle_mod.Oracle(shape, w, 1, 2)
    orc.encode_full(f0)
    orc.encode_incremental(f1)  # leave the caches in a non-trivial state
    kv = {(c, l): orc.cache(c, l) for c in ("K", "V") for l in range(shape.depth)}
    tokens, ref = orc.cache("tokens"), orc.cache("ref")
    tok, counts, idx, sims = orc.encode_incremental(f1)
    assert np.all(counts == 0) and np.all(idx == -1)
    assert np.all(sims >= 0.98)
    assert np.array_equal(tok, tokens)
    for (c, l), arr in kv.items():
        assert np.array_equal(orc.cache(c, l), arr)
    assert np.array_equal(orc.cache("ref"), ref)


def test_cold_start_and_reset(oracle_mod):
    shape = SHAPES[0]
    w = synth.make_weights(shape, 51)
    f0, f1 = synth.stream_random(shape, 4, 2, 52)
    N = shape.n_tokens
    cold = oracle_mod.Oracle(shape, w, 2, 2)
    tok_cold, counts, _, sims = cold.encode_incremental(f0)  # no reference: all tokens
    assert np.all(counts == N) and np.all(sims == -2.0)
    full = oracle_mod.Oracle(shape, w, 2, 2)
    assert np.array_equal(tok_cold, full.encode_full(f0))
    # reset stream 1 (views 2, 3): those recompute everything, stream 0 reuses
    full.reset(1)
    tok, counts, _, _ = full.encode_incremental(f0)
    np.testing.assert_array_equal(counts, [0, 0, N, N])
    assert np.array_equal(tok, tok_cold)
    with pytest.raises(ValueError):
        full.reset(2)


def test_topk_selects_exactly_k(oracle_mod):
    shape = SHAPES[0]
    w = synth.make_weights(shape, 61)
    frames = list(synth.stream_random(shape, 2, 3, 62, change_p=0.5))
    orc = oracle_mod.Oracle(shape, w, 1, 2, select_mode=synth.SEL_TOPK, topk=5)
    orc.encode_full(frames[0])
    for f in frames[1:]:
        _, counts, idx, sims = orc.encode_incremental(f)
        assert np.all(counts == 5)
        for v in range(2):
            order = np.lexsort((np.arange(shape.n_tokens), sims[v]))
            np.testing.assert_array_equal(idx[v, :5], np.sort(order[:5]))


def _drift_frames(shape, n):
    """Patch 0 creeps by 3 grey levels per frame (checkerboard sign); the rest static."""
    rng = np.random.default_rng(71)
    base = rng.integers(60, 190, (1, shape.img_h, shape.img_w, 3)).astype(np.int16)
    P = shape.patch
    sign = (np.indices((P, P, 3)).sum(0) % 2) * 2 - 1
    out = []
    for t in range(n):
        f = base.copy()
        f[0, :P, :P] += (3 * t * sign).astype(np.int16)
        out.append(np.clip(f, 0, 255).astype(np.uint8))
    return out


def test_reference_modes_on_slow_drift(oracle_mod):
    # previous-frame reference never sees a slow drift; last-refresh reference does
    shape = SHAPES[0]
    w = synth.make_weights(shape, 72)
    frames = _drift_frames(shape, 12)
    prev = oracle_mod.Oracle(shape, w, ref_mode=synth.REF_PREV_FRAME)
    last = oracle_mod.Oracle(shape, w, ref_mode=synth.REF_LAST_REFRESH)
    prev.encode_full(frames[0])
    last.encode_full(frames[0])
    hit_prev, hit_last = 0, 0
    for f in frames[1:]:
        _, cp, ip, sp = prev.encode_incremental(f)
        _, cl, il, sl = last.encode_incremental(f)
        assert set(ip[0, :cp[0]]) <= {0} and set(il[0, :cl[0]]) <= {0}
        hit_prev += cp[0]
        hit_last += cl[0]
        assert sl[0, 0] <= sp[0, 0] + 1e-6  # the stale reference is farther away
    assert hit_prev == 0 and hit_last >= 1


def test_selection_equals_repainted_patches(oracle_mod):
    shape = synth.EncoderShape(56, 56, 14, 64, 1, 2, 96)
    w = synth.make_weights(shape, 81)
    frames = list(synth.stream_repaint(shape, 2, 4, 3, 82))
    orc = oracle_mod.Oracle(shape, w, 1, 2)
    orc.encode_full(frames[0])
    for prev, cur in zip(frames, frames[1:]):
        _, counts, idx, _ = orc.encode_incremental(cur)
        truth = synth.pixel_changed_patches(prev, cur, shape.patch)
        for v in range(2):
            np.testing.assert_array_equal(idx[v, :counts[v]], np.nonzero(truth[v])[0])


def test_so400m_layer_shape_on_the_bench_stream(oracle_mod):
    # the SigLIP-So400m block (D 1152, 16 heads of 72, MLP 4304, 256 tokens of 14-px
    # patches) with two of its 27 layers, on the bench's camera stream: full encode and
    # two incremental frames against the fp64 restatement
    import dataclasses
    shape = dataclasses.replace(synth.SO400M_224, depth=2)
    w = synth.make_weights(shape, 0)
    W = restate.weights64(shape, w)
    frames = list(synth.WORKLOADS["so400m_224_1view"].frames(3))
    orc = oracle_mod.Oracle(shape, w, 1, 1)
    tok = orc.encode_full(frames[0])
    t64, K64, V64, e = restate.full(shape, W, frames[0][0])
    assert rel(tok[0], t64) < 1e-5
    for f in frames[1:]:
        tok, counts, idx, sims = orc.encode_incremental(f)
        e1 = restate.embed(shape, W, f[0])
        s64 = torch.nn.functional.cosine_similarity(e1, e, dim=1).numpy()
        np.testing.assert_allclose(sims[0], s64, atol=1e-5)
        mask = s64 < 0.98
        assert np.abs(s64 - 0.98).min() > 1e-3
        np.testing.assert_array_equal(idx[0, :counts[0]], np.nonzero(mask)[0])
        assert 0 < counts[0] < shape.n_tokens
        K64, V64, t64 = restate.run_rows(shape, W, e1, mask, K64, V64, t64)
        e = e1
        assert rel(tok[0], t64) < 1e-5
        for l in range(shape.depth):
            assert rel(orc.cache("K", l)[0], K64[l]) < 1e-5
            assert rel(orc.cache("V", l)[0], V64[l]) < 1e-5


def test_so400m_448_layer_shape_on_the_batched_stream(oracle_mod):
    # 448 px frames (1024 tokens: attention over 1024 keys) with one So400m layer, on
    # view 0 of the batched 16 x 2 stream: full encode and one incremental frame
    import dataclasses
    wl = synth.WORKLOADS["so400m_448_16x2"]
    shape = dataclasses.replace(wl.shape, depth=1)
    w = synth.make_weights(shape, 0)
    W = restate.weights64(shape, w)
    f0, f1 = (f[:1] for f in wl.frames(2))
    orc = oracle_mod.Oracle(shape, w, 1, 1)
    tok = orc.encode_full(f0)
    t64, K64, V64, e = restate.full(shape, W, f0[0])
    assert rel(tok[0], t64) < 1e-5
    tok, counts, idx, sims = orc.encode_incremental(f1)
    e1 = restate.embed(shape, W, f1[0])
    s64 = torch.nn.functional.cosine_similarity(e1, e, dim=1).numpy()
    mask = s64 < 0.98
    assert np.abs(s64 - 0.98).min() > 1e-3
    np.testing.assert_array_equal(idx[0, :counts[0]], np.nonzero(mask)[0])
    assert 0 < counts[0] < shape.n_tokens
    K64, V64, t64 = restate.run_rows(shape, W, e1, mask, K64, V64, t64)
    assert rel(tok[0], t64) < 1e-5
    assert rel(orc.cache("K", 0)[0], K64[0]) < 1e-5


def test_vit_tiny_on_the_square_stream(oracle_mod):
    # the whole ViT-Tiny encoder (12 layers, 3 heads of 64, erf GELU, 196 tokens) on the
    # moving-square stream: full encode, then incremental frames against the restatement
    wl = synth.WORKLOADS["vit_tiny_224_square"]
    shape = wl.shape
    w = synth.make_weights(shape, 0)
    W = restate.weights64(shape, w)
    frames = list(wl.frames(4))
    orc = oracle_mod.Oracle(shape, w, 1, 1)
    tok = orc.encode_full(frames[0])
    t64, K64, V64, e = restate.full(shape, W, frames[0][0])
    assert rel(tok[0], t64) < 1e-5
    for prev, f in zip(frames, frames[1:]):
        tok, counts, idx, sims = orc.encode_incremental(f)
        e1 = restate.embed(shape, W, f[0])
        mask = torch.nn.functional.cosine_similarity(e1, e, dim=1).numpy() < 0.98
        truth = synth.pixel_changed_patches(prev, f, shape.patch)[0]
        np.testing.assert_array_equal(mask, truth)
        np.testing.assert_array_equal(idx[0, :counts[0]], np.nonzero(mask)[0])
        K64, V64, t64 = restate.run_rows(shape, W, e1, mask, K64, V64, t64)
        e = e1
        assert rel(tok[0], t64) < 1e-5
        assert rel(orc.cache("V", shape.depth - 1)[0], V64[-1]) < 1e-5
