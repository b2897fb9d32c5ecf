"""Pins of the oracle's MLP-on-all-tokens reading (Sec. III-B, the passage after Eq. 5:
attention for the updated tokens only, reused tokens inherit their cached attention
outputs, and every token goes through the residual addition and the MLP).  CPU only.

- the full encode is the same under both readings (bitwise): with every token
  updated the two orders of operations are the same arithmetic;
- incremental steps == a masked fp64 ``torch.nn.functional`` restatement (tokens, K, V
  and the cached attention-block outputs);
- all-changed incremental == full encode (bitwise);
- identical frames select nothing and reproduce the previous output bitwise;
- the readings differ exactly where they should: reused tokens keep their cached output
  bitwise under the default reading and are recomputed under this one.
"""
import numpy as np
import pytest
import torch

from paper_2607_12287_gb300 import synth
from tests import restate

SHAPES = [
    synth.EncoderShape(32, 48, 8, 32, 2, 2, 64, synth.GELU_TANH),
    synth.EncoderShape(28, 28, 7, 48, 3, 3, 80, synth.GELU_ERF),
]
MLP_ALL = 1


def rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-30))


@pytest.mark.parametrize("shape", SHAPES)
def test_full_encode_same_under_both_readings(oracle_mod, shape):
    w = synth.make_weights(shape, 51)
    frames = next(synth.stream_random(shape, 2, 1, 52))
    a = oracle_mod.Oracle(shape, w, 1, 2)
    b = oracle_mod.Oracle(shape, w, 1, 2, mlp_tokens=MLP_ALL)
    assert np.array_equal(a.encode_full(frames), b.encode_full(frames))
    for l in range(shape.depth):
        assert np.array_equal(a.cache("K", l), b.cache("K", l))
        assert np.array_equal(a.cache("V", l), b.cache("V", l))


@pytest.mark.parametrize("shape", SHAPES)
def test_incremental_vs_masked_restatement(oracle_mod, shape):
    w = synth.make_weights(shape, 61)
    W = restate.weights64(shape, w)
    frames = list(synth.stream_random(shape, 2, 4, 62, change_p=0.3))
    orc = oracle_mod.Oracle(shape, w, 2, 1, mlp_tokens=MLP_ALL)
    tok0 = orc.encode_full(frames[0])
    state = []
    for v in range(2):
        t64, K64, V64, A64, e64 = restate.full_mlp_all(shape, W, frames[0][v])
        assert rel(tok0[v], t64) < 1e-5
        for l in range(shape.depth):
            assert rel(orc.cache("A", l)[v], A64[l]) < 1e-5
        state.append([K64, V64, A64, e64])
    for f in frames[1:]:
        tok, counts, idx, sims = orc.encode_incremental(f)
        for v in range(2):
            K64, V64, A64, eref = state[v]
            e = restate.embed(shape, W, f[v])
            s64 = torch.nn.functional.cosine_similarity(e, eref, dim=1).numpy()
            mask = s64 < 0.98
            assert np.all(np.abs(s64 - 0.98) > 1e-3), "stream too close to the threshold"
            np.testing.assert_array_equal(idx[v, :counts[v]], np.nonzero(mask)[0])
            K64, V64, A64, t64 = restate.run_rows_mlp_all(shape, W, e, mask, K64, V64, A64)
            state[v] = [K64, V64, A64, e]
            assert rel(tok[v], t64) < 1e-5
            for l in range(shape.depth):
                assert rel(orc.cache("K", l)[v], K64[l]) < 1e-5
                assert rel(orc.cache("V", l)[v], V64[l]) < 1e-5
                assert rel(orc.cache("A", l)[v], A64[l]) < 1e-5
        assert 0 < counts.sum() < 2 * shape.n_tokens


def test_all_changed_incremental_equals_full_bitwise(oracle_mod):
    shape = SHAPES[0]
    w = synth.make_weights(shape, 71)
    f0, f1 = synth.stream_random(shape, 3, 2, 72)
    a = oracle_mod.Oracle(shape, w, 1, 3, threshold=2.0, mlp_tokens=MLP_ALL)
    a.encode_full(f0)
    tok_a, counts, _, _ = a.encode_incremental(f1)
    assert np.all(counts == shape.n_tokens)
    b = oracle_mod.Oracle(shape, w, 1, 3, mlp_tokens=MLP_ALL)
    assert np.array_equal(tok_a, b.encode_full(f1))
    for l in range(shape.depth):
        assert np.array_equal(a.cache("A", l), b.cache("A", l))


def test_identical_frames_reproduce_the_output(oracle_mod):
    shape = SHAPES[1]
    w = synth.make_weights(shape, 81)
    f0 = next(synth.stream_random(shape, 2, 1, 82))
    orc = oracle_mod.Oracle(shape, w, 1, 2, mlp_tokens=MLP_ALL)
    tok0 = orc.encode_full(f0)
    caches = [(orc.cache("K", l), orc.cache("V", l), orc.cache("A", l)) for l in range(shape.depth)]
    tok1, counts, _, _ = orc.encode_incremental(f0)
    assert np.all(counts == 0)
    assert np.array_equal(tok0, tok1)
    for l in range(shape.depth):
        for got, want in zip((orc.cache("K", l), orc.cache("V", l), orc.cache("A", l)), caches[l]):
            assert np.array_equal(got, want)


def test_readings_differ_only_on_reused_tokens(oracle_mod):
    shape = SHAPES[0]
    w = synth.make_weights(shape, 91)
    frames = list(synth.stream_random(shape, 1, 2, 92, change_p=0.3))
    # +-1 grey level everywhere: reused tokens stay far above the threshold but their
    # embeddings move
    noise = np.random.Generator(np.random.PCG64(93)).integers(-1, 2, size=frames[1].shape)
    frames[1] = np.clip(frames[1].astype(np.int16) + noise, 0, 255).astype(np.uint8)
    outs = {}
    for mode in (0, MLP_ALL):
        orc = oracle_mod.Oracle(shape, w, 1, 1, mlp_tokens=mode)
        t0 = orc.encode_full(frames[0])
        t1, counts, idx, sims = orc.encode_incremental(frames[1])
        assert np.all(np.abs(sims - 0.98) > 2e-3)
        outs[mode] = (t0, t1, idx[0, :counts[0]])
    upd = outs[0][2]
    np.testing.assert_array_equal(upd, outs[MLP_ALL][2])
    reused = np.setdiff1d(np.arange(shape.n_tokens), upd)
    assert 0 < len(upd) and 0 < len(reused)
    # default reading: reused tokens keep the cached output byte for byte
    assert np.array_equal(outs[0][1][0, reused], outs[0][0][0, reused])
    # this reading: their residual streams follow the new frame through every MLP
    assert not np.array_equal(outs[MLP_ALL][1][0, reused], outs[MLP_ALL][0][0, reused])
