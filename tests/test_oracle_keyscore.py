"""Pins of the oracle's paper-exact selection options (CPU only): scores from the first
layer's keys (Eq. 3 as printed) and the odd/even chunk schedule (Sec. III-B)."""
import numpy as np
import pytest
import torch

from paper_2607_12287_gb300 import synth
from tests import restate
from tests.test_oracle_encoder import rel

SHAPE = synth.EncoderShape(32, 48, 8, 64, 2, 2, 96, synth.GELU_TANH)


def test_layer0_keys_vs_restatement(oracle_mod):
    w = synth.make_weights(SHAPE, 91)
    W = restate.weights64(SHAPE, w)
    frame = next(synth.stream_random(SHAPE, 1, 1, 92))[0]
    e = restate.embed(SHAPE, W, frame)
    want = restate.layer0_keys(SHAPE, W, e).numpy()
    D = SHAPE.dim
    got = oracle_mod.layer0_keys(e.numpy(), W["pos"].numpy(), W["l0.ln1_g"].numpy(),
                                 W["l0.ln1_b"].numpy(), W["l0.W_qkv"][D:2 * D].numpy(),
                                 W["l0.b_qkv"][D:2 * D].numpy(), SHAPE.ln_eps)
    # fp32 storage with double sums against fp64: any rounding of the LN output to a
    # 16-bit type (relative error ~1e-3) would fail this bound
    assert rel(got, want) < 2e-5
    g64 = got.astype(np.float64)
    cos = (g64 * want).sum(1) / np.linalg.norm(g64, axis=1) / np.linalg.norm(want, axis=1)
    assert cos.min() > 1 - 1e-9
    # the keys are not the embeddings: a dropped projection would be caught here
    assert rel(got, e.numpy()) > 0.5
    # and not the keys of the embeddings without the position embedding
    no_pos = oracle_mod.layer0_keys(e.numpy(), np.zeros_like(W["pos"].numpy()), W["l0.ln1_g"].numpy(),
                                    W["l0.ln1_b"].numpy(), W["l0.W_qkv"][D:2 * D].numpy(),
                                    W["l0.b_qkv"][D:2 * D].numpy(), SHAPE.ln_eps)
    assert rel(no_pos, want) > 1e-2


def test_key_selection_precision_independent_on_bench_stream(oracle_mod):
    """Eq. 3 on first-layer keys decides the updated set in fp32 in the oracle and from a
    bf16 layer-norm output on the GPU.  On the generated So400m camera stream the two
    precisions select the same tokens, and every fp32 score keeps a margin of 2e-3 from
    the threshold, so the GPU's lists can be compared bit-exact with the oracle's."""
    wl = synth.WORKLOADS["so400m_224_1view"]
    shape = wl.shape
    D = shape.dim
    W = restate.weights64(shape, synth.make_weights(shape, 0))
    frames = [f[0] for f in wl.frames(8)]

    def keys(e, round16):
        xn = torch.nn.functional.layer_norm(e + W["pos"], (D,), W["l0.ln1_g"], W["l0.ln1_b"], shape.ln_eps)
        if round16:
            xn = xn.float().bfloat16().double()
        return torch.nn.functional.linear(xn, W["l0.W_qkv"][D:2 * D], W["l0.b_qkv"][D:2 * D])

    prev32 = prev16 = None
    for t, f in enumerate(frames):
        e = restate.embed(shape, W, f)
        k32 = oracle_mod.layer0_keys(e.numpy(), W["pos"].numpy(), W["l0.ln1_g"].numpy(),
                                     W["l0.ln1_b"].numpy(), W["l0.W_qkv"][D:2 * D].numpy(),
                                     W["l0.b_qkv"][D:2 * D].numpy(), shape.ln_eps)
        k16 = keys(e, True)
        if t:
            s32 = np.array([oracle_mod.cosine(a, b) for a, b in zip(k32, prev32)])
            s16 = torch.nn.functional.cosine_similarity(k16, prev16, dim=1).numpy()
            assert np.abs(s32 - wl.threshold).min() > 2e-3, f"frame {t}"
            np.testing.assert_array_equal(oracle_mod.select_threshold(s32, wl.threshold),
                                          np.nonzero(s16 < wl.threshold)[0], err_msg=f"frame {t}")
            assert 0 < (s32 < wl.threshold).sum() < shape.n_tokens
        prev32, prev16 = k32, k16


def test_key_scores_drive_selection(oracle_mod):
    w = synth.make_weights(SHAPE, 93)
    W = restate.weights64(SHAPE, w)
    frames = list(synth.stream_random(SHAPE, 2, 4, 94, change_p=0.3))
    orc = oracle_mod.Oracle(SHAPE, w, 1, 2, score_source=oracle_mod.SCORE_KEY0)
    orc.encode_full(frames[0])
    state = []
    for v in range(2):
        t64, K64, V64, e64 = restate.full(SHAPE, W, frames[0][v])
        state.append([t64, K64, V64, restate.layer0_keys(SHAPE, W, e64)])
    for f in frames[1:]:
        tok, counts, idx, sims = orc.encode_incremental(f)
        for v in range(2):
            t64, K64, V64, kref = state[v]
            e = restate.embed(SHAPE, W, f[v])
            k0 = restate.layer0_keys(SHAPE, W, e)
            s64 = torch.nn.functional.cosine_similarity(k0, kref, dim=1).numpy()
            np.testing.assert_allclose(sims[v], s64, atol=1e-4)
            assert np.all(np.abs(s64 - 0.98) > 1e-3)
            mask = s64 < 0.98
            np.testing.assert_array_equal(idx[v, :counts[v]], np.nonzero(mask)[0])
            K64, V64, t64 = restate.run_rows(SHAPE, W, e, mask, K64, V64, t64)
            state[v] = [t64, K64, V64, k0]
            assert rel(tok[v], t64) < 1e-5
        assert np.array_equal(orc.cache("ref")[0] != 0, np.ones_like(orc.cache("ref")[0], bool))


def test_key_scores_identical_frames(oracle_mod):
    w = synth.make_weights(SHAPE, 95)
    f0, f1 = synth.stream_random(SHAPE, 2, 2, 96)
    orc = oracle_mod.Oracle(SHAPE, w, 1, 2, score_source=oracle_mod.SCORE_KEY0)
    orc.encode_full(f0)
    orc.encode_incremental(f1)
    tok = orc.cache("tokens")
    out, counts, _, sims = orc.encode_incremental(f1)
    assert np.all(counts == 0) and np.all(np.abs(sims - 1) < 1e-6)
    assert np.array_equal(out, tok)


def test_odd_even_schedule(oracle_mod):
    w = synth.make_weights(SHAPE, 97)
    frames = list(synth.stream_random(SHAPE, 2, 5, 98, change_p=0.2))
    sched = oracle_mod.Oracle(SHAPE, w, 1, 2, score_source=oracle_mod.SCORE_KEY0,
                              schedule=oracle_mod.SCHED_ODD_EVEN)
    full = oracle_mod.Oracle(SHAPE, w, 1, 2)
    plain = oracle_mod.Oracle(SHAPE, w, 1, 2, score_source=oracle_mod.SCORE_KEY0)
    N = SHAPE.n_tokens
    for t, f in enumerate(frames):
        out, counts, _, _ = sched.encode_incremental(f)
        if t % 2 == 0:  # odd chunk (1st, 3rd, ...): full forward, every token
            assert np.all(counts == N)
            assert np.array_equal(out, full.encode_full(f))
            plain.encode_full(f)
        else:  # even chunk: incremental against the keys cached by the odd chunk
            ref, rc, _, _ = plain.encode_incremental(f)
            np.testing.assert_array_equal(counts, rc)
            assert np.array_equal(out, ref)
