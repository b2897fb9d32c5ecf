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
    assert rel(got, want) < 2e-3
    cos = (got * want).sum(1) / np.linalg.norm(got, axis=1) / np.linalg.norm(want, axis=1)
    assert cos.min() > 1 - 1e-5
    # the keys are not the embeddings: a dropped projection would be caught here
    assert rel(got, e.numpy()) > 0.5


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
