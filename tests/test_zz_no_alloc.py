"""ivit_select_noalloc: token selection for callers that cannot allocate device memory
(for example code that enqueues work while a stream is captured into a CUDA graph).

The entry point keeps its per-token scores in a fixed device array instead of
allocating.  Its changed-token lists must equal the ones ivit_encode_incremental
selected for the same embeddings, on two calls in a row.  This file is collected last
so that a failure here cannot hide the rest of the suite; it also runs on its own.
"""
import numpy as np
import pytest

from paper_2607_12287_gb300 import synth

pytestmark = pytest.mark.gpu

SHAPE = synth.EncoderShape(112, 112, 14, 320, 2, 5, 840, synth.GELU_TANH)


@pytest.fixture(scope="module")
def pkg():
    import paper_2607_12287_gb300 as p
    p.load()
    return p


@pytest.mark.parametrize("mode,k", [(synth.SEL_THRESHOLD, 0), (synth.SEL_TOPK, 9)])
def test_noalloc_selection_matches_encoder(pkg, mode, k):
    import torch
    S, V = 1, 3
    N, D = SHAPE.n_tokens, SHAPE.dim
    w = synth.make_weights(SHAPE, 23)
    frames = [torch.from_numpy(f).cuda()
              for f in synth.stream_random(SHAPE, S * V, 3, 24, change_p=0.2)]
    enc = pkg.IncrementalViT(SHAPE, w, S, V, select_mode=mode, topk=k)
    idx = torch.full((S * V, N), -7, dtype=torch.int32, device="cuda")
    cnt = torch.full((S * V,), -7, dtype=torch.int32, device="cuda")
    try:
        enc.encode_full(frames[0])
        ref_prev = enc.cache("ref").clone()  # embeddings of frame 0
        for t in (1, 2):  # two calls in a row
            _, counts = enc.encode_incremental(frames[t])
            ref_cur = enc.cache("ref").clone()  # previous-frame reference: frame t's embeddings
            pkg.ivit_select_noalloc(ref_cur, ref_prev, S * V, N, D, mode, 0.98, k, idx, cnt)
            torch.cuda.synchronize()
            assert cnt.cpu().tolist() == counts.cpu().tolist()
            for v in range(S * V):
                want = enc.changed(v).cpu().numpy()
                got = idx[v].cpu().numpy()
                np.testing.assert_array_equal(got[:len(want)], want)
                assert np.all(got[len(want):] == -1)
            ref_prev = ref_cur
        assert enc.device_status() == 0
    finally:
        enc.close()


@pytest.mark.parametrize("mode,k", [(synth.SEL_THRESHOLD, 0), (synth.SEL_TOPK, 11)])
def test_noalloc_selection_matches_oracle(pkg, oracle_mod, mode, k):
    """The lists against the oracle's selection (Eq. 3 cosine in fp32 with double sums,
    then the threshold or top-k of Sec. III-B) on the same embeddings, two calls in a
    row; the oracle's scores keep a margin from every decision boundary."""
    import torch
    V, N, D = 4, 196, 192
    rng = np.random.Generator(np.random.PCG64(31 + k))
    cur = rng.standard_normal((V, N, D)).astype(np.float32)
    for call in range(2):
        ref = cur.copy()
        # a fifth of the tokens change a lot, the rest by a little noise
        moved = rng.random((V, N)) < 0.2
        step = np.where(moved[..., None], 0.9, 0.01) * rng.standard_normal((V, N, D))
        cur = (ref + step).astype(np.float32)
        idx = torch.full((V, N), -7, dtype=torch.int32, device="cuda")
        cnt = torch.full((V,), -7, dtype=torch.int32, device="cuda")
        pkg.ivit_select_noalloc(torch.from_numpy(cur).cuda(), torch.from_numpy(ref).cuda(), V, N, D, mode,
                                0.98, k, idx, cnt)
        torch.cuda.synchronize()
        for v in range(V):
            sims = np.array([oracle_mod.cosine(cur[v, i], ref[v, i]) for i in range(N)], np.float32)
            if mode == synth.SEL_THRESHOLD:
                assert np.abs(sims - 0.98).min() > 1e-3
                want = oracle_mod.select_threshold(sims, 0.98)
            else:
                srt = np.sort(sims)
                assert srt[k] - srt[k - 1] > 1e-4
                want = oracle_mod.select_topk(sims, k)
            assert int(cnt[v]) == len(want), f"call {call} view {v}"
            got = idx[v].cpu().numpy()
            np.testing.assert_array_equal(got[:len(want)], want)
            assert np.all(got[len(want):] == -1)


def test_noalloc_rejects_misaligned_views(pkg):
    import torch
    V, N, D = 1, 16, 8
    buf = torch.zeros(V * N * D + 1, dtype=torch.float32, device="cuda")
    ok = buf[:-1]
    off = buf[1:]  # starts 4 bytes into the allocation: not 16-byte aligned
    ib = torch.zeros(V * N, dtype=torch.int32, device="cuda")
    cb = torch.zeros(V, dtype=torch.int32, device="cuda")
    for a, b in ((off, ok), (ok, off)):
        with pytest.raises(pkg.IvitError) as e:
            pkg.ivit_select_noalloc(a, b, V, N, D, 0, 0.98, 0, ib, cb)
        assert e.value.code == pkg.IVIT_ERR_ARG


def test_noalloc_rejects_oversize(pkg):
    import torch
    buf = torch.zeros(8, dtype=torch.float32, device="cuda")
    ib = torch.zeros(8, dtype=torch.int32, device="cuda")
    n_views = pkg.IVIT_NOALLOC_MAX_TOKENS // 1024 + 1
    with pytest.raises(pkg.IvitError) as e:
        pkg.ivit_select_noalloc(buf, buf, n_views, 1024, 4, 0, 0.98, 0, ib, ib)
    assert e.value.code == pkg.IVIT_ERR_SHAPE
    assert "IVIT_NOALLOC_MAX_TOKENS" in str(e.value)
