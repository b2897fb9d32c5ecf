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


def test_noalloc_rejects_oversize(pkg):
    import torch
    buf = torch.zeros(8, dtype=torch.float32, device="cuda")
    ib = torch.zeros(8, dtype=torch.int32, device="cuda")
    n_views = pkg.IVIT_NOALLOC_MAX_TOKENS // 1024 + 1
    with pytest.raises(pkg.IvitError) as e:
        pkg.ivit_select_noalloc(buf, buf, n_views, 1024, 4, 0, 0.98, 0, ib, ib)
    assert e.value.code == pkg.IVIT_ERR_SHAPE
    assert "IVIT_NOALLOC_MAX_TOKENS" in str(e.value)
