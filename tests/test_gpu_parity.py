"""GPU parity: the CUDA library through its C ABI against the oracle (small shapes that
span several tiles and ragged tails, plus the edge cases of the method)."""
import numpy as np
import pytest

from paper_2607_12287_gb300 import synth
from tests.gpu_util import assert_tokens_close, run_side_by_side

pytestmark = pytest.mark.gpu

# D=320 (2.5 feature tiles), F=840 (6.6 tiles, ragged K for the MLP down projection),
# P=14 (K=588, ragged), dh=64; 3 views of 64 tokens.
SHAPE_A = synth.EncoderShape(112, 112, 14, 320, 2, 5, 840, synth.GELU_TANH)
# N=196 tokens per view, D=192 (1.5 tiles), erf GELU; 2 streams x 1 view = 392 rows.
SHAPE_B = synth.EncoderShape(224, 224, 16, 192, 2, 3, 768, synth.GELU_ERF)
# dh=72 (SigLIP head width), F=1000.
SHAPE_C = synth.EncoderShape(56, 56, 14, 576, 1, 8, 1000, synth.GELU_TANH)


@pytest.fixture(scope="module")
def pkg():
    import paper_2607_12287_gb300 as p
    p.load()
    return p


@pytest.mark.parametrize("shape,S,V", [(SHAPE_A, 1, 3), (SHAPE_B, 2, 1), (SHAPE_C, 1, 2)],
                         ids=["A_d320_3view", "B_n196_2stream", "C_dh72"])
def test_random_repaint_stream(pkg, oracle_mod, shape, S, V):
    w = synth.make_weights(shape, 5)
    frames = list(synth.stream_random(shape, S * V, 4, 6, change_p=0.2))
    run_side_by_side(pkg, oracle_mod, shape, w, frames, S, V, check_caches=True)


def test_identical_frames_select_nothing(pkg, oracle_mod):
    import torch
    shape = SHAPE_A
    w = synth.make_weights(shape, 7)
    f0, f1 = synth.stream_random(shape, 2, 2, 8)
    enc = pkg.IncrementalViT(shape, w, 1, 2)
    d0, d1 = torch.from_numpy(f0).cuda(), torch.from_numpy(f1).cuda()
    enc.encode_full(d0)
    a, _ = enc.encode_incremental(d1)
    b, counts = enc.encode_incremental(d1)  # same frame again: nothing to update
    assert counts.cpu().tolist() == [0, 0]
    assert torch.equal(a, b)
    assert enc.device_status() == 0
    enc.close()


def test_single_token_and_mixed_views(pkg, oracle_mod):
    # view 0 changes one patch, view 1 nothing, view 2 every patch
    shape = SHAPE_A
    w = synth.make_weights(shape, 9)
    rng = np.random.default_rng(10)
    f0 = rng.integers(0, 256, (3, shape.img_h, shape.img_w, 3), dtype=np.uint8)
    f1 = f0.copy()
    f1[0, 14:28, 28:42] = rng.integers(0, 256, (14, 14, 3), dtype=np.uint8)
    f1[2] = rng.integers(0, 256, f1[2].shape, dtype=np.uint8)
    stats = run_side_by_side(pkg, oracle_mod, shape, w, [f0, f1, f1], 1, 3)
    assert stats[1][2].tolist() == [1, 0, shape.n_tokens]
    assert stats[2][2].tolist() == [0, 0, 0]


def test_all_changed_incremental_matches_full(pkg, oracle_mod):
    import torch
    shape = SHAPE_B
    w = synth.make_weights(shape, 11)
    f0, f1 = synth.stream_random(shape, 2, 2, 12)
    a = pkg.IncrementalViT(shape, w, 2, 1, threshold=2.0)  # every sim < 2
    a.encode_full(torch.from_numpy(f0).cuda())
    inc, counts = a.encode_incremental(torch.from_numpy(f1).cuda())
    assert counts.cpu().tolist() == [shape.n_tokens] * 2
    b = pkg.IncrementalViT(shape, w, 2, 1)
    full = b.encode_full(torch.from_numpy(f1).cuda())
    assert_tokens_close(inc.float().cpu().numpy(), full.float().cpu().numpy(), "inc vs full")
    a.close()
    b.close()


def test_cold_start_and_reset(pkg, oracle_mod):
    shape = SHAPE_A
    w = synth.make_weights(shape, 13)
    frames = list(synth.stream_random(shape, 4, 3, 14, change_p=0.1))
    # cold start: the first incremental call encodes everything
    stats = run_side_by_side(pkg, oracle_mod, shape, w, frames, 2, 2, first_full=False)
    assert stats[0][2].tolist() == [shape.n_tokens] * 4


def test_reset_one_stream(pkg, oracle_mod):
    import torch
    shape = SHAPE_A
    w = synth.make_weights(shape, 15)
    f0, f1 = synth.stream_random(shape, 4, 2, 16, change_p=0.1)
    enc = pkg.IncrementalViT(shape, w, 2, 2)
    orc = oracle_mod.Oracle(shape, w, 2, 2)
    enc.encode_full(torch.from_numpy(f0).cuda())
    orc.encode_full(f0)
    enc.reset(1)
    orc.reset(1)
    out, counts = enc.encode_incremental(torch.from_numpy(f1).cuda())
    ref, rc, _, _ = orc.encode_incremental(f1)
    assert counts.cpu().tolist() == rc.tolist()
    assert rc[2] == rc[3] == shape.n_tokens
    assert_tokens_close(out.float().cpu().numpy(), ref, "after reset")
    with pytest.raises(pkg.IvitError):
        enc.reset(2)
    enc.close()


@pytest.mark.parametrize("k", [0, 1, 7, 64])
def test_topk_selection(pkg, oracle_mod, k):
    # k patches repainted per frame (7 when k selects none or all): the k lowest scores
    # are separated from the others by a margin, so the selection is well-posed
    shape = SHAPE_A
    w = synth.make_weights(shape, 17)
    frames = list(synth.stream_repaint(shape, 2, 3, k if 0 < k < shape.n_tokens else 7, 18))
    stats = run_side_by_side(pkg, oracle_mod, shape, w, frames, 1, 2,
                             select_mode=synth.SEL_TOPK, topk=k)
    for s in stats[1:]:
        assert s[2].tolist() == [min(k, shape.n_tokens)] * 2


def test_last_refresh_reference(pkg, oracle_mod):
    shape = SHAPE_C
    w = synth.make_weights(shape, 19)
    frames = list(synth.stream_random(shape, 2, 4, 20, change_p=0.3))
    run_side_by_side(pkg, oracle_mod, shape, w, frames, 1, 2,
                     ref_mode=synth.REF_LAST_REFRESH, check_caches=True)


@pytest.fixture
def forced_path(request, monkeypatch):
    monkeypatch.setenv("IVIT_PATH", request.param)
    return request.param


@pytest.mark.parametrize("forced_path", ["kernels", "persistent", "stream"], indirect=True)
@pytest.mark.parametrize("shape,S,V", [(SHAPE_A, 1, 3), (SHAPE_C, 1, 2)], ids=["A", "C"])
def test_both_execution_paths(pkg, oracle_mod, forced_path, shape, S, V):
    # the per-operation kernel chain, the persistent all-layers kernel and the
    # weight-streaming kernel give the same lists and tokens within tolerance (full
    # encode, cold start and steady state)
    w = synth.make_weights(shape, 25)
    frames = list(synth.stream_random(shape, S * V, 4, 26, change_p=0.15))
    run_side_by_side(pkg, oracle_mod, shape, w, frames, S, V, check_caches=True)
    run_side_by_side(pkg, oracle_mod, shape, w, frames[:2], S, V, first_full=False)


@pytest.mark.parametrize("forced_path", ["kernels", "persistent", "stream"], indirect=True)
@pytest.mark.parametrize("mode,k", [(synth.SEL_THRESHOLD, 0), (synth.SEL_TOPK, 11)])
def test_first_layer_key_scores(pkg, oracle_mod, forced_path, mode, k):
    # Eq. 3 as printed: cosine of the first layer's keys of every token.  Top-k repaints
    # exactly k patches per view so the k lowest scores are well separated from the rest.
    shape = SHAPE_A
    w = synth.make_weights(shape, 27)
    if mode == synth.SEL_TOPK:
        frames = list(synth.stream_repaint(shape, 3, 4, k, 28))
    else:
        frames = list(synth.stream_random(shape, 3, 4, 28, change_p=0.2))
    run_side_by_side(pkg, oracle_mod, shape, w, frames, 1, 3, select_mode=mode, topk=k,
                     score_source=synth.SCORE_KEY0, check_caches=True)


def test_first_layer_key_scores_last_refresh(pkg, oracle_mod):
    shape = SHAPE_C
    w = synth.make_weights(shape, 29)
    frames = list(synth.stream_random(shape, 2, 4, 30, change_p=0.3))
    run_side_by_side(pkg, oracle_mod, shape, w, frames, 1, 2, score_source=synth.SCORE_KEY0,
                     ref_mode=synth.REF_LAST_REFRESH, check_caches=True)


def test_odd_even_schedule(pkg, oracle_mod):
    # every call through ivit_encode_incremental: odd calls encode in full (count N)
    shape = SHAPE_A
    w = synth.make_weights(shape, 31)
    frames = list(synth.stream_random(shape, 2, 5, 32, change_p=0.2))
    stats = run_side_by_side(pkg, oracle_mod, shape, w, frames, 1, 2, first_full=False,
                             score_source=synth.SCORE_KEY0, schedule=synth.SCHED_ODD_EVEN)
    N = shape.n_tokens
    assert [s[2].tolist() for s in stats[0::2]] == [[N, N]] * 3
    assert all(s[2].max() < N for s in stats[1::2])


# ---- the MLP-on-all-tokens reading (attention for updated tokens, MLP for every token)

@pytest.mark.parametrize("shape,S,V", [(SHAPE_A, 1, 3), (SHAPE_B, 2, 1), (SHAPE_C, 1, 2)],
                         ids=["A_d320_3view", "B_n196_2stream", "C_dh72"])
def test_mlp_all_tokens(pkg, oracle_mod, shape, S, V):
    w = synth.make_weights(shape, 105)
    frames = list(synth.stream_random(shape, S * V, 4, 106, change_p=0.2))
    # +-1 noise on every pixel of the later frames: reused tokens' streams move too
    rng = np.random.Generator(np.random.PCG64(107))
    for t in range(1, len(frames)):
        noise = rng.integers(-1, 2, size=frames[t].shape)
        frames[t] = np.clip(frames[t].astype(np.int16) + noise, 0, 255).astype(np.uint8)
    run_side_by_side(pkg, oracle_mod, shape, w, frames, S, V, check_caches=True, mlp_tokens=1)


@pytest.mark.parametrize("mode,k", [(synth.SEL_TOPK, 7), (synth.SEL_THRESHOLD, 0)])
def test_mlp_all_tokens_topk_last_refresh_cold(pkg, oracle_mod, mode, k):
    shape = SHAPE_A
    w = synth.make_weights(shape, 111)
    frames = list(synth.stream_repaint(shape, 2, 4, k or 5, 112))
    run_side_by_side(pkg, oracle_mod, shape, w, frames, 1, 2, select_mode=mode, topk=k,
                     ref_mode=synth.REF_LAST_REFRESH, first_full=False, mlp_tokens=1)


def test_mlp_all_tokens_identical_frames(pkg, oracle_mod):
    import torch
    shape = SHAPE_C
    w = synth.make_weights(shape, 121)
    f0 = next(synth.stream_random(shape, 2, 1, 122))
    enc = pkg.IncrementalViT(shape, w, 1, 2, mlp_tokens=1)
    try:
        fd = torch.from_numpy(f0).cuda()
        t0 = enc.encode_full(fd).clone()
        t1, cnt = enc.encode_incremental(fd)
        assert cnt.cpu().numpy().tolist() == [0, 0]
        # every token is recomputed from the same stream and cached attention outputs,
        # with the full encode's MLP launch shapes: the same bits come out
        assert torch.equal(t0, t1)
        ref = oracle_mod.Oracle(shape, w, 1, 2, mlp_tokens=1).encode_full(f0)
        assert_tokens_close(t1.float().cpu().numpy(), ref, "identical frames")
        assert enc.device_status() == 0
    finally:
        enc.close()


def test_many_keys_online_softmax_groups(pkg, oracle_mod):
    # N = 324 keys per view and 32 views: the full encode has enough items to run one CTA
    # per item, which walks the keys in two groups (256 + 68) with the online softmax
    shape = synth.EncoderShape(288, 288, 16, 128, 2, 2, 256, synth.GELU_TANH)
    w = synth.make_weights(shape, 131)
    frames = list(synth.stream_random(shape, 32, 3, 132, change_p=0.15))
    run_side_by_side(pkg, oracle_mod, shape, w, frames, 16, 2, check_caches=True)


@pytest.mark.parametrize("ref_mode", [synth.REF_PREV_FRAME, synth.REF_LAST_REFRESH])
def test_bulk_copy_gather(pkg, oracle_mod, monkeypatch, ref_mode):
    # the indexed row gather with its rows staged through shared memory by TMA bulk
    # copies (the alternative to the direct 128-bit loads) gives the same lists, tokens
    # and reference caches
    monkeypatch.setenv("IVIT_GATHER", "tma")
    shape = SHAPE_C
    w = synth.make_weights(shape, 143)
    frames = list(synth.stream_random(shape, 2, 4, 144, change_p=0.3))
    run_side_by_side(pkg, oracle_mod, shape, w, frames, 1, 2, ref_mode=ref_mode, check_caches=True)


def test_frames_at_an_odd_address(pkg, monkeypatch):
    # without graphs the patchify kernel reads the caller's frames directly: frames that
    # start at an odd byte address take its byte-load path and must give the same tokens
    import torch
    monkeypatch.setenv("IVIT_NO_GRAPH", "1")
    shape = SHAPE_A
    w = synth.make_weights(shape, 141)
    f0, f1 = synth.stream_random(shape, 2, 2, 142, change_p=0.3)
    outs = []
    for odd in (False, True):
        enc = pkg.IncrementalViT(shape, w, 1, 2)
        try:
            got = []
            for f in (f0, f1):
                buf = torch.zeros(f.size + 1, dtype=torch.uint8, device="cuda")
                fd = buf[1:] if odd else buf[:-1]
                fd.copy_(torch.from_numpy(f).reshape(-1).cuda())
                fd = fd.view(f.shape)
                assert (fd.data_ptr() % 2 == 1) == odd
                got.append(enc.encode_full(fd) if not got else enc.encode_incremental(fd)[0])
            outs.append([g.clone() for g in got])
            assert enc.device_status() == 0
        finally:
            enc.close()
    for a, b in zip(*outs):
        assert torch.equal(a, b)


@pytest.mark.parametrize("forced_path", ["stream"], indirect=True)
@pytest.mark.parametrize("p", [0.1, 0.3])
def test_stream_kernel_row_passes(pkg, oracle_mod, forced_path, p):
    # 2 streams of 196 tokens: about 39 and 118 updated rows per call, so the
    # weight-streaming kernel runs its rows in 2 to 4 passes of 32 (weights kept in the
    # ring across passes, the MLP-down split partials of every pass summed by the last
    # split); erf GELU, a ragged MLP width (768 = 24 slices) and several attention groups
    shape = SHAPE_B
    w = synth.make_weights(shape, 151)
    frames = list(synth.stream_random(shape, 2, 4, 152, change_p=p))
    stats = run_side_by_side(pkg, oracle_mod, shape, w, frames, 2, 1, check_caches=True)
    assert max(int(st[2].sum()) for st in stats[1:]) > 32


def test_timeline_records_every_launch(pkg):
    # timeline mode: the graph is captured again with per-launch stamps; the outputs are
    # bitwise those of the plain graph, each family has its launches, and the kernels'
    # times fit inside the call's span (each starts after the previous one completed)
    import torch
    shape = SHAPE_A
    w = synth.make_weights(shape, 161)
    frames = [torch.from_numpy(f).cuda() for f in synth.stream_random(shape, 3, 4, 162, change_p=0.2)]
    outs = []
    for tl in (False, True):
        enc = pkg.IncrementalViT(shape, w, 1, 3)
        try:
            if tl:
                pkg.ivit_timeline(enc.h, True)
            enc.encode_full(frames[0])
            got = [enc.encode_incremental(f)[0].clone() for f in frames[1:]]
            outs.append(got)
            if tl:
                r = pkg.ivit_timeline_read(enc.h)
                L = shape.depth
                assert r["launches"] == {"gemm": 1 + 4 * L, "attention": L, "layernorm": 2 * L + 1, "other": 4}
                assert all(v > 0 for v in r["ms"].values())
                assert sum(r["ms"].values()) <= r["span_ms"] * 1.02
                assert r["gemm_bytes"] > 2 * shape.dim * 3 * shape.dim * L
                pkg.ivit_timeline(enc.h, False)
                with pytest.raises(pkg.IvitError):
                    pkg.ivit_timeline_read(enc.h)
            assert enc.device_status() == 0
        finally:
            enc.close()
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def test_maximum_view_count(pkg, oracle_mod):
    # 4096 views, the most a handle takes (1024 streams x 4 views of a 4-token encoder):
    # one selection CTA per view, the cold-view mask and the packed-row offsets at their
    # largest, 16384 rows through 256-row GEMM tiles and 4096 attention items
    shape = synth.EncoderShape(16, 16, 8, 64, 1, 1, 128, synth.GELU_TANH)
    w = synth.make_weights(shape, 171)
    frames = list(synth.stream_random(shape, 4096, 3, 172, change_p=0.3))
    stats = run_side_by_side(pkg, oracle_mod, shape, w, frames, 1024, 4, check_caches=True)
    assert all(0 < int(st[2].sum()) < 4096 * shape.n_tokens for st in stats[1:])
