"""Shared helpers of the GPU parity tests: run a stream through the CUDA library and the
oracle side by side and compare, frame by frame.

Bars: the updated-token index lists are bit-exact; final tokens (bf16 math against the
fp32 oracle) have, per view, max |gpu - oracle| / max |oracle| <= 2e-2 and a per-token
cosine similarity >= 0.999.
"""
from __future__ import annotations

import numpy as np

REL_TOL = 2e-2
COS_TOL = 0.999


def token_errors(gpu: np.ndarray, ref: np.ndarray):
    """Per-view normwise max relative error and minimum per-token cosine."""
    g = gpu.astype(np.float64)
    r = ref.astype(np.float64)
    rel = np.abs(g - r).reshape(g.shape[0], -1).max(1) / np.abs(r).reshape(r.shape[0], -1).max(1)
    cos = (g * r).sum(-1) / np.maximum(np.linalg.norm(g, axis=-1) * np.linalg.norm(r, axis=-1), 1e-30)
    return rel, cos.min(axis=1)


def assert_tokens_close(gpu: np.ndarray, ref: np.ndarray, what: str = ""):
    rel, cos = token_errors(gpu, ref)
    assert np.all(rel <= REL_TOL), f"{what}: max rel err per view {rel}"
    assert np.all(cos >= COS_TOL), f"{what}: min token cosine per view {cos}"
    return rel, cos


def run_side_by_side(pkg, oracle_mod, shape, weights, frames, n_streams=1, n_views=1,
                     select_mode=0, threshold=0.98, topk=0, ref_mode=0, margin=2e-3,
                     check_caches=False, first_full=True, score_source=0, schedule=0, mlp_tokens=0,
                     cache_layers="ends"):
    """Feeds ``frames`` (list of uint8 [SV,H,W,3]) to both sides; frame 0 is a full
    encode when ``first_full``.  With ``check_caches`` the per-layer caches of the first
    and last layer (``cache_layers="ends"``) or of every layer (``"all"``) are compared
    after the last frame.  Returns per-frame (rel, cos, counts)."""
    import torch

    enc = pkg.IncrementalViT(shape, weights, n_streams, n_views, select_mode, threshold, topk,
                             ref_mode, score_source, schedule, mlp_tokens)
    orc = oracle_mod.Oracle(shape, weights, n_streams, n_views, select_mode, threshold, topk,
                            ref_mode, score_source, schedule, mlp_tokens)
    sv = n_streams * n_views
    stats = []
    try:
        for t, f in enumerate(frames):
            fd = torch.from_numpy(np.ascontiguousarray(f)).cuda()
            if t == 0 and first_full:
                out = enc.encode_full(fd)
                ref = orc.encode_full(f)
                counts = np.full(sv, shape.n_tokens, np.int32)
            else:
                out, cnt = enc.encode_incremental(fd)
                ref, rc, ridx, sims = orc.encode_incremental(f)
                counts = cnt.cpu().numpy()
                warm = sims[:, 0] > -2  # cold views report -2 and have no margin to check
                if select_mode == 0 and warm.any():
                    gap = np.abs(sims[warm] - threshold).min()
                    assert gap > margin, f"frame {t}: a score is within {gap} of the threshold"
                if select_mode == 1 and 0 < topk < shape.n_tokens:
                    for v in np.nonzero(warm)[0]:  # the k-th and (k+1)-th scores must separate
                        srt = np.sort(sims[v])
                        assert srt[topk] - srt[topk - 1] > margin, (
                            f"frame {t} view {v}: top-{topk} boundary gap {srt[topk] - srt[topk - 1]}")
                np.testing.assert_array_equal(counts, rc, err_msg=f"frame {t}: counts")
                for v in range(sv):
                    np.testing.assert_array_equal(enc.changed(v).cpu().numpy(), ridx[v, :rc[v]],
                                                  err_msg=f"frame {t} view {v}: index list")
            got = out.float().cpu().numpy()
            rel, cos = assert_tokens_close(got, ref, f"frame {t}")
            stats.append((rel, cos, counts))
        if check_caches:
            layers = range(shape.depth) if cache_layers == "all" else sorted({0, shape.depth - 1})
            for l in layers:
                for which in ("K", "V", "A") if mlp_tokens else ("K", "V"):
                    g = enc.cache(which, l).float().cpu().numpy()
                    r = orc.cache(which, l)
                    assert_tokens_close(g, r, f"cache {which} layer {l}")
            g = enc.cache("ref").cpu().numpy()
            r = orc.cache("ref")
            if score_source == 0:  # patch embeddings: exact bf16 products, fp32 sums
                assert np.abs(g - r).max() <= 1e-4 * np.abs(r).max() + 1e-6, "reference embeddings"
            else:  # first-layer keys: a bf16 GEMM over the bf16 LN output
                assert_tokens_close(g, r, "reference keys")
        assert enc.device_status() == 0
    finally:
        enc.close()
        orc.close()
    return stats
