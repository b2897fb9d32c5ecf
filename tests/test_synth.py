"""Host-side checks of the seeded stream generators: the dynamic fractions the workloads
claim hold for every frame of a stream as long as the bench asks for."""
import numpy as np

from paper_2607_12287_gb300 import synth

SQUARE_ROW = 88 + 24  # a pixel row through the moving square (y0 = 88, size 48)


def _changed(frames, patch):
    return [int(synth.pixel_changed_patches(a, b, patch).sum()) for a, b in zip(frames, frames[1:])]


def _square_span(frame):
    """(left edge, width) of the longest run of identical pixels on SQUARE_ROW: the solid
    square (the uniform-noise background has no runs of more than a few pixels)."""
    line = frame[0, SQUARE_ROW].astype(np.int16)
    same = np.all(line[1:] == line[:-1], axis=1)
    best_len, best_start, run, start = 0, 0, 0, 0
    for x, s in enumerate(same):
        if s:
            if run == 0:
                start = x
            run += 1
            if run > best_len:
                best_len, best_start = run, start
        else:
            run = 0
    return best_start, best_len + 1


def test_moving_square_moves_in_every_frame():
    wl = synth.WORKLOADS["vit_tiny_224_square"]
    frames = list(wl.frames(64))
    counts = _changed(frames, wl.shape.patch)
    n = wl.shape.n_tokens
    assert all(0.05 * n <= c <= 0.15 * n for c in counts), counts


def test_moving_square_path():
    # The first frames (those the parity tests use) move the square 16 px per frame to
    # the right from x0 = 8; it turns back before leaving the 224-px image and stays
    # whole inside it.
    wl = synth.WORKLOADS["vit_tiny_224_square"]
    spans = [_square_span(f) for f in wl.frames(48)]
    lefts = [s[0] for s in spans]
    assert lefts[:11] == [8 + 16 * t for t in range(11)]
    assert lefts[11:21] == [8 + 16 * (20 - t) for t in range(11, 21)]
    assert all(w == 48 for _, w in spans)
    assert max(lefts) + 48 <= wl.shape.img_w


def _fractions(wl, n_frames):
    frames = list(wl.frames(n_frames))
    counts = np.array([synth.pixel_changed_patches(a, b, wl.shape.patch).sum(1)
                       for a, b in zip(frames, frames[1:])])  # [steps, views]
    return counts / wl.shape.n_tokens


def test_bench_stream_is_ten_percent_dynamic():
    f = _fractions(synth.WORKLOADS["so400m_224_1view"], 64)
    assert 0.09 <= f.mean() <= 0.11
    assert f.min() > 0 and f.max() <= 0.15


def test_three_view_stream_targets_5_15_30_percent():
    f = _fractions(synth.WORKLOADS["so400m_224_3view"], 64).mean(0)
    assert 0.04 <= f[0] <= 0.08 and 0.14 <= f[1] <= 0.20 and 0.23 <= f[2] <= 0.31, f


def test_batched_448_stream_mix():
    f = _fractions(synth.WORKLOADS["so400m_448_16x2"], 12)
    assert f.shape[1] == 32
    assert 0.06 <= f.mean() <= 0.14
    assert f.min() >= 0.01 and f.max() <= 0.25
    assert f.mean(0).std() > 0.02  # views differ (per-stream random walks of object counts)
