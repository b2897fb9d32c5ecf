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
