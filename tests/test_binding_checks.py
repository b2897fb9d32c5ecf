"""The Python binding rejects tensors the kernels would misread or index out of bounds
(host memory, wrong dtype, non-contiguous, too few elements) before any library call.
CPU-only: device tensors are stood in for by objects with a tensor's attributes."""
import numpy as np
import pytest
import torch

import paper_2607_12287_gb300 as pkg
from paper_2607_12287_gb300 import synth


class FakeCuda:
    """The attributes the binding inspects, as a CUDA tensor would report them."""

    def __init__(self, shape, dtype, contiguous=True):
        self.shape = tuple(shape)
        self.dtype = dtype
        self.device = torch.device("cuda", 0)
        self._contiguous = contiguous

    def numel(self):
        return int(np.prod(self.shape))

    def is_contiguous(self):
        return self._contiguous

    def dim(self):
        return len(self.shape)


def test_require_accepts_a_matching_device_tensor():
    pkg._require(FakeCuda((2, 3), torch.float32), "x", "float32", 6)
    pkg._require(FakeCuda((2, 3), torch.float32), "x", "float32", 4)  # larger is fine
    pkg._require(None, "x", "float32", 6)  # optional output left out
    pkg._require(12345, "x", "float32", 6)  # raw pointer: the caller vouches


@pytest.mark.parametrize("bad,exc", [
    (torch.zeros(6), ValueError),  # host tensor
    (np.zeros(6, np.float32), TypeError),  # numpy (host memory)
    (FakeCuda((6,), torch.float64), TypeError),
    (FakeCuda((6,), torch.float32, contiguous=False), ValueError),
    (FakeCuda((5,), torch.float32), ValueError),
])
def test_require_rejects(bad, exc):
    with pytest.raises(exc):
        pkg._require(bad, "x", "float32", 6)


def test_encode_calls_check_against_the_handle_sizes(monkeypatch):
    shape = synth.EncoderShape(32, 48, 8, 32, 2, 2, 64, synth.GELU_TANH)
    sv, n, d = 2, shape.n_tokens, shape.dim
    handle = 0x5EED
    monkeypatch.setitem(pkg._dims, handle, (sv, shape.img_h * shape.img_w * 3, n, d))
    called = []
    monkeypatch.setattr(pkg, "load", lambda *a: called.append(a) or pytest.fail("library reached"))
    frames = FakeCuda((sv, shape.img_h, shape.img_w, 3), torch.uint8)
    out = FakeCuda((sv, n, d), torch.bfloat16)
    counts = FakeCuda((sv,), torch.int32)
    with pytest.raises(ValueError, match="frames"):
        pkg.ivit_encode_full(handle, FakeCuda((1, shape.img_h, shape.img_w, 3), torch.uint8), out)
    with pytest.raises(TypeError, match="frames"):
        pkg.ivit_encode_full(handle, FakeCuda(frames.shape, torch.float32), out)
    with pytest.raises(TypeError, match="tokens_out"):
        pkg.ivit_encode_incremental(handle, frames, FakeCuda((sv, n, d), torch.float32), counts)
    with pytest.raises(ValueError, match="changed_count"):
        pkg.ivit_encode_incremental(handle, frames, out, FakeCuda((1,), torch.int32))
    with pytest.raises(ValueError, match="frames"):
        pkg.ivit_encode_incremental(handle, FakeCuda(frames.shape, torch.uint8, False), out, counts)
    assert not called


def test_action_combine_checks_every_operand(monkeypatch):
    monkeypatch.setattr(pkg, "load", lambda *a: pytest.fail("library reached"))
    B, A = 4, 14
    ok = lambda: FakeCuda((B, A), torch.float32)
    vec = lambda: FakeCuda((B,), torch.float32)
    with pytest.raises(ValueError, match="x0"):
        pkg.ivit_action_combine(FakeCuda((B * A,), torch.float32), ok(), ok(), vec(), vec(), None, ok())
    with pytest.raises(ValueError, match="v7"):
        pkg.ivit_action_combine(ok(), ok(), FakeCuda((B, A - 1), torch.float32), vec(), vec(), None, ok())
    with pytest.raises(ValueError, match="beta"):
        pkg.ivit_action_combine(ok(), ok(), ok(), vec(), FakeCuda((B - 1,), torch.float32), None, ok())
    with pytest.raises(TypeError, match="b"):
        pkg.ivit_action_combine(ok(), ok(), ok(), vec(), vec(), FakeCuda((B, A), torch.float16), ok())
    with pytest.raises(ValueError, match="xT"):
        pkg.ivit_action_combine(ok(), ok(), ok(), vec(), vec(), None, torch.zeros(B, A))


def test_select_noalloc_checks_sizes_within_the_limit(monkeypatch):
    monkeypatch.setattr(pkg, "load", lambda *a: pytest.fail("library reached"))
    V, N, D = 3, 64, 32
    e = FakeCuda((V, N, D), torch.float32)
    idx, cnt = FakeCuda((V, N), torch.int32), FakeCuda((V,), torch.int32)
    with pytest.raises(ValueError, match="e_ref"):
        pkg.ivit_select_noalloc(e, FakeCuda((V, N, D - 1), torch.float32), V, N, D, 0, 0.98, 0, idx, cnt)
    with pytest.raises(TypeError, match="idx_out"):
        pkg.ivit_select_noalloc(e, e, V, N, D, 0, 0.98, 0, FakeCuda((V, N), torch.int64), cnt)
    with pytest.raises(ValueError, match="counts_out"):
        pkg.ivit_select_noalloc(e, e, V, N, D, 0, 0.98, 0, idx, FakeCuda((V - 1,), torch.int32))


def test_generated_frames_are_row_major():
    # the kernels read frames as dense row-major [views, H, W, 3] bytes
    for wl in list(synth.WORKLOADS.values()) + [synth.sweep_workload(0.05)]:
        for f in wl.frames(2):
            assert f.flags["C_CONTIGUOUS"] and f.dtype == np.uint8, wl.name
