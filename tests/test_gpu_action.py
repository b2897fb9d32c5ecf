"""GPU parity of the 2-step action combine (Sec. III-C, Eq. 9) through the C ABI against
the oracle: 128-bit and scalar paths, no bias, empty batch, and a large batch."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def pkg():
    import paper_2607_12287_gb300 as p
    p.load()
    return p


@pytest.mark.parametrize("B,A,with_b", [(4, 352, True), (3, 350, True), (5, 7, False), (4096, 50 * 7, True)])
def test_action_combine_matches_oracle(pkg, oracle_mod, B, A, with_b):
    import torch
    rng = np.random.Generator(np.random.PCG64(B * 1000 + A))
    x0, v0, v7, b = (rng.standard_normal((B, A)).astype(np.float32) for _ in range(4))
    al, be = (rng.standard_normal(B).astype(np.float32) for _ in range(2))
    want = oracle_mod.action_combine(x0, v0, v7, al, be, b if with_b else None)
    d = lambda a: torch.from_numpy(a).cuda()
    out = torch.full((B, A), float("nan"), dtype=torch.float32, device="cuda")
    pkg.ivit_action_combine(d(x0), d(v0), d(v7), d(al), d(be), d(b) if with_b else None, out)
    got = out.cpu().numpy()
    np.testing.assert_allclose(got, want, rtol=2e-6, atol=2e-6)


def test_action_combine_empty_and_bad_args(pkg):
    import torch
    e = torch.empty((0, 7), dtype=torch.float32, device="cuda")
    pkg.ivit_action_combine(e, e, e, torch.empty(0, device="cuda"), torch.empty(0, device="cuda"), None, e)
    lib = pkg.load()
    assert lib.ivit_action_combine(None, None, None, None, None, None, 2, 3, None, None) == pkg.IVIT_ERR_ARG
    assert lib.ivit_action_combine(None, None, None, None, None, None, -1, 3, None, None) == pkg.IVIT_ERR_ARG


def test_action_combine_offset_views_take_the_scalar_path(pkg, oracle_mod):
    # views starting 4 bytes into their storage are not 16-byte aligned: the library must
    # fall back to scalar accesses instead of faulting on 128-bit ones
    import torch
    B, A = 6, 64
    rng = np.random.Generator(np.random.PCG64(7))
    x0, v0, v7, b = (rng.standard_normal((B, A)).astype(np.float32) for _ in range(4))
    al, be = (rng.standard_normal(B).astype(np.float32) for _ in range(2))
    want = oracle_mod.action_combine(x0, v0, v7, al, be, b)

    def off(a):
        t = torch.zeros(a.size + 1, dtype=torch.float32, device="cuda")
        t[1:] = torch.from_numpy(a.ravel()).cuda()
        return t[1:].view(a.shape)

    outb = torch.full((B * A + 1,), float("nan"), dtype=torch.float32, device="cuda")
    out = outb[1:].view(B, A)
    assert out.data_ptr() % 16 == 4
    pkg.ivit_action_combine(off(x0), off(v0), off(v7), off(al), off(be), off(b), out)
    np.testing.assert_allclose(out.cpu().numpy(), want, rtol=2e-6, atol=2e-6)
