"""Pins of the oracle's 2-step action combine (Sec. III-C, Eq. 9) (CPU only).

- with velocities that lie exactly in the span of the two anchors (the low-rank model of
  the equation before Eq. 9), the combine with alpha = sum_t dt a_t, beta = sum_t dt b_t,
  b = 0 equals the Euler integration of all T steps;
- closed forms: zero coefficients return x_0, b alone shifts, linearity in alpha and beta;
- the Euler integrator against a numpy cumulative sum.
"""
import numpy as np


def test_combine_equals_euler_for_low_rank_velocities(oracle_mod):
    rng = np.random.Generator(np.random.PCG64(5))
    B, A, T, dt = 4, 50 * 7, 10, 0.1
    x0 = rng.standard_normal((B, A)).astype(np.float32)
    v0 = rng.standard_normal((B, A)).astype(np.float32)
    v7 = rng.standard_normal((B, A)).astype(np.float32)
    a = rng.standard_normal((T, B)).astype(np.float32)
    b = rng.standard_normal((T, B)).astype(np.float32)
    v = a[:, :, None] * v0[None] + b[:, :, None] * v7[None]
    v[0], v[7] = v0, v7  # the anchors themselves: a_0 = 1, b_0 = 0, a_7 = 0, b_7 = 1
    a[0], b[0], a[7], b[7] = 1, 0, 0, 1
    euler = oracle_mod.euler(x0, v, dt)
    alpha = (dt * a.astype(np.float64)).sum(0)
    beta = (dt * b.astype(np.float64)).sum(0)
    comb = oracle_mod.action_combine(x0, v0, v7, alpha, beta)
    np.testing.assert_allclose(comb, euler, rtol=1e-5, atol=1e-5)


def test_combine_closed_forms(oracle_mod):
    rng = np.random.Generator(np.random.PCG64(6))
    B, A = 3, 17
    x0, v0, v7, bias = (rng.standard_normal((B, A)).astype(np.float32) for _ in range(4))
    z = np.zeros(B, np.float32)
    np.testing.assert_array_equal(oracle_mod.action_combine(x0, v0, v7, z, z), x0)
    np.testing.assert_allclose(oracle_mod.action_combine(x0, v0, v7, z, z, bias), x0 + bias, rtol=1e-6)
    al = np.array([2.0, -1.0, 0.5], np.float32)
    be = np.array([0.0, 3.0, -2.0], np.float32)
    want = x0.astype(np.float64) + al[:, None] * v0 + be[:, None] * v7 + bias
    np.testing.assert_allclose(oracle_mod.action_combine(x0, v0, v7, al, be, bias), want, rtol=1e-6, atol=1e-6)


def test_euler_matches_cumulative_sum(oracle_mod):
    rng = np.random.Generator(np.random.PCG64(7))
    x0 = rng.standard_normal((2, 9)).astype(np.float32)
    v = rng.standard_normal((6, 2, 9)).astype(np.float32)
    np.testing.assert_allclose(oracle_mod.euler(x0, v, 0.25), x0 + 0.25 * v.sum(0), rtol=1e-6, atol=1e-6)
