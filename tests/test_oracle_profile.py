"""Pins of the oracle's sensitivity-profiling steps (Sec. 4.3): the
norm-adaptive Value perturbation (Eq. 6), the KL divergence averaged over the
evaluation window (Eq. 7) and the calibration-set average (Eq. 8).

Pins: hand-derived closed forms (one-hot rows, two-category and
uniform-versus-spike distributions), invariants (KL(P||P) = 0, invariance of
the softmax to a constant shift of the logits, the norm of the added noise),
and the asymmetry of the divergence, which fails if P and Q are swapped.
"""
import math

import numpy as np
import pytest

from oracle import ripple_oracle as O


def _rng(seed):
    return np.random.default_rng(seed)


# ----------------------------------------------------------- perturbation (Eq. 6)


def test_perturbation_of_one_hot_rows_is_alpha_abs_c_eps():
    # v_u = c_u e_{k_u}: ||v_u||_2 = |c_u|, so v~_u - v_u = alpha |c_u| eps_u,
    # with eps indexed from the first eligible position.
    B, H, T, d = 2, 3, 9, 8
    rng = _rng(1)
    v = np.zeros((B, H, T, d))
    c = rng.uniform(-4.0, 4.0, size=(B, H, T))
    k = rng.integers(0, d, size=(B, H, T))
    for b in range(B):
        for h in range(H):
            for u in range(T):
                v[b, h, u, k[b, h, u]] = c[b, h, u]
    pb, pe, alpha = 2, 7, 0.3
    eps = rng.standard_normal((B, H, pe - pb, d))
    out = O.perturb_values(v, eps, alpha, pb, pe)
    for b in range(B):
        for h in range(H):
            for u in range(T):
                if pb <= u < pe:
                    want = v[b, h, u] + alpha * abs(c[b, h, u]) * eps[b, h, u - pb]
                else:
                    want = v[b, h, u]
                np.testing.assert_allclose(out[b, h, u], want, rtol=0, atol=1e-14)


def test_perturbation_noise_norm_identity():
    # ||v~_u - v_u|| = alpha ||v_u|| ||eps_u|| for every eligible row, and the
    # added noise points along eps_u.
    rng = _rng(2)
    v = rng.standard_normal((2, 2, 16, 64)) * rng.lognormal(0, 1, size=(2, 2, 16, 1))
    eps = rng.standard_normal((2, 2, 10, 64))
    alpha = 0.05
    out = O.perturb_values(v, eps, alpha, 3, 13)
    delta = out[:, :, 3:13] - v[:, :, 3:13]
    vn = np.linalg.norm(v[:, :, 3:13], axis=-1)
    en = np.linalg.norm(eps, axis=-1)
    np.testing.assert_allclose(np.linalg.norm(delta, axis=-1), alpha * vn * en, rtol=1e-12)
    cos = np.sum(delta * eps, axis=-1) / (np.linalg.norm(delta, axis=-1) * en)
    np.testing.assert_allclose(cos, 1.0, rtol=1e-12)


def test_perturbation_leaves_protected_rows_and_alpha_zero_unchanged():
    rng = _rng(3)
    v = rng.standard_normal((1, 2, 12, 16))
    eps = rng.standard_normal((1, 2, 5, 16))
    out = O.perturb_values(v, eps, 0.2, 4, 9)
    assert np.array_equal(out[:, :, :4], v[:, :, :4])
    assert np.array_equal(out[:, :, 9:], v[:, :, 9:])
    assert not np.array_equal(out[:, :, 4:9], v[:, :, 4:9])
    assert np.array_equal(O.perturb_values(v, eps, 0.0, 4, 9), v)
    assert np.array_equal(O.perturb_values(v, np.zeros((1, 2, 0, 16)), 0.2, 6, 6), v)


def test_perturbation_is_positively_homogeneous():
    # scaling the cache by s > 0 scales the perturbed cache by s
    rng = _rng(4)
    v = rng.standard_normal((1, 1, 6, 32))
    eps = rng.standard_normal((1, 1, 6, 32))
    np.testing.assert_allclose(O.perturb_values(2.5 * v, eps, 0.1, 0, 6),
                               2.5 * O.perturb_values(v, eps, 0.1, 0, 6), rtol=1e-12,
                               atol=1e-14)


# ----------------------------------------------------------- window KL (Eq. 7)


def test_two_category_closed_form_and_asymmetry():
    # P = (1/4, 3/4) from logits (0, log 3); Q = (1/2, 1/2) from (0, 0):
    # KL(P||Q) = 1/4 log(1/2) + 3/4 log(3/2); KL(Q||P) = 1/2 log 2 + 1/2 log(2/3)
    p = [[0.0, math.log(3.0)]]
    q = [[0.0, 0.0]]
    kl, d = O.window_kl(p, q)
    assert kl[0] == pytest.approx(0.25 * math.log(0.5) + 0.75 * math.log(1.5), rel=1e-14)
    assert d == pytest.approx(0.1308120359411371, rel=1e-12)
    kl_r, _ = O.window_kl(q, p)
    assert kl_r[0] == pytest.approx(0.5 * math.log(2.0) + 0.5 * math.log(2.0 / 3.0), rel=1e-14)
    assert abs(kl_r[0] - kl[0]) > 0.01


@pytest.mark.parametrize("V,a", [(1000, 5.0), (128256, 12.0), (7, -3.0)])
def test_uniform_versus_spike_closed_forms(V, a):
    # p = 0 (uniform U); q = a at token 0, 0 elsewhere: Q_0 = e^a / Z, Q_v = 1/Z
    # with Z = e^a + V - 1, so KL(U||Q) = log Z - log V - a / V, and
    # KL(Q||U) = log V - H(Q) = log V + (e^a / Z)(a - log Z) - ((V - 1)/Z) log Z.
    p = np.zeros((1, V))
    q = np.zeros((1, V))
    q[0, 0] = a
    Z = math.exp(a) + V - 1
    kl, _ = O.window_kl(p, q)
    assert kl[0] == pytest.approx(math.log(Z) - math.log(V) - a / V, rel=1e-9, abs=1e-15)
    kl_r, _ = O.window_kl(q, p)
    want = math.log(V) + math.exp(a) / Z * (a - math.log(Z)) - (V - 1) / Z * math.log(Z)
    assert kl_r[0] == pytest.approx(want, rel=1e-9, abs=1e-15)


def test_kl_of_identical_and_shifted_logits_is_zero():
    rng = _rng(5)
    p = rng.standard_normal((4, 5000)) * 3.0
    kl, d = O.window_kl(p, p)
    assert np.all(kl == 0.0) and d == 0.0
    shift = np.array([[1.5], [-40.0], [900.0], [0.0]])
    kl, d = O.window_kl(p, p + shift)
    np.testing.assert_allclose(kl, 0.0, atol=1e-12)


def test_window_average_and_nonnegativity():
    # d is the mean over the window positions of the per-position divergences
    p = [[0.0, math.log(3.0)], [0.0, 0.0], [1.0, -1.0]]
    q = [[0.0, 0.0], [0.0, 0.0], [-1.0, 1.0]]
    kl, d = O.window_kl(p, q)
    s1 = 1.0 / (1.0 + math.exp(-2.0))  # P = (s1, 1 - s1), Q = (1 - s1, s1)
    k3 = s1 * math.log(s1 / (1 - s1)) + (1 - s1) * math.log((1 - s1) / s1)
    np.testing.assert_allclose(kl, [0.1308120359411371, 0.0, k3], rtol=1e-12, atol=1e-15)
    assert d == pytest.approx((0.1308120359411371 + k3) / 3.0, rel=1e-12)
    rng = _rng(6)
    kl, _ = O.window_kl(rng.standard_normal((8, 300)) * 4, rng.standard_normal((8, 300)) * 4)
    assert np.all(kl > 0)


def test_large_logits_are_stable():
    # logits near 1e3 (overflow of a naive exp) give the same KL as shifted ones
    rng = _rng(7)
    p = rng.standard_normal((2, 64))
    q = p + 0.1 * rng.standard_normal((2, 64))
    kl0, _ = O.window_kl(p, q)
    kl1, _ = O.window_kl(p + 1000.0, q + 1000.0)
    np.testing.assert_allclose(kl1, kl0, rtol=1e-9)
    assert np.all(np.isfinite(kl1))


# ------------------------------------------------- calibration average (Eq. 8)


def test_sensitivity_profile_is_the_example_average():
    d = [[1.0, 2.0, 0.5], [3.0, 4.0, 0.5], [2.0, 0.0, 0.5]]
    np.testing.assert_array_equal(O.sensitivity_profile(d), [2.0, 2.0, 0.5])
    np.testing.assert_array_equal(O.sensitivity_profile([[0.25, 7.0]]), [0.25, 7.0])
