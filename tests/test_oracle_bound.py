"""Pins of the oracle's BGPO bound (Eq. 10, 13, 14), VRPO ratio (Eq. 7) and Eq. 18."""
import numpy as np
import pytest
from scipy import stats

from oracle import bgpo_oracle as O


def test_lower_bound_below_vrpo_ratio():
    # Lemma 1 (A >= 0) and Lemma 2 (A < 0): R_lb = sum_j g_j <= R_hat (Eq. 8)
    rng = np.random.default_rng(0)
    for n_t in (1, 2, 4, 16):
        ell = rng.standard_normal((200, n_t)) * 3
        ell_old = ell + rng.standard_normal((200, n_t)) * rng.uniform(0, 2, size=(200, 1))
        A = rng.standard_normal(200)
        A[:10] = 0.0
        _, g, _ = O.bound_coeffs(ell, ell_old, A[:, None], n_t, 1.0)
        R_lb = g.sum(axis=1)
        R_hat = O.vrpo_ratio(ell, ell_old, A)
        assert np.all(R_lb <= R_hat + 1e-12 * (1 + np.abs(R_hat)))


def test_taylor_bound_tight_only_at_zero():
    # e^x >= 1 + x with equality only at x = 0: strict for off-policy A > 0
    ell = np.array([[1.0, 2.0]])
    ell_old = np.array([[1.5, 1.0]])
    _, g, _ = O.bound_coeffs(ell, ell_old, np.array([[2.0]]), 2, 1.0)
    assert g.sum() < O.vrpo_ratio(ell, ell_old, np.array([2.0]))[0]


def test_equivalence_value_on_policy():
    # Sec. 3.2: d_j = 0 gives R_lb = R_hat = A
    rng = np.random.default_rng(1)
    for n_t in (1, 3, 16):
        ell = rng.standard_normal((50, n_t)) * 100
        A = rng.standard_normal(50)
        d, g, _ = O.bound_coeffs(ell, ell, A[:, None], n_t, 1.0)
        assert np.array_equal(d, np.zeros_like(d))
        assert np.allclose(g.sum(axis=1), A, rtol=1e-14, atol=1e-15)
        assert np.allclose(O.vrpo_ratio(ell, ell, A), A, rtol=1e-14, atol=1e-15)


def test_coef_is_derivative_of_loss_term():
    # coef = d(-loss_scale * g)/d l, checked by central differences of g itself
    rng = np.random.default_rng(2)
    ell = rng.standard_normal(40)
    ell_old = ell + rng.standard_normal(40) * 0.5
    A = rng.standard_normal(40)
    n_t, ls = 7, 0.125
    _, _, coef = O.bound_coeffs(ell, ell_old, A, n_t, ls)
    h = 1e-6
    _, gp, _ = O.bound_coeffs(ell + h, ell_old, A, n_t, ls)
    _, gm, _ = O.bound_coeffs(ell - h, ell_old, A, n_t, ls)
    fd = -ls * (gp - gm) / (2 * h)
    assert np.allclose(coef, fd, rtol=1e-8, atol=1e-12)


def test_on_policy_coefficient_same_for_both_branches():
    # Sec. 3.2: at d = 0 both branches give dg/dl = A / n_t
    A = np.array([-1.5, -0.1, 0.0, 0.2, 3.0])
    _, _, coef = O.bound_coeffs(np.ones(5), np.ones(5), A, 4, 0.5)
    assert np.allclose(coef, -0.5 * A / 4, rtol=0, atol=1e-16)


def test_nonfinite_raises():
    with pytest.raises(FloatingPointError):
        O.bound_coeffs(np.array([1000.0]), np.array([0.0]), np.array([-1.0]), 1, 1.0)


def test_group_advantage_matches_zscore():
    rng = np.random.default_rng(3)
    r = (rng.random(64) < 0.5).astype(np.float64)
    A = O.group_advantage(r, 8)
    for gidx in range(8):
        grp = r[8 * gidx:8 * gidx + 8]
        if grp.std() == 0:
            assert np.array_equal(A[8 * gidx:8 * gidx + 8], np.zeros(8))
        else:
            assert np.allclose(A[8 * gidx:8 * gidx + 8], stats.zscore(grp, ddof=0), rtol=1e-14)


def test_group_advantage_zero_std_group():
    assert np.array_equal(O.group_advantage(np.ones(4), 4), np.zeros(4))
    A = O.group_advantage(np.array([1.0, 0, 0, 0]), 4)
    assert abs(A.mean()) < 1e-15 and abs(A.std() - 1) < 1e-14
