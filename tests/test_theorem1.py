"""Theorem 1 (RMMC and directional curvature) on a quadratic objective, CPU only.

The oracle's Dion branch on a 1 x n parameter (rank 1) reduces to heavy-ball momentum with a
normalized step, for which Theorem 1's expansion can be written out exactly on
F(x) = x^T H x / 2.  These tests pin that reduction with closed forms, check the oracle's
RMMC against the exact momentum-norm ratio along closed-loop trajectories, and check
Theorem 1's |eta kappa + B_t| against it (exact in one dimension, within the
perpendicular-gradient term rho^2 / (2 a) otherwise).
"""
import math

import numpy as np
import pytest

import oracle.curvadion as oc
import workloads as wl

RNG = np.random.default_rng(77)


@pytest.mark.parametrize("n", [1, 5, 64])
def test_rank1_dion_step_is_normalized_heavy_ball(n):
    """M_t = mu B and X_t = X - eta / (sqrt(n) (||B|| + eps)) B for a 1 x n layer, whatever the
    sign of B Q_{t-1}."""
    for sgn in (1.0, -1.0):
        B = RNG.standard_normal((1, n))
        Qp = RNG.standard_normal((n, 1))
        Qp *= sgn * np.sign((B @ Qp).item())
        X = RNG.standard_normal((1, n))
        res = oc.dion_sync_update(B, Qp, X, 0.9, 0.03, 1e-8)
        assert np.allclose(res.M, 0.9 * B, rtol=0, atol=1e-14)
        step = 0.03 / (math.sqrt(n) * (np.linalg.norm(B) + 1e-8))
        assert step == pytest.approx(oc.rank1_step_size(0.03, n, B, 1e-8), rel=1e-15)
        assert np.allclose(res.X, X - step * B, rtol=0, atol=1e-14)


def closed_loop(n, steps, eta, mu, seed):
    """Oracle trajectory of one 1 x n layer on the quadratic, G_t = H x_t each step."""
    H = wl.quadratic_hessian(n, seed).double().numpy()
    x = wl.quadratic_start(n, seed + 1).double().numpy()
    q = RNG.standard_normal((n, 1))
    layer = oc.LayerState(X=x, M=np.zeros((1, n)), Q=q / np.linalg.norm(q), tau=0.5)
    hp = oc.HParams(mu=mu, eta=eta, eps_rmmc=1e-300, eps_col=1e-300)
    prev, hist = [0.0], []
    for t in range(1, steps + 1):
        G = layer.X @ H
        B = layer.M + G
        o = oc.curvadion_step([layer], [G], prev, hp, t)
        hist.append(dict(x=layer.X.copy(), b=B, rmmc=float(o.rmmc[0])))
        layer, prev = o.layers[0], o.prev_norm
    return H, hist


def test_theorem1_exact_in_one_dimension():
    """n = 1: no gradient component leaves the momentum direction, so RMMC_t = |eta kappa + B_t|
    holds with no remainder (Theorem 1 without its O(eta^2))."""
    eta, mu = 0.05, 0.95
    H, hist = closed_loop(1, 40, eta, mu, seed=3)
    for t in range(1, len(hist)):
        prev = hist[t - 1]
        terms = oc.theorem1_terms(H, prev["x"], prev["b"], mu, oc.rank1_step_size(eta, 1, prev["b"], 1e-300))
        assert terms.rho == 0.0
        assert hist[t]["rmmc"] == pytest.approx(terms.prediction, rel=1e-10, abs=1e-13)
        assert terms.kappa == pytest.approx(float(H[0, 0]), rel=1e-14)


@pytest.mark.parametrize("n,eta", [(64, 0.01), (64, 0.05), (512, 0.02)])
def test_theorem1_identity_and_remainder_bound(n, eta):
    """n > 1: the oracle's RMMC equals |sqrt((1 - B_t - eta kappa)^2 + rho^2) - 1| exactly, and
    Theorem 1's |eta kappa + B_t| is within rho^2 / (2 (1 - B_t - eta kappa)) of it."""
    mu = 0.95
    H, hist = closed_loop(n, 40, eta, mu, seed=5)
    worst_gap = 0.0
    for t in range(1, len(hist)):
        prev = hist[t - 1]
        terms = oc.theorem1_terms(H, prev["x"], prev["b"], mu, oc.rank1_step_size(eta, n, prev["b"], 1e-300))
        a = 1.0 - terms.bias - terms.eta_eff * terms.kappa
        assert a > 0
        assert hist[t]["rmmc"] == pytest.approx(terms.exact, rel=1e-9, abs=1e-12)
        gap = abs(hist[t]["rmmc"] - terms.prediction)
        assert gap <= terms.rho ** 2 / (2 * a) + 1e-12
        worst_gap = max(worst_gap, gap)
    assert worst_gap > 0.0  # the perpendicular term is present for n > 1


def test_theorem1_kappa_is_the_rayleigh_quotient():
    """kappa equals the Rayleigh quotient of H along the momentum, between H's extreme
    eigenvalues, and equals an eigenvalue when the momentum is an eigenvector."""
    n = 32
    H = wl.quadratic_hessian(n, 11).double().numpy()
    lam, U = np.linalg.eigh(H)
    b = RNG.standard_normal((1, n))
    t = oc.theorem1_terms(H, RNG.standard_normal((1, n)), b, 0.9, 0.01)
    assert lam[0] - 1e-12 <= t.kappa <= lam[-1] + 1e-12
    t2 = oc.theorem1_terms(H, RNG.standard_normal((1, n)), 3.0 * U[:, 7][None, :], 0.9, 0.01)
    assert t2.kappa == pytest.approx(lam[7], rel=1e-12)


def test_mutation_step_without_sqrt_n_is_caught(monkeypatch):
    real = oc.rank1_step_size
    monkeypatch.setattr(oc, "rank1_step_size", lambda eta, n, b, eps: real(eta, 1, b, eps))
    with pytest.raises(AssertionError):
        test_rank1_dion_step_is_normalized_heavy_ball(64)
    with pytest.raises(AssertionError):
        test_theorem1_identity_and_remainder_bound(64, 0.05)
