"""Pins of the oracle's SPSA estimator and update (CPU only).

Eq. main-spsa: g_hat = (1/n) sum_j (L(theta+eps z_j) - L(theta-eps z_j))/(2 eps) z_j.
Pins: eps = 0 and lr = 0 special cases, the n = 1 closed form with probes from
an independent Philox, the eps -> 0 limit against the BPTT gradient (itself
pinned to torch autograd and brute-force differences), expert separability,
the large-n limit and the variance law of Prop. 1 (App. F)."""
import numpy as np
import pytest

import philox_ref
from paper_2609_37899_gb300 import inputs

V = 256


def _micro(E=2, H=3, B=2, T=6, N=1, seed=0, std=0.5):
    rng = np.random.default_rng(seed)
    P = inputs.param_count(E, H)
    theta = (rng.standard_normal((N, P)) * std).astype(np.float32)
    bx = rng.integers(0, V, size=(N, B, T + 1), dtype=np.uint8)
    return theta, bx


def test_eps_zero_gives_equal_losses(oracle_mod):
    E, H = 3, 5
    theta, bx = _micro(E, H)
    L, coef = oracle_mod.spsa_losses(theta, E, H, 0.0, 0, 0, bx, n_pert=4)
    base = oracle_mod.loss(theta[0], E, H, bx[0])
    assert (L[..., 0] == L[..., 1]).all()
    assert (L[..., 0] == base).all()
    assert (coef == 0).all()


def test_lr_zero_leaves_theta(oracle_mod):
    E, H = 3, 5
    theta, bx = _micro(E, H, N=2)
    _, _, new = oracle_mod.spsa_step(theta, E, H, 4, np.float32(1e-3), 0.0, 3, 7, bx)
    assert (new == theta.astype(np.float64)).all()


@pytest.mark.skipif(not philox_ref.available(), reason="torch Philox header not found")
def test_update_closed_form_independent_probes(oracle_mod):
    E, H, N, n = 3, 4, 2, 3
    theta, _ = _micro(E, H, N=N)
    P = inputs.param_count(E, H)
    coef = np.array([[0.7, -1.3, 2.0], [0.25, 0.0, -4.0]])
    lr, seed, step = 0.05, 11, 5
    got = oracle_mod.spsa_update(theta, E, H, lr, seed, step, coef)
    for e in range(N):
        z = np.stack([philox_ref.rademacher(seed, step, e, i, 0, P) for i in range(n)]).astype(np.float64)
        want = theta[e].astype(np.float64) - lr * (coef[e] @ z) / n
        np.testing.assert_allclose(got[e], want, rtol=0, atol=1e-15)


def test_coefficient_tends_to_directional_derivative(oracle_mod):
    # (L+ - L-)/(2 eps) = g.z + O(eps^2) (App. F, proof of Prop. 1)
    E, H = 4, 6
    theta, bx = _micro(E, H, B=3, T=8, seed=5, std=0.4)
    th64 = theta.astype(np.float64)
    _, g = oracle_mod.bptt_grad(th64[0], E, H, bx[0])
    P = g.size
    errs = []
    for eps in [1e-1, 3e-2, 1e-2, 3e-3]:
        _, coef = oracle_mod.spsa_losses(th64, E, H, eps, 9, 2, bx, probes=[0, 1, 2])
        want = np.array([g @ oracle_mod.rademacher(9, 2, 0, i, 0, P) for i in range(3)])
        errs.append(np.abs(coef[0] - want).max() / np.abs(want).max())
    slopes = np.diff(np.log(errs)) / np.diff(np.log([1e-1, 3e-2, 1e-2, 3e-3]))
    assert np.all(slopes > 1.8) and np.all(slopes < 2.2), (errs, slopes)
    _, coef = oracle_mod.spsa_losses(th64, E, H, 1e-4, 9, 2, bx, probes=[0, 1, 2])
    want = np.array([g @ oracle_mod.rademacher(9, 2, 0, i, 0, P) for i in range(3)])
    assert np.abs(coef[0] - want).max() / np.abs(want).max() < 1e-6


def test_experts_are_separable(oracle_mod):
    # Eq. separable-training-objective: expert e's losses, coefficients and
    # update depend only on theta_e and its own batch.
    E, H, n = 3, 4, 5
    theta, bx = _micro(E, H, N=3, seed=8)
    L, coef, new = oracle_mod.spsa_step(theta, E, H, n, np.float32(1e-3), 0.1, 1, 1, bx)
    theta2 = theta.copy()
    theta2[1] += 0.3
    bx2 = bx.copy()
    bx2[2] = bx[2][:, ::-1]
    L2, coef2, new2 = oracle_mod.spsa_step(theta2, E, H, n, np.float32(1e-3), 0.1, 1, 1, bx2)
    assert (L2[0] == L[0]).all() and (coef2[0] == coef[0]).all() and (new2[0] == new[0]).all()
    assert (L2[1] != L[1]).any() and (L2[2] != L[2]).any()
    # the summed objective of the ensemble is the sum of the expert losses
    tot = sum(oracle_mod.loss(theta[e], E, H, bx[e]) for e in range(3))
    _, c0 = oracle_mod.spsa_losses(theta, E, H, 0.0, 1, 1, bx, probes=[0])
    L0, _ = oracle_mod.spsa_losses(theta, E, H, 0.0, 1, 1, bx, probes=[0])
    assert L0[:, 0, 0].sum() == pytest.approx(tot, abs=1e-13)


def _g_hat(oracle_mod, theta64, E, H, n, eps, seed, step, bx, lr=1.0):
    L, coef = oracle_mod.spsa_losses(theta64, E, H, eps, seed, step, bx, n_pert=n, n_threads=1)
    new = oracle_mod.spsa_update(theta64, E, H, lr, seed, step, coef)
    return (theta64 - new)[0] / lr


def test_mean_estimate_converges_to_gradient(oracle_mod):
    # E_z[g_hat] = g + O(eps^2) and the error of an average over n_total
    # directions has E||g_hat - g||^2/||g||^2 = (P-1)/n_total.
    E, H = 1, 1
    theta, bx = _micro(E, H, B=2, T=6, seed=11, std=0.8)
    th = theta.astype(np.float64)
    _, g = oracle_mod.bptt_grad(th[0], E, H, bx[0])
    P = g.size
    reps, n = 8, 2048
    acc = np.zeros(P)
    for r in range(reps):
        acc += _g_hat(oracle_mod, th, E, H, n, 1e-3, 21, r, bx)
    gh = acc / reps
    rel2 = np.sum((gh - g) ** 2) / np.sum(g ** 2)
    pred = (P - 1) / (reps * n)
    assert 0.75 < rel2 / pred < 1.3, (rel2, pred)
    cos = gh @ g / np.linalg.norm(gh) / np.linalg.norm(g)
    assert cos > 1.0 / np.sqrt(1.0 + 1.5 * pred)


def test_variance_law(oracle_mod):
    # Prop. 1 / Eq. main-variance: E||g_hat - g||^2/||g||^2 = (d-1)/n_pert + O(eps^2)
    E, H = 2, 2
    theta, bx = _micro(E, H, B=2, T=5, seed=13, std=0.6)
    th = theta.astype(np.float64)
    _, g = oracle_mod.bptt_grad(th[0], E, H, bx[0])
    P = g.size
    for n in (8, 64):
        reps = 2048 // n
        ratios = []
        for r in range(reps):
            gh = _g_hat(oracle_mod, th, E, H, n, 1e-3, 33, 1000 * n + r, bx)
            ratios.append(np.sum((gh - g) ** 2) / np.sum(g ** 2))
        assert np.mean(ratios) == pytest.approx((P - 1) / n, rel=0.12), (n, np.mean(ratios), (P - 1) / n)
