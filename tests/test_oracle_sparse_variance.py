"""The sparse-probe variance prediction of App. G.1 for the oracle's
estimator (CPU).

For a probe z with independent coordinates z_j = a_j s_j (a_j = 1 with
probability q_j, else 0; s_j = +-1 with equal odds) and the small-eps
single-probe estimate X = (g . z) z:
  E[X_j]   = sum_k g_k E[z_j z_k] = q_j g_j,
  E[X_j^2] = sum_k g_k^2 E[z_j^2 z_k^2] = q_j g_j^2 + q_j sum_{k != j} q_k g_k^2,
so with s = sum_j q_j,
  tr Cov(X) = sum_j q_j (1 + s - 2 q_j) g_j^2,
and the average of n independent probes has n times less: the prediction
R_g = sum_j q_j (1 + s - 2 q_j) g_j^2 / (n |g|^2) printed in App. G.1
(q = 1 on normalisation gains, 1/2 elsewhere).  Dense probes (q = 1) give
(P - 1) / n, the law of Prop. 1.

The tests estimate tr Cov from many single-probe estimates c_r z_r of the
oracle (c_r its coefficient, z_r its probe) and compare with the prediction
computed from the exact gradient (the oracle's BPTT gradient for the LSTM
expert, torch autograd for the expert body), within four standard errors
of the sample estimate, and also within 12%.
"""
import numpy as np
import pytest

from paper_2609_37899_gb300 import inputs

V = 256


def predicted_trace(g, q):
    """tr Cov of one probe's estimate: sum_j q_j (1 + s - 2 q_j) g_j^2."""
    s = q.sum()
    return float(np.sum(q * (1.0 + s - 2.0 * q) * g * g))


def sample_trace(X):
    """Unbiased trace of the sample covariance of the rows of X and its
    standard error (from the spread of the per-sample squared deviations)."""
    R = X.shape[0]
    dev = np.sum((X - X.mean(axis=0)) ** 2, axis=1) * (R / (R - 1))
    return float(dev.mean()), float(dev.std(ddof=1) / np.sqrt(R))


def streamed_trace(coefs, probe, P):
    """sample_trace of the rows c_r z_r without holding them: coefs[r] and
    probe(r) (the probe vector z_r) are read twice, first for the mean, then
    for |c_r z_r - mean|^2 = c_r^2 |z_r|^2 - 2 c_r z_r . mean + |mean|^2."""
    R = len(coefs)
    mean = np.zeros(P)
    for r in range(R):
        mean += coefs[r] * probe(r)
    mean /= R
    mm = mean @ mean
    dev = np.empty(R)
    for r in range(R):
        z = probe(r)
        dev[r] = coefs[r] ** 2 * (z @ z) - 2.0 * coefs[r] * (z @ mean) + mm
    dev *= R / (R - 1)
    return float(dev.mean()), float(dev.std(ddof=1) / np.sqrt(R)), mean


def check(measured, se, predicted):
    assert abs(measured - predicted) < 4 * se + 1e-12, (measured, se, predicted)
    assert measured == pytest.approx(predicted, rel=0.12), (measured, predicted)


def test_lstm_sparse_probe_variance(oracle_mod):
    # every coordinate of the LSTM expert is a weight: q = 1/2, so the
    # prediction is (P / 4) |g|^2 per probe
    E, H, B, T = 2, 2, 2, 5
    rng = np.random.default_rng(41)
    P = inputs.param_count(E, H)
    theta = (rng.standard_normal((1, P)) * 0.6).astype(np.float64)
    bx = rng.integers(0, V, size=(1, B, T + 1), dtype=np.uint8)
    _, g = oracle_mod.bptt_grad(theta[0], E, H, bx[0])
    q = np.full(P, 0.5)
    n, steps = 64, 32
    X = []
    for st in range(steps):
        _, c = oracle_mod.spsa_losses(theta, E, H, 1e-4, 5, st, bx, n_pert=n, n_threads=1,
                                      kind="sparse")
        for i in range(n):
            z = oracle_mod.probe(5, st, 0, i, 0, P, kind="sparse").astype(np.float64)
            X.append(c[0, i] * z)
    X = np.asarray(X)
    m, se = sample_trace(X)
    pred = predicted_trace(g, q)
    assert pred == pytest.approx(P / 4 * g @ g, rel=1e-12)
    check(m, se, pred)
    # the mean of the estimate is q g
    slope = X.mean(axis=0) @ g / (g @ g)
    assert abs(slope - 0.5) < 4 * np.sqrt(pred / X.shape[0]) / np.linalg.norm(g)


def test_body_sparse_probe_variance_with_dense_gains(oracle_mod):
    # the expert body: gains always active (q = 1), weights q = 1/2.  The
    # setup makes the gains carry a large share of |g|^2 so that the
    # prediction with the true q differs from the one with q = 1/2 everywhere
    # by several standard errors.
    from test_oracle_body import _setup, _torch_body_grad
    d, D = 4, 1
    theta, head, bx = _setup(d, D, B=2, T=6, seed=23, wstd=0.15)
    th = theta.astype(np.float64)
    _, g = _torch_body_grad(th[0], d, D, head, bx[0])
    P = g.size
    g0 = inputs.body_offsets(d, D)["gains"]
    q = np.where(np.arange(P) < g0, 0.5, 1.0)
    n, steps = 64, 48
    X = []
    for st in range(steps):
        _, c = oracle_mod.body_spsa_losses(th, d, D, head, 1e-4, 9, st, bx, n_pert=n,
                                           kind="sparse", n_threads=1)
        for i in range(n):
            z = oracle_mod.body_probe(9, st, 0, i, d, D, 0, P, kind="sparse").astype(np.float64)
            X.append(c[0, i] * z)
    X = np.asarray(X)
    m, se = sample_trace(X)
    pred = predicted_trace(g, q)
    check(m, se, pred)
    uniform = predicted_trace(g, np.full(P, 0.5))
    assert abs(uniform - pred) > 4 * se, (uniform, pred, se)
