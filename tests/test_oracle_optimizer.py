"""Pins of the oracle's sparse probes and Adam step (App. E, Eq. localspsa).
CPU only.

Sparse probes:
- The sign and activity bits come from an independent Philox: torch's
  PhiloxRNGEngine.h, through tests/philox_ref.py.
- The value distribution is P(0) = 1/2 and P(-1) = P(+1) = 1/4.
- The sparse SPSA estimator's mean is half the gradient: App. E, q_j = 1/2,
  no inverse-probability rescaling.
- Its squared relative error about that mean is P / n_total. For one probe,
  X = (g.z) z has Var[X_p] = |g|^2 / 4 for every p, so
  E|ghat - g/2|^2 / |g/2|^2 = P / n_total.

Adam:
- First update: theta - lr g / (|g| + delta).
- A constant estimate: the bias-corrected moments equal g at every update t.
- Weight decay alone.
- The average over identical accumulation batches equals one batch.
- Opposite coefficients cancel.
"""
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


def _sparse_ref(seed, step, e, i, p0, count):
    """Sparse probe from the independent Philox: the sign of the dense probe
    where the activity stream (probe | 2^31) has its bit set, else 0."""
    sign = philox_ref.rademacher(seed, step, e, i, p0, count).astype(np.int64)
    act = philox_ref.rademacher(seed, step, e, i | 0x80000000, p0, count)  # -1 <=> bit set
    return np.where(act == -1, sign, 0).astype(np.int8)


@pytest.mark.skipif(not philox_ref.available(), reason="torch Philox header not found")
def test_sparse_probe_matches_independent_philox(oracle_mod):
    for (seed, step, e, i, p0, count) in [(7, 3, 0, 1, 0, 300), (2**40 + 5, 2**33 + 9, 3, 77, 61, 500),
                                          (0, 0, 1, 12287, 1000, 257)]:
        got = oracle_mod.probe(seed, step, e, i, p0, count, kind="sparse")
        np.testing.assert_array_equal(got, _sparse_ref(seed, step, e, i, p0, count))
        dense = oracle_mod.probe(seed, step, e, i, p0, count, kind="dense")
        np.testing.assert_array_equal(dense, philox_ref.rademacher(seed, step, e, i, p0, count))


def test_sparse_probe_distribution(oracle_mod):
    n = 200_000
    zs = [oracle_mod.probe(11, s, e, i, 0, n, kind="sparse") for s, e, i in [(0, 0, 0), (1, 2, 5)]]
    for z in zs:
        sd = np.sqrt(0.25 / n)
        assert abs((z == 0).mean() - 0.5) < 5 * sd
        assert abs((z == 1).mean() - 0.25) < 5 * np.sqrt(0.1875 / n)
        assert abs((z == -1).mean() - 0.25) < 5 * np.sqrt(0.1875 / n)
    # independent probes are uncorrelated; a nonzero coordinate is the dense sign
    c = np.mean(zs[0].astype(np.float64) * zs[1])
    assert abs(c) < 5 * np.sqrt(0.25 / n)
    d = oracle_mod.probe(11, 0, 0, 0, 0, n, kind="dense")
    assert np.all((zs[0] == 0) | (zs[0] == d))


def test_sparse_estimator_mean_is_half_gradient(oracle_mod):
    E, H = 1, 1
    theta, bx = _micro(E, H, B=2, T=6, seed=11, std=0.8)
    th = theta.astype(np.float64)
    _, g = oracle_mod.bptt_grad(th[0], E, H, bx[0])
    P = g.size
    reps, n = 8, 2048
    coefs = []
    for r in range(reps):
        _, c = oracle_mod.spsa_losses(th, E, H, 1e-3, 21, r, bx, n_pert=n, n_threads=1,
                                      kind="sparse")
        coefs.append(c)
    coef = np.stack(coefs)  # [A, N, n]
    # with beta1 = 0, t = 1 and no decay the new first moment is the estimate
    # averaged over the A accumulation batches
    zeros = np.zeros_like(th)
    _, m, _ = oracle_mod.adam_update(th, zeros, zeros, E, H, 21, list(range(reps)), coef,
                                     lr=0.0, beta1=0.0, beta2=0.0, delta=1.0, wd=0.0, t=1,
                                     kind="sparse")
    gh = m[0]
    half = 0.5 * g
    rel2 = np.sum((gh - half) ** 2) / np.sum(half ** 2)
    pred = P / (reps * n)
    assert 0.75 < rel2 / pred < 1.3, (rel2, pred)
    slope = gh @ g / (g @ g)
    assert abs(slope - 0.5) < 0.05, slope


@pytest.mark.skipif(not philox_ref.available(), reason="torch Philox header not found")
@pytest.mark.parametrize("kind", ["sparse", "dense"])
def test_adam_first_update_closed_form(oracle_mod, kind):
    E, H, N, n = 3, 4, 2, 3
    theta, _ = _micro(E, H, N=N, seed=3)
    th = theta.astype(np.float64)
    P = inputs.param_count(E, H)
    coef = np.array([[[0.7, -1.3, 2.0], [0.25, 0.0, -4.0]]])
    lr, b1, b2, delta, seed, step = 0.05, 0.9, 0.999, 1e-8, 11, 5
    zeros = np.zeros_like(th)
    got, m, v = oracle_mod.adam_update(th, zeros, zeros, E, H, seed, [step], coef, lr, b1, b2,
                                       delta, 0.0, 1, kind=kind)
    for e in range(N):
        if kind == "sparse":
            z = np.stack([_sparse_ref(seed, step, e, i, 0, P) for i in range(n)])
        else:
            z = np.stack([philox_ref.rademacher(seed, step, e, i, 0, P) for i in range(n)])
        g = coef[0, e] @ z.astype(np.float64) / n
        np.testing.assert_allclose(m[e], (1 - b1) * g, rtol=1e-14, atol=1e-300)
        np.testing.assert_allclose(v[e], (1 - b2) * g * g, rtol=1e-14, atol=1e-300)
        np.testing.assert_allclose(got[e], th[e] - lr * g / (np.abs(g) + delta), rtol=0,
                                   atol=1e-12)
        if kind == "sparse":
            # coordinates no probe touched keep their value
            untouched = np.all(z == 0, axis=0)
            assert untouched.any()
            np.testing.assert_array_equal(got[e][untouched], th[e][untouched])


def test_adam_constant_estimate(oracle_mod):
    # the same estimate at every update: mhat_t = g and vhat_t = g^2 exactly,
    # so every update moves theta by lr g / (|g| + delta)
    E, H, N = 2, 3, 1
    theta, _ = _micro(E, H, N=N, seed=5)
    th0 = theta.astype(np.float64)
    coef = np.array([[[1.5, -0.5, 0.25, 2.0]]])
    lr, b1, b2, delta = 0.01, 0.5, 0.75, 1e-3
    th, m, v = th0, np.zeros_like(th0), np.zeros_like(th0)
    for t in (1, 2, 3):
        th, m, v = oracle_mod.adam_update(th, m, v, E, H, 9, [4], coef, lr, b1, b2, delta, 0.0,
                                          t, kind="sparse")
        _, m1, _ = oracle_mod.adam_update(th0, np.zeros_like(th0), np.zeros_like(th0), E, H, 9,
                                          [4], coef, 0.0, 0.0, 0.0, 1.0, 0.0, 1, kind="sparse")
        g = m1  # beta1 = 0: the estimate itself
        np.testing.assert_allclose(m, (1 - b1 ** t) * g, rtol=1e-12, atol=1e-300)
        np.testing.assert_allclose(v, (1 - b2 ** t) * g * g, rtol=1e-12, atol=1e-300)
        np.testing.assert_allclose(th, th0 - t * lr * g / (np.abs(g) + delta), rtol=0, atol=1e-13)


def test_adam_weight_decay_alone(oracle_mod):
    E, H, N = 2, 3, 2
    theta, _ = _micro(E, H, N=N, seed=8)
    th = theta.astype(np.float64)
    coef = np.zeros((1, N, 2))
    lr, wd, delta = 0.1, 1e-2, 1e-8
    zeros = np.zeros_like(th)
    got, m, _ = oracle_mod.adam_update(th, zeros, zeros, E, H, 1, [0], coef, lr, 0.9, 0.999,
                                       delta, wd, 1, kind="sparse")
    np.testing.assert_allclose(m, 0.1 * wd * th, rtol=1e-14)
    np.testing.assert_allclose(got, th - lr * (wd * th) / (np.abs(wd * th) + delta), atol=1e-15)


def test_adam_accumulation_average(oracle_mod):
    E, H, N = 2, 3, 2
    theta, _ = _micro(E, H, N=N, seed=9)
    th = theta.astype(np.float64)
    zeros = np.zeros_like(th)
    # no signed subset sum of a row is zero: every touched coordinate has an
    # estimate far from 0, where the summation order cannot flip its sign
    c = np.array([[0.3, -1.1, 0.7], [2.0, 0.5, -0.7]])
    args = (0.02, 0.9, 0.999, 1e-8, 0.0, 1)
    one = oracle_mod.adam_update(th, zeros, zeros, E, H, 4, [6], c[None], *args)
    two = oracle_mod.adam_update(th, zeros, zeros, E, H, 4, [6, 6], np.stack([c, c]), *args)
    for a, b in zip(one, two):
        np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-300)
    # opposite coefficients on the same probes cancel up to the rounding of
    # the running sum (~1e-16); with delta = 1e-8 theta moves by < lr 1e-7
    th2, m2, v2 = oracle_mod.adam_update(th, zeros, zeros, E, H, 4, [6, 6], np.stack([c, -c]),
                                         *args)
    assert np.max(np.abs(th2 - th)) < 0.02 * 1e-7
    assert np.max(np.abs(m2)) < 1e-15 and np.max(v2) < 1e-30
