"""Pins of the oracle's two mechanism variants (App. D). CPU only.

Per-probe batches: every probe of an expert draws its own batch.
- Giving every probe the shared batch reproduces the shared-batch step
  exactly.
- Probe i's losses depend on batch i and on no other batch.

Summed-loss control arm: the experts' losses are summed before each finite
difference.
- N = 1 is the per-expert estimator.
- The coefficient tends to sum_e g_e . z_{e,i}, with an O(eps^2) error
  (slope 2), against the BPTT gradient.
- Its error about the gradient obeys the variance law derived here for
  dense probes. For expert e with r = sum_{e' != e} g_e'.z_e' (mean 0,
  variance R = sum_{e' != e} |g_e'|^2, independent of z_e):
    E|ghat_e - g_e|^2 / |g_e|^2 = [(P_e - 1) + P_e R / |g_e|^2] / n,
  against (P_e - 1) / n for the expert's own loss (Prop. 1).
"""
import numpy as np
import pytest

from paper_2609_37899_gb300 import inputs

V = 256


def _micro(E=2, H=3, B=2, T=6, N=1, seed=0, std=0.5):
    rng = np.random.default_rng(seed)
    P = inputs.param_count(E, H)
    theta = (rng.standard_normal((N, P)) * std).astype(np.float32)
    bx = rng.integers(0, V, size=(N, B, T + 1), dtype=np.uint8)
    return theta, bx


@pytest.mark.parametrize("kind", ["dense", "sparse"])
def test_per_probe_batches_equal_to_shared(oracle_mod, kind):
    E, H, N, n = 2, 3, 2, 4
    theta, bx = _micro(E, H, N=N, seed=2)
    shared = oracle_mod.spsa_losses(theta, E, H, 1e-3, 5, 7, bx, n_pert=n, kind=kind)
    per = np.repeat(bx[:, None], n, axis=1)  # [N, n, B, T+1]
    got = oracle_mod.spsa_losses(theta, E, H, 1e-3, 5, 7, per, n_pert=n, kind=kind,
                                 batch_per_probe=True)
    for a, b in zip(shared, got):
        np.testing.assert_array_equal(a, b)


def test_per_probe_batch_is_the_probes_own(oracle_mod):
    E, H, N, n = 2, 3, 1, 3
    theta, _ = _micro(E, H, N=N, seed=4)
    rng = np.random.default_rng(1)
    per = rng.integers(0, V, size=(N, n, 2, 7), dtype=np.uint8)
    L0, c0 = oracle_mod.spsa_losses(theta, E, H, 1e-2, 1, 1, per, n_pert=n, batch_per_probe=True)
    changed = per.copy()
    changed[0, 2] = rng.integers(0, V, size=(2, 7), dtype=np.uint8)  # probe 2's batch only
    L1, c1 = oracle_mod.spsa_losses(theta, E, H, 1e-2, 1, 1, changed, n_pert=n,
                                    batch_per_probe=True)
    np.testing.assert_array_equal(L0[0, :2], L1[0, :2])
    assert np.all(L0[0, 2] != L1[0, 2])
    # and each probe sees exactly its batch: the shared-batch run on batch i
    for i in range(n):
        Li, _ = oracle_mod.spsa_losses(theta, E, H, 1e-2, 1, 1, per[:, i], probes=[i])
        np.testing.assert_array_equal(Li[0, 0], L0[0, i])


def test_summed_loss_single_expert_is_local(oracle_mod):
    E, H = 2, 3
    theta, bx = _micro(E, H, N=1, seed=6)
    a = oracle_mod.spsa_losses(theta, E, H, 1e-3, 3, 2, bx, n_pert=5)
    b = oracle_mod.spsa_losses(theta, E, H, 1e-3, 3, 2, bx, n_pert=5, summed_loss=True)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_allclose(a[1], b[1], rtol=1e-12)


def test_summed_loss_coefficient_limit(oracle_mod):
    # (sum_e L+ - sum_e L-) / (2 eps) = sum_e g_e . z_{e,i} + O(eps^2)
    E, H, N = 2, 2, 3
    theta, bx = _micro(E, H, N=N, seed=8, std=0.6)
    th = theta.astype(np.float64)
    P = th.shape[1]
    want = 0.0
    for e in range(N):
        _, g = oracle_mod.bptt_grad(th[e], E, H, bx[e])
        want += g @ oracle_mod.probe(4, 9, e, 0, 0, P).astype(np.float64)
    errs = []
    for eps in (1e-2, 5e-3, 2.5e-3):
        _, c = oracle_mod.spsa_losses(th, E, H, eps, 4, 9, bx, probes=[0], summed_loss=True)
        assert np.all(c == c[0, 0])  # the same coefficient for every expert
        errs.append(abs(c[0, 0] - want))
    slopes = np.diff(np.log(errs)) / np.diff(np.log([1e-2, 5e-3, 2.5e-3]))
    assert np.all(np.abs(slopes - 2.0) < 0.25), (errs, slopes)


def test_summed_loss_variance_law(oracle_mod):
    E, H, N, n = 1, 1, 2, 64
    theta, bx = _micro(E, H, N=N, B=2, T=5, seed=13, std=0.6)
    th = theta.astype(np.float64)
    P = th.shape[1]
    g = np.stack([oracle_mod.bptt_grad(th[e], E, H, bx[e])[1] for e in range(N)])
    reps = 24
    r_local, r_sum = [], []
    for r in range(reps):
        for summed, acc in ((False, r_local), (True, r_sum)):
            _, c = oracle_mod.spsa_losses(th, E, H, 1e-3, 17, r, bx, n_pert=n, n_threads=1,
                                          summed_loss=summed)
            gh = (th - oracle_mod.spsa_update(th, E, H, 1.0, 17, r, c))  # lr = 1
            acc.append(np.sum((gh - g) ** 2, axis=1) / np.sum(g ** 2, axis=1))
    r_local, r_sum = np.mean(r_local, axis=0), np.mean(r_sum, axis=0)
    for e in range(N):
        R = np.sum(g ** 2) - np.sum(g[e] ** 2)
        pred_sum = ((P - 1) + P * R / np.sum(g[e] ** 2)) / n
        assert r_local[e] == pytest.approx((P - 1) / n, rel=0.2)
        assert r_sum[e] == pytest.approx(pred_sum, rel=0.2), (e, r_sum[e], pred_sum)
