"""Parity of the paper's optimizer step on the GPU (App. E, Eq. localspsa).

The step is split into two parts, each compared with the fp64 oracle on the
same seeded inputs:
- soma_spsa_estimate, with sparse and dense probes. Checked: L+, L- and the
  coefficients (tiny, ragged and a batch of 70 in two chunks in full; SOMA N=2 at
  sampled probes).
- soma_adam_update, given coefficients. Checked: theta', m' and v' against
  the oracle's Adam update of the same coefficients.

The probe stream itself is compared bit-exactly.
"""
import numpy as np
import pytest
import torch

from gpu_common import api, assert_coefs, assert_losses, report
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

V = 256


@pytest.mark.parametrize("kind", ["sparse", "dense"])
@pytest.mark.parametrize("seed,step,e,i,p0,count", [
    (0, 0, 0, 0, 0, 4096), (3, 7, 1, 5, 3, 1000), (2**40 + 1, 2**32 + 9, 255, 12287, 8_299_000, 1160),
])
def test_probe_entries_bit_exact(oracle_mod, kind, seed, step, e, i, p0, count):
    got = api().debug_probe(seed, step, e, i, kind, p0, count).cpu().numpy()
    want = oracle_mod.probe(seed, step, e, i, p0, count, kind=kind)
    assert (got == want).all()


def _estimate(theta, bx, E, H, n, kind, eps, seed, step):
    a = api()
    N, B, T1 = bx.shape
    params = torch.from_numpy(np.ascontiguousarray(theta, dtype=np.float32)).cuda()
    before = params.clone()
    dev_bx = torch.from_numpy(np.ascontiguousarray(bx)).cuda()
    ws = a.alloc_workspace(E, H, N, n, B, T1 - 1)
    losses = torch.full((N, n, 2), float("nan"), device="cuda")
    coef = torch.full((N, n), float("nan"), device="cuda")
    a.spsa_estimate(params, dev_bx, E, H, n, kind, float(eps), seed, step, losses, coef, ws)
    assert a.get_status() == 0
    assert torch.equal(params, before)  # the estimate only reads theta
    return losses.cpu().numpy(), coef.cpu().numpy()


def _batch(N, B, T, seed):
    rng = np.random.default_rng(seed)
    return rng.integers(0, V, size=(N, B, T + 1), dtype=np.uint8)


@pytest.mark.parametrize("E,H,N,n,B,T", [
    (32, 64, 1, 8, 4, 64),     # the tiny workload (tensor path)
    (40, 72, 2, 5, 5, 9),      # ragged: every tile dimension padded
    (16, 32, 1, 3, 70, 4),     # B > 64: two tensor-core chunks (64 + 6)
])
def test_sparse_estimate_full(oracle_mod, E, H, N, n, B, T):
    theta = inputs.init_params(N, E, H, seed=21, std=0.1)
    bx = _batch(N, B, T, seed=E + H)
    L, coef = _estimate(theta, bx, E, H, n, "sparse", 1e-3, 5, 2)
    Lo, co = oracle_mod.spsa_losses(theta, E, H, np.float32(1e-3), 5, 2, bx, n_pert=n,
                                    kind="sparse")
    assert_losses(L, Lo)
    assert_coefs(coef, co)


def test_dense_estimate_equals_step():
    # the same forward as soma_spsa_step: identical losses and coefficients
    from gpu_common import run_step
    c = inputs.CONFIGS["tiny"]
    theta = inputs.config_params("tiny")
    bx = inputs.config_batch("tiny")
    L, coef = _estimate(theta, bx, c["E"], c["H"], c["n_pert"], "dense", c["eps"], 3, 4)
    g = run_step(theta, bx, c["E"], c["H"], c["n_pert"], c["eps"], c["lr"], 3, 4)
    np.testing.assert_array_equal(L, g["losses"])
    np.testing.assert_array_equal(coef, g["coef"])


def test_sparse_estimate_soma_n2_sampled(oracle_mod):
    c = inputs.CONFIGS["soma_n2"]
    E, H, n = c["E"], c["H"], c["n_pert"]
    theta = inputs.config_params("soma_n2")
    bx = inputs.config_batch("soma_n2")
    L, coef = _estimate(theta, bx, E, H, n, "sparse", c["eps"], 0, 1)
    assert np.isfinite(L).all()
    for e, probes in {0: [0, 63], 1: [17]}.items():
        Lo, co = oracle_mod.spsa_losses(theta[e:e + 1], E, H, np.float32(c["eps"]), 0, 1,
                                        bx[e:e + 1], probes=probes, first_expert=e, kind="sparse")
        assert_losses(L[e, probes], Lo[0])
        assert_coefs(coef[e, probes][None], co)


@pytest.mark.parametrize("kind", ["sparse", "dense"])
@pytest.mark.parametrize("E,H,N,n,A,t", [(32, 64, 2, 8, 2, 3), (24, 40, 3, 5, 1, 1),
                                         (64, 256, 1, 8, 2, 7)])
def test_adam_update_matches_oracle(oracle_mod, kind, E, H, N, n, A, t):
    a = api()
    rng = np.random.default_rng(E * H + A)
    P = inputs.param_count(E, H)
    theta = (rng.standard_normal((N, P)) * 0.05).astype(np.float32)
    m = (rng.standard_normal((N, P)) * 1e-3).astype(np.float32)
    # moments from earlier updates: v > 0 keeps the step smooth in g
    v = (rng.random((N, P)) * 1e-4 + 1e-6).astype(np.float32)
    coef = rng.standard_normal((A, N, n)).astype(np.float32)
    steps = [int(x) for x in rng.integers(0, 2**40, size=A)]
    lr, b1, b2, delta, wd = 1e-3, 0.9, 0.999, 1e-8, 1e-4
    dp, dm, dv = (torch.from_numpy(x).cuda() for x in (theta, m, v))
    a.adam_update(dp, dm, dv, E, H, kind, 77, steps, torch.from_numpy(coef).cuda(), lr, b1, b2,
                  delta, wd, t)
    assert a.get_status() == 0
    to, mo, vo = oracle_mod.adam_update(theta, m, v, E, H, 77, steps, coef.astype(np.float64),
                                        np.float32(lr), np.float32(b1), np.float32(b2),
                                        np.float32(delta), np.float32(wd), t, kind=kind)
    gm, gv, gt = dm.cpu().numpy(), dv.cpu().numpy(), dp.cpu().numpy()
    err_m = np.abs(gm - mo).max() / np.abs(mo).max()
    err_v = np.abs(gv - vo).max() / np.abs(vo).max()
    step = np.abs(to - theta)
    err_t = np.abs(gt - to).max() / step.max()
    report("adam_m_rel", err_m)
    report("adam_v_rel", err_v)
    report("adam_theta_rel_step", err_t)
    assert err_m <= 1e-5 and err_v <= 1e-5
    # fp32 rounding of theta (|theta| <= ~0.25: 1.5e-8) plus a relative 1e-4
    # of the step
    assert np.all(np.abs(gt - to) <= 1e-4 * step + 3e-8)


def test_adam_skips_expert_with_nonfinite_coefficient():
    a = api()
    E, H, N, n = 16, 32, 2, 4
    P = inputs.param_count(E, H)
    theta = torch.full((N, P), 0.5, device="cuda")
    m = torch.zeros_like(theta)
    v = torch.zeros_like(theta)
    coef = torch.ones(1, N, n, device="cuda")
    coef[0, 1, 2] = float("nan")
    a.adam_update(theta, m, v, E, H, "sparse", 1, [0], coef, 1e-2, 0.9, 0.999, 1e-8, 0.0, 1)
    assert a.get_status() == 0
    assert (theta[1] == 0.5).all() and not m[1].any() and not v[1].any()
    assert (theta[0] != 0.5).any()


def test_adam_step_through_the_experts_object(oracle_mod):
    # the public wrapper: A = 2 estimates, then one update; each part against
    # the oracle (estimate: coefficients; update: theta' given those)
    from paper_2609_37899_gb300.api import SomaExperts
    c = inputs.CONFIGS["tiny"]
    E, H, n = c["E"], c["H"], c["n_pert"]
    ex = SomaExperts(1, E, H, n, 4, 16)
    theta = inputs.init_params(1, E, H, seed=4, std=0.1)
    ex.params.copy_(torch.from_numpy(theta))
    batches = [torch.from_numpy(_batch(1, 4, 16, seed=s)).cuda() for s in (1, 2)]
    losses, coef = ex.adam_step(batches, 1e-3, 9, [10, 11], t=1, lr=1e-3)
    assert api().get_status() == 0
    coef = coef.cpu().numpy()
    for a, s in enumerate((10, 11)):
        _, co = oracle_mod.spsa_losses(theta, E, H, np.float32(1e-3), 9, s,
                                       batches[a].cpu().numpy(), n_pert=n, kind="sparse")
        assert_coefs(coef[a], co)
    zeros = np.zeros_like(theta, dtype=np.float64)
    to, mo, _ = oracle_mod.adam_update(theta, zeros, zeros, E, H, 9, [10, 11],
                                       coef.astype(np.float64), np.float32(1e-3), np.float32(0.9),
                                       np.float32(0.999), np.float32(1e-8), np.float32(1e-4), 1)
    np.testing.assert_allclose(ex.m.cpu().numpy(), mo, rtol=1e-5, atol=1e-9)
    # at t = 1 every touched coordinate moves by about lr: compare where the
    # estimate is well away from zero
    ok = np.abs(mo) > 1e-3 * np.abs(mo).max()
    got = ex.params.cpu().numpy()
    assert np.all(np.abs(got[ok] - to[ok]) <= 1e-6)
