"""Parity of the paper's expert body on the GPU (Sec. "Model size", App. E).

Checked against the fp64 oracle on the same seeded inputs, through the C ABI:
- the body probe stream (both kinds, windows across the first gain): bit-exact;
- L+, L- and the coefficients: one and several 16-sequence chunks, ragged
  batches, D = 1 and D = 2, dense and sparse probes;
- the SPSA step's theta': against the oracle's own step, and against the
  oracle update of the GPU's coefficients;
- the Adam update given coefficients;
- eps = 0: L+ == L- == the eval loss, bitwise;
- the full workloads (256 experts; B = 16, T = 512 and B = 64, T = 1024) at
  sampled pairs, in the launch configuration the benchmark times.
"""
import numpy as np
import pytest
import torch

from gpu_common import (TOL_THETA, TOL_THETA_GIVEN_COEF, api, assert_coefs, assert_losses,
                        rel_l2, report)
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

V = 256


def _inputs(N, B, T, D=2, seed=0, d=32):
    theta = inputs.init_body(N, d, D, seed)
    g0 = inputs.body_offsets(d, D)["gains"]
    rng = np.random.default_rng(seed + 100)
    theta[:, g0:] = (1.0 + 0.2 * rng.standard_normal((N, theta.shape[1] - g0))).astype(np.float32)
    head = inputs.init_head(d, seed + 1)
    bx = inputs.expert_batch(N, B, T, 2, seed, 0)
    return theta, head, bx


def _estimate(theta, head, bx, D, n, kind, eps, seed, step, d=32):
    a = api()
    N, B, T1 = bx.shape
    params = torch.from_numpy(theta).cuda()
    before = params.clone()
    hd = torch.from_numpy(head).cuda()
    dbx = torch.from_numpy(np.ascontiguousarray(bx)).cuda()
    ws = a.body_alloc_workspace(d, D, N, n, B, T1 - 1)
    losses = torch.full((N, n, 2), float("nan"), device="cuda")
    coef = torch.full((N, n), float("nan"), device="cuda")
    a.body_spsa_estimate(params, hd, dbx, d, D, n, kind, float(eps), seed, step, losses, coef, ws)
    assert a.get_status() == 0
    assert torch.equal(params, before)
    return losses.cpu().numpy(), coef.cpu().numpy()


@pytest.mark.parametrize("kind", ["sparse", "dense"])
@pytest.mark.parametrize("D", [2, 1])
@pytest.mark.parametrize("seed,step,e,i,p0,count", [
    (0, 0, 0, 0, 0, 32928), (7, 3, 5, 63, 16000, 900), (2**40 + 3, 2**33 + 1, 255, 11, 32700, 228),
    (1, 2, 1, 1, 16470, 10),
])
def test_body_probe_bit_exact(oracle_mod, kind, D, seed, step, e, i, p0, count):
    P = inputs.body_param_count(32, D)
    count = min(count, P - p0) if p0 < P else count
    got = api().debug_body_probe(seed, step, e, i, 32, D, kind, p0, count).cpu().numpy()
    want = oracle_mod.body_probe(seed, step, e, i, 32, D, p0, count, kind=kind)
    assert (got == want).all()


@pytest.mark.parametrize("kind", ["sparse", "dense"])
@pytest.mark.parametrize("N,n,B,T,D", [
    (2, 4, 3, 20, 2),    # one chunk, ragged rows
    (1, 3, 19, 9, 2),    # two chunks, the second ragged
    (2, 2, 16, 6, 1),    # one full chunk, one block
    (1, 1, 1, 1, 2),     # one sequence of one target, one probe
    (1, 2, 17, 1, 1),    # a second chunk of one sequence, T = 1
])
def test_body_estimate_matches_oracle(oracle_mod, kind, N, n, B, T, D):
    theta, head, bx = _inputs(N, B, T, D, seed=N * 10 + B)
    L, coef = _estimate(theta, head, bx, D, n, kind, 1e-3, 5, 2)
    Lo, co = oracle_mod.body_spsa_losses(theta, 32, D, head, np.float32(1e-3), 5, 2, bx,
                                         n_pert=n, kind=kind)
    assert_losses(L, Lo)
    assert_coefs(coef, co)


def test_body_eps_zero_is_eval_bitwise(oracle_mod):
    a = api()
    N, n, B, T, D = 3, 4, 18, 11, 2
    theta, head, bx = _inputs(N, B, T, D, seed=4)
    L, coef = _estimate(theta, head, bx, D, n, "sparse", 0.0, 1, 1)
    assert np.all(coef == 0)
    assert np.array_equal(L[..., 0], L[..., 1])
    ws = a.body_alloc_workspace(32, D, N, n, B, T)
    ev = a.body_eval_loss(torch.from_numpy(theta).cuda(), torch.from_numpy(head).cuda(),
                          torch.from_numpy(bx).cuda(), 32, D, ws).cpu().numpy()
    assert a.get_status() == 0
    assert np.array_equal(np.repeat(ev[:, None], n, axis=1), L[..., 0])
    for e in range(N):
        assert abs(ev[e] - oracle_mod.body_loss(theta[e], 32, D, head, bx[e])) <= 2e-4


@pytest.mark.parametrize("kind", ["sparse", "dense"])
def test_body_step_matches_oracle(oracle_mod, kind):
    a = api()
    N, n, B, T, D = 2, 8, 5, 16, 2
    lr, eps = 1e-3, 1e-3
    theta, head, bx = _inputs(N, B, T, D, seed=9)
    params = torch.from_numpy(theta).cuda()
    ws = a.body_alloc_workspace(32, D, N, n, B, T)
    losses = torch.empty(N, n, 2, device="cuda")
    coef = torch.empty(N, n, device="cuda")
    a.body_spsa_step(params, torch.from_numpy(head).cuda(), torch.from_numpy(bx).cuda(), 32, D,
                     n, kind, eps, lr, 3, 7, losses, coef, ws)
    assert a.get_status() == 0
    got = params.cpu().numpy()
    c = coef.cpu().numpy()
    Lo, co = oracle_mod.body_spsa_losses(theta, 32, D, head, np.float32(eps), 3, 7, bx, n_pert=n,
                                         kind=kind)
    assert_losses(losses.cpu().numpy(), Lo)
    assert_coefs(c, co)
    want = oracle_mod.body_spsa_update(theta, 32, D, np.float32(lr), 3, 7, co, kind=kind)
    given = oracle_mod.body_spsa_update(theta, 32, D, np.float32(lr), 3, 7, c.astype(np.float64),
                                        kind=kind)
    err, err_given = rel_l2(got, want), rel_l2(got, given)
    report("body_theta_rel_l2", err)
    report("body_theta_given_coef_rel_l2", err_given)
    assert err <= TOL_THETA and err_given <= TOL_THETA_GIVEN_COEF


def test_body_adam_matches_oracle(oracle_mod):
    a = api()
    N, n, A, t, D = 3, 6, 2, 4, 2
    rng = np.random.default_rng(3)
    P = inputs.body_param_count(32, D)
    theta = (rng.standard_normal((N, P)) * 0.1).astype(np.float32)
    m = (rng.standard_normal((N, P)) * 1e-3).astype(np.float32)
    v = (rng.random((N, P)) * 1e-4 + 1e-6).astype(np.float32)
    coef = rng.standard_normal((A, N, n)).astype(np.float32)
    steps = [11, 2**35 + 3]
    args = (1e-3, 0.9, 0.999, 1e-8, 1e-4)
    dp, dm, dv = (torch.from_numpy(x).cuda() for x in (theta, m, v))
    a.body_adam_update(dp, dm, dv, 32, D, "sparse", 5, steps, torch.from_numpy(coef).cuda(),
                       *args, t)
    assert a.get_status() == 0
    to, mo, vo = oracle_mod.body_adam_update(theta, m, v, 32, D, 5, steps, coef.astype(np.float64),
                                             *(np.float32(x) for x in args), t, kind="sparse")
    gm, gv, gt = dm.cpu().numpy(), dv.cpu().numpy(), dp.cpu().numpy()
    assert np.abs(gm - mo).max() / np.abs(mo).max() <= 1e-5
    assert np.abs(gv - vo).max() / np.abs(vo).max() <= 1e-5
    step = np.abs(to - theta)
    assert np.all(np.abs(gt - to) <= 1e-4 * step + 3e-8)


@pytest.mark.parametrize("name,sample", [
    ("body_n256", {0: [0, 63], 255: [17], 77: [5]}),
    ("body_n256_paper", {3: [0], 200: [63]}),
])
def test_body_full_workload_sampled(oracle_mod, name, sample):
    c = inputs.BODY_CONFIGS[name]
    N, n, B, T, D = c["n_experts"], c["n_pert"], c["batch"], c["seq_len"], c["D"]
    theta = inputs.body_config_params(name)
    head = inputs.init_head(32, 0)
    bx = inputs.body_config_batch(name)
    L, coef = _estimate(theta, head, bx, D, n, "sparse", c["eps"], 0, 1)
    assert np.isfinite(L).all() and np.isfinite(coef).all()
    for e, probes in sample.items():
        Lo, co = oracle_mod.body_spsa_losses(theta[e:e + 1], 32, D, head, np.float32(c["eps"]), 0,
                                             1, bx[e:e + 1], probes=probes, first_expert=e,
                                             kind="sparse")
        assert_losses(L[e, probes], Lo[0])
        # coefficients of a few probes: each within 1e-2 of the largest
        d = np.abs(coef[e, probes] - co[0])
        report("body_full_coef_rel", float(d.max() / np.abs(co[0]).max()))
        assert np.all(d <= 1e-2 * np.abs(co[0]).max())
