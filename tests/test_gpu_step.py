"""Parity of the CUDA path with the fp64 oracle at small sizes (GPU).

Every test calls the C ABI through the ctypes binding; the oracle runs on
the same seeded inputs (tests/gpu_common.py states the tolerances)."""
import numpy as np
import pytest
import torch

from gpu_common import (TOL_THETA, TOL_THETA_GIVEN_COEF, api, assert_coefs, assert_losses,
                        rel_l2, report, run_eval, run_step)
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

V = 256


def test_philox_words_bit_exact(oracle_mod):
    a = api()
    rng = np.random.default_rng(0)
    for seed in [0, 1, 0xFFFFFFFFFFFFFFFF, int(rng.integers(0, 2**63))]:
        ctr = rng.integers(0, 2**32, size=(512, 4), dtype=np.uint64)
        ctr[0] = 0
        ctr[1] = 0xFFFFFFFF
        dev = torch.from_numpy(ctr.astype(np.uint32).view(np.int32)).cuda()
        out = a.debug_philox(seed, dev).cpu().numpy().view(np.uint32)
        key = (seed & 0xFFFFFFFF, seed >> 32)
        for c, o in zip(ctr, out):
            assert (oracle_mod.philox4x32_10(c, key) == o).all()


@pytest.mark.parametrize("seed,step,e,i,p0,count", [
    (0, 0, 0, 0, 0, 4096), (0, 0, 0, 0, 3, 1000), (5, 2**32 + 3, 7, 63, 96, 4100),
    (2**40 + 1, 9, 255, 1023, 8_299_000, 1160), (0, 1, 1, 1, 127, 1),
])
def test_probe_entries_bit_exact(oracle_mod, seed, step, e, i, p0, count):
    got = api().debug_rademacher(seed, step, e, i, p0, count).cpu().numpy()
    want = oracle_mod.rademacher(seed, step, e, i, p0, count)
    assert (got == want).all()


def _full_parity(oracle_mod, theta, bx, E, H, n, eps, lr, seed, step, tol_theta=TOL_THETA):
    g = run_step(theta, bx, E, H, n, eps, lr, seed, step)
    assert g["status"] == 0
    L, coef, new = oracle_mod.spsa_step(theta, E, H, n, np.float32(eps), np.float32(lr), seed,
                                        step, bx)
    assert_losses(g["losses"], L)
    assert_coefs(g["coef"], coef)
    rel = rel_l2(g["theta"], new)
    report(f"theta_rel_l2_eps{eps:g}", rel)
    assert rel <= tol_theta
    # the update kernel alone: the oracle's update of the GPU's coefficients
    new_g = oracle_mod.spsa_update(theta, E, H, np.float32(lr), seed, step,
                                   g["coef"].astype(np.float64))
    assert rel_l2(g["theta"], new_g) <= TOL_THETA_GIVEN_COEF
    return g, (L, coef, new)


def test_tiny_config_full_step(oracle_mod):
    c = inputs.CONFIGS["tiny"]
    theta = inputs.config_params("tiny")
    bx = inputs.config_batch("tiny")
    _full_parity(oracle_mod, theta, bx, c["E"], c["H"], c["n_pert"], c["eps"], c["lr"], 0, 0)


@pytest.mark.parametrize("N,E,H,B,T,n", [
    (3, 5, 37, 3, 7, 3),     # nothing a multiple of a tile
    (2, 33, 65, 35, 40, 2),  # one past every tile edge
    (1, 1, 1, 1, 1, 1),      # degenerate sizes
])
def test_ragged_shapes_full_step(oracle_mod, N, E, H, B, T, n):
    theta = inputs.init_params(N, E, H, seed=N + H, std=0.3)
    bx = inputs.expert_batch(N, B, T, 1, seed=4, step=0)
    _full_parity(oracle_mod, theta, bx, E, H, n, 1e-3, 1e-2, 77, 5)


# The difference operand is stored as dhat = (v+ - v-) / (2 eps), an O(1)
# quantity, so the fp16 rounding of the difference stays relative at any eps.
# The sweep covers the resident kernel (tiny, H <= 64), the persistent kernel
# with one probe per operand group (B = 35) and with two (H = 96, B = 8, an
# odd probe count so the last group holds one probe).
#
# Below eps = 1e-3 the fp32 pre-activations a+- = C +- eps D carry an
# absolute rounding of about 2^-24 |C| against a signal eps |D|, so the
# coefficients, and with them theta' - theta, lose accuracy in proportion to
# 1 / eps (at 1e-4 the coefficient error is about 2e-3, ten times that at
# 1e-3).  The theta' bound of the step (1e-5, stated for eps = 1e-3) is
# scaled by the same factor there.
EPS_SHAPES = {
    "tiny": None,
    "ragged_p1": (2, 33, 65, 35, 40, 2),
    "persistent_p2": (2, 16, 96, 8, 12, 5),
}


@pytest.mark.parametrize("eps", [1e-2, 1e-3, 1e-4])
@pytest.mark.parametrize("shape", list(EPS_SHAPES))
def test_eps_sweep_full_step(oracle_mod, shape, eps):
    if shape == "tiny":
        c = inputs.CONFIGS["tiny"]
        theta = inputs.config_params("tiny")
        bx = inputs.config_batch("tiny")
        E, H, n, lr = c["E"], c["H"], c["n_pert"], c["lr"]
    else:
        N, E, H, B, T, n = EPS_SHAPES[shape]
        theta = inputs.init_params(N, E, H, seed=N + H, std=None)
        bx = inputs.expert_batch(N, B, T, 2, seed=4, step=0)
        lr = 1e-2
    _full_parity(oracle_mod, theta, bx, E, H, n, eps, lr, 11, 3,
                 tol_theta=TOL_THETA * max(1.0, 1e-3 / eps))


def test_eps_zero_is_the_unperturbed_loss():
    E, H, N, n = 16, 40, 2, 4
    theta = inputs.init_params(N, E, H, seed=1, std=0.2)
    bx = inputs.expert_batch(N, 5, 20, 1, seed=2, step=0)
    g = run_step(theta, bx, E, H, n, 0.0, 1e-2, 3, 4)
    assert g["status"] == 0
    assert (g["losses"][..., 0] == g["losses"][..., 1]).all()
    assert (g["coef"] == 0).all()
    assert (g["theta"] == theta).all()
    ev = run_eval(theta, bx, E, H)
    assert (g["losses"][..., 0] == ev[:, None]).all()


def test_eval_loss_matches_oracle(oracle_mod):
    E, H, N = 24, 72, 3
    theta = inputs.init_params(N, E, H, seed=5, std=0.15)
    bx = inputs.expert_batch(N, 6, 33, 2, seed=6, step=0)
    ev = run_eval(theta, bx, E, H)
    for e in range(N):
        assert abs(ev[e] - oracle_mod.loss(theta[e], E, H, bx[e])) <= 2e-4


@pytest.mark.parametrize("B", [1, 130, 257])
def test_eval_loss_unperturbed_layout_matches_oracle(oracle_mod, B):
    # H > 64: the tensor-core sweep in the unperturbed layout, one sweep for
    # the whole batch (groups of 128 sequences, the last one ragged)
    E, H, N = 16, 96, 2
    theta = inputs.init_params(N, E, H, seed=B, std=None)
    bx = inputs.expert_batch(N, B, 9, 2, seed=7, step=0)
    ev = run_eval(theta, bx, E, H)
    for e in range(N):
        assert abs(ev[e] - oracle_mod.loss(theta[e], E, H, bx[e])) <= 2e-4


def test_lr_zero_leaves_params_and_keeps_losses():
    E, H, N, n = 16, 40, 2, 4
    theta = inputs.init_params(N, E, H, seed=1, std=0.2)
    bx = inputs.expert_batch(N, 5, 20, 1, seed=2, step=0)
    g0 = run_step(theta, bx, E, H, n, 1e-3, 0.0, 3, 4)
    g1 = run_step(theta, bx, E, H, n, 1e-3, 1e-2, 3, 4)
    assert (g0["theta"] == theta).all()
    assert (g0["losses"] == g1["losses"]).all() and (g0["coef"] == g1["coef"]).all()
    assert (g1["theta"] != theta).any()


def test_update_kernel_alone(oracle_mod):
    a = api()
    E, H, N, n = 8, 24, 3, 37
    theta = inputs.init_params(N, E, H, seed=9, std=0.1)
    coef = np.random.default_rng(1).standard_normal((N, n)).astype(np.float32)
    params = torch.from_numpy(theta).cuda()
    a.spsa_update(params, E, H, 0.05, 123, 456, torch.from_numpy(coef).cuda())
    got = params.cpu().numpy()
    want = oracle_mod.spsa_update(theta, E, H, np.float32(0.05), 123, 456, coef.astype(np.float64))
    assert rel_l2(got, want) <= 1e-6
    # n = 1 closed form with the oracle's probe entries: theta - lr c z
    params = torch.from_numpy(theta).cuda()
    a.spsa_update(params, E, H, 0.5, 1, 2, torch.from_numpy(coef[:, :1].copy()).cuda())
    got = params.cpu().numpy()
    P = theta.shape[1]
    for e in range(N):
        z = oracle_mod.rademacher(1, 2, e, 0, 0, P).astype(np.float64)
        np.testing.assert_allclose(got[e], theta[e] - np.float32(0.5) * coef[e, 0] * z,
                                   rtol=0, atol=1e-6)


def test_experts_are_separable():
    E, H, N, n = 12, 30, 3, 3
    theta = inputs.init_params(N, E, H, seed=11, std=0.2)
    bx = inputs.expert_batch(N, 4, 16, 1, seed=12, step=0)
    g = run_step(theta, bx, E, H, n, 1e-3, 1e-2, 5, 6)
    theta2 = theta.copy()
    theta2[1] *= 1.5
    bx2 = bx.copy()
    bx2[2] = bx[2][:, ::-1]
    g2 = run_step(theta2, bx2, E, H, n, 1e-3, 1e-2, 5, 6)
    for k in ("losses", "coef", "theta"):
        assert (g2[k][0] == g[k][0]).all()
        assert (g2[k][1] != g[k][1]).any()


def test_deterministic_and_resumable():
    E, H, N, n = 12, 30, 2, 4
    theta = inputs.init_params(N, E, H, seed=13, std=0.2)
    b0 = inputs.expert_batch(N, 4, 16, 1, seed=14, step=0)
    b1 = inputs.expert_batch(N, 4, 16, 1, seed=14, step=1)
    a = api()
    params = torch.from_numpy(theta).cuda()
    ws = a.alloc_workspace(E, H, N, n, 4, 16)
    losses = torch.zeros(N, n, 2, device="cuda")
    a.spsa_step(params, torch.from_numpy(b0).cuda(), E, H, n, 1e-3, 1e-2, 7, 0, losses, None, ws)
    a.spsa_step(params, torch.from_numpy(b1).cuda(), E, H, n, 1e-3, 1e-2, 7, 1, losses, None, ws)
    straight = params.cpu().numpy()
    # checkpoint after the first step: theta plus (seed, step) is the whole state
    g = run_step(theta, b0, E, H, n, 1e-3, 1e-2, 7, 0)
    g2 = run_step(g["theta"], b1, E, H, n, 1e-3, 1e-2, 7, 1)
    assert (g2["theta"] == straight).all()


def test_nonfinite_loss_is_reported_and_skips_the_update():
    E, H, N, n = 8, 16, 2, 3
    theta = inputs.init_params(N, E, H, seed=15, std=0.2)
    theta[0, 2] = np.nan  # Emb[0][2] of expert 0
    bx = inputs.expert_batch(N, 3, 8, 1, seed=16, step=0)
    bx[0, :, :] = 0  # every input byte reads the NaN row
    g = run_step(theta, bx, E, H, n, 1e-3, 1e-2, 1, 1)
    assert g["status"] == 6
    np.testing.assert_array_equal(g["theta"][0], theta[0])
    assert np.isfinite(g["losses"][1]).all() and (g["theta"][1] != theta[1]).any()
    assert api().get_status() == 0  # read-and-clear


def test_init_experts():
    a = api()
    E, H, N = 64, 480, 2
    P = a.param_count(E, H)
    p = torch.empty(N, P, device="cuda")
    a.init_experts(p, E, H, seed=3, std=0.0)
    q = torch.empty(N, P, device="cuda")
    a.init_experts(q, E, H, seed=3, std=0.0)
    assert torch.equal(p, q)
    o = inputs.param_offsets(E, H)
    x = p.cpu().numpy().astype(np.float64)
    assert x[:, o["emb"]:o["w_ih"]].std() == pytest.approx(0.1, rel=0.02)
    assert x[:, o["w_ih"]:o["b"]].std() == pytest.approx(1 / np.sqrt(E + H), rel=0.02)
    assert (x[:, o["b"]:o["w_out"]] == 0).all() and (x[:, o["b_out"]:] == 0).all()
    assert x[:, o["w_out"]:o["b_out"]].std() == pytest.approx(1 / np.sqrt(H), rel=0.02)
    assert abs(x[:, o["w_hh"]:o["b"]].mean()) < 1e-3
    a.init_experts(q, E, H, seed=3, std=0.5)
    assert q.std().item() == pytest.approx(0.5, rel=0.02)


@pytest.mark.parametrize("B", [65, 130, 192])
def test_large_batch_runs_in_chunks(oracle_mod, B):
    # more than 64 sequences per expert: tensor-core sweeps over chunks of at
    # most 64 sequences (65 = 64 + 1, 130 = 64 + 64 + 2, 192 = 3 x 64), each
    # writing its part of the loss partials of the whole batch
    N, E, H, T, n = 2, 3, 70, 4, 3
    theta = inputs.init_params(N, E, H, seed=21, std=0.3)
    bx = inputs.expert_batch(N, B, T, 1, seed=22, step=0)
    _full_parity(oracle_mod, theta, bx, E, H, n, 1e-3, 1e-2, 3, 1)


@pytest.mark.parametrize("n", [160, 304])
def test_many_tasks_per_cta(oracle_mod, n):
    # more probe groups than SMs: every persistent CTA runs several gate and
    # head tasks (and each launch carries the embedding-operand blocks)
    N, E, H, B, T = 1, 64, 96, 8, 6
    theta = inputs.init_params(N, E, H, seed=n, std=None)
    bx = inputs.expert_batch(N, B, T, 2, seed=31, step=0)
    g = run_step(theta, bx, E, H, n, 1e-3, 1e-3, 4, 2)
    assert g["status"] == 0
    probes = [0, 1, 151, 152, 153, n - 2, n - 1]
    L, coef = oracle_mod.spsa_losses(theta, E, H, np.float32(1e-3), 4, 2, bx, probes=probes)
    assert_losses(g["losses"][:, probes], L)
    assert_coefs(g["coef"][:, probes], coef)
