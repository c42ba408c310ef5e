"""The estimator's statistics on the CUDA path (GPU).

Prop. 1 and Eq. main-variance (Sec. "Gradient variance"), the perturbation
average of Eq. perturbation-average and the sparse-probe prediction of
App. G.1, measured from the coefficients the GPU computes at the tiny
workload (1 expert, E=32, H=64, 8 probes, 4 sequences x 64 bytes) over many
independent probe draws, against the exact gradient of the oracle's fp64
BPTT:
 - unbiasedness: E[g_hat . g] / |g|^2 = 1 within four standard errors
   (one step's value has variance about 2/n, from E[(g.z)^4] = 3|g|^4 - 2 sum g^4);
 - the variance law: E|g_hat - g|^2 / |g|^2 = (P - 1)/n within 12%;
 - sparse probes (density 1/2): the single-probe estimates c_r z_r have mean
   g/2 and trace covariance sum_j q_j (1 + s - 2 q_j) g_j^2 = (P / 4) |g|^2,
   and for the expert body, whose gains are always active, the same
   prediction with q = 1 on the gains.
g_hat is the oracle's update applied to the GPU's coefficients (lr = 1),
so the probe vectors come from the oracle's own Philox.
"""
import numpy as np
import pytest
import torch

from gpu_common import api
from paper_2609_37899_gb300 import inputs
from test_oracle_sparse_variance import check, predicted_trace, streamed_trace

pytestmark = pytest.mark.gpu


def _tiny():
    c = inputs.CONFIGS["tiny"]
    return c, inputs.config_params("tiny").astype(np.float64), inputs.config_batch("tiny")


def _gpu_coefs(theta, bx, E, H, n, eps, seed, steps, kind):
    a = api()
    N = theta.shape[0]
    B, T = bx.shape[1], bx.shape[2] - 1
    params = torch.from_numpy(theta.astype(np.float32)).cuda()
    dbx = torch.from_numpy(bx).cuda()
    ws = a.alloc_workspace(E, H, N, n, B, T)
    losses = torch.zeros(N, n, 2, device="cuda")
    out = []
    for st in steps:
        coef = torch.zeros(N, n, device="cuda")
        a.spsa_estimate(params, dbx, E, H, n, kind, eps, seed, st, losses, coef, ws)
        out.append(coef)
    assert a.get_status() == 0
    return [c.cpu().numpy().astype(np.float64) for c in out]


def test_dense_estimator_unbiased_and_variance_law(oracle_mod):
    c, theta, bx = _tiny()
    E, H, n = c["E"], c["H"], c["n_pert"]
    th32 = theta.astype(np.float32).astype(np.float64)
    _, g = oracle_mod.bptt_grad(th32[0], E, H, bx[0])
    P = g.size
    steps = range(256)
    coefs = _gpu_coefs(th32, bx, E, H, n, c["eps"], 17, steps, "dense")
    dots, rels = [], []
    for st, cf in zip(steps, coefs):
        gh = (th32 - oracle_mod.spsa_update(th32, E, H, 1.0, 17, st, cf))[0]
        dots.append(gh @ g / (g @ g))
        rels.append(np.sum((gh - g) ** 2) / np.sum(g ** 2))
    dots = np.asarray(dots)
    se = np.sqrt(2.0 / n / len(steps))
    assert abs(dots.mean() - 1.0) < 4 * se, (dots.mean(), se)
    assert np.mean(rels) == pytest.approx((P - 1) / n, rel=0.12), (np.mean(rels), (P - 1) / n)


def test_sparse_probe_variance_prediction(oracle_mod):
    c, theta, bx = _tiny()
    E, H, n = c["E"], c["H"], c["n_pert"]
    th32 = theta.astype(np.float32).astype(np.float64)
    _, g = oracle_mod.bptt_grad(th32[0], E, H, bx[0])
    P = g.size
    steps = range(256)
    coefs = _gpu_coefs(th32, bx, E, H, n, c["eps"], 23, steps, "sparse")
    cs = [cf[0, i] for cf in coefs for i in range(n)]
    probe = lambda r: oracle_mod.probe(23, steps[r // n], 0, r % n, 0, P,  # noqa: E731
                                       kind="sparse").astype(np.float64)
    m, se, mean = streamed_trace(cs, probe, P)
    pred = predicted_trace(g, np.full(P, 0.5))
    check(m, se, pred)
    slope = mean @ g / (g @ g)
    assert abs(slope - 0.5) < 4 * np.sqrt(pred / len(cs)) / np.linalg.norm(g)


def test_body_sparse_probe_variance_prediction(oracle_mod):
    # the expert body at the kernel's width d = 32: gains q = 1, weights 1/2
    from test_oracle_body import _setup, _torch_body_grad
    a = api()
    d, D, n, B, T = 32, 2, 64, 4, 12
    theta, head, bx = _setup(d, D, B=B, T=T, seed=29, wstd=0.05)
    th = theta.astype(np.float64)
    _, g = _torch_body_grad(th[0], d, D, head, bx[0])
    P = g.size
    g0 = inputs.body_offsets(d, D)["gains"]
    q = np.where(np.arange(P) < g0, 0.5, 1.0)
    params = torch.from_numpy(theta).cuda()
    dhead = torch.from_numpy(head).cuda()
    dbx = torch.from_numpy(bx).cuda()
    ws = a.body_alloc_workspace(d, D, 1, n, B, T)
    losses = torch.zeros(1, n, 2, device="cuda")
    steps = range(48)
    cs = []
    for st in steps:
        coef = torch.zeros(1, n, device="cuda")
        a.body_spsa_estimate(params, dhead, dbx, d, D, n, "sparse", 1e-3, 31, st, losses, coef,
                             ws)
        cs.extend(coef.cpu().numpy().astype(np.float64)[0].tolist())
    assert a.get_status() == 0
    probe = lambda r: oracle_mod.body_probe(31, steps[r // n], 0, r % n, d, D, 0, P,  # noqa: E731
                                            kind="sparse").astype(np.float64)
    m, se, _ = streamed_trace(cs, probe, P)
    pred = predicted_trace(g, q)
    check(m, se, pred)
