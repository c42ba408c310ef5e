"""Pins of the oracle's two-block expert body (Sec. "Model size", App. E).
CPU only.

Independent references:
- The parameter count is the paper's formula M_body = 32 d^2 + 5 d at D = 2,
  its printed 32.9k at d = 32, and its 8.44M ensemble at N = 256.
- The forward is checked against a float64 torch model built from library
  modules, run layer by layer over the whole sequence rather than timestep
  by timestep: torch.nn.LSTM (bias-free), F.layer_norm, F.gelu and
  F.cross_entropy.
- Closed forms: zero weights make every block the identity, which leaves
  the final norm and the tied decode of the embedded byte.  A zero final
  gain gives ln 256.
- The eps -> 0 limit of the coefficient is compared with torch autograd's
  directional derivative (slope 2).
- The probe law uses the independent Philox (tests/philox_ref.py): gains
  take the dense sign, every other coordinate the sparse probe.  The
  estimator's mean is q_j g_j with q = 1 on gains and 1/2 elsewhere (App. E).
- The dense estimator's error obeys the variance law (P - 1) / n of Prop. 1.
- Also checked: eps = 0, experts batched versus alone, and the update's
  closed forms.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import philox_ref
from paper_2609_37899_gb300 import inputs

V = 256


def _torch_body(th, d, D, head, bytes_):
    """Per-token NLL [B, T] of the body from torch library modules (fp64).
    th is a flat torch tensor (autograd flows into it).  Each block runs over
    the whole sequence at once: torch.nn.LSTM (bias-free, gates i, f, g, o)
    on the normalised stream, then the MLP."""
    o = inputs.body_offsets(d, D)
    E = torch.as_tensor(np.asarray(head, dtype=np.float64))
    bx = torch.as_tensor(np.asarray(bytes_, dtype=np.int64))
    x = E[bx[:, :-1]]  # [B, T, d]
    lstm = torch.nn.LSTM(d, d, bias=False, batch_first=True, dtype=torch.float64)
    for k in range(D):
        w = {"weight_ih_l0": th[o[f"w_ih{k}"]:o[f"w_hh{k}"]].view(4 * d, d),
             "weight_hh_l0": th[o[f"w_hh{k}"]:o[f"w1{k}"]].view(4 * d, d)}
        ga = th[o[f"ga{k}"]:o[f"ga{k}"] + d]
        gb = th[o[f"gb{k}"]:o[f"gb{k}"] + d]
        h, _ = torch.func.functional_call(
            lstm, w, (F.layer_norm(x, (d,), weight=ga, bias=None, eps=1e-5),))
        x = x + h
        w1 = th[o[f"w1{k}"]:o[f"w2{k}"]].view(4 * d, d)
        w2 = th[o[f"w2{k}"]:o[f"w2{k}"] + 4 * d * d].view(d, 4 * d)
        x = x + F.linear(F.gelu(F.linear(F.layer_norm(x, (d,), weight=gb, bias=None, eps=1e-5),
                                         w1)), w2)
    y = F.layer_norm(x, (d,), weight=th[o["gf"]:o["end"]], bias=None, eps=1e-5)
    logits = y @ E.T
    return F.cross_entropy(logits.reshape(-1, V), bx[:, 1:].reshape(-1),
                           reduction="none").view(bx.shape[0], -1)


def _torch_body_nll(theta, d, D, head, bytes_):
    with torch.no_grad():
        return _torch_body(torch.as_tensor(np.asarray(theta, dtype=np.float64)), d, D, head,
                           bytes_)


def _torch_body_grad(theta, d, D, head, bytes_):
    th = torch.tensor(np.asarray(theta, dtype=np.float64), requires_grad=True)
    loss = _torch_body(th, d, D, head, bytes_).mean()
    loss.backward()
    return loss.item(), th.grad.numpy()


def _setup(d=8, D=2, N=1, B=3, T=7, seed=0, wstd=None):
    rng = np.random.default_rng(seed)
    theta = inputs.init_body(N, d, D, seed)
    if wstd is not None:
        g0 = inputs.body_offsets(d, D)["gains"]
        theta[:, :g0] = rng.standard_normal((N, g0)) * wstd
    # gains away from 1 so that a swapped gain shows
    g0 = inputs.body_offsets(d, D)["gains"]
    theta[:, g0:] = 1.0 + 0.3 * rng.standard_normal((N, theta.shape[1] - g0))
    head = inputs.init_head(d, seed + 1)
    bx = rng.integers(0, V, size=(N, B, T + 1), dtype=np.uint8)
    return theta.astype(np.float32), head, bx


def test_param_count_matches_paper(oracle_mod):
    for d in (8, 32, 48):
        assert oracle_mod.body_param_count(d, 2) == 32 * d * d + 5 * d == inputs.body_param_count(d)
        assert oracle_mod.body_param_count(d, 3) == 16 * 3 * d * d + 7 * d
    assert oracle_mod.body_param_count(32, 2) == 32928           # "32.9k"
    assert round((V * 32 + 256 * 32928) / 1e6, 2) == 8.44        # M_head + N M_body
    assert oracle_mod.body_gain_offset(32, 2) == 32768


@pytest.mark.parametrize("d,D,B,T", [(8, 2, 3, 9), (32, 2, 2, 17), (4, 1, 2, 5), (6, 3, 2, 6)])
def test_body_loss_matches_torch_modules(oracle_mod, d, D, B, T):
    theta, head, bx = _setup(d, D, B=B, T=T, seed=d + D, wstd=0.5)
    m, nll = oracle_mod.body_loss(theta[0], d, D, head, bx[0], per_token=True)
    want = _torch_body_nll(theta[0], d, D, head, bx[0]).detach().numpy()
    np.testing.assert_allclose(nll, want, rtol=0, atol=1e-12)
    assert abs(m - want.mean()) < 1e-12


def test_zero_weights_leave_the_decoded_embedding(oracle_mod):
    d, D = 8, 2
    theta, head, bx = _setup(d, D, B=2, T=6, seed=3)
    g0 = inputs.body_offsets(d, D)["gains"]
    theta[:, :g0] = 0.0  # every block is the identity
    gf = theta[0, inputs.body_offsets(d, D)["gf"]:].astype(np.float64)
    E = head.astype(np.float64)
    _, nll = oracle_mod.body_loss(theta[0], d, D, head, bx[0], per_token=True)
    for b in range(2):
        for t in range(6):
            x = E[bx[0, b, t]]
            y = (x - x.mean()) / np.sqrt(x.var() + 1e-5) * gf
            lg = E @ y
            want = np.log(np.sum(np.exp(lg - lg.max()))) + lg.max() - lg[bx[0, b, t + 1]]
            assert abs(nll[b, t] - want) < 1e-12
    theta[:, inputs.body_offsets(d, D)["gf"]:] = 0.0
    assert oracle_mod.body_loss(theta[0], d, D, head, bx[0]) == pytest.approx(math.log(256), abs=1e-14)


@pytest.mark.skipif(not philox_ref.available(), reason="torch Philox header not found")
def test_body_probe_law(oracle_mod):
    d, D = 8, 2
    P = inputs.body_param_count(d, D)
    g0 = inputs.body_offsets(d, D)["gains"]
    for (seed, step, e, i) in [(5, 2, 0, 3), (2**40 + 7, 2**33 + 1, 9, 61)]:
        z = oracle_mod.body_probe(seed, step, e, i, d, D, 0, P, kind="sparse")
        sign = philox_ref.rademacher(seed, step, e, i, 0, P)
        act = philox_ref.rademacher(seed, step, e, i | 0x80000000, 0, P)
        np.testing.assert_array_equal(z[g0:], sign[g0:])
        np.testing.assert_array_equal(z[:g0], np.where(act[:g0] == -1, sign[:g0], 0))
        np.testing.assert_array_equal(oracle_mod.body_probe(seed, step, e, i, d, D, 0, P, "dense"),
                                      sign)
        # any window of the stream is the same slice
        np.testing.assert_array_equal(
            oracle_mod.body_probe(seed, step, e, i, d, D, g0 - 5, 11, "sparse"), z[g0 - 5:g0 + 6])
    assert (z[:g0] == 0).mean() == pytest.approx(0.5, abs=0.05)


def test_eps_zero_and_separability(oracle_mod):
    d, D, N = 8, 2, 3
    theta, head, bx = _setup(d, D, N=N, B=2, T=5, seed=7, wstd=0.4)
    L, c = oracle_mod.body_spsa_losses(theta, d, D, head, 0.0, 1, 2, bx, n_pert=3)
    assert np.all(c == 0)
    for e in range(N):
        ref = oracle_mod.body_loss(theta[e], d, D, head, bx[e])
        assert np.all(L[e] == ref)
    La, ca = oracle_mod.body_spsa_losses(theta, d, D, head, 1e-3, 1, 2, bx, n_pert=3)
    for e in range(N):
        Le, ce = oracle_mod.body_spsa_losses(theta[e:e + 1], d, D, head, 1e-3, 1, 2, bx[e:e + 1],
                                             n_pert=3, first_expert=e)
        np.testing.assert_array_equal(Le[0], La[e])
        np.testing.assert_array_equal(ce[0], ca[e])


@pytest.mark.parametrize("kind", ["dense", "sparse"])
def test_coefficient_limit_is_autograd_directional_derivative(oracle_mod, kind):
    d, D = 6, 2
    theta, head, bx = _setup(d, D, B=2, T=6, seed=11, wstd=0.5)
    th = theta.astype(np.float64)
    _, g = _torch_body_grad(th[0], d, D, head, bx[0])
    P = th.shape[1]
    for i in (0, 5):
        z = oracle_mod.body_probe(3, 4, 0, i, d, D, 0, P, kind=kind).astype(np.float64)
        want = g @ z
        errs = []
        for eps in (1e-2, 5e-3, 2.5e-3):
            _, c = oracle_mod.body_spsa_losses(th, d, D, head, eps, 3, 4, bx, probes=[i], kind=kind)
            errs.append(abs(c[0, 0] - want))
        slopes = np.diff(np.log(errs)) / np.diff(np.log([1e-2, 5e-3, 2.5e-3]))
        assert np.all(np.abs(slopes - 2.0) < 0.3), (errs, slopes)
        _, c = oracle_mod.body_spsa_losses(th, d, D, head, 1e-4, 3, 4, bx, probes=[i], kind=kind)
        assert abs(c[0, 0] - want) < 1e-5 * max(1.0, abs(want))


def test_sparse_estimator_mean_q_times_gradient(oracle_mod):
    # E[coef z] = q g: q = 1 on the normalisation gains, 1/2 elsewhere (App. E).
    # The slope of the averaged estimate on each slice S is q up to noise of
    # standard deviation sqrt(q sum_j q_j g_j^2 / n_total) / |g_S| (from
    # E[(g.z)^2 z_p^2] = q_p sum_j q_j g_j^2 + O(g_p^2)).
    d, D = 4, 1
    theta, head, bx = _setup(d, D, B=2, T=5, seed=13, wstd=0.8)
    th = theta.astype(np.float64)
    _, g = _torch_body_grad(th[0], d, D, head, bx[0])
    g0 = inputs.body_offsets(d, D)["gains"]
    qv = np.where(np.arange(g.size) < g0, 0.5, 1.0)
    n, reps = 4096, 6
    gh = np.zeros_like(g)
    for r in range(reps):
        _, c = oracle_mod.body_spsa_losses(th, d, D, head, 1e-4, 21, r, bx, n_pert=n,
                                           kind="sparse", n_threads=1)
        gh += th[0] - oracle_mod.body_spsa_update(th, d, D, 1.0, 21, r, c, kind="sparse")[0]
    gh /= reps
    for sl, q in ((slice(0, g0), 0.5), (slice(g0, None), 1.0)):
        gs, hs = g[sl], gh[sl]
        sd = np.sqrt(q * np.sum(qv * g * g) / (n * reps)) / np.linalg.norm(gs)
        assert sd < 0.05
        slope = hs @ gs / (gs @ gs)
        assert abs(slope - q) < 5 * sd, (q, slope, sd)


def test_update_closed_forms(oracle_mod):
    d, D, N = 4, 2, 2
    theta, _, _ = _setup(d, D, N=N, seed=17)
    th = theta.astype(np.float64)
    P = th.shape[1]
    coef = np.array([[0.7], [-2.5]])
    out = oracle_mod.body_spsa_update(th, d, D, 0.01, 9, 3, coef, kind="sparse")
    for e in range(N):
        z = oracle_mod.body_probe(9, 3, e, 0, d, D, 0, P, kind="sparse")
        np.testing.assert_array_equal(out[e], th[e] - 0.01 * (coef[e, 0] * z))
    assert np.array_equal(oracle_mod.body_spsa_update(th, d, D, 0.0, 9, 3, coef), th)
    # Adam, first update: theta - lr g / (|g| + delta), g the estimate
    cf = np.array([[[0.7, -1.3], [0.25, 2.0]]])
    zeros = np.zeros_like(th)
    to, m, v = oracle_mod.body_adam_update(th, zeros, zeros, d, D, 4, [6], cf, 0.05, 0.9, 0.999,
                                           1e-8, 0.0, 1, kind="sparse")
    for e in range(N):
        z = np.stack([oracle_mod.body_probe(4, 6, e, i, d, D, 0, P) for i in range(2)])
        g = cf[0, e] @ z.astype(np.float64) / 2
        np.testing.assert_allclose(m[e], 0.1 * g, rtol=1e-14, atol=1e-300)
        np.testing.assert_allclose(to[e], th[e] - 0.05 * g / (np.abs(g) + 1e-8), atol=1e-12)
        # gains are always touched; the untouched weights keep their value
        g0 = inputs.body_offsets(d, D)["gains"]
        assert np.all(z[:, g0:] != 0)
        untouched = np.all(z == 0, axis=0)
        np.testing.assert_array_equal(to[e][untouched], th[e][untouched])


def test_dense_estimator_variance_law(oracle_mod):
    # Prop. 1 for the body: with dense probes, E|ghat - g|^2 / |g|^2 = (P - 1) / n
    # (one probe: E[(g.z)^2 |z|^2] = P |g|^2, so E|X - g|^2 = (P - 1) |g|^2)
    d, D = 4, 1
    theta, head, bx = _setup(d, D, B=2, T=5, seed=19, wstd=0.6)
    th = theta.astype(np.float64)
    _, g = _torch_body_grad(th[0], d, D, head, bx[0])
    P, n, reps = g.size, 64, 24
    rel = []
    for r in range(reps):
        _, c = oracle_mod.body_spsa_losses(th, d, D, head, 1e-4, 31, r, bx, n_pert=n,
                                           kind="dense", n_threads=1)
        gh = th[0] - oracle_mod.body_spsa_update(th, d, D, 1.0, 31, r, c, kind="dense")[0]
        rel.append(np.sum((gh - g) ** 2) / np.sum(g ** 2))
    assert np.mean(rel) == pytest.approx((P - 1) / n, rel=0.2), (np.mean(rel), (P - 1) / n)
