"""Pins of the oracle's LSTM forward, loss and BPTT gradient (CPU only).

Independent references: torch.nn.LSTM + F.cross_entropy in float64, torch
autograd, closed forms, brute-force central differences."""
import math

import numpy as np
import pytest
import torch

from paper_2609_37899_gb300 import inputs

V = 256


def _torch_loss(theta, E, H, bytes_, per_token=False):
    """Mean next-byte CE with torch.nn.LSTM (float64), gates i,f,g,o."""
    o = inputs.param_offsets(E, H)
    th = torch.as_tensor(np.asarray(theta, dtype=np.float64))
    emb = th[o["emb"]:o["w_ih"]].view(V, E)
    lstm = torch.nn.LSTM(E, H, batch_first=True, dtype=torch.float64)
    with torch.no_grad():
        lstm.weight_ih_l0.copy_(th[o["w_ih"]:o["w_hh"]].view(4 * H, E))
        lstm.weight_hh_l0.copy_(th[o["w_hh"]:o["b"]].view(4 * H, H))
        lstm.bias_ih_l0.copy_(th[o["b"]:o["w_out"]])
        lstm.bias_hh_l0.zero_()
    w_out = th[o["w_out"]:o["b_out"]].view(V, H)
    b_out = th[o["b_out"]:o["end"]]
    bx = torch.as_tensor(np.asarray(bytes_, dtype=np.int64))
    x = emb[bx[:, :-1]]
    hs, _ = lstm(x)
    logits = hs @ w_out.T + b_out
    nll = torch.nn.functional.cross_entropy(logits.reshape(-1, V), bx[:, 1:].reshape(-1),
                                            reduction="none").view(bx.shape[0], -1)
    return (nll.mean().item(), nll.detach().numpy()) if per_token else nll.mean().item()


@pytest.mark.parametrize("E,H,B,T,std", [(5, 7, 3, 9, 0.3), (32, 64, 4, 64, 0.1), (3, 16, 2, 33, 1.0)])
def test_loss_matches_torch_lstm(oracle_mod, E, H, B, T, std):
    rng = np.random.default_rng(E * 100 + H)
    P = inputs.param_count(E, H)
    theta = rng.standard_normal(P) * std
    bx = rng.integers(0, V, size=(B, T + 1), dtype=np.uint8)
    m, nll = oracle_mod.loss(theta, E, H, bx, per_token=True)
    mt, nllt = _torch_loss(theta, E, H, bx, per_token=True)
    assert abs(m - mt) < 1e-12
    np.testing.assert_allclose(nll, nllt, rtol=0, atol=1e-11)


def test_zero_weights_give_log256(oracle_mod):
    E, H = 4, 6
    theta = np.zeros(inputs.param_count(E, H))
    bx = np.random.default_rng(0).integers(0, V, size=(3, 12), dtype=np.uint8)
    assert oracle_mod.loss(theta, E, H, bx) == pytest.approx(math.log(256.0), abs=1e-15)


def test_output_bias_closed_form_fixes_target_index(oracle_mod):
    # W_out = 0: every logit vector is b_out, so nll_t = lse(b_out) - b_out[y_{t+1}]
    # whatever the recurrence does.  Distinct biases expose a target off by one.
    E, H = 3, 5
    rng = np.random.default_rng(1)
    o = inputs.param_offsets(E, H)
    theta = rng.standard_normal(inputs.param_count(E, H)) * 0.5
    theta[o["w_out"]:o["b_out"]] = 0.0
    beta = rng.standard_normal(V)
    theta[o["b_out"]:o["end"]] = beta
    bx = rng.integers(0, V, size=(4, 10), dtype=np.uint8)
    lse = np.log(np.exp(beta - beta.max()).sum()) + beta.max()
    want = np.mean(lse - beta[bx[:, 1:]])
    assert oracle_mod.loss(theta, E, H, bx) == pytest.approx(want, abs=1e-13)


def test_state_resets_per_sequence(oracle_mod):
    E, H, T = 4, 8, 11
    rng = np.random.default_rng(2)
    theta = rng.standard_normal(inputs.param_count(E, H)) * 0.4
    bx = rng.integers(0, V, size=(5, T + 1), dtype=np.uint8)
    whole = oracle_mod.loss(theta, E, H, bx)
    singles = [oracle_mod.loss(theta, E, H, bx[b:b + 1]) for b in range(5)]
    assert whole == pytest.approx(np.mean(singles), abs=1e-14)


def test_one_step_hand_computed(oracle_mod):
    # E = H = 1, T = 1: write the cell out for one input byte.
    E, H = 1, 1
    o = inputs.param_offsets(E, H)
    theta = np.zeros(inputs.param_count(E, H))
    x_byte, y_byte = 7, 200
    theta[o["emb"] + x_byte] = 0.5                      # x = 0.5
    theta[o["w_ih"]:o["w_hh"]] = [1.0, -2.0, 3.0, 0.25]  # i, f, g, o rows
    theta[o["b"]:o["w_out"]] = [0.1, 0.2, -0.3, 0.4]
    theta[o["w_out"] + y_byte] = 2.0                    # logit_y = 2 h, other logits 0
    a = np.array([0.5 * 1.0 + 0.1, 0.5 * -2.0 + 0.2, 0.5 * 3.0 - 0.3, 0.5 * 0.25 + 0.4])
    sg = lambda u: 1.0 / (1.0 + math.exp(-u))
    c = sg(a[0]) * math.tanh(a[2])                      # f * c0 = 0
    h = sg(a[3]) * math.tanh(c)
    want = math.log(255.0 + math.exp(2.0 * h)) - 2.0 * h
    got = oracle_mod.loss(theta, E, H, np.array([[x_byte, y_byte]], dtype=np.uint8))
    assert got == pytest.approx(want, abs=1e-14)


def _torch_grad(theta, E, H, bytes_):
    o = inputs.param_offsets(E, H)
    th = torch.tensor(np.asarray(theta, dtype=np.float64), requires_grad=True)
    emb = th[o["emb"]:o["w_ih"]].view(V, E)
    w_ih = th[o["w_ih"]:o["w_hh"]].view(4 * H, E)
    w_hh = th[o["w_hh"]:o["b"]].view(4 * H, H)
    b = th[o["b"]:o["w_out"]]
    w_out = th[o["w_out"]:o["b_out"]].view(V, H)
    b_out = th[o["b_out"]:o["end"]]
    bx = torch.as_tensor(np.asarray(bytes_, dtype=np.int64))
    x = emb[bx[:, :-1]]
    lstm = torch.nn.LSTM(E, H, batch_first=True, dtype=torch.float64)
    out, _ = torch.func.functional_call(
        lstm, {"weight_ih_l0": w_ih, "weight_hh_l0": w_hh, "bias_ih_l0": b,
               "bias_hh_l0": torch.zeros_like(b)}, (x,))
    logits = out @ w_out.T + b_out
    loss = torch.nn.functional.cross_entropy(logits.reshape(-1, V), bx[:, 1:].reshape(-1))
    loss.backward()
    return loss.item(), th.grad.numpy()


@pytest.mark.parametrize("E,H,B,T", [(4, 6, 3, 7), (32, 64, 4, 64)])
def test_bptt_matches_torch_autograd(oracle_mod, E, H, B, T):
    rng = np.random.default_rng(3 + H)
    theta = rng.standard_normal(inputs.param_count(E, H)) * 0.2
    bx = rng.integers(0, V, size=(B, T + 1), dtype=np.uint8)
    m, g = oracle_mod.bptt_grad(theta, E, H, bx)
    mt, gt = _torch_grad(theta, E, H, bx)
    assert abs(m - mt) < 1e-12
    np.testing.assert_allclose(g, gt, rtol=0, atol=1e-12 * max(1.0, np.abs(gt).max()))


def test_bptt_matches_brute_force_central_differences(oracle_mod):
    E, H, B, T = 2, 3, 2, 4
    rng = np.random.default_rng(4)
    theta = rng.standard_normal(inputs.param_count(E, H)) * 0.5
    bx = rng.integers(0, V, size=(B, T + 1), dtype=np.uint8)
    _, g = oracle_mod.bptt_grad(theta, E, H, bx)
    h = 1e-5
    fd = np.zeros_like(theta)
    for j in range(theta.size):
        tp = theta.copy(); tp[j] += h
        tm = theta.copy(); tm[j] -= h
        fd[j] = (oracle_mod.loss(tp, E, H, bx, n_threads=1) - oracle_mod.loss(tm, E, H, bx, n_threads=1)) / (2 * h)
    np.testing.assert_allclose(g, fd, rtol=0, atol=1e-9)
