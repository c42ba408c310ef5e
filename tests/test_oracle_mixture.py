"""Pins of the oracle's routed inference (Sec. 3, Eq. main-mixture). CPU only.

- Output-bias-only experts predict softmax(b_out) at every position, so the
  mixture has the closed form -log((1/k) sum_j softmax(b_j)[y]).
- One route reproduces the expert's per-target NLL (the loss pinned against
  torch.nn.LSTM).
- The mixture is invariant to the order of the routes.
- It lies between min_j nll_j and min_j nll_j + log k.
"""
import numpy as np

from paper_2609_37899_gb300 import inputs

V = 256


def _experts(N, E, H, seed, std=0.3):
    return inputs.init_params(N, E, H, seed=seed, std=std).astype(np.float64)


def test_bias_only_experts_closed_form(oracle_mod):
    E, H, N, T, t0 = 3, 4, 3, 9, 2
    P = inputs.param_count(E, H)
    rng = np.random.default_rng(0)
    theta = np.zeros((N, P))
    b = rng.standard_normal((N, V))
    theta[:, P - V:] = b  # b_out is the last block of the layout
    rq = rng.integers(0, V, size=(4, T + 1), dtype=np.uint8)
    routes = np.array([[0, 1, 2], [2, 2, 0], [1, 0, 1], [0, 0, 0]])
    got = oracle_mod.mixture_nll(theta, E, H, rq, routes, t0)
    sm = np.exp(b - b.max(axis=1, keepdims=True))
    sm /= sm.sum(axis=1, keepdims=True)
    for r in range(4):
        for t in range(t0, T):
            y = rq[r, t + 1]
            want = -np.log(np.mean([sm[e, y] for e in routes[r]]))
            assert abs(got[r, t - t0] - want) < 1e-12


def test_single_route_is_the_experts_nll(oracle_mod):
    E, H, N, T = 4, 5, 3, 7
    theta = _experts(N, E, H, 1)
    rq = np.random.default_rng(1).integers(0, V, size=(3, T + 1), dtype=np.uint8)
    routes = np.array([[2], [0], [1]])
    got = oracle_mod.mixture_nll(theta, E, H, rq, routes, 0)
    for r in range(3):
        _, nll = oracle_mod.loss(theta[routes[r, 0]], E, H, rq[r:r + 1], per_token=True)
        np.testing.assert_allclose(got[r], nll[0], rtol=0, atol=1e-12)


def test_route_order_and_bounds(oracle_mod):
    E, H, N, T, t0 = 4, 5, 4, 8, 3
    theta = _experts(N, E, H, 2, std=0.8)
    rq = np.random.default_rng(2).integers(0, V, size=(5, T + 1), dtype=np.uint8)
    routes = np.array([[0, 1, 3], [3, 2, 2], [1, 1, 0], [2, 3, 0], [0, 2, 1]])
    a = oracle_mod.mixture_nll(theta, E, H, rq, routes, t0)
    b = oracle_mod.mixture_nll(theta, E, H, rq, routes[:, ::-1], t0)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-12)
    singles = np.stack([oracle_mod.mixture_nll(theta, E, H, rq, routes[:, j:j + 1], t0)
                        for j in range(3)])
    lo = singles.min(axis=0)
    assert np.all(a >= lo - 1e-12) and np.all(a <= lo + np.log(3) + 1e-12)
    assert np.any(a > lo + 1e-3)  # a real mixture, not one expert
