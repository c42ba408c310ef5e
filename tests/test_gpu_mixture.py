"""Parity of routed inference on the GPU (Sec. 3, Eq. main-mixture) with the
fp64 oracle: per-target NLL of the mixture of the routed experts, including
repeated routes, ragged shapes and expert groups of more than 128 requests
(several 128-sequence groups of the unperturbed layout in one sweep)."""
import numpy as np
import pytest
import torch

from gpu_common import api, report
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

V = 256
# per target: fp16 operands round the logits by ~2^-11 of their size; the
# mean over the scored targets is held to the loss tolerance of the step
TOL_TOKEN = 2e-3
TOL_MEAN = 2e-4


def _run(theta, rq, routes, E, H, t0):
    a = api()
    N = theta.shape[0]
    R, T1 = rq.shape
    params = torch.from_numpy(np.ascontiguousarray(theta, dtype=np.float32)).cuda()
    dev_rq = torch.from_numpy(np.ascontiguousarray(rq)).cuda()
    ws = torch.empty(a.mixture_workspace_bytes(E, H, N, routes, T1 - 1), dtype=torch.uint8,
                     device="cuda")
    out = torch.full((R, T1 - 1 - t0), float("nan"), device="cuda")
    a.mixture_nll(params, dev_rq, E, H, routes, t0, out, ws)
    assert a.get_status() == 0
    return out.cpu().numpy()


@pytest.mark.parametrize("E,H,N,R,T,k,t0", [
    (32, 64, 8, 40, 20, 3, 5),     # tensor path, one sweep
    (40, 72, 3, 17, 11, 2, 0),     # ragged
    (16, 48, 2, 100, 6, 2, 2),     # 100 requests per expert: one partly filled group
    (16, 80, 2, 300, 7, 2, 3),     # about 300 per expert: three groups, the last ragged
    (32, 48, 256, 64, 12, 4, 4),   # the N=256 expert shape, sparse routing
])
def test_mixture_matches_oracle(oracle_mod, E, H, N, R, T, k, t0):
    theta = inputs.init_params(N, E, H, seed=E + N, std=None)
    rng = np.random.default_rng(R + T)
    rq = rng.integers(0, V, size=(R, T + 1), dtype=np.uint8)
    routes = rng.integers(0, N, size=(R, k)).astype(np.int32)
    routes[0, :] = routes[0, 0]  # a request routed k times to one expert
    got = _run(theta, rq, routes, E, H, t0)
    want = oracle_mod.mixture_nll(theta, E, H, rq, routes, t0)
    err = np.abs(got - want)
    report("mixture_token_abs", err.max())
    report("mixture_mean_abs", abs(got.mean() - want.mean()))
    assert err.max() <= TOL_TOKEN
    assert abs(got.mean() - want.mean()) <= TOL_MEAN


def test_mixture_rejects_bad_routes():
    a = api()
    routes = np.array([[0, 3]], dtype=np.int32)  # expert 3 of 2
    with pytest.raises(Exception):
        a.mixture_workspace_bytes(8, 8, 2, routes, 4)
