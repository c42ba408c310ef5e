"""Parity of the two mechanism variants on the GPU (App. D): per-probe batches
and the summed-loss control arm, through soma_spsa_estimate_opts, against the
fp64 oracle on the same seeded inputs (resident, persistent and chunked shapes)."""
import numpy as np
import pytest
import torch

from gpu_common import api, assert_coefs, assert_losses
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

V = 256


def _estimate(theta, bx, E, H, n, kind, eps, seed, step, batch_per_probe, summed_loss):
    a = api()
    N = theta.shape[0]
    B, T1 = bx.shape[-2], bx.shape[-1]
    params = torch.from_numpy(np.ascontiguousarray(theta, dtype=np.float32)).cuda()
    dev_bx = torch.from_numpy(np.ascontiguousarray(bx)).cuda()
    ws = a.alloc_workspace(E, H, N, n, B, T1 - 1)
    losses = torch.full((N, n, 2), float("nan"), device="cuda")
    coef = torch.full((N, n), float("nan"), device="cuda")
    a.spsa_estimate(params, dev_bx, E, H, n, kind, float(eps), seed, step, losses, coef, ws,
                    batch_per_probe=batch_per_probe, summed_loss=summed_loss)
    assert a.get_status() == 0
    return losses.cpu().numpy(), coef.cpu().numpy()


@pytest.mark.parametrize("kind", ["dense", "sparse"])
@pytest.mark.parametrize("batch_per_probe,summed_loss", [(True, False), (False, True), (True, True)])
@pytest.mark.parametrize("E,H,N,n,B,T", [
    (32, 64, 3, 8, 4, 24),     # tensor path
    (40, 72, 2, 5, 5, 9),      # ragged
    (16, 32, 2, 3, 70, 4),     # B > 64: two tensor-core chunks (64 + 6)
])
def test_variant_estimate(oracle_mod, kind, batch_per_probe, summed_loss, E, H, N, n, B, T):
    theta = inputs.init_params(N, E, H, seed=31, std=0.1)
    rng = np.random.default_rng(E + H + n)
    shape = (N, n, B, T + 1) if batch_per_probe else (N, B, T + 1)
    bx = rng.integers(0, V, size=shape, dtype=np.uint8)
    L, coef = _estimate(theta, bx, E, H, n, kind, 1e-3, 8, 3, batch_per_probe, summed_loss)
    Lo, co = oracle_mod.spsa_losses(theta, E, H, np.float32(1e-3), 8, 3, bx, n_pert=n, kind=kind,
                                    batch_per_probe=batch_per_probe, summed_loss=summed_loss)
    assert_losses(L, Lo)
    assert_coefs(coef, co)
    if summed_loss:
        assert np.all(coef == coef[:1])  # one coefficient per probe, shared by the experts
