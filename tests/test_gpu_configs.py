"""Parity at the five workload sizes, in the launch configuration bench.py
times (GPU).

The full-size oracle is too slow to evaluate every probe (one SOMA N=2 step
is ~2e13 fp64 flops), so each test runs the GPU step at full size and checks
 - L+, L- and the coefficients of sampled probes against the oracle;
 - the updated theta against the oracle's update applied to the GPU's own
   coefficients (the update kernel at full size);
 - theta' against the oracle's own complete step where that is affordable
   (the tiny workload, and the N=256 expert shape with 4 experts).
"""
import numpy as np
import pytest

from gpu_common import (TOL_THETA, TOL_THETA_GIVEN_COEF, assert_coefs, assert_losses, rel_l2,
                        run_step)
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

SAMPLES = {
    "soma_n2": [(0, 0), (0, 63), (1, 17)],
    "mono": [(0, 0), (0, 1023)],
    "soma_n8": [(0, 0), (3, 17), (7, 63)],
    "soma_n256": [(0, 0), (1, 63), (77, 5), (128, 31), (200, 62), (255, 0), (255, 63), (31, 40)],
}


@pytest.mark.parametrize("name", list(SAMPLES))
def test_full_size_sampled_parity(oracle_mod, name):
    c = inputs.CONFIGS[name]
    E, H, n = c["E"], c["H"], c["n_pert"]
    theta = inputs.config_params(name)
    bx = inputs.config_batch(name)
    seed, step = 0, 0
    g = run_step(theta, bx, E, H, n, c["eps"], c["lr"], seed, step)
    assert g["status"] == 0
    assert np.isfinite(g["losses"]).all()
    by_expert = {}
    for e, i in SAMPLES[name]:
        by_expert.setdefault(e, []).append(i)
    for e, probes in by_expert.items():
        L, coef = oracle_mod.spsa_losses(theta[e:e + 1], E, H, np.float32(c["eps"]), seed, step,
                                         bx[e:e + 1], probes=probes, first_expert=e)
        assert_losses(g["losses"][e, probes], L[0])
        assert_coefs(g["coef"][e, probes][None], coef)
    new_g = oracle_mod.spsa_update(theta, E, H, np.float32(c["lr"]), seed, step,
                                   g["coef"].astype(np.float64))
    assert rel_l2(g["theta"], new_g) <= TOL_THETA_GIVEN_COEF


def test_n256_expert_shape_full_step(oracle_mod):
    # four experts of the N=256 shape, all 64 probes: the oracle's own theta'
    c = inputs.CONFIGS["soma_n256"]
    E, H, n = c["E"], c["H"], c["n_pert"]
    theta = inputs.config_params("soma_n256", n_experts=4)
    bx = inputs.config_batch("soma_n256", n_experts=4, seq_len=128)
    g = run_step(theta, bx, E, H, n, c["eps"], c["lr"], 0, 0)
    assert g["status"] == 0
    L, coef, new = oracle_mod.spsa_step(theta, E, H, n, np.float32(c["eps"]), np.float32(c["lr"]),
                                        0, 0, bx)
    assert_losses(g["losses"], L)
    assert_coefs(g["coef"], coef)
    assert rel_l2(g["theta"], new) <= TOL_THETA
