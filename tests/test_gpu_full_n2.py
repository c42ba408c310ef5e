"""The whole SOMA N=2 step against the oracle's own complete step (GPU).

2 experts (E=64, H=960, 4,198,400 parameters each), 64 probes, 32
sequences x 256 target bytes per expert: the step bench.py times.  The
fp64 oracle evaluates all 2 x 64 probe pairs (about 1.8e13 flops, a few
minutes on the host cores) and applies its own update, so every quantity of
the step is compared element by element:
 - L+ and L- of all 128 (expert, probe) pairs within 2e-4 nats/byte;
 - every coefficient within 1e-2 relative (per expert in L2, and each one
   against max(|c_i|, rms(c)));
 - theta' within 1e-5 relative L2 of the oracle's theta'.
"""
import numpy as np
import pytest

from gpu_common import TOL_THETA, assert_coefs, assert_losses, rel_l2, report, run_step
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu


def test_soma_n2_full_step_against_the_oracle_step(oracle_mod):
    name = "soma_n2"
    c = inputs.CONFIGS[name]
    E, H, n = c["E"], c["H"], c["n_pert"]
    theta = inputs.config_params(name)
    bx = inputs.config_batch(name)
    seed, step = 0, 0
    g = run_step(theta, bx, E, H, n, c["eps"], c["lr"], seed, step)
    assert g["status"] == 0
    L, coef, new = oracle_mod.spsa_step(theta, E, H, n, np.float32(c["eps"]),
                                        np.float32(c["lr"]), seed, step, bx)
    assert L.shape == (2, 64, 2) and coef.shape == (2, 64)
    assert_losses(g["losses"], L)
    assert_coefs(g["coef"], coef)
    rel = rel_l2(g["theta"], new)
    report("theta_rel_l2_n2_full", rel)
    assert rel <= TOL_THETA
