"""Failure detection without a GPU fault.

Every wait in the library's kernels is bounded: a wait that runs out records
SOMA_ERR_TIMEOUT in the device status word and the kernel winds down, so the
context stays usable.  The test makes a wait run out (a barrier that nothing
completes) and checks the status, then that the next step still runs.
"""
import numpy as np
import pytest

from gpu_common import api, run_step
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

SOMA_ERR_TIMEOUT = 5


def test_bounded_wait_records_timeout_and_context_survives():
    a = api()
    assert a.get_status() == 0
    a.debug_wait_timeout(1000)
    assert a.get_status() == SOMA_ERR_TIMEOUT
    assert a.get_status() == 0  # read and cleared
    c = inputs.CONFIGS["tiny"]
    theta = inputs.config_params("tiny")
    g = run_step(theta, inputs.config_batch("tiny"), c["E"], c["H"], c["n_pert"], c["eps"], c["lr"],
                 0, 0)
    assert g["status"] == 0
    assert np.isfinite(g["losses"]).all()
