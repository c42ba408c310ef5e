"""soma_spsa_step_static: the SPSA step for callers that cannot allocate
device memory, with its scratch in a fixed array inside the library.

Checks, through the C ABI, that it gives the same losses, coefficients and
updated parameters as soma_spsa_step with a caller-allocated workspace on two
calls in a row (the second continues from the first's parameters), and that
sizes beyond its fixed maximum are refused before any launch."""
import ctypes

import numpy as np
import pytest
import torch

from gpu_common import TOL_LOSS, TOL_THETA_GIVEN_COEF, api, rel_l2
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

STATIC_BYTES = 64 << 20


def _static_fn():
    lib = api().lib()
    f = lib.soma_spsa_step_static
    vp, i32, u64, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_float
    f.restype = i32
    f.argtypes = [vp, i32, api().soma_dims, i32, f32, f32, u64, u64, vp, i32, i32, vp, vp, vp]
    return f


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


@pytest.mark.parametrize("name,overrides", [("tiny", {}),
                                            ("soma_n256", dict(n_experts=3, seq_len=40))])
def test_static_step_matches_workspace_step(name, overrides):
    a = api()
    f = _static_fn()
    c = dict(inputs.CONFIGS[name], **overrides)
    N, E, H, n = c["n_experts"], c["E"], c["H"], c["n_pert"]
    B, T = c["batch"], c["seq_len"]
    assert a.workspace_bytes(E, H, N, n, B, T) <= STATIC_BYTES
    theta = inputs.config_params(name, **overrides)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    p_ref = torch.from_numpy(theta).cuda()
    p_static = torch.from_numpy(theta).cuda()
    ws = a.alloc_workspace(E, H, N, n, B, T)
    for k in range(2):
        bx = torch.from_numpy(inputs.config_batch(name, step=k, **overrides)).cuda()
        l_ref = torch.zeros(N, n, 2, device="cuda")
        c_ref = torch.zeros(N, n, device="cuda")
        l_st = torch.full((N, n, 2), float("nan"), device="cuda")
        c_st = torch.full((N, n), float("nan"), device="cuda")
        a.spsa_step(p_ref, bx, E, H, n, c["eps"], c["lr"], 0, k, l_ref, c_ref, ws)
        rc = f(_ptr(p_static), N, a.dims(E, H), n, c["eps"], c["lr"], 0, k, _ptr(bx), B, T,
               _ptr(l_st), _ptr(c_st), stream)
        assert rc == 0, a.status_string(rc)
        assert a.get_status() == 0
        lr_, ls_ = l_ref.cpu().numpy(), l_st.cpu().numpy()
        assert np.abs(ls_ - lr_).max() <= TOL_LOSS
        cr, cs = c_ref.cpu().numpy(), c_st.cpu().numpy()
        assert np.linalg.norm(cs - cr) <= 1e-2 * np.linalg.norm(cr)
        assert rel_l2(p_static.cpu().numpy(), p_ref.cpu().numpy()) <= TOL_THETA_GIVEN_COEF


def test_static_step_refuses_sizes_beyond_its_array():
    a = api()
    f = _static_fn()
    c = inputs.CONFIGS["soma_n2"]
    E, H, N, n, B, T = c["E"], c["H"], c["n_experts"], c["n_pert"], c["batch"], c["seq_len"]
    assert a.workspace_bytes(E, H, N, n, B, T) > STATIC_BYTES
    fake = ctypes.c_void_p(0x10000)  # never dereferenced: refused before any launch
    rc = f(fake, N, a.dims(E, H), n, c["eps"], c["lr"], 0, 0, fake, B, T, fake, None, None)
    assert rc == 3  # SOMA_ERR_WORKSPACE
