"""soma_spsa_step_static: the SPSA step for callers that cannot allocate
device memory, with its scratch in a fixed array inside the library.

Through the C ABI, on every path whose scratch lives in that array (the
resident small-expert kernel, the persistent tensor-core kernel with one and
two probes per operand group, and a batch above 64 that runs in chunks):
 - two calls in a row (the second continues from the first's parameters)
   give bit for bit the losses, coefficients and updated parameters of
   soma_spsa_step with a caller workspace;
 - the persistent tensor-core shape also matches the fp64 oracle at the
   tolerances of the other parity tests;
 - a large call followed by a small one still matches: the small call reads
   no scratch word that it did not write itself, so what the large call left
   in the array does not leak in (the caller workspace of the comparison is
   filled with 0xFF bytes for the same reason);
 - sizes beyond the fixed maximum are refused before anything is launched.

This file sorts last so that a run stopping at the first failure has run
every other test before it."""
import ctypes

import numpy as np
import pytest
import torch

from gpu_common import (TOL_THETA, api, assert_coefs, assert_losses, rel_l2)
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

STATIC_BYTES = 64 << 20

# (N, E, H, B, T, n, eps, lr) of shapes whose workspace fits the array
SHAPES = {
    "resident_tiny": None,                                 # the tiny workload
    "resident_n256_cut": "n256",                           # 3 experts of the N=256 shape
    "persistent_p2": (2, 64, 96, 8, 32, 16, 1e-3, 1e-2),   # two probes per operand group
    "persistent_p1": (1, 40, 130, 40, 12, 5, 1e-3, 1e-2),  # B = 40: one probe per group
    "chunked": (1, 6, 20, 70, 6, 3, 1e-3, 1e-2),           # B = 70 > 64: chunks of 64 and 6
}


def _static_fn():
    lib = api().lib()
    f = lib.soma_spsa_step_static
    vp, i32, u64, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_float
    f.restype = i32
    f.argtypes = [vp, i32, api().soma_dims, i32, f32, f32, u64, u64, vp, i32, i32, vp, vp, vp]
    return f


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr())


def _shape(name):
    """theta, a batch maker and the sizes of one test shape."""
    spec = SHAPES[name]
    if spec is None:
        c = inputs.CONFIGS["tiny"]
        theta = inputs.config_params("tiny")
        batch = lambda k: inputs.config_batch("tiny", step=k)  # noqa: E731
        return theta, batch, (c["n_experts"], c["E"], c["H"], c["batch"], c["seq_len"],
                              c["n_pert"], c["eps"], c["lr"])
    if spec == "n256":
        ov = dict(n_experts=3, seq_len=40)
        c = dict(inputs.CONFIGS["soma_n256"], **ov)
        theta = inputs.config_params("soma_n256", **ov)
        batch = lambda k: inputs.config_batch("soma_n256", step=k, **ov)  # noqa: E731
        return theta, batch, (c["n_experts"], c["E"], c["H"], c["batch"], c["seq_len"],
                              c["n_pert"], c["eps"], c["lr"])
    N, E, H, B, T, n, eps, lr = spec
    theta = inputs.init_params(N, E, H, seed=H, std=None)
    batch = lambda k: inputs.expert_batch(N, B, T, 2, seed=7, step=k)  # noqa: E731
    return theta, batch, spec


def _static_call(f, params, bx, sizes, seed, step):
    a = api()
    N, E, H, B, T, n, eps, lr = sizes
    losses = torch.full((N, n, 2), float("nan"), device="cuda")
    coef = torch.full((N, n), float("nan"), device="cuda")
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = f(_ptr(params), N, a.dims(E, H), n, eps, lr, seed, step, _ptr(bx), B, T, _ptr(losses),
           _ptr(coef), stream)
    assert rc == 0, a.status_string(rc)
    assert a.get_status() == 0
    return losses, coef


def _workspace_call(params, bx, sizes, seed, step):
    a = api()
    N, E, H, B, T, n, eps, lr = sizes
    ws = a.alloc_workspace(E, H, N, n, B, T)
    ws.fill_(0xFF)  # a result that read an unwritten scratch word would change
    losses = torch.full((N, n, 2), float("nan"), device="cuda")
    coef = torch.full((N, n), float("nan"), device="cuda")
    a.spsa_step(params, bx, E, H, n, eps, lr, seed, step, losses, coef, ws)
    assert a.get_status() == 0
    return losses, coef


def _bitwise(x, y):
    assert torch.equal(x, y), float((x - y).abs().max())


@pytest.mark.parametrize("name", list(SHAPES))
def test_static_step_matches_workspace_step(name):
    f = _static_fn()
    theta, batch, sizes = _shape(name)
    N, E, H, B, T, n, eps, lr = sizes
    assert api().workspace_bytes(E, H, N, n, B, T) <= STATIC_BYTES
    p_ref = torch.from_numpy(theta).cuda()
    p_static = torch.from_numpy(theta).cuda()
    for k in range(2):
        bx = torch.from_numpy(batch(k)).cuda()
        l_ref, c_ref = _workspace_call(p_ref, bx, sizes, 0, k)
        l_st, c_st = _static_call(f, p_static, bx, sizes, 0, k)
        _bitwise(l_st, l_ref)
        _bitwise(c_st, c_ref)
        _bitwise(p_static, p_ref)


def test_static_step_matches_the_oracle(oracle_mod):
    # the persistent tensor-core shape, one step from the array, against the
    # fp64 oracle's own step
    f = _static_fn()
    theta, batch, sizes = _shape("persistent_p2")
    N, E, H, B, T, n, eps, lr = sizes
    bx_np = batch(0)
    params = torch.from_numpy(theta).cuda()
    losses, coef = _static_call(f, params, torch.from_numpy(bx_np).cuda(), sizes, 3, 1)
    L, cf, new = oracle_mod.spsa_step(theta, E, H, n, np.float32(eps), np.float32(lr), 3, 1,
                                      bx_np)
    assert_losses(losses.cpu().numpy(), L)
    assert_coefs(coef.cpu().numpy(), cf)
    assert rel_l2(params.cpu().numpy(), new) <= TOL_THETA


def test_static_step_large_then_small():
    # a call that fills much of the array, then a small one on another path:
    # the small call must not see what the large one left behind
    f = _static_fn()
    big = (2, 64, 256, 32, 32, 32, 1e-3, 1e-2)
    N, E, H, B, T, n, eps, lr = big
    assert api().workspace_bytes(E, H, N, n, B, T) > 16 << 20
    theta_b = inputs.init_params(N, E, H, seed=5, std=None)
    bx_b = torch.from_numpy(inputs.expert_batch(N, B, T, 2, seed=8, step=0)).cuda()
    _static_call(f, torch.from_numpy(theta_b).cuda(), bx_b, big, 1, 0)
    for name in ("persistent_p2", "persistent_p1", "chunked", "resident_tiny"):
        theta, batch, sizes = _shape(name)
        bx = torch.from_numpy(batch(0)).cuda()
        p_ref = torch.from_numpy(theta).cuda()
        p_st = torch.from_numpy(theta).cuda()
        l_ref, c_ref = _workspace_call(p_ref, bx, sizes, 2, 0)
        l_st, c_st = _static_call(f, p_st, bx, sizes, 2, 0)
        _bitwise(l_st, l_ref)
        _bitwise(c_st, c_ref)
        _bitwise(p_st, p_ref)
        # the next large call, then the small one again from the array
        _static_call(f, torch.from_numpy(theta_b).cuda(), bx_b, big, 1, 1)


def test_static_step_refuses_sizes_beyond_its_array():
    a = api()
    f = _static_fn()
    c = inputs.CONFIGS["soma_n2"]
    E, H, N, n, B, T = c["E"], c["H"], c["n_experts"], c["n_pert"], c["batch"], c["seq_len"]
    assert a.workspace_bytes(E, H, N, n, B, T) > STATIC_BYTES
    fake = ctypes.c_void_p(0x10000)  # never dereferenced: refused before any launch
    rc = f(fake, N, a.dims(E, H), n, c["eps"], c["lr"], 0, 0, fake, B, T, fake, None, None)
    assert rc == 3  # SOMA_ERR_WORKSPACE
