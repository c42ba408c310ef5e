"""The checked build (libsoma_checked.so) on every path of the library (GPU).

The checked build guards the kernels' shared-memory offsets, tensor-memory
columns and global indices, and puts canary words around every workspace
region.  These tests build it, route the binding to it and run:
 - each entry point on shapes that reach each kernel (the resident
   small-expert kernel, the persistent tensor-core kernel with one and two
   probes per operand group, a batch above 64 in chunks, the 2-expert
   production shape at a shorter sequence, sparse probes, the loss-only
   evaluation, routed inference, the expert body, Adam, the fixed-array
   step): no check fails (status 0, no recorded position), and the results
   agree with the default build's;
 - one failing check that guards no access: SOMA_ERR_BOUNDS and its source
   position are reported, and reading clears them;
 - after a step the canary gaps still hold the canary word.
"""
import contextlib
import ctypes
import os
import re

import numpy as np
import pytest
import torch

from gpu_common import api
from paper_2609_37899_gb300 import inputs

pytestmark = pytest.mark.gpu

CANARY = 0x5A17C0DE
GUARD_WORDS = 64


@pytest.fixture(scope="module")
def checked_path():
    from paper_2609_37899_gb300 import build
    return build.build(checked=True)


@contextlib.contextmanager
def using(path):
    a = api()
    old = a.use_library(path)
    try:
        yield a
    finally:
        a.use_library_handle(old)


def _default_path():
    from paper_2609_37899_gb300 import build
    return build.LIB


def _lstm_step(sizes, kind="dense", seed=3, step=1):
    def run(a):
        N, E, H, B, T, n = sizes
        theta = inputs.init_params(N, E, H, seed=H, std=None)
        params = torch.from_numpy(theta).cuda()
        bx = torch.from_numpy(inputs.expert_batch(N, B, T, 2, seed=7, step=step)).cuda()
        ws = a.alloc_workspace(E, H, N, n, B, T)
        losses = torch.zeros(N, n, 2, device="cuda")
        coef = torch.zeros(N, n, device="cuda")
        if kind == "dense":
            a.spsa_step(params, bx, E, H, n, 1e-3, 1e-2, seed, step, losses, coef, ws)
            return dict(losses=losses, coef=coef, theta=params), ws
        a.spsa_estimate(params, bx, E, H, n, kind, 1e-3, seed, step, losses, coef, ws)
        return dict(losses=losses, coef=coef), ws
    return run


def _eval(sizes):
    def run(a):
        N, E, H, B, T = sizes
        params = torch.from_numpy(inputs.init_params(N, E, H, seed=11, std=None)).cuda()
        bx = torch.from_numpy(inputs.expert_batch(N, B, T, 2, seed=5, step=0)).cuda()
        ws = a.alloc_workspace(E, H, N, 1, B, T)
        out = torch.zeros(N, device="cuda")
        a.eval_loss(params, bx, E, H, out, ws)
        return dict(loss=out), ws
    return run


def _mixture(N=3, E=16, H=48, R=70, k=2, T=9, t0=2):
    def run(a):
        rng = np.random.default_rng(13)
        params = torch.from_numpy(inputs.init_params(N, E, H, seed=2, std=None)).cuda()
        rq = torch.from_numpy(rng.integers(0, 256, size=(R, T + 1), dtype=np.uint8)).cuda()
        routes = rng.integers(0, N, size=(R, k)).astype(np.int32)
        ws = torch.empty(a.mixture_workspace_bytes(E, H, N, routes, T), dtype=torch.uint8,
                         device="cuda")
        out = torch.zeros(R, T - t0, device="cuda")
        a.mixture_nll(params, rq, E, H, routes, t0, out, ws)
        return dict(nll=out), ws
    return run


def _body(d=32, D=2, N=2, n=16, B=4, T=12):
    def run(a):
        from test_oracle_body import _setup
        theta, head, bx = _setup(d, D, N=N, B=B, T=T, seed=29, wstd=0.05)
        params = torch.from_numpy(theta).cuda()
        dhead = torch.from_numpy(head).cuda()
        dbx = torch.from_numpy(bx).cuda()
        ws = a.body_alloc_workspace(d, D, N, n, B, T)
        losses = torch.zeros(N, n, 2, device="cuda")
        coef = torch.zeros(N, n, device="cuda")
        a.body_spsa_step(params, dhead, dbx, d, D, n, "sparse", 1e-3, 1e-2, 31, 0, losses, coef,
                         ws)
        loss = a.body_eval_loss(params, dhead, dbx, d, D, ws)
        return dict(losses=losses, coef=coef, theta=params, loss=loss), ws
    return run


def _adam(N=2, E=24, H=40, n=8):
    def run(a):
        P = a.param_count(E, H)
        params = torch.from_numpy(inputs.init_params(N, E, H, seed=4, std=None)).cuda()
        m = torch.zeros(N, P, device="cuda")
        v = torch.zeros(N, P, device="cuda")
        coef = torch.from_numpy(np.random.default_rng(3).standard_normal((3, N, n))
                                .astype(np.float32)).cuda()
        a.adam_update(params, m, v, E, H, "dense", 5, [0, 1, 2], coef, 1e-3, 0.9, 0.999, 1e-8,
                      0.01, 1)
        return dict(theta=params, m=m, v=v), None
    return run


def _static(sizes=(2, 64, 96, 8, 32, 16)):
    def run(a):
        N, E, H, B, T, n = sizes
        f = a.lib().soma_spsa_step_static
        vp, i32, u64, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_float
        f.restype = i32
        f.argtypes = [vp, i32, a.soma_dims, i32, f32, f32, u64, u64, vp, i32, i32, vp, vp, vp]
        params = torch.from_numpy(inputs.init_params(N, E, H, seed=H, std=None)).cuda()
        bx = torch.from_numpy(inputs.expert_batch(N, B, T, 2, seed=7, step=0)).cuda()
        losses = torch.zeros(N, n, 2, device="cuda")
        coef = torch.zeros(N, n, device="cuda")
        p = lambda t: ctypes.c_void_p(t.data_ptr())  # noqa: E731
        stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
        rc = f(p(params), N, a.dims(E, H), n, 1e-3, 1e-2, 0, 0, p(bx), B, T, p(losses), p(coef),
               stream)
        assert rc == 0, a.status_string(rc)
        return dict(losses=losses, coef=coef, theta=params), None
    return run


CASES = {
    "resident_tiny": _lstm_step((1, 32, 64, 4, 64, 8)),
    "persistent_p2": _lstm_step((2, 64, 96, 8, 32, 16)),
    "persistent_p1": _lstm_step((1, 40, 130, 40, 12, 5)),
    "chunked": _lstm_step((1, 6, 20, 70, 6, 3)),
    "production_t16": _lstm_step((2, 64, 960, 32, 16, 64)),
    "sparse_probes": _lstm_step((2, 64, 96, 8, 20, 16), kind="sparse"),
    "eval_chunked": _eval((2, 20, 72, 66, 7)),
    "mixture": _mixture(),
    "body": _body(),
    "adam": _adam(),
    "static": _static(),
}


def _host(out):
    return {k: v.detach().cpu().numpy().astype(np.float64) for k, v in out.items()}


@pytest.mark.parametrize("name", list(CASES))
def test_no_check_fails_and_results_agree(checked_path, name):
    run = CASES[name]
    with using(_default_path()) as a:
        assert a.lib().soma_checked_build() == 0
        want, _ = run(a)
        assert a.get_status() == 0
        want = _host(want)
    with using(checked_path) as a:
        assert a.lib().soma_checked_build() == 1
        got, ws = run(a)
        status = a.get_status()
        line = a.lib().soma_debug_check_line(None)
        assert (status, line) == (0, 0), (a.STATUS_NAMES.get(status, status), line)
        got = _host(got)
    for k in want:
        np.testing.assert_allclose(got[k], want[k], rtol=1e-5, atol=1e-6, err_msg=k)


def test_a_failing_check_is_reported_and_cleared(checked_path):
    src = os.path.join(os.path.dirname(api().__file__), "csrc", "spsa_misc.cu")
    text = open(src).read().splitlines()
    file_id = int(next(re.search(r"SOMA_CHECK_FILE (\d+)", s).group(1)
                       for s in text if s.startswith("#define SOMA_CHECK_FILE")))
    line = next(i + 1 for i, s in enumerate(text) if "SOMA_CHECK(blockDim.x == 0" in s)
    with using(checked_path) as a:
        assert a.get_status() == 0 and a.lib().soma_debug_check_line(None) == 0
        assert a.lib().soma_debug_check_fail(None) == 0
        assert a.get_status() == 7  # SOMA_ERR_BOUNDS
        assert a.lib().soma_debug_check_line(None) == 10000 * file_id + line
        assert a.get_status() == 0 and a.lib().soma_debug_check_line(None) == 0
    with using(_default_path()) as a:
        # the default build has no checks: the same call reports nothing
        assert a.lib().soma_debug_check_fail(None) == 0
        assert a.get_status() == 0


@pytest.mark.parametrize("name", ["persistent_p2", "chunked", "body"])
def test_canary_gaps_are_intact_after_a_step(checked_path, name):
    with using(checked_path) as a:
        _, ws = CASES[name](a)
        assert a.get_status() == 0
        words = ws.view(torch.int32).cpu().numpy().view(np.uint32)
    hit = (words == CANARY).astype(np.int8)
    # runs of whole 256-byte gaps (64 words, 64-word aligned)
    gaps = hit[: words.size // GUARD_WORDS * GUARD_WORDS].reshape(-1, GUARD_WORDS).all(axis=1)
    assert gaps.sum() >= 3, int(gaps.sum())
    assert gaps[-1], "the gap after the last region"
