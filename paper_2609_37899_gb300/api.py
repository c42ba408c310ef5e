"""ctypes binding of libsoma.so (the C ABI in include/soma_api.h).

Argument marshalling only: every step of the SPSA path runs in the CUDA
kernels behind the C ABI.  PyTorch supplies device memory and streams.  The
library is loaded on first use; if it is missing this module raises -- there
is no fallback of any kind.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libsoma.so")
V = 256

_lock = threading.Lock()
_lib = None

SOMA_OK = 0
STATUS_NAMES = {0: "SOMA_OK", 1: "SOMA_ERR_INVALID_ARG", 2: "SOMA_ERR_UNSUPPORTED",
                3: "SOMA_ERR_WORKSPACE", 4: "SOMA_ERR_CUDA", 5: "SOMA_ERR_TIMEOUT",
                6: "SOMA_ERR_NONFINITE", 7: "SOMA_ERR_BOUNDS"}


class SomaError(RuntimeError):
    def __init__(self, code: int, what: str):
        self.code = code
        super().__init__(f"{what}: {STATUS_NAMES.get(code, code)} ({status_string(code)})")


class soma_dims(ctypes.Structure):
    _fields_ = [("vocab", ctypes.c_int32), ("embed", ctypes.c_int32), ("hidden", ctypes.c_int32)]


TRACE_KINDS = ("gate", "head", "reduce", "update", "prep")


class soma_body_dims(ctypes.Structure):
    _fields_ = [("vocab", ctypes.c_int32), ("width", ctypes.c_int32), ("blocks", ctypes.c_int32)]


class soma_adam_config(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("delta", ctypes.c_float), ("weight_decay", ctypes.c_float),
                ("t", ctypes.c_int32)]


class soma_estimate_options(ctypes.Structure):
    _fields_ = [("probe_kind", ctypes.c_int32), ("batch_per_probe", ctypes.c_int32),
                ("summed_loss", ctypes.c_int32)]


PROBE_KINDS = {"dense": 0, "sparse": 1}
MAX_ACCUM = 64


class soma_kernel_times(ctypes.Structure):
    _fields_ = [("ms", ctypes.c_double * 5), ("launches", ctypes.c_int64 * 5)]


def _sig(lib, name, res, args):
    f = getattr(lib, name)
    f.restype = res
    f.argtypes = args


def lib():
    """The loaded libsoma.so; raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libsoma.so not found at {LIB_PATH}: build it with "
                               "`python -m paper_2609_37899_gb300.build`")
        _lib = _open(LIB_PATH)
        return _lib


def use_library(path: str):
    """Route every call of this module to the library at `path` (for
    instance the checked build, libsoma_checked.so) and return the handle in
    use before, or None; use_library_handle() puts it back."""
    global _lib
    with _lock:
        old = _lib
        _lib = _open(path)
        return old


def use_library_handle(handle):
    global _lib
    with _lock:
        _lib = handle


def _open(path: str):
    """Load one build of the library and declare the C signatures."""
    if True:
        L = ctypes.CDLL(path)
        vp, sz, i32, i64, u64, f32 = (ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int,
                                      ctypes.c_int64, ctypes.c_uint64, ctypes.c_float)
        _sig(L, "soma_param_count", i64, [soma_dims])
        _sig(L, "soma_workspace_bytes", sz, [soma_dims, i32, i32, i32, i32])
        _sig(L, "soma_init_experts", i32, [vp, i32, soma_dims, u64, f32, vp])
        _sig(L, "soma_spsa_step", i32, [vp, i32, soma_dims, i32, f32, f32, u64, u64, vp, i32,
                                        i32, vp, vp, vp, sz, vp])
        _sig(L, "soma_eval_loss", i32, [vp, i32, soma_dims, vp, i32, i32, vp, vp, sz, vp])
        _sig(L, "soma_spsa_update", i32, [vp, i32, soma_dims, i32, f32, u64, u64, vp, vp])
        _sig(L, "soma_get_status", i32, [vp])
        _sig(L, "soma_status_string", ctypes.c_char_p, [i32])
        _sig(L, "soma_trace_enable", i32, [i32])
        _sig(L, "soma_trace_read", i32, [ctypes.POINTER(soma_kernel_times), i32])
        _sig(L, "soma_debug_philox", i32, [u64, vp, vp, i32, vp])
        _sig(L, "soma_debug_rademacher", i32, [u64, u64, i32, i32, i64, i64, vp, vp])
        _sig(L, "soma_debug_tc_gemm", i32, [vp, vp, vp, i32, i32, vp])
        _sig(L, "soma_debug_tc_gemm_ts", i32, [vp, vp, vp, i32, i32, vp])
        _sig(L, "soma_spsa_estimate", i32, [vp, i32, soma_dims, i32, i32, f32, u64, u64, vp, i32,
                                            i32, vp, vp, vp, sz, vp])
        _sig(L, "soma_adam_update", i32, [vp, vp, vp, i32, soma_dims, i32, i32, u64,
                                          ctypes.POINTER(ctypes.c_uint64), i32, vp,
                                          soma_adam_config, vp])
        _sig(L, "soma_debug_probe", i32, [u64, u64, i32, i32, i32, i64, i64, vp, vp])
        i32p = ctypes.POINTER(ctypes.c_int32)
        _sig(L, "soma_mixture_workspace_bytes", sz, [soma_dims, i32, i32p, i32, i32, i32])
        _sig(L, "soma_mixture_nll", i32, [vp, i32, soma_dims, vp, i32, i32, i32p, i32, i32, vp,
                                          vp, sz, vp])
        _sig(L, "soma_spsa_estimate_opts", i32, [vp, i32, soma_dims, i32,
                                                 ctypes.POINTER(soma_estimate_options), f32, u64,
                                                 u64, vp, i32, i32, vp, vp, vp, sz, vp])
        _sig(L, "soma_debug_wait_timeout", i32, [ctypes.c_uint32, vp])
        bd = soma_body_dims
        _sig(L, "soma_body_param_count", i64, [bd])
        _sig(L, "soma_body_workspace_bytes", sz, [bd, i32, i32, i32, i32])
        _sig(L, "soma_body_spsa_estimate", i32, [vp, i32, bd, vp, i32, i32, f32, u64, u64, vp,
                                                 i32, i32, vp, vp, vp, sz, vp])
        _sig(L, "soma_body_spsa_step", i32, [vp, i32, bd, vp, i32, i32, f32, f32, u64, u64, vp,
                                             i32, i32, vp, vp, vp, sz, vp])
        _sig(L, "soma_body_eval_loss", i32, [vp, i32, bd, vp, vp, i32, i32, vp, vp, sz, vp])
        _sig(L, "soma_body_adam_update", i32, [vp, vp, vp, i32, bd, i32, i32, u64,
                                               ctypes.POINTER(ctypes.c_uint64), i32, vp,
                                               soma_adam_config, vp])
        _sig(L, "soma_debug_body_probe", i32, [u64, u64, i32, i32, bd, i32, i64, i64, vp, vp])
        _sig(L, "soma_checked_build", i32, [])
        _sig(L, "soma_debug_check_line", i32, [vp])
        _sig(L, "soma_debug_check_fail", i32, [vp])
        return L


def status_string(code: int) -> str:
    return lib().soma_status_string(code).decode()


def dims(E: int, H: int) -> soma_dims:
    return soma_dims(V, E, H)


def _check(code: int, what: str):
    if code != SOMA_OK:
        raise SomaError(code, what)


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t: torch.Tensor, dtype, name: str, numel: int | None = None) -> ctypes.c_void_p:
    if not t.is_cuda or t.dtype != dtype or not t.is_contiguous():
        raise ValueError(f"{name}: expected a contiguous CUDA {dtype} tensor")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name}: expected {numel} elements, got {t.numel()}")
    return ctypes.c_void_p(t.data_ptr())


def param_count(E: int, H: int) -> int:
    return int(lib().soma_param_count(dims(E, H)))


def workspace_bytes(E: int, H: int, n_experts: int, n_pert: int, batch: int, seq_len: int) -> int:
    return int(lib().soma_workspace_bytes(dims(E, H), n_experts, n_pert, batch, seq_len))


def alloc_workspace(E, H, n_experts, n_pert, batch, seq_len, device="cuda") -> torch.Tensor:
    n = workspace_bytes(E, H, n_experts, n_pert, batch, seq_len)
    if n == 0:
        raise ValueError("invalid sizes for the workspace")
    return torch.empty(n, dtype=torch.uint8, device=device)


def init_experts(params: torch.Tensor, E: int, H: int, seed: int, std: float = 0.0, stream=None):
    n_experts = params.shape[0]
    _check(lib().soma_init_experts(_dev(params, torch.float32, "params",
                                        n_experts * param_count(E, H)),
                                   n_experts, dims(E, H), seed, std, _stream(stream)),
           "soma_init_experts")


def spsa_step(params: torch.Tensor, byte_batch: torch.Tensor, E: int, H: int, n_pert: int,
              eps: float, lr: float, seed: int, step: int, losses: torch.Tensor,
              coef: torch.Tensor | None, workspace: torch.Tensor, stream=None):
    """One SPSA step; params [N, P] fp32 updated in place, losses [N, n_pert, 2],
    coef [N, n_pert] or None, byte_batch [N, B, T+1] uint8 (all on the device)."""
    N, B, T1 = byte_batch.shape
    P = param_count(E, H)
    _check(lib().soma_spsa_step(
        _dev(params, torch.float32, "params", N * P), N, dims(E, H), n_pert, eps, lr, seed, step,
        _dev(byte_batch, torch.uint8, "byte_batch"), B, T1 - 1,
        _dev(losses, torch.float32, "losses", N * n_pert * 2),
        _dev(coef, torch.float32, "coef", N * n_pert) if coef is not None else None,
        _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)),
        "soma_spsa_step")


def spsa_estimate(params: torch.Tensor, byte_batch: torch.Tensor, E: int, H: int, n_pert: int,
                  kind: str, eps: float, seed: int, step: int, losses: torch.Tensor,
                  coef: torch.Tensor, workspace: torch.Tensor, stream=None,
                  batch_per_probe: bool = False, summed_loss: bool = False):
    """Losses [N, n_pert, 2] and coefficients [N, n_pert] of one accumulation
    batch with dense or sparse probes; params are read only.  byte_batch is
    [N, B, T+1], or [N, n_pert, B, T+1] with batch_per_probe; summed_loss
    gives every expert the coefficient of the summed loss (control arm)."""
    N = params.shape[0]
    B, T1 = byte_batch.shape[-2], byte_batch.shape[-1]
    if batch_per_probe:
        assert tuple(byte_batch.shape[:2]) == (N, n_pert), "byte_batch [N, n_pert, B, T+1]"
    P = param_count(E, H)
    opts = soma_estimate_options(PROBE_KINDS[kind], int(batch_per_probe), int(summed_loss))
    _check(lib().soma_spsa_estimate_opts(
        _dev(params, torch.float32, "params", N * P), N, dims(E, H), n_pert, ctypes.byref(opts),
        eps, seed, step, _dev(byte_batch, torch.uint8, "byte_batch"), B, T1 - 1,
        _dev(losses, torch.float32, "losses", N * n_pert * 2),
        _dev(coef, torch.float32, "coef", N * n_pert),
        _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)),
        "soma_spsa_estimate")


def adam_update(params: torch.Tensor, m: torch.Tensor, v: torch.Tensor, E: int, H: int,
                kind: str, seed: int, steps, coef: torch.Tensor, lr: float, beta1: float,
                beta2: float, delta: float, weight_decay: float, t: int, stream=None):
    """The Adam step of Eq. localspsa; coef [A, N, n_pert], steps: A host ints."""
    A, N, n_pert = coef.shape
    P = param_count(E, H)
    st = (ctypes.c_uint64 * A)(*[int(x) for x in steps])
    cfg = soma_adam_config(lr, beta1, beta2, delta, weight_decay, t)
    _check(lib().soma_adam_update(
        _dev(params, torch.float32, "params", N * P), _dev(m, torch.float32, "m", N * P),
        _dev(v, torch.float32, "v", N * P), N, dims(E, H), n_pert, PROBE_KINDS[kind], seed, st,
        A, _dev(coef, torch.float32, "coef", A * N * n_pert), cfg, _stream(stream)),
        "soma_adam_update")


def _routes(routes):
    import numpy as np
    rt = np.ascontiguousarray(routes, dtype=np.int32)
    assert rt.ndim == 2, "routes [R, k]"
    return rt, rt.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def mixture_workspace_bytes(E: int, H: int, n_experts: int, routes, seq_len: int) -> int:
    rt, ptr = _routes(routes)
    n = int(lib().soma_mixture_workspace_bytes(dims(E, H), n_experts, ptr, rt.shape[0],
                                               rt.shape[1], seq_len))
    if n == 0:
        raise SomaError(1, "soma_mixture_workspace_bytes: invalid sizes or routes")
    return n


def mixture_nll(params: torch.Tensor, requests: torch.Tensor, E: int, H: int, routes, t0: int,
                nll_out: torch.Tensor, workspace: torch.Tensor, stream=None):
    """Routed inference (Eq. main-mixture): nll_out [R, T - t0] for requests
    [R, T+1] (device) and host routes [R, k]."""
    rt, ptr = _routes(routes)
    R, T1 = requests.shape
    N = params.shape[0]
    _check(lib().soma_mixture_nll(
        _dev(params, torch.float32, "params", N * param_count(E, H)), N, dims(E, H),
        _dev(requests, torch.uint8, "requests"), R, T1 - 1, ptr, rt.shape[1], t0,
        _dev(nll_out, torch.float32, "nll_out", R * (T1 - 1 - t0)),
        _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)),
        "soma_mixture_nll")


def eval_loss(params: torch.Tensor, byte_batch: torch.Tensor, E: int, H: int,
              loss_out: torch.Tensor, workspace: torch.Tensor, stream=None):
    N, B, T1 = byte_batch.shape
    _check(lib().soma_eval_loss(
        _dev(params, torch.float32, "params", N * param_count(E, H)), N, dims(E, H),
        _dev(byte_batch, torch.uint8, "byte_batch"), B, T1 - 1,
        _dev(loss_out, torch.float32, "loss_out", N),
        _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)),
        "soma_eval_loss")


def spsa_update(params: torch.Tensor, E: int, H: int, lr: float, seed: int, step: int,
                coef: torch.Tensor, stream=None):
    N, n_pert = coef.shape
    _check(lib().soma_spsa_update(
        _dev(params, torch.float32, "params", N * param_count(E, H)), N, dims(E, H), n_pert,
        lr, seed, step, _dev(coef, torch.float32, "coef", N * n_pert), _stream(stream)),
        "soma_spsa_update")


def trace_enable(on: bool = True):
    _check(lib().soma_trace_enable(1 if on else 0), "soma_trace_enable")


def trace_read(reset: bool = True) -> dict:
    """{kind: (total_ms, launches)} of the traced launches (waits for them)."""
    t = soma_kernel_times()
    _check(lib().soma_trace_read(ctypes.byref(t), 1 if reset else 0), "soma_trace_read")
    return {k: (t.ms[j], int(t.launches[j])) for j, k in enumerate(TRACE_KINDS)}


def get_status(stream=None) -> int:
    return int(lib().soma_get_status(_stream(stream)))


def debug_philox(seed: int, counters: torch.Tensor, stream=None) -> torch.Tensor:
    """Philox4x32-10 words [n, 4] (int32 bit patterns) for counters [n, 4] int32."""
    n = counters.shape[0]
    out = torch.empty_like(counters)
    _check(lib().soma_debug_philox(seed, _dev(counters, torch.int32, "counters"),
                                   _dev(out, torch.int32, "out"), n, _stream(stream)),
           "soma_debug_philox")
    return out


def debug_rademacher(seed: int, step: int, expert: int, probe: int, p0: int, count: int,
                     device="cuda", stream=None) -> torch.Tensor:
    z = torch.empty(count, dtype=torch.int8, device=device)
    _check(lib().soma_debug_rademacher(seed, step, expert, probe, p0, count,
                                       _dev(z, torch.int8, "z"), _stream(stream)),
           "soma_debug_rademacher")
    return z


def debug_probe(seed: int, step: int, expert: int, probe: int, kind: str, p0: int, count: int,
                device="cuda", stream=None) -> torch.Tensor:
    z = torch.empty(count, dtype=torch.int8, device=device)
    _check(lib().soma_debug_probe(seed, step, expert, probe, PROBE_KINDS[kind], p0, count,
                                  _dev(z, torch.int8, "z"), _stream(stream)),
           "soma_debug_probe")
    return z


def debug_wait_timeout(max_polls: int, stream=None):
    """Launch a kernel whose bounded wait runs out (see soma_api.h)."""
    _check(lib().soma_debug_wait_timeout(max_polls, _stream(stream)), "soma_debug_wait_timeout")


def debug_tc_gemm(a: torch.Tensor, b: torch.Tensor, stream=None,
                  a_in_tmem: bool = False) -> torch.Tensor:
    """a [128, K] fp16, b [N, K] fp16 (CUDA) -> a @ b.T [128, N] fp32 on the tensor cores;
    with a_in_tmem, a is staged in tensor memory (soma_debug_tc_gemm_ts)."""
    n, k = b.shape
    d = torch.empty(128, n, dtype=torch.float32, device=a.device)
    name = "soma_debug_tc_gemm_ts" if a_in_tmem else "soma_debug_tc_gemm"
    _check(getattr(lib(), name)(_dev(a, torch.float16, "a", 128 * k),
                                _dev(b, torch.float16, "b", n * k),
                                _dev(d, torch.float32, "d"), n, k, _stream(stream)), name)
    return d


class SomaExperts:
    """N experts' parameters and scratch on the current GPU, stepped by the
    C ABI.  Holds device tensors only; each call is one library call."""

    def __init__(self, n_experts: int, E: int, H: int, n_pert: int, batch: int, seq_len: int,
                 device="cuda"):
        self.N, self.E, self.H = n_experts, E, H
        self.n_pert, self.batch, self.seq_len = n_pert, batch, seq_len
        self.P = param_count(E, H)
        self.params = torch.zeros(n_experts, self.P, dtype=torch.float32, device=device)
        self.workspace = alloc_workspace(E, H, n_experts, n_pert, batch, seq_len, device)
        self.losses = torch.zeros(n_experts, n_pert, 2, dtype=torch.float32, device=device)
        self.coef = torch.zeros(n_experts, n_pert, dtype=torch.float32, device=device)
        self.loss = torch.zeros(n_experts, dtype=torch.float32, device=device)

    def init(self, seed: int, std: float = 0.0, stream=None):
        init_experts(self.params, self.E, self.H, seed, std, stream)

    def step(self, byte_batch: torch.Tensor, eps: float, lr: float, seed: int, step: int,
             stream=None):
        spsa_step(self.params, byte_batch, self.E, self.H, self.n_pert, eps, lr, seed, step,
                  self.losses, self.coef, self.workspace, stream)
        return self.losses, self.coef

    def eval(self, byte_batch: torch.Tensor, stream=None):
        eval_loss(self.params, byte_batch, self.E, self.H, self.loss, self.workspace, stream)
        return self.loss

    def adam_step(self, byte_batches, eps: float, seed: int, steps, t: int, lr: float,
                  beta1: float = 0.9, beta2: float = 0.999, delta: float = 1e-8,
                  weight_decay: float = 1e-4, kind: str = "sparse", stream=None,
                  batch_per_probe: bool = False, summed_loss: bool = False):
        """The paper's optimizer step: one estimate per accumulation batch
        (byte_batches[a] with probe step counter steps[a]), then the Adam
        update with bias correction for update t.  Moments live on this
        object (zeros before the first update)."""
        A = len(byte_batches)
        if getattr(self, "m", None) is None:
            self.m = torch.zeros_like(self.params)
            self.v = torch.zeros_like(self.params)
        if getattr(self, "coef_acc", None) is None or self.coef_acc.shape[0] != A:
            self.coef_acc = torch.zeros(A, self.N, self.n_pert, dtype=torch.float32,
                                        device=self.params.device)
            self.losses_acc = torch.zeros(A, self.N, self.n_pert, 2, dtype=torch.float32,
                                          device=self.params.device)
        for a in range(A):
            spsa_estimate(self.params, byte_batches[a], self.E, self.H, self.n_pert, kind, eps,
                          seed, steps[a], self.losses_acc[a], self.coef_acc[a], self.workspace,
                          stream, batch_per_probe=batch_per_probe, summed_loss=summed_loss)
        adam_update(self.params, self.m, self.v, self.E, self.H, kind, seed, steps, self.coef_acc,
                    lr, beta1, beta2, delta, weight_decay, t, stream)
        return self.losses_acc, self.coef_acc


# ---------------------------------------------------------------------------
# The paper's expert body (Sec. "Model size"): D pre-norm residual blocks of
# width d (bias-free LSTM, GELU MLP of width 4d), gain-only LayerNorm, and a
# frozen tied head E [256, d] shared by every expert.
# ---------------------------------------------------------------------------

def body_dims(d: int = 32, D: int = 2) -> soma_body_dims:
    return soma_body_dims(V, d, D)


def body_param_count(d: int = 32, D: int = 2) -> int:
    return int(lib().soma_body_param_count(body_dims(d, D)))


def body_workspace_bytes(d: int, D: int, n_experts: int, n_pert: int, batch: int,
                         seq_len: int) -> int:
    return int(lib().soma_body_workspace_bytes(body_dims(d, D), n_experts, n_pert, batch,
                                               seq_len))


def body_alloc_workspace(d, D, n_experts, n_pert, batch, seq_len, device="cuda") -> torch.Tensor:
    n = body_workspace_bytes(d, D, n_experts, n_pert, batch, seq_len)
    if n == 0:
        raise ValueError("invalid sizes for the workspace")
    return torch.empty(n, dtype=torch.uint8, device=device)


def body_spsa_estimate(params: torch.Tensor, head: torch.Tensor, byte_batch: torch.Tensor,
                       d: int, D: int, n_pert: int, kind: str, eps: float, seed: int, step: int,
                       losses: torch.Tensor | None, coef: torch.Tensor, workspace: torch.Tensor,
                       stream=None):
    """Losses [N, n_pert, 2] and coefficients [N, n_pert] of the body;
    params [N, M_body] are read only, head [256, d], byte_batch [N, B, T+1]."""
    N, B, T1 = byte_batch.shape
    P = body_param_count(d, D)
    _check(lib().soma_body_spsa_estimate(
        _dev(params, torch.float32, "params", N * P), N, body_dims(d, D),
        _dev(head, torch.float32, "head", V * d), n_pert, PROBE_KINDS[kind], eps, seed, step,
        _dev(byte_batch, torch.uint8, "byte_batch"), B, T1 - 1,
        _dev(losses, torch.float32, "losses", N * n_pert * 2) if losses is not None else None,
        _dev(coef, torch.float32, "coef", N * n_pert),
        _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)),
        "soma_body_spsa_estimate")


def body_spsa_step(params: torch.Tensor, head: torch.Tensor, byte_batch: torch.Tensor, d: int,
                   D: int, n_pert: int, kind: str, eps: float, lr: float, seed: int, step: int,
                   losses: torch.Tensor | None, coef: torch.Tensor | None,
                   workspace: torch.Tensor, stream=None):
    """The body's SPSA step: the estimate, then theta -= lr (1/n) sum_i c_i z_i."""
    N, B, T1 = byte_batch.shape
    P = body_param_count(d, D)
    _check(lib().soma_body_spsa_step(
        _dev(params, torch.float32, "params", N * P), N, body_dims(d, D),
        _dev(head, torch.float32, "head", V * d), n_pert, PROBE_KINDS[kind], eps, lr, seed, step,
        _dev(byte_batch, torch.uint8, "byte_batch"), B, T1 - 1,
        _dev(losses, torch.float32, "losses", N * n_pert * 2) if losses is not None else None,
        _dev(coef, torch.float32, "coef", N * n_pert) if coef is not None else None,
        _dev(workspace, torch.uint8, "workspace"), workspace.numel(), _stream(stream)),
        "soma_body_spsa_step")


def body_eval_loss(params: torch.Tensor, head: torch.Tensor, byte_batch: torch.Tensor, d: int,
                   D: int, workspace: torch.Tensor, stream=None) -> torch.Tensor:
    N, B, T1 = byte_batch.shape
    out = torch.empty(N, dtype=torch.float32, device=params.device)
    _check(lib().soma_body_eval_loss(
        _dev(params, torch.float32, "params", N * body_param_count(d, D)), N, body_dims(d, D),
        _dev(head, torch.float32, "head", V * d), _dev(byte_batch, torch.uint8, "byte_batch"),
        B, T1 - 1, _dev(out, torch.float32, "loss"), _dev(workspace, torch.uint8, "workspace"),
        workspace.numel(), _stream(stream)), "soma_body_eval_loss")
    return out


def body_adam_update(params: torch.Tensor, m: torch.Tensor, v: torch.Tensor, d: int, D: int,
                     kind: str, seed: int, steps, coef: torch.Tensor, lr: float, beta1: float,
                     beta2: float, delta: float, weight_decay: float, t: int, stream=None):
    """Eq. localspsa on the body; coef [A, N, n_pert], steps: A host ints."""
    A, N, n_pert = coef.shape
    P = body_param_count(d, D)
    st = (ctypes.c_uint64 * A)(*[int(x) for x in steps])
    cfg = soma_adam_config(lr, beta1, beta2, delta, weight_decay, t)
    _check(lib().soma_body_adam_update(
        _dev(params, torch.float32, "params", N * P), _dev(m, torch.float32, "m", N * P),
        _dev(v, torch.float32, "v", N * P), N, body_dims(d, D), n_pert, PROBE_KINDS[kind], seed,
        st, A, _dev(coef, torch.float32, "coef", A * N * n_pert), cfg, _stream(stream)),
        "soma_body_adam_update")


def debug_body_probe(seed: int, step: int, expert: int, probe: int, d: int, D: int, kind: str,
                     p0: int, count: int, stream=None) -> torch.Tensor:
    z = torch.zeros(count, dtype=torch.int8, device="cuda")
    _check(lib().soma_debug_body_probe(seed, step, expert, probe, body_dims(d, D),
                                       PROBE_KINDS[kind], p0, count,
                                       _dev(z, torch.int8, "z"), _stream(stream)),
           "soma_debug_body_probe")
    return z


class SomaBodies:
    """N expert bodies of the paper's architecture with their shared frozen
    head, parameters, workspace and Adam moments resident on the device."""

    def __init__(self, n_experts: int, n_pert: int, batch: int, seq_len: int, d: int = 32,
                 D: int = 2, device: str = "cuda"):
        self.N, self.d, self.D, self.n_pert = n_experts, d, D, n_pert
        self.P = body_param_count(d, D)
        if self.P < 0:
            raise ValueError("unsupported body dims")
        self.params = torch.zeros(n_experts, self.P, dtype=torch.float32, device=device)
        self.head = torch.zeros(V, d, dtype=torch.float32, device=device)
        self.m = torch.zeros_like(self.params)
        self.v = torch.zeros_like(self.params)
        self.workspace = body_alloc_workspace(d, D, n_experts, n_pert, batch, seq_len, device)
        self.losses = torch.empty(n_experts, n_pert, 2, dtype=torch.float32, device=device)
        self.coef = torch.empty(n_experts, n_pert, dtype=torch.float32, device=device)

    def step(self, byte_batch, eps, lr, seed, step, kind="sparse", stream=None):
        body_spsa_step(self.params, self.head, byte_batch, self.d, self.D, self.n_pert, kind, eps,
                       lr, seed, step, self.losses, self.coef, self.workspace, stream)
        return self.losses, self.coef

    def eval(self, byte_batch, stream=None):
        return body_eval_loss(self.params, self.head, byte_batch, self.d, self.D, self.workspace,
                              stream)

    def adam_step(self, byte_batches, eps, seed, steps, t, lr, beta1=0.9, beta2=0.999,
                  delta=1e-8, weight_decay=1e-4, kind="sparse", stream=None):
        """Eq. localspsa: one estimate per accumulation batch, then Adam."""
        A = len(byte_batches)
        coef = torch.empty(A, self.N, self.n_pert, dtype=torch.float32, device=self.params.device)
        losses = torch.empty(A, self.N, self.n_pert, 2, dtype=torch.float32,
                             device=self.params.device)
        for a, bx in enumerate(byte_batches):
            body_spsa_estimate(self.params, self.head, bx, self.d, self.D, self.n_pert, kind, eps,
                               seed, steps[a], losses[a], coef[a], self.workspace, stream)
        body_adam_update(self.params, self.m, self.v, self.d, self.D, kind, seed, steps, coef, lr,
                         beta1, beta2, delta, weight_decay, t, stream)
        return losses, coef
