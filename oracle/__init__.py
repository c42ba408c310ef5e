"""fp64 CPU oracle for the SOMA SPSA step -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The
product (``paper_2609_37899_gb300``) never imports, links or runs it, and this
package imports nothing from the product.

The arithmetic lives in ``soma_oracle.c`` (plain C, fp64, optional OpenMP over
the sequences of a batch).  This module only compiles it with gcc and
marshals numpy arrays through ctypes.  Parameters are widened from fp32 to
fp64 exactly before they reach the C code, as are ``eps`` and ``lr``.

Paper references (Scaling Zero-Order Pretraining through Model Sharding):
  - Eq. main-spsa (Sec. 4): the central-difference estimator with dense
    Rademacher probes, all probes and both signs on one shared batch;
  - Eq. localspsa (App. E): the same estimator inside the update; here the
    plain-SGD update theta - lr * g_hat (no moments);
  - App. C / Sec. 3: one-layer byte LSTM expert, V = 256;
  - Table experimental-setup: mean cross entropy in nats/byte, hidden state
    reset for every window.

Parity status: every function here is pinned by a CPU test against something
other than itself (published Philox known answers and torch's Philox engine,
torch.nn.LSTM in float64, torch autograd, brute-force central differences,
closed forms).  No function is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "soma_oracle.c")
_SRCS = [_SRC, os.path.join(_HERE, "body_oracle.c")]
_LIB_PATH = os.path.join(_HERE, "liboracle_soma.so")
_lock = threading.Lock()
_lib = None

V = 256


def build(force: bool = False) -> str:
    """Compile soma_oracle.c and body_oracle.c into liboracle_soma.so with gcc
    (-fopenmp)."""
    if (not force and os.path.exists(_LIB_PATH)
            and all(os.path.getmtime(_LIB_PATH) >= os.path.getmtime(f) for f in _SRCS)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-fno-fast-math", "-o", tmp, *_SRCS, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        c_u32p = ctypes.POINTER(ctypes.c_uint32)
        c_dp = ctypes.POINTER(ctypes.c_double)
        c_u8p = ctypes.POINTER(ctypes.c_uint8)
        lib.oracle_philox4x32_10.argtypes = [c_u32p, c_u32p, c_u32p]
        lib.oracle_philox4x32_10.restype = None
        lib.oracle_rademacher.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint32,
                                          ctypes.c_uint32, ctypes.c_int64, ctypes.c_int64,
                                          ctypes.POINTER(ctypes.c_int8)]
        lib.oracle_rademacher.restype = None
        lib.oracle_param_count.argtypes = [ctypes.c_int, ctypes.c_int]
        lib.oracle_param_count.restype = ctypes.c_int64
        lib.oracle_loss.argtypes = [c_dp, ctypes.c_int, ctypes.c_int, c_u8p, ctypes.c_int,
                                    ctypes.c_int, c_dp, ctypes.c_int]
        lib.oracle_loss.restype = ctypes.c_double
        lib.oracle_spsa_losses.argtypes = [c_dp, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                           ctypes.c_int,
                                           ctypes.c_double, ctypes.c_uint64, ctypes.c_uint64,
                                           c_u8p, ctypes.c_int, ctypes.c_int,
                                           ctypes.POINTER(ctypes.c_int32), ctypes.c_int,
                                           c_dp, c_dp, ctypes.c_int]
        lib.oracle_spsa_losses.restype = ctypes.c_int
        lib.oracle_spsa_losses_kind.argtypes = [c_dp, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_double, ctypes.c_int,
                                                ctypes.c_uint64, ctypes.c_uint64,
                                                c_u8p, ctypes.c_int, ctypes.c_int,
                                                ctypes.POINTER(ctypes.c_int32), ctypes.c_int,
                                                c_dp, c_dp, ctypes.c_int]
        lib.oracle_spsa_losses_kind.restype = ctypes.c_int
        lib.oracle_spsa_losses_opts.argtypes = [c_dp, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_double, ctypes.c_int,
                                                ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                                ctypes.c_uint64, ctypes.c_uint64,
                                                c_u8p, ctypes.c_int, ctypes.c_int,
                                                ctypes.POINTER(ctypes.c_int32), ctypes.c_int,
                                                c_dp, c_dp, ctypes.c_int]
        lib.oracle_spsa_losses_opts.restype = ctypes.c_int
        lib.oracle_mixture_nll.argtypes = [c_dp, ctypes.c_int, ctypes.c_int, ctypes.c_int, c_u8p,
                                           ctypes.c_int, ctypes.c_int,
                                           ctypes.POINTER(ctypes.c_int32), ctypes.c_int,
                                           ctypes.c_int, c_dp, ctypes.c_int]
        lib.oracle_mixture_nll.restype = ctypes.c_int
        lib.oracle_probe.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint32,
                                     ctypes.c_uint32, ctypes.c_int, ctypes.c_int64, ctypes.c_int64,
                                     ctypes.POINTER(ctypes.c_int8)]
        lib.oracle_probe.restype = ctypes.c_int
        lib.oracle_adam_update.argtypes = [c_dp, c_dp, c_dp, ctypes.c_int, ctypes.c_int,
                                           ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                           ctypes.c_uint64, ctypes.POINTER(ctypes.c_uint64),
                                           ctypes.c_int, c_dp, ctypes.c_double, ctypes.c_double,
                                           ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                           ctypes.c_int, c_dp, c_dp, c_dp]
        lib.oracle_adam_update.restype = ctypes.c_int
        lib.oracle_spsa_update.argtypes = [c_dp, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                           ctypes.c_int, ctypes.c_double, ctypes.c_uint64,
                                           ctypes.c_uint64, c_dp, c_dp]
        lib.oracle_spsa_update.restype = ctypes.c_int
        lib.oracle_bptt_grad.argtypes = [c_dp, ctypes.c_int, ctypes.c_int, c_u8p, ctypes.c_int,
                                         ctypes.c_int, c_dp]
        lib.oracle_bptt_grad.restype = ctypes.c_double
        c_i32p = ctypes.POINTER(ctypes.c_int32)
        c_i = ctypes.c_int
        lib.oracle_body_param_count.argtypes = [c_i, c_i]
        lib.oracle_body_param_count.restype = ctypes.c_int64
        lib.oracle_body_gain_offset.argtypes = [c_i, c_i]
        lib.oracle_body_gain_offset.restype = ctypes.c_int64
        lib.oracle_body_probe.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint32,
                                          ctypes.c_uint32, c_i, c_i, c_i, ctypes.c_int64,
                                          ctypes.c_int64, ctypes.POINTER(ctypes.c_int8)]
        lib.oracle_body_probe.restype = c_i
        lib.oracle_body_loss.argtypes = [c_dp, c_i, c_i, c_dp, c_u8p, c_i, c_i, c_dp, c_i]
        lib.oracle_body_loss.restype = ctypes.c_double
        lib.oracle_body_spsa_losses.argtypes = [c_dp, c_i, c_i, c_i, c_i, c_dp, ctypes.c_double,
                                                c_i, ctypes.c_uint64, ctypes.c_uint64, c_u8p,
                                                c_i, c_i, c_i32p, c_i, c_dp, c_dp, c_i]
        lib.oracle_body_spsa_losses.restype = c_i
        lib.oracle_body_spsa_update.argtypes = [c_dp, c_i, c_i, c_i, c_i, c_i, ctypes.c_double,
                                                ctypes.c_uint64, ctypes.c_uint64, c_dp, c_dp]
        lib.oracle_body_spsa_update.restype = c_i
        lib.oracle_body_adam_update.argtypes = [c_dp, c_dp, c_dp, c_i, c_i, c_i, c_i, c_i,
                                                ctypes.c_uint64, ctypes.POINTER(ctypes.c_uint64),
                                                c_i, c_dp, ctypes.c_double, ctypes.c_double,
                                                ctypes.c_double, ctypes.c_double,
                                                ctypes.c_double, c_i, c_dp, c_dp, c_dp]
        lib.oracle_body_adam_update.restype = c_i
        _lib = lib
        return lib


def _ptr(a, ctype):
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def _f64(theta) -> np.ndarray:
    # fp32 -> fp64 widening is exact
    return np.ascontiguousarray(np.asarray(theta), dtype=np.float64)


def _u8(bytes_) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(bytes_), dtype=np.uint8)


def param_count(E: int, H: int) -> int:
    return int(_load().oracle_param_count(E, H))


def philox4x32_10(counter, key) -> np.ndarray:
    """Philox4x32-10 of one 4-word counter under a 2-word key (SC'11)."""
    ctr = np.ascontiguousarray(counter, dtype=np.uint32).reshape(4)
    k = np.ascontiguousarray(key, dtype=np.uint32).reshape(2)
    out = np.zeros(4, dtype=np.uint32)
    _load().oracle_philox4x32_10(_ptr(ctr, ctypes.c_uint32), _ptr(k, ctypes.c_uint32),
                                 _ptr(out, ctypes.c_uint32))
    return out


def rademacher(seed: int, step: int, expert: int, probe: int, p0: int, count: int) -> np.ndarray:
    """Probe entries z_{expert,probe}[p0 : p0+count] in {-1, +1} (int8)."""
    z = np.zeros(count, dtype=np.int8)
    _load().oracle_rademacher(seed, step, expert, probe, p0, count,
                              _ptr(z, ctypes.c_int8))
    return z


PROBE_KINDS = {"dense": 0, "sparse": 1}


def probe(seed: int, step: int, expert: int, probe_index: int, p0: int, count: int,
          kind: str = "dense") -> np.ndarray:
    """Probe entries z_{expert,probe}[p0 : p0+count] (int8): dense in {-1, +1},
    sparse in {-1, 0, +1} (App. E)."""
    z = np.zeros(count, dtype=np.int8)
    rc = _load().oracle_probe(seed, step, expert, probe_index, PROBE_KINDS[kind], p0, count,
                              _ptr(z, ctypes.c_int8))
    if rc != 0:
        raise RuntimeError(f"oracle_probe failed ({rc})")
    return z


def loss(theta, E: int, H: int, bytes_, n_threads: int = 0, per_token: bool = False):
    """Mean next-byte cross entropy (nats/byte) of ONE expert.

    theta: [P] parameters; bytes_: [B, T+1] uint8.  Returns the mean, or
    (mean, nll[B, T]) with per_token=True."""
    th = _f64(theta).reshape(-1)
    bx = _u8(bytes_)
    B, T1 = bx.shape
    T = T1 - 1
    assert th.size == param_count(E, H)
    nll = np.zeros((B, T), dtype=np.float64) if per_token else None
    m = _load().oracle_loss(_ptr(th, ctypes.c_double), E, H, _ptr(bx, ctypes.c_uint8), B, T,
                            _ptr(nll, ctypes.c_double) if per_token else None, n_threads)
    return (m, nll) if per_token else m


def spsa_losses(theta, E: int, H: int, eps: float, seed: int, step: int, bytes_,
                probes=None, n_pert: int | None = None, n_threads: int = 0,
                first_expert: int = 0, kind: str = "dense", batch_per_probe: bool = False,
                summed_loss: bool = False):
    """Antithetic losses and coefficients for the selected probes.

    theta [N, P] (fp32 or fp64), bytes_ [N, B, T+1] uint8.  ``probes`` lists
    the probe indices to evaluate (default: range(n_pert)).  ``eps`` is taken
    as given (pass np.float32 values to mirror the fp32 argument of the
    product).  Row e of theta is expert ``first_expert + e`` (the expert index
    keys its probes).  Returns (L [N, n_sel, 2] with L+ then L-, coef [N, n_sel])."""
    th = _f64(theta)
    N = th.shape[0]
    bx = _u8(bytes_)
    assert bx.shape[0] == N
    B, T = bx.shape[-2], bx.shape[-1] - 1
    n_total = bx.shape[1] if batch_per_probe else 0  # bytes [N, n_pert, B, T+1]
    if probes is None:
        probes = range(n_pert)
    sel = np.ascontiguousarray(list(probes), dtype=np.int32)
    L = np.zeros((N, sel.size, 2), dtype=np.float64)
    coef = np.zeros((N, sel.size), dtype=np.float64)
    rc = _load().oracle_spsa_losses_opts(_ptr(th, ctypes.c_double), N, first_expert, E, H,
                                    float(eps), PROBE_KINDS[kind], int(batch_per_probe),
                                    int(summed_loss), n_total, seed, step,
                                    _ptr(bx, ctypes.c_uint8), B, T,
                                    _ptr(sel, ctypes.c_int32), sel.size,
                                    _ptr(L, ctypes.c_double), _ptr(coef, ctypes.c_double),
                                    n_threads)
    if rc != 0:
        raise RuntimeError(f"oracle_spsa_losses failed ({rc})")
    return L, coef


def spsa_update(theta, E: int, H: int, lr: float, seed: int, step: int, coef) -> np.ndarray:
    """theta - lr * (1/n_pert) * sum_i coef[e, i] z_{e,i}, fp64 [N, P]."""
    th = _f64(theta)
    N = th.shape[0]
    cf = np.ascontiguousarray(coef, dtype=np.float64)
    n_pert = cf.shape[1]
    out = np.zeros_like(th)
    rc = _load().oracle_spsa_update(_ptr(th, ctypes.c_double), N, E, H, n_pert, float(lr), seed,
                                    step, _ptr(cf, ctypes.c_double), _ptr(out, ctypes.c_double))
    if rc != 0:
        raise RuntimeError(f"oracle_spsa_update failed ({rc})")
    return out


def spsa_step(theta, E: int, H: int, n_pert: int, eps: float, lr: float, seed: int, step: int,
              bytes_, n_threads: int = 0):
    """One full SPSA step: (L [N, n_pert, 2], coef [N, n_pert], theta' [N, P] fp64)."""
    L, coef = spsa_losses(theta, E, H, eps, seed, step, bytes_, n_pert=n_pert,
                          n_threads=n_threads)
    new = spsa_update(theta, E, H, lr, seed, step, coef)
    return L, coef, new


def adam_update(theta, m, v, E: int, H: int, seed: int, steps, coef, lr: float, beta1: float,
                beta2: float, delta: float, wd: float, t: int, kind: str = "sparse"):
    """The paper's optimizer step (Eq. localspsa with coupled weight decay).

    theta, m, v [N, P]; steps[A] the probe step counter of each accumulation
    batch; coef [A, N, n_pert].  Returns (theta', m', v') in fp64."""
    th = _f64(theta)
    mm = _f64(m)
    vv = _f64(v)
    N = th.shape[0]
    cf = np.ascontiguousarray(coef, dtype=np.float64)
    A, n_pert = cf.shape[0], cf.shape[2]
    st = np.ascontiguousarray(steps, dtype=np.uint64)
    assert st.size == A and cf.shape[1] == N
    to, mo, vo = np.zeros_like(th), np.zeros_like(th), np.zeros_like(th)
    rc = _load().oracle_adam_update(_ptr(th, ctypes.c_double), _ptr(mm, ctypes.c_double),
                                    _ptr(vv, ctypes.c_double), N, E, H, n_pert,
                                    PROBE_KINDS[kind], seed, _ptr(st, ctypes.c_uint64), A,
                                    _ptr(cf, ctypes.c_double), float(lr), float(beta1),
                                    float(beta2), float(delta), float(wd), int(t),
                                    _ptr(to, ctypes.c_double), _ptr(mo, ctypes.c_double),
                                    _ptr(vo, ctypes.c_double))
    if rc != 0:
        raise RuntimeError(f"oracle_adam_update failed ({rc})")
    return to, mo, vo


def mixture_nll(theta, E: int, H: int, requests, routes, t0: int, n_threads: int = 0):
    """Routed-inference NLL [R, T - t0] (Eq. main-mixture): requests [R, T+1]
    uint8, routes [R, k] expert indices into theta [N, P]."""
    th = _f64(theta)
    N = th.shape[0]
    rq = _u8(requests)
    R, T = rq.shape[0], rq.shape[1] - 1
    rt = np.ascontiguousarray(routes, dtype=np.int32)
    k = rt.shape[1]
    out = np.zeros((R, T - t0), dtype=np.float64)
    rc = _load().oracle_mixture_nll(_ptr(th, ctypes.c_double), N, E, H, _ptr(rq, ctypes.c_uint8),
                                    R, T, _ptr(rt, ctypes.c_int32), k, t0,
                                    _ptr(out, ctypes.c_double), n_threads)
    if rc != 0:
        raise RuntimeError(f"oracle_mixture_nll failed ({rc})")
    return out


def bptt_grad(theta, E: int, H: int, bytes_):
    """Exact batch gradient of the mean loss of ONE expert: (loss, grad [P])."""
    th = _f64(theta).reshape(-1)
    bx = _u8(bytes_)
    B, T = bx.shape[0], bx.shape[1] - 1
    g = np.zeros_like(th)
    m = _load().oracle_bptt_grad(_ptr(th, ctypes.c_double), E, H, _ptr(bx, ctypes.c_uint8), B, T,
                                 _ptr(g, ctypes.c_double))
    return m, g


# ---------------------------------------------------------------------------
# The paper's two-block expert body (body_oracle.c): D pre-norm residual
# blocks of width d (bias-free LSTM, then a GELU MLP of width 4d), gain-only
# LayerNorm, and a frozen tied head E [V, d] shared by every expert.
# Probe kinds: "dense" on every coordinate; "sparse" is the paper's training
# law (App. E): gains dense, every other coordinate sparse.
# ---------------------------------------------------------------------------

def body_param_count(d: int, D: int = 2) -> int:
    return int(_load().oracle_body_param_count(d, D))


def body_gain_offset(d: int, D: int = 2) -> int:
    return int(_load().oracle_body_gain_offset(d, D))


def body_probe(seed: int, step: int, expert: int, probe_index: int, d: int, D: int, p0: int,
               count: int, kind: str = "sparse") -> np.ndarray:
    """Body probe entries z[p0 : p0+count] (int8)."""
    z = np.zeros(count, dtype=np.int8)
    rc = _load().oracle_body_probe(seed, step, expert, probe_index, PROBE_KINDS[kind], d, D, p0,
                                   count, _ptr(z, ctypes.c_int8))
    if rc != 0:
        raise RuntimeError(f"oracle_body_probe failed ({rc})")
    return z


def body_loss(theta, d: int, D: int, head, bytes_, n_threads: int = 0,
              per_token: bool = False):
    """Mean next-byte cross entropy of ONE expert body: theta [P], head
    [V, d], bytes_ [B, T+1].  Returns the mean, or (mean, nll [B, T])."""
    th = _f64(theta).reshape(-1)
    hd = _f64(head)
    assert th.size == body_param_count(d, D) and hd.shape == (V, d)
    bx = _u8(bytes_)
    B, T = bx.shape[0], bx.shape[1] - 1
    nll = np.zeros((B, T), dtype=np.float64) if per_token else None
    m = _load().oracle_body_loss(_ptr(th, ctypes.c_double), d, D, _ptr(hd, ctypes.c_double),
                                 _ptr(bx, ctypes.c_uint8), B, T,
                                 _ptr(nll, ctypes.c_double) if per_token else None, n_threads)
    return (m, nll) if per_token else m


def body_spsa_losses(theta, d: int, D: int, head, eps: float, seed: int, step: int, bytes_,
                     probes=None, n_pert: int | None = None, kind: str = "sparse",
                     first_expert: int = 0, n_threads: int = 0):
    """Antithetic losses and coefficients of the selected probes of N expert
    bodies: theta [N, P], bytes_ [N, B, T+1].  Returns (L [N, n_sel, 2],
    coef [N, n_sel])."""
    th = _f64(theta)
    N = th.shape[0]
    hd = _f64(head)
    bx = _u8(bytes_)
    assert bx.shape[0] == N and hd.shape == (V, d)
    B, T = bx.shape[1], bx.shape[2] - 1
    if probes is None:
        probes = range(n_pert)
    sel = np.ascontiguousarray(list(probes), dtype=np.int32)
    L = np.zeros((N, sel.size, 2), dtype=np.float64)
    coef = np.zeros((N, sel.size), dtype=np.float64)
    rc = _load().oracle_body_spsa_losses(_ptr(th, ctypes.c_double), N, first_expert, d, D,
                                         _ptr(hd, ctypes.c_double), float(eps),
                                         PROBE_KINDS[kind], seed, step, _ptr(bx, ctypes.c_uint8),
                                         B, T, _ptr(sel, ctypes.c_int32), sel.size,
                                         _ptr(L, ctypes.c_double), _ptr(coef, ctypes.c_double),
                                         n_threads)
    if rc != 0:
        raise RuntimeError(f"oracle_body_spsa_losses failed ({rc})")
    return L, coef


def body_spsa_update(theta, d: int, D: int, lr: float, seed: int, step: int, coef,
                     kind: str = "sparse") -> np.ndarray:
    """theta - lr (1/n_pert) sum_i coef[e, i] z_{e,i}, fp64 [N, P]."""
    th = _f64(theta)
    N = th.shape[0]
    cf = np.ascontiguousarray(coef, dtype=np.float64)
    out = np.zeros_like(th)
    rc = _load().oracle_body_spsa_update(_ptr(th, ctypes.c_double), N, d, D, cf.shape[1],
                                         PROBE_KINDS[kind], float(lr), seed, step,
                                         _ptr(cf, ctypes.c_double), _ptr(out, ctypes.c_double))
    if rc != 0:
        raise RuntimeError(f"oracle_body_spsa_update failed ({rc})")
    return out


def body_adam_update(theta, m, v, d: int, D: int, seed: int, steps, coef, lr: float,
                     beta1: float, beta2: float, delta: float, wd: float, t: int,
                     kind: str = "sparse"):
    """Eq. localspsa on the body coordinates: (theta', m', v') in fp64."""
    th, mm, vv = _f64(theta), _f64(m), _f64(v)
    N = th.shape[0]
    cf = np.ascontiguousarray(coef, dtype=np.float64)
    A, n_pert = cf.shape[0], cf.shape[2]
    st = np.ascontiguousarray(steps, dtype=np.uint64)
    assert st.size == A and cf.shape[1] == N
    to, mo, vo = np.zeros_like(th), np.zeros_like(th), np.zeros_like(th)
    rc = _load().oracle_body_adam_update(_ptr(th, ctypes.c_double), _ptr(mm, ctypes.c_double),
                                         _ptr(vv, ctypes.c_double), N, d, D, n_pert,
                                         PROBE_KINDS[kind], seed, _ptr(st, ctypes.c_uint64), A,
                                         _ptr(cf, ctypes.c_double), float(lr), float(beta1),
                                         float(beta2), float(delta), float(wd), int(t),
                                         _ptr(to, ctypes.c_double), _ptr(mo, ctypes.c_double),
                                         _ptr(vo, ctypes.c_double))
    if rc != 0:
        raise RuntimeError(f"oracle_body_adam_update failed ({rc})")
    return to, mo, vo
