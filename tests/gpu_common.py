"""Helpers of the GPU parity tests: run the CUDA path through the C ABI and
compare with the oracle at the stated tolerances.

Tolerances (GPU against the fp64 oracle):
  losses L+, L-        |delta| <= 2e-4 nats/byte
  coefficients         ||delta||_2 <= 1e-2 ||c||_2 per expert, and every
                       |delta_i| <= 1e-2 max(|c_i|, rms(c)) (the rms floor
                       keeps a coefficient that happens to be near zero from
                       demanding an absolute accuracy no other one needs)
  updated theta        relative L2 <= 1e-5 against the oracle's own step;
                       <= 2e-6 against the oracle update applied to the
                       GPU's own coefficients (isolates the update kernel)
  Philox words, z      bit-exact
"""
import numpy as np
import torch

TOL_LOSS = 2e-4
TOL_COEF = 1e-2
TOL_THETA = 1e-5
TOL_THETA_GIVEN_COEF = 2e-6


def api():
    from paper_2609_37899_gb300 import api as a
    return a


def run_step(theta, bytes_, E, H, n_pert, eps, lr, seed, step, with_coef=True):
    a = api()
    N = theta.shape[0]
    B, T1 = bytes_.shape[1], bytes_.shape[2]
    params = torch.from_numpy(np.ascontiguousarray(theta, dtype=np.float32)).cuda()
    bx = torch.from_numpy(np.ascontiguousarray(bytes_)).cuda()
    ws = a.alloc_workspace(E, H, N, n_pert, B, T1 - 1)
    losses = torch.full((N, n_pert, 2), float("nan"), device="cuda")
    coef = torch.full((N, n_pert), float("nan"), device="cuda") if with_coef else None
    a.spsa_step(params, bx, E, H, n_pert, float(eps), float(lr), seed, step, losses, coef, ws)
    status = a.get_status()
    return dict(theta=params.cpu().numpy(), losses=losses.cpu().numpy(),
                coef=coef.cpu().numpy() if with_coef else None, status=status)


def run_eval(theta, bytes_, E, H):
    a = api()
    N = theta.shape[0]
    B, T1 = bytes_.shape[1], bytes_.shape[2]
    params = torch.from_numpy(np.ascontiguousarray(theta, dtype=np.float32)).cuda()
    bx = torch.from_numpy(np.ascontiguousarray(bytes_)).cuda()
    ws = a.alloc_workspace(E, H, N, 1, B, T1 - 1)
    out = torch.full((N,), float("nan"), device="cuda")
    a.eval_loss(params, bx, E, H, out, ws)
    assert a.get_status() == 0
    return out.cpu().numpy()


def rel_l2(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / np.linalg.norm(b))


def report(kind, value):
    """Achieved error, printed for `pytest -s`: one line per parity check,
    so the margin of every tolerance can be read off a run."""
    print(f"PARITY {kind} {value:.3e}")


def assert_losses(gpu, ref):
    err = np.abs(np.asarray(gpu, np.float64) - ref).max()
    report("loss_abs", err)
    assert err <= TOL_LOSS, f"loss error {err:.3e} > {TOL_LOSS}"


def assert_coefs(gpu, ref):
    gpu = np.asarray(gpu, np.float64)
    for e in range(ref.shape[0]):
        r = ref[e]
        d = np.abs(gpu[e] - r)
        rms = np.sqrt(np.mean(r ** 2))
        report("coef_rel_l2", np.linalg.norm(d) / np.linalg.norm(r))
        assert np.linalg.norm(d) <= TOL_COEF * np.linalg.norm(r), \
            f"expert {e}: coefficient error {np.linalg.norm(d) / np.linalg.norm(r):.3e}"
        assert np.all(d <= TOL_COEF * np.maximum(np.abs(r), rms)), \
            f"expert {e}: worst coefficient error {np.max(d / np.maximum(np.abs(r), rms)):.3e}"
