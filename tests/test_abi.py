"""The C ABI library builds, loads and exports every declared symbol; host
argument validation needs no GPU (no compute call is made here)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "soma_api.h")


@pytest.fixture(scope="module")
def soma():
    from paper_2609_37899_gb300 import build
    build.build()
    from paper_2609_37899_gb300 import api
    return api


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(soma_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_entry_points():
    names = declared_functions()
    for required in ["soma_init_experts", "soma_spsa_step", "soma_eval_loss",
                     "soma_workspace_bytes", "soma_param_count", "soma_get_status",
                     "soma_status_string", "soma_spsa_update", "soma_debug_philox",
                     "soma_debug_rademacher", "soma_spsa_estimate", "soma_adam_update",
                     "soma_debug_probe", "soma_spsa_estimate_opts", "soma_mixture_nll",
                     "soma_mixture_workspace_bytes", "soma_body_param_count",
                     "soma_body_workspace_bytes", "soma_body_spsa_estimate",
                     "soma_body_spsa_step", "soma_body_eval_loss", "soma_body_adam_update",
                     "soma_debug_body_probe"]:
        assert required in names


def test_library_exports_every_declared_symbol(soma):
    lib = ctypes.CDLL(soma.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_param_count_and_workspace(soma):
    assert soma.param_count(32, 64) == 49_664
    assert soma.param_count(64, 960) == 4_198_400
    assert soma.param_count(32, 48) == 36_288
    assert soma.lib().soma_param_count(soma.soma_dims(255, 32, 64)) == -1
    assert soma.workspace_bytes(32, 64, 1, 8, 4, 64) > 0
    assert soma.workspace_bytes(32, 64, 0, 8, 4, 64) == 0
    assert soma.workspace_bytes(32, 64, 1, 0, 4, 64) == 0
    # grows with every size it depends on
    w = soma.workspace_bytes(64, 960, 2, 64, 32, 256)
    assert soma.workspace_bytes(64, 960, 2, 64, 32, 512) > w
    assert soma.workspace_bytes(64, 960, 2, 128, 32, 256) > w


def test_status_strings(soma):
    for code in range(7):
        assert soma.status_string(code) != "unknown status"
    assert soma.status_string(99) == "unknown status"


def test_host_validation_rejects_before_launch(soma):
    L = soma.lib()
    d = soma.dims(32, 64)
    fake = ctypes.c_void_p(0x10000)  # never dereferenced: validation fails first
    ws = soma.workspace_bytes(32, 64, 1, 8, 4, 64)
    # null params
    assert L.soma_spsa_step(None, 1, d, 8, 1e-3, 1e-2, 0, 0, fake, 4, 64, fake, None, fake, ws,
                            None) == 1
    # misaligned params
    assert L.soma_spsa_step(ctypes.c_void_p(0x10004), 1, d, 8, 1e-3, 1e-2, 0, 0, fake, 4, 64,
                            fake, None, fake, ws, None) == 1
    # negative / non-finite eps, non-finite lr
    assert L.soma_spsa_step(fake, 1, d, 8, -1e-3, 1e-2, 0, 0, fake, 4, 64, fake, None, fake, ws,
                            None) == 1
    assert L.soma_spsa_step(fake, 1, d, 8, float("nan"), 1e-2, 0, 0, fake, 4, 64, fake, None,
                            fake, ws, None) == 1
    assert L.soma_spsa_step(fake, 1, d, 8, 1e-3, float("inf"), 0, 0, fake, 4, 64, fake, None,
                            fake, ws, None) == 1
    # bad dims
    assert L.soma_spsa_step(fake, 1, soma.soma_dims(128, 32, 64), 8, 1e-3, 1e-2, 0, 0, fake, 4,
                            64, fake, None, fake, ws, None) == 2
    assert L.soma_spsa_step(fake, 1, soma.dims(32, 5000), 8, 1e-3, 1e-2, 0, 0, fake, 4, 64,
                            fake, None, fake, ws, None) == 2
    # zero sizes, too many probes
    assert L.soma_spsa_step(fake, 0, d, 8, 1e-3, 1e-2, 0, 0, fake, 4, 64, fake, None, fake, ws,
                            None) == 1
    assert L.soma_spsa_step(fake, 1, d, 20000, 1e-3, 1e-2, 0, 0, fake, 4, 64, fake, None, fake,
                            ws, None) == 1
    # workspace too small or missing
    assert L.soma_spsa_step(fake, 1, d, 8, 1e-3, 1e-2, 0, 0, fake, 4, 64, fake, None, fake,
                            ws - 1, None) == 3
    assert L.soma_spsa_step(fake, 1, d, 8, 1e-3, 1e-2, 0, 0, fake, 4, 64, fake, None, None, ws,
                            None) == 3
    assert L.soma_eval_loss(fake, 1, d, fake, 4, 64, fake, fake, 16, None) == 3
    assert L.soma_init_experts(fake, 1, d, 0, -1.0, None) == 1
    assert L.soma_spsa_update(fake, 1, d, 8, float("nan"), 0, 0, fake, None) == 1
    assert L.soma_debug_rademacher(0, 0, 0, 0, -1, 4, fake, None) == 1
    # the optimizer step's entry points
    est = (fake, 1, d, 8)
    assert L.soma_spsa_estimate(*est, 2, 1e-3, 0, 0, fake, 4, 64, fake, fake, fake, ws,
                                None) == 1  # unknown probe kind
    assert L.soma_spsa_estimate(*est, 1, 1e-3, 0, 0, fake, 4, 64, fake, None, fake, ws,
                                None) == 1  # coef_out is required
    cfg = soma.soma_adam_config(1e-3, 0.9, 0.999, 1e-8, 1e-4, 1)
    steps = (ctypes.c_uint64 * 2)(0, 1)
    assert L.soma_adam_update(fake, fake, fake, 1, d, 8, 1, 0, steps, 0, fake, cfg,
                              None) == 1  # n_acc = 0
    assert L.soma_adam_update(fake, fake, fake, 1, d, 8, 1, 0, steps, 65, fake, cfg,
                              None) == 1  # n_acc > SOMA_MAX_ACCUM
    assert L.soma_adam_update(fake, fake, fake, 1, d, 8, 1, 0, None, 2, fake, cfg, None) == 1
    for bad in (soma.soma_adam_config(1e-3, 1.0, 0.999, 1e-8, 0.0, 1),
                soma.soma_adam_config(1e-3, 0.9, 0.999, 0.0, 0.0, 1),
                soma.soma_adam_config(1e-3, 0.9, 0.999, 1e-8, -1.0, 1),
                soma.soma_adam_config(1e-3, 0.9, 0.999, 1e-8, 0.0, 0)):
        assert L.soma_adam_update(fake, fake, fake, 1, d, 8, 1, 0, steps, 2, fake, bad,
                                  None) == 1
    assert L.soma_debug_probe(0, 0, 0, 0, 3, 0, 4, fake, None) == 1
    # routed inference: routes are checked on the host
    bad = (ctypes.c_int32 * 2)(0, 5)
    assert L.soma_mixture_workspace_bytes(d, 2, bad, 1, 2, 8) == 0
    assert L.soma_mixture_nll(fake, 2, d, fake, 1, 8, bad, 2, 0, fake, fake, 1 << 20, None) == 1
    good = (ctypes.c_int32 * 2)(0, 1)
    assert L.soma_mixture_nll(fake, 2, d, fake, 1, 8, good, 2, 8, fake, fake, 1 << 20,
                              None) == 1  # t0 = seq_len
    assert L.soma_mixture_nll(fake, 2, d, fake, 1, 8, good, 17, 0, fake, fake, 1 << 20,
                              None) == 1  # k > 16


def test_body_sizes_and_validation(soma):
    """The expert body's entry points: sizes and host-side rejection (no launch)."""
    L = soma.lib()
    assert soma.body_param_count(32, 2) == 32 * 32 * 32 + 5 * 32 == 32_928
    assert soma.body_param_count(32, 1) == 16 * 32 * 32 + 3 * 32
    for bad in ((16, 2), (32, 3), (32, 0)):
        assert soma.body_param_count(*bad) == -1
    assert L.soma_body_param_count(soma.soma_body_dims(255, 32, 2)) == -1
    w = soma.body_workspace_bytes(32, 2, 256, 64, 16, 512)
    assert w >= 256 * 64 * 2 * 8 + 256 * 64 * 4
    assert soma.body_workspace_bytes(32, 2, 256, 64, 17, 512) > w  # a second chunk
    assert soma.body_workspace_bytes(32, 2, 0, 64, 16, 512) == 0
    d = soma.body_dims(32, 2)
    fake = ctypes.c_void_p(0x10000)
    ws = 1 << 20
    # unsupported dims, bad kind, negative eps, missing coefficients, workspace
    assert L.soma_body_spsa_step(fake, 1, soma.soma_body_dims(256, 16, 2), fake, 4, 1, 1e-3,
                                 1e-3, 0, 0, fake, 4, 8, fake, fake, fake, ws, None) == 2
    assert L.soma_body_spsa_step(fake, 1, d, fake, 4, 2, 1e-3, 1e-3, 0, 0, fake, 4, 8, fake,
                                 fake, fake, ws, None) == 1
    assert L.soma_body_spsa_step(fake, 1, d, fake, 4, 1, -1e-3, 1e-3, 0, 0, fake, 4, 8, fake,
                                 fake, fake, ws, None) == 1
    assert L.soma_body_spsa_step(fake, 1, d, None, 4, 1, 1e-3, 1e-3, 0, 0, fake, 4, 8, fake,
                                 fake, fake, ws, None) == 1  # no head
    assert L.soma_body_spsa_estimate(fake, 1, d, fake, 4, 1, 1e-3, 0, 0, fake, 4, 8, fake, None,
                                     fake, ws, None) == 1
    assert L.soma_body_spsa_step(fake, 1, d, fake, 4, 1, 1e-3, 1e-3, 0, 0, fake, 4, 8, fake,
                                 fake, fake, 16, None) == 3
    assert L.soma_body_eval_loss(fake, 1, d, fake, fake, 4, 8, fake, fake, 16, None) == 3
    assert L.soma_body_eval_loss(fake, 1, d, fake, fake, 0, 8, fake, fake, ws, None) == 1
    cfg = soma.soma_adam_config(1e-3, 0.9, 0.999, 1e-8, 1e-4, 0)  # t = 0
    steps = (ctypes.c_uint64 * 1)(0)
    assert L.soma_body_adam_update(fake, fake, fake, 1, d, 4, 1, 0, steps, 1, fake, cfg,
                                   None) == 1
    assert L.soma_debug_body_probe(0, 0, 0, 0, d, 1, -1, 4, fake, None) == 1
    assert L.soma_debug_wait_timeout(0, None) == 1
    assert L.soma_debug_wait_timeout((1 << 22) + 1, None) == 1
    assert L.soma_debug_body_probe(0, 0, 0, 0, d, 1, 1 << 30, 4, fake, None) == 1
