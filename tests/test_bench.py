"""The benchmark's host-side arithmetic and its reference arm (CPU only).

- The algorithmic flop counts that the roofline lines divide by, checked
  against the GEMM shapes they stand for.
- The traffic figures' source hashes: comments do not change them, and code
  does.
- `--impl reference` (the oracle on the host cores) prints one JSON line with
  the contract's keys.
"""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2609_37899_gb300 import inputs  # noqa: E402


def test_gate_flops_are_the_gate_gemm():
    c = inputs.CONFIGS["soma_n2"]
    # per (expert, probe, sign) lane and timestep: [B, E+H] x [E+H, 4H]
    lanes = c["n_experts"] * c["n_pert"] * 2
    per_lane = 2 * c["batch"] * (c["E"] + c["H"]) * 4 * c["H"]
    assert bench.gate_flops_per_timestep(c) == lanes * per_lane
    assert bench.gate_flops_per_timestep(c) == 64_424_509_440


def test_body_flops_per_token():
    c = inputs.BODY_CONFIGS["body_n256"]
    d, D = c["d"], c["D"]
    gates = 2 * (2 * d) * (4 * d)          # [u | h] x [2d, 4d]
    mlp = 2 * d * (4 * d) + 2 * (4 * d) * d
    decode = 2 * d * 256
    assert bench.body_flops_per_token(c) == D * (gates + mlp) + decode == 81_920


def test_tokens_per_step():
    c = inputs.CONFIGS["soma_n2"]
    assert bench.tokens_per_step(c) == 2 * 2 * 64 * 32 * 256 == 2_097_152


def test_source_hash_ignores_comments_only(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2609_37899_gb300" / "csrc"
    csrc.mkdir(parents=True)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    f = csrc / "k.cu"
    f.write_text("// a kernel\n__global__ void k(int* x) { x[0] = 1; }\n")
    h0 = bench.source_hash(["k.cu"])
    f.write_text("/* reworded\n   comment */\n__global__ void k(int* x) { x[0] = 1; }  // ok\n\n")
    assert bench.source_hash(["k.cu"]) == h0
    f.write_text("__global__ void k(int* x) { x[0] = 2; }\n")
    assert bench.source_hash(["k.cu"]) != h0


def test_traffic_entries_name_existing_sources():
    for name, t in bench.TRAFFIC.items():
        for f in t["files"]:
            assert os.path.exists(os.path.join(ROOT, "paper_2609_37899_gb300", "csrc", f)), (name, f)
        assert t.get("bytes_per_launch", t.get("bytes_per_phase", 0)) > 0


def test_per_phase_traffic_scales_with_the_phases_of_a_launch(monkeypatch):
    monkeypatch.setattr(bench, "TRAFFIC", {
        "a": {"bytes_per_phase": 10.0, "files": ["forward_tc.cu"],
              "source_hash": bench.source_hash(["forward_tc.cu"])},
        "b": {"bytes_per_launch": 7.0, "files": ["forward_tc.cu"], "source_hash": "stale"}})
    assert bench.launch_traffic("a", 16) == 170.0
    assert bench.launch_traffic("b", 16) is None
    assert bench.launch_traffic("missing", 16) is None


def test_clock_sampler_without_nvidia_smi(monkeypatch):
    def no_smi(*a, **k):
        raise OSError("no nvidia-smi")
    monkeypatch.setattr(bench.subprocess, "Popen", no_smi)
    with bench.ClockSampler(0) as clk:
        pass
    assert clk.summary() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}


@pytest.mark.parametrize("config", ["tiny", "body_tiny"])
def test_reference_arm_prints_the_contract_line(config):
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--config", config, "--steps", "1", "--warmup", "1",
                          "--ref-sample-seqs", "2"],
                         capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr
    lines = [l for l in out.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0
    for k in ("metric", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
