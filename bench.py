#!/usr/bin/env python3
"""Throughput of the SOMA SPSA training step on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl ours|reference]

One step = one call of soma_spsa_step: for every expert and each of its n_pert
probes, the antithetic forward passes of the whole byte-LSTM recurrence at
theta +- eps z over the expert's batch, the per-pass mean cross entropy, the
coefficients and the Philox-regenerating update.  The default workload is the
SOMA N=2 configuration: 2 experts (E=64, H=960, 4,198,400 parameters each),
64 probes, 32 sequences x 256 target bytes per expert, eps = lr = 1e-3.

Prints ONE JSON line (rank 0).  `value` is perturbed LSTM tokens/s over all
ranks (tokens/step = N_experts * 2 * n_pert * B * T per rank), inputs resident
in HBM; `e2e` is the same metric through the public API with the step's bytes
copied from pinned host memory and the losses read back inside the timed
region.  With torchrun (N > 1) every rank steps its own independent set of
experts (no collective on the data path: experts never exchange anything),
so scaling is weak.  `--impl reference` times the fp64 CPU oracle on the
host cores instead (rank 0 only), on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "perturbed LSTM tokens/s & SPSA steps/s per GB300; % of GEMM/HBM roofline"
UNIT = "perturbed tokens/s"

# DRAM traffic of one launch of the dominant kernel from an ncu capture
# (dram__bytes_read.sum + dram__bytes_write.sum), valid only for the kernel
# source it was taken on.
TRAFFIC = {
    # profiles/tc_persistent_kernel_soma_n2.md: one persistent launch of the
    # SOMA N=2 shapes at T=16 (17 phases) captured; per phase, scaled by the
    # T + 1 phases of a launch
    "soma_n2": {"bytes_per_phase": (2194.885e6 + 869.94816e6) / 17,
                "files": ["forward_tc.cu", "tc_primitives.cuh", "soma_device.cuh"],
                "source_hash": "97f08f55d5cc3326"},
    # profiles/res_kernel_soma_n256.md: one full-size launch (T=512)
    "soma_n256": {"bytes_per_launch": 39.452672e6 + 2048,
                  "files": ["resident.cu", "tc_primitives.cuh", "soma_device.cuh"],
                  "source_hash": "7cc9de59fd25da8c"},
    # profiles/body_tc_kernel_body_n256.md: one full-size launch (T=512)
    "body_n256": {"bytes_per_launch": 36.546304e6,
                  "files": ["body_tc.cu", "body_device.cuh", "tc_primitives.cuh",
                            "soma_device.cuh"],
                  "source_hash": "aed1fa16ae461890"},
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default="soma_n2")
    ap.add_argument("--seq-len", type=int, default=None,
                    help="override the workload's sequence length (small profiling cases)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--optimizer", default="sgd", choices=["sgd", "adam"],
                    help="sgd: the SPSA step of Eq. main-spsa (dense probes); adam: the "
                         "paper's optimizer step (Eq. localspsa: --accum estimates, then Adam)")
    ap.add_argument("--probes", default=None, choices=["dense", "sparse"],
                    help="probe kind of --optimizer adam (default sparse, as the paper)")
    ap.add_argument("--accum", type=int, default=1,
                    help="accumulation batches per --optimizer adam update")
    ap.add_argument("--batch-per-probe", action="store_true",
                    help="--optimizer adam: an independent batch for every probe (App. D)")
    ap.add_argument("--summed-loss", action="store_true",
                    help="--optimizer adam: the control arm that sums the experts' losses "
                         "before each finite difference (App. D)")
    ap.add_argument("--inference", action="store_true",
                    help="routed inference (Eq. main-mixture) on the workload's experts instead "
                         "of a training step: --requests requests of seq_len bytes, k = min(4, N) "
                         "random routes each, the last 3/4 of the positions scored")
    ap.add_argument("--requests", type=int, default=4096)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample-seqs", type=int, default=32,
                    help="sequences in the one-probe sample of the cpu_baseline timing")
    ap.add_argument("--ref-sample-seqs", type=int, default=8,
                    help="sequences per step of the --impl reference oracle run")
    return ap.parse_args()


def workload_desc(name, c):
    from paper_2609_37899_gb300 import inputs
    P = inputs.param_count(c["E"], c["H"])
    return (f"{name}: {c['n_experts']} expert(s) x 1-layer byte LSTM (E={c['E']}, H={c['H']}, "
            f"P={P:,}), n_pert={c['n_pert']}, eps={c['eps']}, lr={c['lr']}, "
            f"B={c['batch']} x T={c['seq_len']} bytes per expert, order-{c['order']} "
            f"Zipf(1.1) Markov clusters")


def tokens_per_step(c):
    return c["n_experts"] * 2 * c["n_pert"] * c["batch"] * c["seq_len"]


# fp16 tensor-core operands with fp32 accumulation; gates, cell, softmax,
# losses and the update in fp32 (loss sums in fp64)
DTYPE = "f16/f32"


def gate_kernel_name(B, resident):
    if resident:
        return ("res_kernel (tcgen05, the whole recurrence of a probe pair resident in one CTA: "
                "gate GEMM + cell + head + loss)")
    return ("tc_persistent_kernel (tcgen05; one cooperative launch per sweep, phase t = "
            "gate GEMM + fused cell of timestep t and output head + softmax partials of t - 1)")


def gate_flops_per_timestep(c):
    # one timestep of every (expert, probe, sign) lane: [B, E+H] x [E+H, 4H]
    # per lane, 2 flops per multiply-add (the direct form's algorithmic count)
    return c["n_experts"] * c["n_pert"] * 2 * c["batch"] * 8 * c["H"] * (c["E"] + c["H"])


def head_flops_per_timestep(c):
    # the output head of one timestep of every lane: [B, H] x [H, 256]
    return c["n_experts"] * c["n_pert"] * 2 * c["batch"] * 2 * 256 * c["H"]


def applicable_peak(peaks, clocks):
    """The burst bf16 peak applies when the sampled SM clock sat at its
    maximum with no power cap (the burst figure was measured that way); the
    sustained one otherwise (it was measured under the power cap)."""
    sm, mx = clocks.get("sm_mhz"), clocks.get("sm_max_mhz")
    at_max = sm is not None and mx is not None and sm >= 0.97 * mx
    if at_max and "sw_power_cap" not in clocks.get("reasons", []):
        return "burst", peaks["bf16_tflops"]
    return "sustained", peaks["bf16_tflops_sustained"]


def shard_seeds(rank):
    """Seeds of rank `rank`'s shard.  The parameter init, the data and the
    probe streams all differ between ranks, so N ranks step N disjoint sets of
    experts with no data-path collective (weak scaling)."""
    return {"init": 1000 + rank, "data": rank, "probe": rank}


def max_over_ranks(dist, values, device=None):
    """Timings reduced with MAX over the ranks: the slowest rank sets the
    job's time.  The identity without a process group."""
    if dist is None:
        return [float(v) for v in values]
    import torch
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons every 50 ms while running.  The
    sampler is started and its first sample awaited before the timed region,
    and only the samples taken after that count."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def _read(self):
        for line in self.proc.stdout:
            if line.strip():
                self._all.append((time.monotonic(), line))
                self._first.set()

    def __enter__(self):
        self._all = []
        self._first = threading.Event()
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return self
        self._reader = threading.Thread(target=self._read, daemon=True)
        self._reader.start()
        self._first.wait(timeout=5.0)
        self._t0 = time.monotonic()
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.proc.wait()
            self._reader.join(timeout=5)
            self.lines = [l for (t, l) in self._all if t >= self._t0]

    def summary(self):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "lines", []):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


def cpu_baseline(cfg_name, c, n_seqs, kind="dense"):
    """The fp64 oracle, as it stands, on the host cores: one probe pair of
    expert 0 over `n_seqs` of its sequences (both signs)."""
    import oracle
    from paper_2609_37899_gb300 import inputs
    theta = inputs.config_params(cfg_name)[:1]
    bx = inputs.config_batch(cfg_name)[:1, :n_seqs]
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    oracle.build()
    t0 = time.perf_counter()
    oracle.spsa_losses(theta, c["E"], c["H"], np.float32(c["eps"]), 0, 0, bx, probes=[0],
                       n_threads=cores, kind=kind)
    dt = time.perf_counter() - t0
    toks = 2 * n_seqs * c["seq_len"]
    return {"value": toks / dt, "unit": UNIT, "cores": min(cores, n_seqs), "kind": "oracle",
            "sample": f"expert 0, {kind} probe 0, both signs, {n_seqs} of {c['batch']} sequences x "
                      f"{c['seq_len']} bytes ({toks} perturbed tokens) in {dt:.2f} s; OpenMP "
                      f"over sequences, so {min(cores, n_seqs)} of {cores} cores busy"}


def reference_arm(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import oracle
    from paper_2609_37899_gb300 import inputs
    c = inputs.CONFIGS[args.config]
    n_seqs = min(args.ref_sample_seqs, c["batch"])
    theta = inputs.config_params(args.config)
    bx = inputs.config_batch(args.config)
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    oracle.build()

    def one(k):
        e = k % c["n_experts"]
        i = k % c["n_pert"]
        oracle.spsa_losses(theta[e:e + 1], c["E"], c["H"], np.float32(c["eps"]), 0, 0,
                           bx[e:e + 1, :n_seqs], probes=[i], n_threads=cores, first_expert=e)

    for k in range(args.warmup):
        one(k)
    t0 = time.perf_counter()
    for k in range(args.steps):
        one(args.warmup + k)
    dt = time.perf_counter() - t0
    toks = 2 * n_seqs * c["seq_len"]
    value = toks * args.steps / dt
    sample = (f"per step one probe pair (both signs) of one expert over {n_seqs} of "
              f"{c['batch']} sequences x {c['seq_len']} bytes = {toks} perturbed tokens")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload_desc(args.config, c), "sample": sample},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": min(cores, n_seqs),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def source_hash(files):
    """Hash of the sources a traffic figure was measured on, comments and
    blank lines left out (an edited comment does not change the kernel)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_37899_gb300", "csrc")
    for f in files:
        with open(os.path.join(csrc, f), encoding="utf-8") as fh:
            text = fh.read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        text = re.sub(r"//[^\n]*", "", text)
        code = "\n".join(line.rstrip() for line in text.splitlines() if line.strip())
        h.update(code.encode())
    return h.hexdigest()[:16]


def launch_traffic(config, T):
    """DRAM bytes of one launch of the dominant kernel at sequence length T,
    or None when the sources changed since the capture.  A per-phase figure
    scales to the T + 1 phases of one persistent launch."""
    tr = TRAFFIC.get(config)
    if not tr or tr["source_hash"] != source_hash(tr["files"]):
        return None
    if "bytes_per_phase" in tr:
        return tr["bytes_per_phase"] * (T + 1)
    return tr["bytes_per_launch"]


def our_arm(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    from paper_2609_37899_gb300 import api, build, inputs
    if not os.path.exists(api.LIB_PATH):
        build.build()
    c = dict(inputs.CONFIGS[args.config])
    if args.seq_len:
        c["seq_len"] = args.seq_len
    N, E, H, n, B, T = c["n_experts"], c["E"], c["H"], c["n_pert"], c["batch"], c["seq_len"]
    K, W = args.steps, args.warmup
    adam = args.optimizer == "adam"
    A = args.accum if adam else 1
    kind = (args.probes or "sparse") if adam else "dense"
    if not 1 <= A <= api.MAX_ACCUM:
        raise SystemExit(f"--accum must be in 1..{api.MAX_ACCUM}")
    seeds = shard_seeds(rank)
    experts = api.SomaExperts(N, E, H, n, B, T, device=dev)
    experts.init(seed=seeds["init"], std=c["init_std"] or 0.0)
    # every step gets its own A batches: (W + K) A host batches, pinned, and
    # their HBM-resident copies for the device-timed run
    per_probe = adam and args.batch_per_probe
    summed = adam and args.summed_loss

    def host_batch(k):
        if not per_probe:
            return torch.from_numpy(inputs.config_batch(args.config, seed=seeds["data"], step=k,
                                                        seq_len=c["seq_len"])).pin_memory()
        # [N, n, B, T+1]: probe i of batch k draws its own sequences
        return torch.from_numpy(np.stack(
            [inputs.config_batch(args.config, seed=seeds["data"], step=k * n + i,
                                 seq_len=c["seq_len"])
             for i in range(n)], axis=1)).pin_memory()

    host = [[host_batch(A * s + a) for a in range(A)] for s in range(W + K)]
    resident = [[h.to(dev) for h in hs] for hs in host]

    def do_step(batches, s):
        """One step: the SGD step, or A estimates plus the Adam update t = s + 1
        (App. E hyper-parameters: beta 0.9 / 0.999, delta 1e-8, decay 1e-4)."""
        if not adam:
            return experts.step(batches[0], c["eps"], c["lr"], seeds["probe"], s)[0]
        losses, _ = experts.adam_step(batches, c["eps"], seeds["probe"],
                                      [A * s + a for a in range(A)],
                                      t=s + 1, lr=c["lr"], kind=kind,
                                      batch_per_probe=per_probe, summed_loss=summed)
        return losses
    stream = torch.cuda.current_stream(dev)
    # written between timed steps so that no step starts with the previous
    # step's data in L2 (129 MB)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize(dev)

    for s in range(W):
        do_step(resident[s], s)
    barrier()
    # the timed region: tracing off, so no event is recorded between launches
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        barrier()
        start.record(stream)
        for s in range(K):
            flush.fill_(s & 0xFF)
            do_step(resident[W + s], W + s)
        stop.record(stream)
        barrier()
    ms = start.elapsed_time(stop)
    status = api.get_status()

    # a second pass of the same K steps with the library's trace hooks on: the
    # per-kernel device time (CUDA events on the launching stream around every
    # launch) for kernel_ms and the roofline
    api.trace_enable(True)
    api.trace_read(reset=True)
    barrier()
    for s in range(K):
        flush.fill_(s & 0xFF)
        do_step(resident[W + s], W + s)
    barrier()
    api.trace_enable(False)
    traced = api.trace_read(reset=True)

    # end to end through the public API: H2D of the step's bytes, the step,
    # D2H of its losses, every step
    losses_host = torch.empty(A, N, n, 2, dtype=torch.float32).pin_memory()
    dev_bytes = [torch.empty_like(r) for r in resident[0]]
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for s in range(K):
        flush.fill_(s & 0xFF)
        for a in range(A):
            dev_bytes[a].copy_(host[W + s][a], non_blocking=True)
        losses = do_step(dev_bytes, W + K + s)
        losses_host.copy_(losses.reshape(losses_host.shape), non_blocking=True)
    e1.record(stream)
    barrier()
    ms_e2e = e0.elapsed_time(e1)

    ms, ms_e2e = max_over_ranks(dist, [ms, ms_e2e], dev)
    if rank != 0:
        dist.destroy_process_group()
        return 0

    tok = tokens_per_step(c) * A * world
    value = tok * K / (ms / 1e3)
    gate_ms, gate_n = traced["gate"]
    peaks, peak_src = measured_peaks()
    clocks = clk.summary()
    peak_kind, peak = applicable_peak(peaks, clocks)
    # all algorithmic gate and head work of the traced pass over the dominant
    # kernel's traced time: K steps x A estimates x T timesteps, whether a
    # launch covers one timestep (persistent kernel, the head of the previous
    # timestep inside) or all of them (resident kernel)
    one_launch = traced["prep"][1] == 0  # the resident kernel: no tile preparation
    flops_total = (gate_flops_per_timestep(c) + head_flops_per_timestep(c)) * T * K * A
    achieved = flops_total / (gate_ms / 1e3) / 1e12 if gate_n else None
    traffic = launch_traffic(args.config, T)
    launches = sum(v[1] for v in traced.values())
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": W, "ms_per_step": ms / K, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": DTYPE, "data": "synthetic",
        "steps_per_s": K / (ms / 1e3),
        "config": {
            "workload": workload_desc(args.config, c),
            "optimizer": ("SGD, dense probes (Eq. main-spsa)" if not adam else
                          f"Adam with coupled decay, {kind} probes, {A} accumulation batch(es) "
                          "per update (Eq. localspsa)"
                          + ("; a batch per probe" if per_probe else "")
                          + ("; summed-loss control arm" if summed else "")),
            "tokens_per_step_per_gpu": tokens_per_step(c) * A,
            "seq_len": T,
            "l2": "flushed between timed steps (a 256 MiB buffer is written before each "
                  "step, inside the timed region)",
            "parallelism": f"experts batched in one launch per sweep; {world} independent "
                           "replica(s), no collective",
        },
        "roofline": {
            "bound": "tensor", "kernel": gate_kernel_name(B, one_launch),
            "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
            "frac": (achieved / peak) if achieved else None, "traffic": traffic,
            "peak_source": f"{peak_src} bf16 dense {peak_kind} (MEASURED_PEAKS.json): the "
                           "burst figure when the sampled SM clock sat at its maximum with no "
                           "power cap, the sustained one otherwise",
            "frac_burst": (achieved / peaks["bf16_tflops"]) if achieved else None,
            "frac_sustained": (achieved / peaks["bf16_tflops_sustained"]) if achieved else None,
            "flops": "algorithmic gate + head flops of the direct form: "
                     "8H(E+H) + 512H per perturbed token",
            "flops_per_launch": flops_total / gate_n if gate_n else None,
            "launches": gate_n,
            "kernel_ms_per_launch": gate_ms / gate_n if gate_n else None,
            "share_of_step": gate_ms / ms if ms else None,
            # all K steps' algorithmic flops over the K untraced steps' time
            "step_frac_burst": (flops_total / (ms / 1e3) / 1e12 / peaks["bf16_tflops"])
                               if ms else None,
        },
        "kernel_ms": {k: v[0] / K for k, v in traced.items()},
        "e2e": {"value": tok * K / (ms_e2e / 1e3), "unit": UNIT,
                "h2d_bytes_per_step": int(sum(r.numel() for r in resident[0])),
                "d2h_bytes_per_step": int(A * N * n * 2 * 4)},
        "gpu_launches": launches,
        "clocks": clocks,
        "status": api.STATUS_NAMES.get(status, status),
    }
    if not args.no_cpu_baseline and world == 1:
        line["cpu_baseline"] = cpu_baseline(args.config, c, min(args.cpu_sample_seqs, B), kind)
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def inference_arm(args):
    """Routed inference: scored tokens/s of soma_mixture_nll, routing included."""
    import torch
    from paper_2609_37899_gb300 import api, build, inputs
    if not os.path.exists(api.LIB_PATH):
        build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    c = dict(inputs.CONFIGS[args.config])
    if args.seq_len:
        c["seq_len"] = args.seq_len
    N, E, H, T = c["n_experts"], c["E"], c["H"], c["seq_len"]
    R, k, t0 = args.requests, min(4, c["n_experts"]), c["seq_len"] // 4
    K, W = args.steps, args.warmup
    params = torch.empty(N, api.param_count(E, H), dtype=torch.float32, device=dev)
    api.init_experts(params, E, H, seed=1000, std=c["init_std"] or 0.0)
    rng = np.random.default_rng(7)
    # routes: k distinct experts per request, uniformly (the fitted router is
    # not available); requests: the workload's byte streams
    routes = [np.stack([rng.choice(N, size=k, replace=False) for _ in range(R)]).astype(np.int32)
              for _ in range(W + K)]
    host = []
    for s in range(W + K):
        rows = []
        while sum(len(x) for x in rows) < R:
            rows.append(inputs.config_batch(args.config, seed=1, step=100 * s + len(rows),
                                            seq_len=T).reshape(-1, T + 1))
        host.append(torch.from_numpy(np.concatenate(rows)[:R]).pin_memory())
    resident = [h.to(dev) for h in host]
    ws = torch.empty(max(api.mixture_workspace_bytes(E, H, N, r, T) for r in routes),
                     dtype=torch.uint8, device=dev)
    out = torch.empty(R, T - t0, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    for s in range(W):
        api.mixture_nll(params, resident[s], E, H, routes[s], t0, out, ws)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(0) as clk:
        e0.record(stream)
        for s in range(K):
            flush.fill_(s & 0xFF)
            api.mixture_nll(params, resident[W + s], E, H, routes[W + s], t0, out, ws)
        e1.record(stream)
        torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    out_host = torch.empty_like(out, device="cpu").pin_memory()
    dev_rq = torch.empty_like(resident[0])
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record(stream)
    for s in range(K):
        flush.fill_(s & 0xFF)
        dev_rq.copy_(host[W + s], non_blocking=True)
        api.mixture_nll(params, dev_rq, E, H, routes[W + s], t0, out, ws)
        out_host.copy_(out, non_blocking=True)
    f1.record(stream)
    torch.cuda.synchronize()
    ms_e2e = f0.elapsed_time(f1)
    status = api.get_status()
    tok = R * (T - t0)
    line = {
        "metric": "scored tokens/s, routed inference (Eq. main-mixture)", "value": tok * K / (ms / 1e3),
        "unit": "scored tokens/s", "n_gpus": 1, "steps": K, "warmup": W, "ms_per_step": ms / K,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": DTYPE,
        "data": "synthetic",
        "config": {"workload": workload_desc(args.config, c) + f"; {R} requests x {T} bytes, "
                               f"k={k} uniform random routes, positions {t0}..{T - 1} scored, "
                               "routing (host grouping) inside the timed region",
                   "l2": "flushed between timed steps (256 MiB written before each)"},
        "e2e": {"value": tok * K / (ms_e2e / 1e3), "unit": "scored tokens/s",
                "h2d_bytes_per_step": int(resident[0].numel()),
                "d2h_bytes_per_step": int(out.numel() * 4)},
        "clocks": clk.summary(),
        "status": api.STATUS_NAMES.get(status, status),
    }
    print(json.dumps(line), flush=True)
    return 0


# ---- the paper's expert body -------------------------------------------------

def body_desc(name, c):
    from paper_2609_37899_gb300 import inputs
    P = inputs.body_param_count(c["d"], c["D"])
    return (f"{name}: {c['n_experts']} expert bodies (D={c['D']} pre-norm blocks of width "
            f"d={c['d']}: bias-free LSTM + GELU MLP 4d, gain-only LayerNorm; M_body={P:,}; frozen "
            f"tied head E [256, {c['d']}]), n_pert={c['n_pert']}, eps={c['eps']}, lr={c['lr']}, "
            f"B={c['batch']} x T={c['seq_len']} bytes per expert, order-{c['order']} Zipf(1.1) "
            f"Markov clusters")


def body_flops_per_token(c):
    # per block: LSTM gates [2d] x [2d, 4d] and the MLP [d] x [d, 4d] x [4d, d];
    # the tied decode [d] x [d, 256]; 2 flops per multiply-add
    d = c["d"]
    return c["D"] * (2 * 2 * d * 4 * d + 2 * 2 * d * 4 * d) + 2 * d * 256


def body_cpu_baseline(cfg_name, c, n_seqs, kind):
    import oracle
    from paper_2609_37899_gb300 import inputs
    theta = inputs.body_config_params(cfg_name)[:1]
    head = inputs.init_head(c["d"], 0)
    bx = inputs.body_config_batch(cfg_name)[:1, :n_seqs]
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    oracle.build()
    t0 = time.perf_counter()
    oracle.body_spsa_losses(theta, c["d"], c["D"], head, np.float32(c["eps"]), 0, 0, bx,
                            probes=[0], kind=kind, n_threads=cores)
    dt = time.perf_counter() - t0
    toks = 2 * n_seqs * c["seq_len"]
    return {"value": toks / dt, "unit": UNIT, "cores": min(cores, n_seqs), "kind": "oracle",
            "sample": f"expert 0, {kind} probe 0, both signs, {n_seqs} of {c['batch']} sequences x "
                      f"{c['seq_len']} bytes ({toks} perturbed tokens) in {dt:.2f} s; OpenMP "
                      f"over sequences, so {min(cores, n_seqs)} of {cores} cores busy"}


def body_reference_arm(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import oracle
    from paper_2609_37899_gb300 import inputs
    c = inputs.BODY_CONFIGS[args.config]
    n_seqs = min(args.ref_sample_seqs, c["batch"])
    theta = inputs.body_config_params(args.config)
    head = inputs.init_head(c["d"], 0)
    bx = inputs.body_config_batch(args.config)
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    oracle.build()

    def one(k):
        e, i = k % c["n_experts"], k % c["n_pert"]
        oracle.body_spsa_losses(theta[e:e + 1], c["d"], c["D"], head, np.float32(c["eps"]), 0, 0,
                                bx[e:e + 1, :n_seqs], probes=[i], first_expert=e,
                                n_threads=cores)

    for k in range(args.warmup):
        one(k)
    t0 = time.perf_counter()
    for k in range(args.steps):
        one(args.warmup + k)
    dt = time.perf_counter() - t0
    toks = 2 * n_seqs * c["seq_len"]
    value = toks * args.steps / dt
    sample = (f"per step one probe pair (both signs) of one expert body over {n_seqs} of "
              f"{c['batch']} sequences x {c['seq_len']} bytes = {toks} perturbed tokens")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * dt / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": body_desc(args.config, c), "sample": sample},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": min(cores, n_seqs),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)
    return 0


def body_arm(args):
    """SPSA steps of N expert bodies: the SGD step (Eq. main-spsa), or with
    --optimizer adam the paper's step (sparse probes with dense gains, A
    estimates, Adam: Eq. localspsa)."""
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    from paper_2609_37899_gb300 import api, build, inputs
    if not os.path.exists(api.LIB_PATH):
        build.build()
    c = dict(inputs.BODY_CONFIGS[args.config])
    if args.seq_len:
        c["seq_len"] = args.seq_len
    N, d, D, n, B, T = c["n_experts"], c["d"], c["D"], c["n_pert"], c["batch"], c["seq_len"]
    K, W = args.steps, args.warmup
    adam = args.optimizer == "adam"
    A = args.accum if adam else 1
    kind = (args.probes or "sparse") if adam else (args.probes or "dense")
    seeds = shard_seeds(rank)
    bodies = api.SomaBodies(N, n, B, T, d, D, device=dev)
    bodies.params.copy_(torch.from_numpy(inputs.init_body(N, d, D, seeds["init"])))
    bodies.head.copy_(torch.from_numpy(inputs.init_head(d, 0)))
    host = [[torch.from_numpy(inputs.body_config_batch(args.config, seed=seeds["data"],
                                                       step=A * s + a, seq_len=T)).pin_memory()
             for a in range(A)] for s in range(W + K)]
    resident = [[h.to(dev) for h in hs] for hs in host]

    def do_step(batches, s):
        if not adam:
            return bodies.step(batches[0], c["eps"], c["lr"], seeds["probe"], s, kind=kind)[0]
        return bodies.adam_step(batches, c["eps"], seeds["probe"], [A * s + a for a in range(A)],
                                t=s + 1, lr=c["lr"], kind=kind)[0]

    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize(dev)

    for s in range(W):
        do_step(resident[s], s)
    barrier()
    # the timed region with tracing off; then a traced pass of the same steps
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        barrier()
        start.record(stream)
        for s in range(K):
            flush.fill_(s & 0xFF)
            do_step(resident[W + s], W + s)
        stop.record(stream)
        barrier()
    ms = start.elapsed_time(stop)
    status = api.get_status()
    api.trace_enable(True)
    api.trace_read(reset=True)
    barrier()
    for s in range(K):
        flush.fill_(s & 0xFF)
        do_step(resident[W + s], W + s)
    barrier()
    api.trace_enable(False)
    traced = api.trace_read(reset=True)
    losses_host = torch.empty(A, N, n, 2, dtype=torch.float32).pin_memory()
    dev_bytes = [torch.empty_like(r) for r in resident[0]]
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for s in range(K):
        flush.fill_(s & 0xFF)
        for a in range(A):
            dev_bytes[a].copy_(host[W + s][a], non_blocking=True)
        losses = do_step(dev_bytes, W + K + s)
        losses_host.copy_(losses.reshape(losses_host.shape), non_blocking=True)
    e1.record(stream)
    barrier()
    ms_e2e = e0.elapsed_time(e1)
    ms, ms_e2e = max_over_ranks(dist, [ms, ms_e2e], dev)
    if rank != 0:
        dist.destroy_process_group()
        return 0
    tok = tokens_per_step(c) * A * world
    value = tok * K / (ms / 1e3)
    sweep_ms, sweep_n = traced["gate"]
    flops = body_flops_per_token(c) * tokens_per_step(c) * A * K
    achieved = flops / (sweep_ms / 1e3) / 1e12 if sweep_n else None
    peaks, peak_src = measured_peaks()
    clocks = clk.summary()
    peak_kind, tensor_peak = applicable_peak(peaks, clocks)
    traffic = launch_traffic(args.config, T)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": W, "ms_per_step": ms / K, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": DTYPE, "data": "synthetic",
        "steps_per_s": K / (ms / 1e3),
        "config": {
            "workload": body_desc(args.config, c),
            "optimizer": ("SGD (Eq. main-spsa), " + kind + " probes" if not adam else
                          f"Adam with coupled decay, {kind} probes (gains dense), {A} "
                          "accumulation batch(es) per update (Eq. localspsa)"),
            "tokens_per_step_per_gpu": tokens_per_step(c) * A,
            "seq_len": T,
            "l2": "flushed between timed steps (a 256 MiB buffer is written before each "
                  "step, inside the timed region)",
            "parallelism": f"every (expert, probe, sign) in one launch; {world} independent "
                           "replica(s), no collective",
        },
        "roofline": {
            "bound": "tensor", "kernel": "body_tc_kernel (tcgen05, one CTA per probe pair and "
                                         "16-sequence chunk, the whole recurrence resident; "
                                         "its time includes the decode and the loss)",
            "achieved": achieved, "peak": tensor_peak, "unit": "TFLOP/s",
            "frac": (achieved / tensor_peak) if achieved else None, "traffic": traffic,
            "peak_source": f"{peak_src} bf16 dense {peak_kind} (MEASURED_PEAKS.json): the "
                           "burst figure when the sampled SM clock sat at its maximum with no "
                           "power cap, the sustained one otherwise",
            "frac_burst": (achieved / peaks["bf16_tflops"]) if achieved else None,
            "frac_sustained": (achieved / peaks["bf16_tflops_sustained"]) if achieved else None,
            "flops_per_token": body_flops_per_token(c),
            "launches": sweep_n,
            "kernel_ms_per_launch": sweep_ms / sweep_n if sweep_n else None,
            "share_of_step": sweep_ms / ms if ms else None,
        },
        "kernel_ms": {k: v[0] / K for k, v in traced.items()},
        "e2e": {"value": tok * K / (ms_e2e / 1e3), "unit": UNIT,
                "h2d_bytes_per_step": int(sum(r.numel() for r in resident[0])),
                "d2h_bytes_per_step": int(A * N * n * 2 * 4)},
        "gpu_launches": sum(v[1] for v in traced.values()),
        "clocks": clocks,
        "status": api.STATUS_NAMES.get(status, status),
    }
    if not args.no_cpu_baseline and world == 1:
        line["cpu_baseline"] = body_cpu_baseline(args.config, c, min(args.cpu_sample_seqs, B),
                                                 kind)
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main():
    args = parse()
    from paper_2609_37899_gb300 import inputs
    if args.config in inputs.BODY_CONFIGS:
        return body_reference_arm(args) if args.impl == "reference" else body_arm(args)
    if args.impl == "reference":
        return reference_arm(args)
    if args.inference:
        return inference_arm(args)
    return our_arm(args)


if __name__ == "__main__":
    sys.exit(main())
