"""The N > 1 path on the CPU: two gloo ranks, each stepping its own shard.

Experts never exchange anything (Sec. 6, fully sharded optimisation), so a
multi-GPU run is N ranks, each with its own experts, data and probe streams,
and no collective on the data path.  The timing alone is reduced (MAX over
ranks).  Checked here with world_size 2 and the oracle standing in for each
rank's GPU step:
- bench.py's max_over_ranks gives every rank the slowest rank's time;
- the ranks' shards differ (parameters, data and probes);
- each rank's step, computed inside the process group, equals the same
  shard stepped alone, for the LSTM expert and the paper's expert body;
- the job's token count is the sum over ranks.
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _shard_step(rank):
    """One rank's SPSA steps on its shard (oracle, CPU): LSTM tiny and body."""
    sys.path.insert(0, ROOT)
    import bench
    import oracle
    from paper_2609_37899_gb300 import inputs
    sd = bench.shard_seeds(rank)
    c = inputs.CONFIGS["tiny"]
    theta = inputs.init_params(1, c["E"], c["H"], sd["init"], std=0.1)
    bx = inputs.config_batch("tiny", seed=sd["data"], step=0)
    L, coef, new = oracle.spsa_step(theta, c["E"], c["H"], c["n_pert"], np.float32(c["eps"]),
                                    np.float32(c["lr"]), sd["probe"], 0, bx, n_threads=1)
    b = inputs.BODY_CONFIGS["body_tiny"]
    btheta = inputs.init_body(b["n_experts"], b["d"], b["D"], sd["init"])
    head = inputs.init_head(b["d"], 0)
    bbx = inputs.body_config_batch("body_tiny", seed=sd["data"], seq_len=8)
    BL, bcoef = oracle.body_spsa_losses(btheta, b["d"], b["D"], head, np.float32(b["eps"]),
                                        sd["probe"], 0, bbx, n_pert=2, n_threads=1)
    return dict(theta=theta, bytes=bx, L=L, coef=coef, new=new, BL=BL, bcoef=bcoef,
                tokens=bench.tokens_per_step(c))


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        sys.path.insert(0, ROOT)
        import bench
        r = _shard_step(rank)
        # the only collective: the slowest rank's time
        ms = bench.max_over_ranks(dist, [10.0 + rank, 20.0 - rank])
        objs = [None] * world
        dist.all_gather_object(objs, {k: (v.tolist() if isinstance(v, np.ndarray) else v)
                                      for k, v in r.items()})
        if rank == 0:
            out.put({"ms": ms, "shards": objs})
        else:
            out.put({"ms": ms})
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_step_disjoint_shards():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=300) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # every rank sees the MAX of each timing
    for r in res:
        assert r["ms"] == [11.0, 20.0]
    shards = next(r["shards"] for r in res if "shards" in r)
    a, b = shards
    # disjoint shards: parameters, data and probes differ
    assert not np.array_equal(a["theta"], b["theta"])
    assert not np.array_equal(a["bytes"], b["bytes"])
    assert not np.allclose(a["coef"], b["coef"])
    # each rank's step is the shard's own step: recomputed alone, it agrees
    for rank, got in enumerate(shards):
        alone = _shard_step(rank)
        for k in ("L", "coef", "new", "BL", "bcoef"):
            np.testing.assert_array_equal(np.asarray(got[k]), alone[k])
    # the job's tokens are the sum over ranks (weak scaling)
    assert sum(s["tokens"] for s in shards) == world * a["tokens"]
