"""The batch-sharded multi-rank path on CPU (gloo, world size 2).

Each rank takes its contiguous shard of the global batch and sums the
shared-weight gradient with one all-reduce -- the only exchange of the
data-parallel step.  The ranks call the benchmark's own shard and reduce
functions (bench.dp_shard, bench.dp_sum: the code a multi-GPU bench run
executes); the per-rank compute here is the oracle (no GPU on this host).  The
check is that the shards partition the global batch and that the all-reduced dw
equals the oracle's dw over the whole global batch.
"""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

from oracle import oracle as orc
from paper_2607_11985_gb300 import workloads as wl


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, batch, out):
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    w_ = bench.dp_shard(1, "c128", rank, world, batch=batch)[0]
    dx, dw = orc.backward(w_.spec, w_.x, w_.w, w_.gE)
    t = bench.dp_sum(torch.tensor(dw), world)
    out[rank] = (w_.x.copy(), dx, t.numpy().copy())
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_shards_and_dw_allreduce():
    world, batch = 2, 6
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, batch, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    full = wl.config(1, dtype="c128", batch=batch * world)[0]
    dx_ref, dw_ref = orc.backward(full.spec, full.x, full.w, full.gE)
    xs = np.concatenate([out[r][0] for r in range(world)])
    assert np.array_equal(xs, full.x)
    assert np.allclose(np.concatenate([out[r][1] for r in range(world)]), dx_ref, atol=1e-12)
    for r in range(world):
        assert np.allclose(out[r][2], dw_ref, atol=1e-12)


def test_rank0_shard_equals_single_process_workload():
    a = wl.config(2, rank=0, world=4)[0]
    b = wl.config(2)[0]
    assert np.array_equal(a.x, b.x) and np.array_equal(a.w, b.w) and np.array_equal(a.gE, b.gE)


def test_bench_rank_count_must_match_gpus():
    # a launcher that started a different number of ranks than --gpus asks for
    # is an error, not a silent one-rank measurement
    import subprocess
    import sys
    env = dict(os.environ, WORLD_SIZE="1", RANK="0", LOCAL_RANK="0")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--gpus", "2"], env=env,
                       capture_output=True, text=True, timeout=120)
    assert r.returncode != 0 and "ranks" in r.stderr
