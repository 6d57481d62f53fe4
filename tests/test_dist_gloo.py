"""Batch sharding across ranks, tested with world_size-2 gloo process groups on CPU.

The forward needs no exchange between ranks: each example's output depends
only on that example (Sec. 3.3). Two ranks each compute their shard (with
the CPU oracle standing in for the device path) and the gathered result must
equal the whole batch computed at once; the timing helper must return the
slowest rank's time on every rank.
"""
import os
import socket

import numpy as np
import pytest

from paper_2608_23794_gb300 import dist as mdist
from paper_2608_23794_gb300 import synth

torch = pytest.importorskip("torch")


@pytest.mark.parametrize("n,world", [(5, 2), (64, 2), (7, 3), (2, 4), (0, 2)])
def test_shard_bounds_partition(n, world):
    covered = []
    for r in range(world):
        b, e = mdist.shard_bounds(n, world, r)
        assert 0 <= b <= e <= n
        covered.extend(range(b, e))
        assert e - b in (n // world, n // world + 1)
    assert covered == list(range(n))


def test_job_throughput():
    assert mdist.job_throughput(100.0, 4, 2.0) == 200.0
    with pytest.raises(ValueError):
        mdist.job_throughput(1.0, 1, 0.0)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import torch.distributed as dist

    import oracle
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    info = mdist.rank_info()
    assert (info.rank, info.world) == (rank, world)
    cfg = synth.LayerConfig("shard", 5, 6, 6, 32, 8, 3, "bf16", "nhwc", "relu", 28)
    lay = synth.make_layer(cfg, seed=3)
    pidx, plog, resid = oracle.pack(lay.support_idx, lay.support_logits, cfg.C_in)
    b, e = mdist.shard_bounds(cfg.N, world, rank)
    y = oracle.forward(lay.x[b:e], "nhwc", pidx, plog, resid, lay.W1, lay.b1, lay.w2,
                       float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
    parts = [None] * world
    dist.all_gather_object(parts, (b, e, y))
    slowest = mdist.max_over_ranks(0.5 + rank)
    if rank == 0:
        full = oracle.forward(lay.x, "nhwc", pidx, plog, resid, lay.W1, lay.b1, lay.w2,
                              float(lay.b2[0]), cfg.tau_min, cfg.tau_max)
        joined = np.concatenate([p[2] for p in sorted(parts, key=lambda p: p[0])])
        np.save(os.path.join(out_dir, "ok.npy"),
                np.array([np.array_equal(joined, full), slowest == 0.5 + world - 1]))
    else:
        assert slowest == 0.5 + world - 1
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_shards_equal_whole_batch(tmp_path):
    import torch.multiprocessing as mp
    world = 2
    mp.start_processes(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    ok = np.load(tmp_path / "ok.npy")
    assert ok.all(), ok
