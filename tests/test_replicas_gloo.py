"""Multi-process host logic of bench.py on CPU (gloo, world size 2).

The solver does not shard (every subset of a layer reads subsets of all lower
layers), so N GPUs run N independent replica instances.  What needs checking
without GPUs: each rank gets its own instance, the timing is the maximum
over ranks, and the whole-job value adds the ranks' work.
"""

import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    from paper_2609_13692_gb300 import instances

    w, r, local = bench.dist_env()
    bench.init_dist(w, "gloo")
    seed = bench.replica_seed(r)
    inst = instances.config(1, seed=seed)
    # a rank's "time" depends on its rank; the max must reach every rank
    t = bench.max_over_ranks(1.0 + r, w)
    bench.barrier(w)
    out[rank] = (seed, int(inst.bits.sum() % 1000003), t)
    dist.destroy_process_group()


def test_two_replicas_gloo():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    manager = ctx.Manager()
    out = manager.dict()
    procs = [ctx.Process(target=_worker, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    seeds = [out[r][0] for r in range(world)]
    assert seeds == [0, 1]
    assert out[0][1] != out[1][1]  # different replica instances
    assert out[0][2] == out[1][2] == 2.0  # max over ranks reaches both
