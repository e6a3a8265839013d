"""The multi-GPU bookkeeping of bench.py on two CPU ranks (gloo): each rank serves an
independent batch, the whole-job value divides all ranks' queries by the slowest rank's
time, and nothing but the timing scalar crosses ranks."""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import workloads as W

    cfg = W.get_config(3)
    batch = W.draw_batch(cfg, seed=bench.rank_batch_seed(rank))
    ms = 5.0 + 3.0 * rank                       # rank 1 is the slow one
    worst = bench.max_over_ranks(ms, world)
    value = bench.whole_job_us_per_query(worst, cfg.batch, world)
    out[rank] = (worst, value, tuple(int(d) for d in batch.doc_ids[:40]))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_weak_scaling_bookkeeping():
    world = 2
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 8.0                # max over ranks, seen by every rank
    assert res[0][1] == res[1][1] == pytest.approx(8.0 * 1e3 / (8 * 2))
    assert res[0][2] != res[1][2]                       # independent batches per rank
