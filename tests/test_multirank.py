"""Multi-rank host logic of bench.py on CPU (gloo, world size 2).

The path shards by pages: every rank runs its own independent pages with no
collective on the data path; the only collectives are the timing barrier and
the max over ranks.  These tests run that host logic as two gloo processes.
"""
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch
    import torch.distributed as dist
    import bench
    from paper_2607_18839_gb300 import workloads as W

    dist.init_process_group("gloo", init_method="env://", rank=rank, world_size=world)
    w, r, _ = bench.dist_env()
    assert (w, r) == (world, rank)
    # each rank draws its own pages
    seed_t, seed_l = bench.rank_seeds(1, rank)
    inp = W.make_config("c1", seed=seed_t)
    digest = torch.tensor([float(np.asarray(inp.q, dtype=np.int64).sum() % 1000003)],
                          dtype=torch.float64)
    got = [torch.zeros(1, dtype=torch.float64) for _ in range(world)]
    dist.all_gather(got, digest)
    # slowest rank's time
    ms = 1.0 + rank * 2.5
    slow = bench.max_over_ranks(ms, world, torch.device("cpu"))
    # reference arm under a launcher: rank 0 alone runs and prints
    class A:
        workload = "c1"
        steps = 1
        warmup = 0
        ref_step_seconds = 0.01
    line = bench.run_reference(A, world, rank)
    dist.barrier()
    dist.destroy_process_group()
    with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
        f.write(f"{got[0].item()} {got[1].item()} {slow} {line is not None}\n")
        if line is not None:
            f.write(f"{line['impl']} {line['n_gpus']} {line['value']}\n")


def test_two_ranks_gloo(tmp_path):
    torch = pytest.importorskip("torch")
    import oracle
    oracle.build()  # once, before the ranks start
    port = _free_port()
    ctx = torch.multiprocessing.get_context("spawn")
    procs = [ctx.Process(target=_worker, args=(r, 2, port, str(tmp_path))) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=240)
        assert p.exitcode == 0, f"rank exited with {p.exitcode}"
    rows = [open(tmp_path / f"rank{r}.txt").read().split("\n") for r in range(2)]
    d0, d1, slow0, has0 = rows[0][0].split()
    e0, e1, slow1, has1 = rows[1][0].split()
    assert (d0, d1) == (e0, e1)
    assert d0 != d1, "both ranks drew the same pages"
    assert float(slow0) == float(slow1) == 3.5
    assert has0 == "True" and has1 == "False"
    impl, n_gpus, value = rows[0][1].split()
    assert impl == "reference" and int(n_gpus) == 2 and float(value) > 0


def test_whole_job_value():
    import bench
    # 2 ranks x 64 query tokens per 0.5 ms step
    assert bench.whole_job_value(2, 64, 0.5) == pytest.approx(256000.0)
    assert bench.max_over_ranks(1.25, 1, None) == 1.25
    assert bench.rank_seeds(2, 0) != bench.rank_seeds(2, 1)
