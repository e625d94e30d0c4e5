"""Host logic of the N>1 benchmark path, on CPU with the gloo backend and two
ranks: rendezvous, barrier, max-over-ranks timing, and the weak-scaling shard
assignment (every rank reconstructs its own distinct tensors; no collective on
the data path)."""
import os
import socket

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    from paper_2608_13966_gb300 import workloads as WL
    try:
        w, r = bench.dist_setup(world)
        assert (w, r) == (world, rank)
        assert torch.distributed.get_backend() == "gloo"
        bench.barrier(w)
        # the slowest rank's time is the job's time
        t = bench.max_over_ranks(10.0 + rank, w)
        # each rank's shard holds distinct tensors of the same shapes
        wl = WL.workload("single_int4")
        d = WL.make_tensor(wl, wl.tensors[0], device="cpu", seed=rank)
        sums = [torch.zeros(1, dtype=torch.float64) for _ in range(world)]
        torch.distributed.all_gather(sums, d["w"].double().sum().reshape(1))
        q.put((rank, t, [float(x) for x in sums], tuple(d["w"].shape)))
        torch.distributed.destroy_process_group()
    except Exception as e:  # report instead of hanging the parent
        q.put((rank, "error", repr(e), None))


def test_two_rank_gloo_bench_host_path():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    out.sort()
    for rank, t, sums, shape in out:
        assert t != "error", sums
        assert t == 10.0 + (world - 1)          # max over ranks
        assert shape == (256, 1024)
        assert len(set(sums)) == world          # distinct shards
    assert out[0][2] == out[1][2]               # both ranks saw the same gather


def test_reference_arm_other_ranks_do_no_work(capsys):
    import sys
    sys.path.insert(0, ROOT)
    import bench

    class A:
        workload = "single_int4"
        warmup = 0
        steps = 1
        ref_budget = 0.1
        gpus = 2

    assert bench.reference_arm(A(), 2, 1) is None
    assert capsys.readouterr().out == ""
