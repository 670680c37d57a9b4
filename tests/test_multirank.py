"""The several-GPU path's host logic on CPU ranks (gloo, world size 2):
disjoint trace shards, the max-over-ranks timer, and per-point partial sums
that add up to the single-process sums over all traces."""
import os
import socket

import numpy as np

import oracle
from paper_2505_05286_gb300 import dist as D
from paper_2505_05286_gb300 import workloads as W


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out_dir):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world), RANK=str(rank),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w, r, lr = D.env()
    assert (w, r, lr) == (world, rank, rank)
    per = 2
    wl = W.make_workload(1, n_traces=per, n_queries=60, first_trace=D.first_trace(rank, per))
    wl.grid = W.subset_grid(wl.grid, list(range(0, 64, 5)))
    res = oracle.run(wl)
    P = wl.grid.n_points
    t = res.reshape(per, P)
    sp, ss, sf, nq = D.global_point_sums(t["p95_us"].sum(0), t["slo_met"].sum(0), (t["status"] != 0).sum(0),
                                         sum(tr.n_queries for tr in wl.traces))
    mx = D.max_over_ranks(1.5 + rank)
    np.savez(os.path.join(out_dir, f"rank{rank}.npz"), sp=sp, ss=ss, sf=sf, nq=nq, mx=mx,
             seeds=np.array([D.first_trace(rank, per) + j for j in range(per)]))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, str(tmp_path)), nprocs=2, start_method="spawn", join=True)
    r0, r1 = (np.load(tmp_path / f"rank{r}.npz") for r in (0, 1))
    assert set(r0["seeds"]).isdisjoint(set(r1["seeds"]))
    assert float(r0["mx"]) == float(r1["mx"]) == 2.5
    for k in ("sp", "ss", "sf", "nq"):
        assert np.array_equal(r0[k], r1[k])
    # the same four traces in one process
    wl = W.make_workload(1, n_traces=4, n_queries=60)
    wl.grid = W.subset_grid(wl.grid, list(range(0, 64, 5)))
    res = oracle.run(wl).reshape(4, wl.grid.n_points)
    assert np.array_equal(r0["sp"], res["p95_us"].sum(0))
    assert np.array_equal(r0["ss"], res["slo_met"].sum(0))
    assert int(r0["nq"]) == sum(t.n_queries for t in wl.traces)
    # and the best point of the summed table is the single-process best point
    flat = res.reshape(-1)
    gp, gs, _ = oracle.best(flat, 4, wl.grid.n_points, [t.n_queries for t in wl.traces], W.OBJ_P95)
    assert gp == int(np.argmin(r0["sp"])) and gs == int(r0["sp"].min())


def test_single_process_defaults():
    assert D.env() == (1, 0, 0) or "WORLD_SIZE" in os.environ
    assert D.max_over_ranks(3.0) == 3.0
    assert D.sum_over_ranks(np.array([1, 2], np.int64)).tolist() == [1, 2]
