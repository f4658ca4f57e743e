"""The N>1 bench path on CPU with gloo ranks: the sweep is one table of N x P
rows, rank r simulates its contiguous rows [r*P, (r+1)*P) (no collective in
the data path), the per-point makespans and statuses are gathered to rank 0,
and the step time is the max over ranks.  The oracle stands in for the GPU
kernel: the test checks the partition and the gather, which are host logic."""
import os
import socket

import numpy as np
import torch.multiprocessing as mp

POINTS = 4  # per rank


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _simulate(graph, params):
    from oracle import run as oracle_run
    res = [oracle_run.simulate(graph, params[p]) for p in range(params.shape[0])]
    return np.array([r.makespan for r in res], np.int32), np.array([r.status for r in res], np.int32)


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ws, r, _ = bench.dist_env()
    w = bench.load_workload("gemm512", r, POINTS, world=ws)
    mk, st = _simulate(w.graph, w.params)            # this rank's rows only
    my_ms = 10.0 * (rank + 1)
    worst = bench.reduce_max_over_ranks(my_ms)
    rate = bench.whole_job_rate(bench.node_points_of(w.graph, w.params), ws, worst)
    g = bench.gather_to_rank0([mk, st])
    q.put((rank, ws, r, w.params.tolist(), worst, rate, None if g is None else [x.tolist() for x in g]))
    dist.destroy_process_group()


def _run(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in ps:
        p.start()
    out = sorted((q.get(timeout=300) for _ in ps), key=lambda x: x[0])
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    return out


def test_two_gloo_ranks_partition_one_table_and_gather():
    import bench
    out = _run(2)
    (r0, ws0, rr0, p0, t0, v0, g0), (r1, ws1, rr1, p1, t1, v1, g1) = out
    assert (ws0, ws1, rr0, rr1) == (2, 2, 0, 1)
    # one table of 2 x POINTS rows; each rank holds its contiguous range
    w, table = bench.global_table("gemm512", 2, POINTS)
    assert table.shape[0] == 2 * POINTS
    assert np.array_equal(np.array(p0, np.int32), table[:POINTS])
    assert np.array_equal(np.array(p1, np.int32), table[POINTS:])
    # rank 0's rows are the single-GPU table (weak scaling: P rows per GPU)
    from paper_2607_11262_gb300 import workloads as W
    assert np.array_equal(table[:POINTS], W.workload("gemm512", points=POINTS).params)
    # the gathered arrays on rank 0 equal one process simulating the whole table
    assert g1 is None
    mk, st = _simulate(w.graph, table)
    assert g0[0] == mk.tolist() and g0[1] == st.tolist()
    assert all(s == 0 for s in g0[1]) and all(m > 0 for m in g0[0])
    # the slowest rank's time on both, and the whole-job rate from it
    assert t0 == t1 == 20.0
    assert v0 == v1 == 2 * 2176 * POINTS / 0.020


def test_rank_ranges_cover_the_table():
    import bench
    for total in (0, 1, 7, 64, 4096, 4097):
        for world in (1, 2, 3, 8):
            spans = [bench.rank_range(total, world, r) for r in range(world)]
            assert spans[0][0] == 0 and spans[-1][1] == total
            assert all(a[1] == b[0] for a, b in zip(spans, spans[1:]))


def test_single_process_gather_is_identity():
    import bench
    a = np.arange(5, dtype=np.int32)
    out = bench.gather_to_rank0([a, a * 2])
    assert np.array_equal(out[0], a) and np.array_equal(out[1], a * 2)
