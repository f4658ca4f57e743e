"""The N>1 bench path on CPU: two gloo ranks each simulate their own design
points (no data-path collective) and the step time is the max over ranks."""
import os
import socket

import numpy as np
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from oracle import run as oracle_run
    w = bench.load_workload("gemm512", rank, 4)
    ws, r, _ = bench.dist_env()
    # one "step": this rank's points through the CPU oracle
    mks = [oracle_run.simulate(w.graph, w.params[p]).makespan for p in range(w.params.shape[0])]
    my_ms = 10.0 * (rank + 1)
    worst = bench.reduce_max_over_ranks(my_ms)
    rate = bench.whole_job_rate(bench.node_points_of(w.graph, w.params), ws, worst)
    q.put((rank, ws, r, w.params.tolist(), mks, worst, rate))
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_points_and_take_max_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in ps:
        p.start()
    out = sorted(q.get(timeout=300) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, ws0, rr0, p0, mk0, t0, v0), (r1, ws1, rr1, p1, mk1, t1, v1) = out
    assert (ws0, ws1, rr0, rr1) == (2, 2, 0, 1)
    assert not np.array_equal(np.array(p0), np.array(p1))        # each rank its own design points
    assert np.array(p0).shape == np.array(p1).shape              # same per-rank work (weak scaling)
    assert t0 == t1 == 20.0                                      # slowest rank's time on both
    assert v0 == v1 == 2 * 2176 * 4 / 0.020
    assert all(m > 0 for m in mk0 + mk1)
