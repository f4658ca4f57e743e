"""The scratch contract of gts_simulate_batch: every call leaves the rows it
used all zero (a node's dependency counters are reset when it becomes a warp
head; a point that stops early clears what it used), so a caller that
zero-fills its scratch once may pass GTS_SCRATCH_CLEAN on every later call.
Results are compared bit-exact with the oracle, and the scratch past its
header is read back after every call."""
import numpy as np
import pytest

from oracle import run as oracle_run
from paper_2607_11262_gb300 import workloads as W
from tests import gpu_helpers as H
from tests import tinygraphs as TG

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gts():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts as mod
    mod.load()
    return mod


def _run(gts, graph, params, scratch, flags):
    import torch
    dg = gts.DeviceGraph(graph)
    dp = gts.DeviceParams(dg, params)
    out = gts.simulate(dg, dp, flags=flags | gts.GTS_FULL_TRACE | gts.GTS_WANT_DIGEST | gts.GTS_WANT_CTA_SM
                       | gts.GTS_WANT_BUSY, scratch=scratch)
    torch.cuda.synchronize()
    res = {"status": out.status.cpu().numpy(), "makespan": out.makespan.cpu().numpy(),
           "start": out.start.cpu().numpy(), "finish": out.finish.cpu().numpy(),
           "digest": out.digest.cpu().numpy().astype(np.uint64), "cta_sm": out.cta_sm.cpu().numpy(),
           "busy": out.busy.cpu().numpy()}
    dp.close()
    dg.close()
    return res


def _scratch_for(gts, graph, params):
    dg = gts.DeviceGraph(graph)
    dp = gts.DeviceParams(dg, params)
    s = gts.alloc_scratch(dg, dp)
    dp.close()
    dg.close()
    return s


def _check(graph, params, res):
    for q in range(params.shape[0]):
        H.assert_point_equal(graph, params[q], res, q, oracle_run.simulate(graph, params[q]))


def _clean(gts, scratch):
    import torch
    torch.cuda.synchronize()
    return int(torch.count_nonzero(scratch[gts.GTS_SCRATCH_HEADER_BYTES:]).item()) == 0


def test_clean_scratch_reused_with_error_points(gts):
    """gemm512 rows with overflowing and invalid points in between: results
    bit-exact, the scratch all zero after each of three flagged calls."""
    w = W.workload("gemm512")
    p = w.params.copy()
    p[5, W.P_DRAM_LAT] = 2**31 - 3000   # overflows after some nodes issued
    p[9, W.P_MMA_LAT] = 2**31 - 5000
    p[13, W.P_TMA_BPC] = 0              # invalid row: never starts
    scratch = _scratch_for(gts, w.graph, p)
    assert _clean(gts, scratch)
    first = None
    for _ in range(3):
        res = _run(gts, w.graph, p, scratch, gts.GTS_SCRATCH_CLEAN)
        assert res["status"][5] == res["status"][9] == gts.GTS_ERR_OVERFLOW
        assert res["status"][13] == gts.GTS_ERR_INVALID_PARAMS
        assert _clean(gts, scratch)
        if first is None:
            first = res
            _check(w.graph, p, res)
        else:  # a failed point's trace rows are unspecified (the ABI says so): compare the OK points' rows
            ok = first["status"] == 0
            for k in ("status", "makespan", "digest"):
                assert np.array_equal(res[k], first[k]), k
            for k in ("start", "finish"):
                assert np.array_equal(res[k][ok], first[k][ok]), k


def test_dirty_scratch_without_flag_is_cleared(gts):
    """Without GTS_SCRATCH_CLEAN a scratch full of ones gives the same results,
    and the call leaves every row it used zero."""
    import torch
    w = W.workload("gemm512")
    scratch = _scratch_for(gts, w.graph, w.params)
    scratch.fill_(0xFF)
    res = _run(gts, w.graph, w.params, scratch, 0)
    _check(w.graph, w.params, res)
    torch.cuda.synchronize()
    assert _clean(gts, scratch)  # 64 points, 64 rows: all of them used


def test_deadlocked_points_leave_clean_rows(gts):
    dl = TG.make(3, [(0, 2, W.DATA)], [W.EW, W.EW, W.EW], [0, 0, 0], [1, 1, 0], 1)
    p = np.stack([TG.unit_params(1, 1)] * 5)
    scratch = _scratch_for(gts, dl, p)
    for _ in range(2):
        res = _run(gts, dl, p, scratch, gts.GTS_SCRATCH_CLEAN)
        assert np.all(res["status"] == oracle_run.ERR_DEADLOCK)
        assert _clean(gts, scratch)


def test_one_clean_scratch_across_graphs_of_other_sizes(gts):
    """A scratch left clean by one graph serves another graph with a different
    row size (the rows shift), and stacked sets whose graphs differ in size."""
    rng = np.random.default_rng(7)
    big = W.workload("gemm512")
    scratch = _scratch_for(gts, big.graph, big.params)
    _run(gts, big.graph, big.params, scratch, gts.GTS_SCRATCH_CLEAN)
    gs = [TG.random_graph(rng, int(rng.integers(5, 200)), W_=3, C=3, p_edge=0.05, cta_major=bool(k % 2))
          for k in range(6)]
    st = W.stack(gs, "mixed")
    p = np.stack([TG.small_params(rng, cps=1) for _ in range(24)])
    p[:, W.P_GRAPH_INDEX] = np.arange(24) % 6
    for _ in range(2):
        res = _run(gts, st, p, scratch, gts.GTS_SCRATCH_CLEAN)
        _check(st, p, res)
        assert _clean(gts, scratch)


def test_l2_model_rows_leave_clean_records(gts):
    """With the L2 model each row also holds LRU records per tile: they too are
    zero after the call."""
    rng = np.random.default_rng(91)
    types = (W.LOAD, W.LOAD, W.STORE, W.MMA, W.EW)
    g = TG.random_graph(rng, 40, W_=2, C=2, p_edge=0.1, types=types)
    g.tile = rng.integers(0, 6, g.n_nodes).astype(np.uint32)
    g.n_tiles = 6
    ps = []
    for k in range(8):
        prm = TG.small_params(rng, cps=1)
        prm[W.P_L2_BYTES], prm[W.P_L2_LAT], prm[W.P_L2_BPC] = int(rng.integers(1, 12)), 2, 3
        ps.append(prm)
    p = np.stack(ps)
    scratch = _scratch_for(gts, g, p)
    for _ in range(2):
        res = _run(gts, g, p, scratch, gts.GTS_SCRATCH_CLEAN)
        _check(g, p, res)
        assert _clean(gts, scratch)
