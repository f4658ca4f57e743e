"""libgts with the L2 model (Section 5.2: a fully associative LRU over
tile-derived accesses) against the oracle, bit-exact: hand schedules, random
graphs with tiles (mixed with the issue policies and the NoC), the tiled
persistent GEMM in both rasterization orders, and the L2 study table."""
import json
import os

import numpy as np
import pytest

from oracle import run as oracle_run
from paper_2607_11262_gb300 import workloads as W
from tests import gpu_helpers as H
from tests import tinygraphs as TG

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
TYPE = {n: i for i, n in enumerate(W.TYPE_NAMES)}


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts
    gts.load()


def _check_all(graph, params, res):
    for q in range(res["status"].shape[0]):
        H.assert_point_equal(graph, params[q], res, q, oracle_run.simulate(graph, params[q]))


def test_golden_l2_on_gpu():
    spec = json.load(open(os.path.join(GOLDEN, "l2.json")))
    for case in spec["cases"]:
        nodes = case["nodes"]
        n = len(nodes)
        g = TG.make(n, [(v, v + 1, W.DATA) for v in range(n - 1)], [TYPE[x[0]] for x in nodes], [0] * n, [0] * n,
                    1, work=[x[2] for x in nodes])
        g.tile = np.array([W.NO_TILE if x[1] < 0 else x[1] for x in nodes], np.uint32)
        g.n_tiles = 8
        prm = TG.unit_params(1, 1)
        prm[W.P_DRAM_LAT] = 10
        prm[W.P_L2_BYTES], prm[W.P_L2_LAT], prm[W.P_L2_BPC] = case["l2_bytes"], 3, 2
        res = H.run_gpu(g, prm[None, :])
        assert res["status"][0] == 0, case["name"]
        assert list(res["start"][0]) == case["start"], (case["name"], list(res["start"][0]))
        assert list(res["finish"][0]) == case["finish"], case["name"]
        assert (res["busy"][0][7], res["busy"][0][8]) == (case["hits"], case["loads"]), case["name"]


def test_random_graphs_with_tiles():
    rng = np.random.default_rng(90)
    types = (W.LOAD, W.LOAD, W.STORE, W.MMA, W.EW, W.BAR, W.NOP, W.DSMEM)
    for i in range(80):
        n = int(rng.integers(2, 60))
        g = TG.random_graph(rng, n, W_=int(rng.integers(1, 5)), C=int(rng.integers(1, 6)),
                            p_edge=float(rng.uniform(0.03, 0.3)), cta_major=bool(i % 4), kernels=bool(i % 5 == 0),
                            types=types)
        nt = int(rng.integers(1, 9))
        t = rng.integers(0, nt, n).astype(np.uint32)
        t[rng.random(n) < 0.2] = W.NO_TILE
        g.tile, g.n_tiles = t, nt
        rows = []
        for k in range(6):
            p = W.with_noc(TG.small_params(rng), 2, 1, 1, 2)
            if k:   # row 0 without the L2 model
                p[W.P_L2_BYTES] = int(rng.integers(1, 40))
                p[W.P_L2_LAT] = int(rng.integers(0, 6))
                p[W.P_L2_BPC] = int(rng.integers(1, 6))
            if k >= 4:
                p[W.P_ISSUE_POLICY], p[W.P_SUBPARTITIONS] = k - 3, int(rng.integers(1, 4))
            rows.append(p)
        prms = np.stack(rows)
        _check_all(g, prms, H.run_gpu(g, prms))


def test_l2_gemm_workload_and_study():
    from paper_2607_11262_gb300 import l2gemm, study
    w = W.workload("l2_gemm")
    res = H.run_gpu(w.graph, w.params)
    assert np.all(res["status"] == 0)
    sample = list(range(0, w.params.shape[0], 7))
    refs = oracle_run.simulate_points(w.graph, w.params, sample)
    for q in sample:
        H.assert_point_equal(w.graph, w.params[q], res, q, refs[q])
    rows = study.run_l2_study()
    graph, orders = l2gemm.study_set()
    params = l2gemm.study_params(len(orders))
    refs = oracle_run.simulate_points(graph, params, list(range(params.shape[0])))
    for q, r in enumerate(rows):
        assert (r["makespan"], r["hits"], r["loads"]) == (refs[q].makespan, refs[q].busy[7], refs[q].busy[8])
