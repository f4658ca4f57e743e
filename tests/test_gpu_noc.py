"""libgts with DSMEM nodes over the on-chip NoC of SM groups (Section 5.2
"DSMEM / On-chip NoC") against the oracle, bit-exact: hand schedules, random
graphs (with and without the per-subpartition issue policies) and layered DAGs
spread over several SM groups; busy NoC cycles included."""
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


def test_golden_noc_on_gpu():
    spec = json.load(open(os.path.join(GOLDEN, "noc.json")))
    for case in spec["cases"]:
        nodes = case["nodes"]
        g = TG.make(len(nodes), [], [TYPE[x[0]] for x in nodes], [x[1] for x in nodes], [x[2] for x in nodes],
                    case["warps_per_cta"], work=[x[3] for x in nodes])
        prm = W.with_noc(TG.unit_params(case["num_sms"], case["ctas_per_sm"]), *case["noc"])
        if "smem_bpc" in case:
            prm[W.P_SMEM_BPC] = case["smem_bpc"]
        res = H.run_gpu(g, prm[None, :])
        assert res["status"][0] == 0, case["name"]
        assert list(res["start"][0]) == case["start"], (case["name"], list(res["start"][0]))
        assert list(res["finish"][0]) == case["finish"], case["name"]


def test_random_graphs_with_dsmem():
    rng = np.random.default_rng(61)
    types = (W.LOAD, W.SMEM, W.MMA, W.EW, W.STORE, W.BAR, W.NOP, W.DSMEM, W.DSMEM)
    for i in range(90):
        n = int(rng.integers(2, 60))
        g = TG.random_graph(rng, n, W_=int(rng.integers(1, 5)), C=int(rng.integers(1, 7)),
                            p_edge=float(rng.uniform(0.03, 0.3)), cta_major=bool(i % 4), kernels=bool(i % 5 == 0),
                            types=types)
        rows = []
        for k in range(6):
            p = TG.small_params(rng, num_sms=int(rng.integers(1, 6)))
            p = W.with_noc(p, int(rng.integers(1, 5)), int(rng.integers(0, 6)), int(rng.integers(1, 3)),
                           int(rng.integers(1, 4)))
            if k >= 4:
                p[W.P_ISSUE_POLICY] = k - 3
                p[W.P_SUBPARTITIONS] = int(rng.integers(1, 4))
            rows.append(p)
        prms = np.stack(rows)
        _check_all(g, prms, H.run_gpu(g, prms))


def test_layered_dags_over_sm_groups():
    rng = np.random.default_rng(62)
    gs = []
    for i in range(3):
        g = W.random_layered_dag(70 + i, n_nodes=2000, layers=16, issue_frac=0.2, ctas=12)
        t = g.type.copy()
        t[rng.random(t.shape[0]) < 0.25] = W.DSMEM     # a quarter of the nodes cross the NoC
        g.type = t
        gs.append(g)
    g = W.stack(gs, "noc_mix")
    p = W.stress_params(3)
    p[:, W.P_NUM_SMS] = 12
    p = W.with_noc(p, noc_bpc=1, noc_lat=3, cap_noc=2, cluster_sms=4)
    p[2, W.P_ISSUE_POLICY], p[2, W.P_SUBPARTITIONS] = W.POLICY_GTO, 4
    res = H.run_gpu(g, p)
    assert np.all(res["status"] == 0)
    _check_all(g, p, res)
    assert np.all(res["busy"][:, 6] > 0)


def test_dsmem_without_noc_is_a_row_error():
    rng = np.random.default_rng(63)
    g = TG.random_graph(rng, 12, W_=2, C=2, types=(W.DSMEM, W.EW))
    p = np.stack([TG.small_params(rng), W.with_noc(TG.small_params(rng), 2, 1, 1, 2)])
    res = H.run_gpu(g, p)
    assert list(res["status"]) == [-3, 0]
    _check_all(g, p, res)


def test_noc_fusion_workload_and_study():
    from paper_2607_11262_gb300 import clusters, study
    w = W.workload("noc_fusion")
    res = H.run_gpu(w.graph, w.params)
    assert np.all(res["status"] == 0)
    sample = list(range(0, w.params.shape[0], 9))
    refs = oracle_run.simulate_points(w.graph, w.params, sample)
    for q in sample:
        H.assert_point_equal(w.graph, w.params[q], res, q, refs[q])
    rows = study.run_noc_study(points_per_graph=2)
    graph, cases = clusters.study_set()
    params = clusters.study_params(cases, points_per_graph=2)
    for r in rows:
        a = cases.index((r["cluster"], "noc"))
        b = cases.index((r["cluster"], "dram"))
        ra = oracle_run.simulate(graph, params[2 * a])
        rb = oracle_run.simulate(graph, params[2 * b])
        assert (r["noc_makespan"], r["dram_makespan"]) == (ra.makespan, rb.makespan)
        assert r["speedup"] == pytest.approx(rb.makespan / ra.makespan, rel=1e-12)
