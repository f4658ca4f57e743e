"""libgts under the per-subpartition issue policies (Section 5.3:
greedy-then-oldest and round-robin schedulers, one issue per scheduler per
cycle) against the oracle, bit-exact: hand schedules, random graphs, the
kernel shapes, a batch that mixes policies, and full-size workloads on
sampled points."""
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
KIND = {"DATA": W.DATA, "ISSUE": W.ISSUE}


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts
    gts.load()


def _policies(p, rng, nsub_max=4):
    """Rows cycle through lowest-id, GTO and RR with random scheduler counts."""
    p = np.array(p, copy=True)
    for k in range(p.shape[0]):
        pol = k % 3
        p[k, W.P_ISSUE_POLICY] = pol
        p[k, W.P_SUBPARTITIONS] = 0 if pol == 0 else int(rng.integers(1, nsub_max + 1))
    return p


def _check_all(graph, params, res):
    for q in range(res["status"].shape[0]):
        H.assert_point_equal(graph, params[q], res, q, oracle_run.simulate(graph, params[q]))


def test_golden_issue_policies_on_gpu():
    spec = json.load(open(os.path.join(GOLDEN, "issue_policies.json")))
    for case in spec["cases"]:
        nodes = case["nodes"]
        g = TG.make(len(nodes), [(u, v, KIND[k]) for u, v, k in case["edges"]],
                    [TYPE[x[0]] for x in nodes], [x[1] for x in nodes], [x[2] for x in nodes],
                    case["warps_per_cta"], work=[x[3] for x in nodes])
        prm = TG.unit_params(case["num_sms"], case["ctas_per_sm"])
        prm[W.P_ISSUE_POLICY] = case["policy"]
        prm[W.P_SUBPARTITIONS] = case["subpartitions"]
        res = H.run_gpu(g, prm[None, :])
        assert res["status"][0] == 0, case["name"]
        assert list(res["start"][0]) == case["start"], (case["name"], list(res["start"][0]))


def test_random_graphs_mixed_policies():
    rng = np.random.default_rng(31)
    for i in range(100):
        n = int(rng.integers(1, 60))
        g = TG.random_graph(rng, n, W_=int(rng.integers(1, 6)), C=int(rng.integers(1, 6)),
                            p_edge=float(rng.uniform(0.02, 0.3)), cta_major=bool(i % 4), kernels=bool(i % 3))
        prms = _policies(np.stack([TG.small_params(rng) for _ in range(6)]), rng)
        _check_all(g, prms, H.run_gpu(g, prms))


def test_kernel_shapes_under_policies():
    rng = np.random.default_rng(32)
    per = [3, 3, 3, 2, 2]
    ws = W.assemble("ws", 3, [W.ws_gemm_cta(3, 6), W.ws_gemm_cta(2, 6)],
                    np.array([0 if x == 3 else 1 for x in per]), np.zeros(5, np.uint32))
    p = W.sweep_params(5, 30, [(W.P_NUM_SMS, 1, 6), W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE], 1)
    p[:6, W.P_CTAS_PER_SM] = 2
    p = _policies(p, rng)
    _check_all(ws, p, H.run_gpu(ws, p))
    fa = W.assemble("fa", 3, [W.fa_fwd_cta(7), W.fa_fwd_cta(3)], np.array([0, 1, 0, 1, 1, 0, 0]),
                    np.zeros(7, np.uint32))
    p = _policies(W.sweep_params(6, 24, [(W.P_NUM_SMS, 1, 5), W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE,
                                           W.AX_ALU_RATE], 2), rng)
    _check_all(fa, p, H.run_gpu(fa, p))
    gs = [W.random_layered_dag(60 + i, n_nodes=1500, layers=12, issue_frac=0.3, ctas=6) for i in range(3)]
    g = W.stack(gs, "mix")
    p = W.stress_params(3)
    p[:, W.P_NUM_SMS] = 4
    p[:, W.P_CTAS_PER_SM] = 2
    p = _policies(p, rng, nsub_max=8)
    _check_all(g, p, H.run_gpu(g, p))


@pytest.mark.parametrize("name,points", [("wsgemm_small", 48), ("gemm512", 64), ("pipelines", 96)])
def test_full_size_workloads_under_policies(name, points):
    rng = np.random.default_rng(33)
    w = W.workload(name)
    idx = np.linspace(0, w.params.shape[0] - 1, points).round().astype(int)
    p = _policies(w.params[idx], rng)
    p[1::3, W.P_SUBPARTITIONS] = 4          # the Hopper/Blackwell scheduler count on most GTO rows
    res = H.run_gpu(w.graph, p)
    assert np.all(res["status"] == 0)
    sample = list(range(0, points, max(1, points // 12)))
    refs = oracle_run.simulate_points(w.graph, p, sample)
    for q in sample:
        H.assert_point_equal(w.graph, p[q], res, q, refs[q])


def test_policy_rows_validated_per_point():
    rng = np.random.default_rng(34)
    g = TG.random_graph(rng, 20, W_=2, C=2)
    p = np.stack([TG.small_params(rng) for _ in range(5)])
    p[1, W.P_ISSUE_POLICY], p[1, W.P_SUBPARTITIONS] = 1, 0      # GTO without schedulers
    p[2, W.P_ISSUE_POLICY], p[2, W.P_SUBPARTITIONS] = 3, 1      # unknown policy
    p[3, W.P_SUBPARTITIONS] = 2                                  # schedulers under lowest-id
    p[4, W.P_ISSUE_POLICY], p[4, W.P_SUBPARTITIONS] = 2, 33     # too many schedulers
    res = H.run_gpu(g, p)
    assert res["status"][0] == 0
    assert list(res["status"][1:]) == [-3, -3, -3, -3]
    _check_all(g, p, res)


def test_policy_study_matches_oracle():
    from paper_2607_11262_gb300 import study
    rows = study.run_policy_study(names=("gemm512",), points=3)
    w = W.workload("gemm512")
    idx = np.linspace(0, w.params.shape[0] - 1, 3).round().astype(int)
    base = [oracle_run.simulate(w.graph, w.params[q]).makespan for q in idx]
    code = {"gto": W.POLICY_GTO, "rr": W.POLICY_RR}
    for r in rows:
        ratios = []
        for q, b in zip(idx, base):
            p = w.params[q].copy()
            p[W.P_ISSUE_POLICY], p[W.P_SUBPARTITIONS] = code[r["policy"]], r["schedulers"]
            ratios.append(oracle_run.simulate(w.graph, p).makespan / b)
        assert r["ratio_min"] == pytest.approx(min(ratios), rel=1e-12)
        assert r["ratio_max"] == pytest.approx(max(ratios), rel=1e-12)
