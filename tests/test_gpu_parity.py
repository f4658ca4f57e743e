"""libgts (CUDA, sm_103a) against the CPU oracle: bit-exact start/finish cycles,
makespans, statuses, CTA placement and digests (Section 5 backend semantics)."""
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


def _check_all(graph, params, res, first=0):
    for q in range(res["status"].shape[0]):
        ref = oracle_run.simulate(graph, params[first + q])
        H.assert_point_equal(graph, params[first + q], res, q, ref)


def test_gemm512_all_points():
    w = W.workload("gemm512")
    res = H.run_gpu(w.graph, w.params)
    assert np.all(res["status"] == 0)
    _check_all(w.graph, w.params, res)


def test_golden_hand_schedules_on_gpu():
    spec = json.load(open(os.path.join(GOLDEN, "hand_schedules.json")))
    for case in spec["cases"]:
        nodes = case["nodes"]
        g = TG.make(len(nodes), [(u, v, KIND[k]) for u, v, k in case["edges"]],
                    [TYPE[x[0]] for x in nodes], [x[1] for x in nodes], [x[2] for x in nodes],
                    case["warps_per_cta"], kernels=case["kernels"], work=[x[3] for x in nodes])
        prm = TG.unit_params(case["num_sms"], case["ctas_per_sm"], case["caps"], case["cap_hbm"])[None, :]
        res = H.run_gpu(g, prm)
        assert res["status"][0] == 0, case["name"]
        assert list(res["start"][0]) == case["start"], case["name"]
        assert list(res["finish"][0]) == case["finish"], case["name"]
        assert res["makespan"][0] == case["makespan"], case["name"]
        assert list(res["cta_sm"][0]) == case["cta_sm"], case["name"]


def test_random_small_graphs():
    rng = np.random.default_rng(21)
    for i in range(120):
        n = int(rng.integers(1, 60))
        g = TG.random_graph(rng, n, W_=int(rng.integers(1, 6)), C=int(rng.integers(1, 6)),
                            p_edge=float(rng.uniform(0.02, 0.3)), cta_major=bool(i % 4), kernels=bool(i % 3))
        prms = np.stack([TG.small_params(rng) for _ in range(5)])
        res = H.run_gpu(g, prms)
        _check_all(g, prms, res)


def test_random_intra_cta_graphs():
    rng = np.random.default_rng(22)
    for i in range(80):
        n = int(rng.integers(1, 70))
        g = TG.random_graph(rng, n, W_=int(rng.integers(1, 6)), C=int(rng.integers(1, 7)),
                            p_edge=float(rng.uniform(0.05, 0.4)), cta_major=True, kernels=bool(i % 2),
                            intra_cta=True)
        prms = np.stack([TG.small_params(rng, cps=1) for _ in range(4)]
                        + [TG.small_params(rng, num_sms=4, cps=2) for _ in range(2)])
        _check_all(g, prms, H.run_gpu(g, prms))


def test_small_ws_gemm_many_tiles_ragged():
    # 5 persistent CTAs over 13 tiles (3,3,3,2,2), 6 k-steps, 4-stage ring
    per = [3, 3, 3, 2, 2]
    tpls = [W.ws_gemm_cta(3, 6), W.ws_gemm_cta(2, 6)]
    g = W.assemble("ws", 3, tpls, np.array([0 if x == 3 else 1 for x in per]), np.zeros(5, np.uint32))
    p = W.sweep_params(5, 40, [(W.P_NUM_SMS, 1, 6), W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE], 1)
    p[:7, W.P_CTAS_PER_SM] = 2
    p[7:10, W.P_CAP_HBM] = 3
    res = H.run_gpu(g, p)
    assert np.all(res["status"] == 0)
    _check_all(g, p, res)


def test_small_fa_and_decoder_shapes():
    fa = W.assemble("fa", 3, [W.fa_fwd_cta(7), W.fa_fwd_cta(3)], np.array([0, 1, 0, 1, 1, 0, 0]),
                    np.zeros(7, np.uint32))
    p = W.sweep_params(6, 24, [(W.P_NUM_SMS, 1, 5), W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE, W.AX_ALU_RATE], 1)
    _check_all(fa, p, H.run_gpu(fa, p))
    tpls = [W.ew_cta(loads=(4096,), ew_ops=8192, stores=(4096,)), W.ws_gemm_cta(1, 5), W.fa_fwd_cta(2)]
    ct = [0, 0, 1, 1, 1, 2, 2, 0, 0, 1]
    ck = [0, 0, 1, 1, 1, 2, 2, 3, 3, 4]
    dec = W.assemble("dec", 4, tpls, np.array(ct), np.array(ck, np.uint32))
    p = W.sweep_params(7, 24, [(W.P_NUM_SMS, 1, 4), W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE, W.AX_ALU_RATE], 1)
    p[:4, W.P_CAP_HBM] = 2
    _check_all(dec, p, H.run_gpu(dec, p))


def test_stacked_random_dags():
    g = W.stress_set(5, n_nodes=3000)
    p = W.stress_params(5)
    res = H.run_gpu(g, p)
    assert np.all(res["status"] == 0)
    _check_all(g, p, res)
    # with ISSUE edges and two CTA slots per SM over 4 SMs
    gs = [W.random_layered_dag(40 + i, n_nodes=1500, layers=12, issue_frac=0.3, ctas=6) for i in range(3)]
    g = W.stack(gs, "mix")
    p = W.stress_params(3)
    p[:, W.P_NUM_SMS] = 4
    p[:, W.P_CTAS_PER_SM] = 2
    p[1, W.P_CAP_HBM] = 1
    _check_all(g, p, H.run_gpu(g, p))


def test_batches_offsets_and_makespan_only():
    from paper_2607_11262_gb300 import gts
    w = W.workload("gemm512")
    full = H.run_gpu(w.graph, w.params)
    part = H.run_gpu(w.graph, w.params, first_point=17, n_points=20)
    assert np.array_equal(part["makespan"], full["makespan"][17:37])
    assert np.array_equal(part["start"], full["start"][17:37])
    mo = H.run_gpu(w.graph, w.params, flags=gts.GTS_WANT_DIGEST)
    assert np.array_equal(mo["makespan"], full["makespan"])
    assert np.array_equal(mo["digest"], full["digest"])
    assert np.array_equal(mo["status"], full["status"])


def test_makespan_only_with_tiny_scratch():
    import torch

    from paper_2607_11262_gb300 import gts
    w = W.workload("gemm512")
    dg = gts.DeviceGraph(w.graph)
    dp = gts.DeviceParams(dg, w.params)
    row = ((dg.row_nodes + 1) // 2 * 2) * 8
    head = gts.GTS_SCRATCH_HEADER_BYTES
    scratch = torch.empty(head + 3 * row, dtype=torch.uint8, device="cuda")  # 3 design points at a time
    out = gts.simulate(dg, dp, flags=gts.GTS_WANT_DIGEST, scratch=scratch)
    torch.cuda.synchronize()
    full = H.run_gpu(w.graph, w.params)
    assert np.array_equal(out.makespan.cpu().numpy(), full["makespan"])
    assert np.array_equal(out.digest.cpu().numpy().astype(np.uint64), full["digest"])
    with pytest.raises(gts.GtsError) as e:
        small = torch.empty(head + row - 16, dtype=torch.uint8, device="cuda")
        gts.simulate(dg, dp, flags=0, scratch=small)
    assert e.value.status == gts.GTS_ERR_NOMEM


def test_per_point_errors_do_not_spoil_others():
    w = W.workload("gemm512", points=8)
    p = w.params.copy()
    p[1, W.P_TMA_BPC] = 0               # invalid rate
    p[2, W.P_CAP_ALU] = 0               # invalid cap
    p[3, W.P_GRAPH_INDEX] = 1           # graph index out of range
    p[4, W.P_DRAM_LAT] = 2**31 - 100    # finish overflows int32
    p[5, 21] = 7                        # reserved field
    res = H.run_gpu(w.graph, p)
    assert list(res["status"]) == [0, -3, -3, -3, -6, -3, 0, 0]
    for q in (0, 6, 7):
        H.assert_point_equal(w.graph, p[q], res, q, oracle_run.simulate(w.graph, p[q]))
    assert oracle_run.simulate(w.graph, p[4]).status == oracle_run.ERR_OVERFLOW


def test_deadlock_and_boundary_cycles():
    dl = TG.make(3, [(0, 2, W.DATA)], [W.EW, W.EW, W.EW], [0, 0, 0], [1, 1, 0], 1)
    p = TG.unit_params(1, 1)[None, :]
    res = H.run_gpu(dl, p)
    assert res["status"][0] == oracle_run.simulate(dl, p[0]).status == oracle_run.ERR_DEADLOCK
    edge = TG.make(2, [(0, 1, W.DATA)], [W.NOP, W.NOP], [0, 0], [0, 0], 1, lat_extra=[2**31 - 11, 10])
    res = H.run_gpu(edge, TG.unit_params()[None, :])
    assert res["status"][0] == 0 and res["makespan"][0] == 2**31 - 1
    over = TG.make(2, [(0, 1, W.DATA)], [W.NOP, W.NOP], [0, 0], [0, 0], 1, lat_extra=[2**31 - 11, 11])
    res = H.run_gpu(over, TG.unit_params()[None, :])
    assert res["status"][0] == -6


def test_empty_graph_and_empty_ctas():
    g = TG.make(0, [], [], [], [], 1)
    res = H.run_gpu(g, W.default_params()[None, :])
    assert res["status"][0] == 0 and res["makespan"][0] == 0
    g = TG.make(2, [], [W.EW, W.EW], [0, 0], [0, 2], 1, work=[3, 4])
    p = TG.unit_params(1, 1)[None, :]
    res = H.run_gpu(g, p)
    H.assert_point_equal(g, p[0], res, 0, oracle_run.simulate(g, p[0]))


def test_invalid_graph_and_small_workspace_rejected():
    import torch

    from paper_2607_11262_gb300 import gts
    bad = TG.make(2, [(0, 1, W.DATA)], [W.EW, W.EW], [0, 0], [0, 0], 1)
    bad.col[0] = 0
    with pytest.raises(gts.GtsError) as e:
        gts.DeviceGraph(bad)
    assert e.value.status == gts.GTS_ERR_INVALID_GRAPH
    bad = TG.make(2, [], [W.EW, W.EW], [0, 2], [0, 0], 2)
    with pytest.raises(gts.GtsError) as e:
        gts.DeviceGraph(bad)
    assert e.value.status == gts.GTS_ERR_INVALID_GRAPH
    g = TG.make(2, [(0, 1, W.DATA)], [W.EW, W.EW], [0, 0], [0, 0], 1)
    dg = gts.DeviceGraph(g)
    d = dg.desc
    small = torch.empty(64, dtype=torch.uint8, device="cuda")
    d2 = gts.GraphDesc(d.n_nodes, d.n_edges, d.n_ctas, d.warps_per_cta, d.n_graphs, d.graph_node_off,
                       d.graph_cta_off, d.row_ptr, d.col, d.ekind, d.type, d.warp, d.cta, d.work, d.lat_extra,
                       d.cta_kernel, small.data_ptr(), 64)
    with pytest.raises(gts.GtsError) as e:
        gts.gts_graph_create(d2)
    assert e.value.status == gts.GTS_ERR_NOMEM
