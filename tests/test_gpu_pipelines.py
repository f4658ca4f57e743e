"""GPU parity of the pipeline-organisation study (Section 7.1) and of the
busy-cycle output: every design point of the study workload, bit-exact
against the oracle (start, finish, makespan, CTA placement, digest and busy
server-cycles of every class)."""
import numpy as np
import pytest

from oracle import run as oracle_run
from paper_2607_11262_gb300 import workloads as W
from tests import gpu_helpers as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gts_mod():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts
    gts.load()
    return gts


def test_pipelines_workload_every_point(gts_mod):
    w = W.workload("pipelines")
    res = H.run_gpu(w.graph, w.params)
    assert np.all(res["status"] == 0)
    subs = [w.graph.subgraph(i) for i in range(w.graph.n_graphs)]
    for p in range(w.params.shape[0]):
        gi = int(w.params[p, W.P_GRAPH_INDEX])
        ref = oracle_run.simulate(subs[gi], w.params[p])
        H.assert_point_equal(w.graph, w.params[p], res, p, ref)


def test_study_table_matches_oracle(gts_mod):
    from paper_2607_11262_gb300 import pipelines, study
    rows = study.run_study(points_per_graph=3)
    graph, cases = pipelines.study_set()
    params = pipelines.study_params(len(cases), 3)
    assert [(r["org"], tuple(r["tile"]), r["ablation"]) for r in rows] == cases
    for i, r in enumerate(rows):
        refs = [oracle_run.simulate(graph, params[3 * i + j]) for j in range(3)]
        assert r["makespan"] == refs[0].makespan
        assert r["tensor_busy"] == refs[0].busy[0] and r["tma_busy"] == refs[0].busy[1]
        utils = [x.busy[0] / x.makespan for x in refs]
        assert r["tensor_util"] == pytest.approx(utils[0], rel=1e-12)
        assert r["util_min"] == pytest.approx(min(utils), rel=1e-12)
        assert r["util_max"] == pytest.approx(max(utils), rel=1e-12)
        assert r["util_mean"] == pytest.approx(sum(utils) / 3, rel=1e-12)
    assert max(r["normalised_perf"] for r in rows if r["ablation"] == "full") == 1.0


def test_busy_without_trace_and_flag_checks(gts_mod):
    import torch
    gts = gts_mod
    w = W.workload("gemm512")
    dg = gts.DeviceGraph(w.graph)
    dp = gts.DeviceParams(dg, w.params)
    out = gts.simulate(dg, dp, flags=gts.GTS_WANT_BUSY)
    torch.cuda.synchronize()
    busy = out.busy.cpu().numpy()
    for p in (0, 17, 63):
        ref = oracle_run.simulate(w.graph, w.params[p])
        assert list(busy[p]) == list(ref.busy)
    util = gts.utilisation(busy, out.makespan.cpu().numpy(), w.params)
    assert np.all((util >= 0) & (util <= 1))
    with pytest.raises(gts.GtsError) as e:   # WANT_BUSY without an array
        gts.gts_simulate_batch(dg.handle, dp.handle, 0, 1, gts.GTS_WANT_BUSY, 0, 0, out.makespan.data_ptr(),
                               out.status.data_ptr(), 0, 0, 0, out.scratch.data_ptr(), out.scratch.numel())
    assert e.value.status == gts.GTS_ERR_INVALID_ARG
    dp.close()
    dg.close()
