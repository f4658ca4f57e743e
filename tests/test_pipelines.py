"""The GEMM + SiLU pipeline organisations and the edge-class ablations
(Section 7.1 software-pipelining case study, Section 6.4 ablation), on CPU.

* structure: one CTA, topological ids, warp counts per organisation;
* closed forms of the tile decomposition: total FMAs = tiles x BM x BN x K,
  stored bytes = tiles x BM x BN x 2, loaded bytes = tiles x (BM + BN) x K x 2
  (ping-pong: B twice, tiles x (BM + 2 BN) x K x 2);
* ablations drop exactly their edge classes;
* the stepper equals the oracle (busy cycles included) on tiny instances of
  every organisation and ablation;
* the oracle's single-SM results show the orderings Section 7.1 reports
  (model checks, not parity pins).
"""
import numpy as np
import pytest

from oracle import run, stepper
from paper_2607_11262_gb300 import pipelines as PL
from paper_2607_11262_gb300 import workloads as W


def _edges(g):
    src = np.repeat(np.arange(g.n_nodes), np.diff(g.row_ptr.astype(np.int64)))
    return set(zip(src.tolist(), g.col.tolist(), g.ekind.tolist()))


@pytest.mark.parametrize("org", PL.ORGS)
@pytest.mark.parametrize("tile", [(64, 64, 64), (128, 256, 64), (256, 256, 128)])
def test_structure_and_work_totals(org, tile):
    bm, bn, bk = tile
    g = PL.gemm_silu(org, bm, bn, bk)
    assert g.n_ctas == 1 and np.all(g.cta == 0)
    assert g.warps_per_cta == {"naive_2stage": 2, "ws_3stage": 4}.get(org, 3)
    src = np.repeat(np.arange(g.n_nodes), np.diff(g.row_ptr.astype(np.int64)))
    assert np.all(src < g.col)
    work = g.work.astype(np.int64)
    assert work[g.type == W.MMA].sum() == PL.WAVES * bm * bn * PL.K_DIM
    assert work[g.type == W.STORE].sum() == PL.WAVES * bm * bn * 2
    b_times = 2 if org == "ws_pingpong" else 1
    assert work[g.type == W.LOAD].sum() == PL.WAVES * (bm + b_times * bn) * PL.K_DIM * 2
    assert work[g.type == W.EW].sum() == PL.WAVES * bm * bn * 4
    # every MMA is issued by a math / consumer warp, every producer load by warp 0 (WS)
    if org != "naive_2stage":
        assert set(g.warp[g.type == W.LOAD].tolist()) == {0}
        assert 0 not in set(g.warp[g.type == W.MMA].tolist())
    if org == "ws_3stage":
        assert set(g.warp[g.type == W.EW].tolist()) == {3}


@pytest.mark.parametrize("org", PL.ORGS)
def test_ablations_drop_edge_classes(org):
    full = _edges(PL.gemm_silu(org, 128, 128, 64))
    no_order = _edges(PL.gemm_silu(org, 128, 128, 64, ablation="no_order"))
    no_sync = _edges(PL.gemm_silu(org, 128, 128, 64, ablation="no_sync"))
    data = _edges(PL.gemm_silu(org, 128, 128, 64, ablation="data_only"))
    assert data <= no_order <= full and data <= no_sync <= full
    assert len(no_sync) < len(full)
    if org == "naive_2stage":
        assert len(no_order) < len(full)
    # data-only keeps operand edges: every MMA still depends on a LOAD
    g = PL.gemm_silu(org, 128, 128, 64, ablation="data_only")
    preds = {v: set() for v in range(g.n_nodes)}
    for u, v, _k in data:
        preds[v].add(u)
    for v in np.nonzero(g.type == W.MMA)[0]:
        assert any(g.type[u] == W.LOAD for u in preds[int(v)])


@pytest.mark.parametrize("org", PL.ORGS)
@pytest.mark.parametrize("ablation", list(PL.ABLATIONS))
def test_stepper_equals_oracle_tiny(org, ablation):
    # 2 waves of a 4x4 tile, K split in 2 k-steps; rates/latencies keep it short
    g = PL.gemm_silu(org, 4, 4, 512, ablation=ablation, tiles=2)
    prm = W.default_params()
    prm[W.P_NUM_SMS] = 1
    prm[W.P_HBM_BPC], prm[W.P_TMA_BPC], prm[W.P_MMA_FMA_PC], prm[W.P_ALU_OPS_PC] = 4096, 1024, 1024, 8
    prm[W.P_DRAM_LAT], prm[W.P_MMA_LAT], prm[W.P_BAR_LAT] = 9, 3, 2
    r = run.simulate(g, prm)
    st, mk, start, fin, cta_sm = stepper.simulate_graph(g, prm)
    assert r.status == st == 0
    assert r.makespan == mk and list(r.start) == start and list(r.finish) == fin
    assert list(r.busy) == stepper.busy_cycles(g.type, g.work, g.lat_extra, prm, start, mk)


@pytest.fixture(scope="module")
def single_sm():
    g, cases = PL.study_set()
    prm = PL.study_params(len(cases))
    out = {}
    for i, c in enumerate(cases):
        r = run.simulate(g, prm[i])
        assert r.status == 0
        sub = g.subgraph(i)
        mma = sub.work[sub.type == W.MMA].astype(np.int64)
        assert r.busy[0] == int((-(-mma // int(prm[i, W.P_MMA_FMA_PC]))).sum())
        assert 0 < r.busy[0] <= r.makespan
        out[c] = (r.makespan, r.busy[0] / r.makespan)
    return out


def test_study_orderings_reported_in_the_paper(single_sm):
    mk = {k: v[0] for k, v in single_sm.items()}
    for tile in PL.TILES:
        full = {o: mk[(o, tile, "full")] for o in PL.ORGS}
        # WS cooperative improves on the naive 2-stage kernel at every tile size
        assert full["ws_cooperative"] < full["naive_2stage"], tile
        # WS 3-stage stays near the best organisation
        assert full["ws_3stage"] <= 1.02 * min(full.values()), tile
        # removing constraints only adds (unrealistic) overlap here
        for o in PL.ORGS:
            assert mk[(o, tile, "data_only")] <= mk[(o, tile, "full")], (o, tile)
    # ping-pong: worse than cooperative on small tiles, better on large ones
    assert mk[("ws_pingpong", (64, 64, 64), "full")] > mk[("ws_cooperative", (64, 64, 64), "full")]
    assert mk[("ws_pingpong", (256, 256, 128), "full")] < mk[("ws_cooperative", (256, 256, 128), "full")]


def test_study_params_layout():
    prm = PL.study_params(3, 5)
    assert prm.shape == (15, W.NPARAM)
    assert np.all(prm[:, W.P_NUM_SMS] == 1)
    assert list(prm[:, W.P_GRAPH_INDEX]) == [0] * 5 + [1] * 5 + [2] * 5
    assert np.all(prm[::5, W.P_HBM_BPC] == W.default_params()[W.P_HBM_BPC])
    idx, lo, hi = PL.SINGLE_SM_HBM
    assert np.all((prm[:, idx] >= lo) & (prm[:, idx] <= hi))
    # every graph sees the same hardware points
    blocks = prm.reshape(3, 5, W.NPARAM)
    assert np.array_equal(blocks[0, :, :W.P_GRAPH_INDEX], blocks[2, :, :W.P_GRAPH_INDEX])
