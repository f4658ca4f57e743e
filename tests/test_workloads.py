"""The seeded generator honours the graph contract and the published shapes."""
import numpy as np

from paper_2607_11262_gb300 import workloads as W


def _contract(g):
    n = g.n_nodes
    assert g.row_ptr[0] == 0 and int(g.row_ptr[-1]) == g.n_edges
    src = np.repeat(np.arange(n), np.diff(g.row_ptr.astype(np.int64)))
    assert np.all(g.col.astype(np.int64) > src)          # ids are a topological order
    assert np.all(g.warp < g.warps_per_cta)
    assert np.all(g.cta < g.n_ctas)
    assert np.all(np.diff(g.cta_kernel.astype(np.int64)) >= 0)
    assert np.all(g.type <= W.DSMEM) and np.all(g.ekind <= 1)
    if g.tile is not None:
        named = (g.tile != W.NO_TILE) & ((g.type == W.LOAD) | (g.type == W.STORE))
        assert np.all(g.tile[named] < g.n_tiles)
    for k in range(g.n_graphs):
        n0, n1 = int(g.node_off[k]), int(g.node_off[k + 1])
        e0, e1 = int(g.row_ptr[n0]), int(g.row_ptr[n1])
        assert np.all((g.col[e0:e1] >= n0) & (g.col[e0:e1] < n1))


def test_gemm512_shape():
    w = W.workload("gemm512")
    g = w.graph
    _contract(g)
    assert g.n_nodes == 16 * 136 and g.n_ctas == 16 and g.warps_per_cta == 4
    assert w.params.shape == (64, W.NPARAM)
    assert np.all((w.params[:, W.P_NUM_SMS] >= 8) & (w.params[:, W.P_NUM_SMS] <= 132))
    assert np.all((w.params[:, W.P_MMA_LAT] >= 16) & (w.params[:, W.P_MMA_LAT] <= 64))


def test_small_templates_contract():
    _contract(W.assemble("ws", 3, [W.ws_gemm_cta(2, 6)], np.zeros(3, np.int64), np.zeros(3, np.uint32)))
    _contract(W.assemble("fa", 3, [W.fa_fwd_cta(5)], np.zeros(2, np.int64), np.zeros(2, np.uint32)))
    g = W.random_layered_dag(1, n_nodes=3000, layers=16)
    _contract(g)
    assert g.n_edges >= 3000 - 3000 // 16


def test_stress_stack_and_subgraph():
    g = W.stress_set(3, n_nodes=2000)
    _contract(g)
    assert g.n_graphs == 3 and g.n_nodes == 6000 and g.n_ctas == 24
    s = W.random_layered_dag(2607_5000 + 1, n_nodes=2000)
    sub = g.subgraph(1)
    for k in ("row_ptr", "col", "ekind", "type", "warp", "cta", "work"):
        assert np.array_equal(getattr(sub, k), getattr(s, k)), k


def test_seeded_params_are_reproducible():
    a = W.workload("gemm512").params
    b = W.workload("gemm512").params
    assert np.array_equal(a, b)


# published sizes of the configurations (nodes, edges, points); stress is
# generated at full size only by the GPU tests and the bench (minutes of numpy)
SIZES = {"gemm512": (2176, 4736, 64), "wsgemm8192": (1581056, 1842144, 4096), "fa_fwd": (1724416, 2232320, 1024),
         "decoder": (10059776, 11590144, 512)}


def test_every_named_workload_keeps_the_contract():
    for name in ("gemm512", "wsgemm_small", "wsgemm8192", "fa_fwd", "fa_small", "decoder", "decoder_small",
                 "pipelines", "noc_fusion", "l2_gemm"):
        w = W.workload(name)
        _contract(w.graph)
        assert w.params.shape[1] == W.NPARAM and w.params.dtype == np.int32, name
        assert np.all(w.params[:, W.P_GRAPH_INDEX] < w.graph.n_graphs), name
        if name in SIZES:
            assert (w.graph.n_nodes, w.graph.n_edges, w.params.shape[0]) == SIZES[name], name
    assert np.any(W.workload("noc_fusion").graph.type == W.DSMEM)
    assert W.workload("l2_gemm").graph.n_tiles > 0
