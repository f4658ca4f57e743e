"""gts_graph_create checks the graph contract and packs the graph on the
device.  The packed workspace is compared byte for byte with a plain numpy
statement of the packing (node records, ranges, successor entries, stream
heads, nodes per CTA, graph offsets; zeros elsewhere), for CTA-major and
interleaved graphs, stacked sets, tiles and empty CTAs -- including a graph
whose CTAs interleave so much that the warp streams are linked on the host.
Every contract violation is refused with the lowest offending index named."""
import numpy as np
import pytest

from paper_2607_11262_gb300 import workloads as W
from tests import tinygraphs as TG

pytestmark = pytest.mark.gpu

NONE = 0xFFFFFFFF


@pytest.fixture(scope="module")
def gts():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts as mod
    mod.load()
    return mod


def _up(x):
    return (x + 255) // 256 * 256


def expected_workspace(g, nbytes):
    """The packed graph, restated: record {work, lat_extra, next node of the
    same (cta, warp) stream, type | in-degree << 4}, range {tile + 1 or 0, 0,
    first edge, end edge}, successor {node, kind | its warp << 1 | its cta << 8},
    stream heads, nodes per CTA, graph offsets."""
    n, m, C, Wp, G = g.n_nodes, g.n_edges, g.n_ctas, g.warps_per_cta, g.n_graphs
    ws = np.zeros(nbytes, np.uint8)
    o_rec = 0
    o_rng = o_rec + _up(n * 16)
    o_succ = o_rng + _up(n * 16)
    o_first = o_succ + _up(m * 8)
    o_cnt = o_first + _up(C * Wp * 4)
    o_noff = o_cnt + _up(C * 4)
    o_coff = o_noff + _up((G + 1) * 4)
    indeg = np.bincount(g.col.astype(np.int64), minlength=n).astype(np.uint64) if n else np.zeros(0, np.uint64)
    key = g.cta.astype(np.int64) * Wp + g.warp.astype(np.int64)
    nxt = np.full(n, NONE, np.uint32)
    first = np.full(C * Wp, NONE, np.uint32)
    for v in range(n - 1, -1, -1):
        nxt[v] = first[key[v]]
        first[key[v]] = v
    rec = np.zeros((n, 4), np.uint32)
    rec[:, 0], rec[:, 1], rec[:, 2] = g.work, g.lat_extra, nxt
    rec[:, 3] = g.type.astype(np.uint64) | (indeg << np.uint64(4))
    rng = np.zeros((n, 4), np.uint32)
    if g.tile is not None:
        tiled = (g.tile != NONE) & ((g.type == W.LOAD) | (g.type == W.STORE))
        rng[:, 0] = np.where(tiled, g.tile.astype(np.uint64) + 1, 0)
    rng[:, 2], rng[:, 3] = g.row_ptr[:-1], g.row_ptr[1:]
    succ = np.zeros((m, 2), np.uint32)
    succ[:, 0] = g.col
    succ[:, 1] = (g.ekind.astype(np.uint64) | (g.warp[g.col].astype(np.uint64) << np.uint64(1))
                  | (g.cta[g.col].astype(np.uint64) << np.uint64(8)))
    cnt = np.bincount(g.cta.astype(np.int64), minlength=C).astype(np.uint32)

    def put(off, a):
        b = np.ascontiguousarray(a).view(np.uint8).reshape(-1)
        ws[off:off + b.size] = b
    put(o_rec, rec)
    put(o_rng, rng)
    put(o_succ, succ)
    put(o_first, first)
    put(o_cnt, cnt)
    put(o_noff, g.node_off.astype(np.uint32))
    put(o_coff, g.cta_off.astype(np.uint32))
    return ws


def _check_packed(gts, g):
    dg = gts.DeviceGraph(g)
    got = dg.workspace.cpu().numpy()
    want = expected_workspace(g, got.size)
    if not np.array_equal(got, want):
        bad = np.nonzero(got != want)[0]
        raise AssertionError(f"{g.name}: {bad.size} bytes differ, first at {bad[0]}")
    dg.close()


def test_packed_workspace_matches_restatement(gts):
    rng = np.random.default_rng(5)
    graphs = [W.workload("gemm512").graph, W.workload("wsgemm_small").graph]
    for i in range(12):
        graphs.append(TG.random_graph(rng, int(rng.integers(1, 300)), W_=int(rng.integers(1, 6)),
                                      C=int(rng.integers(1, 9)), p_edge=0.05, cta_major=bool(i % 2),
                                      kernels=bool(i % 3)))
    graphs.append(W.stack(graphs[2:8], "stacked"))
    graphs.append(W.stress_set(3, n_nodes=5000))
    g = TG.make(4, [(0, 3, W.DATA)], [W.EW] * 4, [0, 1, 0, 1], [0, 3, 3, 0], 2, work=[1, 2, 3, 4])  # empty CTAs 1, 2
    graphs.append(g)
    t = TG.random_graph(rng, 80, W_=2, C=3, p_edge=0.08, types=(W.LOAD, W.STORE, W.EW))
    t.tile = rng.integers(0, 5, t.n_nodes).astype(np.uint32)
    t.tile[::7] = NONE
    t.n_tiles = 5
    graphs.append(t)
    for g in graphs:
        _check_packed(gts, g)


def test_interleaved_ctas_link_streams_on_the_host(gts):
    """400 CTAs over 60,000 nodes in random order: the CTAs' id spans sum to
    far above 32 x n, so the stream links take the host path; same bytes."""
    rng = np.random.default_rng(6)
    n, C, Wp = 60_000, 400, 4
    cta = rng.integers(0, C, n).astype(np.uint32)
    src = np.arange(0, n - 1, 3)
    dst = src + 1 + rng.integers(0, 50, src.size)
    keep = dst < n
    g = W.from_edges("interleaved", Wp, rng.integers(0, 7, n).astype(np.uint8),
                     rng.integers(0, Wp, n).astype(np.uint16), cta, rng.integers(1, 9, n).astype(np.uint32),
                     np.zeros(n, np.uint32), np.zeros(C, np.uint32), src[keep], dst[keep],
                     rng.integers(0, 2, keep.sum()).astype(np.uint8))
    _check_packed(gts, g)


def _refused(gts, g, status, words):
    with pytest.raises(gts.GtsError) as e:
        gts.DeviceGraph(g)
    assert e.value.status == status
    msg = gts.gts_last_error()
    for w in words:
        assert w in msg, (msg, w)


def test_each_contract_violation_is_refused(gts):
    base = lambda: TG.make(6, [(0, 2, W.DATA), (1, 4, W.ISSUE), (3, 5, W.DATA)],  # noqa: E731
                           [W.EW, W.LOAD, W.MMA, W.EW, W.STORE, W.BAR], [0, 1, 0, 1, 0, 1], [0, 0, 1, 1, 1, 1], 2,
                           kernels=[0, 1])
    _check_packed(gts, base())
    g = base()
    g.type[4] = 8
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["type", "node 4"])
    g = base()
    g.warp[3] = 2
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["warp", "node 3"])
    g = base()
    g.cta[5] = 2
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["cta", "node 5"])
    g = base()
    g.col[1] = 1                      # edge 1 from node 1 to itself
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["forward", "edge 1"])
    g = base()
    g.col[2] = 6                      # past the last node
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["forward", "edge 2"])
    g = base()
    g.ekind[0] = 2
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["kind", "edge 0"])
    g = base()
    g.cta_kernel[:] = [1, 0]
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["cta_kernel", "CTA 1"])
    g = base()
    g.row_ptr[2], g.row_ptr[3] = 2, 1  # row_ptr decreases between nodes 2 and 3
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["row_ptr"])
    g = base()
    g.tile = np.array([NONE, 7, NONE, NONE, 2, NONE], np.uint32)
    g.n_tiles = 4
    _refused(gts, g, gts.GTS_ERR_INVALID_GRAPH, ["tile", "node 1"])
    # an edge that leaves its graph in a stacked set
    st = W.stack([base(), base()], "two")
    st.col[0] = 8                     # node 0 of graph 0 -> node 8 of graph 1
    _refused(gts, st, gts.GTS_ERR_INVALID_GRAPH, ["forward", "edge 0"])


def test_in_degree_limit(gts):
    """2^24 NOP nodes all feeding one node: one predecessor over the limit."""
    k = 1 << 24
    n = k + 1
    g = W.from_edges("fan_in", 1, np.full(n, W.NOP, np.uint8), np.zeros(n, np.uint16), np.zeros(n, np.uint32),
                     np.zeros(n, np.uint32), np.zeros(n, np.uint32), np.zeros(1, np.uint32),
                     np.arange(k, dtype=np.int64), np.full(k, k, np.int64), np.zeros(k, np.uint8))
    _refused(gts, g, gts.GTS_ERR_UNSUPPORTED, ["predecessors", f"node {k}"])
