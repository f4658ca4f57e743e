"""The tiled persistent GEMM for the L2 model (Section 5.2), on CPU: tile ids
and bytes in closed form, the compulsory-miss closed form of the hit count
with an L2 that holds everything, no hits in a one-byte L2, and the model
check that grouped rasterization hits more often than row-major in a small L2."""
import numpy as np
import pytest

from oracle import run
from paper_2607_11262_gb300 import l2gemm as L
from paper_2607_11262_gb300 import workloads as W

SMALL = dict(M=1024, N=1024, K=512, num_ctas=8)


@pytest.mark.parametrize("order", L.ORDERS)
def test_tiles_and_bytes(order):
    g = L.l2_gemm(order=order, **SMALL)
    mt, nt, kt = 1024 // 128, 1024 // 256, 512 // 64
    assert g.n_tiles == mt * kt + nt * kt + mt * nt
    loads = g.type == W.LOAD
    stores = g.type == W.STORE
    assert np.all(g.tile[loads | stores] < g.n_tiles)
    assert np.all(g.tile[~(loads | stores)] == W.NO_TILE)
    a = loads & (g.tile < mt * kt)
    b = loads & (g.tile >= mt * kt)
    assert np.all(g.work[a] == 128 * 64 * 2) and np.all(g.work[b] == 256 * 64 * 2)
    # every A tile is loaded once per output tile of its row, every B tile once per tile of its column
    assert np.all(np.bincount(g.tile[a], minlength=mt * kt) == nt)
    assert np.all(np.bincount(g.tile[b] - mt * kt, minlength=nt * kt) == mt)
    # each C tile is stored as two halves
    assert np.all(np.bincount(g.tile[stores] - mt * kt - nt * kt, minlength=mt * nt) == 2)


def test_tile_orders_are_permutations():
    for order in L.ORDERS:
        t = L.tile_order(6, 5, order, group=4)
        assert sorted(t) == [(i, j) for i in range(6) for j in range(5)]
    assert L.tile_order(4, 2, "grouped", group=2)[:4] == [(0, 0), (1, 0), (0, 1), (1, 1)]


def _l2(p, mb):
    p = p.copy()
    p[W.P_L2_BYTES], p[W.P_L2_LAT], p[W.P_L2_BPC] = int(mb * (1 << 20)), 380, 4300
    return p


def test_hit_count_closed_forms():
    g = L.l2_gemm(order="row", **SMALL)
    loads = int(np.sum(g.type == W.LOAD))
    distinct = len(np.unique(g.tile[g.type == W.LOAD]))
    big = run.simulate(g, _l2(W.default_params(), 1024))
    assert big.status == 0 and (big.busy[7], big.busy[8]) == (loads - distinct, loads)
    tiny = W.default_params()
    tiny[W.P_L2_BYTES], tiny[W.P_L2_LAT], tiny[W.P_L2_BPC] = 1, 380, 4300
    r = run.simulate(g, tiny)
    assert r.status == 0 and (r.busy[7], r.busy[8]) == (0, loads)


def test_grouped_order_hits_more_in_a_small_l2():
    kw = dict(M=2048, N=4096, K=1024, num_ctas=32)
    row = run.simulate(L.l2_gemm(order="row", **kw), _l2(W.default_params(), 1))
    grp = run.simulate(L.l2_gemm(order="grouped", **kw), _l2(W.default_params(), 1))
    assert row.status == grp.status == 0
    assert grp.busy[7] > row.busy[7]
    assert grp.makespan < row.makespan
