"""A persistent GEMM whose loads name their tiles, for the L2 model (Section 5.2:
a fully associative LRU over tile-derived accesses), and the study of tile
rasterization order against L2 capacity.

C = A x B with BM x BN output tiles and BK-deep k-steps.  Output tiles are
handed to ``num_ctas`` persistent CTAs round-robin in a rasterization order:

* ``row``     -- row-major over (tile row, tile column);
* ``grouped`` -- groups of ``group`` tile rows, column-major inside a group
                 (the usual swizzle that lets concurrently running CTAs share A
                 and B tiles).

Each CTA is warp-specialised (as ``workloads.ws_gemm_cta``): a producer warp
waits on the ring slot's 'empty' barrier and issues two TMA loads per k-step,
the A tile (row block, k) and the B tile (column block, k); two consumer
warpgroups wait on the 'full' barrier and run their MMAs; per output tile each
consumer runs the epilogue and stores its half of the C tile.  Tile ids: A
tiles first, then B tiles, then C tiles.

Input plumbing only: graphs and parameter rows, no scheduling arithmetic.
"""
from __future__ import annotations

import numpy as np

from . import workloads as W

ORDERS = ("row", "grouped")
H100_L2 = dict(l2_bytes=50 * 1024 * 1024, l2_lat=380, l2_bpc=4300)   # Table "GPU configurations"


def tile_order(mt, nt, order, group=8):
    """Output tiles (tile row, tile column) in rasterization order."""
    if order == "row":
        return [(i, j) for i in range(mt) for j in range(nt)]
    if order == "grouped":
        out = []
        for g0 in range(0, mt, group):
            rows = range(g0, min(g0 + group, mt))
            out.extend((i, j) for j in range(nt) for i in rows)
        return out
    raise KeyError(order)


def l2_gemm(M=4096, N=4096, K=4096, BM=128, BN=256, BK=64, num_ctas=132, order="row", group=8, stages=4,
            elem=2, ew_ops_per_elem=1):
    """The GEMM as one tile graph with a tile id on every LOAD and STORE."""
    mt, nt, kt = M // BM, N // BN, K // BK
    a_id = lambda i, k: i * kt + k                                    # noqa: E731
    b_id = lambda j, k: mt * kt + j * kt + k                          # noqa: E731
    c_id = lambda i, j: mt * kt + nt * kt + i * nt + j                # noqa: E731
    n_tiles = mt * kt + nt * kt + mt * nt
    tiles = tile_order(mt, nt, order, group)
    per_cta = [[] for _ in range(num_ctas)]
    for t, ij in enumerate(tiles):
        per_cta[t % num_ctas].append(ij)
    typ, warp, cta, work, tile = [], [], [], [], []
    src, dst, kind = [], [], []

    def node(c, t, w, wk=0, tl=W.NO_TILE):
        typ.append(t)
        warp.append(w)
        cta.append(c)
        work.append(int(wk))
        tile.append(tl)
        return len(typ) - 1

    def edge(u, v):
        assert u < v
        src.append(u)
        dst.append(v)
        kind.append(W.DATA)

    for c in range(num_ctas):
        ring = []
        for i, j in per_cta[c]:
            last = [None, None]
            for k in range(kt):
                be = node(c, W.BAR, 0)
                if len(ring) >= stages:
                    for m in ring[len(ring) - stages]:
                        edge(m, be)
                la = node(c, W.LOAD, 0, BM * BK * elem, a_id(i, k))
                lb = node(c, W.LOAD, 0, BN * BK * elem, b_id(j, k))
                edge(be, la)
                edge(be, lb)
                mm = []
                for q in (1, 2):
                    bf = node(c, W.BAR, q)
                    edge(la, bf)
                    edge(lb, bf)
                    m = node(c, W.MMA, q, BM // 2 * BN * BK)
                    edge(bf, m)
                    mm.append(m)
                ring.append(mm)
                last = mm
            for q in (1, 2):
                ew = node(c, W.EW, q, BM // 2 * BN * ew_ops_per_elem)
                edge(last[q - 1], ew)
                st = node(c, W.STORE, q, BM // 2 * BN * elem, c_id(i, j))
                edge(ew, st)
    n = len(typ)
    return W.from_edges(f"l2_gemm_{order}", 3, np.array(typ, np.uint8), np.array(warp, np.uint16),
                        np.array(cta, np.uint32), np.array(work, np.uint32), np.zeros(n, np.uint32),
                        np.zeros(num_ctas, np.uint32), src, dst, kind, tile=np.array(tile, np.uint32),
                        n_tiles=n_tiles)


def study_set(orders=ORDERS, **kw):
    graphs = [l2_gemm(order=o, **kw) for o in orders]
    return W.stack(graphs, "l2_gemm"), list(orders)


CAPACITIES_MB = (0, 6, 12, 25, 50, 100)


def study_params(n_graphs, capacities_mb=CAPACITIES_MB, points_per_capacity=1, seed=W.SEED0 + 8):
    """H100 rows (132 SMs, one CTA per SM) with the L2 of the paper's table,
    at each capacity (0: no L2 model); further points per capacity draw DRAM
    bandwidth (1-8 TB/s).  The same rows for every graph."""
    rows = []
    rng = np.random.default_rng(seed)
    draws = rng.integers(W.bytes_per_cycle(1.0), W.bytes_per_cycle(8.0) + 1, max(points_per_capacity - 1, 0))
    for cap in capacities_mb:
        for k in range(points_per_capacity):
            p = W.default_params()
            if cap:
                p[W.P_L2_BYTES] = cap * 1024 * 1024
                p[W.P_L2_LAT] = H100_L2["l2_lat"]
                p[W.P_L2_BPC] = H100_L2["l2_bpc"]
            if k:
                p[W.P_HBM_BPC] = draws[k - 1]
            rows.append(p)
    block = np.stack(rows)
    out = []
    for g in range(n_graphs):
        b = block.copy()
        b[:, W.P_GRAPH_INDEX] = g
        out.append(b)
    return np.ascontiguousarray(np.concatenate(out), np.int32)
