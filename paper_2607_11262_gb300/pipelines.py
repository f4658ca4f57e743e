"""Fused GEMM + SiLU persistent kernels in four pipeline organisations, and the
tile-graph mechanism ablations (software-pipelining case study, Section 7.1;
ablation, Section 6.4 "Tile-graph mechanism ablation").

One persistent thread block on one SM computes ``tiles`` output tiles of
BM x BN, one per wave, each over K = 1024 in k-steps of BK (bf16 operands,
bf16 output).  The organisations differ only in which logical warp (a
warpgroup is one logical warp, Section 4.1) issues which node and in the
edges between them:

* ``naive_2stage``   -- no warp specialisation.  Two math warpgroups each own
  BM/2 rows, each issues half of every stage's A/B loads, both wait at a
  barrier for the stage, run their MMA, refill the stage ``stages`` steps
  ahead once both MMAs on it completed, and run the SiLU epilogue and store
  themselves after the mainloop.
* ``ws_cooperative`` -- a TMA producer warpgroup fills a ``stages``-deep ring
  (waiting on the slot's 'empty' barrier), two consumer warpgroups (BM/2 rows
  each) wait on the 'full' barrier, run the MMAs of the same tile, meet at a
  barrier once both finished the tile's mainloop, then both run their
  epilogue.
* ``ws_pingpong``    -- each tile is split into two BM/2-row sub-tiles; the
  producer loads A(BM/2) and the whole B for every k-step of every sub-tile
  (B is loaded twice per tile: more TMA traffic), consumer c computes
  sub-tile c, and the two consumers' mainloops take turns (the first MMA of
  one waits for the issue of the other's last MMA), so one consumer's
  epilogue overlaps the other's mainloop.
* ``ws_3stage``      -- cooperative mainloop plus a dedicated epilogue
  warpgroup fed directly by the consumers' last MMAs; ``acc_buffers``
  accumulator buffers let the consumers start the next tile while the
  epilogue of the previous one runs.

Every edge carries a class used by the ablations (Section 4.1 edge semantics):
``FLOW`` -- a data edge (operands, accumulator chain, epilogue inputs; the
accumulator chain is released at issue, since a tensor pipe accumulates
in-order MMAs back to back);
``ORDER`` -- a general order constraint inside one warp (the epilogue blocks
its warp, a store must drain its staging buffer before the next epilogue
writes it, a warp's own MMA must retire before it refills the stage);
``SYNC`` -- cross-warp/group synchronisation (barrier arrive/wait, the
producer's empty-slot gate, ping-pong turn taking, accumulator-buffer reuse,
the other warpgroup's MMA before a shared stage is refilled, the consumers'
barrier before the cooperative epilogue).

Ablations keep every node and drop edge classes: ``no_order`` drops ORDER,
``no_sync`` drops SYNC, ``data_only`` drops both.  The warp streams' program
order is kept in all of them (the engine always issues a stream in order).

Input plumbing only: graphs and parameter rows, no scheduling arithmetic.
"""
from __future__ import annotations

import numpy as np

from . import workloads as W

FLOW, ORDER, SYNC = 0, 1, 2
ORGS = ("naive_2stage", "ws_cooperative", "ws_pingpong", "ws_3stage")
ABLATIONS = {"full": (), "no_order": (ORDER,), "no_sync": (SYNC,), "data_only": (ORDER, SYNC)}
TILES = ((64, 64, 64), (128, 128, 64), (128, 256, 64), (256, 128, 64), (256, 256, 64), (256, 256, 128))
K_DIM = 1024
WAVES = 10


class _Cta:
    """One thread block's nodes in creation order (= ids) with classed edges."""

    def __init__(self, warps):
        self.warps = warps
        self.t, self.w, self.wk = [], [], []
        self.edges = []          # (u, v, kind, class)
        self.last = [None] * warps

    def node(self, typ, warp, work=0):
        v = len(self.t)
        self.t.append(typ)
        self.w.append(warp)
        self.wk.append(int(work))
        self.last[warp] = v
        return v

    def edge(self, u, v, cls, kind=W.DATA):
        if u is None:
            return
        assert u < v, (u, v)
        self.edges.append((u, v, kind, cls))

    def graph(self, name, drop=()):
        """The CTA as a one-CTA Graph without the edge classes in ``drop``;
        parallel edges are merged (a DATA edge wins over an ISSUE edge)."""
        best = {}
        for u, v, kind, cls in self.edges:
            if cls in drop:
                continue
            best[(u, v)] = min(best.get((u, v), kind), kind)
        keys = sorted(best)
        src = [u for u, _ in keys]
        dst = [v for _, v in keys]
        kind = [best[k] for k in keys]
        n = len(self.t)
        return W.from_edges(name, self.warps, np.array(self.t, np.uint8), np.array(self.w, np.uint16),
                            np.zeros(n, np.uint32), np.array(self.wk, np.uint32), np.zeros(n, np.uint32),
                            np.zeros(1, np.uint32), src, dst, kind)


def _sizes(bm, bn, bk, rows, silu_ops, elem):
    return dict(a=rows * bk * elem, b=bn * bk * elem, mma=rows * bn * bk, ew=rows * bn * silu_ops,
                st=rows * bn * elem)


def _epilogue(c, warp, rows_sz, acc_from, prev_store, peers=()):
    """SiLU + store of one warp's rows; returns (ew, store).  ``peers``: MMAs of
    other warps the epilogue waits for at a barrier."""
    ew = c.node(W.EW, warp, rows_sz["ew"])
    for m in acc_from:
        c.edge(m, ew, FLOW)
    for m in peers:
        c.edge(m, ew, SYNC)
    c.edge(prev_store, ew, ORDER)      # the staging buffer was drained
    st = c.node(W.STORE, warp, rows_sz["st"])
    c.edge(ew, st, FLOW)
    return ew, st


def _naive(bm, bn, bk, tiles, stages, silu_ops, elem):
    c = _Cta(2)
    half = _sizes(bm, bn, bk, bm // 2, silu_ops, elem)
    ks = K_DIM // bk
    total = tiles * ks
    stage_bytes = (bm * bk + bn * bk) * elem
    lbytes = (stage_bytes + 1) // 2
    loads, mmas = {}, {}
    pending = [None, None]             # epilogue node the warp's next op must wait for
    stores = [None, None]

    def issue_load(j):
        loads[j] = []
        for w in (0, 1):
            ld = c.node(W.LOAD, w, lbytes)
            c.edge(pending[w], ld, ORDER)
            if j - stages in mmas:       # refill: both MMAs on the slot retired
                c.edge(mmas[j - stages][w], ld, ORDER)
                c.edge(mmas[j - stages][1 - w], ld, SYNC)
            loads[j].append(ld)
        for w in (0, 1):
            pending[w] = None

    for j in range(min(stages, total)):
        issue_load(j)
    for t in range(tiles):
        for k in range(ks):
            j = t * ks + k
            bars = []
            for w in (0, 1):
                b = c.node(W.BAR, w)
                c.edge(pending[w], b, ORDER)
                for ld in loads[j]:
                    c.edge(ld, b, SYNC)
                bars.append(b)
            mm = []
            for w in (0, 1):
                m = c.node(W.MMA, w, half["mma"])
                c.edge(bars[w], m, SYNC)
                for ld in loads[j]:
                    c.edge(ld, m, FLOW)
                if k:
                    c.edge(mmas[j - 1][w], m, FLOW, W.ISSUE)
                mm.append(m)
            for w in (0, 1):
                pending[w] = None
            mmas[j] = mm
            if j + stages < total:
                issue_load(j + stages)
        for w in (0, 1):
            ew, st = _epilogue(c, w, half, [mmas[t * ks + ks - 1][w]], stores[w])
            stores[w] = st
            pending[w] = ew            # the warp's registers are busy until SiLU is done
    return c


def _ws(bm, bn, bk, tiles, stages, silu_ops, elem, org, acc_buffers):
    pingpong = org == "ws_pingpong"
    three = org == "ws_3stage"
    c = _Cta(4 if three else 3)
    half = _sizes(bm, bn, bk, bm // 2, silu_ops, elem)
    full = _sizes(bm, bn, bk, bm, silu_ops, elem)
    ks = K_DIM // bk
    ring = []                           # per load: the MMAs that consume it
    pending = {1: None, 2: None}
    stores = {1: None, 2: None, 3: None}
    turn = None                         # last MMA issued in the other consumer's mainloop
    epi = []                            # 3-stage: epilogue EW per tile
    epi_pending = None

    def produce(nbytes):
        be = c.node(W.BAR, 0)
        if len(ring) >= stages:
            for m in ring[len(ring) - stages]:
                c.edge(m, be, SYNC)
        ld = c.node(W.LOAD, 0, nbytes)
        c.edge(be, ld, SYNC)
        return ld

    def consume(warp, ld, prev_mma, mma_work, first=None):
        bf = c.node(W.BAR, warp)
        c.edge(pending[warp], bf, ORDER)
        pending[warp] = None
        c.edge(ld, bf, SYNC)
        m = c.node(W.MMA, warp, mma_work)
        c.edge(bf, m, SYNC)
        c.edge(ld, m, FLOW)
        c.edge(prev_mma, m, FLOW, W.ISSUE)
        for u, kind in (first or ()):
            c.edge(u, m, SYNC, kind)
        return m

    for t in range(tiles):
        if pingpong:
            for s, warp in ((0, 1), (1, 2)):
                prev = None
                for k in range(ks):
                    ld = produce(half["a"] + half["b"])
                    first = [(turn, W.ISSUE)] if k == 0 and turn is not None else None
                    prev = consume(warp, ld, prev, half["mma"], first)
                    ring.append([prev])
                turn = prev
                ew, st = _epilogue(c, warp, half, [prev], stores[warp])
                stores[warp] = st
                pending[warp] = ew
        else:
            prev = {1: None, 2: None}
            for k in range(ks):
                ld = produce(full["a"] + full["b"])
                mm = []
                for warp in (1, 2):
                    first = None
                    if three and k == 0 and t >= acc_buffers:
                        first = [(epi[t - acc_buffers], W.DATA)]   # accumulator buffer drained
                    prev[warp] = consume(warp, ld, prev[warp], half["mma"], first)
                    mm.append(prev[warp])
                ring.append(mm)
            if three:
                ew = c.node(W.EW, 3, full["ew"])
                for warp in (1, 2):
                    c.edge(prev[warp], ew, FLOW)
                c.edge(stores[3], ew, ORDER)
                c.edge(epi_pending, ew, ORDER)
                st = c.node(W.STORE, 3, full["st"])
                c.edge(ew, st, FLOW)
                stores[3] = st
                epi_pending = ew
                epi.append(ew)
            else:
                for warp in (1, 2):
                    ew, st = _epilogue(c, warp, half, [prev[warp]], stores[warp], [prev[3 - warp]])
                    stores[warp] = st
                    pending[warp] = ew
    return c


def gemm_silu(org, bm, bn, bk, ablation="full", tiles=WAVES, stages=None, silu_ops=4, elem_bytes=2,
              acc_buffers=2):
    """One persistent GEMM + SiLU thread block as a tile graph (one CTA).
    ``stages`` defaults to 2 for the naive kernel and 4 for the WS ones."""
    if stages is None:
        stages = 2 if org == "naive_2stage" else 4
    if org not in ORGS or ablation not in ABLATIONS:
        raise KeyError((org, ablation))
    if bm % 2 or K_DIM % bk:
        raise ValueError("BM must be even and BK must divide K")
    if org == "naive_2stage":
        c = _naive(bm, bn, bk, tiles, stages, silu_ops, elem_bytes)
    else:
        c = _ws(bm, bn, bk, tiles, stages, silu_ops, elem_bytes, org, acc_buffers)
    return c.graph(f"{org}_{bm}x{bn}x{bk}_{ablation}", ABLATIONS[ablation])


def mma_fmas(bm, bn, tiles=WAVES):
    """FMAs of the whole kernel: tiles x BM x BN x K."""
    return tiles * bm * bn * K_DIM


def study_cases(orgs=ORGS, tiles=TILES, ablations=tuple(ABLATIONS)):
    """(org, tile, ablation) of every graph of the study, in stacking order."""
    return [(o, t, a) for o in orgs for t in tiles for a in ablations]


def study_set(orgs=ORGS, tiles=TILES, ablations=tuple(ABLATIONS), **kw):
    """All study graphs stacked into one graph set; returns (graph, cases)."""
    cases = study_cases(orgs, tiles, ablations)
    graphs = [gemm_silu(o, *t, ablation=a, **kw) for o, t, a in cases]
    return W.stack(graphs, "gemm_silu_pipelines"), cases


SINGLE_SM_HBM = (W.P_HBM_BPC, W.bytes_per_cycle(3.1) // 132, W.bytes_per_cycle(3.1))


def study_params(n_graphs, points_per_graph=1, seed=W.SEED0 + 6):
    """Single-SM Hopper rows (Table "GPU configurations" defaults, 1 SM, 1 CTA).
    Point 0 of every graph uses the defaults (the SM sees the whole DRAM
    bandwidth); points 1.. draw DRAM bandwidth between one SM's share of
    3.1 TB/s and all of it, and the tensor rate between 1024 and 4096 FMA/clk
    (A100 to B200), so the table spans memory- and compute-bound regimes.  The
    draws are made once and shared by every graph, so graphs are compared on
    the same hardware points."""
    base = W.default_params()
    base[W.P_NUM_SMS] = 1
    base[W.P_CTAS_PER_SM] = 1
    block = np.tile(base, (points_per_graph, 1))
    if points_per_graph > 1:
        rng = np.random.default_rng(seed)
        idx, lo, hi = SINGLE_SM_HBM
        block[1:, idx] = rng.integers(lo, hi + 1, points_per_graph - 1)
        block[1:, W.P_MMA_FMA_PC] = rng.integers(1024, 4096 + 1, points_per_graph - 1)
    rows = np.tile(block, (n_graphs, 1))
    rows[:, W.P_GRAPH_INDEX] = np.repeat(np.arange(n_graphs), points_per_graph)
    return np.ascontiguousarray(rows, np.int32)
