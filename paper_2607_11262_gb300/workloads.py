"""Seeded synthetic tile graphs and design-point parameter tables.

A tile graph (Section 4.1) is a DAG G = (V, E) whose nodes are warp-level tile
operations and whose edges are dependencies.  Each node records

* ``type``      -- its operation descriptor (LOAD, SMEM, MMA, EW, STORE, BAR, NOP,
                   DSMEM = a remote shared-memory access over the on-chip NoC),
                   which fixes the hardware unit that serves it (Section 4.1, 5.2);
* ``warp``      -- the CTA-local logical warp (execution group) that issues it;
                   a warpgroup is one logical warp (Section 4.1);
* ``cta``       -- the thread block it belongs to (Section 5.1);
* ``work``      -- the tile size reduced to one scalar: bytes for LOAD/SMEM/STORE,
                   FMAs for MMA, element operations for EW (Section 4.1 tile
                   descriptor);
* ``lat_extra`` -- an additive latency in cycles.

Edges are DATA (released when the producer completes) or ISSUE (an order edge,
released when the producer issues) (Section 4.1, Section 5.1).  Node ids are a
topological order (every edge goes from a lower to a higher id) and the program
order of each (cta, warp) stream is ascending id.  ``cta_kernel`` maps every CTA
to the kernel it belongs to; CTAs of a later kernel start only after every CTA
of the earlier kernels has retired (kernel boundaries, Section 4.2).

The workloads stand in for the paper's GEMM, FlashAttention and Llama decoder
kernels (Section 6.2, 6.3) with the shapes of those kernels; the random layered
DAG set is a stress case.  Everything here is input plumbing: this module holds
no scheduling arithmetic and is shared by the CUDA path and the CPU oracle.
"""
from __future__ import annotations

import dataclasses
import hashlib

import numpy as np

# ---------------------------------------------------------------- vocabulary
LOAD, SMEM, MMA, EW, STORE, BAR, NOP, DSMEM = range(8)
TYPE_NAMES = ("LOAD", "SMEM", "MMA", "EW", "STORE", "BAR", "NOP", "DSMEM")
DATA, ISSUE = 0, 1

NPARAM = 32
(P_NUM_SMS, P_CTAS_PER_SM, P_HBM_BPC, P_DRAM_LAT, P_TMA_BPC, P_TMA_LAT,
 P_SMEM_BPC, P_SMEM_LAT, P_MMA_FMA_PC, P_MMA_LAT, P_ALU_OPS_PC, P_ALU_LAT,
 P_BAR_LAT, P_CAP_TENSOR, P_CAP_TMA, P_CAP_LSU, P_CAP_ALU, P_CAP_BAR,
 P_CAP_HBM, P_GRAPH_INDEX, P_ISSUE_POLICY, P_SUBPARTITIONS, P_NOC_BPC, P_NOC_LAT, P_CAP_NOC,
 P_CLUSTER_SMS, P_L2_BYTES, P_L2_LAT, P_L2_BPC) = range(29)
PARAM_NAMES = ("num_sms", "ctas_per_sm", "hbm_bpc", "dram_lat", "tma_bpc",
               "tma_lat", "smem_bpc", "smem_lat", "mma_fma_pc", "mma_lat",
               "alu_ops_pc", "alu_lat", "bar_lat", "cap_tensor", "cap_tma",
               "cap_lsu", "cap_alu", "cap_bar", "cap_hbm", "graph_index",
               "issue_policy", "subpartitions", "noc_bpc", "noc_lat", "cap_noc",
               "cluster_sms", "l2_bytes", "l2_lat", "l2_bpc") + tuple(f"reserved{i}" for i in range(29, NPARAM))
# issue policies (Section 5.3): one global lowest-id order, or per-subpartition
# greedy-then-oldest / round-robin schedulers issuing one node per cycle
POLICY_LOWEST_ID, POLICY_GTO, POLICY_RR = 0, 1, 2

H100_CORE_HZ = 1.98e9  # H100 SXM core clock, Table "GPU configurations"


def bytes_per_cycle(tb_per_s: float) -> int:
    """DRAM bandwidth in bytes per core cycle at the H100 core clock."""
    return int(tb_per_s * 1e12 // H100_CORE_HZ)


def with_noc(p, noc_bpc=32, noc_lat=180, cap_noc=None, cluster_sms=16):
    """Rows ``p`` with an on-chip NoC: SM groups of ``cluster_sms``, each with
    ``cap_noc`` servers (default: one port per SM of the group) of ``noc_bpc``
    bytes per cycle and ``noc_lat`` cycles.  The paper gives no NoC figures;
    32 B/cycle and 180 cycles per DSMEM access are this framework's Hopper-like
    choice."""
    p = np.array(p, np.int32, copy=True)
    p[..., P_NOC_BPC] = noc_bpc
    p[..., P_NOC_LAT] = noc_lat
    p[..., P_CAP_NOC] = cluster_sms if cap_noc is None else cap_noc
    p[..., P_CLUSTER_SMS] = cluster_sms
    return p


def default_params() -> np.ndarray:
    """One parameter row with H100-like defaults (Table "GPU configurations").

    SM count 132, TC 2048 FMA/clk, SRAM 128 B/cycle at 33 cycles, DRAM 3.1 TB/s
    at 270 cycles, TMA 100 B/cycle.  TMA, MMA, ALU and barrier latencies are not
    given in the paper; the values below are this framework's choice.
    """
    p = np.zeros(NPARAM, dtype=np.int32)
    p[P_NUM_SMS] = 132
    p[P_CTAS_PER_SM] = 1
    p[P_HBM_BPC] = bytes_per_cycle(3.1)
    p[P_DRAM_LAT] = 270
    p[P_TMA_BPC] = 100
    p[P_TMA_LAT] = 0
    p[P_SMEM_BPC] = 128
    p[P_SMEM_LAT] = 33
    p[P_MMA_FMA_PC] = 2048
    p[P_MMA_LAT] = 32
    p[P_ALU_OPS_PC] = 128
    p[P_ALU_LAT] = 8
    p[P_BAR_LAT] = 20
    p[P_CAP_TENSOR] = 1
    p[P_CAP_TMA] = 1
    p[P_CAP_LSU] = 4
    p[P_CAP_ALU] = 4
    p[P_CAP_BAR] = 1
    p[P_CAP_HBM] = 1
    return p


# ---------------------------------------------------------------- graph container
@dataclasses.dataclass
class Graph:
    """A tile graph, or a stacked set of independent tile graphs.

    Node and CTA ids are global over the stack; graph ``g`` owns nodes
    ``node_off[g]:node_off[g+1]`` and CTAs ``cta_off[g]:cta_off[g+1]``, and no
    edge leaves its graph.  Successor lists are CSR (``row_ptr``, ``col``,
    ``ekind``).
    """
    name: str
    warps_per_cta: int
    row_ptr: np.ndarray      # uint32 [n+1]
    col: np.ndarray          # uint32 [m]
    ekind: np.ndarray        # uint8  [m]
    type: np.ndarray         # uint8  [n]
    warp: np.ndarray         # uint16 [n]
    cta: np.ndarray          # uint32 [n]
    work: np.ndarray         # uint32 [n]
    lat_extra: np.ndarray    # uint32 [n]
    cta_kernel: np.ndarray   # uint32 [C]
    node_off: np.ndarray     # uint32 [G+1]
    cta_off: np.ndarray      # uint32 [G+1]
    tile: np.ndarray = None  # uint32 [n] tile a LOAD/STORE reads or writes (NO_TILE: none); None: no tiles
    n_tiles: int = 0         # tile ids are < n_tiles

    @property
    def n_nodes(self) -> int:
        return int(self.type.shape[0])

    @property
    def n_edges(self) -> int:
        return int(self.col.shape[0])

    @property
    def n_ctas(self) -> int:
        return int(self.cta_kernel.shape[0])

    @property
    def n_graphs(self) -> int:
        return int(self.node_off.shape[0] - 1)

    @property
    def max_graph_nodes(self) -> int:
        return int(np.max(np.diff(self.node_off.astype(np.int64)))) if self.n_graphs else 0

    def subgraph(self, g: int) -> "Graph":
        """Graph ``g`` of a stack, with graph-local node and CTA ids."""
        n0, n1 = int(self.node_off[g]), int(self.node_off[g + 1])
        c0, c1 = int(self.cta_off[g]), int(self.cta_off[g + 1])
        e0, e1 = int(self.row_ptr[n0]), int(self.row_ptr[n1])
        return Graph(
            name=f"{self.name}[{g}]", warps_per_cta=self.warps_per_cta,
            row_ptr=(self.row_ptr[n0:n1 + 1] - e0).astype(np.uint32),
            col=(self.col[e0:e1] - n0).astype(np.uint32),
            ekind=self.ekind[e0:e1].copy(), type=self.type[n0:n1].copy(),
            warp=self.warp[n0:n1].copy(), cta=(self.cta[n0:n1] - c0).astype(np.uint32),
            work=self.work[n0:n1].copy(), lat_extra=self.lat_extra[n0:n1].copy(),
            cta_kernel=self.cta_kernel[c0:c1].copy(),
            node_off=np.array([0, n1 - n0], np.uint32),
            cta_off=np.array([0, c1 - c0], np.uint32),
            tile=None if self.tile is None else self.tile[n0:n1].copy(), n_tiles=self.n_tiles)

    def arrays(self):
        return {f.name: getattr(self, f.name) for f in dataclasses.fields(self)
                if isinstance(getattr(self, f.name), np.ndarray)}

    def sha256(self) -> str:
        h = hashlib.sha256()
        for k, a in sorted(self.arrays().items()):
            h.update(k.encode())
            h.update(np.ascontiguousarray(a).tobytes())
        h.update(str(self.warps_per_cta).encode())
        h.update(str(self.n_tiles).encode())
        return h.hexdigest()


NO_TILE = 0xFFFFFFFF


def from_edges(name, warps_per_cta, type_, warp, cta, work, lat_extra, cta_kernel,
               src, dst, kind, node_off=None, cta_off=None, tile=None, n_tiles=0) -> Graph:
    """Build a Graph from an edge list (sorted into CSR by source, then target)."""
    n = int(len(type_))
    src = np.asarray(src, np.int64)
    dst = np.asarray(dst, np.int64)
    kind = np.asarray(kind, np.uint8)
    order = np.lexsort((dst, src))
    src, dst, kind = src[order], dst[order], kind[order]
    row_ptr = np.zeros(n + 1, np.int64)
    np.cumsum(np.bincount(src, minlength=n), out=row_ptr[1:])
    C = int(len(cta_kernel))
    if node_off is None:
        node_off = np.array([0, n], np.uint32)
    if cta_off is None:
        cta_off = np.array([0, C], np.uint32)
    return Graph(name=name, warps_per_cta=int(warps_per_cta),
                 row_ptr=row_ptr.astype(np.uint32), col=dst.astype(np.uint32),
                 ekind=kind, type=np.asarray(type_, np.uint8),
                 warp=np.asarray(warp, np.uint16), cta=np.asarray(cta, np.uint32),
                 work=np.asarray(work, np.uint32), lat_extra=np.asarray(lat_extra, np.uint32),
                 cta_kernel=np.asarray(cta_kernel, np.uint32),
                 node_off=np.asarray(node_off, np.uint32), cta_off=np.asarray(cta_off, np.uint32),
                 tile=None if tile is None else np.asarray(tile, np.uint32), n_tiles=int(n_tiles))


def stack(graphs, name) -> Graph:
    """Concatenate independent graphs into one stacked set (ids made global)."""
    W = max(g.warps_per_cta for g in graphs)
    noff = np.zeros(len(graphs) + 1, np.int64)
    coff = np.zeros(len(graphs) + 1, np.int64)
    eoff = np.zeros(len(graphs) + 1, np.int64)
    for i, g in enumerate(graphs):
        noff[i + 1] = noff[i] + g.n_nodes
        coff[i + 1] = coff[i] + g.n_ctas
        eoff[i + 1] = eoff[i] + g.n_edges
    row_ptr = np.concatenate([g.row_ptr[:-1].astype(np.int64) + eoff[i] for i, g in enumerate(graphs)]
                             + [np.array([eoff[-1]])])
    return Graph(
        name=name, warps_per_cta=W, row_ptr=row_ptr.astype(np.uint32),
        col=np.concatenate([g.col.astype(np.int64) + noff[i] for i, g in enumerate(graphs)]).astype(np.uint32),
        ekind=np.concatenate([g.ekind for g in graphs]),
        type=np.concatenate([g.type for g in graphs]),
        warp=np.concatenate([g.warp for g in graphs]),
        cta=np.concatenate([g.cta.astype(np.int64) + coff[i] for i, g in enumerate(graphs)]).astype(np.uint32),
        work=np.concatenate([g.work for g in graphs]),
        lat_extra=np.concatenate([g.lat_extra for g in graphs]),
        cta_kernel=np.concatenate([g.cta_kernel for g in graphs]),
        node_off=noff.astype(np.uint32), cta_off=coff.astype(np.uint32),
        tile=(None if all(g.tile is None for g in graphs) else np.concatenate(
            [g.tile if g.tile is not None else np.full(g.n_nodes, NO_TILE, np.uint32) for g in graphs])),
        n_tiles=max(g.n_tiles for g in graphs))


# ---------------------------------------------------------------- CTA templates
class CtaTemplate:
    """The tile graph of one CTA, built in program order.

    Nodes get ascending local ids in the order they are added, so adding them
    in program-step order (all warps' step k before any warp's step k+1) keeps
    ids topological.  ``edge`` checks that every edge goes forward.
    """

    def __init__(self, warps: int):
        self.warps = warps
        self.t, self.w, self.wk, self.lx = [], [], [], []
        self.es, self.ed, self.ek = [], [], []

    def node(self, typ, warp, work=0, lat_extra=0):
        assert 0 <= warp < self.warps
        self.t.append(typ)
        self.w.append(warp)
        self.wk.append(work)
        self.lx.append(lat_extra)
        return len(self.t) - 1

    def edge(self, u, v, kind=DATA):
        assert u < v, (u, v)
        self.es.append(u)
        self.ed.append(v)
        self.ek.append(kind)

    def __len__(self):
        return len(self.t)

    def frozen(self):
        return (np.array(self.t, np.uint8), np.array(self.w, np.uint16),
                np.array(self.wk, np.uint32), np.array(self.lx, np.uint32),
                np.array(self.es, np.int64), np.array(self.ed, np.int64),
                np.array(self.ek, np.uint8))


@dataclasses.dataclass
class TemplateSet:
    """A template-shared graph (Section 6.4 "Graph construction"): physical CTA
    graphs stored once, and per logical CTA the template it runs and its kernel.

    Template t owns template nodes ``tpl_node_off[t]:tpl_node_off[t+1]``;
    successors are CSR over template nodes (``col`` indexes template nodes of
    the same template, sorted by source then target).  CTA c's nodes take the
    next block of logical ids in CTA order.  A stacked set gives each graph g
    the CTAs ``graph_cta_off[g]:graph_cta_off[g+1]``.
    """
    name: str
    warps_per_cta: int
    tpl_node_off: np.ndarray   # uint32 [T+1]
    row_ptr: np.ndarray        # uint32 [TN+1]
    col: np.ndarray            # uint32 [TE]
    ekind: np.ndarray          # uint8  [TE]
    type: np.ndarray           # uint8  [TN]
    warp: np.ndarray           # uint16 [TN]
    work: np.ndarray           # uint32 [TN]
    lat_extra: np.ndarray      # uint32 [TN]
    cta_template: np.ndarray   # uint32 [C]
    cta_kernel: np.ndarray     # uint32 [C]
    graph_cta_off: np.ndarray  # uint32 [G+1]

    @property
    def n_templates(self):
        return int(self.tpl_node_off.shape[0] - 1)

    @property
    def n_ctas(self):
        return int(self.cta_template.shape[0])

    @property
    def n_graphs(self):
        return int(self.graph_cta_off.shape[0] - 1)

    def sizes(self):
        """Nodes and edges of each template."""
        off = self.tpl_node_off.astype(np.int64)
        return np.diff(off), np.diff(self.row_ptr.astype(np.int64)[off])

    @property
    def n_nodes(self):
        return int(self.sizes()[0][self.cta_template].sum())

    @property
    def n_edges(self):
        return int(self.sizes()[1][self.cta_template].sum())

    def expand(self) -> Graph:
        """The logical graph (every CTA's copy of its template, CTA-major ids)."""
        off = self.tpl_node_off.astype(np.int64)
        nsz, esz = self.sizes()
        ct = self.cta_template.astype(np.int64)
        cnt = nsz[ct]
        base = np.zeros(len(ct) + 1, np.int64)
        np.cumsum(cnt, out=base[1:])
        n = int(base[-1])
        # template node of every logical node, and its CTA
        cta = np.repeat(np.arange(len(ct)), cnt)
        u = off[ct][cta] + (np.arange(n) - base[:-1][cta])
        rp = self.row_ptr.astype(np.int64)
        deg = rp[u + 1] - rp[u]
        src = np.repeat(np.arange(n), deg)
        first_edge = np.repeat(rp[u], deg)
        x = first_edge + (np.arange(src.shape[0]) - np.repeat(np.cumsum(deg) - deg, deg))
        dst = base[:-1][cta[src]] + (self.col.astype(np.int64)[x] - off[ct[cta[src]]])
        graphs = self.graph_cta_off.astype(np.int64)
        return from_edges(self.name, self.warps_per_cta, self.type[u], self.warp[u], cta.astype(np.uint32),
                          self.work[u], self.lat_extra[u], self.cta_kernel, src, dst, self.ekind[x],
                          node_off=base[graphs].astype(np.uint32), cta_off=self.graph_cta_off)


def template_set(name, warps_per_cta, templates, cta_template, cta_kernel, graph_cta_off=None) -> TemplateSet:
    """CtaTemplates plus the per-CTA table as a TemplateSet."""
    frozen = [t.frozen() for t in templates]
    sizes = [len(f[0]) for f in frozen]
    off = np.zeros(len(frozen) + 1, np.int64)
    np.cumsum(sizes, out=off[1:])
    rows, cols, kinds = [np.zeros(1, np.int64)], [], []
    edges_so_far = 0
    for i, (_t, _w, _wk, _x, es, ed, ek) in enumerate(frozen):
        order = np.lexsort((ed, es))
        es, ed, ek = es[order], ed[order], ek[order]
        cnt = np.bincount(es, minlength=sizes[i])
        rows.append(edges_so_far + np.cumsum(cnt))
        cols.append(off[i] + ed)
        kinds.append(ek)
        edges_so_far += len(es)
    cat = lambda parts, dt: np.concatenate(parts).astype(dt) if parts else np.zeros(0, dt)  # noqa: E731
    C = len(cta_template)
    return TemplateSet(
        name=name, warps_per_cta=int(warps_per_cta), tpl_node_off=off.astype(np.uint32),
        row_ptr=np.concatenate(rows).astype(np.uint32), col=cat(cols, np.uint32), ekind=cat(kinds, np.uint8),
        type=cat([f[0] for f in frozen], np.uint8), warp=cat([f[1] for f in frozen], np.uint16),
        work=cat([f[2] for f in frozen], np.uint32), lat_extra=cat([f[3] for f in frozen], np.uint32),
        cta_template=np.asarray(cta_template, np.uint32), cta_kernel=np.asarray(cta_kernel, np.uint32),
        graph_cta_off=np.array([0, C], np.uint32) if graph_cta_off is None else np.asarray(graph_cta_off, np.uint32))


def assemble(name, warps_per_cta, templates, cta_template, cta_kernel) -> Graph:
    """Replicate CTA templates into one graph (vectorised; CTAs laid out in order).

    ``cta_template[c]`` is the template index of CTA ``c``; CTA ``c``'s nodes get
    the next contiguous block of ids, so ids stay topological across CTAs.
    """
    frozen = [t.frozen() for t in templates]
    sizes = np.array([len(f[0]) for f in frozen], np.int64)
    cta_template = np.asarray(cta_template, np.int64)
    C = len(cta_template)
    cnt = sizes[cta_template]
    off = np.zeros(C + 1, np.int64)
    np.cumsum(cnt, out=off[1:])
    n = int(off[-1])
    typ = np.empty(n, np.uint8)
    warp = np.empty(n, np.uint16)
    work = np.empty(n, np.uint32)
    lx = np.empty(n, np.uint32)
    cta = np.empty(n, np.uint32)
    srcs, dsts, kinds = [], [], []
    for ti, (t, w, wk, x, es, ed, ek) in enumerate(frozen):
        ctas = np.nonzero(cta_template == ti)[0]
        if len(ctas) == 0 or len(t) == 0:
            continue
        base = off[ctas]
        pos = (base[:, None] + np.arange(len(t))[None, :]).ravel()
        k = len(ctas)
        typ[pos] = np.tile(t, k)
        warp[pos] = np.tile(w, k)
        work[pos] = np.tile(wk, k)
        lx[pos] = np.tile(x, k)
        cta[pos] = np.repeat(ctas, len(t)).astype(np.uint32)
        if len(es):
            srcs.append((base[:, None] + es[None, :]).ravel())
            dsts.append((base[:, None] + ed[None, :]).ravel())
            kinds.append(np.tile(ek, k))
    src = np.concatenate(srcs) if srcs else np.zeros(0, np.int64)
    dst = np.concatenate(dsts) if dsts else np.zeros(0, np.int64)
    kind = np.concatenate(kinds) if kinds else np.zeros(0, np.uint8)
    return from_edges(name, warps_per_cta, typ, warp, cta, work, lx, cta_kernel, src, dst, kind)


# ---------------------------------------------------------------- kernel templates
def gemm_2stage_cta(ksteps=8, warps=4, load_bytes=8192, smem_bytes=16384,
                    mma_fma=262144, ew_ops=4096, store_bytes=8192, stages=2):
    """Non-warp-specialised multi-stage GEMM CTA (cp.async style, Section 4.2).

    Every warp loads its share of the A/B k-slice, all warps meet at a CTA
    barrier once the slice has landed, stage their fragments out of shared
    memory and run the MMA.  The load that refills a buffer waits for every
    warp's MMA on the slice the buffer held (buffer reuse, emitted as DATA).
    Epilogue: elementwise then store.
    """
    t = CtaTemplate(warps)
    loads = {}
    mmas = {}

    def issue_load(k):
        for w in range(warps):
            ld = t.node(LOAD, w, load_bytes)
            if k - stages in mmas:
                for m in mmas[k - stages]:
                    t.edge(m, ld)
            loads.setdefault(k, []).append(ld)

    for k in range(min(stages, ksteps)):
        issue_load(k)
    last = [None] * warps
    for k in range(ksteps):
        bars = [t.node(BAR, w) for w in range(warps)]
        for b in bars:
            for ld in loads[k]:
                t.edge(ld, b)
        sm = [t.node(SMEM, w, smem_bytes) for w in range(warps)]
        for w in range(warps):
            t.edge(bars[w], sm[w])
        mm = [t.node(MMA, w, mma_fma) for w in range(warps)]
        for w in range(warps):
            t.edge(sm[w], mm[w])
        mmas[k] = mm
        last = mm
        if k + stages < ksteps:
            issue_load(k + stages)
    ews = [t.node(EW, w, ew_ops) for w in range(warps)]
    for w in range(warps):
        t.edge(last[w], ews[w])
    sts = [t.node(STORE, w, store_bytes) for w in range(warps)]
    for w in range(warps):
        t.edge(ews[w], sts[w])
    return t


def ws_gemm_cta(tiles, ksteps, stages=4, load_bytes=49152, mma_fma=1048576,
                ew_ops=16384, store_bytes=32768):
    """Warp-specialised persistent GEMM CTA (Section 4.2 / Fig. tile-graph (b)).

    Warp 0 is the TMA producer; warps 1 and 2 are the two consumer warpgroups.
    Per k-step the producer waits on the 'empty' barrier of the ring slot and
    issues one TMA load of the A and B slices; each consumer waits on the 'full'
    barrier and issues its MMA.  A slot is refilled only after both consumers'
    MMAs on the tile it held completed (``stages``-deep ring).  Per tile each
    consumer runs an elementwise epilogue and a TMA store.  The ring continues
    across the tiles a persistent CTA processes.
    """
    t = CtaTemplate(3)
    ring = []
    for _ in range(tiles):
        last = None
        for _k in range(ksteps):
            be = t.node(BAR, 0)
            if len(ring) >= stages:
                for m in ring[len(ring) - stages]:
                    t.edge(m, be)
            ld = t.node(LOAD, 0, load_bytes)
            t.edge(be, ld)
            mm = []
            for c in (1, 2):
                bf = t.node(BAR, c)
                t.edge(ld, bf)
                m = t.node(MMA, c, mma_fma)
                t.edge(bf, m)
                mm.append(m)
            ring.append(mm)
            last = mm
        for i, c in enumerate((1, 2)):
            ew = t.node(EW, c, ew_ops)
            t.edge(last[i], ew)
            st = t.node(STORE, c, store_bytes)
            t.edge(ew, st)
    return t


def fa_fwd_cta(kv_blocks, stages=2, q_bytes=32768, kv_bytes=32768, qk_fma=1048576,
               softmax_ops=32768, pv_fma=1048576, norm_ops=8192, o_bytes=16384):
    """FlashAttention-3 style forward CTA for one 128-row Q block.

    Warp 0 (producer) loads Q once, then per KV block waits on the 'empty'
    barrier and issues TMA loads of K and V.  Warps 1 and 2 (consumer
    warpgroups, 64 rows each) per KV block: wait for K, QK^T MMA, online softmax
    (elementwise), wait for V, PV MMA.  Consumer 1's QK^T issues only after
    consumer 0's QK^T issued and consumer 0's next QK^T only after consumer 1's
    PV issued (warpgroup ping-pong ordering, ISSUE edges).  A K/V slot is
    refilled after both consumers' PV MMAs on it completed.  Epilogue per
    consumer: normalisation and an O store.
    """
    t = CtaTemplate(3)
    q = t.node(LOAD, 0, q_bytes)
    ring = []
    prev_pv1 = None
    last_pv = [None, None]
    for j in range(kv_blocks):
        be = t.node(BAR, 0)
        if j >= stages:
            for m in ring[j - stages]:
                t.edge(m, be)
        lk = t.node(LOAD, 0, kv_bytes)
        t.edge(be, lk)
        lv = t.node(LOAD, 0, kv_bytes)
        pvs = []
        qk0 = None
        for i, c in enumerate((1, 2)):
            bk = t.node(BAR, c)
            t.edge(lk, bk)
            if j == 0:
                t.edge(q, bk)
            qk = t.node(MMA, c, qk_fma)
            t.edge(bk, qk)
            if i == 0:
                qk0 = qk
                if prev_pv1 is not None:
                    t.edge(prev_pv1, qk, ISSUE)
            else:
                t.edge(qk0, qk, ISSUE)
            sm = t.node(EW, c, softmax_ops)
            t.edge(qk, sm)
            bv = t.node(BAR, c)
            t.edge(lv, bv)
            pv = t.node(MMA, c, pv_fma)
            t.edge(bv, pv)
            t.edge(sm, pv)
            pvs.append(pv)
        ring.append(pvs)
        prev_pv1 = pvs[1]
        last_pv = pvs
    for i, c in enumerate((1, 2)):
        ew = t.node(EW, c, norm_ops)
        t.edge(last_pv[i], ew)
        st = t.node(STORE, c, o_bytes)
        t.edge(ew, st)
    return t


def ew_cta(warps=4, loads=(131072,), ew_ops=262144, stores=(131072,)):
    """Row-parallel elementwise kernel CTA (RMSNorm, SiLU*mul, residual add).

    Each warp loads its rows, runs the elementwise op once every load landed
    and stores the results.
    """
    t = CtaTemplate(warps)
    lds = [[t.node(LOAD, w, b) for w in range(warps)] for b in loads]
    ews = [t.node(EW, w, ew_ops) for w in range(warps)]
    for w in range(warps):
        for row in lds:
            t.edge(row[w], ews[w])
    for b in stores:
        for w in range(warps):
            st = t.node(STORE, w, b)
            t.edge(ews[w], st)
    return t


# ---------------------------------------------------------------- the five workloads
def _build(name, warps, templates, cta_template, cta_kernel, templated):
    """The logical graph, or with ``templated`` the template-shared form."""
    if templated:
        return template_set(name, warps, templates, cta_template, cta_kernel)
    return assemble(name, warps, templates, cta_template, cta_kernel)


def gemm512(templated=False):
    """GEMM M=N=K=512 fp16, 128x128x64 CTA tiles (4x4 = 16 CTAs), 4 warps, 2-stage."""
    tpl = gemm_2stage_cta(ksteps=512 // 64)
    return _build("gemm512", 4, [tpl], np.zeros(16, np.int64), np.zeros(16, np.uint32), templated)


def ws_gemm(M=8192, N=8192, K=8192, num_ctas=132, name="wsgemm8192", templated=False):
    """Warp-specialised persistent GEMM (bf16, 128x256x64 tiles).

    (M/128)*(N/256) output tiles over ``num_ctas`` persistent CTAs (tile t ->
    CTA t mod num_ctas), 4-stage ring, K/64 k-steps per tile.
    """
    tiles = (M // 128) * (N // 256)
    per = np.array([tiles // num_ctas + (1 if c < tiles % num_ctas else 0) for c in range(num_ctas)])
    kinds = sorted(set(per.tolist()), reverse=True)
    tpls = [ws_gemm_cta(k, K // 64) for k in kinds]
    ct = np.array([kinds.index(x) for x in per], np.int64)
    return _build(name, 3, tpls, ct, np.zeros(num_ctas, np.uint32), templated)


def wsgemm8192(num_ctas=132, templated=False):
    """M=N=K=8192: 2048 tiles over 132 persistent CTAs, 128 k-steps per tile."""
    return ws_gemm(8192, 8192, 8192, num_ctas, templated=templated)


def fa_fwd(batch=4, heads=32, seq=4096, head_dim=128, q_block=128, kv_block=128, templated=False):
    """FlashAttention forward, non-causal: one CTA per (batch, head, Q block)."""
    assert head_dim == 128
    nq = seq // q_block
    tpl = fa_fwd_cta(seq // kv_block)
    C = batch * heads * nq
    return _build("fa_fwd", 3, [tpl], np.zeros(C, np.int64), np.zeros(C, np.uint32), templated)


def decoder_layer(hidden=4096, heads=32, ffn=11008, tokens=16384, seq=2048, templated=False):
    """One Llama-style decoder layer for prefill of ``tokens`` tokens (fp16).

    Kernels in stream order (each a kernel-boundary gate for the next):
    RMSNorm, QKV GEMM, causal attention, O GEMM, residual add + RMSNorm,
    gate/up GEMM, SiLU*mul, down GEMM, residual add.
    GEMMs use the warp-specialised tile template with one tile per CTA
    (128x256x64); elementwise kernels process 64 rows per CTA with 4 warps.
    """
    rows_per_cta = 64
    ew_ctas = tokens // rows_per_cta
    rows_w = rows_per_cta // 4
    tpls, cta_t, cta_k = [], [], []

    def add(tpl, count, kernel):
        tpls.append(tpl)
        cta_t.extend([len(tpls) - 1] * count)
        cta_k.extend([kernel] * count)

    def gemm(n_out, k_in, kernel):
        count = (tokens // 128) * (n_out // 256)
        add(ws_gemm_cta(1, k_in // 64), count, kernel)

    hb = rows_w * hidden * 2
    add(ew_cta(loads=(hb,), ew_ops=rows_w * hidden * 4, stores=(hb,)), ew_ctas, 0)
    gemm(3 * hidden, hidden, 1)
    nq = seq // 128
    batch = tokens // seq
    att = [fa_fwd_cta(i + 1) for i in range(nq)]
    base = len(tpls)
    tpls.extend(att)
    for _b in range(batch):
        for _h in range(heads):
            for i in range(nq):
                cta_t.append(base + i)
                cta_k.append(2)
    gemm(hidden, hidden, 3)
    add(ew_cta(loads=(hb, hb), ew_ops=rows_w * hidden * 5, stores=(hb, hb)), ew_ctas, 4)
    gemm(2 * ffn + (256 - (2 * ffn) % 256) % 256, hidden, 5)
    fb = rows_w * ffn * 2
    add(ew_cta(loads=(2 * fb,), ew_ops=rows_w * ffn * 4, stores=(fb,)), ew_ctas, 6)
    gemm(hidden, ffn, 7)
    add(ew_cta(loads=(hb, hb), ew_ops=rows_w * hidden, stores=(hb,)), ew_ctas, 8)
    return _build("decoder", 4, tpls, np.array(cta_t), np.array(cta_k, np.uint32), templated)


def random_layered_dag(seed, n_nodes=100_000, layers=64, fan_in=(1, 4), lat_log2=(2.0, 12.0),
                       warps=16, ctas=8, issue_frac=0.0, name="stress") -> Graph:
    """Random layered DAG (stress case).

    Ids are layer-major; every node after the first layer draws k ~ U{fan_in}
    distinct predecessors uniformly from all earlier layers.  Latency
    floor(2^U(lat_log2)) cycles is carried as ``work`` so that occupancy equals
    latency when every rate is 1 and every base latency 0.  Type is uniform over
    LOAD, MMA, EW, STORE and the issuing (cta, warp) uniform over ctas x warps.
    With ``issue_frac`` > 0 that fraction of edges are ISSUE edges.
    """
    rng = np.random.default_rng(seed)
    sizes = np.full(layers, n_nodes // layers, np.int64)
    sizes[: n_nodes % layers] += 1
    lstart = np.zeros(layers + 1, np.int64)
    np.cumsum(sizes, out=lstart[1:])
    node_layer = np.repeat(np.arange(layers), sizes)
    lat = np.floor(2.0 ** rng.uniform(lat_log2[0], lat_log2[1], n_nodes)).astype(np.int64)
    typ = rng.choice(np.array([LOAD, MMA, EW, STORE], np.uint8), n_nodes)
    flat = rng.integers(0, warps * ctas, n_nodes)
    cta = (flat // warps).astype(np.uint32)
    warp = (flat % warps).astype(np.uint16)
    srcs, dsts = [], []
    later = np.arange(lstart[1], n_nodes)
    k = rng.integers(fan_in[0], fan_in[1] + 1, later.shape[0])
    avail = lstart[node_layer[later]]   # number of nodes in earlier layers
    kmax = fan_in[1]
    cand = np.floor(rng.random((later.shape[0], kmax)) * avail[:, None]).astype(np.int64)
    # resample duplicates among the first k picks until each row is distinct
    for _ in range(100):
        dup = np.zeros(cand.shape, bool)
        for a in range(kmax):
            for b in range(a):
                dup[:, a] |= cand[:, a] == cand[:, b]
        dup &= np.arange(kmax)[None, :] < k[:, None]
        if not dup.any():
            break
        r, c = np.nonzero(dup)
        cand[r, c] = np.floor(rng.random(r.shape[0]) * avail[r]).astype(np.int64)
    sel = np.arange(kmax)[None, :] < k[:, None]
    srcs = cand[sel]
    dsts = np.repeat(later, k)
    kinds = np.zeros(srcs.shape[0], np.uint8)
    if issue_frac > 0:
        kinds = (rng.random(srcs.shape[0]) < issue_frac).astype(np.uint8)
    return from_edges(name, warps, typ, warp, cta, lat.astype(np.uint32),
                      np.zeros(n_nodes, np.uint32), np.zeros(ctas, np.uint32), srcs, dsts, kinds)


def stress_set(instances=256, n_nodes=100_000, seed0=2607_5000) -> Graph:
    """``instances`` distinct random layered DAGs (seeds seed0 + i) as one stack."""
    return stack([random_layered_dag(seed0 + i, n_nodes) for i in range(instances)], "stress")


def stress_params(instances=256) -> np.ndarray:
    """One row per stress instance: 8 SMs x 1 CTA, every rate 1, base latency 0,
    4 HBM servers and 1 server of every per-SM class; row i runs graph i."""
    p = np.tile(default_params(), (instances, 1))
    p[:, P_NUM_SMS] = 8
    p[:, P_CTAS_PER_SM] = 1
    for i in (P_HBM_BPC, P_TMA_BPC, P_SMEM_BPC, P_MMA_FMA_PC, P_ALU_OPS_PC):
        p[:, i] = 1
    for i in (P_DRAM_LAT, P_TMA_LAT, P_SMEM_LAT, P_MMA_LAT, P_ALU_LAT, P_BAR_LAT):
        p[:, i] = 0
    for i in (P_CAP_TENSOR, P_CAP_TMA, P_CAP_LSU, P_CAP_ALU, P_CAP_BAR):
        p[:, i] = 1
    p[:, P_CAP_HBM] = 4
    p[:, P_GRAPH_INDEX] = np.arange(instances)
    return p


def sweep_params(seed, points, axes, ctas_per_sm) -> np.ndarray:
    """``points`` rows around the defaults; each axis (index, lo, hi) is drawn
    uniformly over the integers lo..hi with numpy's PCG64 seeded by ``seed``."""
    rng = np.random.default_rng(seed)
    p = np.tile(default_params(), (points, 1))
    p[:, P_CTAS_PER_SM] = ctas_per_sm
    for idx, lo, hi in axes:
        p[:, idx] = rng.integers(lo, hi + 1, points)
    return p


SEED0 = 2607_0000
AX_SMS = (P_NUM_SMS, 8, 132)
AX_HBM = (P_HBM_BPC, bytes_per_cycle(1.0), bytes_per_cycle(8.0))
AX_TMA_LAT = (P_TMA_LAT, 128, 1024)
AX_MMA_RATE = (P_MMA_FMA_PC, 1024, 4096)
AX_ALU_RATE = (P_ALU_OPS_PC, 64, 128)


@dataclasses.dataclass
class Workload:
    name: str
    description: str
    graph: Graph
    params: np.ndarray


TEMPLATED = ("gemm512", "wsgemm8192", "wsgemm_small", "fa_fwd", "fa_small", "decoder", "decoder_small")


def workload(name: str, points: int | None = None, instances: int | None = None,
             templated: bool = False) -> Workload:
    """One of the named workloads (graph + parameter table).

    ``points`` truncates the parameter table (the rows are drawn for the full
    size, so a prefix is the same rows); ``instances`` shrinks the stress set;
    ``templated`` returns the graph as a TemplateSet (the workloads in
    TEMPLATED, whose CTAs run shared templates).
    """
    if templated and name not in TEMPLATED:
        raise ValueError(f"{name} has no template-shared form")
    if name == "gemm512":
        g = gemm512(templated)
        p = sweep_params(SEED0 + 1, 64, [AX_SMS, AX_HBM, (P_MMA_LAT, 16, 64)], 2)
        d = "GEMM 512^3 fp16, 128x128x64 tiles, 4 warps, 2-stage; 64 points"
    elif name == "wsgemm8192":
        g = wsgemm8192(templated=templated)
        p = sweep_params(SEED0 + 2, 4096, [AX_SMS, AX_HBM, AX_TMA_LAT, AX_MMA_RATE], 1)
        d = "WS persistent GEMM 8192^3 bf16, 128x256x64, 1 producer + 2 consumer WGs, 4-stage ring, 132 CTAs; 4096 points"
    elif name == "wsgemm_small":
        g = ws_gemm(2048, 2048, 1024, 132, "wsgemm_small", templated=templated)
        p = sweep_params(SEED0 + 2, 4096, [AX_SMS, AX_HBM, AX_TMA_LAT, AX_MMA_RATE], 1)
        d = "WS GEMM 2048x2048x1024 (profiling-size case of the wsgemm8192 kernel shape); 4096 points"
    elif name == "fa_fwd":
        g = fa_fwd(templated=templated)
        p = sweep_params(SEED0 + 3, 1024, [AX_SMS, AX_HBM, AX_TMA_LAT, AX_MMA_RATE, AX_ALU_RATE], 1)
        d = "FlashAttention fwd B4 H32 S4096 d128 fp16, non-causal; 1024 points"
    elif name == "fa_small":
        g = fa_fwd(batch=1, heads=16, seq=2048, templated=templated)
        p = sweep_params(SEED0 + 3, 1024, [AX_SMS, AX_HBM, AX_TMA_LAT, AX_MMA_RATE, AX_ALU_RATE], 1)
        d = "FlashAttention fwd B1 H16 S2048 d128 (profiling-size case of the fa_fwd shape); 1024 points"
    elif name == "decoder_small":
        g = decoder_layer(hidden=1024, heads=8, ffn=2816, tokens=2048, seq=512, templated=templated)
        p = sweep_params(SEED0 + 4, 512, [AX_SMS, AX_HBM, AX_TMA_LAT, AX_MMA_RATE, AX_ALU_RATE], 1)
        d = "decoder layer hidden 1024, 8 heads, FFN 2816, 4x512 tokens (profiling-size case of the decoder shape); 512 points"
    elif name == "decoder":
        g = decoder_layer(templated=templated)
        p = sweep_params(SEED0 + 4, 512, [AX_SMS, AX_HBM, AX_TMA_LAT, AX_MMA_RATE, AX_ALU_RATE], 1)
        d = "Llama-style decoder layer prefill, hidden 4096, 32 heads, FFN 11008, 8x2048 tokens; 512 points"
    elif name == "stress":
        k = 256 if instances is None else instances
        g = stress_set(k)
        p = stress_params(k)
        d = f"{k} random layered DAGs x 100k nodes, 64 layers, fan-in 1-4, latency 4-4096"
    elif name == "pipelines":
        from . import pipelines
        g, cases = pipelines.study_set()
        p = pipelines.study_params(len(cases), 64)
        d = (f"GEMM+SiLU pipeline study: 4 organisations x {len(pipelines.TILES)} tiles x 4 ablations, "
             "10 waves on 1 SM; 64 points per graph (DRAM and tensor rate swept)")
    elif name == "l2_gemm":
        from . import l2gemm
        g, orders = l2gemm.study_set()
        p = l2gemm.study_params(len(orders), points_per_capacity=8)
        d = ("persistent WS GEMM 4096^3 bf16, 128x256x64, 132 CTAs, A/B/C loads and stores naming tiles, row-major "
             "and grouped rasterization; L2 0-100 MB (LRU over tiles), 8 DRAM rates each")
    elif name == "noc_fusion":
        from . import clusters
        g, cases = clusters.study_set()
        p = clusters.study_params(cases, points_per_graph=32)
        d = ("cluster-fused attention decode (H 4096, 32 heads, d 128, KV 1024), clusters of 2-16 CTAs, "
             "NoC vs DRAM exchanges; 32 points per graph (NoC and DRAM rates swept)")
    else:
        raise KeyError(name)
    if points is not None:
        p = p[:points]
    return Workload(name, d, g, np.ascontiguousarray(p, np.int32))


WORKLOADS = ("gemm512", "wsgemm8192", "fa_fwd", "decoder", "stress")
STUDIES = ("pipelines", "noc_fusion", "l2_gemm")
