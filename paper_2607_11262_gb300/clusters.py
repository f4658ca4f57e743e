"""Cluster-fused attention decode with on-chip (NoC) or DRAM communication
(case study "NoC-enabled Fusion and Mapping", Section 7.2).

One decode step of one attention layer (batch 1, hidden H, ``heads`` heads of
dimension d, KV length S).  Every head runs on a cluster of ``k`` thread
blocks (one logical warp each); block r of a head works on 1/k of the head:
a slice of the QKV-projection outputs, S/k keys and values (split-KV
attention), and H/k outputs of the output projection.  The blocks of a
cluster exchange intermediates five times -- a reduce after RMSNorm, a gather
after the QKV projection, two reduces inside attention (the running max and
the exp-sum), and a reduce of the partial outputs after the rescale:

* ``noc``:  each block writes its payload into every peer's shared memory
  (one DSMEM node per peer), waits at a cluster barrier for the peers'
  writes (cross-block DATA edges into its BAR node), and combines;
* ``dram``: each block stores its payload to global memory, waits at the
  barrier for the peers' stores, loads the k-1 peer payloads back and
  combines.

All weight and KV loads are issued up front (prefetch) and the compute nodes
wait for them.  Node ids are numbered stage by stage across all blocks (all
blocks' stage-s nodes before any stage-(s+1) node), so the cross-block edges
of the exchanges go forward and each block's program order is ascending.

Input plumbing only: graphs and parameter rows, no scheduling arithmetic.
"""
from __future__ import annotations

import numpy as np

from . import workloads as W

MODES = ("noc", "dram")
CLUSTER_SIZES = (2, 4, 8, 16)


def fused_attention(k, mode, hidden=4096, heads=32, head_dim=128, kv_len=1024, elem=2):
    """The fused attention decode kernel as one tile graph (heads * k CTAs)."""
    if mode not in MODES or k < 2:
        raise ValueError((k, mode))
    H, d, S = hidden, head_dim, kv_len
    C = heads * k
    typ, warp, cta, work = [], [], [], []
    src, dst, kind = [], [], []

    def node(t, c, w=0):
        typ.append(t)
        warp.append(0)
        cta.append(c)
        work.append(int(w))
        return len(typ) - 1

    def edge(u, v):
        assert u < v
        src.append(u)
        dst.append(v)
        kind.append(W.DATA)

    def stage(fn):
        """Adds one stage's nodes for every block (stage-major ids)."""
        return [fn(c) for c in range(C)]

    def exchange(prev, payload):
        """Cluster exchange of ``payload`` bytes per block after node prev[c];
        returns each block's combine node."""
        def peers(c):
            h = c // k
            return [h * k + j for j in range(k) if h * k + j != c]
        if mode == "noc":
            writes = stage(lambda c: [node(W.DSMEM, c, payload) for _ in range(k - 1)])
            for c in range(C):
                for x in writes[c]:
                    edge(prev[c], x)
            bars = stage(lambda c: node(W.BAR, c))
            for c in range(C):
                for p, x in zip(peers(c), range(k - 1)):
                    # block c's x-th write goes to its x-th peer p
                    edge(writes[c][x], bars[p])
            done = bars
        else:
            stores = stage(lambda c: node(W.STORE, c, payload))
            for c in range(C):
                edge(prev[c], stores[c])
            bars = stage(lambda c: node(W.BAR, c))
            for c in range(C):
                for p in peers(c):
                    edge(stores[p], bars[c])
            loads = stage(lambda c: node(W.LOAD, c, (k - 1) * payload))
            for c in range(C):
                edge(bars[c], loads[c])
            done = loads
        comb = stage(lambda c: node(W.EW, c, (k - 1) * max(payload // elem, 1)))
        for c in range(C):
            edge(done[c], comb[c])
        return comb

    def step(prev, t, w, *deps):
        out = stage(lambda c: node(t, c, w))
        for c in range(C):
            edge(prev[c], out[c])
            for dd in deps:
                edge(dd[c], out[c])
        return out

    # prefetch: x, this block's QKV-weight slice, K and V slices, Wo slice
    x = stage(lambda c: node(W.LOAD, c, H * elem))
    wqkv = stage(lambda c: node(W.LOAD, c, H * 3 * d // k * elem))
    kk = stage(lambda c: node(W.LOAD, c, S // k * d * elem))
    vv = stage(lambda c: node(W.LOAD, c, S // k * d * elem))
    wo = stage(lambda c: node(W.LOAD, c, d * H // k * elem))
    sq = step(x, W.EW, H // k)                        # partial sum of squares
    r1 = exchange(sq, 16)                             # reduce after RMSNorm
    nrm = step(r1, W.EW, H)                           # normalise x
    qkv = step(nrm, W.MMA, H * 3 * d // k, wqkv)      # QKV projection slice
    g = exchange(qkv, 3 * d // k * elem)              # gather q, k, v
    rope = step(g, W.EW, 3 * d)
    qk = step(rope, W.MMA, S // k * d, kk)            # scores on this block's keys
    mx = step(qk, W.EW, S // k)                       # local max
    r2 = exchange(mx, 16)                             # reduce: max
    ex = step(r2, W.EW, 2 * S // k)                   # exp and local sum
    r3 = exchange(ex, 16)                             # reduce: exp-sum
    pv = step(r3, W.MMA, S // k * d, vv, ex)          # partial output
    rs = step(pv, W.EW, d)                            # rescale
    r4 = exchange(rs, d * 4)                          # reduce partial outputs (fp32)
    out = step(r4, W.MMA, d * H // k, wo)             # output projection slice
    step(out, W.STORE, H // k * 4)                    # fp32 partial of this head
    n = len(typ)
    return W.from_edges(f"fused_attn_k{k}_{mode}", 1, np.array(typ, np.uint8), np.array(warp, np.uint16),
                        np.array(cta, np.uint32), np.array(work, np.uint32), np.zeros(n, np.uint32),
                        np.zeros(C, np.uint32), src, dst, kind)


def study_cases(sizes=CLUSTER_SIZES, modes=MODES):
    return [(k, m) for k in sizes for m in modes]


def study_set(sizes=CLUSTER_SIZES, modes=MODES, **kw):
    cases = study_cases(sizes, modes)
    return W.stack([fused_attention(k, m, **kw) for k, m in cases], "fused_attention"), cases


def study_params(cases, heads=32, points_per_graph=1, seed=W.SEED0 + 7):
    """H100-like rows with the Hopper-like NoC of ``workloads.with_noc`` (groups
    of 16 SMs, one 32 B/cycle port per SM, 180 cycles); CTA slots per SM so
    that every block of the kernel is resident.  Point 0 of each graph uses
    these defaults; further points draw NoC bandwidth (8-64 B/cycle), NoC
    latency (60-400 cycles) and DRAM bandwidth (1-8 TB/s), shared by every
    graph."""
    base = W.with_noc(W.default_params())
    block = np.tile(base, (points_per_graph, 1))
    if points_per_graph > 1:
        rng = np.random.default_rng(seed)
        m = points_per_graph - 1
        block[1:, W.P_NOC_BPC] = rng.integers(8, 65, m)
        block[1:, W.P_NOC_LAT] = rng.integers(60, 401, m)
        block[1:, W.P_HBM_BPC] = rng.integers(W.bytes_per_cycle(1.0), W.bytes_per_cycle(8.0) + 1, m)
    rows = []
    for i, (k, _m) in enumerate(cases):
        b = block.copy()
        b[:, W.P_CTAS_PER_SM] = -(-heads * k // int(base[W.P_NUM_SMS]))
        b[:, W.P_GRAPH_INDEX] = i
        rows.append(b)
    return np.ascontiguousarray(np.concatenate(rows), np.int32)
