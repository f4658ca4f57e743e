"""Small seeded graphs for the oracle pins and the GPU parity edge cases (test helper)."""
from __future__ import annotations

import itertools

import numpy as np

from paper_2607_11262_gb300 import workloads as W


def unit_params(num_sms=1, cps=1, caps=1, cap_hbm=1):
    """Every rate 1 and every base latency 0: a LOAD/SMEM/MMA/EW/STORE node then
    occupies its unit(s) for ``work`` cycles and, with lat_extra 0, has latency
    ``work`` too."""
    p = W.default_params()
    p[W.P_NUM_SMS] = num_sms
    p[W.P_CTAS_PER_SM] = cps
    for i in (W.P_HBM_BPC, W.P_TMA_BPC, W.P_SMEM_BPC, W.P_MMA_FMA_PC, W.P_ALU_OPS_PC):
        p[i] = 1
    for i in (W.P_DRAM_LAT, W.P_TMA_LAT, W.P_SMEM_LAT, W.P_MMA_LAT, W.P_ALU_LAT, W.P_BAR_LAT):
        p[i] = 0
    for i in (W.P_CAP_TENSOR, W.P_CAP_TMA, W.P_CAP_LSU, W.P_CAP_ALU, W.P_CAP_BAR):
        p[i] = caps
    p[W.P_CAP_HBM] = cap_hbm
    return p


def small_params(rng, num_sms=None, cps=None):
    """Random small-latency parameter row (keeps cycle counts tiny)."""
    p = W.default_params()
    p[W.P_NUM_SMS] = num_sms if num_sms is not None else rng.integers(1, 4)
    p[W.P_CTAS_PER_SM] = cps if cps is not None else rng.integers(1, 3)
    for i in (W.P_HBM_BPC, W.P_TMA_BPC, W.P_SMEM_BPC, W.P_MMA_FMA_PC, W.P_ALU_OPS_PC):
        p[i] = rng.integers(1, 5)
    for i in (W.P_DRAM_LAT, W.P_TMA_LAT, W.P_SMEM_LAT, W.P_MMA_LAT, W.P_ALU_LAT, W.P_BAR_LAT):
        p[i] = rng.integers(0, 4)
    for i in (W.P_CAP_TENSOR, W.P_CAP_TMA, W.P_CAP_LSU, W.P_CAP_ALU, W.P_CAP_BAR, W.P_CAP_HBM):
        p[i] = rng.integers(1, 3)
    return p


def make(n, edges, types, warps, ctas, W_, kernels=None, work=None, lat_extra=None, name="tiny"):
    """Graph from explicit lists; ``edges`` = [(u, v, kind)]."""
    C = (max(ctas) + 1) if len(ctas) else 1
    if kernels is None:
        kernels = [0] * C
    if work is None:
        work = [1] * n
    if lat_extra is None:
        lat_extra = [0] * n
    src = [e[0] for e in edges]
    dst = [e[1] for e in edges]
    kind = [e[2] for e in edges]
    return W.from_edges(name, W_, types, warps, ctas, work, lat_extra, kernels, src, dst, kind)


def random_graph(rng, n, W_=None, C=None, p_edge=0.25, p_issue=0.3, max_work=6, cta_major=True,
                 kernels=False, types=(0, 1, 2, 3, 4, 5, 6), intra_cta=False):
    """Random DAG over ids 0..n-1 (edges only go forward; with ``intra_cta``
    only between nodes of the same CTA)."""
    W_ = W_ if W_ is not None else int(rng.integers(1, 4))
    C = C if C is not None else int(rng.integers(1, 4))
    if cta_major:
        ctas = sorted(int(x) for x in rng.integers(0, C, n))
    else:
        ctas = [int(x) for x in rng.integers(0, C, n)]
    edges = []
    for v in range(n):
        for u in range(v):
            if intra_cta and ctas[u] != ctas[v]:
                continue
            if rng.random() < p_edge:
                edges.append((u, v, int(rng.random() < p_issue)))
    C_eff = max(ctas) + 1 if n else C
    C_eff = max(C_eff, C)
    warps = [int(x) for x in rng.integers(0, W_, n)]
    tys = [int(x) for x in rng.choice(np.array(types), n)]
    work = [int(x) for x in rng.integers(0, max_work + 1, n)]
    lx = [int(x) for x in rng.integers(0, 3, n)]
    if kernels:
        kern = sorted(int(x) for x in rng.integers(0, 3, C_eff))
    else:
        kern = [0] * C_eff
    return W.from_edges("rand", W_, tys, warps, ctas, work, lx, kern,
                        [e[0] for e in edges], [e[1] for e in edges], [e[2] for e in edges])


def all_edge_sets(n):
    """Every DAG on n ordered nodes with each forward pair absent, DATA or ISSUE."""
    pairs = [(u, v) for v in range(n) for u in range(v)]
    for choice in itertools.product((None, 0, 1), repeat=len(pairs)):
        yield [(u, v, k) for (u, v), k in zip(pairs, choice) if k is not None]
