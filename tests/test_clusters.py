"""The cluster-fused attention decode of Section 7.2 (NoC vs DRAM exchanges),
on CPU: graph structure and closed forms of the bytes each variant moves,
the stepper against the oracle on a tiny instance, and the model check that
on-chip exchanges never lose to DRAM round trips at the default point."""
import numpy as np
import pytest

from oracle import run, stepper
from paper_2607_11262_gb300 import clusters as CL
from paper_2607_11262_gb300 import workloads as W

PAYLOADS = lambda k, d=128, e=2: [16, 3 * d // k * e, 16, 16, d * 4]  # noqa: E731  the five exchanges


@pytest.mark.parametrize("k", [2, 4, 8])
def test_structure_and_exchange_bytes(k):
    heads = 3
    noc = CL.fused_attention(k, "noc", heads=heads)
    dram = CL.fused_attention(k, "dram", heads=heads)
    C = heads * k
    for g in (noc, dram):
        assert g.n_ctas == C and g.warps_per_cta == 1
        src = np.repeat(np.arange(g.n_nodes), np.diff(g.row_ptr.astype(np.int64)))
        assert np.all(src < g.col)
        assert np.sum(g.type == W.BAR) == 5 * C            # one barrier per exchange per block
        # every barrier waits for exactly the k-1 peers of its cluster
        bars = np.nonzero(g.type == W.BAR)[0]
        indeg = np.bincount(g.col, minlength=g.n_nodes)
        assert np.all(indeg[bars] == k - 1)
        for b in bars:
            peers = src[g.col == b]
            assert np.all(g.cta[peers] // k == g.cta[b] // k) and np.all(g.cta[peers] != g.cta[b])
    per_block = sum(PAYLOADS(k))
    work = noc.work.astype(np.int64)
    assert work[noc.type == W.DSMEM].sum() == C * (k - 1) * per_block
    assert np.sum(dram.type == W.DSMEM) == 0
    dw = dram.work.astype(np.int64)
    # DRAM: each block stores each payload once and loads its k-1 peers' payloads back
    assert dw[dram.type == W.STORE].sum() == C * (per_block + 4096 // k * 4)
    assert dw[dram.type == W.LOAD].sum() - work[noc.type == W.LOAD].sum() == C * (k - 1) * per_block


def test_stepper_equals_oracle_tiny():
    g = CL.fused_attention(2, "noc", hidden=8, heads=2, head_dim=4, kv_len=4)
    h = CL.fused_attention(2, "dram", hidden=8, heads=2, head_dim=4, kv_len=4)
    prm = W.with_noc(W.default_params(), noc_bpc=2, noc_lat=3, cap_noc=1, cluster_sms=2)
    prm[W.P_NUM_SMS] = 4
    prm[W.P_DRAM_LAT], prm[W.P_MMA_LAT], prm[W.P_SMEM_LAT], prm[W.P_BAR_LAT] = 5, 2, 1, 1
    for graph in (g, h):
        r = run.simulate(graph, prm)
        st, mk, start, fin, cta_sm = stepper.simulate_graph(graph, prm)
        assert r.status == st == 0
        assert r.makespan == mk and list(r.start) == start and list(r.finish) == fin
        assert list(r.busy) == stepper.busy_cycles(graph.type, graph.work, graph.lat_extra, prm, start, mk)


def test_noc_never_loses_at_the_default_point():
    g, cases = CL.study_set()
    prm = CL.study_params(cases)
    mk = {c: run.simulate(g, prm[i]).makespan for i, c in enumerate(cases)}
    for k in CL.CLUSTER_SIZES:
        assert mk[(k, "noc")] < mk[(k, "dram")], k


def test_study_params_make_every_block_resident():
    cases = CL.study_cases()
    prm = CL.study_params(cases, points_per_graph=3)
    assert prm.shape == (len(cases) * 3, W.NPARAM)
    for i, (k, _m) in enumerate(cases):
        rows = prm[3 * i:3 * i + 3]
        assert np.all(rows[:, W.P_NUM_SMS] * rows[:, W.P_CTAS_PER_SM] >= 32 * k)
        assert np.all(rows[:, W.P_GRAPH_INDEX] == i)
        assert np.all(rows[:, W.P_CLUSTER_SMS] == 16)
