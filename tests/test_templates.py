"""Template-shared graphs (Section 6.4 "Graph construction") on CPU: the
expansion of a TemplateSet is exactly the logical graph the generator builds
(every array equal), for the named workloads, stacked sets and empty
templates; a TemplateSet stores far fewer nodes than it represents."""
import numpy as np
import pytest

from paper_2607_11262_gb300 import workloads as W


def _same(a, b):
    for k, v in a.arrays().items():
        assert np.array_equal(v, getattr(b, k)), k
        assert v.dtype == getattr(b, k).dtype, k
    assert a.warps_per_cta == b.warps_per_cta


@pytest.mark.parametrize("name", W.TEMPLATED)
def test_expansion_is_the_logical_graph(name):
    ts = W.workload(name, templated=True).graph
    g = W.workload(name).graph
    assert (ts.n_nodes, ts.n_edges, ts.n_ctas) == (g.n_nodes, g.n_edges, g.n_ctas)
    assert int(ts.tpl_node_off[-1]) * 16 <= g.n_nodes      # at least 16x fewer stored nodes
    _same(ts.expand(), g)


def test_stacked_set_and_empty_templates():
    a = W.gemm_2stage_cta(ksteps=3, warps=2)
    b = W.ws_gemm_cta(2, 3)
    empty = W.CtaTemplate(3)
    tpls = [a, b, empty]
    ct = np.array([0, 2, 1, 1, 0, 2, 1])
    ck = np.array([0, 0, 1, 1, 0, 1, 1], np.uint32)
    ts = W.template_set("mix", 3, tpls, ct, ck, graph_cta_off=[0, 4, 7])
    # reference: two graphs assembled separately and stacked
    g1 = W.assemble("g1", 3, tpls, ct[:4], ck[:4])
    g2 = W.assemble("g2", 3, tpls, ct[4:], ck[4:])
    ref = W.stack([g1, g2], "mix")
    _same(ts.expand(), ref)
    assert ts.n_graphs == 2 and ts.n_ctas == 7


def test_template_csr_is_sorted_and_local():
    ts = W.workload("wsgemm_small", templated=True).graph
    off = ts.tpl_node_off.astype(np.int64)
    for t in range(ts.n_templates):
        for u in range(off[t], off[t + 1]):
            succ = ts.col[ts.row_ptr[u]:ts.row_ptr[u + 1]].astype(np.int64)
            assert np.all(np.diff(succ) >= 0)
            assert np.all((succ > u) & (succ < off[t + 1]))


def _random_template(rng, warps):
    t = W.CtaTemplate(warps)
    n = int(rng.integers(0, 12))
    for _ in range(n):
        t.node(int(rng.integers(0, 7)), int(rng.integers(0, warps)), int(rng.integers(0, 5000)), int(rng.integers(0, 9)))
    for v in range(1, n):
        for u in rng.choice(v, size=min(v, int(rng.integers(0, 3))), replace=False):
            t.edge(int(u), v, int(rng.integers(0, 2)))
    return t


def _by_hand(name, warps, tpls, ct, ck):
    """The logical graph written out CTA by CTA: CTA c's copy of its template
    takes the next block of ids, edges shifted by that block's base."""
    typ, wp, wk, lx, cta, src, dst, kind = [], [], [], [], [], [], [], []
    for c, t in enumerate(ct):
        tp = tpls[t]
        base = len(typ)
        for u in range(len(tp)):
            typ.append(tp.t[u]); wp.append(tp.w[u]); wk.append(tp.wk[u]); lx.append(tp.lx[u]); cta.append(c)
        for u, v, k in zip(tp.es, tp.ed, tp.ek):
            src.append(base + u); dst.append(base + v); kind.append(k)
    return W.from_edges(name, warps, typ, wp, cta, wk, lx, ck, src, dst, kind)


def test_random_template_sets_expand_to_the_hand_built_graph():
    rng = np.random.default_rng(77)
    for trial in range(60):
        warps = int(rng.integers(1, 5))
        tpls = [_random_template(rng, warps) for _ in range(int(rng.integers(1, 5)))]
        C = int(rng.integers(1, 12))
        ct = rng.integers(0, len(tpls), C)
        ck = np.sort(rng.integers(0, 3, C)).astype(np.uint32)
        ts = W.template_set(f"r{trial}", warps, tpls, ct, ck)
        ref = _by_hand(f"r{trial}", warps, tpls, ct, ck)
        _same(ts.expand(), ref)
        _same(W.assemble(f"r{trial}", warps, tpls, ct, ck), ref)
