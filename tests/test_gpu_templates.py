"""Template-shared graphs on the GPU: gts_graph_create_templated expands the
templates into exactly the packed workspace gts_graph_create builds from the
logical graph (byte for byte), so simulations agree bit-exactly; malformed
template sets are refused."""
import numpy as np
import pytest

from paper_2607_11262_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gts_mod():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts
    gts.load()
    return gts


@pytest.mark.parametrize("name,points", [("gemm512", 64), ("wsgemm_small", 256), ("fa_fwd", 16),
                                         ("wsgemm8192", 8), ("decoder", 4)])
def test_templated_equals_explicit(gts_mod, name, points):
    import torch
    gts = gts_mod
    ex = W.workload(name, points=points)
    ts = W.workload(name, points=points, templated=True)
    dge = gts.DeviceGraph(ex.graph)
    dgt = gts.DeviceGraph(ts.graph)
    k = dge.workspace.numel()
    assert dgt.workspace.numel() > k
    assert torch.equal(dge.workspace, dgt.workspace[:k])           # same packed graph, byte for byte
    assert (dge.row_nodes, dge.row_ctas) == (dgt.row_nodes, dgt.row_ctas)
    flags = gts.GTS_FULL_TRACE | gts.GTS_WANT_DIGEST | gts.GTS_WANT_CTA_SM | gts.GTS_WANT_BUSY
    outs = []
    for dg in (dge, dgt):
        dp = gts.DeviceParams(dg, ex.params)
        out = gts.simulate(dg, dp, flags=flags)
        torch.cuda.synchronize()
        outs.append(out)
    a, b = outs
    assert np.all(a.status.cpu().numpy() == 0)
    for f in ("status", "makespan", "start", "finish", "digest", "cta_sm", "busy"):
        assert torch.equal(getattr(a, f), getattr(b, f)), f


def _broken(ts, **changes):
    import dataclasses
    return dataclasses.replace(ts, **{k: np.asarray(v, getattr(ts, k).dtype) for k, v in changes.items()})


def test_malformed_template_sets_are_refused(gts_mod):
    gts = gts_mod
    ts = W.workload("gemm512", templated=True).graph
    bad_col = ts.col.copy()
    bad_col[0] = 0                                           # edge backwards
    bad_type = ts.type.copy()
    bad_type[3] = 9
    bad_warp = ts.warp.copy()
    bad_warp[5] = 4
    bad_ct = ts.cta_template.copy()
    bad_ct[2] = 1                                            # no template 1
    bad_kernel = ts.cta_kernel.copy()
    bad_kernel[:8] = 1                                       # kernel id decreases
    for case in (dict(col=bad_col), dict(type=bad_type), dict(warp=bad_warp), dict(cta_template=bad_ct),
                 dict(cta_kernel=bad_kernel)):
        with pytest.raises(gts.GtsError) as e:
            gts.DeviceGraph(_broken(ts, **case))
        assert e.value.status == gts.GTS_ERR_INVALID_GRAPH, case.keys()


def _random_template(rng, warps, n, fan=False):
    t = W.CtaTemplate(warps)
    for v in range(n):
        t.node(int(rng.integers(0, 7)), int(rng.integers(0, warps)), work=int(rng.integers(0, 9)),
               lat_extra=int(rng.integers(0, 3)))
    for v in range(1, n):
        for u in rng.choice(v, size=min(v, int(rng.integers(0, 3))), replace=False):
            t.edge(int(u), v, int(rng.integers(0, 2)))
    if fan and n > 40:  # node 0 feeds every later node: more than 32 successors
        have = set(zip(t.es, t.ed))
        for v in range(1, n):
            if (0, v) not in have:
                t.edge(0, v, W.DATA)
    return t


def test_random_template_sets(gts_mod):
    """Random template sets (several templates, one unused, a node with more than
    32 successors, stacked graphs, kernel gates), expanded on the device and
    simulated: bit-exact against the oracle on the expanded logical graph."""
    import torch

    from oracle import run as oracle_run
    from tests import gpu_helpers as H
    from tests import tinygraphs as TG
    gts = gts_mod
    rng = np.random.default_rng(31)
    for case in range(6):
        warps = int(rng.integers(1, 5))
        tpls = [_random_template(rng, warps, int(rng.integers(1, 60)), fan=(k == 0)) for k in range(4)]
        C = int(rng.integers(2, 14))
        ct = rng.integers(0, 3, C)          # template 3 is never used
        kern = np.sort(rng.integers(0, 3, C)) if case % 2 else np.zeros(C, np.int64)
        goff = None
        if case >= 3:                       # two stacked graphs
            cut = int(rng.integers(1, C))
            goff = [0, cut, C]
            kern = np.concatenate([np.sort(kern[:cut]), np.sort(kern[cut:])])
        ts = W.template_set(f"rand{case}", warps, tpls, ct, kern, goff)
        g = ts.expand()
        prms = np.stack([TG.small_params(rng) for _ in range(8)])
        if goff is not None:
            prms[:, W.P_GRAPH_INDEX] = np.arange(8) % 2
        res = H.run_gpu(ts, prms)
        torch.cuda.synchronize()
        for q in range(prms.shape[0]):
            H.assert_point_equal(g, prms[q], res, q, oracle_run.simulate(g, prms[q]))
