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
