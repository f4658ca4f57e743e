"""Longest-processing-time-first point order (gts_params_set_order): the
order in which warps take design points changes no result -- whole batches,
sub-ranges (the order is skipped outside them), a scratch that holds fewer
rows than there are points, and mixed lean / extended rows."""
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


def _run(gts, dg, params, ordered, first=0, n=None, scratch=None):
    import torch
    dp = gts.DeviceParams(dg, params, ordered=ordered)
    flags = gts.GTS_FULL_TRACE | gts.GTS_WANT_DIGEST | gts.GTS_WANT_CTA_SM | gts.GTS_WANT_BUSY
    out = gts.simulate(dg, dp, first_point=first, n_points=n, flags=flags, scratch=scratch)
    torch.cuda.synchronize()
    res = {f: getattr(out, f).cpu().numpy() for f in ("status", "makespan", "start", "finish", "digest", "cta_sm",
                                                       "busy")}
    order = None if dp.order is None else dp.order.cpu().numpy()
    dp.close()
    return res, order


def _same(a, b):
    """Equal results; start/finish/CTA placement only for OK points (unspecified otherwise)."""
    assert np.array_equal(a["status"], b["status"])
    ok = a["status"] == 0
    for k in a:
        assert np.array_equal(a[k][ok], b[k][ok]), k


def test_order_is_by_estimated_cost(gts_mod):
    gts = gts_mod
    w = W.workload("wsgemm_small", points=300)
    dg = gts.DeviceGraph(w.graph)
    _res, order = _run(gts, dg, w.params, True)
    assert sorted(order.tolist()) == list(range(300))
    sms = w.params[order, W.P_NUM_SMS]
    assert np.all(np.diff(sms) <= 0)      # one graph: cost falls with the simulated SM count


@pytest.mark.parametrize("first,n", [(0, None), (37, 101), (299, 1)])
def test_ordered_equals_unordered(gts_mod, first, n):
    gts = gts_mod
    w = W.workload("wsgemm_small", points=300)
    dg = gts.DeviceGraph(w.graph)
    a, _ = _run(gts, dg, w.params, False, first, n)
    b, _ = _run(gts, dg, w.params, True, first, n)
    _same(a, b)


def test_ordered_with_few_rows_and_mixed_instances(gts_mod):
    import torch
    gts = gts_mod
    w = W.workload("gemm512")
    p = w.params.copy()
    p[::3, W.P_ISSUE_POLICY], p[::3, W.P_SUBPARTITIONS] = W.POLICY_GTO, 4   # extended instance for the batch
    p[5, W.P_TMA_BPC] = 0                                                    # one invalid row
    dg = gts.DeviceGraph(w.graph)
    row = ((dg.row_nodes + 1) // 2 * 2) * 8
    few = torch.empty(gts.GTS_SCRATCH_HEADER_BYTES + 5 * row, dtype=torch.uint8, device="cuda")
    a, _ = _run(gts, dg, p, False)
    b, _ = _run(gts, dg, p, True, scratch=few)
    _same(a, b)
    assert a["status"][5] == gts.GTS_ERR_INVALID_PARAMS
