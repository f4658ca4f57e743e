"""Full-size workloads in the launch configuration the benchmark times.

Every design point of each workload is simulated on the GPU in one batch with
the full trace; a sample of points spread over the parameter ranges is checked
bit-exact against the oracle (computed in parallel host processes), and every
point is checked for properties that hold at any size: status OK, makespan =
max finish, every start >= 0 and finish >= start.
"""
import numpy as np
import pytest

from oracle import run as oracle_run
from paper_2607_11262_gb300 import workloads as W
from tests import gpu_helpers as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gts_mod():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts
    gts.load()
    return gts


def _sample(params, k):
    """k points spread over the SM-count range (smallest, largest, and between)."""
    order = np.argsort(params[:, W.P_NUM_SMS], kind="stable")
    idx = np.unique(np.linspace(0, len(order) - 1, k).round().astype(int))
    return sorted(int(order[i]) for i in idx)


@pytest.mark.parametrize("name,k", [("gemm512", 64), ("wsgemm8192", 6), ("fa_fwd", 4), ("decoder", 2),
                                    ("stress", 8)])
def test_full_size_workload(gts_mod, name, k):
    import torch
    gts = gts_mod
    w = W.workload(name)
    dg = gts.DeviceGraph(w.graph)
    dp = gts.DeviceParams(dg, w.params)
    flags = gts.GTS_FULL_TRACE | gts.GTS_WANT_DIGEST | gts.GTS_WANT_CTA_SM | gts.GTS_WANT_BUSY
    out = gts.simulate(dg, dp, flags=flags)
    torch.cuda.synchronize()
    status = out.status.cpu().numpy()
    assert np.all(status == 0), np.unique(status)
    # properties of every point, checked on the device
    sizes = torch.from_numpy(np.diff(w.graph.node_off.astype(np.int64))[w.params[:, W.P_GRAPH_INDEX]]).cuda()
    col = torch.arange(dg.row_nodes, device="cuda")[None, :]
    valid = col < sizes[:, None]
    fin = torch.where(valid, out.finish, torch.zeros_like(out.finish))
    assert torch.equal(fin.max(dim=1).values, out.makespan)
    assert bool(((out.start >= 0) | ~valid).all())
    assert bool(((out.finish >= out.start) | ~valid).all())
    # a sample of points bit-exact against the oracle
    pts = _sample(w.params, min(k, w.params.shape[0]))
    refs = oracle_run.simulate_points(w.graph, w.params, pts)
    res = {"status": status, "makespan": out.makespan.cpu().numpy()}
    sel = torch.tensor(pts, device="cuda")
    start = out.start.index_select(0, sel).cpu().numpy()
    finish = out.finish.index_select(0, sel).cpu().numpy()
    cta_sm = out.cta_sm.index_select(0, sel).cpu().numpy()
    digest = out.digest.cpu().numpy().astype(np.uint64)
    busy = out.busy.cpu().numpy()
    for j, p in enumerate(pts):
        one = {"status": res["status"][[p]], "makespan": res["makespan"][[p]], "start": start[[j]],
               "finish": finish[[j]], "cta_sm": cta_sm[[j]], "digest": digest[[p]], "busy": busy[[p]]}
        H.assert_point_equal(w.graph, w.params[p], one, 0, refs[p])
    del out
    dp.close()
    dg.close()
    torch.cuda.empty_cache()
