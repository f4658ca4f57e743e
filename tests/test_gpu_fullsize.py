"""Full-size workloads in the launch configuration the benchmark times, every
design point checked against the oracle.

Each workload runs on the GPU in one batch with the full trace, digests, CTA
placement and busy counters.  Every point's status, makespan, (start, finish)
digest and placement/busy digest must equal the oracle's, stored by
tests/golden/make_fullsize_golden.py (oracle only) under tests/golden/.  On top
of that, points at both ends and the middle of every swept parameter axis are
compared element by element (start, finish, CTA placement, busy cycles) with
the oracle run here, and every point is checked for properties that hold at
any size: makespan = max finish, start >= 0, finish >= start.
"""
import hashlib
import json
import os

import numpy as np
import pytest

from oracle import run as oracle_run
from paper_2607_11262_gb300 import workloads as W
from tests import gpu_helpers as H

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def gts_mod():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts
    gts.load()
    return gts


def axis_sample(params):
    """Points at the minimum, median and maximum of every column that varies
    over the table (the swept axes), first occurrence of each."""
    pts = set()
    for k in range(params.shape[1]):
        col = params[:, k]
        if np.all(col == col[0]):
            continue
        order = np.argsort(col, kind="stable")
        pts |= {int(order[0]), int(order[len(order) // 2]), int(order[-1])}
    return sorted(pts) if pts else [0]


def test_axis_sample_covers_both_ends_and_middle():
    p = W.workload("wsgemm8192").params
    s = axis_sample(p)
    for k in (W.P_NUM_SMS, W.P_HBM_BPC, W.P_TMA_LAT, W.P_MMA_FMA_PC):
        vals = p[s, k]
        assert vals.min() == p[:, k].min() and vals.max() == p[:, k].max()


@pytest.mark.parametrize("name", list(W.WORKLOADS))
def test_full_size_workload_every_point(gts_mod, name):
    import torch
    gts = gts_mod
    gold = json.load(open(os.path.join(GOLDEN, f"fullsize_{name}.json")))
    w = W.workload(name)
    # the stored values belong to these exact inputs
    assert gold["graph_sha256"] == w.graph.sha256(), "generator graph differs from the golden file's"
    assert gold["params_sha256"] == hashlib.sha256(np.ascontiguousarray(w.params, np.int32).tobytes()).hexdigest()
    P = w.params.shape[0]
    assert gold["points"] == P
    dg = gts.DeviceGraph(w.graph)
    dp = gts.DeviceParams(dg, w.params)
    flags = gts.GTS_FULL_TRACE | gts.GTS_WANT_DIGEST | gts.GTS_WANT_CTA_SM | gts.GTS_WANT_BUSY
    out = gts.simulate(dg, dp, flags=flags)
    torch.cuda.synchronize()
    status = out.status.cpu().numpy()
    makespan = out.makespan.cpu().numpy()
    digest = out.digest.cpu().numpy().astype(np.uint64)
    cta_sm = out.cta_sm.cpu().numpy()
    busy = out.busy.cpu().numpy()
    sizes = np.diff(w.graph.node_off.astype(np.int64))[w.params[:, W.P_GRAPH_INDEX]]
    csizes = np.diff(w.graph.cta_off.astype(np.int64))[w.params[:, W.P_GRAPH_INDEX]]
    # ---- every point against the stored oracle results
    bad = []
    for p in range(P):
        got = (int(status[p]), int(makespan[p]), f"{int(digest[p]):016x}",
               f"{H.aux_digest(cta_sm[p][:csizes[p]], busy[p]):016x}")
        want = (gold["status"][p], gold["makespan"][p], gold["digest"][p], gold["aux"][p])
        if got != want:
            bad.append((p, got, want))
    assert not bad, f"{len(bad)} of {P} points differ; first: {bad[0]}"
    assert np.all(status == 0)
    # ---- properties of every point, checked on the device
    sz = torch.from_numpy(sizes).cuda()
    colidx = torch.arange(dg.row_nodes, device="cuda")[None, :]
    valid = colidx < sz[:, None]
    fin = torch.where(valid, out.finish, torch.zeros_like(out.finish))
    assert torch.equal(fin.max(dim=1).values, out.makespan)
    assert bool(((out.start >= 0) | ~valid).all())
    assert bool(((out.finish >= out.start) | ~valid).all())
    # ---- ends and middle of every swept axis, element by element against the oracle
    pts = axis_sample(w.params)
    refs = oracle_run.simulate_points(w.graph, w.params, pts)
    sel = torch.tensor(pts, device="cuda")
    start = out.start.index_select(0, sel).cpu().numpy()
    finish = out.finish.index_select(0, sel).cpu().numpy()
    for j, p in enumerate(pts):
        one = {"status": status[[p]], "makespan": makespan[[p]], "start": start[[j]], "finish": finish[[j]],
               "cta_sm": cta_sm[[p]], "digest": digest[[p]], "busy": busy[[p]]}
        H.assert_point_equal(w.graph, w.params[p], one, 0, refs[p])
    del out
    dp.close()
    dg.close()
    torch.cuda.empty_cache()
