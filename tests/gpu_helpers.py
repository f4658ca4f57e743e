"""Shared helpers of the GPU tests: run libgts, compare with the oracle."""
from __future__ import annotations

import numpy as np

MASK64 = (1 << 64) - 1


def digest(start, finish):
    """The ABI's per-point digest computed on the host from oracle rows:
    sum over v of splitmix64-finalise((v << 32 | start) ^ (finish * golden)) mod 2^64."""
    v = np.arange(len(start), dtype=np.uint64)
    s = np.asarray(start, np.int64).astype(np.uint32).astype(np.uint64)
    f = np.asarray(finish, np.int64).astype(np.uint32).astype(np.uint64)
    with np.errstate(over="ignore"):
        z = ((v << np.uint64(32)) | s) ^ (f * np.uint64(0x9E3779B97F4A7C15))
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        z = z ^ (z >> np.uint64(31))
        return int(np.sum(z, dtype=np.uint64))


def _mix(z):
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def aux_digest(cta_sm, busy):
    """A host-side digest of one point's CTA placement and busy counters:
    sum over c of mix(c << 32 | cta_sm[c]) plus sum over k of mix((k + 1) << 56 ^ busy[k]),
    mod 2^64 (mix = the splitmix64 finaliser).  Used only to compare the GPU's
    outputs with stored oracle results."""
    c = np.arange(len(cta_sm), dtype=np.uint64)
    s = np.asarray(cta_sm, np.int64).astype(np.uint32).astype(np.uint64)
    k = np.arange(len(busy), dtype=np.uint64) + np.uint64(1)
    b = np.asarray(busy, np.int64).astype(np.uint64)
    with np.errstate(over="ignore"):
        t1 = np.sum(_mix((c << np.uint64(32)) | s), dtype=np.uint64)
        t2 = np.sum(_mix((k << np.uint64(56)) ^ b), dtype=np.uint64)
        return int((int(t1) + int(t2)) & MASK64)


def run_gpu(graph, params, flags=None, first_point=0, n_points=None):
    import torch

    from paper_2607_11262_gb300 import gts
    if flags is None:
        flags = gts.GTS_FULL_TRACE | gts.GTS_WANT_DIGEST | gts.GTS_WANT_CTA_SM | gts.GTS_WANT_BUSY
    dg = gts.DeviceGraph(graph)
    dp = gts.DeviceParams(dg, params)
    out = gts.simulate(dg, dp, first_point=first_point, n_points=n_points, flags=flags)
    torch.cuda.synchronize()
    res = {"status": out.status.cpu().numpy(), "makespan": out.makespan.cpu().numpy()}
    if out.start is not None:
        res["start"] = out.start.cpu().numpy()
        res["finish"] = out.finish.cpu().numpy()
    if out.digest is not None:
        res["digest"] = out.digest.cpu().numpy().astype(np.uint64)
    if out.cta_sm is not None:
        res["cta_sm"] = out.cta_sm.cpu().numpy()
    if out.busy is not None:
        res["busy"] = out.busy.cpu().numpy()
    del out
    dp.close()
    dg.close()
    return res


def graph_sizes(graph, g):
    n = int(graph.node_off[g + 1] - graph.node_off[g])
    c = int(graph.cta_off[g + 1] - graph.cta_off[g])
    return n, c


def assert_point_equal(graph, params, res, q, ref, check_trace=True):
    """Bit-exact comparison of GPU point q (param row = q + first) with oracle result ``ref``."""
    assert int(res["status"][q]) == ref.status, (q, int(res["status"][q]), ref.status)
    if ref.status != 0:
        return
    assert int(res["makespan"][q]) == ref.makespan, (q, int(res["makespan"][q]), ref.makespan)
    gi = int(params[19]) if graph.n_graphs > 1 else 0
    n, c = graph_sizes(graph, gi)
    if check_trace and "start" in res:
        s = res["start"][q][:n]
        f = res["finish"][q][:n]
        if not (np.array_equal(s, ref.start) and np.array_equal(f, ref.finish)):
            bad = np.nonzero((s != ref.start) | (f != ref.finish))[0]
            v = int(bad[0])
            raise AssertionError(f"point {q}: {len(bad)} nodes differ; first node {v}: gpu ({s[v]}, {f[v]}) "
                                 f"oracle ({ref.start[v]}, {ref.finish[v]})")
    if "cta_sm" in res:
        assert np.array_equal(res["cta_sm"][q][:c], ref.cta_sm), q
    if "digest" in res:
        assert int(res["digest"][q]) == digest(ref.start, ref.finish), q
    if "busy" in res:
        assert list(res["busy"][q]) == list(ref.busy), (q, list(res["busy"][q]), list(ref.busy))
