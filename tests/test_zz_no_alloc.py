"""gts_simulate_batch_noalloc -- the entry point for callers that cannot
allocate device memory when they call it (a plug-in inside a host application
that owns every device allocation, or a service whose device memory is fixed
at start-up so its allocator must not grow) -- gives the same results as
gts_simulate_batch with caller scratch, call after call, and allocates
nothing.

This file is collected last on purpose: it shares the library's static scratch
with nothing else and must pass alone in a fresh process or after the rest.
"""
import numpy as np
import pytest

from paper_2607_11262_gb300 import workloads as W
from tests import tinygraphs as TG

pytestmark = pytest.mark.gpu

FLAGS = 1 | 2 | 4 | 8  # full trace, digest, CTA placement, busy cycles


@pytest.fixture(scope="module")
def gts_mod():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts
    gts.load()
    return gts


def _noalloc(gts, dg, dp, out, first=0, n=None):
    import torch
    n = dp.n_points - first if n is None else n
    p = lambda t: 0 if t is None else t.data_ptr()  # noqa: E731
    gts.gts_simulate_batch_noalloc(dg.handle, dp.handle, first, n, FLAGS, p(out.start), p(out.finish),
                                   p(out.makespan), p(out.status), p(out.digest), p(out.cta_sm), p(out.busy),
                                   torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return {k: getattr(out, k).cpu().numpy().copy() for k in ("makespan", "status", "start", "finish", "digest",
                                                               "cta_sm", "busy")}


def _reference(gts, dg, dp):
    import torch
    out = gts.simulate(dg, dp, flags=FLAGS)
    torch.cuda.synchronize()
    return {k: getattr(out, k).cpu().numpy().copy() for k in ("makespan", "status", "start", "finish", "digest",
                                                               "cta_sm", "busy")}


def _same(a, b):
    for k in a:
        assert np.array_equal(a[k], b[k]), k   # integer cycles: bit-exact


@pytest.mark.parametrize("case", ["gemm512", "ws_small", "stacked_dags"])
def test_noalloc_matches_caller_scratch_twice(gts_mod, case):
    gts = gts_mod
    if case == "gemm512":
        w = W.workload("gemm512")
        graph, params = w.graph, w.params
    elif case == "ws_small":
        w = W.workload("wsgemm_small", points=300)
        graph, params = w.graph, w.params
    else:
        graph = W.stress_set(4, n_nodes=2500)
        params = W.stress_params(4)
    dg = gts.DeviceGraph(graph)
    dp = gts.DeviceParams(dg, params)
    ref = _reference(gts, dg, dp)
    assert np.all(ref["status"] == 0)
    out = gts.alloc_outputs(dg, dp.n_points, FLAGS)
    first = _noalloc(gts, dg, dp, out)
    _same(first, ref)
    out.makespan.fill_(-7)
    out.start.fill_(-7)
    second = _noalloc(gts, dg, dp, out)  # the static array keeps the first call's contents
    _same(second, ref)


def test_noalloc_partial_range_and_too_large(gts_mod):
    gts = gts_mod
    w = W.workload("gemm512")
    dg = gts.DeviceGraph(w.graph)
    dp = gts.DeviceParams(dg, w.params)
    ref = _reference(gts, dg, dp)
    out = gts.alloc_outputs(dg, 20, FLAGS)
    part = _noalloc(gts, dg, dp, out, first=10, n=20)
    for k in part:
        assert np.array_equal(part[k], ref[k][10:30]), k


def _nop_graph(n):
    return W.from_edges("nops", 1, np.full(n, W.NOP, np.uint8), np.zeros(n, np.uint16), np.zeros(n, np.uint32),
                        np.zeros(n, np.uint32), np.zeros(n, np.uint32), np.zeros(1, np.uint32), [], [], [])


def test_noalloc_size_limit_exact(gts_mod):
    """The header (16 B) and one row (8 B per node, rounded to an even count)
    must fit in GTS_STATIC_SCRATCH_BYTES: 4,194,302 nodes do, 4,194,303 not."""
    gts = gts_mod
    limit = (gts.GTS_STATIC_SCRATCH_BYTES - gts.GTS_SCRATCH_HEADER_BYTES) // 8
    assert limit == 4_194_302
    for n, ok in ((limit, True), (limit + 1, False)):
        dg = gts.DeviceGraph(_nop_graph(n))
        dp = gts.DeviceParams(dg, TG.unit_params()[None, :])
        out = gts.alloc_outputs(dg, 1, 0)
        call = lambda: gts.gts_simulate_batch_noalloc(dg.handle, dp.handle, 0, 0, 0, 0, 0,  # noqa: E731
                                                      out.makespan.data_ptr(), out.status.data_ptr(), 0, 0, 0, 0)
        if ok:
            call()  # size accepted (no point requested, so nothing runs)
        else:
            with pytest.raises(gts.GtsError) as e:
                call()
            assert e.value.status == gts.GTS_ERR_NOMEM
            assert "static scratch" in gts.gts_last_error()
        dp.close()
        dg.close()


def test_noalloc_allocates_no_device_memory(gts_mod):
    """After a first call (which loads the module and looks up the array), a
    call leaves the device's free memory unchanged."""
    import torch
    gts = gts_mod
    w = W.workload("gemm512")
    dg = gts.DeviceGraph(w.graph)
    dp = gts.DeviceParams(dg, w.params)
    out = gts.alloc_outputs(dg, dp.n_points, FLAGS)
    first = _noalloc(gts, dg, dp, out)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    again = _noalloc(gts, dg, dp, out)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    _same(again, first)
