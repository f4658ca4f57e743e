"""The lean kernel instance with split SM records, which the library launches
when every row's SMs hold fewer than 8 warp slots, against the oracle and
against the whole-record instance.

An SM with exactly one issuable HBM head keeps that head apart in its record
and takes its effective cycle max(key, H) when the record is read; an SM with
several HBM heads keeps the whole record and is rescanned when the HBM
horizon passes its least HBM key.  These graphs are LOAD/STORE heavy with
several warps per CTA, so both forms occur and the horizon moves often."""
import numpy as np
import pytest

from oracle import run as oracle_run
from paper_2607_11262_gb300 import workloads as W
from tests import gpu_helpers as H
from tests import tinygraphs as TG

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_11262_gb300 import gts
    gts.load()


HBM_HEAVY = (W.LOAD, W.LOAD, W.STORE, W.MMA, W.EW, W.BAR)


def _rows(rng, k, cps):
    rows = []
    for _ in range(k):
        p = TG.small_params(rng, num_sms=int(rng.integers(1, 5)), cps=cps)
        p[W.P_CAP_HBM] = int(rng.integers(1, 4))
        p[W.P_HBM_BPC] = int(rng.integers(1, 3))   # slow HBM: heads wait on the horizon
        rows.append(p)
    return np.stack(rows)


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_split_instance_against_the_oracle(seed):
    """Rows of 3 warps x 2 CTA slots (6 slots per SM): the split instance."""
    rng = np.random.default_rng(9100 + seed)
    g = TG.random_graph(rng, 120, W_=3, C=6, p_edge=0.06, types=HBM_HEAVY)
    prms = _rows(rng, 12, 2)
    res = H.run_gpu(g, prms)
    for q in range(prms.shape[0]):
        H.assert_point_equal(g, prms[q], res, q, oracle_run.simulate(g, prms[q]))


def test_split_and_whole_instances_agree():
    """The same rows in a batch that also holds a row of 8 slots per SM (which
    makes the library launch the whole-record instance) give identical
    results to the batch of those rows alone (split instance)."""
    rng = np.random.default_rng(9200)
    g = TG.random_graph(rng, 150, W_=4, C=6, p_edge=0.05, types=HBM_HEAVY)
    small = _rows(rng, 10, 1)                 # 4 slots per SM
    wide = TG.small_params(rng, num_sms=2, cps=2)   # 8 slots per SM
    mixed = np.concatenate([small, wide[None, :]])
    a = H.run_gpu(g, small)
    b = H.run_gpu(g, mixed)
    n = small.shape[0]
    for k in ("status", "makespan", "digest"):
        assert np.array_equal(a[k], b[k][:n]), k
    ok = a["status"] == 0   # a failed point's trace rows are unspecified
    assert ok.any()
    for k in ("start", "finish", "cta_sm", "busy"):
        assert np.array_equal(a[k][ok], b[k][:n][ok]), k
    H.assert_point_equal(g, wide, b, small.shape[0], oracle_run.simulate(g, wide))


def test_wsgemm_shape_rows_run_split():
    """The ws GEMM profiling case (3 warps per CTA, 1 CTA per SM) on a few
    points, spread over the SM-count axis, against the oracle."""
    w = W.workload("wsgemm_small")
    order = np.argsort(w.params[:, W.P_NUM_SMS], kind="stable")
    pts = w.params[order[[0, len(order) // 2, len(order) - 1]]]
    res = H.run_gpu(w.graph, pts)
    for q in range(pts.shape[0]):
        H.assert_point_equal(w.graph, pts[q], res, q, oracle_run.simulate(w.graph, pts[q]))
