"""libgts at the limits of its layout, against the oracle: nodes with more
successors than a warp has lanes (several release rounds, and the successor
count the slot cannot hold), wide joins, 128 logical warps per CTA, 32
servers of every class, many CTA slots per SM, and a row whose on-chip state
does not fit one warp's shared memory (GTS_ERR_UNSUPPORTED for that point
only)."""
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


def _check_all(graph, params, res):
    for q in range(res["status"].shape[0]):
        H.assert_point_equal(graph, params[q], res, q, oracle_run.simulate(graph, params[q]))


@pytest.mark.parametrize("fan", [30, 31, 32, 33, 64, 100, 300])
def test_fan_out_and_fan_in(fan):
    # node 0 releases `fan` nodes spread over warps and CTAs (DATA and ISSUE
    # edges), which all join into one sink
    rng = np.random.default_rng(fan)
    n = fan + 2
    C, Wn = 3, 4
    cta = [0] + sorted(int(x) for x in rng.integers(0, C, fan)) + [C - 1]
    warp = [0] + [int(x) for x in rng.integers(0, Wn, fan)] + [0]
    types = [W.LOAD] + [int(x) for x in rng.choice([W.MMA, W.EW, W.SMEM, W.NOP, W.BAR], fan)] + [W.STORE]
    edges = [(0, v, int(rng.integers(0, 2))) for v in range(1, fan + 1)] + [(v, n - 1, W.DATA)
                                                                           for v in range(1, fan + 1)]
    g = TG.make(n, edges, types, warp, cta, Wn, work=[int(x) for x in rng.integers(1, 9, n)])
    prms = np.stack([TG.small_params(rng, num_sms=s, cps=c) for s, c in ((1, 1), (3, 1), (2, 2), (1, 3))])
    _check_all(g, prms, H.run_gpu(g, prms))


def test_128_warps_per_cta_and_32_servers():
    rng = np.random.default_rng(7)
    g = TG.random_graph(rng, 400, W_=128, C=2, p_edge=0.01, max_work=12)
    p = TG.small_params(rng, num_sms=2, cps=1)
    for i in (W.P_CAP_TENSOR, W.P_CAP_TMA, W.P_CAP_LSU, W.P_CAP_ALU, W.P_CAP_BAR, W.P_CAP_HBM):
        p[i] = 32
    q = p.copy()
    q[W.P_CAP_HBM] = 1
    prms = np.stack([p, q, TG.small_params(rng, num_sms=1, cps=2)])
    _check_all(g, prms, H.run_gpu(g, prms))


def test_many_cta_slots_per_sm():
    rng = np.random.default_rng(8)
    g = TG.random_graph(rng, 300, W_=2, C=40, p_edge=0.02, intra_cta=True, kernels=True)
    prms = np.stack([TG.small_params(rng, num_sms=s, cps=c) for s, c in ((1, 16), (2, 20), (3, 7), (40, 1))])
    _check_all(g, prms, H.run_gpu(g, prms))


def test_row_too_large_for_one_warp_is_unsupported():
    # 6,000 SMs x 1 CTA slot with 6,000 one-node CTAs: about 44 bytes of
    # on-chip state per SM, more than one warp may keep in shared memory; the
    # other rows still run
    n = 6000
    g = W.from_edges("wide", 1, np.full(n, W.NOP, np.uint8), np.zeros(n, np.uint16), np.arange(n, dtype=np.uint32),
                     np.zeros(n, np.uint32), np.zeros(n, np.uint32), np.zeros(n, np.uint32), [], [], [])
    big = TG.unit_params(n, 1)
    small = TG.unit_params(8, 4)
    res = H.run_gpu(g, np.stack([small, big, small]))
    assert list(res["status"]) == [0, -9, 0]
    ref = oracle_run.simulate(g, small)
    H.assert_point_equal(g, small, res, 0, ref)
    assert oracle_run.simulate(g, big).status == 0   # the oracle has no such limit
