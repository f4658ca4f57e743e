"""Pins of the CPU oracle against things other than itself (no GPU needed).

* hand-worked schedules and per-type latencies (tests/golden/);
* brute force: an independent cycle-by-cycle stepper on every tiny DAG;
* closed forms: a DATA chain sums its latencies; unlimited resources give the
  DAG longest path (networkx Bellman-Ford on negated weights); one server with
  occupancy = latency leaves no idle cycle;
* bounds and invariants: critical path and per-resource work lower-bound the
  makespan; finish = start + latency; no unit over capacity at any cycle; warp
  starts are non-decreasing; Graham's (2 - 1/m) bound against a brute-force
  optimum of P|prec|Cmax;
* per-subpartition issue policies (greedy-then-oldest, round-robin): hand
  schedules, stepper == oracle, one issue per scheduler per cycle;
* DSMEM nodes over the on-chip NoC of SM groups: hand schedules, stepper ==
  oracle, parameter checks;
* busy server-cycles: equal to the stepper's cycle-by-cycle count of held
  servers; a single saturated server is busy for the whole makespan; busy
  cycles never exceed servers x makespan;
* error statuses.
"""
import json
import os

import networkx as nx
import numpy as np
import pytest

from oracle import run, stepper
from paper_2607_11262_gb300 import workloads as W
from tests import tinygraphs as TG

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
TYPE = {n: i for i, n in enumerate(W.TYPE_NAMES)}
KIND = {"DATA": W.DATA, "ISSUE": W.ISSUE}


def both(g, prm):
    """Oracle result and the stepper's (status, makespan, start, finish, cta_sm,
    busy cycles counted cycle by cycle)."""
    r = run.simulate(g, prm)
    s = stepper.simulate_graph(g, prm)
    busy = stepper.busy_cycles(g.type, g.work, g.lat_extra, prm, s[2], s[1]) if s[0] == 0 else None
    return r, s + (busy,)


def assert_same(r, s):
    st, mk, start, fin, cta_sm, busy = s
    assert r.status == st
    if st == 0:
        assert r.makespan == mk
        assert list(r.start) == start
        assert list(r.finish) == fin
        assert list(r.cta_sm) == cta_sm
        assert list(r.busy) == busy


# ------------------------------------------------------------------ golden
def test_golden_single_node_latency():
    spec = json.load(open(os.path.join(GOLDEN, "single_node_latency.json")))
    for case in spec["cases"]:
        g = TG.make(1, [], [TYPE[case["type"]]], [0], [0], 1, work=[case["work"]],
                    lat_extra=[case["lat_extra"]])
        r = run.simulate(g, W.default_params())
        assert r.status == 0
        assert r.makespan == case["makespan"], case
        assert (r.start[0], r.finish[0]) == (0, case["makespan"])


def test_golden_hand_schedules():
    spec = json.load(open(os.path.join(GOLDEN, "hand_schedules.json")))
    for case in spec["cases"]:
        nodes = case["nodes"]
        g = TG.make(len(nodes), [(u, v, KIND[k]) for u, v, k in case["edges"]],
                    [TYPE[x[0]] for x in nodes], [x[1] for x in nodes], [x[2] for x in nodes],
                    case["warps_per_cta"], kernels=case["kernels"], work=[x[3] for x in nodes])
        prm = TG.unit_params(case["num_sms"], case["ctas_per_sm"], case["caps"], case["cap_hbm"])
        r, s = both(g, prm)
        assert r.status == 0, case["name"]
        assert list(r.start) == case["start"], case["name"]
        assert list(r.finish) == case["finish"], case["name"]
        assert r.makespan == case["makespan"], case["name"]
        assert list(r.cta_sm) == case["cta_sm"], case["name"]
        assert_same(r, s)


def test_golden_issue_policies():
    spec = json.load(open(os.path.join(GOLDEN, "issue_policies.json")))
    for case in spec["cases"]:
        nodes = case["nodes"]
        g = TG.make(len(nodes), [(u, v, KIND[k]) for u, v, k in case["edges"]],
                    [TYPE[x[0]] for x in nodes], [x[1] for x in nodes], [x[2] for x in nodes],
                    case["warps_per_cta"], work=[x[3] for x in nodes])
        prm = TG.unit_params(case["num_sms"], case["ctas_per_sm"])
        prm[W.P_ISSUE_POLICY] = case["policy"]
        prm[W.P_SUBPARTITIONS] = case["subpartitions"]
        r, s = both(g, prm)
        assert r.status == 0, case["name"]
        assert list(r.start) == case["start"], (case["name"], list(r.start))
        assert_same(r, s)


def test_golden_noc():
    spec = json.load(open(os.path.join(GOLDEN, "noc.json")))
    for case in spec["cases"]:
        nodes = case["nodes"]
        g = TG.make(len(nodes), [], [TYPE[x[0]] for x in nodes], [x[1] for x in nodes], [x[2] for x in nodes],
                    case["warps_per_cta"], work=[x[3] for x in nodes])
        prm = W.with_noc(TG.unit_params(case["num_sms"], case["ctas_per_sm"]), *case["noc"])
        if "smem_bpc" in case:
            prm[W.P_SMEM_BPC] = case["smem_bpc"]
        r, s = both(g, prm)
        assert r.status == 0, case["name"]
        assert list(r.start) == case["start"], (case["name"], list(r.start))
        assert list(r.finish) == case["finish"], case["name"]
        assert r.makespan == case["makespan"], case["name"]
        assert r.busy[6] == sum(-(-x[3] // case["noc"][0]) for x in nodes if x[0] == "DSMEM")
        assert_same(r, s)


def test_stepper_equals_oracle_noc():
    rng = np.random.default_rng(60)
    types = (W.LOAD, W.SMEM, W.MMA, W.EW, W.BAR, W.NOP, W.DSMEM, W.DSMEM)
    for i in range(140):
        n = int(rng.integers(2, 20))
        g = TG.random_graph(rng, n, p_edge=float(rng.uniform(0.05, 0.3)), cta_major=bool(i % 3),
                            kernels=bool(i % 4 == 0), types=types)
        prm = TG.small_params(rng)
        prm = W.with_noc(prm, int(rng.integers(1, 4)), int(rng.integers(0, 4)), int(rng.integers(1, 3)),
                         int(rng.integers(1, 4)))
        if i % 3 == 1:
            prm = _with_policy(prm, int(rng.integers(1, 3)), int(rng.integers(1, 4)))
        r, s = both(g, prm)
        assert_same(r, s)


def test_noc_parameter_checks():
    g = TG.make(2, [], [W.DSMEM, W.NOP], [0, 0], [0, 0], 1, work=[4, 0])
    h = TG.make(2, [], [W.SMEM, W.NOP], [0, 0], [0, 0], 1, work=[4, 0])
    base = TG.unit_params(1, 1)
    assert run.simulate(g, base).status == run.ERR_INVALID_PARAMS        # DSMEM node, no NoC
    assert run.simulate(h, base).status == 0                              # no DSMEM node, no NoC
    assert run.simulate(g, W.with_noc(base, 1, 0, 1, 1)).status == 0
    for fields in ((0, 0, 1, 1), (1, -1, 1, 1), (1, 0, 0, 1), (1, 0, 33, 1), (1, 0, 1, 33), (1, 0, 1, 0),
                   (0, 5, 0, 0)):
        prm = base.copy()
        prm[W.P_NOC_BPC:W.P_CLUSTER_SMS + 1] = fields
        assert run.simulate(h, prm).status == run.ERR_INVALID_PARAMS, fields


def _l2_graph(case_nodes):
    n = len(case_nodes)
    g = TG.make(n, [(v, v + 1, W.DATA) for v in range(n - 1)], [TYPE[x[0]] for x in case_nodes], [0] * n,
                [0] * n, 1, work=[x[2] for x in case_nodes])
    g.tile = np.array([W.NO_TILE if x[1] < 0 else x[1] for x in case_nodes], np.uint32)
    g.n_tiles = 8
    return g


def _l2_params(l2_bytes, l2_lat=3, l2_bpc=2):
    prm = TG.unit_params(1, 1)
    prm[W.P_DRAM_LAT] = 10
    prm[W.P_L2_BYTES], prm[W.P_L2_LAT], prm[W.P_L2_BPC] = l2_bytes, l2_lat, l2_bpc
    return prm


def test_golden_l2():
    spec = json.load(open(os.path.join(GOLDEN, "l2.json")))
    for case in spec["cases"]:
        g = _l2_graph(case["nodes"])
        prm = _l2_params(case["l2_bytes"])
        r = run.simulate(g, prm)
        assert r.status == 0, case["name"]
        assert list(r.start) == case["start"], (case["name"], list(r.start))
        assert list(r.finish) == case["finish"], (case["name"], list(r.finish))
        assert (r.busy[7], r.busy[8], r.busy[5]) == (case["hits"], case["loads"], case["hbm_busy"]), case["name"]
        info = {}
        st, mk, start, fin, _ = stepper.simulate_graph(g, prm, info=info)
        assert (st, list(r.start), list(r.finish)) == (0, start, fin)
        assert list(r.busy) == stepper.busy_cycles(g.type, g.work, g.lat_extra, prm, start, mk, info)


def test_stepper_equals_oracle_l2():
    # the stepper decides hits by stack distance over its log of accesses, the
    # oracle by an explicit LRU list
    rng = np.random.default_rng(80)
    types = (W.LOAD, W.LOAD, W.LOAD, W.STORE, W.MMA, W.EW, W.NOP)
    for i in range(150):
        n = int(rng.integers(2, 24))
        g = TG.random_graph(rng, n, p_edge=float(rng.uniform(0.05, 0.35)), cta_major=bool(i % 3),
                            kernels=bool(i % 5 == 0), types=types, max_work=9)
        nt = int(rng.integers(1, 6))
        t = rng.integers(0, nt, n).astype(np.uint32)
        t[rng.random(n) < 0.15] = W.NO_TILE
        g.tile, g.n_tiles = t, nt
        prm = TG.small_params(rng)
        prm[W.P_L2_BYTES] = int(rng.integers(1, 30))
        prm[W.P_L2_LAT] = int(rng.integers(0, 5))
        prm[W.P_L2_BPC] = int(rng.integers(1, 6))
        if i % 4 == 1:
            prm = _with_policy(prm, int(rng.integers(1, 3)), int(rng.integers(1, 3)))
        r = run.simulate(g, prm)
        info = {}
        st, mk, start, fin, cta_sm = stepper.simulate_graph(g, prm, info=info)
        assert r.status == st
        if st == 0:
            assert r.makespan == mk and list(r.start) == start and list(r.finish) == fin
            assert list(r.busy) == stepper.busy_cycles(g.type, g.work, g.lat_extra, prm, start, mk, info)


def test_l2_closed_forms():
    rng = np.random.default_rng(81)
    for _ in range(20):
        k = int(rng.integers(2, 12))
        w = [int(x) for x in rng.integers(1, 6, k)]
        # every LOAD a new tile: no hits; one tile reloaded with room for it: all but the first hit
        distinct = _l2_graph([["LOAD", v, w[v]] for v in range(k)])
        distinct.n_tiles = k
        same = _l2_graph([["LOAD", 0, 5] for _ in range(k)])
        r1 = run.simulate(distinct, _l2_params(1000))
        r2 = run.simulate(same, _l2_params(5))
        assert (r1.busy[7], r1.busy[8]) == (0, k)
        assert (r2.busy[7], r2.busy[8]) == (k - 1, k)
        # a chain of misses: makespan = sum of (tma_lat + l2_lat + dram_lat + work); hits: 3 + 5 each
        assert r1.makespan == sum(13 + x for x in w)
        assert r2.makespan == 18 + (k - 1) * 8


def test_l2_parameter_checks():
    g = _l2_graph([["LOAD", 0, 4]])
    assert run.simulate(g, _l2_params(8)).status == 0
    for fields in ((0, 3, 0), (0, 0, 2), (8, -1, 2), (8, 3, 0), (-1, 3, 2)):
        prm = _l2_params(*fields) if fields[0] >= 0 else _l2_params(8)
        if fields[0] < 0:
            prm[W.P_L2_BYTES] = -1
        assert run.simulate(g, prm).status == run.ERR_INVALID_PARAMS, fields
    bad = g.subgraph(0)
    bad.tile = np.array([9], np.uint32)       # tile id >= n_tiles
    assert run.simulate(bad, _l2_params(8)).status == run.ERR_INVALID_GRAPH


def _with_policy(prm, policy, nsub):
    prm = prm.copy()
    prm[W.P_ISSUE_POLICY] = policy
    prm[W.P_SUBPARTITIONS] = nsub
    return prm


@pytest.mark.parametrize("policy", [W.POLICY_GTO, W.POLICY_RR])
def test_stepper_equals_oracle_policies(policy):
    rng = np.random.default_rng(40 + policy)
    for n in (1, 2, 3):
        for edges in TG.all_edge_sets(n):
            types = [int(x) for x in rng.integers(0, 7, n)]
            warps = [int(x) for x in rng.integers(0, 3, n)]
            ctas = sorted(int(x) for x in rng.integers(0, 2, n))
            g = TG.make(n, edges, types, warps, ctas, 3, work=[int(x) for x in rng.integers(0, 4, n)])
            prm = _with_policy(TG.small_params(rng, 1, 2), policy, int(rng.integers(1, 4)))
            r, s = both(g, prm)
            assert_same(r, s)
    for i in range(120):
        n = int(rng.integers(5, 22))
        g = TG.random_graph(rng, n, p_edge=float(rng.uniform(0.05, 0.35)), cta_major=bool(i % 3),
                            kernels=bool(i % 2))
        prm = _with_policy(TG.small_params(rng), policy, int(rng.integers(1, 5)))
        r, s = both(g, prm)
        assert_same(r, s)


@pytest.mark.parametrize("policy", [W.POLICY_GTO, W.POLICY_RR])
def test_one_issue_per_scheduler_per_cycle(policy):
    # W independent zero-latency warps of k nodes on one scheduler: the n nodes
    # start at 0, 1, ..., n-1 (no idle cycle, never two in one cycle); with s
    # schedulers every cycle issues min(s, warps left) nodes
    rng = np.random.default_rng(50 + policy)
    for _ in range(20):
        Wn = int(rng.integers(1, 6))
        k = int(rng.integers(1, 5))
        n = Wn * k
        g = TG.make(n, [], [W.NOP] * n, [v % Wn for v in range(n)], [0] * n, Wn, work=[0] * n)
        r = run.simulate(g, _with_policy(TG.unit_params(1, 1), policy, 1))
        assert r.status == 0
        assert sorted(r.start) == list(range(n))
        if Wn > 1:
            r2 = run.simulate(g, _with_policy(TG.unit_params(1, 1), policy, Wn))
            assert list(r2.start) == [v // Wn for v in range(n)]


def test_policy_parameter_checks():
    g = TG.make(2, [], [W.NOP, W.NOP], [0, 1], [0, 0], 2, work=[0, 0])
    base = TG.unit_params(1, 1)
    for policy, nsub in ((0, 1), (1, 0), (2, 33), (3, 1), (-1, 0)):
        assert run.simulate(g, _with_policy(base, policy, nsub)).status == run.ERR_INVALID_PARAMS
    bad = base.copy()
    bad[W.NPARAM - 1] = 1          # reserved
    assert run.simulate(g, bad).status == run.ERR_INVALID_PARAMS
    for policy, nsub in ((0, 0), (1, 1), (2, 32)):
        assert run.simulate(g, _with_policy(base, policy, nsub)).status == 0


# ------------------------------------------------------------------ brute force
@pytest.mark.parametrize("n", [1, 2, 3, 4])
def test_stepper_equals_oracle_exhaustive(n):
    rng = np.random.default_rng(100 + n)
    prms = [TG.unit_params(1, 1, 1, 1), TG.small_params(rng, 2, 1), TG.small_params(rng, 1, 2)]
    count = 0
    for edges in TG.all_edge_sets(n):
        for a in range(2 if n == 4 else 4):
            types = [int(x) for x in rng.integers(0, 7, n)]
            warps = [int(x) for x in rng.integers(0, 2, n)]
            ctas = sorted(int(x) for x in rng.integers(0, 2, n))
            work = [int(x) for x in rng.integers(0, 4, n)]
            g = TG.make(n, edges, types, warps, ctas, 2, kernels=[0, a % 2][: max(ctas) + 1], work=work)
            for prm in prms:
                r, s = both(g, prm)
                assert_same(r, s)
                count += 1
    assert count > 0


def test_stepper_equals_oracle_random():
    rng = np.random.default_rng(7)
    for i in range(160):
        n = int(rng.integers(5, 22))
        g = TG.random_graph(rng, n, p_edge=float(rng.uniform(0.05, 0.35)), cta_major=bool(i % 3),
                            kernels=bool(i % 2))
        prm = TG.small_params(rng)
        r, s = both(g, prm)
        assert_same(r, s)


def test_stepper_equals_oracle_small_gemm_cta():
    # one CTA of the 2-stage GEMM template with 2 k-steps and tiny work sizes
    tpl = W.gemm_2stage_cta(ksteps=3, warps=2, load_bytes=3, smem_bytes=2, mma_fma=4, ew_ops=2, store_bytes=3)
    g = W.assemble("g", 2, [tpl], np.zeros(2, np.int64), np.zeros(2, np.uint32))
    rng = np.random.default_rng(3)
    for _ in range(4):
        r, s = both(g, TG.small_params(rng))
        assert_same(r, s)


# ------------------------------------------------------------------ closed forms
def test_chain_makespan_is_sum_of_latencies():
    rng = np.random.default_rng(11)
    for _ in range(40):
        n = int(rng.integers(1, 60))
        types = [int(x) for x in rng.choice([W.LOAD, W.SMEM, W.MMA, W.EW, W.STORE], n)]
        work = [int(x) for x in rng.integers(1, 50, n)]
        W_ = int(rng.integers(1, 4))
        warps = [int(x) for x in rng.integers(0, W_, n)]
        ctas = sorted(int(x) for x in rng.integers(0, 4, n))
        edges = [(v, v + 1, W.DATA) for v in range(n - 1)]
        g = TG.make(n, edges, types, warps, ctas, W_, work=work)
        prm = TG.unit_params(int(rng.integers(1, 3)), int(rng.integers(1, 3)), int(rng.integers(1, 4)),
                             int(rng.integers(1, 4)))
        r = run.simulate(g, prm)
        assert r.status == 0
        assert r.makespan == sum(work)
        assert list(r.finish - r.start) == work


def _longest_path_starts(g, L):
    """Earliest start of every node with unlimited units and slots: longest path
    over DATA edges (weight L(u)), ISSUE edges (weight 0), warp program order
    (weight 0) and kernel-boundary gates (weight L(u) from every node of an
    earlier kernel), from a source at time 0."""
    n = g.n_nodes
    G = nx.DiGraph()
    src = n
    G.add_node(src)
    for v in range(n):
        G.add_edge(src, v, weight=0)

    def add(u, v, w):
        # keep the longest parallel edge, negated for a shortest-path solver
        if G.has_edge(u, v):
            G[u][v]["weight"] = min(G[u][v]["weight"], -w)
        else:
            G.add_edge(u, v, weight=-w)
    for u in range(n):
        for e in range(int(g.row_ptr[u]), int(g.row_ptr[u + 1])):
            add(u, int(g.col[e]), 0 if g.ekind[e] == W.ISSUE else L[u])
    last = {}
    for v in range(n):
        s = (int(g.cta[v]), int(g.warp[v]))
        if s in last:
            add(last[s], v, 0)
        last[s] = v
    kern = g.cta_kernel[g.cta]
    for u in range(n):
        for v in range(n):
            if kern[u] < kern[v]:
                add(u, v, L[u])
    d = nx.single_source_bellman_ford_path_length(G, src, weight="weight")
    return [-d[v] for v in range(n)]


def test_unlimited_resources_give_longest_path():
    rng = np.random.default_rng(12)
    for i in range(60):
        n = int(rng.integers(1, 30))
        g = TG.random_graph(rng, n, p_edge=float(rng.uniform(0.05, 0.4)), kernels=bool(i % 2),
                            types=(W.LOAD, W.SMEM, W.MMA, W.EW, W.STORE), max_work=20)
        g.lat_extra[:] = 0
        g.work[:] = np.maximum(g.work, 1)
        L = [int(x) for x in g.work]  # unit rates, zero base latency
        prm = TG.unit_params(num_sms=g.n_ctas, cps=1, caps=n + 1, cap_hbm=n + 1)
        r = run.simulate(g, prm)
        assert r.status == 0
        exp = _longest_path_starts(g, L)
        assert list(r.start) == exp
        assert r.makespan == max([exp[v] + L[v] for v in range(n)], default=0)


def test_single_server_no_idle():
    rng = np.random.default_rng(13)
    for _ in range(40):
        n = int(rng.integers(1, 40))
        g = TG.random_graph(rng, n, W_=int(rng.integers(1, 5)), C=1, p_edge=float(rng.uniform(0, 0.3)),
                            types=(W.MMA,), max_work=9)
        g.work[:] = np.maximum(g.work, 1)
        g.lat_extra[:] = 0
        r = run.simulate(g, TG.unit_params(1, 1, 1, 1))
        assert r.status == 0
        assert r.makespan == int(g.work.sum())
        assert r.busy[0] == r.makespan          # the tensor server never idles
        assert list(r.busy[1:]) == [0] * 8


# ------------------------------------------------------------------ bounds and invariants
def _occupancy_unit(g):
    """Unit-rate occupancies: per-SM class and HBM occupancy both equal work;
    BAR occupies 1; NOP nothing."""
    cls = {W.LOAD: "tma", W.STORE: "tma", W.SMEM: "lsu", W.MMA: "tensor", W.EW: "alu", W.BAR: "bar"}
    out = []
    for v in range(g.n_nodes):
        t = int(g.type[v])
        out.append((cls.get(t), 1 if t == W.BAR else int(g.work[v]),
                    int(g.work[v]) if t in (W.LOAD, W.STORE) else None))
    return out


def test_invariants_random_graphs():
    rng = np.random.default_rng(14)
    for i in range(80):
        n = int(rng.integers(1, 80))
        g = TG.random_graph(rng, n, p_edge=float(rng.uniform(0.02, 0.2)), kernels=bool(i % 2), max_work=12)
        caps = int(rng.integers(1, 3))
        cap_hbm = int(rng.integers(1, 3))
        prm = TG.unit_params(int(rng.integers(1, 3)), int(rng.integers(1, 3)), caps, cap_hbm)
        r = run.simulate(g, prm)
        assert r.status == 0
        occ = _occupancy_unit(g)
        L = [max([0] + [x for x in (o[1] if o[0] else None, o[2]) if x is not None]) + int(g.lat_extra[v])
             for v, o in enumerate(occ)]
        # finish = start + L
        assert list(r.finish - r.start) == L
        # predecessors respected
        for u in range(n):
            for e in range(int(g.row_ptr[u]), int(g.row_ptr[u + 1])):
                v = int(g.col[e])
                assert r.start[v] >= (r.start[u] if g.ekind[e] == W.ISSUE else r.finish[u])
        # warp program order
        last = {}
        for v in range(n):
            s = (int(g.cta[v]), int(g.warp[v]))
            if s in last:
                assert r.start[v] >= r.start[last[s]]
            last[s] = v
        # critical path lower bound
        crit = max([a + b for a, b in zip(_longest_path_starts(g, L), L)], default=0)
        assert r.makespan >= crit
        # capacity at every cycle and per-resource work bound
        sm = [int(r.cta_sm[int(g.cta[v])]) for v in range(n)]
        for t in range(int(r.makespan) + 1):
            use = {}
            h = 0
            for v in range(n):
                c, o, ho = occ[v]
                if c and r.start[v] <= t < r.start[v] + o:
                    use[(sm[v], c)] = use.get((sm[v], c), 0) + 1
                if ho is not None and r.start[v] <= t < r.start[v] + ho:
                    h += 1
            assert all(k <= caps for k in use.values())
            assert h <= cap_hbm
        work = {}
        for v in range(n):
            c, o, _ = occ[v]
            if c:
                work[(sm[v], c)] = work.get((sm[v], c), 0) + o
        assert all(w <= caps * r.makespan for w in work.values())
        assert sum(o[2] for o in occ if o[2] is not None) <= cap_hbm * r.makespan
        # busy server-cycles: per class the unit-rate occupancies; within capacity
        names = ("tensor", "tma", "lsu", "alu", "bar")
        for k, c in enumerate(names):
            assert r.busy[k] == sum(o[1] for o in occ if o[0] == c)
        assert r.busy[5] == sum(o[2] for o in occ if o[2] is not None)
        assert all(r.busy[k] <= caps * int(prm[0]) * r.makespan for k in range(5))
        assert r.busy[5] <= cap_hbm * r.makespan


def _opt_makespan(p, preds, m):
    """Brute-force optimum of P|prec|Cmax (m machines, processing times p):
    search over semi-active schedules (starts at 0 or at a completion)."""
    n = len(p)
    from functools import lru_cache

    @lru_cache(maxsize=None)
    def best(done, running):
        # running: tuple of (job, remaining) sorted
        if len(done) == n:
            return 0
        started = done | frozenset(j for j, _ in running)
        avail = [j for j in range(n) if j not in started and all(u in done for u in preds[j])]
        free = m - len(running)
        out = float("inf")
        from itertools import combinations
        for k in range(min(free, len(avail)), -1, -1):
            for pick in combinations(avail, k):
                run_ = list(running) + [(j, p[j]) for j in pick]
                if not run_:
                    continue
                dt = min(r for _, r in run_)
                fin = frozenset(j for j, r in run_ if r == dt)
                rest = tuple(sorted((j, r - dt) for j, r in run_ if r > dt))
                out = min(out, dt + best(done | fin, rest))
        return out
    return best(frozenset(), tuple())


def test_graham_list_scheduling_bound():
    rng = np.random.default_rng(15)
    for _ in range(25):
        n = int(rng.integers(2, 8))
        m = int(rng.integers(2, 4))
        edges = [(u, v, W.DATA) for v in range(n) for u in range(v) if rng.random() < 0.3]
        work = [int(x) for x in rng.integers(1, 6, n)]
        g = TG.make(n, edges, [W.MMA] * n, list(range(n)), [0] * n, n, work=work)
        r = run.simulate(g, TG.unit_params(1, 1, m, 1))
        assert r.status == 0
        preds = [[u for u, v, _ in edges if v == j] for j in range(n)]
        opt = _opt_makespan(work, preds, m)
        assert opt <= r.makespan <= (2 - 1 / m) * opt + 1e-9


# ------------------------------------------------------------------ error statuses
def test_error_statuses():
    g = TG.make(2, [(0, 1, W.DATA)], [W.EW, W.EW], [0, 0], [0, 0], 1)
    p = W.default_params()
    p[W.P_ALU_OPS_PC] = 0
    assert run.simulate(g, p).status == run.ERR_INVALID_PARAMS
    p = W.default_params()
    p[W.P_CAP_HBM] = 0
    assert run.simulate(g, p).status == run.ERR_INVALID_PARAMS
    p = W.default_params()
    p[W.P_BAR_LAT] = -1
    assert run.simulate(g, p).status == run.ERR_INVALID_PARAMS
    bad = TG.make(2, [(0, 1, W.DATA)], [W.EW, W.EW], [0, 0], [0, 0], 1)
    bad.col[0] = 0  # self edge
    assert run.simulate(bad, W.default_params()).status == run.ERR_INVALID_GRAPH
    bad = TG.make(2, [], [W.EW, 9], [0, 0], [0, 0], 1)
    assert run.simulate(bad, W.default_params()).status == run.ERR_INVALID_GRAPH
    bad = TG.make(2, [], [W.EW, W.EW], [0, 3], [0, 0], 2)
    assert run.simulate(bad, W.default_params()).status == run.ERR_INVALID_GRAPH
    # overflow: a LOAD of 2^32-1 bytes at 1 B/cycle
    big = TG.make(1, [], [W.LOAD], [0], [0], 1, work=[2**32 - 1])
    assert run.simulate(big, TG.unit_params()).status == run.ERR_OVERFLOW
    # finish exactly 2^31-1 is representable
    edge = TG.make(1, [], [W.NOP], [0], [0], 1, lat_extra=[2**31 - 1])
    r = run.simulate(edge, TG.unit_params())
    assert r.status == 0 and r.makespan == 2**31 - 1
    # deadlock: CTA0's node waits on CTA1's node, CTA1 cannot launch (1 slot)
    dl = TG.make(2, [(0, 1, W.DATA)], [W.EW, W.EW], [0, 0], [1, 0], 1)
    assert run.simulate(dl, TG.unit_params(1, 1)).status == run.ERR_DEADLOCK
    s = stepper.simulate_graph(dl, TG.unit_params(1, 1))
    assert s[0] == run.ERR_DEADLOCK


def test_empty_graph_and_empty_ctas():
    g = TG.make(0, [], [], [], [], 1)
    r = run.simulate(g, W.default_params())
    assert r.status == 0 and r.makespan == 0
    # CTA 1 has no nodes: it launches and retires at once
    g = TG.make(2, [], [W.EW, W.EW], [0, 0], [0, 2], 1, work=[3, 4])
    prm = TG.unit_params(1, 1)
    r, s = both(g, prm)
    assert_same(r, s)
    assert list(r.start) == [0, 3] and list(r.cta_sm) == [0, 0, 0]
