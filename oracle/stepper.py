"""Cycle-by-cycle stepper for tiny tile graphs (TEST INFRASTRUCTURE ONLY).

A second, independent statement of the scheduling definition (Section 5.1 to
5.3) used to pin the C oracle on tiny inputs.  It differs from the oracle on
purpose in everything but the definition:

* time advances one cycle at a time (t = 0, 1, 2, ...), no event skipping;
* nothing is tracked incrementally: readiness, warp heads, resource usage and
  CTA residency are recomputed from the partial schedule at every decision;
* a resource class is free at t when fewer than ``cap`` of the nodes already
  started on it satisfy start <= t < start + occupancy (counting, not the
  server free-time multiset the oracle keeps);
* under the per-subpartition issue policies, a scheduler has issued at t when
  a node of its warp slots started at t, and the slot it issued from last is
  that of its latest-started node (read off the schedule, no scheduler state);
* the L2 keeps no cache state: a LOAD hits when its tile was accessed before
  and survived every trim since, i.e. after each later access its bytes plus
  the bytes (as of then) of the other tiles accessed since still fit in the
  capacity -- the LRU stack-distance property (Mattson et al. 1970) for
  entries of changing sizes, read off the log of accesses in issue order.

Pure Python; only for graphs of a few dozen nodes with short latencies.
"""
from __future__ import annotations

LOAD, SMEM, MMA, EW, STORE, BAR, NOP, DSMEM = range(8)
ISSUE = 1


def node_costs(ty, work, lat_extra, prm):
    """(per-SM class or None, its occupancy, HBM occupancy or None, NoC
    occupancy or None, latency)."""
    def cdiv(a, b):
        return -(-a // b)
    num = {"hbm": prm[2], "tma": prm[4], "smem": prm[6], "mma": prm[8], "alu": prm[10]}
    nocc = None
    if ty == LOAD:
        cls, occ, hocc, base = "tma", cdiv(work, num["tma"]), cdiv(work, num["hbm"]), prm[5] + prm[3]
    elif ty == STORE:
        cls, occ, hocc, base = "tma", cdiv(work, num["tma"]), cdiv(work, num["hbm"]), prm[5]
    elif ty == SMEM:
        cls, occ, hocc, base = "lsu", cdiv(work, num["smem"]), None, prm[7]
    elif ty == MMA:
        cls, occ, hocc, base = "tensor", cdiv(work, num["mma"]), None, prm[9]
    elif ty == EW:
        cls, occ, hocc, base = "alu", cdiv(work, num["alu"]), None, prm[11]
    elif ty == BAR:
        cls, occ, hocc, base = "bar", 1, None, prm[12]
    elif ty == DSMEM:   # the local shared-memory port plus the SM group's NoC
        cls, occ, hocc, base = "lsu", cdiv(work, num["smem"]), None, prm[7] + prm[23]
        nocc = cdiv(work, prm[22])
    else:
        cls, occ, hocc, base = None, 0, None, 0
    lat = base + lat_extra + max([0] + ([occ] if cls else []) + [x for x in (hocc, nocc) if x is not None])
    return cls, occ, hocc, nocc, lat


NO_TILE = 0xFFFFFFFF


def simulate(row_ptr, col, ekind, type_, warp, cta, work, lat_extra, cta_kernel, warps_per_cta, prm,
             t_limit=None, tile=None, info=None):
    """Returns (status, makespan, start list, finish list, cta_sm list).

    status: 0 ok, -6 a finish above 2^31-1, -8 no progress possible.  With a
    dict ``info``, also fills info["hbm_occ"] (memory-side occupancy per node
    as issued) and info["l2"] = [LOAD hits, LOADs naming a tile].
    """
    n = len(type_)
    C = len(cta_kernel)
    prm = [int(x) for x in prm]
    num_sms, cps = prm[0], prm[1]
    policy, nsub = prm[20], prm[21]
    per = cps * warps_per_cta
    cap = {"tensor": prm[13], "tma": prm[14], "lsu": prm[15], "alu": prm[16], "bar": prm[17]}
    cap_hbm = prm[18]
    cap_noc, group = prm[24], prm[25]
    l2_cap, l2_lat, l2_bpc = prm[26], prm[27], prm[28]
    accesses = []          # (tile, bytes) of LOAD/STORE nodes naming a tile, in issue order
    dyn = {}               # node -> (memory-side occupancy, latency) decided at issue
    l2_count = [0, 0]

    def tile_of(v):
        if tile is None or int(type_[v]) not in (LOAD, STORE) or int(tile[v]) == NO_TILE:
            return None
        return int(tile[v])

    def l2_hit(x):
        last = [k for k, (y, _b) in enumerate(accesses) if y == x]
        if not last:
            return False
        since, worst = {}, 0
        for y, b in accesses[last[-1] + 1:]:
            since[y] = b
            worst = max(worst, sum(since.values()))
        return worst + accesses[last[-1]][1] <= l2_cap
    costs = [node_costs(int(type_[v]), int(work[v]), int(lat_extra[v]), prm) for v in range(n)]
    preds = [[] for _ in range(n)]
    for u in range(n):
        for e in range(int(row_ptr[u]), int(row_ptr[u + 1])):
            preds[int(col[e])].append((u, int(ekind[e])))
    members = [[v for v in range(n) if int(cta[v]) == c] for c in range(C)]
    start = [None] * n
    cta_sm = [-1] * C
    cta_slot = [-1] * C
    launched = [False] * C
    total_lat = sum(c[4] for c in costs)
    if l2_cap:   # with the L2 a LOAD can take up to l2_lat + work cycles more
        total_lat += sum(l2_lat + int(work[v]) for v in range(n) if int(type_[v]) == LOAD)
    if t_limit is None:   # every cycle without an issue lies under some node's latency or issue slot
        t_limit = total_lat + n + 2

    def finish(v):
        return start[v] + (dyn[v][1] if v in dyn else costs[v][4])

    def hocc_of(u):
        return dyn[u][0] if u in dyn else costs[u][2]

    def retired(c, t):
        return launched[c] and all(start[v] is not None and finish(v) <= t for v in members[c])

    def is_head(v):
        return all(start[u] is not None for u in members[int(cta[v])]
                   if u < v and int(warp[u]) == int(warp[v]))

    def busy(cls, sm, t):
        k = 0
        for u in range(n):
            if start[u] is None or costs[u][0] != cls or cta_sm[int(cta[u])] != sm:
                continue
            if start[u] <= t < start[u] + costs[u][1]:
                k += 1
        return k

    def busy_hbm(t):
        return sum(1 for u in range(n) if start[u] is not None and hocc_of(u) is not None
                   and start[u] <= t < start[u] + hocc_of(u))

    def busy_noc(grp, t):
        return sum(1 for u in range(n) if start[u] is not None and costs[u][3] is not None
                   and cta_sm[int(cta[u])] // group == grp and start[u] <= t < start[u] + costs[u][3])

    def sched(v):
        """(SM, scheduler, warp slot) of node v's warp."""
        c = int(cta[v])
        slot = cta_slot[c] * warps_per_cta + int(warp[v])
        return cta_sm[c], slot % nsub, slot

    def scheduler_picks(cands, t):
        """Per scheduler that has not issued at t, its first candidate in policy order."""
        groups = {}
        for v in cands:
            groups.setdefault(sched(v)[:2], []).append(v)
        picks = []
        for key, vs in groups.items():
            mine = [u for u in range(n) if start[u] is not None and sched(u)[:2] == key]
            if any(start[u] == t for u in mine):
                continue
            last = sched(max(mine, key=lambda u: start[u]))[2] if mine else None

            def order(v):
                slot = sched(v)[2]
                if policy == 1:   # greedy-then-oldest
                    return (slot != last, int(cta[v]) * warps_per_cta + int(warp[v]))
                return slot if last is None else (slot - last - 1) % per   # round-robin
            picks.append(min(vs, key=order))
        return picks

    def issuable(v, t):
        c = int(cta[v])
        if start[v] is not None or not launched[c] or not is_head(v):
            return False
        rel = 0
        for u, k in preds[v]:
            if start[u] is None:
                return False
            rel = max(rel, start[u] if k == ISSUE else finish(u))
        if rel > t:
            return False
        cls, _occ, hocc, nocc, _lat = costs[v]
        if cls is not None and busy(cls, cta_sm[c], t) >= cap[cls]:
            return False
        if hocc is not None and busy_hbm(t) >= cap_hbm:
            return False
        if nocc is not None and busy_noc(cta_sm[c] // group, t) >= cap_noc:
            return False
        return True

    t = 0
    while True:
        changed = True
        while changed:
            changed = False
            # CTA launches in ascending order, each on the lowest SM with a free slot
            while True:
                c = sum(launched)
                if c >= C:
                    break
                if any(int(cta_kernel[d]) < int(cta_kernel[c]) and not retired(d, t) for d in range(c)):
                    break
                occupied = [0] * num_sms
                for d in range(c):
                    if not retired(d, t):
                        occupied[cta_sm[d]] += 1
                free = [s for s in range(num_sms) if occupied[s] < cps]
                if not free:
                    break
                launched[c] = True
                cta_sm[c] = free[0]
                taken = {cta_slot[d] for d in range(c) if cta_sm[d] == free[0] and not retired(d, t)}
                cta_slot[c] = min(k for k in range(cps) if k not in taken)
                changed = True
            cands = [v for v in range(n) if issuable(v, t)]
            if cands and nsub:
                cands = scheduler_picks(cands, t)
            if cands:
                v = min(cands)
                x = tile_of(v)
                if l2_cap and int(type_[v]) == LOAD:
                    hit = x is not None and l2_hit(x)
                    w = int(work[v])
                    ho = -(-w // (l2_bpc if hit else prm[2]))
                    occ = costs[v][1]
                    dyn[v] = (ho, prm[5] + l2_lat + (0 if hit else prm[3]) + int(lat_extra[v]) + max(occ, ho))
                    if x is not None:
                        l2_count[0] += hit
                        l2_count[1] += 1
                if l2_cap and x is not None:
                    accesses.append((x, int(work[v])))
                start[v] = t
                if finish(v) > 2**31 - 1:
                    return -6, 0, start, [None] * n, cta_sm
                changed = True
        if all(s is not None for s in start):
            fin = [finish(v) for v in range(n)]
            if info is not None:
                info["hbm_occ"] = [hocc_of(v) for v in range(n)]
                info["l2"] = list(l2_count)
            return 0, max(fin, default=0), start, fin, cta_sm
        t += 1
        if t > t_limit:
            return -8, 0, start, [None] * n, cta_sm


CLASS_ORDER = ("tensor", "tma", "lsu", "alu", "bar", "hbm", "noc")


def busy_cycles(type_, work, lat_extra, prm, start, makespan, info=None):
    """Busy server-cycles of each class, measured on a finished schedule by
    sweeping every cycle t in [0, makespan) and counting the servers held at t
    (a node holds one server of its class on [start, start + occupancy), one
    HBM server on [start, start + HBM occupancy) and one NoC server on
    [start, start + NoC occupancy)).  Returned in the order TENSOR, TMA, LSU,
    ALU, BAR, HBM, NoC, then the L2 counts of ``info`` (from ``simulate``;
    its memory-side occupancies replace the static ones)."""
    prm = [int(x) for x in prm]
    costs = [node_costs(int(type_[v]), int(work[v]), int(lat_extra[v]), prm) for v in range(len(type_))]
    if info is not None:
        costs = [(c[0], c[1], info["hbm_occ"][v], c[3], c[4]) for v, c in enumerate(costs)]
    total = dict.fromkeys(CLASS_ORDER, 0)
    for t in range(makespan):
        for v, (cls, occ, hocc, nocc, _lat) in enumerate(costs):
            if cls is not None and start[v] <= t < start[v] + occ:
                total[cls] += 1
            if hocc is not None and start[v] <= t < start[v] + hocc:
                total["hbm"] += 1
            if nocc is not None and start[v] <= t < start[v] + nocc:
                total["noc"] += 1
    return [total[k] for k in CLASS_ORDER] + (list(info["l2"]) if info is not None else [0, 0])


def simulate_graph(g, prm, **kw):
    """Same, for a single workloads.Graph."""
    return simulate(g.row_ptr, g.col, g.ekind, g.type, g.warp, g.cta, g.work, g.lat_extra, g.cta_kernel,
                    g.warps_per_cta, prm, tile=g.tile, **kw)
