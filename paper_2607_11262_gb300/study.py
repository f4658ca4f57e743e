"""Case studies on the GPU: software pipelining and the tile-graph ablation
(Section 7.1 "Software Pipelining Impact"; Section 6.4 ablation), NoC-enabled
fusion (Section 7.2), and the L2 model (Section 5.2) under two tile orders.

Every (organisation, tile, ablation) graph of ``pipelines.study_set`` runs on
one simulated Hopper SM through libgts; the table reports, per graph, the
makespan, the tensor-pipe utilisation (busy tensor cycles / makespan, from the
engine's busy-cycle output) and the performance normalised to the fastest
organisation of the same tile.  With ``--points-per-graph`` > 1 the extra
design points sweep DRAM bandwidth and tensor rate, and the table adds the
utilisation's minimum, mean and maximum over the sweep.

The NoC study runs the cluster-fused attention decode of ``clusters`` with
NoC and with DRAM exchanges for every cluster size and reports both makespans,
the speedup and the NoC utilisation (busy NoC cycles / (servers x makespan)).

The L2 study runs the persistent GEMM of ``l2gemm`` in row-major and grouped
rasterization at L2 capacities of 0-100 MB and reports makespan and hit rate.

The policy study reruns workloads' design points under the per-subpartition
issue policies (greedy-then-oldest, round-robin; Section 5.3) with 1, 2 and 4
schedulers per SM and compares each makespan with the lowest-id order.

    python -m paper_2607_11262_gb300.study [--study pipelines|noc|l2|policies] [--points-per-graph 64] [--json out.json]
"""
from __future__ import annotations

import argparse
import json

import numpy as np

from . import clusters, gts, l2gemm, pipelines, workloads


def run_study(points_per_graph=1, device="cuda"):
    """Runs the study; returns a list of dicts, one per graph, in stacking order."""
    import torch
    gts.load()
    graph, cases = pipelines.study_set()
    params = pipelines.study_params(len(cases), points_per_graph)
    dg = gts.DeviceGraph(graph, device=device)
    dp = gts.DeviceParams(dg, params)
    out = gts.simulate(dg, dp, flags=gts.GTS_WANT_BUSY)
    torch.cuda.synchronize()
    status = out.status.cpu().numpy()
    if np.any(status != gts.GTS_OK):
        raise gts.GtsError(int(status[status != 0][0]), "a study point did not simulate")
    mk = out.makespan.cpu().numpy()
    busy = out.busy.cpu().numpy()
    util = gts.utilisation(busy, mk, params)[:, gts.GTS_BUSY_TENSOR]
    dp.close()
    dg.close()
    rows = []
    for i, (org, tile, abl) in enumerate(cases):
        sl = slice(i * points_per_graph, (i + 1) * points_per_graph)
        rows.append(dict(org=org, tile=list(tile), ablation=abl, makespan=int(mk[sl][0]),
                         tensor_util=float(util[sl][0]), tensor_busy=int(busy[sl][0, gts.GTS_BUSY_TENSOR]),
                         tma_busy=int(busy[sl][0, gts.GTS_BUSY_TMA]),
                         util_min=float(util[sl].min()), util_mean=float(util[sl].mean()),
                         util_max=float(util[sl].max())))
    best = {}
    for r in rows:
        if r["ablation"] == "full":
            k = tuple(r["tile"])
            best[k] = min(best.get(k, r["makespan"]), r["makespan"])
    for r in rows:
        r["normalised_perf"] = best[tuple(r["tile"])] / r["makespan"]
    return rows


def run_noc_study(points_per_graph=1, device="cuda"):
    """NoC-vs-DRAM fusion study; one dict per cluster size, makespans of the
    default point and the speedup over the sweep (min / mean / max)."""
    import torch
    gts.load()
    graph, cases = clusters.study_set()
    params = clusters.study_params(cases, points_per_graph=points_per_graph)
    dg = gts.DeviceGraph(graph, device=device)
    dp = gts.DeviceParams(dg, params)
    out = gts.simulate(dg, dp, flags=gts.GTS_WANT_BUSY)
    torch.cuda.synchronize()
    status = out.status.cpu().numpy()
    if np.any(status != gts.GTS_OK):
        raise gts.GtsError(int(status[status != 0][0]), "a study point did not simulate")
    mk = out.makespan.cpu().numpy().reshape(len(cases), points_per_graph)
    util = gts.utilisation(out.busy.cpu().numpy(), out.makespan.cpu().numpy(), params)
    util = util.reshape(len(cases), points_per_graph, gts.GTS_BUSY_CLASSES)
    dp.close()
    dg.close()
    rows = []
    for k in clusters.CLUSTER_SIZES:
        a, b = cases.index((k, "noc")), cases.index((k, "dram"))
        sp = mk[b] / mk[a]
        rows.append(dict(cluster=k, noc_makespan=int(mk[a][0]), dram_makespan=int(mk[b][0]),
                         speedup=float(sp[0]), speedup_min=float(sp.min()), speedup_mean=float(sp.mean()),
                         speedup_max=float(sp.max()), noc_util=float(util[a][0, gts.GTS_BUSY_NOC]),
                         hbm_util_noc=float(util[a][0, gts.GTS_BUSY_HBM]),
                         hbm_util_dram=float(util[b][0, gts.GTS_BUSY_HBM])))
    return rows


def run_l2_study(device="cuda"):
    """L2 capacity x tile order; one dict per (order, capacity)."""
    import torch
    gts.load()
    graph, orders = l2gemm.study_set()
    params = l2gemm.study_params(len(orders))
    dg = gts.DeviceGraph(graph, device=device)
    dp = gts.DeviceParams(dg, params)
    out = gts.simulate(dg, dp, flags=gts.GTS_WANT_BUSY)
    torch.cuda.synchronize()
    status = out.status.cpu().numpy()
    if np.any(status != gts.GTS_OK):
        raise gts.GtsError(int(status[status != 0][0]), "a study point did not simulate")
    mk = out.makespan.cpu().numpy()
    busy = out.busy.cpu().numpy()
    dp.close()
    dg.close()
    rows = []
    for q in range(params.shape[0]):
        loads = int(busy[q, gts.GTS_BUSY_L2_LOADS])
        rows.append(dict(order=orders[int(params[q, 19])], l2_mb=int(params[q, 26]) >> 20, makespan=int(mk[q]),
                         hits=int(busy[q, gts.GTS_BUSY_L2_HITS]), loads=loads,
                         hit_rate=float(busy[q, gts.GTS_BUSY_L2_HITS]) / loads if loads else 0.0))
    return rows


POLICY_CASES = (("gto", 1), ("gto", 2), ("gto", 4), ("rr", 1), ("rr", 2), ("rr", 4))


def run_policy_study(names=("gemm512", "wsgemm_small", "fa_fwd"), points=64, device="cuda"):
    """Makespan under each issue policy relative to lowest-id, per workload:
    one dict per (workload, policy, schedulers) with the ratio's min / mean /
    max over the points."""
    import torch
    gts.load()
    code = {"gto": workloads.POLICY_GTO, "rr": workloads.POLICY_RR}
    rows = []
    for name in names:
        w = workloads.workload(name)
        idx = np.linspace(0, w.params.shape[0] - 1, min(points, w.params.shape[0])).round().astype(int)
        base = w.params[idx]
        variants = [base]
        for pol, nsub in POLICY_CASES:
            p = base.copy()
            p[:, workloads.P_ISSUE_POLICY] = code[pol]
            p[:, workloads.P_SUBPARTITIONS] = nsub
            variants.append(p)
        table = np.ascontiguousarray(np.concatenate(variants), np.int32)
        dg = gts.DeviceGraph(w.graph, device=device)
        dp = gts.DeviceParams(dg, table)
        out = gts.simulate(dg, dp, flags=0)
        torch.cuda.synchronize()
        status = out.status.cpu().numpy()
        if np.any(status != gts.GTS_OK):
            raise gts.GtsError(int(status[status != 0][0]), "a study point did not simulate")
        mk = out.makespan.cpu().numpy().reshape(len(variants), len(idx)).astype(np.float64)
        dp.close()
        dg.close()
        for k, (pol, nsub) in enumerate(POLICY_CASES):
            r = mk[k + 1] / mk[0]
            rows.append(dict(workload=name, policy=pol, schedulers=nsub, points=len(idx), ratio_min=float(r.min()),
                             ratio_mean=float(r.mean()), ratio_max=float(r.max())))
    return rows


def format_policy_table(rows):
    lines = [f"{'workload':<14}{'policy':<8}{'schedulers':>11}{'makespan / lowest-id (min / mean / max)':>42}"]
    for r in rows:
        lines.append(f"{r['workload']:<14}{r['policy']:<8}{r['schedulers']:>11}"
                     f"{r['ratio_min']:>24.3f} / {r['ratio_mean']:.3f} / {r['ratio_max']:.3f}")
    return "\n".join(lines)


def format_l2_table(rows):
    lines = [f"{'order':<10}{'L2 MB':>7}{'cycles':>12}{'hits':>9}{'loads':>9}{'hit rate':>10}"]
    for r in rows:
        lines.append(f"{r['order']:<10}{r['l2_mb']:>7}{r['makespan']:>12}{r['hits']:>9}{r['loads']:>9}"
                     f"{100 * r['hit_rate']:>9.1f}%")
    return "\n".join(lines)


def format_noc_table(rows):
    lines = [f"{'cluster':>8}{'NoC cycles':>12}{'DRAM cycles':>13}{'speedup':>9}{'sweep min/mean/max':>22}"
             f"{'NoC util':>10}{'HBM util NoC/DRAM':>19}"]
    for r in rows:
        lines.append(f"{r['cluster']:>8}{r['noc_makespan']:>12}{r['dram_makespan']:>13}{r['speedup']:>9.3f}"
                     f"{r['speedup_min']:>10.3f}/{r['speedup_mean']:.3f}/{r['speedup_max']:.3f}"
                     f"{100 * r['noc_util']:>9.1f}%{100 * r['hbm_util_noc']:>11.1f}/{100 * r['hbm_util_dram']:.1f}%")
    return "\n".join(lines)


def format_table(rows):
    lines = [f"{'organisation':<16}{'tile':<15}{'ablation':<11}{'makespan':>10}{'perf':>7}{'tensor':>8}"
             f"{'sweep min/mean/max':>22}"]
    for r in rows:
        tile = "x".join(str(x) for x in r["tile"])
        lines.append(f"{r['org']:<16}{tile:<15}{r['ablation']:<11}{r['makespan']:>10d}{r['normalised_perf']:>7.3f}"
                     f"{100 * r['tensor_util']:>7.1f}%{100 * r['util_min']:>8.1f}/{100 * r['util_mean']:.1f}/"
                     f"{100 * r['util_max']:.1f}%")
    return "\n".join(lines)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--study", default="pipelines", choices=["pipelines", "noc", "l2", "policies"])
    ap.add_argument("--points-per-graph", type=int, default=1)
    ap.add_argument("--json", default=None)
    args = ap.parse_args()
    if args.study == "noc":
        rows = run_noc_study(args.points_per_graph)
        print(format_noc_table(rows))
    elif args.study == "l2":
        rows = run_l2_study()
        print(format_l2_table(rows))
    elif args.study == "policies":
        rows = run_policy_study(points=args.points_per_graph)
        print(format_policy_table(rows))
    else:
        rows = run_study(args.points_per_graph)
        print(format_table(rows))
    if args.json:
        with open(args.json, "w") as f:
            json.dump(rows, f, indent=1)


if __name__ == "__main__":
    main()
