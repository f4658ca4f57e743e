"""Benchmark: batched tile-graph simulation throughput on GB300.

One step = one gts_simulate_batch over every design point of the workload
(full per-node start/finish trace), i.e. one pass of the whole hot path.
Default workload: the warp-specialised persistent GEMM 8192^3 tile graph
(1.58M nodes) x 4096 design points.  Prints ONE JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle on the host cores

Under torchrun (N > 1) the sweep is one table of N x P rows: rank 0's rows are
the workload's own table, rank r's rows are drawn with a rank-specific seed.
Rank r simulates the contiguous rows [r*P, (r+1)*P) on its own GPU (P per GPU:
weak scaling) with no collective in the data path; after the timed steps the
per-point makespans, statuses and digests are gathered to rank 0 and the step
time is the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "simulated tile-graph nodes/sec"
UNIT = "node-points/s"
KERNEL_SRC = os.path.join(ROOT, "paper_2607_11262_gb300", "csrc", "gts.cu")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic_k_simulate.txt")
ISSUE_FILE = os.path.join(ROOT, "profiles", "issue_k_simulate.txt")
SCHEDULERS_PER_SM = 4  # warp schedulers per SM; each issues at most one warp-instruction per cycle


def node_points_of(graph, params):
    """Simulated nodes summed over the design points (each point runs its graph)."""
    if graph.n_graphs == 1:
        return graph.n_nodes * int(params.shape[0])
    sizes = np.diff(graph.node_off.astype(np.int64))
    return int(sizes[params[:, 19]].sum())


def algorithmic_bytes(graph, params, full_trace=True):
    """Bytes the batch must move at minimum: the graph read once (node fields
    1+2+4+4+4+2 B, row pointers, 5 B per edge), the parameter rows, and per
    point its trace (start + finish, 8 B per node), makespan and status."""
    n, m = graph.n_nodes, graph.n_edges
    graph_bytes = n * (1 + 2 + 4 + 4 + 4 + 2) + (n + 1) * 4 + m * 5
    P = int(params.shape[0])
    row = 4 * int(params.shape[1])
    return graph_bytes + row * P + (8 * node_points_of(graph, params) if full_trace else 0) + 8 * P


def profiled(path, name):
    """A profile figure file, if it was taken on this kernel source and workload."""
    if not os.path.exists(path):
        return None
    f = json.load(open(path))
    return f if f.get("source_sha256_16") == source_hash() and name in f.get("applies_to", []) else None


def code_tokens(text):
    """C/C++/CUDA source with comments removed and whitespace runs collapsed
    (string and character literals kept), so that a comment edit keeps the
    hash and any change to the code changes it."""
    out, i, n = [], 0, len(text)

    def space():
        if out and out[-1] != " ":
            out.append(" ")

    while i < n:
        c = text[i]
        if c in "\"'":
            j = i + 1
            while j < n and text[j] != c:
                j += 2 if text[j] == "\\" else 1
            out.append(text[i:j + 1])
            i = j + 1
        elif text.startswith("//", i):
            j = text.find("\n", i)
            i = n if j < 0 else j
        elif text.startswith("/*", i):
            j = text.find("*/", i + 2)
            i = n if j < 0 else j + 2
            space()
        elif c.isspace():
            j = i
            while j < n and text[j].isspace():
                j += 1
            space()
            i = j
        else:
            out.append(c)
            i += 1
    return "".join(out).strip()


def source_hash():
    """First 16 hex digits of the SHA-256 of the kernel source's code (comments excluded)."""
    return hashlib.sha256(code_tokens(open(KERNEL_SRC).read()).encode()).hexdigest()[:16]


class Clocks:
    """nvidia-smi sampling of SM clock and throttle reasons during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.lines = []
        self.reader = None

    def start(self):
        import threading
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.dev}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.reader = threading.Thread(target=lambda: self.lines.extend(self.proc.stdout), daemon=True)
        self.reader.start()

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.reader.join(timeout=5)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in list(self.lines):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for nm, val in zip(names, f[5:9]):
                if val.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def reduce_max_over_ranks(value, device=None):
    """Max of a per-rank float over the process group (identity without one)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(node_points_per_rank, world, ms_per_step):
    """Whole-job throughput: every rank's node-points over the slowest rank's time."""
    return node_points_per_rank * world / (ms_per_step / 1e3)


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    return ws, int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0"))


POLICIES = {"lowest_id": 0, "gto": 1, "rr": 2}


def rank_params(name, rank, w):
    """The rows of rank ``rank`` in the N-rank sweep: the workload's own table
    for rank 0, a table of the same size and axes drawn with a rank-specific
    seed for rank r > 0 (stress: the same instances on every rank)."""
    from paper_2607_11262_gb300 import workloads as W
    if rank == 0 or name == "stress":
        return w.params
    if name == "pipelines":
        from paper_2607_11262_gb300 import pipelines
        return pipelines.study_params(w.graph.n_graphs, 64, seed=W.SEED0 + 6 + 100 * rank)
    if name == "l2_gemm":
        from paper_2607_11262_gb300 import l2gemm
        return l2gemm.study_params(w.graph.n_graphs, points_per_capacity=8, seed=W.SEED0 + 8 + 100 * rank)
    if name == "noc_fusion":
        from paper_2607_11262_gb300 import clusters
        return clusters.study_params(clusters.study_cases(), points_per_graph=32, seed=W.SEED0 + 7 + 100 * rank)
    axes = {"gemm512": [W.AX_SMS, W.AX_HBM, (W.P_MMA_LAT, 16, 64)],
            "wsgemm8192": [W.AX_SMS, W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE],
            "wsgemm_small": [W.AX_SMS, W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE]}.get(
        name, [W.AX_SMS, W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE, W.AX_ALU_RATE])
    cps = int(w.params[0, W.P_CTAS_PER_SM])
    seed = W.SEED0 + 100 * rank + (W.WORKLOADS.index(name) + 1 if name in W.WORKLOADS else 2)
    return W.sweep_params(seed, w.params.shape[0], axes, cps)


def global_table(name, world, points=None, policy="lowest_id", subpartitions=4):
    """(workload, rows of all ``world`` ranks concatenated: [world * P][32])."""
    from paper_2607_11262_gb300 import workloads as W
    w = W.workload(name)
    parts = []
    for r in range(world):
        p = np.array(rank_params(name, r, w), np.int32, copy=True)
        if points is not None:
            p = p[:points]
        p[:, W.P_ISSUE_POLICY] = POLICIES[policy]
        p[:, W.P_SUBPARTITIONS] = 0 if policy == "lowest_id" else subpartitions
        parts.append(p)
    return w, np.ascontiguousarray(np.concatenate(parts))


def rank_range(total, world, rank):
    """Contiguous rows [lo, hi) of rank ``rank`` (equal shares; the last rank
    takes the remainder)."""
    per = total // world
    lo = rank * per
    return lo, (total if rank == world - 1 else lo + per)


def load_workload(name, rank, points, policy="lowest_id", subpartitions=4, world=1):
    """This rank's workload: the graph and its contiguous rows of the N-rank table."""
    w, table = global_table(name, max(world, rank + 1), points, policy, subpartitions)
    lo, hi = rank_range(table.shape[0], max(world, rank + 1), rank)
    w.params = np.ascontiguousarray(table[lo:hi])
    return w


def gather_to_rank0(arrays, device=None):
    """Concatenation over ranks (in rank order) of each per-point array, on
    rank 0 (numpy); None on the other ranks.  Without a process group, the
    arrays themselves.  Every rank must pass arrays of the same lengths."""
    import torch
    import torch.distributed as dist

    def as_tensor(a):
        return a.contiguous() if isinstance(a, torch.Tensor) else torch.as_tensor(np.ascontiguousarray(a))
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [as_tensor(a).cpu().numpy() for a in arrays]
    world, rank = dist.get_world_size(), dist.get_rank()
    out = []
    for a in arrays:
        t = as_tensor(a).to(device if device is not None else "cpu")
        parts = [torch.empty_like(t) for _ in range(world)]
        dist.all_gather(parts, t)
        out.append(np.concatenate([x.cpu().numpy() for x in parts]) if rank == 0 else None)
    return out if rank == 0 else None


def workload_config(w, args, world):
    """The ``config`` object both arms print for a workload."""
    return {"workload": w.name, "description": w.description, "nodes": w.graph.max_graph_nodes,
            "edges": w.graph.n_edges, "design_points_per_gpu": int(w.params.shape[0]), "full_trace": True,
            "issue_policy": args.policy, "subpartitions": 0 if args.policy == "lowest_id" else args.subpartitions,
            "l2": "inputs+outputs larger than L2 (trace rows alone exceed it)",
            "parallelism": f"design points sharded over {world} GPU(s)"}


def spread_points(params, k, offset=0):
    """``k`` point indices spread evenly over the simulated-SM-count axis (the
    axis that sets a point's cost), starting ``offset`` points into that order,
    so successive samples take different points."""
    from paper_2607_11262_gb300 import workloads as W
    P = int(params.shape[0])
    k = max(1, min(int(k), P))
    order = np.argsort(params[:, W.P_NUM_SMS], kind="stable")
    stride = P / k
    return sorted({int(order[(int(j * stride) + offset) % P]) for j in range(k)})


def cpu_baseline(graph, params, seconds=15.0, procs=None):
    """The oracle, as it stands, on the host cores over a bounded sample of the
    workload's points spread over the SM-count axis (spawned worker processes,
    one point per process at a time)."""
    from oracle import run as oracle_run
    procs = procs or (os.cpu_count() or 1)
    probe = spread_points(params, 1, offset=params.shape[0] // 2)[0]
    t0 = time.time()
    oracle_run.simulate(graph, params[probe])   # one median-cost point to size the sample
    t_one = time.time() - t0
    k = int(max(1, min(params.shape[0], procs * max(1, round(seconds / max(t_one, 1e-3))))))
    k = max(1, min(k, procs * 4))
    pts = spread_points(params, k)
    pool = oracle_run.PointPool(graph, min(procs, len(pts)))
    wall, reps = 0.0, 0
    while reps == 0 or wall < seconds / 3:  # a small workload is repeated until the clock means something
        t0 = time.time()
        res = pool.run(params, pts)
        wall += time.time() - t0
        reps += 1
        assert all(r.status == 0 for r in res.values())
    pool.close()
    nodes = node_points_of(graph, params[pts]) * reps
    return {"value": nodes / wall, "unit": UNIT, "cores": min(procs, len(pts)), "kind": "oracle",
            "sample": f"{len(pts)} of {params.shape[0]} design points spread over the SM-count axis"
                      + (f", {reps} times" if reps > 1 else "") + f", {min(procs, len(pts))} processes, {wall:.1f} s wall"}


def run_reference(args):
    """The oracle as the reference arm: every step simulates a bounded sample
    of the workload's points (one per host core, a different part of the
    SM-count axis each step) and is timed as it runs; the rate is node-points
    of the samples over their wall time."""
    from oracle import run as oracle_run
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    w = load_workload(args.workload, 0, args.points, args.policy, args.subpartitions)
    g = w.graph
    P = int(w.params.shape[0])
    procs = os.cpu_count() or 1
    per_step = max(1, min(P, procs * args.ref_points_per_core))
    pool = oracle_run.PointPool(g, min(procs, per_step))
    wall, nodes, samples = [], [], []
    for i in range(args.warmup + args.steps):
        pts = spread_points(w.params, per_step, offset=i * max(1, P // (per_step * (args.warmup + args.steps))))
        t0 = time.perf_counter()
        res = pool.run(w.params, pts)
        dt = time.perf_counter() - t0
        assert all(r.status == 0 for r in res.values())
        if i >= args.warmup:
            wall.append(dt)
            nodes.append(node_points_of(g, w.params[pts]))
            samples.append(len(pts))
    pool.close()
    v = float(sum(nodes) / sum(wall))
    ms_per_step = float(np.mean(wall)) * 1e3
    cores = min(procs, per_step)
    line = {"metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": workload_config(w, args, ws),
            "impl": "reference",
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"{per_step} of {P} design points per step (a different part of the "
                                       f"SM-count axis each step), {cores} processes"},
            "step_sample_points": per_step,
            "full_sweep_ms_extrapolated": node_points_of(g, w.params) / v * 1e3,
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gts", choices=["gts", "reference"])
    ap.add_argument("--workload", default="wsgemm8192")
    ap.add_argument("--points", type=int, default=None)
    ap.add_argument("--policy", default="lowest_id", choices=sorted(POLICIES))
    ap.add_argument("--subpartitions", type=int, default=4)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end leg (e2e is then null)")
    ap.add_argument("--ref-seconds", type=float, default=15.0)
    ap.add_argument("--ref-points-per-core", type=int, default=1)
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)

    import torch
    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    from paper_2607_11262_gb300 import gts
    gts.load()

    w = load_workload(args.workload, rank, args.points, args.policy, args.subpartitions, world=ws)
    g = w.graph
    P = int(w.params.shape[0])
    node_points = node_points_of(g, w.params)
    flags = gts.GTS_FULL_TRACE | gts.GTS_SCRATCH_CLEAN
    stream = torch.cuda.Stream()

    with torch.cuda.stream(stream):
        dg = gts.DeviceGraph(g, stream=stream)
        dp = gts.DeviceParams(dg, w.params, stream=stream)
        out = gts.alloc_outputs(dg, P, flags)
        scratch = gts.alloc_scratch(dg, dp, flags, stream=stream)  # zero-filled once; every batch leaves it so
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]

    def barrier():
        if ws > 1:
            torch.distributed.barrier()

    for _ in range(args.warmup):
        gts.simulate(dg, dp, flags=flags, out=out, scratch=scratch, stream=stream)
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    clocks = Clocks(local)
    clocks.start()
    for i in range(args.steps):
        ev[i][0].record(stream)
        gts.simulate(dg, dp, flags=flags, out=out, scratch=scratch, stream=stream)
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    ck = clocks.stop()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = float(sum(step_ms))
    total_ms = reduce_max_over_ranks(total_ms, device="cuda")
    # the only exchange: per-point makespans and statuses to rank 0
    gathered = gather_to_rank0([out.makespan, out.status], device="cuda")
    if rank == 0:
        mk_all, st_all = gathered
        assert np.all(st_all == 0), f"non-OK statuses: {np.unique(st_all)}"
    ms_per_step = total_ms / args.steps
    value = whole_job_rate(node_points, ws, ms_per_step)

    # ---- e2e: host buffers through the C ABI, copies inside the timed region
    e2e = None
    if (rank == 0 or ws > 1) and not args.no_e2e:
        from paper_2607_11262_gb300 import workloads as W
        templates = W.workload(args.workload, templated=True).graph if args.workload in W.TEMPLATED else None
        e2e = measure_e2e(g, w.params, gts, stream, templates=templates)

    if rank != 0:
        if ws > 1:
            torch.distributed.destroy_process_group()
        return
    alg = algorithmic_bytes(g, w.params)
    kernel_s = ms_per_step / 1e3
    peaks = json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json"))) if os.path.exists(
        os.path.join(ROOT, "MEASURED_PEAKS.json")) else {}
    peak = float(peaks.get("hbm_gbs", 6800.0))
    achieved = alg / kernel_s / 1e9
    traffic = None
    tf = profiled(TRAFFIC_FILE, w.name)
    if tf:
        traffic = tf["bytes_per_node_point"] * node_points + tf.get("bytes_fixed", 0)
    # issue-slot roofline: warp-instructions per node (ncu) x node rate against
    # SMs x schedulers x the SM clock seen during the timed steps
    issue = None
    fi = profiled(ISSUE_FILE, w.name)
    if fi and ck and ck.get("sm_mhz"):
        sms = torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count
        got = fi["warp_instr_per_node_point"] * node_points / kernel_s
        cap = sms * SCHEDULERS_PER_SM * ck["sm_mhz"] * 1e6
        issue = {"achieved": got / 1e9, "peak": cap / 1e9, "unit": "Gwarp-instr/s", "frac": got / cap,
                 "warp_instr_per_node": fi["warp_instr_per_node_point"],
                 "peak_basis": f"{sms} SMs x {SCHEDULERS_PER_SM} schedulers x {ck['sm_mhz']:.0f} MHz"}
    cb = None
    if not args.no_cpu_baseline:
        cb = cpu_baseline(g, w.params, seconds=args.ref_seconds)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "int32", "data": "synthetic",
        "config": workload_config(w, args, ws),
        "design_points_per_s": P * ws / kernel_s,
        "hbm_gbs_algorithmic": achieved,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "peak_source": "measured" if peaks else "fallback",
                     "frac_of_8tbps": achieved / 8000.0, "issue": issue},
        "cpu_baseline": cb, "e2e": e2e, "gpu_launches": args.steps, "clocks": ck,
        "kernel_source": source_hash(),
        "gathered": {"points": int(st_all.shape[0]), "ok": int((st_all == 0).sum()),
                     "makespan_max": int(mk_all.max()) if mk_all.size else 0},
    }
    print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def measure_e2e(graph, params, gts, stream, reps=2, templates=None, chunk_bytes=1 << 30, copy_streams=4):
    """Same metric through the public API from pinned host buffers, every step:
    graph and parameter upload (host->device), graph packing, the batch, and
    the device->host read of the whole result -- the start/finish trace of
    every point, then the makespans and statuses.  The trace crosses the link
    in chunks of rows, spread over ``copy_streams`` streams that each reuse one
    pinned buffer of ``chunk_bytes`` (a consumer would write each chunk out or
    reduce it as it arrives; 52 GB of trace per wsgemm8192 step is not kept in
    host memory).  With ``templates``
    (the same graph as a TemplateSet) the graph goes in template-shared form:
    templates and the CTA table are uploaded and libgts expands them."""
    import torch
    P = int(params.shape[0])
    node_points = node_points_of(graph, params)
    src = templates if templates is not None else graph
    keys = gts.DeviceGraph.TEMPLATE_FIELDS if templates is not None else gts.DeviceGraph.FIELDS

    def pinned(a):
        a = np.ascontiguousarray(a)
        a = a.view(np.int32 if a.dtype == np.uint32 else (np.int16 if a.dtype == np.uint16 else a.dtype))
        return torch.from_numpy(a).pin_memory()
    host = {k: pinned(getattr(src, k)) for k in keys}
    hp = torch.from_numpy(np.ascontiguousarray(params, np.int32).reshape(-1)).pin_memory()
    h_mk = torch.empty(P, dtype=torch.int32).pin_memory()
    h_st = torch.empty(P, dtype=torch.int32).pin_memory()
    ring = [torch.empty(chunk_bytes // 4, dtype=torch.int32).pin_memory() for _ in range(copy_streams)]
    copiers = [torch.cuda.Stream() for _ in range(copy_streams)]
    # inputs, plus the processing order libgts uploads (4 B per point, gts_params_set_order)
    h2d = sum(t.numel() * t.element_size() for t in host.values()) + hp.numel() * 4 + 4 * P
    flags = gts.GTS_FULL_TRACE | gts.GTS_SCRATCH_CLEAN
    times, d2h = [], 0
    dev = torch.device("cuda")
    for _ in range(reps):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        with torch.cuda.stream(stream):
            dt = {k: v.to(dev, non_blocking=True) for k, v in host.items()}
            dpar = hp.to(dev, non_blocking=True)
            dg = gts.DeviceGraph.from_device_tensors(src, dt, stream=stream)
            dpp = gts.DeviceParams.from_device_tensor(dg, dpar, P, stream=stream)
            out = gts.alloc_outputs(dg, P, flags)
            scratch = gts.alloc_scratch(dg, dpp, flags, stream=stream)
            gts.simulate(dg, dpp, flags=flags, out=out, scratch=scratch, stream=stream)
            done = torch.cuda.Event()
            done.record(stream)
            rows = max(1, (chunk_bytes // 4) // max(dg.row_nodes, 1))
            d2h, k = 0, 0
            for cs in copiers:
                cs.wait_event(done)
            for trace in (out.start, out.finish):
                for r0 in range(0, P, rows):
                    part = trace[r0:r0 + rows].reshape(-1)
                    with torch.cuda.stream(copiers[k]):
                        ring[k][:part.numel()].copy_(part, non_blocking=True)
                    d2h += part.numel() * 4
                    k = (k + 1) % copy_streams
            for cs in copiers:
                stream.wait_stream(cs)
            h_mk.copy_(out.makespan, non_blocking=True)
            h_st.copy_(out.status, non_blocking=True)
            d2h += 8 * P
        stream.synchronize()
        times.append(time.perf_counter() - t0)
        assert bool((h_st == 0).all()), "non-OK statuses in the end-to-end run"
        del out, dpp, dg, dt, dpar, scratch
    t = min(times)
    return {"value": node_points / t, "unit": UNIT, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "seconds_per_step": t, "graph_input": "template-shared" if templates is not None else "logical",
            "trace_to_host": f"start and finish rows in {2 * ((P + rows - 1) // rows)} chunks over {copy_streams} "
                             f"copy streams, each into its own {chunk_bytes >> 20} MiB pinned buffer"}


if __name__ == "__main__":
    main()
