"""Benchmark: batched tile-graph simulation throughput on GB300.

One step = one gts_simulate_batch over every design point of the workload
(full per-node start/finish trace), i.e. one pass of the whole hot path.
Default workload: the warp-specialised persistent GEMM 8192^3 tile graph
(1.58M nodes) x 4096 design points.  Prints ONE JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle on the host cores

Under torchrun (N > 1) every rank simulates its own 4096 design points (drawn
with a rank-specific seed) on its own GPU: no data-path collective; the
per-rank times are reduced with a max at the end.
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


def load_workload(name, rank, points, policy="lowest_id", subpartitions=4):
    from paper_2607_11262_gb300 import workloads as W
    w = W.workload(name)
    if rank > 0 and name == "pipelines":
        from paper_2607_11262_gb300 import pipelines
        w.params = pipelines.study_params(w.graph.n_graphs, 64, seed=W.SEED0 + 6 + 100 * rank)
    elif rank > 0 and name == "l2_gemm":
        from paper_2607_11262_gb300 import l2gemm
        w.params = l2gemm.study_params(w.graph.n_graphs, points_per_capacity=8, seed=W.SEED0 + 8 + 100 * rank)
    elif rank > 0 and name == "noc_fusion":
        from paper_2607_11262_gb300 import clusters
        w.params = clusters.study_params(clusters.study_cases(), points_per_graph=32, seed=W.SEED0 + 7 + 100 * rank)
    elif rank > 0 and name != "stress":
        # weak scaling: every rank gets its own design points of the same sweep
        axes = {"gemm512": [W.AX_SMS, W.AX_HBM, (W.P_MMA_LAT, 16, 64)],
                "wsgemm8192": [W.AX_SMS, W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE]}.get(
            name, [W.AX_SMS, W.AX_HBM, W.AX_TMA_LAT, W.AX_MMA_RATE, W.AX_ALU_RATE])
        cps = int(w.params[0, W.P_CTAS_PER_SM])
        w.params = W.sweep_params(W.SEED0 + 100 * rank + W.WORKLOADS.index(name) + 1, w.params.shape[0], axes, cps)
    if points is not None:
        w.params = w.params[:points]
    w.params = np.ascontiguousarray(w.params)
    w.params[:, W.P_ISSUE_POLICY] = POLICIES[policy]
    w.params[:, W.P_SUBPARTITIONS] = 0 if policy == "lowest_id" else subpartitions
    return w


def workload_config(w, args, world):
    """The ``config`` object both arms print for a workload."""
    return {"workload": w.name, "description": w.description, "nodes": w.graph.max_graph_nodes,
            "edges": w.graph.n_edges, "design_points_per_gpu": int(w.params.shape[0]), "full_trace": True,
            "issue_policy": args.policy, "subpartitions": 0 if args.policy == "lowest_id" else args.subpartitions,
            "l2": "inputs+outputs larger than L2 (trace rows alone exceed it)",
            "parallelism": f"design points sharded over {world} GPU(s)"}


def cpu_baseline(graph, params, seconds=15.0, procs=None):
    """The oracle, as it stands, on the host cores over a bounded sample of the
    workload's points (spawned worker processes, one point per process)."""
    from oracle import run as oracle_run
    procs = procs or (os.cpu_count() or 1)
    t0 = time.time()
    oracle_run.simulate(graph, params[0])       # one point to size the sample
    t_one = time.time() - t0
    k = int(max(1, min(params.shape[0], procs * max(1, round(seconds / max(t_one, 1e-3))))))
    k = max(1, min(k, procs * 4))
    pts = list(range(k))
    pool = oracle_run.PointPool(graph, min(procs, k))
    t0 = time.time()
    res = pool.run(params, pts)
    wall = time.time() - t0
    pool.close()
    assert all(r.status == 0 for r in res.values())
    nodes = node_points_of(graph, params[pts])
    return {"value": nodes / wall, "unit": UNIT, "cores": min(procs, k), "kind": "oracle",
            "sample": f"{k} of {params.shape[0]} design points, {min(procs, k)} processes, {wall:.1f} s wall"}


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    w = load_workload(args.workload, 0, args.points, args.policy, args.subpartitions)
    g = w.graph
    vals, times = [], []
    node_points = node_points_of(g, w.params)
    for i in range(args.warmup + args.steps):
        cb = cpu_baseline(g, w.params, seconds=args.ref_seconds)
        if i >= args.warmup:
            vals.append(cb["value"])
            times.append(cb)
    v = float(np.median(vals))
    line = {"metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": node_points / v * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": workload_config(w, args, ws),
            "impl": "reference", "cpu_baseline": dict(times[-1], value=v),
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
    ap.add_argument("--ref-seconds", type=float, default=15.0)
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

    w = load_workload(args.workload, rank, args.points, args.policy, args.subpartitions)
    g = w.graph
    P = int(w.params.shape[0])
    node_points = node_points_of(g, w.params)
    flags = gts.GTS_FULL_TRACE
    stream = torch.cuda.Stream()

    with torch.cuda.stream(stream):
        dg = gts.DeviceGraph(g, stream=stream)
        dp = gts.DeviceParams(dg, w.params, stream=stream)
        out = gts.alloc_outputs(dg, P, flags)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]

    def barrier():
        if ws > 1:
            torch.distributed.barrier()

    for _ in range(args.warmup):
        gts.simulate(dg, dp, flags=flags, out=out, stream=stream)
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    clocks = Clocks(local)
    clocks.start()
    for i in range(args.steps):
        ev[i][0].record(stream)
        gts.simulate(dg, dp, flags=flags, out=out, stream=stream)
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    barrier()
    torch.cuda.synchronize()
    ck = clocks.stop()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = float(sum(step_ms))
    st = out.status.cpu().numpy()
    assert np.all(st == 0), f"non-OK statuses: {np.unique(st)}"
    total_ms = reduce_max_over_ranks(total_ms, device="cuda")
    ms_per_step = total_ms / args.steps
    value = whole_job_rate(node_points, ws, ms_per_step)

    # ---- e2e: host buffers through the C ABI, copies inside the timed region
    e2e = None
    if rank == 0 or ws > 1:
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
    }
    print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def measure_e2e(graph, params, gts, stream, reps=2, templates=None):
    """Same metric through the public API from pinned host buffers: graph and
    parameter upload (host->device), graph packing, the batch, and the
    device->host read of the per-point makespans and statuses, every step.
    With ``templates`` (the same graph as a TemplateSet) the graph goes in
    template-shared form: templates and the CTA table are uploaded and libgts
    expands them on the device."""
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
    # inputs, plus the processing order libgts uploads (4 B per point, gts_params_set_order)
    h2d = sum(t.numel() * t.element_size() for t in host.values()) + hp.numel() * 4 + 4 * P
    d2h = P * 8
    flags = gts.GTS_FULL_TRACE
    times = []
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
            gts.simulate(dg, dpp, flags=flags, out=out, stream=stream)
            h_mk.copy_(out.makespan, non_blocking=True)
            h_st.copy_(out.status, non_blocking=True)
        stream.synchronize()
        times.append(time.perf_counter() - t0)
        del out, dpp, dg, dt, dpar
    t = min(times)
    return {"value": node_points / t, "unit": UNIT, "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "seconds_per_step": t, "graph_input": "template-shared" if templates is not None else "logical"}


if __name__ == "__main__":
    main()
