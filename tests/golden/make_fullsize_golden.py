"""Write the per-point golden results of the five full-size workloads.

Every design point of gemm512, wsgemm8192, fa_fwd, decoder and stress is run
through the CPU oracle (``oracle/``) in spawned worker processes.  For each
point the file stores the status, the makespan, the ABI digest of the
(start, finish) rows (``tests.gpu_helpers.digest``) and a digest of the CTA
placement and busy server-cycles (``tests.gpu_helpers.aux_digest``).  The
GPU test ``tests/test_gpu_fullsize.py`` compares every point of the same
batch, run in the launch configuration the benchmark times, against these.

Inputs come from the seeded generator only; the file records the generator's
fingerprint (graph and parameter-table SHA-256), so a changed generator makes
the GPU test fail instead of comparing against stale values.  Nothing here
touches the CUDA library.

    python tests/golden/make_fullsize_golden.py [--workers N] [name ...]

Each workload is written to ``tests/golden/fullsize_<name>.json`` as soon as it
is done.  About 40,000 core-seconds in all (wsgemm8192 ~18k, decoder ~13k,
fa_fwd ~9k, stress and gemm512 seconds).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import multiprocessing as mp
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from oracle import run as oracle_run  # noqa: E402
from paper_2607_11262_gb300 import workloads as W  # noqa: E402
from tests import gpu_helpers as H  # noqa: E402

HERE = os.path.dirname(os.path.abspath(__file__))
_graph = None


def _init(name):
    global _graph
    _graph = W.workload(name).graph
    oracle_run._load()


def _one(args):
    p, row = args
    r = oracle_run.simulate(_graph, row)
    if r.status != 0:
        return p, r.status, 0, 0, 0
    return p, r.status, r.makespan, H.digest(r.start, r.finish), H.aux_digest(r.cta_sm, r.busy)


def fingerprint(w) -> dict:
    return {"graph_sha256": w.graph.sha256(),
            "params_sha256": hashlib.sha256(np.ascontiguousarray(w.params, np.int32).tobytes()).hexdigest()}


def path_for(name: str) -> str:
    return os.path.join(HERE, f"fullsize_{name}.json")


def make(name: str, workers: int) -> None:
    t0 = time.time()
    w = W.workload(name)
    P = w.params.shape[0]
    # costliest first (the simulated SM count drives a point's cost), so the
    # pool's tail is short
    order = np.argsort(-w.params[:, W.P_NUM_SMS], kind="stable")
    status = np.zeros(P, np.int64)
    makespan = np.zeros(P, np.int64)
    dig = [0] * P
    aux = [0] * P
    with mp.get_context("spawn").Pool(workers, initializer=_init, initargs=(name,)) as pool:
        done = 0
        for p, st, mk, d, a in pool.imap_unordered(_one, [(int(p), w.params[p]) for p in order]):
            status[p], makespan[p], dig[p], aux[p] = st, mk, d, a
            done += 1
            if done % max(1, P // 16) == 0:
                print(f"{name}: {done}/{P} points, {time.time() - t0:.0f} s", flush=True)
    out = {
        "what": ("oracle results of every design point of the full-size workload; digest = ABI digest of the "
                 "(start, finish) rows, aux = digest of the CTA placement and busy server-cycles"),
        "written_by": "tests/golden/make_fullsize_golden.py (oracle only)",
        "workload": name,
        "points": P,
        "n_nodes": w.graph.n_nodes,
        **fingerprint(w),
        "status": status.tolist(),
        "makespan": makespan.tolist(),
        "digest": [f"{d:016x}" for d in dig],
        "aux": [f"{a:016x}" for a in aux],
        "oracle_seconds": round(time.time() - t0, 1),
        "workers": workers,
    }
    tmp = path_for(name) + ".tmp"
    with open(tmp, "w") as f:
        json.dump(out, f, separators=(",", ":"))
    os.replace(tmp, path_for(name))
    print(f"{name}: wrote {path_for(name)} in {time.time() - t0:.0f} s", flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workers", type=int, default=os.cpu_count() or 1)
    ap.add_argument("names", nargs="*", default=["stress", "gemm512", "fa_fwd", "decoder", "wsgemm8192"])
    a = ap.parse_args()
    for name in a.names:
        make(name, a.workers)


if __name__ == "__main__":
    main()
