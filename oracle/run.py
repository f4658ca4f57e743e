"""ctypes driver for the C oracle (TEST INFRASTRUCTURE ONLY).

``simulate`` runs one design point on one graph; ``simulate_points`` fans
points out over worker processes started with the ``spawn`` method.  Status
codes mirror the library's numeric values (0 ok, -2 invalid graph,
-3 invalid params, -5 no memory, -6 overflow, -8 deadlock).
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "gts_oracle.c")
BUILD_DIR = os.path.join(HERE, "_build")
LIB = os.path.join(BUILD_DIR, "liboracle.so")

OK, ERR_INVALID_ARG, ERR_INVALID_GRAPH, ERR_INVALID_PARAMS = 0, -1, -2, -3
ERR_NOMEM, ERR_OVERFLOW, ERR_DEADLOCK = -5, -6, -8

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C99, -O2) into oracle/_build/."""
    os.makedirs(BUILD_DIR, exist_ok=True)
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        tmp = LIB + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c99", "-Wall", "-shared", "-fPIC", "-o", tmp, SRC])
        os.replace(tmp, LIB)
    return LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            p = ctypes.c_void_p
            i64 = ctypes.c_int64
            lib.oracle_simulate.argtypes = [i64, i64, i64, i64] + [p] * 16 + [i64]
            lib.oracle_simulate.restype = ctypes.c_int
            _lib = lib
    return _lib


@dataclasses.dataclass
class Result:
    status: int
    makespan: int
    start: np.ndarray    # int64 [n]
    finish: np.ndarray   # int64 [n]
    cta_sm: np.ndarray   # int32 [C]
    busy: np.ndarray = None  # int64 [9]: busy server-cycles of TENSOR, TMA, LSU, ALU, BAR, HBM, NoC; L2 load hits,
    #                          loads naming a tile


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def simulate_arrays(row_ptr, col, ekind, type_, warp, cta, work, lat_extra, cta_kernel,
                    warps_per_cta, params, tile=None, n_tiles=0) -> Result:
    """One design point on one graph given as plain arrays (graph-local ids)."""
    lib = _load()
    a = dict(row_ptr=np.ascontiguousarray(row_ptr, np.uint32), col=np.ascontiguousarray(col, np.uint32),
             ekind=np.ascontiguousarray(ekind, np.uint8), type=np.ascontiguousarray(type_, np.uint8),
             warp=np.ascontiguousarray(warp, np.uint16), cta=np.ascontiguousarray(cta, np.uint32),
             work=np.ascontiguousarray(work, np.uint32), lat_extra=np.ascontiguousarray(lat_extra, np.uint32),
             cta_kernel=np.ascontiguousarray(cta_kernel, np.uint32))
    prm = np.ascontiguousarray(params, np.int32)
    assert prm.shape == (32,)
    tl = None if tile is None else np.ascontiguousarray(tile, np.uint32)
    n = a["type"].shape[0]
    m = a["col"].shape[0]
    C = a["cta_kernel"].shape[0]
    start = np.empty(max(n, 1), np.int64)
    finish = np.empty(max(n, 1), np.int64)
    cta_sm = np.empty(max(C, 1), np.int32)
    mk = ctypes.c_int64(0)
    busy = np.zeros(9, np.int64)
    st = lib.oracle_simulate(n, m, C, int(warps_per_cta), _ptr(a["row_ptr"]), _ptr(a["col"]), _ptr(a["ekind"]),
                             _ptr(a["type"]), _ptr(a["warp"]), _ptr(a["cta"]), _ptr(a["work"]),
                             _ptr(a["lat_extra"]), _ptr(a["cta_kernel"]), _ptr(prm), _ptr(start), _ptr(finish),
                             ctypes.byref(mk), _ptr(cta_sm), _ptr(busy), None if tl is None else _ptr(tl),
                             int(n_tiles))
    return Result(int(st), int(mk.value), start[:n], finish[:n], cta_sm[:C], busy)


def simulate(graph, params_row) -> Result:
    """One design point.  ``graph`` is a workloads.Graph (a stacked set is cut to
    the row's graph_index); returned ids are graph-local."""
    prm = np.asarray(params_row, np.int32)
    g = graph
    if graph.n_graphs > 1 or int(graph.node_off[0]) != 0:
        gi = int(prm[19])
        if not 0 <= gi < graph.n_graphs:
            return Result(ERR_INVALID_PARAMS, 0, np.zeros(0, np.int64), np.zeros(0, np.int64), np.zeros(0, np.int32))
        g = graph.subgraph(gi)
    return simulate_arrays(g.row_ptr, g.col, g.ekind, g.type, g.warp, g.cta, g.work, g.lat_extra,
                           g.cta_kernel, g.warps_per_cta, prm, g.tile, g.n_tiles)


# ------------------------------------------------------------ process pool
_pool_graph = None


def _pool_init(graph):
    global _pool_graph
    _pool_graph = graph
    _load()


def _pool_run(args):
    p, row = args
    r = simulate(_pool_graph, row)
    return p, r


def _pool_ready(_):
    return os.getpid()


class PointPool:
    """A started pool of oracle worker processes holding one graph.

    Start-up (spawning, shipping the graph, loading the library) happens in the
    constructor, so ``run`` times only the simulation of the points."""

    def __init__(self, graph, processes):
        import multiprocessing as mp
        self.processes = max(1, int(processes))
        self.pool = mp.get_context("spawn").Pool(self.processes, initializer=_pool_init, initargs=(graph,))
        self.pool.map(_pool_ready, range(self.processes * 2))

    def run(self, params, points):
        return dict(self.pool.imap_unordered(_pool_run, [(p, params[p]) for p in points]))

    def close(self):
        self.pool.close()
        self.pool.join()


def simulate_points(graph, params, points, processes=None):
    """Oracle results for the listed points, computed in ``processes`` worker
    processes (spawned, so the pool is safe to start after CUDA init)."""
    import multiprocessing as mp
    points = list(points)
    if processes is None:
        processes = min(len(points), os.cpu_count() or 1)
    if processes <= 1 or len(points) <= 1:
        return {p: simulate(graph, params[p]) for p in points}
    ctx = mp.get_context("spawn")
    with ctx.Pool(processes, initializer=_pool_init, initargs=(graph,)) as pool:
        out = dict(pool.imap_unordered(_pool_run, [(p, params[p]) for p in points]))
    return out
