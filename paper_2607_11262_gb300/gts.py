"""Python binding of libgts (argument marshalling only).

Functions named like the C ABI in include/gts.h take plain integers (device
pointers, sizes, stream handles) and return handles or raise ``GtsError``.
``DeviceGraph`` / ``DeviceParams`` / ``simulate`` add torch-owned device
buffers around them: torch supplies device memory and streams, every step of
the simulation runs in libgts's CUDA kernels.  There is no CPU fallback: if
libgts is not built, importing works but every call raises.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libgts.so")

GTS_OK = 0
GTS_ERR_INVALID_ARG = -1
GTS_ERR_INVALID_GRAPH = -2
GTS_ERR_INVALID_PARAMS = -3
GTS_ERR_CUDA = -4
GTS_ERR_NOMEM = -5
GTS_ERR_OVERFLOW = -6
GTS_ERR_STEP_LIMIT = -7
GTS_ERR_DEADLOCK = -8
GTS_ERR_UNSUPPORTED = -9

GTS_FULL_TRACE = 1
GTS_WANT_DIGEST = 2
GTS_WANT_CTA_SM = 4
GTS_WANT_BUSY = 8
GTS_SCRATCH_CLEAN = 16

GTS_BUSY_CLASSES = 9
(GTS_BUSY_TENSOR, GTS_BUSY_TMA, GTS_BUSY_LSU, GTS_BUSY_ALU, GTS_BUSY_BAR, GTS_BUSY_HBM, GTS_BUSY_NOC,
 GTS_BUSY_L2_HITS, GTS_BUSY_L2_LOADS) = range(9)
BUSY_NAMES = ("tensor", "tma", "lsu", "alu", "bar", "hbm", "noc", "l2_hits", "l2_loads")

GTS_NPARAM = 32
GTS_POLICY_LOWEST_ID, GTS_POLICY_GTO, GTS_POLICY_RR = 0, 1, 2

GTS_STATIC_SCRATCH_BYTES = 32 << 20
GTS_SCRATCH_HEADER_BYTES = 16

EXPORTS = ("gts_graph_workspace_bytes", "gts_graph_create", "gts_graph_destroy", "gts_template_workspace_bytes",
           "gts_graph_create_templated", "gts_params_upload", "gts_params_set_order",
           "gts_params_destroy", "gts_row_nodes", "gts_row_ctas", "gts_scratch_bytes", "gts_simulate_batch",
           "gts_read_results", "gts_results_destroy", "gts_simulate_batch_noalloc", "gts_last_error")


class GtsError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"libgts status {status}: {msg}")
        self.status = status


class GraphDesc(ctypes.Structure):
    _fields_ = [("n_nodes", ctypes.c_uint32), ("n_edges", ctypes.c_uint32), ("n_ctas", ctypes.c_uint32),
                ("warps_per_cta", ctypes.c_uint32), ("n_graphs", ctypes.c_uint32),
                ("graph_node_off", ctypes.c_void_p), ("graph_cta_off", ctypes.c_void_p),
                ("row_ptr", ctypes.c_void_p), ("col", ctypes.c_void_p), ("ekind", ctypes.c_void_p),
                ("type", ctypes.c_void_p), ("warp", ctypes.c_void_p), ("cta", ctypes.c_void_p),
                ("work", ctypes.c_void_p), ("lat_extra", ctypes.c_void_p), ("cta_kernel", ctypes.c_void_p),
                ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t),
                ("tile", ctypes.c_void_p), ("n_tiles", ctypes.c_uint32)]


class TemplateDesc(ctypes.Structure):
    _fields_ = [("n_templates", ctypes.c_uint32), ("n_tpl_nodes", ctypes.c_uint32), ("n_tpl_edges", ctypes.c_uint32),
                ("n_nodes", ctypes.c_uint32), ("n_edges", ctypes.c_uint32), ("n_ctas", ctypes.c_uint32),
                ("warps_per_cta", ctypes.c_uint32), ("n_graphs", ctypes.c_uint32),
                ("graph_cta_off", ctypes.c_void_p), ("tpl_node_off", ctypes.c_void_p), ("tpl_row_ptr", ctypes.c_void_p),
                ("tpl_col", ctypes.c_void_p), ("tpl_ekind", ctypes.c_void_p), ("tpl_type", ctypes.c_void_p),
                ("tpl_warp", ctypes.c_void_p), ("tpl_work", ctypes.c_void_p), ("tpl_lat_extra", ctypes.c_void_p),
                ("cta_template", ctypes.c_void_p), ("cta_kernel", ctypes.c_void_p),
                ("workspace", ctypes.c_void_p), ("workspace_bytes", ctypes.c_size_t)]


_lib = None


def load():
    """The loaded libgts (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"libgts is not built ({LIB_PATH}); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    vp, u32, i32, sz = ctypes.c_void_p, ctypes.c_uint32, ctypes.c_int32, ctypes.c_size_t
    pp = ctypes.POINTER(ctypes.c_void_p)
    lib.gts_graph_workspace_bytes.argtypes = [u32, u32, u32, u32, u32]
    lib.gts_graph_workspace_bytes.restype = sz
    lib.gts_graph_create.argtypes = [ctypes.POINTER(GraphDesc), vp, pp]
    lib.gts_graph_create.restype = i32
    lib.gts_graph_destroy.argtypes = [vp]
    lib.gts_graph_destroy.restype = i32
    lib.gts_template_workspace_bytes.argtypes = [u32, u32, u32, u32, u32, u32, u32]
    lib.gts_template_workspace_bytes.restype = sz
    lib.gts_graph_create_templated.argtypes = [ctypes.POINTER(TemplateDesc), vp, pp]
    lib.gts_graph_create_templated.restype = i32
    lib.gts_params_upload.argtypes = [vp, vp, u32, vp, pp]
    lib.gts_params_upload.restype = i32
    lib.gts_params_destroy.argtypes = [vp]
    lib.gts_params_destroy.restype = i32
    lib.gts_params_set_order.argtypes = [vp, vp, vp]
    lib.gts_params_set_order.restype = i32
    lib.gts_row_nodes.argtypes = [vp]
    lib.gts_row_nodes.restype = u32
    lib.gts_row_ctas.argtypes = [vp]
    lib.gts_row_ctas.restype = u32
    lib.gts_scratch_bytes.argtypes = [vp, vp, u32]
    lib.gts_scratch_bytes.restype = sz
    lib.gts_simulate_batch.argtypes = [vp, vp, u32, u32, u32, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp, pp]
    lib.gts_simulate_batch.restype = i32
    lib.gts_read_results.argtypes = [vp, vp, vp, vp, u32]
    lib.gts_read_results.restype = i32
    lib.gts_results_destroy.argtypes = [vp]
    lib.gts_results_destroy.restype = i32
    lib.gts_simulate_batch_noalloc.argtypes = [vp, vp, u32, u32, u32, vp, vp, vp, vp, vp, vp, vp, vp]
    lib.gts_simulate_batch_noalloc.restype = i32
    lib.gts_last_error.argtypes = []
    lib.gts_last_error.restype = ctypes.c_char_p
    _lib = lib
    return lib


def _check(status):
    if status != GTS_OK:
        raise GtsError(status, load().gts_last_error().decode())


# ---------------------------------------------------------------- raw ABI (same names)
def gts_graph_workspace_bytes(n_nodes, n_edges, n_ctas, warps_per_cta, n_graphs):
    return int(load().gts_graph_workspace_bytes(n_nodes, n_edges, n_ctas, warps_per_cta, n_graphs))


def gts_graph_create(desc: GraphDesc, stream: int = 0):
    h = ctypes.c_void_p()
    _check(load().gts_graph_create(ctypes.byref(desc), stream, ctypes.byref(h)))
    return h.value


def gts_graph_destroy(graph):
    _check(load().gts_graph_destroy(graph))


def gts_template_workspace_bytes(n_templates, n_tpl_nodes, n_nodes, n_edges, n_ctas, warps_per_cta, n_graphs):
    return int(load().gts_template_workspace_bytes(n_templates, n_tpl_nodes, n_nodes, n_edges, n_ctas,
                                                   warps_per_cta, n_graphs))


def gts_graph_create_templated(desc: TemplateDesc, stream: int = 0):
    h = ctypes.c_void_p()
    _check(load().gts_graph_create_templated(ctypes.byref(desc), stream, ctypes.byref(h)))
    return h.value


def gts_params_upload(graph, d_params: int, n_points: int, stream: int = 0):
    h = ctypes.c_void_p()
    _check(load().gts_params_upload(graph, d_params, n_points, stream, ctypes.byref(h)))
    return h.value


def gts_params_destroy(params):
    _check(load().gts_params_destroy(params))


def gts_params_set_order(params, d_order: int, stream: int = 0):
    _check(load().gts_params_set_order(params, d_order, stream))


def gts_row_nodes(graph):
    return int(load().gts_row_nodes(graph))


def gts_row_ctas(graph):
    return int(load().gts_row_ctas(graph))


def gts_scratch_bytes(graph, params, flags):
    return int(load().gts_scratch_bytes(graph, params, flags))


def gts_simulate_batch(graph, params, first_point, n_points, flags, d_start, d_finish, d_makespan, d_status,
                       d_digest, d_cta_sm, d_busy, d_scratch, scratch_bytes, stream=0, want_handle=False):
    h = ctypes.c_void_p()
    _check(load().gts_simulate_batch(graph, params, first_point, n_points, flags, d_start, d_finish, d_makespan,
                                     d_status, d_digest, d_cta_sm, d_busy, d_scratch, scratch_bytes, stream,
                                     ctypes.byref(h) if want_handle else None))
    return h.value if want_handle else None


def gts_read_results(results, h_makespan, h_status, h_digest, n_points):
    _check(load().gts_read_results(results, h_makespan, h_status, h_digest, n_points))


def gts_results_destroy(results):
    _check(load().gts_results_destroy(results))


def gts_simulate_batch_noalloc(graph, params, first_point, n_points, flags, d_start, d_finish, d_makespan,
                               d_status, d_digest, d_cta_sm, d_busy, stream=0):
    """gts_simulate_batch without caller scratch: libgts uses its own fixed
    device array (GTS_STATIC_SCRATCH_BYTES) and allocates nothing."""
    _check(load().gts_simulate_batch_noalloc(graph, params, first_point, n_points, flags, d_start, d_finish,
                                             d_makespan, d_status, d_digest, d_cta_sm, d_busy, stream))


def gts_last_error():
    return load().gts_last_error().decode()


# ---------------------------------------------------------------- torch-owned buffers
class _null:
    def __enter__(self):
        return None

    def __exit__(self, *a):
        return False


def _stream_handle(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def _to_device(a, dev):
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    elif a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).to(dev)


class DeviceGraph:
    """A workloads.Graph (or a template-shared workloads.TemplateSet) resident on
    the GPU, validated and packed by libgts."""

    FIELDS = ("row_ptr", "col", "ekind", "type", "warp", "cta", "work", "lat_extra", "cta_kernel",
              "node_off", "cta_off")
    TEMPLATE_FIELDS = ("tpl_node_off", "row_ptr", "col", "ekind", "type", "warp", "work", "lat_extra",
                       "cta_template", "cta_kernel", "graph_cta_off")

    def __init__(self, graph, device="cuda", stream=None, tensors=None):
        """``tensors`` (optional): the graph's arrays already on the device,
        keyed like FIELDS (uint32 arrays as int32, uint16 as int16)."""
        import torch
        self.graph = graph
        dev = torch.device(device)
        if hasattr(graph, "tpl_node_off"):
            self._create_templated(graph, dev, stream, tensors)
            return

        def t(a):
            return _to_device(a, dev)
        if tensors is None:
            tensors = {k: t(getattr(graph, k)) for k in self.FIELDS}
            if getattr(graph, "tile", None) is not None:
                tensors["tile"] = t(graph.tile)
        else:
            dev = next(iter(tensors.values())).device
        self.tensors = tensors
        n, m, C, W, G = graph.n_nodes, graph.n_edges, graph.n_ctas, graph.warps_per_cta, graph.n_graphs
        nbytes = gts_graph_workspace_bytes(n, m, C, W, G)
        if nbytes == 0:
            raise GtsError(GTS_ERR_INVALID_ARG, "graph size out of range")
        with torch.cuda.stream(stream) if stream is not None else _null():
            self.workspace = torch.zeros(nbytes, dtype=torch.uint8, device=dev)  # padding included
        T = self.tensors
        d = GraphDesc(n, m, C, W, G, T["node_off"].data_ptr(), T["cta_off"].data_ptr(), T["row_ptr"].data_ptr(),
                      T["col"].data_ptr(), T["ekind"].data_ptr(), T["type"].data_ptr(), T["warp"].data_ptr(),
                      T["cta"].data_ptr(), T["work"].data_ptr(), T["lat_extra"].data_ptr(),
                      T["cta_kernel"].data_ptr(), self.workspace.data_ptr(), nbytes,
                      T["tile"].data_ptr() if "tile" in T else None, int(getattr(graph, "n_tiles", 0) or 0))
        self.desc = d
        self.handle = gts_graph_create(d, _stream_handle(stream))
        self.row_nodes = gts_row_nodes(self.handle)
        self.row_ctas = gts_row_ctas(self.handle)

    def _create_templated(self, ts, dev, stream, tensors=None):
        import torch
        if tensors is None:
            tensors = {k: _to_device(getattr(ts, k), dev) for k in self.TEMPLATE_FIELDS}
        else:
            dev = next(iter(tensors.values())).device
        self.tensors = T = tensors
        TN, TE = int(ts.tpl_node_off[-1]), int(ts.col.shape[0])
        # logical totals; an out-of-range template index is left for libgts to refuse
        nsz, esz = ts.sizes()
        ct = np.minimum(ts.cta_template.astype(np.int64), max(ts.n_templates - 1, 0))
        n, m = (int(nsz[ct].sum()), int(esz[ct].sum())) if ts.n_templates else (0, 0)
        C, W, G = ts.n_ctas, ts.warps_per_cta, ts.n_graphs
        nbytes = gts_template_workspace_bytes(ts.n_templates, TN, n, m, C, W, G)
        if nbytes == 0:
            raise GtsError(GTS_ERR_INVALID_ARG, "template set size out of range")
        with torch.cuda.stream(stream) if stream is not None else _null():
            self.workspace = torch.zeros(nbytes, dtype=torch.uint8, device=dev)  # padding included
        d = TemplateDesc(ts.n_templates, TN, TE, n, m, C, W, G, T["graph_cta_off"].data_ptr(),
                         T["tpl_node_off"].data_ptr(), T["row_ptr"].data_ptr(), T["col"].data_ptr(),
                         T["ekind"].data_ptr(), T["type"].data_ptr(), T["warp"].data_ptr(), T["work"].data_ptr(),
                         T["lat_extra"].data_ptr(), T["cta_template"].data_ptr(), T["cta_kernel"].data_ptr(),
                         self.workspace.data_ptr(), nbytes)
        self.desc = d
        self.handle = gts_graph_create_templated(d, _stream_handle(stream))
        self.row_nodes = gts_row_nodes(self.handle)
        self.row_ctas = gts_row_ctas(self.handle)

    @classmethod
    def from_device_tensors(cls, graph, tensors, stream=None):
        """``tensors`` keyed like FIELDS, or like TEMPLATE_FIELDS for a TemplateSet."""
        return cls(graph, stream=stream, tensors=tensors)

    def close(self):
        if getattr(self, "handle", None):
            gts_graph_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class DeviceParams:
    """A [P][GTS_NPARAM] int32 parameter table resident on the GPU."""

    def __init__(self, dgraph: DeviceGraph, params, stream=None, tensor=None, n_points=None, ordered=True):
        """``ordered``: hand points to the warps largest estimated cost first
        (gts_params_set_order); results are the same either way."""
        import torch
        self.dgraph = dgraph
        if tensor is None:
            p = np.ascontiguousarray(params, np.int32)
            if p.ndim != 2 or p.shape[1] != GTS_NPARAM:
                raise ValueError(f"params must be [n_points][{GTS_NPARAM}] int32, got {p.shape}")
            self.n_points = int(p.shape[0])
            self.tensor = torch.from_numpy(p.reshape(-1)).to(dgraph.workspace.device)
        else:
            self.n_points = int(n_points)
            self.tensor = tensor
        self.handle = gts_params_upload(dgraph.handle, self.tensor.data_ptr(), self.n_points, _stream_handle(stream))
        self.order = None
        if ordered and self.n_points:
            self.order = torch.empty(self.n_points, dtype=torch.int32, device=self.tensor.device)
            gts_params_set_order(self.handle, self.order.data_ptr(), _stream_handle(stream))

    @classmethod
    def from_device_tensor(cls, dgraph, tensor, n_points, stream=None, ordered=True):
        return cls(dgraph, None, stream=stream, tensor=tensor, n_points=n_points, ordered=ordered)

    def close(self):
        if getattr(self, "handle", None):
            gts_params_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


@dataclasses.dataclass
class BatchOutput:
    makespan: object
    status: object
    start: object = None
    finish: object = None
    digest: object = None
    cta_sm: object = None
    busy: object = None


def alloc_outputs(dgraph: DeviceGraph, n_points: int, flags: int):
    import torch
    dev = dgraph.workspace.device
    out = BatchOutput(makespan=torch.empty(n_points, dtype=torch.int32, device=dev),
                      status=torch.empty(n_points, dtype=torch.int32, device=dev))
    if flags & GTS_FULL_TRACE:
        out.start = torch.empty((n_points, dgraph.row_nodes), dtype=torch.int32, device=dev)
        out.finish = torch.empty((n_points, dgraph.row_nodes), dtype=torch.int32, device=dev)
    if flags & GTS_WANT_DIGEST:
        out.digest = torch.empty(n_points, dtype=torch.int64, device=dev)
    if flags & GTS_WANT_CTA_SM:
        out.cta_sm = torch.empty((n_points, dgraph.row_ctas), dtype=torch.int32, device=dev)
    if flags & GTS_WANT_BUSY:
        out.busy = torch.empty((n_points, GTS_BUSY_CLASSES), dtype=torch.int64, device=dev)
    return out


def _ptr(t):
    return 0 if t is None else t.data_ptr()


def alloc_scratch(dgraph: DeviceGraph, dparams: DeviceParams, flags=0, stream=None):
    """A zero-filled scratch of gts_scratch_bytes; pass it to ``simulate`` with
    GTS_SCRATCH_CLEAN in the flags, call after call (libgts leaves it clean)."""
    import torch
    nb = gts_scratch_bytes(dgraph.handle, dparams.handle, flags)
    with torch.cuda.stream(stream) if stream is not None else _null():
        return torch.zeros(max(nb, 16), dtype=torch.uint8, device=dgraph.workspace.device)


def simulate(dgraph: DeviceGraph, dparams: DeviceParams, first_point=0, n_points=None,
             flags=GTS_FULL_TRACE | GTS_WANT_DIGEST | GTS_WANT_CTA_SM, out: BatchOutput = None,
             scratch=None, stream=None) -> BatchOutput:
    """Enqueue one gts_simulate_batch on ``stream`` (default: torch's current)."""
    import torch
    if n_points is None:
        n_points = dparams.n_points - first_point
    if out is None:
        out = alloc_outputs(dgraph, n_points, flags)
    if scratch is None:  # zero-filled, so the kernel need not clear it (GTS_SCRATCH_CLEAN)
        nb = gts_scratch_bytes(dgraph.handle, dparams.handle, flags)
        scratch = torch.zeros(max(nb, 16), dtype=torch.uint8, device=dgraph.workspace.device)
        flags |= GTS_SCRATCH_CLEAN
    gts_simulate_batch(dgraph.handle, dparams.handle, first_point, n_points, flags, _ptr(out.start),
                       _ptr(out.finish), _ptr(out.makespan), _ptr(out.status), _ptr(out.digest),
                       _ptr(out.cta_sm), _ptr(out.busy), _ptr(scratch), 0 if scratch is None else scratch.numel(),
                       _stream_handle(stream))
    out.scratch = scratch
    return out


def utilisation(busy, makespan, params):
    """Reporting only: the engine's output is the busy server-cycles per class
    (GTS_WANT_BUSY, computed in libgts); this turns them into the ratio the
    paper reports (Section 7.1) for tables and plots, after the simulation.
    Per-class utilisation of each point from its busy server-cycles:
    busy_r / (servers_r * makespan), servers_r = cap_r * num_sms for the per-SM
    classes, cap_hbm for HBM and cap_noc * ceil(num_sms / cluster_sms) for the
    NoC; 0 where the makespan is 0 or the row has no NoC.  The two L2 entries
    are counts, not cycles: column GTS_BUSY_L2_HITS holds the hit rate (hits /
    loads naming a tile) and GTS_BUSY_L2_LOADS 0.  numpy in, numpy out
    ([n_points][GTS_BUSY_CLASSES] float64)."""
    import numpy as np
    busy = np.asarray(busy, np.float64)
    prm = np.asarray(params, np.int64)
    mk = np.asarray(makespan, np.float64)
    servers = np.empty((prm.shape[0], GTS_BUSY_CLASSES), np.float64)
    servers[:, :5] = prm[:, 13:18] * prm[:, 0:1]
    servers[:, 5] = prm[:, 18]
    groups = np.where(prm[:, 25] > 0, -(-prm[:, 0] // np.maximum(prm[:, 25], 1)), 0)
    servers[:, 6] = prm[:, 24] * groups
    den = servers[:, :7] * mk[:, None]
    out = np.zeros_like(busy)
    np.divide(busy[:, :7], den, out=out[:, :7], where=den > 0)
    np.divide(busy[:, 7], busy[:, 8], out=out[:, 7], where=busy[:, 8] > 0)
    return out
