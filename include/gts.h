/*
 * gts.h -- C ABI of libgts, a batched graph-driven tile-graph simulator for
 * sm_103a (GB300).
 *
 * The library computes what the graph-driven simulation backend of
 * GPU-Tile-Sim computes (Section 5): given a warp-centric tile graph
 * G = (V, E) (Section 4.1) and a hardware description, the start and finish
 * cycle of every node and the kernel makespan.  It does so for many
 * independent hardware/tiling design points in one launch, one design point
 * per warp.
 *
 * Semantics (Section 5.1 execution flow, Section 5.2 throughput models,
 * Section 5.3 runtime control), with the framework's fixed readings:
 *  - each logical warp issues its nodes in program order (ascending id);
 *  - a DATA edge u->v releases v when u completes, an ISSUE (order) edge when
 *    u issues, in the same cycle;
 *  - a node of type LOAD/STORE takes one TMA server of its SM and one of the
 *    global HBM servers, SMEM one LSU server, MMA one TENSOR server, EW one
 *    ALU server, BAR one BAR server, NOP none; each for its occupancy
 *    ceil(work / rate) cycles (BAR: 1 cycle); the node's latency is
 *    L = base(type) + lat_extra + max occupancy, and finish = start + L;
 *  - CTAs launch in ascending id, each on the lowest SM with a free slot,
 *    at the cycle a slot frees; a CTA retires when all its nodes completed;
 *    a CTA of kernel k launches only after every CTA of kernels < k retired;
 *  - at every cycle the scheduler issues, one at a time, the lowest node id
 *    among warp heads whose predecessors are released and whose units have a
 *    free server, launching CTAs first, until nothing changes; then it moves to
 *    the next event cycle.
 *  Cycles are int32; a finish above 2^31-1 is reported as GTS_ERR_OVERFLOW.
 *
 * Conventions:
 *  - Every pointer named d_* or held in gts_graph_desc is a DEVICE pointer on
 *    the current CUDA device, owned by the caller; h_* pointers are host
 *    pointers.  The library never allocates device memory: the caller supplies
 *    the graph workspace and the simulation scratch, sized by the *_bytes()
 *    queries.  Handles borrow the caller's buffers and must not outlive them.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *    Calls enqueue work on it and return without waiting, except
 *    gts_graph_create, gts_params_upload and gts_read_results, which wait for
 *    the stream.
 *  - Host-side errors are returned as a status; gts_last_error() then holds a
 *    message for the calling thread.  Per-design-point errors (bad parameter
 *    row, overflow, deadlock, step limit) are written to d_status[p]; the other
 *    points are still simulated.  No call throws, traps or spins without bound.
 */
#ifndef GTS_H
#define GTS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t gts_status;
#define GTS_OK                  0
#define GTS_ERR_INVALID_ARG    (-1)  /* null pointer, size out of range, bad flags */
#define GTS_ERR_INVALID_GRAPH  (-2)  /* graph breaks the contract below */
#define GTS_ERR_INVALID_PARAMS (-3)  /* parameter row: rate/cap/count < 1, latency < 0, bad graph index */
#define GTS_ERR_CUDA           (-4)  /* a CUDA runtime call failed */
#define GTS_ERR_NOMEM          (-5)  /* workspace or scratch smaller than required */
#define GTS_ERR_OVERFLOW       (-6)  /* some finish cycle exceeds 2^31-1 (per point) */
#define GTS_ERR_STEP_LIMIT     (-7)  /* per-point loop bound reached (never for valid input) */
#define GTS_ERR_DEADLOCK       (-8)  /* no event left while nodes remain (per point) */
#define GTS_ERR_UNSUPPORTED    (-9)  /* row needs more on-chip state than one warp may hold */

/* Node operation types (Section 4.1 operation descriptor). */
#define GTS_LOAD  0   /* global/TMA -> shared; work = bytes; TMA + HBM; base tma_lat + dram_lat */
#define GTS_SMEM  1   /* shared <-> registers; work = bytes; LSU; base smem_lat */
#define GTS_MMA   2   /* tensor-core MMA; work = FMAs; TENSOR; base mma_lat */
#define GTS_EW    3   /* elementwise / softmax / norm; work = ops; ALU; base alu_lat */
#define GTS_STORE 4   /* shared/registers -> global; work = bytes; TMA + HBM; base tma_lat */
#define GTS_BAR   5   /* mbarrier / named-barrier wait; BAR for 1 cycle; base bar_lat */
#define GTS_NOP   6   /* pure synchronisation point; no unit; base 0 */
#define GTS_DSMEM 7   /* remote shared-memory access inside an SM group (DSMEM, Section 5.2 "DSMEM / On-chip
                         NoC"); work = bytes; LSU on its own SM + one NoC server of its SM group;
                         base smem_lat + noc_lat */

/* Edge kinds (Section 4.1 data and order edges). */
#define GTS_EDGE_DATA  0  /* released when the producer completes */
#define GTS_EDGE_ISSUE 1  /* released when the producer issues */

/* Parameter row: GTS_NPARAM int32 per design point (Table "GPU configurations"
 * quantities in cycles and bytes/FMAs/ops per cycle). */
#define GTS_NPARAM 32
#define GTS_P_NUM_SMS      0
#define GTS_P_CTAS_PER_SM  1
#define GTS_P_HBM_BPC      2   /* global DRAM bytes per cycle (one HBM server) */
#define GTS_P_DRAM_LAT     3
#define GTS_P_TMA_BPC      4
#define GTS_P_TMA_LAT      5
#define GTS_P_SMEM_BPC     6
#define GTS_P_SMEM_LAT     7
#define GTS_P_MMA_FMA_PC   8
#define GTS_P_MMA_LAT      9
#define GTS_P_ALU_OPS_PC  10
#define GTS_P_ALU_LAT     11
#define GTS_P_BAR_LAT     12
#define GTS_P_CAP_TENSOR  13   /* servers per SM */
#define GTS_P_CAP_TMA     14
#define GTS_P_CAP_LSU     15
#define GTS_P_CAP_ALU     16
#define GTS_P_CAP_BAR     17
#define GTS_P_CAP_HBM     18   /* global HBM servers */
#define GTS_P_GRAPH_INDEX 19   /* which graph of a stacked set this point runs */
#define GTS_P_ISSUE_POLICY 20  /* GTS_POLICY_*, see below */
#define GTS_P_SUBPARTITIONS 21 /* issue schedulers per SM: 1..32 for GTO / RR, 0 for LOWEST_ID */
#define GTS_P_NOC_BPC      22  /* on-chip NoC bytes per cycle per NoC server */
#define GTS_P_NOC_LAT      23  /* NoC latency added to a DSMEM node's base */
#define GTS_P_CAP_NOC      24  /* NoC servers per SM group (1..32) */
#define GTS_P_CLUSTER_SMS  25  /* SMs per NoC group: SM s is in group s / cluster_sms (1..32) */
/* NoC fields 22..25 are all 0 (no NoC: a graph with DSMEM nodes is then GTS_ERR_INVALID_PARAMS
 * for that row) or noc_bpc >= 1, noc_lat >= 0, 1 <= cap_noc <= 32, 1 <= cluster_sms <= 32. */
#define GTS_P_L2_BYTES     26  /* L2 capacity in bytes; 0: no L2 model */
#define GTS_P_L2_LAT       27  /* L2 latency, cycles */
#define GTS_P_L2_BPC       28  /* L2 bytes per cycle per memory-side server */
/* L2 fields 26..28 are all 0, or l2_bytes >= 1, l2_lat >= 0, l2_bpc >= 1.
 * 29..31 reserved, must be 0.
 *
 * L2 model (Section 5.2: a fully associative LRU cache over tile-derived
 * accesses).  With l2_bytes > 0, every design point keeps an LRU list of the
 * tiles its LOAD and STORE nodes name (gts_graph_desc.tile), each entry sized
 * by the bytes of its latest access, updated in issue order; after an access
 * the least recently used tiles are dropped until the total is <= l2_bytes.
 *  - LOAD whose tile is resident (hit): base tma_lat + l2_lat, holds a
 *    memory-side server ceil(work / l2_bpc) cycles;
 *  - any other LOAD (miss, or no tile): base tma_lat + l2_lat + dram_lat,
 *    ceil(work / hbm_bpc) cycles;
 *  - STORE: timing as without L2; its tile becomes the most recent entry.
 * The memory-side servers are the cap_hbm servers ("HBM" below): hits and
 * misses share them.  Without the L2 model a LOAD has base tma_lat + dram_lat. */

/*
 * Issue policies (Section 5.3: ready nodes sit in per-subpartition queues
 * served by greedy-then-oldest or round-robin schedulers).
 *  GTS_POLICY_LOWEST_ID: one global order -- at each cycle, the lowest node id
 *    among issuable warp heads issues, one at a time, until none is left; no
 *    per-cycle issue limit.
 *  GTS_POLICY_GTO / GTS_POLICY_RR: every SM has `subpartitions` schedulers.
 *    The warp slot l = (CTA's slot on its SM) * warps_per_cta + warp belongs to
 *    scheduler l mod subpartitions.  A scheduler issues at most one node per
 *    cycle: among its issuable warp heads, the first in its order --
 *      GTO: the slot it issued from last (greedy) if issuable, else the oldest
 *           warp (lowest CTA id * warps_per_cta + warp);
 *      RR:  slots in cyclic order starting after the slot it issued from last
 *           (from slot 0 before its first issue).
 *    Within a cycle the schedulers' picks issue in ascending node id, one at a
 *    time, each followed by the state update, until no scheduler that has not
 *    issued in this cycle has an issuable head.
 */
#define GTS_POLICY_LOWEST_ID 0
#define GTS_POLICY_GTO       1
#define GTS_POLICY_RR        2

/* Flags of gts_simulate_batch. */
#define GTS_FULL_TRACE  1u  /* write d_start / d_finish [n_points][row_nodes] */
#define GTS_WANT_DIGEST 2u  /* write d_digest[n_points] */
#define GTS_WANT_CTA_SM 4u  /* write d_cta_sm [n_points][row_ctas] (-1: never launched) */
#define GTS_WANT_BUSY   8u  /* write d_busy [n_points][GTS_BUSY_CLASSES] */
#define GTS_SCRATCH_CLEAN 16u /* d_scratch past its header is all zero (see gts_scratch_bytes) */

/* Busy server-cycles per resource class (Section 5.2 throughput servers):
 * d_busy[q*GTS_BUSY_CLASSES + r] = sum over the point's nodes v that use class
 * r of occ_r(v), the cycles v holds one server of r.  Class r's utilisation
 * over the run (Section 7.1 reports it for the tensor cores) is
 * busy_r / (servers_r * makespan), with servers_r = cap_r * num_sms for the
 * per-SM classes, cap_hbm for HBM and cap_noc * ceil(num_sms / cluster_sms)
 * for the NoC. */
#define GTS_BUSY_CLASSES 9
#define GTS_BUSY_TENSOR  0
#define GTS_BUSY_TMA     1
#define GTS_BUSY_LSU     2
#define GTS_BUSY_ALU     3
#define GTS_BUSY_BAR     4
#define GTS_BUSY_HBM     5
#define GTS_BUSY_NOC     6
#define GTS_BUSY_L2_HITS 7   /* not cycles: LOAD nodes that hit in L2 (L2 model only) */
#define GTS_BUSY_L2_LOADS 8  /* not cycles: LOAD nodes that named a tile (L2 model only) */

typedef struct gts_graph gts_graph;
typedef struct gts_params gts_params;
typedef struct gts_results gts_results;

/*
 * A tile graph, or a stack of n_graphs independent tile graphs (Section 4.1).
 * Ids are global over the stack; graph g owns nodes graph_node_off[g] ..
 * graph_node_off[g+1]-1 and CTAs graph_cta_off[g] .. graph_cta_off[g+1]-1.
 * Contract (checked by gts_graph_create, else GTS_ERR_INVALID_GRAPH):
 *  - successors are CSR: row_ptr[0] = 0, row_ptr non-decreasing,
 *    row_ptr[n_nodes] = n_edges; col[e] is the successor, ekind[e] its kind;
 *  - every edge u->v has u < v and stays inside its graph (ids are a
 *    topological order);
 *  - type < 8, warp < warps_per_cta, cta inside the node's graph;
 *  - cta_kernel is non-decreasing within each graph.
 * The program order of each (cta, warp) stream is ascending id.
 * Limits: n_nodes < 2^31, n_ctas < 2^24, warps_per_cta <= 128, in-degree
 * < 2^24 (GTS_ERR_UNSUPPORTED beyond).
 */
typedef struct {
  uint32_t n_nodes, n_edges, n_ctas, warps_per_cta, n_graphs;
  const uint32_t *graph_node_off;   /* [n_graphs+1]; NULL allowed when n_graphs == 1 */
  const uint32_t *graph_cta_off;    /* [n_graphs+1]; NULL allowed when n_graphs == 1 */
  const uint32_t *row_ptr;          /* [n_nodes+1] */
  const uint32_t *col;              /* [n_edges] */
  const uint8_t  *ekind;            /* [n_edges] GTS_EDGE_* */
  const uint8_t  *type;             /* [n_nodes] GTS_LOAD.. */
  const uint16_t *warp;             /* [n_nodes] CTA-local logical warp */
  const uint32_t *cta;              /* [n_nodes] */
  const uint32_t *work;             /* [n_nodes] bytes / FMAs / ops */
  const uint32_t *lat_extra;        /* [n_nodes] extra latency, cycles */
  const uint32_t *cta_kernel;       /* [n_ctas] */
  void *workspace;                  /* device, 16-byte aligned, >= gts_graph_workspace_bytes(...) */
  size_t workspace_bytes;
  const uint32_t *tile;             /* [n_nodes] tile a LOAD/STORE reads or writes, < n_tiles, or
                                       0xFFFFFFFF (none); ignored on other types; NULL: no tiles */
  uint32_t n_tiles;                 /* tile ids of each graph of the stack are < n_tiles */
} gts_graph_desc;

/* Bytes of device workspace gts_graph_create needs for a graph of this size
 * (Section 4.1 tile graph: packed node records, successor lists, the first
 * node of every (CTA, warp) stream, nodes per CTA, and the check's status
 * words and per-CTA temporaries, zero once the call returns).  Returns 0 when
 * a size is out of range. */
size_t gts_graph_workspace_bytes(uint32_t n_nodes, uint32_t n_edges, uint32_t n_ctas,
                                 uint32_t warps_per_cta, uint32_t n_graphs);

/* Checks the graph contract and builds the derived device arrays into
 * desc->workspace (Section 4.1 graph, Section 5.1 per-TB streams), on the
 * device: the graph never leaves it.  The host reads the graph offsets, the
 * two ends of row_ptr and a few status words back; graphs whose CTAs
 * interleave over id spans longer than 32 x n_nodes in total also have their
 * CTA and warp arrays and node records copied through the host to link the
 * warp streams.  Waits for `stream`.  *out borrows desc->cta_kernel and
 * desc->workspace.
 * Errors: INVALID_ARG, INVALID_GRAPH (message names the check and the lowest
 * offending index), UNSUPPORTED (in-degree), NOMEM (workspace too small), CUDA. */
gts_status gts_graph_create(const gts_graph_desc *desc, void *stream, gts_graph **out);
/* Frees the host handle of a graph (Section 4.1); the workspace and the
 * arrays it borrowed stay the caller's. */
gts_status gts_graph_destroy(gts_graph *graph);

/*
 * Template-shared graphs (Section 6.4 "Graph construction": the CTAs of a
 * regular kernel run isomorphic tile graphs, so one physical CTA graph is
 * stored once and every logical CTA refers to it).  T templates hold
 * n_tpl_nodes nodes in total; template t owns nodes tpl_node_off[t] ..
 * tpl_node_off[t+1]-1, with successor lists in CSR (tpl_row_ptr, tpl_col as an
 * index into the same template's nodes, tpl_ekind).  Logical CTA c runs
 * template cta_template[c]; its nodes get the next block of logical ids in CTA
 * order (CTA-major), so node u of template t in CTA c has id
 *   base_c + (u - tpl_node_off[t]),  base_c = sum over c' < c of |template of c'|.
 * Edges stay inside a CTA.  Stacked sets: graph g owns CTAs graph_cta_off[g] ..
 * graph_cta_off[g+1]-1 and the nodes of those CTAs.  n_nodes / n_edges are the
 * logical totals (checked).  All arrays are DEVICE pointers owned by the caller.
 * Contract (else GTS_ERR_INVALID_GRAPH): template edges go forward inside their
 * template, type < 8, warp < warps_per_cta, ekind < 2, cta_template[c] < T,
 * cta_kernel non-decreasing within each graph.
 */
typedef struct {
  uint32_t n_templates, n_tpl_nodes, n_tpl_edges;
  uint32_t n_nodes, n_edges, n_ctas, warps_per_cta, n_graphs;
  const uint32_t *graph_cta_off;   /* [n_graphs+1]; NULL allowed when n_graphs == 1 */
  const uint32_t *tpl_node_off;    /* [n_templates+1] */
  const uint32_t *tpl_row_ptr;     /* [n_tpl_nodes+1] */
  const uint32_t *tpl_col;         /* [n_tpl_edges] */
  const uint8_t  *tpl_ekind;       /* [n_tpl_edges] GTS_EDGE_* */
  const uint8_t  *tpl_type;        /* [n_tpl_nodes] */
  const uint16_t *tpl_warp;        /* [n_tpl_nodes] */
  const uint32_t *tpl_work;        /* [n_tpl_nodes] */
  const uint32_t *tpl_lat_extra;   /* [n_tpl_nodes] */
  const uint32_t *cta_template;    /* [n_ctas] */
  const uint32_t *cta_kernel;      /* [n_ctas] */
  void *workspace;                 /* device, 16-byte aligned, >= gts_template_workspace_bytes(...) */
  size_t workspace_bytes;
} gts_template_desc;

/* Device workspace of gts_graph_create_templated: the packed logical graph
 * (as gts_graph_workspace_bytes) plus the expansion tables.  0 when a size is
 * out of range. */
size_t gts_template_workspace_bytes(uint32_t n_templates, uint32_t n_tpl_nodes, uint32_t n_nodes, uint32_t n_edges,
                                    uint32_t n_ctas, uint32_t warps_per_cta, uint32_t n_graphs);

/* Checks the templates and the CTA table on the host (they are copied there;
 * the logical graph never is), then expands the logical graph on the device
 * into desc->workspace, in the same packed form gts_graph_create builds from
 * the expanded graph.  Waits for `stream`.  *out borrows desc->cta_kernel and
 * desc->workspace.  Errors: INVALID_ARG, INVALID_GRAPH, UNSUPPORTED (in-degree),
 * NOMEM (workspace), CUDA. */
gts_status gts_graph_create_templated(const gts_template_desc *desc, void *stream, gts_graph **out);

/* Registers a table of design points (one hardware description per point:
 * the Section 5.2 throughput and latency parameters, with the meanings and
 * H100 / A100 / B200 values of Section 6.1, Table "GPU configurations used in
 * evaluation"; fields listed above): d_params is [n_points][GTS_NPARAM]
 * int32 on the device, borrowed by *out.  Copies it to the host to size the
 * per-warp on-chip state of each row; waits for `stream`.  Rows that break the
 * parameter rules are not an error here: gts_simulate_batch reports them as
 * GTS_ERR_INVALID_PARAMS in d_status.  Errors: INVALID_ARG, CUDA. */
gts_status gts_params_upload(gts_graph *graph, const int32_t *d_params, uint32_t n_points,
                             void *stream, gts_params **out);
/* Frees the host handle of a parameter table; d_params stays the caller's. */
gts_status gts_params_destroy(gts_params *params);

/* Attaches a processing order to a parameter table.  The paper has no
 * counterpart: it orders the independent design points of a sweep (the
 * design-space use of Section 7) over the GPU's warps and changes no result.  Fills d_order (device,
 * [n_points] uint32, caller-owned, borrowed by params) with the point indices
 * sorted by estimated cost, largest first (nodes of the row's graph x (743 +
 * simulated SMs), x 3.5 for rows that need the extended model), and makes
 * gts_simulate_batch hand points to its warps in that order, each warp taking
 * the next point when it finishes one (longest processing time first, which
 * keeps the last wave short).  Results do not depend on the order.  Without
 * one, warp w takes points w, w + warps, ... .  Waits for `stream`.
 * Errors: INVALID_ARG, CUDA. */
gts_status gts_params_set_order(gts_params *params, uint32_t *d_order, void *stream);

/* Per-point output row lengths (the per-node start and finish cycles and the
 * thread-block placement of Section 5.1): start/finish rows hold
 * gts_row_nodes() entries (the largest graph of the stack), cta_sm rows
 * gts_row_ctas(). */
uint32_t gts_row_nodes(const gts_graph *graph);
uint32_t gts_row_ctas(const gts_graph *graph);

/* Device scratch gts_simulate_batch wants: GTS_SCRATCH_HEADER_BYTES (the
 * next-point counter of an ordered batch), then one row per concurrently
 * simulated design point -- dependency counters (Section 5.3 dependency-driven
 * runtime control: released predecessors and latest release cycle, 8 bytes per
 * node of the largest graph, rounded up to 16 bytes) and, for a graph with tiles, one
 * 16-byte L2 list record per tile.  Returns the size that lets every resident
 * warp work; a smaller scratch (the header and at least one row) runs fewer
 * points at a time.
 * Every call leaves the rows it used all zero: a node's dependency counters
 * go back to zero when the node becomes a warp head, and a design point that
 * stops early (error status) clears what it used.  With GTS_SCRATCH_CLEAN the
 * caller vouches that the scratch past the header is all zero -- zero-filled
 * once when allocated and since then passed only to gts_simulate_batch -- and
 * no row is cleared up front.  Without it each warp clears its row before its
 * first design point, which writes the whole scratch once per call.  A flag
 * given for a scratch that is not clean gives wrong results, not a fault.
 * Calls sharing one scratch must not overlap on the GPU. */
#define GTS_SCRATCH_HEADER_BYTES 16
size_t gts_scratch_bytes(const gts_graph *graph, const gts_params *params, uint32_t flags);

/*
 * Simulates design points first_point .. first_point+n_points-1 of `params`
 * on `graph`: the graph-driven simulation backend of Section 5 (5.1 execution
 * flow, 5.2 throughput-oriented hardware model, 5.3 dependency-driven runtime
 * control), with the semantics stated at the top of this file.  Output arrays are indexed by q = p - first_point:
 *   d_makespan[q], d_status[q]                      (required)
 *   d_start[q*row_nodes + v], d_finish[...]         (GTS_FULL_TRACE; graph-local v)
 *   d_digest[q]                                     (GTS_WANT_DIGEST)
 *   d_cta_sm[q*row_ctas + c]                        (GTS_WANT_CTA_SM; graph-local c)
 *   d_busy[q*GTS_BUSY_CLASSES + r]                  (GTS_WANT_BUSY; see above)
 * Start/finish/digest/cta_sm/busy of a point whose status is not GTS_OK are
 * unspecified.  The digest is sum over v of splitmix64-finalise(
 * (v << 32 | (uint32)start) ^ ((uint64)(uint32)finish * 0x9E3779B97F4A7C15)) mod 2^64.
 * d_scratch (16-byte aligned, scratch_bytes long) is required; see
 * gts_scratch_bytes.  Every other device pointer is aligned to its element
 * type, as C requires of typed pointers (4 bytes for the int32 arrays, 8 for
 * d_digest and d_busy); d_busy's alignment is checked (INVALID_ARG).  Enqueues on `stream` and returns; *out (may be NULL)
 * remembers the arrays for gts_read_results.  Errors: INVALID_ARG, NOMEM
 * (scratch smaller than one row), CUDA.
 */
gts_status gts_simulate_batch(gts_graph *graph, gts_params *params,
                              uint32_t first_point, uint32_t n_points, uint32_t flags,
                              int32_t *d_start, int32_t *d_finish,
                              int32_t *d_makespan, int32_t *d_status,
                              uint64_t *d_digest, int32_t *d_cta_sm, int64_t *d_busy,
                              void *d_scratch, size_t scratch_bytes,
                              void *stream, gts_results **out);

/* Waits for the batch and copies its per-point arrays -- the kernel makespan
 * of each design point (Section 5.1: the cycle the last node completes), its
 * status and digest -- to the host (any h_* may be NULL; n_points <= the
 * batch's).  Errors: INVALID_ARG, CUDA. */
gts_status gts_read_results(gts_results *results, int32_t *h_makespan, int32_t *h_status,
                            uint64_t *h_digest, uint32_t n_points);
/* Frees a results handle; the device arrays stay the caller's. */
gts_status gts_results_destroy(gts_results *results);

/*
 * No-allocation variant of gts_simulate_batch.  The paper has no counterpart:
 * it is an interface for callers that cannot allocate device memory when they
 * call it -- a plug-in running inside a host application that owns every
 * device allocation and hands out no scratch, or a service whose device memory
 * is fixed at start-up so that its allocator must not grow while requests run.
 * Instead of caller scratch it uses one fixed array of GTS_STATIC_SCRATCH_BYTES
 * that lives in the library's own device memory: every GPU that loads the
 * library holds it until the process exits.  The caller still passes every
 * input and output.
 *  - The array's device address is looked up (cudaGetSymbolAddress) on the
 *    first call in each device context, with that device current, and kept
 *    with the context's id; a call in a new context (after cudaDeviceReset)
 *    looks it up again.  The first call may load the library's module on the
 *    device: make it before any stream capture.  No call allocates or frees
 *    device memory.
 *  - The scratch header and one row (see gts_scratch_bytes) must fit in
 *    GTS_STATIC_SCRATCH_BYTES, else GTS_ERR_NOMEM: at most 4,194,302 nodes in
 *    the largest graph without tiles.  Fewer design points then run at a time
 *    than with a large caller scratch (as many as rows fit in the array).
 *  - All calls share the array, which keeps the last call's contents; each
 *    warp clears its row before its first design point (GTS_SCRATCH_CLEAN is
 *    ignored here), so nothing carries over between calls.  Calls that overlap
 *    on the GPU (other streams, other threads) race on it and must be ordered
 *    by the caller.
 *  - No results handle is returned: read d_makespan / d_status directly.
 * Errors: as gts_simulate_batch, plus NOMEM for a graph too large.
 */
#define GTS_STATIC_SCRATCH_BYTES (32u << 20)
gts_status gts_simulate_batch_noalloc(gts_graph *graph, gts_params *params,
                                      uint32_t first_point, uint32_t n_points, uint32_t flags,
                                      int32_t *d_start, int32_t *d_finish,
                                      int32_t *d_makespan, int32_t *d_status,
                                      uint64_t *d_digest, int32_t *d_cta_sm, int64_t *d_busy,
                                      void *stream);

/* Message for the calling thread's last non-OK host-side status ("" if none).
 * Error reporting of this C ABI; the paper has no counterpart. */
const char *gts_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* GTS_H */
