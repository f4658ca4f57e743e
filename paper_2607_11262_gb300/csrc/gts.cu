// gts.cu -- libgts: batched graph-driven tile-graph simulation on sm_103a.
//
// One warp simulates one design point (one hardware parameter row) of the
// graph-driven simulation backend (Section 5): the warp keeps the event
// frontier -- the head node of every logical warp stream of every resident
// CTA -- plus the per-SM unit servers, the global HBM servers and the CTA
// slots in shared memory, and advances the schedule with warp ballot / shuffle
// / min-reduction primitives.  The tile graph is shared read-only by all
// points; each point's start/finish rows live in global memory (the output
// trace, or caller scratch).
//
// Semantics are those stated in include/gts.h.  Design notes:
//  * Issue selection (Section 5.3, lowest-id reading): every frontier slot
//    caches key = max(rdy, earliest free server of its per-SM class), or INF
//    while a predecessor is unissued; a head is issuable at t when key <= t
//    and, for LOAD/STORE, some HBM server is free at t.  The warp takes the
//    minimum node id over issuable heads (one __reduce_min_sync).
//  * Dependency release (Section 5.1): an issued node pushes its release time
//    (issue cycle for ISSUE edges, finish for DATA edges) only into
//    successors that are currently warp heads; a node that becomes a head
//    pulls the state of its already-issued predecessors from the point's
//    start/finish rows (start = -1 marks "not issued").  Every predecessor is
//    thus counted exactly once.
//  * Time advance: the next cycle is the minimum over heads of their key
//    (raised to the HBM availability for LOAD/STORE) and over finished CTAs of
//    their retirement cycle; no cycle in between can issue or launch.
//  * Server identity is unobservable, so "take any free server" takes the
//    first free one.
//  * Every loop is bounded: the per-point step count is capped by
//    8*n + 4*C + 64 (each step launches a CTA, issues a node or moves to a
//    distinct finish / server-free cycle, of which there are at most 3n);
//    reaching it writes GTS_ERR_STEP_LIMIT.  No kernel waits on another.
#include "gts.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <cstring>
#include <new>
#include <string>
#include <vector>

namespace {

constexpr uint32_t NONE = 0xFFFFFFFFu;     // no node / no CTA
constexpr uint32_t INF = 0xFFFFFFFFu;      // key of a head that cannot issue
constexpr uint32_t HBM_BIT = 0x80000000u;  // on a slot's node id: node uses HBM
constexpr uint32_t ID_MASK = 0x7FFFFFFFu;
constexpr uint32_t FULL = 0xFFFFFFFFu;
constexpr int MAX_WPB = 4;                  // warps (design points) per block
constexpr uint32_t MAX_SMEM_BYTES = 227u * 1024u;
constexpr uint32_t MAX_W = 128;

// per-SM resource classes (Section 5.2)
enum : uint32_t { RC_TENSOR = 0, RC_TMA = 1, RC_LSU = 2, RC_ALU = 3, RC_BAR = 4, RC_N = 5, RC_NONE = 7 };

thread_local std::string g_err;

gts_status fail(gts_status s, const std::string &msg) {
  g_err = msg;
  return s;
}

gts_status cuda_fail(cudaError_t e, const char *what) {
  return fail(GTS_ERR_CUDA, std::string(what) + ": " + cudaGetErrorString(e));
}

// ----------------------------------------------------------------- device graph
struct DevGraph {
  const uint4 *rec;            // [n] x=work y=lat_extra z=next node of the stream w=type|warp<<4
  const uint4 *rng;            // [n] x,y = predecessor list range; z,w = successor list range
  const uint2 *succ;           // [m] x=successor id, y=kind | warp<<1 | cta<<8
  const uint32_t *pred;        // [m] predecessor id | kind<<31
  const uint32_t *stream_first;// [C*W] first node of stream (c, w) or NONE
  const uint32_t *cta_cnt;     // [C] nodes per CTA
  const uint32_t *cta_kernel;  // [C]
  const uint32_t *node_off;    // [G+1]
  const uint32_t *cta_off;     // [G+1]
  uint32_t W, G, row_nodes, row_ctas, cross_cta;
};

// ----------------------------------------------------------------- per-point layout
// Shared-memory words of one design point.  Frontier slot s = (cta slot) * W
// + warp; CTA slot j lives on SM j / ctas_per_sm (SM-major, so the lowest free
// slot is on the lowest SM with room).  Only min(num_sms*cps, C) CTA slots can
// ever be occupied (a launch always takes the lowest free slot).
struct Layout {
  uint32_t S, Scta, NS, SC, cap_hbm;
  uint32_t cap[RC_N], off[RC_N];
  uint32_t o_prm, o_hid, o_key, o_rdy, o_np, o_L, o_occ, o_hocc, o_next, o_sb, o_se, o_meta;
  uint32_t o_cid, o_crem, o_cend, o_ckern, o_sv, o_hs, words;
};

__host__ __device__ inline int check_row(const int32_t *p, uint32_t G) {
  if (p[GTS_P_NUM_SMS] < 1 || p[GTS_P_CTAS_PER_SM] < 1) return GTS_ERR_INVALID_PARAMS;
  const int rates[5] = {GTS_P_HBM_BPC, GTS_P_TMA_BPC, GTS_P_SMEM_BPC, GTS_P_MMA_FMA_PC, GTS_P_ALU_OPS_PC};
  for (int i = 0; i < 5; i++)
    if (p[rates[i]] < 1) return GTS_ERR_INVALID_PARAMS;
  const int lats[6] = {GTS_P_DRAM_LAT, GTS_P_TMA_LAT, GTS_P_SMEM_LAT, GTS_P_MMA_LAT, GTS_P_ALU_LAT, GTS_P_BAR_LAT};
  for (int i = 0; i < 6; i++)
    if (p[lats[i]] < 0) return GTS_ERR_INVALID_PARAMS;
  for (int i = GTS_P_CAP_TENSOR; i <= GTS_P_CAP_HBM; i++)
    if (p[i] < 1) return GTS_ERR_INVALID_PARAMS;
  if (p[GTS_P_GRAPH_INDEX] < 0 || (uint32_t)p[GTS_P_GRAPH_INDEX] >= G) return GTS_ERR_INVALID_PARAMS;
  for (int i = 20; i < GTS_NPARAM; i++)
    if (p[i] != 0) return GTS_ERR_INVALID_PARAMS;
  return GTS_OK;
}

// Fills `L` for a valid row on a graph with CG CTAs; false if the point needs
// more than one warp's shared-memory budget.
__host__ __device__ inline bool make_layout(const int32_t *p, uint32_t CG, uint32_t W, Layout &L) {
  const uint64_t cps = (uint64_t)p[GTS_P_CTAS_PER_SM];
  uint64_t slots = (uint64_t)p[GTS_P_NUM_SMS] * cps;
  if (slots > CG) slots = CG;
  L.Scta = (uint32_t)slots;
  L.S = L.Scta * W;
  L.NS = (uint32_t)((slots + cps - 1) / cps);
  uint64_t sc = 0;
  for (int r = 0; r < (int)RC_N; r++) {
    const uint64_t c = (uint64_t)p[GTS_P_CAP_TENSOR + r];
    if (c > 65536) return false;
    L.cap[r] = (uint32_t)c;
    L.off[r] = (uint32_t)sc;
    sc += c;
  }
  L.SC = (uint32_t)sc;
  if ((uint64_t)p[GTS_P_CAP_HBM] > 65536) return false;
  L.cap_hbm = (uint32_t)p[GTS_P_CAP_HBM];
  uint64_t w = 0;
  L.o_prm = (uint32_t)w; w += GTS_NPARAM;
  L.o_hid = (uint32_t)w; w += L.S;
  L.o_key = (uint32_t)w; w += L.S;
  L.o_rdy = (uint32_t)w; w += L.S;
  L.o_np = (uint32_t)w; w += L.S;
  L.o_L = (uint32_t)w; w += L.S;
  L.o_occ = (uint32_t)w; w += L.S;
  L.o_hocc = (uint32_t)w; w += L.S;
  L.o_next = (uint32_t)w; w += L.S;
  L.o_sb = (uint32_t)w; w += L.S;
  L.o_se = (uint32_t)w; w += L.S;
  L.o_meta = (uint32_t)w; w += L.S;
  L.o_cid = (uint32_t)w; w += L.Scta;
  L.o_crem = (uint32_t)w; w += L.Scta;
  L.o_cend = (uint32_t)w; w += L.Scta;
  L.o_ckern = (uint32_t)w; w += L.Scta;
  L.o_sv = (uint32_t)w; w += (uint64_t)L.NS * L.SC;
  L.o_hs = (uint32_t)w; w += L.cap_hbm;
  w = (w + 3) & ~(uint64_t)3;  // 16-byte multiple
  if (w * 4 > MAX_SMEM_BYTES) return false;
  L.words = (uint32_t)w;
  return true;
}

// ----------------------------------------------------------------- device helpers
__device__ __forceinline__ uint32_t cdiv(uint32_t a, uint32_t b) { return a / b + (a % b != 0u); }

__device__ __forceinline__ uint64_t mix64(uint64_t z) {  // splitmix64 finaliser (Steele, Lea, Flood 2014)
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

struct Point {
  uint32_t *sp;      // this warp's shared-memory words
  Layout L;
  uint32_t W, cps, n0, c0, c1;
  int32_t *st, *fi;  // point rows (graph-local index)
};

// Per-node unit, occupancy and latency (Section 5.2 throughput model).
__device__ __forceinline__ void node_cost(const Point &P, uint32_t type, uint32_t work, uint32_t lx, uint32_t &cls,
                                          uint32_t &occ, uint32_t &hocc, uint32_t &lat, bool &hbm) {
  const int32_t *prm = reinterpret_cast<const int32_t *>(P.sp + P.L.o_prm);
  uint32_t base = 0;
  cls = RC_NONE;
  occ = 0;
  hocc = 0;
  hbm = false;
  switch (type) {
    case GTS_LOAD:
      cls = RC_TMA; occ = cdiv(work, (uint32_t)prm[GTS_P_TMA_BPC]);
      hbm = true; hocc = cdiv(work, (uint32_t)prm[GTS_P_HBM_BPC]);
      base = (uint32_t)prm[GTS_P_TMA_LAT] + (uint32_t)prm[GTS_P_DRAM_LAT];
      break;
    case GTS_SMEM:
      cls = RC_LSU; occ = cdiv(work, (uint32_t)prm[GTS_P_SMEM_BPC]); base = (uint32_t)prm[GTS_P_SMEM_LAT];
      break;
    case GTS_MMA:
      cls = RC_TENSOR; occ = cdiv(work, (uint32_t)prm[GTS_P_MMA_FMA_PC]); base = (uint32_t)prm[GTS_P_MMA_LAT];
      break;
    case GTS_EW:
      cls = RC_ALU; occ = cdiv(work, (uint32_t)prm[GTS_P_ALU_OPS_PC]); base = (uint32_t)prm[GTS_P_ALU_LAT];
      break;
    case GTS_STORE:
      cls = RC_TMA; occ = cdiv(work, (uint32_t)prm[GTS_P_TMA_BPC]);
      hbm = true; hocc = cdiv(work, (uint32_t)prm[GTS_P_HBM_BPC]);
      base = (uint32_t)prm[GTS_P_TMA_LAT];
      break;
    case GTS_BAR:
      cls = RC_BAR; occ = 1; base = (uint32_t)prm[GTS_P_BAR_LAT];
      break;
    default:
      break;
  }
  const uint64_t L = (uint64_t)base + lx + (occ > hocc ? occ : hocc);
  lat = L > 0x80000000ull ? 0x80000000u : (uint32_t)L;  // any value >= 2^31 overflows at issue
}

// Earliest cycle slot i's head could issue, ignoring HBM; INF if blocked.
__device__ __forceinline__ uint32_t slot_key(const Point &P, uint32_t i) {
  const uint32_t *sp = P.sp;
  const uint32_t h = sp[P.L.o_hid + i];
  if (h == NONE || sp[P.L.o_np + i] != 0u) return INF;
  uint32_t k = sp[P.L.o_rdy + i];
  const uint32_t cls = sp[P.L.o_meta + i] & 7u;
  if (cls != RC_NONE) {
    const uint32_t sm = (i / P.W) / P.cps;
    const uint32_t *sv = sp + P.L.o_sv + sm * P.L.SC + P.L.off[cls];
    uint32_t a = sv[0];
    for (uint32_t q = 1; q < P.L.cap[cls]; q++) a = min(a, sv[q]);
    k = max(k, a);
  }
  return k;
}

// Slot i takes node v as its head (v == NONE: stream exhausted).  The caller's
// lane alone does the work (used for CTA launches: one lane per stream).
__device__ void load_head_lane(const DevGraph &g, const Point &P, uint32_t i, uint32_t v) {
  uint32_t *sp = P.sp;
  if (v == NONE) {
    sp[P.L.o_hid + i] = NONE;
    sp[P.L.o_key + i] = INF;
    return;
  }
  const uint4 r = g.rec[v];
  const uint4 q = g.rng[v];
  uint32_t cnt = 0;
  int32_t rdy = 0;
  for (uint32_t e = q.x; e < q.y; e++) {
    const uint32_t pe = g.pred[e];
    const uint32_t u = (pe & ID_MASK) - P.n0;
    const int32_t s = P.st[u];
    if (s < 0) cnt++;
    else rdy = max(rdy, (pe >> 31) ? s : P.fi[u]);
  }
  uint32_t cls, occ, hocc, lat;
  bool hbm;
  node_cost(P, r.w & 15u, r.x, r.y, cls, occ, hocc, lat, hbm);
  sp[P.L.o_hid + i] = v | (hbm ? HBM_BIT : 0u);
  sp[P.L.o_np + i] = cnt;
  sp[P.L.o_rdy + i] = (uint32_t)rdy;
  sp[P.L.o_L + i] = lat;
  sp[P.L.o_occ + i] = occ;
  sp[P.L.o_hocc + i] = hocc;
  sp[P.L.o_next + i] = r.z;
  sp[P.L.o_sb + i] = q.z;
  sp[P.L.o_se + i] = q.w;
  sp[P.L.o_meta + i] = cls;
}

// Same, with the whole warp pulling the predecessors (one per lane).
__device__ void load_head_warp(const DevGraph &g, const Point &P, uint32_t i, uint32_t v, int lane) {
  uint32_t *sp = P.sp;
  if (v == NONE) {
    if (lane == 0) {
      sp[P.L.o_hid + i] = NONE;
      sp[P.L.o_key + i] = INF;
    }
    return;
  }
  const uint4 r = g.rec[v];
  const uint4 q = g.rng[v];
  uint32_t cnt = 0;
  int32_t rdy = 0;
  for (uint32_t e = q.x + lane; e < q.y; e += 32) {
    const uint32_t pe = g.pred[e];
    const uint32_t u = (pe & ID_MASK) - P.n0;
    const int32_t s = P.st[u];
    if (s < 0) cnt++;
    else rdy = max(rdy, (pe >> 31) ? s : P.fi[u]);
  }
  cnt = __reduce_add_sync(FULL, cnt);
  rdy = __reduce_max_sync(FULL, rdy);
  if (lane == 0) {
    uint32_t cls, occ, hocc, lat;
    bool hbm;
    node_cost(P, r.w & 15u, r.x, r.y, cls, occ, hocc, lat, hbm);
    sp[P.L.o_hid + i] = v | (hbm ? HBM_BIT : 0u);
    sp[P.L.o_np + i] = cnt;
    sp[P.L.o_rdy + i] = (uint32_t)rdy;
    sp[P.L.o_L + i] = lat;
    sp[P.L.o_occ + i] = occ;
    sp[P.L.o_hocc + i] = hocc;
    sp[P.L.o_next + i] = r.z;
    sp[P.L.o_sb + i] = q.z;
    sp[P.L.o_se + i] = q.w;
    sp[P.L.o_meta + i] = cls;
  }
}

// Retire finished CTAs and launch as many CTAs as fit at cycle t (Section 5.1
// TB scheduler; kernel-boundary gate).  Returns false on step-limit.
__device__ bool launch_ctas(const DevGraph &g, Point &P, int32_t t, uint32_t &next_cta, uint64_t &steps,
                            uint64_t step_limit, int32_t *cta_sm_row, int lane) {
  uint32_t *sp = P.sp;
  for (;;) {
    for (uint32_t j = lane; j < P.L.Scta; j += 32) {
      if (sp[P.L.o_cid + j] != NONE && sp[P.L.o_crem + j] == 0u && (int32_t)sp[P.L.o_cend + j] <= t)
        sp[P.L.o_cid + j] = NONE;
    }
    __syncwarp();
    if (next_cta >= P.c1) return true;
    const uint32_t kc = g.cta_kernel[next_cta];
    bool blocked = false;
    uint32_t freeslot = NONE;
    for (uint32_t j = lane; j < P.L.Scta; j += 32) {
      if (sp[P.L.o_cid + j] != NONE) {
        if (sp[P.L.o_ckern + j] < kc) blocked = true;
      } else {
        freeslot = min(freeslot, j);
      }
    }
    if (__any_sync(FULL, blocked)) return true;
    freeslot = __reduce_min_sync(FULL, freeslot);
    if (freeslot == NONE) return true;
    if (++steps > step_limit) return false;
    if (lane == 0) {
      sp[P.L.o_cid + freeslot] = next_cta;
      sp[P.L.o_crem + freeslot] = g.cta_cnt[next_cta];
      sp[P.L.o_cend + freeslot] = 0u;
      sp[P.L.o_ckern + freeslot] = kc;
      if (cta_sm_row) cta_sm_row[next_cta - P.c0] = (int32_t)(freeslot / P.cps);
    }
    for (uint32_t w = lane; w < P.W; w += 32) {
      const uint32_t i = freeslot * P.W + w;
      load_head_lane(g, P, i, g.stream_first[(size_t)next_cta * P.W + w]);
      sp[P.L.o_key + i] = slot_key(P, i);
    }
    __syncwarp();
    next_cta++;
  }
}

__global__ void __launch_bounds__(MAX_WPB * 32)
k_simulate(DevGraph g, const int32_t *__restrict__ params, uint32_t first_point, uint32_t n_points, uint32_t flags,
           int32_t *d_start, int32_t *d_finish, int32_t *d_makespan, int32_t *d_status, uint64_t *d_digest,
           int32_t *d_cta_sm, int32_t *scratch, uint32_t n_warps, uint32_t budget_words) {
  extern __shared__ __align__(16) uint32_t smem[];
  const int lane = threadIdx.x & 31;
  const uint32_t wib = threadIdx.x >> 5;
  const uint32_t gw = blockIdx.x * (blockDim.x >> 5) + wib;
  if (gw >= n_warps) return;
  Point P;
  P.sp = smem + wib * budget_words;
  P.W = g.W;
  uint32_t *sp = P.sp;

  for (uint32_t q = gw; q < n_points; q += n_warps) {
    const uint32_t p = first_point + q;
    // ---- parameter row -> shared memory
    if (lane < GTS_NPARAM) sp[lane] = (uint32_t)params[(size_t)p * GTS_NPARAM + lane];
    __syncwarp();
    const int32_t *prm = reinterpret_cast<const int32_t *>(sp);
    int status = check_row(prm, g.G);
    const uint32_t gi = status == GTS_OK ? (uint32_t)prm[GTS_P_GRAPH_INDEX] : 0u;
    P.n0 = g.node_off[gi];
    const uint32_t n1 = g.node_off[gi + 1];
    P.c0 = g.cta_off[gi];
    P.c1 = g.cta_off[gi + 1];
    const uint32_t nG = n1 - P.n0, CG = P.c1 - P.c0;
    if (status == GTS_OK) {
      if (!make_layout(prm, CG, P.W, P.L) || P.L.words > budget_words) status = GTS_ERR_UNSUPPORTED;
    }
    if (status != GTS_OK) {
      if (lane == 0) {
        d_status[q] = status;
        d_makespan[q] = 0;
        if (d_digest) d_digest[q] = 0;
      }
      __syncwarp();
      continue;
    }
    P.cps = (uint32_t)prm[GTS_P_CTAS_PER_SM];
    if (flags & GTS_FULL_TRACE) {
      P.st = d_start + (size_t)q * g.row_nodes;
      P.fi = d_finish + (size_t)q * g.row_nodes;
    } else {
      P.st = scratch + (size_t)gw * 2 * g.row_nodes;
      P.fi = P.st + g.row_nodes;
    }
    int32_t *cta_sm_row = (flags & GTS_WANT_CTA_SM) ? d_cta_sm + (size_t)q * g.row_ctas : nullptr;

    // ---- clear state
    for (uint32_t i = lane; i < P.L.S; i += 32) {
      sp[P.L.o_hid + i] = NONE;
      sp[P.L.o_key + i] = INF;
    }
    for (uint32_t j = lane; j < P.L.Scta; j += 32) sp[P.L.o_cid + j] = NONE;
    for (uint32_t k = lane; k < P.L.NS * P.L.SC; k += 32) sp[P.L.o_sv + k] = 0u;
    for (uint32_t k = lane; k < P.L.cap_hbm; k += 32) sp[P.L.o_hs + k] = 0u;
    for (uint32_t v = lane; v < nG; v += 32) P.st[v] = -1;
    if (cta_sm_row)
      for (uint32_t c = lane; c < CG; c += 32) cta_sm_row[c] = -1;
    __syncwarp();

    const uint64_t step_limit = 8ull * nG + 4ull * CG + 64ull;
    uint64_t steps = 0;
    uint32_t next_cta = P.c0, issued = 0;
    int32_t t = 0, mk = 0;
    uint32_t H = 0;  // earliest free HBM server
    uint64_t digest = 0;
    bool ok = launch_ctas(g, P, t, next_cta, steps, step_limit, cta_sm_row, lane);
    if (!ok) status = GTS_ERR_STEP_LIMIT;

    while (status == GTS_OK) {
      // ---- issue, lowest id first, until nothing is issuable at t
      for (;;) {
        const bool hbm_ok = H <= (uint32_t)t;
        uint32_t best = NONE, bslot = 0;
        for (uint32_t i = lane; i < P.L.S; i += 32) {
          if (sp[P.L.o_key + i] <= (uint32_t)t) {
            const uint32_t h = sp[P.L.o_hid + i];
            if (!(h & HBM_BIT) || hbm_ok) {
              const uint32_t id = h & ID_MASK;
              if (id < best) { best = id; bslot = i; }
            }
          }
        }
        const uint32_t v = __reduce_min_sync(FULL, best);
        if (v == NONE) break;
        const uint32_t owner = __ffs(__ballot_sync(FULL, best == v)) - 1;
        const uint32_t i = __shfl_sync(FULL, bslot, owner);
        if (++steps > step_limit) { status = GTS_ERR_STEP_LIMIT; break; }
        const uint32_t lat = sp[P.L.o_L + i];
        const int64_t f64 = (int64_t)t + (int64_t)lat;
        if (f64 > 0x7FFFFFFFll) { status = GTS_ERR_OVERFLOW; break; }
        const int32_t f = (int32_t)f64;
        const uint32_t hid = sp[P.L.o_hid + i];
        const uint32_t cls = sp[P.L.o_meta + i] & 7u;
        const uint32_t cs = i / P.W;
        const uint32_t sm = cs / P.cps;
        // take one server of the node's per-SM class
        if (cls != RC_NONE) {
          uint32_t *sv = sp + P.L.o_sv + sm * P.L.SC + P.L.off[cls];
          const uint32_t occ = sp[P.L.o_occ + i];
          for (uint32_t b = 0; b < P.L.cap[cls]; b += 32) {
            const uint32_t k = b + lane;
            const bool fr = k < P.L.cap[cls] && sv[k] <= (uint32_t)t;
            const uint32_t bal = __ballot_sync(FULL, fr);
            if (bal) {
              if (lane == (int)(__ffs(bal) - 1)) sv[k] = (uint32_t)t + occ;
              break;
            }
          }
        }
        // take one global HBM server
        if (hid & HBM_BIT) {
          uint32_t *hs = sp + P.L.o_hs;
          const uint32_t hocc = sp[P.L.o_hocc + i];
          for (uint32_t b = 0; b < P.L.cap_hbm; b += 32) {
            const uint32_t k = b + lane;
            const bool fr = k < P.L.cap_hbm && hs[k] <= (uint32_t)t;
            const uint32_t bal = __ballot_sync(FULL, fr);
            if (bal) {
              if (lane == (int)(__ffs(bal) - 1)) hs[k] = (uint32_t)t + hocc;
              break;
            }
          }
          __syncwarp();
          uint32_t hm = INF;
          for (uint32_t k = lane; k < P.L.cap_hbm; k += 32) hm = min(hm, hs[k]);
          H = __reduce_min_sync(FULL, hm);
        }
        const uint32_t vl = v - P.n0;
        if (lane == 0) {
          P.st[vl] = t;
          P.fi[vl] = f;
          sp[P.L.o_crem + cs] -= 1u;
          sp[P.L.o_cend + cs] = (uint32_t)max((int32_t)sp[P.L.o_cend + cs], f);
          digest += mix64(((uint64_t)vl << 32 | (uint32_t)t) ^ ((uint64_t)(uint32_t)f * 0x9E3779B97F4A7C15ull));
        }
        mk = max(mk, f);
        issued++;
        // release successors that are warp heads right now
        const uint32_t sb = sp[P.L.o_sb + i], se = sp[P.L.o_se + i];
        const uint32_t myc = sp[P.L.o_cid + cs];
        for (uint32_t e = sb + lane; e < se; e += 32) {
          const uint2 s = g.succ[e];
          const uint32_t wc = s.y >> 8;
          uint32_t tcs = NONE;
          if (wc == myc) {
            tcs = cs;
          } else {
            for (uint32_t j = 0; j < P.L.Scta; j++)
              if (sp[P.L.o_cid + j] == wc) { tcs = j; break; }
          }
          if (tcs != NONE) {
            const uint32_t j = tcs * P.W + ((s.y >> 1) & 127u);
            if ((sp[P.L.o_hid + j] & ID_MASK) == s.x) {
              atomicSub(&sp[P.L.o_np + j], 1u);
              atomicMax(reinterpret_cast<int *>(&sp[P.L.o_rdy + j]), (s.y & 1u) ? t : f);
            }
          }
        }
        __syncwarp();
        // the stream advances to its next node
        load_head_warp(g, P, i, sp[P.L.o_next + i], lane);
        __syncwarp();
        // refresh the keys the issue may have changed
        if (g.cross_cta) {
          for (uint32_t k = lane; k < P.L.S; k += 32) sp[P.L.o_key + k] = slot_key(P, k);
        } else {
          const uint32_t per = P.cps * P.W;
          const uint32_t k0 = sm * per, k1 = min(k0 + per, P.L.S);
          for (uint32_t k = k0 + lane; k < k1; k += 32) sp[P.L.o_key + k] = slot_key(P, k);
        }
        __syncwarp();
        if (sp[P.L.o_crem + cs] == 0u && (int32_t)sp[P.L.o_cend + cs] <= t) {
          if (!launch_ctas(g, P, t, next_cta, steps, step_limit, cta_sm_row, lane)) {
            status = GTS_ERR_STEP_LIMIT;
            break;
          }
        }
      }
      if (status != GTS_OK || issued == nG) break;
      // ---- advance to the next event cycle
      uint32_t tn = INF;
      for (uint32_t k = lane; k < P.L.S; k += 32) {
        uint32_t key = sp[P.L.o_key + k];
        if (key != INF) {
          if (sp[P.L.o_hid + k] & HBM_BIT) key = max(key, H);
          tn = min(tn, key);
        }
      }
      for (uint32_t j = lane; j < P.L.Scta; j += 32) {
        if (sp[P.L.o_cid + j] != NONE && sp[P.L.o_crem + j] == 0u) {
          const uint32_t ce = sp[P.L.o_cend + j];
          if (ce > (uint32_t)t) tn = min(tn, ce);
        }
      }
      tn = __reduce_min_sync(FULL, tn);
      if (tn == INF) { status = GTS_ERR_DEADLOCK; break; }
      if (++steps > step_limit) { status = GTS_ERR_STEP_LIMIT; break; }
      t = (int32_t)tn;
      if (!launch_ctas(g, P, t, next_cta, steps, step_limit, cta_sm_row, lane)) {
        status = GTS_ERR_STEP_LIMIT;
        break;
      }
    }
    if (lane == 0) {
      d_status[q] = status;
      d_makespan[q] = status == GTS_OK ? mk : 0;
      if (d_digest) d_digest[q] = status == GTS_OK ? digest : 0ull;
    }
    __syncwarp();
  }
}

size_t align_up(size_t x) { return (x + 255) & ~(size_t)255; }

struct WsLayout {
  size_t rec, rng, succ, pred, first, cnt, noff, coff, total;
};

bool ws_layout(uint64_t n, uint64_t m, uint64_t C, uint64_t W, uint64_t G, WsLayout &w) {
  if (n >= 0x7FFFFFFEull || C >= (1ull << 24) || W < 1 || W > MAX_W || G < 1 || G > C + n + 1) return false;
  size_t o = 0;
  w.rec = o; o += align_up(n * 16);
  w.rng = o; o += align_up(n * 16);
  w.succ = o; o += align_up(m * 8);
  w.pred = o; o += align_up(m * 4);
  w.first = o; o += align_up(C * W * 4);
  w.cnt = o; o += align_up(C * 4);
  w.noff = o; o += align_up((G + 1) * 4);
  w.coff = o; o += align_up((G + 1) * 4);
  w.total = o + 256;
  return true;
}

template <class T>
cudaError_t d2h(std::vector<T> &dst, const T *src, size_t count, cudaStream_t s) {
  dst.resize(count);
  if (count == 0) return cudaSuccess;
  if (!src) return cudaErrorInvalidValue;
  return cudaMemcpyAsync(dst.data(), src, count * sizeof(T), cudaMemcpyDeviceToHost, s);
}

}  // namespace

struct gts_graph {
  uint32_t n, m, C, W, G;
  DevGraph dg;
  int device;
  std::vector<uint32_t> node_off, cta_off;
};

struct gts_params {
  gts_graph *graph;
  const int32_t *d_params;
  uint32_t n_points;
  std::vector<uint32_t> words;  // per row: shared words, 0 if the row is invalid or too large
};

struct gts_results {
  int32_t *d_makespan, *d_status;
  uint64_t *d_digest;
  uint32_t n_points;
  cudaStream_t stream;
};

extern "C" {

const char *gts_last_error(void) { return g_err.c_str(); }

size_t gts_graph_workspace_bytes(uint32_t n_nodes, uint32_t n_edges, uint32_t n_ctas, uint32_t warps_per_cta,
                                 uint32_t n_graphs) {
  WsLayout w;
  if (!ws_layout(n_nodes, n_edges, n_ctas, warps_per_cta, n_graphs, w)) return 0;
  return w.total;
}

uint32_t gts_row_nodes(const gts_graph *g) { return g ? g->dg.row_nodes : 0u; }
uint32_t gts_row_ctas(const gts_graph *g) { return g ? g->dg.row_ctas : 0u; }

gts_status gts_graph_create(const gts_graph_desc *d, void *stream, gts_graph **out) {
  g_err.clear();
  if (!d || !out) return fail(GTS_ERR_INVALID_ARG, "null desc or out");
  *out = nullptr;
  const uint64_t n = d->n_nodes, m = d->n_edges, C = d->n_ctas, W = d->warps_per_cta, G = d->n_graphs;
  WsLayout wl;
  if (!ws_layout(n, m, C, W, G, wl))
    return fail(GTS_ERR_INVALID_ARG, "size out of range (n < 2^31-1, C < 2^24, 1 <= W <= 128, n_graphs >= 1)");
  if (!d->row_ptr || (n && (!d->type || !d->warp || !d->cta || !d->work || !d->lat_extra)) ||
      (m && (!d->col || !d->ekind)) || (C && !d->cta_kernel))
    return fail(GTS_ERR_INVALID_ARG, "null graph array");
  if (G > 1 && (!d->graph_node_off || !d->graph_cta_off))
    return fail(GTS_ERR_INVALID_ARG, "stacked graph needs graph_node_off and graph_cta_off");
  if (!d->workspace) return fail(GTS_ERR_INVALID_ARG, "null workspace");
  if (d->workspace_bytes < wl.total)
    return fail(GTS_ERR_NOMEM, "workspace too small: need " + std::to_string(wl.total) + " bytes");
  cudaStream_t s = (cudaStream_t)stream;
  std::vector<uint32_t> row_ptr, col, cta, work, lx, kern, noff, coff;
  std::vector<uint8_t> ek, ty;
  std::vector<uint16_t> wp;
  cudaError_t e = cudaSuccess;
  if (e == cudaSuccess) e = d2h(row_ptr, d->row_ptr, n + 1, s);
  if (e == cudaSuccess) e = d2h(col, d->col, m, s);
  if (e == cudaSuccess) e = d2h(ek, d->ekind, m, s);
  if (e == cudaSuccess) e = d2h(ty, d->type, n, s);
  if (e == cudaSuccess) e = d2h(wp, d->warp, n, s);
  if (e == cudaSuccess) e = d2h(cta, d->cta, n, s);
  if (e == cudaSuccess) e = d2h(work, d->work, n, s);
  if (e == cudaSuccess) e = d2h(lx, d->lat_extra, n, s);
  if (e == cudaSuccess) e = d2h(kern, d->cta_kernel, C, s);
  if (e == cudaSuccess) {
    if (G > 1 || d->graph_node_off) e = d2h(noff, d->graph_node_off, G + 1, s);
    else noff = {0u, (uint32_t)n};
  }
  if (e == cudaSuccess) {
    if (G > 1 || d->graph_cta_off) e = d2h(coff, d->graph_cta_off, G + 1, s);
    else coff = {0u, (uint32_t)C};
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "graph_create: copy to host");

  // ---- contract
  if (noff[0] != 0 || noff[G] != n || coff[0] != 0 || coff[G] != C)
    return fail(GTS_ERR_INVALID_GRAPH, "graph offsets must start at 0 and end at n_nodes / n_ctas");
  for (uint64_t k = 0; k < G; k++)
    if (noff[k + 1] < noff[k] || coff[k + 1] < coff[k])
      return fail(GTS_ERR_INVALID_GRAPH, "graph offsets decrease at graph " + std::to_string(k));
  if (row_ptr[0] != 0 || row_ptr[n] != m) return fail(GTS_ERR_INVALID_GRAPH, "row_ptr[0] != 0 or row_ptr[n] != n_edges");
  uint32_t row_nodes = 0, row_ctas = 0, cross = 0;
  for (uint64_t k = 0; k < G; k++) {
    const uint32_t n0 = noff[k], n1 = noff[k + 1], c0 = coff[k], c1 = coff[k + 1];
    row_nodes = std::max(row_nodes, n1 - n0);
    row_ctas = std::max(row_ctas, c1 - c0);
    for (uint32_t v = n0; v < n1; v++) {
      if (row_ptr[v + 1] < row_ptr[v]) return fail(GTS_ERR_INVALID_GRAPH, "row_ptr decreases at node " + std::to_string(v));
      if (ty[v] > GTS_NOP) return fail(GTS_ERR_INVALID_GRAPH, "bad type at node " + std::to_string(v));
      if (wp[v] >= W) return fail(GTS_ERR_INVALID_GRAPH, "warp >= warps_per_cta at node " + std::to_string(v));
      if (cta[v] < c0 || cta[v] >= c1) return fail(GTS_ERR_INVALID_GRAPH, "cta outside its graph at node " + std::to_string(v));
      for (uint32_t x = row_ptr[v]; x < row_ptr[v + 1]; x++) {
        if (col[x] <= v || col[x] >= n1)
          return fail(GTS_ERR_INVALID_GRAPH, "edge " + std::to_string(x) + " must go forward inside its graph");
        if (ek[x] > 1) return fail(GTS_ERR_INVALID_GRAPH, "bad edge kind at edge " + std::to_string(x));
        if (cta[col[x]] != cta[v]) cross = 1;
      }
    }
    for (uint32_t c = c0 + 1; c < c1; c++)
      if (kern[c] < kern[c - 1]) return fail(GTS_ERR_INVALID_GRAPH, "cta_kernel decreases at CTA " + std::to_string(c));
  }

  // ---- derived arrays
  std::vector<uint32_t> indeg(n + 1, 0), pptr(n + 1, 0), pred(m), first(C * W, NONE), nxt(n, NONE), cnt(C, 0);
  for (uint64_t x = 0; x < m; x++) indeg[col[x]]++;
  for (uint64_t v = 0; v < n; v++) pptr[v + 1] = pptr[v] + indeg[v];
  {
    std::vector<uint32_t> cur(pptr.begin(), pptr.end() - 1);
    for (uint64_t u = 0; u < n; u++)
      for (uint32_t x = row_ptr[u]; x < row_ptr[u + 1]; x++)
        pred[cur[col[x]]++] = (uint32_t)u | ((uint32_t)ek[x] << 31);
  }
  for (uint64_t v = n; v-- > 0;) {
    const uint64_t key = (uint64_t)cta[v] * W + wp[v];
    nxt[v] = first[key];
    first[key] = (uint32_t)v;
  }
  for (uint64_t v = 0; v < n; v++) cnt[cta[v]]++;
  std::vector<uint4> rec(n), rng(n);
  for (uint64_t v = 0; v < n; v++) {
    rec[v] = make_uint4(work[v], lx[v], nxt[v], (uint32_t)ty[v] | ((uint32_t)wp[v] << 4));
    rng[v] = make_uint4(pptr[v], pptr[v + 1], row_ptr[v], row_ptr[v + 1]);
  }
  std::vector<uint2> succ(m);
  for (uint64_t x = 0; x < m; x++)
    succ[x] = make_uint2(col[x], (uint32_t)ek[x] | ((uint32_t)wp[col[x]] << 1) | (cta[col[x]] << 8));

  char *ws = (char *)d->workspace;
  e = cudaSuccess;
  auto up = [&](size_t off, const void *src, size_t bytes) {
    if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(ws + off, src, bytes, cudaMemcpyHostToDevice, s);
  };
  up(wl.rec, rec.data(), n * 16);
  up(wl.rng, rng.data(), n * 16);
  up(wl.succ, succ.data(), m * 8);
  up(wl.pred, pred.data(), m * 4);
  up(wl.first, first.data(), C * W * 4);
  up(wl.cnt, cnt.data(), C * 4);
  up(wl.noff, noff.data(), (G + 1) * 4);
  up(wl.coff, coff.data(), (G + 1) * 4);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "graph_create: copy to device");

  gts_graph *g = new (std::nothrow) gts_graph();
  if (!g) return fail(GTS_ERR_INVALID_ARG, "host allocation failed");
  g->n = (uint32_t)n; g->m = (uint32_t)m; g->C = (uint32_t)C; g->W = (uint32_t)W; g->G = (uint32_t)G;
  cudaGetDevice(&g->device);
  g->node_off = noff;
  g->cta_off = coff;
  DevGraph &dg = g->dg;
  dg.rec = (const uint4 *)(ws + wl.rec);
  dg.rng = (const uint4 *)(ws + wl.rng);
  dg.succ = (const uint2 *)(ws + wl.succ);
  dg.pred = (const uint32_t *)(ws + wl.pred);
  dg.stream_first = (const uint32_t *)(ws + wl.first);
  dg.cta_cnt = (const uint32_t *)(ws + wl.cnt);
  dg.cta_kernel = d->cta_kernel;
  dg.node_off = (const uint32_t *)(ws + wl.noff);
  dg.cta_off = (const uint32_t *)(ws + wl.coff);
  dg.W = (uint32_t)W;
  dg.G = (uint32_t)G;
  dg.row_nodes = row_nodes;
  dg.row_ctas = row_ctas;
  dg.cross_cta = cross;
  *out = g;
  return GTS_OK;
}

gts_status gts_graph_destroy(gts_graph *g) {
  delete g;
  return GTS_OK;
}

gts_status gts_params_upload(gts_graph *g, const int32_t *d_params, uint32_t n_points, void *stream,
                             gts_params **out) {
  g_err.clear();
  if (!g || !out || (n_points && !d_params)) return fail(GTS_ERR_INVALID_ARG, "null graph, params or out");
  *out = nullptr;
  std::vector<int32_t> h;
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = d2h(h, d_params, (size_t)n_points * GTS_NPARAM, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "params_upload: copy to host");
  gts_params *P = new (std::nothrow) gts_params();
  if (!P) return fail(GTS_ERR_INVALID_ARG, "host allocation failed");
  P->graph = g;
  P->d_params = d_params;
  P->n_points = n_points;
  P->words.assign(n_points, 0u);
  for (uint32_t p = 0; p < n_points; p++) {
    const int32_t *row = h.data() + (size_t)p * GTS_NPARAM;
    if (check_row(row, g->G) != GTS_OK) continue;
    const uint32_t gi = (uint32_t)row[GTS_P_GRAPH_INDEX];
    Layout L;
    if (make_layout(row, g->cta_off[gi + 1] - g->cta_off[gi], g->W, L)) P->words[p] = L.words;
  }
  *out = P;
  return GTS_OK;
}

gts_status gts_params_destroy(gts_params *p) {
  delete p;
  return GTS_OK;
}

namespace {
struct Plan {
  uint32_t words, wpb, smem, blocks, warps;
};

gts_status plan_launch(const gts_graph *g, const gts_params *P, uint32_t first, uint32_t np, uint32_t flags,
                       size_t scratch_bytes, bool limit_by_scratch, Plan &pl) {
  uint32_t words = 64;
  for (uint32_t p = first; p < first + np; p++) words = std::max(words, P->words[p]);
  const uint32_t bytes = words * 4;
  pl.words = words;
  pl.wpb = std::max(1u, std::min((uint32_t)MAX_WPB, MAX_SMEM_BYTES / bytes));
  pl.smem = pl.wpb * bytes;
  cudaError_t e = cudaFuncSetAttribute(k_simulate, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)pl.smem);
  if (e != cudaSuccess) return cuda_fail(e, "simulate: set shared memory size");
  int nb = 0, dev = 0, sms = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, k_simulate, (int)pl.wpb * 32, pl.smem);
  if (e == cudaSuccess) e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_fail(e, "simulate: occupancy query");
  uint64_t warps = (uint64_t)std::max(nb, 1) * sms * pl.wpb;
  warps = std::min<uint64_t>(warps, np);
  if (limit_by_scratch && !(flags & GTS_FULL_TRACE)) {
    const uint64_t row = (uint64_t)g->dg.row_nodes * 8;
    const uint64_t fit = row ? scratch_bytes / row : warps;
    if (fit == 0) return fail(GTS_ERR_NOMEM, "scratch smaller than one point's start/finish rows");
    warps = std::min(warps, fit);
  }
  pl.warps = (uint32_t)std::max<uint64_t>(warps, 1);
  pl.blocks = (pl.warps + pl.wpb - 1) / pl.wpb;
  return GTS_OK;
}
}  // namespace

size_t gts_scratch_bytes(const gts_graph *g, const gts_params *P, uint32_t flags) {
  if (!g || !P) return 0;
  if (flags & GTS_FULL_TRACE) return 0;
  Plan pl;
  if (plan_launch(g, P, 0, P->n_points, flags, 0, false, pl) != GTS_OK) return 0;
  return (size_t)pl.warps * g->dg.row_nodes * 8;
}

gts_status gts_simulate_batch(gts_graph *g, gts_params *P, uint32_t first_point, uint32_t n_points, uint32_t flags,
                              int32_t *d_start, int32_t *d_finish, int32_t *d_makespan, int32_t *d_status,
                              uint64_t *d_digest, int32_t *d_cta_sm, void *d_scratch, size_t scratch_bytes,
                              void *stream, gts_results **out) {
  g_err.clear();
  if (out) *out = nullptr;
  if (!g || !P || P->graph != g) return fail(GTS_ERR_INVALID_ARG, "null or mismatched graph / params");
  if (flags & ~(GTS_FULL_TRACE | GTS_WANT_DIGEST | GTS_WANT_CTA_SM)) return fail(GTS_ERR_INVALID_ARG, "unknown flag");
  if ((uint64_t)first_point + n_points > P->n_points) return fail(GTS_ERR_INVALID_ARG, "point range outside the table");
  if (!d_makespan || !d_status) return fail(GTS_ERR_INVALID_ARG, "d_makespan and d_status are required");
  if ((flags & GTS_FULL_TRACE) && (!d_start || !d_finish)) return fail(GTS_ERR_INVALID_ARG, "FULL_TRACE needs d_start and d_finish");
  if ((flags & GTS_WANT_DIGEST) && !d_digest) return fail(GTS_ERR_INVALID_ARG, "WANT_DIGEST needs d_digest");
  if ((flags & GTS_WANT_CTA_SM) && !d_cta_sm) return fail(GTS_ERR_INVALID_ARG, "WANT_CTA_SM needs d_cta_sm");
  if (!(flags & GTS_FULL_TRACE) && !d_scratch && g->dg.row_nodes) return fail(GTS_ERR_NOMEM, "scratch required without FULL_TRACE");
  cudaStream_t s = (cudaStream_t)stream;
  if (n_points) {
    Plan pl;
    gts_status st = plan_launch(g, P, first_point, n_points, flags, scratch_bytes, true, pl);
    if (st != GTS_OK) return st;
    k_simulate<<<pl.blocks, pl.wpb * 32, pl.smem, s>>>(
        g->dg, P->d_params, first_point, n_points, flags, d_start, d_finish, d_makespan, d_status,
        (flags & GTS_WANT_DIGEST) ? d_digest : nullptr, (flags & GTS_WANT_CTA_SM) ? d_cta_sm : nullptr,
        (int32_t *)d_scratch, pl.warps, pl.words);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "simulate: launch");
  }
  if (out) {
    gts_results *r = new (std::nothrow) gts_results();
    if (!r) return fail(GTS_ERR_INVALID_ARG, "host allocation failed");
    r->d_makespan = d_makespan;
    r->d_status = d_status;
    r->d_digest = (flags & GTS_WANT_DIGEST) ? d_digest : nullptr;
    r->n_points = n_points;
    r->stream = s;
    *out = r;
  }
  return GTS_OK;
}

gts_status gts_read_results(gts_results *r, int32_t *h_makespan, int32_t *h_status, uint64_t *h_digest,
                            uint32_t n_points) {
  g_err.clear();
  if (!r) return fail(GTS_ERR_INVALID_ARG, "null results");
  if (n_points > r->n_points) return fail(GTS_ERR_INVALID_ARG, "n_points exceeds the batch");
  if (h_digest && !r->d_digest) return fail(GTS_ERR_INVALID_ARG, "batch ran without WANT_DIGEST");
  cudaError_t e = cudaSuccess;
  if (n_points) {
    if (h_makespan) e = cudaMemcpyAsync(h_makespan, r->d_makespan, n_points * 4, cudaMemcpyDeviceToHost, r->stream);
    if (e == cudaSuccess && h_status)
      e = cudaMemcpyAsync(h_status, r->d_status, n_points * 4, cudaMemcpyDeviceToHost, r->stream);
    if (e == cudaSuccess && h_digest)
      e = cudaMemcpyAsync(h_digest, r->d_digest, n_points * 8, cudaMemcpyDeviceToHost, r->stream);
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(r->stream);
  if (e != cudaSuccess) return cuda_fail(e, "read_results");
  return GTS_OK;
}

gts_status gts_results_destroy(gts_results *r) {
  delete r;
  return GTS_OK;
}

}  // extern "C"
