// gts.cu -- libgts: batched graph-driven tile-graph simulation on sm_103a.
//
// One warp simulates one design point (one hardware parameter row) of the
// graph-driven simulation backend (Section 5).  The warp keeps in shared
// memory the event frontier -- the head node of every logical warp stream of
// every resident CTA -- with each head's release state, the per-SM unit
// servers, the global HBM servers, the CTA slots, and one summary per
// simulated SM; it advances the schedule with warp min-reductions.  The tile
// graph is shared read-only by all points.  Per point, a global scratch row
// holds the dependency counters of nodes that are not warp heads yet.
//
// Semantics are those stated in include/gts.h.  Design notes:
//  * Issue keys (Section 5.3, lowest-id reading).  A head's key is the
//    earliest cycle >= now at which its predecessors are released and its
//    per-SM unit has a free server (INF while a predecessor is unissued); for
//    LOAD/STORE the effective cycle is max(key, H), H the earliest free HBM
//    server.  Every unissued head keeps effective cycle >= t (keys are clamped
//    to the cycle they are computed at; a head that could issue at t but did
//    not has had its key recomputed when its unit or H changed), so the next
//    event is the minimum of (effective cycle << 32 | node id) over all
//    heads: if its cycle is t, the node is the lowest-id issuable head;
//    otherwise it is the next event cycle.  Each simulated SM keeps that
//    minimum over its heads; lane l owns SMs l, l+32, ... and keeps the
//    minimum over them in registers; the warp takes the minimum over lanes
//    with two __reduce_min_sync.  After an issue the issuing SM's keys and
//    summary are recomputed warp-parallel together with its owner lane's
//    minimum (one pass, two independent reductions, for SMs of <= 16 slots);
//    when H moves, the SMs whose HBM heads it overtakes are recomputed (each
//    lane its own SMs, or one SM at a time a slot per lane when SMs hold 8
//    slots or more).  When every SM has fewer than 8 slots, an SM whose only
//    issuable HBM head is one keeps that head apart in its summary and takes
//    its effective cycle max(key, H) when the summary is read, so such SMs
//    need no recomputation when H moves.  A release into a head of another
//    CTA recomputes every SM (the extended instance: the SMs it reached).
//  * The issue itself runs in every lane on broadcast values (no divergence);
//    only global atomics and scratch-counter reads are lane 0's.
//  * Dependency release (Section 5.1).  An issued node releases each
//    successor at its issue cycle (ISSUE edge) or finish (DATA edge): into the
//    frontier if the successor is a warp head, else into the successor's
//    scratch counters (count of released predecessors, max release cycle)
//    with fire-and-forget global atomics.  A node that becomes a head reads
//    its counters once; everything after that reaches it in shared memory.
//    Lane 0 performs every release and every counter read of a point, so
//    program order orders them; CTA launches, whose heads are read by other
//    lanes, fence first.
//  * Occupancy ceil(work / rate) uses exact division by invariant integers
//    (Lemire, Kaser, Kurz 2019: floor(n/d) = floor(ceil(2^64/d) * n / 2^64)
//    for 32-bit n and d), with the per-point constants computed once; slot,
//    CTA-slot and SM indices (< 2^16) use the 32-bit form of the same method.
//  * Server identity is unobservable, so "take any free server" takes the
//    first free one.
//  * Every loop is bounded: the per-point step count is capped by
//    8*n + 4*C + 64 (each step launches a CTA, issues a node or moves to a
//    distinct finish / server-free / retirement cycle, of which there are at
//    most 3n); reaching it writes GTS_ERR_STEP_LIMIT.  No warp waits on
//    another warp.
#include "gts.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstring>
#include <new>
#include <string>
#include <vector>

namespace {

constexpr uint32_t NONE = 0xFFFFFFFFu;     // no node / no CTA
constexpr uint32_t INF = 0xFFFFFFFFu;      // key of a head that cannot issue
constexpr uint64_t INF64 = ~0ull;
constexpr uint32_t HBM_BIT = 0x80000000u;  // on a slot's node id: node uses HBM
constexpr uint32_t ID_MASK = 0x7FFFFFFFu;
constexpr uint32_t FULL = 0xFFFFFFFFu;
constexpr int MAX_WPB = 4;                  // warps (design points) per block, at most
constexpr uint32_t MAX_SMEM_BYTES = 227u * 1024u;
constexpr uint32_t MAX_W = 128;
constexpr uint32_t MAX_INDEG = (1u << 24) - 1;
constexpr uint32_t DEG_BIG = 31;            // successor count field: 31 = read it from the graph

// per-SM resource classes (Section 5.2)
enum : uint32_t { RC_TENSOR = 0, RC_TMA = 1, RC_LSU = 2, RC_ALU = 3, RC_BAR = 4, RC_N = 5, RC_NONE = 7 };
// class code of a DSMEM node: an LSU server on its SM plus a NoC server of its SM group
constexpr uint32_t RC_DSM = 5;
// class_mask bit: some node crosses the NoC (servers of unused classes are not kept)
constexpr uint32_t CM_NOC = 1u << 5;
// Per node type (LOAD, SMEM, MMA, EW, STORE, BAR, NOP, DSMEM), one nibble
// each: its class code, and the rate that sets its per-SM occupancy (0 HBM,
// 1 TMA, 2 SMEM, 3 MMA, 4 ALU, 5 = one cycle, 6 = none).  LOAD and STORE also
// take an HBM server.
constexpr uint32_t TYPE_CLASS = 0x57413021u;
constexpr uint32_t TYPE_RATE = 0x26514321u;
constexpr uint32_t TYPE_HBM = 0x11u;
static_assert(GTS_P_TMA_BPC == GTS_P_HBM_BPC + 2 && GTS_P_SMEM_BPC == GTS_P_HBM_BPC + 4 &&
                  GTS_P_MMA_FMA_PC == GTS_P_HBM_BPC + 6 && GTS_P_ALU_OPS_PC == GTS_P_HBM_BPC + 8,
              "rate k of the division-constant table sits at parameter index GTS_P_HBM_BPC + 2k");

thread_local char g_err[512];

gts_status fail(gts_status s, const char *msg) {
  size_t k = 0;
  for (; msg[k] && k + 1 < sizeof(g_err); k++) g_err[k] = msg[k];
  g_err[k] = 0;
  return s;
}

gts_status fail(gts_status s, const std::string &msg) { return fail(s, msg.c_str()); }

void clear_error() { g_err[0] = 0; }

gts_status cuda_fail(cudaError_t e, const char *what) {
  char buf[256];
  size_t k = 0;
  for (const char *p = what; *p && k < 200; p++) buf[k++] = *p;
  buf[k++] = ':';
  buf[k++] = ' ';
  for (const char *p = cudaGetErrorString(e); *p && k + 1 < sizeof(buf); p++) buf[k++] = *p;
  buf[k] = 0;
  return fail(GTS_ERR_CUDA, (const char *)buf);
}

// ----------------------------------------------------------------- device graph
struct DevGraph {
  const uint4 *rec;            // [n] x=work y=lat_extra z=next node of the stream w=type | indegree<<4
  const uint4 *rng;            // [n] z,w = successor list range (x, y unused)
  const uint2 *succ;           // [m] x=successor id, y=kind | warp<<1 | cta<<8
  const uint32_t *stream_first;// [C*W] first node of stream (c, w) or NONE
  const uint32_t *cta_cnt;     // [C] nodes per CTA
  const uint32_t *cta_kernel;  // [C]
  const uint32_t *node_off;    // [G+1]
  const uint32_t *cta_off;     // [G+1]
  uint32_t W, G, row_nodes, row_ctas, cross_cta;
  uint32_t n_tiles;     // tile ids of LOAD/STORE nodes (rng.x = tile + 1; 0: none)
  uint32_t class_mask;  // bit r < 5: some node uses per-SM class r; CM_NOC: some node crosses the NoC
};

// ----------------------------------------------------------------- per-point layout
// Shared-memory words of one design point.  Frontier slot i = (CTA slot) * W +
// warp; CTA slot j lives on SM j / ctas_per_sm (SM-major, so the lowest free
// slot is on the lowest SM with room).  Only min(num_sms*cps, C) CTA slots can
// ever be occupied (a launch always takes the lowest free slot).
constexpr uint32_t O_MAG = GTS_NPARAM;       // 7 x 2 words: division constants of the 5 rates, NoC and L2 rates
constexpr uint32_t O_BASE = GTS_NPARAM + 14; // 8 words: base latency per node type, then LOAD hit / miss with L2
constexpr uint32_t O_L2B = O_BASE + 8;
constexpr uint32_t O_DYN = GTS_NPARAM + 24;  // first per-point array
static_assert(O_MAG % 2 == 0, "division constants are 8-byte words");
// slot record (4 words, one 16-byte vector): id|HBM, rdy, pending<<8 | deg<<3 | class, next node of the stream.
// The successor-list start is read from the node's range record when it issues, which keeps a point at 4 words
// per warp slot (at 132 SMs x 3 warps, 8 two-warp blocks fit on an SM instead of 7).
constexpr uint32_t F_HID = 0, F_RDY = 1, F_META = 2, F_NXT = 3, SLOT_WORDS = 4;
static_assert(O_DYN % 4 == 0 && SLOT_WORDS == 4 && F_NXT == 3, "warp slots are read and written as 16-byte vectors");
// SM record (4 words): best id, best effective cycle, best slot, min key of its HBM heads
constexpr uint32_t SM_WORDS = 4;
static_assert(SM_WORDS % 2 == 0, "SM records are read as 8-byte pairs");
// CTA slot record (3 words): CTA id, nodes not issued, max finish
constexpr uint32_t C_ID = 0, C_REM = 1, C_END = 2, CTA_WORDS = 3;

// Scheduler record (2 words, per-subpartition policies only): first cycle it
// may issue again, warp slot on the SM it issued from last (NONE: never)
constexpr uint32_t Q_AVAIL = 0, Q_LAST = 1, SUB_WORDS = 2;

struct Layout {
  uint32_t S, Scta, NS, SC, cap_hbm, per, nsub, csms, cap_noc;
  uint32_t o_slot, o_sm, o_cta, o_sv, o_hs, o_sub, o_ns, words;
};

__host__ __device__ inline int check_row(const int32_t *p, uint32_t G, uint32_t class_mask) {
  if (p[GTS_P_NUM_SMS] < 1 || p[GTS_P_CTAS_PER_SM] < 1) return GTS_ERR_INVALID_PARAMS;
  for (int i = 0; i < 5; i++)
    if (p[GTS_P_HBM_BPC + 2 * i] < 1) return GTS_ERR_INVALID_PARAMS;
  const int lats[6] = {GTS_P_DRAM_LAT, GTS_P_TMA_LAT, GTS_P_SMEM_LAT, GTS_P_MMA_LAT, GTS_P_ALU_LAT, GTS_P_BAR_LAT};
  for (int i = 0; i < 6; i++)
    if (p[lats[i]] < 0) return GTS_ERR_INVALID_PARAMS;
  for (int i = GTS_P_CAP_TENSOR; i <= GTS_P_CAP_HBM; i++)
    if (p[i] < 1) return GTS_ERR_INVALID_PARAMS;
  if (p[GTS_P_GRAPH_INDEX] < 0 || (uint32_t)p[GTS_P_GRAPH_INDEX] >= G) return GTS_ERR_INVALID_PARAMS;
  const int32_t pol = p[GTS_P_ISSUE_POLICY], nsub = p[GTS_P_SUBPARTITIONS];
  if (pol == GTS_POLICY_LOWEST_ID) {
    if (nsub != 0) return GTS_ERR_INVALID_PARAMS;
  } else if (pol == GTS_POLICY_GTO || pol == GTS_POLICY_RR) {
    if (nsub < 1 || nsub > 32) return GTS_ERR_INVALID_PARAMS;
  } else {
    return GTS_ERR_INVALID_PARAMS;
  }
  const int32_t csms = p[GTS_P_CLUSTER_SMS], cap_noc = p[GTS_P_CAP_NOC];
  if (csms != 0) {
    if (p[GTS_P_NOC_BPC] < 1 || p[GTS_P_NOC_LAT] < 0 || cap_noc < 1 || cap_noc > 32 || csms > 32)
      return GTS_ERR_INVALID_PARAMS;
  } else if (p[GTS_P_NOC_BPC] != 0 || p[GTS_P_NOC_LAT] != 0 || cap_noc != 0) {
    return GTS_ERR_INVALID_PARAMS;
  }
  if ((class_mask & CM_NOC) && csms == 0) return GTS_ERR_INVALID_PARAMS;  // DSMEM nodes, no NoC
  if (p[GTS_P_L2_BYTES] != 0) {
    if (p[GTS_P_L2_BYTES] < 1 || p[GTS_P_L2_LAT] < 0 || p[GTS_P_L2_BPC] < 1) return GTS_ERR_INVALID_PARAMS;
  } else if (p[GTS_P_L2_LAT] != 0 || p[GTS_P_L2_BPC] != 0) {
    return GTS_ERR_INVALID_PARAMS;
  }
  for (int i = GTS_P_L2_BPC + 1; i < GTS_NPARAM; i++)
    if (p[i] != 0) return GTS_ERR_INVALID_PARAMS;
  return GTS_OK;
}

// Fills `L` for a valid row on a graph with CG CTAs; false if the point needs
// more than one warp's shared-memory budget.  Servers per class are limited
// to 32 (one lane each).
__host__ __device__ inline bool make_layout(const int32_t *p, uint32_t CG, uint32_t W, uint32_t class_mask,
                                          Layout &L) {
  const uint64_t cps = (uint64_t)p[GTS_P_CTAS_PER_SM];
  uint64_t slots = (uint64_t)p[GTS_P_NUM_SMS] * cps;
  if (slots > CG) slots = CG;
  L.Scta = (uint32_t)slots;
  L.S = L.Scta * W;
  L.NS = (uint32_t)((slots + cps - 1) / cps);
  if (cps * W > 0xFFFFull) return false;
  L.per = (uint32_t)(cps * W);
  uint64_t sc = 0;
  for (int r = 0; r < (int)RC_N; r++) {
    const uint64_t c = (uint64_t)p[GTS_P_CAP_TENSOR + r];
    if (!((class_mask >> r) & 1u)) continue;
    if (c > 32) return false;
    sc += c;
  }
  L.SC = (uint32_t)sc;
  if ((uint64_t)p[GTS_P_CAP_HBM] > 32) return false;
  L.cap_hbm = (uint32_t)p[GTS_P_CAP_HBM];
  uint64_t w = O_DYN;
  L.o_slot = (uint32_t)w; w += (uint64_t)L.S * SLOT_WORDS;
  w = (w + 1) & ~(uint64_t)1;  // SM records are read as 8-byte pairs
  L.o_sm = (uint32_t)w; w += (uint64_t)L.NS * SM_WORDS;
  L.o_cta = (uint32_t)w; w += (uint64_t)L.Scta * CTA_WORDS;
  L.o_sv = (uint32_t)w; w += (uint64_t)L.NS * L.SC;
  L.o_hs = (uint32_t)w; w += L.cap_hbm;
  L.nsub = (uint32_t)p[GTS_P_SUBPARTITIONS];
  L.o_sub = (uint32_t)w; w += (uint64_t)L.NS * L.nsub * SUB_WORDS;
  L.csms = (uint32_t)p[GTS_P_CLUSTER_SMS];
  L.cap_noc = (class_mask & CM_NOC) ? (uint32_t)p[GTS_P_CAP_NOC] : 0u;
  L.o_ns = (uint32_t)w;  // NoC servers per SM group
  if (L.cap_noc) w += (uint64_t)((L.NS + L.csms - 1) / L.csms) * L.cap_noc;
  w = (w + 3) & ~(uint64_t)3;  // 16-byte multiple
  if (w * 4 > MAX_SMEM_BYTES) return false;
  L.words = (uint32_t)w;
  return true;
}

// ----------------------------------------------------------------- device helpers
// ceil(2^64 / d) for d >= 2 (0 encodes d == 1).
__device__ __forceinline__ uint64_t div_const(uint32_t d) { return d <= 1u ? 0ull : ~0ull / d + 1ull; }

// ceil(n / d) given M = div_const(d).
__device__ __forceinline__ uint32_t cdiv_c(uint32_t n, uint32_t d, uint64_t M) {
  if (M == 0ull) return n;
  const uint32_t q = (uint32_t)__umul64hi(M, (uint64_t)n);
  return q + (q * d != n ? 1u : 0u);
}

// floor(n / d) for n < 2^16 from m = div16_const(d) = ceil(2^32 / d) (0 for d = 1):
// n*m/2^32 exceeds n/d by less than n/2^32 < 2^-16, never enough to carry past the
// next integer when d < 2^16; for larger d both sides are 0.
__host__ __device__ __forceinline__ uint32_t div16_const(uint32_t d) { return d <= 1u ? 0u : 0xFFFFFFFFu / d + 1u; }
__device__ __forceinline__ uint32_t div16(uint32_t n, uint32_t m) { return m ? __umulhi(n, m) : n; }

__device__ __forceinline__ uint64_t mix64(uint64_t z) {  // splitmix64 finaliser (Steele, Lea, Flood 2014)
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint2 ld_counters(const uint2 *p) {  // strong load of a scratch counter pair
  uint2 r;
  asm volatile("ld.relaxed.gpu.global.v2.u32 {%0, %1}, [%2];" : "=r"(r.x), "=r"(r.y) : "l"(p) : "memory");
  return r;
}

__device__ __forceinline__ void st_counters_zero(uint2 *p) {  // a counter pair back to (0, 0)
  asm volatile("st.relaxed.gpu.global.v2.u32 [%0], {%1, %1};" ::"l"(p), "r"(0u) : "memory");
}

__device__ __forceinline__ uint64_t pack(uint32_t eff, uint32_t id) { return (uint64_t)eff << 32 | id; }

// Warp-wide minimum of a u64 (all lanes get it) and the lowest lane holding it.
__device__ __forceinline__ uint64_t warp_min64(uint64_t x, uint32_t &lane_of) {
  const uint32_t hi = __reduce_min_sync(FULL, (uint32_t)(x >> 32));
  const uint32_t lo = __reduce_min_sync(FULL, (uint32_t)(x >> 32) == hi ? (uint32_t)x : NONE);
  const uint64_t m = pack(hi, lo);
  lane_of = __ffs(__ballot_sync(FULL, x == m)) - 1;
  return m;
}

struct Pt {
  uint32_t *sp;  // this warp's shared-memory words
  Layout L;
  uint32_t W, cps, n0, c0, c1;
  int32_t *st, *fi;  // trace rows (graph-local index) or null
  uint2 *scr;        // scratch counters (graph-local index)
  uint64_t offs;     // byte r: offset of class r's servers inside an SM's servers
  uint32_t caps;     // 6 bits per class: servers of class r (0: class unused)
  uint32_t policy;   // GTS_POLICY_*; L.nsub > 0 for the per-subpartition policies
  uint32_t mW, mCps; // div16 constants of W and ctas_per_sm; slot and CTA-slot indices stay below
                     // 2^16 because the 4-word slot records of a point fit in MAX_SMEM_BYTES
  uint32_t mSub, mCsms;  // div16 constants of the scheduler count and the SMs per NoC group
  __device__ __forceinline__ uint32_t cls_off(uint32_t r) const { return (uint32_t)(offs >> (8 * r)) & 255u; }
  __device__ __forceinline__ uint32_t cls_cap(uint32_t r) const { return (caps >> (6 * r)) & 63u; }
  __device__ __forceinline__ uint32_t *slot(uint32_t i) const { return sp + L.o_slot + i * SLOT_WORDS; }
  __device__ __forceinline__ uint32_t *smrec(uint32_t s) const { return sp + L.o_sm + s * SM_WORDS; }
  __device__ __forceinline__ uint32_t *cta(uint32_t j) const { return sp + L.o_cta + j * CTA_WORDS; }
  __device__ __forceinline__ uint32_t *sub(uint32_t s, uint32_t u) const {
    return sp + L.o_sub + (s * L.nsub + u) * SUB_WORDS;
  }
};

// Occupancies and latency of a node (Section 5.2 throughput model): per-SM
// class, HBM and NoC occupancy; latency = base + lat_extra + the largest.
// l2: 0 no L2 model, 1 LOAD missed, 2 LOAD hit (L2 model, Section 5.2).
template <bool EXT>
__device__ __forceinline__ void node_cost(const uint32_t *sp, uint32_t type, uint32_t work, uint32_t lx,
                                          uint32_t &occ, uint32_t &hocc, uint32_t &nocc, uint64_t &lat,
                                          uint32_t l2 = 0u) {
  const uint32_t rt = (TYPE_RATE >> (4 * type)) & 15u;
  occ = rt == 5u ? 1u : 0u;
  if (rt < 5u) occ = cdiv_c(work, sp[GTS_P_HBM_BPC + 2 * rt], *reinterpret_cast<const uint64_t *>(sp + O_MAG + 2 * rt));
  hocc = 0u;
  if ((TYPE_HBM >> type) & 1u) hocc = cdiv_c(work, sp[GTS_P_HBM_BPC], *reinterpret_cast<const uint64_t *>(sp + O_MAG));
  nocc = 0u;
  if (EXT && type == GTS_DSMEM) nocc = cdiv_c(work, sp[GTS_P_NOC_BPC], *reinterpret_cast<const uint64_t *>(sp + O_MAG + 10));
  uint32_t base = sp[O_BASE + type];
  if (EXT && l2 != 0u && type == GTS_LOAD) {  // a hit is served by L2, a miss goes through L2 to DRAM
    if (l2 == 2u) hocc = cdiv_c(work, sp[GTS_P_L2_BPC], *reinterpret_cast<const uint64_t *>(sp + O_MAG + 12));
    base = sp[O_L2B + (l2 == 2u ? 0u : 1u)];
  }
  lat = (uint64_t)base + lx + max(max(occ, hocc), nocc);
}

// Dependency counters are read, released into and reset under an L2
// evict_last policy: a design point's live counters (the nodes near its warp
// heads) are re-touched soon after their first release, while the trace,
// written once and never read back, goes out as streaming stores.
__device__ __forceinline__ uint64_t keep_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ uint2 ld_counters_keep(const uint2 *p, uint64_t pol) {
  uint2 r;
  asm volatile("ld.relaxed.gpu.global.L2::cache_hint.v2.u32 {%0, %1}, [%2], %3;"
               : "=r"(r.x), "=r"(r.y) : "l"(p), "l"(pol) : "memory");
  return r;
}
__device__ __forceinline__ void red_keep(uint2 *c, uint32_t r, uint64_t pol) {  // one released predecessor at r
  asm volatile("red.relaxed.gpu.global.add.L2::cache_hint.u32 [%0], 1, %1;" ::"l"(&c->x), "l"(pol) : "memory");
  asm volatile("red.relaxed.gpu.global.max.L2::cache_hint.u32 [%0], %1, %2;" ::"l"(&c->y), "r"(r), "l"(pol) : "memory");
}
__device__ __forceinline__ void st_counters_zero_keep(uint2 *p, uint64_t pol) {
  asm volatile("st.relaxed.gpu.global.L2::cache_hint.v2.u32 [%0], {%1, %1}, %2;" ::"l"(p), "r"(0u), "l"(pol) : "memory");
}

// Key of slot i computed at cycle t (>= t; INF if it cannot issue yet).
template <bool EXT>
__device__ __forceinline__ uint32_t slot_key(const Pt &P, uint32_t i, uint32_t sm, uint32_t t) {
  const uint4 e = *reinterpret_cast<const uint4 *>(P.slot(i));  // {id|HBM, rdy, meta, next}
  const uint32_t h = e.x;
  const uint32_t meta = e.z;
  if (h == NONE || (meta >> 8) != 0u) return INF;
  uint32_t k = max(e.y, t);
  const uint32_t cls = meta & 7u;
  if (cls != RC_NONE) {
    const uint32_t sc = EXT && cls == RC_DSM ? RC_LSU : cls;
    const uint32_t *sv = P.sp + P.L.o_sv + sm * P.L.SC + P.cls_off(sc);
    const uint32_t cap = P.cls_cap(sc);
    uint32_t a = sv[0];
    for (uint32_t q = 1; q < cap; q++) a = min(a, sv[q]);
    k = max(k, a);
    if (EXT && cls == RC_DSM) {  // and a NoC server of the SM's group
      const uint32_t *ns = P.sp + P.L.o_ns + div16(sm, P.mCsms) * P.L.cap_noc;
      a = ns[0];
      for (uint32_t q = 1; q < P.L.cap_noc; q++) a = min(a, ns[q]);
      k = max(k, a);
    }
  }
  return k;
}

// One lane: SM s's record under per-subpartition schedulers (Section 5.3,
// greedy-then-oldest / round-robin).  Scheduler u's event is
// E_u = max(first cycle it may issue, least effective key of its heads); its
// pick is the first head in policy order among those whose effective key is
// <= E_u.  The record holds the least (E_u, id of the pick) over u.
template <bool EXT>
__device__ __forceinline__ void rescan_sm_sub(const Pt &P, uint32_t s, uint32_t t, uint32_t H) {
  const uint32_t per = P.L.per, nsub = P.L.nsub, i0 = s * per;
  const uint32_t nl = min(per, P.L.S - i0);
  uint64_t best = INF64;
  uint32_t bsl = 0, hmin = INF;
  for (uint32_t u = 0; u < nsub; u++) {
    const uint32_t *sq = P.sub(s, u);
    uint32_t m = INF;
    for (uint32_t l = u; l < nl; l += nsub) {
      const uint32_t k = slot_key<EXT>(P, i0 + l, s, t);
      if (k == INF) continue;
      if (P.slot(i0 + l)[F_HID] & HBM_BIT) {
        hmin = min(hmin, k);
        m = min(m, max(k, H));
      } else {
        m = min(m, k);
      }
    }
    if (m == INF) continue;
    const uint32_t E = max(m, sq[Q_AVAIL]), last = sq[Q_LAST];
    uint64_t bp = INF64;  // (policy key << 32 | slot)
    for (uint32_t l = u; l < nl; l += nsub) {
      const uint32_t k = slot_key<EXT>(P, i0 + l, s, t);
      if (k == INF) continue;
      const uint32_t e = (P.slot(i0 + l)[F_HID] & HBM_BIT) ? max(k, H) : k;
      if (e > E) continue;
      uint32_t key;
      if (P.policy == GTS_POLICY_GTO) {  // greedy slot, then the oldest warp (CTA id, warp)
        const uint32_t cs = div16(i0 + l, P.mW);  // CTA slot; i0 is a multiple of W
        key = (l == last ? 0u : 0x80000000u) | (P.cta(cs)[C_ID] * P.W + (i0 + l - cs * P.W));
      } else {                            // round-robin after the last slot
        const uint32_t x = l + per - last - 1u;  // l, last < per
        key = last == NONE ? l : (x >= per ? x - per : x);
      }
      bp = min(bp, pack(key, l));
    }
    const uint32_t lc = (uint32_t)bp;
    const uint64_t val = pack(E, P.slot(i0 + lc)[F_HID] & ID_MASK);
    if (val < best) {
      best = val;
      bsl = i0 + lc;
    }
  }
  uint32_t *o = P.smrec(s);
  o[0] = (uint32_t)best;
  o[1] = (uint32_t)(best >> 32);
  o[2] = bsl;
  o[3] = hmin;
}

// Warp-parallel form of rescan_sm_sub for SMs of at most 32 slots (one slot
// per lane): each lane keys its slot once; per scheduler one reduction gives
// E_u and a second its pick (policy keys are distinct within a scheduler).
template <bool EXT>
__device__ __forceinline__ void rescan_sm_sub_warp(const Pt &P, uint32_t s, uint32_t t, uint32_t H, int lane) {
  const uint32_t per = P.L.per, nsub = P.L.nsub, i0 = s * per;
  const uint32_t nl = min(per, P.L.S - i0);
  const uint32_t l = (uint32_t)lane;
  uint32_t e = INF, hk = INF, id = 0, u = NONE;
  if (l < nl) {
    const uint32_t k = slot_key<EXT>(P, i0 + l, s, t);
    const uint32_t h = P.slot(i0 + l)[F_HID];
    id = h & ID_MASK;
    u = l - div16(l, P.mSub) * nsub;
    if (k != INF) {
      const bool hb = (h & HBM_BIT) != 0u;
      e = hb ? max(k, H) : k;
      hk = hb ? k : INF;
    }
  }
  const uint32_t hmin = __reduce_min_sync(FULL, hk);
  uint64_t best = INF64;
  uint32_t bsl = 0;
  for (uint32_t v = 0; v < nsub && v < nl; v++) {
    const uint32_t m = __reduce_min_sync(FULL, u == v ? e : INF);
    if (m == INF) continue;
    const uint32_t *sq = P.sub(s, v);
    const uint32_t E = max(m, sq[Q_AVAIL]), last = sq[Q_LAST];
    const bool cand = u == v && e <= E;
    uint32_t key = INF;
    if (cand) {
      if (P.policy == GTS_POLICY_GTO) {  // greedy slot, then the oldest warp (CTA id, warp)
        const uint32_t cs = div16(i0 + l, P.mW);
        key = (l == last ? 0u : 0x80000000u) | (P.cta(cs)[C_ID] * P.W + (i0 + l - cs * P.W));
      } else {                            // round-robin after the last slot
        const uint32_t x = l + per - last - 1u;
        key = last == NONE ? l : (x >= per ? x - per : x);
      }
    }
    const uint32_t kmin = __reduce_min_sync(FULL, key);
    const uint32_t wl = __ffs(__ballot_sync(FULL, cand && key == kmin)) - 1;
    const uint64_t val = pack(E, __shfl_sync(FULL, id, wl));
    if (val < best) {
      best = val;
      bsl = i0 + wl;
    }
  }
  if (lane == 0) {
    uint32_t *o = P.smrec(s);
    o[0] = (uint32_t)best;
    o[1] = (uint32_t)(best >> 32);
    o[2] = bsl;
    o[3] = hmin;
  }
}

// Warp-parallel: the keys of SM s's heads at cycle t and the SM's summary
// record.  All lanes call it.
template <bool EXT>
__device__ __forceinline__ void refresh_sm(const Pt &P, uint32_t s, uint32_t t, uint32_t H, int lane) {
  if (EXT && P.L.nsub) {
    if (P.L.per <= 32u) rescan_sm_sub_warp<EXT>(P, s, t, H, lane);
    else if (lane == 0) rescan_sm_sub<EXT>(P, s, t, H);
    __syncwarp();
    return;
  }
  const uint32_t i0 = s * P.L.per, i1 = min(i0 + P.L.per, P.L.S);
  uint64_t best = INF64;
  uint32_t bsl = 0, hmin = INF;
  for (uint32_t base = i0; base < i1; base += 32) {
    const uint32_t i = base + lane;
    uint64_t val = INF64;
    if (i < i1) {
      const uint32_t k = slot_key<EXT>(P, i, s, t);
      const uint32_t h = P.slot(i)[F_HID];
      if (k != INF) {
        const bool hb = (h & HBM_BIT) != 0u;
        val = pack(hb ? max(k, H) : k, h & ID_MASK);
        if (hb) hmin = min(hmin, k);
      }
    }
    uint32_t who;
    const uint64_t m = warp_min64(val, who);
    if (m < best) {
      best = m;
      bsl = base + who;
    }
  }
  hmin = __reduce_min_sync(FULL, hmin);
  if (lane == 0) {
    uint32_t *o = P.smrec(s);
    o[0] = (uint32_t)best;
    o[1] = (uint32_t)(best >> 32);
    o[2] = bsl;
    o[3] = hmin;
  }
  __syncwarp();
}

// Warp-parallel, SMs of at most 16 slots and at most 512 SMs: SM s's record
// (as refresh_sm) and the owner lane's best (as refresh_owner after it) in
// one pass.  Lanes below per key SM s's slots; lane 16 + j reads the record of
// the owner's j-th SM (owner + 32 j) unless it is s; the two minima are
// independent reductions over the same values.
template <bool EXT>
__device__ __forceinline__ void refresh_sm_owner(const Pt &P, uint32_t s, uint32_t t, uint32_t H, int lane, uint64_t &b,
                                                 uint32_t &bsl) {
  const uint32_t per = P.L.per, i0 = s * per, owner = s & 31u, l = (uint32_t)lane;
  uint64_t vs = INF64, vo = INF64;
  uint32_t hk = INF, so = 0;
  if (l < per && i0 + l < P.L.S) {
    const uint32_t k = slot_key<EXT>(P, i0 + l, s, t);
    if (k != INF) {
      const uint32_t h = P.slot(i0 + l)[F_HID];
      const bool hb = (h & HBM_BIT) != 0u;
      vs = pack(hb ? max(k, H) : k, h & ID_MASK);
      if (hb) hk = k;
    }
  } else if (l >= 16u) {
    const uint32_t sj = owner + 32u * (l - 16u);
    if (sj < P.L.NS && sj != s) {
      const uint2 o = *reinterpret_cast<const uint2 *>(P.smrec(sj));
      vo = pack(o.y, o.x);
      so = P.smrec(sj)[2];
    }
  }
  uint32_t wa, wb;
  const uint64_t ma = warp_min64(vs, wa);
  const uint64_t mb = warp_min64(vs < vo ? vs : vo, wb);
  const uint32_t hmin = __reduce_min_sync(FULL, hk);
  const uint32_t sb = __shfl_sync(FULL, l < 16u ? i0 + l : so, wb);
  if (lane == 0) {
    uint32_t *o = P.smrec(s);
    o[0] = (uint32_t)ma;
    o[1] = (uint32_t)(ma >> 32);
    o[2] = ma == INF64 ? 0u : i0 + wa;
    o[3] = hmin;
  }
  if (l == owner) {
    b = mb;
    bsl = mb == INF64 ? 0u : sb;
  }
  __syncwarp();
}

// One lane: recompute the record of SM s at cycle t and horizon H.
template <bool EXT>
__device__ __forceinline__ void rescan_sm_lane(const Pt &P, uint32_t s, uint32_t t, uint32_t H) {
  if (EXT && P.L.nsub) {
    rescan_sm_sub<EXT>(P, s, t, H);
    return;
  }
  const uint32_t i0 = s * P.L.per, i1 = min(i0 + P.L.per, P.L.S);
  uint64_t best = INF64;
  uint32_t bsl = 0, hmin = INF;
  for (uint32_t i = i0; i < i1; i++) {
    const uint32_t k = slot_key<EXT>(P, i, s, t);
    if (k == INF) continue;
    const uint32_t h = P.slot(i)[F_HID];
    const bool hb = (h & HBM_BIT) != 0u;
    const uint64_t val = pack(hb ? max(k, H) : k, h & ID_MASK);
    if (hb) hmin = min(hmin, k);
    if (val < best) { best = val; bsl = i; }
  }
  uint32_t *o = P.smrec(s);
  o[0] = (uint32_t)best;
  o[1] = (uint32_t)(best >> 32);
  o[2] = bsl;
  o[3] = hmin;
}

// Lane's best (packed, slot) over the SMs it owns, computed by that lane.
__device__ __forceinline__ uint64_t lane_best(const Pt &P, int lane, uint32_t &slot) {
  uint64_t b = INF64;
  slot = 0;
  for (uint32_t s = lane; s < P.L.NS; s += 32) {
    const uint2 o = *reinterpret_cast<const uint2 *>(P.smrec(s));
    const uint64_t v = pack(o.y, o.x);
    if (v < b) { b = v; slot = P.smrec(s)[2]; }
  }
  return b;
}

// Warp-parallel: the best over the SMs owned by lane `owner`; the owner lane
// stores it in (b, bsl).
__device__ __forceinline__ void refresh_owner(const Pt &P, uint32_t owner, int lane, uint64_t &b, uint32_t &bsl) {
  uint64_t best = INF64;
  uint32_t slot = 0;
  for (uint32_t base = owner; base < P.L.NS; base += 32 * 32) {
    const uint32_t s = base + 32u * lane;
    uint64_t val = INF64;
    if (s < P.L.NS) {
      const uint2 o = *reinterpret_cast<const uint2 *>(P.smrec(s));
      val = pack(o.y, o.x);
    }
    uint32_t who;
    const uint64_t m = warp_min64(val, who);
    const uint32_t ws = __shfl_sync(FULL, s < P.L.NS ? P.smrec(s)[2] : 0u, who);
    if (m < best) { best = m; slot = ws; }
  }
  if ((uint32_t)lane == owner) { b = best; bsl = slot; }
}

// ---- split SM records (plain instance, SMs of fewer than 8 slots).  An SM
// with exactly one issuable HBM head keeps it apart from its other heads:
// words 0-1 hold the best NON-HBM head (effective cycle, id), word 2 that
// head's slot | the HBM head's slot << 16, word 3 the HBM head's key.  The HBM
// head's effective cycle max(key, H) is taken where the record is read, so a
// horizon move needs no rescan of such an SM.  Any other SM keeps the whole
// record (best head at the horizon of its last refresh, slot | SPLIT_NONE,
// least HBM key) and is rescanned when H passes that key.
constexpr uint32_t SPLIT_NONE = 0xFFFF0000u;

__device__ __forceinline__ void put_split_rec(const Pt &P, uint32_t s, uint64_t nh, uint32_t nhslot, uint64_t all,
                                              uint32_t allslot, uint32_t hcnt, uint32_t hslot, uint32_t hmin) {
  uint32_t *o = P.smrec(s);
  const bool one = hcnt == 1u;
  const uint64_t v = one ? nh : all;
  o[0] = (uint32_t)v;
  o[1] = (uint32_t)(v >> 32);
  o[2] = (v == INF64 ? 0u : (one ? nhslot : allslot)) | (one ? hslot << 16 : SPLIT_NONE);
  o[3] = hmin;
}

// Best (effective cycle << 32 | id) of SM s at horizon H, and its slot.
__device__ __forceinline__ uint64_t split_sm_best(const Pt &P, uint32_t s, uint32_t H, uint32_t &slot) {
  const uint32_t *o = P.smrec(s);
  const uint2 a = *reinterpret_cast<const uint2 *>(o);
  const uint2 c = *reinterpret_cast<const uint2 *>(o + 2);
  uint64_t v = pack(a.y, a.x);
  slot = c.x & 0xFFFFu;
  if ((c.x >> 16) != 0xFFFFu) {
    const uint64_t hv = pack(max(c.y, H), P.slot(c.x >> 16)[F_HID] & ID_MASK);
    if (hv < v) {
      v = hv;
      slot = c.x >> 16;
    }
  }
  return v;
}

// Warp-parallel refresh of SM s (all its slots in one round of lanes).
__device__ __forceinline__ void split_refresh_sm(const Pt &P, uint32_t s, uint32_t t, uint32_t H, int lane) {
  const uint32_t i0 = s * P.L.per, i = i0 + lane;
  uint64_t val = INF64;
  uint32_t hk = INF;
  bool hf = false;
  if (lane < (int)P.L.per && i < P.L.S) {
    const uint32_t k = slot_key<false>(P, i, s, t);
    const uint32_t h = P.slot(i)[F_HID];
    if (k != INF) {
      hf = (h & HBM_BIT) != 0u;
      val = pack(hf ? max(k, H) : k, h & ID_MASK);
      if (hf) hk = k;
    }
  }
  const uint32_t hcnt = __popc(__ballot_sync(FULL, hf));
  uint32_t who;
  const uint64_t m = warp_min64(hcnt == 1u && hf ? INF64 : val, who);
  const uint32_t hmin = __reduce_min_sync(FULL, hk);
  if (hcnt == 1u ? hf : lane == 0) put_split_rec(P, s, m, i0 + who, m, i0 + who, hcnt, i, hmin);
  __syncwarp();
}

// Warp-parallel, as refresh_sm_owner: SM s's record and the owner lane's best
// (b, bsl) from two independent reductions over the same values.
__device__ __forceinline__ void split_refresh_sm_owner(const Pt &P, uint32_t s, uint32_t t, uint32_t H, int lane,
                                                       uint64_t &b, uint32_t &bsl) {
  const uint32_t per = P.L.per, i0 = s * per, owner = s & 31u, l = (uint32_t)lane;
  uint64_t vs = INF64, vo = INF64;
  uint32_t hk = INF, so = 0;
  bool hf = false;
  if (l < per && i0 + l < P.L.S) {
    const uint32_t k = slot_key<false>(P, i0 + l, s, t);
    if (k != INF) {
      const uint32_t h = P.slot(i0 + l)[F_HID];
      hf = (h & HBM_BIT) != 0u;
      vs = pack(hf ? max(k, H) : k, h & ID_MASK);
      if (hf) hk = k;
    }
  } else if (l >= 16u) {
    const uint32_t sj = owner + 32u * (l - 16u);
    if (sj < P.L.NS && sj != s) vo = split_sm_best(P, sj, H, so);
  }
  const bool one = __popc(__ballot_sync(FULL, hf)) == 1u;
  uint32_t wa, wb;
  const uint64_t ma = warp_min64(one && hf ? INF64 : vs, wa);
  const uint64_t mb = warp_min64(vs < vo ? vs : vo, wb);
  const uint32_t hmin = __reduce_min_sync(FULL, hk);
  const uint32_t sb = __shfl_sync(FULL, l < 16u ? i0 + l : so, wb);
  if (one ? hf : lane == 0) {
    uint32_t *o = P.smrec(s);
    o[0] = (uint32_t)ma;
    o[1] = (uint32_t)(ma >> 32);
    o[2] = (ma == INF64 ? 0u : i0 + wa) | (one ? (i0 + l) << 16 : SPLIT_NONE);
    o[3] = hmin;
  }
  if (l == owner) {
    b = mb;
    bsl = mb == INF64 ? 0u : sb;
  }
  __syncwarp();
}

// One lane: recompute the record of SM s at cycle t and horizon H.
__device__ __forceinline__ void split_rescan_sm_lane(const Pt &P, uint32_t s, uint32_t t, uint32_t H) {
  const uint32_t i0 = s * P.L.per, i1 = min(i0 + P.L.per, P.L.S);
  uint64_t best = INF64, nbest = INF64;
  uint32_t bsl = 0, nsl = 0, hmin = INF, hcnt = 0, hslot = 0;
  for (uint32_t i = i0; i < i1; i++) {
    const uint32_t k = slot_key<false>(P, i, s, t);
    if (k == INF) continue;
    const uint32_t h = P.slot(i)[F_HID];
    const bool hb = (h & HBM_BIT) != 0u;
    const uint64_t val = pack(hb ? max(k, H) : k, h & ID_MASK);
    if (hb) {
      hmin = min(hmin, k);
      hcnt++;
      hslot = i;
    } else if (val < nbest) {
      nbest = val;
      nsl = i;
    }
    if (val < best) { best = val; bsl = i; }
  }
  put_split_rec(P, s, nbest, nsl, best, bsl, hcnt, hslot, hmin);
}

__device__ __forceinline__ uint64_t split_lane_best(const Pt &P, int lane, uint32_t H, uint32_t &slot) {
  uint64_t b = INF64;
  slot = 0;
  for (uint32_t s = lane; s < P.L.NS; s += 32) {
    uint32_t sl;
    const uint64_t v = split_sm_best(P, s, H, sl);
    if (v < b) { b = v; slot = sl; }
  }
  return b;
}

__device__ __forceinline__ void split_refresh_owner(const Pt &P, uint32_t owner, int lane, uint32_t H, uint64_t &b,
                                                    uint32_t &bsl) {
  uint64_t best = INF64;
  uint32_t slot = 0;
  for (uint32_t base = owner; base < P.L.NS; base += 32 * 32) {
    const uint32_t s = base + 32u * lane;
    uint64_t val = INF64;
    uint32_t sl = 0;
    if (s < P.L.NS) val = split_sm_best(P, s, H, sl);
    uint32_t who;
    const uint64_t m = warp_min64(val, who);
    const uint32_t ws = __shfl_sync(FULL, sl, who);
    if (m < best) { best = m; slot = ws; }
  }
  if ((uint32_t)lane == owner) { b = best; bsl = slot; }
}

// Refresh entry points of the kernel: the split forms in the instance that
// keeps split SM records, the plain ones otherwise.
template <bool EXT, bool SPL>
__device__ __forceinline__ void r_sm(const Pt &P, uint32_t s, uint32_t t, uint32_t H, int lane) {
  if constexpr (SPL) split_refresh_sm(P, s, t, H, lane); else refresh_sm<EXT>(P, s, t, H, lane);
}
template <bool EXT, bool SPL>
__device__ __forceinline__ void r_sm_owner(const Pt &P, uint32_t s, uint32_t t, uint32_t H, int lane, uint64_t &b,
                                           uint32_t &bsl) {
  if constexpr (SPL) split_refresh_sm_owner(P, s, t, H, lane, b, bsl); else refresh_sm_owner<EXT>(P, s, t, H, lane, b, bsl);
}
template <bool EXT, bool SPL>
__device__ __forceinline__ void r_rescan(const Pt &P, uint32_t s, uint32_t t, uint32_t H) {
  if constexpr (SPL) split_rescan_sm_lane(P, s, t, H); else rescan_sm_lane<EXT>(P, s, t, H);
}
template <bool SPL>
__device__ __forceinline__ uint64_t r_lane_best(const Pt &P, int lane, uint32_t H, uint32_t &slot) {
  if constexpr (SPL) return split_lane_best(P, lane, H, slot); else return lane_best(P, lane, slot);
}
template <bool SPL>
__device__ __forceinline__ void r_owner(const Pt &P, uint32_t owner, int lane, uint32_t H, uint64_t &b, uint32_t &bsl) {
  if constexpr (SPL) split_refresh_owner(P, owner, lane, H, b, bsl); else refresh_owner(P, owner, lane, b, bsl);
}
// SM s's record must be rescanned once H passes its least HBM key (whole records only).
template <bool SPL>
__device__ __forceinline__ bool r_stale(const Pt &P, uint32_t s, uint32_t H) {
  if constexpr (SPL) {
    const uint2 c = *reinterpret_cast<const uint2 *>(P.smrec(s) + 2);
    return c.y < H && (c.x >> 16) == 0xFFFFu;
  } else {
    return P.smrec(s)[3] < H;
  }
}

// Slot i takes node v as its head (v == NONE: stream exhausted); adj_cnt /
// adj_rdy are releases the caller applied directly.  Every lane writes the
// same values.
__device__ __forceinline__ void set_head(const Pt &P, uint32_t i, uint32_t v, uint4 r, uint4 q, uint2 c,
                                         uint32_t adj_cnt, uint32_t adj_rdy) {
  uint32_t *sl = P.slot(i);
  if (v == NONE) {
    sl[F_HID] = NONE;
    sl[F_META] = RC_NONE;
    return;
  }
  const uint32_t type = r.w & 15u;
  const uint32_t pend = (r.w >> 4) - c.x - adj_cnt;
  const uint32_t deg = min(q.w - q.z, DEG_BIG);
  *reinterpret_cast<uint4 *>(sl) = make_uint4(v | (((TYPE_HBM >> type) & 1u) ? HBM_BIT : 0u), max(c.y, adj_rdy),
                                              ((TYPE_CLASS >> (4 * type)) & 15u) | (deg << 3) | (pend << 8), r.z);
}

struct Clock {
  uint32_t t;          // current cycle
  uint32_t H;          // earliest free HBM server
  uint32_t next_ret;   // earliest retirement cycle among finished, still resident CTAs
  uint32_t next_cta;   // next CTA to launch (global id)
  uint64_t steps, limit;
};

// Retire finished CTAs and launch as many CTAs as fit at cycle t (Section 5.1
// TB scheduler; kernel-boundary gate).  Returns false on step-limit.
template <bool EXT, bool SPL>
__device__ bool launch_ctas(const DevGraph &g, Pt &P, Clock &C, int32_t *cta_sm_row, int lane, uint64_t &b,
                            uint32_t &bsl) {
  const uint32_t t = C.t;
  for (;;) {
    uint32_t nr = INF;
    for (uint32_t j = lane; j < P.L.Scta; j += 32) {
      uint32_t *cr = P.cta(j);
      if (cr[C_ID] != NONE && cr[C_REM] == 0u) {
        if (cr[C_END] <= t) cr[C_ID] = NONE;
        else nr = min(nr, cr[C_END]);
      }
    }
    C.next_ret = __reduce_min_sync(FULL, nr);
    __syncwarp();
    if (C.next_cta >= P.c1) return true;
    const uint32_t kc = g.cta_kernel[C.next_cta];
    bool blocked = false;
    uint32_t freeslot = NONE;
    for (uint32_t j = lane; j < P.L.Scta; j += 32) {
      const uint32_t *cr = P.cta(j);
      if (cr[C_ID] != NONE) {
        if (g.cta_kernel[cr[C_ID]] < kc) blocked = true;
      } else {
        freeslot = min(freeslot, j);
      }
    }
    if (__any_sync(FULL, blocked)) return true;
    freeslot = __reduce_min_sync(FULL, freeslot);
    if (freeslot == NONE) return true;
    if (++C.steps > C.limit) return false;
    const uint32_t c = C.next_cta;
    const uint32_t cnt = g.cta_cnt[c];
    if (lane == 0) {
      uint32_t *cr = P.cta(freeslot);
      cr[C_ID] = c;
      cr[C_REM] = cnt;
      cr[C_END] = 0u;
      if (cta_sm_row) cta_sm_row[c - P.c0] = (int32_t)div16(freeslot, P.mCps);
      __threadfence();  // lane 0's earlier counter releases before the heads are read below
    }
    __syncwarp();
    __threadfence();
    for (uint32_t w = lane; w < P.W; w += 32) {
      const uint32_t i = freeslot * P.W + w;
      const uint32_t v = g.stream_first[(size_t)c * P.W + w];
      uint4 r = make_uint4(0, 0, 0, 0), q = r;
      uint2 cc = make_uint2(0, 0);
      if (v != NONE) {
        r = g.rec[v];
        q = g.rng[v];
        cc = ld_counters(P.scr + (v - P.n0));
        if (cc.x | cc.y) st_counters_zero(P.scr + (v - P.n0));  // read once: leave the row clean
      }
      set_head(P, i, v, r, q, cc, 0u, 0u);
    }
    __syncwarp();
    const uint32_t s = div16(freeslot, P.mCps);
    r_sm<EXT, SPL>(P, s, t, C.H, lane);
    r_owner<SPL>(P, s & 31u, lane, C.H, b, bsl);
    C.next_cta++;
  }
}

// One access of the L2 model's LRU list of a design point (Section 5.2): tile
// x becomes the most recent entry, sized b; least recent entries are dropped
// until the total is <= cap.  T[x] = {previous (more recent), next (less
// recent), bytes, listed}; head / tail / used live in the calling lane.
// Returns whether x was listed before the access (a hit).  One lane calls it.
__device__ __forceinline__ uint32_t l2_access(uint4 *T, uint32_t x, uint32_t b, uint32_t &head, uint32_t &tail,
                                              uint64_t &used, uint64_t cap) {
  uint32_t *Tw = reinterpret_cast<uint32_t *>(T);
  const uint4 e = T[x];
  if (e.w) {  // unlink
    if (e.x != NONE) Tw[4 * e.x + 1] = e.y; else head = e.y;
    if (e.y != NONE) Tw[4 * e.y + 0] = e.x; else tail = e.x;
    used -= e.z;
  }
  T[x] = make_uint4(NONE, head, b, 1u);
  if (head != NONE) Tw[4 * head + 0] = x; else tail = x;
  head = x;
  used += b;
  while (used > cap) {  // every entry dropped leaves used <= cap at the latest
    const uint32_t y = tail;
    const uint4 ey = T[y];
    tail = ey.x;
    if (tail != NONE) Tw[4 * tail + 1] = NONE; else head = NONE;
    Tw[4 * y + 3] = 0u;
    used -= ey.z;
  }
  return e.w;
}

// The next design point of a warp (batch-relative), or NONE: from the shared
// counter over `order` (skipping points outside the batch), else the warp's
// own stride.
__device__ __noinline__ uint32_t next_point_of(const uint32_t *order, uint32_t n_order, uint32_t *counter,
                                               uint32_t first, uint32_t n, uint32_t q, uint32_t stride, int lane) {
  if (!order) return q + stride < n ? q + stride : NONE;
  for (;;) {
    uint32_t k = 0;
    if (lane == 0) k = atomicAdd(counter, 1u);
    k = __shfl_sync(FULL, k, 0);
    if (k >= n_order) return NONE;
    const uint32_t pa = order[k];
    if (pa >= first && pa - first < n) return pa - first;
  }
}

__device__ __forceinline__ uint32_t first_point_of(const uint32_t *order, uint32_t n_order, uint32_t *counter,
                                                   uint32_t first, uint32_t n, uint32_t gw, int lane) {
  if (!order) return gw < n ? gw : NONE;
  return next_point_of(order, n_order, counter, first, n, 0u, 0u, lane);
}

// EXT: the kernel instance that also runs the per-subpartition issue policies
// and the NoC of DSMEM nodes; the host launches a plain instance when no row
// asks for a policy and the graph has no DSMEM node.  SPL: the plain instance
// that keeps split SM records, launched when every row's SMs have fewer than 8
// warp slots (the record forms are described above split_sm_best); the other
// plain instance keeps whole records only.  A warp's registers come
// from one SM sub-partition's 16K-register file, allocated 8 per thread at a
// time: 4 warps fit per sub-partition up to 128 registers, 3 up to 168, 2
// above.  The plain instance is held to 128 (16 warps per SM; shared memory
// also allows 16 on rows of 132 SMs x 3 warps), the extended one to 168 (12
// warps per SM).
template <bool EXT, bool SPL>
__global__ void __launch_bounds__(MAX_WPB * 32, EXT ? 3 : 4)
k_simulate(DevGraph g, const int32_t *__restrict__ params, uint32_t first_point, uint32_t n_points, uint32_t flags,
           int32_t *d_start, int32_t *d_finish, int32_t *d_makespan, int32_t *d_status, uint64_t *d_digest,
           int32_t *d_cta_sm, int64_t *d_busy, uint2 *scratch, uint32_t n_warps, uint32_t budget_words,
           const uint32_t *__restrict__ order, uint32_t n_order) {
  extern __shared__ __align__(16) uint32_t smem[];
  const int lane = threadIdx.x & 31;
  const uint32_t wib = threadIdx.x >> 5;
  const uint32_t gw = blockIdx.x * (blockDim.x >> 5) + wib;
  if (gw >= n_warps) return;
  Pt P;
  P.sp = smem + wib * budget_words;
  P.W = g.W;
  uint32_t *sp = P.sp;
  const bool want_digest = d_digest != nullptr;
  // The warp's scratch row is all zero between its points: a node's counter
  // pair is reset when the node becomes a warp head (after that, releases
  // reach it in shared memory), and a point that stops early clears the part
  // it used.  A row is cleared once, before the warp's first point, unless
  // the caller vouches that the scratch is already clean.
  bool row_clean = (flags & GTS_SCRATCH_CLEAN) != 0u;

  // points: the next one in `order` (a counter in the scratch header), or
  // gw, gw + n_warps, ... without an order
  uint32_t *next_point = reinterpret_cast<uint32_t *>(scratch);
  for (uint32_t q = first_point_of(order, n_order, next_point, first_point, n_points, gw, lane); q != NONE;
       q = next_point_of(order, n_order, next_point, first_point, n_points, q, n_warps, lane)) {
    const uint32_t p = first_point + q;
    // ---- parameter row -> shared memory
    if (lane < GTS_NPARAM) sp[lane] = (uint32_t)params[(size_t)p * GTS_NPARAM + lane];
    __syncwarp();
    const int32_t *prm = reinterpret_cast<const int32_t *>(sp);
    int status = check_row(prm, g.G, g.class_mask);
    const uint32_t gi = status == GTS_OK ? (uint32_t)prm[GTS_P_GRAPH_INDEX] : 0u;
    P.n0 = g.node_off[gi];
    const uint32_t nG = g.node_off[gi + 1] - P.n0;
    P.c0 = g.cta_off[gi];
    P.c1 = g.cta_off[gi + 1];
    const uint32_t CG = P.c1 - P.c0;
    const bool l2on = EXT && status == GTS_OK && prm[GTS_P_L2_BYTES] != 0;
    if (status == GTS_OK) {
      if (!make_layout(prm, CG, P.W, g.class_mask, P.L) || P.L.words > budget_words ||
          (!EXT && (P.L.nsub || P.L.cap_noc || prm[GTS_P_L2_BYTES] != 0)) || (SPL && P.L.per >= 8u))
        status = GTS_ERR_UNSUPPORTED;
    }
    if (status != GTS_OK) {
      if (lane == 0) {
        d_status[q] = status;
        d_makespan[q] = 0;
        if (want_digest) d_digest[q] = 0;
      }
      if (d_busy && lane < GTS_BUSY_CLASSES) d_busy[(size_t)q * GTS_BUSY_CLASSES + lane] = 0;
      __syncwarp();
      continue;
    }
    P.cps = (uint32_t)prm[GTS_P_CTAS_PER_SM];
    P.mW = div16_const(P.W);
    P.mCps = div16_const(P.cps);
    P.mSub = EXT ? div16_const(P.L.nsub) : 0u;
    P.mCsms = EXT ? div16_const(P.L.csms) : 0u;
    P.policy = (uint32_t)prm[GTS_P_ISSUE_POLICY];
    P.st = (flags & GTS_FULL_TRACE) ? d_start + (size_t)q * g.row_nodes : nullptr;
    P.fi = (flags & GTS_FULL_TRACE) ? d_finish + (size_t)q * g.row_nodes : nullptr;
    P.scr = scratch + GTS_SCRATCH_HEADER_BYTES / 8 + (size_t)gw * (((g.row_nodes + 1u) & ~1u) + 2u * g.n_tiles);
    uint4 *l2t = reinterpret_cast<uint4 *>(P.scr + ((g.row_nodes + 1u) & ~1u));  // L2 list records per tile
    int32_t *cta_sm_row = (flags & GTS_WANT_CTA_SM) ? d_cta_sm + (size_t)q * g.row_ctas : nullptr;

    // ---- per-point constants and cleared state
    {  // servers are kept only for the classes the graph uses (caps <= 32, offsets < 160)
      uint32_t off = 0;
      P.offs = 0;
      P.caps = 0;
      for (uint32_t r = 0; r < RC_N; r++) {
        const uint32_t c = ((g.class_mask >> r) & 1u) ? (uint32_t)prm[GTS_P_CAP_TENSOR + r] : 0u;
        P.offs |= (uint64_t)off << (8 * r);
        P.caps |= c << (6 * r);
        off += c;
      }
    }
    if (lane < (int)RC_N) {
      *reinterpret_cast<uint64_t *>(sp + O_MAG + 2 * lane) = div_const((uint32_t)prm[GTS_P_HBM_BPC + 2 * lane]);
    } else if (lane == (int)RC_N) {
      *reinterpret_cast<uint64_t *>(sp + O_MAG + 10) = div_const((uint32_t)prm[GTS_P_NOC_BPC]);
    } else if (lane == (int)RC_N + 1) {
      *reinterpret_cast<uint64_t *>(sp + O_MAG + 12) = div_const((uint32_t)prm[GTS_P_L2_BPC]);
    } else if (lane == 30) {  // LOAD base with the L2 model: hit, miss
      sp[O_L2B] = (uint32_t)prm[GTS_P_TMA_LAT] + (uint32_t)prm[GTS_P_L2_LAT];
      sp[O_L2B + 1] = (uint32_t)prm[GTS_P_TMA_LAT] + (uint32_t)prm[GTS_P_L2_LAT] + (uint32_t)prm[GTS_P_DRAM_LAT];
    }
    if (lane < 8) {  // base latency per type: LOAD, SMEM, MMA, EW, STORE, BAR, NOP
      uint32_t bl = 0;
      switch (lane) {
        case GTS_LOAD: bl = (uint32_t)prm[GTS_P_TMA_LAT] + (uint32_t)prm[GTS_P_DRAM_LAT]; break;
        case GTS_SMEM: bl = (uint32_t)prm[GTS_P_SMEM_LAT]; break;
        case GTS_MMA: bl = (uint32_t)prm[GTS_P_MMA_LAT]; break;
        case GTS_EW: bl = (uint32_t)prm[GTS_P_ALU_LAT]; break;
        case GTS_STORE: bl = (uint32_t)prm[GTS_P_TMA_LAT]; break;
        case GTS_BAR: bl = (uint32_t)prm[GTS_P_BAR_LAT]; break;
        case GTS_DSMEM: bl = (uint32_t)prm[GTS_P_SMEM_LAT] + (uint32_t)prm[GTS_P_NOC_LAT]; break;
        default: break;
      }
      sp[O_BASE + lane] = bl;
    }
    for (uint32_t i = lane; i < P.L.S; i += 32) {
      uint32_t *sl = P.slot(i);
      sl[F_HID] = NONE;
      sl[F_META] = RC_NONE;
    }
    for (uint32_t s = lane; s < P.L.NS; s += 32) {
      uint32_t *o = P.smrec(s);
      o[0] = NONE; o[1] = INF; o[2] = SPL ? SPLIT_NONE : 0u; o[3] = INF;
    }
    for (uint32_t j = lane; j < P.L.Scta; j += 32) P.cta(j)[C_ID] = NONE;
    for (uint32_t k = lane; k < P.L.NS * P.L.SC; k += 32) sp[P.L.o_sv + k] = 0u;
    for (uint32_t k = lane; k < P.L.cap_hbm; k += 32) sp[P.L.o_hs + k] = 0u;
    if (P.L.cap_noc)
      for (uint32_t k = lane; k < ((P.L.NS + P.L.csms - 1) / P.L.csms) * P.L.cap_noc; k += 32) sp[P.L.o_ns + k] = 0u;
    for (uint32_t k = lane; k < P.L.NS * P.L.nsub; k += 32) {
      sp[P.L.o_sub + k * SUB_WORDS + Q_AVAIL] = 0u;
      sp[P.L.o_sub + k * SUB_WORDS + Q_LAST] = NONE;
    }
    if (!row_clean) {  // the whole row: counters of the largest graph, then the L2 list records
      uint4 *z = reinterpret_cast<uint4 *>(P.scr);
      const uint32_t nz = ((g.row_nodes + 1u) >> 1) + g.n_tiles;
      for (uint32_t k = lane; k < nz; k += 32) z[k] = make_uint4(0, 0, 0, 0);
      row_clean = true;
    }
    if (cta_sm_row)
      for (uint32_t c = lane; c < CG; c += 32) cta_sm_row[c] = -1;
    __threadfence();
    __syncwarp();

    Clock C;
    C.t = 0;
    C.H = 0;
    C.next_ret = INF;
    C.next_cta = P.c0;
    C.steps = 0;
    C.limit = 8ull * nG + 4ull * CG + 64ull;
    uint32_t issued = 0;
    int32_t mk = 0;
    uint64_t digest = 0;
    uint64_t busy = 0;  // lane r < 5: server-cycles of per-SM class r; 5: HBM; 6: NoC; 7, 8: L2 hits, loads
    uint32_t l2_head = NONE, l2_tail = NONE;  // the L2 list (lane 0)
    uint64_t l2_used = 0;
    const uint64_t l2_cap = l2on ? (uint64_t)prm[GTS_P_L2_BYTES] : 0ull;
    uint64_t b = INF64;  // this lane's best (effective cycle << 32 | id) over its SMs
    uint32_t bsl = 0;    // ... and its slot
    if (!launch_ctas<EXT, SPL>(g, P, C, cta_sm_row, lane, b, bsl)) status = GTS_ERR_STEP_LIMIT;

    while (status == GTS_OK && issued < nG) {
      // ---- next event: minimum of (effective cycle, node id) over all heads
      uint32_t owner;
      const uint64_t m = warp_min64(b, owner);
      const uint32_t E = (uint32_t)(m >> 32);
      if (E > C.t) {
        const uint32_t tn = min(E, C.next_ret);
        if (tn == INF) { status = GTS_ERR_DEADLOCK; break; }
        if (++C.steps > C.limit) { status = GTS_ERR_STEP_LIMIT; break; }
        C.t = tn;
        if (C.next_ret <= C.t) {  // a CTA retires first: launch, then choose again
          if (!launch_ctas<EXT, SPL>(g, P, C, cta_sm_row, lane, b, bsl)) { status = GTS_ERR_STEP_LIMIT; break; }
          continue;
        }
        // otherwise the minimum just found is the first issue at the new cycle
      }
      // ---- issue v, the lowest-id issuable head, at cycle t (all lanes, same values)
      if (++C.steps > C.limit) { status = GTS_ERR_STEP_LIMIT; break; }
      const uint32_t v = (uint32_t)m;
      const uint32_t i = __shfl_sync(FULL, bsl, owner);
      const uint32_t t = C.t;
      const uint32_t cs = div16(i, P.mW);
      const uint32_t sm = div16(cs, P.mCps);
      const uint32_t *sl = P.slot(i);
      const uint4 se = *reinterpret_cast<const uint4 *>(sl);
      const uint32_t hidv = se.x, meta = se.z, nx = se.w;
      const uint32_t cls = meta & 7u;
      // one round of loads: the issued node's record and range (its successor-list
      // start), the next head's record, range and counters; then the successor entries
      const uint64_t pol = keep_policy();
      const uint4 rv = g.rec[v];
      const uint4 qv = g.rng[v];
      const uint32_t tkey = l2on ? qv.x : 0u;  // tile + 1 of the node (0: none)
      const uint32_t sb = qv.z;
      uint4 rn = make_uint4(0, 0, 0, 0), qn = rn;
      uint2 cn = make_uint2(0, 0);
      if (nx != NONE) {
        rn = g.rec[nx];
        qn = g.rng[nx];
        if (lane == 0) cn = ld_counters_keep(P.scr + (nx - P.n0), pol);
      }
      uint32_t deg = (meta >> 3) & 31u;
      if (deg == DEG_BIG) deg = qv.w - sb;
      uint2 ew = make_uint2(NONE, 0);
      if ((uint32_t)lane < deg) ew = g.succ[sb + lane];
      uint32_t occ, hocc, nocc;
      uint64_t lat;
      uint32_t l2 = 0u;  // L2 model: 1 LOAD missed, 2 LOAD hit
      if (EXT && l2on) {
        const uint32_t ty = rv.w & 15u;
        const bool mem = (ty == GTS_LOAD || ty == GTS_STORE) && tkey != 0u;
        uint32_t hit = 0u;
        if (lane == 0 && mem) hit = l2_access(l2t, tkey - 1u, rv.x, l2_head, l2_tail, l2_used, l2_cap);
        hit = __shfl_sync(FULL, hit, 0);
        if (ty == GTS_LOAD) {
          l2 = hit ? 2u : 1u;
          busy += ((uint32_t)lane == GTS_BUSY_L2_HITS && hit) || ((uint32_t)lane == GTS_BUSY_L2_LOADS && mem) ? 1u : 0u;
        }
      }
      node_cost<EXT>(sp, rv.w & 15u, rv.x, rv.y, occ, hocc, nocc, lat, l2);
      const uint64_t f64 = (uint64_t)t + lat;
      if (f64 > 0x7FFFFFFFull) { status = GTS_ERR_OVERFLOW; break; }
      const uint32_t f = (uint32_t)f64;
      const uint32_t scls = EXT && cls == RC_DSM ? RC_LSU : cls;  // the per-SM class it takes
      busy += (uint32_t)lane == scls ? occ
            : (uint32_t)lane == GTS_BUSY_HBM ? hocc : ((uint32_t)lane == GTS_BUSY_NOC ? nocc : 0u);
      // take one free server of the node's class on its SM (lane k tests server k)
      if (cls != RC_NONE) {
        uint32_t *sv = sp + P.L.o_sv + sm * P.L.SC + P.cls_off(scls);
        const bool fr = (uint32_t)lane < P.cls_cap(scls) && sv[lane] <= t;
        const uint32_t bal = __ballot_sync(FULL, fr);
        if (lane == __ffs(bal) - 1) sv[lane] = t + occ;
      }
      bool noc_touch = false;  // a NoC server of the SM's group was taken
      if (EXT && cls == RC_DSM) {
        uint32_t *ns = sp + P.L.o_ns + div16(sm, P.mCsms) * P.L.cap_noc;
        const bool fr = (uint32_t)lane < P.L.cap_noc && ns[lane] <= t;
        const uint32_t bal = __ballot_sync(FULL, fr);
        if (lane == __ffs(bal) - 1) ns[lane] = t + nocc;
        noc_touch = P.L.csms > 1u;
      }
      if (EXT && P.L.nsub && lane == 0) {  // the issuing scheduler: one issue per cycle, remember the slot
        const uint32_t l = i - sm * P.L.per;
        uint32_t *sq = P.sub(sm, l - div16(l, P.mSub) * P.L.nsub);
        sq[Q_AVAIL] = t + 1u;
        sq[Q_LAST] = l;
      }
      // take one free global HBM server
      const uint32_t prevH = C.H;
      if (hidv & HBM_BIT) {
        uint32_t *hs = sp + P.L.o_hs;
        const bool in = (uint32_t)lane < P.L.cap_hbm;
        uint32_t hv = in ? hs[lane] : INF;
        const uint32_t bal = __ballot_sync(FULL, in && hv <= t);
        if (lane == __ffs(bal) - 1) {
          hv = t + hocc;
          hs[lane] = hv;
        }
        C.H = __reduce_min_sync(FULL, hv);
      }
      if (lane == 0) {
        if (P.st) {
          __stcs(P.st + (v - P.n0), (int32_t)t);
          __stcs(P.fi + (v - P.n0), (int32_t)f);
        }
        if (want_digest) digest += mix64(((uint64_t)(v - P.n0) << 32 | t) ^ ((uint64_t)f * 0x9E3779B97F4A7C15ull));
      }
      uint32_t *cr = P.cta(cs);
      const uint32_t rem = cr[C_REM] - 1u;
      const uint32_t cend = max(cr[C_END], f);
      const uint32_t myc = cr[C_ID];
      __syncwarp();
      cr[C_REM] = rem;
      cr[C_END] = cend;
      mk = max(mk, (int32_t)f);
      issued++;
      // ---- release successors, one per lane: into warp heads with shared-memory
      // atomics; into scratch counters by lane 0 (which also reads them later)
      uint32_t adj_cnt = 0, adj_rdy = 0;
      bool cross_touch = false;
      uint32_t xs = NONE;  // SM of the head in another CTA slot this lane released into (one round only)
      for (uint32_t base = 0; base < deg; base += 32) {
        if (base) ew = (base + lane < deg) ? g.succ[sb + base + lane] : make_uint2(NONE, 0);
        const bool mine = base + lane < deg;
        const uint32_t rel = (ew.y & 1u) ? t : f;
        const bool to_next = mine && ew.x == nx;  // the stream's next node becomes the head right below
        bool to_head = false, cross = false;
        const uint32_t wc = ew.y >> 8;
        uint32_t tcs = (mine && !to_next && wc == myc) ? cs : NONE;
        // successors in other CTAs: find each one's CTA slot, all lanes searching together
        uint32_t xm = g.cross_cta ? __ballot_sync(FULL, mine && !to_next && wc != myc) : 0u;
        while (xm) {
          const int j = __ffs(xm) - 1;
          xm &= xm - 1;
          const uint32_t wcj = __shfl_sync(FULL, wc, j);
          uint32_t found = NONE;
          for (uint32_t b0 = 0; b0 < P.L.Scta; b0 += 32) {
            const uint32_t jj = b0 + lane;
            const uint32_t hit = __ballot_sync(FULL, jj < P.L.Scta && P.cta(jj)[C_ID] == wcj);
            if (hit) {
              found = b0 + __ffs(hit) - 1;
              break;
            }
          }
          if (lane == j) tcs = found;
        }
        if (mine && !to_next) {
          if (tcs != NONE) {
            uint32_t *ts = P.slot(tcs * P.W + ((ew.y >> 1) & 127u));
            if ((ts[F_HID] & ID_MASK) == ew.x) {
              atomicSub(&ts[F_META], 256u);
              atomicMax(&ts[F_RDY], rel);
              to_head = true;
              cross = tcs != cs;
              if (EXT && cross) xs = div16(tcs, P.mCps);
            }
          }
        }
        adj_cnt += __reduce_add_sync(FULL, to_next ? 1u : 0u);
        adj_rdy = max(adj_rdy, __reduce_max_sync(FULL, to_next ? rel : 0u));
        cross_touch |= __any_sync(FULL, cross);
        uint32_t todo = __ballot_sync(FULL, mine && !to_next && !to_head);
        while (todo) {
          const int j = __ffs(todo) - 1;
          todo &= todo - 1;
          const uint32_t w = __shfl_sync(FULL, ew.x, j);
          const uint32_t r = __shfl_sync(FULL, rel, j);
          if (lane == 0) {
            uint2 *c = P.scr + (w - P.n0);
            red_keep(c, r, pol);
          }
        }
      }
      __syncwarp();
      if (lane == 0 && (cn.x | cn.y)) st_counters_zero_keep(P.scr + (nx - P.n0), pol);  // read once: leave the row clean
      cn.x = __shfl_sync(FULL, cn.x, 0);  // the next head's counters (its scratch row is not released into above)
      cn.y = __shfl_sync(FULL, cn.y, 0);
      set_head(P, i, nx, rn, qn, cn, adj_cnt, adj_rdy);
      __syncwarp();
      // ---- refresh keys and summaries the issue may have changed
      if (EXT && cross_touch && deg <= 32u) {  // releases reached heads of other CTAs: their SMs and this one
        r_sm<EXT, SPL>(P, sm, t, C.H, lane);
        bool own = (uint32_t)lane == (sm & 31u);
        uint32_t xm = __ballot_sync(FULL, xs != NONE && xs != sm);
        uint32_t done = sm;
        while (xm) {
          const int j = __ffs(xm) - 1;
          xm &= xm - 1;
          const uint32_t s2 = __shfl_sync(FULL, xs, j);
          if (s2 == done) continue;
          done = s2;
          r_sm<EXT, SPL>(P, s2, t, C.H, lane);
          own |= (uint32_t)lane == (s2 & 31u);
        }
        if (C.H != prevH) {  // and the SMs whose HBM heads the new horizon overtakes
          for (uint32_t s = lane; s < P.L.NS; s += 32) {
            if (r_stale<SPL>(P, s, C.H)) {
              r_rescan<EXT, SPL>(P, s, t, C.H);
              own = true;
            }
          }
        }
        if (EXT && noc_touch) {  // the group's other SMs may hold DSMEM heads keyed on that server
          const uint32_t g0 = div16(sm, P.mCsms) * P.L.csms, g1 = min(g0 + P.L.csms, P.L.NS);
          for (uint32_t s = g0 + lane; s < g1; s += 32) r_rescan<EXT, SPL>(P, s, t, C.H);
          __syncwarp();
          for (uint32_t s = g0; s < g1; s++) own |= (s & 31u) == (uint32_t)lane;
        }
        __syncwarp();
        if (own) b = r_lane_best<SPL>(P, lane, C.H, bsl);
      } else if (cross_touch) {  // a node with many successors: recompute everything
        for (uint32_t s = lane; s < P.L.NS; s += 32) r_rescan<EXT, SPL>(P, s, t, C.H);
        __syncwarp();
        b = r_lane_best<SPL>(P, lane, C.H, bsl);
      } else if (C.H == prevH && (SPL || P.L.per <= 16u) && P.L.NS <= 512u && !(EXT && P.L.nsub)) {
        r_sm_owner<EXT, SPL>(P, sm, t, C.H, lane, b, bsl);
        if (EXT && noc_touch) {  // the group's other SMs may hold DSMEM heads keyed on that server
          const uint32_t g0 = div16(sm, P.mCsms) * P.L.csms, g1 = min(g0 + P.L.csms, P.L.NS);
          for (uint32_t s = g0 + lane; s < g1; s += 32)
            if (s != sm) r_rescan<EXT, SPL>(P, s, t, C.H);
          __syncwarp();
          bool mine = false;
          for (uint32_t s = g0; s < g1; s++) mine |= s != sm && (s & 31u) == (uint32_t)lane;
          if (mine) b = r_lane_best<SPL>(P, lane, C.H, bsl);
        }
      } else {
        r_sm<EXT, SPL>(P, sm, t, C.H, lane);
        if (!SPL && C.H != prevH && P.L.per >= 8u && !(EXT && P.L.nsub)) {
          // SMs of many slots: one SM at a time, a slot per lane
          bool own = (uint32_t)lane == (sm & 31u);
          for (uint32_t s0 = 0; s0 < P.L.NS; s0 += 32) {
            const uint32_t s = s0 + lane;
            uint32_t xm = __ballot_sync(FULL, s < P.L.NS && s != sm && r_stale<SPL>(P, s, C.H));
            while (xm) {
              const uint32_t s2 = s0 + __ffs(xm) - 1;
              xm &= xm - 1;
              r_sm<EXT, SPL>(P, s2, t, C.H, lane);
              own |= (uint32_t)lane == (s2 & 31u);
            }
          }
          if (own) b = r_lane_best<SPL>(P, lane, C.H, bsl);
        } else if (SPL && C.H != prevH) {
          // split records: one pass per lane rescans its whole records that H
          // overtook and takes its best at the new H from every record it owns
          uint64_t nb = INF64;
          uint32_t ns = 0;
          for (uint32_t s = lane; s < P.L.NS; s += 32) {
            if (s != sm && r_stale<SPL>(P, s, C.H)) r_rescan<EXT, SPL>(P, s, t, C.H);
            uint32_t sl;
            const uint64_t v = split_sm_best(P, s, C.H, sl);
            if (v < nb) { nb = v; ns = sl; }
          }
          b = nb;
          bsl = ns;
        } else if (C.H != prevH) {
          // SMs whose HBM heads H overtakes change their effective cycles
          bool any = false;
          for (uint32_t s = lane; s < P.L.NS; s += 32) {
            if (s != sm && r_stale<SPL>(P, s, C.H)) {
              r_rescan<EXT, SPL>(P, s, t, C.H);
              any = true;
            }
          }
          // split records take the new H where they are read: every lane's best may move
          if (SPL || any || (uint32_t)lane == (sm & 31u)) b = r_lane_best<SPL>(P, lane, C.H, bsl);
        } else {
          r_owner<SPL>(P, sm & 31u, lane, C.H, b, bsl);
        }
        if (EXT && noc_touch) {  // the group's other SMs may hold DSMEM heads keyed on that server
          const uint32_t g0 = div16(sm, P.mCsms) * P.L.csms, g1 = min(g0 + P.L.csms, P.L.NS);
          for (uint32_t s = g0 + lane; s < g1; s += 32)
            if (s != sm) r_rescan<EXT, SPL>(P, s, t, C.H);
          __syncwarp();
          bool mine = false;  // this lane owns one of them
          for (uint32_t s = g0; s < g1; s++) mine |= s != sm && (s & 31u) == (uint32_t)lane;
          if (mine) b = r_lane_best<SPL>(P, lane, C.H, bsl);
        }
      }
      __syncwarp();
      if (rem == 0u) {
        if (cend <= t) {
          if (!launch_ctas<EXT, SPL>(g, P, C, cta_sm_row, lane, b, bsl)) { status = GTS_ERR_STEP_LIMIT; break; }
        } else {
          C.next_ret = min(C.next_ret, cend);
        }
      }
    }
    // leave the row clean: a point that stopped early may hold counters of
    // nodes that never became heads; the L2 list records are always used
    if (status != GTS_OK || l2on) {
      __threadfence();  // lane 0's releases and list updates come before the clears
      __syncwarp();
      uint4 *z = reinterpret_cast<uint4 *>(P.scr);
      const uint32_t nz = status != GTS_OK ? (nG + 1u) >> 1 : 0u;
      for (uint32_t k = lane; k < nz; k += 32) z[k] = make_uint4(0, 0, 0, 0);
      if (l2on)
        for (uint32_t k = lane; k < g.n_tiles; k += 32) l2t[k] = make_uint4(0, 0, 0, 0);
    }
    __threadfence();
    if (lane == 0) {
      d_status[q] = status;
      d_makespan[q] = status == GTS_OK ? mk : 0;
      if (want_digest) d_digest[q] = status == GTS_OK ? digest : 0ull;
    }
    if (d_busy && lane < GTS_BUSY_CLASSES) d_busy[(size_t)q * GTS_BUSY_CLASSES + lane] = status == GTS_OK ? (int64_t)busy : 0;
    __syncwarp();
  }
}

size_t align_up(size_t x) { return (x + 255) & ~(size_t)255; }

struct WsLayout {
  size_t rec, rng, succ, first, cnt, noff, coff, stat, chi, total;
};

// Status words of the device-side graph check (GK_* index: first offending
// node / edge / CTA, NONE if none), then its reductions.
enum : uint32_t {
  GK_ROWPTR = 0, GK_TYPE, GK_WARP, GK_CTA, GK_TILE, GK_EDGE, GK_KIND, GK_KERNEL, GK_INDEG, GK_NCHECKS,
  GK_CLASS = GK_NCHECKS, GK_CROSS,
  GK_SPAN_LO = 12, GK_SPAN_HI = 13,  // one 64-bit word: 8-byte aligned (the status block is 256-byte aligned)
  GK_WORDS = 16
};
static_assert(GK_CROSS < GK_SPAN_LO && GK_SPAN_LO % 2 == 0 && GK_SPAN_HI == GK_SPAN_LO + 1 && GK_SPAN_HI < GK_WORDS,
              "the span sum is an aligned 64-bit word after the other status words");

bool ws_layout(uint64_t n, uint64_t m, uint64_t C, uint64_t W, uint64_t G, WsLayout &w) {
  if (n >= 0x7FFFFFFEull || C >= (1ull << 24) || W < 1 || W > MAX_W || G < 1 || G > C + n + 1) return false;
  size_t o = 0;
  w.rec = o; o += align_up(n * 16);
  w.rng = o; o += align_up(n * 16);
  w.succ = o; o += align_up(m * 8);
  w.first = o; o += align_up(C * W * 4);
  w.cnt = o; o += align_up(C * 4);
  w.noff = o; o += align_up((G + 1) * 4);
  w.coff = o; o += align_up((G + 1) * 4);
  o += 256;
  // used only while gts_graph_create runs, zero afterwards
  w.stat = o; o += align_up(GK_WORDS * 4);
  w.chi = o; o += align_up(C * 4);
  w.total = o;
  return true;
}

// ---------------------------------------------------------------- device-side graph check and packing
// Graph of node / CTA x: the g with off[g] <= x < off[g+1] (off non-decreasing, off[0] = 0 <= x < off[G]).
__device__ __forceinline__ uint32_t graph_of(const uint32_t *off, uint32_t G, uint32_t x) {
  uint32_t lo = 0, hi = G;  // off[lo] <= x < off[hi]
  while (hi - lo > 1) {
    const uint32_t mid = (lo + hi) >> 1;
    if (off[mid] <= x) lo = mid; else hi = mid;
  }
  return lo;
}

struct GraphIn {  // the caller's arrays (gts_graph_desc)
  const uint32_t *row_ptr, *col, *cta, *work, *lx, *kern, *tile;
  const uint8_t *ek, *ty;
  const uint16_t *wp;
  uint32_t n, m, C, W, G, n_tiles;
};

// Contract checks of the Section 4.1 graph, one thread per node (edges of the
// node in the same thread).  Records the first offending index per check;
// touches memory only at indices it has checked.  Also counts in-degrees
// (into rng[].y), nodes per CTA, the first node of every (CTA, warp) stream
// and the last node of every CTA, and ORs the unit classes in use and whether
// an edge crosses CTAs.
__global__ void k_graph_check(GraphIn in, const uint32_t *noff, const uint32_t *coff, uint32_t *stat, uint4 *rng,
                              uint32_t *first, uint32_t *cnt, uint32_t *chi) {
  const uint32_t lane = threadIdx.x & 31u;
  uint32_t cls_or = 0u, cross = 0u;
  for (uint32_t v0 = blockIdx.x * blockDim.x; v0 < in.n; v0 += gridDim.x * blockDim.x) {
    const uint32_t v = v0 + threadIdx.x;
    if (v < in.n) {
      const uint32_t g = graph_of(noff, in.G, v);
      const uint32_t n1 = noff[g + 1], c0 = coff[g], c1 = coff[g + 1];
      const uint32_t a = in.row_ptr[v], b = in.row_ptr[v + 1];
      const bool rows_ok = a <= b && b <= in.m;
      if (!rows_ok) atomicMin(&stat[GK_ROWPTR], v);
      const uint32_t ty = in.ty[v], wp = in.wp[v], c = in.cta[v];
      if (ty > GTS_DSMEM) atomicMin(&stat[GK_TYPE], v);
      else {
        const uint32_t k = (TYPE_CLASS >> (4 * ty)) & 15u;
        if (k < RC_N) cls_or |= 1u << k;
        if (k == RC_DSM) cls_or |= (1u << RC_LSU) | CM_NOC;
      }
      if (wp >= in.W) atomicMin(&stat[GK_WARP], v);
      const bool cta_ok = c >= c0 && c < c1;
      if (!cta_ok) atomicMin(&stat[GK_CTA], v);
      if (in.tile && (ty == GTS_LOAD || ty == GTS_STORE) && in.tile[v] != NONE && in.tile[v] >= in.n_tiles)
        atomicMin(&stat[GK_TILE], v);
      if (cta_ok) {
        atomicAdd(&cnt[c], 1u);
        atomicMax(&chi[c], v);
        if (wp < in.W) atomicMin(&first[(size_t)c * in.W + wp], v);
      }
      if (rows_ok) {
        for (uint32_t x = a; x < b; x++) {
          const uint32_t w = in.col[x];
          if (w <= v || w >= n1) {
            atomicMin(&stat[GK_EDGE], x);
          } else {
            atomicAdd(&rng[w].y, 1u);
            if (in.cta[w] != c) cross = 1u;
          }
          if (in.ek[x] > 1u) atomicMin(&stat[GK_KIND], x);
        }
      }
    }
  }
  cls_or = __reduce_or_sync(FULL, cls_or);
  cross = __reduce_or_sync(FULL, cross);
  if (lane == 0) {
    if (cls_or) atomicOr(&stat[GK_CLASS], cls_or);
    if (cross) atomicOr(&stat[GK_CROSS], 1u);
  }
}

// Second pass, after every in-degree and stream head is known: in-degree
// limit per node, kernel ids non-decreasing within each graph per CTA, and
// the sum over CTAs of their id span (last - first node + 1), the work of the
// stream-link pass below.
__global__ void k_graph_check2(GraphIn in, const uint32_t *coff, uint32_t *stat, const uint4 *rng,
                               const uint32_t *first, const uint32_t *cnt, const uint32_t *chi) {
  unsigned long long span = 0ull;
  const uint32_t N = max(in.n, in.C);
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < N; i += gridDim.x * blockDim.x) {
    if (i < in.n && rng[i].y > MAX_INDEG) atomicMin(&stat[GK_INDEG], i);
    if (i < in.C) {
      if (i > 0 && graph_of(coff, in.G, i) == graph_of(coff, in.G, i - 1) && in.kern[i] < in.kern[i - 1])
        atomicMin(&stat[GK_KERNEL], i);
      if (cnt[i]) {
        uint32_t lo = NONE;
        for (uint32_t w = 0; w < in.W; w++) lo = min(lo, first[(size_t)i * in.W + w]);
        span += (unsigned long long)(chi[i] - lo) + 1ull;
      }
    }
  }
  for (int o = 16; o > 0; o >>= 1) span += __shfl_down_sync(FULL, span, o);
  if ((threadIdx.x & 31u) == 0 && span) {
    unsigned long long *s64 = reinterpret_cast<unsigned long long *>(stat + GK_SPAN_LO);
    atomicAdd(s64, span);
  }
}

// Packed node records, ranges and successor entries (the layout k_simulate
// reads), one thread per node.  The stream link (rec.z) is filled by
// k_graph_streams.
__global__ void k_graph_pack(GraphIn in, uint4 *rec, uint4 *rng, uint2 *succ) {
  for (uint32_t v = blockIdx.x * blockDim.x + threadIdx.x; v < in.n; v += gridDim.x * blockDim.x) {
    const uint32_t a = in.row_ptr[v], b = in.row_ptr[v + 1], ty = in.ty[v];
    const uint32_t indeg = rng[v].y;
    const bool tiled = in.tile && in.tile[v] != NONE && (ty == GTS_LOAD || ty == GTS_STORE);
    rec[v] = make_uint4(in.work[v], in.lx[v], NONE, ty | (indeg << 4));
    rng[v] = make_uint4(tiled ? in.tile[v] + 1u : 0u, 0u, a, b);
    for (uint32_t x = a; x < b; x++) {
      const uint32_t w = in.col[x];
      succ[x] = make_uint2(w, (uint32_t)in.ek[x] | ((uint32_t)in.wp[w] << 1) | (in.cta[w] << 8));
    }
  }
}

// Program order of every (CTA, warp) stream (Section 5.1: each warp issues its
// nodes in ascending id): rec[v].z = the next node of v's stream.  One warp
// per CTA walks the CTA's id span downwards, 32 ids at a time; lanes holding
// nodes of the CTA group by warp (match), each takes the next higher lane of
// its group, and the group's lowest lane leaves its id for the chunk below.
__global__ void k_graph_streams(GraphIn in, const uint32_t *first, const uint32_t *cnt, const uint32_t *chi,
                                uint4 *rec) {
  extern __shared__ uint32_t carry_all[];  // W per warp
  const uint32_t lane = threadIdx.x & 31u, wib = threadIdx.x >> 5, wpb = blockDim.x >> 5;
  uint32_t *carry = carry_all + wib * in.W;
  for (uint32_t c = blockIdx.x * wpb + wib; c < in.C; c += gridDim.x * wpb) {
    if (cnt[c] == 0u) continue;
    uint32_t lo = NONE;
    for (uint32_t w = lane; w < in.W; w += 32) {
      carry[w] = NONE;
      lo = min(lo, first[(size_t)c * in.W + w]);
    }
    lo = __reduce_min_sync(FULL, lo);
    const uint32_t hi = chi[c];
    __syncwarp();
    for (uint32_t top = hi + 1u; top > lo;) {
      const uint32_t base = top - lo >= 32u ? top - 32u : lo;
      const uint32_t v = base + lane;
      const bool mine = v < top && in.cta[v] == c;
      const uint32_t key = mine ? (uint32_t)in.wp[v] : NONE;
      const uint32_t peers = __match_any_sync(FULL, key);
      if (mine) {
        const uint32_t higher = peers & ~((2u << lane) - 1u);
        rec[v].z = higher ? base + (uint32_t)__ffs(higher) - 1u : carry[key];
      }
      __syncwarp();
      if (mine && lane == (uint32_t)__ffs(peers) - 1u) carry[key] = v;
      __syncwarp();
      top = base;
    }
  }
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
  std::vector<uint8_t> sched;   // per row: asks for a per-subpartition issue policy or the L2 model
  std::vector<double> cost;     // per row: estimated simulation cost (0 for invalid rows)
  std::vector<uint8_t> wide;    // per row: SMs of 8 or more warp slots (no split SM records)
  const uint32_t *d_order = nullptr;  // processing order (gts_params_set_order), borrowed
};

struct gts_results {
  int32_t *d_makespan, *d_status;
  uint64_t *d_digest;
  uint32_t n_points;
  cudaStream_t stream;
};

namespace {

// The library's handle over a packed workspace.
gts_status make_handle(const WsLayout &wl, char *ws, uint64_t n, uint64_t m, uint64_t C, uint64_t W, uint64_t G,
                       const std::vector<uint32_t> &noff, const std::vector<uint32_t> &coff, const uint32_t *d_kernel,
                       uint32_t row_nodes, uint32_t row_ctas, uint32_t cross, uint32_t class_mask, uint32_t n_tiles,
                       gts_graph **out) {
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
  dg.stream_first = (const uint32_t *)(ws + wl.first);
  dg.cta_cnt = (const uint32_t *)(ws + wl.cnt);
  dg.cta_kernel = d_kernel;
  dg.node_off = (const uint32_t *)(ws + wl.noff);
  dg.cta_off = (const uint32_t *)(ws + wl.coff);
  dg.W = (uint32_t)W;
  dg.G = (uint32_t)G;
  dg.row_nodes = row_nodes;
  dg.row_ctas = row_ctas;
  dg.cross_cta = cross;
  dg.class_mask = class_mask;
  dg.n_tiles = n_tiles;
  *out = g;
  return GTS_OK;
}

// Expansion tables of a template-shared graph, after the packed graph.
struct TplLayout {
  size_t base, ebase, indeg, next, first, total;
};

bool tpl_layout(uint64_t T, uint64_t TN, uint64_t n, uint64_t m, uint64_t C, uint64_t W, uint64_t G, WsLayout &w,
                TplLayout &x) {
  if (!ws_layout(n, m, C, W, G, w) || T < 1 || T > TN + 1 || TN >= 0x7FFFFFFEull) return false;
  size_t o = w.total;
  x.base = o; o += align_up(C * 4);
  x.ebase = o; o += align_up(C * 4);
  x.indeg = o; o += align_up(TN * 4);
  x.next = o; o += align_up(TN * 4);
  x.first = o; o += align_up(T * W * 4);
  x.total = o;
  return true;
}

// One block per logical CTA (grid-stride): copy its template's nodes and
// edges into the packed arrays at the CTA's node and edge base, turning
// template indices into logical ids.
__global__ void k_expand(const uint32_t *__restrict__ cta_tpl, const uint32_t *__restrict__ tpl_off,
                         const uint32_t *__restrict__ row_ptr, const uint32_t *__restrict__ col,
                         const uint8_t *__restrict__ ek, const uint8_t *__restrict__ ty,
                         const uint16_t *__restrict__ wp, const uint32_t *__restrict__ work,
                         const uint32_t *__restrict__ lx, const uint32_t *__restrict__ cbase,
                         const uint32_t *__restrict__ cebase, const uint32_t *__restrict__ tindeg,
                         const uint32_t *__restrict__ tnext, const uint32_t *__restrict__ tfirst, uint32_t C, uint32_t W,
                         uint4 *rec, uint4 *rng, uint2 *succ, uint32_t *first, uint32_t *cnt) {
  for (uint32_t c = blockIdx.x; c < C; c += gridDim.x) {
    const uint32_t t = cta_tpl[c], u0 = tpl_off[t], u1 = tpl_off[t + 1];
    const uint32_t base = cbase[c], eb = cebase[c], x0 = row_ptr[u0];
    for (uint32_t u = u0 + threadIdx.x; u < u1; u += blockDim.x) {
      const uint32_t v = base + (u - u0), nx = tnext[u];
      rec[v] = make_uint4(work[u], lx[u], nx == NONE ? NONE : base + (nx - u0), (uint32_t)ty[u] | (tindeg[u] << 4));
      const uint32_t a = row_ptr[u], b = row_ptr[u + 1];
      rng[v] = make_uint4(0u, 0u, eb + (a - x0), eb + (b - x0));
      for (uint32_t x = a; x < b; x++) {
        const uint32_t w = col[x];
        succ[eb + (x - x0)] = make_uint2(base + (w - u0), (uint32_t)ek[x] | ((uint32_t)wp[w] << 1) | (c << 8));
      }
    }
    for (uint32_t w = threadIdx.x; w < W; w += blockDim.x) {
      const uint32_t f = tfirst[(size_t)t * W + w];
      first[(size_t)c * W + w] = f == NONE ? NONE : base + (f - u0);
    }
    if (threadIdx.x == 0) cnt[c] = u1 - u0;
  }
}

}  // namespace

extern "C" {

const char *gts_last_error(void) { return g_err; }

size_t gts_graph_workspace_bytes(uint32_t n_nodes, uint32_t n_edges, uint32_t n_ctas, uint32_t warps_per_cta,
                                 uint32_t n_graphs) {
  WsLayout w;
  if (!ws_layout(n_nodes, n_edges, n_ctas, warps_per_cta, n_graphs, w)) return 0;
  return w.total;
}

uint32_t gts_row_nodes(const gts_graph *g) { return g ? g->dg.row_nodes : 0u; }
uint32_t gts_row_ctas(const gts_graph *g) { return g ? g->dg.row_ctas : 0u; }

gts_status gts_graph_create(const gts_graph_desc *d, void *stream, gts_graph **out) {
  clear_error();
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
  if ((uintptr_t)d->workspace % 16 != 0) return fail(GTS_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
  if (d->workspace_bytes < wl.total)
    return fail(GTS_ERR_NOMEM, "workspace too small: need " + std::to_string(wl.total) + " bytes");
  if (d->tile && (d->n_tiles == 0 || d->n_tiles > (1u << 28)))
    return fail(GTS_ERR_INVALID_ARG, "tiles need 1 <= n_tiles <= 2^28");
  cudaStream_t s = (cudaStream_t)stream;
  char *ws = (char *)d->workspace;
  // ---- the graph offsets and the ends of row_ptr come to the host (a few words)
  std::vector<uint32_t> noff, coff, ends;
  cudaError_t e = d2h(ends, d->row_ptr, 1, s);
  uint32_t last = 0;
  if (e == cudaSuccess) e = cudaMemcpyAsync(&last, d->row_ptr + n, 4, cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) {
    if (G > 1 || d->graph_node_off) e = d2h(noff, d->graph_node_off, G + 1, s);
    else noff = {0u, (uint32_t)n};
  }
  if (e == cudaSuccess) {
    if (G > 1 || d->graph_cta_off) e = d2h(coff, d->graph_cta_off, G + 1, s);
    else coff = {0u, (uint32_t)C};
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "graph_create: copy offsets to host");
  if (noff[0] != 0 || noff[G] != n || coff[0] != 0 || coff[G] != C)
    return fail(GTS_ERR_INVALID_GRAPH, "graph offsets must start at 0 and end at n_nodes / n_ctas");
  for (uint64_t k = 0; k < G; k++)
    if (noff[k + 1] < noff[k] || coff[k + 1] < coff[k])
      return fail(GTS_ERR_INVALID_GRAPH, "graph offsets decrease at graph " + std::to_string(k));
  if (ends[0] != 0 || last != m) return fail(GTS_ERR_INVALID_GRAPH, "row_ptr[0] != 0 or row_ptr[n] != n_edges");
  uint32_t row_nodes = 0, row_ctas = 0;
  for (uint64_t k = 0; k < G; k++) {
    row_nodes = std::max(row_nodes, noff[k + 1] - noff[k]);
    row_ctas = std::max(row_ctas, coff[k + 1] - coff[k]);
  }

  // ---- contract checks on the device (Section 4.1 graph): one status read back
  GraphIn in;
  in.row_ptr = d->row_ptr; in.col = d->col; in.cta = d->cta; in.work = d->work; in.lx = d->lat_extra;
  in.kern = d->cta_kernel; in.tile = d->tile; in.ek = d->ekind; in.ty = d->type; in.wp = d->warp;
  in.n = (uint32_t)n; in.m = (uint32_t)m; in.C = (uint32_t)C; in.W = (uint32_t)W; in.G = (uint32_t)G;
  in.n_tiles = d->tile ? d->n_tiles : 0u;
  uint32_t *stat = (uint32_t *)(ws + wl.stat);
  uint32_t *chi = (uint32_t *)(ws + wl.chi);
  uint32_t *first = (uint32_t *)(ws + wl.first);
  uint32_t *cnt = (uint32_t *)(ws + wl.cnt);
  uint4 *rec = (uint4 *)(ws + wl.rec);
  uint4 *rng = (uint4 *)(ws + wl.rng);
  const uint32_t *d_noff = (const uint32_t *)(ws + wl.noff), *d_coff = (const uint32_t *)(ws + wl.coff);
  auto up = [&](size_t off, const void *src, size_t bytes) {
    if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(ws + off, src, bytes, cudaMemcpyHostToDevice, s);
  };
  auto zero = [&](size_t off, int value, size_t bytes) {
    if (e == cudaSuccess && bytes) e = cudaMemsetAsync(ws + off, value, bytes, s);
  };
  up(wl.noff, noff.data(), (G + 1) * 4);
  up(wl.coff, coff.data(), (G + 1) * 4);
  zero(wl.stat, 0xFF, GK_NCHECKS * 4);
  zero(wl.stat + GK_NCHECKS * 4, 0, (GK_WORDS - GK_NCHECKS) * 4);
  zero(wl.rng, 0, n * 16);
  zero(wl.first, 0xFF, C * W * 4);
  zero(wl.cnt, 0, C * 4);
  zero(wl.chi, 0, C * 4);
  int dev = 0, sms = 1;
  if (e == cudaSuccess) e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const uint32_t grid = (uint32_t)std::max<int>(1, sms * 8);
  if (e == cudaSuccess && n) {
    k_graph_check<<<grid, 256, 0, s>>>(in, d_noff, d_coff, stat, rng, first, cnt, chi);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess && (n || C)) {
    k_graph_check2<<<grid, 256, 0, s>>>(in, d_coff, stat, rng, first, cnt, chi);
    e = cudaGetLastError();
  }
  uint32_t st[GK_WORDS];
  if (e == cudaSuccess) e = cudaMemcpyAsync(st, stat, sizeof(st), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "graph_create: device checks");
  static const char *what[GK_NCHECKS] = {"row_ptr decreases or exceeds n_edges at node ", "bad type at node ",
                                         "warp >= warps_per_cta at node ", "cta outside its graph at node ",
                                         "tile >= n_tiles at node ",
                                         "edge must go forward inside its graph: edge ",
                                         "bad edge kind at edge ", "cta_kernel decreases at CTA ",
                                         "more than 2^24-1 predecessors at node "};
  for (uint32_t k = 0; k < GK_NCHECKS; k++)
    if (st[k] != NONE)
      return fail(k == GK_INDEG ? GTS_ERR_UNSUPPORTED : GTS_ERR_INVALID_GRAPH, what[k] + std::to_string(st[k]));

  // ---- packing and stream links on the device
  if (n) {
    k_graph_pack<<<grid, 256, 0, s>>>(in, rec, rng, (uint2 *)(ws + wl.succ));
    e = cudaGetLastError();
  }
  const uint64_t span = (uint64_t)st[GK_SPAN_LO] | (uint64_t)st[GK_SPAN_HI] << 32;
  if (e == cudaSuccess && n && span <= 32ull * n + (1ull << 22)) {
    const uint32_t wpb = 8;
    k_graph_streams<<<(uint32_t)std::min<uint64_t>((C + wpb - 1) / wpb, 65535), wpb * 32, wpb * W * 4, s>>>(
        in, first, cnt, chi, rec);
    e = cudaGetLastError();
  } else if (e == cudaSuccess && n) {
    // CTAs interleave over long id ranges (rare): link the streams on the
    // host from the CTA and warp of every node, then patch the packed records
    std::vector<uint32_t> hc;
    std::vector<uint16_t> hw;
    std::vector<uint4> hrec;
    e = d2h(hc, d->cta, n, s);
    if (e == cudaSuccess) e = d2h(hw, d->warp, n, s);
    if (e == cudaSuccess) e = d2h(hrec, (const uint4 *)rec, n, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e == cudaSuccess) {
      std::vector<uint32_t> head(C * W, NONE);
      for (uint64_t v = n; v-- > 0;) {
        const uint64_t key = (uint64_t)hc[v] * W + hw[v];
        hrec[v].z = head[key];
        head[key] = (uint32_t)v;
      }
      e = cudaMemcpyAsync(rec, hrec.data(), n * 16, cudaMemcpyHostToDevice, s);
      if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    }
  }
  // the check's temporaries back to zero (the workspace past the packed graph reads as zeros)
  zero(wl.stat, 0, wl.total - wl.stat);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "graph_create: packing");
  return make_handle(wl, ws, n, m, C, W, G, noff, coff, d->cta_kernel, row_nodes, row_ctas, st[GK_CROSS] ? 1u : 0u,
                     st[GK_CLASS], d->tile ? d->n_tiles : 0u, out);
}

size_t gts_template_workspace_bytes(uint32_t n_templates, uint32_t n_tpl_nodes, uint32_t n_nodes, uint32_t n_edges,
                                    uint32_t n_ctas, uint32_t warps_per_cta, uint32_t n_graphs) {
  WsLayout w;
  TplLayout x;
  if (!tpl_layout(n_templates, n_tpl_nodes, n_nodes, n_edges, n_ctas, warps_per_cta, n_graphs, w, x)) return 0;
  return x.total;
}

gts_status gts_graph_create_templated(const gts_template_desc *d, void *stream, gts_graph **out) {
  clear_error();
  if (!d || !out) return fail(GTS_ERR_INVALID_ARG, "null desc or out");
  *out = nullptr;
  const uint64_t T = d->n_templates, TN = d->n_tpl_nodes, TE = d->n_tpl_edges;
  const uint64_t n = d->n_nodes, m = d->n_edges, C = d->n_ctas, W = d->warps_per_cta, G = d->n_graphs;
  WsLayout wl;
  TplLayout xl;
  if (!tpl_layout(T, TN, n, m, C, W, G, wl, xl) || TE >= 0xFFFFFFFFull)
    return fail(GTS_ERR_INVALID_ARG, "size out of range (1 <= templates, n < 2^31-1, C < 2^24, 1 <= W <= 128)");
  if (!d->tpl_node_off || !d->tpl_row_ptr || (TN && (!d->tpl_type || !d->tpl_warp || !d->tpl_work || !d->tpl_lat_extra)) ||
      (TE && (!d->tpl_col || !d->tpl_ekind)) || (C && (!d->cta_template || !d->cta_kernel)))
    return fail(GTS_ERR_INVALID_ARG, "null template array");
  if (G > 1 && !d->graph_cta_off) return fail(GTS_ERR_INVALID_ARG, "stacked set needs graph_cta_off");
  if (!d->workspace) return fail(GTS_ERR_INVALID_ARG, "null workspace");
  if ((uintptr_t)d->workspace % 16 != 0) return fail(GTS_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
  if (d->workspace_bytes < xl.total)
    return fail(GTS_ERR_NOMEM, "workspace too small: need " + std::to_string(xl.total) + " bytes");
  cudaStream_t s = (cudaStream_t)stream;
  std::vector<uint32_t> toff, row_ptr, col, work, lx, ctpl, kern, coff;
  std::vector<uint8_t> ek, ty;
  std::vector<uint16_t> wp;
  cudaError_t e = cudaSuccess;
  if (e == cudaSuccess) e = d2h(toff, d->tpl_node_off, T + 1, s);
  if (e == cudaSuccess) e = d2h(row_ptr, d->tpl_row_ptr, TN + 1, s);
  if (e == cudaSuccess) e = d2h(col, d->tpl_col, TE, s);
  if (e == cudaSuccess) e = d2h(ek, d->tpl_ekind, TE, s);
  if (e == cudaSuccess) e = d2h(ty, d->tpl_type, TN, s);
  if (e == cudaSuccess) e = d2h(wp, d->tpl_warp, TN, s);
  if (e == cudaSuccess) e = d2h(work, d->tpl_work, TN, s);
  if (e == cudaSuccess) e = d2h(lx, d->tpl_lat_extra, TN, s);
  if (e == cudaSuccess) e = d2h(ctpl, d->cta_template, C, s);
  if (e == cudaSuccess) e = d2h(kern, d->cta_kernel, C, s);
  if (e == cudaSuccess) {
    if (G > 1 || d->graph_cta_off) e = d2h(coff, d->graph_cta_off, G + 1, s);
    else coff = {0u, (uint32_t)C};
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "graph_create_templated: copy to host");

  // ---- contract on the templates
  if (toff[0] != 0 || toff[T] != TN) return fail(GTS_ERR_INVALID_GRAPH, "tpl_node_off must run from 0 to n_tpl_nodes");
  if (row_ptr[0] != 0 || row_ptr[TN] != TE) return fail(GTS_ERR_INVALID_GRAPH, "tpl_row_ptr must run from 0 to n_tpl_edges");
  std::vector<uint32_t> tmask(T, 0u), tindeg(TN, 0u), tnext(TN, NONE), tfirst(T * W, NONE);
  for (uint64_t t = 0; t < T; t++) {
    if (toff[t + 1] < toff[t]) return fail(GTS_ERR_INVALID_GRAPH, "tpl_node_off decreases at template " + std::to_string(t));
    const uint32_t u0 = toff[t], u1 = toff[t + 1];
    for (uint32_t u = u0; u < u1; u++) {
      if (row_ptr[u + 1] < row_ptr[u]) return fail(GTS_ERR_INVALID_GRAPH, "tpl_row_ptr decreases at node " + std::to_string(u));
      if (ty[u] > GTS_DSMEM) return fail(GTS_ERR_INVALID_GRAPH, "bad type at template node " + std::to_string(u));
      if (wp[u] >= W) return fail(GTS_ERR_INVALID_GRAPH, "warp >= warps_per_cta at template node " + std::to_string(u));
      const uint32_t cls_v = (TYPE_CLASS >> (4 * ty[u])) & 15u;
      if (cls_v < RC_N) tmask[t] |= 1u << cls_v;
      if (cls_v == RC_DSM) tmask[t] |= (1u << RC_LSU) | CM_NOC;
      for (uint32_t x = row_ptr[u]; x < row_ptr[u + 1]; x++) {
        if (col[x] <= u || col[x] >= u1)
          return fail(GTS_ERR_INVALID_GRAPH, "template edge " + std::to_string(x) + " must go forward inside its template");
        if (ek[x] > 1) return fail(GTS_ERR_INVALID_GRAPH, "bad edge kind at template edge " + std::to_string(x));
        if (++tindeg[col[x]] > MAX_INDEG)
          return fail(GTS_ERR_UNSUPPORTED, "template node " + std::to_string(col[x]) + " has more than 2^24-1 predecessors");
      }
    }
    for (uint32_t u = u1; u-- > u0;) {  // program order of each warp stream: ascending
      tnext[u] = tfirst[t * W + wp[u]];
      tfirst[t * W + wp[u]] = u;
    }
  }
  // ---- the CTA table: node and edge bases (CTA-major), graph ranges
  if (coff[0] != 0 || coff[G] != C) return fail(GTS_ERR_INVALID_GRAPH, "graph_cta_off must run from 0 to n_ctas");
  std::vector<uint32_t> cbase(C), cebase(C), noff(G + 1);
  uint64_t nb = 0, eb = 0;
  uint32_t row_nodes = 0, row_ctas = 0, class_mask = 0;
  for (uint64_t k = 0; k < G; k++) {
    if (coff[k + 1] < coff[k]) return fail(GTS_ERR_INVALID_GRAPH, "graph_cta_off decreases at graph " + std::to_string(k));
    noff[k] = (uint32_t)nb;
    for (uint32_t c = coff[k]; c < coff[k + 1]; c++) {
      const uint32_t t = ctpl[c];
      if (t >= T) return fail(GTS_ERR_INVALID_GRAPH, "cta_template out of range at CTA " + std::to_string(c));
      if (c > coff[k] && kern[c] < kern[c - 1])
        return fail(GTS_ERR_INVALID_GRAPH, "cta_kernel decreases at CTA " + std::to_string(c));
      cbase[c] = (uint32_t)nb;
      cebase[c] = (uint32_t)eb;
      nb += toff[t + 1] - toff[t];
      eb += row_ptr[toff[t + 1]] - row_ptr[toff[t]];
      class_mask |= tmask[t];
      if (nb > n || eb > m) return fail(GTS_ERR_INVALID_GRAPH, "templates hold more nodes or edges than n_nodes / n_edges");
    }
    row_nodes = std::max(row_nodes, (uint32_t)(nb - noff[k]));
    row_ctas = std::max(row_ctas, coff[k + 1] - coff[k]);
  }
  noff[G] = (uint32_t)nb;
  if (nb != n || eb != m) return fail(GTS_ERR_INVALID_GRAPH, "n_nodes / n_edges differ from the templates' totals");

  // ---- tables to the device, then the expansion
  char *ws = (char *)d->workspace;
  auto up = [&](size_t off, const void *src, size_t bytes) {
    if (e == cudaSuccess && bytes) e = cudaMemcpyAsync(ws + off, src, bytes, cudaMemcpyHostToDevice, s);
  };
  up(xl.base, cbase.data(), C * 4);
  up(xl.ebase, cebase.data(), C * 4);
  up(xl.indeg, tindeg.data(), TN * 4);
  up(xl.next, tnext.data(), TN * 4);
  up(xl.first, tfirst.data(), T * W * 4);
  up(wl.noff, noff.data(), (G + 1) * 4);
  up(wl.coff, coff.data(), (G + 1) * 4);
  if (e == cudaSuccess && C) {
    const uint32_t blocks = (uint32_t)std::min<uint64_t>(C, 65535);
    k_expand<<<blocks, 256, 0, s>>>(d->cta_template, d->tpl_node_off, d->tpl_row_ptr, d->tpl_col, d->tpl_ekind,
                                    d->tpl_type, d->tpl_warp, d->tpl_work, d->tpl_lat_extra,
                                    (const uint32_t *)(ws + xl.base), (const uint32_t *)(ws + xl.ebase),
                                    (const uint32_t *)(ws + xl.indeg), (const uint32_t *)(ws + xl.next),
                                    (const uint32_t *)(ws + xl.first), (uint32_t)C, (uint32_t)W, (uint4 *)(ws + wl.rec),
                                    (uint4 *)(ws + wl.rng), (uint2 *)(ws + wl.succ), (uint32_t *)(ws + wl.first),
                                    (uint32_t *)(ws + wl.cnt));
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "graph_create_templated: expansion");
  return make_handle(wl, ws, n, m, C, W, G, noff, coff, d->cta_kernel, row_nodes, row_ctas, 0u, class_mask, 0u, out);
}

gts_status gts_graph_destroy(gts_graph *g) {
  delete g;
  return GTS_OK;
}

gts_status gts_params_upload(gts_graph *g, const int32_t *d_params, uint32_t n_points, void *stream,
                             gts_params **out) {
  clear_error();
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
  P->sched.assign(n_points, 0u);
  P->cost.assign(n_points, 0.0);
  P->wide.assign(n_points, 0);
  for (uint32_t p = 0; p < n_points; p++) {
    const int32_t *row = h.data() + (size_t)p * GTS_NPARAM;
    if (check_row(row, g->G, g->dg.class_mask) != GTS_OK) continue;
    P->sched[p] = row[GTS_P_ISSUE_POLICY] != GTS_POLICY_LOWEST_ID || row[GTS_P_L2_BYTES] != 0;
    const uint32_t gi = (uint32_t)row[GTS_P_GRAPH_INDEX];
    Layout L;
    if (make_layout(row, g->cta_off[gi + 1] - g->cta_off[gi], g->W, g->dg.class_mask, L)) {
      P->words[p] = L.words;
      P->wide[p] = L.per >= 8u;
      // per issue the work grows slowly with the simulated SMs; the extended model costs about 3.5x
      P->cost[p] = (double)(g->node_off[gi + 1] - g->node_off[gi]) * (743.0 + L.NS) * (P->sched[p] ? 3.5 : 1.0);
    }
  }
  *out = P;
  return GTS_OK;
}

gts_status gts_params_set_order(gts_params *P, uint32_t *d_order, void *stream) {
  clear_error();
  if (!P || (P->n_points && !d_order)) return fail(GTS_ERR_INVALID_ARG, "null params or order");
  std::vector<uint32_t> order(P->n_points);
  for (uint32_t p = 0; p < P->n_points; p++) order[p] = p;
  std::stable_sort(order.begin(), order.end(), [&](uint32_t a, uint32_t b) { return P->cost[a] > P->cost[b]; });
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e = cudaSuccess;
  if (P->n_points) e = cudaMemcpyAsync(d_order, order.data(), (size_t)P->n_points * 4, cudaMemcpyHostToDevice, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "params_set_order: copy to device");
  P->d_order = d_order;
  return GTS_OK;
}

gts_status gts_params_destroy(gts_params *p) {
  delete p;
  return GTS_OK;
}

namespace {
// Per-warp scratch: one (released-predecessor count, max release cycle) pair
// per node of the largest graph, rounded to 16 bytes.
// ... plus, for a graph with tiles, one 16-byte L2 list record per tile.
// At least 16 bytes, so that a graph without nodes still has a row size to divide by.
uint64_t scratch_row_bytes(const gts_graph *g) {
  return std::max<uint64_t>(16, (((uint64_t)g->dg.row_nodes + 1) & ~1ull) * 8 + 16ull * g->dg.n_tiles);
}

struct Plan {
  uint32_t words, wpb, smem, blocks, warps;
  bool sched;  // launch the extended instance (issue policies, NoC, L2)
  bool split;  // plain instance with split SM records (every row's SMs have fewer than 8 slots)
};

gts_status plan_launch(const gts_graph *g, const gts_params *P, uint32_t first, uint32_t np, uint32_t flags,
                       size_t scratch_bytes, bool limit_by_scratch, Plan &pl) {
  (void)flags;
  uint32_t words = 64;
  pl.sched = false;
  bool wide = false;
  for (uint32_t p = first; p < first + np; p++) {
    words = std::max(words, P->words[p]);
    pl.sched = pl.sched || P->sched[p];
    wide = wide || P->wide[p];
  }
  pl.sched = pl.sched || (g->dg.class_mask & CM_NOC) != 0u;
  pl.split = !pl.sched && !wide;
  const uint32_t bytes = words * 4;
  pl.words = words;
  const void *kern = pl.sched ? (const void *)k_simulate<true, false>
                   : pl.split ? (const void *)k_simulate<false, true> : (const void *)k_simulate<false, false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)MAX_SMEM_BYTES);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
  int dev = 0, sms = 0;
  if (e == cudaSuccess) e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_fail(e, "simulate: kernel attributes");
  // warps per block: whichever keeps the most design points resident per SM
  uint32_t best_w = 0;
  pl.wpb = 1;
  for (uint32_t wpb = MAX_WPB; wpb >= 1; wpb--) {
    if (wpb * bytes > MAX_SMEM_BYTES) continue;
    int nb = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kern, (int)wpb * 32, wpb * bytes);
    if (e != cudaSuccess) return cuda_fail(e, "simulate: occupancy query");
    if ((uint32_t)nb * wpb > best_w) {
      best_w = (uint32_t)nb * wpb;
      pl.wpb = wpb;
    }
  }
  uint64_t warps = (uint64_t)std::max(best_w, 1u) * sms;
  // a batch smaller than one wave: one design point per block, so that the
  // block scheduler (which fills SMs breadth first) spreads the points evenly
  if (np < warps) pl.wpb = 1u;
  warps = std::min<uint64_t>(warps, np);
  if (limit_by_scratch) {
    const uint64_t row = scratch_row_bytes(g);
    const uint64_t fit = scratch_bytes > GTS_SCRATCH_HEADER_BYTES ? (scratch_bytes - GTS_SCRATCH_HEADER_BYTES) / row : 0;
    if (fit == 0) return fail(GTS_ERR_NOMEM, "scratch smaller than one design point's counter row");
    warps = std::min(warps, fit);
  }
  pl.warps = (uint32_t)std::max<uint64_t>(warps, 1);
  pl.wpb = std::min(pl.wpb, pl.warps);
  pl.smem = pl.wpb * bytes;
  pl.blocks = (pl.warps + pl.wpb - 1) / pl.wpb;
  return GTS_OK;
}
}  // namespace

size_t gts_scratch_bytes(const gts_graph *g, const gts_params *P, uint32_t flags) {
  if (!g || !P) return 0;
  Plan pl;
  if (plan_launch(g, P, 0, P->n_points, flags, 0, false, pl) != GTS_OK) return 0;
  return GTS_SCRATCH_HEADER_BYTES + (size_t)pl.warps * scratch_row_bytes(g);
}

gts_status gts_simulate_batch(gts_graph *g, gts_params *P, uint32_t first_point, uint32_t n_points, uint32_t flags,
                              int32_t *d_start, int32_t *d_finish, int32_t *d_makespan, int32_t *d_status,
                              uint64_t *d_digest, int32_t *d_cta_sm, int64_t *d_busy, void *d_scratch,
                              size_t scratch_bytes, void *stream, gts_results **out) {
  clear_error();
  if (out) *out = nullptr;
  if (!g || !P || P->graph != g) return fail(GTS_ERR_INVALID_ARG, "null or mismatched graph / params");
  if (flags & ~(GTS_FULL_TRACE | GTS_WANT_DIGEST | GTS_WANT_CTA_SM | GTS_WANT_BUSY | GTS_SCRATCH_CLEAN))
    return fail(GTS_ERR_INVALID_ARG, "unknown flag");
  if ((uint64_t)first_point + n_points > P->n_points) return fail(GTS_ERR_INVALID_ARG, "point range outside the table");
  if (!d_makespan || !d_status) return fail(GTS_ERR_INVALID_ARG, "d_makespan and d_status are required");
  if ((flags & GTS_FULL_TRACE) && g->dg.row_nodes && (!d_start || !d_finish))
    return fail(GTS_ERR_INVALID_ARG, "FULL_TRACE needs d_start and d_finish");
  if ((flags & GTS_WANT_DIGEST) && !d_digest) return fail(GTS_ERR_INVALID_ARG, "WANT_DIGEST needs d_digest");
  if ((flags & GTS_WANT_CTA_SM) && g->dg.row_ctas && !d_cta_sm) return fail(GTS_ERR_INVALID_ARG, "WANT_CTA_SM needs d_cta_sm");
  if ((flags & GTS_WANT_BUSY) && !d_busy) return fail(GTS_ERR_INVALID_ARG, "WANT_BUSY needs d_busy");
  if ((flags & GTS_WANT_BUSY) && (uintptr_t)d_busy % 8 != 0) return fail(GTS_ERR_INVALID_ARG, "d_busy must be 8-byte aligned");
  if (!d_scratch) return fail(GTS_ERR_NOMEM, "scratch required (gts_scratch_bytes)");
  if ((uintptr_t)d_scratch % 16 != 0) return fail(GTS_ERR_INVALID_ARG, "scratch must be 16-byte aligned");
  cudaStream_t s = (cudaStream_t)stream;
  if (n_points) {
    Plan pl;
    gts_status st = plan_launch(g, P, first_point, n_points, flags, scratch_bytes, true, pl);
    if (st != GTS_OK) return st;
    if (P->d_order) {  // the next-point counter
      const cudaError_t em = cudaMemsetAsync(d_scratch, 0, GTS_SCRATCH_HEADER_BYTES, s);
      if (em != cudaSuccess) return cuda_fail(em, "simulate: clear the point counter");
    }
    auto kern = pl.sched ? k_simulate<true, false> : pl.split ? k_simulate<false, true> : k_simulate<false, false>;
    kern<<<pl.blocks, pl.wpb * 32, pl.smem, s>>>(
        g->dg, P->d_params, first_point, n_points, flags, d_start, d_finish, d_makespan, d_status,
        (flags & GTS_WANT_DIGEST) ? d_digest : nullptr, (flags & GTS_WANT_CTA_SM) ? d_cta_sm : nullptr,
        (flags & GTS_WANT_BUSY) ? d_busy : nullptr, (uint2 *)d_scratch, pl.warps, pl.words, P->d_order,
        P->d_order ? P->n_points : 0u);
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
  clear_error();
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

// ----------------------------------------------------------------- no-allocation entry point
// Scratch for gts_simulate_batch_noalloc: a fixed array in the library's own
// device memory, created when the module loads in a device's context and held
// until the process exits.  In host code the symbol is only a handle; its
// device address comes from cudaGetSymbolAddress, looked up once per device
// and context: the context's process-unique id (cuCtxGetId) is kept with the
// address, so a call after cudaDeviceReset (a new context, the module loaded
// anew) looks the address up again instead of using the old one.
static __device__ __align__(256) uint2 g_static_scratch[GTS_STATIC_SCRATCH_BYTES / sizeof(uint2)];

namespace {
constexpr int MAX_DEVICES = 64;
struct StaticScratch {
  unsigned long long ctx_id;
  void *ptr;
};
StaticScratch g_static[MAX_DEVICES];
std::atomic<int> g_static_lock{0};
typedef int (*ctx_get_id_fn)(void *ctx, unsigned long long *id);  // CUresult cuCtxGetId(CUcontext, ...)
ctx_get_id_fn g_ctx_get_id = nullptr;

// Id of the current context, or 0 when none is current yet.
gts_status current_ctx_id(unsigned long long *id) {
  *id = 0;
  if (!g_ctx_get_id) {
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    const cudaError_t e = cudaGetDriverEntryPointByVersion("cuCtxGetId", &fn, 12000, cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
      return fail(GTS_ERR_CUDA, "simulate_noalloc: driver entry point cuCtxGetId unavailable");
    g_ctx_get_id = (ctx_get_id_fn)fn;
  }
  if (g_ctx_get_id(nullptr, id) != 0) *id = 0;
  return GTS_OK;
}

// Address of the static scratch in the current device's context (set-up on
// the first call in each device context).
gts_status static_scratch(void **out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "simulate_noalloc: current device");
  if (dev < 0 || dev >= MAX_DEVICES) return fail(GTS_ERR_UNSUPPORTED, "simulate_noalloc: device ordinal above 63");
  while (g_static_lock.exchange(1, std::memory_order_acquire)) {
  }
  unsigned long long id = 0;
  gts_status st = current_ctx_id(&id);
  if (st == GTS_OK && (id == 0 || g_static[dev].ctx_id != id || !g_static[dev].ptr)) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);  // makes the device's context current if none was
    if (e != cudaSuccess) {
      st = cuda_fail(e, "simulate_noalloc: static scratch address");
    } else {
      if (id == 0) current_ctx_id(&id);
      g_static[dev].ctx_id = id;
      g_static[dev].ptr = p;
    }
  }
  *out = g_static[dev].ptr;
  g_static_lock.store(0, std::memory_order_release);
  return st;
}
}  // namespace

extern "C" {

gts_status gts_simulate_batch_noalloc(gts_graph *g, gts_params *P, uint32_t first_point, uint32_t n_points,
                                      uint32_t flags, int32_t *d_start, int32_t *d_finish, int32_t *d_makespan,
                                      int32_t *d_status, uint64_t *d_digest, int32_t *d_cta_sm, int64_t *d_busy,
                                      void *stream) {
  clear_error();
  if (!g) return fail(GTS_ERR_INVALID_ARG, "null graph");
  if (GTS_SCRATCH_HEADER_BYTES + scratch_row_bytes(g) > GTS_STATIC_SCRATCH_BYTES)
    return fail(GTS_ERR_NOMEM, "simulate_noalloc: one scratch row (8 bytes per node of the largest graph, 16 per "
                               "tile) does not fit in the static scratch (GTS_STATIC_SCRATCH_BYTES)");
  void *scr = nullptr;
  gts_status st = static_scratch(&scr);
  if (st != GTS_OK) return st;
  // the shared array is cleared row by row before use (never vouched clean)
  flags &= ~GTS_SCRATCH_CLEAN;
  return gts_simulate_batch(g, P, first_point, n_points, flags, d_start, d_finish, d_makespan, d_status, d_digest,
                            d_cta_sm, d_busy, scr, GTS_STATIC_SCRATCH_BYTES, stream, nullptr);
}

}  // extern "C"
