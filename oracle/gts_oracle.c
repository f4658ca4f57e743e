/*
 * gts_oracle.c -- reference list scheduler for warp-centric tile graphs.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the CPU oracle that the CUDA path is
 * checked against.  Only the tests, the smoke check and the benchmark's CPU
 * baseline and reference arm may load it; the product path never does.  It
 * shares no code, header or table with the CUDA library.
 *
 * What it computes (graph-driven simulation backend, Section 5):
 *   Given a tile graph G = (V, E) (Section 4.1) and one hardware parameter row,
 *   produce the integer start and finish cycle of every node and the makespan.
 *
 *   - A node is issued by its logical warp in program order (ascending id
 *     within its (cta, warp) stream).
 *   - A DATA edge u->v releases v when u completes; an ISSUE (order) edge
 *     releases v when u issues (Section 5.1, Section 5.3).
 *   - Compute and memory units are throughput servers (Section 5.2): a node of
 *     type ty takes one server of each resource class it uses for its
 *     occupancy occ = ceil(work / rate) cycles; its latency is
 *     L = base(ty) + lat_extra + max over used classes of occ.  Per-SM classes:
 *     TENSOR, TMA, LSU, ALU, BAR; one global class: HBM; one class per group
 *     of cluster_sms consecutive SMs: the on-chip NoC that DSMEM nodes (remote
 *     shared-memory accesses, Section 5.2 "DSMEM / On-chip NoC") cross.
 *   - Thread blocks are bound to SMs in ascending CTA order, each to the lowest
 *     SM with a free slot; a CTA retires when all its nodes completed and then
 *     frees its slot (Section 5.1).  A CTA of kernel k launches only after
 *     every CTA of kernels < k retired (kernel boundaries, Section 4.2).
 *   - The issue scheduler picks, at the current cycle t, the LOWEST node id
 *     among issuable warp heads, one node at a time, launching CTAs first,
 *     until nothing changes at t; then t jumps to the next event time.
 *   - Optional per-subpartition schedulers (Section 5.3: per-subpartition
 *     queues under greedy-then-oldest or round-robin): each SM has nsub
 *     schedulers; warp slot l = (CTA's slot on its SM) * W + warp belongs to
 *     scheduler l mod nsub, which issues at most one node per cycle -- the
 *     first of its issuable heads in policy order (GTO: the slot it issued
 *     from last, then the oldest warp, CTA id * W + warp; RR: cyclic slot
 *     order after its last slot).  The schedulers' picks go in ascending node
 *     id, one at a time.
 *
 * Readings where the paper is silent (the framework's fixed choices):
 *   lowest-id issue in place of GTO/round-robin; an ISSUE edge lets the
 *   successor start in the same cycle; contention delays only the start,
 *   finish = start + L exactly; a server taken at t is busy on [t, t+occ);
 *   CTA launch latency 0; times are int64 here and any finish above
 *   2^31-1 is reported as overflow.
 *
 * L2 (optional, Section 5.2: a fully associative LRU cache over tile-derived
 * accesses): LOAD and STORE nodes may name a tile; an LRU list of tiles, each
 * sized by its latest access, is updated at every such issue and trimmed from
 * the least recent end to l2_bytes.  A LOAD whose tile is in the list hits:
 * base tma_lat + l2_lat and ceil(work / l2_bpc) cycles on a memory-side (HBM)
 * server; every other LOAD pays tma_lat + l2_lat + dram_lat and
 * ceil(work / hbm_bpc).  STORE timing is unchanged.
 *
 * Busy server-cycles (optional output): for each resource class the sum of
 * the occupancies of the nodes served by it -- the cycles its servers were
 * held (Section 5.2).  Utilisation (Section 7.1 reports the tensor cores')
 * is that divided by servers x makespan.
 *
 * Plain on purpose: every step scans the resident CTAs, their warp heads and
 * all servers; no heaps, no incremental structures.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_ERR_INVALID_ARG (-1)
#define OR_ERR_INVALID_GRAPH (-2)
#define OR_ERR_INVALID_PARAMS (-3)
#define OR_ERR_NOMEM (-5)
#define OR_ERR_OVERFLOW (-6)
#define OR_ERR_DEADLOCK (-8)

/* operation types (Section 4.1 operation descriptor) */
enum { OT_LOAD = 0, OT_SMEM = 1, OT_MMA = 2, OT_EW = 3, OT_STORE = 4, OT_BAR = 5, OT_NOP = 6, OT_DSMEM = 7,
       OT_COUNT = 8 };
/* per-SM resource classes (Section 5.2) */
enum { RC_TENSOR = 0, RC_TMA = 1, RC_LSU = 2, RC_ALU = 3, RC_BAR = 4, RC_COUNT = 5 };

/* parameter row layout */
enum {
  PR_NUM_SMS = 0, PR_CTAS_PER_SM, PR_HBM_BPC, PR_DRAM_LAT, PR_TMA_BPC, PR_TMA_LAT,
  PR_SMEM_BPC, PR_SMEM_LAT, PR_MMA_FMA_PC, PR_MMA_LAT, PR_ALU_OPS_PC, PR_ALU_LAT,
  PR_BAR_LAT, PR_CAP_TENSOR, PR_CAP_TMA, PR_CAP_LSU, PR_CAP_ALU, PR_CAP_BAR,
  PR_CAP_HBM, PR_GRAPH_INDEX, PR_ISSUE_POLICY, PR_SUBPARTITIONS, PR_NOC_BPC, PR_NOC_LAT, PR_CAP_NOC,
  PR_CLUSTER_SMS, PR_L2_BYTES, PR_L2_LAT, PR_L2_BPC, PR_COUNT = 32
};
enum { POL_LOWEST_ID = 0, POL_GTO = 1, POL_RR = 2 };

#define INT32_LIMIT ((int64_t)2147483647)

static int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

int oracle_simulate(
    int64_t n, int64_t m, int64_t n_ctas, int64_t W,
    const uint32_t *row_ptr, const uint32_t *col, const uint8_t *ekind,
    const uint8_t *type, const uint16_t *warp, const uint32_t *cta,
    const uint32_t *work, const uint32_t *lat_extra, const uint32_t *cta_kernel,
    const int32_t *prm,
    int64_t *start, int64_t *finish, int64_t *makespan, int32_t *cta_sm,
    int64_t *busy /* [RC_COUNT + 4]: per-SM classes, HBM, NoC, L2 load hits, tracked loads; may be NULL */,
    const uint32_t *tile /* [n] tile of a LOAD/STORE or 0xFFFFFFFF; may be NULL */, int64_t n_tiles)
{
  int64_t v, e, c, w, k, r;
  int status = OR_OK;
  if (n < 0 || m < 0 || n_ctas < 0 || W < 1 || !prm || !makespan) return OR_ERR_INVALID_ARG;
  int64_t busy_acc[RC_COUNT + 4] = {0, 0, 0, 0, 0, 0, 0, 0, 0};
  if (busy)
    for (r = 0; r < RC_COUNT + 4; r++) busy[r] = 0;

  /* ---- parameter row (Table "GPU configurations" quantities) ---- */
  const int64_t num_sms = prm[PR_NUM_SMS], cps = prm[PR_CTAS_PER_SM];
  const int64_t rate[RC_COUNT] = {prm[PR_MMA_FMA_PC], prm[PR_TMA_BPC], prm[PR_SMEM_BPC], prm[PR_ALU_OPS_PC], 1};
  const int64_t cap[RC_COUNT] = {prm[PR_CAP_TENSOR], prm[PR_CAP_TMA], prm[PR_CAP_LSU], prm[PR_CAP_ALU], prm[PR_CAP_BAR]};
  const int64_t hbm_bpc = prm[PR_HBM_BPC], cap_hbm = prm[PR_CAP_HBM];
  if (num_sms < 1 || cps < 1 || hbm_bpc < 1 || cap_hbm < 1) return OR_ERR_INVALID_PARAMS;
  for (r = 0; r < RC_COUNT; r++)
    if (rate[r] < 1 || cap[r] < 1) return OR_ERR_INVALID_PARAMS;
  if (prm[PR_DRAM_LAT] < 0 || prm[PR_TMA_LAT] < 0 || prm[PR_SMEM_LAT] < 0 || prm[PR_MMA_LAT] < 0 ||
      prm[PR_ALU_LAT] < 0 || prm[PR_BAR_LAT] < 0)
    return OR_ERR_INVALID_PARAMS;
  const int64_t policy = prm[PR_ISSUE_POLICY], nsub = prm[PR_SUBPARTITIONS];
  if (policy == POL_LOWEST_ID) {
    if (nsub != 0) return OR_ERR_INVALID_PARAMS;
  } else if (policy == POL_GTO || policy == POL_RR) {
    if (nsub < 1 || nsub > 32) return OR_ERR_INVALID_PARAMS;
  } else {
    return OR_ERR_INVALID_PARAMS;
  }
  const int64_t noc_bpc = prm[PR_NOC_BPC], cap_noc = prm[PR_CAP_NOC], csms = prm[PR_CLUSTER_SMS];
  const int noc = csms != 0;                 /* the row configures an on-chip NoC */
  if (noc) {
    if (noc_bpc < 1 || prm[PR_NOC_LAT] < 0 || cap_noc < 1 || cap_noc > 32 || csms < 1 || csms > 32)
      return OR_ERR_INVALID_PARAMS;
  } else if (noc_bpc != 0 || prm[PR_NOC_LAT] != 0 || cap_noc != 0) {
    return OR_ERR_INVALID_PARAMS;
  }
  const int64_t l2_cap = prm[PR_L2_BYTES], l2_lat = prm[PR_L2_LAT], l2_bpc = prm[PR_L2_BPC];
  const int l2on = l2_cap != 0;              /* the row models the L2 */
  if (l2on) {
    if (l2_cap < 1 || l2_lat < 0 || l2_bpc < 1) return OR_ERR_INVALID_PARAMS;
  } else if (l2_lat != 0 || l2_bpc != 0) {
    return OR_ERR_INVALID_PARAMS;
  }
  for (k = PR_L2_BPC + 1; k < PR_COUNT; k++)
    if (prm[k] != 0) return OR_ERR_INVALID_PARAMS;
  if (n_tiles < 0 || (tile && n_tiles < 1)) return OR_ERR_INVALID_ARG;
  const int64_t ngrp = noc ? (num_sms + csms - 1) / csms : 1;  /* NoC groups */
  const int64_t per = cps * W;               /* warp slots per SM */
  const int64_t nq = num_sms * (nsub ? nsub : 1);

  /* ---- graph contract ---- */
  if (row_ptr[0] != 0 || (int64_t)row_ptr[n] != m) return OR_ERR_INVALID_GRAPH;
  for (v = 0; v < n; v++) {
    if (row_ptr[v + 1] < row_ptr[v]) return OR_ERR_INVALID_GRAPH;
    if (type[v] >= OT_COUNT || (int64_t)warp[v] >= W || (int64_t)cta[v] >= n_ctas) return OR_ERR_INVALID_GRAPH;
    for (e = row_ptr[v]; e < (int64_t)row_ptr[v + 1]; e++)
      if ((int64_t)col[e] <= v || (int64_t)col[e] >= n || ekind[e] > 1) return OR_ERR_INVALID_GRAPH;
    if (tile && tile[v] != 0xFFFFFFFFu && (type[v] == OT_LOAD || type[v] == OT_STORE) && (int64_t)tile[v] >= n_tiles)
      return OR_ERR_INVALID_GRAPH;
  }
  for (c = 1; c < n_ctas; c++)
    if (cta_kernel[c] < cta_kernel[c - 1]) return OR_ERR_INVALID_GRAPH;
  for (v = 0; v < n; v++)
    if (type[v] == OT_DSMEM && !noc) return OR_ERR_INVALID_PARAMS;  /* the row has no NoC to serve it */

  /* ---- per-node occupancy and latency (Section 5.2, Section 5.3) ---- */
  int8_t *cls = malloc((size_t)(n ? n : 1));
  int64_t *occ = malloc(sizeof(int64_t) * (size_t)(n ? n : 1));
  int64_t *hocc = malloc(sizeof(int64_t) * (size_t)(n ? n : 1));
  int64_t *lat = malloc(sizeof(int64_t) * (size_t)(n ? n : 1));
  int64_t *npend = calloc((size_t)(n ? n : 1), sizeof(int64_t));
  int64_t *rdy = calloc((size_t)(n ? n : 1), sizeof(int64_t));
  int64_t *nxt = malloc(sizeof(int64_t) * (size_t)(n ? n : 1));
  int64_t *head = malloc(sizeof(int64_t) * (size_t)(n_ctas > 0 ? n_ctas * W : 1));
  int64_t *rem = calloc((size_t)(n_ctas ? n_ctas : 1), sizeof(int64_t));
  int64_t *endt = calloc((size_t)(n_ctas ? n_ctas : 1), sizeof(int64_t));
  int64_t *sm_of = malloc(sizeof(int64_t) * (size_t)(n_ctas ? n_ctas : 1));
  int64_t *res = malloc(sizeof(int64_t) * (size_t)(n_ctas ? n_ctas : 1)); /* launched, not yet seen retired */
  int64_t *res_cnt = malloc(sizeof(int64_t) * (size_t)num_sms);
  int64_t *slot_of = malloc(sizeof(int64_t) * (size_t)(n_ctas ? n_ctas : 1)); /* CTA's slot on its SM */
  int64_t *sub_avail = calloc((size_t)nq, sizeof(int64_t)); /* scheduler may issue from this cycle on */
  int64_t *sub_last = malloc(sizeof(int64_t) * (size_t)nq);  /* warp slot it issued from last, -1 none */
  int64_t *cand = malloc(sizeof(int64_t) * (size_t)nq);
  int64_t *cand_key = malloc(sizeof(int64_t) * (size_t)nq);
  int64_t *srv[RC_COUNT];
  int64_t *hsrv = calloc((size_t)cap_hbm, sizeof(int64_t));
  int64_t *nsrv = calloc((size_t)(ngrp * (noc ? cap_noc : 1)), sizeof(int64_t)); /* NoC servers per group */
  int64_t *nocc = malloc(sizeof(int64_t) * (size_t)(n ? n : 1));
  const int64_t nt = tile ? n_tiles : 1;     /* L2 list over tiles: links, membership, entry bytes */
  int64_t *l2_prev = malloc(sizeof(int64_t) * (size_t)nt), *l2_next = malloc(sizeof(int64_t) * (size_t)nt);
  int64_t *l2_in = calloc((size_t)nt, sizeof(int64_t)), *l2_sz = calloc((size_t)nt, sizeof(int64_t));
  int64_t l2_head = -1, l2_tail = -1, l2_used = 0;
  for (r = 0; r < RC_COUNT; r++) srv[r] = calloc((size_t)(num_sms * cap[r]), sizeof(int64_t));
  int nomem = !cls || !occ || !hocc || !lat || !npend || !rdy || !nxt || !head || !rem || !endt ||
              !sm_of || !res || !res_cnt || !hsrv || !slot_of || !sub_avail || !sub_last || !cand || !cand_key ||
              !nsrv || !nocc || !l2_prev || !l2_next || !l2_in || !l2_sz;
  for (r = 0; r < RC_COUNT; r++) nomem |= !srv[r];
  if (nomem) { status = OR_ERR_NOMEM; goto out; }

  for (v = 0; v < n; v++) {
    const int64_t wk = work[v];
    int64_t base = 0, mx = 0;
    cls[v] = -1;
    occ[v] = 0;
    hocc[v] = -1; /* -1: does not use HBM */
    nocc[v] = -1; /* -1: does not cross the NoC */
    switch (type[v]) {
      case OT_LOAD:  cls[v] = RC_TMA; occ[v] = cdiv(wk, rate[RC_TMA]); hocc[v] = cdiv(wk, hbm_bpc);
                     base = prm[PR_TMA_LAT] + prm[PR_DRAM_LAT]; break;
      case OT_SMEM:  cls[v] = RC_LSU; occ[v] = cdiv(wk, rate[RC_LSU]); base = prm[PR_SMEM_LAT]; break;
      case OT_MMA:   cls[v] = RC_TENSOR; occ[v] = cdiv(wk, rate[RC_TENSOR]); base = prm[PR_MMA_LAT]; break;
      case OT_EW:    cls[v] = RC_ALU; occ[v] = cdiv(wk, rate[RC_ALU]); base = prm[PR_ALU_LAT]; break;
      case OT_STORE: cls[v] = RC_TMA; occ[v] = cdiv(wk, rate[RC_TMA]); hocc[v] = cdiv(wk, hbm_bpc);
                     base = prm[PR_TMA_LAT]; break;
      case OT_BAR:   cls[v] = RC_BAR; occ[v] = 1; base = prm[PR_BAR_LAT]; break;
      case OT_DSMEM: cls[v] = RC_LSU; occ[v] = cdiv(wk, rate[RC_LSU]); nocc[v] = cdiv(wk, noc_bpc);
                     base = prm[PR_SMEM_LAT] + prm[PR_NOC_LAT]; break;
      default:       break; /* NOP: no resource, base 0 */
    }
    if (cls[v] >= 0 && occ[v] > mx) mx = occ[v];
    if (hocc[v] > mx) mx = hocc[v];
    if (nocc[v] > mx) mx = nocc[v];
    lat[v] = base + (int64_t)lat_extra[v] + mx;
  }

  /* ---- streams: program order of each (cta, warp) is ascending id ---- */
  for (k = 0; k < n_ctas * W; k++) head[k] = -1;
  for (v = n - 1; v >= 0; v--) {
    const int64_t s = (int64_t)cta[v] * W + warp[v];
    nxt[v] = head[s];
    head[s] = v;
  }
  for (v = 0; v < n; v++)
    for (e = row_ptr[v]; e < (int64_t)row_ptr[v + 1]; e++) npend[col[e]]++;
  for (v = 0; v < n; v++) rem[cta[v]]++;
  for (c = 0; c < n_ctas; c++) { sm_of[c] = -1; slot_of[c] = -1; if (cta_sm) cta_sm[c] = -1; }
  for (k = 0; k < nq; k++) sub_last[k] = -1;
  for (v = 0; v < n; v++) { start[v] = -1; finish[v] = -1; }

  int64_t t = 0, issued = 0, next_cta = 0, nres = 0, mkspan = 0;
  for (;;) {
    /* ---- fixpoint at cycle t: CTA launches first, then one issue ---- */
    int progress = 1;
    while (progress) {
      progress = 0;
      /* (1) CTA launch, strictly ascending CTA id (head of line) */
      for (;;) {
        int64_t j = 0;
        for (k = 0; k < nres; k++) {             /* drop CTAs retired by t */
          const int64_t cc = res[k];
          if (!(rem[cc] == 0 && endt[cc] <= t)) res[j++] = cc;
        }
        nres = j;
        if (next_cta >= n_ctas) break;
        c = next_cta;
        int gate = 1;
        for (k = 0; k < nres; k++)
          if (cta_kernel[res[k]] < cta_kernel[c]) gate = 0;
        if (!gate) break;
        for (k = 0; k < num_sms; k++) res_cnt[k] = 0;
        for (k = 0; k < nres; k++) res_cnt[sm_of[res[k]]]++;
        int64_t sm = -1;
        for (k = 0; k < num_sms; k++)
          if (res_cnt[k] < cps) { sm = k; break; }
        if (sm < 0) break;
        int64_t slot = 0;                        /* lowest free slot on that SM */
        for (;; slot++) {
          int used = 0;
          for (k = 0; k < nres; k++)
            if (sm_of[res[k]] == sm && slot_of[res[k]] == slot) used = 1;
          if (!used) break;
        }
        sm_of[c] = sm;
        slot_of[c] = slot;
        if (cta_sm) cta_sm[c] = (int32_t)sm;
        res[nres++] = c;
        next_cta++;
        progress = 1;
      }
      /* (2) issue the lowest-id issuable warp head (per-subpartition
       *     policies: the lowest id among the schedulers' picks) */
      int64_t best = -1;
      for (k = 0; k < nq; k++) cand[k] = -1;
      for (k = 0; k < nres; k++) {
        const int64_t cc = res[k], sm = sm_of[cc];
        for (w = 0; w < W; w++) {
          const int64_t h = head[cc * W + w];
          if (h < 0 || npend[h] != 0 || rdy[h] > t) continue;
          const int64_t l = slot_of[cc] * W + w, q = nsub ? sm * nsub + l % nsub : 0;
          if (nsub && sub_avail[q] > t) continue; /* this scheduler already issued at t */
          if (cls[h] >= 0) {
            int ok = 0;
            for (int64_t q = 0; q < cap[cls[h]]; q++)
              if (srv[cls[h]][sm * cap[cls[h]] + q] <= t) ok = 1;
            if (!ok) continue;
          }
          if (hocc[h] >= 0) {
            int ok = 0;
            for (int64_t q = 0; q < cap_hbm; q++)
              if (hsrv[q] <= t) ok = 1;
            if (!ok) continue;
          }
          if (nocc[h] >= 0) {
            int ok = 0;
            for (int64_t q = 0; q < cap_noc; q++)
              if (nsrv[(sm / csms) * cap_noc + q] <= t) ok = 1;
            if (!ok) continue;
          }
          if (!nsub) {
            if (best < 0 || h < best) best = h;
            continue;
          }
          int64_t key;
          if (policy == POL_GTO)
            key = (l == sub_last[q] ? 0 : ((int64_t)1 << 40)) + cc * W + w;
          else
            key = sub_last[q] < 0 ? l : ((l - sub_last[q] - 1) % per + per) % per;
          if (cand[q] < 0 || key < cand_key[q]) { cand[q] = h; cand_key[q] = key; }
        }
      }
      if (nsub)
        for (k = 0; k < nq; k++)
          if (cand[k] >= 0 && (best < 0 || cand[k] < best)) best = cand[k];
      if (best >= 0) {
        v = best;
        c = cta[v];
        const int64_t sm = sm_of[c];
        int64_t lv = lat[v], hv = hocc[v];
        const int64_t tv = (tile && (type[v] == OT_LOAD || type[v] == OT_STORE) && tile[v] != 0xFFFFFFFFu)
                               ? (int64_t)tile[v] : -1;
        if (l2on && type[v] == OT_LOAD) {      /* hit or miss decides latency and memory-side occupancy */
          const int hit = tv >= 0 && l2_in[tv];
          hv = hit ? cdiv(work[v], l2_bpc) : cdiv(work[v], hbm_bpc);
          lv = prm[PR_TMA_LAT] + l2_lat + (hit ? 0 : prm[PR_DRAM_LAT]) + (int64_t)lat_extra[v] +
               (occ[v] > hv ? occ[v] : hv);
          if (tv >= 0) { busy_acc[RC_COUNT + 3]++; if (hit) busy_acc[RC_COUNT + 2]++; }
        }
        if (l2on && tv >= 0) {                 /* the tile becomes the most recent entry */
          if (l2_in[tv]) {
            if (l2_prev[tv] >= 0) l2_next[l2_prev[tv]] = l2_next[tv]; else l2_head = l2_next[tv];
            if (l2_next[tv] >= 0) l2_prev[l2_next[tv]] = l2_prev[tv]; else l2_tail = l2_prev[tv];
            l2_used -= l2_sz[tv];
          }
          l2_prev[tv] = -1;
          l2_next[tv] = l2_head;
          if (l2_head >= 0) l2_prev[l2_head] = tv; else l2_tail = tv;
          l2_head = tv;
          l2_in[tv] = 1;
          l2_sz[tv] = work[v];
          l2_used += work[v];
          while (l2_used > l2_cap) {           /* drop least recent entries */
            const int64_t y = l2_tail;
            l2_tail = l2_prev[y];
            if (l2_tail >= 0) l2_next[l2_tail] = -1; else l2_head = -1;
            l2_in[y] = 0;
            l2_used -= l2_sz[y];
          }
        }
        const int64_t f = t + lv;
        if (f > INT32_LIMIT) { status = OR_ERR_OVERFLOW; goto out; }
        start[v] = t;
        finish[v] = f;
        if (nsub) {
          const int64_t l = slot_of[c] * W + warp[v], q = sm * nsub + l % nsub;
          sub_avail[q] = t + 1;
          sub_last[q] = l;
        }
        if (f > mkspan) mkspan = f;
        if (cls[v] >= 0) busy_acc[cls[v]] += occ[v];
        if (hv >= 0) busy_acc[RC_COUNT] += hv;
        if (nocc[v] >= 0) busy_acc[RC_COUNT + 1] += nocc[v];
        if (cls[v] >= 0) { /* take any free server of the class on this SM */
          for (int64_t q = 0; q < cap[cls[v]]; q++) {
            int64_t *s = &srv[cls[v]][sm * cap[cls[v]] + q];
            if (*s <= t) { *s = t + occ[v]; break; }
          }
        }
        if (hv >= 0) {
          for (int64_t q = 0; q < cap_hbm; q++)
            if (hsrv[q] <= t) { hsrv[q] = t + hv; break; }
        }
        if (nocc[v] >= 0) { /* any free NoC server of the SM's group */
          for (int64_t q = 0; q < cap_noc; q++) {
            int64_t *s = &nsrv[(sm / csms) * cap_noc + q];
            if (*s <= t) { *s = t + nocc[v]; break; }
          }
        }
        for (e = row_ptr[v]; e < (int64_t)row_ptr[v + 1]; e++) {
          const int64_t u = col[e];
          const int64_t rel = ekind[e] ? t : f;   /* ISSUE edge: at issue; DATA: at completion */
          npend[u]--;
          if (rel > rdy[u]) rdy[u] = rel;
        }
        head[c * W + warp[v]] = nxt[v];
        rem[c]--;
        if (f > endt[c]) endt[c] = f;
        issued++;
        progress = 1;
      }
    }
    if (issued == n) break;
    /* ---- advance to the next event time ---- */
    int64_t tn = INT64_MAX;
    for (k = 0; k < nres; k++) {
      const int64_t cc = res[k];
      for (w = 0; w < W; w++) {
        const int64_t h = head[cc * W + w];
        if (h >= 0 && npend[h] == 0 && rdy[h] > t && rdy[h] < tn) tn = rdy[h];
      }
      if (rem[cc] == 0 && endt[cc] > t && endt[cc] < tn) tn = endt[cc];
    }
    for (r = 0; r < RC_COUNT; r++)
      for (k = 0; k < num_sms * cap[r]; k++)
        if (srv[r][k] > t && srv[r][k] < tn) tn = srv[r][k];
    for (k = 0; k < cap_hbm; k++)
      if (hsrv[k] > t && hsrv[k] < tn) tn = hsrv[k];
    if (noc)
      for (k = 0; k < ngrp * cap_noc; k++)
        if (nsrv[k] > t && nsrv[k] < tn) tn = nsrv[k];
    if (nsub)
      for (k = 0; k < nq; k++)
        if (sub_avail[k] > t && sub_avail[k] < tn) tn = sub_avail[k];
    if (tn == INT64_MAX) { status = OR_ERR_DEADLOCK; goto out; }
    t = tn;
  }
  *makespan = mkspan;
  if (busy)
    for (r = 0; r < RC_COUNT + 4; r++) busy[r] = busy_acc[r];

out:
  free(cls); free(occ); free(hocc); free(lat); free(npend); free(rdy); free(nxt); free(head);
  free(rem); free(endt); free(sm_of); free(res); free(res_cnt); free(hsrv);
  free(slot_of); free(sub_avail); free(sub_last); free(cand); free(cand_key); free(nsrv); free(nocc);
  free(l2_prev); free(l2_next); free(l2_in); free(l2_sz);
  for (r = 0; r < RC_COUNT; r++) free(srv[r]);
  return status;
}
