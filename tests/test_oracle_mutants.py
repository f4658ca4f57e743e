"""Plausible mistakes planted in a copy of the oracle's C source must each fail
one of the oracle's pins (tests/test_oracle_pins.py): a dropped term, a wrong
comparison or index, a released edge at the wrong cycle, a policy key turned
around, an L2 rule broken.  The committed oracle is never edited: every mutant
is compiled from an edited copy into oracle/_build/mutants/ and swapped in for
the duration of the pins.  A mutant that no pin catches names a gap in the pins.
"""
import ctypes
import os
import subprocess

from oracle import run
from paper_2607_11262_gb300 import workloads as W
from tests import test_oracle_pins as PINS

MUTANT_DIR = os.path.join(run.BUILD_DIR, "mutants")

# (name, text of gts_oracle.c, replacement, replace every occurrence)
MUTANTS = [
    # dependency release (Section 5.1)
    ("ISSUE edge released at finish", "const int64_t rel = ekind[e] ? t : f;", "const int64_t rel = f;", False),
    ("DATA edge released at issue", "const int64_t rel = ekind[e] ? t : f;", "const int64_t rel = t;", False),
    ("release keeps the earliest cycle", "if (rel > rdy[u]) rdy[u] = rel;",
     "if (rdy[u] == 0 || rel < rdy[u]) rdy[u] = rel;", False),
    # issue order (lowest id) and resources
    ("highest id first", "if (best < 0 || h < best) best = h;", "if (best < 0 || h > best) best = h;", False),
    ("HBM servers not checked", "for (int64_t q = 0; q < cap_hbm; q++)\n              if (hsrv[q] <= t) ok = 1;",
     "ok = 1;", False),
    ("unit servers not checked",
     "for (int64_t q = 0; q < cap[cls[h]]; q++)\n              if (srv[cls[h]][sm * cap[cls[h]] + q] <= t) ok = 1;",
     "ok = 1;", False),
    # latency and occupancy (Section 5.2)
    ("occupancy rounded down", "return (a + b - 1) / b;", "return a / b;", False),
    ("BAR holds no cycle", "occ[v] = 1; base = prm[PR_BAR_LAT]", "occ[v] = 0; base = prm[PR_BAR_LAT]", False),
    ("lat_extra dropped", "lat[v] = base + (int64_t)lat_extra[v] + mx;", "lat[v] = base + mx;", False),
    ("occupancies summed, not maxed", "if (hocc[v] > mx) mx = hocc[v];", "if (hocc[v] > 0) mx += hocc[v];", False),
    ("LOAD without TMA latency", "base = prm[PR_TMA_LAT] + prm[PR_DRAM_LAT]; break;", "base = prm[PR_DRAM_LAT]; break;",
     False),
    ("STORE pays DRAM latency", "hocc[v] = cdiv(wk, hbm_bpc);\n                     base = prm[PR_TMA_LAT]; break;",
     "hocc[v] = cdiv(wk, hbm_bpc);\n                     base = prm[PR_TMA_LAT] + prm[PR_DRAM_LAT]; break;", False),
    ("MMA on the ALU servers", "case OT_MMA:   cls[v] = RC_TENSOR;", "case OT_MMA:   cls[v] = RC_ALU;", False),
    ("HBM busy until finish", "if (hsrv[q] <= t) { hsrv[q] = t + hv; break; }",
     "if (hsrv[q] <= t) { hsrv[q] = t + lv; break; }", False),
    # CTA launch and retirement (Section 5.1 TB scheduler)
    ("no kernel-boundary gate", "if (cta_kernel[res[k]] < cta_kernel[c]) gate = 0;", "(void)0;", False),
    ("CTA on the highest free SM", "if (res_cnt[k] < cps) { sm = k; break; }", "if (res_cnt[k] < cps) { sm = k; }",
     False),
    ("CTA retires at its last issue", "if (!(rem[cc] == 0 && endt[cc] <= t)) res[j++] = cc;",
     "if (!(rem[cc] == 0)) res[j++] = cc;", False),
    # time advance
    ("server free times are no events", "if (srv[r][k] > t && srv[r][k] < tn) tn = srv[r][k];", "(void)0;", False),
    # busy counters
    ("HBM busy cycles not counted", "if (hv >= 0) busy_acc[RC_COUNT] += hv;", "(void)0;", False),
    # per-subpartition policies (Section 5.3)
    ("GTO prefers the youngest warp", "key = (l == sub_last[q] ? 0 : ((int64_t)1 << 40)) + cc * W + w;",
     "key = (l == sub_last[q] ? 0 : ((int64_t)1 << 40)) - cc * W - w;", False),
    ("GTO not greedy", "key = (l == sub_last[q] ? 0 : ((int64_t)1 << 40)) + cc * W + w;", "key = cc * W + w;", False),
    ("RR restarts at the last slot", "((l - sub_last[q] - 1) % per + per) % per", "((l - sub_last[q]) % per + per) % per",
     False),
    ("two issues per scheduler per cycle", "sub_avail[q] = t + 1;", "sub_avail[q] = t;", False),
    ("slot-to-scheduler map by division", "q = nsub ? sm * nsub + l % nsub : 0", "q = nsub ? sm * nsub + (l / nsub) % nsub : 0",
     False),
    # DSMEM over the NoC (Section 5.2)
    ("NoC group by modulo", "(sm / csms) * cap_noc", "(sm % ngrp) * cap_noc", True),
    ("DSMEM without NoC latency", "base = prm[PR_SMEM_LAT] + prm[PR_NOC_LAT]; break;", "base = prm[PR_SMEM_LAT]; break;",
     False),
    ("NoC occupancy not in the latency", "if (nocc[v] > mx) mx = nocc[v];", "(void)0;", False),
    # L2 (Section 5.2, LRU over tiles)
    ("L2 hit pays DRAM latency", "(hit ? 0 : prm[PR_DRAM_LAT])", "prm[PR_DRAM_LAT]", False),
    ("L2 hit at DRAM bandwidth", "hv = hit ? cdiv(work[v], l2_bpc) : cdiv(work[v], hbm_bpc);",
     "hv = cdiv(work[v], hbm_bpc);", False),
    ("STORE does not allocate in L2", "if (l2on && tv >= 0) {", "if (l2on && tv >= 0 && type[v] == OT_LOAD) {", False),
    ("L2 capacity off by one", "while (l2_used > l2_cap) {", "while (l2_used >= l2_cap) {", False),
    ("L2 hit keeps its recency", "if (l2on && tv >= 0) {", "if (l2on && tv >= 0 && !l2_in[tv]) {", False),
]

# the pins, fastest first; each is a plain function of tests/test_oracle_pins.py
PIN_CALLS = [
    ("golden single-node latency", PINS.test_golden_single_node_latency, ()),
    ("golden hand schedules", PINS.test_golden_hand_schedules, ()),
    ("chain sums latencies", PINS.test_chain_makespan_is_sum_of_latencies, ()),
    ("golden issue policies", PINS.test_golden_issue_policies, ()),
    ("golden NoC", PINS.test_golden_noc, ()),
    ("golden L2", PINS.test_golden_l2, ()),
    ("L2 closed forms", PINS.test_l2_closed_forms, ()),
    ("one issue per scheduler per cycle (GTO)", PINS.test_one_issue_per_scheduler_per_cycle, (W.POLICY_GTO,)),
    ("one issue per scheduler per cycle (RR)", PINS.test_one_issue_per_scheduler_per_cycle, (W.POLICY_RR,)),
    ("single server without idle", PINS.test_single_server_no_idle, ()),
    ("unlimited resources: longest path", PINS.test_unlimited_resources_give_longest_path, ()),
    ("Graham bound", PINS.test_graham_list_scheduling_bound, ()),
    ("stepper, exhaustive n=3", PINS.test_stepper_equals_oracle_exhaustive, (3,)),
    ("stepper, small GEMM CTA", PINS.test_stepper_equals_oracle_small_gemm_cta, ()),
    ("stepper, random", PINS.test_stepper_equals_oracle_random, ()),
    ("stepper, policies GTO", PINS.test_stepper_equals_oracle_policies, (W.POLICY_GTO,)),
    ("stepper, policies RR", PINS.test_stepper_equals_oracle_policies, (W.POLICY_RR,)),
    ("stepper, NoC", PINS.test_stepper_equals_oracle_noc, ()),
    ("stepper, L2", PINS.test_stepper_equals_oracle_l2, ()),
    ("invariants on random graphs", PINS.test_invariants_random_graphs, ()),
    ("stepper, exhaustive n=4", PINS.test_stepper_equals_oracle_exhaustive, (4,)),
]


def _source():
    return open(run.SRC).read()


def _build_mutant(k, text):
    os.makedirs(MUTANT_DIR, exist_ok=True)
    src = os.path.join(MUTANT_DIR, f"mutant{k:02d}.c")
    lib = os.path.join(MUTANT_DIR, f"libmutant{k:02d}_{os.getpid()}.so")
    with open(src, "w") as f:
        f.write(text)
    subprocess.check_call(["gcc", "-O2", "-std=c99", "-shared", "-fPIC", "-o", lib, src])
    m = ctypes.CDLL(lib)
    m.oracle_simulate.argtypes = [ctypes.c_int64] * 4 + [ctypes.c_void_p] * 16 + [ctypes.c_int64]
    m.oracle_simulate.restype = ctypes.c_int
    return m, lib


def _first_failing_pin(lib):
    saved = run._load()
    run._lib = lib
    try:
        for name, fn, args in PIN_CALLS:
            try:
                fn(*args)
            except Exception:  # an assertion, or a result the pin cannot even read
                return name
        return None
    finally:
        run._lib = saved


def test_mutations_apply_to_the_oracle_source():
    src = _source()
    for name, a, b, every in MUTANTS:
        assert a in src, name
        assert a != b, name


def test_unmutated_oracle_passes_every_pin_here():
    assert _first_failing_pin(run._load()) is None


def test_every_planted_mistake_fails_a_pin():
    src = _source()
    missed, caught = [], {}
    for k, (name, a, b, every) in enumerate(MUTANTS):
        text = src.replace(a, b) if every else src.replace(a, b, 1)
        m, lib = _build_mutant(k, text)
        try:
            pin = _first_failing_pin(m)
        finally:
            os.remove(lib)
        if pin is None:
            missed.append(name)
        else:
            caught[name] = pin
    assert not missed, f"planted mistakes no pin catches: {missed}"
    assert len(caught) == len(MUTANTS)
