"""CPU oracle for the graph-driven simulation backend (Section 5).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg and reference arm (the oracle timed on the host
cores) are the only callers.  It shares no code with the
CUDA library; the two meet only at the seeded inputs.

* ``gts_oracle.c`` / ``run.py`` -- the plain single-threaded event-driven
  scheduler (int64 cycles) and its ctypes driver.
* ``stepper.py`` -- an independent pure-Python cycle-by-cycle stepper for tiny
  graphs, written from the same definition without event skipping.
"""
