"""The C-ABI library builds for sm_103a, loads without a GPU and exports every
function include/gts.h declares (no compute calls)."""
import ctypes
import os
import re

import pytest

from paper_2607_11262_gb300 import build as B
from paper_2607_11262_gb300 import gts

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared(header):
    src = open(header).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return set(re.findall(r"^[A-Za-z_][\w\s\*]*?\b(gts_\w+)\s*\(", src, flags=re.M))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(B.LIB):
        B.build()
    return ctypes.CDLL(B.LIB)


def test_header_declarations_match_binding():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            names |= declared(os.path.join(ROOT, "include", f))
    assert names, "no declarations found"
    assert set(gts.EXPORTS) <= names


def test_every_declared_symbol_is_exported(lib):
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            for name in declared(os.path.join(ROOT, "include", f)):
                assert hasattr(lib, name), name


def test_binding_loads_and_sizes_without_gpu(lib):
    gts.load()
    # pure host arithmetic: workspace sizing and argument checks
    assert gts.gts_graph_workspace_bytes(10, 12, 2, 3, 1) > 10 * 32
    assert gts.gts_graph_workspace_bytes(10, 12, 2, 200, 1) == 0     # too many warps per CTA
    assert gts.gts_graph_workspace_bytes(10, 12, 2, 3, 0) == 0       # no graph
    assert gts.load().gts_graph_create(None, None, None) == gts.GTS_ERR_INVALID_ARG
    assert "null" in gts.gts_last_error()
    assert gts.load().gts_simulate_batch(None, None, 0, 0, 0, None, None, None, None, None, None, None, None, 0,
                                         None, None) == gts.GTS_ERR_INVALID_ARG


def test_oracle_builds_and_is_separate():
    from oracle import run
    assert os.path.exists(run.build())
    src = open(run.SRC).read()
    assert "gts.h" not in src and "libgts" not in src
    for f in ("gts.py", "build.py", "workloads.py"):
        txt = open(os.path.join(ROOT, "paper_2607_11262_gb300", f)).read()
        assert not re.search(r"^\s*(from|import)\s+oracle", txt, flags=re.M), f


C_CLIENT = r"""
#include <stdio.h>
#include "gts.h"

int main(void) {
  /* host-only calls: sizes and the error text need no GPU */
  printf("%zu %zu %zu\n", gts_graph_workspace_bytes(10, 12, 2, 3, 1), gts_graph_workspace_bytes(10, 12, 2, 200, 1),
         gts_template_workspace_bytes(2, 20, 40, 50, 4, 3, 1));
  printf("%d %d\n", gts_graph_create(NULL, NULL, NULL), gts_last_error() != NULL);
  return 0;
}
"""


def test_header_is_plain_c_and_a_c_client_links(lib):
    # a C99 program (pedantic, warnings as errors) includes the header, links
    # libgts and gets the binding's answers from the host-only calls
    import shutil
    import subprocess
    if shutil.which("gcc") is None:
        pytest.skip("no C compiler")
    out_dir = os.path.join(os.path.dirname(B.LIB), "c_client")
    os.makedirs(out_dir, exist_ok=True)
    src = os.path.join(out_dir, "client.c")
    exe = os.path.join(out_dir, f"client_{os.getpid()}")
    with open(src, "w") as f:
        f.write(C_CLIENT)
    lib_dir = os.path.dirname(B.LIB)
    subprocess.check_call(["gcc", "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror", "-I", os.path.join(ROOT, "include"),
                           "-o", exe, src, os.path.join(lib_dir, os.path.basename(B.LIB)), f"-Wl,-rpath,{lib_dir}"])
    try:
        got = subprocess.run([exe], capture_output=True, text=True, check=True).stdout.split()
    finally:
        os.remove(exe)
    want = [gts.gts_graph_workspace_bytes(10, 12, 2, 3, 1), gts.gts_graph_workspace_bytes(10, 12, 2, 200, 1),
            gts.gts_template_workspace_bytes(2, 20, 40, 50, 4, 3, 1)]
    assert [int(x) for x in got[:3]] == want
    assert int(got[3]) == gts.GTS_ERR_INVALID_ARG and got[4] == "1"
