"""The CUDA path and the oracle stay independent: the package (Python and
CUDA/C sources) never names the oracle, the oracle imports nothing of the
package, and bench.py reaches the oracle only in its CPU-baseline leg and its reference
arm (the oracle timed on the host cores)."""
import ast
import glob
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2607_11262_gb300")


def imported_modules(path):
    tree = ast.parse(open(path).read())
    out = set()
    for node in ast.walk(tree):
        if isinstance(node, ast.Import):
            out |= {a.name.split(".")[0] for a in node.names}
        elif isinstance(node, ast.ImportFrom) and node.module:
            out.add(node.module.split(".")[0])
    return out


def test_package_never_imports_the_oracle():
    for path in glob.glob(os.path.join(PKG, "*.py")):
        assert "oracle" not in imported_modules(path), path


def test_native_sources_never_name_the_oracle():
    for path in glob.glob(os.path.join(PKG, "csrc", "*")) + glob.glob(os.path.join(ROOT, "include", "*.h")):
        assert not re.search(r"oracle", open(path).read(), re.I), path


def test_oracle_imports_nothing_of_the_package():
    for path in glob.glob(os.path.join(ROOT, "oracle", "*.py")):
        assert not imported_modules(path) & {"paper_2607_11262_gb300", "bench", "__graft_entry__"}, path
    src = open(os.path.join(ROOT, "oracle", "gts_oracle.c")).read()
    assert '#include "gts.h"' not in src and "gts_" not in src.replace("gts_oracle", "")


def test_bench_reaches_the_oracle_only_in_its_cpu_legs():
    tree = ast.parse(open(os.path.join(ROOT, "bench.py")).read())
    users = set()
    for fn in ast.walk(tree):
        if isinstance(fn, ast.FunctionDef):
            for node in ast.walk(fn):
                if isinstance(node, ast.ImportFrom) and node.module and node.module.split(".")[0] == "oracle":
                    users.add(fn.name)
    top = {n.module for n in tree.body if isinstance(n, ast.ImportFrom) and n.module}
    assert "oracle" not in {m.split(".")[0] for m in top}
    assert users == {"cpu_baseline", "run_reference"}, users
