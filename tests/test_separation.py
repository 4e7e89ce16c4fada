"""The oracle and the CUDA path share no code, and only the permitted places use the oracle: the
tests, __graft_entry__.smoke() and bench.py's CPU baseline and reference arm. Static checks of
the sources (no GPU, no imports of the modules under test)."""
import ast
import glob
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2501_19090_gb300")


def _imports(path):
    """(module, enclosing function name or None) for every import statement in a Python file."""
    tree = ast.parse(open(path).read(), path)
    out = []

    def walk(node, fn):
        for child in ast.iter_child_nodes(node):
            if isinstance(child, (ast.FunctionDef, ast.AsyncFunctionDef)):
                walk(child, child.name if fn is None else fn)
            elif isinstance(child, ast.Import):
                out.extend((a.name, fn) for a in child.names)
            elif isinstance(child, ast.ImportFrom):
                out.append(((child.module or "") if not child.level else "." + (child.module or ""), fn))
            else:
                walk(child, fn)

    walk(tree, None)
    return out


def test_product_python_never_imports_the_oracle():
    for path in glob.glob(os.path.join(PKG, "*.py")):
        for mod, _ in _imports(path):
            assert not mod.split(".")[0] == "oracle", f"{path} imports {mod}"


def test_product_native_sources_never_include_the_oracle():
    for path in glob.glob(os.path.join(PKG, "csrc", "*")) + glob.glob(os.path.join(ROOT, "include", "*")):
        for line in open(path, errors="replace"):
            if re.match(r"\s*#\s*include", line):
                assert "oracle" not in line, f"{path}: {line.strip()}"


def test_oracle_imports_only_numpy_scipy_and_the_standard_library():
    allowed = {"numpy", "scipy", "dataclasses", "__future__", "math", "fractions", "itertools", "typing"}
    for path in glob.glob(os.path.join(ROOT, "oracle", "*.py")):
        for mod, _ in _imports(path):
            if mod.startswith("."):
                continue                                   # the oracle's own modules
            assert mod.split(".")[0] in allowed, f"{path} imports {mod}"


def test_bench_and_entry_use_the_oracle_only_where_permitted():
    permitted = {os.path.join(ROOT, "bench.py"): {"cpu_baseline", "run_reference"},
                 os.path.join(ROOT, "__graft_entry__.py"): {"smoke"}}
    for path, fns in permitted.items():
        uses = [fn for mod, fn in _imports(path) if mod.split(".")[0] == "oracle"]
        assert uses, f"{path}: expected the oracle in {sorted(fns)}"
        assert set(uses) <= fns, f"{path} imports the oracle in {sorted(set(uses) - fns)}"
