"""The oracle and the CUDA path stay apart: the package never imports the oracle (or the
tests), the oracle imports nothing but numpy and the standard library, bench.py reaches the
oracle only from its host-core baseline worker, and the shared input generator holds none
of the method's arithmetic."""

import ast
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2606_00144_gb300")
ORACLE = os.path.join(ROOT, "oracle")


def py_files(folder):
    return sorted(os.path.join(folder, f) for f in os.listdir(folder) if f.endswith(".py"))


def imports(path):
    """(top-level module name, enclosing function or None, relative level) of every import."""
    tree = ast.parse(open(path).read(), path)
    out = []

    def visit(node, func):
        for child in ast.iter_child_nodes(node):
            f = child.name if isinstance(child, (ast.FunctionDef, ast.AsyncFunctionDef)) else func
            if isinstance(child, ast.Import):
                out.extend((a.name.split(".")[0], func, 0) for a in child.names)
            elif isinstance(child, ast.ImportFrom):
                out.append(((child.module or "").split(".")[0], func, child.level))
            visit(child, f)

    visit(tree, None)
    return out


def test_package_never_imports_the_oracle_or_the_tests():
    for path in py_files(PKG):
        for mod, _, level in imports(path):
            if level == 0:
                assert mod not in ("oracle", "tests"), f"{os.path.relpath(path, ROOT)} imports {mod}"


def test_cuda_sources_do_not_mention_the_oracle():
    csrc = os.path.join(PKG, "csrc")
    for f in sorted(os.listdir(csrc)):
        text = open(os.path.join(csrc, f)).read().lower()
        assert "oracle" not in text, f"csrc/{f} mentions the oracle"


def test_oracle_imports_only_numpy_and_the_standard_library():
    allowed = {"__future__", "math", "numpy"}
    for path in py_files(ORACLE):
        for mod, _, level in imports(path):
            if level == 0:
                assert mod in allowed, f"{os.path.relpath(path, ROOT)} imports {mod}"
            else:
                assert mod == "budgetdraft_oracle", f"{os.path.relpath(path, ROOT)} imports .{mod}"


def test_bench_reaches_the_oracle_only_from_its_host_core_worker():
    sites = [(mod, func) for mod, func, level in imports(os.path.join(ROOT, "bench.py")) if mod == "oracle"]
    assert sites, "bench.py no longer times the oracle"
    assert all(func == "_oracle_worker" for _, func in sites), sites


def test_input_generator_holds_none_of_the_methods_arithmetic():
    """workload.py feeds both sides; it draws and rounds inputs and nothing else."""
    text = open(os.path.join(PKG, "workload.py")).read()
    for name in ("softmax", "logsumexp", "topk", "argmax", "argsort", "scaled_dot_product", ".exp(", "ctypes",
                 "binding"):
        assert name not in text, f"workload.py uses {name}"
