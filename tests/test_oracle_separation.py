"""The oracle and the CUDA path share no code (static import scan, CPU only).

The product package never imports the oracle and the oracle never imports the product
package; the seeded input generators (`paper_2607_11185_gb300/workloads.py`) are the one shared
module and hold none of the method's arithmetic, and the oracle does not import them either
(tests pass it the inputs).  Outside the tests, only the bench's CPU-baseline and reference legs
and `smoke()` may reach the oracle.
"""
import ast
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _imports(path):
    """(module, enclosing top-level function or None) for every import in a Python file."""
    tree = ast.parse(open(path).read(), path)
    out = []

    def visit(node, fn):
        for child in ast.iter_child_nodes(node):
            f = fn
            if isinstance(child, (ast.FunctionDef, ast.AsyncFunctionDef)) and fn is None:
                f = child.name
            if isinstance(child, ast.Import):
                out.extend((a.name, f) for a in child.names)
            elif isinstance(child, ast.ImportFrom):
                mod = child.module or ""
                if child.level:                       # relative import inside a package
                    mod = "." + mod
                out.extend((f"{mod}.{a.name}" if mod else a.name, f) for a in child.names)
                out.append((mod, f))
            visit(child, f)

    visit(tree, None)
    return out


def _py_files(d):
    for base, _, files in os.walk(os.path.join(ROOT, d)):
        if "__pycache__" in base:
            continue
        for f in files:
            if f.endswith(".py"):
                yield os.path.join(base, f)


def test_product_package_never_imports_the_oracle():
    for path in _py_files("paper_2607_11185_gb300"):
        for mod, _ in _imports(path):
            assert not mod.split(".")[0] == "oracle", (path, mod)
    for d in ("paper_2607_11185_gb300/csrc", "include"):
        for base, _, files in os.walk(os.path.join(ROOT, d)):
            for f in files:
                if f.endswith((".cu", ".cuh", ".h", ".c", ".cpp")):
                    text = open(os.path.join(base, f)).read()
                    assert "oracle/" not in text and '#include "oracle' not in text, f


def test_oracle_never_imports_the_product():
    for path in _py_files("oracle"):
        for mod, _ in _imports(path):
            assert not mod.split(".")[0] == "paper_2607_11185_gb300", (path, mod)
            assert mod.split(".")[0] not in ("bench", "__graft_entry__"), (path, mod)


def test_oracle_reached_only_from_the_allowed_legs():
    allowed = {
        "bench.py": {"oracle_sample", "oracle_one_core", "run_reference"},
        "__graft_entry__.py": {"smoke"},
    }
    for name, fns in allowed.items():
        for mod, fn in _imports(os.path.join(ROOT, name)):
            if mod.split(".")[0] == "oracle":
                assert fn in fns, (name, mod, fn)
    # the one-core leg runs the oracle in a child interpreter: its source names the oracle,
    # and it is one of the allowed functions above
    src = open(os.path.join(ROOT, "bench.py")).read()
    tree = ast.parse(src)
    for node in tree.body:
        if isinstance(node, ast.FunctionDef) and "from oracle" in ast.get_source_segment(src, node):
            assert node.name in allowed["bench.py"], node.name
