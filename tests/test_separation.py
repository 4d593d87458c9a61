"""The oracle and the CUDA path stay apart, read from the source (CPU only).

* the library package never imports the oracle, and the oracle never imports
  the library;
* the seeded input generator imports neither;
* outside ``tests/`` only the bench's CPU-timing functions and ``smoke()``
  reach the oracle;
* the CUDA sources and the public header never refer to it;
* a missing ``libarckv.so`` raises instead of falling back to anything.
"""
import ast
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parent.parent
PKG = ROOT / "paper_2609_36835_gb300"


def _imports(path: Path):
    """(top-level module name, enclosing function or None) for every import."""
    tree = ast.parse(path.read_text(), str(path))
    out = []

    def visit(node, fn):
        for child in ast.iter_child_nodes(node):
            here = child.name if isinstance(child, (ast.FunctionDef, ast.AsyncFunctionDef)) else fn
            if isinstance(child, ast.Import):
                out.extend((a.name.split(".")[0], fn) for a in child.names)
            elif isinstance(child, ast.ImportFrom) and child.level == 0 and child.module:
                out.append((child.module.split(".")[0], fn))
            visit(child, here)

    visit(tree, None)
    return out


def _py(folder: Path):
    return sorted(p for p in folder.rglob("*.py") if "__pycache__" not in p.parts)


def test_library_does_not_import_the_oracle():
    for p in _py(PKG):
        assert "oracle" not in {m for m, _ in _imports(p)}, p


def test_oracle_does_not_import_the_library():
    for p in _py(ROOT / "oracle"):
        mods = {m for m, _ in _imports(p)}
        assert not mods & {"paper_2609_36835_gb300", "torch", "ctypes"}, (p, mods)


def test_input_generator_imports_neither_side():
    for p in _py(ROOT / "synth"):
        mods = {m for m, _ in _imports(p)}
        assert not mods & {"oracle", "paper_2609_36835_gb300"}, (p, mods)


def test_oracle_reached_only_from_tests_smoke_and_the_cpu_baseline():
    allowed = {("bench.py", "oracle_pair_seconds"), ("bench.py", "oracle_segments"), ("__graft_entry__.py", "smoke")}
    seen = set()
    for p in sorted(ROOT.glob("*.py")):
        for mod, fn in _imports(p):
            if mod == "oracle":
                seen.add((p.name, fn))
    assert seen and seen <= allowed, seen


@pytest.mark.parametrize("folder", [PKG / "csrc", ROOT / "include"])
def test_native_sources_never_refer_to_the_oracle(folder):
    for p in sorted(folder.iterdir()):
        if p.suffix in {".cu", ".cuh", ".h", ".cpp", ".c"}:
            assert "oracle" not in p.read_text().lower(), p


def test_missing_library_raises(monkeypatch, tmp_path):
    import paper_2609_36835_gb300 as pk
    monkeypatch.setattr(pk, "_lib", None)
    monkeypatch.setattr(pk, "_LIB_PATH", tmp_path / "libarckv.so")
    with pytest.raises(RuntimeError, match="missing"):
        pk.load_library()
