"""The product path and the oracle stay apart, and the product path has no fallback (host only).

* Nothing in the package (Python or CUDA) imports, includes or links the oracle, and the
  oracle imports nothing from the package.
* `bench.py` reaches the oracle only inside its CPU legs (no module-level import).
* When the compiled library cannot be built, the binding raises instead of computing
  anything another way.
"""
import ast
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2506_02475_gb300")
ORACLE = os.path.join(ROOT, "oracle")


def _imports(path):
    tree = ast.parse(open(path).read())
    names = []
    for node in ast.walk(tree):
        if isinstance(node, ast.Import):
            names += [a.name.split(".")[0] for a in node.names]
        elif isinstance(node, ast.ImportFrom) and node.module and node.level == 0:
            names.append(node.module.split(".")[0])
    return names


def _files(top, exts):
    for d, _, fs in os.walk(top):
        if "_build" in d or "__pycache__" in d:
            continue
        for f in fs:
            if f.endswith(exts):
                yield os.path.join(d, f)


def test_package_never_imports_or_includes_the_oracle():
    for f in _files(PKG, (".py",)):
        assert "oracle" not in _imports(f), f
    for f in _files(PKG, (".cu", ".cuh", ".h", ".cpp")):
        for line in open(f):
            if line.lstrip().startswith("#include"):
                assert "oracle" not in line, (f, line)


def test_oracle_never_imports_the_package():
    pkg = os.path.basename(PKG)
    for f in _files(ORACLE, (".py",)):
        assert pkg not in _imports(f), f
    for f in _files(ORACLE, (".c", ".h")):
        for line in open(f):
            if line.lstrip().startswith("#include"):
                assert pkg not in line and "csrc" not in line, (f, line)


def test_bench_reaches_the_oracle_only_inside_functions():
    tree = ast.parse(open(os.path.join(ROOT, "bench.py")).read())
    top = []
    for node in tree.body:
        if isinstance(node, ast.Import):
            top += [a.name.split(".")[0] for a in node.names]
        elif isinstance(node, ast.ImportFrom) and node.module:
            top.append(node.module.split(".")[0])
    assert "oracle" not in top


def test_binding_raises_when_the_library_cannot_be_built(monkeypatch, tmp_path):
    from paper_2506_02475_gb300 import binding

    def no_build(*a, **k):
        raise RuntimeError("nvcc not found")

    monkeypatch.setattr(binding, "_lib", None)
    monkeypatch.setattr(binding._build, "LIB", str(tmp_path / "missing" / "libcomba.so"))
    monkeypatch.setattr(binding._build, "build", no_build)
    with pytest.raises(RuntimeError, match="nvcc not found"):
        binding.lib()
