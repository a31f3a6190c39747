"""The oracle and the CUDA path share no code: no module of either imports, includes or loads
the other (the seeded input generators in synth/ are the only common dependency, and they hold
none of the method's arithmetic)."""
import ast
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = "paper_2607_26253_gb300"


def _files(sub, exts):
    for d, _, fs in os.walk(os.path.join(ROOT, sub)):
        if "__pycache__" in d or "_build" in d:
            continue
        for f in fs:
            if f.endswith(exts):
                yield os.path.join(d, f)


def _py_imports(path):
    tree = ast.parse(open(path).read(), path)
    for node in ast.walk(tree):
        if isinstance(node, ast.Import):
            for a in node.names:
                yield a.name
        elif isinstance(node, ast.ImportFrom):
            yield (node.module or "") if node.level == 0 else "." + (node.module or "")


def test_product_path_does_not_use_the_oracle():
    for path in _files(PKG, (".py",)):
        for mod in _py_imports(path):
            assert not mod.split(".")[0] == "oracle", (path, mod)
    for path in _files(PKG, (".cu", ".cuh", ".h", ".c")):
        text = open(path).read()
        assert not re.search(r'#include\s+["<][^">]*oracle', text), path


def test_oracle_does_not_use_the_product_path():
    for path in _files("oracle", (".py",)):
        for mod in _py_imports(path):
            assert not mod.split(".")[0] in (PKG, "bench", "__graft_entry__"), (path, mod)
    for path in _files("oracle", (".c", ".h")):
        text = open(path).read()
        assert not re.search(r'#include\s+["<][^">]*(csrc|sara\.h)', text), path
        assert "libsara" not in text, path


def test_input_generators_import_neither_side():
    for path in _files("synth", (".py",)):
        for mod in _py_imports(path):
            assert mod.split(".")[0] not in ("oracle", PKG), (path, mod)
