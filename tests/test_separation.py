"""The CUDA path and the oracle share no code, and the product path has no
CPU fallback.  No GPU.

- No file of the package (Python or CUDA) imports or includes the oracle, and
  the oracle imports nothing of the package.
- The seeded input generators (synth/) import neither.
- The binding fails loudly, before any compute, when the library is missing.
"""
import ast
import glob
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = "paper_2608_02474_gb300"


def _imports(path):
    tree = ast.parse(open(path).read(), filename=path)
    out = set()
    for node in ast.walk(tree):
        if isinstance(node, ast.Import):
            out.update(a.name.split(".")[0] for a in node.names)
        elif isinstance(node, ast.ImportFrom) and node.module and node.level == 0:
            out.add(node.module.split(".")[0])
    return out


def _py(folder):
    return glob.glob(os.path.join(ROOT, folder, "**", "*.py"), recursive=True)


def test_package_never_imports_the_oracle():
    files = _py(PKG)
    assert files
    for f in files:
        assert "oracle" not in _imports(f), f
    for f in glob.glob(os.path.join(ROOT, PKG, "csrc", "*")):
        text = open(f, errors="replace").read()
        assert "oracle" not in text.lower(), f


def test_oracle_never_imports_the_package():
    for f in _py("oracle"):
        assert PKG not in _imports(f), f


def test_input_generators_import_neither_side():
    for f in _py("synth"):
        imps = _imports(f)
        assert "oracle" not in imps and PKG not in imps, f


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    from paper_2608_02474_gb300 import echocache as ec
    monkeypatch.setattr(ec, "_LIB", None)
    monkeypatch.setattr(ec, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="missing"):
        ec.lib()
