"""The product path has no fallback: without libheadguard.so every entry point
raises, and nothing in the package imports the CPU oracle."""
import ast
import os

import pytest

import paper_2609_35800_gb300 as hg
from paper_2609_35800_gb300 import build

PKG = os.path.dirname(os.path.abspath(hg.__file__))


def test_missing_library_raises(monkeypatch, tmp_path):
    monkeypatch.setattr(build, "LIB", str(tmp_path / "libheadguard.so"))
    monkeypatch.setattr(hg, "_lib", None)
    with pytest.raises(RuntimeError, match="not built"):
        hg.library()
    with pytest.raises(RuntimeError, match="not built"):
        hg.hg_status_string(0)
    with pytest.raises(RuntimeError, match="not built"):
        hg.hg_cache_layout(hg.Shape(), hg.QuantConfig(), [[0]])


def test_package_never_imports_the_oracle():
    for name in sorted(os.listdir(PKG)):
        if not name.endswith(".py"):
            continue
        tree = ast.parse(open(os.path.join(PKG, name)).read())
        for node in ast.walk(tree):
            if isinstance(node, ast.Import):
                mods = [a.name for a in node.names]
            elif isinstance(node, ast.ImportFrom):
                mods = [node.module or ""]
            else:
                continue
            assert not any(m == "oracle" or m.startswith("oracle.") for m in mods), (name, mods)


def test_kernel_sources_never_include_the_oracle():
    csrc = os.path.join(PKG, "csrc")
    for name in sorted(os.listdir(csrc)):
        txt = open(os.path.join(csrc, name)).read()
        assert "hg_oracle" not in txt and "oracle/" not in txt, name
