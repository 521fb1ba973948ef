"""The oracle and the CUDA path are independent, and the product path has no
CPU fallback (checked on the sources, CPU only).

* Nothing in the package (binding, build script, kernels, headers) imports,
  includes, links or loads anything from ``oracle/``; the oracle includes no
  header of the package or of ``include/`` and imports none of its modules.
* The seeded input module that both sides use holds none of the method's
  arithmetic (no softmax, exponent, pooling or attention; it does not call
  the binding or the oracle).
* The binding raises when its library cannot be loaded: it never routes a
  call anywhere else.
"""
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2607_06827_gb300")
ORACLE = os.path.join(ROOT, "oracle")
SOURCE_EXT = (".py", ".cu", ".cuh", ".h", ".c", ".cpp")


def _sources(top):
    for dirpath, dirnames, files in os.walk(top):
        dirnames[:] = [d for d in dirnames if d not in ("__pycache__", "_build", "build")]
        for f in files:
            if f.endswith(SOURCE_EXT):
                yield os.path.join(dirpath, f)


def _code(path):
    return open(path, encoding="utf-8").read()


def test_package_never_touches_the_oracle():
    pattern = re.compile(
        r"^\s*(import\s+oracle\b|from\s+oracle\b|#\s*include\s+[\"<][^\">]*oracle)"
        r"|liboracle|speechkv_oracle\.c|oracle_[a-z_]+\s*\(",
        re.M)
    files = list(_sources(PKG)) + list(_sources(os.path.join(ROOT, "include")))
    assert files
    for path in files:
        hits = pattern.findall(_code(path))
        assert not hits, f"{os.path.relpath(path, ROOT)} refers to the oracle: {hits}"


def test_oracle_never_touches_the_package():
    include = re.compile(r'^\s*#\s*include\s+"([^"]+)"', re.M)
    imports = re.compile(r"^\s*(from|import)\s+(paper_2607_06827_gb300|tests)\b", re.M)
    files = list(_sources(ORACLE))
    assert any(p.endswith(".c") for p in files)
    for path in files:
        text = _code(path)
        assert not include.findall(text), f"{os.path.relpath(path, ROOT)} includes a local header"
        assert not imports.findall(text), f"{os.path.relpath(path, ROOT)} imports the package"
        assert "speechkv.h" not in text and "libspeechkv" not in text


def test_input_module_holds_no_method_arithmetic():
    text = _code(os.path.join(PKG, "inputs.py"))
    code = re.sub(r'"""(.*?)"""', "", text, flags=re.S)      # docstrings
    code = re.sub(r"#.*", "", code)                          # comments
    code = re.sub(r"^\s*@.*$", "", code, flags=re.M)          # decorators
    for banned in ("softmax", "exp(", "logsumexp", "einsum", "matmul", "@",
                   "speechkv", "oracle", "compressed_len", "pool"):
        assert banned not in code, f"inputs.py uses {banned!r}"


def test_binding_raises_without_its_library(tmp_path, monkeypatch):
    from paper_2607_06827_gb300 import speechkv
    monkeypatch.setattr(speechkv, "_lib", None)  # as in a fresh process
    missing = str(tmp_path / "libspeechkv.so")
    with pytest.raises(RuntimeError, match="no fallback"):
        speechkv.load(missing)
