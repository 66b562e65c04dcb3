"""The product path (CPU checks): the binding fails loudly when the CUDA
library is missing instead of falling back to anything, and no file of the
product package reads, imports or links the oracle."""
import ast
import os

import pytest
import torch

from paper_2608_13524_gb300 import dart
from workloads import TOY

PKG = os.path.dirname(os.path.abspath(dart.__file__))


def test_missing_library_raises(monkeypatch, tmp_path):
    monkeypatch.setattr(dart, "LIB_PATH", str(tmp_path / "libdart.so"))
    monkeypatch.setattr(dart, "_lib", None)
    with pytest.raises(RuntimeError, match="not found"):
        dart.lib()
    w = torch.zeros(4, dtype=torch.float32)
    with pytest.raises(RuntimeError, match="not found"):
        dart.Dart(TOY, w, w, w)


def test_product_package_does_not_use_the_oracle():
    for root, _, files in os.walk(PKG):
        if "_build" in root or "__pycache__" in root:
            continue
        for f in files:
            p = os.path.join(root, f)
            if f.endswith(".py"):
                tree = ast.parse(open(p).read())
                for node in ast.walk(tree):
                    if isinstance(node, ast.Import):
                        assert not any(a.name.split(".")[0] == "oracle" for a in node.names), p
                    elif isinstance(node, ast.ImportFrom):
                        assert (node.module or "").split(".")[0] != "oracle", p
            elif f.endswith((".cu", ".cuh", ".h", ".cpp", ".c")):
                assert "oracle" not in open(p).read().lower(), p
