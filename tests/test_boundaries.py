"""Structural rules of the repository, checked on CPU: the CUDA product path
and the CPU oracle share no code and neither imports the other; the product
path fails loudly without its library (no CPU fallback); every compute entry
point of the C ABI cites the passage it implements; the bench drops a DRAM
traffic figure taken on other kernel source."""
import ast
import importlib
import json
import os
import re
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2605_31035_gb300")


def _imports(path):
    tree = ast.parse(open(path).read())
    names = set()
    for node in ast.walk(tree):
        if isinstance(node, ast.Import):
            names.update(a.name.split(".")[0] for a in node.names)
        elif isinstance(node, ast.ImportFrom) and node.module and node.level == 0:
            names.add(node.module.split(".")[0])
    return names


def test_product_package_never_imports_the_oracle():
    for f in os.listdir(PKG):
        if f.endswith(".py"):
            assert "oracle" not in _imports(os.path.join(PKG, f)), f


def test_cuda_sources_include_nothing_from_the_oracle():
    csrc = os.path.join(PKG, "csrc")
    for f in os.listdir(csrc):
        text = open(os.path.join(csrc, f)).read()
        for inc in re.findall(r'#include\s+[<"]([^>"]+)[>"]', text):
            assert "oracle" not in inc, (f, inc)


def test_oracle_imports_nothing_from_the_product_path():
    odir = os.path.join(ROOT, "oracle")
    for f in os.listdir(odir):
        if f.endswith(".py"):
            assert "paper_2605_31035_gb300" not in _imports(os.path.join(odir, f)), f
    text = open(os.path.join(odir, "mixfp4_oracle.c")).read()
    assert "csrc" not in " ".join(re.findall(r'#include\s+[<"]([^>"]+)[>"]', text))


def test_binding_fails_loudly_without_the_library(tmp_path, monkeypatch):
    from paper_2605_31035_gb300 import ops
    monkeypatch.setattr(ops, "_lib", None)
    monkeypatch.setattr(ops, "_LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="missing"):
        ops.lib()


CITATION = re.compile(r"\b(Sec\.|Alg\.|Algorithm|App\.|Eq\.|Table)\s*\d|\bApp\. [A-Z]|Algorithm 1|reading R\d+")


def test_every_compute_entry_point_cites_the_paper():
    """Each declaration's comment block names a section, algorithm,
    appendix, equation, table or reading, or defines the entry point through
    another declared one (whose block is checked in turn)."""
    text = open(os.path.join(ROOT, "include", "mixfp4.h")).read()
    utility = {"mixfp4_status_string", "mixfp4_version", "mixfp4_selftest_bounded_wait"}
    blocks = {}
    for m in re.finditer(r"/\*(.*?)\*/\s*((?:int|const char\s*\*)\s+(mixfp4_\w+)\s*\(.*?\);(?:\s*int\s+(mixfp4_\w+)\s*\(.*?\);)?)",
                         text, flags=re.S):
        for name in (m.group(3), m.group(4)):
            if name:
                blocks[name] = m.group(1)
    declared = set(re.findall(r"\b(mixfp4_\w+)\s*\(", re.sub(r"/\*.*?\*/", "", text, flags=re.S)))
    for name in sorted(declared - utility):
        assert name in blocks, f"{name} has no comment block"
        refers = any(o != name and re.search(rf"\b{o}\b", blocks[name]) for o in declared)
        assert CITATION.search(blocks[name]) or refers, name


def test_stale_traffic_figure_is_dropped(tmp_path, monkeypatch):
    import sys
    sys.path.insert(0, ROOT)
    bench = importlib.import_module("bench")
    entry = json.load(open(os.path.join(ROOT, "profiles", "ncu_traffic.json")))["gemm_attn"]
    assert bench.ncu_traffic("gemm_attn", "gemm.cu") == entry["dram_bytes_per_launch"]
    fake_root = tmp_path / "r"
    shutil.copytree(os.path.join(ROOT, "profiles"), fake_root / "profiles")
    os.makedirs(fake_root / "paper_2605_31035_gb300" / "csrc")
    (fake_root / "paper_2605_31035_gb300" / "csrc" / "gemm.cu").write_text("// another kernel\n")
    monkeypatch.setattr(bench, "ROOT", str(fake_root))
    assert bench.ncu_traffic("gemm_attn", "gemm.cu") is None


def test_binding_rejects_bad_arguments_before_the_library(monkeypatch):
    """The binding's checks raise ValueError (they stay on under python -O)
    and run before any library call: a CPU tensor, a wrong dtype, a bad block
    size or output dtype never reaches the C ABI."""
    import torch
    from paper_2605_31035_gb300 import ops

    def no_lib():
        raise AssertionError("the library must not be reached")
    monkeypatch.setattr(ops, "lib", no_lib)
    x_cpu = torch.zeros(4, 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="CUDA"):
        ops.mixfp4_quantize(x_cpu)
    with pytest.raises(ValueError, match="CUDA"):
        ops.mixfp4_quantize_2d(x_cpu.float())
    with pytest.raises(ValueError):
        ops.mixfp4_fake_quantize(x_cpu, 15, 16)
    with pytest.raises(ValueError):
        ops.mixfp4_quantize_rht(x_cpu, signs=torch.zeros(8, dtype=torch.uint8))
