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
    current = entry["source_sha"] == bench.kernel_hash("gemm.cu")
    assert bench.ncu_traffic("gemm_attn", "gemm.cu") == (entry["dram_bytes_per_launch"] if current else None)
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


def test_binding_rejects_bad_operands_and_outputs(monkeypatch):
    """GEMM, dequantize, split and quantizer outputs: a CPU operand, a
    wrong-shape or wrong-dtype C, a short workspace or a mismatched QTensor
    raise ValueError before any library call (a bad pointer never reaches a
    kernel).  Device placement is checked first; to reach the shape and dtype
    checks on this CPU-only host, the device check is relaxed to "all on the
    same device" for the second half."""
    import torch
    from paper_2605_31035_gb300 import ops

    def no_lib():
        raise AssertionError("the library must not be reached")
    monkeypatch.setattr(ops, "lib", no_lib)

    def qt(rows, K, dtype=torch.uint8):
        return ops.QTensor(torch.zeros(rows, K // 2, dtype=dtype), torch.zeros(rows, K // 16, dtype=dtype),
                           torch.ones(1))
    a, b = qt(8, 256), qt(16, 256)
    with pytest.raises(ValueError, match="CUDA"):
        ops.mixfp4_gemm(a, b)
    with pytest.raises(ValueError, match="CUDA"):
        ops.mixfp4_dequantize(a)
    with pytest.raises(ValueError, match="CUDA"):
        ops.mixfp4_split_native(a)
    with pytest.raises(ValueError, match="CUDA"):
        ops.mixfp4_gemm_native_fewrows(a, b)

    def same_device(t, device, what):
        ops._require(isinstance(t, torch.Tensor) and t.device == device, f"{what} must be on {device}")
    monkeypatch.setattr(ops, "_check_dev", same_device)
    with pytest.raises(ValueError, match="out must be a float32"):
        ops.mixfp4_gemm(a, b, out=torch.zeros(8, 15))
    with pytest.raises(ValueError, match="out must be a float32"):
        ops.mixfp4_gemm(a, b, out=torch.zeros(8, 16, dtype=torch.float64))
    with pytest.raises(ValueError, match="out must be a float32"):
        ops.mixfp4_gemm(a, b, out=torch.zeros(16, 8).t())
    with pytest.raises(ValueError, match="share K"):
        ops.mixfp4_gemm(a, qt(16, 512))
    with pytest.raises(ValueError, match="status_word"):
        ops.mixfp4_gemm(a, b, status_word=torch.zeros(1, dtype=torch.float32))
    bad = ops.QTensor(a.codes, torch.zeros(8, 8, dtype=torch.uint8), a.tensor_scale)
    with pytest.raises(ValueError, match="scales"):
        ops.mixfp4_gemm(bad, b)
    with pytest.raises(ValueError, match="codes"):
        ops.mixfp4_gemm(qt(8, 256, torch.int8), b)
    with pytest.raises(ValueError, match="tensor_scale"):
        ops.mixfp4_gemm(ops.QTensor(a.codes, a.scales, torch.ones(1, dtype=torch.float64)), b)
    with pytest.raises(ValueError, match="at most 64 rows"):
        ops.mixfp4_gemm_native_fewrows(qt(65, 256), b)
    with pytest.raises(ValueError, match="dense float32"):
        ops.mixfp4_dequantize(a, out=torch.zeros(8, 128))
    x = torch.zeros(8, 256, dtype=torch.bfloat16)
    monkeypatch.setattr(ops, "_check_x", lambda t: None)
    with pytest.raises(ValueError, match="out.codes"):
        ops.mixfp4_quantize(x, out=qt(8, 128))
    with pytest.raises(ValueError, match="workspace"):
        ops.mixfp4_quantize(x, out=qt(8, 256), workspace=torch.zeros(1, dtype=torch.uint8))
    with pytest.raises(ValueError, match="tensor_scale"):
        ops.mixfp4_quantize(x, out=qt(8, 256), tensor_scale=torch.ones(2))
    with pytest.raises(ValueError, match="out.codes"):
        ops.mixfp4_quantize_colwise(x, out=qt(8, 256))
    with pytest.raises(ValueError, match="choice"):
        ops.mixfp4_fake_quantize(x, 3, 16, choice=torch.zeros(8, 8, dtype=torch.int32))
