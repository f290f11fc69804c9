"""Host-side logic of bench.py that needs no GPU: the kernel code hash that keys the recorded
DRAM traffic, the count of this library's kernels per timed step, and the metric names."""
import os
import shutil

import pytest

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_kernel_hash_ignores_comments_and_whitespace_but_not_code(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2609_33601_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in ("operand.cuh", "ptx.cuh"):
        shutil.copy(os.path.join(ROOT, "paper_2609_33601_gb300", "csrc", f), csrc / f)
    src = "// a kernel\n__global__ void k(int* p) {\n  p[0] = 1;  /* one */\n}\n"
    (csrc / "k.cu").write_text(src)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.kernel_hash("k.cu")
    (csrc / "k.cu").write_text("/* the same kernel,\n   documented */\n__global__ void k(int* p) {\n    p[0] = 1;\n}\n")
    assert bench.kernel_hash("k.cu") == h0
    (csrc / "k.cu").write_text(src.replace("p[0] = 1", "p[0] = 2"))
    assert bench.kernel_hash("k.cu") != h0


def test_recorded_traffic_matches_the_current_kernels():
    # the traffic figures in bench.py were taken on the current kernel code (profiles/)
    assert ("dllm", bench.kernel_hash("gemm.cu")) in bench.KERNEL_TRAFFIC
    assert ("sweep_m1", bench.kernel_hash("skinny.cu")) in bench.KERNEL_TRAFFIC


@pytest.mark.parametrize("M,few,fused,ternary,expect", [
    (1, True, False, False, 2),      # quantiser + few-token kernel
    (16, True, False, False, 2),
    (64, True, False, False, 3),     # + operand expansion (pre-expanded tokens)
    (1024, False, False, False, 3),  # quantiser + operand expansion + GEMM
    (1024, False, False, True, 4),   # + ternary -> INT4 rewrite
    (64, True, False, True, 3),
    (4608, False, True, False, 2),   # quantise-to-operand + GEMM
    (1, True, True, False, 2),
])
def test_launches_per_step(M, few, fused, ternary, expect):
    assert bench.launches_per_step(M, few, fused, ternary) == expect


def test_metric_names():
    class A:
        weights = "int4"
    assert bench.metric_name(A) == "W4A4 linear TOPS"
    A.weights = "ternary"
    assert bench.metric_name(A) == "W1.58A4 linear TOPS"
