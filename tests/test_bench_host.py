"""Host-side logic of bench.py that needs no GPU: the kernel code hash that keys the recorded
DRAM traffic, the count of this library's kernels per timed step, the metric names, and the
CPU-oracle baseline (all-cores and single-thread samples)."""
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


def test_recorded_traffic_applies_only_to_the_code_it_was_captured_on(monkeypatch):
    # a DRAM-traffic figure is keyed by workload and kernel code hash: it is reported for that
    # exact code, and null once the code changes (until a new ncu capture is recorded)
    h = bench.kernel_hash("gemm.cu")
    monkeypatch.setattr(bench, "KERNEL_TRAFFIC", {("flux_qkv", h): 123.0, ("dllm", "0" * 16): 5.0})
    assert bench.recorded_traffic("flux_qkv", "gemm.cu") == 123.0
    assert bench.recorded_traffic("dllm", "gemm.cu") is None
    assert bench.recorded_traffic("flux_out", "gemm.cu") is None


@pytest.mark.parametrize("M,fused,nvfp4,expect", [
    (1, False, False, 2),      # quantiser + few-token kernel
    (16, False, False, 2),
    (64, False, False, 3),     # + operand expansion (pre-expanded tokens)
    (1024, False, False, 3),   # quantiser + operand expansion + GEMM (INT4 or ternary weights)
    (4608, True, False, 2),    # quantise-to-operand + GEMM
    (1, True, False, 2),
    (1024, False, True, 4),    # NVFP4: quantiser + two operand images + GEMM
])
def test_launches_per_step(M, fused, nvfp4, expect):
    assert bench.launches_per_step(M, fused, nvfp4) == expect


def test_metric_names():
    class A:
        weights = "int4"
    assert bench.metric_name(A) == "W4A4 linear TOPS"
    A.weights = "ternary"
    assert bench.metric_name(A) == "W1.58A4 linear TOPS"


def test_oracle_results_do_not_depend_on_its_thread_count():
    import numpy as np
    import oracle
    from paper_2609_33601_gb300 import workloads as wl
    w = wl.make("tiny", seed=3)
    qw, sw = oracle.quantize_f32(w.w, w.G)
    threads = oracle.max_threads()
    outs = []
    try:
        for n in (1, 3, max(threads, 2)):
            oracle.set_threads(n)
            qa, sa = oracle.quantize_bf16(w.x_bits, w.G)
            outs.append((qa, sa) + oracle.linear(qa, sa, qw, sw, w.bias, w.G))
    finally:
        oracle.set_threads(threads)
    assert oracle.max_threads() == threads
    for o in outs[1:]:
        assert all(np.array_equal(a, b) for a, b in zip(outs[0], o))


def test_cpu_baseline_reports_an_all_cores_and_a_single_thread_sample(monkeypatch):
    import oracle
    monkeypatch.setitem(bench.WORKLOADS, "tiny", ("tiny: 64 x 256 -> 256, group64", 64, 256, 256, 64, "tiny"))
    threads = oracle.max_threads()
    o = bench.OracleSample("tiny")
    o.calibrate(0.05)
    cb = o.describe(o.run(o.rows), single_s=0.02)
    assert cb["kind"] == "oracle" and cb["value"] > 0 and 1 <= cb["cores"] <= threads
    st = cb["single_thread"]
    assert st["cores"] == 1 and st["value"] > 0
    assert oracle.max_threads() == threads  # restored
    assert "single_thread" not in o.describe(o.run(o.rows))


class _FakeNvml:
    """Stands in for NvmlClocks: a fixed SM clock, its maximum, reason bits and power."""

    def __init__(self, bits):
        self.bits = bits
        self.calls = 0

    def sample(self):
        self.calls += 1
        return 1965, 2070, self.bits, 1180.5


def test_clock_sampler_decodes_nvml_reason_bits():
    import time
    with bench.ClockSampler(0, nvml=_FakeNvml(0x4 | 0x8 | 0x1)) as c:  # power cap, hw slowdown, idle
        time.sleep(0.05)
    s = c.summary()
    assert s["source"] == "nvml" and s["samples"] >= 2
    assert s["sm_mhz"] == 1965 and s["sm_max_mhz"] == 2070 and s["power_w"] == 1180.5
    # the idle bit is not a throttle reason; the two others keep nvidia-smi's names
    assert s["reasons"] == ["hw_slowdown", "sw_power_cap"]
    with bench.ClockSampler(0, nvml=_FakeNvml(0)) as c:
        time.sleep(0.02)
    assert c.summary()["reasons"] == []


def test_clock_sampler_reports_an_unsampled_region():
    class Dead:
        def sample(self):
            return None
    with bench.ClockSampler(0, nvml=Dead()) as c:
        pass
    assert c.summary()["reasons"] == ["unsampled"]
