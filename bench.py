"""Benchmark of the naive W4A4 linear layer (JustQuant, arxiv 2609.33601) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload flux_qkv] [--impl ours|reference]

One step = one pass of the deployed hot path over one batch: the activation quantiser
(jq_quantize_act) followed by the W4A4 GEMM with its dequantise + bias epilogue
(jq_w4a4_linear).  The default workload is the largest single-GPU configuration, the FLUX-style
12B DiT's fused QKV+MLP-in projection (M=4608 tokens x K=3072 -> N=21504, group64, the FLUX
setting of Sec. 4.2 and the Appendix "FLUX experimental details").  Weights are packed once,
offline, as the paper's deployment does.  Rotating input/weight sets, together several times
larger than the 129 MB L2, make every step stream its operands from HBM.  Metric: W4A4 linear
TOPS (2*M*N*K per step), whole job over all ranks.

Other workloads (--workload): the dLLM gate/up projection (group128), the FLUX output
projection (also as the fused call, --fused), the M sweep of the memory-to-compute crossover,
and, as their own lines, the memory-bound kernels alone: the activation quantiser, the
training-side fake quantisation and the straight-through backward (GB/s against the HBM copy
rate).

Under torchrun each rank runs its own replica of the workload (the layer shards along tokens
with no exchange), so scaling is weak and no collective sits on the data path; a barrier and a
max-reduction of the timings bracket the timed region.

--impl reference times the CPU oracle (oracle/, the plain C reference of the same layer) on
the host cores, on a bounded row sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOADS = {
    # name: (description, M, K, N, G, generator in workloads.py)
    "dllm": ("dLLM 8B gate/up projection: M=1024 tokens x K=4096 -> N=12288, group128", 1024, 4096, 12288, 128,
             "dllm"),
    "flux_qkv": ("FLUX 12B DiT fused QKV+MLP-in: M=4608 x K=3072 -> N=21504, group64", 4608, 3072, 21504, 64,
                 "flux_qkv"),
    "flux_out": ("FLUX 12B DiT output projection: M=4608 x K=15360 -> N=3072, group64", 4608, 15360, 3072, 64,
                 "flux_out"),
    "dllm_gk": ("dLLM 8B gate/up projection, per-token/per-channel scales: M=1024 x K=4096 -> N=12288, group = K",
                1024, 4096, 12288, 4096, "dllm"),
    # M-sweep points below the memory-to-compute crossover (per-token / per-channel: group = K);
    # these run the few-token kernel and are bound by streaming the packed weights from HBM
    "sweep_m1": ("M sweep: M=1 token x K=4096 -> N=12288, per-token/per-channel (group = K)", 1, 4096, 12288,
                 4096, "sweep_a"),
    "sweep_m16": ("M sweep: M=16 tokens x K=4096 -> N=12288, per-token/per-channel (group = K)", 16, 4096, 12288,
                  4096, "sweep_a"),
    "sweep_m64": ("M sweep: M=64 tokens x K=4096 -> N=12288, per-token/per-channel (group = K)", 64, 4096, 12288,
                  4096, "sweep_a"),
}
# DiT-XL/2 block linears (16 images of 256 tokens, group128) with the neighbour operation that
# feeds each one fused into the activation quantiser: the adaLN modulation before the attention's
# QKV projection and the MLP's first linear, the tanh GELU before the MLP's second linear; the
# attention output projection takes the plain quantiser.
DIT = {
    "dit_qkv": ("DiT-XL/2 attention QKV: 16 images x 256 tokens = 4096 x 1152 -> 3456, group128, "
                "modulation fused into the quantiser", 4096, 1152, 3456, 128, "dit", "modulate"),
    "dit_proj": ("DiT-XL/2 attention output projection: 4096 x 1152 -> 1152, group128", 4096, 1152, 1152, 128, "dit",
                 None),
    "dit_fc1": ("DiT-XL/2 MLP in: 4096 x 1152 -> 4608, group128, modulation fused into the quantiser", 4096, 1152,
                4608, 128, "dit", "modulate"),
    "dit_fc2": ("DiT-XL/2 MLP out: 4096 x 4608 -> 1152, group128, tanh GELU fused into the quantiser", 4096, 4608,
                1152, 128, "dit", "gelu"),
}
for _n, _v in DIT.items():
    WORKLOADS[_n] = _v[:6]
DIT_PROLOGUE = {n: v[6] for n, v in DIT.items()}
# The whole M sweep of the memory-to-compute crossover, at both shapes (per-token/per-channel
# scales, group = K): M <= 64 runs the few-token kernel, larger M the GEMM.
SWEEP_M = (1, 16, 64, 256, 1024, 4096, 16384)
for _m in SWEEP_M:
    WORKLOADS[f"sweep_a_m{_m}"] = (f"M sweep A: M={_m} x K=4096 -> N=12288, group = K", _m, 4096, 12288, 4096,
                                   "sweep_a")
    WORKLOADS[f"sweep_b_m{_m}"] = (f"M sweep B: M={_m} x K=3072 -> N=3072, group = K", _m, 3072, 3072, 3072,
                                   "sweep_b")
FEW_TOKENS = 64  # M at or below this takes the few-token (weight-streaming) kernel
PEAKS_PATH = os.path.join(ROOT, "MEASURED_PEAKS.json")
FP8_PER_BF16 = 2.0  # nominal dense FP8 / BF16 tensor-core ratio on GB300 (4.5 / 2.25 PFLOP/s)

# DRAM traffic of one launch of the dominant kernel (dram__bytes_read.sum + dram__bytes_write.sum)
# from an ncu capture of that kernel, keyed by workload and by the hash of the kernel code the
# capture was taken on (kernel_hash); once the code changes the figure no longer applies and the
# bench reports null until a new capture is recorded here.
KERNEL_TRAFFIC: dict = {}


def recorded_traffic(workload: str, kernel_file: str):
    """The captured DRAM bytes per launch for this workload on the current kernel code, or None."""
    return KERNEL_TRAFFIC.get((workload, kernel_hash(kernel_file)))


def kernel_hash(kernel_file: str) -> str:
    """Hash of a kernel's code (its .cu file and the two headers it is built from), comments and
    whitespace removed, so that only a change of the code itself retires a traffic figure."""
    import re
    h = hashlib.sha256()
    for f in (kernel_file, "operand.cuh", "ptx.cuh"):
        with open(os.path.join(ROOT, "paper_2609_33601_gb300", "csrc", f)) as fh:
            text = fh.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)  # block comments
        text = re.sub(r"//[^\n]*", " ", text)                 # line comments
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()[:16]


def max_over_ranks(values, device):
    """Each timing's maximum over the ranks (one replica of the workload per rank): the
    whole job is as slow as its slowest rank.  The identity on a single process."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.cpu()]


def whole_job_tops(world: int, ops_per_step: float, steps: int, seconds: float) -> float:
    """Whole-job throughput of `world` replicas that each ran `steps` steps of `ops_per_step`
    operations in at most `seconds` (the max over ranks)."""
    return world * ops_per_step * steps / seconds / 1e12


def metric_name(args) -> str:
    return {"ternary": "W1.58A4 linear TOPS", "nvfp4": "NVFP4 W4A4 linear TOPS"}.get(args.weights, "W4A4 linear TOPS")


def launches_per_step(M: int, fused: bool, nvfp4: bool = False) -> int:
    """Kernels of this library per timed step: the activation quantiser (or, fused, the
    quantise-to-operand kernel), the operand expansion when the linear kernel reads the operand
    image (more than 16 tokens), and the linear kernel itself (ternary weights are read as
    2-bit codes by both linear kernels)."""
    if fused:
        return 2
    if nvfp4:  # quantiser, the two operand images, GEMM
        return 4
    return 1 + (1 if M > 16 else 0) + 1


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


class NvmlClocks:
    """SM clock, its maximum, the clock-event (throttle) reason bits and the power draw of one
    GPU, read through NVML (libnvidia-ml, installed with the driver) by ctypes: read-only
    queries, a few microseconds each, so the timed region gets sampled many times."""

    CLOCK_SM = 1  # NVML_CLOCK_SM

    def __init__(self, index: int, uuid: str | None = None):
        import ctypes
        c = ctypes
        lib = c.CDLL("libnvidia-ml.so.1")
        lib.nvmlDeviceGetHandleByIndex_v2.argtypes = [c.c_uint, c.POINTER(c.c_void_p)]
        lib.nvmlDeviceGetUUID.argtypes = [c.c_void_p, c.c_char_p, c.c_uint]
        lib.nvmlDeviceGetClockInfo.argtypes = [c.c_void_p, c.c_int, c.POINTER(c.c_uint)]
        lib.nvmlDeviceGetMaxClockInfo.argtypes = [c.c_void_p, c.c_int, c.POINTER(c.c_uint)]
        lib.nvmlDeviceGetPowerUsage.argtypes = [c.c_void_p, c.POINTER(c.c_uint)]
        reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None)
        if reasons is None:
            reasons = lib.nvmlDeviceGetCurrentClocksThrottleReasons
        reasons.argtypes = [c.c_void_p, c.POINTER(c.c_ulonglong)]
        if lib.nvmlInit_v2() != 0:
            raise OSError("nvmlInit_v2 failed")
        self._c, self._lib, self._reasons = c, lib, reasons
        try:
            self.handle = self._find(index, uuid)
        except Exception:
            lib.nvmlShutdown()
            raise

    def _find(self, index, uuid):
        """The device whose UUID is the CUDA device's (CUDA and NVML may number GPUs differently),
        else NVML index `index`."""
        c, lib = self._c, self._lib
        count = c.c_uint(0)
        if uuid and lib.nvmlDeviceGetCount_v2(c.byref(count)) == 0:
            buf = c.create_string_buffer(96)
            for i in range(count.value):
                h = c.c_void_p()
                if (lib.nvmlDeviceGetHandleByIndex_v2(i, c.byref(h)) == 0
                        and lib.nvmlDeviceGetUUID(h, buf, 96) == 0
                        and buf.value.decode().lower().endswith(uuid.lower())):
                    return h
        h = c.c_void_p()
        if lib.nvmlDeviceGetHandleByIndex_v2(index, c.byref(h)) != 0:
            raise OSError(f"no NVML device {index}")
        return h

    def sample(self):
        c, lib, h = self._c, self._lib, self.handle
        sm, mx, pw, r = c.c_uint(), c.c_uint(), c.c_uint(), c.c_ulonglong()
        if (lib.nvmlDeviceGetClockInfo(h, self.CLOCK_SM, c.byref(sm)) != 0
                or lib.nvmlDeviceGetMaxClockInfo(h, self.CLOCK_SM, c.byref(mx)) != 0
                or self._reasons(h, c.byref(r)) != 0):
            return None
        power = pw.value / 1000.0 if lib.nvmlDeviceGetPowerUsage(h, c.byref(pw)) == 0 else None
        return sm.value, mx.value, r.value, power

    def close(self):
        self._lib.nvmlShutdown()


# NVML clock-event reason bits (nvmlClocksEventReason*) and the names nvidia-smi gives them.
CLOCK_REASON_BITS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
                     0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}


class ClockSampler:
    """Samples SM clocks and throttle reasons while the timed region runs: through NVML every
    5 ms, or, where NVML cannot be loaded, with nvidia-smi (one sample per call, ~0.2 s apart)."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, gpu_index: int, uuid: str | None = None, nvml=None):
        self.gpu = gpu_index
        self.uuid = uuid
        self.samples = []  # (sm MHz, max MHz, reason names, power W)
        self.source = None
        self._nvml = nvml
        self._stop = threading.Event()
        self._thread = None

    def _run_nvml(self):
        while not self._stop.is_set():
            s = self._nvml.sample()
            if s is not None:
                sm, mx, bits, power = s
                self.samples.append((float(sm), float(mx),
                                     [n for b, n in CLOCK_REASON_BITS.items() if bits & b], power))
            self._stop.wait(0.005)

    def _run_smi(self):
        gpu = f"GPU-{self.uuid}" if self.uuid and not self.uuid.startswith("GPU-") else (self.uuid or self.gpu)
        while not self._stop.is_set():
            try:
                out = subprocess.run(["nvidia-smi", f"--id={gpu}", f"--query-gpu={self.QUERY}",
                                      "--format=csv,noheader,nounits"], capture_output=True, text=True, timeout=5)
                if out.returncode == 0 and out.stdout.strip():
                    v = [x.strip() for x in out.stdout.strip().split(",")]
                    num = lambda t: float(t) if t.replace(".", "").isdigit() else None  # noqa: E731
                    self.samples.append((num(v[1]), num(v[2]),
                                         [n for n, a in zip(self.NAMES, v[5:9]) if a.lower() == "active"],
                                         num(v[3])))
            except Exception:
                return
            self._stop.wait(0.2)

    def __enter__(self):
        if self._nvml is None:
            try:
                self._nvml = NvmlClocks(self.gpu, self.uuid)
            except Exception:
                self._nvml = None
        self.source = "nvml" if self._nvml is not None else "nvidia-smi"
        self._thread = threading.Thread(target=self._run_nvml if self._nvml is not None else self._run_smi,
                                        daemon=True)
        self._thread.start()
        return self

    def __exit__(self, *exc):
        self._stop.set()
        if self._thread:
            self._thread.join(timeout=10)
        if isinstance(self._nvml, NvmlClocks):
            self._nvml.close()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "source": self.source}
        sm = [s[0] for s in self.samples if s[0] is not None]
        mx = [s[1] for s in self.samples if s[1] is not None]
        pw = [s[3] for s in self.samples if s[3] is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted({n for s in self.samples for n in s[2]}), "samples": len(self.samples),
                "power_w": round(statistics.median(pw), 1) if pw else None, "source": self.source}


def device_uuid(torch, dev) -> str | None:
    """The CUDA device's UUID (to find the same GPU in NVML), where this PyTorch reports it."""
    try:
        return str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        return None


def measured_peaks():
    try:
        with open(PEAKS_PATH) as f:
            p = json.load(f)
        return float(p["bf16_tflops"]), float(p["hbm_gbs"]), "measured"
    except Exception:
        return 1900.0, 6800.0, "fallback"


# ----------------------------------------------------------------------------- reference arm

class OracleSample:
    """The CPU oracle, as it stands, on a bounded row sample of the workload: quantise the
    sampled activation rows and evaluate the linear layer for them (the weights are packed
    once, outside the timing, as on the GPU)."""

    def __init__(self, name: str, seed: int = 7, ternary: bool = False, fmt: str | None = None):
        import oracle
        from paper_2609_33601_gb300 import workloads as wl
        self.oracle = oracle
        self.wl = wl
        self.name = name
        self.fmt = fmt or ("ternary" if ternary else "int4")
        self.desc, self.M, self.K, self.N, self.G, gen = WORKLOADS[name]
        w = wl.make(gen, seed=seed, M=self.M, K=self.K, N=self.N, G=self.G)
        self.x_bits, self.bias = w.x_bits, w.bias
        if self.fmt == "nvfp4":  # weights with their own tensor scale; activations with a calibrated one
            self.gw = oracle.nvfp4_tensor_scale(w.w)
            self.qw, self.sw = oracle.quantize_nvfp4(w.w, self.gw)
            self.ga = oracle.nvfp4_tensor_scale(wl.bf16_bits_to_f32(self.x_bits))
        else:
            quant = oracle.quantize_ternary_f32 if self.fmt == "ternary" else oracle.quantize_f32
            self.qw, self.sw = quant(w.w, self.G)
        self.rows = 8
        self.run_s = 0.0
        self.tokens_per_sample = wl.DIT_TOKENS_PER_IMAGE
        self.mod = wl.dit_modulation(seed, -(-self.M // self.tokens_per_sample), self.K)

    def run(self, rows: int) -> float:
        t0 = time.perf_counter()
        if self.fmt == "nvfp4":
            qa2, sa = self.oracle.quantize_nvfp4(self.wl.bf16_bits_to_f32(self.x_bits[:rows]), self.ga)
            self.oracle.linear_nvfp4(qa2, sa, self.ga, self.qw, self.sw, self.gw, self.bias)
            return time.perf_counter() - t0
        prologue = DIT_PROLOGUE.get(self.name)
        if prologue == "modulate":
            _, qa, sa = self.oracle.modulate_quantize_bf16(self.x_bits[:rows], self.mod[0], self.mod[1],
                                                           self.tokens_per_sample, self.G)
        elif prologue == "gelu":
            _, qa, sa = self.oracle.gelu_quantize_bf16(self.x_bits[:rows], self.G)
        else:
            qa, sa = self.oracle.quantize_bf16(self.x_bits[:rows], self.G)
        self.oracle.linear(qa, sa, self.qw, self.sw, self.bias, self.G)
        return time.perf_counter() - t0

    def calibrate(self, target_s: float) -> int:
        rows = 8
        while True:
            dt = self.run(rows)
            if dt >= 0.8 * target_s or rows >= self.M:
                break
            rows = min(self.M, max(rows * 2, int(rows * target_s / max(dt, 1e-3))))
        self.rows = rows
        return rows

    def ops(self, rows: int | None = None) -> float:
        return 2.0 * (self.rows if rows is None else rows) * self.N * self.K

    def single_thread(self, target_s: float) -> dict:
        """The same oracle on one host thread, on a row sample sized for about target_s."""
        threads = self.oracle.max_threads()
        self.oracle.set_threads(1)
        try:
            used = min(threads, self.rows)  # the all-cores sample ran on this many threads
            rows = max(1, min(self.rows, int(self.rows * target_s / max(self.run_s * used, 1e-3))))
            dt = self.run(rows)
        finally:
            self.oracle.set_threads(threads)
        return {"value": self.ops(rows) / dt / 1e12, "cores": 1,
                "sample": f"{rows} token rows, {dt:.2f} s"}

    def describe(self, dt: float, single_s: float = 0.0) -> dict:
        self.run_s = dt
        cores = self.oracle.max_threads()
        out = {"value": self.ops() / dt / 1e12, "unit": "TOPS", "cores": min(cores, self.rows), "kind": "oracle",
               "host_threads": os.cpu_count(),
               "sample": f"{self.rows} of {self.M} token rows of the {self.name} workload (all N={self.N} "
                         f"outputs), quantise + linear, {dt:.2f} s per sample"}
        if single_s > 0:
            out["single_thread"] = self.single_thread(single_s)
        return out


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    o = OracleSample(args.workload, fmt=args.weights)
    per_step = min(args.ref_seconds, 120.0 / (args.steps + args.warmup))
    o.calibrate(per_step)
    for _ in range(args.warmup):
        o.run(o.rows)
    times = [o.run(o.rows) for _ in range(args.steps)]
    mean = sum(times) / len(times)
    cb = o.describe(mean, single_s=args.ref_single_seconds)
    value = cb["value"]
    line = {"impl": "reference", "metric": metric_name(args), "value": value, "unit": "TOPS", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": mean * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int4", "data": "synthetic",
            "config": {"workload": o.desc, "M": o.M, "K": o.K, "N": o.N, "group": o.G},
            "cpu_baseline": cb, "e2e": {"value": value, "unit": "TOPS", "h2d_bytes_per_step": 0,
                                        "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_stream_reference(args):
    """The reference arm of a memory-bound kernel line: the oracle's version on the host cores."""
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    o = StreamOracle(args.workload)
    cb = o.baseline(min(args.ref_seconds, 120.0 / (args.steps + args.warmup)))
    line = {"impl": "reference", "metric": STREAM_METRIC[o.op], "value": cb["value"], "unit": "GB/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if o.op != "fq_weight" else "f32",
            "data": "synthetic", "config": {"workload": o.desc, "rows": o.M, "K": o.K, "group": o.G},
            "cpu_baseline": cb, "e2e": {"value": cb["value"], "unit": "GB/s", "h2d_bytes_per_step": 0,
                                        "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- context

def cublas_context(torch, dev, sets, M, N, K, args, world):
    """cuBLAS bf16 GEMM of the same shape (y = x W^T, bf16 weights), for context: rotating bf16
    weight sets together larger than L2, K launches captured in a CUDA graph, timed with CUDA
    events like the linear layer."""
    wbytes = N * K * 2
    n_w = max(2, -(-300_000_000 // wbytes))
    if n_w * wbytes > 4_000_000_000:
        return {"skipped": "bf16 weight sets would exceed 4 GB"}
    gen = torch.Generator(device=dev)
    gen.manual_seed(5)
    ws = [(torch.randn((N, K), device=dev, generator=gen) * 0.02).to(torch.bfloat16) for _ in range(n_w)]
    xs = [sets[i % len(sets)][0] for i in range(n_w)]
    out = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
    cap = torch.cuda.Stream()
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(cap):
        for i in range(args.warmup):
            torch.matmul(xs[i % n_w], ws[i % n_w].t(), out=out)
    cap.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=cap):
        for i in range(args.steps):
            torch.matmul(xs[i % n_w], ws[i % n_w].t(), out=out)
    g.replay()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    g.replay()
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / args.steps
    del ws, g
    torch.cuda.empty_cache()
    return {"value": world * 2.0 * M * N * K / (ms * 1e-3) / 1e12, "unit": "TFLOP/s", "ms_per_call": ms,
            "what": "torch.matmul bf16 x[M,K] @ W[N,K]^T, same M, N, K"}


def copy_context(torch, dev, nbytes, args, world):
    """What a device-to-device copy of as many bytes as the linear layer moves takes, for the
    HBM-bound lines (the measured HBM peak is a copy rate): rotating source and destination
    buffers (together larger than L2), K copies captured in a CUDA graph and timed with CUDA
    events like the linear layer; GB/s counts the bytes read and written.  At a few MB a
    launch's fixed costs, not HBM, set the copy's rate too."""
    n = max(4096, (nbytes // 16) * 16)
    n_b = max(2, -(-300_000_000 // (2 * n)))
    src = [torch.ones(n, dtype=torch.uint8, device=dev) for _ in range(n_b)]
    dst = [torch.empty(n, dtype=torch.uint8, device=dev) for _ in range(n_b)]
    cap = torch.cuda.Stream()
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(cap):
        for i in range(args.warmup):
            dst[i % n_b].copy_(src[i % n_b])
    cap.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=cap):
        for i in range(args.steps):
            dst[i % n_b].copy_(src[i % n_b])
    g.replay()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record()
    g.replay()
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / args.steps
    del src, dst, g
    torch.cuda.empty_cache()
    return {"value": world * 2 * n / (ms * 1e-3) / 1e9, "unit": "GB/s", "ms_per_call": ms, "bytes": n,
            "what": "device-to-device copy of the linear's algorithmic bytes (rotating buffers > L2), K copies "
                    "in a CUDA graph; GB/s counts bytes read + written, like the measured HBM peak"}


def prologue_context(torch, jq, sets, mods, prologue, G, T, q, s_a, args):
    """The DiT neighbour operation fused into the quantiser against the same operation done
    separately (PyTorch bf16 ops writing the activation, then jq_quantize_act reading it back),
    each as a CUDA graph of K launches over the rotating inputs."""
    n = len(sets)

    def graph_ms(fn):
        cap = torch.cuda.Stream()
        cap.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(cap):
            for i in range(args.warmup):
                fn(i, cap)
        cap.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap):
            for i in range(args.steps):
                fn(i, cap)
        g.replay()
        torch.cuda.synchronize()
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record()
        g.replay()
        t1.record()
        torch.cuda.synchronize()
        return t0.elapsed_time(t1) / args.steps

    def fused(i, st):
        x = sets[i % n][0]
        if prologue == "modulate":
            jq.jq_modulate_quantize_act(x, mods[i % n][0], mods[i % n][1], T, G, q, s_a, stream=st)
        else:
            jq.jq_gelu_quantize_act(x, G, q, s_a, stream=st)

    def separate(i, st):
        x = sets[i % n][0]
        M = x.shape[0]
        if prologue == "modulate":
            sh, sc = mods[i % n]
            rows = torch.arange(M, device=x.device) // T
            z = (x.float() * (1.0 + sc[rows]) + sh[rows]).to(torch.bfloat16)
        else:
            z = torch.nn.functional.gelu(x, approximate="tanh")
        jq.jq_quantize_act(z, G, q, s_a, stream=st)

    f, sep = graph_ms(fused), graph_ms(separate)
    return {"fused_us": f * 1e3, "separate_us": sep * 1e3,
            "what": f"{prologue} fused into the activation quantiser vs the PyTorch {prologue} writing bf16 "
                    "followed by jq_quantize_act (per launch, CUDA graph)"}


# ----------------------------------------------------------------------------- memory-bound kernels

# The HBM-bound kernels of the library timed alone: name -> (description, op, rows, K, G, generator).
# op: "quantize" (jq_quantize_act), "fq_act" (jq_fake_quant_act), "fq_weight"
# (jq_fake_quant_weight, fp32 rows), "ste" (jq_ste_backward over rows x K gradients).
STREAM_WORKLOADS = {
    "quant_dllm": ("activation quantiser on the dLLM activations: 1024 x 4096 bf16, group128", "quantize", 1024,
                   4096, 128, "dllm"),
    "quant_flux_out": ("activation quantiser on the FLUX output projection's input: 4608 x 15360 bf16, group64",
                       "quantize", 4608, 15360, 64, "flux_out"),
    "fq_act_dllm": ("training-side fake quantisation of activations: 1024 x 4096 bf16, group128", "fq_act", 1024,
                    4096, 128, "dllm"),
    "fq_act_flux_out": ("training-side fake quantisation of activations: 4608 x 15360 bf16, group64", "fq_act",
                        4608, 15360, 64, "flux_out"),
    "fq_w_flux_qkv": ("training-side fake quantisation of the student's fp32 weights: 21504 x 3072, group64",
                      "fq_weight", 21504, 3072, 64, "flux_qkv"),
    "ste_dllm": ("straight-through backward: 1024 x 4096 bf16 gradients and their pass-through mask", "ste", 1024,
                 4096, 128, "dllm"),
    "ste_flux_out": ("straight-through backward: 4608 x 15360 bf16 gradients and their pass-through mask", "ste",
                     4608, 15360, 64, "flux_out"),
}
STREAM_METRIC = {"quantize": "activation quantiser GB/s", "fq_act": "fake-quant (activations) GB/s",
                 "fq_weight": "fake-quant (weights) GB/s", "ste": "STE backward GB/s"}


def stream_bytes(op: str, rows: int, K: int, G: int) -> float:
    """Algorithmic HBM bytes of one launch: every input read once, every output written once."""
    n = rows * K
    if op == "quantize":
        return 2 * n + n / 2 + 4 * n / G      # bf16 in; packed codes, scales out
    if op == "fq_act":
        return 2 * n + 2 * n + n + 4 * n / G  # bf16 in; bf16 x-hat, mask, scales out
    if op == "fq_weight":
        return 4 * n + 4 * n + n + 4 * n / G  # fp32 in; fp32 w-hat, mask, scales out
    if op == "ste":
        return 2 * n + n + 2 * n              # bf16 gradient and mask in; bf16 gradient out
    raise KeyError(op)


class StreamOracle:
    """The CPU oracle's version of a memory-bound kernel on a bounded row sample."""

    def __init__(self, name: str, seed: int = 7):
        import oracle
        from paper_2609_33601_gb300 import workloads as wl
        self.oracle = oracle
        self.desc, self.op, self.M, self.K, self.G, gen = STREAM_WORKLOADS[name]
        rows = min(self.M, 512)
        if self.op == "fq_weight":
            self.x = wl.make(gen, seed=seed, M=1, N=rows, K=self.K, G=self.G).w
        else:
            self.x = wl.make(gen, seed=seed, M=rows, K=self.K, G=self.G, with_weights=False).x_bits
        self.mask = (np.arange(self.x.size).reshape(self.x.shape) % 7 != 0).astype(np.uint8)
        self.rows = 8

    def run(self, rows: int) -> float:
        t0 = time.perf_counter()
        x = self.x[:rows]
        if self.op == "quantize":
            self.oracle.quantize_bf16(x, self.G)
        elif self.op == "fq_act":
            self.oracle.fake_quant_bf16(x, self.G)
        elif self.op == "fq_weight":
            self.oracle.fake_quant_f32(x, self.G)
        else:
            self.oracle.ste_backward_bf16(x, self.mask[:rows])
        return time.perf_counter() - t0

    def baseline(self, target_s: float) -> dict:
        rows = 8
        while True:
            dt = self.run(rows)
            if dt >= 0.8 * target_s or rows >= len(self.x):
                break
            rows = min(len(self.x), max(rows * 2, int(rows * target_s / max(dt, 1e-4))))
        reps = max(1, int(target_s / max(dt, 1e-4)))
        t = sum(self.run(rows) for _ in range(reps)) / reps
        return {"value": stream_bytes(self.op, rows, self.K, self.G) / t / 1e9, "unit": "GB/s",
                "cores": min(self.oracle.max_threads(), rows), "kind": "oracle", "host_threads": os.cpu_count(),
                "sample": f"{rows} of {self.M} rows, {reps} repetition(s) of {t:.3f} s"}


def run_stream(args):
    """Times one memory-bound kernel alone: a CUDA graph of K launches over rotating buffers that
    together exceed L2 several times over, so every launch reads and writes HBM."""
    import torch

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2609_33601_gb300 import build as jq_build
    jq_build.build()
    import paper_2609_33601_gb300 as jq
    from paper_2609_33601_gb300 import workloads as wl

    desc, op, M, K, G, gen = STREAM_WORKLOADS[args.workload]
    dev = torch.device("cuda", local)
    alg = stream_bytes(op, M, K, G)
    n_sets = max(3, -(-int(1.2e9) // int(alg)))
    if op == "fq_weight":
        base = torch.from_numpy(wl.make(gen, seed=100 + rank, M=1, N=M, K=K, G=G).w).to(dev)
    else:
        base = torch.from_numpy(wl.make(gen, seed=100 + rank, M=M, K=K, G=G, with_weights=False).x_bits
                                .view(np.int16)).to(dev).view(torch.bfloat16)
    mask0 = (torch.arange(M * K, device=dev).reshape(M, K) % 7 != 0).to(torch.uint8)
    sets = []
    for i in range(n_sets):
        # each set its own inputs and outputs (the row order rolled, so no two sets share lines)
        x = torch.roll(base, shifts=i * 37, dims=0).contiguous()
        if op == "quantize":
            outs = (torch.empty((M, K // 2), dtype=torch.uint8, device=dev),
                    torch.empty((M, K // G), dtype=torch.float32, device=dev))
        elif op == "ste":
            outs = (torch.roll(mask0, shifts=i, dims=0).contiguous(),)
        else:
            outs = ()
        sets.append((x, outs))
    torch.cuda.synchronize()

    def launch(i, st):
        x, outs = sets[i % n_sets]
        if op == "quantize":
            jq.jq_quantize_act(x, G, outs[0], outs[1], stream=st)
        elif op == "fq_act":
            jq.jq_fake_quant_act(x, G, stream=st)
        elif op == "fq_weight":
            jq.jq_fake_quant_weight(x, G, stream=st)
        else:
            jq.jq_ste_backward(x, outs[0], stream=st)

    stream = torch.cuda.current_stream()
    for i in range(args.warmup):
        launch(i, stream)
    torch.cuda.synchronize()
    # the fake-quant calls allocate their outputs: capture them in the graph's private pool
    cap = torch.cuda.Stream()
    cap.wait_stream(stream)
    with torch.cuda.stream(cap):
        for i in range(args.warmup):
            launch(i, cap)
    cap.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=cap):
        for i in range(args.steps):
            launch(i, cap)
    g.replay()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local, device_uuid(torch, dev)) as clocks:
        t0.record(stream)
        g.replay()
        t1.record(stream)
        torch.cuda.synchronize()
    (ms,) = max_over_ranks([t0.elapsed_time(t1)], dev)
    assert jq.jq_device_status() == 0, "a kernel reported a bounded-wait timeout"

    # end to end through the public API: host input copied in and the outputs copied out per step
    x_host = sets[0][0].cpu().pin_memory()
    x_dev = torch.empty_like(sets[0][0])
    host_outs = {}

    def e2e_step(i):
        x_dev.copy_(x_host, non_blocking=True)
        if op == "quantize":
            q, sa = jq.jq_quantize_act(x_dev, G)
            res = (q, sa)
        elif op == "fq_act":
            res = jq.jq_fake_quant_act(x_dev, G)
        elif op == "fq_weight":
            res = jq.jq_fake_quant_weight(x_dev, G)
        else:
            res = (jq.jq_ste_backward(x_dev, sets[0][1][0]),)
        for j, r in enumerate(res):
            if j not in host_outs:
                host_outs[j] = torch.empty(r.shape, dtype=r.dtype).pin_memory()
            host_outs[j].copy_(r, non_blocking=True)

    for i in range(args.warmup):
        e2e_step(i)
    torch.cuda.synchronize()
    e0 = time.perf_counter()
    for i in range(args.steps):
        e2e_step(i)
    torch.cuda.synchronize()
    (e2e_s,) = max_over_ranks([time.perf_counter() - e0], dev)
    h2d = sets[0][0].numel() * sets[0][0].element_size()
    d2h = sum(t.numel() * t.element_size() for t in host_outs.values())

    _, hbm_peak, peak_src = measured_peaks()
    gbs = world * alg * args.steps / (ms * 1e-3) / 1e9
    per_launch = alg / (ms / args.steps * 1e-3) / 1e9
    if rank != 0:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return 0
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        cpu = StreamOracle(args.workload).baseline(args.ref_seconds)
    line = {
        "metric": STREAM_METRIC[op], "value": gbs, "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16" if op != "fq_weight" else "f32", "data": "synthetic",
        "config": {"workload": desc, "rows": M, "K": K, "group": G, "launch": "CUDA graph of the K launches",
                   "parallelism": f"replicas x{world}",
                   "l2": f"{n_sets} rotating input/output sets, {n_sets * alg / 1e9:.2f} GB in all"},
        "roofline": {"bound": "hbm", "achieved": per_launch, "peak": hbm_peak, "unit": "GB/s",
                     "frac": per_launch / hbm_peak, "traffic": None, "algorithmic_bytes": alg,
                     "kernel": f"{op} kernel alone, CUDA events around a graph of K launches",
                     "peak_source": f"{peak_src} HBM copy bandwidth {hbm_peak} GB/s"},
        "cpu_baseline": cpu,
        "e2e": {"value": world * alg * args.steps / e2e_s / 1e9, "unit": "GB/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "copies": "pinned host buffers, on the compute stream around the kernel"},
        "gpu_launches": args.steps,
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


# ----------------------------------------------------------------------------- our arm

def run_ours(args):
    import torch

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    from paper_2609_33601_gb300 import build as jq_build
    jq_build.build()
    import paper_2609_33601_gb300 as jq
    from paper_2609_33601_gb300 import workloads as wl

    desc, M, K, N, G, gen = WORKLOADS[args.workload]
    nv = args.weights == "nvfp4"
    few = M <= FEW_TOKENS and not nv  # NVFP4 has no few-token kernel: every M takes its GEMM
    dev = torch.device("cuda", local)
    sets = []
    # rotating weight sets: together several times larger than the 126 MB L2
    n_sets = args.sets if args.sets > 0 else max(6, -(-400_000_000 // (N * K // 2 + M * K * 2)))
    for i in range(n_sets):
        w = wl.make(gen, seed=100 + 17 * rank + i, M=M, K=K, N=N, G=G)
        x = torch.from_numpy(w.x_bits.view(np.int16)).to(dev).view(torch.bfloat16)
        if nv:  # codes, (block-scale bytes, device tensor scale)
            codes_w, scales_w, g_w = jq.jq_nvfp4_pack_weight(torch.from_numpy(w.w).to(dev))
            qw, sw = codes_w, (scales_w, g_w)
            if i == 0:  # the activations' tensor scale, calibrated once on the first input set
                ga = float(np.float32(np.abs(wl.bf16_bits_to_f32(w.x_bits)).max()) / np.float32(2688.0))
        else:
            pack = jq.jq_pack_weight_ternary if args.weights == "ternary" else jq.jq_pack_weight
            qw, sw = pack(torch.from_numpy(w.w).to(dev), G)
        b = None if w.bias is None else torch.from_numpy(w.bias).to(dev)
        sets.append((x, qw, sw, b))
        del w
    torch.cuda.synchronize()
    q = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
    s_a = torch.empty((M, K // G), dtype=torch.float32, device=dev)
    y = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
    fused = args.fused
    ternary = args.weights == "ternary"
    need = (jq.jq_nvfp4_workspace_size(M, N, K) if nv else
            jq.jq_w158a4_workspace_size(M, N, K, G) if ternary else jq.jq_workspace_size(M, N, K, G, fused))
    ws = torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
    linear_call = jq.jq_w158a4_linear if ternary else jq.jq_w4a4_linear
    if nv:
        codes_a = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
        scales_a = torch.empty((M, K // 16), dtype=torch.uint8, device=dev)

        def linear_call(q_, s_, qw_, sw_, b_, g_, y=None, workspace=None, stream=None):
            return jq.jq_nvfp4_linear(codes_a, scales_a, ga, qw_, sw_[0], sw_[1], b_, y=y, workspace=workspace,
                                      stream=stream)
    stream = torch.cuda.current_stream()

    prologue = DIT_PROLOGUE.get(args.workload)
    T = wl.DIT_TOKENS_PER_IMAGE
    if prologue == "modulate":
        mods = [tuple(torch.from_numpy(a).to(dev) for a in wl.dit_modulation(300 + 31 * rank + i, -(-M // T), K))
                for i in range(n_sets)]

    def quantize(i, st):
        x = sets[i % n_sets][0]
        if nv:
            jq.jq_nvfp4_quantize_act(x, ga, codes_a, scales_a, stream=st)
        elif prologue == "modulate":
            sh, sc = mods[i % n_sets]
            jq.jq_modulate_quantize_act(x, sh, sc, T, G, q, s_a, stream=st)
        elif prologue == "gelu":
            jq.jq_gelu_quantize_act(x, G, q, s_a, stream=st)
        else:
            jq.jq_quantize_act(x, G, q, s_a, stream=st)

    def linear(i, st):
        x, qw, sw, b = sets[i % n_sets]
        if fused:  # bf16 activations straight into the GEMM operand
            jq.jq_fused_quant_linear(x, qw, sw, b, G, y=y, workspace=ws, stream=st)
        else:
            linear_call(q, s_a, qw, sw, b, G, y=y, workspace=ws, stream=st)

    def step(i, st=None):
        if not fused:
            quantize(i, st or stream)
        linear(i, st or stream)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    assert jq.jq_device_status() == 0, "a kernel reported a bounded-wait timeout"

    # The K timed steps are captured once into a CUDA graph and replayed: the host's per-call cost
    # (Python, ctypes, argument checks, launch) would otherwise gate the device on the short
    # launches of the few-token workloads.  A second graph holds the K linear launches alone, for
    # the per-launch duration of the dominant kernel.
    cap = torch.cuda.Stream()
    cap.wait_stream(stream)
    with torch.cuda.stream(cap):
        for i in range(args.warmup):
            step(i, cap)
    cap.synchronize()
    g_steps, g_linear = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(g_steps, stream=cap):
        for i in range(args.steps):
            step(i, cap)
    with torch.cuda.graph(g_linear, stream=cap):
        for i in range(args.steps):
            linear(i, cap)
    g_steps.replay()
    g_linear.replay()
    torch.cuda.synchronize()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    l_start, l_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    torch.cuda.synchronize()
    with ClockSampler(local, device_uuid(torch, dev)) as clocks:
        t_start.record(stream)
        g_steps.replay()
        t_end.record(stream)
        torch.cuda.synchronize()
        l_start.record(stream)
        g_linear.replay()
        l_end.record(stream)
        torch.cuda.synchronize()
    barrier()
    total_ms = t_start.elapsed_time(t_end)
    gemm_ms = l_start.elapsed_time(l_end) / args.steps
    total_ms, gemm_ms = max_over_ranks([total_ms, gemm_ms], dev)
    assert jq.jq_device_status() == 0, "a kernel reported a bounded-wait timeout"

    # End to end through the public API: every step copies its activations in from pinned host
    # memory and its result out to pinned host memory, inside the timed region.  As in a serving
    # loop, when a step moves at least 1 MB the copies run on their own streams and overlap the
    # neighbouring steps' kernels (two device buffers each for x and y, ordered by events); for
    # smaller steps the host's per-step cost of that bookkeeping outweighs the copies, and the
    # copies simply precede and follow the kernels on the compute stream.
    pipelined = M * K * 2 + M * N * 2 >= 1 << 20
    nb = 2
    x_host = [sets[i][0].cpu().pin_memory() for i in range(min(2, n_sets))]
    y_host = [torch.empty((M, N), dtype=torch.bfloat16).pin_memory() for _ in range(nb)]
    x_dev = [torch.empty((M, K), dtype=torch.bfloat16, device=dev) for _ in range(nb)]
    y_dev = [torch.empty((M, N), dtype=torch.bfloat16, device=dev) for _ in range(nb)]
    h2d, d2h = torch.cuda.Stream(), torch.cuda.Stream()
    x_free = [None] * nb  # the kernels that read x_dev[k] are done
    y_free = [None] * nb  # the copy out of y_dev[k] is done

    def quantize_x(x, i, st):
        if nv:
            jq.jq_nvfp4_quantize_act(x, ga, codes_a, scales_a, stream=st)
        elif prologue == "modulate":
            sh, sc = mods[i % n_sets]
            jq.jq_modulate_quantize_act(x, sh, sc, T, G, q, s_a, stream=st)
        elif prologue == "gelu":
            jq.jq_gelu_quantize_act(x, G, q, s_a, stream=st)
        else:
            jq.jq_quantize_act(x, G, q, s_a, stream=st)

    def e2e_step(i):
        k = i % nb
        if not pipelined:
            x_dev[0].copy_(x_host[i % len(x_host)], non_blocking=True)
            _, qw, sw, b = sets[i % n_sets]
            if fused:
                jq.jq_fused_quant_linear(x_dev[0], qw, sw, b, G, y=y_dev[0], workspace=ws, stream=stream)
            else:
                quantize_x(x_dev[0], i, stream)
                linear_call(q, s_a, qw, sw, b, G, y=y_dev[0], workspace=ws, stream=stream)
            y_host[0].copy_(y_dev[0], non_blocking=True)
            return
        with torch.cuda.stream(h2d):
            if x_free[k] is not None:
                h2d.wait_event(x_free[k])
            x_dev[k].copy_(x_host[i % len(x_host)], non_blocking=True)
            x_in = torch.cuda.Event()
            x_in.record(h2d)
        stream.wait_event(x_in)
        if y_free[k] is not None:
            stream.wait_event(y_free[k])
        _, qw, sw, b = sets[i % n_sets]
        if fused:
            jq.jq_fused_quant_linear(x_dev[k], qw, sw, b, G, y=y_dev[k], workspace=ws, stream=stream)
        else:
            quantize_x(x_dev[k], i, stream)
            linear_call(q, s_a, qw, sw, b, G, y=y_dev[k], workspace=ws, stream=stream)
        done = torch.cuda.Event()
        done.record(stream)
        x_free[k] = done
        with torch.cuda.stream(d2h):
            d2h.wait_event(done)
            y_host[k].copy_(y_dev[k], non_blocking=True)
            out = torch.cuda.Event()
            out.record(d2h)
        y_free[k] = out

    for i in range(args.warmup):
        e2e_step(i)
    torch.cuda.synchronize()
    barrier()
    e0 = time.perf_counter()
    for i in range(args.steps):
        e2e_step(i)
    torch.cuda.synchronize()
    e2e_s = time.perf_counter() - e0
    (e2e_s,) = max_over_ranks([e2e_s], dev)

    ops_step = 2.0 * M * N * K
    value = whole_job_tops(world, ops_step, args.steps, total_ms * 1e-3)
    e2e_value = whole_job_tops(world, ops_step, args.steps, e2e_s)
    bf16_peak, hbm_peak, peak_src = measured_peaks()
    fp8_peak = bf16_peak * FP8_PER_BF16
    kernel_file = "skinny.cu" if few else "gemm.cu"
    traffic = None if (fused or nv) else recorded_traffic(args.workload + ("/ternary" if ternary else ""),
                                                          kernel_file)
    # algorithmic bytes of one linear call: packed weights and their scales, packed activation
    # codes and scales (the fused call reads bf16 activations instead), bias, bf16 output
    groups = K // G
    act_bytes = M * K * 2 if fused else M * K // 2 + M * groups * 4
    wbytes = N * K // 4 if ternary else N * K // 2  # 2-bit ternary or 4-bit INT4 weight codes
    alg_bytes = wbytes + groups * N * 4 + act_bytes + (0 if sets[0][3] is None else N * 4) + M * N * 2
    tensor_peak, tensor_src = fp8_peak, f"{peak_src} bf16 {bf16_peak} TFLOP/s x nominal FP8/BF16 ratio {FP8_PER_BF16}"
    if nv:  # E2M1 codes and E4M3 block-scale bytes of both operands; the layer's MMA is bf16
        alg_bytes = (M + N) * (K // 2 + K // 16) + (0 if sets[0][3] is None else N * 4) + M * N * 2
        tensor_peak, tensor_src = bf16_peak, f"{peak_src} bf16 {bf16_peak} TFLOP/s (the layer's MMA is bf16)"
    # the bound is whichever of the tensor time and the HBM time is larger
    t_tensor, t_hbm = ops_step / (tensor_peak * 1e12), alg_bytes / (hbm_peak * 1e9)
    what = ("jq_nvfp4_linear (bf16 operand images of the exact block-scaled values + tcgen05 kind::f16 GEMM)"
            if nv else
            "jq_w158a4_linear (few-token kernel, 2-bit weights)" if ternary and few else
            "jq_w158a4_linear (operand expansion + tcgen05 GEMM reading the 2-bit codes)" if ternary else
            "jq_fused_quant_linear (quantise-to-operand + tcgen05 GEMM)" if fused else
            "jq_w4a4_linear (few-token weight-streaming kernel)" if few else
            "jq_w4a4_linear (operand expansion + tcgen05 GEMM)")
    if t_hbm > t_tensor:
        achieved = alg_bytes / (gemm_ms * 1e-3) / 1e9
        roofline = {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s", "frac": achieved / hbm_peak,
                    "traffic": traffic, "algorithmic_bytes": alg_bytes,
                    "kernel": what + ", CUDA events around a graph of K launches",
                    "peak_source": f"{peak_src} HBM copy bandwidth {hbm_peak} GB/s"}
    else:
        achieved = ops_step / (gemm_ms * 1e-3) / 1e12
        roofline = {"bound": "tensor", "achieved": achieved, "peak": tensor_peak, "unit": "TFLOP/s",
                    "frac": achieved / tensor_peak, "frac_of_bf16_peak": achieved / bf16_peak,
                    "traffic": traffic, "algorithmic_bytes": alg_bytes,
                    "kernel": what + ", CUDA events around a graph of K launches",
                    "peak_source": tensor_src}
    context = None
    if not args.no_context:
        context = {"cublas_bf16": cublas_context(torch, dev, sets, M, N, K, args, world)}
        if few:
            context["copy_same_bytes"] = copy_context(torch, dev, alg_bytes, args, world)
        if prologue is not None:
            context["prologue"] = prologue_context(torch, jq, sets, mods if prologue == "modulate" else None, prologue,
                                                   G, T, q, s_a, args)

    if rank != 0:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return 0
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        o = OracleSample(args.workload, fmt=args.weights)
        o.calibrate(args.ref_seconds)
        cpu = o.describe(o.run(o.rows), single_s=args.ref_single_seconds)
    line = {
        "metric": metric_name(args), "value": value, "unit": "TOPS", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "nvfp4" if nv else "int4", "data": "synthetic",
        "config": {"workload": desc, "M": M, "K": K, "N": N, "group": G,
                   "step": ("jq_nvfp4_quantize_act + jq_nvfp4_linear" if nv else
                            "jq_fused_quant_linear" if fused else
                            "jq_quantize_act + jq_w158a4_linear" if ternary else
                            "jq_modulate_quantize_act + jq_w4a4_linear" if prologue == "modulate" else
                            "jq_gelu_quantize_act + jq_w4a4_linear" if prologue == "gelu" else
                            "jq_quantize_act + jq_w4a4_linear"),
                   "weights": ("NVFP4 (E2M1, E4M3 scale per 16, fp32 tensor scale)" if nv else
                               "ternary (2-bit)" if ternary else "INT4"),
                   "launch": "CUDA graph of the K steps",
                   "parallelism": f"replicas x{world}",
                   "l2": f"{n_sets} rotating input/weight sets larger than L2"},
        "roofline": roofline,
        "context": context,
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": "TOPS", "h2d_bytes_per_step": M * K * 2, "d2h_bytes_per_step": M * N * 2,
                "copies": ("pinned host buffers, on two copy streams overlapping the neighbouring steps' kernels"
                           if pipelined else "pinned host buffers, on the compute stream around the kernels")},
        "gpu_launches": launches_per_step(M, fused, nv) * args.steps,
        "clocks": clocks.summary(),
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS) + sorted(STREAM_WORKLOADS), default="flux_qkv")
    ap.add_argument("--sets", type=int, default=0, help="rotating input/weight sets (0: enough for > 3x L2)")
    ap.add_argument("--ref-seconds", type=float, default=10.0, help="CPU seconds per oracle sample")
    ap.add_argument("--ref-single-seconds", type=float, default=5.0,
                    help="CPU seconds for the oracle's single-thread sample (0: skip it)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--fused", action="store_true", help="time jq_fused_quant_linear (bf16 activations in)")
    ap.add_argument("--weights", choices=["int4", "ternary", "nvfp4"], default="int4",
                    help="ternary: the W1.58A4 layer (jq_pack_weight_ternary + jq_w158a4_linear); nvfp4: the "
                         "NVFP4 W4A4 layer (jq_nvfp4_pack_weight + jq_nvfp4_quantize_act + jq_nvfp4_linear)")
    ap.add_argument("--no-context", action="store_true", help="skip the cuBLAS bf16 GEMM of the same shape")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.fused and args.weights != "int4":
        ap.error("--fused is an INT4-weight call")
    if args.weights == "nvfp4" and (args.workload in DIT_PROLOGUE or args.workload in STREAM_WORKLOADS):
        ap.error("--weights nvfp4 runs the plain linear layer workloads")
    if args.workload in STREAM_WORKLOADS:
        if args.impl == "reference":
            return run_stream_reference(args)
        return run_stream(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
