"""Seeded synthetic inputs shaped like the paper's W4A4 linears.

This module only *generates data*: it holds none of the quantiser / GEMM
arithmetic, and both the CPU oracle and the CUDA path consume exactly the
bytes it returns.  The paper's own workloads (FLUX.1 on MJHQ prompts, LLaDA /
ELF on GSM8K / OpenWebText) are not available, so these tensors stand in for
them with the layer shapes of a FLUX-12B-style DiT (hidden 3072, fused
QKV+MLP-in 3072 -> 21504, output 15360 -> 3072) and an 8B LLaMA-style dLLM
(hidden 4096, MLP 12288), which are the model families the paper quantises
(Sec. 4.1 experimental summary table: FLUX.1 12B, LLaDA 8B).

Group sizes follow the paper: group64 for FLUX transformer-block linears
(Sec. 4.2 "FLUX"; Appendix "FLUX experimental details"), group128 for the
dLLM family (Appendix "ELF-B and LLaDA-8B experimental details").

Recipe (all draws from numpy PCG64 ``default_rng(seed)``; activations are
drawn in fp64/fp32 and rounded once to bf16, round-to-nearest-even):

* ``tiny``  : X ~ N(0,1) [64, 256], 4 seeded outlier channels x20;
              W ~ N(0, 0.02) fp32 [256, 256]; bias ~ N(0, 0.01).
* ``dllm``  : X ~ N(0,1) [1024, 4096]; 1% of channels (41) replaced by
              Student-t(nu=3) x10; W ~ N(0, 0.02) [12288, 4096]; no bias.
* ``flux_qkv``: X ~ N(0,1) * c_k with c_k log-uniform in [0.1, 30] per
              channel, [4608, 3072]; W ~ N(0, 0.02) [21504, 3072];
              bias ~ N(0, 0.01).
* ``flux_out``: X [4608, 15360]: channels [0, 3072) ~ N(0,1) (attention
              output), channels [3072, 15360) = GELU(N(0,1)) with the exact
              erf GELU in fp64 (MLP hidden); W ~ N(0, 0.02) [3072, 15360];
              bias ~ N(0, 0.01).
* ``sweep_a`` / ``sweep_b``: M tokens x (K=4096 -> N=12288) or
              (K=3072 -> N=3072); X ~ N(0,1) with 1% of channels x20;
              W ~ N(0, 0.02); no bias.
* ``dit``   : DiT-XL/2 block linears (hidden 1152, MLP 4608, 256 tokens per
              256x256 image: 16 images = 4096 tokens), group128 (Appendix
              "DiT-XL/2 experimental details").  X ~ N(0,1) (layer-normalised
              tokens, or the MLP's pre-activation for the GELU); the adaLN
              modulation's shift and scale per image ~ N(0, 0.5^2)
              (``dit_modulation``); W ~ N(0, 0.02); bias ~ N(0, 0.01).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

WORKLOADS = {
    # name: (M, K, N, G, has_bias)
    "tiny": (64, 256, 256, 64, True),
    "dllm": (1024, 4096, 12288, 128, False),
    "flux_qkv": (4608, 3072, 21504, 64, True),
    "flux_out": (4608, 15360, 3072, 64, True),
    "sweep_a": (None, 4096, 12288, 128, False),
    "sweep_b": (None, 3072, 3072, 64, False),
    "dit": (4096, 1152, 3456, 128, True),
}
DIT_TOKENS_PER_IMAGE = 256  # 256x256 images, 32x32 latent, patch 2
SWEEP_M = (1, 16, 64, 256, 1024, 4096, 16384)


@dataclasses.dataclass
class Workload:
    name: str
    M: int
    K: int
    N: int
    G: int
    x_bits: np.ndarray      # uint16 [M, K]: bf16 bit patterns of the activations
    w: np.ndarray           # float32 [N, K]: full-precision weights
    bias: np.ndarray | None  # float32 [N] or None

    @property
    def ops(self) -> float:
        return 2.0 * self.M * self.N * self.K


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (nearest, ties to even) and return the bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _gelu_exact(x64: np.ndarray) -> np.ndarray:
    try:
        from scipy.special import erf
        return 0.5 * x64 * (1.0 + erf(x64 / math.sqrt(2.0)))
    except ImportError:  # pragma: no cover - scipy is present on both machines
        v = np.vectorize(math.erf)
        return 0.5 * x64 * (1.0 + v(x64 / math.sqrt(2.0)))


def _activations(name: str, rng: np.random.Generator, M: int, K: int) -> np.ndarray:
    if name == "tiny":
        x = rng.standard_normal((M, K), dtype=np.float32)
        ch = rng.choice(K, size=4, replace=False)
        x[:, ch] *= 20.0
    elif name == "dllm":
        x = rng.standard_normal((M, K), dtype=np.float32)
        n_out = max(1, int(round(0.01 * K)))
        ch = rng.choice(K, size=n_out, replace=False)
        x[:, ch] = (rng.standard_t(3.0, size=(M, n_out)) * 10.0).astype(np.float32)
    elif name == "flux_qkv":
        c = np.exp(rng.uniform(math.log(0.1), math.log(30.0), size=K)).astype(np.float32)
        x = rng.standard_normal((M, K), dtype=np.float32) * c[None, :]
    elif name == "flux_out":
        attn = 3072
        x = np.empty((M, K), np.float32)
        x[:, :attn] = rng.standard_normal((M, attn), dtype=np.float32)
        h = rng.standard_normal((M, K - attn))
        x[:, attn:] = _gelu_exact(h).astype(np.float32)
    elif name == "dit":
        x = rng.standard_normal((M, K), dtype=np.float32)
    elif name in ("sweep_a", "sweep_b", "custom"):
        x = rng.standard_normal((M, K), dtype=np.float32)
        n_out = max(1, int(round(0.01 * K)))
        ch = rng.choice(K, size=n_out, replace=False)
        x[:, ch] *= 20.0
    else:
        raise KeyError(name)
    return f32_to_bf16_bits(x)


def make(name: str, seed: int = 0, M: int | None = None, K: int | None = None,
         N: int | None = None, G: int | None = None, bias: bool | None = None,
         with_weights: bool = True) -> Workload:
    """Build one seeded workload.  Shapes default to the named config; any of
    M, K, N, G may be overridden (e.g. a smaller M for a bounded sample)."""
    if name == "custom":
        dM, dK, dN, dG, db = (M, K, N, G, bool(bias))
    else:
        dM, dK, dN, dG, db = WORKLOADS[name]
    M = dM if M is None else M
    K = dK if K is None else K
    N = dN if N is None else N
    G = dG if G is None else G
    db = db if bias is None else bias
    if M is None:
        raise ValueError(f"workload {name} needs an explicit M (one of {SWEEP_M})")
    rng = np.random.default_rng(seed)
    x_bits = _activations(name, rng, M, K)
    if with_weights:
        w = (rng.standard_normal((N, K), dtype=np.float32) * np.float32(0.02)).astype(np.float32)
        b = (rng.standard_normal(N, dtype=np.float32) * np.float32(0.01)).astype(np.float32) if db else None
    else:
        w = np.zeros((0, K), np.float32)
        b = None
    return Workload(name, M, K, N, G, x_bits, w, b)


def random_codes(rng: np.random.Generator, rows: int, K: int, low: int = -8, high: int = 7) -> np.ndarray:
    """Uniform random INT4 codes in [low, high], as int8 [rows, K] (for GEMM
    tests that feed the full code range, including -8, straight to the GEMM)."""
    return rng.integers(low, high + 1, size=(rows, K), dtype=np.int8)


def dit_modulation(seed: int, samples: int, K: int):
    """The adaLN modulation's per-image shift and scale, fp32 [samples, K] each, ~ N(0, 0.5^2)."""
    rng = np.random.default_rng(seed)
    shift = (rng.standard_normal((samples, K)) * 0.5).astype(np.float32)
    scale = (rng.standard_normal((samples, K)) * 0.5).astype(np.float32)
    return shift, scale
