"""GPU parity of the NVFP4 W4A4 path (the LLaDA-8B format) through the C ABI.

Bit-exact: the E2M1 codes (packed bytes), the E4M3 block scales (decoded from their bytes by a
decoder written here from the format) and the weights' tensor scale, against the oracle.  bf16
outputs: against the oracle's fp64 evaluation, within one bf16 ulp plus the fp32 summation bound
over the K products the layer sums (every product is exact: each operand value q * s_b is exact
in bf16), (K + 2) * 2^-24 * (sum_k |term| + |bias|).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl
from tests.helpers import report_escape, ulp_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _device():
    assert torch.cuda.is_available(), "the gpu tests need a CUDA device"
    jq._load()
    yield
    assert jq.jq_device_status() == 0


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def e4m3_decode(b: np.ndarray) -> np.ndarray:
    """E4M3 bytes (no sign, finite) -> float64: exponent bits 3-6 (bias 7), 3 mantissa bits;
    exponent 0 is subnormal, m * 2^-9."""
    b = b.astype(np.int64)
    e, m = (b >> 3) & 15, b & 7
    return np.where(e == 0, m * 2.0 ** -9, (8 + m) * np.exp2((e - 10).astype(np.float64)))


def special_activations(M, K, rng):
    """N(0,1) bf16 rows and rows that stress the rule: zeros, a block with one nonzero, values
    whose quotient lands on E2M1 midpoints, tiny values whose block scale underflows, huge ones."""
    x = rng.standard_normal((M, K)).astype(np.float32)
    if M > 6:
        x[0] = 0.0
        x[1, :] = 0.0
        x[1, 5] = 3.0
        x[2] = np.tile(np.array([6, 5, 3.5, 2.5, 1.75, 1.25, 0.75, 0.25], np.float32), K // 8)  # midpoints x 1
        x[3] *= np.float32(1e-30)
        x[4] *= np.float32(1e4)
        x[5, : K // 2] = -x[5, K // 2:]
    return wl.f32_to_bf16_bits(x)


@pytest.mark.parametrize("M,K", [(1, 64), (7, 128), (130, 192), (64, 4096), (257, 1024)])
@pytest.mark.parametrize("g_rule", ["amax", "fixed", "zero"])
def test_nvfp4_quantize_act_bit_exact(M, K, g_rule):
    rng = np.random.default_rng(M * 7 + K)
    xb = special_activations(M, K, rng)
    xf = wl.bf16_bits_to_f32(xb)
    g = {"amax": oracle.nvfp4_tensor_scale(xf), "fixed": 0.0123, "zero": 0.0}[g_rule]
    codes2, s_ref = oracle.quantize_nvfp4(xf, g)
    codes, scales = jq.jq_nvfp4_quantize_act(dev(xb).view(torch.bfloat16), g)
    torch.cuda.synchronize()
    assert np.array_equal(codes.cpu().numpy(), oracle.pack_nvfp4(codes2)), "codes differ from the oracle"
    assert np.array_equal(e4m3_decode(scales.cpu().numpy()), s_ref.astype(np.float64)), "block scales differ"


def test_nvfp4_quantize_act_padded_rows():
    rng = np.random.default_rng(11)
    M, K, ld = 33, 256, 320
    full = wl.f32_to_bf16_bits(rng.standard_normal((M, ld)).astype(np.float32))
    g = 0.004
    codes2, s_ref = oracle.quantize_nvfp4(wl.bf16_bits_to_f32(full[:, :K]), g)
    x = dev(full).view(torch.bfloat16)[:, :K]
    codes, scales = jq.jq_nvfp4_quantize_act(x, g)
    torch.cuda.synchronize()
    assert np.array_equal(codes.cpu().numpy(), oracle.pack_nvfp4(codes2))
    assert np.array_equal(e4m3_decode(scales.cpu().numpy()), s_ref.astype(np.float64))


@pytest.mark.parametrize("N,K", [(8, 64), (264, 192), (520, 1024), (96, 4096)])
def test_nvfp4_pack_weight_bit_exact(N, K):
    rng = np.random.default_rng(N + K)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    w[0] = 0.0
    w[1, 3] = 0.7  # the tensor maximum: its block gets the largest scale, its code +-6
    if N > 4:
        w[2] *= np.float32(1e-20)
        w[3, :16] = np.float32(1e-42)  # fp32 subnormals
    g_ref = oracle.nvfp4_tensor_scale(w)
    codes2, s_ref = oracle.quantize_nvfp4(w, g_ref)
    codes, scales, g_w = jq.jq_nvfp4_pack_weight(dev(w))
    torch.cuda.synchronize()
    assert np.float32(g_w.cpu().numpy()[0]) == np.float32(g_ref), "tensor scale differs from the oracle"
    assert np.array_equal(codes.cpu().numpy(), oracle.pack_nvfp4(codes2)), "codes differ from the oracle"
    assert np.array_equal(e4m3_decode(scales.cpu().numpy()), s_ref.astype(np.float64)), "block scales differ"


def nvfp4_tolerance(y64, qa2, sa, ga, qw2, sw, gw, bias):
    """ulp_bf16(y64) + (K + 2) * 2^-24 * (sum_k |qa sa_b qw sw_b| ga gw + |bias|)."""
    K = qa2.shape[1]
    a = np.abs(qa2.astype(np.float64)) / 2 * np.repeat(sa.astype(np.float64), 16, axis=1)
    w = np.abs(qw2.astype(np.float64)) / 2 * np.repeat(sw.astype(np.float64), 16, axis=1)
    mag = (a @ w.T) * float(ga) * float(gw)
    if bias is not None:
        mag = mag + np.abs(bias.astype(np.float64))[None, :]
    return ulp_bf16(y64) + (K + 2) * 2.0 ** -24 * mag


def run_linear(M, N, K, with_bias, seed, label):
    rng = np.random.default_rng(seed)
    xb = special_activations(M, K, rng)
    xf = wl.bf16_bits_to_f32(xb)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    bias = (rng.standard_normal(N) * 0.01).astype(np.float32) if with_bias else None
    ga = oracle.nvfp4_tensor_scale(xf)
    qa2, sa = oracle.quantize_nvfp4(xf, ga)
    gw = oracle.nvfp4_tensor_scale(w)
    qw2, sw = oracle.quantize_nvfp4(w, gw)
    y64, _ = oracle.linear_nvfp4(qa2, sa, ga, qw2, sw, gw, bias)
    codes_a, scales_a = jq.jq_nvfp4_quantize_act(dev(xb).view(torch.bfloat16), ga)
    codes_w, scales_w, g_w = jq.jq_nvfp4_pack_weight(dev(w))
    y = jq.jq_nvfp4_linear(codes_a, scales_a, ga, codes_w, scales_w, g_w, None if bias is None else dev(bias))
    torch.cuda.synchronize()
    yg = wl.bf16_bits_to_f32(y.view(torch.int16).cpu().numpy().view(np.uint16)).astype(np.float64)
    err = np.abs(yg - y64)
    tol = nvfp4_tolerance(y64, qa2, sa, ga, qw2, sw, gw, bias)
    bad = err > tol
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{label}: {bad.sum()} elements out of tolerance, e.g. "
                             + "; ".join(f"[{m},{n}] gpu={yg[m, n]!r} ref={y64[m, n]!r} tol={tol[m, n]:.3g}"
                                         for m, n in idx))
    ulp = ulp_bf16(y64)
    report_escape(label, int((err > ulp).sum()), err.size, float((err / ulp).max()), enforce=False)


@pytest.mark.parametrize("M,N,K,with_bias", [(1, 256, 64, True), (130, 264, 192, False), (256, 512, 4096, True),
                                             (300, 1032, 1024, True), (64, 8, 128, False)])
def test_nvfp4_linear_matches_oracle(M, N, K, with_bias):
    run_linear(M, N, K, with_bias, M + N + K, f"nvfp4 {M}x{K}->{N}")


def test_nvfp4_linear_zero_activation_scale_gives_the_bias():
    rng = np.random.default_rng(5)
    M, N, K = 40, 264, 256
    xb = wl.f32_to_bf16_bits(rng.standard_normal((M, K)).astype(np.float32))
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    bias = (rng.standard_normal(N) * 0.01).astype(np.float32)
    codes_a, scales_a = jq.jq_nvfp4_quantize_act(dev(xb).view(torch.bfloat16), 0.0)
    codes_w, scales_w, g_w = jq.jq_nvfp4_pack_weight(dev(w))
    y = jq.jq_nvfp4_linear(codes_a, scales_a, 0.0, codes_w, scales_w, g_w, dev(bias))
    torch.cuda.synchronize()
    want = np.broadcast_to(wl.f32_to_bf16_bits(bias), (M, N))
    assert np.array_equal(y.view(torch.int16).cpu().numpy().view(np.uint16), want)


def test_nvfp4_linear_dllm_shape_all_rows():
    """The dLLM gate/up shape, 1024 x 4096 -> 12288, every output element."""
    run_linear(1024, 12288, 4096, False, 7, "nvfp4 dllm 1024x4096->12288")
