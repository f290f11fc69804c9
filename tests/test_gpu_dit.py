"""GPU parity of the DiT neighbour operations fused with the activation quantiser (C ABI).

jq_modulate_quantize_act (adaLN modulation) and jq_gelu_quantize_act (tanh GELU) must give the
oracle's codes and scales bit for bit: the modulation is exact IEEE arithmetic on both sides; the
GELU is the oracle's fp32 sequence rounded to bf16, which the kernel looks up in a table of all
65536 bf16 inputs filled on the device by its own evaluation of that sequence (checked here for
every finite input; tests/test_oracle_dit_pins.py pins the oracle's side to a high-precision
reference).  Shapes follow DiT-XL/2 (hidden 1152, MLP 4608, 256 tokens per
256x256 image, group128); ragged token counts, strided rows, group64 and one group are covered.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl
from tests.helpers import check_linear_full

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _device():
    assert torch.cuda.is_available(), "the gpu tests need a CUDA device"
    jq._load()
    yield
    assert jq.jq_device_status() == 0


def dev_bf16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def modulation_inputs(M, K, T, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((M, K)).astype(np.float32)
    x[0] = 0.0
    if M > 2:
        x[1, ::3] = 1e-39      # bf16 subnormals
        x[2] *= np.float32(1e30)
    samples = -(-M // T)
    shift = (rng.standard_normal((samples, K)) * 0.5).astype(np.float32)
    scale = (rng.standard_normal((samples, K)) * 0.5).astype(np.float32)
    scale[0, :32] = -1.0       # z = shift
    shift[0, 32:64] = 0.0
    scale[0, 32:64] = 0.0      # z = x
    scale[-1, :16] = 1e30      # huge products
    return wl.f32_to_bf16_bits(x), shift, scale


@pytest.mark.parametrize("M,K,T,G", [(256 * 3 + 17, 1152, 256, 128), (300, 4608, 256, 128), (64, 1152, 16, 64),
                                     (40, 1152, 7, 1152), (1, 256, 1, 128)])
def test_modulate_quantize_bit_exact(M, K, T, G):
    x, shift, scale = modulation_inputs(M, K, T, seed=M + K)
    _, codes, s = oracle.modulate_quantize_bf16(x, shift, scale, T, G)
    q, sa = jq.jq_modulate_quantize_act(dev_bf16(x), dev(shift), dev(scale), T, G)
    assert np.array_equal(q.cpu().numpy(), oracle.pack(codes))
    assert np.array_equal(sa.cpu().numpy().view(np.uint32), s.view(np.uint32))


def test_modulate_quantize_strided_rows():
    M, K, T, G = 130, 1152, 64, 128
    x, shift, scale = modulation_inputs(M, K, T, seed=5)
    xp = np.zeros((M, K + 64), np.uint16)
    xp[:, :K] = x
    _, codes, s = oracle.modulate_quantize_bf16(x, shift, scale, T, G)
    q, sa = jq.jq_modulate_quantize_act(dev_bf16(xp)[:, :K], dev(shift), dev(scale), T, G)
    assert np.array_equal(q.cpu().numpy(), oracle.pack(codes))
    assert np.array_equal(sa.cpu().numpy(), s)


def gelu_inputs():
    pos = np.arange(0, 0x7F80, dtype=np.uint16)
    vals = wl.bf16_bits_to_f32(pos)
    keep = pos[vals <= 16.0]
    sweep = np.concatenate([keep, keep | np.uint16(0x8000)])          # every bf16 in [-16, 16], +-0
    extra = wl.f32_to_bf16_bits(np.array([-8.0, -8.0625, -9.0, -10.0, -12.0, -20.0, -52.0, -100.0, -3e38, 20.0, 50.0,
                                          1e6, 3e38, 1e-38, -1e-38, 1e-30], np.float32))
    rng = np.random.default_rng(3)
    rand = wl.f32_to_bf16_bits((rng.standard_normal(4096 * 8) * 3).astype(np.float32))
    h = np.concatenate([sweep, extra, rand])
    return np.resize(h, (-(-len(h) // 1152)) * 1152).reshape(-1, 1152)


@pytest.mark.parametrize("G", [128, 64, 1152])
def test_gelu_quantize_bit_exact(G):
    h = gelu_inputs()
    z, codes, s = oracle.gelu_quantize_bf16(h, G)
    q, sa = jq.jq_gelu_quantize_act(dev_bf16(h), G)
    got = q.cpu().numpy()
    want = oracle.pack(codes)
    if not np.array_equal(got, want):
        rows = np.unique(np.argwhere(got != want)[:, 0])[:3]
        raise AssertionError(f"codes differ in rows {rows}; first inputs there: {h[rows[0], :8]}")
    assert np.array_equal(sa.cpu().numpy().view(np.uint32), s.view(np.uint32))


def test_gelu_every_finite_bf16_through_the_group_scale():
    """Every finite bf16 h, each alone in a group of 64 (the rest zeros, GELU(0) = 0): the group
    scale is |GELU(h)| / 7 and the code carries the sign, so equal scales and codes mean the fused
    GELU's bf16 value equals the oracle's for every input the kernel can see."""
    allb = np.arange(0, 0x10000, dtype=np.uint32).astype(np.uint16)
    vals = wl.bf16_bits_to_f32(allb)
    h_vals = allb[np.isfinite(vals)]
    G, K = 64, 4096
    rows = -(-len(h_vals) // (K // G))
    h = np.zeros((rows * (K // G), G), np.uint16)
    h[: len(h_vals), 0] = h_vals
    h = h.reshape(rows, K)
    z, codes, s = oracle.gelu_quantize_bf16(h, G)
    q, sa = jq.jq_gelu_quantize_act(dev_bf16(h), G)
    assert np.array_equal(q.cpu().numpy(), oracle.pack(codes)), "codes differ"
    got = sa.cpu().numpy().view(np.uint32)
    want = s.view(np.uint32)
    if not np.array_equal(got, want):
        bad = np.argwhere(got.reshape(-1) != want.reshape(-1))[:5, 0]
        raise AssertionError(f"{(got != want).sum()} group scales differ, e.g. inputs {h.reshape(-1, G)[bad, 0]}")


CAPTURE_FIRST = r"""
import sys
import numpy as np
import torch
sys.path.insert(0, sys.argv[1])
import oracle
import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl
rng = np.random.default_rng(9)
h = wl.f32_to_bf16_bits((rng.standard_normal((512, 4608)) * 2).astype(np.float32))
hd = torch.from_numpy(h.view(np.int16)).cuda().view(torch.bfloat16)
jq._load()
g = torch.cuda.CUDAGraph()
s = torch.cuda.Stream()
s.wait_stream(torch.cuda.current_stream())
with torch.cuda.stream(s):
    with torch.cuda.graph(g, stream=s):
        q, sa = jq.jq_gelu_quantize_act(hd, 128)
g.replay()
torch.cuda.synchronize()
_, codes, scales = oracle.gelu_quantize_bf16(h, 128)
ok = np.array_equal(q.cpu().numpy(), oracle.pack(codes)) and np.array_equal(sa.cpu().numpy(), scales)
q2, sa2 = jq.jq_gelu_quantize_act(hd, 128)  # an eager call after the capture
torch.cuda.synchronize()
ok = ok and np.array_equal(q2.cpu().numpy(), oracle.pack(codes)) and jq.jq_device_status() == 0
print("OK" if ok else "MISMATCH")
"""


def test_gelu_first_call_inside_a_graph_capture():
    """In a fresh process whose first fused GELU call is captured into a CUDA graph (the GELU
    table not yet filled on the device), the replayed graph and a later eager call both give the
    oracle's codes and scales."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, "-c", CAPTURE_FIRST, root], capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    assert out.stdout.strip().endswith("OK"), out.stdout[-500:] + out.stderr[-1000:]


def test_modulate_quantize_then_linear_at_the_dit_qkv_shape():
    """DiT-XL/2 attention input projection, 4 images of 256 tokens: 1024 x 1152 -> 3456, group128,
    through jq_modulate_quantize_act and jq_w4a4_linear; every output against the oracle."""
    M, K, N, T, G = 1024, 1152, 3456, 256, 128
    x, shift, scale = modulation_inputs(M, K, T, seed=11)
    w = wl.make("custom", seed=12, M=1, K=K, N=N, G=G, bias=True)
    _, codes, s = oracle.modulate_quantize_bf16(x, shift, scale, T, G)
    qw_codes, sw = oracle.quantize_f32(w.w, G)
    q, sa = jq.jq_modulate_quantize_act(dev_bf16(x), dev(shift), dev(scale), T, G)
    qw, sw_dev = jq.jq_pack_weight(dev(w.w), G)
    y = jq.jq_w4a4_linear(q, sa, qw, sw_dev, dev(w.bias), G)
    yb = y.view(torch.int16).cpu().numpy().view(np.uint16)
    check_linear_full(yb, codes, s, qw_codes, sw, w.bias, G, "dit qkv modulate")


def test_empty_batch_is_a_noop():
    x = torch.zeros((0, 256), dtype=torch.bfloat16, device="cuda")
    q, s = jq.jq_gelu_quantize_act(x, 128)
    assert q.shape == (0, 128) and s.shape == (0, 2)
