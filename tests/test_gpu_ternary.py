"""GPU parity of the W1.58A4 path (ternary weights, INT4 activations) through the C ABI.

Bit-exact: packed ternary codes and their scales against the oracle's absmean rule.  bf16
outputs: the same tolerance rule as the W4A4 layer (tests/helpers.py), against the oracle's
fp64 evaluation with the ternary codes.  M <= 16: the few-token kernel converts the packed
token codes itself; 16 < M <= 64: it reads them pre-expanded; M > 64: the ternary codes are
rewritten as INT4 and the GEMM runs.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl
from tests.helpers import check_linear, check_linear_full

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _device():
    assert torch.cuda.is_available(), "the gpu tests need a CUDA device"
    jq._load()
    yield
    assert jq.jq_device_status() == 0


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host_bits(y):
    return y.view(torch.int16).cpu().numpy().view(np.uint16)


def special_weights(N, K, G, rng):
    """Typical N(0, 0.02) weights with rows that stress the rule: a zero row, a zero group,
    constant groups, exact ties at s = 1, an outlier, huge and tiny magnitudes."""
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    w[0] = 0.0
    w[1, :G] = 0.0
    w[2] = -0.3
    t = np.tile(np.array([0.5, 1.5, 1.0, 1.0], np.float32), K // 4)  # mean |w| = 1: ties at +-0.5, +-1.5
    w[3] = t
    w[4, K // 3] = 50.0
    w[5] *= np.float32(1e30)
    w[6] *= np.float32(1e-30)
    return w


@pytest.mark.parametrize("N,K,G", [(520, 512, 64), (264, 512, 128), (96, 1024, 1024), (8, 15360, 64),
                                   (16, 4096, 4096)])
def test_pack_weight_ternary_bit_exact(N, K, G):
    rng = np.random.default_rng(N + K + G)
    w = special_weights(N, K, G, rng)
    codes, s = oracle.quantize_ternary_f32(w, G)
    qw2, sw = jq.jq_pack_weight_ternary(dev(w), G)
    torch.cuda.synchronize()
    assert np.array_equal(sw.cpu().numpy(), np.ascontiguousarray(s.T)), "scales differ from the oracle"
    assert np.array_equal(qw2.cpu().numpy(), oracle.pack_ternary(codes)), "packed codes differ from the oracle"


@pytest.mark.parametrize("M", [1, 9, 16, 40, 64, 200, 300])
@pytest.mark.parametrize("N,K,G,bias", [(264, 512, 64, True), (136, 1024, 128, False), (264, 2048, 2048, True)])
def test_w158a4_linear_matches_oracle(M, N, K, G, bias):
    rng = np.random.default_rng(7 * M + K + G)
    w = wl.make("custom", seed=M + N, M=M, K=K, N=N, G=G, bias=bias)
    x = w.x_bits
    qa, sa = oracle.quantize_bf16(x, G)
    qw, sw = oracle.quantize_ternary_f32(special_weights(N, K, G, rng), G)
    y64, _ = oracle.linear(qa, sa, qw, sw, w.bias, G)
    acc = oracle.group_partials(qa, qw, G)
    b = None if w.bias is None else dev(w.bias)
    y = jq.jq_w158a4_linear(dev(oracle.pack(qa)), dev(sa), dev(oracle.pack_ternary(qw)), dev(np.ascontiguousarray(sw.T)),
                            b, G)
    check_linear(host_bits(y), y64, acc, sa, sw, w.bias, f"M={M}")


@pytest.mark.parametrize("M", [16, 64, 1024])
def test_w158a4_dllm_shape_all_rows(M):
    """The dLLM gate/up shape (K=4096 -> N=12288, group128) with GPU-packed ternary weights, in
    the launch configuration the benchmark times: every output against the oracle, every packed
    weight byte and scale against the oracle's."""
    w = wl.make("dllm", seed=3, M=M)
    G = 128
    codes, s = oracle.quantize_ternary_f32(w.w, G)
    qw2, sw = jq.jq_pack_weight_ternary(dev(w.w), G)
    xd = torch.from_numpy(w.x_bits.view(np.int16)).cuda().view(torch.bfloat16)
    q, s_a = jq.jq_quantize_act(xd, G)
    y = jq.jq_w158a4_linear(q, s_a, qw2, sw, None, G)
    torch.cuda.synchronize()
    assert np.array_equal(qw2.cpu().numpy(), oracle.pack_ternary(codes))
    assert np.array_equal(sw.cpu().numpy(), np.ascontiguousarray(s.T))
    qa, sa = oracle.quantize_bf16(w.x_bits, G)
    check_linear_full(host_bits(y), qa, sa, codes, s, None, G, f"w158a4 dllm M={M}")
