"""GPU parity of the training-side fake quantisation and straight-through backward.

jq_fake_quant_act, jq_fake_quant_weight and jq_ste_backward against the oracle
(oracle_fake_quant_bf16, oracle_fake_quant_f32, oracle_ste_backward_bf16) on the same seeded inputs, bit for bit: the scales, the 0/1 mask and
the bf16 xhat (one rounding of the exact product q*s) are all decided in the same fp32 steps
on both sides, so nothing here needs a tolerance.  Shapes cover several 2048-element row
chunks with a ragged last chunk, one group per row with a partly filled warp (K = 384), rows
beyond one wave of blocks, clamping learned scales, all-zero groups, the hand-built case whose
exact product sits a quarter fp32 ulp above a bf16 midpoint, and the dLLM gate/up activation
shape (1024 x 4096, group128).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu, pytest.mark.late]


def _to_dev_bf16(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def _bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def _check(xb, G, s_in=None, what=""):
    s_dev = None if s_in is None else torch.from_numpy(s_in).cuda()
    xhat, mask, s = jq.jq_fake_quant_act(_to_dev_bf16(xb), G, s_dev)
    torch.cuda.synchronize()
    ox, om, os_ = oracle.fake_quant_bf16(xb, G, s_in)
    assert (s.cpu().numpy().view(np.uint32) == os_.view(np.uint32)).all(), f"{what}: scales"
    assert (mask.cpu().numpy() == om).all(), f"{what}: mask"
    bad = np.argwhere(_bits(xhat) != ox)
    assert bad.size == 0, f"{what}: {len(bad)} xhat mismatches, first at {bad[:3].tolist()}"
    return om


def _gen(seed, M, K):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((M, K)).astype(np.float32)
    x[:, rng.choice(K, max(1, K // 100), replace=False)] *= 20.0  # outlier channels
    return wl.f32_to_bf16_bits(x)


# Four rows per block from 2432 rows on (152 SMs), else one: a ragged last block at 2433 rows.
@pytest.mark.parametrize("M,K,G", [(64, 256, 64), (64, 256, 128), (64, 256, 256), (37, 384, 384),
                                   (37, 384, 128), (5, 6144, 64), (3, 6144, 6144), (1500, 128, 128),
                                   (2433, 256, 64), (2436, 384, 384), (2437, 1024, 128)])
def test_amax_rule_matches_the_oracle(M, K, G):
    xb = _gen(M * 7 + K + G, M, K)
    xb[min(2, M - 1), :G] = 0  # an all-zero group
    om = _check(xb, G, what=f"{M}x{K} G={G}")
    assert om.all()


@pytest.mark.parametrize("M,K,G", [(33, 256, 64), (9, 2304, 128), (4, 384, 384), (2435, 256, 64)])
def test_given_scales_clamp_like_the_oracle(M, K, G):
    xb = _gen(100 + M, M, K)
    rng = np.random.default_rng(M)
    s_in = rng.uniform(0.02, 0.5, (M, K // G)).astype(np.float32)
    om = _check(xb, G, s_in, what=f"given scales {M}x{K} G={G}")
    assert not om.all()  # these scales clamp the outlier channels


def test_single_rounding_case_and_the_tiny_workload():
    s = np.float32(9624430 * 2.0 ** -26)
    x = np.zeros((2, 128), np.float32)
    x[0, :2] = [1.0, -1.0]
    xb = wl.f32_to_bf16_bits(x)
    s_in = np.full((2, 1), s, np.float32)
    xhat, _, _ = jq.jq_fake_quant_act(_to_dev_bf16(xb), 128, torch.from_numpy(s_in).cuda())
    assert [f"{v:04X}" for v in _bits(xhat)[0, :2]] == ["3F81", "BF81"]
    w = wl.make("tiny", seed=2)
    _check(w.x_bits, w.G, what="tiny workload")


def test_dllm_gate_up_activation_shape():
    w = wl.make("dllm", seed=1)
    _check(w.x_bits, 128, what="dLLM 1024x4096 G=128")


@pytest.mark.parametrize("n", [1, 7, 8, 1003, 1 << 20])
def test_ste_backward_matches_the_oracle(n):
    rng = np.random.default_rng(n)
    g = wl.f32_to_bf16_bits(rng.standard_normal(n).astype(np.float32))
    m = (rng.random(n) < 0.7).astype(np.uint8)
    out = jq.jq_ste_backward(_to_dev_bf16(g), torch.from_numpy(m).cuda())
    want = oracle.ste_backward_bf16(g.reshape(1, -1), m.reshape(1, -1)).reshape(-1)
    assert (_bits(out) == want).all()


def test_forward_mask_feeds_the_backward():
    xb = _gen(7, 16, 512)
    s_in = np.full((16, 512 // 64), 0.1, np.float32)
    x = _to_dev_bf16(xb)
    _, mask, _ = jq.jq_fake_quant_act(x, 64, torch.from_numpy(s_in).cuda())
    grad = torch.randn((16, 512), device="cuda").to(torch.bfloat16)
    gx = jq.jq_ste_backward(grad, mask)
    keep = mask.bool()
    assert torch.equal(gx[keep], grad[keep]) and (gx[~keep].view(torch.int16) == 0).all()


@pytest.mark.parametrize("N,K,G,given", [(256, 256, 64, False), (96, 384, 384, False), (300, 4096, 128, False),
                                         (1300, 128, 128, False), (40, 2304, 128, True), (2434, 3072, 64, False),
                                         (2441, 512, 128, True)])
def test_weight_fake_quant_matches_the_oracle(N, K, G, given):
    rng = np.random.default_rng(N + K)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    w[1, :G] = 0  # an all-zero group
    s_in = rng.uniform(0.001, 0.006, (N, K // G)).astype(np.float32) if given else None
    what, mask, s = jq.jq_fake_quant_weight(torch.from_numpy(w).cuda(), G,
                                            None if s_in is None else torch.from_numpy(s_in).cuda())
    ow, om, os_ = oracle.fake_quant_f32(w, G, s_in)
    assert (s.cpu().numpy().view(np.uint32) == os_.view(np.uint32)).all()
    assert (mask.cpu().numpy() == om).all()
    assert (what.cpu().numpy().view(np.uint32) == ow.view(np.uint32)).all()
    assert om.all() != given  # the amax rule never clamps; these small given scales do
