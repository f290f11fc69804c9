"""The Python binding's argument checks (no GPU needed).

The C ABI receives bare pointers and sizes, so it cannot see that a tensor is smaller than the
call implies, strided, of another type or on another device; the binding refuses such tensors
before anything reaches the library.  Host tensors of the right form get through these checks
and stop at the next one (CUDA tensors only), which is how these tests tell the two apart.
"""
import pytest
import torch

import paper_2609_33601_gb300 as jq

M, N, K, G = 5, 16, 256, 64
CUDA_ONLY = "CUDA tensors only"


def u8(*shape):
    return torch.zeros(shape, dtype=torch.uint8)


def f32(*shape):
    return torch.zeros(shape, dtype=torch.float32)


def bf16(*shape):
    return torch.zeros(shape, dtype=torch.bfloat16)


def good_linear():
    return dict(q=u8(M, K // 2), s_a=f32(M, K // G), qw=u8(N, K // 2), s_w=f32(K // G, N), bias=f32(N))


def call_linear(a, **kw):
    return jq.jq_w4a4_linear(a["q"], a["s_a"], a["qw"], a["s_w"], a["bias"], G, **kw)


def test_well_formed_arguments_reach_the_device_check():
    with pytest.raises(ValueError, match=CUDA_ONLY):
        call_linear(good_linear())
    with pytest.raises(ValueError, match=CUDA_ONLY):
        call_linear(good_linear(), y=bf16(M, N), workspace=u8(1 << 16))
    a = good_linear()
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_w4a4_linear_noalloc(a["q"], a["s_a"], a["qw"], a["s_w"], None, G)
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_fused_quant_linear(bf16(M, K), a["qw"], a["s_w"], a["bias"], G)
    padded = bf16(M, K + 64)[:, :K]  # rows padded: allowed through ldx
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_quantize_act(padded, G)
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_quantize_act(bf16(M, K), G, u8(M, K // 2), f32(M, K // G))
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_pack_weight(f32(N, K), G)
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_pack_weight_ternary(f32(N, K), G)
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_w158a4_linear(a["q"], a["s_a"], u8(N, K // 4), a["s_w"], None, G)
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_w4a4_group_partials(a["q"], a["qw"], G)
    # one group (per token / per channel): scales [M, 1] and [1, N]
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_w4a4_linear(a["q"], f32(M, 1), a["qw"], f32(1, N), None, K)
    # an empty batch is well formed
    with pytest.raises(ValueError, match=CUDA_ONLY):
        jq.jq_w4a4_linear(u8(0, K // 2), f32(0, K // G), a["qw"], a["s_w"], None, G)


@pytest.mark.parametrize("name,bad", [
    ("s_a", f32(M, K // G - 1)),                # too few groups
    ("s_a", f32(M - 1, K // G)),                # too few tokens
    ("s_a", f32(K // G, M).t()),                # transposed view: not contiguous
    ("s_a", torch.zeros((M, K // G), dtype=torch.float64)),
    ("s_w", f32(N, K // G)),                    # token-major instead of group-major
    ("s_w", f32(K // G, N - 8)),
    ("bias", f32(N - 1)),
    ("bias", torch.zeros(N, dtype=torch.bfloat16)),
    ("qw", u8(N, K // 4)),                      # ternary-sized weights to the INT4 call
    ("qw", torch.zeros((N, K // 2), dtype=torch.int8)),
    ("q", u8(M, K)[:, ::2]),                    # strided codes
])
def test_malformed_linear_arguments_are_refused_by_name(name, bad):
    a = good_linear()
    a[name] = bad
    with pytest.raises(ValueError) as e:
        call_linear(a)
    msg = str(e.value)
    assert CUDA_ONLY not in msg
    assert ("packed weights" if name == "qw" else name) in msg


@pytest.mark.parametrize("kw", [dict(y=bf16(M, N - 8)), dict(y=f32(M, N)), dict(y=bf16(N, M).t()),
                                dict(workspace=f32(1024)), dict(workspace=u8(32, 32))])
def test_malformed_output_and_workspace_are_refused(kw):
    with pytest.raises(ValueError) as e:
        call_linear(good_linear(), **kw)
    assert CUDA_ONLY not in str(e.value) and next(iter(kw)) in str(e.value)


def test_other_entry_points_refuse_malformed_tensors():
    a = good_linear()
    cases = [
        lambda: jq.jq_quantize_act(f32(M, K), G),                                  # not bf16
        lambda: jq.jq_quantize_act(bf16(K, M).t(), G),                             # column-major
        lambda: jq.jq_quantize_act(bf16(M, K), G, u8(M, K // 4)),                  # q too small
        lambda: jq.jq_quantize_act(bf16(M, K), G, None, f32(M, K // 128)),         # s_a for another group
        lambda: jq.jq_pack_weight(f32(K, N).t(), G),                               # strided weights
        lambda: jq.jq_pack_weight(torch.zeros((N, K), dtype=torch.float64), G),
        lambda: jq.jq_pack_weight_ternary(bf16(N, K), G),
        lambda: jq.jq_fused_quant_linear(bf16(M, K), u8(N, K // 4), a["s_w"], None, G),
        lambda: jq.jq_fused_quant_linear(bf16(M, K), a["qw"], f32(N, K // G), None, G),
        lambda: jq.jq_w158a4_linear(a["q"], a["s_a"], a["qw"], a["s_w"], None, G),  # INT4-sized weights
        lambda: jq.jq_w4a4_group_partials(a["q"], u8(N - 8, K // 4), G),
        lambda: jq.jq_w4a4_group_partials(a["q"], a["qw"], 100),                   # group does not divide K
        lambda: jq.jq_w4a4_linear_noalloc(a["q"], a["s_a"], a["qw"], f32(N, K // G), None, G),
    ]
    for i, c in enumerate(cases):
        with pytest.raises(ValueError) as e:
            c()
        assert CUDA_ONLY not in str(e.value), i


def test_tensors_on_different_devices_are_refused():
    a = good_linear()
    a["s_w"] = torch.zeros((K // G, N), dtype=torch.float32, device="meta")
    with pytest.raises(ValueError) as e:
        call_linear(a)
    assert "s_w" in str(e.value) and CUDA_ONLY not in str(e.value)


def test_tensors_of_another_gpu_than_the_current_one_are_refused():
    """The C calls launch on the current CUDA device; tensors (or a stream) of another device
    would be addressed there as foreign pointers, so the binding names the mismatch first."""
    cuda1 = torch.device("cuda", 1)
    assert jq._device_mismatch(torch.device("cuda", 0), 0) is None
    assert jq._device_mismatch(cuda1, 1, cuda1) is None
    why = jq._device_mismatch(cuda1, 0)
    assert why is not None and "cuda:1" in why and "current CUDA device is cuda:0" in why
    why = jq._device_mismatch(torch.device("cuda", 0), 0, cuda1)
    assert why is not None and "stream" in why
