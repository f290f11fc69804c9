"""GPU parity: the CUDA path through the C ABI against the CPU oracle, on seeded inputs.

Bit-exact: packed codes, scales, per-group integer partials.  bf16 outputs: within
ulp_bf16(y64) + (K/G + 2) * 2^-24 * (sum_g |acc*s_a*s_w| + |bias|) of the oracle's fp64 value
(see helpers.tolerance).  Shapes span several output tiles with ragged M and N tails; the
full-size configs run in the launch configuration bench.py times and are checked in full
(every code, scale and output), with the number of outputs that needed the fp32-summation
term of the tolerance recorded (helpers.report_escape).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl
from tests.helpers import Reference, check_linear, check_linear_full, report_escape

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _device():
    assert torch.cuda.is_available(), "the gpu tests need a CUDA device"
    jq._load()  # raises if libjq.so is missing: there is no fallback
    yield
    assert jq.jq_device_status() == 0


def dev_bf16(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch.bfloat16)


def dev(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def host_bits(y: torch.Tensor) -> np.ndarray:
    return y.view(torch.int16).cpu().numpy().view(np.uint16)


def special_rows(K: int, rng, extreme: bool = True) -> np.ndarray:
    """Rows that stress the quantiser: zeros, constants, exact ties, subnormals, an outlier,
    huge magnitudes (s_a > 2^110), and (extreme) the top of the bf16 range."""
    rows = []
    rows.append(np.zeros(K, np.float32))
    rows.append(np.full(K, -0.75, np.float32))
    t = np.tile(np.array([7.0, 0.5, 1.5, 2.5, -3.5, -0.5, 6.5, 4.5], np.float32), K // 8)  # s = 1: ties
    rows.append(t)
    sub = (rng.standard_normal(K) * 1e-39).astype(np.float32)  # bf16 subnormals
    rows.append(sub)
    o = rng.standard_normal(K).astype(np.float32)
    o[K // 3] = 3000.0
    rows.append(o)
    rows.append((rng.standard_normal(K) * 1e35).astype(np.float32))
    if extreme:
        big = np.full(K, 3.3e38, np.float32)
        big[1::2] = -1e38
        rows.append(big)
    return wl.f32_to_bf16_bits(np.stack(rows))


def act_bits(M, K, seed, special=True, extreme=True):
    rng = np.random.default_rng(seed)
    x = wl.make("custom", seed=seed, M=M, K=K, N=8, G=K, with_weights=False).x_bits
    if special:
        sp = special_rows(K, rng, extreme)
        x = x.copy()
        x[: len(sp)] = sp[: min(len(sp), M)]
    return x


# ----------------------------------------------------------------- quantiser ----

@pytest.mark.parametrize("M,K,G,pad", [(300, 512, 64, 0), (300, 512, 128, 0), (300, 512, 512, 0),
                                       (9, 15360, 64, 0), (7, 4096, 4096, 0), (1, 128, 128, 0),
                                       (37, 256, 64, 72), (63, 384, 64, 0),
                                       (64, 15360, 64, 0), (130, 1152, 64, 0), (130, 384, 128, 40),
                                       (65, 4096, 128, 8), (200, 128, 64, 0),
                                       # at least 4 tiles of 64 x 256 per SM: the TMA-staged kernel,
                                       # with a ragged last row tile and a half-empty last column tile
                                       (4100, 2432, 64, 40), (4100, 2432, 128, 0)])
def test_quantize_act_bit_exact(M, K, G, pad):
    x = act_bits(M, K, seed=M + K + G)
    ref_codes, ref_s = oracle.quantize_bf16(x, G)
    if pad:
        xp = np.zeros((M, K + pad), np.uint16)
        xp[:, :K] = x
        xd = dev_bf16(xp)[:, :K]
    else:
        xd = dev_bf16(x)
    q, s = jq.jq_quantize_act(xd, G)
    assert np.array_equal(q.cpu().numpy(), oracle.pack(ref_codes))
    assert np.array_equal(s.cpu().numpy().view(np.uint32), ref_s.view(np.uint32))


@pytest.mark.parametrize("G", [64, 128])
def test_quantize_act_exhaustive_bf16(G):
    """Every positive finite bf16 value, grouped with amaxes spread over the whole exponent
    range (and their negatives): codes and scales must equal the oracle's exactly.  This pins
    the reciprocal-multiply fast path with its near-tie fallback to the IEEE quotient."""
    allb = np.arange(1, 0x7F80, dtype=np.uint16)
    allf = wl.bf16_bits_to_f32(allb)
    amaxes = np.unique(np.concatenate([np.linspace(1, 0x7F7F, 150).astype(np.uint16),
                                       wl.f32_to_bf16_bits(np.array([1.0, 7.0, 3.5, 448.0], np.float32))]))
    rows = []
    per = G - 1
    for a in amaxes:
        xs = allb[allf <= wl.bf16_bits_to_f32(np.array([a]))[0]]
        n = (len(xs) + per - 1) // per
        blk = np.zeros((n, G), np.uint16)
        blk[:, 0] = a
        flat = np.zeros(n * per, np.uint16)
        flat[: len(xs)] = xs
        blk[:, 1:] = flat.reshape(n, per)
        rows.append(blk)
    x = np.concatenate(rows)
    x = np.concatenate([x, x ^ np.uint16(0x8000)])  # negatives
    M = x.shape[0] - x.shape[0] % 2
    x = x[:M].reshape(M // 2, 2 * G) if G == 64 else x
    ref_codes, ref_s = oracle.quantize_bf16(x, G)
    q, s = jq.jq_quantize_act(dev_bf16(x), G)
    assert np.array_equal(q.cpu().numpy(), oracle.pack(ref_codes))
    assert np.array_equal(s.cpu().numpy().view(np.uint32), ref_s.view(np.uint32))


@pytest.mark.parametrize("G", [64, 128])
def test_quantize_act_exhaustive_bf16_tiled(G):
    """The same values as test_quantize_act_exhaustive_bf16 (every positive finite bf16 under
    amaxes over the whole range, and their negatives), laid out as rows of 2048 and repeated so
    that the input takes the TMA-staged kernel (at least four 64 x 256 tiles per SM)."""
    allb = np.arange(1, 0x7F80, dtype=np.uint16)
    allf = wl.bf16_bits_to_f32(allb)
    amaxes = np.unique(np.concatenate([np.linspace(1, 0x7F7F, 150).astype(np.uint16),
                                       wl.f32_to_bf16_bits(np.array([1.0, 7.0, 3.5, 448.0], np.float32))]))
    per = G - 1
    rows = []
    for a in amaxes:
        xs = allb[allf <= wl.bf16_bits_to_f32(np.array([a]))[0]]
        n = (len(xs) + per - 1) // per
        blk = np.zeros((n, G), np.uint16)
        blk[:, 0] = a
        flat = np.zeros(n * per, np.uint16)
        flat[: len(xs)] = xs
        blk[:, 1:] = flat.reshape(n, per)
        rows.append(blk)
    groups = np.concatenate(rows)
    groups = np.concatenate([groups, groups ^ np.uint16(0x8000)])
    K = 2048
    reps = -(-(10 * 2 ** 20) // groups.size)  # >= 10 M elements: > 4 tiles per SM
    flat = np.tile(groups.reshape(-1), reps)
    flat = flat[: (flat.size // K) * K]
    x = flat.reshape(-1, K)
    ref_codes, ref_s = oracle.quantize_bf16(x, G)
    q, s = jq.jq_quantize_act(dev_bf16(x), G)
    assert np.array_equal(q.cpu().numpy(), oracle.pack(ref_codes))
    assert np.array_equal(s.cpu().numpy().view(np.uint32), ref_s.view(np.uint32))


@pytest.mark.slow
def test_quantize_act_every_bf16_pair():
    """Every positive finite bf16 amax with every bf16 x of magnitude up to it, both signs (about
    1.07e9 pairs), in groups of 128 that each hold one amax: codes and scales must equal the
    oracle's exactly.  This covers the compiled reciprocal shortcut and its fallback everywhere
    (tests/test_fast_division_argument.py checks the argument behind it on the CPU)."""
    G, per = 128, 127
    allb = np.arange(1, 0x7F80, dtype=np.uint16)  # positive finite bf16, increasing in value
    for chunk in np.array_split(np.arange(allb.size), 24):
        blocks = []
        for ia in chunk:
            xs = np.concatenate([allb[: ia + 1], allb[: ia + 1] ^ np.uint16(0x8000)])
            n = -(-xs.size // per)
            blk = np.zeros((n, G), np.uint16)
            blk[:, 0] = allb[ia]
            flat = np.zeros(n * per, np.uint16)
            flat[: xs.size] = xs
            blk[:, 1:] = flat.reshape(n, per)
            blocks.append(blk)
        x = np.concatenate(blocks)
        ref_codes, ref_s = oracle.quantize_bf16(x, G)
        q, s = jq.jq_quantize_act(dev_bf16(x), G)
        assert np.array_equal(q.cpu().numpy(), oracle.pack(ref_codes)), f"amax index {chunk[0]}..{chunk[-1]}"
        assert np.array_equal(s.cpu().numpy().view(np.uint32), ref_s.view(np.uint32))


@pytest.mark.parametrize("N,K,G", [(520, 512, 64), (264, 512, 128), (96, 1024, 1024), (8, 15360, 64)])
def test_pack_weight_bit_exact(N, K, G):
    rng = np.random.default_rng(N + K)
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    w[0] = 0.0
    w[1, ::2] = 1e-42   # fp32 subnormals
    w[2] = np.float32(-3.0e38)
    w[3, 5] = 40.0
    ref_codes, ref_s = oracle.quantize_f32(w, G)
    qw, s_w = jq.jq_pack_weight(dev(w), G)
    assert np.array_equal(qw.cpu().numpy(), oracle.pack(ref_codes))
    assert np.array_equal(s_w.cpu().numpy().view(np.uint32), np.ascontiguousarray(ref_s.T).view(np.uint32))


# ------------------------------------------------------------ integer partials ----

@pytest.mark.parametrize("M,N,K,G", [(300, 520, 512, 64), (300, 520, 512, 128), (300, 520, 512, 512),
                                     (128, 256, 128, 128), (1, 8, 128, 64), (130, 264, 4096, 4096)])
def test_group_partials_bit_exact(M, N, K, G):
    rng = np.random.default_rng(M * N + K)
    qa = wl.random_codes(rng, M, K)        # the full code range, -8 included
    qw = wl.random_codes(rng, N, K)
    qa[0] = -8
    qw[0] = -8
    ref = oracle.group_partials(qa, qw, G)
    acc = jq.jq_w4a4_group_partials(dev(oracle.pack(qa)), dev(oracle.pack(qw)), G)
    assert np.array_equal(acc.cpu().numpy(), ref)


# --------------------------------------------------------------- linear layer ----

def run_linear(ref: Reference, x_bits, fused: bool):
    qw, sw = dev(ref.packed_w), dev(ref.s_w_groupmajor)
    b = None if ref.bias is None else dev(ref.bias)
    if fused:
        return jq.jq_fused_quant_linear(dev_bf16(x_bits), qw, sw, b, ref.G)
    return jq.jq_w4a4_linear(dev(ref.packed_a), dev(ref.s_a), qw, sw, b, ref.G)


# M <= 16: the few-token kernel converts the packed token codes itself; 16 < M <= 64: it reads
# the tokens pre-expanded (operand image + corrections); M > 64: the GEMM
@pytest.mark.parametrize("M,N,K,G,bias", [(300, 520, 512, 64, True), (300, 520, 512, 128, False),
                                          (300, 520, 512, 512, True), (64, 256, 256, 64, True),
                                          (1, 8, 128, 128, True), (129, 8, 256, 64, False),
                                          (17, 264, 1024, 128, True), (40, 520, 512, 512, False),
                                          (64, 136, 2048, 2048, True), (33, 264, 768, 64, False),
                                          # an odd number of 128-deep K stages (the ring's last slot
                                          # holds one stage): DiT-XL/2's hidden size 1152 = 9 x 128
                                          (300, 264, 384, 64, True), (300, 264, 384, 128, False),
                                          (300, 264, 384, 384, True), (257, 520, 1152, 128, True),
                                          (257, 136, 1152, 1152, False), (40, 264, 1152, 128, True),
                                          # the GEMM's tile width follows the tile count (128 for
                                          # the small shapes above); 224 here, ragged in M and N
                                          (1000, 12200, 256, 64, False), (1000, 12200, 1152, 128, True),
                                          # and 256 (several rounds of tiles, ragged in M and N)
                                          (4500, 3000, 512, 64, True)])
def test_linear_matches_oracle(M, N, K, G, bias):
    w = wl.make("custom", seed=11 + M, M=M, K=K, N=N, G=G, bias=bias)
    x = act_bits(M, K, seed=3 + M, extreme=False) if M >= 8 else w.x_bits
    ref = Reference(x, w.w, w.bias, G)
    y64, _ = ref.linear()
    acc = ref.partials()
    for fused in (False, True):
        y = run_linear(ref, x, fused)
        check_linear(host_bits(y), y64, acc, ref.s_a, ref.s_w_rows, ref.bias, f"fused={fused}")


def test_fused_is_bit_identical_to_separate():
    w = wl.make("custom", seed=5, M=333, K=1024, N=264, G=64, bias=True)
    ref = Reference(w.x_bits, w.w, w.bias, 64)
    a = host_bits(run_linear(ref, w.x_bits, fused=False))
    b = host_bits(run_linear(ref, w.x_bits, fused=True))
    assert np.array_equal(a, b)


def test_full_code_range_linear():
    """Codes straight to the GEMM, -8 included, arbitrary positive scales."""
    rng = np.random.default_rng(21)
    M, N, K, G = 200, 264, 512, 64
    qa, qw = wl.random_codes(rng, M, K), wl.random_codes(rng, N, K)
    sa = rng.uniform(1e-3, 4.0, (M, K // G)).astype(np.float32)
    sw = rng.uniform(1e-4, 0.1, (N, K // G)).astype(np.float32)
    bias = rng.standard_normal(N).astype(np.float32)
    y64, _ = oracle.linear(qa, sa, qw, sw, bias, G)
    acc = oracle.group_partials(qa, qw, G)
    y = jq.jq_w4a4_linear(dev(oracle.pack(qa)), dev(sa), dev(oracle.pack(qw)), dev(np.ascontiguousarray(sw.T)),
                          dev(bias), G)
    check_linear(host_bits(y), y64, acc, sa, sw, bias)


@pytest.mark.parametrize("M", [1, 16, 33, 64, 200])
@pytest.mark.parametrize("K,G", [(4096, 4096), (16384, 16384), (4096, 128), (2048, 64)])
def test_large_partial_sums_cancel(M, K, G):
    """Running sums climb to ~49 K/2 and fall back to a small exact integer.

    Weight row n is +7 over the first half of K and -7 over the second (one code changed so that
    the row sums to -(n % 5)); token rows are all 7 or all -8.  With unit scales y = acc exactly,
    so an accumulation that dropped low bits of a large intermediate sum (or a mistaken code
    offset) shows up as a wrong small integer.  M <= 64 and M > 64 take different kernels.
    """
    N = 264
    qw = np.full((N, K), 7, np.int8)
    qw[:, K // 2:] = -7
    qw[:, 1] -= (np.arange(N) % 5).astype(np.int8)
    qa = np.where((np.arange(M) % 2 == 0)[:, None], np.int8(7), np.int8(-8)) * np.ones((M, K), np.int8)
    sa = np.ones((M, K // G), np.float32)
    sw = np.ones((N, K // G), np.float32)
    y64, _ = oracle.linear(qa, sa, qw, sw, None, G)
    acc = oracle.group_partials(qa, qw, G).sum(axis=2)
    assert np.abs(acc).max() <= 8 * 4 * 7  # the exact result is small; the running sums are not
    y = jq.jq_w4a4_linear(dev(oracle.pack(qa)), dev(sa), dev(oracle.pack(qw)), dev(np.ascontiguousarray(sw.T)),
                          None, G)
    assert np.array_equal(wl.bf16_bits_to_f32(host_bits(y)), acc.astype(np.float32))
    check_linear(host_bits(y), y64, oracle.group_partials(qa, qw, G), sa, sw, None)


@pytest.mark.parametrize("M", [16, 200])
def test_one_group_at_the_largest_k(M):
    """G = K at the largest K the library accepts, 262016 (2047 K stages of 128, an odd count).

    Codes in [4, 7] on both sides: the exact partial stays below 49 K < 2^24, but a sum of
    offset-code products (q_w + 8) q_a would climb to about 74 K > 2^24, where fp32 drops odd
    integers, so a run this long must keep the sign-magnitude form.  Both M take the GEMM (the
    few-token kernel takes one group only up to K = 139776)."""
    K, N = 262016, 136
    rng = np.random.default_rng(M + 5)
    qa = rng.integers(4, 8, (M, K), dtype=np.int8)
    qw = rng.integers(4, 8, (N, K), dtype=np.int8)
    ref = oracle.group_partials(qa, qw, K)
    pa, pw = dev(oracle.pack(qa)), dev(oracle.pack(qw))
    acc = jq.jq_w4a4_group_partials(pa, pw, K)
    assert np.array_equal(acc.cpu().numpy(), ref)
    sa = np.ones((M, 1), np.float32)
    sw = np.ones((N, 1), np.float32)
    y64, _ = oracle.linear(qa, sa, qw, sw, None, K)
    y = jq.jq_w4a4_linear(pa, dev(sa), pw, dev(np.ascontiguousarray(sw.T)), None, K)
    check_linear(host_bits(y), y64, ref, sa, sw, None)


def test_zero_weights_and_zero_activations():
    M, N, K, G = 130, 264, 256, 128
    w = wl.make("custom", seed=2, M=M, K=K, N=N, G=G, bias=True)
    x = w.x_bits.copy()
    x[7] = 0
    wt = w.w.copy()
    wt[9] = 0.0
    ref = Reference(x, wt, w.bias, G)
    y = host_bits(run_linear(ref, x, fused=False))
    yb = wl.bf16_bits_to_f32(y)
    assert np.array_equal(yb[7], wl.bf16_bits_to_f32(wl.f32_to_bf16_bits(w.bias)))
    assert np.array_equal(yb[:, 9], np.full(M, wl.bf16_bits_to_f32(wl.f32_to_bf16_bits(w.bias[9:10]))[0]))


@pytest.mark.parametrize("M", [16, 40])
def test_huge_activation_scale_path(M):
    """s_a above 2^110 takes the epilogue's overflow-safe ordering."""
    N, K, G = 256, 256, 64
    rng = np.random.default_rng(8)
    x = wl.f32_to_bf16_bits((rng.standard_normal((M, K)) * 2e35).astype(np.float32))
    w = (rng.standard_normal((N, K)) * 1e-3).astype(np.float32)
    ref = Reference(x, w, None, G)
    assert ref.s_a.max() > 2.0 ** 110
    y64, _ = ref.linear()
    check_linear(host_bits(run_linear(ref, x, fused=False)), y64, ref.partials(), ref.s_a, ref.s_w_rows, None)


def test_empty_batch_is_a_noop():
    qw = torch.zeros((8, 64), dtype=torch.uint8, device="cuda")
    sw = torch.zeros((2, 8), dtype=torch.float32, device="cuda")
    q = torch.zeros((0, 64), dtype=torch.uint8, device="cuda")
    sa = torch.zeros((0, 2), dtype=torch.float32, device="cuda")
    y = jq.jq_w4a4_linear(q, sa, qw, sw, None, 64)
    assert y.shape == (0, 8)


# ------------------------------------------------------ full-size configs (every output) ----

FULL = [("dllm", 128), ("dllm", 4096), ("flux_qkv", 64), ("flux_out", 64), ("tiny", 64), ("tiny", 256)]


@pytest.mark.parametrize("name,G", FULL)
def test_full_size_config(name, G):
    w = wl.make(name, seed=1)
    ref = Reference(w.x_bits, w.w, w.bias, G)
    xd = dev_bf16(w.x_bits)
    q, s = jq.jq_quantize_act(xd, G)
    assert np.array_equal(q.cpu().numpy(), ref.packed_a)
    assert np.array_equal(s.cpu().numpy().view(np.uint32), ref.s_a.view(np.uint32))
    qw, sw = jq.jq_pack_weight(dev(w.w), G)
    assert np.array_equal(qw.cpu().numpy(), ref.packed_w)
    assert np.array_equal(sw.cpu().numpy().view(np.uint32), ref.s_w_groupmajor.view(np.uint32))
    b = None if w.bias is None else dev(w.bias)
    y_sep = host_bits(jq.jq_w4a4_linear(q, s, qw, sw, b, G))
    y_fus = host_bits(jq.jq_fused_quant_linear(xd, qw, sw, b, G))
    assert np.array_equal(y_sep, y_fus)
    check_linear_full(y_sep, ref.qa, ref.s_a, ref.qw, ref.s_w_rows, ref.bias, G, f"{name} G={G}")


# The memory-to-compute crossover sweep at full size: both shapes (K=4096 -> N=12288 and
# K=3072 -> N=3072, per-token/per-channel scales) at token counts that take each kernel
# (1 and 64 tokens: the few-token kernel with and without pre-expanded tokens; 4096 and 16384:
# the GEMM).  Every code, scale and output against the oracle.
SWEEP_FULL = [("sweep_a", M) for M in (1, 64, 4096, 16384)] + [("sweep_b", M) for M in (1, 64, 4096, 16384)]


@pytest.mark.parametrize("name,M", SWEEP_FULL)
def test_sweep_full_size(name, M):
    K = 4096 if name == "sweep_a" else 3072
    G = K
    w = wl.make(name, seed=2, M=M, G=G)
    xd = dev_bf16(w.x_bits)
    q, s = jq.jq_quantize_act(xd, G)
    qw, sw = jq.jq_pack_weight(dev(w.w), G)
    y = host_bits(jq.jq_w4a4_linear(q, s, qw, sw, None, G))
    codes_a, s_a = oracle.quantize_bf16(w.x_bits, G)
    assert np.array_equal(q.cpu().numpy(), oracle.pack(codes_a))
    assert np.array_equal(s.cpu().numpy().view(np.uint32), s_a.view(np.uint32))
    codes_w, s_w = oracle.quantize_f32(w.w, G)
    assert np.array_equal(qw.cpu().numpy(), oracle.pack(codes_w))
    assert np.array_equal(sw.cpu().numpy().view(np.uint32), np.ascontiguousarray(s_w.T).view(np.uint32))
    check_linear_full(y, codes_a, s_a, codes_w, s_w, None, G, f"{name} M={M}")
