"""Pins for the CPU oracle: checks against things other than the oracle itself.

The paper prints no numeric example of its quantiser (it names only "INT4
weights/activations, group128" and "W4A4 group64": Appendix experimental
detail tables, Sec. 4.2 "FLUX"), so the pins are:

* hand-worked examples whose expected values are derived by hand in the
  comments from the symmetric INT4 rule (stored in tests/golden/);
* an independent exact-rational evaluation of the rule (Python Fractions with
  our own fp32 round-to-nearest-even) -- this pins that the oracle's division
  is the correctly rounded IEEE one and that rint breaks ties to even;
* mathematical invariants of round-to-nearest quantisation;
* brute force on tiny shapes (pure-Python loops, a different loop order);
* special cases that reduce to library routines (numpy fp64 matmul of the
  dequantised groups; the int64 matmul when all scales are 1);
* a hand-derived bf16 rounding table.

Shapes are deliberately non-square with distinct per-group scales and nonzero
bias, so a transposed operand, a wrong group index, a dropped bias or a
flipped sign breaks at least one test.
"""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2609_33601_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- helpers ----

def f32_rne(fr: Fraction) -> float:
    """Exact rational -> nearest fp32 (ties to even), written from the IEEE-754
    definition (24-bit significand, subnormals below 2^-126)."""
    if fr == 0:
        return 0.0
    sign = -1 if fr < 0 else 1
    a = abs(fr)
    e = a.numerator.bit_length() - a.denominator.bit_length()
    if Fraction(2) ** e > a:
        e -= 1
    # now 2^e <= a < 2^(e+1)
    ulp_e = max(e, -126) - 23
    q = a / Fraction(2) ** ulp_e
    n = math.floor(q)
    rem = q - n
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and n % 2 == 1):
        n += 1
    return sign * float(Fraction(n) * Fraction(2) ** ulp_e)


def quant_ref(xs):
    """Exact-rational evaluation of the symmetric INT4 rule on one group."""
    xs = [float(np.float32(v)) for v in xs]
    amax = max(abs(v) for v in xs)
    if amax == 0:
        return [0] * len(xs), 0.0
    s = f32_rne(Fraction(amax) / 7)
    out = []
    for v in xs:
        t = f32_rne(Fraction(v) / Fraction(s))
        q = round(t)  # Python rounds half to even
        out.append(max(-8, min(7, q)))
    return out, s


def bits(a):
    return wl.f32_to_bf16_bits(np.asarray(a, np.float32))


def load_golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ------------------------------------------------------ hand-worked pins ----

def test_worked_example_quantise_and_pack():
    g = load_golden("worked_example_g8.json")
    x = np.array([g["x"]], np.float32)
    codes, scales = oracle.quantize_bf16(bits(x), group=8)
    assert scales[0, 0] == np.float32(g["scale"])
    assert codes[0].tolist() == g["codes"]
    packed = oracle.pack(codes)
    assert packed[0].tolist() == [int(b, 16) for b in g["packed_hex"]]
    assert oracle.unpack(packed)[0].tolist() == g["codes"]
    # dequantisation error reaches s/2 exactly at the two ties
    deq = codes[0].astype(np.float64) * scales[0, 0]
    assert np.max(np.abs(deq - x[0])) == g["scale"] / 2


def test_worked_example_linear():
    g = load_golden("worked_example_g8.json")
    x = np.array([g["x"]], np.float32)
    qa, sa = oracle.quantize_bf16(bits(x), group=8)
    qw = np.ones((1, 8), np.int8)
    sw = np.array([[g["linear"]["s_w"]]], np.float32)
    bias = np.array([g["linear"]["bias"]], np.float32)
    acc = oracle.group_partials(qa, qw, 8)
    assert acc[0, 0, 0] == g["linear"]["acc"]
    y64, yb = oracle.linear(qa, sa, qw, sw, bias, 8)
    assert y64[0, 0] == g["linear"]["y"]
    assert yb[0, 0] == int(g["linear"]["y_bf16_hex"], 16)


def test_division_reading_pins_fl_x_over_s():
    # amax = 1 -> s = fl(1/7) = 0x3E124925 (slightly above 1/7), so
    # fl(0.5 / s) = 3.4999998 < 3.5 and the code is 3; the real-arithmetic
    # 0.5 * 7 = 3.5 would round (to even) to 4.
    g = load_golden("division_reading.json")
    codes, scales = oracle.quantize_bf16(bits([[g["amax"], g["x"]]]), group=2)
    assert scales.view(np.uint32)[0, 0] == int(g["scale_bits_hex"], 16)
    assert codes[0].tolist() == [7, g["code"]]


# ------------------------------------------- exact-rational cross-check ----

@pytest.mark.parametrize("seed", [0, 1, 2])
def test_quantiser_matches_exact_rational_rule(seed):
    rng = np.random.default_rng(seed)
    G = 16
    x = rng.standard_normal((40, G)).astype(np.float32) * rng.choice([1e-3, 1.0, 37.0], size=(40, 1))
    x[3] = 0.0                      # all-zero group
    x[5] = 2.5                      # constant group
    x[7, :4] = [7.0, 3.5, -3.5, 0.5]  # exact ties once scaled by s = 1
    xb = bits(x)
    codes, scales = oracle.quantize_bf16(xb, group=G)
    xf = wl.bf16_bits_to_f32(xb)
    for r in range(x.shape[0]):
        q_ref, s_ref = quant_ref(xf[r])
        assert scales[r, 0] == np.float32(s_ref), r
        assert codes[r].tolist() == q_ref, r


def test_quantiser_exhaustive_positive_bf16():
    """Every positive finite bf16 x, paired with a group amax >= x, at several
    amax values: codes equal the exact-rational rule, are monotone in x and
    are one of floor/ceil of the real quotient."""
    allb = np.arange(1, 0x7F80, dtype=np.uint16)
    allf = wl.bf16_bits_to_f32(allb)
    for amax in (1.0, 3.5, 448.0, 1.0e-38, 3.3e38):
        am_b = bits([amax])[0]
        am = float(wl.bf16_bits_to_f32(np.array([am_b]))[0])
        sel = allb[allf <= am]
        rows = np.stack([np.full(sel.shape, am_b, np.uint16), sel], axis=1)
        codes, scales = oracle.quantize_bf16(rows, group=2)
        s = float(scales[0, 0])
        assert s == f32_rne(Fraction(am) / 7)
        assert np.all(codes[:, 0] == 7)
        q = codes[:, 1].astype(np.int64)
        assert np.all(np.diff(q) >= 0)
        assert q.min() >= 0 and q.max() <= 7
        xs = wl.bf16_bits_to_f32(sel).astype(np.float64)
        real = np.array([float(Fraction(float(v)) / Fraction(s)) for v in xs])
        assert np.all((q == np.floor(real)) | (q == np.ceil(real)))
        # exact-rational rule on a strided subsample (every 7th value + the ends)
        idx = np.unique(np.concatenate([np.arange(0, len(sel), 7), [len(sel) - 1]]))
        for i in idx:
            t = f32_rne(Fraction(float(xs[i])) / Fraction(s))
            assert q[i] == round(t), (amax, xs[i])


# ---------------------------------------------------------- invariants ----

def test_quantiser_invariants():
    w = wl.make("tiny", seed=3)
    for G in (64, 128, 256):
        codes, s = oracle.quantize_bf16(w.x_bits, group=G)
        xf = wl.bf16_bits_to_f32(w.x_bits).astype(np.float64).reshape(w.M, w.K // G, G)
        c = codes.astype(np.float64).reshape(w.M, w.K // G, G)
        assert codes.min() >= -7 and codes.max() <= 7          # symmetric: never -8
        err = np.abs(xf - c * s.astype(np.float64)[..., None])
        assert np.all(err <= s[..., None] / 2 * (1 + 2.0 ** -20))
        # the element reaching amax maps to +-7
        arg = np.abs(xf).argmax(axis=2)
        top = np.take_along_axis(c, arg[..., None], axis=2)[..., 0]
        assert np.all(np.abs(top) == 7)
        # sign symmetry q(-x) = -q(x)
        neg = w.x_bits ^ np.uint16(0x8000)
        codes_n, s_n = oracle.quantize_bf16(neg, group=G)
        assert np.array_equal(codes_n, -codes) and np.array_equal(s_n, s)


def test_zero_and_constant_groups():
    x = np.zeros((3, 128), np.float32)
    x[1] = -0.75
    x[2, :64] = 5.0
    codes, s = oracle.quantize_bf16(bits(x), group=64)
    assert np.all(codes[0] == 0) and np.all(s[0] == 0)
    assert np.all(codes[1] == -7)
    assert np.all(codes[2, :64] == 7) and np.all(codes[2, 64:] == 0) and s[2, 1] == 0


def test_strided_rows_match_contiguous():
    w = wl.make("tiny", seed=4)
    big = np.zeros((w.M, w.K + 64), np.uint16)
    big[:, :w.K] = w.x_bits
    a = oracle.quantize_bf16(big[:, :w.K], group=64)
    b = oracle.quantize_bf16(w.x_bits, group=64)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_weight_quantiser_equals_activation_rule_on_bf16_exact_values():
    rng = np.random.default_rng(5)
    xb = bits(rng.standard_normal((17, 128)))
    xf = wl.bf16_bits_to_f32(xb)
    ca, sa = oracle.quantize_bf16(xb, group=64)
    cw, sw = oracle.quantize_f32(xf, group=64)
    assert np.array_equal(ca, cw) and np.array_equal(sa, sw)


@pytest.mark.parametrize("seed", [0, 1])
def test_weight_quantiser_matches_exact_rational_rule_on_fp32_values(seed):
    """The fp32 weight path on values that are not bf16-exact (24 significant bits), against the
    exact-rational rule directly: random magnitudes over many binades, fp32 subnormals, groups
    whose quotients fall on exact ties (x = (k + 1/2) s with s = amax/7 representable), and
    values one fp32 ulp either side of such ties."""
    rng = np.random.default_rng(100 + seed)
    G = 16
    w = (rng.standard_normal((48, G)) * np.exp(rng.uniform(-30, 30, (48, 1)))).astype(np.float32)
    w[0] = 0.0
    w[1, :] = np.float32(3e-42)                       # fp32 subnormal group
    w[1, 5] = np.float32(7e-42)
    s = np.float32(0.25)                              # amax 1.75 gives s = fl32(1.75 / 7) = 0.25
    w[2] = np.float32(0.0)
    w[2, :8] = np.array([1.75, 0.625, -0.625, 0.875, -1.125, 0.375, 0.125, -0.125], np.float32)
    w[3] = w[2]
    w[3, 1:8] = np.nextafter(w[2, 1:8], np.float32(np.inf))     # just above the ties
    w[4] = w[2]
    w[4, 1:8] = np.nextafter(w[2, 1:8], np.float32(-np.inf))    # just below
    assert np.float32(np.float32(1.75) / np.float32(7)) == s
    codes, scales = oracle.quantize_f32(w, group=G)
    for r in range(w.shape[0]):
        q_ref, s_ref = quant_ref(w[r])
        assert scales[r, 0] == np.float32(s_ref), r
        assert codes[r].tolist() == q_ref, r


# ---------------------------------------------------------------- packing ----

def test_pack_all_byte_values_round_trip():
    allbytes = np.arange(256, dtype=np.uint8).reshape(1, 256)
    codes = oracle.unpack(allbytes)
    lo = np.arange(256) & 0xF
    hi = np.arange(256) >> 4
    sx = lambda v: np.where(v >= 8, v - 16, v)
    assert codes[0, 0::2].tolist() == sx(lo).tolist()
    assert codes[0, 1::2].tolist() == sx(hi).tolist()
    assert np.array_equal(oracle.pack(codes), allbytes)


# ------------------------------------------------ GEMM / epilogue pins ----

def test_group_partials_brute_force():
    rng = np.random.default_rng(6)
    M, N, K, G = 3, 5, 32, 8
    qa = wl.random_codes(rng, M, K)
    qw = wl.random_codes(rng, N, K)
    acc = oracle.group_partials(qa, qw, G)
    for m in range(M):
        for n in range(N):
            for g in range(K // G):
                s = 0
                for k in reversed(range(g * G, (g + 1) * G)):
                    s += int(qa[m, k]) * int(qw[n, k])
                assert acc[m, n, g] == s


def test_partials_extreme_codes():
    M, N, K, G = 2, 3, 256, 128
    qa = np.full((M, K), -8, np.int8)
    qw = np.full((N, K), -8, np.int8)
    qw[1] = 7
    acc = oracle.group_partials(qa, qw, G)
    assert np.all(acc[:, 0] == 64 * G) and np.all(acc[:, 1] == -56 * G)


def test_linear_matches_numpy_fp64_dequant_matmul():
    rng = np.random.default_rng(7)
    M, N, K, G = 37, 29, 256, 64
    qa = wl.random_codes(rng, M, K)
    qw = wl.random_codes(rng, N, K)
    sa = rng.uniform(0.01, 2.0, size=(M, K // G)).astype(np.float32)
    sw = rng.uniform(0.001, 0.1, size=(N, K // G)).astype(np.float32)
    bias = rng.standard_normal(N).astype(np.float32)
    y64, yb = oracle.linear(qa, sa, qw, sw, bias, G)
    ref = np.zeros((M, N))
    for g in range(K // G):
        A = qa[:, g * G:(g + 1) * G].astype(np.float64) * sa[:, g:g + 1].astype(np.float64)
        B = qw[:, g * G:(g + 1) * G].astype(np.float64) * sw[:, g:g + 1].astype(np.float64)
        ref += A @ B.T
    ref += bias.astype(np.float64)[None, :]
    np.testing.assert_allclose(y64, ref, rtol=1e-12, atol=1e-12)
    # bias broadcasts over rows (a transposed or dropped bias fails this)
    y0, _ = oracle.linear(qa, sa, qw, sw, None, G)
    np.testing.assert_allclose(y64 - y0, np.broadcast_to(bias.astype(np.float64), (M, N)), rtol=0, atol=1e-12)


def test_unit_scales_reduce_to_integer_matmul():
    rng = np.random.default_rng(8)
    M, N, K, G = 11, 13, 384, 128
    qa = wl.random_codes(rng, M, K)
    qw = wl.random_codes(rng, N, K)
    y64, _ = oracle.linear(qa, np.ones((M, K // G), np.float32), qw, np.ones((N, K // G), np.float32), None, G)
    assert np.array_equal(y64, (qa.astype(np.int64) @ qw.astype(np.int64).T).astype(np.float64))


def test_per_token_special_case():
    """G = K is per-token activations x per-output-channel weights:
    y = (qa . qw) * s_a[m] * s_w[n] + bias[n]."""
    w = wl.make("tiny", seed=9)
    K = w.K
    qa, sa = oracle.quantize_bf16(w.x_bits, group=K)
    qw, sw = oracle.quantize_f32(w.w, group=K)
    assert sa.shape == (w.M, 1) and sw.shape == (w.N, 1)
    amax_row = np.abs(wl.bf16_bits_to_f32(w.x_bits)).max(axis=1)
    assert np.array_equal(sa[:, 0], (amax_row / np.float32(7)).astype(np.float32))
    y64, _ = oracle.linear(qa, sa, qw, sw, w.bias, K)
    dot = qa.astype(np.int64) @ qw.astype(np.int64).T
    ref = dot * sa.astype(np.float64) * sw[:, 0].astype(np.float64)[None, :] + w.bias.astype(np.float64)
    np.testing.assert_allclose(y64, ref, rtol=1e-13, atol=1e-13)


# -------------------------------------------------------------- bf16 RNE ----

@pytest.mark.parametrize("v,expect", [
    (1.0, 0x3F80),
    (1.0 + 2.0 ** -8, 0x3F80),                 # tie -> even (mantissa 0)
    (1.0 + 3 * 2.0 ** -8, 0x3F82),             # tie between mantissa 1 and 2 -> 2
    (1.0 + 2.0 ** -8 + 2.0 ** -30, 0x3F81),    # just above the tie
    (1.0 + 2.0 ** -8 - 2.0 ** -30, 0x3F80),    # just below the tie
    (-2.5, 0xC020),
    (-0.0, 0x8000),
    (2.0 ** -133, 0x0001),                     # smallest subnormal
    (2.0 ** -134, 0x0000),                     # tie between 0 and 2^-133 -> 0
    (3 * 2.0 ** -134, 0x0002),                 # tie between 1 and 2 quanta -> 2
    (2.0 ** -126 * (1 - 2.0 ** -9), 0x0080),   # rounds up to the smallest normal
    (255.0 * 2.0 ** 120, 0x7F7F),              # largest finite
    (255.5 * 2.0 ** 120, 0x7F80),              # tie past the largest finite -> inf
    (3.0e40, 0x7F80),
])
def test_bf16_rne_table(v, expect):
    assert oracle.bf16_rne(v) == expect


# ------------------------------------------------ ternary weights (W1.58A4) ----

def ternary_ref(ws):
    """Exact-rational evaluation of the absmean ternary rule on one group: s = fl32(mean |w|)
    with the mean taken exactly, q = clamp(round(fl32(w/s)), -1, 1).  The oracle sums the group
    in fp64, which matches this unless the exact mean sits within ~G * 2^-53 (relative) of an
    fp32 rounding boundary."""
    ws = [float(np.float32(v)) for v in ws]
    mean = sum(Fraction(abs(v)) for v in ws) / len(ws)
    if mean == 0:
        return [0] * len(ws), 0.0
    s = f32_rne(mean)
    out = []
    for v in ws:
        t = f32_rne(Fraction(v) / Fraction(s))
        out.append(max(-1, min(1, round(t))))
    return out, s


def test_ternary_worked_example():
    g = load_golden("ternary_example.json")
    codes, s = oracle.quantize_ternary_f32(np.array([g["w"]], np.float32), 8)
    assert codes[0].tolist() == g["codes"] and float(s[0, 0]) == g["scale"]
    codes, s = oracle.quantize_ternary_f32(np.array([g["tie_w"]], np.float32), 4)
    assert codes[0].tolist() == g["tie_codes"] and float(s[0, 0]) == g["tie_scale"]
    packed = oracle.pack_ternary(np.array([g["pack_codes"]], np.int8))
    assert [f"{b:02X}" for b in packed[0]] == g["packed_hex"]
    assert oracle.unpack_ternary(packed)[0].tolist() == g["pack_codes"]
    lin = g["linear"]
    qw, sw = oracle.quantize_ternary_f32(np.array([g["w"]], np.float32), 8)
    qa = np.ones((1, 8), np.int8)
    y64, yb = oracle.linear(qa, np.array([[lin["s_a"]]], np.float32), qw, sw, np.array([lin["bias"]], np.float32), 8)
    assert oracle.group_partials(qa, qw, 8)[0, 0, 0] == lin["acc"]
    assert y64[0, 0] == lin["y"] and f"{int(yb[0, 0]):04X}" == lin["y_bf16_hex"]


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_ternary_matches_exact_rational_rule(seed):
    rng = np.random.default_rng(100 + seed)
    G = 64
    rows = []
    rows.append((rng.standard_normal(G) * 0.02).astype(np.float32))             # typical weights
    rows.append((rng.standard_normal(G) * 10.0 ** rng.uniform(-30, 30)).astype(np.float32))  # extreme magnitudes
    r = rng.integers(-3, 4, G).astype(np.float32) * np.float32(0.5)               # many exact ties
    r[0] = 3.0
    rows.append(r)
    o = (rng.standard_normal(G) * 0.02).astype(np.float32)
    o[5] = 4.0                                                                       # one outlier
    rows.append(o)
    w = np.stack(rows)
    codes, s = oracle.quantize_ternary_f32(w, G)
    for i in range(w.shape[0]):
        q_ref, s_ref = ternary_ref(w[i])
        assert float(s[i, 0]) == s_ref, i
        assert codes[i].tolist() == q_ref, i


def test_ternary_invariants():
    rng = np.random.default_rng(7)
    N, K, G = 24, 384, 128
    w = (rng.standard_normal((N, K)) * 0.02).astype(np.float32)
    codes, s = oracle.quantize_ternary_f32(w, G)
    assert codes.min() >= -1 and codes.max() <= 1
    # s is the group's mean |w| (fp64 sum, then fp32): within one fp32 rounding of numpy's
    m = np.abs(w.astype(np.float64)).reshape(N, K // G, G).mean(axis=2)
    assert np.all(np.abs(s - m) <= m * 2.0 ** -23)
    # sign symmetry, and scaling by a power of two moves only the scale
    c2, s2 = oracle.quantize_ternary_f32(-w, G)
    assert np.array_equal(c2, -codes) and np.array_equal(s2, s)
    c3, s3 = oracle.quantize_ternary_f32(w * np.float32(8.0), G)
    assert np.array_equal(c3, codes) and np.array_equal(s3, s * np.float32(8.0))
    # every code is the nearest level of w/s within [-1, 1]
    t = w.reshape(N, K // G, G) / s[:, :, None]
    assert np.all(np.abs(np.clip(t, -1.5, 1.5) - codes.reshape(N, K // G, G)) <= 0.5 + 1e-6)


def test_ternary_zero_and_constant_groups():
    w = np.zeros((2, 32), np.float32)
    w[1, :16] = -0.25
    w[1, 16:] = 3.0
    codes, s = oracle.quantize_ternary_f32(w, 16)
    assert np.all(codes[0] == 0) and np.all(s[0] == 0)
    assert s[1].tolist() == [0.25, 3.0]
    assert codes[1].tolist() == [-1] * 16 + [1] * 16


def test_ternary_pack_round_trip_and_layout():
    rng = np.random.default_rng(3)
    codes = rng.integers(-1, 2, (7, 160)).astype(np.int8)
    packed = oracle.pack_ternary(codes)
    assert packed.shape == (7, 40)
    assert np.array_equal(oracle.unpack_ternary(packed), codes)
    # every byte value a packed ternary row can hold (3^4 = 81 of them) round-trips, and a byte
    # holds elements 2j, 2j+1, 8+2j, 9+2j of its 16-element word
    vals = np.array([[a, b, c, d] for a in range(3) for b in range(3) for c in range(3) for d in range(3)])
    for j in range(4):
        row = np.zeros((len(vals), 16), np.int8)
        row[:, 2 * j], row[:, 2 * j + 1], row[:, 8 + 2 * j], row[:, 9 + 2 * j] = (vals - 1).T
        p = oracle.pack_ternary(row)
        expect = vals[:, 0] | vals[:, 1] << 2 | vals[:, 2] << 4 | vals[:, 3] << 6
        assert np.array_equal(p[:, j], expect.astype(np.uint8))
        assert np.all(np.delete(p, j, axis=1) == 0x55)  # the other bytes: all codes 0 (q+1 = 1)
        assert np.array_equal(oracle.unpack_ternary(p), row)


def test_w158a4_linear_matches_numpy_fp64_dequant_matmul():
    rng = np.random.default_rng(12)
    M, N, K, G = 9, 40, 256, 128
    x = wl.f32_to_bf16_bits(rng.standard_normal((M, K)).astype(np.float32))
    qa, sa = oracle.quantize_bf16(x, G)
    qw, sw = oracle.quantize_ternary_f32((rng.standard_normal((N, K)) * 0.02).astype(np.float32), G)
    bias = (rng.standard_normal(N) * 0.01).astype(np.float32)
    y64, _ = oracle.linear(qa, sa, qw, sw, bias, G)
    a = (qa.reshape(M, K // G, G) * sa[:, :, None].astype(np.float64)).reshape(M, K)
    w = (qw.reshape(N, K // G, G) * sw[:, :, None].astype(np.float64)).reshape(N, K)
    ref = a @ w.T + bias.astype(np.float64)
    assert np.allclose(y64, ref, rtol=1e-12, atol=1e-15)
