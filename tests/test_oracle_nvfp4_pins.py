"""Pins for the NVFP4 oracle (the format of the paper's LLaDA-8B "NVFP4 W4A4" rows).

The paper names the format (Appendix table "ELF-B and LLaDA-8B experimental
details") and defines none of it, so the oracle follows the published NVFP4
format: E2M1 elements, one E4M3 scale per 16 consecutive reduction-axis
elements, one fp32 tensor scale.  Pins, none of which reuses the oracle's
arithmetic:

* a hand-worked example (tests/golden/nvfp4_example.json) that hits all seven
  E2M1 midpoints, an E4M3 scale that has to round, the packed bytes and one
  linear output;
* E2M1 and E4M3 reference roundings done by enumerating every finite value
  from the formats' bit fields (sign / exponent / mantissa) and taking the
  nearest in exact rational arithmetic, ties to the even mantissa; the oracle
  rounds by scaling and rint instead, so a wrong bias, quantum or tie rule
  shows up;
* an exact-rational evaluation of the whole block rule on random rows;
* invariants (sign symmetry, power-of-two scale invariance, the tensor-max
  element landing on +-6 with block scale 448, the half-gap error bound);
* zero and underflow cases;
* the linear layer against exact rationals and against a numpy fp64
  dequantise-then-matmul.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from test_oracle_pins import f32_rne

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------- formats ----

def e2m1_table():
    """(value, mantissa bit) of the 8 non-negative E2M1 values from the bit fields:
    exponent bias 1, 1 mantissa bit, exponent field 0 subnormal (m * 0.5)."""
    out = []
    for e in range(4):
        for m in range(2):
            v = Fraction(m, 2) if e == 0 else (1 + Fraction(m, 2)) * Fraction(2) ** (e - 1)
            out.append((v, m))
    return out


def e4m3_table():
    """(value, mantissa lsb) of the non-negative finite E4M3 values from the bit fields:
    exponent bias 7, 3 mantissa bits, exponent field 0 subnormal (m/8 * 2^-6); the code with
    all exponent and mantissa bits set is NaN and is left out."""
    out = []
    for e in range(16):
        for m in range(8):
            if e == 15 and m == 7:
                continue
            v = Fraction(m, 8) * Fraction(2) ** -6 if e == 0 else (1 + Fraction(m, 8)) * Fraction(2) ** (e - 7)
            out.append((v, m & 1))
    return out


E2M1 = e2m1_table()
E4M3 = e4m3_table()


def nearest_even(a: Fraction, table):
    """Nearest table value to a >= 0 (saturating at the largest), ties to mantissa lsb 0."""
    top = max(v for v, _ in table)
    if a >= top:
        return top
    best = min(table, key=lambda t: (abs(t[0] - a), t[1]))
    return best[0]


def nvfp4_block_ref(xs, g):
    """Exact-rational evaluation of one 16-element block: (2q list, block scale s_b)."""
    xs = [float(np.float32(v)) for v in xs]
    g = float(np.float32(g))
    if g == 0:
        return [0] * len(xs), 0.0
    amax = max(abs(v) for v in xs)
    six_g = f32_rne(6 * Fraction(g))
    s = nearest_even(Fraction(f32_rne(Fraction(amax) / Fraction(six_g))), E4M3)
    S = f32_rne(s * Fraction(g))
    if S == 0:
        return [0] * len(xs), float(s)
    out = []
    for v in xs:
        t = f32_rne(Fraction(v) / Fraction(S))
        q = nearest_even(abs(Fraction(t)), E2M1)
        out.append(int(2 * q) * (-1 if t < 0 else 1))
    return out, float(s)


def bf16_of(fr: Fraction) -> int:
    """Exact rational -> bf16 bits, nearest even (8 significant bits), for normal values."""
    sign = 0x8000 if fr < 0 else 0
    a = abs(fr)
    if a == 0:
        return sign
    e = a.numerator.bit_length() - a.denominator.bit_length()
    if Fraction(2) ** e > a:
        e -= 1
    q = a / Fraction(2) ** (e - 7)
    n = int(q)
    rem = q - n
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and n % 2 == 1):
        n += 1
    if n == 256:
        n, e = 128, e + 1
    return sign | ((e + 127) << 7) | (n - 128)


def load_golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


# ------------------------------------------------------------------ tests ----

def test_format_tables_match_published_extremes():
    """Facts of the formats: E2M1 holds {0, .5, 1, 1.5, 2, 3, 4, 6}; E4M3 tops out at 448,
    its smallest subnormal is 2^-9, its smallest normal 2^-6, and it has 126 positive finite
    values."""
    assert [float(v) for v, _ in E2M1] == [0, 0.5, 1, 1.5, 2, 3, 4, 6]
    vals = sorted(v for v, _ in E4M3)
    assert vals[-1] == 448 and vals[1] == Fraction(1, 512) and len(vals) == 127
    assert Fraction(1, 64) in vals and Fraction(7, 512) in vals and Fraction(480) not in vals


def test_nvfp4_worked_example():
    gd = load_golden("nvfp4_example.json")
    x = np.array([gd["x"]], np.float32)
    q2, s = oracle.quantize_nvfp4(x, gd["g"])
    assert s[0].tolist() == gd["block_scales"]
    assert q2[0].tolist() == gd["codes2"]
    packed = oracle.pack_nvfp4(q2)
    assert [f"{b:02X}" for b in packed[0]] == gd["packed_hex"]
    assert np.array_equal(oracle.unpack_nvfp4(packed), q2)
    lin = gd["linear"]
    qw2 = np.array([lin["qw2"]], np.int8)
    sw = np.array([lin["s_w"]], np.float32)
    y64, yb = oracle.linear_nvfp4(q2, s, gd["g"], qw2, sw, lin["g_w"], np.array([lin["bias"]], np.float32))
    assert y64[0, 0] == lin["y"]
    assert f"{int(yb[0, 0]):04X}" == lin["y_bf16_hex"]


def test_e2m1_rounding_sweep_at_unit_scale():
    """g = 1 and a block maximum of 6 make s_b = 1 and S_b = 1, so the codes are the E2M1
    rounding of x itself: sweep x over a 1/64 grid of [-6, 6] (all midpoints included)."""
    grid = np.arange(-6 * 64, 6 * 64 + 1) / 64.0
    vals = grid[np.abs(grid) < 6]
    pad = (-len(vals)) % 15
    vals = np.concatenate([vals, np.zeros(pad)]).reshape(-1, 15)
    x = np.concatenate([np.full((vals.shape[0], 1), 6.0), vals], axis=1).astype(np.float32)
    q2, s = oracle.quantize_nvfp4(x, 1.0)
    assert np.all(s == 1.0)
    for r in range(x.shape[0]):
        for k in range(16):
            v = Fraction(float(x[r, k]))
            ref = int(2 * nearest_even(abs(v), E2M1)) * (-1 if v < 0 else 1)
            assert q2[r, k] == ref, (float(v), q2[r, k], ref)


def test_e4m3_scale_rounding_sweep():
    """g = 1: s_b = e4m3(fl32(amax / 6)).  With amax = 6 v for v with few significant bits,
    amax / 6 = v exactly, so s_b must be the E4M3 rounding of v: sweep every E4M3 value, every
    midpoint between neighbours and points just beside them, plus values past 448."""
    vals = sorted(v for v, _ in E4M3)
    probes = []
    for lo, hi in zip(vals, vals[1:]):
        mid = (lo + hi) / 2
        eps = (hi - lo) / 64
        probes += [lo, mid, mid - eps, mid + eps]
    probes += [Fraction(448), Fraction(456), Fraction(464), Fraction(470), Fraction(1000),
               Fraction(1, 1024), Fraction(3, 2048)]
    probes = [p for p in probes if p > 0]
    x = np.zeros((len(probes), 16), np.float32)
    for i, p in enumerate(probes):
        assert Fraction(float(np.float32(float(6 * p)))) == 6 * p  # exact in fp32
        x[i, 0] = float(6 * p)
    _, s = oracle.quantize_nvfp4(x, 1.0)
    for i, p in enumerate(probes):
        assert Fraction(float(s[i, 0])) == nearest_even(p, E4M3), (float(p), float(s[i, 0]))


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_nvfp4_matches_exact_rational_rule(seed):
    rng = np.random.default_rng(seed)
    rows, K = 24, 64
    kind = seed % 4
    if kind == 0:
        x = rng.standard_normal((rows, K))
    elif kind == 1:  # heavy-tailed, with per-row outliers
        x = rng.standard_t(2, (rows, K)) * rng.uniform(0.01, 10, (rows, 1))
    elif kind == 2:  # tiny magnitudes: scales in the E4M3 subnormal range
        x = rng.standard_normal((rows, K)) * 1e-4
    else:  # coarse dyadic values: many exact E2M1 ties
        x = rng.integers(-48, 49, (rows, K)) / 8.0
    x = x.astype(np.float32)
    g = oracle.nvfp4_tensor_scale(x) if seed < 2 else float(np.float32(rng.uniform(0.001, 0.05)))
    q2, s = oracle.quantize_nvfp4(x, g)
    for r in range(rows):
        for b in range(K // 16):
            ref_q, ref_s = nvfp4_block_ref(x[r, b * 16:(b + 1) * 16], g)
            assert float(s[r, b]) == ref_s
            assert q2[r, b * 16:(b + 1) * 16].tolist() == ref_q


def test_tensor_scale_and_tensor_max_element():
    """g = fl32(amax / 2688); the block holding the tensor's largest magnitude gets the
    largest E4M3 scale, 448, and that element quantises to +-6."""
    rng = np.random.default_rng(11)
    for _ in range(20):
        w = (rng.standard_normal((8, 64)) * rng.uniform(1e-3, 1e3)).astype(np.float32)
        g = oracle.nvfp4_tensor_scale(w)
        amax = float(np.abs(w).max())
        assert g == f32_rne(Fraction(amax) / 2688)
        q2, s = oracle.quantize_nvfp4(w, g)
        r, k = np.unravel_index(np.argmax(np.abs(w)), w.shape)
        assert s[r, k // 16] == 448.0
        assert abs(int(q2[r, k])) == 12 and np.sign(q2[r, k]) == np.sign(w[r, k])
        assert s.max() <= 448.0


def test_nvfp4_invariants():
    rng = np.random.default_rng(12)
    x = (rng.standard_normal((32, 128)) * rng.uniform(0.1, 5, (32, 1))).astype(np.float32)
    g = oracle.nvfp4_tensor_scale(x)
    q2, s = oracle.quantize_nvfp4(x, g)
    # sign symmetry
    qn, sn = oracle.quantize_nvfp4(-x, g)
    assert np.array_equal(qn, -q2) and np.array_equal(sn, s)
    # scaling x and g by a power of two changes nothing
    q4, s4 = oracle.quantize_nvfp4(x * np.float32(4), g * 4)
    assert np.array_equal(q4, q2) and np.array_equal(s4, s)
    # codes are monotone in x within a block
    for r in range(4):
        blk = x[r, :16]
        order = np.argsort(blk, kind="stable")
        assert np.all(np.diff(q2[r, :16][order].astype(int)) >= 0)
    # error bound: |q - x/S| <= half the E2M1 gap around x/S (0.25 below 2, 0.5 below 4, 1 above)
    S = (s.astype(np.float64) * np.float32(g)).astype(np.float32).repeat(16, axis=1)
    t = np.abs(x.astype(np.float64) / S.astype(np.float64))
    err = np.abs(np.abs(q2.astype(np.float64)) / 2 - t)
    half_gap = np.where(t < 2, 0.25, np.where(t < 4, 0.5, 1.0))
    assert np.all(err <= half_gap + 1e-6)


def test_nvfp4_zero_and_underflow_cases():
    rng = np.random.default_rng(13)
    x = rng.standard_normal((3, 32)).astype(np.float32)
    q2, s = oracle.quantize_nvfp4(x, 0.0)  # no tensor scale: everything is zero
    assert not q2.any() and not s.any()
    x[1, 16:] = 0.0  # an all-zero block
    q2, s = oracle.quantize_nvfp4(x, 0.01)
    assert s[1, 1] == 0.0 and not q2[1, 16:].any()
    # a block whose amax / (6 g) is below half the smallest E4M3 subnormal: s_b = 0, codes 0
    y = np.zeros((1, 16), np.float32)
    y[0, 0] = 6.0 * 2.0 ** -11
    q2, s = oracle.quantize_nvfp4(y, 1.0)
    assert s[0, 0] == 0.0 and not q2.any()


def test_nvfp4_pack_encoding_and_round_trip():
    """The 4-bit E2M1 encoding decoded from its bit fields (bit 3 sign, bits 1-2 exponent,
    bit 0 mantissa) matches unpack; pack(unpack(b)) == b for every byte except the negative
    zero nibble 8, which packs back as 0."""
    allb = np.arange(256, dtype=np.uint8).reshape(1, 256)
    codes = oracle.unpack_nvfp4(allb)
    for b in range(256):
        for half, nib in enumerate((b & 15, b >> 4)):
            e, m = (nib >> 1) & 3, nib & 1
            mag = Fraction(m, 2) if e == 0 else (1 + Fraction(m, 2)) * Fraction(2) ** (e - 1)
            val = -mag if nib & 8 else mag
            assert codes[0, 2 * b + half] == 2 * val
    back = oracle.pack_nvfp4(codes)[0]
    fix = lambda n: 0 if n == 8 else n
    assert back.tolist() == [fix(b & 15) | (fix(b >> 4) << 4) for b in range(256)]


def test_linear_nvfp4_matches_exact_rationals():
    rng = np.random.default_rng(14)
    M, N, K = 5, 7, 64
    xa = rng.standard_normal((M, K)).astype(np.float32)
    xw = (rng.standard_normal((N, K)) * 0.05).astype(np.float32)
    ga, gw = oracle.nvfp4_tensor_scale(xa), oracle.nvfp4_tensor_scale(xw)
    qa2, sa = oracle.quantize_nvfp4(xa, ga)
    qw2, sw = oracle.quantize_nvfp4(xw, gw)
    bias = rng.standard_normal(N).astype(np.float32)
    y64, yb = oracle.linear_nvfp4(qa2, sa, ga, qw2, sw, gw, bias)
    for m in range(M):
        for n in range(N):
            y, mag = Fraction(0), Fraction(0)
            gg = Fraction(float(np.float32(ga))) * Fraction(float(np.float32(gw)))
            for b in range(K // 16):
                acc = sum(Fraction(int(qa2[m, k]), 2) * Fraction(int(qw2[n, k]), 2)
                          for k in range(b * 16, (b + 1) * 16))
                term = acc * Fraction(float(sa[m, b])) * Fraction(float(sw[n, b])) * gg
                y, mag = y + term, mag + abs(term)
            y += Fraction(float(bias[n]))
            mag += abs(Fraction(float(bias[n])))
            # fp64 summation of K/16 + 1 terms: error below (K/16 + 4) 2^-53 of their magnitude sum
            assert abs(Fraction(y64[m, n]) - y) <= mag * Fraction(K // 16 + 4, 2 ** 53)
            if abs(Fraction(y64[m, n]) - y) * 2 ** 20 < abs(y):  # far from any bf16 midpoint
                assert int(yb[m, n]) == bf16_of(y)


def test_linear_nvfp4_matches_numpy_dequant_matmul():
    rng = np.random.default_rng(15)
    M, N, K = 19, 23, 256
    qa2 = rng.choice([-12, -8, -6, -4, -3, -2, -1, 0, 1, 2, 3, 4, 6, 8, 12], (M, K)).astype(np.int8)
    qw2 = rng.choice([-12, -8, -6, -4, -3, -2, -1, 0, 1, 2, 3, 4, 6, 8, 12], (N, K)).astype(np.int8)
    e4m3_vals = np.array([float(v) for v, _ in E4M3], np.float32)
    sa = rng.choice(e4m3_vals, (M, K // 16))
    sw = rng.choice(e4m3_vals, (N, K // 16))
    ga, gw = float(np.float32(0.013)), float(np.float32(0.0007))
    bias = rng.standard_normal(N).astype(np.float32)
    y64, _ = oracle.linear_nvfp4(qa2, sa, ga, qw2, sw, gw, bias)
    A = qa2.astype(np.float64) / 2 * np.repeat(sa.astype(np.float64), 16, axis=1)
    B = qw2.astype(np.float64) / 2 * np.repeat(sw.astype(np.float64), 16, axis=1)
    ref = (A @ B.T) * np.float64(np.float32(ga)) * np.float64(np.float32(gw)) + bias.astype(np.float64)
    np.testing.assert_allclose(y64, ref, rtol=1e-11, atol=1e-12)
    # unit scales: the integer matmul of the doubled codes, divided by 4
    y1, _ = oracle.linear_nvfp4(qa2, np.ones_like(sa), 1.0, qw2, np.ones_like(sw), 1.0, None)
    assert np.array_equal(y1 * 4, (qa2.astype(np.int64) @ qw2.astype(np.int64).T).astype(np.float64))
