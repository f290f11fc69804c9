"""Pins of the oracle's DiT-XL/2 neighbour operations fused with the activation quantiser.

The paper deploys DiT-XL/2 (a 0.6B DiT; Sec. 1's remark that small matrices and non-GEMM time
limit the speed-up, and the Appendix table "DiT-XL/2 experimental details" with W4A4 /
W1.58A4, group128).  In its blocks the linears are fed by the adaLN modulation
x (1 + scale) + shift and by the MLP's tanh GELU.  The readings (jq_oracle.c): the modulation in
IEEE single steps without contraction, rounded once to bf16; the GELU as a fixed sequence of IEEE
single operations (the logistic form, an own exponential), rounded to bf16; then the activation
rule.  Pinned here by
  * an exact-rational evaluation of the modulation with fp32 / bf16 roundings written from the
    formats (not a retyping of the oracle's expression in the same arithmetic), on random,
    extreme and tie-constructed inputs, and its identities (scale 0 and shift 0 give x; scale -1
    gives bf16(shift); scale 2^j - 1 with shift 0 scales x exactly);
  * a 50-digit mpmath evaluation of 0.5 h (1 + tanh(sqrt(2/pi)(h + 0.044715 h^3))): the fp32
    sequence within its error bound of it for every bf16 h in [-9, 16], its bf16 result equal to
    the exact value rounded once except within that bound of a rounding boundary, extreme
    magnitudes, and the GELU's invariants;
  * a hand-worked modulated group with its codes and scale;
  * planted mistakes (a fused multiply-add, a double rounding through bf16, the cancelling
    1 + tanh(u) form in fp64) that each fail one of these checks.
"""
import math
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2609_33601_gb300 import workloads as wl
from tests.test_oracle_pins import f32_rne


def bf16_rne_bits(fr: Fraction, neg_zero: bool = False) -> int:
    """Exact rational -> bf16 bits, nearest with ties to even (8-bit significand, subnormals
    below 2^-126 in steps of 2^-133); written from the format."""
    if fr == 0:
        return 0x8000 if neg_zero else 0
    sign = 0x8000 if fr < 0 else 0
    a = abs(fr)
    e = a.numerator.bit_length() - a.denominator.bit_length()
    if Fraction(2) ** e > a:
        e -= 1
    ulp_e = max(e, -126) - 7
    q = a / Fraction(2) ** ulp_e
    n = math.floor(q)
    rem = q - n
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and n % 2 == 1):
        n += 1
    v = float(Fraction(n) * Fraction(2) ** ulp_e)
    return sign | int(np.array([v], np.float32).view(np.uint32)[0] >> 16)


def modulate_ref(x: float, shift: float, scale: float) -> int:
    """bf16 bits of bf16(fl32(fl32(x * fl32(1 + scale)) + shift)), exact rationals."""
    one_plus = f32_rne(1 + Fraction(scale))
    t = f32_rne(Fraction(x) * Fraction(one_plus))
    z = f32_rne(Fraction(t) + Fraction(shift))
    neg_zero = z == 0 and math.copysign(1.0, z) < 0
    return bf16_rne_bits(Fraction(z), neg_zero)


def b2f(b):
    return wl.bf16_bits_to_f32(np.asarray(b, np.uint16))


def run_modulate(xb, sh, sc, T, G=64):
    return oracle.modulate_quantize_bf16(np.asarray(xb, np.uint16).reshape(1, -1) if np.ndim(xb) == 1 else xb,
                                         sh, sc, T, G)


def test_modulation_matches_exact_rational_evaluation():
    rng = np.random.default_rng(7)
    M, K, T = 6, 256, 2
    x = wl.f32_to_bf16_bits((rng.standard_normal((M, K)) * np.exp(rng.uniform(-20, 20, (M, K)))).astype(np.float32))
    sh = (rng.standard_normal((3, K)) * np.exp(rng.uniform(-20, 5, (3, K)))).astype(np.float32)
    sc = (rng.standard_normal((3, K)) * np.exp(rng.uniform(-30, 2, (3, K)))).astype(np.float32)
    sc[0, :8] = -1.0
    sc[1, :8] = 0.0
    sh[1, :8] = 0.0
    z, _, _ = oracle.modulate_quantize_bf16(x, sh, sc, T, 64)
    xf = b2f(x)
    for m in range(M):
        b = m // T
        for k in range(K):
            assert z[m, k] == modulate_ref(float(xf[m, k]), float(sh[b, k]), float(sc[b, k])), (m, k)


def test_modulation_identities():
    rng = np.random.default_rng(1)
    K = 128
    x = wl.f32_to_bf16_bits(rng.standard_normal((4, K)).astype(np.float32))
    zero = np.zeros((2, K), np.float32)
    z, codes, s = oracle.modulate_quantize_bf16(x, zero, zero, 2, 64)
    assert np.array_equal(z, x)  # x (1 + 0) + 0 = x exactly
    ref_codes, ref_s = oracle.quantize_bf16(x, 64)
    assert np.array_equal(codes, ref_codes) and np.array_equal(s, ref_s)
    sh = rng.standard_normal((2, K)).astype(np.float32)
    z, _, _ = oracle.modulate_quantize_bf16(x, sh, np.full((2, K), -1.0, np.float32), 2, 64)
    assert np.array_equal(z, wl.f32_to_bf16_bits(np.repeat(sh, 2, axis=0)))  # x * 0 + shift
    z, _, _ = oracle.modulate_quantize_bf16(x, zero, np.full((2, K), 7.0, np.float32), 2, 64)
    assert np.array_equal(b2f(z), b2f(x) * 8)  # a power of two scales exactly


def test_modulation_is_a_single_bf16_rounding_of_unfused_fp32_steps():
    # x = 1 + 2^-7 (bf16 exact), scale = 2^-8: x (1 + scale) = 1 + 3 * 2^-8 + 2^-15 exactly, which
    # fp32 holds; + shift = -2^-15 cancels the last term, so z = 1 + 3 * 2^-8, whose bf16 rounding
    # is a tie that goes to the even 1 + 2^-6 (0x3F82).  A fused multiply-add gives the same here,
    # so a second case makes the contraction visible: x = 1 + 2^-7, scale = 2^-23 + 2^-30 (fp32
    # exact): 1 + scale rounds to 1 + 2^-23, and the products differ by more than the shift's ulp.
    x = wl.f32_to_bf16_bits(np.array([1 + 2.0 ** -7], np.float32))
    z, _, _ = oracle.modulate_quantize_bf16(x.reshape(1, 1).repeat(64, 1), np.full((1, 64), -2.0 ** -15, np.float32),
                                            np.full((1, 64), 2.0 ** -8, np.float32), 1, 64)
    assert int(z[0, 0]) == 0x3F82
    # unfused steps vs a fused multiply-add on a case built so the two round differently
    xs, sc_, sh_ = 1.0 + 2.0 ** -7, 2.0 ** -22 + 2.0 ** -30, -(1.0 + 2.0 ** -7)
    one_plus = f32_rne(1 + Fraction(sc_))
    fused = bf16_rne_bits(Fraction(xs) * Fraction(one_plus) + Fraction(sh_))
    unfused = modulate_ref(xs, sh_, sc_)
    assert fused != unfused
    zz, _, _ = oracle.modulate_quantize_bf16(wl.f32_to_bf16_bits(np.full((1, 64), xs, np.float32)),
                                             np.full((1, 64), sh_, np.float32), np.full((1, 64), sc_, np.float32), 1, 64)
    assert int(zz[0, 0]) == unfused


def test_modulate_quantize_hand_worked_group():
    # x = [1, -1, 0.5, 2, 0, ...] (group of 8 repeated to 64), scale 1 (x2), shift 0.5 on the
    # first sample: z = 2x + 0.5 = [2.5, -1.5, 1.5, 4.5, 0.5, ...]; amax = 4.5, s = 4.5/7;
    # z / s = [3.888.., -2.333.., 2.333.., 7, 0.777..] -> codes [4, -2, 2, 7, 1].
    base = np.array([1, -1, 0.5, 2, 0, 1, -1, 0.5], np.float32)
    x = wl.f32_to_bf16_bits(np.tile(base, 8).reshape(1, 64))
    z, codes, s = oracle.modulate_quantize_bf16(x, np.full((1, 64), 0.5, np.float32), np.full((1, 64), 1.0, np.float32),
                                                1, 64)
    assert np.array_equal(b2f(z[0, :8]), np.array([2.5, -1.5, 1.5, 4.5, 0.5, 2.5, -1.5, 1.5], np.float32))
    assert s[0, 0] == np.float32(4.5) / np.float32(7)
    assert list(codes[0, :8]) == [4, -2, 2, 7, 1, 4, -2, 2]


def test_tokens_map_to_their_sample():
    rng = np.random.default_rng(3)
    M, K, T = 10, 128, 4  # samples 0, 1, 2 (the last one partial)
    x = wl.f32_to_bf16_bits(rng.standard_normal((M, K)).astype(np.float32))
    sh = rng.standard_normal((3, K)).astype(np.float32)
    sc = rng.standard_normal((3, K)).astype(np.float32)
    z, _, _ = oracle.modulate_quantize_bf16(x, sh, sc, T, 128)
    for m in range(M):
        zr, _, _ = oracle.modulate_quantize_bf16(x[m:m + 1], sh[m // T:m // T + 1], sc[m // T:m // T + 1], 1, 128)
        assert np.array_equal(z[m], zr[0])


# ------------------------------------------------------------------------ GELU ----

def gelu_mp(h: float):
    """The exact tanh GELU of h as a 60-digit mpmath value."""
    import mpmath
    mpmath.mp.dps = 60
    hm = mpmath.mpf(h)
    u = mpmath.sqrt(2 / mpmath.pi) * (hm + mpmath.mpf("0.044715") * hm ** 3)
    return hm / 2 * (1 + mpmath.tanh(u))


def mp_fraction(g) -> Fraction:
    import mpmath
    if g == 0:
        return Fraction(0)
    p, q = abs(mpmath.mpf(g)).man_exp  # mpmath's mantissa is unsigned
    return (-1 if g < 0 else 1) * Fraction(int(p)) * (Fraction(2) ** int(q))


def all_bf16_in(lo, hi):
    pos = np.arange(0, 0x7F80, dtype=np.uint16)
    vals = b2f(pos)
    keep = pos[(vals >= 0) & (vals <= hi)]
    neg = keep[1:] | np.uint16(0x8000)
    negv = b2f(neg)
    return np.concatenate([keep, neg[negv >= lo]])


# The fp32 evaluation's error against the exact GELU, relative, over h >= -9: at most
# 2^-24 (8 + 4 |u|) by the rounding analysis of its steps (the constants' representation, the
# cubic, the reduction r = x - n ln2 whose error grows with |n| ~ 2.9 |u|, the degree-8 Taylor
# polynomial, the logistic and the product), u = 0.8 (h + 0.045 h^3).
def gelu_bound(h: float) -> float:
    u = abs(0.7978845608 * (h + 0.044715 * h ** 3))
    return (8 + 4 * u) * 2.0 ** -24


@pytest.mark.slow
def test_gelu_fp32_is_within_its_bound_of_the_50_digit_value():
    hs = all_bf16_in(-9.0, 16.0)
    worst = 0.0
    for hb in hs:
        h = float(b2f(np.array([hb], np.uint16))[0])
        g = oracle.gelu_tanh_f32(h)
        ex = gelu_mp(h)
        if ex == 0:
            assert g == 0
            continue
        rel = abs(float(Fraction(g) - mp_fraction(ex)) / float(abs(mp_fraction(ex))))
        worst = max(worst, rel / gelu_bound(h))
        assert rel <= gelu_bound(h), (h, g, float(ex), rel / 2.0 ** -24)
    assert worst > 0.01  # the bound is not vacuous: the errors are of its order


@pytest.mark.slow
def test_gelu_bf16_equals_the_single_rounding_except_within_the_bound_of_a_midpoint():
    """bf16 of the fp32 GELU (the reading) against the exact GELU rounded once: they may differ
    only where the exact value lies within the fp32 error bound of a bf16 rounding boundary."""
    hs = all_bf16_in(-9.0, 16.0)
    z, _, _ = oracle.gelu_quantize_bf16(np.resize(hs, (len(hs) + 63) // 64 * 64).reshape(-1, 64), 64)
    z = z.reshape(-1)[: len(hs)]
    differ = 0
    for hb, zb in zip(hs, z):
        h = float(b2f(np.array([hb], np.uint16))[0])
        ex = mp_fraction(gelu_mp(h))
        single = bf16_rne_bits(ex, neg_zero=(ex == 0 and math.copysign(1.0, h) < 0))
        if int(zb) != single:
            differ += 1
            lo = bf16_rne_bits(ex * (1 - Fraction(gelu_bound(h))))
            hi = bf16_rne_bits(ex * (1 + Fraction(gelu_bound(h))))
            assert lo != hi, (h, hex(int(zb)), hex(single))  # a boundary lies within the bound
    # about one input in 300: mostly the bf16 subnormals with an odd quantum, where GELU(h) is
    # 0.5 h (a bf16 tie, which fp32 holds exactly and rounds to even) plus ~0.4 h^2
    assert differ <= len(hs) // 100


def test_gelu_extreme_and_special_values():
    # +-0 keep their sign; large h returns h; deep negative h gives a (signed) tiny value or zero
    for h, want in [(0.0, 0x0000), (-0.0, 0x8000), (8.0, None), (20.0, None), (1e6, None), (3e38, None)]:
        hb = int(wl.f32_to_bf16_bits(np.array([h], np.float32))[0])
        z, _, _ = oracle.gelu_quantize_bf16(np.full((1, 64), hb, np.uint16), 64)
        assert int(z[0, 0]) == (hb if want is None else want), h
    for h in (-9.5, -10.0, -12.0, -20.0, -100.0, -3e38):
        g = oracle.gelu_tanh_f32(h)
        assert g <= 0 and abs(g) < 2.0 ** -100
    # the sample used by the module docstring's remark: GELU(-10) is about -1.2e-37
    assert abs(oracle.gelu_tanh_f32(-10.0) / float(gelu_mp(-10.0)) - 1) < 2.0 ** -20


def test_gelu_invariants():
    hs = all_bf16_in(-16.0, 16.0)
    hb = np.resize(hs, (len(hs) + 63) // 64 * 64).reshape(-1, 64)
    z, codes, s = oracle.gelu_quantize_bf16(hb, 64)
    zf = b2f(z.reshape(-1)[: len(hs)])
    hf = b2f(hs)
    assert np.all(zf[hf <= 0] <= 0) and np.all(zf[hf >= 0] >= 0)
    assert np.all(zf[hf >= 8] == hf[hf >= 8])  # GELU(h) = h (1 - tiny) rounds to h for h >= 8
    pos = np.argsort(hf[hf >= 0])
    assert np.all(np.diff(zf[hf >= 0][pos]) >= 0)  # monotone on h >= 0
    ref_codes, ref_s = oracle.quantize_bf16(z, 64)
    assert np.array_equal(codes, ref_codes) and np.array_equal(s, ref_s)


def test_gelu_worked_values():
    # GELU(1) = 0.841192 (the tanh form), bf16 0x3F57 (0.83984375 / 0.84375: nearer 0.83984375)
    z, _, _ = oracle.gelu_quantize_bf16(wl.f32_to_bf16_bits(np.full((1, 64), 1.0, np.float32)), 64)
    assert int(z[0, 0]) == 0x3F57
    # GELU(-1) = -0.158808: bf16 0xBE23 (-0.1591796875; the neighbour -0.158203125 is farther)
    z, _, _ = oracle.gelu_quantize_bf16(wl.f32_to_bf16_bits(np.full((1, 64), -1.0, np.float32)), 64)
    assert int(z[0, 0]) == 0xBE23


def test_planted_cancelling_tanh_form_loses_the_value():
    # 0.5 h (1 + tanh(u)) evaluated as written (even in fp64) loses the value where 1 + tanh(u)
    # cancels: at h = -10 the GELU is about -1.2e-37, the written form gives 0; the oracle's
    # logistic form keeps it (checked against the 50-digit value above)
    h = -10.0
    u = math.sqrt(2 / math.pi) * (h + 0.044715 * h ** 3)
    assert 0.5 * h * (1 + math.tanh(u)) == 0.0
    assert oracle.gelu_tanh_f32(h) != 0.0
