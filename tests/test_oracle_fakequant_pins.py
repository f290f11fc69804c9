"""Pins for the oracle's training-side fake quantisation and straight-through estimator.

The paper trains the student's quantised blocks by gradient descent (Algorithm 1, Stage 1) and
names the straight-through estimator as the gradient rule of 4-bit activations (Sec. 3, "Why
QAT fails"), but prints no formula.  The reading: xhat = q*s with the deployed quantiser's code
q and the group scale s (amax/7, or a given scale), formed exactly and rounded once; the
backward passes the gradient where the unclamped code lies in [-8, 7].  Pinned by:

* hand-worked examples (tests/golden/fake_quant_example.json), one of them built so that
  rounding to fp32 before bf16 gives a different answer than the single rounding;
* a brute-force evaluation on tiny shapes in a different implementation (numpy IEEE fp32
  division, exact rationals, a bf16 rounding written here from the format's definition);
* invariants: with the amax scale no code is clamped, |x - xhat| <= s/2 (+ the output rounding),
  xhat requantises to the same codes, sign symmetry;
* consistency with the deployed integer path: the fp64 product of the fake-quantised operands
  reproduces the W4A4 layer's exact result within fp32 rounding of the operands.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2609_33601_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden():
    with open(os.path.join(GOLDEN, "fake_quant_example.json")) as f:
        return json.load(f)


def bf16_bits(vals):
    """Exactly representable values -> bf16 bits (top half of the fp32 pattern)."""
    return (np.asarray(vals, np.float32).view(np.uint32) >> 16).astype(np.uint16)


def bits_to_f32(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32)


def bf16_rne_fraction(v: Fraction) -> int:
    """Exact rational -> bf16 bits, nearest even: 8 significant bits, normal exponents down to
    2^-126, subnormal quantum 2^-133 (finite results only)."""
    neg = v < 0
    a = -v if neg else v
    if a == 0:
        return 0x8000 if neg else 0
    e = 0
    while a >= Fraction(2) ** (e + 1):
        e += 1
    while a < Fraction(2) ** e:
        e -= 1
    q_exp = max(e - 7, -133)
    t = a / Fraction(2) ** q_exp
    n = t.numerator // t.denominator
    rem = t - n
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and n % 2 == 1):
        n += 1
    r = np.float32(float(Fraction(n) * Fraction(2) ** q_exp))
    b = int(np.array([r], np.float32).view(np.uint32)[0] >> 16)
    return b | (0x8000 if neg else 0)


def brute_fake_quant(xb, G, s_given=None):
    """Element-by-element restatement: numpy fp32 division (IEEE), np.rint (half to even),
    exact rational product, bf16 rounding above."""
    M, K = xb.shape
    x = bits_to_f32(xb)
    xhat = np.zeros((M, K), np.uint16)
    mask = np.zeros((M, K), np.uint8)
    for m in range(M):
        for g in range(K // G):
            seg = x[m, g * G:(g + 1) * G]
            if s_given is None:
                amax = np.float32(np.max(np.abs(seg)))
                if amax == 0:
                    mask[m, g * G:(g + 1) * G] = 1
                    continue
                s = np.float32(amax / np.float32(7.0))
            else:
                s = np.float32(s_given[m, g])
            for k in range(G):
                r = float(np.rint(np.float32(seg[k] / s)))
                mask[m, g * G + k] = 1 if -8 <= r <= 7 else 0
                q = min(max(r, -8.0), 7.0)
                xhat[m, g * G + k] = bf16_rne_fraction(Fraction(q) * Fraction(float(s)))
    return xhat, mask


# ------------------------------------------------------------- hand-worked --

def test_hand_worked_amax_rule():
    g = _golden()
    xhat, mask, s = oracle.fake_quant_bf16(bf16_bits([g["x"]]), 8)
    assert s[0, 0] == np.float32(g["amax_rule"]["scale"])
    assert bits_to_f32(xhat[0]).tolist() == g["amax_rule"]["xhat"]
    assert mask[0].tolist() == g["amax_rule"]["mask"]


def test_hand_worked_given_scale_clamps_and_masks():
    g = _golden()
    s_in = np.array([[g["given_scale"]["scale"]]], np.float32)
    xhat, mask, s = oracle.fake_quant_bf16(bf16_bits([g["x"]]), 8, s_in)
    assert s[0, 0] == s_in[0, 0]
    assert bits_to_f32(xhat[0]).tolist() == g["given_scale"]["xhat"]
    assert mask[0].tolist() == g["given_scale"]["mask"]
    what, mask32, _ = oracle.fake_quant_f32(np.array([g["x"]], np.float32), 8, s_in)
    assert what[0].tolist() == g["given_scale"]["xhat"] and mask32[0].tolist() == g["given_scale"]["mask"]


def test_hand_worked_ste_backward():
    g = _golden()
    mask = np.array([g["given_scale"]["mask"]], np.uint8)
    out = oracle.ste_backward_bf16(bf16_bits([g["ste_backward"]["grad"]]), mask)
    assert out[0].tolist() == bf16_bits(g["ste_backward"]["grad_x"]).tolist()
    # masked entries are +0, never -0 (the gradients there are positive and negative)
    assert (out[mask == 0] == 0).all()


def test_single_rounding_of_the_exact_product():
    g = _golden()["single_rounding"]
    s = np.float32(g["scale_numerator"] * 2.0 ** g["scale_exp2"])
    assert float(s) == g["scale_numerator"] * 2.0 ** g["scale_exp2"]  # an fp32 value
    x = np.zeros((1, 64), np.float32)
    x[0, :2] = g["x"]
    s_in = np.array([[s]], np.float32)
    xhat, mask, _ = oracle.fake_quant_bf16(bf16_bits(x), 64, s_in)
    assert [f"{v:04X}" for v in xhat[0, :2]] == g["xhat_bf16_hex"]
    assert mask.all()
    what, _, _ = oracle.fake_quant_f32(x, 64, s_in)
    assert [f"{v:08X}" for v in what[0, :2].view(np.uint32)] == g["what_f32_hex"]
    # the independent rounding agrees with the hand derivation
    assert bf16_rne_fraction(7 * Fraction(float(s))) == int(g["xhat_bf16_hex"][0], 16)


# -------------------------------------------------------------- brute force --

@pytest.mark.parametrize("G", [8, 16])
def test_brute_force_tiny(G):
    rng = np.random.default_rng(11)
    xb = bf16_bits(rng.standard_normal((3, 32)).astype(np.float32) * np.float32(3.0))
    xb[1, :G] = 0  # a group whose amax is 0
    for s_in in (None, (rng.uniform(0.05, 0.6, (3, 32 // G))).astype(np.float32)):
        xhat, mask, _ = oracle.fake_quant_bf16(xb, G, s_in)
        bx, bm = brute_fake_quant(xb, G, s_in)
        assert (xhat == bx).all() and (mask == bm).all()
    assert not bm.all()  # the small given scales do clamp somewhere
    assert (xhat != 0x8000).all()  # a zero code dequantises to +0, also for negative x


# --------------------------------------------------------------- invariants --

@pytest.mark.parametrize("G", [64, 128, 256])
def test_invariants_on_the_tiny_workload(G):
    w = wl.make("tiny", seed=3)
    xb = w.x_bits
    xhat, mask, s = oracle.fake_quant_bf16(xb, G)
    assert mask.all()  # the amax scale never reaches the clamp
    codes, s_dep = oracle.quantize_bf16(xb, G)
    assert (s.view(np.uint32) == s_dep.view(np.uint32)).all()  # the deployed quantiser's scales
    x = bits_to_f32(xb).astype(np.float64)
    xh = bits_to_f32(xhat).astype(np.float64)
    srep = np.repeat(s.astype(np.float64), G, axis=1)
    ulp_half = np.abs(xh) * 2.0 ** -8  # half a bf16 ulp is at most 2^-8 |v|
    assert (np.abs(x - xh) <= srep / 2 + ulp_half).all()
    # requantising xhat gives the same codes
    codes2, _ = oracle.quantize_bf16(xhat, G)
    assert (codes2 == codes).all()
    # sign symmetry
    xhat_n, mask_n, _ = oracle.fake_quant_bf16(xb ^ np.uint16(0x8000), G)
    nz = xhat != 0
    assert (xhat_n[nz] == (xhat[nz] ^ np.uint16(0x8000))).all() and (mask_n == mask).all()
    # the STE backward with an all-ones mask is the identity
    grad = bf16_bits(np.random.default_rng(5).standard_normal(xb.shape).astype(np.float32))
    assert (oracle.ste_backward_bf16(grad, mask) == grad).all()


def test_fake_quant_linear_reproduces_the_deployed_layer():
    """The fp64 product of fake-quantised fp32 operands against the W4A4 layer's exact result:
    each operand is q*s rounded once to fp32, so the two differ by at most 2^-23 relative per
    product term."""
    w = wl.make("tiny", seed=9)
    G = w.G
    x32 = bits_to_f32(w.x_bits)
    ah, amask, sa = oracle.fake_quant_f32(x32, G)
    wh, wmask, sw = oracle.fake_quant_f32(w.w, G)
    assert amask.all() and wmask.all()
    qa, sa_dep = oracle.quantize_bf16(w.x_bits, G)
    qw, sw_dep = oracle.quantize_f32(w.w, G)
    assert (sa == sa_dep).all() and (sw == sw_dep).all()
    y64, _ = oracle.linear(qa, sa_dep, qw, sw_dep, w.bias, G)
    yf = ah.astype(np.float64) @ wh.astype(np.float64).T + w.bias.astype(np.float64)
    bound = (np.abs(ah.astype(np.float64)) @ np.abs(wh.astype(np.float64)).T) * 2.0 ** -22 + 1e-300
    assert (np.abs(yf - y64) <= bound * 1.01 + 1e-12 * np.abs(y64)).all()
    # a dropped scale, sign or bias moves the result far outside that bound
    assert not (np.abs(-yf - y64) <= bound).all()


def test_fp32_weight_path_rounds_to_nearest():
    g = _golden()["fp32_rounding"]
    s = np.float32(g["scale_numerator"] * 2.0 ** g["scale_exp2"])
    w = np.zeros((1, 64), np.float32)
    w[0, :2] = g["x"]
    s_in = np.array([[s]], np.float32)
    what, mask, _ = oracle.fake_quant_f32(w, 64, s_in)
    assert [f"{v:08X}" for v in what[0, :2].view(np.uint32)] == g["what_f32_hex"] and mask.all()
    xhat, _, _ = oracle.fake_quant_bf16(bf16_bits(w), 64, s_in)
    assert [f"{v:04X}" for v in xhat[0, :2]] == g["xhat_bf16_hex"]
