"""The quantiser's division shortcut, checked over every pair of positive finite bf16 values.

The rule needs q = clamp(rint(fl32(x / s)), -8, 7) with s = fl32(amax / 7).  The activation
quantiser avoids a division per element: with r = RN(1/s) it rounds y = RN(x * r) instead, and
falls back to the IEEE quotient when y lies within 2^-19 of a half-integer (and for subnormal
s).  The argument: |y - x/s| < 2^-20 and |fl32(x/s) - x/s| <= 2^-22 while |x/s| <= 7 (1 + 2^-23),
so outside that band both round to the same integer.

This test checks the argument itself, not the compiled kernel (whose outputs the GPU tests
compare with the oracle): over every positive finite bf16 amax and every bf16 x with
|x| <= amax (both signs, about 1.07e9 pairs), the shortcut with its fallback must give the
exact rule's code.  The compiler may contract x * r into the add that rounds it or into the
subtraction that measures the distance to the rounded value, so all four contractions are
checked; in each the exact product x * r is formed in fp64 (24 x 24 significant bits fit).
"""
import numpy as np
import pytest

MAGIC = np.float32(1.5 * 2 ** 23 + 8)  # the kernel's rounding constant (its low nibble is q + 8)
GUARD = np.float32(0.5 - 2.0 ** -19)


@pytest.mark.slow
def test_reciprocal_shortcut_matches_the_exact_quotient_for_every_bf16_pair():
    pos = (np.arange(1, 0x7F80, dtype=np.uint32) << 16).view(np.float32)  # every positive finite bf16
    mismatches = {"mul/mul": 0, "fma-round": 0, "fma-distance": 0, "fma-both": 0}
    pairs = fallbacks = 0
    for i, amax in enumerate(pos):
        s = np.float32(amax / np.float32(7.0))
        if not (s >= np.float32(2.0 ** -126)):
            continue  # subnormal scale: the kernel divides exactly
        x = np.concatenate([pos[: i + 1], -pos[: i + 1], np.zeros(1, np.float32)])
        exact = np.clip(np.rint(x / s), -8, 7)  # IEEE single division, ties to even
        r = np.float32(np.float32(1.0) / s)
        prod = x.astype(np.float64) * np.float64(r)  # exact
        y = (x * r).astype(np.float32)
        y64 = y.astype(np.float64)
        for variant in mismatches:
            fused_round = variant in ("fma-round", "fma-both")
            fused_dist = variant in ("fma-distance", "fma-both")
            t = np.rint(prod) if fused_round else np.rint(y64)  # t - MAGIC, an integer
            d = ((prod if fused_dist else y64) - t).astype(np.float32)
            fast = np.abs(d) <= GUARD
            q = np.where(fast, np.clip(t, -8, 7), exact)
            mismatches[variant] += int(np.count_nonzero(q != exact))
            if variant == "mul/mul":
                fallbacks += int(np.count_nonzero(~fast))
        pairs += x.size
    assert pairs > 1_000_000_000
    assert mismatches == {k: 0 for k in mismatches}, mismatches
    assert fallbacks < pairs // 1000  # the exact division stays rare


def test_tiled_kernel_tie_test_covers_the_band():
    """The TMA-staged quantiser flags a near-tie by fma(d, d, -c) >= 0 with d = y - rint(y), whose
    sign is that of the exact d^2 - c.  Every element of the band above (|d| > 1/2 - 2^-19) must
    be flagged, so c must lie below (1/2 - 2^-19)^2; and c close to 1/4 keeps the extra
    fallbacks rare.  The constant is read from the kernel source."""
    import os
    import re
    from fractions import Fraction
    src = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                            "paper_2609_33601_gb300", "csrc", "quantize.cu")).read()
    lit = re.search(r"constexpr float kTieSq = (0x[0-9a-fA-F.]+p-?\d+)f;", src).group(1)
    c = Fraction(float.fromhex(lit))
    assert float(np.float32(float(c))) == float(c), "the constant is an fp32 value"
    band = Fraction(1, 2) - Fraction(1, 2 ** 19)
    assert c < band * band
    assert c > Fraction(1, 4) - Fraction(1, 2 ** 18)
