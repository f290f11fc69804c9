"""The Stage-1 schedule of Theseus QAD (paper_2609_33601_gb300/theseus.py) against the paper's
own numbers: the widths of the 28-block DiT (Sec. 3) and every allocation of Table 1
(tests/golden/theseus_table1.json), plus the properties the rule must have at any size."""
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

from paper_2609_33601_gb300 import theseus

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "theseus_table1.json")


def gamma_of(text: str):
    return math.inf if text == "inf" else Fraction(text)


def table1():
    with open(GOLDEN) as f:
        return json.load(f)


def test_widths_of_the_28_block_dit():
    gd = table1()
    assert theseus.binary_merge_widths(gd["L"]) == tuple(gd["widths"])


@pytest.mark.parametrize("row", table1()["rows"], ids=lambda r: r["gamma"])
def test_table1_allocations(row):
    gd = table1()
    assert theseus.allocate(gd["T1"], gamma_of(row["gamma"]), len(gd["widths"])) == tuple(row["N"])


def test_the_033_row_is_one_third():
    # 0.33 itself would put 6710 steps at width 1, not the 6676 Table 1 prints
    assert theseus.allocate(10000, Fraction(33, 100), 6)[0] != 6676
    assert theseus.allocate(10000, 1 / 3, 6) == (6676, 2225, 742, 247, 82, 28)  # the float 1/3 agrees


def test_schedule_of_the_28_block_dit_at_gamma_2():
    sched = theseus.stage_one_schedule(28, 10000, 2)
    assert [e["width"] for e in sched] == [1, 2, 4, 8, 16, 28]
    assert [e["steps"] for e in sched] == [159, 317, 635, 1270, 2540, 5079]
    assert [w for _, w in sched[3]["segments"]] == [8, 8, 8, 4]
    assert [w for _, w in sched[4]["segments"]] == [16, 12]


@pytest.mark.parametrize("L", range(1, 70))
def test_segments_tile_every_level(L):
    levels = theseus.binary_merge_segments(L)
    for level in levels:
        b = 0
        for start, width in level:
            assert start == b and width >= 1
            b += width
        assert b == L
    assert levels[0] == [(i, 1) for i in range(L)] and levels[-1] == [(0, L)]
    # the widths are the powers of two below L, then L
    assert theseus.binary_merge_widths(L) == tuple([2 ** k for k in range(L.bit_length()) if 2 ** k < L] + [L])


def test_allocation_properties():
    rng = np.random.default_rng(4)
    for _ in range(300):
        T1 = int(rng.integers(0, 100000))
        levels = int(rng.integers(1, 9))
        g = Fraction(int(rng.integers(1, 400)), int(rng.integers(1, 400)))
        N = theseus.allocate(T1, g, levels)
        assert sum(N) == T1 and len(N) == levels
        w = [g ** k for k in range(levels)]
        for k in range(levels):
            quota = T1 * w[k] / sum(w)
            assert math.floor(quota) <= N[k] <= math.ceil(quota)  # each level within one step of its quota
        # gamma and 1/gamma give mirrored quotas, hence mirrored counts unless remainders tie
        quotas = [T1 * x / sum(w) for x in w]
        fracs = [q - math.floor(q) for q in quotas]
        if len(set(fracs)) == levels:
            assert theseus.allocate(T1, 1 / g, levels) == tuple(reversed(N))
    assert theseus.allocate(7, 0, 3) == (7, 0, 0) and theseus.allocate(7, math.inf, 3) == (0, 0, 7)
    assert theseus.allocate(0, 2, 4) == (0, 0, 0, 0)
    with pytest.raises(ValueError):
        theseus.allocate(10, -1, 3)
