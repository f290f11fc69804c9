"""Shared helpers for the parity tests: oracle references and the bf16 tolerance rule."""
from __future__ import annotations

import json
import os

import numpy as np

import oracle
from paper_2609_33601_gb300 import workloads as wl


def ulp_bf16(v: np.ndarray) -> np.ndarray:
    """Spacing of bf16 values at |v| (8 significant bits; subnormal quantum 2^-133)."""
    a = np.abs(np.asarray(v, np.float64))
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    e = np.maximum(e, -126.0)
    return np.where(a >= 2.0 ** -126, np.exp2(e - 7.0), 2.0 ** -133)


def tolerance(y64: np.ndarray, acc: np.ndarray, s_a: np.ndarray, s_w_rows: np.ndarray,
              bias: np.ndarray | None) -> np.ndarray:
    """|y_gpu - y64| <= ulp_bf16(y64) + (K/G + 2) * 2^-24 * (sum_g |acc * s_a * s_w| + |bias|).

    The first term is the 1-ulp bf16 target; the second is the standard bound for summing the
    K/G group terms (plus bias) in fp32, which matters only under cancellation.
    acc: int32 [M, N, K/G]; s_a: [M, K/G]; s_w_rows: [N, K/G] (per output channel)."""
    ng = acc.shape[2]
    mag = np.einsum("mng,mg,ng->mn", np.abs(acc.astype(np.float64)), np.abs(s_a.astype(np.float64)),
                    np.abs(s_w_rows.astype(np.float64)))
    if bias is not None:
        mag = mag + np.abs(bias.astype(np.float64))[None, :]
    return ulp_bf16(y64) + (ng + 2) * 2.0 ** -24 * mag


def check_linear(y_gpu_bits: np.ndarray, y64: np.ndarray, acc, s_a, s_w_rows, bias, label=""):
    """Asserts the tolerance rule element by element; returns (max ulp error, #needing term 2)."""
    yg = wl.bf16_bits_to_f32(y_gpu_bits).astype(np.float64)
    err = np.abs(yg - y64)
    tol = tolerance(y64, acc, s_a, s_w_rows, bias)
    bad = err > tol
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{label}: {bad.sum()} elements out of tolerance, e.g. "
                             + "; ".join(f"[{m},{n}] gpu={yg[m, n]!r} ref={y64[m, n]!r} tol={tol[m, n]:.3g}"
                                         for m, n in idx))
    ulp = ulp_bf16(y64)
    worst, beyond = float((err / ulp).max()) if err.size else 0.0, int((err > ulp).sum())
    report_escape(label or "check_linear", beyond, err.size, worst, enforce=False)
    return worst, beyond


class Reference:
    """Oracle-side quantities for one (activations, weights, bias, G) problem."""

    def __init__(self, x_bits: np.ndarray, w: np.ndarray, bias, G: int):
        self.G = G
        self.qa, self.s_a = oracle.quantize_bf16(x_bits, G)
        self.qw, self.s_w_rows = oracle.quantize_f32(w, G)
        self.bias = bias
        self.packed_a = oracle.pack(self.qa)
        self.packed_w = oracle.pack(self.qw)

    @property
    def s_w_groupmajor(self) -> np.ndarray:
        return np.ascontiguousarray(self.s_w_rows.T)

    def linear(self, rows=None):
        qa = self.qa if rows is None else self.qa[rows]
        sa = self.s_a if rows is None else self.s_a[rows]
        return oracle.linear(qa, sa, self.qw, self.s_w_rows, self.bias, self.G)

    def partials(self, rows=None):
        qa = self.qa if rows is None else self.qa[rows]
        return oracle.group_partials(qa, self.qw, self.G)


def report_escape(label: str, beyond_ulp: int, elements: int, worst_ulp: float, enforce: bool = True) -> None:
    """Records how many outputs needed the fp32-summation term of the tolerance (those more than
    one bf16 ulp from the oracle).  With JQ_PARITY_REPORT set, one JSON line per check is
    appended to that file; the count is also asserted to stay rare (the term is there for
    cancellation near zero, roughly one output in 10^4 on random data, not for a systematic
    error; enforce=False only records it)."""
    path = os.environ.get("JQ_PARITY_REPORT")
    if path:
        with open(path, "a") as f:
            f.write(json.dumps({"check": label, "elements": elements, "beyond_1_ulp": beyond_ulp,
                                "max_error_ulp": worst_ulp}) + "\n")
    assert not enforce or beyond_ulp <= max(16, elements // 1000), (
        f"{label}: {beyond_ulp} of {elements} outputs needed the fp32 summation term")


def check_linear_full(y_gpu_bits: np.ndarray, qa: np.ndarray, s_a: np.ndarray, qw: np.ndarray,
                      s_w_rows: np.ndarray, bias, G: int, label: str = ""):
    """Every output of a full-size problem against the oracle, by the same rule as check_linear.

    The oracle's fp64 result covers all M x N outputs; the second term of the tolerance needs
    the per-group partials, which would be M x N x K/G integers at full size, so they are formed
    only for the outputs more than one bf16 ulp from the oracle (expected to be very few).
    Returns (max error in ulps, number of outputs beyond one ulp) and records the count."""
    y64, _ = oracle.linear(qa, s_a, qw, s_w_rows, bias, G)
    yg = wl.bf16_bits_to_f32(y_gpu_bits).astype(np.float64)
    err = np.abs(yg - y64)
    ulp = ulp_bf16(y64)
    beyond = np.argwhere(err > ulp)
    if len(beyond):
        for start in range(0, len(beyond), 4096):
            idx = beyond[start:start + 4096]
            m, n = idx[:, 0], idx[:, 1]
            acc = np.stack([oracle.group_partials(qa[mi:mi + 1], qw[ni:ni + 1], G)[0, 0] for mi, ni in zip(m, n)])
            mag = np.sum(np.abs(acc.astype(np.float64)) * np.abs(s_a[m].astype(np.float64))
                         * np.abs(s_w_rows[n].astype(np.float64)), axis=1)
            if bias is not None:
                mag = mag + np.abs(np.asarray(bias, np.float64))[n]
            tol = ulp[m, n] + (acc.shape[1] + 2) * 2.0 ** -24 * mag
            bad = err[m, n] > tol
            if bad.any():
                k = np.argmax(bad)
                raise AssertionError(f"{label}: {int(bad.sum())} outputs out of tolerance, e.g. [{m[k]},{n[k]}] "
                                     f"gpu={yg[m[k], n[k]]!r} ref={y64[m[k], n[k]]!r} tol={tol[k]:.3g}")
    worst = float((err / ulp).max()) if err.size else 0.0
    report_escape(label, len(beyond), err.size, worst)
    return worst, len(beyond)
