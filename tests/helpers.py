"""Shared helpers for the parity tests: oracle references and the bf16 tolerance rule."""
from __future__ import annotations

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
    return float((err / ulp).max()), int((err > ulp).sum())


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
