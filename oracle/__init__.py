"""CPU oracle for the naive W4A4 linear layer (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the cpu-baseline/reference
leg of ``bench.py`` may import this package.  The product library never does.

The arithmetic lives in ``jq_oracle.c`` (plain C, compiled with gcc, no
fast-math, no FMA contraction); this module only compiles it and marshals
numpy arrays through ctypes.  Layout conventions used here:

* activation codes / weight codes: ``int8 [rows, K]`` (one code per element);
* packed codes: ``uint8 [rows, K/2]``, element 2j in the low nibble;
* packed ternary codes (W1.58A4 weights): ``uint8 [rows, K/4]``, q + 1 in 2 bits
  (byte layout in ``jq_oracle.c``);
* activation scales ``s_a``: ``float32 [M, K/G]``;
* weight scales ``s_w``: ``float32 [N, K/G]`` (per output channel);
* NVFP4 (E2M1 elements, E4M3 block scales per 16 along K, one fp32 tensor
  scale): element codes as ``int8`` holding twice the E2M1 value (integers in
  [-12, 12]); block scales ``float32 [rows, K/16]`` (each an E4M3 value);
  packed ``uint8 [rows, K/2]`` in the 4-bit E2M1 encoding, element 2j in the
  low nibble;
* bf16 values travel as their ``uint16`` bit patterns;
* DiT neighbour operations fused with the quantiser (adaLN modulation, tanh
  GELU): the modulated / activated bf16 bits come back beside the codes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "jq_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

_CFLAGS = ["-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC", "-shared", "-std=c11"]


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/liboracle.so`` (gcc, seconds)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < max(
        os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "jq_oracle.h"))
    ):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", *_CFLAGS, "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            i64, vp = ctypes.c_int64, ctypes.c_void_p
            lib.oracle_bf16_rne.argtypes = [ctypes.c_double]
            lib.oracle_bf16_rne.restype = ctypes.c_uint16
            lib.oracle_quantize_bf16.argtypes = [vp, i64, i64, i64, i64, vp, vp]
            lib.oracle_quantize_f32.argtypes = [vp, i64, i64, i64, vp, vp]
            lib.oracle_quantize_ternary_f32.argtypes = [vp, i64, i64, i64, vp, vp]
            lib.oracle_pack_ternary.argtypes = [vp, i64, i64, vp]
            lib.oracle_unpack_ternary.argtypes = [vp, i64, i64, vp]
            lib.oracle_pack.argtypes = [vp, i64, i64, vp]
            lib.oracle_unpack.argtypes = [vp, i64, i64, vp]
            lib.oracle_group_partials.argtypes = [vp, vp, i64, i64, i64, i64, vp]
            lib.oracle_linear.argtypes = [vp, vp, vp, vp, vp, i64, i64, i64, i64, vp, vp]
            f32 = ctypes.c_float
            lib.oracle_set_threads.argtypes = [ctypes.c_int]
            lib.oracle_set_threads.restype = None
            lib.oracle_max_threads.argtypes = []
            lib.oracle_max_threads.restype = ctypes.c_int
            lib.oracle_nvfp4_tensor_scale.argtypes = [vp, i64]
            lib.oracle_nvfp4_tensor_scale.restype = f32
            lib.oracle_quantize_nvfp4.argtypes = [vp, i64, i64, f32, vp, vp]
            lib.oracle_pack_nvfp4.argtypes = [vp, i64, i64, vp]
            lib.oracle_unpack_nvfp4.argtypes = [vp, i64, i64, vp]
            lib.oracle_linear_nvfp4.argtypes = [vp, vp, f32, vp, vp, f32, vp, i64, i64, i64, vp, vp]
            lib.oracle_fake_quant_bf16.argtypes = [vp, i64, i64, i64, vp, vp, vp, vp]
            lib.oracle_fake_quant_f32.argtypes = [vp, i64, i64, i64, vp, vp, vp, vp]
            lib.oracle_ste_backward_bf16.argtypes = [vp, vp, i64, vp]
            lib.oracle_gelu_tanh_f32.argtypes = [ctypes.c_float]
            lib.oracle_gelu_tanh_f32.restype = ctypes.c_float
            lib.oracle_modulate_quantize_bf16.argtypes = [vp, i64, i64, i64, vp, vp, i64, i64, vp, vp, vp]
            lib.oracle_gelu_quantize_bf16.argtypes = [vp, i64, i64, i64, i64, vp, vp, vp]
            for f in ("oracle_fake_quant_bf16", "oracle_fake_quant_f32", "oracle_ste_backward_bf16",
                      "oracle_quantize_bf16", "oracle_quantize_f32", "oracle_pack", "oracle_unpack",
                      "oracle_group_partials", "oracle_linear", "oracle_quantize_ternary_f32",
                      "oracle_pack_ternary", "oracle_unpack_ternary", "oracle_quantize_nvfp4",
                      "oracle_pack_nvfp4", "oracle_unpack_nvfp4", "oracle_linear_nvfp4",
                      "oracle_modulate_quantize_bf16", "oracle_gelu_quantize_bf16"):
                getattr(lib, f).restype = None
            _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def set_threads(n: int) -> None:
    """OpenMP threads for the oracle's row-parallel loops (results do not depend on it)."""
    _load().oracle_set_threads(int(n))


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def bf16_rne(v: float) -> int:
    """fp64 -> bf16 bits, round to nearest even."""
    return int(_load().oracle_bf16_rne(float(v)))


def quantize_bf16(x_bits: np.ndarray, group: int):
    """bf16 activations (uint16 bits, [M, K] or a strided view) -> (codes int8 [M,K], s_a f32 [M,K/G])."""
    x_bits = np.asarray(x_bits)
    assert x_bits.dtype == np.uint16 and x_bits.ndim == 2
    M, K = x_bits.shape
    assert K % group == 0
    if x_bits.strides[1] != 2 or x_bits.strides[0] % 2:
        x_bits = np.ascontiguousarray(x_bits)
    ldx = x_bits.strides[0] // 2
    codes = np.empty((M, K), np.int8)
    scales = np.empty((M, K // group), np.float32)
    _load().oracle_quantize_bf16(_p(x_bits), M, K, ldx, group, _p(codes), _p(scales))
    return codes, scales


def quantize_f32(w: np.ndarray, group: int):
    """fp32 weights [N, K] -> (codes int8 [N,K], s_w f32 [N,K/G])."""
    w = _c(w, np.float32)
    N, K = w.shape
    assert K % group == 0
    codes = np.empty((N, K), np.int8)
    scales = np.empty((N, K // group), np.float32)
    _load().oracle_quantize_f32(_p(w), N, K, group, _p(codes), _p(scales))
    return codes, scales


def pack(codes: np.ndarray) -> np.ndarray:
    codes = _c(codes, np.int8)
    R, K = codes.shape
    assert K % 2 == 0
    out = np.empty((R, K // 2), np.uint8)
    _load().oracle_pack(_p(codes), R, K, _p(out))
    return out


def unpack(packed: np.ndarray) -> np.ndarray:
    packed = _c(packed, np.uint8)
    R, H = packed.shape
    out = np.empty((R, 2 * H), np.int8)
    _load().oracle_unpack(_p(packed), R, 2 * H, _p(out))
    return out


def quantize_ternary_f32(w: np.ndarray, group: int):
    """fp32 weights [N, K] -> (ternary codes int8 [N,K] in {-1,0,1}, s_w f32 [N,K/G]) (absmean rule)."""
    w = _c(w, np.float32)
    N, K = w.shape
    assert K % group == 0
    codes = np.empty((N, K), np.int8)
    scales = np.empty((N, K // group), np.float32)
    _load().oracle_quantize_ternary_f32(_p(w), N, K, group, _p(codes), _p(scales))
    return codes, scales


def pack_ternary(codes: np.ndarray) -> np.ndarray:
    """ternary codes int8 [rows, K] (K % 16 == 0) -> uint8 [rows, K/4] (2 bits per code, q + 1)."""
    codes = _c(codes, np.int8)
    R, K = codes.shape
    assert K % 16 == 0 and codes.min(initial=0) >= -1 and codes.max(initial=0) <= 1
    out = np.empty((R, K // 4), np.uint8)
    _load().oracle_pack_ternary(_p(codes), R, K, _p(out))
    return out


def unpack_ternary(packed: np.ndarray) -> np.ndarray:
    packed = _c(packed, np.uint8)
    R, Q = packed.shape
    out = np.empty((R, 4 * Q), np.int8)
    _load().oracle_unpack_ternary(_p(packed), R, 4 * Q, _p(out))
    return out


def group_partials(qa: np.ndarray, qw: np.ndarray, group: int) -> np.ndarray:
    """Exact per-group integer partials, int32 [M, N, K/G]."""
    qa, qw = _c(qa, np.int8), _c(qw, np.int8)
    M, K = qa.shape
    N, K2 = qw.shape
    assert K == K2 and K % group == 0
    acc = np.empty((M, N, K // group), np.int32)
    _load().oracle_group_partials(_p(qa), _p(qw), M, N, K, group, _p(acc))
    return acc


def linear(qa, s_a, qw, s_w, bias, group: int):
    """(y64 float64 [M,N], y_bf16 uint16 [M,N]) of the dequantising linear layer."""
    qa, qw = _c(qa, np.int8), _c(qw, np.int8)
    s_a, s_w = _c(s_a, np.float32), _c(s_w, np.float32)
    M, K = qa.shape
    N = qw.shape[0]
    assert s_a.shape == (M, K // group) and s_w.shape == (N, K // group)
    b = None if bias is None else _c(bias, np.float32)
    y64 = np.empty((M, N), np.float64)
    yb = np.empty((M, N), np.uint16)
    _load().oracle_linear(_p(qa), _p(s_a), _p(qw), _p(s_w), _p(b), M, N, K, group, _p(y64), _p(yb))
    return y64, yb


def nvfp4_tensor_scale(x: np.ndarray) -> float:
    """fp32 per-tensor NVFP4 scale fl32(amax |x| / 2688) (2688 = 6 * 448)."""
    x = _c(x, np.float32)
    return float(_load().oracle_nvfp4_tensor_scale(_p(x), x.size))


def quantize_nvfp4(x: np.ndarray, g: float):
    """fp32 [rows, K] (K % 16 == 0), tensor scale g -> (2q int8 [rows,K], E4M3 block scales f32 [rows,K/16])."""
    x = _c(x, np.float32)
    R, K = x.shape
    assert K % 16 == 0
    codes2 = np.empty((R, K), np.int8)
    scales = np.empty((R, K // 16), np.float32)
    _load().oracle_quantize_nvfp4(_p(x), R, K, ctypes.c_float(g), _p(codes2), _p(scales))
    return codes2, scales


def pack_nvfp4(codes2: np.ndarray) -> np.ndarray:
    codes2 = _c(codes2, np.int8)
    R, K = codes2.shape
    assert K % 2 == 0
    assert np.isin(np.abs(codes2.astype(np.int16)), [0, 1, 2, 3, 4, 6, 8, 12]).all()
    out = np.empty((R, K // 2), np.uint8)
    _load().oracle_pack_nvfp4(_p(codes2), R, K, _p(out))
    return out


def unpack_nvfp4(packed: np.ndarray) -> np.ndarray:
    packed = _c(packed, np.uint8)
    R, H = packed.shape
    out = np.empty((R, 2 * H), np.int8)
    _load().oracle_unpack_nvfp4(_p(packed), R, 2 * H, _p(out))
    return out


def linear_nvfp4(qa2, sa, ga: float, qw2, sw, gw: float, bias):
    """(y64 float64 [M,N], y_bf16 uint16 [M,N]) of the NVFP4 linear layer (block scales per 16 along K)."""
    qa2, qw2 = _c(qa2, np.int8), _c(qw2, np.int8)
    sa, sw = _c(sa, np.float32), _c(sw, np.float32)
    M, K = qa2.shape
    N = qw2.shape[0]
    assert K % 16 == 0 and sa.shape == (M, K // 16) and sw.shape == (N, K // 16)
    b = None if bias is None else _c(bias, np.float32)
    y64 = np.empty((M, N), np.float64)
    yb = np.empty((M, N), np.uint16)
    _load().oracle_linear_nvfp4(_p(qa2), _p(sa), ctypes.c_float(ga), _p(qw2), _p(sw), ctypes.c_float(gw),
                                _p(b), M, N, K, _p(y64), _p(yb))
    return y64, yb


def fake_quant_bf16(x_bits: np.ndarray, group: int, s_in=None):
    """Fake quantisation of bf16 activations for training (forward of the STE reading).

    x_bits uint16 [M, K] -> (xhat uint16 bf16 bits [M, K], mask uint8 [M, K], scales f32 [M, K/G]).
    s_in: None for the amax/7 rule, else [M, K/G] positive finite scales to use instead."""
    x_bits = _c(x_bits, np.uint16)
    M, K = x_bits.shape
    assert K % group == 0
    s = None if s_in is None else _c(s_in, np.float32)
    assert s is None or s.shape == (M, K // group)
    xhat = np.empty((M, K), np.uint16)
    mask = np.empty((M, K), np.uint8)
    s_out = np.empty((M, K // group), np.float32)
    _load().oracle_fake_quant_bf16(_p(x_bits), M, K, group, _p(s), _p(xhat), _p(mask), _p(s_out))
    return xhat, mask, s_out


def fake_quant_f32(w: np.ndarray, group: int, s_in=None):
    """Fake quantisation of fp32 weights: -> (what f32 [N, K], mask uint8 [N, K], scales f32 [N, K/G])."""
    w = _c(w, np.float32)
    N, K = w.shape
    assert K % group == 0
    s = None if s_in is None else _c(s_in, np.float32)
    assert s is None or s.shape == (N, K // group)
    what = np.empty((N, K), np.float32)
    mask = np.empty((N, K), np.uint8)
    s_out = np.empty((N, K // group), np.float32)
    _load().oracle_fake_quant_f32(_p(w), N, K, group, _p(s), _p(what), _p(mask), _p(s_out))
    return what, mask, s_out


def ste_backward_bf16(grad_bits: np.ndarray, mask: np.ndarray) -> np.ndarray:
    """STE backward: bf16 gradient bits where mask is 1, +0 where it is 0 (same shape)."""
    grad_bits = _c(grad_bits, np.uint16)
    mask = _c(mask, np.uint8)
    assert grad_bits.shape == mask.shape
    out = np.empty_like(grad_bits)
    _load().oracle_ste_backward_bf16(_p(grad_bits), _p(mask), grad_bits.size, _p(out))
    return out


def gelu_tanh_f32(h: float) -> float:
    """The tanh-approximate GELU of one fp32 value, in the oracle's fp32 steps."""
    return float(_load().oracle_gelu_tanh_f32(ctypes.c_float(h)))


def _rows(a):
    a = np.asarray(a)
    assert a.dtype == np.uint16 and a.ndim == 2
    if a.strides[1] != 2 or a.strides[0] % 2:
        a = np.ascontiguousarray(a)
    return a, a.strides[0] // 2


def modulate_quantize_bf16(x_bits: np.ndarray, shift: np.ndarray, scale: np.ndarray, tokens_per_sample: int,
                           group: int):
    """adaLN modulation fused with the activation quantiser (DiT-XL/2 block linears).

    x_bits uint16 [M, K] (bf16 bits, rows may be strided); shift, scale f32 [B, K] with
    B = ceil(M / tokens_per_sample) -> (z uint16 [M, K] the modulated bf16 bits,
    codes int8 [M, K], scales f32 [M, K/G])."""
    x_bits, ldx = _rows(x_bits)
    M, K = x_bits.shape
    assert K % group == 0 and tokens_per_sample > 0
    sh, sc = _c(shift, np.float32), _c(scale, np.float32)
    assert sh.shape == sc.shape and sh.shape[1] == K and sh.shape[0] * tokens_per_sample >= M
    z = np.empty((M, K), np.uint16)
    codes = np.empty((M, K), np.int8)
    scales = np.empty((M, K // group), np.float32)
    _load().oracle_modulate_quantize_bf16(_p(x_bits), M, K, ldx, _p(sh), _p(sc), tokens_per_sample, group, _p(z),
                                          _p(codes), _p(scales))
    return z, codes, scales


def gelu_quantize_bf16(h_bits: np.ndarray, group: int):
    """tanh-approximate GELU fused with the activation quantiser (the input of a DiT MLP's second
    linear): h_bits uint16 [M, K] -> (z uint16 [M, K] = bf16 of the fp32-evaluated GELU(h),
    codes int8 [M, K], scales f32 [M, K/G])."""
    h_bits, ldh = _rows(h_bits)
    M, K = h_bits.shape
    assert K % group == 0
    z = np.empty((M, K), np.uint16)
    codes = np.empty((M, K), np.int8)
    scales = np.empty((M, K // group), np.float32)
    _load().oracle_gelu_quantize_bf16(_p(h_bits), M, K, ldh, group, _p(z), _p(codes), _p(scales))
    return z, codes, scales
