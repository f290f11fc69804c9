"""GB300-native naive W4A4 linear layer of JustQuant (arxiv 2609.33601).

Python binding of ``libjq.so`` (the C ABI in ``include/jq.h``).  The functions carry the C
names and only marshal arguments: torch tensors provide device memory and the current CUDA
stream, and every step of the computation runs in the library's sm_103a kernels.  There is no
CPU or PyTorch fallback: if ``libjq.so`` is missing or the device is not an sm_103 GPU, the
calls raise.

    q, s_a  = jq_quantize_act(x_bf16, group)              # INT4 codes, per (token, K-group) scales
    qw, s_w = jq_pack_weight(w_fp32, group)               # offline
    y       = jq_w4a4_linear(q, s_a, qw, s_w, bias, group)
    y       = jq_fused_quant_linear(x_bf16, qw, s_w, bias, group)

Layouts: x bf16 [M, K] (row stride may exceed K); q uint8 [M, K/2]; s_a fp32 [M, K/G];
qw uint8 [N, K/2]; s_w fp32 [K/G, N]; bias fp32 [N] or None; y bf16 [M, N].
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

__all__ = [
    "JQError", "library_path", "jq_quantize_act", "jq_pack_weight", "jq_workspace_size", "jq_w4a4_linear",
    "jq_fused_quant_linear", "jq_w4a4_group_partials", "jq_device_status", "jq_status_string",
    "jq_w4a4_linear_noalloc", "jq_pack_weight_ternary", "jq_w158a4_workspace_size", "jq_w158a4_linear",
    "jq_debug_wait_timeout", "jq_fake_quant_act", "jq_fake_quant_weight",
    "jq_ste_backward", "jq_modulate_quantize_act", "jq_gelu_quantize_act", "jq_nvfp4_quantize_act", "jq_nvfp4_pack_weight",
    "jq_nvfp4_workspace_size", "jq_nvfp4_linear",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
library_path = os.path.join(_HERE, "libjq.so")

JQ_STATUS = {0: "JQ_OK", 1: "JQ_ERR_INVALID_ARG", 2: "JQ_ERR_MISALIGNED", 3: "JQ_ERR_UNSUPPORTED",
             4: "JQ_ERR_CUDA", 5: "JQ_ERR_TIMEOUT", 6: "JQ_ERR_WORKSPACE"}

_lock = threading.Lock()
_lib = None


class JQError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} failed: {JQ_STATUS.get(code, code)}")
        self.code = code


def _load() -> ctypes.CDLL:
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(library_path):
                raise RuntimeError(
                    f"{library_path} is not built; run `python -m paper_2609_33601_gb300.build` "
                    "(needs nvcc for sm_103a). There is no fallback implementation.")
            lib = ctypes.CDLL(library_path)
            i64, i32, vp, sz = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_size_t
            sig = {
                "jq_quantize_act": [vp, i64, i64, i64, i32, vp, vp, vp],
                "jq_pack_weight": [vp, i64, i64, i32, vp, vp, vp],
                "jq_w4a4_linear": [vp, vp, vp, vp, vp, vp, i64, i64, i64, i32, vp, sz, vp],
                "jq_fused_quant_linear": [vp, i64, vp, vp, vp, vp, i64, i64, i64, i32, vp, sz, vp],
                "jq_w4a4_group_partials": [vp, vp, vp, i64, i64, i64, i32, vp, sz, vp],
                "jq_device_status": [vp, i32],
                "jq_debug_wait_timeout": [vp],
                "jq_fake_quant_act": [vp, i64, i64, i32, vp, vp, vp, vp, vp],
                "jq_ste_backward": [vp, vp, i64, vp, vp],
                "jq_fake_quant_weight": [vp, i64, i64, i32, vp, vp, vp, vp, vp],
                "jq_w4a4_linear_noalloc": [vp, vp, vp, vp, vp, vp, i64, i64, i64, i32, vp],
                "jq_pack_weight_ternary": [vp, i64, i64, i32, vp, vp, vp],
                "jq_w158a4_linear": [vp, vp, vp, vp, vp, vp, i64, i64, i64, i32, vp, sz, vp],
                "jq_modulate_quantize_act": [vp, i64, i64, i64, vp, vp, i64, i32, vp, vp, vp],
                "jq_gelu_quantize_act": [vp, i64, i64, i64, i32, vp, vp, vp],
                "jq_nvfp4_quantize_act": [vp, i64, i64, i64, ctypes.c_float, vp, vp, vp],
                "jq_nvfp4_pack_weight": [vp, i64, i64, vp, vp, vp, vp],
                "jq_nvfp4_linear": [vp, vp, ctypes.c_float, vp, vp, vp, vp, vp, i64, i64, i64, vp, sz, vp],
            }
            for name, args in sig.items():
                f = getattr(lib, name)
                f.argtypes = args
                f.restype = ctypes.c_int
            lib.jq_workspace_size.argtypes = [i64, i64, i64, i32, i32]
            lib.jq_workspace_size.restype = ctypes.c_size_t
            lib.jq_w158a4_workspace_size.argtypes = [i64, i64, i64, i32]
            lib.jq_w158a4_workspace_size.restype = ctypes.c_size_t
            lib.jq_nvfp4_workspace_size.argtypes = [i64, i64, i64]
            lib.jq_nvfp4_workspace_size.restype = ctypes.c_size_t
            lib.jq_status_string.argtypes = [ctypes.c_int]
            lib.jq_status_string.restype = ctypes.c_char_p
            _lib = lib
    return _lib


def _check(name: str, code: int) -> None:
    if code != 0:
        raise JQError(name, code)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _device_mismatch(device, current: int, stream_device=None) -> str | None:
    """Why tensors on `device` cannot go to a library call made with CUDA device `current` and a
    stream of `stream_device`, or None when they can.  The C calls launch on the current device
    and address its memory, so tensors of another GPU would be read there as foreign pointers."""
    if device.index is not None and device.index != current:
        return (f"the tensors are on {device} but the current CUDA device is cuda:{current}; "
                f"call inside `with torch.cuda.device({device.index}):`")
    if stream_device is not None and stream_device != device:
        return f"the stream belongs to {stream_device}, the tensors to {device}"
    return None


def _need_cuda(*ts, stream=None):
    """Every tensor is a CUDA tensor on the current device, and the stream (if given) is one of
    that device (the tensors' agreement with one another is checked by _expect)."""
    dev = None
    for t in ts:
        if t is not None and not t.is_cuda:
            raise ValueError("libjq works on CUDA tensors only")
        if t is not None and dev is None:
            dev = t.device
    if dev is not None:
        why = _device_mismatch(dev, torch.cuda.current_device(), None if stream is None else stream.device)
        if why is not None:
            raise ValueError(f"libjq: {why}")


def _groups(K: int, group: int):
    """K/group, or None when group does not divide K (the library then rejects the call)."""
    return K // group if group > 0 and K % group == 0 else None


def _expect(fn: str, name: str, t, dtype, shape, device) -> None:
    """The library receives bare pointers, so a tensor smaller than the call implies, strided,
    of another type or on another device would be read or written out of bounds: refuse it
    here.  shape entries of None are not checked (the scale shapes when group is invalid)."""
    if t is None:
        return
    if None in shape:
        shape_ok = t.dim() == len(shape) and all(w is None or h == w for h, w in zip(t.shape, shape))
    else:
        shape_ok = t.shape == shape
    if not (shape_ok and t.dtype == dtype and t.is_contiguous() and t.device == device):
        raise ValueError(f"{fn}: {name} must be a contiguous {dtype} tensor of shape {list(shape)} on {device}; "
                         f"got {t.dtype} {list(t.shape)} (contiguous={t.is_contiguous()}) on {t.device}")


def _expect_workspace(fn: str, ws, device) -> None:
    """Any 1-D contiguous uint8 device buffer (the library checks its size)."""
    if ws is not None and not (ws.dtype == torch.uint8 and ws.dim() == 1 and ws.is_contiguous()
                               and ws.device == device):
        raise ValueError(f"{fn}: workspace must be a contiguous 1-D uint8 tensor on {device}; "
                         f"got {ws.dtype} {list(ws.shape)} on {ws.device}")


def _expect_x(fn: str, x) -> None:
    if not (x.dtype == torch.bfloat16 and x.dim() == 2 and x.stride(1) == 1):
        raise ValueError(f"{fn}: x must be a 2-D bfloat16 tensor with unit column stride (rows may be padded); "
                         f"got {x.dtype} {list(x.shape)} strides {list(x.stride())}")


def _codes_shapes(fn: str, q, qw, codes_per_byte: int):
    """(M, K, N) from packed activation codes q [M, K/2] and packed weights qw [N, K/codes_per_byte],
    after checking both."""
    if q.dim() != 2 or qw.dim() != 2:
        raise ValueError(f"{fn}: q and the packed weights must be 2-D, got {list(q.shape)} and {list(qw.shape)}")
    M, K = q.shape[0], q.shape[1] * 2
    N = qw.shape[0]
    _expect(fn, "q", q, torch.uint8, (M, K // 2), q.device)
    _expect(fn, "packed weights", qw, torch.uint8, (N, K // codes_per_byte), q.device)
    return M, K, N


def _expect_linear(fn: str, M: int, N: int, K: int, group: int, device, s_a, s_w, bias, y, workspace) -> None:
    ng = _groups(K, group)
    _expect(fn, "s_a", s_a, torch.float32, (M, ng), device)
    _expect(fn, "s_w", s_w, torch.float32, (ng, N), device)
    _expect(fn, "bias", bias, torch.float32, (N,), device)
    _expect(fn, "y", y, torch.bfloat16, (M, N), device)
    _expect_workspace(fn, workspace, device)


def jq_status_string(code: int) -> str:
    return _load().jq_status_string(code).decode()


def jq_workspace_size(M: int, N: int, K: int, group: int, fused: bool = False) -> int:
    return int(_load().jq_workspace_size(M, N, K, group, 1 if fused else 0))


def _workspace(M, N, K, group, fused, device, workspace):
    need = jq_workspace_size(M, N, K, group, fused)
    if workspace is None:
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=device)
    return workspace, workspace.numel() * workspace.element_size()


def jq_quantize_act(x: torch.Tensor, group: int, q: torch.Tensor | None = None, s_a: torch.Tensor | None = None,
                    stream=None):
    """bf16 activations [M, K] (row stride >= K) -> (packed codes uint8 [M, K/2], scales fp32 [M, K/G])."""
    fn = "jq_quantize_act"
    _expect_x(fn, x)
    M, K = x.shape
    _expect(fn, "q", q, torch.uint8, (M, K // 2), x.device)
    _expect(fn, "s_a", s_a, torch.float32, (M, _groups(K, group)), x.device)
    _need_cuda(x, stream=stream)
    if q is None:
        q = torch.empty((M, K // 2), dtype=torch.uint8, device=x.device)
    if s_a is None:
        s_a = torch.empty((M, K // group if group else 0), dtype=torch.float32, device=x.device)
    _check("jq_quantize_act", _load().jq_quantize_act(_ptr(x), M, K, x.stride(0), group, _ptr(q), _ptr(s_a),
                                                      _stream(stream)))
    return q, s_a


def jq_modulate_quantize_act(x: torch.Tensor, shift: torch.Tensor, scale: torch.Tensor, tokens_per_sample: int,
                             group: int, q: torch.Tensor | None = None, s_a: torch.Tensor | None = None, stream=None):
    """adaLN modulation fused with the activation quantiser (DiT block linears): the codes and
    scales of bf16(x * (1 + scale[b]) + shift[b]) for token m of sample b = m // tokens_per_sample.

    x bf16 [M, K] (row stride >= K); shift, scale fp32 [ceil(M / tokens_per_sample), K]
    -> (packed codes uint8 [M, K/2], scales fp32 [M, K/G])."""
    fn = "jq_modulate_quantize_act"
    _expect_x(fn, x)
    M, K = x.shape
    if tokens_per_sample <= 0:
        raise ValueError(f"{fn}: tokens_per_sample must be positive")
    samples = -(-M // tokens_per_sample)
    _expect(fn, "shift", shift, torch.float32, (samples, K), x.device)
    _expect(fn, "scale", scale, torch.float32, (samples, K), x.device)
    _expect(fn, "q", q, torch.uint8, (M, K // 2), x.device)
    _expect(fn, "s_a", s_a, torch.float32, (M, _groups(K, group)), x.device)
    _need_cuda(x, shift, scale, stream=stream)
    if q is None:
        q = torch.empty((M, K // 2), dtype=torch.uint8, device=x.device)
    if s_a is None:
        s_a = torch.empty((M, K // group if group else 0), dtype=torch.float32, device=x.device)
    _check(fn, _load().jq_modulate_quantize_act(_ptr(x), M, K, x.stride(0), _ptr(shift), _ptr(scale),
                                                tokens_per_sample, group, _ptr(q), _ptr(s_a), _stream(stream)))
    return q, s_a


def jq_gelu_quantize_act(h: torch.Tensor, group: int, q: torch.Tensor | None = None,
                         s_a: torch.Tensor | None = None, stream=None):
    """tanh GELU fused with the activation quantiser (the input of a DiT MLP's second linear):
    the codes and scales of bf16(GELU(h)).  h bf16 [M, K] -> (uint8 [M, K/2], fp32 [M, K/G])."""
    fn = "jq_gelu_quantize_act"
    _expect_x(fn, h)
    M, K = h.shape
    _expect(fn, "q", q, torch.uint8, (M, K // 2), h.device)
    _expect(fn, "s_a", s_a, torch.float32, (M, _groups(K, group)), h.device)
    _need_cuda(h, stream=stream)
    if q is None:
        q = torch.empty((M, K // 2), dtype=torch.uint8, device=h.device)
    if s_a is None:
        s_a = torch.empty((M, K // group if group else 0), dtype=torch.float32, device=h.device)
    _check(fn, _load().jq_gelu_quantize_act(_ptr(h), M, K, h.stride(0), group, _ptr(q), _ptr(s_a), _stream(stream)))
    return q, s_a


def jq_pack_weight(w: torch.Tensor, group: int, stream=None):
    """fp32 weights [N, K] -> (packed codes uint8 [N, K/2], scales fp32 [K/G, N])."""
    if w.dim() != 2:
        raise ValueError(f"jq_pack_weight: w must be 2-D, got shape {list(w.shape)}")
    N, K = w.shape
    _expect("jq_pack_weight", "w", w, torch.float32, (N, K), w.device)
    _need_cuda(w, stream=stream)
    qw = torch.empty((N, K // 2), dtype=torch.uint8, device=w.device)
    s_w = torch.empty((K // group if group else 0, N), dtype=torch.float32, device=w.device)
    _check("jq_pack_weight", _load().jq_pack_weight(_ptr(w), N, K, group, _ptr(qw), _ptr(s_w), _stream(stream)))
    return qw, s_w


def jq_w4a4_linear(q, s_a, qw, s_w, bias, group: int, y=None, workspace=None, stream=None):
    """y = bf16(sum_g acc * s_a * s_w + bias) from packed activation and weight codes."""
    fn = "jq_w4a4_linear"
    M, K, N = _codes_shapes(fn, q, qw, 2)
    _expect_linear(fn, M, N, K, group, q.device, s_a, s_w, bias, y, workspace)
    _need_cuda(q, s_a, qw, s_w, bias, stream=stream)
    if y is None:
        y = torch.empty((M, N), dtype=torch.bfloat16, device=q.device)
    ws, ws_bytes = _workspace(M, N, K, group, False, q.device, workspace)
    _check("jq_w4a4_linear", _load().jq_w4a4_linear(_ptr(q), _ptr(s_a), _ptr(qw), _ptr(s_w), _ptr(bias), _ptr(y),
                                                    M, N, K, group, _ptr(ws), ws_bytes, _stream(stream)))
    return y


def jq_w4a4_linear_noalloc(q, s_a, qw, s_w, bias, group: int, y=None, stream=None):
    """jq_w4a4_linear without a workspace, for callers that cannot allocate device memory: the
    library keeps the scratch in its own fixed 16 MiB device array.  More than 64 tokens (and
    one-group problems with K above 139776) need
    ceil(M/128)*128*K + round_up(4*M*(K/G), 256) <= 16 MiB
    (the operand image, then one fp32 correction per token and group); larger calls raise
    JQError(JQ_ERR_WORKSPACE).  Calls share that array, so order them on one stream.  (Only the
    output tensor is allocated here, by the caller's side, when y is None.)"""
    fn = "jq_w4a4_linear_noalloc"
    M, K, N = _codes_shapes(fn, q, qw, 2)
    _expect_linear(fn, M, N, K, group, q.device, s_a, s_w, bias, y, None)
    _need_cuda(q, s_a, qw, s_w, bias, stream=stream)
    if y is None:
        y = torch.empty((M, N), dtype=torch.bfloat16, device=q.device)
    _check("jq_w4a4_linear_noalloc",
           _load().jq_w4a4_linear_noalloc(_ptr(q), _ptr(s_a), _ptr(qw), _ptr(s_w), _ptr(bias), _ptr(y), M, N, K,
                                          group, _stream(stream)))
    return y


def jq_fused_quant_linear(x, qw, s_w, bias, group: int, y=None, workspace=None, stream=None):
    """Same result as jq_w4a4_linear(*jq_quantize_act(x, group), ...), straight from bf16 x."""
    fn = "jq_fused_quant_linear"
    _expect_x(fn, x)
    M, K = x.shape
    if qw.dim() != 2:
        raise ValueError(f"{fn}: qw must be 2-D, got shape {list(qw.shape)}")
    N = qw.shape[0]
    _expect(fn, "qw", qw, torch.uint8, (N, K // 2), x.device)
    _expect_linear(fn, M, N, K, group, x.device, None, s_w, bias, y, workspace)
    _need_cuda(x, qw, s_w, bias, stream=stream)
    if y is None:
        y = torch.empty((M, N), dtype=torch.bfloat16, device=x.device)
    ws, ws_bytes = _workspace(M, N, K, group, True, x.device, workspace)
    _check("jq_fused_quant_linear",
           _load().jq_fused_quant_linear(_ptr(x), x.stride(0), _ptr(qw), _ptr(s_w), _ptr(bias), _ptr(y), M, N, K,
                                         group, _ptr(ws), ws_bytes, _stream(stream)))
    return y


def jq_w4a4_group_partials(q, qw, group: int, workspace=None, stream=None):
    """Exact per-group integer partials int32 [M, N, K/G] (verification export)."""
    fn = "jq_w4a4_group_partials"
    M, K, N = _codes_shapes(fn, q, qw, 2)
    if _groups(K, group) is None:
        raise ValueError(f"{fn}: group {group} does not divide K = {K}")
    _expect_workspace(fn, workspace, q.device)
    _need_cuda(q, qw, stream=stream)
    acc = torch.empty((M, N, K // group), dtype=torch.int32, device=q.device)
    ws, ws_bytes = _workspace(M, N, K, group, False, q.device, workspace)
    _check("jq_w4a4_group_partials",
           _load().jq_w4a4_group_partials(_ptr(q), _ptr(qw), _ptr(acc), M, N, K, group, _ptr(ws), ws_bytes,
                                          _stream(stream)))
    return acc


def jq_pack_weight_ternary(w: torch.Tensor, group: int, stream=None):
    """fp32 weights [N, K] -> (packed ternary codes uint8 [N, K/4], scales fp32 [K/G, N])."""
    if w.dim() != 2:
        raise ValueError(f"jq_pack_weight_ternary: w must be 2-D, got shape {list(w.shape)}")
    N, K = w.shape
    _expect("jq_pack_weight_ternary", "w", w, torch.float32, (N, K), w.device)
    _need_cuda(w, stream=stream)
    qw2 = torch.empty((N, K // 4), dtype=torch.uint8, device=w.device)
    s_w = torch.empty((K // group if group else 0, N), dtype=torch.float32, device=w.device)
    _check("jq_pack_weight_ternary",
           _load().jq_pack_weight_ternary(_ptr(w), N, K, group, _ptr(qw2), _ptr(s_w), _stream(stream)))
    return qw2, s_w


def jq_w158a4_workspace_size(M: int, N: int, K: int, group: int) -> int:
    return int(_load().jq_w158a4_workspace_size(M, N, K, group))


def jq_w158a4_linear(q, s_a, qw2, s_w, bias, group: int, y=None, workspace=None, stream=None):
    """W1.58A4: y = bf16(sum_g acc * s_a * s_w + bias) from packed INT4 activations and packed
    ternary weights."""
    fn = "jq_w158a4_linear"
    M, K, N = _codes_shapes(fn, q, qw2, 4)
    _expect_linear(fn, M, N, K, group, q.device, s_a, s_w, bias, y, workspace)
    _need_cuda(q, s_a, qw2, s_w, bias, stream=stream)
    if y is None:
        y = torch.empty((M, N), dtype=torch.bfloat16, device=q.device)
    if workspace is None:
        workspace = torch.empty(max(jq_w158a4_workspace_size(M, N, K, group), 16), dtype=torch.uint8, device=q.device)
    ws_bytes = workspace.numel() * workspace.element_size()
    _check("jq_w158a4_linear",
           _load().jq_w158a4_linear(_ptr(q), _ptr(s_a), _ptr(qw2), _ptr(s_w), _ptr(bias), _ptr(y), M, N, K, group,
                                    _ptr(workspace), ws_bytes, _stream(stream)))
    return y


def jq_nvfp4_quantize_act(x: torch.Tensor, g_a: float, codes=None, scales=None, stream=None):
    """NVFP4 activations: bf16 [M, K] (K % 64 == 0) with the tensor scale g_a ->
    (E2M1 codes uint8 [M, K/2], E4M3 block-scale bytes uint8 [M, K/16])."""
    fn = "jq_nvfp4_quantize_act"
    _expect_x(fn, x)
    M, K = x.shape
    dev = x.device
    _expect(fn, "codes", codes, torch.uint8, (M, K // 2), dev)
    _expect(fn, "scales", scales, torch.uint8, (M, K // 16), dev)
    _need_cuda(x, stream=stream)
    if codes is None:
        codes = torch.empty((M, K // 2), dtype=torch.uint8, device=dev)
    if scales is None:
        scales = torch.empty((M, K // 16), dtype=torch.uint8, device=dev)
    _check(fn, _load().jq_nvfp4_quantize_act(_ptr(x), M, K, x.stride(0), float(g_a), _ptr(codes), _ptr(scales),
                                             _stream(stream)))
    return codes, scales


def jq_nvfp4_pack_weight(w: torch.Tensor, stream=None):
    """NVFP4 weights: fp32 [N, K] -> (codes uint8 [N, K/2], block-scale bytes uint8 [N, K/16],
    tensor scale fp32 [1] on the device)."""
    fn = "jq_nvfp4_pack_weight"
    if w.dim() != 2:
        raise ValueError(f"{fn}: w must be 2-D, got shape {list(w.shape)}")
    N, K = w.shape
    _expect(fn, "w", w, torch.float32, (N, K), w.device)
    _need_cuda(w, stream=stream)
    codes = torch.empty((N, K // 2), dtype=torch.uint8, device=w.device)
    scales = torch.empty((N, K // 16), dtype=torch.uint8, device=w.device)
    g_w = torch.empty(4, dtype=torch.float32, device=w.device)  # one used; 16 bytes for the alignment rule
    _check(fn, _load().jq_nvfp4_pack_weight(_ptr(w), N, K, _ptr(codes), _ptr(scales), _ptr(g_w), _stream(stream)))
    return codes, scales, g_w[:1]


def jq_nvfp4_workspace_size(M: int, N: int, K: int) -> int:
    return int(_load().jq_nvfp4_workspace_size(M, N, K))


def jq_nvfp4_linear(codes_a, scales_a, g_a: float, codes_w, scales_w, g_w, bias, y=None, workspace=None,
                    stream=None):
    """NVFP4 W4A4: y = bf16(sum_b (sum qa qw) sa_b sw_b g_a g_w + bias) from the quantiser's and
    the packer's outputs (g_w: the packer's one-element device tensor)."""
    fn = "jq_nvfp4_linear"
    M, K, N = _codes_shapes(fn, codes_a, codes_w, 2)
    dev = codes_a.device
    _expect(fn, "scales_a", scales_a, torch.uint8, (M, K // 16), dev)
    _expect(fn, "scales_w", scales_w, torch.uint8, (N, K // 16), dev)
    _expect(fn, "g_w", g_w, torch.float32, (1,), dev)
    _expect(fn, "bias", bias, torch.float32, (N,), dev)
    _expect(fn, "y", y, torch.bfloat16, (M, N), dev)
    _expect_workspace(fn, workspace, dev)
    _need_cuda(codes_a, scales_a, codes_w, scales_w, g_w, bias, stream=stream)
    if y is None:
        y = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
    if workspace is None:
        workspace = torch.empty(max(jq_nvfp4_workspace_size(M, N, K), 16), dtype=torch.uint8, device=dev)
    ws_bytes = workspace.numel() * workspace.element_size()
    _check(fn, _load().jq_nvfp4_linear(_ptr(codes_a), _ptr(scales_a), float(g_a), _ptr(codes_w), _ptr(scales_w),
                                       _ptr(g_w), _ptr(bias), _ptr(y), M, N, K, _ptr(workspace), ws_bytes,
                                       _stream(stream)))
    return y


def jq_debug_wait_timeout(stream=None) -> None:
    """Enqueues the failure-handling probe: a kernel whose bounded wait runs out after about a
    second and records JQ_ERR_TIMEOUT for jq_device_status (nothing faults or hangs)."""
    _check("jq_debug_wait_timeout", _load().jq_debug_wait_timeout(_stream(stream)))


def jq_device_status(reset: bool = True, stream=None) -> int:
    """Synchronises the stream; returns the library's status code (5 = a kernel timed out)."""
    return int(_load().jq_device_status(_stream(stream), 1 if reset else 0))


def jq_fake_quant_act(x: torch.Tensor, group: int, s_in: torch.Tensor | None = None, stream=None):
    """Training-side fake quantisation of bf16 activations [M, K] (dense rows).

    Returns (xhat bf16 [M, K], mask uint8 [M, K], scales fp32 [M, K/G]); s_in, if given, is
    [M, K/G] fp32 positive scales used in place of the amax/7 rule."""
    fn = "jq_fake_quant_act"
    _expect_x(fn, x)
    M, K = x.shape
    if not x.is_contiguous():
        raise ValueError(f"{fn}: x must have dense rows")
    _expect(fn, "s_in", s_in, torch.float32, (M, _groups(K, group)), x.device)
    _need_cuda(x, stream=stream)
    xhat = torch.empty((M, K), dtype=torch.bfloat16, device=x.device)
    mask = torch.empty((M, K), dtype=torch.uint8, device=x.device)
    s_out = torch.empty((M, K // group if group else 0), dtype=torch.float32, device=x.device)
    _check(fn, _load().jq_fake_quant_act(_ptr(x), M, K, group, _ptr(s_in), _ptr(xhat), _ptr(mask), _ptr(s_out),
                                         _stream(stream)))
    return xhat, mask, s_out


def jq_fake_quant_weight(w: torch.Tensor, group: int, s_in: torch.Tensor | None = None, stream=None):
    """Training-side fake quantisation of fp32 weights [N, K]: (what fp32 [N, K], mask uint8 [N, K],
    scales fp32 [N, K/G]); s_in, if given, is [N, K/G] fp32 positive scales."""
    fn = "jq_fake_quant_weight"
    if w.dim() != 2:
        raise ValueError(f"{fn}: w must be 2-D, got shape {list(w.shape)}")
    N, K = w.shape
    _expect(fn, "w", w, torch.float32, (N, K), w.device)
    _expect(fn, "s_in", s_in, torch.float32, (N, _groups(K, group)), w.device)
    _need_cuda(w, stream=stream)
    what = torch.empty((N, K), dtype=torch.float32, device=w.device)
    mask = torch.empty((N, K), dtype=torch.uint8, device=w.device)
    s_out = torch.empty((N, K // group if group else 0), dtype=torch.float32, device=w.device)
    _check(fn, _load().jq_fake_quant_weight(_ptr(w), N, K, group, _ptr(s_in), _ptr(what), _ptr(mask), _ptr(s_out),
                                            _stream(stream)))
    return what, mask, s_out


def jq_ste_backward(grad: torch.Tensor, mask: torch.Tensor, stream=None):
    """Straight-through backward: the bf16 gradient where mask != 0, +0 elsewhere (same shape)."""
    fn = "jq_ste_backward"
    if grad.dtype != torch.bfloat16 or not grad.is_contiguous():
        raise ValueError(f"{fn}: grad must be a contiguous bf16 tensor")
    _expect(fn, "mask", mask, torch.uint8, tuple(grad.shape), grad.device)
    if mask is None:
        raise ValueError(f"{fn}: mask is required")
    _need_cuda(grad, mask, stream=stream)
    out = torch.empty_like(grad)
    _check(fn, _load().jq_ste_backward(_ptr(grad), _ptr(mask), grad.numel(), _ptr(out), _stream(stream)))
    return out
