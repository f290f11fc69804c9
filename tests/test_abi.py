"""Host-side checks of the C ABI (no GPU needed): the library builds and loads, exports every
entry point include/jq.h declares, and rejects bad arguments synchronously, before touching a
device, with the documented status codes."""
import ctypes
import os
import re

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "jq.h")

OK, INVALID, MISALIGNED, UNSUPPORTED, CUDA, TIMEOUT, WORKSPACE = range(7)


@pytest.fixture(scope="module")
def lib():
    from paper_2609_33601_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(jq_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for need in ("jq_quantize_act", "jq_pack_weight", "jq_w4a4_linear", "jq_fused_quant_linear",
                 "jq_status_string", "jq_workspace_size", "jq_w4a4_group_partials", "jq_device_status",
                 "jq_pack_weight_ternary", "jq_w158a4_linear", "jq_w158a4_workspace_size"):
        assert need in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    lib.jq_status_string.restype = ctypes.c_char_p
    lib.jq_status_string.argtypes = [ctypes.c_int]
    names = [lib.jq_status_string(i).decode() for i in range(7)]
    assert names == ["JQ_OK", "JQ_ERR_INVALID_ARG", "JQ_ERR_MISALIGNED", "JQ_ERR_UNSUPPORTED", "JQ_ERR_CUDA",
                     "JQ_ERR_TIMEOUT", "JQ_ERR_WORKSPACE"]


def test_workspace_size(lib):
    f = lib.jq_workspace_size
    f.argtypes = [ctypes.c_int64] * 3 + [ctypes.c_int32] * 2
    f.restype = ctypes.c_size_t
    # operand image (whole 128-row tiles of K bytes), then one fp32 per token and group (the
    # activation-sum corrections), then for the fused path the activation scales; 256-byte parts
    assert f(1024, 12288, 4096, 128, 0) == 1024 * 4096 + 1024 * 32 * 4
    assert f(1024, 12288, 4096, 128, 1) == 1024 * 4096 + 2 * 1024 * 32 * 4
    assert f(3, 8, 256, 64, 0) == 128 * 256 + 256
    assert f(0, 8, 256, 64, 0) == 0


def _fake(addr):
    return ctypes.c_void_p(addr)


def test_argument_checks_reject_before_launch(lib):
    i64, i32, vp, sz = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_size_t
    lib.jq_quantize_act.argtypes = [vp, i64, i64, i64, i32, vp, vp, vp]
    lib.jq_pack_weight.argtypes = [vp, i64, i64, i32, vp, vp, vp]
    lib.jq_w4a4_linear.argtypes = [vp, vp, vp, vp, vp, vp, i64, i64, i64, i32, vp, sz, vp]
    lib.jq_fused_quant_linear.argtypes = [vp, i64, vp, vp, vp, vp, i64, i64, i64, i32, vp, sz, vp]
    A = _fake(0x10000)       # 16-byte aligned fake device addresses: never dereferenced here
    odd = _fake(0x10008)
    q = lib.jq_quantize_act
    assert q(None, 4, 256, 256, 64, A, A, None) == INVALID
    assert q(A, 4, 256, 256, 32, A, A, None) == INVALID          # unsupported group
    assert q(A, 4, 192, 192, 64, A, A, None) == INVALID          # K % 128 != 0
    assert q(A, 4, 256, 128, 64, A, A, None) == INVALID          # ldx < K
    assert q(A, -1, 256, 256, 64, A, A, None) == INVALID
    assert q(A, 0, 256, 256, 64, None, None, None) == OK         # M == 0 is a no-op
    assert q(odd, 4, 256, 256, 64, A, A, None) == MISALIGNED
    assert q(A, 4, 256, 260, 64, A, A, None) == MISALIGNED       # row pitch 520 B
    assert q(A, 4, 262144, 262144, 262144, A, A, None) == INVALID  # K too large for exact sums
    p = lib.jq_pack_weight
    assert p(None, 8, 256, 64, A, A, None) == INVALID
    assert p(A, 8, 256, 100, A, A, None) == INVALID
    assert p(A, 8, 256, 64, odd, A, None) == MISALIGNED
    L = lib.jq_w4a4_linear
    big = 1 << 30
    assert L(A, A, A, A, None, A, 4, 12, 256, 64, A, big, None) == INVALID     # N % 8
    assert L(A, A, A, A, None, A, 4, 16, 256, 96, A, big, None) == INVALID     # group
    assert L(None, A, A, A, None, A, 4, 16, 256, 64, A, big, None) == INVALID
    assert L(A, A, A, A, odd, A, 4, 16, 256, 64, A, big, None) == MISALIGNED   # bias
    assert L(A, A, A, A, None, A, 4, 16, 256, 64, None, big, None) == WORKSPACE
    assert L(A, A, A, A, None, A, 4, 16, 256, 64, A, 16, None) == WORKSPACE
    assert L(A, A, A, A, None, A, 0, 16, 256, 64, None, 0, None) == OK        # M == 0
    F = lib.jq_fused_quant_linear
    assert F(A, 200, A, A, None, A, 4, 16, 256, 64, A, big, None) == INVALID   # ldx < K
    assert F(A, 260, A, A, None, A, 4, 16, 256, 64, A, big, None) == MISALIGNED
    assert F(A, 256, A, A, None, A, 4, 16, 256, 64, A, 1024, None) == WORKSPACE


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-device path; a GPU is present")
def test_valid_arguments_without_a_device_report_unsupported(lib):
    i64, i32, vp = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p
    lib.jq_quantize_act.argtypes = [vp, i64, i64, i64, i32, vp, vp, vp]
    A = _fake(0x10000)
    assert lib.jq_quantize_act(A, 4, 256, 256, 64, A, A, None) == UNSUPPORTED
    lib.jq_debug_wait_timeout.argtypes = [vp]
    assert lib.jq_debug_wait_timeout(None) == UNSUPPORTED  # the failure probe launches nothing either


def test_binding_fails_loudly_without_cuda_tensors():
    import paper_2609_33601_gb300 as jq
    x = torch.zeros((4, 256), dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        jq.jq_quantize_act(x, 64)


def test_w158a4_entry_points(lib):
    i64, i32, vp, sz = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_size_t
    lib.jq_pack_weight_ternary.argtypes = [vp, i64, i64, i32, vp, vp, vp]
    lib.jq_w158a4_linear.argtypes = [vp, vp, vp, vp, vp, vp, i64, i64, i64, i32, vp, sz, vp]
    lib.jq_w158a4_workspace_size.argtypes = [i64, i64, i64, i32]
    lib.jq_w158a4_workspace_size.restype = sz
    lib.jq_workspace_size.argtypes = [i64, i64, i64, i32, i32]
    lib.jq_workspace_size.restype = sz
    ws, ws4 = lib.jq_w158a4_workspace_size, lib.jq_workspace_size
    # as the INT4 linear at every size: both kernels read the 2-bit codes in place
    assert ws(64, 12288, 4096, 128) == ws4(64, 12288, 4096, 128, 0)
    assert ws(1024, 12288, 4096, 128) == ws4(1024, 12288, 4096, 128, 0)
    assert ws(4608, 3072, 15360, 15360) == ws4(4608, 3072, 15360, 15360, 0)
    assert ws(0, 8, 256, 64) == 0
    A, odd = _fake(0x10000), _fake(0x10008)
    P = lib.jq_pack_weight_ternary
    assert P(None, 8, 256, 64, A, A, None) == INVALID
    assert P(A, 8, 256, 100, A, A, None) == INVALID
    assert P(A, 8, 192, 64, A, A, None) == INVALID
    assert P(A, 8, 256, 64, odd, A, None) == MISALIGNED
    assert P(A, 0, 256, 64, None, None, None) == OK
    L = lib.jq_w158a4_linear
    big = 1 << 30
    assert L(A, A, A, A, None, A, 4, 12, 256, 64, A, big, None) == INVALID     # N % 8
    assert L(None, A, A, A, None, A, 4, 16, 256, 64, A, big, None) == INVALID
    assert L(A, A, odd, A, None, A, 4, 16, 256, 64, A, big, None) == MISALIGNED
    assert L(A, A, A, A, None, A, 100, 16, 256, 64, A, 16, None) == WORKSPACE
    assert L(A, A, A, A, None, A, 0, 16, 256, 64, None, 0, None) == OK


C_CLIENT = r"""
#include <stdio.h>
#include <string.h>
#include "jq.h"

int main(void) {
  int bad = 0;
  if (strcmp(jq_status_string(JQ_ERR_WORKSPACE), "JQ_ERR_WORKSPACE") != 0) bad |= 1;
  if (jq_workspace_size(1024, 12288, 4096, 128, 0) != (size_t)1024 * 4096 + 1024 * 32 * 4) bad |= 2;
  /* argument checks run before any device is touched */
  if (jq_w4a4_linear(NULL, NULL, NULL, NULL, NULL, NULL, 16, 256, 4096, 128, NULL, 0, NULL) != JQ_ERR_INVALID_ARG)
    bad |= 4;
  if (jq_quantize_act(NULL, 4, 100, 100, 64, NULL, NULL, NULL) != JQ_ERR_INVALID_ARG) bad |= 8;
  if (jq_w4a4_linear(NULL, NULL, NULL, NULL, NULL, NULL, 0, 256, 4096, 128, NULL, 0, NULL) != JQ_OK) bad |= 16;
  printf("%d\n", bad);
  return bad;
}
"""


def test_header_is_plain_c_and_links_from_a_c_program(lib, tmp_path):
    """A C99 client compiled with gcc -pedantic -Werror against include/jq.h links to libjq.so
    and gets the documented answers from calls that need no GPU."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    from paper_2609_33601_gb300 import build
    libpath = build.build()
    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    subprocess.run([gcc, "-std=c99", "-pedantic", "-Wall", "-Wextra", "-Werror", "-I", os.path.dirname(HEADER),
                    str(src), "-o", str(exe), libpath, f"-Wl,-rpath,{os.path.dirname(libpath)}"],
                   check=True, capture_output=True, text=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "0", (r.returncode, r.stdout, r.stderr)


def test_fake_quant_and_ste_entry_points_check_arguments(lib):
    i64, i32, vp = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p
    lib.jq_fake_quant_act.argtypes = [vp, i64, i64, i32, vp, vp, vp, vp, vp]
    lib.jq_ste_backward.argtypes = [vp, vp, i64, vp, vp]
    A = _fake(0x10000)
    odd = _fake(0x10008)
    fq = lib.jq_fake_quant_act
    assert fq(None, 4, 256, 64, None, A, A, A, None) == INVALID
    assert fq(A, 4, 256, 64, None, A, None, A, None) == INVALID      # the mask is required
    assert fq(A, 4, 256, 32, None, A, A, A, None) == INVALID         # unsupported group
    assert fq(A, 4, 192, 64, None, A, A, A, None) == INVALID         # K % 128 != 0
    assert fq(A, -1, 256, 64, None, A, A, A, None) == INVALID
    assert fq(A, 0, 256, 64, None, None, None, None, None) == OK     # M == 0 is a no-op
    assert fq(A, 4, 256, 64, odd, A, A, A, None) == MISALIGNED       # given scales
    assert fq(A, 4, 256, 64, None, A, odd, A, None) == MISALIGNED    # mask
    lib.jq_fake_quant_weight.argtypes = [vp, i64, i64, i32, vp, vp, vp, vp, vp]
    fw = lib.jq_fake_quant_weight
    assert fw(None, 4, 256, 64, None, A, A, A, None) == INVALID
    assert fw(A, 4, 256, 96, None, A, A, A, None) == INVALID
    assert fw(A, 0, 256, 64, None, None, None, None, None) == OK
    assert fw(A, 4, 256, 64, None, odd, A, A, None) == MISALIGNED
    if not torch.cuda.is_available():
        assert fw(A, 4, 256, 64, None, A, A, A, None) == UNSUPPORTED
    st = lib.jq_ste_backward
    assert st(A, A, -1, A, None) == INVALID
    assert st(None, A, 8, A, None) == INVALID
    assert st(A, A, 0, None, None) == OK                             # n == 0 is a no-op
    assert st(A, odd, 8, A, None) == MISALIGNED
    if not torch.cuda.is_available():
        assert fq(A, 4, 256, 64, None, A, A, A, None) == UNSUPPORTED
        assert st(A, A, 13, A, None) == UNSUPPORTED


def test_fake_quant_binding_refuses_wrong_tensors():
    import paper_2609_33601_gb300 as jq
    x = torch.zeros((4, 256), dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="s_in"):
        jq.jq_fake_quant_act(x, 64, torch.zeros((4, 3), dtype=torch.float32))
    with pytest.raises(ValueError, match="dense rows"):
        jq.jq_fake_quant_act(torch.zeros((4, 512), dtype=torch.bfloat16)[:, :256], 64)
    with pytest.raises(ValueError, match="CUDA tensors only"):
        jq.jq_fake_quant_act(x, 64)
    with pytest.raises(ValueError, match="s_in"):
        jq.jq_fake_quant_weight(torch.zeros((8, 256)), 128, torch.zeros((8, 1)))
    with pytest.raises(ValueError, match="CUDA tensors only"):
        jq.jq_fake_quant_weight(torch.zeros((8, 256)), 128)
    with pytest.raises(ValueError, match="mask"):
        jq.jq_ste_backward(x, torch.zeros((4, 255), dtype=torch.uint8))
    with pytest.raises(ValueError, match="CUDA tensors only"):
        jq.jq_ste_backward(x, torch.zeros((4, 256), dtype=torch.uint8))


def test_dit_neighbour_entry_points_check_arguments(lib):
    """jq_modulate_quantize_act / jq_gelu_quantize_act refuse bad arguments before any launch."""
    vp = ctypes.c_void_p
    lib.jq_modulate_quantize_act.argtypes = [vp, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, vp, vp,
                                             ctypes.c_int64, ctypes.c_int32, vp, vp, vp]
    lib.jq_gelu_quantize_act.argtypes = [vp, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int32, vp, vp,
                                         vp]
    p = vp(4096)
    odd = vp(4100)
    mod = lib.jq_modulate_quantize_act
    assert mod(p, 4, 256, 256, p, p, 1, 64, p, p, None) == 3          # valid: no sm_103 device here
    assert mod(p, 0, 256, 256, p, p, 1, 64, p, p, None) == 0          # empty batch
    assert mod(p, 4, 256, 256, p, p, 0, 64, p, p, None) == 1          # tokens_per_sample <= 0
    assert mod(p, 4, 256, 256, None, p, 1, 64, p, p, None) == 1       # no shift
    assert mod(p, 4, 256, 256, p, None, 1, 64, p, p, None) == 1       # no scale
    assert mod(p, 4, 256, 128, p, p, 1, 64, p, p, None) == 1          # ldx < K
    assert mod(p, 4, 256, 256, p, p, 1, 96, p, p, None) == 1          # unsupported group
    assert mod(p, 4, 256, 256, odd, p, 1, 64, p, p, None) == 2        # misaligned x
    assert mod(p, 4, 256, 256, p, odd, 1, 64, p, p, None) == 2        # misaligned shift
    gelu = lib.jq_gelu_quantize_act
    assert gelu(p, 4, 256, 256, 128, p, p, None) == 3
    assert gelu(p, 4, 256, 260, 128, p, p, None) == 2                 # ldh * 2 not a multiple of 16
    assert gelu(None, 4, 256, 256, 128, p, p, None) == 1
    assert gelu(p, 4, 200, 256, 128, p, p, None) == 1                 # K not a multiple of 128


def test_nvfp4_entry_points_check_arguments(lib):
    """jq_nvfp4_quantize_act / _pack_weight / _linear refuse bad arguments before any launch."""
    vp, i64, f32, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
    lib.jq_nvfp4_quantize_act.argtypes = [vp, i64, i64, i64, f32, vp, vp, vp]
    lib.jq_nvfp4_pack_weight.argtypes = [vp, i64, i64, vp, vp, vp, vp]
    lib.jq_nvfp4_linear.argtypes = [vp, vp, f32, vp, vp, vp, vp, vp, i64, i64, i64, vp, sz, vp]
    lib.jq_nvfp4_workspace_size.argtypes = [i64, i64, i64]
    lib.jq_nvfp4_workspace_size.restype = sz
    p, odd = vp(4096), vp(4100)
    qa = lib.jq_nvfp4_quantize_act
    assert qa(p, 4, 192, 192, 0.01, p, p, None) == 3               # valid (K % 64 == 0): no sm_103 device here
    assert qa(p, 0, 192, 192, 0.01, p, p, None) == 0               # empty batch
    assert qa(p, 4, 200, 200, 0.01, p, p, None) == 1               # K not a multiple of 64
    assert qa(p, 4, 192, 128, 0.01, p, p, None) == 1               # ldx < K
    assert qa(p, 4, 192, 192, -1.0, p, p, None) == 1               # negative tensor scale
    assert qa(p, 4, 192, 192, float("inf"), p, p, None) == 1       # infinite tensor scale
    assert qa(p, 4, 192, 192, float("nan"), p, p, None) == 1       # NaN tensor scale
    assert qa(odd, 4, 192, 192, 0.01, p, p, None) == 2             # misaligned x
    assert qa(p, 4, 192, 196, 0.01, p, p, None) == 2               # ldx * 2 not a multiple of 16
    pw = lib.jq_nvfp4_pack_weight
    assert pw(p, 8, 128, p, p, p, None) == 3
    assert pw(p, 8, 128, p, p, None, None) == 1                    # no output for g_w
    assert pw(p, 8, 128, p, p, odd, None) == 2
    need = lib.jq_nvfp4_workspace_size(64, 256, 128)
    assert need == 128 * 128 * 2 + 256 * 128 * 2                  # two bf16 operand images, whole 128-row tiles
    assert lib.jq_nvfp4_workspace_size(64, 256, 100) == 0
    ln = lib.jq_nvfp4_linear
    assert ln(p, p, 1.0, p, p, p, None, p, 64, 256, 128, p, need, None) == 3
    assert ln(p, p, 1.0, p, p, p, None, p, 64, 252, 128, p, need, None) == 1   # N % 8 != 0
    assert ln(p, p, 1.0, p, p, None, None, p, 64, 256, 128, p, need, None) == 1  # no g_w
    assert ln(p, p, 1.0, p, p, p, None, p, 64, 256, 128, p, need - 1, None) == 6  # short workspace
    assert ln(p, p, 1.0, p, p, p, None, odd, 64, 256, 128, p, need, None) == 2   # misaligned y
    assert ln(p, p, 1.0, p, p, p, None, p, 0, 256, 128, None, 0, None) == 0      # empty
