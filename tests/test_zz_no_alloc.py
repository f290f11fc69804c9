"""GPU test of jq_w4a4_linear_noalloc, the entry point for callers that cannot allocate device
memory (a host callback, a plug-in whose framework owns every allocation, a serving loop that
must not allocate after start-up): it keeps its scratch in a fixed device array inside the
library instead of a caller-provided workspace.

Two calls in a row on different shapes, each compared with jq_w4a4_linear (which uses a
workspace) and with the CPU oracle under the tolerance the parity tests use; then the size
limit; then 17-64 tokens, where the few-token kernel converts the tokens itself.  This file is collected last so that a run stopping at the first failure has already run
every other test; it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl
from tests.helpers import Reference, check_linear

pytestmark = pytest.mark.gpu

JQ_ERR_WORKSPACE = 6
MAX_SCRATCH = 16 * 1024 * 1024


@pytest.fixture(scope="module", autouse=True)
def _device():
    assert torch.cuda.is_available(), "the gpu tests need a CUDA device"
    jq._load()
    yield
    assert jq.jq_device_status() == 0


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _bits(y):
    return y.view(torch.int16).cpu().numpy().view(np.uint16)


def _problem(M, N, K, G, bias, seed):
    w = wl.make("custom", seed=seed, M=M, K=K, N=N, G=G, bias=bias)
    ref = Reference(w.x_bits, w.w, w.bias, G)
    args = (_dev(ref.packed_a), _dev(ref.s_a), _dev(ref.packed_w), _dev(ref.s_w_groupmajor),
            None if ref.bias is None else _dev(ref.bias))
    return ref, args


def test_noalloc_matches_workspace_linear_on_two_calls_in_a_row():
    cases = [(300, 520, 512, 64, True, 1), (1024, 264, 4096, 128, False, 2)]
    probs = [_problem(*c) for c in cases]
    # two no-allocation calls back to back, sharing the library's scratch array
    outs = [jq.jq_w4a4_linear_noalloc(*args, ref.G) for ref, args in probs]
    torch.cuda.synchronize()
    for (ref, args), y_na in zip(probs, outs):
        y_ws = jq.jq_w4a4_linear(*args, ref.G)
        a, b = _bits(y_na), _bits(y_ws)
        y64, _ = ref.linear()
        check_linear(a, y64, ref.partials(), ref.s_a, ref.s_w_rows, ref.bias, "noalloc")
        check_linear(b, y64, ref.partials(), ref.s_a, ref.s_w_rows, ref.bias, "workspace")
        assert np.array_equal(a, b)  # same kernels, same operands: identical bits


def test_noalloc_rejects_problems_beyond_its_scratch():
    lib = jq._load()
    small = torch.zeros(256, dtype=torch.uint8, device="cuda")
    p = ctypes.c_void_p(small.data_ptr())
    K = 4096
    M = MAX_SCRATCH // K + 1  # one 128-row tile too many
    rc = lib.jq_w4a4_linear_noalloc(p, p, p, p, None, p, M, 8, K, 128, None)
    assert rc == JQ_ERR_WORKSPACE
    torch.cuda.synchronize()


@pytest.mark.parametrize("M,N,K,G,bias", [(17, 264, 1024, 128, True), (40, 520, 512, 64, False),
                                          (64, 136, 2048, 2048, True)])
def test_noalloc_few_tokens_convert_the_tokens_in_the_kernel(M, N, K, G, bias):
    """Up to 64 tokens the no-allocation call has no workspace for pre-expanded tokens, so the
    few-token kernel converts the packed token codes itself; with more than 16 tokens that is
    the only caller of that form (jq_w4a4_linear hands it the tokens pre-expanded).  Same
    result as jq_w4a4_linear, and within the oracle's tolerance."""
    ref, args = _problem(M, N, K, G, bias, seed=M + 3)
    y_na = _bits(jq.jq_w4a4_linear_noalloc(*args, G))
    y_ws = _bits(jq.jq_w4a4_linear(*args, G))
    y64, _ = ref.linear()
    check_linear(y_na, y64, ref.partials(), ref.s_a, ref.s_w_rows, ref.bias, f"noalloc M={M}")
    assert np.array_equal(y_na, y_ws)


def test_noalloc_largest_accepted_problem_fills_the_scratch():
    """At K = 4096, group128 the scratch holds the operand image (whole 128-row tiles of K bytes)
    and then one fp32 correction per token and group, rounded up to 256 bytes: M = 3968 needs
    16,760,832 of the 16,777,216 bytes, so the corrections end within 17 KB of the array's last
    byte.  That call must give the same bits as jq_w4a4_linear; one more token (M = 3969 starts a
    32nd image tile) must be refused before any launch."""
    K, G, N = 4096, 128, 264
    M = 3968
    assert -(-M // 128) * 128 * K + -(-(4 * M * (K // G)) // 256) * 256 == 16_760_832 <= MAX_SCRATCH
    ref, args = _problem(M, N, K, G, True, seed=9)
    y_na = _bits(jq.jq_w4a4_linear_noalloc(*args, G))
    y_ws = _bits(jq.jq_w4a4_linear(*args, G))
    assert np.array_equal(y_na, y_ws)
    rows = np.array([0, 1, 2047, 3840, M - 1])
    y64, _ = ref.linear(rows)
    check_linear(y_na[rows], y64, ref.partials(rows), ref.s_a[rows], ref.s_w_rows, ref.bias, "noalloc M=3968")
    lib = jq._load()
    small = torch.zeros(256, dtype=torch.uint8, device="cuda")
    p = ctypes.c_void_p(small.data_ptr())
    assert lib.jq_w4a4_linear_noalloc(p, p, p, p, None, p, M + 1, N, K, G, None) == JQ_ERR_WORKSPACE
    torch.cuda.synchronize()
