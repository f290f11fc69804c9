"""Failure detection on the GPU without a GPU fault.

Every wait in the library's kernels is bounded: after about 2^31 SM cycles it gives up, records
JQ_ERR_TIMEOUT in a device status word and lets the kernel return.  jq_debug_wait_timeout runs
that same bounded wait on an mbarrier phase nothing completes, so the wait runs out for real;
the host must then read JQ_ERR_TIMEOUT, reset it, and keep using the context.  Nothing here
traps, faults or hangs.
"""
import time

import numpy as np
import pytest
import torch

import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl
from tests.helpers import Reference, check_linear

pytestmark = pytest.mark.gpu

JQ_ERR_TIMEOUT = 5


@pytest.mark.slow  # waits about a second by design; runs after the parity tests
def test_a_wait_that_runs_out_is_reported_and_the_context_stays_usable():
    assert torch.cuda.is_available()
    assert jq.jq_device_status(reset=True) == 0
    t0 = time.monotonic()
    jq.jq_debug_wait_timeout()
    assert jq.jq_device_status(reset=True) == JQ_ERR_TIMEOUT  # synchronises the stream
    assert time.monotonic() - t0 < 60  # the wait gave up; nothing hung
    assert jq.jq_device_status() == 0  # reset
    # the context still works: a small linear layer matches the oracle
    w = wl.make("tiny", seed=4)
    ref = Reference(w.x_bits, w.w, w.bias, w.G)
    x = torch.from_numpy(w.x_bits.view(np.int16)).cuda().view(torch.bfloat16)
    qw, sw = jq.jq_pack_weight(torch.from_numpy(w.w).cuda(), w.G)
    y = jq.jq_fused_quant_linear(x, qw, sw, torch.from_numpy(w.bias).cuda(), w.G)
    y64, _ = ref.linear()
    check_linear(y.view(torch.int16).cpu().numpy().view(np.uint16), y64, ref.partials(), ref.s_a, ref.s_w_rows,
                 ref.bias, "after a timeout")
    assert jq.jq_device_status() == 0
