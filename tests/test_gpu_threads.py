"""First use of the library from two host threads at once (GPU).

The launchers set kernel attributes and probe occupancy once per device, under a mutex
(kernels.cuh, PerDevice), and the device probe behind every call is locked the same way.  A
fresh process is needed for a true first use, so the check runs in a child process: two threads
each make their first calls at the same moment, on their own streams -- one a GEMM-sized
problem, one a few-token problem -- and both results must match the oracle.
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys, threading
sys.path.insert(0, ROOT)
import numpy as np, torch
import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl
from tests.helpers import Reference, check_linear

torch.cuda.set_device(0)
cases = [dict(M=300, K=1024, N=520, G=64), dict(M=40, K=2048, N=264, G=128),
         dict(M=300, K=1024, N=520, G=1024), dict(M=9, K=512, N=136, G=512)]
refs, inputs = [], []
for i, c in enumerate(cases):
    w = wl.make("custom", seed=40 + i, bias=True, **c)
    ref = Reference(w.x_bits, w.w, w.bias, c["G"])
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    refs.append(ref)
    inputs.append((dev(ref.packed_a), dev(ref.s_a), dev(ref.packed_w), dev(ref.s_w_groupmajor), dev(ref.bias)))
torch.cuda.synchronize()
start = threading.Barrier(2)
out = [None] * len(cases)
errors = []

def worker(t):
    try:
        torch.cuda.set_device(0)
        st = torch.cuda.Stream()
        start.wait()
        with torch.cuda.stream(st):
            for i in range(t, len(cases), 2):  # thread 0: the two GEMM cases, thread 1: the few-token ones
                out[i] = jq.jq_w4a4_linear(*inputs[i], refs[i].G, stream=st)
        st.synchronize()
    except Exception as e:  # reported by the main thread
        errors.append(repr(e))

ts = [threading.Thread(target=worker, args=(t,)) for t in range(2)]
[t.start() for t in ts]
[t.join() for t in ts]
assert not errors, errors
assert jq.jq_device_status() == 0
for i, ref in enumerate(refs):
    y = out[i].view(torch.int16).cpu().numpy().view(np.uint16)
    y64, _ = ref.linear()
    check_linear(y, y64, ref.partials(), ref.s_a, ref.s_w_rows, ref.bias, f"thread case {i}")
print("threads ok")
"""


def test_first_calls_from_two_threads_at_once():
    code = "ROOT = %r\n" % ROOT + CHILD
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0 and "threads ok" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]
