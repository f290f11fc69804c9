"""GPU: layers chained on one stream with no host synchronisation in between.

The kernels use programmatic dependent launch: a kernel may start while the previous one in the
stream is still running (the linear layer starts streaming its weights during the activation
quantiser) and waits for it before touching data that kernel writes or reads.  These tests chain
three layers, each layer's output being the next layer's input, and reuse one set of code and
scale buffers for every layer, so that a missing wait would show up as a read of a half-written
or already-overwritten buffer.  The results must be bit-identical to the same calls with a
device synchronisation after each one (which the parity tests check against the oracle), both
when issued eagerly and when replayed from a CUDA graph.
"""
import numpy as np
import pytest
import torch

import paper_2609_33601_gb300 as jq
from paper_2609_33601_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

LAYERS = 3


@pytest.fixture(scope="module", autouse=True)
def _device():
    assert torch.cuda.is_available(), "the gpu tests need a CUDA device"
    jq._load()
    yield
    assert jq.jq_device_status() == 0


def _layers(K, G, seed):
    out = []
    for layer in range(LAYERS):
        w = wl.make("custom", seed=seed + layer, M=1, K=K, N=K, G=G, bias=True)
        qw, sw = jq.jq_pack_weight(torch.from_numpy(w.w).cuda(), G)
        out.append((qw, sw, torch.from_numpy(w.bias).cuda()))
    torch.cuda.synchronize()
    return out


def _bits(t):
    return t.view(torch.int16).cpu().numpy()


# M <= 64 runs the few-token kernel, larger M the GEMM (operand expansion + tcgen05 GEMM)
@pytest.mark.parametrize("M,K,G", [(1, 4096, 4096), (16, 2048, 128), (64, 1024, 64), (300, 2048, 128),
                                   (300, 2048, 2048), (520, 1024, 64)])
def test_chained_layers_match_synchronised_calls(M, K, G):
    layers = _layers(K, G, seed=M + K + G)
    x0 = wl.make("custom", seed=7 * M + G, M=M, K=K, N=8, G=G, with_weights=False).x_bits
    x0 = torch.from_numpy(x0.view(np.int16)).cuda().view(torch.bfloat16)
    q = torch.empty((M, K // 2), dtype=torch.uint8, device="cuda")
    s_a = torch.empty((M, K // G), dtype=torch.float32, device="cuda")
    ws = torch.empty(max(jq.jq_workspace_size(M, K, K, G, False), 16), dtype=torch.uint8, device="cuda")
    ys = [torch.empty((M, K), dtype=torch.bfloat16, device="cuda") for _ in range(LAYERS)]

    def chain(sync, stream=None):
        x = x0
        for (qw, sw, b), y in zip(layers, ys):
            jq.jq_quantize_act(x, G, q, s_a, stream=stream)
            if sync:
                torch.cuda.synchronize()
            jq.jq_w4a4_linear(q, s_a, qw, sw, b, G, y=y, workspace=ws, stream=stream)
            if sync:
                torch.cuda.synchronize()
            x = y

    chain(sync=True)
    ref = [_bits(y) for y in ys]
    for y in ys:
        y.fill_(0)
    torch.cuda.synchronize()
    for _ in range(3):
        chain(sync=False)
    torch.cuda.synchronize()
    for layer, (r, y) in enumerate(zip(ref, ys)):
        assert np.array_equal(r, _bits(y)), f"layer {layer}: eager chain differs from synchronised calls"

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        chain(sync=False, stream=s)
    for y in ys:
        y.fill_(0)
    torch.cuda.synchronize()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    for layer, (r, y) in enumerate(zip(ref, ys)):
        assert np.array_equal(r, _bits(y)), f"layer {layer}: graph replay differs from synchronised calls"
