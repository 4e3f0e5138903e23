"""Ordering under programmatic dependent launch: the layer's kernels may be
scheduled before their predecessor in the stream ends, so each must wait for
it before touching global memory. Back-to-back layer calls that share one
workspace (the second call's router overwrites the k / ids / gates the first
call's combine reads) and plain torch kernels that rewrite the input in place
between calls must give exactly the outputs of the same calls run one at a
time with a synchronisation in between."""
import numpy as np
import pytest

from paper_2608_04401_gb300 import synth

from gpu_util import to_dev_bf16

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def moe():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2608_04401_gb300 as m
    m.build()
    m.library()
    return m


@pytest.mark.parametrize("T", [8, 64, 300])
def test_back_to_back_layers_with_input_rewrites(moe, T):
    import torch
    d, N, I, K = 512, 64, 256, 8
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=4242 + T)
    x = to_dev_bf16(inp["x"])
    wr = to_dev_bf16(inp["w_router"])
    wgu = to_dev_bf16(inp["w_gate_up"])
    wd = to_dev_bf16(inp["w_down"])
    ws = torch.empty(moe.layer_workspace_size(T, d, N, I, K), dtype=torch.uint8, device="cuda")
    scales = [1.0, -0.5, 2.0, 0.25]

    # reference: each call alone, with a synchronisation around it
    ref = []
    for sc in scales:
        xi = (x.float() * sc).to(torch.bfloat16)
        torch.cuda.synchronize()
        y, _ = moe.moe_layer_forward(xi, wr, wgu, wd, K=K, ws=ws, return_intermediates=True)
        torch.cuda.synchronize()
        ref.append(y.clone())

    # the same calls back to back on one stream, the input rewritten in place
    # by torch kernels between them, no synchronisation until the end
    xs = x.clone()
    outs = []
    ys = [torch.empty(T, d, dtype=torch.bfloat16, device="cuda") for _ in scales]
    for sc, y in zip(scales, ys):
        xs.copy_((x.float() * sc).to(torch.bfloat16))
        moe.moe_layer_forward(xs, wr, wgu, wd, K=K, y=y, ws=ws)
        outs.append(y)
    torch.cuda.synchronize()
    moe.read_device_error(ws)
    for i, (a, b) in enumerate(zip(outs, ref)):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16)), f"call {i} differs"


def test_graph_replays_with_input_rewrites(moe):
    """A captured layer replayed after the input changed sees the new input."""
    import torch
    T, d, N, I, K = 256, 512, 64, 256, 8
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=77)
    x = to_dev_bf16(inp["x"])
    wr = to_dev_bf16(inp["w_router"])
    wgu = to_dev_bf16(inp["w_gate_up"])
    wd = to_dev_bf16(inp["w_down"])
    ws = torch.empty(moe.layer_workspace_size(T, d, N, I, K), dtype=torch.uint8, device="cuda")
    xs = x.clone()
    y = torch.empty(T, d, dtype=torch.bfloat16, device="cuda")
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        moe.moe_layer_forward(xs, wr, wgu, wd, K=K, y=y, ws=ws)
    torch.cuda.current_stream().wait_stream(side)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        moe.moe_layer_forward(xs, wr, wgu, wd, K=K, y=y, ws=ws)
    for sc in (1.0, -2.0, 0.5):
        xs.copy_((x.float() * sc).to(torch.bfloat16))
        g.replay()
        got = y.clone()
        torch.cuda.synchronize()
        ref, _ = moe.moe_layer_forward(xs, wr, wgu, wd, K=K, return_intermediates=True)
        torch.cuda.synchronize()
        assert torch.equal(got.view(torch.int16), ref.view(torch.int16)), f"scale {sc}"
