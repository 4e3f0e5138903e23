"""GPU parity of the decode-shaped expert GEMMs (T <= 64: weights as the M
operand, the expert's rows as N) against numpy fp64 on the same dispatch,
including expert sizes 0, 1, 31-33, 63 and 64 rows, and of the whole layer at
decode sizes (T = 1 ... 64, which moe_layer_forward routes to these GEMMs, and
T = 65, which it does not) against the oracle."""
import numpy as np
import pytest

import oracle
from paper_2608_04401_gb300 import synth

from gpu_util import assert_layer_close, bf16_tensor_to_f64, to_dev, to_dev_bf16

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


def f64(bits):
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


def _swiglu64(xs, wgu, I):
    g = xs @ wgu[:I].T
    u = xs @ wgu[I:].T
    return g / (1.0 + np.exp(-g)) * u


@pytest.mark.parametrize("N,d,I,case,T", [
    (64, 512, 256, "random", 64),
    (64, 2048, 1024, "random", 64),
    (128, 1024, 512, "random", 64),
    (64, 512, 256, "edges", 64),
    (64, 512, 256, "random", 1),
    (64, 1024, 512, "random", 16),
    (128, 512, 256, "random", 32),
    (64, 512, 256, "edges", 16),
    (64, 512, 256, "edges", 32),
])
def test_decode_gemm_steps(moe, N, d, I, case, T):
    """T <= 16, <= 32 and <= 64 take 16-, 32- and 64-column token tiles."""
    import torch
    rng = np.random.default_rng(N + d + I + T)
    K = 8
    if case == "random":
        r = oracle.route(synth.boosted_logits(rng, T, N), K=K)
        k, ids = r["k"], r["ids"]
    else:
        # expert e has sizes[e] rows: tokens t < sizes[e] select it
        # (capped at T, plus one expert of T - 1 rows: the full and the
        # one-short tile of each width)
        sizes = {0: 64, 2: 1, 5: 31, 6: 32, 7: 33, 9: 63, N - 1: 64}
        sizes = {e: min(n, T) for e, n in sizes.items()}
        sizes[3] = T - 1
        ids = np.zeros((T, K), np.int32)
        k = np.zeros(T, np.int32)
        for t in range(T):
            mine = [e for e, s in sizes.items() if t < s]
            k[t] = len(mine)
            rest = [e for e in range(N) if e not in mine][: K - len(mine)]
            ids[t] = mine + rest
    x = synth.bf16_bits(rng.standard_normal((T, d)).astype(np.float32))
    wgu, wd = synth.expert_weights(N + 7, N, d, I)
    off, perm, pp, ws = moe.moe_dispatch(to_dev(k), to_dev(ids), N)
    P = T * K
    xs = moe.gather_rows(to_dev_bf16(x), perm, off, P)
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    h = moe.expert_gate_up_decode(xs, to_dev_bf16(wgu), off, T, err=err)
    o = moe.expert_down_decode(h, to_dev_bf16(wd), off, T, err=err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    offs = off.cpu().numpy()
    n = int(offs[-1])
    xsf = f64(x)[perm.cpu().numpy()[:n]]
    h_ref = np.zeros((n, I))
    o_ref = np.zeros((n, d))
    for e in range(N):
        a, b = offs[e], offs[e + 1]
        assert b - a <= T
        if b > a:
            h_ref[a:b] = _swiglu64(xsf[a:b], f64(wgu[e]), I)
            o_ref[a:b] = h_ref[a:b] @ f64(wd[e]).T
    assert_layer_close(bf16_tensor_to_f64(h[:n]), h_ref, "h")
    # down GEMM on the GPU's own h (isolates the down contraction)
    o_own = bf16_tensor_to_f64(h[:n]).astype(np.float64)
    o_ref2 = np.zeros((n, d))
    for e in range(N):
        a, b = offs[e], offs[e + 1]
        if b > a:
            o_ref2[a:b] = o_own[a:b] @ f64(wd[e]).T
    assert_layer_close(bf16_tensor_to_f64(o[:n]), o_ref2, "o")
    assert_layer_close(bf16_tensor_to_f64(o[:n]), o_ref, "o vs fp64 chain")


def test_decode_gemm_rejects_large_batches(moe):
    import torch
    xs = torch.zeros(65 * 8, 512, dtype=torch.bfloat16, device="cuda")
    w = torch.zeros(64, 512, 512, dtype=torch.bfloat16, device="cuda")
    off = torch.zeros(65, dtype=torch.int32, device="cuda")
    with pytest.raises(moe.MoeError):
        moe.expert_gate_up_decode(xs, w, off, 65)


@pytest.mark.parametrize("T", [1, 2, 17, 63, 64, 65])
def test_layer_decode_sizes(moe, T):
    """The whole layer at decode sizes: every token against the oracle (GPU
    routing bit-exact on its own logits, outputs within the tolerance)."""
    import torch
    inp = synth.layer_inputs(T=T, d=2048, N=64, I=1024, seed=500 + T)
    x = to_dev_bf16(inp["x"])
    ws = torch.empty(moe.layer_workspace_size(T, 2048, 64, 1024, 8), dtype=torch.uint8, device="cuda")
    y, it = moe.moe_layer_forward(x, to_dev_bf16(inp["w_router"]), to_dev_bf16(inp["w_gate_up"]),
                                  to_dev_bf16(inp["w_down"]), K=8, ws=ws, return_intermediates=True)
    moe.read_device_error(ws)
    lg = it["logits"].cpu().numpy()
    # T <= 64: the split router GEMM on CUDA cores; T = 65: the tensor-core router
    ref_lg = oracle.router_logits(inp["x"], inp["w_router"]).astype(np.float64)
    abs_sum = np.abs(f64(inp["x"])) @ np.abs(f64(inp["w_router"])).T
    assert np.all(np.abs(lg.astype(np.float64) - ref_lg) <= 2048 * 2.0 ** -24 * abs_sum + 1e-30)
    r = oracle.route(lg, K=8)
    assert np.array_equal(r["k"], it["k"].cpu().numpy())
    assert np.array_equal(r["ids"], it["ids"].cpu().numpy())
    rows = np.arange(T)
    ref = oracle.layer_rows(inp["x"], inp["w_router"], inp["w_gate_up"], inp["w_down"], rows=rows, K=8)
    same = (ref["k"] == r["k"]) & np.all(ref["ids"] == r["ids"], axis=1)
    assert same.sum() >= max(1, int(0.9 * T))
    assert_layer_close(bf16_tensor_to_f64(y)[same], ref["y"][same])


@pytest.mark.parametrize("T,N,d,I,K,mode", [(16, 128, 1024, 512, 8, 0), (40, 128, 1024, 512, 8, 1),
                                            (9, 64, 512, 256, 4, 0), (64, 64, 512, 256, 2, 0),
                                            (64, 128, 1024, 512, 8, 0), (24, 64, 4096, 128, 8, 0),
                                            (33, 64, 256, 128, 8, 0)])
def test_layer_small_batches_shapes(moe, T, N, d, I, K, mode):
    """Small batches with 128 experts, other caps and top-K mode: the split
    router GEMM with warp routing (its largest shared-memory case at T = 64,
    N = 128; 2 to 32 slices of d), the decode GEMMs, every token vs the
    oracle."""
    import torch
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=900 + T + N)
    ws = torch.empty(moe.layer_workspace_size(T, d, N, I, K), dtype=torch.uint8, device="cuda")
    y, it = moe.moe_layer_forward(to_dev_bf16(inp["x"]), to_dev_bf16(inp["w_router"]),
                                  to_dev_bf16(inp["w_gate_up"]), to_dev_bf16(inp["w_down"]), K=K,
                                  mode=mode, ws=ws, return_intermediates=True)
    moe.read_device_error(ws)
    # the split router GEMM's logits: fp32 sums of d products (64-column
    # slices added in order) within the recursive-sum bound d 2^-24 sum|x w|
    lg = it["logits"].cpu().numpy().astype(np.float64)
    ref_lg = oracle.router_logits(inp["x"], inp["w_router"]).astype(np.float64)
    abs_sum = np.abs(f64(inp["x"])) @ np.abs(f64(inp["w_router"])).T
    assert np.all(np.abs(lg - ref_lg) <= d * 2.0 ** -24 * abs_sum + 1e-30)
    r = oracle.route(it["logits"].cpu().numpy(), K=K, mode=mode)
    assert np.array_equal(r["k"], it["k"].cpu().numpy())
    assert np.array_equal(r["ids"], it["ids"].cpu().numpy())
    assert np.array_equal(r["gates"].view(np.uint32), it["gates"].cpu().numpy().view(np.uint32))
    rows = np.arange(T)
    ref = oracle.layer_rows(inp["x"], inp["w_router"], inp["w_gate_up"], inp["w_down"], rows=rows,
                            K=K, mode=mode)
    same = (ref["k"] == r["k"]) & np.all(ref["ids"] == r["ids"], axis=1)
    assert same.sum() >= max(1, int(0.9 * T))
    assert_layer_close(bf16_tensor_to_f64(y)[same], ref["y"][same])
