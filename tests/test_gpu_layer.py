"""GPU parity of the layer's contractions and of the whole MoE layer forward
against the CPU oracle (and numpy fp64 for the isolated GEMM steps).

Routing inside the layer runs on the GPU's fp32 router logits, which differ
from the oracle's fp64-accumulated logits in the last bits; a token whose
elbow decision flips is counted (the flip fraction is bounded) and left out
of the element-wise output comparison. All other tokens must match within
rel-Frobenius <= 5e-3 and |delta| <= 2e-2 * max|ref|."""
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


@pytest.mark.parametrize("T,d,N", [(64, 2048, 64), (200, 2048, 64), (130, 4096, 128), (1, 512, 64)])
def test_router_logits(moe, T, d, N):
    inp = synth.layer_inputs(T=T, d=d, N=N, I=128, seed=T + d, with_experts=False)
    got = moe.router_logits(to_dev_bf16(inp["x"]), to_dev_bf16(inp["w_router"])).cpu().numpy()
    ref = oracle.router_logits(inp["x"], inp["w_router"]).astype(np.float64)
    abs_sum = np.abs(f64(inp["x"])) @ np.abs(f64(inp["w_router"])).T
    # fp32 accumulation of d products: |err| <= d * 2^-24 * sum|x w| (recursive-sum bound)
    err = np.abs(got - ref)
    assert np.all(err <= d * 2.0 ** -24 * abs_sum + 1e-30), err.max()


def _swiglu64(xs, wgu, I):
    g = xs @ wgu[:I].T
    u = xs @ wgu[I:].T
    return g / (1.0 + np.exp(-g)) * u


@pytest.mark.parametrize("N,counts", [
    (64, "random"),
    (64, "edges"),
    (128, "random"),
])
def test_grouped_gemm_steps(moe, N, counts):
    """gather -> expert gate/up (SwiGLU) -> expert down -> combine, each step
    against numpy fp64 on the same dispatch."""
    import torch
    rng = np.random.default_rng(N)
    d, I, K = 512, 256, 8
    if counts == "random":
        T = 700
        r = oracle.route(synth.boosted_logits(rng, T, N), K=K)
        k, ids = r["k"], r["ids"]
        gates = r["gates"]
    else:
        # expert sizes 0, 1, 65, 127, 128, 129, 192, 193, 300: ragged last
        # m-tiles of 1, 44, 64, 65, 127 and 128 rows
        sizes = {3: 1, 5: 127, 6: 128, 7: 129, 9: 192, 11: 300, 13: 65, 15: 193}
        T = 300
        ids = np.zeros((T, K), np.int32)
        k = np.zeros(T, np.int32)
        for t in range(T):
            mine = [e for e, s in sizes.items() if t < s]
            k[t] = len(mine)
            rest = [e for e in range(N) if e not in mine][: K - len(mine)]
            ids[t] = mine + rest
        gates = np.where(np.arange(K)[None, :] < k[:, None],
                         rng.uniform(0.05, 0.5, (T, K)), 0.0).astype(np.float32)
    x = synth.bf16_bits(rng.standard_normal((T, d)).astype(np.float32))
    wgu, wd = synth.expert_weights(N, N, d, I)
    dk, dids = to_dev(k), to_dev(ids)
    off, perm, pp, ws = moe.moe_dispatch(dk, dids, N)
    toff = moe.dispatch_tile_offsets(ws, T, N, K)
    P = T * K
    xs = moe.gather_rows(to_dev_bf16(x), perm, off, P)
    offs = off.cpu().numpy()
    nrows = int(offs[-1])
    perm_h = perm.cpu().numpy()[:nrows]
    assert np.array_equal(xs[:nrows].view(torch.int16).cpu().numpy(), x.view(np.int16)[perm_h])

    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    h = moe.expert_gate_up(xs, to_dev_bf16(wgu), off, toff, err=err)
    o = moe.expert_down(h, to_dev_bf16(wd), off, toff, err=err)
    y = moe.combine(o, dk, pp, to_dev(gates))
    torch.cuda.synchronize()
    assert int(err.item()) == 0

    xsf = f64(x)[perm_h]
    h_ref = np.zeros((nrows, I))
    o_ref = np.zeros((nrows, d))
    h_gpu = bf16_tensor_to_f64(h[:nrows])
    for e in range(N):
        a, b = offs[e], offs[e + 1]
        if b > a:
            h_ref[a:b] = _swiglu64(xsf[a:b], f64(wgu[e]), I)
            o_ref[a:b] = h_ref[a:b] @ f64(wd[e]).T
    assert_layer_close(h_gpu, h_ref, "h")
    assert_layer_close(bf16_tensor_to_f64(o[:nrows]), o_ref, "o")
    pos = pp.cpu().numpy()
    y_ref = np.zeros((T, d))
    for t in range(T):
        for s in range(k[t]):
            y_ref[t] += float(gates[t, s]) * o_ref[pos[t, s]]
    assert_layer_close(bf16_tensor_to_f64(y), y_ref, "y")


def _run_layer(moe, inp, K=8, mode=0, renorm=0, residual=None):
    import torch
    x = to_dev_bf16(inp["x"])
    wr = to_dev_bf16(inp["w_router"])
    wgu = to_dev_bf16(inp["w_gate_up"])
    wd = to_dev_bf16(inp["w_down"])
    res = None if residual is None else to_dev_bf16(residual)
    T, d = inp["x"].shape
    N = inp["w_router"].shape[0]
    I = inp["w_gate_up"].shape[1] // 2
    ws = torch.empty(moe.layer_workspace_size(T, d, N, I, K), dtype=torch.uint8, device="cuda")
    y, it = moe.moe_layer_forward(x, wr, wgu, wd, K=K, mode=mode, renorm=renorm, residual=res,
                                  ws=ws, return_intermediates=True)
    moe.read_device_error(ws)
    out = {n: v.cpu().numpy() for n, v in it.items()}
    out["y"] = bf16_tensor_to_f64(y)
    return out


def _compare_layer(inp, got, rows, K=8, mode=0, renorm=0, residual=None, max_flip=0.01):
    ref = oracle.layer_rows(inp["x"], inp["w_router"], inp["w_gate_up"], inp["w_down"], rows=rows,
                            K=K, mode=mode, renorm=renorm, residual_bits=residual)
    same = (got["k"][rows] == ref["k"]) & np.all(got["ids"][rows] == ref["ids"], axis=1)
    assert (1.0 - same.mean()) <= max_flip, f"routing flips on {np.count_nonzero(~same)} rows"
    assert same.sum() > 0
    fro, mx = assert_layer_close(got["y"][rows][same], ref["y"][same])
    # logits within the fp32 accumulation bound of d products
    d = inp["x"].shape[1]
    abs_sum = np.abs(f64(inp["x"][rows])) @ np.abs(f64(inp["w_router"])).T
    assert np.all(np.abs(got["logits"][rows] - ref["logits"]) <= d * 2.0 ** -24 * abs_sum + 1e-30)
    return ref, same, fro, mx


@pytest.mark.parametrize("mode,renorm", [(0, 0), (1, 0), (0, 1)])
def test_layer_small(moe, mode, renorm):
    """The 64-token OLMoE-shaped layer, every token against the oracle."""
    w = synth.WORKLOADS["layer_t64"]
    inp = synth.layer_inputs(T=w["T"], d=w["d"], N=w["N"], I=w["I"], seed=w["seed"])
    got = _run_layer(moe, inp, mode=mode, renorm=renorm)
    rows = np.arange(w["T"])
    ref, same, _, _ = _compare_layer(inp, got, rows, mode=mode, renorm=renorm, max_flip=0.02)
    # the layer's own routing outputs are consistent with its logits (bit-exact)
    r = oracle.route(got["logits"], K=8, mode=mode, renorm=renorm)
    assert np.array_equal(r["k"], got["k"]) and np.array_equal(r["ids"], got["ids"])
    assert np.array_equal(r["gates"].view(np.uint32), got["gates"].view(np.uint32))
    d = oracle.dispatch(got["k"], got["ids"], w["N"])
    assert np.array_equal(d["offsets"], got["offsets"])
    # also within tolerance of the storage-rounded oracle
    ref2 = oracle.layer_rows(inp["x"], inp["w_router"], inp["w_gate_up"], inp["w_down"], rows=rows,
                             mode=mode, renorm=renorm, round_h=True, round_y=True)
    assert_layer_close(got["y"][same], ref2["y"][same])


@pytest.mark.parametrize("T", [1, 3, 129])
def test_layer_ragged_with_residual(moe, T):
    inp = synth.layer_inputs(T=T, d=512, N=64, I=256, seed=77 + T)
    res = synth.bf16_bits(np.random.default_rng(T).standard_normal(inp["x"].shape).astype(np.float32))
    got = _run_layer(moe, inp, residual=res)
    _compare_layer(inp, got, np.arange(T), residual=res, max_flip=0.05)


@pytest.mark.parametrize("mode", [0, 1])
def test_layer_prefill_all_tokens(moe, mode):
    """The 16,384-token prefill layer in the launch configuration the benchmark
    times, every token against the oracle: routing of every token (flip
    fraction between the GPU's fp32 and the oracle's fp64 logits), the
    layer's own routing bit-exact on its logits, the dispatch offsets, and
    the outputs of every token whose routing agrees, element by element."""
    w = synth.WORKLOADS["layer_t16k"]
    inp = synth.layer_inputs(T=w["T"], d=w["d"], N=w["N"], I=w["I"], seed=w["seed"])
    got = _run_layer(moe, inp, mode=mode)
    r = oracle.route(got["logits"], K=8, mode=mode)
    assert np.array_equal(r["k"], got["k"]) and np.array_equal(r["ids"], got["ids"])
    assert np.array_equal(r["gates"].view(np.uint32), got["gates"].view(np.uint32))
    d_ref = oracle.dispatch(got["k"], got["ids"], w["N"])
    assert np.array_equal(d_ref["offsets"], got["offsets"])
    _, same, _, _ = _compare_layer(inp, got, np.arange(w["T"]), mode=mode, max_flip=1e-3)
    assert same.mean() >= 1.0 - 1e-3


def test_layer_wide_all_tokens(moe):
    """N = 128 experts, d = 4096, I = 1536, 20 % flat tokens (large k, ragged
    loads), every one of the 8,192 tokens against the oracle."""
    w = synth.WORKLOADS["layer_wide"]
    inp = synth.layer_inputs(T=w["T"], d=w["d"], N=w["N"], I=w["I"], seed=w["seed"],
                             flat_frac=w["flat_frac"])
    got = _run_layer(moe, inp)
    r = oracle.route(got["logits"], K=8)
    assert np.array_equal(r["k"], got["k"]) and np.array_equal(r["ids"], got["ids"])
    d_ref = oracle.dispatch(got["k"], got["ids"], w["N"])
    assert np.array_equal(d_ref["offsets"], got["offsets"])
    _, same, _, _ = _compare_layer(inp, got, np.arange(w["T"]), max_flip=2e-3)
    assert same.mean() >= 1.0 - 2e-3


@pytest.mark.parametrize("N,K,mode", [(64, 1, 1), (64, 3, 0), (128, 4, 0), (128, 5, 1)])
def test_layer_prefill_other_caps(moe, N, K, mode):
    """The prefill path (T > 64: multi-chunk dispatch, gathered gate/up GEMM,
    down GEMM, combine) with caps K < 8, every token against the oracle."""
    T, d, I = 1000, 512, 256
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=2100 + N + K)
    got = _run_layer(moe, inp, K=K, mode=mode)
    r = oracle.route(got["logits"], K=K, mode=mode)
    assert np.array_equal(r["k"], got["k"]) and np.array_equal(r["ids"], got["ids"])
    d_ref = oracle.dispatch(got["k"], got["ids"], N)
    assert np.array_equal(d_ref["offsets"], got["offsets"])
    _compare_layer(inp, got, np.arange(T), K=K, mode=mode, max_flip=0.02)


@pytest.mark.parametrize("T,mode", [(300, 0), (300, 1), (20, 0)])
def test_layer_d_multiple_of_128(moe, T, mode):
    """d = 384 (a multiple of 128, not of 256: the down GEMM's 128-column
    output tiles), prefill and decode paths, every token against the oracle."""
    N, d, I = 64, 384, 256
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=3300 + T)
    got = _run_layer(moe, inp, mode=mode)
    r = oracle.route(got["logits"], K=8, mode=mode)
    assert np.array_equal(r["k"], got["k"]) and np.array_equal(r["ids"], got["ids"])
    _compare_layer(inp, got, np.arange(T), mode=mode, max_flip=0.02)
