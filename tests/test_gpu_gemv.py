"""GPU parity of the CUDA-core expert contractions for batches of T <= 4
tokens (the one-token latency regime: each touched expert's weight rows spread
over many blocks, the token rows read from x through the dispatch permutation)
against numpy fp64 on the same dispatch, and of the whole layer at T = 1
(which moe_layer_forward routes to them) and T = 2, 4 against the oracle."""
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


@pytest.mark.parametrize("T,N,d,I,K", [(1, 64, 2048, 1024, 8), (2, 64, 512, 256, 8),
                                       (3, 128, 1024, 512, 5), (4, 64, 4096, 1536, 8),
                                       (4, 128, 256, 4096, 8), (1, 128, 384, 128, 1)])
def test_gemv_steps(moe, T, N, d, I, K):
    import torch
    rng = np.random.default_rng(T * 31 + N + d + I + K)
    r = oracle.route(synth.boosted_logits(rng, T, N), K=K)
    k, ids = r["k"], r["ids"]
    x = synth.bf16_bits(rng.standard_normal((T, d)).astype(np.float32))
    wgu, wd = synth.expert_weights(N + d, N, d, I)
    off, perm, pp, ws = moe.moe_dispatch(to_dev(k), to_dev(ids), N)
    P = T * K
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    h = moe.expert_gate_up_gemv(to_dev_bf16(x), perm, to_dev_bf16(wgu), off, P, K=K, err=err)
    o = moe.expert_down_gemv(h, to_dev_bf16(wd), off, T, K=K, err=err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    offs = off.cpu().numpy()
    n = int(offs[-1])
    xsf = f64(x)[perm.cpu().numpy()[:n]]
    h_ref = np.zeros((n, I))
    o_own = np.zeros((n, d))
    hg = bf16_tensor_to_f64(h[:n])
    for e in range(N):
        a, b = offs[e], offs[e + 1]
        if b > a:
            g = xsf[a:b] @ f64(wgu[e][:I]).T
            u = xsf[a:b] @ f64(wgu[e][I:]).T
            h_ref[a:b] = g / (1.0 + np.exp(-g)) * u
            o_own[a:b] = hg[a:b] @ f64(wd[e]).T
    assert_layer_close(hg, h_ref, "h")
    assert_layer_close(bf16_tensor_to_f64(o[:n]), o_own, "o")


@pytest.mark.parametrize("T,mode,N", [(1, 0, 64), (1, 1, 64), (1, 0, 128), (2, 1, 64), (4, 0, 128)])
def test_layer_gemv_sizes(moe, T, mode, N):
    """The whole layer at T = 1 (the CUDA-core contractions) and at T = 2, 4
    (the tensor-core decode tiles), every token against the oracle; routing
    bit-exact on the layer's own logits."""
    import torch
    d, I = (2048, 1024) if N == 64 else (1024, 512)
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=800 + T + N)
    x = to_dev_bf16(inp["x"])
    ws = torch.empty(moe.layer_workspace_size(T, d, N, I, 8), dtype=torch.uint8, device="cuda")
    y, it = moe.moe_layer_forward(x, to_dev_bf16(inp["w_router"]), to_dev_bf16(inp["w_gate_up"]),
                                  to_dev_bf16(inp["w_down"]), K=8, mode=mode, ws=ws,
                                  return_intermediates=True)
    moe.read_device_error(ws)
    r = oracle.route(it["logits"].cpu().numpy(), K=8, mode=mode)
    assert np.array_equal(r["k"], it["k"].cpu().numpy())
    assert np.array_equal(r["ids"], it["ids"].cpu().numpy())
    ref = oracle.layer_rows(inp["x"], inp["w_router"], inp["w_gate_up"], inp["w_down"],
                            rows=np.arange(T), K=8, mode=mode)
    same = (ref["k"] == r["k"]) & np.all(ref["ids"] == r["ids"], axis=1)
    assert same.all()
    assert_layer_close(bf16_tensor_to_f64(y), ref["y"])


@pytest.mark.parametrize("T,d,I,N,mode,K,res", [(1, 256, 2048, 64, 0, 8, False),
                                                (1, 4096, 256, 128, 1, 8, True),
                                                (1, 384, 384, 64, 1, 3, True),
                                                (1, 1024, 4096, 128, 0, 1, False),
                                                (2, 4096, 1536, 128, 0, 8, True),
                                                (2, 512, 256, 64, 1, 5, False),
                                                (2, 2048, 1024, 128, 1, 8, False)])
def test_layer_few_token_shapes(moe, T, d, I, N, mode, K, res):
    """Layers of one and two tokens on other shapes (down items of 16 to 64
    columns, one to sixteen experts, two rows for experts both tokens chose,
    with a residual): y against the oracle, routing bit-exact on the layer's
    own logits, and the device error word clean."""
    import torch
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=900 + T + d + I + K)
    x = to_dev_bf16(inp["x"])
    resid = synth.bf16_bits(np.random.default_rng(d + I).standard_normal((T, d)).astype(np.float32))
    ws = torch.empty(moe.layer_workspace_size(T, d, N, I, K), dtype=torch.uint8, device="cuda")
    y, it = moe.moe_layer_forward(x, to_dev_bf16(inp["w_router"]), to_dev_bf16(inp["w_gate_up"]),
                                  to_dev_bf16(inp["w_down"]), K=K, mode=mode, ws=ws,
                                  residual=to_dev_bf16(resid) if res else None,
                                  return_intermediates=True)
    moe.read_device_error(ws)
    r = oracle.route(it["logits"].cpu().numpy(), K=K, mode=mode)
    assert np.array_equal(r["k"], it["k"].cpu().numpy())
    assert np.array_equal(r["ids"], it["ids"].cpu().numpy())
    ref = oracle.layer_rows(inp["x"], inp["w_router"], inp["w_gate_up"], inp["w_down"],
                            rows=np.arange(T), K=K, mode=mode,
                            residual_bits=resid if res else None)
    assert np.array_equal(ref["k"], r["k"]) and np.array_equal(ref["ids"], r["ids"])
    assert_layer_close(bf16_tensor_to_f64(y), ref["y"])


@pytest.mark.parametrize("N,mode,renorm", [(64, 0, 1), (128, 1, 0), (64, 1, 1)])
def test_layer_two_identical_tokens(moe, N, mode, renorm):
    """Two copies of one token: every expert in use has two rows (both rows of
    the expert item, and two pairs per column block in the combine), with
    renorm = 1 and both modes; routing equal for both tokens and bit-exact on
    the layer's logits, y equal for both tokens and within tolerance of the
    oracle."""
    import torch
    d, I, K = 1024, 512, 8
    inp = synth.layer_inputs(T=1, d=d, N=N, I=I, seed=777 + N + mode)
    x2 = np.concatenate([inp["x"], inp["x"]], axis=0)
    ws = torch.empty(moe.layer_workspace_size(2, d, N, I, K), dtype=torch.uint8, device="cuda")
    y, it = moe.moe_layer_forward(to_dev_bf16(x2), to_dev_bf16(inp["w_router"]),
                                  to_dev_bf16(inp["w_gate_up"]), to_dev_bf16(inp["w_down"]), K=K,
                                  mode=mode, renorm=renorm, ws=ws, return_intermediates=True)
    moe.read_device_error(ws)
    k, ids = it["k"].cpu().numpy(), it["ids"].cpu().numpy()
    assert k[0] == k[1] and np.array_equal(ids[0], ids[1])
    offs = it["offsets"].cpu().numpy()
    cnt = np.diff(offs)
    assert set(cnt[cnt > 0].tolist()) == {2}
    r = oracle.route(it["logits"].cpu().numpy(), K=K, mode=mode, renorm=renorm)
    assert np.array_equal(r["k"], k) and np.array_equal(r["ids"], ids)
    yv = bf16_tensor_to_f64(y)
    assert np.array_equal(yv[0], yv[1])
    ref = oracle.layer_rows(x2, inp["w_router"], inp["w_gate_up"], inp["w_down"], rows=np.arange(2),
                            K=K, mode=mode, renorm=renorm)
    if np.array_equal(ref["k"], k) and np.array_equal(ref["ids"], ids):
        assert_layer_close(yv, ref["y"])


def test_gemv_rejects_large_batches(moe):
    import torch
    x = torch.zeros(5, 512, dtype=torch.bfloat16, device="cuda")
    w = torch.zeros(64, 512, 512, dtype=torch.bfloat16, device="cuda")
    perm = torch.zeros(40, dtype=torch.int32, device="cuda")
    off = torch.zeros(65, dtype=torch.int32, device="cuda")
    with pytest.raises(moe.MoeError):
        moe.expert_gate_up_gemv(x, perm, w, off, 40)
