"""The layer's fused stages against their unfused counterparts, bit for bit:
the router GEMM with routing in its epilogue vs router GEMM + elbow_route, and
the gate/up GEMM that gathers its token rows vs gather + dense gate/up GEMM."""
import numpy as np
import pytest

import oracle
from paper_2608_04401_gb300 import synth

from gpu_util import to_dev, to_dev_bf16

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


@pytest.mark.parametrize("T,d,N,mode", [(64, 2048, 64, 0), (200, 512, 64, 0), (130, 512, 128, 0),
                                        (1000, 2048, 64, 1), (3000, 1024, 128, 0)])
def test_router_route_matches_steps(moe, T, d, N, mode):
    import torch
    inp = synth.layer_inputs(T=T, d=d, N=N, I=128, seed=T + N, with_experts=False)
    x, wr = to_dev_bf16(inp["x"]), to_dev_bf16(inp["w_router"])
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    k, ids, gates, lg, cc = moe.router_route(x, wr, mode=mode, err=err)
    lg_ref = moe.router_logits(x, wr)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    assert torch.equal(lg.view(torch.int32), lg_ref.view(torch.int32))
    k2, ids2, g2 = moe.elbow_route(lg_ref, mode=mode)
    assert torch.equal(k, k2) and torch.equal(ids, ids2)
    assert torch.equal(gates.view(torch.int32), g2.view(torch.int32))
    # per-chunk expert counts of the selected pairs
    kn, idn = k.cpu().numpy(), ids.cpu().numpy()
    want = np.zeros((N, (T + 127) // 128), np.int32)
    for t in range(T):
        for s in range(kn[t]):
            want[idn[t, s], t // 128] += 1
    assert np.array_equal(cc.cpu().numpy(), want)
    # and the routing agrees with the oracle given these logits
    r = oracle.route(lg.cpu().numpy(), K=8, mode=mode)
    assert np.array_equal(r["k"], kn) and np.array_equal(r["ids"], idn)


@pytest.mark.parametrize("N,T", [(64, 300), (64, 2000), (128, 700)])
def test_gate_up_gathered_matches_dense(moe, N, T):
    import torch
    rng = np.random.default_rng(N * T)
    d, I, K = 512, 256, 8
    r = oracle.route(synth.boosted_logits(rng, T, N), K=K)
    x = to_dev_bf16(synth.bf16_bits(rng.standard_normal((T, d)).astype(np.float32)))
    wgu, _ = synth.expert_weights(7, N, d, I)
    wgu = to_dev_bf16(wgu)
    off, perm, pp, ws = moe.moe_dispatch(to_dev(r["k"]), to_dev(r["ids"]), N)
    toff = moe.dispatch_tile_offsets(ws, T, N, K)
    P = T * K
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    xs = moe.gather_rows(x, perm, off, P)
    h_dense = moe.expert_gate_up(xs, wgu, off, toff, err=err)
    h_gath = moe.expert_gate_up_gathered(x, perm, wgu, off, toff, P, err=err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    n = int(off[-1].item())
    assert torch.equal(h_dense[:n].view(torch.int16), h_gath[:n].view(torch.int16))


@pytest.mark.parametrize("T,N", [(64, 64), (5000, 64), (3000, 128)])
def test_dispatch_counted_matches_dispatch(moe, T, N):
    """Router counts written straight into the dispatch workspace give the
    same dispatch as counting again."""
    import torch
    inp = synth.layer_inputs(T=T, d=512, N=N, I=128, seed=T * 3 + N, with_experts=False)
    x, wr = to_dev_bf16(inp["x"]), to_dev_bf16(inp["w_router"])
    ws = torch.empty(moe.dispatch_workspace_size(T, N, 8), dtype=torch.uint8, device="cuda")
    cc = moe.dispatch_chunk_counts(ws, T, N, 8)
    k, ids, gates, _, _ = moe.router_route(x, wr, with_logits=False, chunk_counts=cc)
    # counts [N][ceil(T/128)]: the pairs of expert e among tokens 128 c .. 128 c + 127
    kh, idh = k.cpu().numpy(), ids.cpu().numpy()
    sel = np.arange(8)[None, :] < kh[:, None]
    want = np.zeros((N, (T + 127) // 128), np.int64)
    np.add.at(want, (idh[sel], np.repeat(np.arange(T) // 128, kh)), 1)
    assert np.array_equal(cc.cpu().numpy(), want)
    off_a, perm_a, pp_a = moe.moe_dispatch_counted(k, ids, N, ws)
    off_b, perm_b, pp_b, _ = moe.moe_dispatch(k, ids, N)
    torch.cuda.synchronize()
    assert torch.equal(off_a, off_b) and torch.equal(pp_a, pp_b)
    n = int(off_b[-1].item())
    assert torch.equal(perm_a[:n], perm_b[:n])
