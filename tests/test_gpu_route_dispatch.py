"""GPU parity of routing (elbow_route) and dispatch (moe_dispatch) against the
CPU oracle: bit-exact k, ids, gates, offsets, perm and pair_pos on the same
seeded fp32 logits, including the full 1,048,576-token routing stress."""
import numpy as np
import pytest

import oracle
from paper_2608_04401_gb300 import synth

from gpu_util import to_dev

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


def _route_both(moe, lg, K=8, mode=0, renorm=0, eps=1e-8):
    k, ids, gates = moe.elbow_route(to_dev(lg), K=K, eps=eps, mode=mode, renorm=renorm)
    ref = oracle.route(lg, K=K, eps=eps, mode=mode, renorm=renorm)
    return (k.cpu().numpy(), ids.cpu().numpy(), gates.cpu().numpy()), ref


def _assert_route_equal(got, ref):
    k, ids, gates = got
    bad = np.nonzero(k != ref["k"])[0]
    assert bad.size == 0, f"k differs at {bad[:10]} (of {bad.size})"
    assert np.array_equal(ids, ref["ids"])
    assert np.array_equal(gates.view(np.uint32), ref["gates"].view(np.uint32))


@pytest.mark.parametrize("N", [64, 128])
@pytest.mark.parametrize("T", [1, 127, 129, 5000])
def test_route_bitexact_sizes(moe, N, T):
    rng = np.random.default_rng(T * 7 + N)
    lg = synth.boosted_logits(rng, T, N)
    _assert_route_equal(*_route_both(moe, lg))


@pytest.mark.parametrize("K,mode,renorm", [(8, 1, 0), (8, 0, 1), (1, 0, 0), (3, 0, 0), (5, 1, 1)])
def test_route_bitexact_params(moe, K, mode, renorm):
    rng = np.random.default_rng(K * 10 + mode + 3 * renorm)
    for N in (64, 128):
        lg = synth.boosted_logits(rng, 3001, N)
        _assert_route_equal(*_route_both(moe, lg, K=K, mode=mode, renorm=renorm))


def test_route_edge_cases(moe):
    N = 64
    rows = []
    rows.append(np.zeros(N))                      # uniform: k = 1
    rows.append(np.full(N, 3.25))                 # uniform, nonzero
    for m in (1, 2, 5, 7, 8, 20, 62, 63):          # step curves
        r = np.zeros(N); r[:m] = 6.0; rows.append(r)
    r = np.zeros(N); r[[3, 9, 40]] = 4.0; rows.append(r)   # ties among the head
    r = np.full(N, -500.0); r[11] = 0.0; rows.append(r)    # tail underflows to 0
    r = np.arange(N, dtype=np.float64) * 0.01; rows.append(r)  # nearly linear curve
    r = np.zeros(N); r[::2] = 1e-7; rows.append(r)   # distinct logits, equal probabilities
    r = np.linspace(-60, 30, N); rows.append(r)      # wide range
    rng = np.random.default_rng(0)
    # logit ranges around 87 (rows whose range is within 87 run the exponential
    # without its clamps) and around the exponential's underflow limits
    # (-87.3, -104)
    for zlow in (-85.99, -86.0, -86.01, -86.999, -87.0, -87.001, -87.4, -87.8, -103.9, -104.0,
                 -104.3, -104.6):
        r = rng.uniform(-3.0, 0.0, N); r[0] = 0.0; r[7] = zlow; rows.append(r)
        r = rng.uniform(zlow, zlow + 1.5, N); r[3] = 0.0; r[4] = -0.5; rows.append(r)
    q = np.round(rng.standard_normal((200, N)) * 2) / 2   # many exact ties
    lg = np.concatenate([np.array(rows), q]).astype(np.float32)
    for K in (8, 2):
        for mode in (0, 1):
            _assert_route_equal(*_route_both(moe, lg, K=K, mode=mode))
    lg128 = np.concatenate([lg, lg], axis=1)
    _assert_route_equal(*_route_both(moe, lg128))
    # eps = 0 on a non-degenerate batch
    _assert_route_equal(*_route_both(moe, q.astype(np.float32), eps=0.0))


@pytest.mark.parametrize("N", [64, 128])
def test_route_near_ties_and_flat_curves(moe, N):
    """Curves that defeat shortcuts: values a few ulps apart in the top ranks,
    exact ties around rank 31, flat and linear curves, wide heads of 24-40
    boosted experts, and tails that underflow."""
    rng = np.random.default_rng(N + 99)
    T = 4096
    lg = rng.standard_normal((T, N)).astype(np.float32)
    # 1) near ties: a base value plus perturbations of a few ulps
    lg[0:512] = (2.0 + rng.integers(-3, 4, (512, N)) * np.float32(2.0 ** -22)).astype(np.float32)
    # 2) exact ties everywhere in the top 40 ranks
    lg[512:1024] = np.round(rng.uniform(-1, 1, (512, N)) * 4) / 4
    # 3) flat / linear curves, permuted
    for t in range(1024, 1536):
        lg[t] = rng.permutation(np.linspace(0, rng.uniform(0.1, 4.0), N))
    # 4) wide heads
    for t in range(1536, 2048):
        hsz = rng.integers(24, 41)
        lg[t] = rng.standard_normal(N) * 0.3
        lg[t, rng.choice(N, hsz, replace=False)] += rng.uniform(0.5, 1.0, hsz)
    # 5) spikes over a -60..-200 tail (partial underflow of the exponent)
    lg[2048:2560] = rng.uniform(-200, -60, (512, N))
    lg[2048:2560, 0] = 0.0
    lg = lg.astype(np.float32)
    for K, mode in ((8, 0), (8, 1), (4, 0), (1, 0)):
        _assert_route_equal(*_route_both(moe, lg, K=K, mode=mode))


def test_route_full_stress(moe):
    """The 1,048,576 x 64 routing stress, compared token by token."""
    w = synth.WORKLOADS["route_t1m"]
    rng = np.random.Generator(np.random.PCG64(w["seed"]))
    lg = synth.boosted_logits(rng, w["T"], w["N"])
    got, ref = _route_both(moe, lg, K=w["K"])
    _assert_route_equal(got, ref)
    assert 1.0 < ref["k"].mean() < 8.0


def _dispatch_both(moe, k, ids, N):
    import torch
    off, perm, pp, ws = moe.moe_dispatch(to_dev(k), to_dev(ids), N)
    torch.cuda.synchronize()
    ref = oracle.dispatch(k, ids, N)
    off = off.cpu().numpy()
    assert np.array_equal(off, ref["offsets"])
    P = int(off[-1])
    assert np.array_equal(perm.cpu().numpy()[:P], ref["perm"])
    assert np.array_equal(pp.cpu().numpy(), ref["pair_pos"])
    # m-tile prefix sums left in the workspace
    T, K = ids.shape
    toff = moe.dispatch_tile_offsets(ws, T, N, K).cpu().numpy()
    cnt = np.diff(ref["offsets"])
    assert np.array_equal(toff, np.concatenate([[0], np.cumsum((cnt + 127) // 128)]))
    return ref


@pytest.mark.parametrize("N,T,kind", [(64, 700, "routed"), (128, 2049, "routed"),
                                        (64, 2049, "same"), (128, 1700, "same")])
def test_dispatch_ignores_stale_workspace(moe, N, T, kind):
    """Every part of the dispatch workspace is written before it is read: a
    workspace full of 0xff bytes gives the same dispatch, with and without the
    router's counts. kind "same": every token selects experts 0..7 (128 pairs
    of each of them per chunk, 0 of every other expert)."""
    import torch
    rng = np.random.default_rng(T + 7 * N)
    lg = synth.boosted_logits(rng, T, N)
    if kind == "same":
        k = np.full(T, 8, np.int32)
        ids = np.tile(np.arange(8, dtype=np.int32), (T, 1))
    else:
        r = oracle.route(lg, K=8)
        k, ids = r["k"], r["ids"]
    ref = oracle.dispatch(k, ids, N)
    P = int(ref["offsets"][-1])
    ws = torch.full((moe.dispatch_workspace_size(T, N, 8),), 255, dtype=torch.uint8, device="cuda")
    off, perm, pp, _ = moe.moe_dispatch(to_dev(k), to_dev(ids), N, ws=ws)
    torch.cuda.synchronize()
    assert np.array_equal(off.cpu().numpy(), ref["offsets"])
    assert np.array_equal(perm.cpu().numpy()[:P], ref["perm"])
    assert np.array_equal(pp.cpu().numpy(), ref["pair_pos"])
    if kind == "routed":
        ws.fill_(255)
        cc = moe.dispatch_chunk_counts(ws, T, N, 8)
        k2, ids2, _ = moe.elbow_route_with_counts(to_dev(lg), cc)
        off2, perm2, pp2 = moe.moe_dispatch_counted(k2, ids2, N, ws)
        torch.cuda.synchronize()
        assert np.array_equal(off2.cpu().numpy(), ref["offsets"])
        assert np.array_equal(perm2.cpu().numpy()[:P], ref["perm"])
        assert np.array_equal(pp2.cpu().numpy(), ref["pair_pos"])


@pytest.mark.parametrize("N,T", [(64, 100), (128, 100), (64, 3000), (128, 3000)])
def test_dispatch_drops_out_of_range_ids(moe, N, T):
    """Pairs whose id lies outside [0, N) are dropped (not counted, not in perm,
    pair_pos -1); the other pairs keep the stable expert-major order."""
    import torch
    rng = np.random.default_rng(T + N + 11)
    r = oracle.route(synth.boosted_logits(rng, T, N), K=8)
    k, ids = r["k"], r["ids"].copy()
    sel = np.arange(8)[None, :] < k[:, None]
    bad = sel & (rng.random(ids.shape) < 0.05)
    ids[bad] = rng.choice(np.array([-1, -7, N, N + 3, 1 << 20], np.int32), bad.sum())
    off, perm, pp, _ = moe.moe_dispatch(to_dev(k), to_dev(ids), N)
    torch.cuda.synchronize()
    good = sel & ~bad
    t_idx, s_idx = np.nonzero(good)
    e_idx = ids[t_idx, s_idx]
    order = np.lexsort((t_idx, e_idx))  # by expert, then token
    want_off = np.concatenate([[0], np.cumsum(np.bincount(e_idx, minlength=N))])
    want_pp = np.full(ids.shape, -1, np.int64)
    want_pp[t_idx[order], s_idx[order]] = np.arange(len(order))
    assert np.array_equal(off.cpu().numpy(), want_off)
    assert np.array_equal(perm.cpu().numpy()[:len(order)], t_idx[order])
    assert np.array_equal(pp.cpu().numpy(), want_pp)


@pytest.mark.parametrize("N", [64, 128])
@pytest.mark.parametrize("K", [1, 3, 5, 7])
@pytest.mark.parametrize("T", [100, 3001])
def test_dispatch_other_caps(moe, N, K, T):
    """K < 8: rows of ids that are not 32 bytes (element loads instead of the
    16-byte ones), in the one-block and the multi-chunk dispatch."""
    rng = np.random.default_rng(T + N + 31 * K)
    r = oracle.route(synth.boosted_logits(rng, T, N), K=K)
    _dispatch_both(moe, r["k"], r["ids"], N)


@pytest.mark.parametrize("N", [64, 128])
@pytest.mark.parametrize("T", [1, 33, 2047, 2048, 2049, 20000])
def test_dispatch_bitexact(moe, N, T):
    rng = np.random.default_rng(T + N)
    r = oracle.route(synth.boosted_logits(rng, T, N), K=8)
    _dispatch_both(moe, r["k"], r["ids"], N)


def test_dispatch_edges(moe):
    N, K = 64, 8
    T = 5000
    ids = np.tile(np.arange(K, dtype=np.int32), (T, 1))
    _dispatch_both(moe, np.ones(T, np.int32), ids, N)             # all on expert 0
    _dispatch_both(moe, np.full(T, K, np.int32), ids, N)           # fixed top-8
    _dispatch_both(moe, np.zeros(T, np.int32), ids, N)             # no pairs
    ids2 = ids.copy(); ids2[:, 0] = 63; ids2[:, 7] = 0
    _dispatch_both(moe, np.full(T, 3, np.int32), ids2, N)          # last expert
    ids3 = np.tile(np.arange(120, 128, dtype=np.int32), (T, 1))
    _dispatch_both(moe, np.full(T, K, np.int32), ids3, 128)
    # T = 0
    import torch
    off, perm, pp, ws = moe.moe_dispatch(torch.zeros(0, dtype=torch.int32, device="cuda"),
                                         torch.zeros(0, K, dtype=torch.int32, device="cuda"), N)
    assert np.all(off.cpu().numpy() == 0)


@pytest.mark.parametrize("N,T,K", [(64, 150001, 8), (128, 300007, 8), (128, 99999, 5),
                                   (64, 1000003, 3)])
def test_dispatch_single_pass_ranges(moe, N, T, K):
    """The single-pass dispatch with several 32-token units per warp (running
    positions carried from unit to unit), ragged last block, both N and
    K < 8 (element loads and stores)."""
    rng = np.random.default_rng(T + N + K)
    r = oracle.route(synth.boosted_logits(rng, T, N), K=K)
    _dispatch_both(moe, r["k"], r["ids"], N)


def test_dispatch_workspace_error_word(moe):
    """The single-pass dispatch clears its workspace's error word and leaves it
    clear: moe_read_device_error on the dispatch workspace reports MOE_OK, and
    a second call on the same workspace gives the same bit-exact result."""
    import torch
    rng = np.random.default_rng(4242)
    r = oracle.route(synth.boosted_logits(rng, 50000, 64), K=8)
    k, ids = to_dev(r["k"]), to_dev(r["ids"])
    ws = torch.full((moe.dispatch_workspace_size(50000, 64, 8),), 0xFF, dtype=torch.uint8,
                    device="cuda")
    out1 = moe.moe_dispatch(k, ids, 64, ws)
    moe.read_device_error(ws)
    out2 = moe.moe_dispatch(k, ids, 64, ws)
    moe.read_device_error(ws)
    P = int(out1[0][-1].item())
    assert torch.equal(out1[0], out2[0]) and torch.equal(out1[2], out2[2])
    assert torch.equal(out1[1][:P], out2[1][:P])  # perm past offsets[N] is left untouched
    ref = oracle.dispatch(r["k"], r["ids"], 64)
    assert np.array_equal(out2[2].cpu().numpy(), ref["pair_pos"])


def test_dispatch_full_stress(moe):
    w = synth.WORKLOADS["route_t1m"]
    rng = np.random.Generator(np.random.PCG64(w["seed"] + 1))
    lg = synth.boosted_logits(rng, w["T"], w["N"])
    r = oracle.route(lg, K=8)
    _dispatch_both(moe, r["k"], r["ids"], w["N"])


@pytest.mark.parametrize("N,T", [(64, 1000), (128, 3000), (64, 70000)])
def test_route_with_counts_then_counted_dispatch(moe, N, T):
    """The router's per-chunk counts let the dispatch skip its counting pass;
    routing and dispatch stay bit-exact against the oracle."""
    import torch
    rng = np.random.default_rng(N + T)
    lg = synth.boosted_logits(rng, T, N)
    ws = torch.empty(moe.dispatch_workspace_size(T, N, 8), dtype=torch.uint8, device="cuda")
    cc = moe.dispatch_chunk_counts(ws, T, N, 8)
    k, ids, gates = moe.elbow_route_with_counts(to_dev(lg), cc)
    torch.cuda.synchronize()
    ref = oracle.route(lg, K=8)
    # counts [N][ceil(T/128)]: the pairs of expert e among tokens 128 c .. 128 c + 127
    sel = np.arange(8)[None, :] < ref["k"][:, None]
    want = np.zeros((N, (T + 127) // 128), np.int64)
    np.add.at(want, (ref["ids"][sel], np.repeat(np.arange(T) // 128, ref["k"])), 1)
    assert np.array_equal(cc.cpu().numpy(), want)
    off, perm, pp = moe.moe_dispatch_counted(k, ids, N, ws)
    torch.cuda.synchronize()
    _assert_route_equal((k.cpu().numpy(), ids.cpu().numpy(), gates.cpu().numpy()), ref)
    d = oracle.dispatch(ref["k"], ref["ids"], N)
    assert np.array_equal(off.cpu().numpy(), d["offsets"])
    n = int(d["offsets"][-1])
    assert np.array_equal(perm.cpu().numpy()[:n], d["perm"])
    assert np.array_equal(pp.cpu().numpy(), d["pair_pos"])


# ------------------------------------------- one warp per token (small batches)
def _route_warp_both(moe, lg, K=8, mode=0, renorm=0, eps=1e-8):
    k, ids, gates = moe.elbow_route_warp(to_dev(lg), K=K, eps=eps, mode=mode, renorm=renorm)
    ref = oracle.route(lg, K=K, eps=eps, mode=mode, renorm=renorm)
    return (k.cpu().numpy(), ids.cpu().numpy(), gates.cpu().numpy()), ref


@pytest.mark.parametrize("N", [64, 128])
@pytest.mark.parametrize("K,mode,renorm", [(8, 0, 0), (8, 1, 0), (8, 0, 1), (1, 0, 0), (3, 0, 1)])
def test_route_warp_bitexact(moe, N, K, mode, renorm):
    rng = np.random.default_rng(N * 3 + K + 7 * mode + renorm)
    lg = synth.boosted_logits(rng, 3001, N)
    _assert_route_equal(*_route_warp_both(moe, lg, K=K, mode=mode, renorm=renorm))


@pytest.mark.parametrize("N", [64, 128])
def test_route_warp_edge_cases(moe, N):
    """The curves that stress the thread kernel's shortcuts, through the warp
    kernel: near ties, exact ties, flat and linear curves, wide heads, tails
    that underflow, uniform rows, step curves."""
    rng = np.random.default_rng(N + 5)
    rows = [np.zeros(N), np.full(N, 2.5)]
    for m in (1, 2, 7, 8, 9, N // 2, N - 2, N - 1):
        r = np.zeros(N); r[:m] = 6.0; rows.append(r)
    r = np.full(N, -500.0); r[3] = 0.0; rows.append(r)
    r = np.linspace(-60, 30, N); rows.append(r)
    lg = rng.standard_normal((1024, N)).astype(np.float32)
    lg[0:256] = (2.0 + rng.integers(-3, 4, (256, N)) * np.float32(2.0 ** -22)).astype(np.float32)
    lg[256:512] = np.round(rng.uniform(-1, 1, (256, N)) * 4) / 4
    lg[512:768] = rng.uniform(-200, -60, (256, N)); lg[512:768, 0] = 0.0
    lg = np.concatenate([np.array(rows, np.float32), lg]).astype(np.float32)
    for K, mode in ((8, 0), (8, 1), (2, 0)):
        _assert_route_equal(*_route_warp_both(moe, lg, K=K, mode=mode))


def test_route_warp_full_stress(moe):
    """The 1,048,576-token stress through the warp kernel, token by token."""
    w = synth.WORKLOADS["route_t1m"]
    rng = np.random.Generator(np.random.PCG64(w["seed"] + 2))
    lg = synth.boosted_logits(rng, w["T"], w["N"])
    _assert_route_equal(*_route_warp_both(moe, lg, K=w["K"]))
