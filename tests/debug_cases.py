"""Cases for the bounds-checked debug build (run by test_gpu_debug.py in a
child process with ELBOW_MOE_DEBUG=1, which makes the binding load that build).

Every output buffer the library writes is allocated with a tail of sentinel
bytes (a canary) that must be unchanged afterwards, and the device bounds
checks of the debug build must count no violation: small batches T = 1..33
(the decode path), a few prefill batches, N in {64, 128}, K in {1..8}. A last
case plants an out-of-range pair position in the combine's input and checks
that the debug build counts it while the canary stays intact (the release
clamp keeps the access inside the array)."""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))
sys.path.insert(0, HERE)

import torch  # noqa: E402

import oracle  # noqa: E402
import paper_2608_04401_gb300 as moe  # noqa: E402
from paper_2608_04401_gb300 import synth  # noqa: E402
from gpu_util import to_dev_bf16  # noqa: E402

CANARY = 0x5A
PAD = 4096  # canary bytes after each output


def padded(numel, dtype):
    """A [numel] tensor view at the head of a buffer whose PAD-byte tail is the canary."""
    esz = torch.empty(0, dtype=dtype).element_size()
    raw = torch.full((numel * esz + PAD,), CANARY, dtype=torch.uint8, device="cuda")
    return raw, raw[: numel * esz].view(dtype)


def tail_ok(raw, numel_bytes):
    torch.cuda.synchronize()
    return bool(torch.all(raw[numel_bytes:] == CANARY).item())


def layer_case(T, N, K, mode, d=256, I=128):
    """One layer forward: y and the workspace canary-padded, no violation, the
    routing bit-exact on the layer's own logits, outputs within tolerance."""
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=9000 + 17 * T + N + K)
    x, wr = to_dev_bf16(inp["x"]), to_dev_bf16(inp["w_router"])
    wgu, wd = to_dev_bf16(inp["w_gate_up"]), to_dev_bf16(inp["w_down"])
    need = moe.layer_workspace_size(T, d, N, I, K)
    ws_raw, ws = padded(need, torch.uint8)
    y_raw, y = padded(T * d, torch.bfloat16)
    y = y.view(T, d)
    _, it = moe.moe_layer_forward(x, wr, wgu, wd, K=K, mode=mode, y=y, ws=ws,
                                  return_intermediates=True)
    moe.read_device_error(ws)
    assert moe.debug_violations() == 0, ("layer", T, N, K)
    assert tail_ok(ws_raw, need) and tail_ok(y_raw, T * d * 2), ("layer canary", T, N, K)
    lg = it["logits"].cpu().numpy()
    r = oracle.route(lg, K=K, mode=mode)
    assert np.array_equal(r["k"], it["k"].cpu().numpy()), ("k", T, N, K)
    assert np.array_equal(r["ids"], it["ids"].cpu().numpy()), ("ids", T, N, K)
    ref = oracle.layer_rows(inp["x"], inp["w_router"], inp["w_gate_up"], inp["w_down"], K=K,
                            mode=mode)
    same = (ref["k"] == r["k"]) & np.all(ref["ids"] == r["ids"], axis=1)
    got = y.float().cpu().numpy().astype(np.float64)[same]
    want = ref["y"][same]
    fro = np.linalg.norm(got - want) / max(np.linalg.norm(want), 1e-30)
    assert fro <= 5e-3, ("layer output", T, N, K, fro)


def dispatch_case(T, N, K, seed):
    """moe_dispatch with every output canary-padded, no violation, and the
    oracle's dispatch bit for bit."""
    rng = np.random.default_rng(seed)
    ids = np.argsort(rng.random((T, N)), axis=1)[:, :K].astype(np.int32)
    k = rng.integers(1, K + 1, size=T).astype(np.int32)
    lib = moe.library()
    dk = torch.from_numpy(k).cuda()
    dids = torch.from_numpy(ids).cuda()
    o_raw, off = padded(N + 1, torch.int32)
    p_raw, perm = padded(max(1, T * K), torch.int32)
    q_raw, pp = padded(T * K, torch.int32)
    wsz = moe.dispatch_workspace_size(T, N, K)
    w_raw, ws = padded(wsz, torch.uint8)
    st = lib.moe_dispatch(moe._p(dk), moe._p(dids), T, N, K, moe._p(off), moe._p(perm), moe._p(pp),
                          moe._p(ws), wsz, moe._stream())
    assert st == 0, st
    assert moe.debug_violations() == 0, ("dispatch", T, N, K)
    for raw, nb in ((o_raw, 4 * (N + 1)), (p_raw, 4 * max(1, T * K)), (q_raw, 4 * T * K),
                    (w_raw, wsz)):
        assert tail_ok(raw, nb), ("dispatch canary", T, N, K)
    ref = oracle.dispatch(k, ids, N)
    P = int(ref["offsets"][-1])
    assert np.array_equal(off.cpu().numpy(), ref["offsets"])
    assert np.array_equal(perm.cpu().numpy()[:P], ref["perm"][:P])
    assert np.array_equal(pp.cpu().numpy(), ref["pair_pos"].reshape(-1))


def steps_case(T, N, K, d=256, I=128):
    """The step-level entry points on one routed batch, each output
    canary-padded: the gathered gate/up and down GEMMs (T > 64) or the row
    gather and the decode-shaped GEMMs (T <= 64), then the combine."""
    lib = moe.library()
    P_ = moe._p
    s = moe._stream()
    rng = np.random.default_rng(500 + T + N + K)
    inp = synth.layer_inputs(T=T, d=d, N=N, I=I, seed=700 + T + N + K)
    x, wgu, wd = (to_dev_bf16(inp[n]) for n in ("x", "w_gate_up", "w_down"))
    lg = torch.from_numpy(synth.boosted_logits(rng, T, N)).cuda()
    k, ids, gates = moe.elbow_route(lg, K=K)
    off, perm, pp, dws = moe.moe_dispatch(k, ids, N)
    toff = moe.dispatch_tile_offsets(dws, T, N, K)
    P = T * K
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    h_raw, h = padded(P * I, torch.bfloat16)
    o_raw, o = padded(P * d, torch.bfloat16)
    if T > 64:
        assert lib.moe_expert_gate_up_gathered(P_(x), T, P_(perm), P_(wgu), P_(off), P_(toff), P, d,
                                               N, I, P_(h), P_(err), s) == 0
        assert lib.moe_expert_down(P_(h), P_(wd), P_(off), P_(toff), P, d, N, I, P_(o), P_(err),
                                   s) == 0
        outs = [(h_raw, 2 * P * I), (o_raw, 2 * P * d)]
    else:
        xs_raw, xs = padded(P * d, torch.bfloat16)
        assert lib.moe_gather_rows(P_(x), P_(perm), P_(off), T, P, d, N, P_(xs), s) == 0
        assert lib.moe_expert_gate_up_decode(P_(xs), P_(wgu), P_(off), T, P, d, N, I, P_(h),
                                             P_(err), s) == 0
        assert lib.moe_expert_down_decode(P_(h), P_(wd), P_(off), T, P, d, N, I, P_(o), P_(err),
                                          s) == 0
        outs = [(xs_raw, 2 * P * d), (h_raw, 2 * P * I), (o_raw, 2 * P * d)]
    y_raw, y = padded(T * d, torch.bfloat16)
    assert lib.moe_combine(P_(o), P_(k), P_(pp), P_(gates), None, T, d, K, P_(y), s) == 0
    outs.append((y_raw, 2 * T * d))
    assert moe.debug_violations() == 0, ("steps", T, N, K)
    assert int(err.item()) == 0
    for raw, nb in outs:
        assert tail_ok(raw, nb), ("steps canary", T, N, K)
    assert bool(torch.isfinite(y.float()).all().item())


def planted_case():
    """An out-of-range pair position given to the combine: the debug build
    counts it (the release clamp keeps the read inside o) and y's canary stays."""
    lib = moe.library()
    P_ = moe._p
    T, d, K = 40, 256, 4
    k = torch.full((T,), K, dtype=torch.int32, device="cuda")
    pp = torch.arange(T * K, dtype=torch.int32, device="cuda").view(T, K).contiguous()
    pp[3, 1] = T * K + 5
    gates = torch.full((T, K), 0.25, dtype=torch.float32, device="cuda")
    o = torch.ones(T * K, d, dtype=torch.bfloat16, device="cuda")
    y_raw, y = padded(T * d, torch.bfloat16)
    assert lib.moe_combine(P_(o), P_(k), P_(pp), P_(gates), None, T, d, K, P_(y),
                           moe._stream()) == 0
    v = moe.debug_violations()
    assert v >= 1, v
    assert tail_ok(y_raw, 2 * T * d)
    assert moe.debug_violations() == 0  # the count was reset


def main():
    assert os.environ.get("ELBOW_MOE_DEBUG") == "1"
    moe.build(debug=True)
    assert moe._LIB_PATH.endswith(os.path.join("debug", "libelbow_moe.so"))
    torch.cuda.set_device(0)
    n = 0
    for T in list(range(1, 34)) + [65, 200, 1000]:
        for N in (64, 128):
            K = 1 + (T + N // 64) % 8
            mode = T % 2
            layer_case(T, N, K, mode)
            dispatch_case(T, N, K, seed=T * 7 + N)
            steps_case(T, N, K)
            n += 3
    for K in range(1, 9):
        layer_case(33, 64, K, 0)
        dispatch_case(129, 64, K, seed=K)
        n += 2
    planted_case()
    print(f"debug build: {n + 1} cases, no bounds violation, canaries intact")


if __name__ == "__main__":
    main()
