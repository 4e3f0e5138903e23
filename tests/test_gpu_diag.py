"""GPU parity of the routing diagnostics (moe_route_diagnostics) against the
oracle: the uncapped elbow index bit-exact, the elbow angle of Sec. 2.3
within 1e-4 degrees (fp64 arccos on both sides, rounded to fp32), the
histograms and per-expert loads exact, and the load-change quantities of
Sec. 2.4 / App. A.3 within 1e-12."""
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


def _logits(N, T, seed):
    rng = np.random.default_rng(seed)
    lg = synth.boosted_logits(rng, T, N)
    edge = [np.zeros(N), np.full(N, 2.0)]
    for m in (1, 2, 7, 8, 9, N // 2, N - 2, N - 1):
        r = np.zeros(N); r[:m] = 6.0; edge.append(r)
    edge.append(np.round(rng.standard_normal(N) * 2) / 2)
    edge.append(np.linspace(-30, 0, N))
    return np.concatenate([lg, np.array(edge, np.float32)]).astype(np.float32)


@pytest.mark.parametrize("N,K", [(64, 8), (128, 8), (64, 4)])
def test_diagnostics_vs_oracle(moe, N, K):
    lg = _logits(N, 4000, N + K)
    st, el, th = moe.route_diagnostics(to_dev(lg), K=K)
    el, th = el.cpu().numpy(), th.cpu().numpy()
    ref = oracle.elbow_angle(lg)
    assert np.array_equal(el, ref["elbow"])
    assert np.max(np.abs(th.astype(np.float64) - ref["theta"])) <= 1e-4
    T = lg.shape[0]
    k = np.minimum(el + 1, K)
    assert st["tokens"] == T
    assert np.array_equal(st["k_hist"], np.bincount(k, minlength=9))
    assert np.array_equal(st["elbow_hist"], np.bincount(el, minlength=N))
    assert np.array_equal(st["theta_hist"], np.bincount(np.floor(th).astype(np.int64), minlength=181))
    assert st["sharp_elbows"] == int(np.count_nonzero(th <= 135.0))
    r = oracle.route(lg, K=K)
    assert np.array_equal(r["k"], k)
    assert np.array_equal(st["load_top"], np.bincount(r["ids"].ravel(), minlength=N))
    sel = r["ids"][np.arange(K)[None, :] < r["k"][:, None]]
    assert np.array_equal(st["load_elb"], np.bincount(sel, minlength=N))
    lb = oracle.load_balance(r["k"], r["ids"], N)
    for a, b in (("mean_k", None), ("delta", "delta"), ("l1", "l1"), ("l1_bound", "l1_bound"),
                 ("top1_change", "max_change"), ("cv2_change", "cv2_change"),
                 ("cv2_bound", "cv2_bound"), ("top1_share_change_pct", "top1_share_change_pct"),
                 ("cv_change_pct", "cv_change_pct")):
        want = r["k"].mean() if b is None else lb[b]
        assert abs(st[a] - want) <= 1e-12 * max(1.0, abs(want)), (a, st[a], want)
    # Theorem 1 and Corollaries 1-2 on this batch
    assert st["l1"] <= st["l1_bound"] and st["top1_change"] <= st["l1_bound"]
    assert st["cv2_change"] <= st["cv2_bound"]


def test_diagnostics_empty_and_stress(moe):
    import torch
    st, _, _ = moe.route_diagnostics(torch.zeros(0, 64, dtype=torch.float32, device="cuda"))
    assert st["tokens"] == 0 and st["k_hist"].sum() == 0 and st["load_top"].sum() == 0
    # the 1,048,576-token stress: consistent with the routing kernel's own outputs
    w = synth.WORKLOADS["route_t1m"]
    rng = np.random.Generator(np.random.PCG64(w["seed"]))
    lg = to_dev(synth.boosted_logits(rng, w["T"], w["N"]))
    k, ids, _ = moe.elbow_route(lg, K=w["K"])
    st, el, th = moe.route_diagnostics(lg, K=w["K"])
    k = k.cpu().numpy()
    assert np.array_equal(np.minimum(el.cpu().numpy() + 1, w["K"]), k)
    assert np.array_equal(st["k_hist"], np.bincount(k, minlength=9))
    ids = ids.cpu().numpy()
    assert np.array_equal(st["load_top"], np.bincount(ids.ravel(), minlength=w["N"]))
    assert st["l1"] <= st["l1_bound"]
    assert 0.99 <= st["sharp_elbows"] / w["T"] <= 1.0
