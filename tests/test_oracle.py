"""Pins of the CPU oracle against what the paper and the mathematics fix.

Every check here is independent of the oracle's own code: closed forms worked
by hand (tests/golden), the geometric Kneedle definition evaluated in fp64,
library routines that compute special cases (numpy sort, bincount, matmul),
exact identities of App. A.3, and an exhaustive error sweep of the routing
exponential against double-precision exp.
"""
import math
import os

import numpy as np
import pytest

import oracle
from paper_2608_04401_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ------------------------------------------------------------------ EXP spec
def test_exp_error_exhaustive():
    """EXP within 2 ulp of exp() on every fp32 in [-104, 0] with a normal result."""
    err, worst = oracle.exp_max_ulp(-104.0, 0.0)
    assert err <= 2.0, (err, worst)


def test_exp_special_values():
    assert oracle.exp([0.0])[0] == np.float32(1.0)
    assert oracle.exp([-np.inf])[0] == 0.0
    assert oracle.exp([-104.5])[0] == 0.0
    # n < -126 flushes to zero (documented): exp(-88) ~ 6e-39 is below 2^-126
    assert oracle.exp([-88.0])[0] == 0.0
    z = np.float32(-87.0)
    assert abs(float(oracle.exp([z])[0]) - math.exp(float(z))) <= 2 ** -149 * 8 + math.exp(float(z)) * 2 ** -22


# ------------------------------------------------------------ Algorithm 1
def _golden_steps():
    rows = []
    with open(os.path.join(GOLDEN, "step_curves.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            N, m, K, hi, lo, e, k = line.split()
            rows.append((int(N), int(m), int(K), float(hi), float(lo), int(e), int(k)))
    return rows


@pytest.mark.parametrize("N,m,K,hi,lo,e,k", _golden_steps())
def test_step_curves(N, m, K, hi, lo, e, k):
    lg = np.full((1, N), lo, np.float32)
    lg[0, :m] = hi
    r = oracle.route(lg, K=K, with_sorted=True)
    assert r["elbow"][0] == e
    assert r["k"][0] == k


def test_step_curves_any_position():
    """The step's members need not be the first experts: e = m wherever they sit."""
    rng = np.random.default_rng(5)
    for _ in range(50):
        N = int(rng.choice([16, 64, 128]))
        m = int(rng.integers(1, N - 1))
        lg = np.zeros((1, N), np.float32)
        members = rng.choice(N, size=m, replace=False)
        lg[0, members] = 5.0
        r = oracle.route(lg, K=8, with_sorted=True)
        assert r["elbow"][0] == m
        assert r["k"][0] == min(m + 1, 8)
        # ties broken by ascending expert id (reading R3)
        assert list(r["ids"][0][: min(m, 8)]) == sorted(members)[: min(m, 8)]


def test_three_level_closed_form():
    """Levels A > B > C with counts m1, m2, rest. With beta = p'_B:
    D peaks at i = m1 (value 1 - beta - x'_{m1}) or at i = m1 + m2 (value
    1 - x'_{m1+m2}); the first wins iff beta < m2 / (N - 1)."""
    N = 64
    cases = 0
    for m1 in (1, 2, 4):
        for m2 in (2, 5, 9):
            for b in np.linspace(-3.0, 3.0, 13):
                lg = np.full((1, N), -2.0, np.float32)
                lg[0, :m1] = 6.0
                lg[0, m1:m1 + m2] = b
                # beta from the fp64 softmax (levels are exact ratios of exps)
                a, bb, c = math.exp(6.0), math.exp(float(np.float32(b))), math.exp(-2.0)
                beta = (bb - c) / (a - c)
                thr = m2 / (N - 1)
                if abs(beta - thr) < 1e-4:
                    continue
                want = m1 if beta < thr else m1 + m2
                r = oracle.route(lg, K=64, with_sorted=True)
                assert r["elbow"][0] == want, (m1, m2, b, beta, thr)
                cases += 1
    assert cases > 50


def _kneedle_fp64(logits_row):
    """Kneedle knee in fp64: points (x'_i, p'_i) of the descending curve, knee =
    the point farthest below the straight line through the first and last
    points (perpendicular distance via the 2-D cross product)."""
    l = logits_row.astype(np.float64)
    p = np.exp(l - l.max())
    p /= p.sum()
    order = sorted(range(len(p)), key=lambda j: (-p[j], j))
    ps = p[order]
    n = len(ps)
    xs = np.arange(n) / (n - 1)
    pn = (ps - ps[-1]) / (ps[0] - ps[-1])
    (x0, y0), (x1, y1) = (xs[0], pn[0]), (xs[-1], pn[-1])
    # signed distance, positive below the chord of a descending curve
    dist = ((x1 - x0) * (y0 - pn) - (xs - x0) * (y0 - y1)) / math.hypot(x1 - x0, y1 - y0)
    return dist, order, ps


def test_bruteforce_small_n():
    """Tiny N, random logits: the oracle's elbow is the fp64 Kneedle knee, and its
    sorted order is the fp64 descending order, wherever fp32 cannot flip them."""
    rng = np.random.default_rng(11)
    checked = 0
    for N in (4, 8, 16, 32):
        lg = (rng.standard_normal((400, N)) * rng.uniform(0.3, 3.0, (400, 1))).astype(np.float32)
        r = oracle.route(lg, K=N, with_sorted=True)
        for t in range(lg.shape[0]):
            dist, order, ps = _kneedle_fp64(lg[t])
            top2 = np.sort(dist)[-2:]
            if top2[1] - top2[0] > 1e-5:
                assert r["elbow"][t] == int(np.argmax(dist))
                checked += 1
            gaps = -np.diff(ps)
            if gaps.min() > 1e-6 * ps[0]:
                assert list(r["ids"][t]) == order[:N]
    assert checked > 1000


def test_bruteforce_permutations():
    """All orderings of one multiset of logits give the same elbow and, up to the
    rounding of the position-ordered softmax sum, the same sorted curve; the ids
    follow the permutation (the sort is a total order)."""
    import itertools
    base = np.array([3.0, 0.5, 1.5, 0.5, -1.0, 2.0], np.float32)
    N = 8
    ref = None
    for perm in itertools.permutations(range(6)):
        lg = np.full((1, N), -3.0, np.float32)
        lg[0, list(perm)] = base
        r = oracle.route(lg, K=N, with_sorted=True)
        if ref is None:
            ref = (r["sorted_p"][0].copy(), r["elbow"][0])
        np.testing.assert_allclose(r["sorted_p"][0], ref[0], rtol=2.0 ** -21)
        assert r["elbow"][0] == ref[1]
        want = sorted(range(N), key=lambda j: (-float(lg[0, j]), j))
        assert list(r["ids"][0]) == want


# ------------------------------------------------------ selection and gates
@pytest.mark.parametrize("N,K", [(64, 8), (128, 8), (64, 1), (16, 16), (128, 3)])
def test_selection_invariants(N, K):
    rng = np.random.default_rng(N * 100 + K)
    lg = synth.boosted_logits(rng, 3000, N)
    el = oracle.route(lg, K=K, with_sorted=True)
    tk = oracle.route(lg, K=K, mode=oracle.MODE_TOPK)
    k = el["k"]
    assert np.all((1 <= k) & (k <= K))
    assert np.all(tk["k"] == K)
    # same sort in both modes: elbow-K is a prefix of top-K (Sec. 2.1)
    assert np.array_equal(el["ids"], tk["ids"])
    # capped count follows the elbow (Sec. 2.1, reading R2)
    assert np.array_equal(k, np.minimum(el["elbow"] + 1, K))
    # ids are the first K of the descending order; distinct
    for t in range(0, lg.shape[0], 7):
        assert len(set(el["ids"][t])) == K
    # gates: the sorted probabilities for s < k, zero after; non-increasing
    s = np.arange(K)[None, :]
    sp = el["sorted_p"][:, :K]
    assert np.array_equal(el["gates"], np.where(s < k[:, None], sp, 0).astype(np.float32))
    assert np.array_equal(tk["gates"], sp)
    assert np.all(np.diff(el["gates"], axis=1) <= 0)
    # top-K against numpy's fp64 softmax + stable argsort where fp32 cannot reorder
    l64 = lg.astype(np.float64)
    p64 = np.exp(l64 - l64.max(1, keepdims=True))
    p64 /= p64.sum(1, keepdims=True)
    order = np.argsort(-p64, axis=1, kind="stable")[:, :K + 1]
    top = np.take_along_axis(p64, order, 1)
    clear = np.all(-np.diff(top, axis=1) > 1e-5 * top[:, :1], axis=1)
    assert clear.mean() > 0.5
    assert np.array_equal(el["ids"][clear], order[clear, :K])
    np.testing.assert_allclose(tk["gates"], top[:, :K], rtol=3e-6, atol=1e-12)
    # softmax sums to one within N * 2^-23 (each p_j carries <= 2.5 ulp)
    assert np.all(np.abs(el["sorted_p"].astype(np.float64).sum(1) - 1.0) <= N * 2.0 ** -23)


def test_renorm_gates():
    rng = np.random.default_rng(3)
    lg = synth.boosted_logits(rng, 2000, 64)
    r = oracle.route(lg, K=8, renorm=1)
    tot = r["gates"].astype(np.float64).sum(1)
    assert np.all(np.abs(tot - 1.0) <= 8 * 2.0 ** -23)
    base = oracle.route(lg, K=8)
    assert np.array_equal(r["k"], base["k"]) and np.array_equal(r["ids"], base["ids"])
    # k = 1 with renorm: the single gate is exactly 1
    one = oracle.route(lg, K=1, renorm=1)
    assert np.all(one["gates"][:, 0] == 1.0)


@pytest.mark.parametrize("shift", [512.0, -512.0])
def test_softmax_shift_invariance(shift):
    """Softmax is invariant under adding one constant to all logits. On logits of a
    2^-10 grid within +-32 the shifted logits, and their differences to the
    shifted maximum, are exact in fp32, so the routing must be bit-identical;
    a softmax that skipped the max subtraction would overflow (+512) or underflow
    (-512) here."""
    rng = np.random.default_rng(77)
    for N in (64, 128):
        lg = (np.round(rng.normal(0.0, 4.0, (300, N)) * 1024.0) / 1024.0).clip(-32, 32)
        lg = lg.astype(np.float32)
        a = oracle.route(lg, K=8)
        b = oracle.route((lg + np.float32(shift)).astype(np.float32), K=8)
        assert np.array_equal(a["k"], b["k"]) and np.array_equal(a["ids"], b["ids"])
        assert np.array_equal(a["gates"].view(np.uint32), b["gates"].view(np.uint32))


def test_flat_and_degenerate():
    N = 64
    # all logits equal: R = 0, k = 1 (documented degenerate case)
    r = oracle.route(np.full((3, N), 2.5, np.float32), K=8, with_sorted=True)
    assert np.all(r["k"] == 1) and np.all(r["elbow"] == 0)
    assert list(r["ids"][0]) == list(range(8))
    # huge spread: tail probabilities underflow to exactly 0
    lg = np.full((1, N), -500.0, np.float32)
    lg[0, 7] = 0.0
    r = oracle.route(lg, K=8, with_sorted=True)
    assert r["sorted_p"][0, 0] == 1.0 and np.all(r["sorted_p"][0, 1:] == 0)
    assert r["k"][0] == 2 and r["ids"][0, 0] == 7


# ----------------------------------------------- load balance (App. A.3)
def _tree_sum_f32(v):
    """The balanced tree sum of R6 in fp32: v_i += v_{i+h}, h = N/2 .. 1."""
    v = np.array(v, dtype=np.float32)
    h = v.shape[-1] // 2
    while h >= 1:
        v[..., :h] = v[..., :h] + v[..., h:2 * h]
        h //= 2
    return v[..., 0]


@pytest.mark.parametrize("N", [64, 128])
def test_printed_quotients_rounded_once(N):
    """Every quotient of the printed formulas is the correctly rounded fp32
    quotient: p_j = e_j / s (the softmax of Sec. 2) and p'_i = (p_(i) - p_min) /
    den (Alg. 1's normalisation). An fp64 quotient of two fp32 numbers rounded
    to fp32 is the correctly rounded fp32 quotient (53 >= 2 * 24 + 2 bits, so
    the double rounding is innocuous: Figueroa, 1995), which a product with a
    rounded reciprocal is not in general. D_i = (1 - p'_i) - x'_i, each
    difference rounded once."""
    rng = np.random.default_rng(700 + N)
    T = 96
    lg = np.concatenate([synth.boosted_logits(rng, T // 2, N),
                         rng.standard_normal((T // 2, N)).astype(np.float32)])
    cur = oracle.elbow_curve(lg, eps=1e-8)
    f32, f64 = np.float32, np.float64
    m = lg.max(axis=1, keepdims=True)
    e = oracle.exp((lg - m).astype(np.float32))
    s = _tree_sum_f32(e)
    p = (e.astype(f64) / s[:, None].astype(f64)).astype(f32)
    assert np.array_equal(np.sort(p, axis=1)[:, ::-1], cur["p"])
    sp = cur["p"]
    pmin = sp[:, -1:]
    den = (f32(sp[:, :1] - pmin) + f32(1e-8)).astype(f32)
    a = (sp - pmin).astype(f32)
    pn = (a.astype(f64) / den.astype(f64)).astype(f32)
    assert np.array_equal(pn, cur["pn"])
    x = (np.arange(N, dtype=f32) / f32(N - 1)).astype(f32)
    D = ((f32(1.0) - pn).astype(f32) - x).astype(f32)
    assert np.array_equal(D, cur["D"])
    # the reading matters: the reciprocal products differ from the quotients
    # in some of these values, so the check above can tell the two apart
    p_rcp = (e * (f32(1.0) / s)[:, None]).astype(f32)
    assert np.count_nonzero(p_rcp != p) > 0


def test_theorem1_and_corollaries():
    """Theorem 1 and Corollaries 1-2 hold exactly on the empirical loads of any
    batch, and q_elb - q_top = delta/(1-delta) (q_top - r) (the proof's identity)."""
    for seed, N in ((1, 64), (2, 128)):
        rng = np.random.default_rng(seed)
        lg = synth.boosted_logits(rng, 4000, N)
        r = oracle.route(lg, K=8)
        lb = oracle.load_balance(r["k"], r["ids"], N)
        d = lb["delta"]
        assert 0 < d < 1
        assert lb["l1"] <= lb["l1_bound"] + 1e-12
        assert lb["max_change"] <= lb["l1_bound"] + 1e-12
        assert lb["cv2_change"] <= lb["cv2_bound"] + 1e-12
        R = lb["L_top"] - lb["L_elb"]
        assert np.all(R >= -1e-15)
        rr = R / (d * 8)
        np.testing.assert_allclose(lb["q_elb"] - lb["q_top"], d / (1 - d) * (lb["q_top"] - rr), atol=1e-12)
        np.testing.assert_allclose(lb["L_top"].sum(), 8.0)
        np.testing.assert_allclose(lb["L_elb"].sum(), r["k"].mean())


def test_load_balance_hand_example():
    """Two tokens, N = 4, K = 2: token 0 keeps expert 0 of (0, 1), token 1 keeps
    both of (0, 2). By hand: q_top = (1/2, 1/4, 1/4, 0), q_elb = (2/3, 0, 1/3, 0),
    delta = 1/4, l1 = 1/2 <= 2/3, top-1 share change |2/3 - 1/2| = 1/6, CV^2 = 1/2
    and 11/9 with Corollary 2's bound 2 N delta / (1 - delta)^2 = 32/9, top-1 share
    change (1/2 - 2/3) / (1/2) = -100/3 %, CV change (sqrt(1/2) - sqrt(11/9)) / sqrt(1/2)."""
    lb = oracle.load_balance(np.array([1, 2]), np.array([[0, 1], [0, 2]]), 4)
    np.testing.assert_allclose(lb["q_top"], [0.5, 0.25, 0.25, 0.0], atol=1e-15)
    np.testing.assert_allclose(lb["q_elb"], [2 / 3, 0.0, 1 / 3, 0.0], atol=1e-15)
    assert abs(lb["delta"] - 0.25) < 1e-15
    assert abs(lb["l1"] - 0.5) < 1e-15 and abs(lb["l1_bound"] - 2 / 3) < 1e-15
    assert abs(lb["max_change"] - 1 / 6) < 1e-15
    assert abs(lb["cv2_change"] - (11 / 9 - 0.5)) < 1e-14
    assert abs(lb["cv2_bound"] - 32 / 9) < 1e-14
    assert abs(lb["top1_share_change_pct"] + 100 / 3) < 1e-12
    want = (np.sqrt(0.5) - np.sqrt(11 / 9)) / np.sqrt(0.5) * 100
    assert abs(lb["cv_change_pct"] - want) < 1e-12


# ------------------------------------------------------ elbow angle (Sec. 2.3)
@pytest.mark.parametrize("N", [64, 128])
def test_elbow_angle_step_curves(N):
    """A step of m equal high values has its elbow at e = m with p'_e = 0, so
    v1 = (-x, -1), v2 = (1 - x, 0) and theta = 90 deg + atan(x), x = m/(N-1)."""
    for m in (1, 2, 3, 7, 8, 20, N // 2, N - 2):
        lg = np.zeros((1, N), np.float32)
        lg[0, :m] = 6.0
        a = oracle.elbow_angle(lg)
        assert a["elbow"][0] == m
        x = float(np.float32(m) / np.float32(N - 1))
        assert abs(float(a["theta"][0]) - (90.0 + np.degrees(np.arctan(x)))) < 2e-5


def test_elbow_angle_uniform_and_range():
    """The uniform curve: e = 0, p' = 0, v1 = (0, -1), v2 = (1, 0): 90 degrees.
    Every angle lies in [0, 180]."""
    a = oracle.elbow_angle(np.zeros((3, 64), np.float32))
    assert np.all(a["elbow"] == 0) and np.all(a["theta"] == 90.0)
    lg = synth.boosted_logits(np.random.default_rng(4), 3000, 64)
    a = oracle.elbow_angle(lg)
    assert np.all((a["theta"] >= 0) & (a["theta"] <= 180))


@pytest.mark.parametrize("N", [64, 128])
def test_elbow_angle_vs_atan2(N):
    """Recomputed from the sorted curve with atan2 (the angle between the two
    directions, no dot product or arccos), on random curves; the uncapped
    elbow index agrees with the routing's."""
    rng = np.random.default_rng(N + 5)
    lg = synth.boosted_logits(rng, 500, N)
    a = oracle.elbow_angle(lg)
    r = oracle.route(lg, K=8, with_sorted=True)
    assert np.array_equal(a["elbow"], r["elbow"])
    assert np.array_equal(r["k"], np.minimum(a["elbow"] + 1, 8))
    f = np.float32
    for t in range(500):
        sp = r["sorted_p"][t]
        e = int(a["elbow"][t])
        den = f(f(sp[0] - sp[-1]) + f(1e-8))
        pn = f(np.float64(f(sp[e] - sp[-1])) / np.float64(den))
        x = float(f(e) / f(N - 1))
        y = 1.0 - float(pn)
        a1 = np.arctan2(-y, -x)
        a2 = np.arctan2(1.0 - y, 1.0 - x)
        th = abs(np.degrees(a1 - a2))
        th = 360.0 - th if th > 180.0 else th
        assert abs(th - float(a["theta"][t])) < 2e-4, (t, th, a["theta"][t])


# --------------------------------------------------------------- dispatch
def _check_dispatch(k, ids, N):
    out = oracle.dispatch(k, ids, N)
    T, K = ids.shape
    s = np.arange(K)[None, :]
    valid = s < k[:, None]
    e_pairs = ids[valid]
    t_pairs = np.repeat(np.arange(T), k)
    # counts and offsets: exclusive scan of the histogram
    cnt = np.bincount(e_pairs, minlength=N)
    assert np.array_equal(out["offsets"], np.concatenate([[0], np.cumsum(cnt)]).astype(np.int32))
    # stable counting sort of the pairs by expert = stable argsort
    want = t_pairs[np.argsort(e_pairs, kind="stable")]
    assert np.array_equal(out["perm"], want)
    pp = out["pair_pos"]
    assert np.all(pp[~valid] == -1)
    assert np.array_equal(out["perm"][pp[valid]], t_pairs)
    assert sorted(pp[valid].tolist()) == list(range(len(t_pairs)))
    return out


def test_dispatch_random():
    rng = np.random.default_rng(9)
    for N, K, T in ((64, 8, 5000), (128, 8, 3000), (64, 1, 1000), (8, 8, 300)):
        ids = np.argsort(rng.random((T, N)), axis=1)[:, :K].astype(np.int32)
        k = rng.integers(1, K + 1, size=T).astype(np.int32)
        _check_dispatch(k, ids, N)


def test_dispatch_edges():
    N, K = 64, 8
    # every token on expert 5 first
    T = 1000
    ids = np.tile(np.arange(K, dtype=np.int32), (T, 1))
    ids[:, 0] = 5
    ids[:, 5] = 0
    out = _check_dispatch(np.ones(T, np.int32), ids, N)
    assert out["offsets"][5] == 0 and out["offsets"][6] == T
    # empty batch
    out = _check_dispatch(np.zeros(0, np.int32), np.zeros((0, K), np.int32), N)
    assert np.all(out["offsets"] == 0)
    # k = 0 tokens are allowed by the dispatch (no pairs)
    _check_dispatch(np.zeros(10, np.int32), np.tile(np.arange(K, dtype=np.int32), (10, 1)), N)
    # invalid: duplicate expert inside a token
    bad = np.tile(np.arange(K, dtype=np.int32), (2, 1))
    bad[1, 3] = bad[1, 1]
    with pytest.raises(ValueError):
        oracle.dispatch(np.full(2, K, np.int32), bad, N)


# ------------------------------------------------------------------ layer
def _mlp64(xf, wgu, wd, e, I):
    g = xf @ wgu[e, :I].T
    u = xf @ wgu[e, I:].T
    h = g / (1.0 + np.exp(-g)) * u
    return h @ wd[e].T


def _small_layer(seed, T=24, d=64, N=8, I=32):
    rng = np.random.default_rng(seed)
    wr, w_hat = synth.router_weights(rng, N, d)
    x = synth.tokens(rng, T, w_hat)
    wgu, wd = synth.expert_weights(seed, N, d, I)
    f = lambda b: synth.bf16_bits_to_f32(b).astype(np.float64)
    return x, wr, wgu, wd, f(x), f(wr), f(wgu), f(wd)


def test_router_logits_vs_matmul():
    x, wr, *_ , xf, wrf, _, _ = _small_layer(1)
    lg = oracle.router_logits(x, wr)
    want = (xf @ wrf.T).astype(np.float32)
    np.testing.assert_allclose(lg, want, rtol=2 ** -23, atol=1e-30)


def test_layer_single_expert_is_dense_swiglu():
    """K = 1, renorm = 1: each token gets gate 1 on its top expert, so the layer is
    the dense SwiGLU MLP of that expert (numpy fp64 matmul)."""
    x, wr, wgu, wd, xf, wrf, wguf, wdf = _small_layer(2)
    I = wgu.shape[1] // 2
    out = oracle.layer_rows(x, wr, wgu, wd, K=1, renorm=1)
    assert np.all(out["k"] == 1) and np.all(out["gates"][:, 0] == 1.0)
    for t in range(x.shape[0]):
        want = _mlp64(xf[t:t + 1], wguf, wdf, out["ids"][t, 0], I)[0]
        np.testing.assert_allclose(out["y"][t], want, rtol=1e-10, atol=1e-12)


def test_layer_combine_vs_matmul():
    """General K: y_t = sum_{s<k_t} g_{t,s} MLP_{ids[t,s]}(x_t), with the residual."""
    x, wr, wgu, wd, xf, wrf, wguf, wdf = _small_layer(3)
    I = wgu.shape[1] // 2
    res = synth.bf16_bits(np.random.default_rng(4).standard_normal(x.shape).astype(np.float32))
    for mode in (oracle.MODE_ELBOW, oracle.MODE_TOPK):
        out = oracle.layer_rows(x, wr, wgu, wd, K=4, mode=mode, residual_bits=res)
        r = oracle.route(out["logits"], K=4, mode=mode)
        assert np.array_equal(r["k"], out["k"]) and np.array_equal(r["ids"], out["ids"])
        for t in range(x.shape[0]):
            want = synth.bf16_bits_to_f32(res[t]).astype(np.float64).copy()
            for s in range(out["k"][t]):
                want += float(out["gates"][t, s]) * _mlp64(xf[t:t + 1], wguf, wdf, out["ids"][t, s], I)[0]
            np.testing.assert_allclose(out["y"][t], want, rtol=1e-10, atol=1e-12)
    # routed rows are independent: a subset of rows reproduces the same outputs
    sub = oracle.layer_rows(x, wr, wgu, wd, rows=[5, 0, 17], K=4)
    full = oracle.layer_rows(x, wr, wgu, wd, K=4)
    assert np.array_equal(sub["y"], full["y"][[5, 0, 17]])


def test_layer_storage_rounding_is_small():
    """Rounding h and the expert outputs to bf16 (the kernels' storage precision)
    moves the output by far less than the parity tolerance."""
    x, wr, wgu, wd, *_ = _small_layer(6, T=16, d=128, N=8, I=64)
    a = oracle.layer_rows(x, wr, wgu, wd, K=8)["y"]
    b = oracle.layer_rows(x, wr, wgu, wd, K=8, round_h=True, round_y=True)["y"]
    assert np.linalg.norm(a - b) / np.linalg.norm(a) < 5e-3


def test_synthetic_tokens_have_elbows():
    """The signal-noise generator (Sec. 2.2) gives a head of boosted experts: the
    elbow sits at |S_t| for most tokens and mean k is well inside [1, K]."""
    inp = synth.layer_inputs(T=256, d=256, N=64, I=64, seed=7, with_experts=False)
    lg = oracle.router_logits(inp["x"], inp["w_router"])
    r = oracle.route(lg, K=8)
    assert 3.0 < r["k"].mean() < 8.0


# ------------------------------------------- tail randomisation (Sec. 2.2)
def _p_by_id(lg):
    """Every expert's probability, read off a full top-N routing (N slots)."""
    T, N = lg.shape
    r = oracle.route(lg, K=N, mode=oracle.MODE_TOPK)
    p = np.empty((T, N), np.float32)
    np.put_along_axis(p, r["ids"], r["gates"], axis=1)
    return p


@pytest.mark.parametrize("N", [64, 128])
def test_randomized_tail_invariants(N):
    rng = np.random.default_rng(N + 21)
    T, K = 3000, 8
    lg = synth.boosted_logits(rng, T, N)
    rnd = rng.integers(0, 2**32, size=(T, K), dtype=np.uint32)
    base = oracle.route(lg, K=K)
    p = _p_by_id(lg)
    for mode in (oracle.MODE_RAND_TAIL, oracle.MODE_RAND_HEAD):
        r = oracle.route_randomized(lg, rnd, K=K, mode=mode)
        assert np.all(r["k"] == K)
        for t in range(T):
            k, ids, top = base["k"][t], r["ids"][t], base["ids"][t]
            assert len(set(ids.tolist())) == K
            if mode == oracle.MODE_RAND_TAIL:
                assert np.array_equal(ids[:k], top[:k])          # the head is kept
                assert not set(ids[k:]) & set(top[:k])           # tail picks have rank >= k
            else:
                assert np.array_equal(ids[k:], top[k:])          # ranks k..K-1 are kept
                assert not set(ids[:k]) & set(top)               # head picks have rank >= K
            assert np.array_equal(r["gates"][t], p[t, ids])      # gate = the expert's own p


def test_randomized_zero_draws_take_smallest_ids():
    """rand = 0 selects, slot after slot, the smallest remaining id."""
    N, K = 64, 8
    lg = np.zeros((1, N), np.float32)
    lg[0, [40, 50, 60]] = 6.0                     # head of 3: ranks 0..2 = 40, 50, 60; k = 4
    base = oracle.route(lg, K=K)
    k = int(base["k"][0])
    assert k == 4
    r = oracle.route_randomized(lg, np.zeros((1, K), np.uint32), K=K, mode=oracle.MODE_RAND_TAIL)
    # rank 3 is expert 0 (ties by ascending id); the tail draws the smallest ids outside the head
    assert r["ids"][0].tolist() == base["ids"][0, :k].tolist() + [1, 2, 3, 4]
    r = oracle.route_randomized(lg, np.zeros((1, K), np.uint32), K=K, mode=oracle.MODE_RAND_HEAD)
    top = set(base["ids"][0].tolist())
    first = [j for j in range(N) if j not in top][:k]
    assert r["ids"][0, :k].tolist() == first and r["ids"][0, k:].tolist() == base["ids"][0, k:].tolist()


def test_randomized_draw_is_uniform():
    """One token repeated: the first tail draw is uniform over the N - k experts
    of rank >= k (chi-square, 60 cells, far inside the 1e-6 tail)."""
    N, K, T = 64, 8, 60000
    row = np.zeros(N, np.float32)
    row[[5, 9, 33]] = 6.0
    lg = np.tile(row, (T, 1))
    rnd = np.random.default_rng(7).integers(0, 2**32, size=(T, K), dtype=np.uint32)
    r = oracle.route_randomized(lg, rnd, K=K, mode=oracle.MODE_RAND_TAIL)
    k = int(oracle.route(lg[:1], K=K)["k"][0])
    first = r["ids"][:, k]
    cnt = np.bincount(first, minlength=N)
    head = oracle.route(lg[:1], K=K)["ids"][0, :k]
    assert np.all(cnt[head] == 0)
    cells = np.delete(cnt, head)
    exp_c = T / (N - k)
    chi2 = float(((cells - exp_c) ** 2 / exp_c).sum())
    assert chi2 < 130.0, chi2      # dof = N - k - 1 = 59; P(chi2 > 130) < 1e-6


def test_randomized_renorm_and_full_head():
    rng = np.random.default_rng(3)
    lg = synth.boosted_logits(rng, 500, 64)
    rnd = rng.integers(0, 2**32, size=(500, 8), dtype=np.uint32)
    r = oracle.route_randomized(lg, rnd, mode=oracle.MODE_RAND_TAIL, renorm=1)
    np.testing.assert_allclose(r["gates"].astype(np.float64).sum(1), 1.0, atol=1e-6)
    base = oracle.route(lg, K=8, mode=oracle.MODE_TOPK)
    k = oracle.route(lg, K=8)["k"]
    full = k == 8                              # no tail: nothing to randomise
    r0 = oracle.route_randomized(lg, rnd, mode=oracle.MODE_RAND_TAIL)
    assert np.array_equal(r0["ids"][full], base["ids"][full])
    assert np.array_equal(r0["gates"][full], base["gates"][full])
