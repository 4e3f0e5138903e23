"""The routing divides with its own correctly rounded quotients (one
reciprocal per divisor, then Markstein's fused multiply-add correction), so
that p_j = e_j / s and p'_i = (p_(i) - p_min) / den are the quotients the
printed formulas define, rounded once. Checked against CUDA's __fdiv_rn and
against the fp64 quotient rounded to fp32 (the correctly rounded fp32
quotient: 53 >= 2 * 24 + 2, Figueroa 1995) on the ranges the routing uses:
numerators in [0, 1] (softmax numerators, normalised differences), divisors
in [1, 128] (softmax sums) and [2^-32, 2] (Alg. 1's p_max - p_min + eps),
with the hard cases of the correction: divisors with all-ones significands,
numerators near the top of a binade, quotients near midpoints, and numerators
below the correction's range (taken by __fdiv_rn)."""
import numpy as np
import pytest

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


def _f32_bits(lo, hi, n, rng):
    """n fp32 values with uniformly random bit patterns in [lo, hi] (lo, hi > 0)."""
    blo = np.array(lo, np.float32).view(np.uint32)
    bhi = np.array(hi, np.float32).view(np.uint32)
    return rng.integers(int(blo), int(bhi) + 1, size=n, dtype=np.uint64).astype(np.uint32).view(np.float32)


def _cases(rng, n):
    a, b = [], []
    # softmax: e in [2^-90, 1] (log-uniform bits), s in [1, 128]
    a.append(_f32_bits(2.0 ** -90, 1.0, n, rng)); b.append(_f32_bits(1.0, 128.0, n, rng))
    # normalisation: numerators in [2^-60, 1], denominators in [2^-32, 2]
    a.append(_f32_bits(2.0 ** -60, 1.0, n, rng)); b.append(_f32_bits(2.0 ** -32, 2.0, n, rng))
    # divisors whose significand is all ones or all ones but one (|b y - 1| largest)
    sig = np.array([0x7FFFFF, 0x7FFFFE, 0x7FFFFD, 0x400001, 0x000001], np.uint32)
    exps = rng.integers(127 - 32, 127 + 8, size=n).astype(np.uint32)
    bb = ((exps << 23) | sig[rng.integers(0, len(sig), size=n)]).view(np.float32)
    a.append(_f32_bits(2.0 ** -40, 1.0, n, rng)); b.append(bb)
    # numerators with all-ones significands (quotients at the top of a binade)
    ea = rng.integers(127 - 60, 127, size=n).astype(np.uint32)
    a.append(((ea << 23) | np.uint32(0x7FFFFF)).view(np.float32)); b.append(_f32_bits(1.0, 128.0, n, rng))
    # quotients on or next to a midpoint of the float grid: a = b * m rounded,
    # with m an fp32 value plus half an ulp
    m = _f32_bits(0.5, 1.0, n, rng).astype(np.float64) * (1.0 + 2.0 ** -24)
    bq = _f32_bits(1.0, 64.0, n, rng)
    a.append((bq.astype(np.float64) * m).astype(np.float32)); b.append(bq)
    # zeros and numerators below the correction's range (2^-90)
    a.append(np.concatenate([np.zeros(16, np.float32), _f32_bits(2.0 ** -126, 2.0 ** -90, n - 16, rng)]))
    b.append(_f32_bits(1.0, 128.0, n, rng))
    return np.concatenate(a), np.concatenate(b)


def test_quotients_are_correctly_rounded(moe):
    import torch
    rng = np.random.default_rng(2026)
    a, b = _cases(rng, 1 << 20)
    out = moe.check_quotients(torch.from_numpy(a).cuda(), torch.from_numpy(b).cuda()).cpu().numpy()
    ref = (a.astype(np.float64) / b.astype(np.float64)).astype(np.float32)
    for col in range(3):
        bad = np.flatnonzero(out[:, col].view(np.uint32) != ref.view(np.uint32))
        assert bad.size == 0, (col, a[bad[:4]], b[bad[:4]], out[bad[:4]], ref[bad[:4]])
    # the plain reciprocal product is not the quotient on these inputs (the
    # check can tell the two apart)
    rcp = (a * (np.float32(1.0) / b)).astype(np.float32)
    assert np.count_nonzero(rcp != ref) > 1000
