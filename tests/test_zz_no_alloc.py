"""moe_dispatch_noalloc, the dispatch entry point for callers that cannot
allocate device memory while they dispatch (it keeps its scratch in a fixed
array inside the library), must give exactly what moe_dispatch gives with a
caller workspace. Calls follow each other on the one shared array, a large one
before smaller ones, so that contents one call leaves there would show up in
the next: the multi-chunk path (count, scan, scatter), the single-chunk path
(T <= 128, no count or scan), T = 0, and caps K < 8 (element loads of the ids).
This file is collected last."""
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


def _inputs(seed, T, N, K):
    rng = np.random.default_rng(seed)
    ids = np.argsort(rng.random((T, N)), axis=1)[:, :K].astype(np.int32)
    k = rng.integers(1, K + 1, size=T).astype(np.int32)
    return k, ids


def _compare(moe, k, ids, N):
    import torch
    T, K = ids.shape
    dk = torch.from_numpy(k).cuda()
    dids = torch.from_numpy(ids).cuda()
    off_a, perm_a, pp_a = moe.moe_dispatch_noalloc(dk, dids, N)
    off_b, perm_b, pp_b, _ = moe.moe_dispatch(dk, dids, N)
    torch.cuda.synchronize()
    off_a, off_b = off_a.cpu().numpy(), off_b.cpu().numpy()
    assert np.array_equal(off_a, off_b)
    P = int(off_b[-1])
    assert P == int(k.sum())
    assert np.array_equal(perm_a.cpu().numpy()[:P], perm_b.cpu().numpy()[:P])
    assert np.array_equal(pp_a.cpu().numpy(), pp_b.cpu().numpy())


@pytest.mark.parametrize("N", [64, 128])
def test_noalloc_matches_workspace_dispatch(moe, N):
    K = 8
    # second call smaller than the first, so stale chunk counts would show up
    for seed, T in ((1, 262144), (2, 4097)):
        k, ids = _inputs(seed + N, T, N, K)
        _compare(moe, k, ids, N)


@pytest.mark.parametrize("K", [1, 5, 8])
def test_noalloc_small_and_ragged_batches(moe, K):
    N = 64
    for seed, T in ((11, 4097), (12, 129), (13, 128), (14, 1), (15, 0), (16, 129)):
        k, ids = _inputs(seed * 10 + K, T, N, K)
        _compare(moe, k, ids, N)


def test_noalloc_rejects_oversize(moe):
    import ctypes
    lib = moe.library()
    fake = ctypes.c_void_p(256)
    assert lib.moe_dispatch_noalloc(fake, fake, (1 << 18) + 1, 64, 8, fake, fake, fake, None) == 2


def test_noalloc_binding_checks_buffers(moe):
    import torch
    k, ids = _inputs(3, 300, 64, 8)
    dk = torch.from_numpy(k).cuda()
    dids = torch.from_numpy(ids).cuda()
    small = torch.empty(10, dtype=torch.int32, device="cuda")
    for kw in ({"offsets": small}, {"perm": small}, {"pair_pos": small}):
        with pytest.raises(ValueError):
            moe.moe_dispatch_noalloc(dk, dids, 64, **kw)
    with pytest.raises(TypeError):
        moe.moe_dispatch_noalloc(dk, dids, 64, perm=torch.empty(300 * 8, dtype=torch.int64,
                                                                 device="cuda"))
    with pytest.raises(ValueError):
        moe.moe_dispatch_noalloc(dk[:299], dids, 64)
