"""moe_dispatch_noalloc, the dispatch entry point for callers that cannot
allocate device memory while they dispatch (it keeps its scratch in a fixed
array inside the library), must give exactly what moe_dispatch gives with a
caller workspace. Two calls in a row with different inputs check that the
contents left in the shared array by one call do not leak into the next.
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


@pytest.mark.parametrize("N", [64, 128])
def test_noalloc_matches_workspace_dispatch(moe, N):
    import torch
    K = 8
    # second call smaller than the first, so stale chunk counts would show up
    for seed, T in ((1, 262144), (2, 4097)):
        k, ids = _inputs(seed + N, T, N, K)
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


def test_noalloc_rejects_oversize(moe):
    import ctypes
    lib = moe.library()
    fake = ctypes.c_void_p(256)
    assert lib.moe_dispatch_noalloc(fake, fake, (1 << 18) + 1, 64, 8, fake, fake, fake, None) == 2
