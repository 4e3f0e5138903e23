"""GPU parity of the tail / head randomisation of Sec. 2.2
(elbow_route_randomized) against the oracle: ids, gates and k bit-exact on the
same logits and the same uint32 random numbers."""
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


@pytest.mark.parametrize("N", [64, 128])
@pytest.mark.parametrize("mode", [2, 3])
@pytest.mark.parametrize("renorm", [0, 1])
def test_randomized_bitexact(moe, N, mode, renorm):
    import torch
    rng = np.random.default_rng(N * 10 + mode + renorm)
    T, K = 3001, 8
    lg = synth.boosted_logits(rng, T, N)
    lg[:5] = 0.0                       # uniform curves (k = 1)
    lg[5, :N - 1] = 4.0                # elbow far out (k = K)
    rnd = rng.integers(0, 2**32, size=(T, K), dtype=np.uint32)
    rnd[6] = 0xFFFFFFFF
    rd = torch.from_numpy(rnd.view(np.int32)).cuda()
    k, ids, gates = moe.elbow_route_randomized(to_dev(lg), rd, K=K, mode=mode, renorm=renorm)
    ref = oracle.route_randomized(lg, rnd, K=K, mode=mode, renorm=renorm)
    assert np.array_equal(k.cpu().numpy(), ref["k"])
    assert np.array_equal(ids.cpu().numpy(), ref["ids"])
    assert np.array_equal(gates.cpu().numpy().view(np.uint32), ref["gates"].view(np.uint32))


def test_randomized_small_k(moe):
    import torch
    rng = np.random.default_rng(5)
    T, K = 777, 3
    lg = synth.boosted_logits(rng, T, 64)
    rnd = rng.integers(0, 2**32, size=(T, K), dtype=np.uint32)
    rd = torch.from_numpy(rnd.view(np.int32)).cuda()
    for mode in (2, 3):
        k, ids, gates = moe.elbow_route_randomized(to_dev(lg), rd, K=K, mode=mode)
        ref = oracle.route_randomized(lg, rnd, K=K, mode=mode)
        assert np.array_equal(ids.cpu().numpy(), ref["ids"])
        assert np.array_equal(gates.cpu().numpy().view(np.uint32), ref["gates"].view(np.uint32))
