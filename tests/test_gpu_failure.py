"""Failure detection without a GPU fault: the bounded wait that every GEMM
pipeline uses gives up on a barrier that nothing arrives on, reports
MOE_ERR_DEVICE_TIMEOUT through the device error word, and leaves the context
usable (routing afterwards is still bit-exact)."""
import time

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


def test_bounded_wait_times_out_and_context_survives(moe):
    import torch
    err = torch.zeros(4, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    status = moe.check_bounded_wait(err, seconds=0.2)
    dt = time.perf_counter() - t0
    assert status == 5                      # MOE_ERR_DEVICE_TIMEOUT
    assert int(err[0].item()) != 0
    assert 0.15 <= dt < 5.0, dt
    # the context is still usable
    lg = synth.boosted_logits(np.random.default_rng(9), 1000, 64)
    k, ids, gates = moe.elbow_route(to_dev(lg))
    ref = oracle.route(lg, K=8)
    assert np.array_equal(k.cpu().numpy(), ref["k"])
    assert np.array_equal(ids.cpu().numpy(), ref["ids"])
    # and a clean call clears the word
    ws = torch.zeros(64, dtype=torch.int32, device="cuda")
    assert moe.library().moe_read_device_error(ws.data_ptr(), None) == 0
