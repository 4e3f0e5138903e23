"""GPU parity of a stack of OLMoE-shaped MoE layers with the residual add
between layers (x_{l+1} = bf16(x_l + MoE_l(x_l)), no attention), the 16-layer
stack's shapes at T = 4096 with its first three layers.

Teacher-forced per layer: the oracle gets the GPU's own bf16 input x_l of
layer l and is compared with the GPU's x_{l+1} on sampled tokens, within the
layer tolerance (tokens whose elbow decision flips between the GPU's fp32
logits and the oracle's fp64 logits are counted and left out). The
free-running difference against an oracle-only chain is not gated."""
import numpy as np
import pytest

import oracle
from paper_2608_04401_gb300 import synth

from gpu_util import assert_layer_close, to_dev, to_dev_bf16

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


def _bits(t):
    import torch
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def test_stack_teacher_forced(moe):
    import torch
    w = synth.WORKLOADS["stack16_t4k"]
    T, d, N, I, K = w["T"], w["d"], w["N"], w["I"], w["K"]
    L = 3
    x0, routers = synth.stack_inputs(T, d, N, L, w["seed"])
    ws = torch.empty(moe.layer_workspace_size(T, d, N, I, K), dtype=torch.uint8, device="cuda")
    rows = np.unique(np.concatenate([[0, T - 1], np.random.default_rng(3).choice(T, 24, replace=False)]))
    cur = to_dev_bf16(x0)
    mean_k = []
    for l in range(L):
        wgu, wd = synth.expert_weights(synth.stack_expert_seed(w["seed"], l), N, d, I)
        x_in = _bits(cur)
        nxt, it = moe.moe_layer_forward(cur, to_dev_bf16(routers[l]), to_dev_bf16(wgu),
                                        to_dev_bf16(wd), K=K, residual=cur, ws=ws,
                                        return_intermediates=True)
        moe.read_device_error(ws)
        got_k = it["k"].cpu().numpy()
        got_ids = it["ids"].cpu().numpy()
        mean_k.append(float(got_k.mean()))
        # the layer's routing is bit-exact on its own fp32 logits
        r = oracle.route(it["logits"].cpu().numpy(), K=K)
        assert np.array_equal(r["k"], got_k) and np.array_equal(r["ids"], got_ids)
        # teacher-forced output on sampled tokens
        ref = oracle.layer_rows(x_in, routers[l], wgu, wd, rows=rows, K=K, residual_bits=x_in)
        same = (got_k[rows] == ref["k"]) & np.all(got_ids[rows] == ref["ids"], axis=1)
        assert same.mean() >= 0.9, f"layer {l}: routing flips on {np.count_nonzero(~same)} rows"
        y = nxt.float().cpu().numpy().astype(np.float64)
        assert_layer_close(y[rows][same], ref["y"][same], f"layer {l}")
        # the residual path: the output differs from the input only by the MoE term
        assert np.all(np.isfinite(y))
        cur = nxt
    assert all(1.0 <= m <= K for m in mean_k)
