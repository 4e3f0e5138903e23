"""Helpers shared by the GPU tests: moving synthetic inputs to the device and
the output tolerance of the layer (relative Frobenius error <= 5e-3 and
per-element |delta| <= 2e-2 * max|ref|, bf16 storage with fp32 accumulation)."""
import numpy as np

REL_FRO = 5e-3
REL_MAX = 2e-2


def to_dev_bf16(bits: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def to_dev(a: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def bf16_tensor_to_f64(t) -> np.ndarray:
    return t.float().cpu().numpy().astype(np.float64)


def assert_layer_close(got: np.ndarray, ref: np.ndarray, what: str = "y"):
    ref = np.asarray(ref, np.float64)
    got = np.asarray(got, np.float64)
    assert got.shape == ref.shape
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    fro = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    mx = np.abs(got - ref).max() / max(np.abs(ref).max(), 1e-30)
    assert fro <= REL_FRO and mx <= REL_MAX, f"{what}: rel_fro={fro:.3e} rel_max={mx:.3e}"
    return fro, mx
