"""GB300 (sm_103a) elbow-routed MoE layer: thin Python binding of the C ABI.

Every function here marshals torch CUDA tensors into the C entry points of
libelbow_moe.so (declared in include/elbow_moe.h) and allocates the outputs
with torch; all arithmetic runs in the library's CUDA kernels. There is no
fallback: if the library is missing or a CUDA device is absent, calls raise.

Names follow the C ABI: elbow_route, moe_dispatch, moe_layer_forward, and the
step-level entry points router_logits, gather_rows, expert_gate_up,
expert_down, combine.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

__all__ = [
    "MODE_ELBOW", "MODE_TOPK", "MoeError", "library", "build", "route_diagnostics", "RouteDiag", "check_bounded_wait", "check_quotients", "elbow_route_warp",
    "elbow_route_randomized", "MODE_RAND_TAIL", "MODE_RAND_HEAD",
    "elbow_route", "moe_dispatch", "moe_dispatch_noalloc", "dispatch_workspace_size", "layer_workspace_size",
    "moe_layer_forward", "read_device_error", "router_logits", "gather_rows",
    "expert_gate_up", "expert_down", "combine",
]

MODE_ELBOW = 0
MODE_TOPK = 1

_HERE = os.path.dirname(os.path.abspath(__file__))
# ELBOW_MOE_DEBUG=1 in the environment loads the bounds-checked debug build
# (build(debug=True)) instead of the release library
_DEBUG = os.environ.get("ELBOW_MOE_DEBUG", "") == "1"
_LIB_PATH = os.path.join(_HERE, "_lib", "debug" if _DEBUG else "", "libelbow_moe.so")
_lock = threading.Lock()
_lib = None


class MoeError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = library().moe_status_string(status).decode() if _lib is not None else str(status)
        super().__init__(f"{where}: {msg}")


class RouteParams(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int), ("eps", ctypes.c_float), ("mode", ctypes.c_int),
                ("renorm", ctypes.c_int)]


class RouteDiag(ctypes.Structure):
    """Host mirror of moe_route_diag (include/elbow_moe.h)."""
    _fields_ = [("tokens", ctypes.c_int64), ("sharp_elbows", ctypes.c_int64),
                ("k_hist", ctypes.c_int64 * 9), ("elbow_hist", ctypes.c_int64 * 128),
                ("theta_hist", ctypes.c_int64 * 181), ("load_top", ctypes.c_int64 * 128),
                ("load_elb", ctypes.c_int64 * 128), ("mean_k", ctypes.c_double),
                ("delta", ctypes.c_double), ("l1", ctypes.c_double), ("l1_bound", ctypes.c_double),
                ("top1_change", ctypes.c_double), ("cv2_change", ctypes.c_double),
                ("cv2_bound", ctypes.c_double), ("top1_share_change_pct", ctypes.c_double),
                ("cv_change_pct", ctypes.c_double)]


def build(force: bool = False, debug: bool = None) -> str:
    """Compile libelbow_moe.so in-tree (nvcc, sm_103a); debug (default: as
    ELBOW_MOE_DEBUG says) builds the bounds-checked library."""
    from . import buildlib
    return buildlib.build(force=force, debug=_DEBUG if debug is None else debug)


def debug_violations() -> int:
    """Debug build only: synchronises the device and returns (and resets) the
    number of failed device bounds checks since the last call."""
    v = ctypes.c_uint32(0)
    _check(library().moe_debug_violations(ctypes.byref(v)), "moe_debug_violations")
    return int(v.value)


def library():
    """Load libelbow_moe.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"{_LIB_PATH} is missing: run paper_2608_04401_gb300.build()")
        lib = ctypes.CDLL(_LIB_PATH)
        P, i64, i32, f32, sz = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float,
                                ctypes.c_size_t)
        RP = ctypes.POINTER(RouteParams)
        sig = {
            "moe_status_string": ([i32], ctypes.c_char_p),
            "elbow_route": ([P, i64, i32, RP, P, P, P, P], i32),
            "elbow_route_with_counts": ([P, i64, i32, RP, P, P, P, P, P], i32),
            "elbow_route_warp": ([P, i64, i32, RP, P, P, P, P], i32),
            "moe_route_diagnostics": ([P, i64, i32, RP, P, P, P, P], i32),
            "elbow_route_randomized": ([P, i64, i32, RP, P, P, P, P, P], i32),
            "moe_dispatch_workspace_size": ([i64, i32, i32], sz),
            "moe_dispatch": ([P, P, i64, i32, i32, P, P, P, P, sz, P], i32),
            "moe_dispatch_tile_offsets": ([P, i64, i32, i32], P),
            "moe_dispatch_noalloc": ([P, P, i64, i32, i32, P, P, P, P], i32),
            "moe_check_quotients": ([P, P, i64, P, P], i32),
            "moe_debug_violations": ([P], i32),
            "moe_dispatch_chunk_counts": ([P, i64, i32, i32], P),
            "moe_dispatch_counted": ([P, P, i64, i32, i32, P, P, P, P, sz, P], i32),
            "moe_layer_workspace_size": ([i64, i32, i32, i32, i32], sz),
            "moe_layer_forward": ([P, P, P, P, i64, i32, i32, i32, RP, P, P, P, P, P, P, P, P, sz, P],
                                  i32),
            "moe_read_device_error": ([P, P], i32),
            "moe_check_bounded_wait": ([P, ctypes.c_double, P], i32),
            "moe_router_logits": ([P, P, i64, i32, i32, P, P, P], i32),
            "moe_expert_gate_up": ([P, P, P, P, i64, i32, i32, i32, P, P, P], i32),
            "moe_expert_down": ([P, P, P, P, i64, i32, i32, i32, P, P, P], i32),
            "moe_gather_rows": ([P, P, P, i64, i64, i32, i32, P, P], i32),
            "moe_combine": ([P, P, P, P, P, i64, i32, i32, P, P], i32),
            "moe_router_route": ([P, P, i64, i32, i32, RP, P, P, P, P, P, P, P], i32),
            "moe_expert_gate_up_gathered": ([P, i64, P, P, P, P, i64, i32, i32, i32, P, P, P], i32),
            "moe_expert_gate_up_decode": ([P, P, P, i64, i64, i32, i32, i32, P, P, P], i32),
            "moe_expert_down_decode": ([P, P, P, i64, i64, i32, i32, i32, P, P, P], i32),
            "moe_expert_gate_up_gemv": ([P, i64, P, P, P, i64, i32, i32, i32, i32, P, P, P], i32),
            "moe_expert_down_gemv": ([P, P, P, i64, i64, i32, i32, i32, i32, P, P, P], i32),
        }
        for name, (args, res) in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _lib = lib
        return lib


def _torch():
    import torch
    return torch


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(status: int, where: str):
    if status != 0:
        raise MoeError(status, where)


def _cuda(t, dtype, name):
    torch = _torch()
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _params(K, eps, mode, renorm):
    return ctypes.byref(RouteParams(int(K), float(eps), int(mode), int(renorm)))


def elbow_route(logits, K: int = 8, eps: float = 1e-8, mode: int = MODE_ELBOW, renorm: int = 0,
                stream=None):
    """Route fp32 logits [T, N]: returns (k [T] int32, ids [T, K] int32, gates [T, K] fp32)."""
    torch = _torch()
    lib = library()
    _cuda(logits, torch.float32, "logits")
    T, N = logits.shape
    k = torch.empty(T, dtype=torch.int32, device=logits.device)
    ids = torch.empty(T, K, dtype=torch.int32, device=logits.device)
    gates = torch.empty(T, K, dtype=torch.float32, device=logits.device)
    _check(lib.elbow_route(_p(logits), T, N, _params(K, eps, mode, renorm), _p(k), _p(ids),
                           _p(gates), _stream(stream)), "elbow_route")
    return k, ids, gates


def elbow_route_warp(logits, K: int = 8, eps: float = 1e-8, mode: int = MODE_ELBOW, renorm: int = 0,
                     stream=None):
    """elbow_route with one warp per token (same results; the small-batch kernel)."""
    torch = _torch()
    _cuda(logits, torch.float32, "logits")
    T, N = logits.shape
    k = torch.empty(T, dtype=torch.int32, device=logits.device)
    ids = torch.empty(T, K, dtype=torch.int32, device=logits.device)
    gates = torch.empty(T, K, dtype=torch.float32, device=logits.device)
    _check(library().elbow_route_warp(_p(logits), T, N, _params(K, eps, mode, renorm), _p(k),
                                      _p(ids), _p(gates), _stream(stream)), "elbow_route_warp")
    return k, ids, gates


def _check_chunk_counts(cc, T, N):
    """The per-chunk counts a router writes: int32 [N, ceil(T/128)], contiguous."""
    torch = _torch()
    _cuda(cc, torch.int32, "chunk_counts")
    if tuple(cc.shape) != (N, _num_chunks(T)):
        raise ValueError(f"chunk_counts must be a contiguous [{N}, {_num_chunks(T)}] int32 tensor")


def _num_chunks(T):
    """128-token chunks of the dispatch counts."""
    return (T + 127) // 128


def elbow_route_with_counts(logits, chunk_counts, K: int = 8, eps: float = 1e-8,
                            mode: int = MODE_ELBOW, renorm: int = 0, stream=None):
    """elbow_route that also writes the per-chunk expert counts (an int32 tensor of
    [N, ceil(T/128)], e.g. dispatch_chunk_counts(ws, ...)). Returns (k, ids, gates)."""
    torch = _torch()
    lib = library()
    _cuda(logits, torch.float32, "logits")
    T, N = logits.shape
    k = torch.empty(T, dtype=torch.int32, device=logits.device)
    ids = torch.empty(T, K, dtype=torch.int32, device=logits.device)
    gates = torch.empty(T, K, dtype=torch.float32, device=logits.device)
    _check_chunk_counts(chunk_counts, T, N)
    _check(lib.elbow_route_with_counts(_p(logits), T, N, _params(K, eps, mode, renorm), _p(k),
                                       _p(ids), _p(gates), _p(chunk_counts), _stream(stream)),
           "elbow_route_with_counts")
    return k, ids, gates


MODE_RAND_TAIL = 2
MODE_RAND_HEAD = 3


def elbow_route_randomized(logits, rand, K: int = 8, eps: float = 1e-8, mode: int = MODE_RAND_TAIL,
                           renorm: int = 0, stream=None):
    """Tail (MODE_RAND_TAIL) or head (MODE_RAND_HEAD) randomisation with the
    uint32 random numbers rand [T, K] (an int32 tensor holding the bits is
    accepted too). Returns (k, ids, gates)."""
    torch = _torch()
    _cuda(logits, torch.float32, "logits")
    T, N = logits.shape
    if rand.dtype not in (torch.int32, getattr(torch, "uint32", torch.int32)) or \
            tuple(rand.shape) != (T, K) or not rand.is_contiguous() or rand.device != logits.device:
        raise ValueError(f"rand must be a contiguous [{T}, {K}] 32-bit tensor on {logits.device}")
    k = torch.empty(T, dtype=torch.int32, device=logits.device)
    ids = torch.empty(T, K, dtype=torch.int32, device=logits.device)
    gates = torch.empty(T, K, dtype=torch.float32, device=logits.device)
    _check(library().elbow_route_randomized(_p(logits), T, N, _params(K, eps, mode, renorm),
                                            _p(rand), _p(k), _p(ids), _p(gates), _stream(stream)),
           "elbow_route_randomized")
    return k, ids, gates


def check_quotients(a, b, stream=None):
    """The routing's correctly rounded quotients a / b on the device: returns
    [n, 3] fp32 = (scalar form, packed two-lane form, CUDA's __fdiv_rn)."""
    torch = _torch()
    _cuda(a, torch.float32, "a")
    _cuda(b, torch.float32, "b")
    if a.numel() != b.numel():
        raise ValueError("a and b must have the same size")
    out = torch.empty(a.numel(), 3, dtype=torch.float32, device=a.device)
    _check(library().moe_check_quotients(_p(a), _p(b), a.numel(), _p(out), _stream(stream)),
           "moe_check_quotients")
    return out


def check_bounded_wait(err, seconds: float = 0.2, stream=None) -> int:
    """Run the GEMMs' bounded wait on a barrier nothing arrives on; returns the
    status moe_read_device_error reports afterwards (MOE_ERR_DEVICE_TIMEOUT = 5)."""
    lib = library()
    _check(lib.moe_check_bounded_wait(_p(err), float(seconds), _stream(stream)),
           "moe_check_bounded_wait")
    return int(lib.moe_read_device_error(_p(err), _stream(stream)))


def route_diagnostics(logits, K: int = 8, eps: float = 1e-8, per_token: bool = True,
                      diag=None, stream=None):
    """Routing diagnostics of fp32 logits [T, N] (moe_route_diagnostics).
    Returns (stats dict, elbow [T] int32 or None, theta [T] fp32 degrees or None);
    `diag` may be a device uint8 tensor of sizeof(RouteDiag) bytes to reuse."""
    torch = _torch()
    _cuda(logits, torch.float32, "logits")
    T, N = logits.shape
    dev = logits.device
    if diag is None:
        diag = torch.empty(ctypes.sizeof(RouteDiag), dtype=torch.uint8, device=dev)
    el = torch.empty(T, dtype=torch.int32, device=dev) if per_token else None
    th = torch.empty(T, dtype=torch.float32, device=dev) if per_token else None
    _check(library().moe_route_diagnostics(_p(logits), T, N, _params(K, eps, MODE_ELBOW, 0),
                                           _p(el), _p(th), _p(diag), _stream(stream)),
           "moe_route_diagnostics")
    host = RouteDiag.from_buffer_copy(diag.cpu().numpy().tobytes())
    out = {}
    for name, _ in RouteDiag._fields_:
        v = getattr(host, name)
        out[name] = np.array(v[:], dtype=np.int64) if hasattr(v, "__len__") else v
    for name in ("elbow_hist", "load_top", "load_elb"):
        out[name] = out[name][:N]
    return out, el, th


def dispatch_workspace_size(T: int, N: int, K: int) -> int:
    return int(library().moe_dispatch_workspace_size(T, N, K))


def moe_dispatch(k, ids, N: int, ws=None, stream=None):
    """Stable token-to-expert dispatch: returns (offsets [N+1], perm [T*K], pair_pos [T, K],
    ws). perm is valid up to offsets[N]; ws holds the m-tile offsets."""
    torch = _torch()
    lib = library()
    _cuda(k, torch.int32, "k")
    _cuda(ids, torch.int32, "ids")
    T, K = ids.shape
    dev = ids.device
    need = dispatch_workspace_size(T, N, K)
    if ws is None:
        ws = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
    offsets = torch.empty(N + 1, dtype=torch.int32, device=dev)
    perm = torch.empty(max(1, T * K), dtype=torch.int32, device=dev)
    pair_pos = torch.empty(T, K, dtype=torch.int32, device=dev)
    _check(lib.moe_dispatch(_p(k), _p(ids), T, N, K, _p(offsets), _p(perm), _p(pair_pos), _p(ws),
                            ws.numel(), _stream(stream)), "moe_dispatch")
    return offsets, perm, pair_pos, ws


def dispatch_chunk_counts(ws, T: int, N: int, K: int):
    """View of the [N, ceil(T/128)] per-chunk expert counts inside a dispatch workspace
    (chunk c = tokens 128 c .. 128 c + 127)."""
    torch = _torch()
    ptr = library().moe_dispatch_chunk_counts(_p(ws), T, N, K)
    off = ptr - ws.data_ptr()
    nblk = _num_chunks(T)
    return ws[off: off + 4 * N * nblk].view(torch.int32).view(N, nblk)


def moe_dispatch_counted(k, ids, N: int, ws, stream=None):
    """moe_dispatch using the per-chunk counts already in ws (from router_route)."""
    torch = _torch()
    lib = library()
    T, K = ids.shape
    dev = ids.device
    offsets = torch.empty(N + 1, dtype=torch.int32, device=dev)
    perm = torch.empty(max(1, T * K), dtype=torch.int32, device=dev)
    pair_pos = torch.empty(T, K, dtype=torch.int32, device=dev)
    _check(lib.moe_dispatch_counted(_p(k), _p(ids), T, N, K, _p(offsets), _p(perm), _p(pair_pos),
                                    _p(ws), ws.numel(), _stream(stream)), "moe_dispatch_counted")
    return offsets, perm, pair_pos


def moe_dispatch_noalloc(k, ids, N: int, offsets=None, perm=None, pair_pos=None, stream=None):
    """moe_dispatch without a workspace (the library's fixed scratch array is used).
    Output buffers may be passed in; returns (offsets, perm, pair_pos)."""
    torch = _torch()
    lib = library()
    _cuda(k, torch.int32, "k")
    _cuda(ids, torch.int32, "ids")
    if ids.dim() != 2:
        raise ValueError("ids must be [T, K]")
    T, K = ids.shape
    dev = ids.device
    if k.numel() != T or k.device != dev:
        raise ValueError(f"k must hold T = {T} counts on {dev}")
    if offsets is None:
        offsets = torch.empty(N + 1, dtype=torch.int32, device=dev)
    if perm is None:
        perm = torch.empty(max(1, T * K), dtype=torch.int32, device=dev)
    if pair_pos is None:
        pair_pos = torch.empty(T, K, dtype=torch.int32, device=dev)
    # the C entry point cannot see buffer sizes: every caller-supplied buffer is
    # checked here, before the kernels could write past its end
    for name, buf, need in (("offsets", offsets, N + 1), ("perm", perm, max(1, T * K)),
                            ("pair_pos", pair_pos, T * K)):
        _cuda(buf, torch.int32, name)
        if buf.device != dev:
            raise ValueError(f"{name} must be on {dev}")
        if buf.numel() < need:
            raise ValueError(f"{name} holds {buf.numel()} entries, needs {need}")
    _check(lib.moe_dispatch_noalloc(_p(k), _p(ids), T, N, K, _p(offsets), _p(perm), _p(pair_pos),
                                    _stream(stream)), "moe_dispatch_noalloc")
    return offsets, perm, pair_pos


def dispatch_tile_offsets(ws, T: int, N: int, K: int):
    """The [N+1] m-tile offsets a moe_dispatch left in its workspace (a view)."""
    torch = _torch()
    ptr = library().moe_dispatch_tile_offsets(_p(ws), T, N, K)
    off = ptr - ws.data_ptr()
    return ws[off: off + 4 * (N + 1)].view(torch.int32)


def layer_workspace_size(T: int, d: int, N: int, I: int, K: int) -> int:
    return int(library().moe_layer_workspace_size(T, d, N, I, K))


def moe_layer_forward(x, w_router, w_gate_up, w_down, K: int = 8, eps: float = 1e-8,
                      mode: int = MODE_ELBOW, renorm: int = 0, residual=None, y=None, ws=None,
                      return_intermediates: bool = False, stream=None):
    """One MoE layer forward. x [T, d], w_router [N, d], w_gate_up [N, 2I, d],
    w_down [N, d, I] (bf16 CUDA tensors). Returns y [T, d] bf16, or
    (y, dict(logits, k, ids, gates, offsets)) with return_intermediates."""
    torch = _torch()
    lib = library()
    bf = torch.bfloat16
    for t, n in ((x, "x"), (w_router, "w_router"), (w_gate_up, "w_gate_up"), (w_down, "w_down")):
        _cuda(t, bf, n)
    if residual is not None:
        _cuda(residual, bf, "residual")
    T, d = x.shape
    N = w_router.shape[0]
    I = w_gate_up.shape[1] // 2
    dev = x.device
    if y is None:
        y = torch.empty(T, d, dtype=bf, device=dev)
    need = layer_workspace_size(T, d, N, I, K)
    if ws is None:
        ws = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
    inter = None
    if return_intermediates:
        inter = dict(logits=torch.empty(T, N, dtype=torch.float32, device=dev),
                     k=torch.empty(T, dtype=torch.int32, device=dev),
                     ids=torch.empty(T, K, dtype=torch.int32, device=dev),
                     gates=torch.empty(T, K, dtype=torch.float32, device=dev),
                     offsets=torch.empty(N + 1, dtype=torch.int32, device=dev))
    g = (lambda n: _p(inter[n])) if inter else (lambda n: None)
    _check(lib.moe_layer_forward(_p(x), _p(w_router), _p(w_gate_up), _p(w_down), T, d, N, I,
                                 _params(K, eps, mode, renorm), _p(residual), _p(y), g("logits"),
                                 g("k"), g("ids"), g("gates"), g("offsets"), _p(ws), ws.numel(),
                                 _stream(stream)), "moe_layer_forward")
    return (y, inter) if return_intermediates else y


def read_device_error(ws, stream=None):
    """Synchronise the stream and raise MoeError if a layer kernel timed out."""
    _check(library().moe_read_device_error(_p(ws), _stream(stream)), "device")


def router_logits(x, w_router, err=None, stream=None):
    torch = _torch()
    _cuda(x, torch.bfloat16, "x")
    _cuda(w_router, torch.bfloat16, "w_router")
    T, d = x.shape
    N = w_router.shape[0]
    out = torch.empty(T, N, dtype=torch.float32, device=x.device)
    _check(library().moe_router_logits(_p(x), _p(w_router), T, d, N, _p(out), _p(err),
                                       _stream(stream)), "moe_router_logits")
    return out


def router_route(x, w_router, K: int = 8, eps: float = 1e-8, mode: int = MODE_ELBOW,
                 renorm: int = 0, with_logits: bool = True, with_counts: bool = True, err=None,
                 chunk_counts=None, stream=None):
    """Router GEMM with the elbow routing in its epilogue. Returns
    (k, ids, gates, logits or None, chunk_counts [N, ceil(T/128)] or None)."""
    torch = _torch()
    _cuda(x, torch.bfloat16, "x")
    _cuda(w_router, torch.bfloat16, "w_router")
    T, d = x.shape
    N = w_router.shape[0]
    dev = x.device
    k = torch.empty(T, dtype=torch.int32, device=dev)
    ids = torch.empty(T, K, dtype=torch.int32, device=dev)
    gates = torch.empty(T, K, dtype=torch.float32, device=dev)
    lg = torch.empty(T, N, dtype=torch.float32, device=dev) if with_logits else None
    cc = chunk_counts
    if cc is None and with_counts:
        cc = torch.zeros(N, _num_chunks(T), dtype=torch.int32, device=dev)
    if cc is not None:
        _check_chunk_counts(cc, T, N)
    _check(library().moe_router_route(_p(x), _p(w_router), T, d, N, _params(K, eps, mode, renorm),
                                      _p(lg), _p(k), _p(ids), _p(gates), _p(cc), _p(err),
                                      _stream(stream)), "moe_router_route")
    return k, ids, gates, lg, cc


def expert_gate_up_gathered(x, perm, w_gate_up, offsets, tile_off, P: int, err=None, stream=None):
    torch = _torch()
    T, d = x.shape
    N, I2, _ = w_gate_up.shape
    h = torch.empty(max(P, 1), I2 // 2, dtype=torch.bfloat16, device=x.device)
    _check(library().moe_expert_gate_up_gathered(_p(x), T, _p(perm), _p(w_gate_up), _p(offsets),
                                                 _p(tile_off), P, d, N, I2 // 2, _p(h), _p(err),
                                                 _stream(stream)), "moe_expert_gate_up_gathered")
    return h


def expert_gate_up_decode(xs, w_gate_up, offsets, T: int, err=None, stream=None):
    """Decode-shaped gate/up GEMM (T <= 64): h [P, I] from the dispatched rows xs [P, d]."""
    torch = _torch()
    P, d = xs.shape
    N, I2, _ = w_gate_up.shape
    h = torch.empty(max(P, 1), I2 // 2, dtype=torch.bfloat16, device=xs.device)
    _check(library().moe_expert_gate_up_decode(_p(xs), _p(w_gate_up), _p(offsets), T, P, d, N,
                                               I2 // 2, _p(h), _p(err), _stream(stream)),
           "moe_expert_gate_up_decode")
    return h


def expert_down_decode(h, w_down, offsets, T: int, err=None, stream=None):
    """Decode-shaped down GEMM (T <= 64): o [P, d] from h [P, I]."""
    torch = _torch()
    P, I = h.shape
    N, d, _ = w_down.shape
    o = torch.empty(max(P, 1), d, dtype=torch.bfloat16, device=h.device)
    _check(library().moe_expert_down_decode(_p(h), _p(w_down), _p(offsets), T, P, d, N, I, _p(o),
                                            _p(err), _stream(stream)), "moe_expert_down_decode")
    return o


def expert_gate_up_gemv(x, perm, w_gate_up, offsets, P: int, K: int = 8, err=None, stream=None):
    """h [P, I] for batches of T <= 4 tokens (CUDA-core contractions reading x through perm)."""
    torch = _torch()
    bf = torch.bfloat16
    _cuda(x, bf, "x")
    _cuda(w_gate_up, bf, "w_gate_up")
    _cuda(perm, torch.int32, "perm")
    _cuda(offsets, torch.int32, "offsets")
    T, d = x.shape
    N, I2, _ = w_gate_up.shape
    I = I2 // 2
    h = torch.zeros(max(P, 1), I, dtype=bf, device=x.device)
    _check(library().moe_expert_gate_up_gemv(_p(x), T, _p(perm), _p(offsets), _p(w_gate_up), P, d,
                                             N, I, K, _p(h), _p(err), _stream(stream)),
           "moe_expert_gate_up_gemv")
    return h


def expert_down_gemv(h, w_down, offsets, T: int, K: int = 8, err=None, stream=None):
    """o [P, d] for batches of T <= 4 tokens (CUDA-core contractions)."""
    torch = _torch()
    bf = torch.bfloat16
    _cuda(h, bf, "h")
    _cuda(w_down, bf, "w_down")
    _cuda(offsets, torch.int32, "offsets")
    P, I = h.shape
    N, d, _ = w_down.shape
    o = torch.zeros(P, d, dtype=bf, device=h.device)
    _check(library().moe_expert_down_gemv(_p(h), _p(offsets), _p(w_down), T, P, d, N, I, K, _p(o),
                                          _p(err), _stream(stream)),
           "moe_expert_down_gemv")
    return o


def gather_rows(x, perm, offsets, P: int, stream=None):
    torch = _torch()
    T, d = x.shape
    N = offsets.numel() - 1
    xs = torch.empty(max(P, 1), d, dtype=x.dtype, device=x.device)
    _check(library().moe_gather_rows(_p(x), _p(perm), _p(offsets), T, P, d, N, _p(xs),
                                     _stream(stream)), "moe_gather_rows")
    return xs


def expert_gate_up(xs, w_gate_up, offsets, tile_off, err=None, stream=None):
    torch = _torch()
    P, d = xs.shape
    N, I2, _ = w_gate_up.shape
    h = torch.empty(P, I2 // 2, dtype=torch.bfloat16, device=xs.device)
    _check(library().moe_expert_gate_up(_p(xs), _p(w_gate_up), _p(offsets), _p(tile_off), P, d, N,
                                        I2 // 2, _p(h), _p(err), _stream(stream)),
           "moe_expert_gate_up")
    return h


def expert_down(h, w_down, offsets, tile_off, err=None, stream=None):
    torch = _torch()
    P, I = h.shape
    N, d, _ = w_down.shape
    o = torch.empty(P, d, dtype=torch.bfloat16, device=h.device)
    _check(library().moe_expert_down(_p(h), _p(w_down), _p(offsets), _p(tile_off), P, d, N, I,
                                     _p(o), _p(err), _stream(stream)), "moe_expert_down")
    return o


def combine(o, k, pair_pos, gates, residual=None, stream=None):
    torch = _torch()
    T, K = pair_pos.shape
    d = o.shape[1]
    y = torch.empty(T, d, dtype=torch.bfloat16, device=o.device)
    _check(library().moe_combine(_p(o), _p(k), _p(pair_pos), _p(gates), _p(residual), T, d, K,
                                 _p(y), _stream(stream)), "moe_combine")
    return y
