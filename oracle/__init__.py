"""CPU oracle for the elbow-routed MoE layer (ctypes wrapper of elbow_oracle.c).

TEST INFRASTRUCTURE. Only the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package. The product path
(the CUDA library and its binding) never imports it and shares no code with it.

Functions and the passages they follow:
  route          Alg. 1 (softmax, descending sort, Kneedle deviation, elbow)
                 and the capped selection k = min(e, K) of Sec. 2.1
  dispatch       stable token-to-expert grouping of the selected pairs
  router_logits  l(x) = W_r x of Sec. 2, fp64 accumulation rounded to fp32
  layer_rows     the whole MoE layer forward (App. A.4) for chosen tokens, fp64
  load_balance   L_i, q_i, delta and the bounds of Theorem 1 / Corollaries 1-2
                 (App. A.3), the percentage changes of Sec. 2.4
  elbow_angle    the uncapped elbow index and the elbow angle of Sec. 2.3
  elbow_curve    Alg. 1's sorted p, normalised p' and deviation D per rank
  route_randomized  the tail / head randomisation experiment of Sec. 2.2
  exp / exp_max_ulp  the fp32 routing exponential and its error sweep
  threads / set_threads  the OpenMP thread count (timing support)
The readings taken where the paper is silent or garbled are listed in the
header of elbow_oracle.c.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "elbow_oracle.c")
_OUT = os.path.join(_HERE, "_lib", "libelbow_oracle.so")
_lock = threading.Lock()
_lib = None

MODE_ELBOW = 0
MODE_TOPK = 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no FP contraction)."""
    if not force and os.path.exists(_OUT) and os.path.getmtime(_OUT) >= os.path.getmtime(_SRC):
        return _OUT
    os.makedirs(os.path.dirname(_OUT), exist_ok=True)
    tmp = _OUT + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
           "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _OUT)
    return _OUT


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        # ORACLE_LIBRARY: a library built from a modified copy of elbow_oracle.c
        # (test support: the mutation tests check that the pins reject it)
        lib = ctypes.CDLL(os.environ.get("ORACLE_LIBRARY") or build())
        P = ctypes.c_void_p
        i64, i32, f32 = ctypes.c_int64, ctypes.c_int, ctypes.c_float
        lib.oracle_max_threads.argtypes = []
        lib.oracle_max_threads.restype = i32
        lib.oracle_set_threads.argtypes = [i32]
        lib.oracle_set_threads.restype = None
        lib.oracle_exp.argtypes = [f32]
        lib.oracle_exp.restype = f32
        lib.oracle_exp_max_ulp.argtypes = [f32, f32, P]
        lib.oracle_exp_max_ulp.restype = ctypes.c_double
        lib.oracle_route.argtypes = [P, i64, i32, i32, f32, i32, i32, P, P, P, P, P]
        lib.oracle_route.restype = i32
        lib.oracle_route_randomized.argtypes = [P, i64, i32, i32, f32, i32, i32, P, P, P, P]
        lib.oracle_route_randomized.restype = i32
        lib.oracle_elbow_curve.argtypes = [P, i64, i32, f32, P, P, P]
        lib.oracle_elbow_curve.restype = i32
        lib.oracle_elbow_angle.argtypes = [P, i64, i32, f32, P, P]
        lib.oracle_elbow_angle.restype = i32
        lib.oracle_angle_deg.argtypes = [i32, i32, f32]
        lib.oracle_angle_deg.restype = ctypes.c_double
        lib.oracle_dispatch.argtypes = [P, P, i64, i32, i32, P, P, P]
        lib.oracle_dispatch.restype = i32
        lib.oracle_router_logits.argtypes = [P, P, i64, i32, i32, P, i64, P]
        lib.oracle_router_logits.restype = None
        lib.oracle_layer_rows.argtypes = [P, P, P, P, i64, i32, i32, i32, i32, f32, i32, i32,
                                          P, P, i64, i32, P, P, P, P, P]
        lib.oracle_layer_rows.restype = i32
        _lib = lib
        return lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def threads() -> int:
    """OpenMP threads the oracle's parallel loops use."""
    return int(_load().oracle_max_threads())


def set_threads(n: int) -> None:
    """Set the OpenMP threads of the oracle's parallel loops (timing support)."""
    _load().oracle_set_threads(int(n))


def exp(z):
    """The routing exponential EXP on each fp32 element of z."""
    lib = _load()
    z = np.asarray(z, dtype=np.float32)
    return np.array([lib.oracle_exp(float(v)) for v in z.ravel()], dtype=np.float32).reshape(z.shape)


def exp_max_ulp(lo: float, hi: float):
    """(max ulp error of EXP over every fp32 in [lo, hi], worst z)."""
    lib = _load()
    wz = ctypes.c_float(0.0)
    err = lib.oracle_exp_max_ulp(lo, hi, ctypes.byref(wz))
    return err, wz.value


def elbow_curve(logits, eps: float = 1e-8):
    """Alg. 1's curve per token in sorted order: dict(p, pn, D), each [T, N]."""
    lib = _load()
    lg = _c(logits, np.float32)
    T, N = lg.shape
    out = {n: np.empty((T, N), np.float32) for n in ("p", "pn", "D")}
    if lib.oracle_elbow_curve(_ptr(lg), T, N, eps, _ptr(out["p"]), _ptr(out["pn"]),
                              _ptr(out["D"])) != 0:
        raise ValueError("oracle_elbow_curve: unsupported arguments")
    return out


def route(logits, K: int = 8, eps: float = 1e-8, mode: int = MODE_ELBOW, renorm: int = 0,
          with_sorted: bool = False):
    """Route fp32 logits [T, N]. Returns dict(k, ids, gates[, sorted_p, elbow])."""
    lib = _load()
    lg = _c(logits, np.float32)
    T, N = lg.shape
    k = np.empty(T, np.int32)
    ids = np.empty((T, K), np.int32)
    gates = np.empty((T, K), np.float32)
    sp = np.empty((T, N), np.float32) if with_sorted else None
    el = np.empty(T, np.int32) if with_sorted else None
    rc = lib.oracle_route(_ptr(lg), T, N, K, eps, mode, renorm, _ptr(k), _ptr(ids), _ptr(gates),
                          _ptr(sp), _ptr(el))
    if rc != 0:
        raise ValueError("oracle_route: unsupported arguments")
    out = dict(k=k, ids=ids, gates=gates)
    if with_sorted:
        out["sorted_p"] = sp
        out["elbow"] = el
    return out


def dispatch(k, ids, N: int):
    """Stable dispatch of the selected pairs. Returns dict(offsets, perm, pair_pos)."""
    lib = _load()
    k = _c(k, np.int32)
    ids = _c(ids, np.int32)
    T, K = ids.shape
    offsets = np.empty(N + 1, np.int32)
    perm = np.full(max(1, T * K), -1, np.int32)
    pair_pos = np.empty((T, K), np.int32)
    rc = lib.oracle_dispatch(_ptr(k), _ptr(ids), T, N, K, _ptr(offsets), _ptr(perm), _ptr(pair_pos))
    if rc != 0:
        raise ValueError("oracle_dispatch: invalid k or ids")
    return dict(offsets=offsets, perm=perm[: int(offsets[N])], pair_pos=pair_pos)


def router_logits(x_bits, w_router_bits, rows=None):
    """fp32 logits (fp64 accumulation) for the chosen rows of x (bf16 bits)."""
    lib = _load()
    x = _c(x_bits, np.uint16)
    wr = _c(w_router_bits, np.uint16)
    T, d = x.shape
    N = wr.shape[0]
    rows = np.arange(T, dtype=np.int64) if rows is None else _c(rows, np.int64)
    out = np.empty((len(rows), N), np.float32)
    lib.oracle_router_logits(_ptr(x), _ptr(wr), T, d, N, _ptr(rows), len(rows), _ptr(out))
    return out


def layer_rows(x_bits, w_router_bits, w_gate_up_bits, w_down_bits, rows=None, K: int = 8,
               eps: float = 1e-8, mode: int = MODE_ELBOW, renorm: int = 0, residual_bits=None,
               round_h: bool = False, round_y: bool = False):
    """fp64 MoE layer forward for chosen token rows (all rows by default).

    Returns dict(y [n, d] float64, logits, k, ids, gates)."""
    lib = _load()
    x = _c(x_bits, np.uint16)
    wr = _c(w_router_bits, np.uint16)
    wgu = _c(w_gate_up_bits, np.uint16)
    wd = _c(w_down_bits, np.uint16)
    T, d = x.shape
    N = wr.shape[0]
    I = wgu.shape[1] // 2
    rows = np.arange(T, dtype=np.int64) if rows is None else _c(rows, np.int64)
    n = len(rows)
    res = None if residual_bits is None else _c(residual_bits, np.uint16)
    y = np.empty((n, d), np.float64)
    lg = np.empty((n, N), np.float32)
    k = np.empty(n, np.int32)
    ids = np.empty((n, K), np.int32)
    gates = np.empty((n, K), np.float32)
    flags = (1 if round_h else 0) | (2 if round_y else 0)
    rc = lib.oracle_layer_rows(_ptr(x), _ptr(wr), _ptr(wgu), _ptr(wd), T, d, N, I, K, eps, mode,
                               renorm, _ptr(res), _ptr(rows), n, flags, _ptr(y), _ptr(lg), _ptr(k),
                               _ptr(ids), _ptr(gates))
    if rc != 0:
        raise ValueError("oracle_layer_rows: unsupported arguments")
    return dict(y=y, logits=lg, k=k, ids=ids, gates=gates)


MODE_RAND_TAIL = 2
MODE_RAND_HEAD = 3


def route_randomized(logits, rand, K: int = 8, eps: float = 1e-8, mode: int = MODE_RAND_TAIL,
                     renorm: int = 0):
    """Tail (mode 2) or head (mode 3) randomisation of Sec. 2.2 with the uint32
    random numbers rand [T, K]. Returns dict(k, ids, gates)."""
    lib = _load()
    lg = _c(logits, np.float32)
    rnd = _c(rand, np.uint32)
    T, N = lg.shape
    assert rnd.shape == (T, K)
    k = np.empty(T, np.int32)
    ids = np.empty((T, K), np.int32)
    gates = np.empty((T, K), np.float32)
    if lib.oracle_route_randomized(_ptr(lg), T, N, K, eps, mode, renorm, _ptr(rnd), _ptr(k),
                                   _ptr(ids), _ptr(gates)) != 0:
        raise ValueError("oracle_route_randomized: unsupported arguments")
    return dict(k=k, ids=ids, gates=gates)


def elbow_angle(logits, eps: float = 1e-8):
    """Per token of fp32 logits [T, N]: the uncapped elbow index (argmax of D
    over all ranks) and the elbow angle in degrees (Sec. 2.3, reading R11)."""
    lib = _load()
    lg = _c(logits, np.float32)
    T, N = lg.shape
    e = np.empty(T, np.int32)
    th = np.empty(T, np.float32)
    if lib.oracle_elbow_angle(_ptr(lg), T, N, eps, _ptr(e), _ptr(th)) != 0:
        raise ValueError("oracle_elbow_angle: unsupported arguments")
    return dict(elbow=e, theta=th)


def angle_deg(e: int, N: int, pn_e: float) -> float:
    """The elbow angle (degrees, fp64) at rank e of an N-point curve with p'_e = pn_e."""
    return float(_load().oracle_angle_deg(int(e), int(N), float(np.float32(pn_e))))


def load_balance(k_elb, ids, N: int):
    """Expert loads under elbow-K and top-K routing of the same tokens (App. A.3).

    L_i = mean over tokens of 1{i selected}; q = L / sum(L); delta = 1 - E[k]/K.
    Returns the distributions, delta, and the three quantities Theorem 1 and
    Corollaries 1-2 bound, with their bounds."""
    k_elb = np.asarray(k_elb)
    ids = np.asarray(ids)
    T, K = ids.shape
    L_top = np.zeros(N)
    L_elb = np.zeros(N)
    for t in range(T):
        for s in range(K):
            L_top[ids[t, s]] += 1.0
            if s < k_elb[t]:
                L_elb[ids[t, s]] += 1.0
    L_top /= T
    L_elb /= T
    q_top = L_top / L_top.sum()
    q_elb = L_elb / L_elb.sum()
    delta = 1.0 - k_elb.mean() / K
    cv2 = lambda q: N * float(np.dot(q, q)) - 1.0
    cv_top, cv_elb = np.sqrt(max(cv2(q_top), 0.0)), np.sqrt(max(cv2(q_elb), 0.0))
    return dict(
        L_top=L_top, L_elb=L_elb, q_top=q_top, q_elb=q_elb, delta=delta,
        l1=float(np.abs(q_elb - q_top).sum()),
        l1_bound=2 * delta / (1 - delta),
        max_change=abs(q_elb.max() - q_top.max()),
        cv2_change=abs(cv2(q_elb) - cv2(q_top)),
        cv2_bound=2 * N * delta / (1 - delta) ** 2,
        # the percentages of Sec. 2.4
        top1_share_change_pct=(q_top.max() - q_elb.max()) / q_top.max() * 100.0,
        cv_change_pct=(cv_top - cv_elb) / cv_top * 100.0 if cv_top > 0 else 0.0,
    )
