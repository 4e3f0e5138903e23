"""The C-ABI library builds, loads and exports every entry point that
include/elbow_moe.h declares; host-side argument validation returns the
documented status codes. No kernel is launched here (no GPU needed)."""
import ctypes
import os
import re

import pytest

import paper_2608_04401_gb300 as moe

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "elbow_moe.h")


@pytest.fixture(scope="module")
def lib():
    moe.build()
    return moe.library()


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s+\*?([a-z_][a-z0-9_]*)\s*\(",
                       src, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("elbow_route", "moe_dispatch", "moe_layer_forward", "moe_layer_workspace_size",
              "moe_status_string", "moe_read_device_error"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for n in _declared():
        assert hasattr(lib, n), n


def test_status_strings(lib):
    for s in range(6):
        assert lib.moe_status_string(s).startswith(b"MOE_")


def _rp(K=8, eps=1e-8, mode=0, renorm=0):
    return ctypes.byref(moe.RouteParams(K, eps, mode, renorm))


def test_route_validation(lib):
    fake = ctypes.c_void_p(256)
    # unsupported N, K
    assert lib.elbow_route(fake, 10, 65, _rp(), fake, fake, fake, None) == 2
    assert lib.elbow_route(fake, 10, 64, _rp(K=9), fake, fake, fake, None) == 2
    assert lib.elbow_route(fake, 10, 64, _rp(K=0), fake, fake, fake, None) == 2
    # bad params / pointers
    assert lib.elbow_route(fake, 10, 64, _rp(mode=3), fake, fake, fake, None) == 1
    assert lib.elbow_route(fake, 10, 64, _rp(eps=-1.0), fake, fake, fake, None) == 1
    assert lib.elbow_route(None, 10, 64, _rp(), fake, fake, fake, None) == 1
    assert lib.elbow_route(ctypes.c_void_p(258), 10, 64, _rp(), fake, fake, fake, None) == 1
    assert lib.elbow_route(fake, -1, 64, _rp(), fake, fake, fake, None) == 1
    # T * K pair counts must fit in int32: T < 2^28
    assert lib.elbow_route(fake, 1 << 28, 64, _rp(), fake, fake, fake, None) == 1
    assert lib.elbow_route(fake, 10, 64, None, fake, fake, fake, None) == 1
    # T = 0 is a no-op that launches nothing
    assert lib.elbow_route(None, 0, 64, _rp(), None, None, None, None) == 0


def test_dispatch_validation(lib):
    fake = ctypes.c_void_p(256)
    need = lib.moe_dispatch_workspace_size(1000, 64, 8)
    assert need > 0
    assert lib.moe_dispatch(fake, fake, 1000, 64, 8, fake, fake, fake, fake, need - 1, None) == 3
    assert lib.moe_dispatch(fake, fake, 1000, 96, 8, fake, fake, fake, fake, need, None) == 2
    assert lib.moe_dispatch(fake, fake, 1000, 64, 8, None, fake, fake, fake, need, None) == 1
    big = lib.moe_dispatch_workspace_size((1 << 28) - 1, 64, 8)
    assert big > 0 and lib.moe_dispatch_workspace_size(1 << 28, 64, 8) == 0
    assert lib.moe_dispatch(fake, fake, 1 << 28, 64, 8, fake, fake, fake, fake, big, None) == 1


def test_layer_validation(lib):
    fake = ctypes.c_void_p(256)
    ws = lib.moe_layer_workspace_size(64, 2048, 64, 1024, 8)
    # h [T*K, I] and the expert outputs [T*K, d], bf16
    assert ws > 64 * 8 * (2048 * 2 + 1024 * 2)
    args = lambda T=64, d=2048, N=64, I=1024, rp=None, wsb=ws: (
        fake, fake, fake, fake, T, d, N, I, rp or _rp(), None, fake, None, None, None, None, None,
        fake, wsb, None)
    assert lib.moe_layer_forward(*args(d=2000)) == 2
    # d a multiple of 128 is supported (the check reaches the workspace size);
    # a multiple of 64 only is not
    ws384 = lib.moe_layer_workspace_size(64, 384, 64, 1024, 8)
    assert ws384 > 0
    assert lib.moe_layer_forward(*args(d=384, wsb=ws384 - 1)) == 3
    assert lib.moe_layer_forward(*args(d=320)) == 2
    assert lib.moe_layer_forward(*args(I=1000)) == 2
    assert lib.moe_layer_forward(*args(N=32)) == 2
    assert lib.moe_layer_forward(*args(wsb=ws - 1)) == 3
    assert lib.moe_layer_forward(*args(rp=_rp(renorm=2))) == 1
    assert lib.moe_layer_workspace_size(64, 2048, 63, 1024, 8) == 0
    assert lib.moe_layer_workspace_size(1 << 28, 2048, 64, 1024, 8) == 0
    assert lib.moe_layer_workspace_size(64, 2048, 64, 1024, 9) == 0


def test_diagnostics_validation(lib):
    fake = ctypes.c_void_p(256)
    assert lib.moe_route_diagnostics(fake, 10, 64, _rp(), None, None, None, None) == 1
    assert lib.moe_route_diagnostics(fake, 10, 64, _rp(), None, None, ctypes.c_void_p(260), None) == 1
    assert lib.moe_route_diagnostics(fake, 10, 96, _rp(), None, None, fake, None) == 2
    assert ctypes.sizeof(moe.RouteDiag) == 8 * (2 + 9 + 128 + 181 + 128 + 128) + 8 * 9


def test_randomized_validation(lib):
    fake = ctypes.c_void_p(256)
    # modes other than 2 / 3, missing rand
    assert lib.elbow_route_randomized(fake, 10, 64, _rp(mode=0), fake, fake, fake, fake, None) == 1
    assert lib.elbow_route_randomized(fake, 10, 64, _rp(mode=2), None, fake, fake, fake, None) == 1
    assert lib.elbow_route_randomized(fake, 10, 64, _rp(mode=3, K=9), fake, fake, fake, fake, None) == 2
    # elbow_route itself rejects the randomisation modes
    assert lib.elbow_route(fake, 10, 64, _rp(mode=2), fake, fake, fake, None) == 1


def test_bounded_wait_check_validation(lib):
    assert lib.moe_check_bounded_wait(None, 0.1, None) == 1
    assert lib.moe_check_bounded_wait(ctypes.c_void_p(258), 0.1, None) == 1
    assert lib.moe_check_bounded_wait(ctypes.c_void_p(256), 0.0, None) == 1
    assert lib.moe_check_bounded_wait(ctypes.c_void_p(256), 11.0, None) == 1



def test_misaligned_int32_arrays_are_rejected(lib):
    """4-byte arrays (counts, offsets, positions, gates, error words) that are
    not 4-byte aligned return MOE_ERR_INVALID_ARG before anything is enqueued."""
    fake = ctypes.c_void_p(256)
    odd = ctypes.c_void_p(258)
    need = lib.moe_dispatch_workspace_size(1000, 64, 8)
    assert lib.moe_dispatch(odd, fake, 1000, 64, 8, fake, fake, fake, fake, need, None) == 1
    assert lib.moe_dispatch(fake, fake, 1000, 64, 8, fake, odd, fake, fake, need, None) == 1
    assert lib.moe_dispatch(fake, fake, 1000, 64, 8, fake, fake, odd, fake, need, None) == 1
    assert lib.moe_dispatch(fake, fake, 1000, 64, 8, odd, fake, fake, fake, need, None) == 1
    assert lib.moe_combine(fake, fake, fake, odd, None, 10, 2048, 8, fake, None) == 1
    assert lib.moe_combine(fake, fake, odd, fake, None, 10, 2048, 8, fake, None) == 1
    assert lib.moe_combine(fake, fake, fake, fake, None, 1 << 28, 2048, 8, fake, None) == 1
    assert lib.moe_expert_down(fake, fake, odd, fake, 100, 2048, 64, 1024, fake, None, None) == 1
    assert lib.moe_expert_down(fake, fake, fake, fake, 100, 2048, 64, 1024, fake, odd, None) == 1
    assert lib.moe_gather_rows(fake, odd, fake, 10, 80, 2048, 64, fake, None) == 1
    ws = lib.moe_layer_workspace_size(64, 2048, 64, 1024, 8)
    assert lib.moe_layer_forward(fake, fake, fake, fake, 64, 2048, 64, 1024, _rp(), None, fake,
                                 None, odd, None, None, None, fake, ws, None) == 1


def test_quotient_check_validation(lib):
    fake = ctypes.c_void_p(256)
    assert lib.moe_check_quotients(fake, fake, 0, fake, None) == 0
    assert lib.moe_check_quotients(fake, fake, -1, fake, None) == 1
    assert lib.moe_check_quotients(None, fake, 4, fake, None) == 1
    assert lib.moe_check_quotients(fake, ctypes.c_void_p(258), 4, fake, None) == 1


def test_debug_violations_release_build(lib):
    """The release build has no device bounds checks: the report says so."""
    v = ctypes.c_uint32(7)
    assert lib.moe_debug_violations(ctypes.byref(v)) == 2 and v.value == 0
    assert lib.moe_debug_violations(None) == 1


def test_gemv_validation(lib):
    fake = ctypes.c_void_p(256)
    # T > 4, d > 4096, N unsupported
    assert lib.moe_expert_gate_up_gemv(fake, 5, fake, fake, fake, 40, 512, 64, 256, 8, fake, None,
                                       None) == 2
    assert lib.moe_expert_gate_up_gemv(fake, 1, fake, fake, fake, 8, 8192, 64, 256, 8, fake, None,
                                       None) == 2
    assert lib.moe_expert_down_gemv(fake, fake, fake, 1, 8, 512, 96, 256, 8, fake, None, None) == 2
    assert lib.moe_expert_down_gemv(fake, fake, fake, 1, 8, 512, 64, 256, 8, ctypes.c_void_p(257),
                                    None, None) == 1
    assert lib.moe_expert_down_gemv(fake, fake, fake, 1, 8, 512, 64, 256, 8, fake,
                                    ctypes.c_void_p(258), None) == 1
    assert lib.moe_expert_gate_up_gemv(fake, 0, fake, fake, fake, 0, 512, 64, 256, 8, fake, None,
                                       None) == 0
