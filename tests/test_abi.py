"""The C-ABI library: it builds for sm_103a, loads, exports every declared entry point,
and rejects bad arguments on the host (no GPU needed: no compute call is made)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADERS = [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include"))
           if f.endswith(".h")]


def declared_functions():
    names = set()
    for h in HEADERS:
        text = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names |= set(re.findall(r"^[A-Za-z_][\w\s\*]*?\b(flex_\w+)\s*\(", text, flags=re.M))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    from paper_2606_27748_gb300 import build, flexattn
    build.build()
    return flexattn.load()


def test_header_declares_the_entry_points():
    names = declared_functions()
    for n in ("flex_featmap", "flex_linattn_fwd", "flex_linattn_bwd", "flex_check_status",
              "flex_workspace_bytes", "flex_strerror"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_binding_names_match_header():
    from paper_2606_27748_gb300 import flexattn
    assert set(flexattn.EXPORTS) <= set(declared_functions())


def test_host_validation_without_gpu(lib):
    from paper_2606_27748_gb300.flexattn import FlexShape, FLEX_EINVAL, FLEX_EWORKSPACE
    ok = FlexShape(2, 3, 100, 64, 64, 1)
    assert lib.flex_workspace_bytes(ctypes.byref(ok), 1, 0) >= 256
    assert lib.flex_workspace_bytes(ctypes.byref(ok), 1, 1) > lib.flex_workspace_bytes(
        ctypes.byref(ok), 1, 0)
    bad = FlexShape(2, 3, 0, 64, 64, 1)
    assert lib.flex_workspace_bytes(ctypes.byref(bad), 1, 0) == 0
    p = ctypes.c_void_p(4096)  # never dereferenced: validation fails first
    # null shape / N < 1 / null input
    # (shape, q, k, v, W1, W2, tau, causal, out, den, ws, ws_bytes, stream)
    assert lib.flex_linattn_fwd(None, p, p, p, p, None, None, 1, p, None, p, 1 << 20,
                                None) == FLEX_EINVAL
    assert lib.flex_linattn_fwd(ctypes.byref(bad), p, p, p, p, None, None, 1, p, None, p,
                                1 << 20, None) == FLEX_EINVAL
    assert lib.flex_linattn_fwd(ctypes.byref(ok), None, p, p, p, None, None, 1, p, None, p,
                                1 << 20, None) == FLEX_EINVAL
    # misaligned pointer (an input, or tau off 4 bytes)
    mis = ctypes.c_void_p(4096 + 2)
    assert lib.flex_linattn_fwd(ctypes.byref(ok), mis, p, p, p, None, None, 1, p, None, p,
                                1 << 20, None) == FLEX_EINVAL
    assert lib.flex_linattn_fwd(ctypes.byref(ok), p, p, p, p, None, mis, 1, p, None, p,
                                1 << 20, None) == FLEX_EINVAL
    # workspace too small
    assert lib.flex_linattn_fwd(ctypes.byref(ok), p, p, p, p, None, None, 1, p, None, p, 16,
                                None) == FLEX_EWORKSPACE
    # (shape, q, k, v, W1, W2, tau, causal, out, den, dout, dq, dk, dv, dW1, dW2, dtau, ws,
    #  ws_bytes, stream): W2 given without dW2 (and the reverse); tau without dtau (and the
    # reverse)
    args = [p] * 3 + [p, p, None, 1, p, p, p, p, p, p, p]
    assert lib.flex_linattn_bwd(ctypes.byref(ok), *args, None, None, p, 1 << 24,
                                None) == FLEX_EINVAL
    args = [p] * 3 + [p, None, None, 1, p, p, p, p, p, p, p]
    assert lib.flex_linattn_bwd(ctypes.byref(ok), *args, p, None, p, 1 << 24,
                                None) == FLEX_EINVAL
    args = [p] * 3 + [p, None, p, 1, p, p, p, p, p, p, p]
    assert lib.flex_linattn_bwd(ctypes.byref(ok), *args, None, None, p, 1 << 24,
                                None) == FLEX_EINVAL
    args = [p] * 3 + [p, None, None, 1, p, p, p, p, p, p, p]
    assert lib.flex_linattn_bwd(ctypes.byref(ok), *args, None, p, p, 1 << 24,
                                None) == FLEX_EINVAL
    assert lib.flex_strerror(FLEX_EINVAL)


def test_decode_host_validation_without_gpu(lib):
    from paper_2606_27748_gb300.flexattn import FlexShape, FLEX_EINVAL, FLEX_EWORKSPACE
    p = ctypes.c_void_p(4096)  # never dereferenced: validation fails first
    one = FlexShape(2, 3, 1, 64, 64, 1)
    two = FlexShape(2, 3, 2, 64, 64, 1)  # more than one token per sequence
    need = lib.flex_decode_workspace_bytes(ctypes.byref(one))
    # header + phi(q), phi(k): B H x 2 x 2M fp32
    assert need == 256 + 2 * 3 * 2 * 128 * 4
    assert lib.flex_decode_workspace_bytes(ctypes.byref(two)) == 0
    # (shape, q, k, v, W1, W2, tau, S, z, out, den, ws, ws_bytes, stream)
    assert lib.flex_linattn_decode(ctypes.byref(two), p, p, p, p, None, None, p, p, p, None,
                                   p, need, None) == FLEX_EINVAL
    assert lib.flex_linattn_decode(ctypes.byref(one), p, p, p, p, None, None, None, p, p, None,
                                   p, need, None) == FLEX_EINVAL
    assert lib.flex_linattn_decode(ctypes.byref(one), p, p, p, p, None, None, p, p,
                                   ctypes.c_void_p(4097), None, p, need, None) == FLEX_EINVAL
    assert lib.flex_linattn_decode(ctypes.byref(one), p, p, p, p, None, None, p, p, p, None,
                                   p, need - 1, None) == FLEX_EWORKSPACE
    assert lib.flex_linattn_decode(ctypes.byref(one), p, p, p, p, None, None, p, p, p, None,
                                   None, need, None) == FLEX_EINVAL
    assert lib.flex_linattn_decode(ctypes.byref(one), p, p, p, p, None,
                                   ctypes.c_void_p(4097 + 2), p, p, p, None, p, need,
                                   None) == FLEX_EINVAL


def test_awd_host_validation_without_gpu(lib):
    from paper_2606_27748_gb300.flexattn import (FlexShape, FLEX_EINVAL, FLEX_EUNSUPPORTED,
                                                 FLEX_EWORKSPACE)
    p = ctypes.c_void_p(4096)  # never dereferenced: validation fails first
    ok = FlexShape(2, 3, 300, 64, 64, 1)
    f32 = FlexShape(2, 3, 300, 64, 64, 0)
    need = lib.flex_awd_workspace_bytes(ctypes.byref(ok))
    assert need > 256 and lib.flex_awd_workspace_bytes(ctypes.byref(f32)) == 0
    # (shape, q, k, W1, W2, tau, causal, loss, ws, ws_bytes, stream)
    assert lib.flex_awd_loss(ctypes.byref(ok), None, p, p, None, None, 0, p, p, need,
                             None) == FLEX_EINVAL
    assert lib.flex_awd_loss(ctypes.byref(f32), p, p, p, None, None, 0, p, p, need,
                             None) == FLEX_EUNSUPPORTED
    assert lib.flex_awd_loss(ctypes.byref(ok), p, p, p, None, None, 0, p, p, need - 1,
                             None) == FLEX_EWORKSPACE
    assert lib.flex_awd_loss(ctypes.byref(ok), p, p, p, None, ctypes.c_void_p(4098), 0, p, p,
                             need, None) == FLEX_EINVAL


def test_awd_bwd_host_validation_without_gpu(lib):
    from paper_2606_27748_gb300.flexattn import (FlexShape, FLEX_EINVAL, FLEX_EUNSUPPORTED,
                                                 FLEX_EWORKSPACE)
    p = ctypes.c_void_p(4096)  # never dereferenced: validation fails first
    ok = FlexShape(2, 3, 300, 64, 64, 1)
    f32 = FlexShape(2, 3, 300, 64, 64, 0)
    need = lib.flex_awd_bwd_workspace_bytes(ctypes.byref(ok))
    assert need > lib.flex_awd_workspace_bytes(ctypes.byref(ok))
    assert lib.flex_awd_bwd_workspace_bytes(ctypes.byref(f32)) == 0
    f = lib.flex_awd_loss_bwd
    # (shape, q, k, W1, W2, tau, causal, dloss, loss, dW1, dW2, dtau, ws, ws_bytes, stream)
    assert f(ctypes.byref(ok), p, p, p, None, None, 0, None, p, p, None, None, p, need,
             None) == FLEX_EINVAL                                   # no dloss
    assert f(ctypes.byref(ok), p, p, p, p, None, 0, p, p, p, None, None, p, need,
             None) == FLEX_EINVAL                                   # W2 without dW2
    assert f(ctypes.byref(ok), p, p, p, None, None, 0, p, p, p, p, None, p, need,
             None) == FLEX_EINVAL                                   # dW2 without W2
    assert f(ctypes.byref(ok), p, p, p, None, p, 0, p, p, p, None, None, p, need,
             None) == FLEX_EINVAL                                   # tau without dtau
    assert f(ctypes.byref(f32), p, p, p, None, None, 0, p, p, p, None, None, p, need,
             None) == FLEX_EUNSUPPORTED
    assert f(ctypes.byref(ok), p, p, p, None, None, 0, p, p, p, None, None, p, need - 1,
             None) == FLEX_EWORKSPACE
    assert f(ctypes.byref(ok), p, p, p, None, None, 0, p, p, ctypes.c_void_p(4100), None, None,
             p, need, None) == FLEX_EINVAL                          # misaligned dW1


def test_debug_stall_validation_without_gpu(lib):
    from paper_2606_27748_gb300.flexattn import FLEX_EINVAL, FLEX_EWORKSPACE
    p = ctypes.c_void_p(4096)  # 256-byte aligned, never dereferenced: validation fails first
    assert lib.flex_debug_stall(None, 256, 1000, None) == FLEX_EINVAL
    assert lib.flex_debug_stall(ctypes.c_void_p(4100), 256, 1000, None) == FLEX_EINVAL
    assert lib.flex_debug_stall(p, 256, -1, None) == FLEX_EINVAL
    assert lib.flex_debug_stall(p, 255, 1000, None) == FLEX_EWORKSPACE
