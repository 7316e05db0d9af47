"""The C-ABI library loads, exports every entry point qtea.h declares, and fails loudly
without a GPU (CPU-only checks: no kernel is launched here)."""
import ctypes
import os
import re

import pytest

import paper_2609_00224_gb300 as qt

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    text = open(os.path.join(ROOT, "include", "qtea.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(qtea_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("qtea_pack_layout", "qtea_gemv", "qtea_free", "qtea_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol():
    lib = ctypes.CDLL(qt._build.build())
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings():
    for code in range(9):
        assert qt.status_string(code) and qt.status_string(code) != "unknown status"
    assert qt.status_string(99) == "unknown status"


def test_host_side_argument_checks_need_no_gpu():
    lib = qt.load()
    out = ctypes.c_void_p()
    assert lib.qtea_pack_layout(None, 4, 8, 8, 0, 0, None, None) == qt.QTEA_ERR_INVALID_ARG
    assert lib.qtea_pack_layout(None, -1, 8, 8, 0, 0, None, ctypes.byref(out)) == qt.QTEA_ERR_INVALID_ARG
    assert lib.qtea_pack_layout(None, 6, 8, 8, 4, 0, None, ctypes.byref(out)) == qt.QTEA_ERR_INVALID_ARG  # N % 4
    assert lib.qtea_pack_layout(None, 4, 8, 8, 9, 0, None, ctypes.byref(out)) == qt.QTEA_ERR_INVALID_ARG  # s > K
    assert lib.qtea_pack_layout(ctypes.c_void_p(16), 4, 8, 8, 0, 7, None,
                                ctypes.byref(out)) == qt.QTEA_ERR_INVALID_ARG  # no such format
    assert lib.qtea_pack_layout(ctypes.c_void_p(16), 4, 256, 64, 0, 0, None,
                                ctypes.byref(out)) == qt.QTEA_ERR_UNSUPPORTED  # groups other than K or 128
    assert lib.qtea_set_layout_options(None, qt.QTEA_OPT_BIAS) == qt.QTEA_ERR_INVALID_ARG
    assert lib.qtea_gemv(None, None, None, None, None, None, None, None, 1, None) == qt.QTEA_ERR_INVALID_ARG
    q = lib.qtea_quantize
    P = ctypes.c_void_p(16)
    assert q(None, P, 4, 8, 8, 0, 0, 2, 2, P, P, P, None, None, None, None) == qt.QTEA_ERR_INVALID_ARG  # no W
    assert q(P, P, 6, 8, 8, 4, 0, 2, 2, P, P, P, P, P, P, None) == qt.QTEA_ERR_INVALID_ARG  # N % 4 with s > 0
    assert q(P, P, 4, 8, 8, 9, 0, 2, 2, P, P, P, P, P, P, None) == qt.QTEA_ERR_INVALID_ARG  # s > K
    assert q(P, P, 4, 8, 8, 2, 0, 2, 2, P, P, P, None, P, P, None) == qt.QTEA_ERR_INVALID_ARG  # no salient list
    assert q(P, P, 4, 256, 64, 0, 0, 2, 2, P, P, P, None, None, None, None) == qt.QTEA_ERR_UNSUPPORTED  # group
    assert q(P, P, 4, 8, 8, 0, 4, 2, 2, P, P, P, None, None, None, None) == qt.QTEA_ERR_INVALID_ARG  # option
    assert q(P, P, 4, 8, 8, 0, 0, -1, 2, P, P, P, None, None, None, None) == qt.QTEA_ERR_INVALID_ARG  # iters
    out4 = (ctypes.c_int * 4)(9, 9, 9, 9)
    nul = (ctypes.c_void_p * 8)()  # one problem, every pointer NULL: no layout
    assert lib.qtea_gemv_plan(None, -1, 1, out4) == qt.QTEA_ERR_INVALID_ARG
    assert lib.qtea_gemv_plan(nul, 1, 1, None) == qt.QTEA_ERR_INVALID_ARG
    assert lib.qtea_gemv_plan(nul, 1, 0, out4) == qt.QTEA_ERR_INVALID_ARG  # M < 1
    assert lib.qtea_gemv_plan(nul, 1, 1, out4) == qt.QTEA_ERR_INVALID_ARG  # no layout
    assert list(out4) == [9, 9, 9, 9]  # unchanged on error
    assert lib.qtea_gemv_plan(None, 0, 1, None) == qt.QTEA_OK
    lib.qtea_free(None)


@pytest.mark.skipif(__import__("torch").cuda.is_available(), reason="checks the no-GPU failure path")
def test_compute_entry_points_fail_without_gpu():
    lib = qt.load()
    out = ctypes.c_void_p()
    rc = lib.qtea_pack_layout(ctypes.c_void_p(16), 4, 8, 8, 0, 0, None, ctypes.byref(out))
    assert rc == qt.QTEA_ERR_CUDA and not out.value
    # the allocation-free entry's state query needs the device too, and reports it
    assert lib.qtea_gemv_m1_static_status(1, None) == qt.QTEA_ERR_CUDA
