"""The C ABI on the host: the library loads, exports every declared symbol, and rejects bad
arguments before touching CUDA (so these run without a GPU)."""
import ctypes
import math
import os

import pytest

from paper_2608_03447_gb300 import asd, build

NULL = None


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(asd.LIBRARY) or any(
            os.path.getmtime(s) > os.path.getmtime(asd.LIBRARY) for s in build.sources()):
        build.build()
    return asd.load()


def test_every_declared_symbol_is_exported(lib):
    declared = asd.declared_functions()
    assert {"asd_verify", "asd_verify_strict", "asd_workspace_size", "asd_workspace_init",
            "asd_status_string"} <= set(declared)
    for name in declared:
        assert hasattr(lib, name), f"{name} is declared in include/asd.h but not exported"


def test_status_strings(lib):
    for code in range(0, 9):
        assert asd.status_string(code)
    assert asd.status_string(12345) == "unknown status code"


def test_workspace_size(lib):
    n = asd.workspace_size(32, 8, 151936, asd.BF16)
    assert n >= 32 * 9 * 12 + 32 * 12 and n % 256 == 0
    n0 = asd.workspace_size(0, 8, 10, asd.F32)
    assert n0 > 0
    sz = ctypes.c_size_t(0)
    assert lib.asd_workspace_size(1, 32, 10, asd.F32, ctypes.byref(sz)) == 2   # K > 31
    assert lib.asd_workspace_size(1, -1, 10, asd.F32, ctypes.byref(sz)) == 2
    assert lib.asd_workspace_size(1, 4, 0, asd.F32, ctypes.byref(sz)) == 2     # V < 1
    assert lib.asd_workspace_size(1, 4, 10, 7, ctypes.byref(sz)) == 3          # dtype
    assert lib.asd_workspace_size(1, 4, 10, asd.F32, None) == 1


def test_resident_inputs_flag_is_a_flag_not_a_dtype(lib):
    """ASD_RESIDENT_INPUTS rides in the dtype argument: it changes no size or validation, and any other
    high bit is still an unknown dtype."""
    sz, sz_flag = ctypes.c_size_t(0), ctypes.c_size_t(0)
    for dt in (asd.F32, asd.BF16):
        assert lib.asd_workspace_size(8, 4, 1000, dt, ctypes.byref(sz)) == 0
        assert lib.asd_workspace_size(8, 4, 1000, dt | asd.RESIDENT_INPUTS, ctypes.byref(sz_flag)) == 0
        assert sz.value == sz_flag.value
        n, n_flag = ctypes.c_int(0), ctypes.c_int(0)
        for (B, K, V) in ((32, 8, 151936), (4, 8, 1024)):
            assert lib.asd_verify_launches(B, K, V, dt, ctypes.byref(n)) == 0
            assert lib.asd_verify_launches(B, K, V, dt | asd.RESIDENT_INPUTS, ctypes.byref(n_flag)) == 0
            assert n.value == n_flag.value
    assert lib.asd_workspace_size(8, 4, 1000, asd.F32 | 0x200, ctypes.byref(sz)) == 3
    assert _verify(lib, dtype=asd.F32 | 0x200) == 3
    assert _verify(lib, dtype=asd.F32 | asd.RESIDENT_INPUTS, B=0) == 0
    assert _verify(lib, dtype=asd.BF16 | asd.RESIDENT_INPUTS, K=32) == 2


def _verify(lib, **kw):
    a = dict(logits=0x1000, dtype=asd.F32, B=2, K=3, V=10, draft=0x2000, ledger=0x3000, gate=1.0, cap=2,
             acc=0x4000, com=0x5000, rec=0x6000, ya=NULL, rr=NULL, st=NULL, ws=0x7000, wsb=1 << 20)
    a.update(kw)
    return lib.asd_verify(a["logits"], a["dtype"], a["B"], a["K"], a["V"], a["draft"], a["ledger"], a["gate"],
                          a["cap"], a["acc"], a["com"], a["rec"], a["ya"], a["rr"], a["st"], a["ws"], a["wsb"], None)


def test_verify_rejects_bad_arguments_without_launching(lib):
    # fake (never dereferenced) pointers: every case returns before any CUDA call
    assert _verify(lib, dtype=5) == 3
    assert _verify(lib, K=32) == 2
    assert _verify(lib, V=0) == 2
    assert _verify(lib, B=-1) == 2
    assert _verify(lib, logits=NULL) == 1
    assert _verify(lib, draft=NULL) == 1
    assert _verify(lib, ledger=NULL) == 1
    assert _verify(lib, acc=NULL) == 1
    assert _verify(lib, ws=NULL) == 1
    assert _verify(lib, gate=-0.5) == 4
    assert _verify(lib, gate=math.nan) == 4
    assert _verify(lib, cap=-1) == 4
    assert _verify(lib, wsb=16) == 5
    assert _verify(lib, ws=0x7004) == 6                      # workspace not 16-byte aligned
    assert _verify(lib, logits=0x1001) == 6                  # fp32 logits not 4-byte aligned
    assert _verify(lib, dtype=asd.BF16, logits=0x1001) == 6  # bf16 logits not 2-byte aligned
    assert _verify(lib, B=0) == 0                            # empty batch: nothing to do


def test_strict_rejects_bad_arguments(lib):
    def strict(**kw):
        a = dict(logits=0x1000, dtype=asd.F32, B=2, K=3, V=10, draft=0x2000, acc=0x4000, com=0x5000,
                 rec=0x6000, ws=0x7000, wsb=1 << 20)
        a.update(kw)
        return lib.asd_verify_strict(a["logits"], a["dtype"], a["B"], a["K"], a["V"], a["draft"], a["acc"],
                                     a["com"], a["rec"], None, None, None, a["ws"], a["wsb"], None)
    assert strict(draft=NULL) == 1
    assert strict(K=0, draft=NULL, B=0) == 0
    assert strict(K=40) == 2
    assert strict(wsb=0) == 5


def test_lmhead_entry_points_reject_bad_arguments(lib):
    """The fused LM-head entry points validate shapes, pointers and alignment before any CUDA call."""
    sz = ctypes.c_size_t(0)
    assert lib.asd_lmhead_workspace_size(4, 8, 1000, 64, ctypes.byref(sz)) == 0 and sz.value > 0
    assert lib.asd_lmhead_workspace_size(4, 8, 1000, 60, ctypes.byref(sz)) == 2   # H not a multiple of 8

    def partials(**kw):
        a = dict(h=0x1000, w=0x2000, H=64, B=2, K=3, Vs=100, off=0, V=400, draft=0x3000, out=0x4000,
                 ws=0x7000, wsb=1 << 20)
        a.update(kw)
        return lib.asd_lmhead_partials(a["h"], a["w"], a["H"], a["B"], a["K"], a["Vs"], a["off"], a["V"],
                                       a["draft"], a["out"], a["ws"], a["wsb"], None)
    assert partials(off=301) == 2          # shard past the vocabulary
    assert partials(off=-1) == 2
    assert partials(Vs=0) == 2
    assert partials(K=32) == 2
    assert partials(H=12) == 2             # rows not 16-byte pitched
    assert partials(h=NULL) == 1
    assert partials(out=NULL) == 1
    assert partials(draft=NULL) == 1
    assert partials(ws=NULL) == 1
    assert partials(wsb=16) == 5
    assert partials(w=0x2008) == 6         # weight not 16-byte aligned
    assert partials(B=0) == 0              # empty batch: nothing to do


def test_workspace_init_null(lib):
    assert lib.asd_workspace_init(None, 256, None) == 1


def test_binding_fails_loudly_without_library(tmp_path):
    with pytest.raises(RuntimeError):
        asd._declare  # the module is importable without the library
        import importlib
        mod = importlib.reload(asd)
        try:
            mod._lib = None
            mod.load(str(tmp_path / "missing.so"))
        finally:
            importlib.reload(asd)


def test_launch_options_round_trip(lib):
    """asd_set_launch_options / asd_get_launch_options: host-only state, read by every later call."""
    try:
        assert asd.get_launch_options() == {"path": "auto", "fused_select": False, "pdl": True}
        n = ctypes.c_int(-1)
        assert lib.asd_verify_launches(32, 8, 151936, asd.BF16, ctypes.byref(n)) == 0 and n.value == 2
        asd.set_launch_options(path="stream", fused_select=True, pdl=False)
        assert asd.get_launch_options() == {"path": "stream", "fused_select": True, "pdl": False}
        assert lib.asd_verify_launches(32, 8, 151936, asd.BF16, ctypes.byref(n)) == 0 and n.value == 1
        asd.set_launch_options(path="tma", fused_select=True)
        assert lib.asd_verify_launches(4, 8, 1024, asd.F32, ctypes.byref(n)) == 0 and n.value == 1
        asd.set_launch_options(path="tma")
        assert lib.asd_verify_launches(4, 8, 1024, asd.F32, ctypes.byref(n)) == 0 and n.value == 2

        class Bad(ctypes.Structure):
            _fields_ = [("path", ctypes.c_int), ("a", ctypes.c_int), ("b", ctypes.c_int)]
        assert lib.asd_set_launch_options(ctypes.byref(Bad(7, 0, 0))) == 4  # ASD_ERR_CONTROL
        assert asd.get_launch_options()["path"] == "tma"  # a rejected call changes nothing
        assert lib.asd_get_launch_options(None) == 1      # ASD_ERR_NULL
    finally:
        asd.reset_launch_options()
    assert asd.get_launch_options()["path"] == "auto"
