"""C-ABI checks that need no GPU: the library loads, exports every entry point
declared in include/aspis.h, and its host-only calls behave (Algorithm 2
assignment bit-identical to the oracle's; argument errors)."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from conftest import ROOT

ap = pytest.importorskip("paper_2108_02416_gb300")


def declared_functions():
    src = open(os.path.join(ROOT, "include", "aspis.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(aspis_[a-z_]+)\s*\(", src)))


def test_header_symbols_exported():
    names = declared_functions()
    assert "aspis_check" in names and "aspis_aggregate" in names and len(names) >= 11
    lib = ctypes.CDLL(ap.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), f"{n} declared in aspis.h but not exported"


def test_struct_sizes_match_header():
    assert ctypes.sizeof(ap.Detection) == 36
    assert ctypes.sizeof(ap._Assignment) == 4 + 4 + 8 * 3 + 8 * 4


def test_status_strings():
    assert ap.status_str(0) == "ok"
    assert ap.status_str(5).startswith("clique")
    assert ap.lib.aspis_abi_version() == 2


@pytest.mark.parametrize("K,r", [(2, 2), (7, 3), (9, 4), (15, 3), (15, 5), (21, 3), (24, 3),
                                 (31, 2), (31, 3), (12, 8), (20, 7)])
def test_assign_bit_exact_vs_oracle(K, r):
    a = ap.aspis_assign(K, r, device=False)
    o = oracle.assign(K, r)
    assert (a.f, a.l, a.pair_share) == (o.f, o.l, oracle.binom(K - 2, r - 2))
    assert np.array_equal(a.file_workers(), o.file_workers)
    assert np.array_equal(a.worker_files(), o.worker_files)
    assert np.array_equal(a.slot_of(), o.slot_of)


@pytest.mark.parametrize("K,r,code", [(7, 1, ap.E_INVAL), (3, 4, ap.E_INVAL), (32, 3, ap.E_RANGE),
                                      (31, 9, ap.E_RANGE), (1, 1, ap.E_INVAL)])
def test_assign_rejects(K, r, code):
    with pytest.raises(ap.AspisError) as ei:
        ap.aspis_assign(K, r, device=False)
    assert ei.value.status == code


def test_device_calls_reject_without_mirror():
    """Arguments are checked before anything touches the GPU."""
    a = ap.aspis_assign(7, 3, device=False)
    P = ctypes.c_void_p
    assert ap.lib.aspis_check(P(16), 8, 8, a.ref, P(16), P(16), None) == ap.E_INVAL
    assert ap.lib.aspis_select(P(16), P(16), a.ref, P(16), None) == ap.E_INVAL
    assert ap.lib.aspis_aggregate(P(16), 8, 8, a.ref, P(16), P(16), 0, P(16), None) == ap.E_INVAL
    assert ap.lib.aspis_detect(None, 7, P(16), None) == ap.E_INVAL
    assert ap.lib.aspis_detect(P(16), 32, P(16), None) == ap.E_RANGE
    assert ap.lib.aspis_detect(P(16), 1, P(16), None) == ap.E_INVAL


def test_every_declared_call_through_ctypes():
    """Every entry point of include/aspis.h called through ctypes without a
    GPU: the host-only calls for real, the device calls on arguments that
    are refused before anything is enqueued."""
    P, i64 = ctypes.c_void_p, ctypes.c_int64
    lib = ap.lib
    a = ap.aspis_assign(7, 3, device=False)
    null = P(None)
    f32 = ctypes.c_float
    calls = {
        "aspis_status_str": lambda: lib.aspis_status_str(ap.E_RANGE).decode().startswith("size"),
        "aspis_abi_version": lambda: lib.aspis_abi_version() == 2,
        "aspis_workspace_bytes": lambda: (lib.aspis_workspace_bytes(a.ref) == 0 and
                                          lib.aspis_workspace_bytes(None) == 0),
        "aspis_assign": lambda: _assign_and_free(lib),
        "aspis_assignment_free": lambda: _assign_and_free(lib),
        "aspis_assignment_to_device": lambda: lib.aspis_assignment_to_device(None) == ap.E_INVAL,
        "aspis_check": lambda: lib.aspis_check(null, 8, 8, a.ref, null, null, None) == ap.E_INVAL,
        "aspis_graph": lambda: lib.aspis_graph(null, a.ref, null, None) == ap.E_INVAL,
        "aspis_detect": lambda: lib.aspis_detect(null, 7, null, None) == ap.E_INVAL,
        "aspis_select": lambda: lib.aspis_select(null, null, a.ref, null, None) == ap.E_INVAL,
        "aspis_aggregate": lambda: lib.aspis_aggregate(null, 8, 8, a.ref, null, null, 0, null,
                                                       None) == ap.E_INVAL,
        "aspis_round": lambda: lib.aspis_round(null, 8, 8, a.ref, null, null, null, null, 0, null,
                                               None) == ap.E_INVAL,
        "aspis_round_host": lambda: lib.aspis_round_host(null, null, 8, 8, a.ref, null, null, null,
                                                         null, 0, null, null, null,
                                                         None) == ap.E_INVAL,
        "aspis_round_static": lambda: lib.aspis_round_static(null, 8, 8, a.ref, null, 0, null,
                                                             None) == ap.E_INVAL,
        "aspis_detect_wide": lambda: lib.aspis_detect_wide(null, 5, null, None) == ap.E_INVAL,
        "aspis_round_tolerant": lambda: lib.aspis_round_tolerant(
            null, 8, 8, a.ref, f32(0.0), null, null, null, null, null, null, i64(8), 0, null,
            None) == ap.E_INVAL,
        "aspis_sgd": lambda: lib.aspis_sgd(null, null, null, 8, f32(0.1), f32(0.0),
                                           None) == ap.E_INVAL,
    }
    assert set(calls) == set(declared_functions()), "a declared call has no check here"
    for name, call in calls.items():
        assert call(), name


def _assign_and_free(lib):
    out = ap._Assignment()
    if lib.aspis_assign(9, 4, ctypes.byref(out)) != ap.OK or out.f != 126:
        return False
    lib.aspis_assignment_free(ctypes.byref(out))
    return out.f == 0 and not out.file_workers


def test_no_oracle_on_product_path():
    """The product package never imports the oracle."""
    pkg = os.path.join(ROOT, "paper_2108_02416_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cpp", ".cuh", ".h")):
                text = open(os.path.join(dirpath, fn)).read()
                assert "oracle" not in text.lower(), f"{fn} mentions the oracle"
