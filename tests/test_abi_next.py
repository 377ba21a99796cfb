"""Argument checks of the entry points added for the rows after the step
(tolerant round, round from host memory), exercised without a GPU: each case
is rejected before anything reaches the device.  The assignment carries a
fake device-mirror address that is never dereferenced (argument errors
return first) and is cleared before the assignment is freed."""
import ctypes
import contextlib

import pytest

ap = pytest.importorskip("paper_2108_02416_gb300")
P = ctypes.c_void_p
FAKE = 0x100000                     # 16-byte aligned, never dereferenced


@contextlib.contextmanager
def fake_mirror(K, r):
    a = ap.aspis_assign(K, r, device=False)
    a._a.dev_file_workers = FAKE
    try:
        yield a
    finally:
        a._a.dev_file_workers = None


def tolerant(a, d=8, ld=8, tau=0.0, ldm=8, mode=0, **null):
    args = dict(copies=P(FAKE), file_neq=P(FAKE), adj=P(FAKE), det=P(FAKE), slot_mask=P(FAKE),
                sel=P(FAKE), means=P(FAKE), out=P(FAKE))
    for k in null:
        args[k] = None
    return ap.lib.aspis_round_tolerant(args["copies"], d, ld, a.ref, tau, args["file_neq"],
                                       args["adj"], args["det"], args["slot_mask"], args["sel"],
                                       args["means"], ldm, mode, args["out"], None)


def test_tolerant_round_argument_errors():
    with fake_mirror(7, 3) as a:
        assert tolerant(a, tau=-1.0) == ap.E_INVAL
        assert tolerant(a, tau=float("nan")) == ap.E_INVAL
        assert tolerant(a, mode=2) == ap.E_INVAL
        assert tolerant(a, ldm=7) == ap.E_INVAL
        assert tolerant(a, d=0) == ap.E_INVAL
        assert tolerant(a, ld=7) == ap.E_INVAL
        for k in ("copies", "file_neq", "adj", "det", "slot_mask", "sel", "means", "out"):
            assert tolerant(a, **{k: True}) == ap.E_INVAL, k
    with fake_mirror(20, 5) as a:                  # f = 15504 > 6144 files
        assert tolerant(a) == ap.E_RANGE
    a = ap.aspis_assign(7, 3, device=False)        # no device mirror at all
    assert tolerant(a) == ap.E_INVAL


def test_round_host_argument_errors():
    with fake_mirror(7, 3) as a:
        def call(mode=0, host=FAKE, hout=FAKE, hdet=FAKE, fneq=FAKE):
            return ap.lib.aspis_round_host(P(host), P(FAKE), 8, 8, a.ref, P(fneq), P(FAKE), P(FAKE),
                                           P(FAKE), mode, P(FAKE), P(hout), P(hdet), None)
        assert call(mode=3) == ap.E_INVAL
        assert call(host=0) == ap.E_INVAL
        assert call(hout=0) == ap.E_INVAL
        assert call(hdet=0) == ap.E_INVAL
        assert call(fneq=0) == ap.E_INVAL
    with fake_mirror(20, 5) as a:
        assert ap.lib.aspis_round_host(P(FAKE), P(FAKE), 8, 8, a.ref, P(FAKE), P(FAKE), P(FAKE),
                                       P(FAKE), 0, P(FAKE), P(FAKE), P(FAKE), None) == ap.E_RANGE
