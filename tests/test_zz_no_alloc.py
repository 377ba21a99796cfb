"""aspis_round_static: the round for callers that cannot allocate device
memory (a runtime lending the library buffers from its own pool, a process
whose allocator is locked or budgeted).  It keeps the round's intermediates in
the library's fixed device array instead of caller buffers, so its results
must equal aspis_round's on the same copies, call after call, although each
call reuses the array the previous one left behind.

This file is collected last on purpose: the GPU test calls the library's
first use of that array on the device, and a run that stops at the first
failure has then already run every other test."""
import ctypes
import dataclasses

import numpy as np
import pytest

import synth

ap = pytest.importorskip("paper_2108_02416_gb300")


def test_static_round_rejects_too_many_files():
    """f above the array's capacity is refused before anything is enqueued
    (no GPU needed: the check comes first)."""
    a = ap.aspis_assign(31, 4, device=False)          # f = C(31,4) = 31465
    assert a.f > ap.STATIC_MAX_FILES
    P = ctypes.c_void_p
    st = ap.lib.aspis_round_static(P(256), 16, 16, a.ref, P(256), 0, P(256), None)
    assert st == ap.E_RANGE
    b = ap.aspis_assign(7, 3, device=False)
    assert ap.lib.aspis_round_static(P(256), 16, 16, b.ref, P(256), 2, P(256), None) == ap.E_INVAL


@pytest.mark.gpu
@pytest.mark.parametrize("name,d,mode", [
    ("k15_r3_d11m_strong_alie", 65_543, ap.MEDIAN),   # Case 2, ragged tail
    ("k15_r3_d1m_weak_reversed", 40_001, ap.MEDIAN),  # Case 1, one file dropped
    ("k15_r3_d1m_weak_reversed", 40_001, ap.MEAN),
    ("k15_r5_d1m_strong_alie", 9_001, ap.MEDIAN),     # f = 3003
])
def test_static_round_matches_round_twice(name, d, mode):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    dev = torch.device("cuda:0")
    w = dataclasses.replace(synth.CONFIGS[name], d=d)
    a = ap.aspis_assign(w.K, w.r)                     # with device mirror, for aspis_round
    a_host = ap.aspis_assign(w.K, w.r, device=False)  # host tables only
    copies = synth.build_copies_torch(w, a.file_workers(), dev)
    torch.cuda.synchronize()

    ref = ap.RoundBuffers(a, w.d, dev)
    ap.aspis_round(copies, w.d, a, ref.file_neq, ref.adj, ref.det, ref.sel, ref.out, mode)
    torch.cuda.synchronize()
    want_det = ref.detection()
    want = ref.out.cpu().numpy()
    assert want_det.status == ap.OK

    for call in range(2):
        det = torch.zeros(ap.DETECTION_BYTES, dtype=torch.uint8, device=dev)
        out = torch.full((w.d,), float("nan"), dtype=torch.float32, device=dev)
        ap.aspis_round_static(copies, w.d, a_host, det, out, mode)
        torch.cuda.synchronize()
        got_det = ap.Detection.from_tensor(det)
        for field in ("clique_mask", "omega", "n_max_cliques", "success", "n_sel", "status"):
            assert getattr(got_det, field) == getattr(want_det, field), (call, field)
        got = out.cpu().numpy()
        if mode == ap.MEDIAN:
            assert np.array_equal(got.view(np.uint32), want.view(np.uint32)), call
        else:
            err = np.abs(got.astype(np.float64) - want.astype(np.float64))
            assert (err <= 1e-6 * np.abs(want.astype(np.float64)) + 1e-30).all(), call
