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

import oracle
import synth

ap = pytest.importorskip("paper_2108_02416_gb300")

# K=21, r=4: f = 5985 files, near the array's 6144-file limit
K21R4 = synth.Workload("k21_r4_strong_alie", K=21, r=4, d=2053, q=4, attack="strong",
                       distortion="alie", z=1.0, seed=8)


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
    ("k21_r4_strong_alie", 2_053, ap.MEDIAN),         # f = 5985
])
def test_static_round_matches_round_twice(name, d, mode):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    dev = torch.device("cuda:0")
    base = K21R4 if name == K21R4.name else synth.CONFIGS[name]
    w = dataclasses.replace(base, d=d)
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

    # the oracle on the same bytes: a direct check, not only through aspis_round
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers)
    orc = oracle.run_round(host, oa, w.d, mode)
    rows = np.array([host[i, orc.sel[i], : w.d] for i in range(oa.f) if orc.sel[i] >= 0])
    scale = np.abs(rows.astype(np.float64)).mean(0)

    for call in range(2):
        det = torch.zeros(ap.DETECTION_BYTES, dtype=torch.uint8, device=dev)
        out = torch.full((w.d,), float("nan"), dtype=torch.float32, device=dev)
        ap.aspis_round_static(copies, w.d, a_host, det, out, mode)
        torch.cuda.synchronize()
        got_det = ap.Detection.from_tensor(det)
        for field in ("clique_mask", "omega", "n_max_cliques", "success", "n_sel", "status"):
            assert getattr(got_det, field) == getattr(want_det, field), (call, field)
        assert (got_det.omega, got_det.n_max_cliques, got_det.clique_mask,
                bool(got_det.success), got_det.n_sel) == \
            (orc.det.omega, orc.det.n_max, orc.det.clique, orc.det.success, orc.n_sel), call
        got = out.cpu().numpy()
        if mode == ap.MEDIAN:
            assert np.array_equal(got.view(np.uint32), want.view(np.uint32)), call
            assert np.array_equal(got.view(np.uint32), orc.out.view(np.uint32)), call
        else:
            err = np.abs(got.astype(np.float64) - want.astype(np.float64))
            assert (err <= 1e-6 * np.abs(want.astype(np.float64)) + 1e-30).all(), call
            ref = np.maximum(np.abs(orc.out.astype(np.float64)), scale)
            err = np.abs(got.astype(np.float64) - orc.out.astype(np.float64))
            assert (err <= 1e-6 * ref + 1e-30).all(), call
