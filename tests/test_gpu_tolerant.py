"""The round for copies that are not bit-identical (aspis_round_tolerant)
against the oracle: mismatch words, graph, clique and slot masks bit for bit;
the kept files' averages, and the median and mean over them, within
1e-6 * max(|oracle|, mean |copy|) + 1e-30 of the oracle's arithmetic means
(the kernel averages in fp32).
Cases: tau = 0 on bit-identical copies (equal to the exact round), honest
copies with per-copy noise below tau under the weak, optimal and
all-adversary attacks (Case 1 averages, Case 2 clusters, r = 2 to 6), the
Fall-of-Empires distortion, NaNs, the 4-byte paths, and the full ResNet-18
length."""
import dataclasses

import numpy as np
import pytest

import oracle
import synth
from _gpu_round import as_u32, assert_mean_close

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)
ap = pytest.importorskip("paper_2108_02416_gb300")
DEV = torch.device("cuda:0")


def run(host, w, tau, mode=0, offset=0, ldm_pad=0):
    a = ap.aspis_assign(w.K, w.r)
    base = torch.zeros(host.size + offset, dtype=torch.float32, device=DEV)
    copies = base[offset:].view(host.shape)
    copies.copy_(torch.from_numpy(host))
    buf = ap.TolerantBuffers(a, w.d, DEV)
    if ldm_pad:
        buf.means = torch.zeros((a.f, w.d + ldm_pad), dtype=torch.float32, device=DEV)
    ap.aspis_round_tolerant(copies, w.d, a, tau, buf.file_neq, buf.adj, buf.det, buf.slot_mask,
                            buf.sel, buf.means, buf.out, mode)
    torch.cuda.synchronize()
    return buf


def check(buf, want, host, mode=0, exact_means=False):
    det = buf.detection()
    assert det.status == ap.OK, ap.status_str(det.status)
    assert np.array_equal(as_u32(buf.file_neq), want.file_neq), "file_neq"
    assert np.array_equal(as_u32(buf.adj), want.adj), "adjacency"
    assert (det.omega, det.n_max_cliques, det.clique_mask, bool(det.success)) == \
        (want.det.omega, want.det.n_max, want.det.clique, want.det.success), "clique"
    mask = buf.slot_mask.cpu().numpy()
    assert np.array_equal(mask, want.slot_mask), "slot masks"
    assert np.array_equal(buf.sel.cpu().numpy(), np.where(want.slot_mask != 0, 0, -1)), "sel"
    assert det.n_sel == want.n_kept
    d = want.means.shape[1]
    kept = mask != 0
    means = buf.means[:, :d].cpu().numpy()
    # per kept file and coordinate: max(|average|, mean |chosen copy|)
    scale = np.fmax(np.abs(want.means[kept].astype(np.float64)), chosen_abs_mean(host, want)[kept])
    scale = np.where(np.isnan(scale), 0.0, scale)       # NaN copies: compared as NaN below
    err = np.abs(means[kept].astype(np.float64) - want.means[kept].astype(np.float64))
    bad = ~(err <= 1e-6 * scale + 1e-30) & ~(np.isnan(means[kept]) & np.isnan(want.means[kept]))
    assert not bad.any(), f"averages differ at {np.argwhere(bad)[:5]}"
    # an order statistic moves by at most the largest change of its inputs
    col_scale = scale.max(axis=0) if scale.size else np.zeros(d)
    got = buf.out.cpu().numpy().astype(np.float64)
    ref = want.out.astype(np.float64)
    if mode == 0:
        err = np.abs(got - ref)
        bad = ~(err <= 1e-6 * col_scale + 1e-30) & ~(np.isnan(got) & np.isnan(ref))
        assert not bad.any(), f"lower median differs at {np.nonzero(bad)[0][:5]}"
        if exact_means:
            assert np.array_equal(as_u32(buf.out), want.out.view(np.uint32)), "lower median bits"
    else:
        assert_mean_close(buf.out.cpu().numpy(), want.out, col_scale)


def chosen_abs_mean(host, want):
    """[f, d] mean |x| over the chosen copies of each file (0 where dropped)."""
    f, r, _ = host.shape
    d = want.means.shape[1]
    out = np.zeros((f, d))
    for i in range(f):
        slots = [s for s in range(r) if (int(want.slot_mask[i]) >> s) & 1]
        if slots:
            out[i] = np.abs(host[i, slots, :d].astype(np.float64)).mean(axis=0)
    return out


CASES = [
    ("k7_r3_d4096_alie", 4097, 0.0, 0.0),
    ("k15_r3_d1m_weak_reversed", 3001, 0.0, 0.0),
    ("k15_r3_d11m_strong_alie", 3001, 0.0, 0.0),
    ("k15_r5_d1m_strong_alie", 1027, 0.0, 0.0),
    ("k7_r3_d4096_alie", 4097, 1e-6, 1e-4),
    ("k15_r3_d1m_weak_reversed", 3001, 1e-6, 1e-4),
    ("k15_r3_d11m_strong_alie", 3001, 1e-6, 1e-4),
    ("k15_r5_d1m_strong_alie", 1027, 1e-6, 1e-4),
    ("k21_r3_d2m_strong_alie", 513, 1e-6, 1e-4),
    ("k15_r3_d11m_strong_alie", 3001, 1e-4, 1e-6),    # noise above tau: honest copies split
]


@pytest.mark.parametrize("name,d,noise,tau", CASES)
@pytest.mark.parametrize("mode", [0, 1])
def test_tolerant_round(name, d, noise, tau, mode):
    w = dataclasses.replace(synth.CONFIGS[name], d=d, copy_noise=noise)
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers)
    want = oracle.run_round_tolerant(host, oa, tau, w.d, mode)
    # identical copies average to themselves on both sides: the median is exact
    check(run(host, w, tau, mode), want, host, mode, exact_means=noise == 0.0)
    if noise == 0.0 and tau == 0.0 and mode == 0:
        exact = oracle.run_round(host, oa, w.d, 0)
        assert np.array_equal(want.out.view(np.uint32), exact.out.view(np.uint32))


@pytest.mark.parametrize("offset,ldm_pad", [(1, 0), (0, 3), (1, 1)])
def test_tolerant_unaligned_paths(offset, ldm_pad):
    w = dataclasses.replace(synth.CONFIGS["k15_r3_d11m_strong_alie"], d=2049, ld_align=1,
                            copy_noise=1e-6)
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers)
    want = oracle.run_round_tolerant(host, oa, 1e-4, w.d, 0)
    check(run(host, w, 1e-4, 0, offset, ldm_pad), want, host, 0)


@pytest.mark.parametrize("K,r,q,attack", [(6, 2, 2, "weak"), (8, 2, 3, "strong"), (8, 4, 3, "strong"),
                                          (9, 4, 4, "weak"), (9, 6, 4, "strong")])
def test_tolerant_other_r(K, r, q, attack):
    w = synth.Workload("tol_r", K=K, r=r, d=1003, q=q, attack=attack, distortion="alie", seed=K + r,
                       copy_noise=1e-6)
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers)
    want = oracle.run_round_tolerant(host, oa, 1e-4, w.d, 0)
    check(run(host, w, 1e-4), want, host)


def test_tolerant_foe_and_nans():
    w = synth.Workload("foe", K=9, r=3, d=777, q=3, attack="strong", distortion="foe", z=0.5,
                       seed=5, copy_noise=1e-6)
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers)
    want = oracle.run_round_tolerant(host, oa, 1e-4, w.d, 0)
    check(run(host, w, 1e-4), want, host)
    host[3, 1, 5] = np.nan                     # one copy is no longer close to anything
    host[10, :, 7] = np.nan                    # identical NaNs are not close either
    want = oracle.run_round_tolerant(host, oa, 1e-4, w.d, 0)
    check(run(host, w, 1e-4), want, host)


def test_tolerant_rejects_bad_tau():
    w = dataclasses.replace(synth.CONFIGS["k7_r3_d4096_alie"], d=64)
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers)
    for tau in (-1.0, float("nan")):
        with pytest.raises(ap.AspisError) as e:
            run(host, w, tau)
        assert e.value.status == ap.E_INVAL


def test_tolerant_full_length_equals_exact_round():
    """ResNet-18 length, optimal attack: with tau = 0 the tolerant round's
    output equals the exact round's bit for bit (both checked against the
    oracle elsewhere), and its averages equal the chosen copies."""
    w = synth.CONFIGS["k15_r3_d11m_strong_alie"]
    a = ap.aspis_assign(w.K, w.r)
    copies = synth.build_copies_torch(w, a.file_workers(), DEV)
    exact = ap.RoundBuffers(a, w.d, DEV)
    ap.aspis_round(copies, w.d, a, exact.file_neq, exact.adj, exact.det, exact.sel, exact.out)
    buf = ap.TolerantBuffers(a, w.d, DEV)
    ap.aspis_round_tolerant(copies, w.d, a, 0.0, buf.file_neq, buf.adj, buf.det, buf.slot_mask,
                            buf.sel, buf.means, buf.out)
    torch.cuda.synchronize()
    assert torch.equal(buf.out.view(torch.int32), exact.out.view(torch.int32))
    sel = exact.sel.cpu().numpy()
    rng = np.random.default_rng(0)
    for i in rng.choice(a.f, 8, replace=False):
        if sel[i] >= 0:
            assert torch.equal(buf.means[i, : w.d].view(torch.int32),
                               copies[i, int(sel[i]), : w.d].view(torch.int32))
