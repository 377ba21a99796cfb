"""Pins for the variant with copies that are not bit-identical (Section 5,
after Algorithm 1: average the honest copies in Case 1, average the largest
cluster of copies in Case 2) and for the new generator options (Fall of
Empires, per-copy noise).  Readings: copies are close iff every coordinate
differs by at most tau in fp32; clusters are connected components of
"close"; the average is the arithmetic mean of the chosen copies, rounded
once to fp32."""
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth


def f32(x):
    return np.float32(x)


def two_copy_file(a, b, r=2):
    c = np.zeros((1, r, len(a)), np.float32)
    c[0, 0] = a
    c[0, 1] = b
    return c


def test_close_relation_edges():
    tau = 0.25
    assert oracle.file_agreement_tol(two_copy_file([1.0, 2.0], [1.25, 2.0]), tau)[0] == 0
    above = np.nextafter(f32(1.25), f32(2.0))
    assert oracle.file_agreement_tol(two_copy_file([1.0, 2.0], [above, 2.0]), tau)[0] == 1
    nan = f32(np.nan)
    assert oracle.file_agreement_tol(two_copy_file([nan], [nan]), 1.0)[0] == 1     # NaN never close
    inf = f32(np.inf)
    assert oracle.file_agreement_tol(two_copy_file([inf], [inf]), 1.0)[0] == 1     # inf - inf is NaN
    assert oracle.file_agreement_tol(two_copy_file([0.0], [-0.0]), 0.0)[0] == 0    # |+0 - -0| = 0
    with pytest.raises(ValueError):
        oracle.file_agreement_tol(two_copy_file([0.0], [0.0]), -1.0)


@pytest.mark.parametrize("name", ["k7_r3_d4096_alie", "k15_r3_d1m_weak_reversed",
                                  "k15_r3_d11m_strong_alie", "k15_r5_d1m_strong_alie"])
def test_zero_tolerance_is_bitwise_equality(name):
    """With tau = 0 and copies free of NaN and signed-zero differences,
    "close" is bitwise equality, and the whole tolerant round (clusters,
    averages of identical copies) reproduces the exact round bit for bit."""
    import dataclasses
    w = dataclasses.replace(synth.CONFIGS[name], d=257)
    a = oracle.assign(w.K, w.r)
    copies = synth.build_copies_np(w, a.file_workers)
    exact = oracle.run_round(copies, a, w.d, 0)
    tol = oracle.run_round_tolerant(copies, a, 0.0, w.d, 0)
    assert np.array_equal(tol.file_neq, exact.file_neq)
    assert np.array_equal(tol.adj, exact.adj)
    assert tol.det == exact.det
    assert tol.n_kept == exact.n_sel
    assert np.array_equal(tol.slot_mask != 0, exact.sel >= 0)
    assert np.array_equal(tol.out.view(np.uint32), exact.out.view(np.uint32))


def test_clusters_single_linkage_and_ties():
    # r = 5: close pairs 0~2, 2~4 (0 and 4 not close) and 1~3: clusters {0,2,4}, {1,3}
    a = oracle.assign(5, 5)
    close = {(0, 2), (2, 4), (1, 3)}
    word = 0
    p = 0
    for s in range(5):
        for t in range(s + 1, 5):
            if (s, t) not in close:
                word |= 1 << p
            p += 1
    mask, n = oracle.select_tol(np.array([word], np.uint32), a, 0, False)
    assert mask[0] == 0b10101 and n == 1
    # r = 4, clusters {0,1} and {2,3} tie: the one with the lower slot
    a4 = oracle.assign(4, 4)
    word = 0
    p = 0
    for s in range(4):
        for t in range(s + 1, 4):
            if (s, t) not in {(0, 1), (2, 3)}:
                word |= 1 << p
            p += 1
    mask, _ = oracle.select_tol(np.array([word], np.uint32), a4, 0, False)
    assert mask[0] == 0b0011
    # all apart: a single slot, the lowest
    mask, _ = oracle.select_tol(np.array([0b111111], np.uint32), a4, 0, False)
    assert mask[0] == 0b0001


def test_case1_masks_and_dropped_files():
    a = oracle.assign(6, 3)
    clique = 0b000111                         # workers 0, 1, 2 honest
    mask, n = oracle.select_tol(np.zeros(a.f, np.uint32), a, clique, True)
    for i in range(a.f):
        want = sum(1 << s for s in range(3) if (clique >> int(a.file_workers[i, s])) & 1)
        assert mask[i] == want
    assert n == sum(1 for i in range(a.f) if mask[i])
    assert n == a.f - 1                       # only the file {3, 4, 5} has no honest worker


def test_means_exact_cases():
    inf, nan = np.inf, np.nan
    # identical copies give their value exactly, including -0, inf and NaN payloads
    x = np.array([-0.0, inf, -inf, 1e-45, 3.0e38, 1.0 / 3.0], np.float32)
    nan_bits = np.array([0x7FC00123], np.uint32).view(np.float32)
    x = np.concatenate([x, nan_bits])
    c = np.stack([x, x, x])[None]             # one file, r = 3, all identical
    m = oracle.file_means(c, np.array([0b111], np.uint8))
    assert np.array_equal(m[0].view(np.uint32), x.view(np.uint32))
    # dyadic values: the mean is exact
    c = np.array([[[1.0, 8.0], [1.5, 8.0], [2.0, 4.0], [2.5, 4.0]]], np.float32)
    m = oracle.file_means(c, np.array([0b1111], np.uint8))
    assert m[0].tolist() == [1.75, 6.0]
    m = oracle.file_means(c, np.array([0b0101], np.uint8))           # slots 0 and 2
    assert m[0].tolist() == [1.5, 6.0]
    m = oracle.file_means(c, np.array([0b1000], np.uint8))           # one copy: itself
    assert m[0].tolist() == [2.5, 4.0]


@pytest.mark.parametrize("spread", [1e-3, 1.0, 1e6])
def test_means_are_the_exact_mean_rounded(spread):
    """The average is the exact rational mean of the chosen copies within
    one ulp of the result (one rounding of a double sum and quotient), for
    close copies, copies of mixed sign and copies of very different size."""
    rng = np.random.default_rng(2)
    f, r, d = 40, 5, 64
    base = rng.standard_normal((f, 1, d)).astype(np.float32)
    c = (base + rng.standard_normal((f, r, d)).astype(np.float32) * spread).astype(np.float32)
    masks = rng.integers(1, 32, f).astype(np.uint8)
    m = oracle.file_means(c, masks)
    for i in range(f):
        slots = [s for s in range(r) if (masks[i] >> s) & 1]
        for j in range(d):
            exact = sum(Fraction(float(c[i, s, j])) for s in slots) / len(slots)
            got = Fraction(float(m[i, j]))
            assert abs(got - exact) <= Fraction(float(np.spacing(np.float32(abs(m[i, j]))))), \
                (i, j)


def test_noisy_honest_copies_keep_the_graph():
    """Honest copies with independent noise far below tau: the tolerant graph,
    clique and kept files equal those of the noiseless exact round, and the
    output stays within the noise of the noiseless output."""
    import dataclasses
    for name in ["k15_r3_d1m_weak_reversed", "k15_r3_d11m_strong_alie"]:
        w = dataclasses.replace(synth.CONFIGS[name], d=300)
        wn = dataclasses.replace(w, copy_noise=1e-6)
        a = oracle.assign(w.K, w.r)
        clean = oracle.run_round(synth.build_copies_np(w, a.file_workers), a, w.d, 0)
        noisy_copies = synth.build_copies_np(wn, a.file_workers)
        exact_noisy = oracle.run_round(noisy_copies, a, w.d, 0)
        assert exact_noisy.det.omega < clean.det.omega          # bitwise equality breaks down
        tol = oracle.run_round_tolerant(noisy_copies, a, 1e-4, w.d, 0)
        assert np.array_equal(tol.adj, clean.adj)
        assert tol.det == clean.det
        assert tol.n_kept == clean.n_sel
        assert np.max(np.abs(tol.out - clean.out)) < 1e-5


def test_foe_and_copy_noise_generators():
    import dataclasses
    w = synth.Workload("foe", K=7, r=3, d=50, q=2, attack="all_alie", distortion="foe", z=0.5,
                       seed=3, adversaries=(0, 1))
    a = oracle.assign(7, 3)
    c = synth.build_copies_np(w, a.file_workers)
    honest = np.stack([synth.honest_np(w.seed, i, 0, w.d) for i in range(a.f)]).astype(np.float64)
    want = (-0.5 * honest.mean(axis=0)).astype(np.float32)
    mask = synth.corrupted_mask(w, a.file_workers)
    for i, s in zip(*np.nonzero(mask)):
        assert np.allclose(c[i, s, : w.d], want, rtol=0, atol=1e-9)
    wn = dataclasses.replace(w, distortion="reversed", copy_noise=1e-3)
    cn = synth.build_copies_np(wn, a.file_workers)
    torch = pytest.importorskip("torch")
    ct = synth.build_copies_torch(wn, a.file_workers, torch.device("cpu"))
    assert np.array_equal(cn.view(np.uint32), ct.numpy().view(np.uint32))
    for i in range(a.f):                                     # honest copies now differ
        h = [s for s in range(3) if not mask[i, s]]
        if len(h) >= 2:
            assert not np.array_equal(cn[i, h[0]], cn[i, h[1]])
            assert np.max(np.abs(cn[i, h[0], : w.d] - cn[i, h[1], : w.d])) < 1e-2
