"""GPU parity: every step of the CUDA path against the CPU oracle on the same
seeded inputs, at sizes the oracle finishes in seconds (several tiles, ragged
tails), plus the degenerate and edge cases of the method."""
import math

import numpy as np
import pytest

import oracle
import synth
from _gpu_round import as_u32, assert_mean_close, assert_round_matches, gpu_round

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)
ap = pytest.importorskip("paper_2108_02416_gb300")
DEV = torch.device("cuda:0")


def run_case(w, mode=0, ld=None, pad=0.0, offset=0):
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers, pad_value=pad)
    if ld is not None and ld != host.shape[2]:
        h2 = np.full((oa.f, w.r, ld), pad, np.float32)
        h2[:, :, : w.d] = host[:, :, : w.d]
        host = h2
    want = oracle.run_round(host, oa, w.d, mode)
    a = ap.aspis_assign(w.K, w.r)
    flat = torch.empty(host.size + offset, dtype=torch.float32, device=DEV)
    dev = flat[offset:].view(host.shape)
    dev.copy_(torch.from_numpy(host))
    buf = gpu_round(ap, torch, dev, w.d, a, mode)
    return buf, want, host


# ------------------------------------------------ the five workloads, small d

SMALL = [
    synth.Workload("cfg1", K=7, r=3, d=4096, q=2, attack="all_alie", seed=0, adversaries=(0, 1)),
    synth.Workload("cfg2s", K=15, r=3, d=4099, q=3, attack="weak", distortion="reversed", seed=1),
    synth.Workload("cfg3s", K=15, r=3, d=8197, q=3, attack="strong", z=1.0, seed=2),
    synth.Workload("cfg4s", K=21, r=3, d=2053, q=5, attack="strong", z=1.5, seed=3),
    synth.Workload("cfg5s", K=15, r=5, d=1031, q=4, attack="strong", z=1.0, seed=4),
]


@pytest.mark.parametrize("w", SMALL, ids=[w.name for w in SMALL])
def test_round_parity_small(w):
    buf, want, _ = run_case(w)
    assert_round_matches(ap, buf, want)


@pytest.mark.parametrize("w", SMALL[:3], ids=[w.name for w in SMALL[:3]])
def test_round_parity_mean(w):
    buf, want, host = run_case(w, mode=1)
    assert_round_matches(ap, buf, want, mode=1, check_out=False)
    rows = np.array([host[i, want.sel[i], : w.d] for i in range(len(want.sel)) if want.sel[i] >= 0])
    assert_mean_close(buf.out.cpu().numpy(), want.out, np.abs(rows.astype(np.float64)).mean(0))


def test_theorem1_counts_on_gpu():
    """Optimal attack: two maximum cliques and (1/2) C(2q, r) corrupted picks."""
    w = synth.Workload("t1", K=15, r=3, d=67, q=4, attack="strong", seed=9)
    buf, want, _ = run_case(w)
    det = buf.detection()
    assert det.n_max_cliques == 2 and det.omega == w.K - w.q and not det.success
    oa = oracle.assign(w.K, w.r)
    mask = synth.corrupted_mask(w, oa.file_workers)
    sel = buf.sel.cpu().numpy()
    assert 2 * sum(bool(mask[i, sel[i]]) for i in range(oa.f)) == math.comb(2 * w.q, w.r)


# ------------------------------------------------------- ragged / unaligned


@pytest.mark.parametrize("d", [1, 2, 3, 4, 5, 7, 31, 33, 127, 129, 16387])
@pytest.mark.parametrize("layout", ["ld32", "ld_eq_d", "offset1"])
def test_ragged_and_unaligned(d, layout):
    w = synth.Workload("rag", K=8, r=3, d=d, q=3, attack="strong", seed=d)
    if layout == "ld32":
        buf, want, _ = run_case(w, pad=np.float32(np.nan))
    elif layout == "ld_eq_d":
        buf, want, _ = run_case(w, ld=d)
    else:
        buf, want, _ = run_case(w, offset=1, pad=-5.0)
    assert_round_matches(ap, buf, want)


def test_padding_ignored_even_when_copies_differ_there():
    w = synth.Workload("pad", K=9, r=4, d=45, q=0, seed=5)
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers)
    rng = np.random.default_rng(0)
    host[:, :, w.d:] = rng.standard_normal(host[:, :, w.d:].shape).astype(np.float32)
    want = oracle.run_round(host, oa, w.d)
    a = ap.aspis_assign(w.K, w.r)
    buf = gpu_round(ap, torch, torch.from_numpy(host).to(DEV), w.d, a)
    assert_round_matches(ap, buf, want)
    assert int(as_u32(buf.file_neq).max()) == 0


# ------------------------------------------------------- every redundancy


@pytest.mark.parametrize("K,r,q", [(10, 2, 4), (9, 4, 3), (11, 5, 5), (12, 6, 4), (9, 7, 3),
                                   (10, 8, 4), (31, 2, 8), (31, 3, 6)])
def test_all_r(K, r, q):
    w = synth.Workload("r", K=K, r=r, d=203, q=q, attack="strong", seed=K * r)
    buf, want, _ = run_case(w)
    assert_round_matches(ap, buf, want)
    w = synth.Workload("rw", K=K, r=r, d=203, q=q, attack="weak", distortion="reversed",
                       seed=K + r)
    buf, want, _ = run_case(w)
    assert_round_matches(ap, buf, want)


# ---------------------------------------------- signed zeros, NaN, ties


def test_special_values_and_ties():
    K, r, d = 9, 3, 257
    oa = oracle.assign(K, r)
    rng = np.random.default_rng(42)
    palette = np.array([0x00000000, 0x80000000, 0x3f800000, 0xbf800000, 0x7fc00000,
                        0x7fc00001, 0xffc00000, 0x7f800000, 0xff800000, 0x00000001,
                        0x80000001], np.uint32)
    base = palette[rng.integers(0, len(palette), (oa.f, d))].view(np.float32)
    host = np.repeat(base[:, None, :], r, axis=1).copy()
    # a few files where one copy differs only by the sign of a zero or a NaN payload
    host.view(np.uint32)[3, 1, 7] ^= 0x80000000
    host.view(np.uint32)[5, 2, 100] = 0x7fc00002
    want = oracle.run_round(host, oa, d)
    a = ap.aspis_assign(K, r)
    buf = gpu_round(ap, torch, torch.from_numpy(host).to(DEV), d, a)
    assert_round_matches(ap, buf, want)


def test_median_all_equal_and_two_values():
    K, r, d = 7, 3, 96
    oa = oracle.assign(K, r)
    host = np.zeros((oa.f, r, d), np.float32)
    host[:, :, :32] = 1.5                                  # all equal
    host[: oa.f // 2, :, 32:64] = -2.0                     # two values, 17 / 18 split
    host[oa.f // 2:, :, 32:64] = 3.0
    host[:, :, 64:] = np.arange(oa.f, dtype=np.float32)[:, None, None] * 1e-38  # subnormals
    want = oracle.run_round(host, oa, d)
    a = ap.aspis_assign(K, r)
    buf = gpu_round(ap, torch, torch.from_numpy(host).to(DEV), d, a)
    assert_round_matches(ap, buf, want)


def test_no_majority_plurality():
    """r=5 files whose copies split 2-2-1 or are all different (no strict
    majority): plurality with the lower-slot tie-break, as in the oracle."""
    K, r, d = 8, 5, 12
    oa = oracle.assign(K, r)
    rng = np.random.default_rng(1)
    host = np.repeat(rng.standard_normal((oa.f, 1, d)).astype(np.float32), r, axis=1)
    for i in range(oa.f):
        pattern = [[0, 0, 1, 1, 2], [0, 1, 2, 3, 4], [1, 1, 0, 0, 0], [0, 1, 1, 0, 2]][i % 4]
        for s in range(r):
            host[i, s] += np.float32(pattern[s])
    want = oracle.run_round(host, oa, d)
    a = ap.aspis_assign(K, r)
    buf = gpu_round(ap, torch, torch.from_numpy(host).to(DEV), d, a)
    assert_round_matches(ap, buf, want)


# ------------------------------------------------------------ detection


def detect_gpu(adj, K, budget=0):
    det = torch.zeros(ap.DETECTION_BYTES, dtype=torch.uint8, device=DEV)
    if budget:
        det.view(torch.int32)[7] = budget
    ap.aspis_detect(torch.from_numpy(adj.view(np.int32)).to(DEV), K, det)
    torch.cuda.synchronize()
    return ap.Detection.from_tensor(det)


def random_adj(K, p, rng):
    adj = np.zeros(K, np.uint32)
    for j in range(K):
        for k in range(j + 1, K):
            if rng.random() < p:
                adj[j] |= np.uint32(1 << k)
                adj[k] |= np.uint32(1 << j)
    return adj


def test_detect_random_graphs():
    rng = np.random.default_rng(3)
    for trial in range(150):
        K = int(rng.integers(2, 32))
        p = float(rng.choice([0.05, 0.3, 0.5, 0.7, 0.9, 0.98]))
        adj = random_adj(K, p, rng)
        want = oracle.max_cliques_bk(adj, K)
        got = detect_gpu(adj, K)
        assert got.status == ap.OK
        assert (got.omega, got.n_max_cliques, got.clique_mask) == (want.omega, want.n_max, want.clique)
        assert got.success == (want.n_max == 1)


@pytest.mark.parametrize("parts", [2, 5, 10])
def test_detect_moon_moser(parts):
    K = 3 * parts
    adj = np.array([sum(1 << k for k in range(K) if k // 3 != j // 3) for j in range(K)], np.uint32)
    got = detect_gpu(adj, K)
    assert got.status == ap.OK
    assert (got.omega, got.n_max_cliques) == (parts, 3 ** parts)
    assert got.clique_mask == sum(1 << (3 * p) for p in range(parts))


def test_detect_degenerate_graphs():
    for K in (2, 3, 17, 31):
        got = detect_gpu(np.zeros(K, np.uint32), K)
        assert (got.omega, got.n_max_cliques, got.clique_mask, got.success) == (1, K, 1, 0)
        full = np.array([((1 << K) - 1) & ~(1 << j) for j in range(K)], np.uint32)
        got = detect_gpu(full, K)
        assert (got.omega, got.n_max_cliques, got.clique_mask, got.success) == (K, 1, (1 << K) - 1, 1)


def test_detect_budget_exhaustion_reports_limit():
    K = 30
    adj = np.array([sum(1 << k for k in range(K) if k // 3 != j // 3) for j in range(K)], np.uint32)
    got = detect_gpu(adj, K, budget=10)
    assert got.status == ap.E_LIMIT and got.success == 0
    got = detect_gpu(adj, K)          # the default budget finishes the same graph
    assert got.status == ap.OK and got.n_max_cliques == 3 ** 10


# ------------------------------------------------------- statuses / errors


def test_empty_selection_reports_status_and_leaves_out():
    K, r, d = 7, 3, 40
    a = ap.aspis_assign(K, r)
    copies = torch.randn(a.f, r, 64, device=DEV)
    sel = torch.full((a.f,), -1, dtype=torch.int8, device=DEV)
    det = torch.zeros(ap.DETECTION_BYTES, dtype=torch.uint8, device=DEV)
    out = torch.full((d,), 7.0, device=DEV)
    ap.aspis_aggregate(copies, d, a, sel, det, out)
    torch.cuda.synchronize()
    assert ap.Detection.from_tensor(det).status == ap.E_EMPTY
    assert bool((out == 7.0).all())


def test_aggregate_rejects_too_many_files():
    a = ap.aspis_assign(18, 6)                    # f = 18564 > ASPIS_MAX_AGG_FILES
    copies = torch.zeros(a.f, 6, 4, device=DEV)
    buf = ap.RoundBuffers(a, 4, DEV)
    with pytest.raises(ap.AspisError) as ei:
        ap.aspis_aggregate(copies, 4, a, buf.sel, buf.det, buf.out)
    assert ei.value.status == ap.E_RANGE
    # the check step has no such limit
    ap.aspis_check(copies, 4, a, buf.file_neq, buf.adj)
    torch.cuda.synchronize()
    assert int(as_u32(buf.file_neq).max()) == 0


def test_large_f_check_and_select_parity():
    """f = 18564 files (K=18, r=6): check, detect and select against the oracle."""
    w = synth.Workload("bigf", K=18, r=6, d=9, q=5, attack="strong", seed=11)
    oa = oracle.assign(w.K, w.r)
    host = synth.build_copies_np(w, oa.file_workers)
    want = oracle.run_round(host, oa, w.d, aggregate_out=False)
    a = ap.aspis_assign(w.K, w.r)
    dev = torch.from_numpy(host).to(DEV)
    buf = ap.RoundBuffers(a, w.d, DEV)
    ap.aspis_check(dev, w.d, a, buf.file_neq, buf.adj)
    ap.aspis_detect(buf.adj, w.K, buf.det)
    ap.aspis_select(buf.file_neq, buf.det, a, buf.sel)
    torch.cuda.synchronize()
    assert_round_matches(ap, buf, want, check_out=False)


def test_two_rounds_same_buffers():
    """Buffers are reused round after round: nothing leaks between rounds."""
    w1 = synth.Workload("a", K=15, r=3, d=999, q=3, attack="strong", seed=21)
    w2 = synth.Workload("b", K=15, r=3, d=999, q=3, attack="weak", distortion="reversed", seed=22)
    a = ap.aspis_assign(15, 3)
    oa = oracle.assign(15, 3)
    buf = ap.RoundBuffers(a, 999, DEV)
    for w in (w1, w2, w1):
        host = synth.build_copies_np(w, oa.file_workers)
        want = oracle.run_round(host, oa, w.d)
        ap.aspis_round(torch.from_numpy(host).to(DEV), w.d, a, buf.file_neq, buf.adj, buf.det,
                       buf.sel, buf.out)
        torch.cuda.synchronize()
        assert_round_matches(ap, buf, want)


def test_round_host_entry_point():
    w = SMALL[1]
    oa = oracle.assign(w.K, w.r)
    host = torch.from_numpy(synth.build_copies_np(w, oa.file_workers)).pin_memory()
    want = oracle.run_round(host.numpy(), oa, w.d)
    a = ap.aspis_assign(w.K, w.r)
    buf = ap.RoundBuffers(a, w.d, DEV)
    dev = torch.empty_like(host, device=DEV)
    hout = torch.empty(w.d, dtype=torch.float32).pin_memory()
    hdet = torch.zeros(ap.DETECTION_BYTES, dtype=torch.uint8).pin_memory()
    ap.aspis_round_host(host, dev, w.d, a, buf.file_neq, buf.adj, buf.det, buf.sel, buf.out,
                        hout, hdet)
    torch.cuda.synchronize()
    assert np.array_equal(hout.numpy().view(np.uint32), want.out.view(np.uint32))
    det = ap.Detection.from_buffer_copy(bytes(hdet.numpy().tobytes()))
    assert det.success == want.det.success and det.n_sel == want.n_sel


@pytest.mark.parametrize("kind", ["pinned", "pinned_offset", "pageable"])
def test_round_host_large_copy_paths(kind):
    """Above 64 MiB the host copy takes the copy kernel (pinned, aligned) or
    the copy engines (pinned at an odd offset, pageable); results are the
    oracle's either way."""
    import dataclasses
    w = dataclasses.replace(synth.CONFIGS["k15_r3_d11m_strong_alie"], d=20000)   # 109 MB
    oa = oracle.assign(w.K, w.r)
    arr = synth.build_copies_np(w, oa.file_workers)
    want = oracle.run_round(arr, oa, w.d)
    if kind == "pageable":
        host = torch.from_numpy(arr)
    else:
        base = torch.empty(arr.size + 1, dtype=torch.float32).pin_memory()
        off = 1 if kind == "pinned_offset" else 0
        host = base[off: off + arr.size].view(arr.shape)
        host.copy_(torch.from_numpy(arr))
    a = ap.aspis_assign(w.K, w.r)
    buf = ap.RoundBuffers(a, w.d, DEV)
    dev = torch.empty(arr.shape, dtype=torch.float32, device=DEV)
    hout = torch.empty(w.d, dtype=torch.float32).pin_memory()
    hdet = torch.zeros(ap.DETECTION_BYTES, dtype=torch.uint8).pin_memory()
    ap.aspis_round_host(host, dev, w.d, a, buf.file_neq, buf.adj, buf.det, buf.sel, buf.out,
                        hout, hdet)
    torch.cuda.synchronize()
    assert torch.equal(dev.cpu().view(torch.int32), torch.from_numpy(arr).view(torch.int32))
    assert np.array_equal(hout.numpy().view(np.uint32), want.out.view(np.uint32))


def test_generator_torch_cuda_matches_numpy():
    """The shared input generator gives the same bits on the GPU and the CPU."""
    w = synth.Workload("g", K=7, r=3, d=1000, q=2, attack="strong", seed=5)
    oa = oracle.assign(7, 3)
    host = synth.build_copies_np(w, oa.file_workers)
    dev = synth.build_copies_torch(w, oa.file_workers, DEV)
    assert np.array_equal(dev.cpu().numpy().view(np.uint32), host.view(np.uint32))


# ------------------------------------------------ exact fallback paths of the median


def _median_case(vals, r=2):
    """vals: float32 [n, d] chosen values; run aggregate with every copy of a
    file equal, so that every file is kept as is (rows past n repeat the last)."""
    n, d = vals.shape
    K = next(k for k in range(r, 200) if math.comb(k, r) >= n)
    f = math.comb(K, r)
    host = np.zeros((f, r, d), np.float32)
    rows = np.concatenate([vals, np.repeat(vals[-1:], f - n, axis=0)]) if f > n else vals
    host[:] = rows[:, None, :]
    oa = oracle.assign(K, r)
    want = oracle.run_round(host, oa, d)
    a = ap.aspis_assign(K, r)
    buf = gpu_round(ap, torch, torch.from_numpy(host).to(DEV), d, a)
    assert_round_matches(ap, buf, want)
    return buf


def test_median_nan_inf_outside_sampled_rows():
    rng = np.random.default_rng(12)
    n, d = 455, 96
    vals = rng.standard_normal((n, d)).astype(np.float32)
    u = vals.view(np.uint32)
    for c in range(d):
        rows = rng.choice(np.arange(100, n), size=3, replace=False)
        kind = c % 6
        pat = [0xffc00000, 0x7fc00000, 0xff800000, 0x7f800000, 0xffc00123, 0x80000000][kind]
        u[rows, c] = pat
    _median_case(vals)


def test_median_heavy_ties_overflow_bin():
    rng = np.random.default_rng(13)
    n, d = 455, 64
    vals = rng.standard_normal((n, d)).astype(np.float32)
    med = np.sort(vals, axis=0)[(n - 1) // 2]
    for c in range(d):
        rows = rng.choice(np.arange(64, n), size=60, replace=False)
        vals[rows, c] = med[c]               # 60 ties straddle the median
    _median_case(vals)


@pytest.mark.parametrize("case", ["plain", "one_warp_15", "one_warp_30", "ties_200", "nan_inf"])
def test_two_pass_median_edge_cases(case):
    """More kept files (3276) than any tag layout holds: the two-pass median.
    Members of the median's bin concentrated in the rows of one warp (rows
    12 apart) overflow its own 10 list rows into the shared ones (15) or past
    them into the exact passes (30); 200 ties exceed the list; NaN and
    infinities sit outside the sampled rows."""
    rng = np.random.default_rng(40)
    n, d = 3276, 256                                     # C(28, 3): every row a distinct file
    vals = rng.standard_normal((n, d)).astype(np.float32)
    if case.startswith("one_warp"):
        k = int(case.split("_")[-1])
        rows = np.arange(24, 24 + 12 * k, 12)           # the rows of one warp
        for c in range(d):
            med = float(np.sort(vals[:, c])[(n - 1) // 2])
            vals[rows, c] = (med + np.arange(k) * 1e-7).astype(np.float32)
    elif case == "ties_200":
        for c in range(d):
            med = float(np.sort(vals[:, c])[(n - 1) // 2])
            vals[rng.choice(np.arange(24, n), size=200, replace=False), c] = med
    elif case == "nan_inf":
        u = vals.view(np.uint32)
        for c in range(d):
            rows = rng.choice(np.arange(100, n), size=3, replace=False)
            u[rows, c] = [0xffc00000, 0x7fc00000, 0xff800000, 0x7f800000][c % 4]
    _median_case(vals, r=3)


def test_median_candidates_concentrated_in_one_lane():
    rng = np.random.default_rng(14)
    n, d = 455, 64
    vals = rng.standard_normal((n, d)).astype(np.float32)
    for c in range(d):
        med = float(np.sort(vals[:, c])[(n - 1) // 2])
        rows = np.arange(64, n, 8)[:20]      # one row group: one lane holds them all
        vals[rows, c] = (med + np.arange(20) * 1e-6).astype(np.float32)
    _median_case(vals)


def test_median_wide_range_and_subnormals():
    rng = np.random.default_rng(15)
    n, d = 300, 64
    mag = 10.0 ** rng.uniform(-44, 38, (n, d))
    vals = (rng.choice([-1.0, 1.0], (n, d)) * mag).astype(np.float32)
    _median_case(vals)


# ------------------------------------------- value-space refinement of a crowded bin


def _crowd(vals, rng, rows_from, count, spread, ties=0):
    """Put `count` distinct values within `spread` of each column's median
    (the first `ties` of them equal to it), away from the sampled rows."""
    n, d = vals.shape
    for c in range(d):
        med = float(np.sort(vals[:, c])[(n - 1) // 2])
        rows = rng.choice(np.arange(rows_from, n), size=count, replace=False)
        off = np.linspace(-spread, spread, count)
        off[:ties] = 0.0
        vals[rows, c] = (med + off).astype(np.float32)


def test_median_refines_crowded_bin():
    """More than 32 distinct values in the median's bin: one refinement level."""
    rng = np.random.default_rng(21)
    vals = rng.standard_normal((455, 96)).astype(np.float32)
    _crowd(vals, rng, 64, 120, 1e-3)
    _median_case(vals)


def test_median_refines_twice():
    """A crowd inside the crowd: two refinement levels before the final list."""
    rng = np.random.default_rng(22)
    vals = rng.standard_normal((455, 64)).astype(np.float32)
    _crowd(vals, rng, 64, 200, 1e-2)
    _crowd(vals, rng, 64, 90, 1e-5)
    _median_case(vals)


def test_median_refine_ties_at_median():
    """Crowded bin whose members around the target rank are all equal."""
    rng = np.random.default_rng(23)
    vals = rng.standard_normal((455, 64)).astype(np.float32)
    _crowd(vals, rng, 64, 100, 1e-4, ties=70)
    _median_case(vals)


def test_median_crowded_overflow_bin_goes_to_key_space():
    """The median sits above every sampled value, among values reaching +inf:
    the members' value range is not finite, so key-space bins take over."""
    rng = np.random.default_rng(24)
    n, d = 455, 32
    vals = np.empty((n, d), np.float32)
    vals[:16] = rng.uniform(-1.0, 1.0, (16, d))          # the sampled rows
    big = 10.0 ** rng.uniform(0.5, 38, (n - 16, d))
    vals[16:] = big.astype(np.float32)
    vals[rng.choice(np.arange(16, n), 20, replace=False), :] = np.inf
    _median_case(vals)


@pytest.mark.parametrize("r", [3, 5])
def test_median_refine_many_rows(r):
    """Thousands of kept files: several warps share a coordinate."""
    rng = np.random.default_rng(25 + r)
    n = 2024 if r == 3 else 3003
    vals = (0.01 * rng.standard_normal((n, 40))).astype(np.float32)
    _crowd(vals, rng, 256, 300, 1e-5, ties=40)
    _median_case(vals, r=r)


def test_median_values_far_below_a_narrow_sample():
    """Values some millions of bin widths below the sampled range map to a
    small negative fma result; they must count in the lowest bin."""
    rng = np.random.default_rng(27)
    n, d = 455, 32
    vals = (1.0 + rng.uniform(0.0, 1.26e-4, (n, d))).astype(np.float32)
    for c in range(d):
        rows = rng.choice(np.arange(16, n), 150, replace=False)
        vals[rows[:100], c] = np.float32(-9.0 - c)
        vals[rows[100:], c] = np.float32(3.0 + c)
    _median_case(vals)


# --------------------------------- 8-bit bin counters that overflow, very large f


@pytest.mark.parametrize("n,equal", [(455, 300), (600, 280), (1200, 300)])
def test_median_bin_counter_overflow(n, equal):
    """More than 255 equal values in one bin overflow an 8-bit counter; the
    bin search sees the coordinate's total change and the exact path decides
    (n = 600 and 1200 keep 680 and 1330 files: bin maps widened 1.25 and
    1.5 times around the sampled range)."""
    rng = np.random.default_rng(n)
    d = 64
    vals = rng.standard_normal((n, d)).astype(np.float32)
    for c in range(d):
        rows = rng.choice(np.arange(32, n), size=equal, replace=False)
        vals[rows, c] = np.float32(0.125 + c * 1e-3)      # inside the sampled range
    buf = _median_case(vals, r=2 if n <= 465 else 3)     # K <= 31 files
    assert buf.detection().median_exact == d


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("layout", ["aligned", "offset1"])
def test_round_k21_r4_near_the_file_limit(mode, layout):
    """K=21, r=4: f = 5985 files, more than any tag layout of the median holds
    in shared memory.  Aligned rows take the two-pass median (no tags), rows
    that are not 16-byte aligned the radix-select path (every coordinate by
    the exact passes); the tag-free mean takes both."""
    w = synth.Workload("k21r4", K=21, r=4, d=1029, q=4, attack="strong", z=1.0, seed=12)
    buf, want, host = run_case(w, mode=mode, offset=1 if layout == "offset1" else 0)
    if mode == 0:
        assert_round_matches(ap, buf, want)
        if layout == "offset1":
            assert buf.detection().median_exact == w.d
        else:
            assert buf.detection().median_exact < w.d
    else:
        assert_round_matches(ap, buf, want, mode=1, check_out=False)
        rows = np.array([host[i, want.sel[i], : w.d] for i in range(len(want.sel))
                         if want.sel[i] >= 0])
        assert_mean_close(buf.out.cpu().numpy(), want.out, np.abs(rows.astype(np.float64)).mean(0))


# ------------------------------------------------ coordinate-split round on one GPU


def test_graph_entry_point_matches_oracle():
    w = synth.CONFIGS["k15_r3_d1m_weak_reversed"]
    oa = oracle.assign(w.K, w.r)
    a = ap.aspis_assign(w.K, w.r)
    rng = np.random.default_rng(31)
    for _ in range(20):
        words = rng.integers(0, 1 << 3, oa.f).astype(np.uint32) * (rng.random(oa.f) < 0.05)
        words = words.astype(np.uint32)
        adj = torch.zeros(w.K, dtype=torch.int32, device=DEV)
        ap.aspis_graph(torch.from_numpy(words.view(np.int32)).to(DEV), a, adj)
        torch.cuda.synchronize()
        want = oracle.graph(oracle.pair_agreement(words, oa), w.K, w.r)
        assert np.array_equal(as_u32(adj), want)


@pytest.mark.parametrize("name", ["k7_r3_d4096_alie", "k15_r3_d11m_strong_alie"])
def test_coordinate_split_round_equals_whole_round(name):
    """Two coordinate slices on one device, combined as two ranks would:
    OR of the mismatch words, then identical graph / cliques / selection and
    per-slice aggregation.  Must equal the whole round and the oracle."""
    from paper_2108_02416_gb300 import shard
    import dataclasses
    w = dataclasses.replace(synth.CONFIGS[name], d=5000)
    oa = oracle.assign(w.K, w.r)
    a = ap.aspis_assign(w.K, w.r)
    full = torch.from_numpy(synth.build_copies_np(w, oa.file_workers, 0, w.d)).to(DEV)
    parts = []
    for p in range(2):
        c0, c1 = shard.shard_bounds(w.d, 2, p)
        ops = shard.DeviceOps(a, DEV)
        parts.append((c0, c1, ops, full[:, :, c0:c1].contiguous()))
    words = shard.or_combine([ops.compare(x, c1 - c0).clone() for c0, c1, ops, x in parts])
    outs = []
    for c0, c1, ops, x in parts:
        adj = ops.graph(words)
        det = ops.detect(adj)
        sel = ops.select(words, det)
        outs.append(ops.aggregate(x, c1 - c0, sel, det))
    torch.cuda.synchronize()
    want = oracle.run_round(full.cpu().numpy(), oa, w.d)
    assert np.array_equal(as_u32(words), want.file_neq)
    for c0, c1, ops, x in parts:
        assert np.array_equal(as_u32(ops.buf.adj), want.adj)
        assert np.array_equal(ops.buf.sel.cpu().numpy(), want.sel)
    out = torch.cat(outs).cpu().numpy()
    assert np.array_equal(out.view(np.uint32), want.out.view(np.uint32))
