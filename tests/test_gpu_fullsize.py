"""Full-size parity: the five benchmark workloads at their real sizes, run
through the C ABI exactly as bench.py runs them (aspis_check, aspis_detect,
aspis_select, aspis_aggregate on one side stream).

The oracle recomputes every file's agreement word on the host (files are
streamed through a pinned buffer), then the graph, the maximum cliques and
the selection, all compared exactly.  The median is compared bit for bit on
every coordinate: the copies the oracle selects are gathered on the device in
chunks of coordinates and the oracle aggregates each chunk on the host."""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)
ap = pytest.importorskip("paper_2108_02416_gb300")
DEV = torch.device("cuda:0")


def oracle_file_neq(copies, d, files_per_chunk):
    """Oracle agreement words for all files, streaming chunks of files to host."""
    f, r, ld = copies.shape
    out = np.zeros(f, np.uint32)
    stage = torch.empty((files_per_chunk, r, d), dtype=torch.float32, pin_memory=True)
    for i0 in range(0, f, files_per_chunk):
        i1 = min(f, i0 + files_per_chunk)
        stage[: i1 - i0].copy_(copies[i0:i1, :, :d])
        out[i0:i1] = oracle.file_agreement(stage[: i1 - i0].numpy(), d)
    return out


def oracle_round(copies, w, oa):
    """Oracle agreement, graph, cliques and selection for the device copies."""
    row_bytes = w.r * w.d * 4
    fneq = oracle_file_neq(copies, w.d, max(1, int(2e9 // row_bytes)))
    alpha = oracle.pair_agreement(fneq, oa)
    adj = oracle.graph(alpha, w.K, w.r)
    odet = oracle.detect(adj, w.K)
    sel, n_sel = oracle.select(fneq, oa, odet.clique, odet.success)
    return fneq, adj, odet, sel, n_sel


def gather_chosen(copies, w, sel, cols):
    """[n_sel, len(cols)] values of the chosen copies at the given coordinates."""
    kept = np.nonzero(sel >= 0)[0]
    rows_idx = torch.from_numpy(kept * w.r + sel[kept].astype(np.int64)).to(DEV)
    flat = copies.view(-1, copies.shape[2])
    sub = flat[:, torch.from_numpy(cols).to(DEV)]          # columns first: small
    return sub.index_select(0, rows_idx).cpu().numpy()


@pytest.mark.parametrize("name", list(synth.CONFIGS))
def test_fullsize_round(name):
    w = synth.CONFIGS[name]
    oa = oracle.assign(w.K, w.r)
    a = ap.aspis_assign(w.K, w.r)
    assert np.array_equal(a.file_workers(), oa.file_workers)
    copies = synth.build_copies_torch(w, oa.file_workers, DEV)
    buf = ap.RoundBuffers(a, w.d, DEV)
    stream = torch.cuda.Stream(device=DEV)
    stream.wait_stream(torch.cuda.current_stream())      # inputs were made on the default stream
    with torch.cuda.stream(stream):
        ap.aspis_check(copies, w.d, a, buf.file_neq, buf.adj, stream)
        ap.aspis_detect(buf.adj, w.K, buf.det, stream)
        ap.aspis_select(buf.file_neq, buf.det, a, buf.sel, stream)
        ap.aspis_aggregate(copies, w.d, a, buf.sel, buf.det, buf.out, ap.MEDIAN, stream)
    torch.cuda.synchronize()
    det = buf.detection()
    assert det.status == ap.OK

    fneq, adj, odet, sel, n_sel = oracle_round(copies, w, oa)

    assert np.array_equal(buf.file_neq.cpu().numpy().view(np.uint32), fneq)
    assert np.array_equal(buf.adj.cpu().numpy().view(np.uint32), adj)
    assert (det.omega, det.n_max_cliques, det.clique_mask, bool(det.success)) == \
        (odet.omega, odet.n_max, odet.clique, odet.success)
    assert np.array_equal(buf.sel.cpu().numpy(), sel) and det.n_sel == n_sel

    got = buf.out.cpu().numpy().view(np.uint32)
    bad = []
    for c0, want in oracle_median_chunks(copies, w, sel):
        diff = np.nonzero(got[c0: c0 + len(want)] != want.view(np.uint32))[0]
        bad.extend((c0 + diff[:8]).tolist())
    assert not bad, f"median differs at coordinates {bad[:8]}"
    # how many coordinates the kernel settled by its exact key-space path
    print(f"{name}: {det.median_exact} of {w.d} coordinates by the exact path")
    del copies
    torch.cuda.empty_cache()


def oracle_median_chunks(copies, w, sel, max_bytes=1 << 28):
    """(c0, oracle lower median of coordinates [c0, c0 + m)) for consecutive
    chunks covering all d coordinates: the oracle's chosen rows are gathered on
    the device, copied to the host and aggregated there by the oracle."""
    kept = np.nonzero(sel >= 0)[0]
    n = len(kept)
    rows_idx = torch.from_numpy(kept * w.r + sel[kept].astype(np.int64)).to(DEV)
    flat = copies.view(-1, copies.shape[2])
    step = max(4096, max_bytes // (4 * n) // 32 * 32)
    slot0 = np.zeros(n, np.int8)           # one row per kept file: slot 0
    for c0 in range(0, w.d, step):
        c1 = min(w.d, c0 + step)
        chunk = flat[:, c0:c1].index_select(0, rows_idx)
        host = chunk.contiguous().cpu().numpy().reshape(n, 1, c1 - c0)
        yield c0, oracle.aggregate(host, slot0, 0, 0, c1 - c0)


def test_fullsize_mean_sampled():
    """Mean aggregator at a full size (Case 1 workload), sampled coordinates."""
    w = synth.CONFIGS["k15_r3_d1m_weak_reversed"]
    oa = oracle.assign(w.K, w.r)
    a = ap.aspis_assign(w.K, w.r)
    copies = synth.build_copies_torch(w, oa.file_workers, DEV)
    buf = ap.RoundBuffers(a, w.d, DEV)
    ap.aspis_round(copies, w.d, a, buf.file_neq, buf.adj, buf.det, buf.sel, buf.out, ap.MEAN)
    torch.cuda.synchronize()
    _, _, _, sel, _ = oracle_round(copies, w, oa)
    assert np.array_equal(buf.sel.cpu().numpy(), sel)
    rng = np.random.default_rng(3)
    cols = np.unique(rng.integers(0, w.d, 2048)).astype(np.int64)
    gathered = gather_chosen(copies, w, sel, cols)
    want = oracle.mean(gathered)
    got = buf.out.cpu().numpy()[cols]
    scale = np.abs(gathered.astype(np.float64)).mean(0)
    err = np.abs(got.astype(np.float64) - want.astype(np.float64))
    assert (err <= 1e-6 * np.maximum(np.abs(want.astype(np.float64)), scale) + 1e-30).all()
