"""Helpers for the GPU parity tests: run one round through the C ABI and run
the oracle on the same bytes."""
import numpy as np


def as_u32(t):
    return t.detach().cpu().numpy().view(np.uint32)


def gpu_round(ap, torch, copies_dev, d, a, mode=0, stream=None):
    """copies_dev: CUDA float32 [f, r, ld] (any storage offset)."""
    buf = ap.RoundBuffers(a, d, copies_dev.device)
    ap.aspis_round(copies_dev, d, a, buf.file_neq, buf.adj, buf.det, buf.sel, buf.out, mode,
                   stream)
    torch.cuda.synchronize()
    return buf


def assert_round_matches(ap, buf, want, mode=0, check_out=True):
    det = buf.detection()
    assert det.status == ap.OK, ap.status_str(det.status)
    assert np.array_equal(as_u32(buf.file_neq), want.file_neq), "file_neq"
    assert np.array_equal(as_u32(buf.adj), want.adj), "adjacency"
    got = (det.omega, det.n_max_cliques, det.clique_mask, bool(det.success))
    assert got == (want.det.omega, want.det.n_max, want.det.clique, want.det.success), "clique"
    assert np.array_equal(buf.sel.cpu().numpy(), want.sel), "sel"
    assert det.n_sel == want.n_sel, "n_sel"
    if check_out:
        out = buf.out.cpu().numpy()
        if mode == 0:
            assert np.array_equal(out.view(np.uint32), want.out.view(np.uint32)), \
                f"median mismatch at {np.nonzero(out.view(np.uint32) != want.out.view(np.uint32))[0][:10]}"
        else:
            assert_mean_close(out, want.out, None)


def assert_mean_close(got, want, scale):
    """|gpu - oracle| <= 1e-6 * max(|oracle|, mean|x|) + 1e-30 (mean mode)."""
    ref = np.abs(want.astype(np.float64))
    if scale is not None:
        ref = np.maximum(ref, scale)
    err = np.abs(got.astype(np.float64) - want.astype(np.float64))
    bad = err > 1e-6 * ref + 1e-30
    assert not bad.any(), f"mean mismatch at {np.nonzero(bad)[0][:10]}"
