"""Tables 2-4 end to end through the CUDA path: for every (K, r, attack, q)
row the round's compare, clique search and selection kernels run on
synthetic copies (weak attack: reversed gradients; optimal attack of
Theorem 1: ALIE), and the distortion fraction eps = c/f (files dropped or
represented by a distorted copy) must equal the printed value to its three
decimals; the selection must equal the oracle's, file by file."""
import math

import numpy as np
import pytest

import oracle
import synth
from conftest import read_golden

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)
ap = pytest.importorskip("paper_2108_02416_gb300")
DEV = torch.device("cuda:0")

ROWS = [r.split() for r in read_golden("epsilon_tables.txt")]


@pytest.fixture(scope="module")
def assignments():
    return {}


@pytest.mark.parametrize("row", ROWS, ids=["-".join(r[:4]) for r in ROWS])
def test_epsilon_through_kernels(row, assignments):
    K, r, attack, q, eps = int(row[0]), int(row[1]), row[2], int(row[3]), float(row[4])
    misprint = "misprint" in row
    if (K, r) not in assignments:
        assignments[(K, r)] = (ap.aspis_assign(K, r), oracle.assign(K, r))
    a, oa = assignments[(K, r)]
    w = synth.Workload("eps", K=K, r=r, d=64, q=q,
                       attack="strong" if attack == "optimal" else "weak",
                       distortion="alie" if attack == "optimal" else "reversed", seed=q)
    fw = a.file_workers()
    assert np.array_equal(fw, oa.file_workers)
    host = synth.build_copies_np(w, fw)
    copies = torch.from_numpy(host).to(DEV)
    buf = ap.RoundBuffers(a, w.d, DEV)
    ap.aspis_check(copies, w.d, a, buf.file_neq, buf.adj)
    ap.aspis_detect(buf.adj, K, buf.det)
    ap.aspis_select(buf.file_neq, buf.det, a, buf.sel)
    torch.cuda.synchronize()
    sel = buf.sel.cpu().numpy()
    want = oracle.run_round(host, oa, w.d, aggregate_out=False)
    assert np.array_equal(sel, want.sel)
    mask = synth.corrupted_mask(w, fw)
    c = sum(1 for i in range(a.f) if sel[i] < 0 or mask[i, sel[i]])
    if misprint:
        assert c == math.comb(q, r) == 0 and eps > 0
    else:
        assert abs(c / a.f - eps) <= 0.0005 + 1e-12, (K, r, attack, q, c / a.f, eps)
