"""Property tier: random rounds through the C ABI against the oracle, bit for
bit (mismatch words, graph, clique, selection, lower median).  Random K <= 12,
r in 2..5, d not a multiple of 4; a random adversary set whose members
corrupt random subsets of their files (many or few) or, as in Theorem 1,
exactly the files inside A u D that hold r' adversaries; sometimes colluding
(one shared distorted vector) and sometimes not (each its own), so Case 1,
Case 2, the plurality rule and dropped files all occur.  Honest copies of a file are
identical, so the honest workers always form a clique (checked)."""
import numpy as np
import pytest

import oracle
from _gpu_round import assert_round_matches, gpu_round

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)
ap = pytest.importorskip("paper_2108_02416_gb300")
DEV = torch.device("cuda:0")


def random_round(seed):
    rng = np.random.default_rng(seed)
    r = int(rng.integers(2, 6))
    K = int(rng.integers(max(r + 1, 4), 13))
    d = int(rng.integers(9, 400))
    if d % 4 == 0:
        d += 1
    q = int(rng.integers(0, (K - 1) // 2 + 1))
    A = set(rng.choice(K, size=q, replace=False).tolist()) if q else set()
    oa = oracle.assign(K, r)
    f = oa.f
    g = rng.standard_normal((f, d)).astype(np.float32)
    copies = np.repeat(g[:, None, :], r, axis=1).copy()
    collude = bool(rng.integers(0, 2))
    shared = rng.standard_normal(d).astype(np.float32)
    mode = seed % 3                  # 0: random files, 1: few files, 2: Theorem 1 style
    p = float(rng.uniform(0.2, 1.0)) if mode == 0 else float(rng.uniform(0.01, 0.1))
    rest = [j for j in range(K) if j not in A]
    D = set(rng.choice(rest, size=min(q, len(rest)), replace=False).tolist()) if q else set()
    rp = (r + 1) // 2
    for i in range(f):
        ws = [int(x) for x in oa.file_workers[i]]
        target = all(x in A or x in D for x in ws) and sum(x in A for x in ws) >= rp
        for s in range(r):
            wk = ws[s]
            hit = target if mode == 2 else rng.random() < p
            if wk in A and hit:
                if collude:
                    copies[i, s] = shared
                else:
                    copies[i, s] = rng.standard_normal(d).astype(np.float32)
                    # a corruption that differs only in the last coordinate
                    if rng.random() < 0.2:
                        copies[i, s] = g[i]
                        copies[i, s, d - 1] = np.nextafter(g[i, d - 1], np.float32(np.inf))
    return K, r, d, A, oa, copies


@pytest.mark.parametrize("seed", range(24))
def test_random_round(seed):
    K, r, d, A, oa, host = random_round(seed)
    want = oracle.run_round(host, oa, d, 0)
    honest = sum(1 << j for j in range(K) if j not in A)
    for j in range(K):                       # honest workers form a clique
        if j not in A:
            assert (int(want.adj[j]) | (1 << j)) & honest == honest
    a = ap.aspis_assign(K, r)
    buf = gpu_round(ap, torch, torch.from_numpy(host).to(DEV), d, a)
    if want.n_sel == 0:
        assert buf.detection().status == ap.E_EMPTY
        return
    assert_round_matches(ap, buf, want)
