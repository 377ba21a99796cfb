"""Algorithm 3 beyond 32 workers: aspis_detect_wide against the oracle's
128-bit Bron-Kerbosch (omega, number of maximum cliques, the smallest
maximum clique, the number of maximal cliques) on random graphs across the
word boundaries, the K = 100, r = 5 attack graphs of the clique-timing
experiment (Table 5), closed-form multipartite graphs, one-sided rows, and
the node budget.  Argument errors are checked without a GPU."""
import ctypes
import random

import numpy as np
import pytest

import oracle
import synth

ap = pytest.importorskip("paper_2108_02416_gb300")


def test_wide_detection_layout_and_argument_errors():
    assert ap.WIDE_DETECTION_BYTES == 64
    P = ctypes.c_void_p
    fake = P(0x10000)
    assert ap.lib.aspis_detect_wide(fake, 0, fake, None) == ap.E_INVAL
    assert ap.lib.aspis_detect_wide(None, 10, fake, None) == ap.E_INVAL
    assert ap.lib.aspis_detect_wide(fake, 10, None, None) == ap.E_INVAL
    assert ap.lib.aspis_detect_wide(fake, 129, fake, None) == ap.E_RANGE


torch = pytest.importorskip("torch")
DEV = torch.device("cuda:0")
gpu = pytest.mark.gpu
needs_gpu = pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")


def gnp(K, p, seed):
    rnd = random.Random(seed)
    rows = [0] * K
    for a in range(K):
        for b in range(a + 1, K):
            if rnd.random() < p:
                rows[a] |= 1 << b
                rows[b] |= 1 << a
    return rows


def run_wide(rows, K, flags=0, budget=0):
    words = oracle.masks_to_words(rows, K)
    adj = torch.from_numpy(words.view(np.int32).copy()).to(DEV)
    det = ap.wide_detection_buffer(DEV, node_budget=budget, flags=flags)
    ap.aspis_detect_wide(adj, K, det)
    torch.cuda.synchronize()
    return ap.DetectionWide.from_tensor(det)


def assert_matches(rows, K, flags=0):
    want = oracle.max_cliques_wide(oracle.masks_to_words(rows, K), K)
    got = run_wide(rows, K, flags)
    assert got.status == ap.OK
    assert (got.omega, got.n_max_cliques, got.clique_mask) == (want.omega, want.n_max, want.clique)
    assert got.success == (1 if want.n_max == 1 else 0)
    if flags & ap.WIDE_ALL_MAXIMAL:
        assert got.n_maximal == want.n_maximal
    else:
        assert want.n_max <= got.n_maximal <= want.n_maximal
    return got


CASES = [(1, 0.0), (2, 1.0), (31, 0.5), (32, 0.5), (33, 0.5), (63, 0.3), (64, 0.3), (65, 0.6),
         (100, 0.2), (100, 0.45), (127, 0.1), (128, 0.3), (128, 0.02), (48, 0.85)]


@gpu
@needs_gpu
@pytest.mark.parametrize("K,p", CASES)
@pytest.mark.parametrize("flags", [0, 1])
def test_wide_random_graphs(K, p, flags):
    assert_matches(gnp(K, p, K * 7 + int(p * 100)), K, flags)


@gpu
@needs_gpu
@pytest.mark.parametrize("q", [5, 15, 25, 35, 45])
@pytest.mark.parametrize("attack", ["weak", "strong"])
@pytest.mark.parametrize("flags", [0, 1])
def test_wide_table5_graphs(q, attack, flags):
    w = synth.Workload("t5", K=100, r=5, d=1, q=q, attack=attack, seed=q)
    got = assert_matches(synth.attack_graph(w), 100, flags)
    assert got.omega == 100 - q
    assert got.n_max_cliques == (1 if attack == "weak" else 2)


@gpu
@needs_gpu
def test_wide_multipartite_closed_form():
    K = 128
    perm = list(range(K))
    random.Random(9).shuffle(perm)
    parts = [perm[3 * i: 3 * i + 3] for i in range(6)] + [[v] for v in perm[18:]]
    part_of = {v: i for i, part in enumerate(parts) for v in part}
    rows = [sum(1 << b for b in range(K) if part_of[b] != part_of[a]) for a in range(K)]
    for flags in (0, 1):
        got = assert_matches(rows, K, flags)
        assert (got.omega, got.n_max_cliques) == (K - 12, 3 ** 6)
        assert got.clique_mask == sum(1 << min(part) for part in parts)


@gpu
@needs_gpu
def test_wide_moon_moser_and_budget():
    K = 36                                   # 3^12 maximum cliques of size 12
    rows = [sum(1 << b for b in range(K) if b // 3 != a // 3) for a in range(K)]
    got = assert_matches(rows, K, ap.WIDE_ALL_MAXIMAL)
    assert got.n_max_cliques == 3 ** 12 and got.n_maximal == 3 ** 12
    small = run_wide(rows, K, budget=10)
    assert small.status == ap.E_LIMIT and small.success == 0


@gpu
@needs_gpu
def test_wide_one_sided_rows_and_self_loops():
    K = 70
    rows = gnp(K, 0.5, 3)
    rnd = random.Random(4)
    for _ in range(300):                     # drop one direction of some edges
        a, b = rnd.randrange(K), rnd.randrange(K)
        rows[a] &= ~(1 << b)
    for a in range(K):                       # self loops and bits beyond K
        rows[a] |= (1 << a) | (1 << (K + a % 50))
    assert_matches(rows, K, 0)
    assert_matches(rows, K, 1)


@gpu
@needs_gpu
def test_wide_agrees_with_narrow_detector():
    for seed in range(6):
        K = 20 + seed * 2
        rows = gnp(K, 0.6, seed)
        adj = torch.from_numpy(np.array(rows, np.uint32).view(np.int32)).to(DEV)
        det = torch.zeros(ap.DETECTION_BYTES, dtype=torch.uint8, device=DEV)
        ap.aspis_detect(adj, K, det)
        torch.cuda.synchronize()
        narrow = ap.Detection.from_tensor(det)
        wide = run_wide(rows, K)
        assert (wide.omega, wide.n_max_cliques, wide.clique_mask) == \
            (narrow.omega, narrow.n_max_cliques, narrow.clique_mask)
