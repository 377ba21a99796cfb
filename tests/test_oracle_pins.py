"""Pins for the CPU oracle: each test checks the oracle against something the
paper or mathematics fixes independently of the oracle's own code (printed
values, closed forms, brute force, NetworkX, sorting)."""
import itertools
import math
import random
import statistics
import struct

import numpy as np
import pytest

import oracle
import synth
from conftest import read_golden


def bits_to_f32(u):
    return struct.unpack("<f", struct.pack("<I", u))[0]


def f32_bits(x):
    return struct.unpack("<I", struct.pack("<f", x))[0]


# ------------------------------------------------------------ Algorithm 2


def test_assign_counts_golden():
    for row in read_golden("assignment_counts.txt"):
        K, r, f, l, share = (int(x) for x in row.split()[:5])
        a = oracle.assign(K, r)
        assert (a.f, a.l) == (f, l)
        sets = [set(np.nonzero(np.isin(np.arange(a.f), a.worker_files[j]))[0])
                for j in range(K)]
        for j1 in range(K):
            assert len(sets[j1]) == l
            for j2 in range(j1 + 1, K):
                assert len(sets[j1] & sets[j2]) == share


@pytest.mark.parametrize("K,r", [(2, 2), (5, 2), (6, 3), (7, 3), (8, 8), (9, 4), (12, 5),
                                 (15, 3), (15, 5), (21, 3), (31, 3), (20, 8)])
def test_assign_matches_lexicographic_enumeration(K, r):
    a = oracle.assign(K, r)
    expect = list(itertools.combinations(range(K), r))
    assert a.f == len(expect) == math.comb(K, r)
    assert a.l == math.comb(K - 1, r - 1)
    assert [tuple(int(x) for x in row) for row in a.file_workers] == expect
    # worker_files lists each worker's files ascending; slot_of is its slot there
    for j in range(K):
        files = a.worker_files[j]
        assert list(files) == sorted(files)
        for k, i in enumerate(files):
            assert a.file_workers[i][a.slot_of[j][k]] == j


def test_example1_file0():
    a = oracle.assign(7, 3)
    assert tuple(a.file_workers[0]) == (0, 1, 2)      # S_0 = {U1,U2,U3} <-> B_{t,0}


def test_assign_rejects_r1():
    with pytest.raises(ValueError):
        oracle.assign(7, 1)


# ------------------------------------------------------ per-file agreement


def pair_index(r, s, t):
    return [(a, b) for a in range(r) for b in range(a + 1, r)].index((s, t))


@pytest.mark.parametrize("r", [2, 3, 5, 8])
def test_file_agreement_single_bit_flips(r):
    d, ld = 37, 40
    f = 6
    rng = np.random.default_rng(r)
    base = rng.standard_normal((f, d)).astype(np.float32)
    copies = np.repeat(base[:, None, :], r, axis=1)
    copies = np.concatenate([copies, np.zeros((f, r, ld - d), np.float32)], axis=2)
    # file 1: flip lowest mantissa bit of coordinate 0 in slot r-1
    # file 2: flip sign bit at the last coordinate in slot 0
    # file 3: flip at an odd coordinate in slot 1
    # file 4: padding differs only beyond d -> equal
    # file 5: +0 vs -0 at coordinate 5 in slot 0
    u = copies.view(np.uint32)
    u[1, r - 1, 0] ^= 1
    u[2, 0, d - 1] ^= 0x80000000
    u[3, 1, 13] ^= 0x10
    u[4, 0, d:] = 0xdeadbeef
    copies[5, :, 5] = 0.0
    u[5, 0, 5] = 0x80000000
    neq = oracle.file_agreement(copies, d)
    full = (1 << (r * (r - 1) // 2)) - 1

    def expect_one_slot_differs(s):
        w = 0
        for t in range(r):
            if t != s:
                w |= 1 << pair_index(r, min(s, t), max(s, t))
        return w

    assert neq[0] == 0
    assert neq[1] == expect_one_slot_differs(r - 1)
    assert neq[2] == expect_one_slot_differs(0)
    assert neq[3] == expect_one_slot_differs(1)
    assert neq[4] == 0
    assert neq[5] == expect_one_slot_differs(0)
    assert all(int(w) & ~full == 0 for w in neq)


def test_file_agreement_nan_payloads():
    d = 4
    copies = np.zeros((2, 3, d), np.float32)
    u = copies.view(np.uint32)
    u[0, :, 2] = 0x7fc00000           # identical NaNs: equal bit patterns
    u[1, :, 2] = 0x7fc00000
    u[1, 2, 2] = 0x7fc00001           # different payload: not equal
    neq = oracle.file_agreement(copies)
    assert neq[0] == 0
    assert neq[1] == (1 << pair_index(3, 0, 2)) | (1 << pair_index(3, 1, 2))


# ------------------------------------------------ graph and Figure 3 cases


def _round_for(K, r, d, corrupt):
    """copies for workload where corrupt(i, workers) -> list of per-slot
    corrupted values (None = honest)."""
    a = oracle.assign(K, r)
    rng = np.random.default_rng(K * 100 + r)
    g = rng.standard_normal((a.f, d)).astype(np.float32)
    copies = np.repeat(g[:, None, :], r, axis=1).copy()
    for i in range(a.f):
        vals = corrupt(i, [int(x) for x in a.file_workers[i]])
        for s, v in enumerate(vals):
            if v is not None:
                copies[i, s] = v
    return a, copies


def test_figure3_graphs():
    rows = {r.split()[0]: r.split() for r in read_golden("figure3_k7.txt")}
    A = {0, 1, 2}
    bad = np.full(8, 7.0, np.float32)
    # weak: every copy held by an adversary is distorted (colluding: same value)
    a, copies = _round_for(7, 3, 8, lambda i, ws: [bad if w in A else None for w in ws])
    res = oracle.run_round(copies, a)
    om, nm, masks = int(rows["weak"][1]), int(rows["weak"][2]), [int(x) for x in rows["weak"][3].split(",")]
    assert (res.det.omega, res.det.n_max, res.det.clique) == (om, nm, masks[0])
    for det in (oracle.max_cliques_brute(res.adj, 7), oracle.max_cliques_bk(res.adj, 7)):
        assert (det.omega, det.n_max, det.clique) == (om, nm, masks[0])
    # optimal: all adversaries disagree with D = {U4,U5,U6} (Theorem 1 construction)
    D = {3, 4, 5}

    def strong(i, ws):
        inside = all(w in A | D for w in ws)
        n_adv = sum(w in A for w in ws)
        return [bad if (w in A and inside and n_adv >= 2) else None for w in ws]

    a, copies = _round_for(7, 3, 8, strong)
    res = oracle.run_round(copies, a)
    om, nm, masks = int(rows["optimal"][1]), int(rows["optimal"][2]), [int(x) for x in rows["optimal"][3].split(",")]
    assert (res.det.omega, res.det.n_max, res.det.clique) == (om, nm, min(masks))
    nx = pytest.importorskip("networkx")
    G = nx.Graph()
    G.add_nodes_from(range(7))
    G.add_edges_from((j, k) for j in range(7) for k in range(7) if (int(res.adj[j]) >> k) & 1)
    found = sorted(sum(1 << v for v in c) for c in nx.find_cliques(G) if len(c) == om)
    assert found == masks


def test_graph_edge_rule_one_shared_file():
    """A pair that disagrees on exactly one of its C(K-2,r-2) shared files has
    no edge; every other pair keeps its edge (edge iff alpha = C(K-2,r-2))."""
    K, r = 8, 3
    a = oracle.assign(K, r)
    copies = np.zeros((a.f, r, 3), np.float32)
    copies[:] = np.arange(a.f, dtype=np.float32)[:, None, None]
    i = next(i for i in range(a.f) if tuple(a.file_workers[i]) == (2, 5, 7))
    copies[i, 1, 2] = -1.0        # worker 5 disagrees with 2 and 7 on this file only
    fneq = oracle.file_agreement(copies)
    alpha = oracle.pair_agreement(fneq, a)
    share = math.comb(K - 2, r - 2)
    assert alpha[5, 2] == alpha[5, 7] == share - 1
    adj = oracle.graph(alpha, K, r)
    for j in range(K):
        for k in range(K):
            has = (int(adj[j]) >> k) & 1
            broken = {j, k} in ({2, 5}, {5, 7})
            assert has == (j != k and not broken)


# ------------------------------------------------------ maximum cliques


def py_max_cliques(adj, K):
    """Brute force written in the test: every subset, check all pairs."""
    best, cnt, first = 0, 0, 0
    for size in range(K, 0, -1):
        for sub in itertools.combinations(range(K), size):
            if all((int(adj[u]) >> v) & 1 for u, v in itertools.combinations(sub, 2)):
                m = sum(1 << v for v in sub)
                if size > best:
                    best, cnt, first = size, 1, m
                elif size == best:
                    cnt += 1
                    first = min(first, m)
        if best:
            break
    return best, cnt, first


def random_graph(K, p, rng):
    adj = np.zeros(K, np.uint32)
    for j in range(K):
        for k in range(j + 1, K):
            if rng.random() < p:
                adj[j] |= np.uint32(1 << k)
                adj[k] |= np.uint32(1 << j)
    return adj


def test_cliques_exhaustive_small():
    for K in range(1, 6):
        pairs = list(itertools.combinations(range(K), 2))
        for e in range(1 << len(pairs)):
            adj = np.zeros(K, np.uint32)
            for b, (u, v) in enumerate(pairs):
                if (e >> b) & 1:
                    adj[u] |= np.uint32(1 << v)
                    adj[v] |= np.uint32(1 << u)
            want = py_max_cliques(adj, K)
            for det in (oracle.max_cliques_brute(adj, K), oracle.max_cliques_bk(adj, K)):
                assert (det.omega, det.n_max, det.clique) == want


def test_cliques_random_vs_networkx():
    nx = pytest.importorskip("networkx")
    rng = random.Random(7)
    for trial in range(300):
        K = rng.randint(2, 20)
        p = rng.choice([0.1, 0.3, 0.5, 0.7, 0.9, 0.97])
        adj = random_graph(K, p, rng)
        G = nx.Graph()
        G.add_nodes_from(range(K))
        G.add_edges_from((j, k) for j in range(K) for k in range(j + 1, K) if (int(adj[j]) >> k) & 1)
        cl = list(nx.find_cliques(G))
        om = max(len(c) for c in cl)
        maxs = [sum(1 << v for v in c) for c in cl if len(c) == om]
        want = (om, len(maxs), min(maxs))
        assert (lambda d: (d.omega, d.n_max, d.clique))(oracle.max_cliques_bk(adj, K)) == want
        if K <= 16:
            assert (lambda d: (d.omega, d.n_max, d.clique))(oracle.max_cliques_brute(adj, K)) == want


@pytest.mark.parametrize("parts", [1, 2, 4, 7, 10])
def test_cliques_moon_moser(parts):
    """Complete multipartite graph with parts of 3: 3^parts maximum cliques,
    each of size parts; the smallest mask takes vertex 0 of every part."""
    K = 3 * parts
    adj = np.zeros(K, np.uint32)
    for j in range(K):
        for k in range(K):
            if j // 3 != k // 3:
                adj[j] |= np.uint32(1 << k)
    det = oracle.max_cliques_bk(adj, K)
    assert det.omega == parts
    assert det.n_max == 3 ** parts
    assert det.clique == sum(1 << (3 * p) for p in range(parts))


def test_cliques_degenerate():
    for K in (1, 2, 9, 31, 32):
        empty = np.zeros(K, np.uint32)
        d = oracle.max_cliques_bk(empty, K)
        assert (d.omega, d.n_max, d.clique) == (1, K, 1)
        full = np.array([((1 << K) - 1) & ~(1 << j) & 0xffffffff for j in range(K)], np.uint32)
        d = oracle.max_cliques_bk(full, K)
        assert (d.omega, d.n_max, d.clique) == (K, 1, (1 << K) - 1)


# ------------------------------------------------------------ selection


def _one_file_select(r, classes, success=False, clique=0, workers=None):
    """classes: class label per slot (equal labels = bitwise-equal copies)."""
    w = 0
    for s in range(r):
        for t in range(s + 1, r):
            if classes[s] != classes[t]:
                w |= 1 << pair_index(r, s, t)
    a = oracle.Assignment(K=max(8, r), r=r, f=1, l=0,
                          file_workers=np.array([workers or list(range(r))], np.uint8),
                          worker_files=np.zeros((1, 1), np.int32), slot_of=np.zeros((1, 1), np.uint8))
    sel, n = oracle.select(np.array([w], np.uint32), a, clique, success)
    return int(sel[0]), n


def test_select_majority_cases():
    assert _one_file_select(3, [0, 0, 1]) == (0, 1)
    assert _one_file_select(3, [1, 0, 0]) == (1, 1)
    assert _one_file_select(3, [0, 1, 0]) == (0, 1)
    assert _one_file_select(5, [0, 1, 0, 1, 0]) == (0, 1)
    assert _one_file_select(5, [1, 0, 0, 1, 0]) == (1, 1)       # majority {1,2,4}
    assert _one_file_select(3, [0, 1, 2]) == (0, 1)             # no majority: lowest slot
    assert _one_file_select(4, [0, 1, 1, 0]) == (0, 1)          # tie 2-2: class of slot 0
    assert _one_file_select(4, [0, 1, 1, 2]) == (1, 1)          # plurality {1,2}
    assert _one_file_select(8, [3, 3, 1, 1, 1, 2, 2, 2]) == (2, 1)


def test_select_case1():
    # workers (4, 6, 9); clique holds 6 and 9 -> lowest slot in H is 1
    assert _one_file_select(3, [0, 0, 0], True, (1 << 6) | (1 << 9), [4, 6, 9]) == (1, 1)
    assert _one_file_select(3, [0, 1, 2], True, 1 << 9, [4, 6, 9]) == (2, 1)
    assert _one_file_select(3, [0, 0, 0], True, 1 << 5, [4, 6, 9]) == (-1, 0)   # dropped


# -------------------------------------- end-to-end pins from Sections 4-5


def _copies_for(w, a, d=5):
    w = synth.Workload(**{**w.__dict__, "d": d})
    return w, synth.build_copies_np(w, a.file_workers)


@pytest.mark.parametrize("K,r,q", [(7, 3, 3), (15, 3, 3), (15, 3, 6), (15, 5, 4), (21, 3, 5)])
def test_weak_attack_detected(K, r, q):
    """Section 4.1: adversaries are excluded, H is the unique maximum clique,
    and only the C(q,r) files held entirely by adversaries are lost."""
    a = oracle.assign(K, r)
    w = synth.Workload("t", K=K, r=r, d=5, q=q, attack="weak", distortion="reversed", seed=K + q)
    w, copies = _copies_for(w, a)
    A, _ = synth.adversary_sets(w)
    res = oracle.run_round(copies, a)
    H = sum(1 << j for j in range(K) if j not in A)
    assert res.det.n_max == 1 and res.det.clique == H and res.det.omega == K - q
    dropped = [i for i in range(a.f) if res.sel[i] < 0]
    assert len(dropped) == math.comb(q, r)
    assert all(set(int(x) for x in a.file_workers[i]) <= set(A) for i in dropped)
    assert res.n_sel == a.f - math.comb(q, r)
    mask = synth.corrupted_mask(w, a.file_workers)
    assert not any(mask[i, res.sel[i]] for i in range(a.f) if res.sel[i] >= 0)


@pytest.mark.parametrize("K,r,q", [(7, 3, 3), (15, 3, 2), (15, 3, 3), (15, 3, 7), (21, 3, 5),
                                   (15, 5, 4), (13, 5, 6)])
def test_optimal_attack_theorem1(K, r, q):
    """Theorem 1: two maximum cliques of size K-q, detection fails, and the
    majority vote is corrupted on exactly (1/2) C(2q, r) files."""
    a = oracle.assign(K, r)
    w = synth.Workload("t", K=K, r=r, d=5, q=q, attack="strong", distortion="alie", seed=K * q)
    w, copies = _copies_for(w, a)
    res = oracle.run_round(copies, a)
    assert res.det.n_max == 2 and res.det.omega == K - q and not res.det.success
    mask = synth.corrupted_mask(w, a.file_workers)
    c = sum(bool(mask[i, res.sel[i]]) for i in range(a.f))
    assert 2 * c == math.comb(2 * q, r)
    assert res.n_sel == a.f


def test_epsilon_tables_golden():
    """Tables 2-4: eps^Aspis = c/f for the weak and optimal attacks, end to
    end through the oracle (rounded to the paper's three decimals)."""
    cache = {}
    for row in read_golden("epsilon_tables.txt"):
        parts = row.split()
        K, r, attack, q, eps = int(parts[0]), int(parts[1]), parts[2], int(parts[3]), float(parts[4])
        misprint = "misprint" in parts
        a = cache.setdefault((K, r), oracle.assign(K, r))
        w = synth.Workload("t", K=K, r=r, d=2, q=q,
                           attack="strong" if attack == "optimal" else "weak",
                           distortion="alie" if attack == "optimal" else "reversed", seed=q)
        copies = synth.build_copies_np(w, a.file_workers)
        res = oracle.run_round(copies, a, aggregate_out=False)
        mask = synth.corrupted_mask(w, a.file_workers)
        c = sum(1 for i in range(a.f) if res.sel[i] < 0 or mask[i, res.sel[i]])
        got = c / a.f
        if misprint:
            assert c == math.comb(q, r) == 0 and eps > 0
        else:
            assert abs(got - eps) <= 0.0005 + 1e-12, (K, attack, q, got, eps)


def test_honest_workers_form_clique_random_adversaries():
    """Section 4: honest copies are identical, so H is always a clique, whatever
    the adversaries return."""
    rng = random.Random(3)
    for trial in range(40):
        K = rng.randint(4, 12)
        r = rng.randint(2, min(5, K))
        q = rng.randint(0, (K - 1) // 2)
        A = set(rng.sample(range(K), q))
        a = oracle.assign(K, r)

        def corrupt(i, ws):
            return [np.float32([rng.choice([1.0, 2.0, 3.0])] * 3) if (w in A and rng.random() < 0.5)
                    else None for w in ws]

        a, copies = _round_for(K, r, 3, corrupt)
        res = oracle.run_round(copies, a, aggregate_out=False)
        H = [j for j in range(K) if j not in A]
        for j in H:
            for k in H:
                if j != k:
                    assert (int(res.adj[j]) >> k) & 1
        assert res.det.omega >= K - q


# -------------------------------------------------- coordinate-wise median


def test_median_total_order_golden():
    for row in read_golden("median_total_order.txt"):
        ins, exp = row.split(";")
        vals = np.array([int(x, 16) for x in ins.strip().split(",")], np.uint32).view(np.float32)
        out = oracle.lower_median(vals[:, None])
        assert int(out.view(np.uint32)[0]) == int(exp.strip(), 16), row


def test_median_matches_statistics_median_low():
    rng = random.Random(11)
    for trial in range(200):
        n = rng.randint(1, 60)
        m = rng.randint(1, 5)
        vals = np.array([[rng.uniform(-5, 5) for _ in range(m)] for _ in range(n)], np.float32)
        vals[vals == 0] = 1.0
        out = oracle.lower_median(vals)
        for c in range(m):
            assert out[c] == statistics.median_low([float(x) for x in vals[:, c]])


def test_aggregate_uses_selected_copies_only():
    a = oracle.assign(6, 3)
    rng = np.random.default_rng(5)
    copies = rng.standard_normal((a.f, 3, 9)).astype(np.float32)
    sel = rng.integers(-1, 3, a.f).astype(np.int8)
    out = oracle.aggregate(copies, sel, 0, 0, 7)
    rows = np.array([copies[i, sel[i], :7] for i in range(a.f) if sel[i] >= 0])
    want = np.sort(rows, axis=0)[(len(rows) - 1) // 2]
    assert np.array_equal(out, want)
    mean = oracle.aggregate(copies, sel, 1, 2, 9)
    for c in range(2, 9):
        exact = math.fsum(float(x) for x in copies[[i for i in range(a.f) if sel[i] >= 0],
                                                     sel[sel >= 0], c]) / len(rows)
        assert abs(float(mean[c - 2]) - exact) <= 2 ** -23 * abs(exact) + 1e-30


def test_aggregate_empty_rejected():
    copies = np.zeros((3, 2, 4), np.float32)
    with pytest.raises(ValueError):
        oracle.aggregate(copies, np.full(3, -1, np.int8))


def test_mean_against_fsum():
    rng = random.Random(2)
    vals = np.array([[rng.gauss(0, 1) * 10 ** rng.randint(-3, 3) for _ in range(4)]
                     for _ in range(301)], np.float32)
    out = oracle.mean(vals)
    for c in range(4):
        exact = math.fsum(float(x) for x in vals[:, c]) / 301
        assert abs(float(out[c]) - exact) <= 2 ** -24 * abs(exact) * 1.0001 + 1e-30


def test_config1_end_to_end_shape():
    """K=7, r=3, adversaries 0 and 1 replace every copy with ALIE: detection
    succeeds with H = {2..6} and all 35 files keep an honest copy."""
    w = synth.CONFIGS["k7_r3_d4096_alie"]
    a = oracle.assign(w.K, w.r)
    copies = synth.build_copies_np(w, a.file_workers)
    res = oracle.run_round(copies, a, w.d)
    assert res.det.success and res.det.clique == 0b1111100 and res.n_sel == 35
    assert int(res.adj[0]) == 0b10 and int(res.adj[1]) == 0b01
    # median output is one of the selected values at each coordinate
    chosen = np.array([copies[i, res.sel[i], : w.d] for i in range(a.f)])
    assert all(res.out[c] in chosen[:, c] for c in range(0, w.d, 97))
