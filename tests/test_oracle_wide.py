"""Pins for Algorithm 3 beyond 32 workers (oracle.max_cliques_wide, K <= 128)
and for the closed-form attack graphs of graph-only workloads
(synth.attack_graph): NetworkX enumeration, complete multipartite graphs
with a closed-form clique count, the two attacks of Section 4 on the
K = 100, r = 5 graphs of the clique-timing experiment (Table 5), and the
graph computed from actual copies for small K."""
import itertools
import random

import numpy as np
import pytest

import oracle
import synth


def rows_from_edges(K, edges):
    rows = [0] * K
    for a, b in edges:
        rows[a] |= 1 << b
        rows[b] |= 1 << a
    return rows


def gnp(K, p, seed):
    rnd = random.Random(seed)
    return rows_from_edges(K, [(a, b) for a in range(K) for b in range(a + 1, K) if rnd.random() < p])


def summary_from_cliques(cliques):
    """omega, number of maximum cliques, smallest maximum mask, number of maximal cliques"""
    masks = [sum(1 << v for v in c) for c in cliques]
    omega = max(len(c) for c in cliques)
    top = [m for m, c in zip(masks, cliques) if len(c) == omega]
    return omega, len(top), min(top), len(masks)


def check(rows, K, want):
    got = oracle.max_cliques_wide(oracle.masks_to_words(rows, K), K)
    assert (got.omega, got.n_max, got.clique, got.n_maximal) == want


@pytest.mark.parametrize("K,p,seed", [(40, 0.8, 1), (64, 0.6, 2), (100, 0.4, 3), (128, 0.3, 4),
                                      (128, 0.05, 5), (33, 0.5, 6)])
def test_wide_against_networkx(K, p, seed):
    nx = pytest.importorskip("networkx")
    rows = gnp(K, p, seed)
    g = nx.Graph()
    g.add_nodes_from(range(K))
    g.add_edges_from((a, b) for a in range(K) for b in range(a + 1, K) if (rows[a] >> b) & 1)
    check(rows, K, summary_from_cliques(list(nx.find_cliques(g))))


def test_wide_complete_multipartite_closed_form():
    # parts of sizes 3 (six of them) and 1 (the rest), spread over all four
    # words by a seeded permutation: the maximal cliques are the transversals,
    # 3^6 of them, each of size K - 12
    K = 128
    perm = list(range(K))
    random.Random(9).shuffle(perm)
    parts = [perm[3 * i: 3 * i + 3] for i in range(6)] + [[v] for v in perm[18:]]
    part_of = {v: i for i, part in enumerate(parts) for v in part}
    rows = rows_from_edges(K, [(a, b) for a in range(K) for b in range(a + 1, K)
                               if part_of[a] != part_of[b]])
    canon = sum(1 << min(part) for part in parts)
    check(rows, K, (len(parts), 3 ** 6, canon, 3 ** 6))


def test_wide_degenerate_graphs():
    check([0] * 128, 128, (1, 128, 1, 128))                        # no edges: every vertex
    full = (1 << 128) - 1
    check([full & ~(1 << j) for j in range(128)], 128, (128, 1, full, 1))
    check([0], 1, (1, 1, 1, 1))
    # one-sided rows do not make an edge; self loops and bits >= K are ignored
    rows = [(1 << 1) | (1 << 0) | (1 << 70), 0, 0]
    check(rows, 3, (1, 3, 1, 3))


def test_wide_equals_narrow_oracle_on_small_graphs():
    for seed in range(40):
        K = 5 + seed % 27
        rows = gnp(K, 0.3 + 0.5 * (seed % 3) / 2, seed)
        narrow = oracle.max_cliques_bk(np.array(rows, np.uint32), K)
        wide = oracle.max_cliques_wide(oracle.masks_to_words(rows, K), K)
        assert (wide.omega, wide.n_max, wide.clique) == (narrow.omega, narrow.n_max, narrow.clique)


@pytest.mark.parametrize("q", [5, 15, 25, 35, 45])
def test_table5_graphs_closed_form(q):
    """The K = 100, r = 5 graphs of the clique-timing experiment.  Weak attack:
    honest workers H and the adversaries A are the two maximal cliques and H is
    the unique maximum.  Optimal attack (Theorem 1): A u R and D u R, both of
    size K - q, with R the workers outside A u D."""
    K = 100
    weak = synth.Workload("t5w", K=K, r=5, d=1, q=q, attack="weak", seed=q)
    A, _ = synth.adversary_sets(weak)
    H = sum(1 << k for k in range(K) if k not in A)
    check(synth.attack_graph(weak), K, (K - q, 1, H, 2))
    strong = synth.Workload("t5s", K=K, r=5, d=1, q=q, attack="strong", seed=q)
    A, D = synth.adversary_sets(strong)
    R = sum(1 << k for k in range(K) if k not in A and k not in D)
    a_r, d_r = R | sum(1 << k for k in A), R | sum(1 << k for k in D)
    check(synth.attack_graph(strong), K, (K - q, 2, min(a_r, d_r), 2))


@pytest.mark.parametrize("K,r,q,attack", [(7, 3, 2, "weak"), (9, 3, 3, "strong"), (9, 5, 3, "strong"),
                                          (11, 5, 4, "strong"), (12, 3, 5, "strong"), (10, 3, 1, "strong"),
                                          (12, 5, 2, "strong"), (10, 5, 4, "weak")])
def test_attack_graph_matches_graph_from_copies(K, r, q, attack):
    """synth.attack_graph equals the graph the oracle computes from the
    copies themselves (file comparison, pair agreement counts, edge rule)."""
    w = synth.Workload("g", K=K, r=r, d=16, q=q, attack=attack, seed=K + q)
    a = oracle.assign(K, r)
    copies = synth.build_copies_np(w, a.file_workers)
    neq = oracle.file_agreement(copies, w.d)
    adj = oracle.graph(oracle.pair_agreement(neq, a), K, r)
    assert [int(x) for x in adj] == synth.attack_graph(w)
