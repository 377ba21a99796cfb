"""Coordinate-sharded round on CPU ranks (gloo, world size 2): the package's
protocol with the oracle's steps must reproduce the unsharded oracle round;
a rank that leaves before the exchange must give PEER_FAILED, not a hang."""
import multiprocessing as mp
import os
import socket

import numpy as np
import pytest

import oracle
import synth

torch = pytest.importorskip("torch")
shard = pytest.importorskip("paper_2108_02416_gb300.shard")


def test_shard_bounds_cover_in_aligned_blocks():
    for d in (0, 1, 31, 32, 33, 1000, 4099, 11173962):
        for world in (1, 2, 3, 4, 8):
            rng = [shard.shard_bounds(d, world, p) for p in range(world)]
            assert rng[0][0] == 0 and rng[-1][1] == d
            for (a0, a1), (b0, b1) in zip(rng, rng[1:]):
                assert a1 == b0 and a0 <= a1
            for c0, c1 in rng:
                assert c0 % 32 == 0 and (c1 % 32 == 0 or c1 == d)
            sizes = [c1 - c0 for c0, c1 in rng]
            assert max(sizes) - min(sizes) <= 32 or d < 32 * world


def test_or_combine():
    a = torch.tensor([1, 0, 4], dtype=torch.int32)
    b = torch.tensor([2, 0, 4], dtype=torch.int32)
    assert shard.or_combine([a, b]).tolist() == [3, 0, 4]


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _run(cfg, d, mode, tmp_path, drop_rank=-1, world=2, timeout_s=20.0):
    from _shard_worker import run_rank
    ctx = mp.get_context("spawn")
    port = _free_port()
    procs = [ctx.Process(target=run_rank, args=(p, world, port, cfg, d, mode, str(tmp_path),
                                                drop_rank, timeout_s)) for p in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    alive = [p for p in procs if p.is_alive()]
    for p in alive:
        p.kill()
        p.join()
    assert not alive, "a rank did not finish"
    return [dict(np.load(os.path.join(tmp_path, f"rank{p}.npz"))) if p != drop_rank else None
            for p in range(world)]


@pytest.mark.parametrize("cfg,d,mode", [
    ("k7_r3_d4096_alie", 4099, 0),             # Case 1: unique maximum clique
    ("k15_r3_d11m_strong_alie", 2000, 0),      # Case 2: majority + median
    ("k15_r3_d1m_weak_reversed", 1000, 1),     # Case 1, mean
])
def test_sharded_round_matches_unsharded(cfg, d, mode, tmp_path):
    import dataclasses
    res = _run(cfg, d, mode, tmp_path)
    w = dataclasses.replace(synth.CONFIGS[cfg], d=d)
    oa = oracle.assign(w.K, w.r)
    full = oracle.run_round(synth.build_copies_np(w, oa.file_workers, 0, d), oa, d, mode)
    for r in res:
        assert str(r["status"]) == shard.OK
        assert np.array_equal(r["file_neq"], full.file_neq)
        assert np.array_equal(r["adj"], full.adj)
        assert int(r["clique"]) == full.det.clique
        assert np.array_equal(r["sel"], full.sel)
        assert float(r["mx"]) == 2.0                   # max over the two ranks
    out = np.concatenate([r["out"] for r in res])
    assert np.array_equal(out.view(np.uint32), full.out.view(np.uint32))


def test_dropped_rank_reports_peer_failure(tmp_path):
    import time
    t0 = time.time()
    res = _run("k7_r3_d4096_alie", 512, 0, tmp_path, drop_rank=1, timeout_s=5.0)
    assert str(res[0]["status"]) == shard.PEER_FAILED
    assert res[0]["out"].size == 0
    assert time.time() - t0 < 100
