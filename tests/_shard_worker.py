"""Rank body of the coordinate-sharded round for the gloo tests: the five
steps are the oracle's (CPU), the protocol is the package's shard module."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


class OracleOps:
    def __init__(self, oa, mode=0):
        self.oa, self.mode = oa, mode

    def zero_words(self):
        import torch
        return torch.zeros(self.oa.f, dtype=torch.int32)

    def compare(self, copies, d):
        import oracle
        import torch
        return torch.from_numpy(oracle.file_agreement(copies, d).view(np.int32).copy())

    def graph(self, words):
        import oracle
        w = words.numpy().view(np.uint32)
        return oracle.graph(oracle.pair_agreement(w, self.oa), self.oa.K, self.oa.r)

    def detect(self, adj):
        import oracle
        return oracle.detect(adj, self.oa.K)

    def select(self, words, det):
        import oracle
        sel, _ = oracle.select(words.numpy().view(np.uint32), self.oa, det.clique, det.success)
        return sel

    def aggregate(self, copies, d, sel, det):
        import oracle
        return oracle.aggregate(copies, sel, self.mode, 0, d)


def run_rank(rank, world, port, cfg, d, mode, out_dir, drop_rank, timeout_s):
    import datetime

    import torch.distributed as dist

    import oracle
    import synth
    from paper_2108_02416_gb300 import shard

    dist.init_process_group("gloo", rank=rank, world_size=world,
                            init_method=f"tcp://127.0.0.1:{port}",
                            timeout=datetime.timedelta(seconds=60))
    import dataclasses
    w = dataclasses.replace(synth.CONFIGS[cfg], d=d)
    oa = oracle.assign(w.K, w.r)
    c0, c1 = shard.shard_bounds(d, world, rank)
    if rank == drop_rank:
        os._exit(0)                  # leaves before the exchange, without a word
    local = synth.build_copies_np(w, oa.file_workers, c0, c1) if c1 > c0 else \
        np.zeros((oa.f, oa.r, 0), np.float32)
    res = shard.sharded_round(local, c1 - c0, c0, OracleOps(oa, mode), timeout_s=timeout_s)
    np.savez(os.path.join(out_dir, f"rank{rank}.npz"), status=res.status, c0=c0, c1=c1,
             file_neq=(res.file_neq.numpy().view(np.uint32) if res.file_neq is not None
                       else np.zeros(0, np.uint32)),
             adj=res.adj if res.adj is not None else np.zeros(0, np.uint32),
             clique=(res.det.clique if res.det is not None else -1),
             sel=res.sel if res.sel is not None else np.zeros(0, np.int8),
             out=res.out if res.out is not None else np.zeros(0, np.float32),
             mx=shard.max_over_ranks(float(rank + 1)) if res.status == shard.OK else -1.0)
    if res.status == shard.OK:
        dist.destroy_process_group()
    os._exit(0)
