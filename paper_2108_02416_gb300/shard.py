"""The PS round split by coordinate range over several processes, one GPU each.

Rank p of P holds copies[:, :, c0_p:c1_p] (every file, every copy, a slice of
the coordinates).  The steps of Algorithm 1 then need one exchange:

  1. compare the copies of every file on the local slice (aspis_check);
  2. OR-combine the per-file mismatch words of all ranks: a pair of copies
     differs iff it differs in some slice, so the combined words are those of
     the whole vectors (Section 4's alpha_i compares whole gradients);
  3. graph, maximum cliques and selection from the combined words: the same
     deterministic result on every rank (aspis_graph, aspis_detect,
     aspis_select);
  4. aggregate the local slice (aspis_aggregate): rank p owns the output
     coordinates [c0_p, c1_p).

Splitting by file instead would need an all-to-all of copies before the
coordinate-wise median, so coordinates are the split that keeps the data
where it is.  The exchange moves f * 4 bytes per rank.

A rank that has gone away is found at the exchange by a bounded wait; the
round then reports PEER_FAILED and returns no result, it does not hang.

The step functions are passed in (``ops``), so the protocol is the same for
the device path (``DeviceOps``, through libaspis) and for any other
implementation of the five steps.
"""
from __future__ import annotations

import datetime
from dataclasses import dataclass
from typing import Any, Optional

OK = "ok"
PEER_FAILED = "peer_failed"


def shard_bounds(d: int, world: int, rank: int, align: int = 32):
    """Coordinate range [c0, c1) of `rank`: contiguous, in whole blocks of
    `align` coordinates (the aggregation tile), as even as the blocks allow.
    A rank may get an empty range when d is small."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} of {world}")
    if d < 0 or align < 1:
        raise ValueError("d >= 0 and align >= 1 required")
    blocks = (d + align - 1) // align
    b0 = blocks * rank // world
    b1 = blocks * (rank + 1) // world
    return min(d, b0 * align), min(d, b1 * align)


def or_combine(words):
    """Bitwise OR of equally shaped integer tensors."""
    out = words[0].clone()
    for x in words[1:]:
        out.bitwise_or_(x)
    return out


def _default_group_timeout(timeout_s):
    return datetime.timedelta(seconds=float(timeout_s))


def exchange_file_neq(file_neq, group=None, timeout_s: float = 30.0):
    """All ranks' mismatch words, OR-combined.  Raises PeerFailure when a
    rank does not reach the exchange within `timeout_s` (gloo: a monitored
    barrier names it; other backends rely on the process group's own
    timeout)."""
    import torch.distributed as dist

    if not dist.is_available() or not dist.is_initialized():
        return file_neq                 # one process holds every coordinate
    world = dist.get_world_size(group)
    if world == 1:
        return file_neq
    try:
        if dist.get_backend(group) == "gloo":
            dist.monitored_barrier(group, timeout=_default_group_timeout(timeout_s),
                                   wait_all_ranks=True)
        parts = [file_neq.new_empty(file_neq.shape) for _ in range(world)]
        dist.all_gather(parts, file_neq.contiguous(), group=group)
    except Exception as e:          # a dead or stuck peer surfaces as a runtime error
        raise PeerFailure(str(e)) from e
    return or_combine(parts)


class PeerFailure(RuntimeError):
    """Another rank did not take part in the exchange."""


@dataclass
class ShardResult:
    status: str
    c0: int
    c1: int
    file_neq: Any = None      # combined [f] words (ops' tensor type)
    adj: Any = None
    det: Any = None
    sel: Any = None
    out: Any = None           # aggregate of coordinates [c0, c1)
    error: Optional[str] = None


def sharded_round(local_copies, d_local: int, c0: int, ops, group=None,
                  timeout_s: float = 30.0) -> ShardResult:
    """One round on this rank's slice; see the module docstring.

    local_copies  [f][r][ld] slice of coordinates [c0, c0 + d_local)
    ops           compare(copies, d) -> words; graph(words) -> adj;
                  detect(adj) -> det; select(words, det) -> sel;
                  aggregate(copies, d, sel, det) -> out
    """
    c1 = c0 + d_local
    if d_local > 0:
        words = ops.compare(local_copies, d_local)
    else:
        words = ops.zero_words()
    try:
        words = exchange_file_neq(words, group, timeout_s)
    except PeerFailure as e:
        return ShardResult(PEER_FAILED, c0, c1, error=str(e))
    adj = ops.graph(words)
    det = ops.detect(adj)
    sel = ops.select(words, det)
    out = ops.aggregate(local_copies, d_local, sel, det) if d_local > 0 else None
    return ShardResult(OK, c0, c1, words, adj, det, sel, out)


class DeviceOps:
    """The five steps through libaspis on one device (stream-ordered)."""

    def __init__(self, a, device="cuda", mode: int = 0, stream=None):
        import torch

        from . import RoundBuffers

        self.a, self.mode, self.stream = a, mode, stream
        self.buf = RoundBuffers(a, 1, device)
        self.device = torch.device(device)

    def zero_words(self):
        import torch
        return torch.zeros(self.a.f, dtype=torch.int32, device=self.device)

    def compare(self, copies, d):
        from . import aspis_check
        aspis_check(copies, d, self.a, self.buf.file_neq, self.buf.adj, self.stream)
        return self.buf.file_neq

    def graph(self, words):
        from . import aspis_graph
        aspis_graph(words, self.a, self.buf.adj, self.stream)
        return self.buf.adj

    def detect(self, adj):
        from . import aspis_detect
        aspis_detect(adj, self.a.K, self.buf.det, self.stream)
        return self.buf.det

    def select(self, words, det):
        from . import aspis_select
        aspis_select(words, det, self.a, self.buf.sel, self.stream)
        return self.buf.sel

    def aggregate(self, copies, d, sel, det):
        import torch

        from . import aspis_aggregate
        out = torch.empty(d, dtype=torch.float32, device=self.device)
        aspis_aggregate(copies, d, self.a, sel, det, out, self.mode, self.stream)
        return out


def max_over_ranks(x: float, device=None, group=None) -> float:
    """Largest `x` over the ranks (1 rank: x itself); used for step times."""
    import torch
    import torch.distributed as dist

    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size(group) == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    return float(t.item())
