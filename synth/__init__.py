"""Seeded synthetic inputs for the Aspis detection-and-aggregation step.

This module is shared by the tests, the benchmark and the oracle's callers.  It
holds none of the method's arithmetic: it draws honest file gradients, picks the
adversaries and writes the copies each worker returns, given the file -> worker
table (which the caller obtains from the assignment it is testing).

Random numbers come from one counter-based generator, SplitMix64's output
function (Steele, Lea & Flood, "Fast splittable pseudorandom number
generators", OOPSLA 2014), keyed by (seed, stream, index).  A standard normal
is approximated by the Irwin-Hall sum of twelve 32-bit uniforms minus 6; every
step is exact integer or exact double arithmetic up to one final rounding, so
the numpy and the torch (CPU or CUDA) backends produce identical bits.

Workload recipe (the paper trains ResNet-18 on CIFAR-10 with K = 15 / 21
workers and r = 3; synthetic vectors stand in for the gradients):
  b[c]   = 0.01  * z_b[c]                (one shared "batch gradient" per round)
  n_f[c] = 0.001 * z_f[c]                (per-file noise)
  g_f[c] = fp32(b[c] + n_f[c])           (all honest copies of file f are g_f)
Distortions (Section 6.1): ALIE fp32(mean_f g - z * std_f g) (population std,
double, file order); reversed gradient fp32(-c * g_f); Fall of Empires (inner
product manipulation) fp32(-z * mean_f g).  Colluding adversaries return
identical corrupted vectors.  For the variant with copies that are not
bit-identical, copy_noise > 0 gives honest copy (i, s) the value
fp32(g_i + copy_noise * z_{i,s}) instead of g_i.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Sequence

import numpy as np

_M64 = (1 << 64) - 1
PHI = 0x9E3779B97F4A7C15
C1 = 0xBF58476D1CE4E5B9
C2 = 0x94D049BB133111EB

STREAM_B = 0
STREAM_PERM = 1
STREAM_FILE0 = 16
STREAM_COPY0 = 1 << 40          # + 8 i + s: per-copy noise of honest copies


def _mix64_int(z: int) -> int:
    z &= _M64
    z = ((z ^ (z >> 30)) * C1) & _M64
    z = ((z ^ (z >> 27)) * C2) & _M64
    return z ^ (z >> 31)


def stream_key(seed: int, stream: int) -> int:
    """64-bit key of one random stream."""
    k0 = _mix64_int((seed * PHI + 1) & _M64)
    return _mix64_int(k0 ^ ((stream * PHI) & _M64))


def _to_signed(x: int) -> int:
    return x - (1 << 64) if x >= (1 << 63) else x


# ------------------------------------------------------------------ numpy


def _mix64_np(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * np.uint64(C1)
    z = (z ^ (z >> np.uint64(27))) * np.uint64(C2)
    return z ^ (z >> np.uint64(31))


def normal_np(seed: int, stream: int, c0: int, c1: int) -> np.ndarray:
    """Irwin-Hall standard normals for indices [c0, c1) of one stream (float64)."""
    key = np.uint64(stream_key(seed, stream))
    idx = np.arange(c0, c1, dtype=np.uint64)
    acc = np.zeros(c1 - c0, np.uint64)
    with np.errstate(over="ignore"):
        for k in range(6):
            x = _mix64_np(key + (idx * np.uint64(6) + np.uint64(k + 1)) * np.uint64(PHI))
            acc += (x & np.uint64(0xFFFFFFFF)) + (x >> np.uint64(32))
    return acc.astype(np.float64) * (2.0 ** -32) - 6.0


def honest_np(seed: int, i: int, c0: int, c1: int, b: np.ndarray | None = None) -> np.ndarray:
    """g_i[c0:c1] as float32."""
    if b is None:
        b = 0.01 * normal_np(seed, STREAM_B, c0, c1)
    n = 0.001 * normal_np(seed, STREAM_FILE0 + i, c0, c1)
    return (b + n).astype(np.float32)


# ------------------------------------------------------------------ torch


def _mix64_torch(z):
    import torch  # noqa: F401

    def lsr(x, s):
        return (x >> s) & ((1 << (64 - s)) - 1)

    z = (z ^ lsr(z, 30)) * _to_signed(C1)
    z = (z ^ lsr(z, 27)) * _to_signed(C2)
    return z ^ lsr(z, 31)


def normal_torch(seed: int, stream: int, c0: int, c1: int, device):
    """Same numbers as :func:`normal_np`, computed with torch int64 ops."""
    import torch
    key = _to_signed(stream_key(seed, stream))
    idx = torch.arange(c0, c1, dtype=torch.int64, device=device)
    acc = torch.zeros(c1 - c0, dtype=torch.int64, device=device)
    for k in range(6):
        x = _mix64_torch(key + (idx * 6 + (k + 1)) * _to_signed(PHI))
        acc += (x & 0xFFFFFFFF) + ((x >> 32) & 0xFFFFFFFF)
    return acc.to(torch.float64) * (2.0 ** -32) - 6.0


def honest_torch(seed: int, i: int, c0: int, c1: int, device, b=None):
    if b is None:
        b = 0.01 * normal_torch(seed, STREAM_B, c0, c1, device)
    n = 0.001 * normal_torch(seed, STREAM_FILE0 + i, c0, c1, device)
    return (b + n).to(__import__("torch").float32)


# --------------------------------------------------------------- workloads


@dataclass
class Workload:
    """One round's synthetic workload.

    attack:
      "none"          every copy honest
      "all_alie"      listed adversaries replace every copy with the ALIE vector
      "weak"          adversaries (random by seed) corrupt every copy they hold
      "strong"        optimal attack of Theorem 1: A and a disagreement set D
                      (both random by seed); an adversary corrupts its copy of
                      file F iff F is inside A u D and |F n A| >= r' = (r+1)/2
    distortion: "alie" (z), "foe" (z = the Fall-of-Empires epsilon) or
      "reversed" (scale)
    copy_noise: std of the per-copy noise of honest copies (0 = bit-identical)
    """
    name: str
    K: int
    r: int
    d: int
    q: int = 0
    attack: str = "none"
    distortion: str = "alie"
    z: float = 1.0
    scale: float = 10.0
    seed: int = 0
    adversaries: Sequence[int] | None = None
    ld_align: int = 32
    copy_noise: float = 0.0
    extra: dict = field(default_factory=dict)

    @property
    def ld(self) -> int:
        a = self.ld_align
        return (self.d + a - 1) // a * a

    @property
    def f(self) -> int:
        from math import comb
        return comb(self.K, self.r)


def worker_permutation(seed: int, K: int) -> list[int]:
    key = stream_key(seed, STREAM_PERM)
    h = [_mix64_int(key + (j + 1) * PHI) for j in range(K)]
    return sorted(range(K), key=lambda j: (h[j], j))


def adversary_sets(w: Workload) -> tuple[list[int], list[int]]:
    """(A, D): the adversaries and, for the strong attack, the honest workers
    they all disagree with."""
    if w.attack == "none" or w.q == 0:
        return [], []
    if w.adversaries is not None:
        return sorted(w.adversaries), []
    perm = worker_permutation(w.seed, w.K)
    A = sorted(perm[: w.q])
    D = sorted(perm[w.q: 2 * w.q]) if w.attack == "strong" else []
    return A, D


def corrupted_mask(w: Workload, file_workers: np.ndarray) -> np.ndarray:
    """bool [f, r]: True where the returned copy is adversarial."""
    A, D = adversary_sets(w)
    Aset, ADset = set(A), set(A) | set(D)
    fw = np.asarray(file_workers)
    f, r = fw.shape
    mask = np.zeros((f, r), bool)
    if not A:
        return mask
    rp = (w.r + 1) // 2
    for i in range(f):
        ws = [int(x) for x in fw[i]]
        if w.attack in ("all_alie", "weak"):
            mask[i] = [x in Aset for x in ws]
        elif w.attack == "strong":
            n_adv = sum(x in Aset for x in ws)
            if all(x in ADset for x in ws) and n_adv >= rp:
                mask[i] = [x in Aset for x in ws]
        else:
            raise ValueError(w.attack)
    return mask


def random_graph(K: int, p: float, seed: int) -> list[int]:
    """Neighbour masks of an Erdos-Renyi graph G(K, p): every pair (j, k)
    is an edge with probability p, drawn from a seeded generator.  Used as a
    clique-search input with many maximal cliques."""
    rng = np.random.default_rng(seed)
    coin = rng.random((K, K)) < p
    rows = [0] * K
    for j in range(K):
        for k in range(j + 1, K):
            if coin[j, k]:
                rows[j] |= 1 << k
                rows[k] |= 1 << j
    return rows


def attack_graph(w: Workload) -> list[int]:
    """Neighbour masks (bit k = worker k) of the agreement graph that the
    workload's attack leaves, for any K, without materialising the C(K,r)
    files: an edge (j, k) is missing iff some file held by both carries
    different copies from j and k.
      weak / all_alie: every copy an adversary holds is distorted, the same
        way by all colluders, so exactly the adversary-honest pairs disagree.
      strong: adversary a and worker k of D disagree iff some file inside
        A u D holds both and at least r' = (r+1)/2 adversaries; all other
        pairs agree (adversaries return honest copies elsewhere).
    Used for graph-only workloads (the clique search alone, as in the
    K = 100 timing experiment); for small K the tests check it against the
    graph computed from actual copies."""
    A, D = adversary_sets(w)
    K, r = w.K, w.r
    missing = set()
    if A and w.attack in ("all_alie", "weak"):
        H = [k for k in range(K) if k not in set(A)]
        missing = {(a, h) for a in A for h in H}
    elif A and w.attack == "strong":
        rp = (r + 1) // 2
        q_a, q_d = len(A), len(D)
        # the r - 2 other members: x more adversaries (x >= r' - 1) and
        # r - 2 - x more workers of D
        ok = any(rp - 1 <= x <= q_a - 1 and 0 <= r - 2 - x <= q_d - 1 for x in range(r - 1))
        if ok:
            missing = {(a, k) for a in A for k in D}
    elif A:
        raise ValueError(w.attack)
    rows = [0] * K
    for j in range(K):
        for k in range(K):
            if j != k and (j, k) not in missing and (k, j) not in missing:
                rows[j] |= 1 << k
    return rows


def _alie_np(w: Workload, c0: int, c1: int) -> np.ndarray:
    b = 0.01 * normal_np(w.seed, STREAM_B, c0, c1)
    f = w.f
    s = np.zeros(c1 - c0)
    for i in range(f):
        s += honest_np(w.seed, i, c0, c1, b).astype(np.float64)
    mu = s / f
    if w.distortion == "foe":
        return (-w.z * mu).astype(np.float32)
    v = np.zeros(c1 - c0)
    for i in range(f):
        t = honest_np(w.seed, i, c0, c1, b).astype(np.float64) - mu
        v += t * t
    sd = np.sqrt(v / f)
    return (mu - w.z * sd).astype(np.float32)


def _alie_torch(w: Workload, c0: int, c1: int, device):
    import torch
    b = 0.01 * normal_torch(w.seed, STREAM_B, c0, c1, device)
    f = w.f
    s = torch.zeros(c1 - c0, dtype=torch.float64, device=device)
    for i in range(f):
        s += honest_torch(w.seed, i, c0, c1, device, b).to(torch.float64)
    mu = s / f
    if w.distortion == "foe":
        return (-w.z * mu).to(torch.float32)
    v = torch.zeros_like(s)
    for i in range(f):
        t = honest_torch(w.seed, i, c0, c1, device, b).to(torch.float64) - mu
        v += t * t
    sd = torch.sqrt(v / f)
    return (mu - w.z * sd).to(torch.float32)


def build_copies_np(w: Workload, file_workers: np.ndarray, c0: int = 0,
                    c1: int | None = None, pad_value: float = 0.0) -> np.ndarray:
    """float32 [f, r, ld'] with the copies of coordinates [c0, c1).

    With the default c0=0, c1=d the last axis is ld (padding filled with
    pad_value); for a slice it is c1-c0.
    """
    full = c1 is None and c0 == 0
    c1 = w.d if c1 is None else c1
    fw = np.asarray(file_workers)
    f, r = fw.shape
    width = w.ld if full else c1 - c0
    out = np.full((f, r, width), pad_value, np.float32)
    mask = corrupted_mask(w, fw)
    bad = None
    if mask.any() and w.distortion in ("alie", "foe"):
        bad = _alie_np(w, c0, c1)
    b = 0.01 * normal_np(w.seed, STREAM_B, c0, c1)
    for i in range(f):
        g = honest_np(w.seed, i, c0, c1, b)
        for s in range(r):
            if not mask[i, s]:
                if w.copy_noise:
                    z = normal_np(w.seed, STREAM_COPY0 + 8 * i + s, c0, c1)
                    out[i, s, : c1 - c0] = (g.astype(np.float64) + w.copy_noise * z).astype(np.float32)
                else:
                    out[i, s, : c1 - c0] = g
            elif w.distortion in ("alie", "foe"):
                out[i, s, : c1 - c0] = bad
            else:
                out[i, s, : c1 - c0] = (g.astype(np.float64) * -w.scale).astype(np.float32)
    return out


def build_copies_torch(w: Workload, file_workers: np.ndarray, device, out=None,
                       pad_value: float = 0.0, c0: int = 0, c1: int | None = None):
    """The same copies as :func:`build_copies_np`, written into a device
    tensor [f, r, ld] (allocated unless ``out`` is given).  Generation is done
    one file at a time so the working set stays a few vectors.  With c0/c1
    only coordinates [c0, c1) are made (a tensor [f, r, round_up(c1 - c0,
    ld_align)]); every value equals the one of the whole-vector build."""
    import torch
    fw = np.asarray(file_workers)
    f, r = fw.shape
    c1 = w.d if c1 is None else c1
    if not 0 <= c0 <= c1 <= w.d:
        raise ValueError(f"slice [{c0}, {c1}) of d={w.d}")
    d = c1 - c0
    ld = w.ld if (c0, c1) == (0, w.d) else max(w.ld_align, -(-d // w.ld_align) * w.ld_align)
    if out is None:
        out = torch.empty((f, r, ld), dtype=torch.float32, device=device)
    if ld > d:
        out[:, :, d:] = pad_value
    if d == 0:
        return out
    mask = corrupted_mask(w, fw)
    bad = None
    if mask.any() and w.distortion in ("alie", "foe"):
        bad = _alie_torch(w, c0, c1, device)
    b = 0.01 * normal_torch(w.seed, STREAM_B, c0, c1, device)
    for i in range(f):
        g = honest_torch(w.seed, i, c0, c1, device, b)
        for s in range(r):
            if not mask[i, s]:
                if w.copy_noise:
                    z = normal_torch(w.seed, STREAM_COPY0 + 8 * i + s, c0, c1, device)
                    out[i, s, :d].copy_((g.to(torch.float64) + w.copy_noise * z).to(torch.float32))
                else:
                    out[i, s, :d].copy_(g)
            elif w.distortion in ("alie", "foe"):
                out[i, s, :d].copy_(bad)
            else:
                out[i, s, :d].copy_((g.to(torch.float64) * -w.scale).to(torch.float32))
    return out


# The five benchmark workloads (K, r, d, attack) of the Aspis evaluation,
# shaped like a flattened ResNet-18 gradient where d = 11,173,962.
CONFIGS = {
    "k7_r3_d4096_alie": Workload("k7_r3_d4096_alie", K=7, r=3, d=4096, q=2,
                                 attack="all_alie", distortion="alie", z=1.0, seed=0,
                                 adversaries=(0, 1)),
    "k15_r3_d1m_weak_reversed": Workload("k15_r3_d1m_weak_reversed", K=15, r=3, d=1_048_576,
                                         q=3, attack="weak", distortion="reversed",
                                         scale=10.0, seed=1),
    "k15_r3_d11m_strong_alie": Workload("k15_r3_d11m_strong_alie", K=15, r=3, d=11_173_962,
                                        q=3, attack="strong", distortion="alie", z=1.0,
                                        seed=2),
    "k21_r3_d2m_strong_alie": Workload("k21_r3_d2m_strong_alie", K=21, r=3, d=2_097_152,
                                       q=5, attack="strong", distortion="alie", z=1.5, seed=3),
    "k15_r5_d1m_strong_alie": Workload("k15_r5_d1m_strong_alie", K=15, r=5, d=1_048_576,
                                       q=4, attack="strong", distortion="alie", z=1.0, seed=4),
}
