"""CPU oracle for the Aspis detection-and-aggregation step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product library never calls it, and it shares no code with the
CUDA path.  The arithmetic lives in ``aspis_oracle.c`` (plain C, pthreads);
this module only compiles it and marshals numpy arrays.

Functions follow the paper (Konstantinidis & Ramamoorthy, "Aspis: Robust
Detection for Distributed Learning"):

* :func:`assign`            -- Algorithm 2 (subset-based assignment), Example 1
* :func:`file_agreement`    -- alpha_i^{(j1,j2)}, Section 4 (first display)
* :func:`pair_agreement`    -- alpha^{(j1,j2)}, Section 4 (second display)
* :func:`graph`             -- edge iff alpha == C(K-2, r-2), Algorithm 3
* :func:`max_cliques_brute` / :func:`max_cliques_bk` -- Algorithm 3
* :func:`max_cliques_wide`  -- Algorithm 3 for up to 128 workers, all maximal cliques counted
* :func:`select`            -- Algorithm 1, Case 1 / Case 2 (Eq. 2)
* :func:`aggregate`, :func:`lower_median`, :func:`mean` -- Algorithm 1 updates
* :func:`sgd`               -- the model update with the aggregate (Eq. 1, momentum)
* :func:`run_round_tolerant` -- the variant for copies that are not bit-identical
  (Section 5: average the honest copies / the largest cluster)
* :func:`run_round`         -- the whole step in the paper's order
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from dataclasses import dataclass

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "aspis_oracle.c")
_LIB_PATH = os.path.join(_HERE, "_build", "liboracle.so")
_lock = threading.Lock()
_lib = None

OK, EINVAL, ERANGE, EEMPTY = 0, 1, 2, 6


def build_oracle(force: bool = False) -> str:
    """Compile ``aspis_oracle.c`` into ``oracle/_build/liboracle.so``."""
    os.makedirs(os.path.dirname(_LIB_PATH), exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread",
                           _SRC, "-o", tmp, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build_oracle())
            P = ctypes.c_void_p
            i64, i32 = ctypes.c_int64, ctypes.c_int
            lib.oracle_binom.argtypes = [i64, i64]
            lib.oracle_binom.restype = i64
            lib.oracle_assign.argtypes = [i32, i32, P, P, P]
            lib.oracle_file_agreement.argtypes = [P, i64, i32, i64, i64, P, i32]
            lib.oracle_pair_agreement.argtypes = [P, P, i64, i32, i32, P]
            lib.oracle_graph.argtypes = [P, i32, i32, P]
            lib.oracle_max_cliques_brute.argtypes = [P, i32, P, P, P]
            lib.oracle_max_cliques_bk.argtypes = [P, i32, P, P, P, P]
            lib.oracle_select.argtypes = [P, P, i64, i32, ctypes.c_uint32, i32, P]
            lib.oracle_select.restype = i64
            lib.oracle_aggregate.argtypes = [P, i64, i32, i64, P, i32, i64, i64, P, i32]
            lib.oracle_lower_median.argtypes = [P, i64, i64, P]
            lib.oracle_mean.argtypes = [P, i64, i64, P]
            lib.oracle_max_cliques_wide.argtypes = [P, i32, P, P, P, P]
            lib.oracle_sgd.argtypes = [P, P, P, i64, ctypes.c_float, ctypes.c_float]
            lib.oracle_file_agreement_tol.argtypes = [P, i64, i32, i64, i64, ctypes.c_float, P, i32]
            lib.oracle_select_tol.argtypes = [P, P, i64, i32, ctypes.c_uint32, i32, P]
            lib.oracle_select_tol.restype = i64
            lib.oracle_file_means.argtypes = [P, i64, i32, i64, i64, P, P]
            _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data)


def _threads(nthreads):
    return int(nthreads) if nthreads else (os.cpu_count() or 1)


def binom(n: int, k: int) -> int:
    return int(_load().oracle_binom(n, k))


@dataclass
class Assignment:
    K: int
    r: int
    f: int
    l: int
    file_workers: np.ndarray   # uint8 [f, r]
    worker_files: np.ndarray   # int32 [K, l]
    slot_of: np.ndarray        # uint8 [K, l]


def assign(K: int, r: int) -> Assignment:
    """Algorithm 2: file i <-> i-th r-subset of workers, lexicographic."""
    f, l = binom(K, r), binom(K - 1, r - 1)
    fw = np.zeros((max(f, 1), r), np.uint8)
    wf = np.zeros((K, max(l, 1)), np.int32)
    so = np.zeros((K, max(l, 1)), np.uint8)
    rc = _load().oracle_assign(K, r, _ptr(fw), _ptr(wf), _ptr(so))
    if rc != OK:
        raise ValueError(f"oracle_assign(K={K}, r={r}) failed: {rc}")
    return Assignment(K, r, f, l, fw[:f], wf[:, :l], so[:, :l])


def file_agreement(copies: np.ndarray, d: int | None = None, nthreads=None) -> np.ndarray:
    """copies: float32 [f, r, ld]; returns uint32 [f] per-file mismatch words."""
    copies = np.ascontiguousarray(copies, dtype=np.float32)
    f, r, ld = copies.shape
    d = ld if d is None else d
    out = np.zeros(f, np.uint32)
    rc = _load().oracle_file_agreement(_ptr(copies), f, r, d, ld, _ptr(out), _threads(nthreads))
    if rc != OK:
        raise ValueError(f"oracle_file_agreement failed: {rc}")
    return out


def pair_agreement(file_neq: np.ndarray, a: Assignment) -> np.ndarray:
    file_neq = np.ascontiguousarray(file_neq, dtype=np.uint32)
    fw = np.ascontiguousarray(a.file_workers, dtype=np.uint8)
    alpha = np.zeros((a.K, a.K), np.int64)
    rc = _load().oracle_pair_agreement(_ptr(file_neq), _ptr(fw), a.f, a.r, a.K, _ptr(alpha))
    if rc != OK:
        raise ValueError(f"oracle_pair_agreement failed: {rc}")
    return alpha


def graph(alpha: np.ndarray, K: int, r: int) -> np.ndarray:
    alpha = np.ascontiguousarray(alpha, dtype=np.int64)
    adj = np.zeros(K, np.uint32)
    rc = _load().oracle_graph(_ptr(alpha), K, r, _ptr(adj))
    if rc != OK:
        raise ValueError(f"oracle_graph failed: {rc}")
    return adj


@dataclass
class Detection:
    omega: int
    n_max: int
    clique: int
    calls: int = 0

    @property
    def success(self) -> bool:
        return self.n_max == 1


def max_cliques_brute(adj: np.ndarray, K: int) -> Detection:
    adj = np.ascontiguousarray(adj, dtype=np.uint32)
    om, nm, cn = ctypes.c_int32(), ctypes.c_uint32(), ctypes.c_uint32()
    rc = _load().oracle_max_cliques_brute(_ptr(adj), K, ctypes.byref(om), ctypes.byref(nm),
                                          ctypes.byref(cn))
    if rc != OK:
        raise ValueError(f"oracle_max_cliques_brute failed: {rc}")
    return Detection(om.value, nm.value, cn.value)


def max_cliques_bk(adj: np.ndarray, K: int) -> Detection:
    adj = np.ascontiguousarray(adj, dtype=np.uint32)
    om, nm, cn, calls = ctypes.c_int32(), ctypes.c_uint32(), ctypes.c_uint32(), ctypes.c_uint64()
    rc = _load().oracle_max_cliques_bk(_ptr(adj), K, ctypes.byref(om), ctypes.byref(nm),
                                       ctypes.byref(cn), ctypes.byref(calls))
    if rc != OK:
        raise ValueError(f"oracle_max_cliques_bk failed: {rc}")
    return Detection(om.value, nm.value, cn.value, calls.value)


@dataclass
class WideDetection:
    omega: int
    n_max: int
    clique: int          # the maximum clique with the smallest mask value, bit k = worker k
    n_maximal: int       # all maximal cliques

    @property
    def success(self) -> bool:
        return self.n_max == 1


def max_cliques_wide(adj: np.ndarray, K: int) -> WideDetection:
    """Algorithm 3 for K <= 128: adj is [K, 4] uint32 (worker k = bit k % 32 of
    word k // 32); an edge needs both rows to list it."""
    adj = np.ascontiguousarray(adj, dtype=np.uint32).reshape(K, 4)
    om, nm, nmax = ctypes.c_int32(), ctypes.c_uint64(), ctypes.c_uint64()
    canon = np.zeros(4, np.uint32)
    rc = _load().oracle_max_cliques_wide(_ptr(adj), K, ctypes.byref(om), ctypes.byref(nm),
                                         _ptr(canon), ctypes.byref(nmax))
    if rc != OK:
        raise ValueError(f"oracle_max_cliques_wide failed: {rc}")
    clique = sum(int(canon[i]) << (32 * i) for i in range(4))
    return WideDetection(om.value, nm.value, clique, nmax.value)


def masks_to_words(rows, K: int) -> np.ndarray:
    """[K, 4] uint32 adjacency words from K Python-int neighbour masks."""
    out = np.zeros((K, 4), np.uint32)
    for j, m in enumerate(rows):
        for i in range(4):
            out[j, i] = (int(m) >> (32 * i)) & 0xFFFFFFFF
    return out


def select(file_neq: np.ndarray, a: Assignment, clique: int, success: bool):
    """Algorithm 1 selection; returns (sel int8 [f], n_sel)."""
    file_neq = np.ascontiguousarray(file_neq, dtype=np.uint32)
    fw = np.ascontiguousarray(a.file_workers, dtype=np.uint8)
    sel = np.zeros(max(a.f, 1), np.int8)
    n = _load().oracle_select(_ptr(file_neq), _ptr(fw), a.f, a.r, ctypes.c_uint32(clique),
                              1 if success else 0, _ptr(sel))
    return sel[: a.f], int(n)


def aggregate(copies: np.ndarray, sel: np.ndarray, mode: int = 0, c0: int = 0,
              c1: int | None = None, nthreads=None) -> np.ndarray:
    """Coordinate-wise lower median (mode 0) or mean (mode 1) over [c0, c1)."""
    copies = np.ascontiguousarray(copies, dtype=np.float32)
    f, r, ld = copies.shape
    c1 = ld if c1 is None else c1
    sel = np.ascontiguousarray(sel, dtype=np.int8)
    out = np.zeros(max(c1 - c0, 1), np.float32)
    rc = _load().oracle_aggregate(_ptr(copies), f, r, ld, _ptr(sel), mode, c0, c1, _ptr(out),
                                  _threads(nthreads))
    if rc == EEMPTY:
        raise ValueError("no file kept: aggregation is empty")
    if rc != OK:
        raise ValueError(f"oracle_aggregate failed: {rc}")
    return out[: c1 - c0]


def lower_median(vals: np.ndarray) -> np.ndarray:
    """Column-wise lower median of a dense float32 [n, m] matrix (bit-exact)."""
    vals = np.ascontiguousarray(vals, dtype=np.float32)
    n, m = vals.shape
    out = np.zeros(max(m, 1), np.float32)
    rc = _load().oracle_lower_median(_ptr(vals), n, m, _ptr(out))
    if rc != OK:
        raise ValueError(f"oracle_lower_median failed: {rc}")
    return out[:m]


def mean(vals: np.ndarray) -> np.ndarray:
    vals = np.ascontiguousarray(vals, dtype=np.float32)
    n, m = vals.shape
    out = np.zeros(max(m, 1), np.float32)
    rc = _load().oracle_mean(_ptr(vals), n, m, _ptr(out))
    if rc != OK:
        raise ValueError(f"oracle_mean failed: {rc}")
    return out[:m]


def sgd(g: np.ndarray, w: np.ndarray, v: np.ndarray | None, eta: float, mu: float):
    """One update w, v <- (Eq. 1 with momentum) on copies; returns (w', v').

    eta and mu are rounded to fp32 first, as the library receives them.
    With mu == 0, v is returned unchanged (None stays None)."""
    g = np.ascontiguousarray(g, dtype=np.float32)
    w2 = np.array(w, dtype=np.float32, copy=True)
    v2 = None if v is None else np.array(v, dtype=np.float32, copy=True)
    m = g.size
    if w2.size != m or (v2 is not None and v2.size != m):
        raise ValueError("g, w and v must have the same length")
    rc = _load().oracle_sgd(_ptr(g), _ptr(w2), None if v2 is None else _ptr(v2), m,
                            float(np.float32(eta)), float(np.float32(mu)))
    if rc != OK:
        raise ValueError(f"oracle_sgd failed: {rc}")
    return w2, v2


@dataclass
class RoundResult:
    file_neq: np.ndarray
    alpha: np.ndarray
    adj: np.ndarray
    det: Detection
    sel: np.ndarray
    n_sel: int
    out: np.ndarray | None


def detect(adj: np.ndarray, K: int) -> Detection:
    """Algorithm 3 on the agreement graph (brute force when K <= 20)."""
    return max_cliques_brute(adj, K) if K <= 20 else max_cliques_bk(adj, K)


def run_round(copies: np.ndarray, a: Assignment, d: int | None = None, mode: int = 0,
              nthreads=None, aggregate_out: bool = True) -> RoundResult:
    """The whole detection-and-aggregation step on one round's copies."""
    f, r, ld = copies.shape
    d = ld if d is None else d
    file_neq = file_agreement(copies, d, nthreads)
    alpha = pair_agreement(file_neq, a)
    adj = graph(alpha, a.K, a.r)
    det = detect(adj, a.K)
    sel, n_sel = select(file_neq, a, det.clique, det.success)
    out = None
    if aggregate_out and n_sel > 0:
        out = aggregate(copies, sel, mode, 0, d, nthreads)
    return RoundResult(file_neq, alpha, adj, det, sel, n_sel, out)


# ------------------------------------------------ copies that are not bit-identical

def file_agreement_tol(copies: np.ndarray, tau: float, d: int | None = None,
                       nthreads=None) -> np.ndarray:
    """Per-file mismatch words under the tolerance: bit p set iff the copies
    of slot pair p are not within tau on every coordinate (fp32)."""
    copies = np.ascontiguousarray(copies, dtype=np.float32)
    f, r, ld = copies.shape
    d = ld if d is None else d
    out = np.zeros(max(f, 1), np.uint32)
    rc = _load().oracle_file_agreement_tol(_ptr(copies), f, r, d, ld, float(np.float32(tau)),
                                           _ptr(out), _threads(nthreads))
    if rc != OK:
        raise ValueError(f"oracle_file_agreement_tol failed: {rc}")
    return out[:f]


def select_tol(file_neq: np.ndarray, a: Assignment, clique: int, success: bool):
    """(slot_mask[f] uint8, files kept): the copies averaged for each file."""
    file_neq = np.ascontiguousarray(file_neq, dtype=np.uint32)
    fw = np.ascontiguousarray(a.file_workers, dtype=np.uint8)
    mask = np.zeros(max(a.f, 1), np.uint8)
    n = _load().oracle_select_tol(_ptr(file_neq), _ptr(fw), a.f, a.r, ctypes.c_uint32(clique),
                                  1 if success else 0, _ptr(mask))
    return mask[: a.f], int(n)


def file_means(copies: np.ndarray, slot_mask: np.ndarray, d: int | None = None) -> np.ndarray:
    """[f, d] averages of the chosen copies of every file (zeros where dropped)."""
    copies = np.ascontiguousarray(copies, dtype=np.float32)
    f, r, ld = copies.shape
    d = ld if d is None else d
    mask = np.ascontiguousarray(slot_mask, dtype=np.uint8)
    out = np.zeros((max(f, 1), max(d, 1)), np.float32)
    rc = _load().oracle_file_means(_ptr(copies), f, r, d, ld, _ptr(mask), _ptr(out))
    if rc != OK:
        raise ValueError(f"oracle_file_means failed: {rc}")
    return out[:f, :d]


@dataclass
class TolerantResult:
    file_neq: np.ndarray
    adj: np.ndarray
    det: Detection
    slot_mask: np.ndarray
    n_kept: int
    means: np.ndarray
    out: np.ndarray | None


def run_round_tolerant(copies: np.ndarray, a: Assignment, tau: float, d: int | None = None,
                       mode: int = 0, nthreads=None) -> TolerantResult:
    """The round with "close within tau" in place of bitwise equality; the
    kept files' averaged copies are reduced by the lower median (mode 0) or
    the mean (mode 1)."""
    f, r, ld = copies.shape
    d = ld if d is None else d
    file_neq = file_agreement_tol(copies, tau, d, nthreads)
    adj = graph(pair_agreement(file_neq, a), a.K, a.r)
    det = detect(adj, a.K)
    mask, n = select_tol(file_neq, a, det.clique, det.success)
    means = file_means(copies, mask, d)
    out = None
    if n > 0:
        kept = means[mask != 0]
        out = lower_median(kept) if mode == 0 else mean(kept)
    return TolerantResult(file_neq, adj, det, mask, n, means, out)
