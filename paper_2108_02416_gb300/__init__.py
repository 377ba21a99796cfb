"""Python binding of libaspis (C ABI in ``include/aspis.h``).

Argument marshalling only: every step of the PS round runs in the library's
CUDA kernels.  PyTorch supplies device memory and streams.  There is no CPU
fallback; if ``libaspis.so`` is missing, importing the binding raises.
Build it with ``python paper_2108_02416_gb300/build.py`` (or
``__graft_entry__.build()``).

The call names mirror the C entry points:

  aspis_assign(K, r) -> Assignment          Algorithm 2
  aspis_check(copies, d, a, file_neq, adj)  per-file agreement + graph G
  aspis_detect(adj, K, det)                 Algorithm 3 (maximum cliques)
  aspis_select(file_neq, det, a, sel)       Algorithm 1 (Case 1 / Case 2)
  aspis_aggregate(copies, d, a, sel, det, out, mode)   coordinate-wise median / mean
  aspis_round(...)                          the four device steps on one stream
  aspis_round_host(...)                     the same from pinned host memory
  aspis_round_static(copies, d, a, det, out, mode)   the round with no device allocation
  aspis_sgd(g, w, v, eta, mu)               the model update with the aggregate (Eq. 1, momentum)
  aspis_detect_wide(adj, K, det)            Algorithm 3 for K <= 128 (graph given directly)
  aspis_round_tolerant(copies, d, a, tau, ...)   the round for copies that are not bit-identical
"""
from __future__ import annotations

import ctypes
import os

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libaspis.so")

OK, E_INVAL, E_RANGE, E_ALIGN, E_CUDA, E_LIMIT, E_EMPTY, E_NOT_IMPLEMENTED = range(8)
MAX_K, MAX_R, MAX_AGG_FILES = 31, 8, 6144
STATIC_MAX_FILES = 6144
MEDIAN, MEAN = 0, 1


class AspisError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_str(status)} ({status})")


class _Assignment(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("r", ctypes.c_int32), ("f", ctypes.c_int64),
                ("l", ctypes.c_int64), ("pair_share", ctypes.c_int64),
                ("file_workers", ctypes.POINTER(ctypes.c_uint8)),
                ("worker_files", ctypes.POINTER(ctypes.c_int32)),
                ("slot_of", ctypes.POINTER(ctypes.c_uint8)),
                ("dev_file_workers", ctypes.c_void_p)]


class Detection(ctypes.Structure):
    """Host image of ``aspis_detection`` (36 bytes)."""
    _fields_ = [("clique_mask", ctypes.c_uint32), ("omega", ctypes.c_int32),
                ("n_max_cliques", ctypes.c_uint32), ("success", ctypes.c_int32),
                ("n_sel", ctypes.c_int32), ("status", ctypes.c_int32),
                ("search_nodes", ctypes.c_uint32), ("node_budget", ctypes.c_uint32),
                ("median_exact", ctypes.c_uint32)]

    @classmethod
    def from_tensor(cls, t):
        """Read a device/host uint8 tensor holding an aspis_detection."""
        raw = bytes(t.detach().to("cpu").contiguous().numpy().tobytes())
        return cls.from_buffer_copy(raw)

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


DETECTION_BYTES = ctypes.sizeof(Detection)

WIDE_MAX_K = 128
WIDE_ALL_MAXIMAL = 1


class DetectionWide(ctypes.Structure):
    """Host image of ``aspis_detection_wide`` (64 bytes)."""
    _fields_ = [("clique_words", ctypes.c_uint32 * 4), ("n_max_cliques", ctypes.c_uint64),
                ("n_maximal", ctypes.c_uint64), ("search_nodes", ctypes.c_uint64),
                ("omega", ctypes.c_int32), ("success", ctypes.c_int32),
                ("status", ctypes.c_int32), ("node_budget", ctypes.c_uint32),
                ("flags", ctypes.c_uint32), ("reserved", ctypes.c_uint32)]

    @classmethod
    def from_tensor(cls, t):
        raw = bytes(t.detach().to("cpu").contiguous().numpy().tobytes())
        return cls.from_buffer_copy(raw)

    @property
    def clique_mask(self) -> int:
        """the reported clique as one integer, bit k = worker k"""
        return sum(int(self.clique_words[i]) << (32 * i) for i in range(4))


WIDE_DETECTION_BYTES = ctypes.sizeof(DetectionWide)


def wide_detection_buffer(device, node_budget: int = 0, flags: int = 0):
    """A device uint8 tensor holding an aspis_detection_wide with the inputs set."""
    import torch
    d = DetectionWide()
    d.node_budget = node_budget
    d.flags = flags
    host = torch.frombuffer(bytearray(bytes(d)), dtype=torch.uint8)
    return host.to(device)


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it first (python "
                          "paper_2108_02416_gb300/build.py or __graft_entry__.build()); "
                          "there is no CPU fallback")
    lib = ctypes.CDLL(LIB_PATH)
    P, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
    A = ctypes.POINTER(_Assignment)
    sig = {
        "aspis_status_str": ([i32], ctypes.c_char_p),
        "aspis_abi_version": ([], i32),
        "aspis_workspace_bytes": ([A], ctypes.c_size_t),
        "aspis_assign": ([i32, i32, A], i32),
        "aspis_assignment_to_device": ([A], i32),
        "aspis_assignment_free": ([A], None),
        "aspis_check": ([P, i64, i64, A, P, P, P], i32),
        "aspis_graph": ([P, A, P, P], i32),
        "aspis_detect": ([P, i32, P, P], i32),
        "aspis_select": ([P, P, A, P, P], i32),
        "aspis_aggregate": ([P, i64, i64, A, P, P, i32, P, P], i32),
        "aspis_round": ([P, i64, i64, A, P, P, P, P, i32, P, P], i32),
        "aspis_round_host": ([P, P, i64, i64, A, P, P, P, P, i32, P, P, P, P], i32),
        "aspis_round_static": ([P, i64, i64, A, P, i32, P, P], i32),
        "aspis_sgd": ([P, P, P, i64, ctypes.c_float, ctypes.c_float, P], i32),
        "aspis_detect_wide": ([P, i32, P, P], i32),
        "aspis_round_tolerant": ([P, i64, i64, A, ctypes.c_float, P, P, P, P, P, P, i64, i32, P, P],
                                 i32),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    return lib


lib = _load()


def status_str(status: int) -> str:
    return lib.aspis_status_str(int(status)).decode()


def _ok(status: int, where: str):
    if status != OK:
        raise AspisError(status, where)


class Assignment:
    """Owns an ``aspis_assignment`` (host tables + device mirror)."""

    def __init__(self, K: int, r: int, device: bool = True):
        self._a = _Assignment()
        _ok(lib.aspis_assign(K, r, ctypes.byref(self._a)), "aspis_assign")
        if device:
            self.to_device()

    def to_device(self):
        _ok(lib.aspis_assignment_to_device(ctypes.byref(self._a)), "aspis_assignment_to_device")
        return self

    @property
    def ref(self):
        return ctypes.byref(self._a)

    K = property(lambda s: s._a.K)
    r = property(lambda s: s._a.r)
    f = property(lambda s: s._a.f)
    l = property(lambda s: s._a.l)
    pair_share = property(lambda s: s._a.pair_share)

    def file_workers(self):
        import numpy as np
        return np.ctypeslib.as_array(self._a.file_workers, (self.f * self.r,)).reshape(self.f, self.r).copy()

    def worker_files(self):
        import numpy as np
        return np.ctypeslib.as_array(self._a.worker_files, (self.K * self.l,)).reshape(self.K, self.l).copy()

    def slot_of(self):
        import numpy as np
        return np.ctypeslib.as_array(self._a.slot_of, (self.K * self.l,)).reshape(self.K, self.l).copy()

    def close(self):
        if getattr(self, "_a", None) is not None and self._a.K:
            lib.aspis_assignment_free(ctypes.byref(self._a))

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def aspis_assign(K: int, r: int, device: bool = True) -> Assignment:
    return Assignment(K, r, device)


def _stream(stream):
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t, dtype=None, name="tensor"):
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _ld(copies, a: Assignment):
    if copies.dim() != 3 or copies.shape[0] != a.f or copies.shape[1] != a.r:
        raise ValueError(f"copies must be [f={a.f}, r={a.r}, ld], got {tuple(copies.shape)}")
    return int(copies.shape[2])


def aspis_check(copies, d: int, a: Assignment, file_neq, adj, stream=None):
    import torch
    ld = _ld(copies, a)
    _ok(lib.aspis_check(_dev(copies, torch.float32, "copies"), d, ld, a.ref,
                        _dev(file_neq, torch.int32, "file_neq"), _dev(adj, torch.int32, "adj"),
                        _stream(stream)), "aspis_check")


def aspis_graph(file_neq, a: Assignment, adj, stream=None):
    import torch
    _ok(lib.aspis_graph(_dev(file_neq, torch.int32, "file_neq"), a.ref,
                        _dev(adj, torch.int32, "adj"), _stream(stream)), "aspis_graph")


def aspis_detect(adj, K: int, det, stream=None):
    import torch
    _ok(lib.aspis_detect(_dev(adj, torch.int32, "adj"), K, _dev(det, torch.uint8, "det"),
                         _stream(stream)), "aspis_detect")


def aspis_select(file_neq, det, a: Assignment, sel, stream=None):
    import torch
    _ok(lib.aspis_select(_dev(file_neq, torch.int32, "file_neq"), _dev(det, torch.uint8, "det"),
                         a.ref, _dev(sel, torch.int8, "sel"), _stream(stream)), "aspis_select")


def aspis_aggregate(copies, d: int, a: Assignment, sel, det, out, mode: int = MEDIAN, stream=None):
    import torch
    ld = _ld(copies, a)
    _ok(lib.aspis_aggregate(_dev(copies, torch.float32, "copies"), d, ld, a.ref,
                            _dev(sel, torch.int8, "sel"), _dev(det, torch.uint8, "det"), mode,
                            _dev(out, torch.float32, "out"), _stream(stream)), "aspis_aggregate")


def aspis_round(copies, d: int, a: Assignment, file_neq, adj, det, sel, out, mode: int = MEDIAN,
                stream=None):
    import torch
    ld = _ld(copies, a)
    _ok(lib.aspis_round(_dev(copies, torch.float32, "copies"), d, ld, a.ref,
                        _dev(file_neq, torch.int32, "file_neq"), _dev(adj, torch.int32, "adj"),
                        _dev(det, torch.uint8, "det"), _dev(sel, torch.int8, "sel"), mode,
                        _dev(out, torch.float32, "out"), _stream(stream)), "aspis_round")


def aspis_round_host(host_copies, dev_copies, d: int, a: Assignment, file_neq, adj, det, sel,
                     dev_out, host_out, host_det, mode: int = MEDIAN, stream=None):
    """host_copies / host_out / host_det: CPU tensors (pinned for full speed)."""
    import torch
    ld = _ld(dev_copies, a)
    for t, nm in ((host_copies, "host_copies"), (host_out, "host_out"), (host_det, "host_det")):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{nm} must be a contiguous CPU tensor")
    if host_copies.numel() != dev_copies.numel() or host_copies.dtype != torch.float32:
        raise ValueError("host_copies must match dev_copies (float32)")
    _ok(lib.aspis_round_host(ctypes.c_void_p(host_copies.data_ptr()),
                             _dev(dev_copies, torch.float32, "dev_copies"), d, ld, a.ref,
                             _dev(file_neq, torch.int32, "file_neq"), _dev(adj, torch.int32, "adj"),
                             _dev(det, torch.uint8, "det"), _dev(sel, torch.int8, "sel"), mode,
                             _dev(dev_out, torch.float32, "dev_out"),
                             ctypes.c_void_p(host_out.data_ptr()),
                             ctypes.c_void_p(host_det.data_ptr()), _stream(stream)),
        "aspis_round_host")


def aspis_round_static(copies, d: int, a: Assignment, det, out, mode: int = MEDIAN, stream=None):
    """The round for callers that cannot allocate device memory: the
    intermediates live in the library's fixed device array (see aspis.h);
    ``a`` needs no device mirror.  Calls that may overlap on the GPU race."""
    import torch
    ld = _ld(copies, a)
    _ok(lib.aspis_round_static(_dev(copies, torch.float32, "copies"), d, ld, a.ref,
                               _dev(det, torch.uint8, "det"), mode,
                               _dev(out, torch.float32, "out"), _stream(stream)),
        "aspis_round_static")


def aspis_detect_wide(adj, K: int, det, stream=None):
    """Algorithm 3 for K <= 128 workers: ``adj`` is a device uint32 [K, 4]
    tensor (worker k = bit k % 32 of word k // 32), ``det`` a device uint8
    tensor from :func:`wide_detection_buffer`."""
    import torch
    if adj.numel() < 4 * K:
        raise ValueError("adj must hold K rows of 4 words")
    if adj.dtype not in (torch.int32, getattr(torch, "uint32", torch.int32)):
        raise ValueError(f"adj must hold 32-bit words, got {adj.dtype}")
    _ok(lib.aspis_detect_wide(_dev(adj, None, "adj"), K, _dev(det, torch.uint8, "det"),
                              _stream(stream)),
        "aspis_detect_wide")


def aspis_round_tolerant(copies, d: int, a: Assignment, tau: float, file_neq, adj, det, slot_mask,
                         sel, means, out, mode: int = MEDIAN, stream=None):
    """The round with "close within tau" in place of bitwise equality and the
    kept files' averaged copies aggregated (see aspis.h).  ``means`` is a
    device float32 [f, ldm] tensor with ldm >= d."""
    import torch
    ld = _ld(copies, a)
    if means.dim() != 2 or means.shape[0] != a.f or means.shape[1] < d:
        raise ValueError(f"means must be [f={a.f}, ldm >= d], got {tuple(means.shape)}")
    _ok(lib.aspis_round_tolerant(_dev(copies, torch.float32, "copies"), d, ld, a.ref, float(tau),
                                 _dev(file_neq, torch.int32, "file_neq"), _dev(adj, torch.int32, "adj"),
                                 _dev(det, torch.uint8, "det"), _dev(slot_mask, torch.uint8, "slot_mask"),
                                 _dev(sel, torch.int8, "sel"), _dev(means, torch.float32, "means"),
                                 int(means.shape[1]), mode, _dev(out, torch.float32, "out"),
                                 _stream(stream)),
        "aspis_round_tolerant")


def aspis_sgd(g, w, v, eta: float, mu: float = 0.9, stream=None):
    """w, v <- one SGD step with heavy-ball momentum on the aggregate g
    (in place; see aspis.h).  ``v`` may be None when ``mu == 0``."""
    import torch
    n = g.numel()
    if w.numel() != n or (v is not None and v.numel() != n):
        raise ValueError("g, w and v must have the same number of elements")
    vp = None if v is None else _dev(v, torch.float32, "v")
    _ok(lib.aspis_sgd(_dev(g, torch.float32, "g"), _dev(w, torch.float32, "w"), vp, n,
                      float(eta), float(mu), _stream(stream)),
        "aspis_sgd")


class RoundBuffers:
    """Device buffers of one round for an assignment (allocated by torch)."""

    def __init__(self, a: Assignment, d: int, device="cuda"):
        import torch
        self.file_neq = torch.zeros(a.f, dtype=torch.int32, device=device)
        self.adj = torch.zeros(a.K, dtype=torch.int32, device=device)
        self.det = torch.zeros(DETECTION_BYTES, dtype=torch.uint8, device=device)
        self.sel = torch.zeros(a.f, dtype=torch.int8, device=device)
        self.out = torch.zeros(d, dtype=torch.float32, device=device)

    def detection(self) -> Detection:
        return Detection.from_tensor(self.det)


class TolerantBuffers(RoundBuffers):
    """RoundBuffers plus the slot masks and the [f, round_up(d, 4)] averages
    of the tolerant round."""

    def __init__(self, a: Assignment, d: int, device):
        import torch
        super().__init__(a, d, device)
        self.slot_mask = torch.zeros(a.f, dtype=torch.uint8, device=device)
        self.means = torch.zeros((a.f, (d + 3) // 4 * 4), dtype=torch.float32, device=device)
