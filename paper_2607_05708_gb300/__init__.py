"""GB300 (sm_103a) hot path of MemAttention's memory system (arXiv 2607.05708).

Thin Python binding of the C ABI in ``include/akashic_mem.h``
(``libakashic_mem.so``, built in-tree by ``_build.build()``).  It only
marshals arguments: every step of retrieval (score, relation propagation,
top-k, page resolve) and of the relation update (cosine top-M, CSR insert)
runs in the library's CUDA kernels.  PyTorch is used for device memory and
streams.  There is no CPU fallback: without the built library every call
raises.
"""
from __future__ import annotations

import ctypes
import os

from ._build import LIB as LIB_PATH
from ._build import build

__all__ = ["MemStore", "AkashicError", "load_library", "build", "EXPORTS", "STATUS", "PHASES",
           "softmax_scores_noalloc", "sort_pairs"]

STATUS = {0: "OK", 1: "EINVAL", 2: "ENOMEM", 3: "ECAPACITY", 4: "ECUDA", 5: "ETIMEOUT",
          6: "EDEVICE", 7: "ERANGE"}
PHASES = ("score", "propagate", "select", "relate", "graph", "relocate", "compact", "bound",
          "last_hop", "csr_insert", "transpose", "hub_plan")

# Every function declared in include/akashic_mem.h.
EXPORTS = (
    "akashic_mem_create", "akashic_mem_destroy", "akashic_mem_append_chunks",
    "akashic_mem_update_relations", "akashic_mem_retrieve", "akashic_mem_export_csr",
    "akashic_mem_size", "akashic_mem_sync", "akashic_mem_set_profiling",
    "akashic_mem_phase_times", "akashic_mem_last_error", "akashic_mem_softmax_scores_noalloc",
    "akashic_mem_set_namespace", "akashic_mem_retrieve_scoped", "akashic_mem_delete",
    "akashic_mem_relocate", "akashic_mem_compact_pages", "akashic_mem_page_stats",
    "akashic_mem_export_pages", "akashic_mem_check_wait_timeout", "akashic_mem_sort_pairs",
)


class AkashicError(RuntimeError):
    def __init__(self, status: int, message: str):
        self.status = status
        self.code = STATUS.get(status, str(status))
        super().__init__(f"akashic_mem {self.code}: {message}")


class _Config(ctypes.Structure):
    _fields_ = [("dim", ctypes.c_int32), ("capacity", ctypes.c_int64),
                ("chunks_per_page", ctypes.c_int32), ("device", ctypes.c_int32),
                ("temperature", ctypes.c_float), ("relation_scale", ctypes.c_float)]


_lib = None


def load_library(path: str | None = None):
    """Load libakashic_mem.so (raises if it has not been built)."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise ImportError(f"{p} is missing: build the CUDA library first "
                          "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(p)
    V, I32, I64, F = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float
    P64 = ctypes.POINTER(ctypes.c_int64)
    sig = {
        "akashic_mem_create": ([ctypes.POINTER(_Config), ctypes.POINTER(V)], ctypes.c_int),
        "akashic_mem_destroy": ([V], None),
        "akashic_mem_append_chunks": ([V, V, I64, V, V, V, V, P64, V], ctypes.c_int),
        "akashic_mem_update_relations": ([V, I64, I64, I32, I32, V], ctypes.c_int),
        "akashic_mem_retrieve": ([V, V, I32, I32, F, I32, V, V, V, V, V], ctypes.c_int),
        "akashic_mem_retrieve_scoped": ([V, V, I32, I32, F, I32, V, I32, V, V, V, V, V],
                                        ctypes.c_int),
        "akashic_mem_set_namespace": ([V, I64, I64, V, V], ctypes.c_int),
        "akashic_mem_delete": ([V, V, I64, V], ctypes.c_int),
        "akashic_mem_relocate": ([V, V, I32, I32, F, V], ctypes.c_int),
        "akashic_mem_compact_pages": ([V, F, F, P64, V], ctypes.c_int),
        "akashic_mem_page_stats": ([V, P64], ctypes.c_int),
        "akashic_mem_export_pages": ([V, V, V], ctypes.c_int),
        "akashic_mem_export_csr": ([V, P64, P64, V, V, V, V, V], ctypes.c_int),
        "akashic_mem_size": ([V, P64, P64], ctypes.c_int),
        "akashic_mem_sync": ([V, V], ctypes.c_int),
        "akashic_mem_check_wait_timeout": ([V, ctypes.c_uint32, V], ctypes.c_int),
        "akashic_mem_sort_pairs": ([V, V, I64, I32, V], ctypes.c_int),
        "akashic_mem_set_profiling": ([V, I32], ctypes.c_int),
        "akashic_mem_phase_times": ([V, ctypes.POINTER(ctypes.c_float), ctypes.POINTER(I32)],
                                    ctypes.c_int),
        "akashic_mem_last_error": ([], ctypes.c_char_p),
        "akashic_mem_softmax_scores_noalloc": ([V, I64, I32, V, I32, F, V, V, V, V, V],
                                               ctypes.c_int),
    }
    for name, (args, res) in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    if path is None:
        _lib = lib
    return lib


def _check(rc: int):
    if rc != 0:
        msg = load_library().akashic_mem_last_error().decode(errors="replace")
        raise AkashicError(rc, msg)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(torch, stream, device):
    s = stream if stream is not None else torch.cuda.current_stream(device)
    return ctypes.c_void_p(s.cuda_stream)


def softmax_scores_noalloc(emb, q, u, z, temperature=0.0, shift=None, status=None, stream=None):
    """Scores for callers that cannot allocate: fills the caller's u [n, B]
    and z [B] (softmax = u[:, b] / z[b]) through
    akashic_mem_softmax_scores_noalloc, which uses a fixed scratch array and
    allocates nothing.  emb: int16 [n, dim], q: int16 [B, dim] with B in
    {32, 64, 128, 256}, all CUDA tensors on the current device."""
    import torch
    for t, name in ((emb, "emb"), (q, "q"), (u, "u"), (z, "z")):
        if not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA tensor")
    s = stream if stream is not None else torch.cuda.current_stream(emb.device)
    _check(load_library().akashic_mem_softmax_scores_noalloc(
        _ptr(emb), emb.shape[0], emb.shape[1], _ptr(q), q.shape[0], float(temperature), _ptr(u),
        _ptr(z), _ptr(shift), _ptr(status), ctypes.c_void_p(s.cuda_stream)))


def sort_pairs(keys, vals, bits=32, stream=None):
    """Stable in-place sort of (keys, vals), int32 CUDA tensors of equal
    length, by the low `bits` bits of the keys, through akashic_mem_sort_pairs
    (the library's own sort primitive)."""
    import torch
    for t, name in ((keys, "keys"), (vals, "vals")):
        if not t.is_cuda or not t.is_contiguous() or t.dtype != torch.int32:
            raise ValueError(f"{name} must be a contiguous int32 CUDA tensor")
    if keys.numel() != vals.numel():
        raise ValueError("keys and vals differ in length")
    s = stream if stream is not None else torch.cuda.current_stream(keys.device)
    _check(load_library().akashic_mem_sort_pairs(_ptr(keys), _ptr(vals), keys.numel(), int(bits),
                                                 ctypes.c_void_p(s.cuda_stream)))


class MemStore:
    """A chunk store on one GPU; methods mirror the C ABI one to one."""

    def __init__(self, dim: int, capacity: int, chunks_per_page: int = 64, device: int = 0,
                 temperature: float = 0.0, relation_scale: float = 0.0):
        import torch
        self._torch = torch
        self.device = device
        self.dim = dim
        lib = load_library()
        cfg = _Config(dim, capacity, chunks_per_page, device, temperature, relation_scale)
        h = ctypes.c_void_p()
        _check(lib.akashic_mem_create(ctypes.byref(cfg), ctypes.byref(h)))
        self._h = h

    @classmethod
    def from_arrays(cls, emb, page_of=None, row_ptr=None, col=None, aff=None, *, dim=None,
                    capacity=None, chunks_per_page=64, device=0, temperature=0.0,
                    relation_scale=0.0, stream=None):
        """Create a store and append host (numpy) arrays: emb uint16 [n, dim] bf16 bits,
        page_of int32 [n], optional out-edge CSR row_ptr/col/aff of those rows."""
        import numpy as np
        import torch
        dev = torch.device("cuda", device)
        n, d = emb.shape
        st = cls(d if dim is None else dim, capacity or n, chunks_per_page, device, temperature,
                 relation_scale)

        def up(a, dt):
            if a is None:
                return None
            return torch.from_numpy(np.ascontiguousarray(a).view(dt)).to(dev)

        st.append_chunks(up(emb, np.int16), up(page_of, np.int32),
                         up(row_ptr, np.int64), up(col, np.int32), up(aff, np.float32),
                         stream=stream)
        return st

    # -- helpers
    def _dev(self, t, dtype, name, numel=None):
        torch = self._torch
        if t is None:
            return None
        if not t.is_cuda or t.device.index != self.device:
            raise ValueError(f"{name} must be a CUDA tensor on device {self.device}")
        if t.dtype != dtype:
            raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")
        if numel is not None and t.numel() < numel:
            raise ValueError(f"{name} needs {numel} elements")
        return t

    def close(self):
        if getattr(self, "_h", None) and self._h.value:
            load_library().akashic_mem_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- ABI
    def append_chunks(self, emb, page_of=None, row_ptr=None, col=None, aff=None, stream=None) -> int:
        """emb: int16 [n, dim] (bf16 bits); page_of int32 [n]; optional CSR of the new rows."""
        torch = self._torch
        self._dev(emb, torch.int16, "emb")
        n = emb.shape[0]
        self._dev(page_of, torch.int32, "page_of", n)
        self._dev(row_ptr, torch.int64, "row_ptr", n + 1)
        self._dev(col, torch.int32, "col")
        self._dev(aff, torch.float32, "aff")
        first = ctypes.c_int64(-1)
        _check(load_library().akashic_mem_append_chunks(
            self._h, _ptr(emb), n, _ptr(page_of), _ptr(row_ptr), _ptr(col), _ptr(aff),
            ctypes.byref(first), _stream(torch, stream, self.device)))
        return first.value

    def update_relations(self, first: int, n: int, M: int, reciprocal: bool = True, stream=None):
        _check(load_library().akashic_mem_update_relations(
            self._h, first, n, M, int(bool(reciprocal)), _stream(self._torch, stream, self.device)))

    def relocate(self, S, tau_assoc: float = 0.7, stream=None):
        """Relocation of co-retrieved chunks (S: int64 [n_req, s_len] device tensor)."""
        torch = self._torch
        self._dev(S, torch.int64, "S")
        n_req, s_len = (S.shape[0], S.shape[1]) if S.dim() == 2 else (1, S.shape[0])
        _check(load_library().akashic_mem_relocate(self._h, _ptr(S), n_req, s_len,
                                                   float(tau_assoc),
                                                   _stream(torch, stream, self.device)))

    def compact_pages(self, theta: float = 0.75, tau_assoc: float = 0.7, stream=None) -> int:
        rel = ctypes.c_int64()
        _check(load_library().akashic_mem_compact_pages(
            self._h, float(theta), float(tau_assoc), ctypes.byref(rel),
            _stream(self._torch, stream, self.device)))
        return rel.value

    def page_stats(self) -> dict:
        out = (ctypes.c_int64 * 5)()
        _check(load_library().akashic_mem_page_stats(self._h, out))
        keys = ("pages_in_use", "slots_total", "slots_live", "chunk_writes", "appended")
        return dict(zip(keys, list(out)))

    def export_pages(self, stream=None):
        torch = self._torch
        n, _ = self.size()
        out = torch.empty(max(n, 1), dtype=torch.int32, device=torch.device("cuda", self.device))
        _check(load_library().akashic_mem_export_pages(self._h, _ptr(out),
                                                       _stream(torch, stream, self.device)))
        return out[:n]

    def delete(self, ids, stream=None):
        """Delete chunks (int64 device tensor of chunk IDs)."""
        torch = self._torch
        self._dev(ids, torch.int64, "ids")
        _check(load_library().akashic_mem_delete(self._h, _ptr(ids), ids.numel(),
                                                 _stream(torch, stream, self.device)))

    def set_namespace(self, first: int, ns, stream=None):
        """Tags of chunk IDs [first, first+len(ns)) (int32 device tensor)."""
        torch = self._torch
        self._dev(ns, torch.int32, "ns")
        _check(load_library().akashic_mem_set_namespace(
            self._h, first, ns.numel(), _ptr(ns), _stream(torch, stream, self.device)))

    def retrieve(self, q, k: int, alpha: float, hops: int, ids=None, scores=None, page_ids=None,
                 n_pages=None, stream=None, q_ns=None, sort_by_time: bool = False):
        """q: int16 [B, dim] bf16 bits.  Returns (ids int64 [B,k], scores f32 [B,k],
        page_ids int32 [B,k], n_pages int32 [B]); outputs are allocated unless given.
        q_ns (int32 [B] device tensor) scopes each query to its namespace;
        sort_by_time returns the winners in ascending chunk ID."""
        torch = self._torch
        self._dev(q, torch.int16, "q")
        B = q.shape[0]
        dev = q.device
        if ids is None:
            ids = torch.empty((B, k), dtype=torch.int64, device=dev)
        if scores is None:
            scores = torch.empty((B, k), dtype=torch.float32, device=dev)
        if page_ids is None:
            page_ids = torch.empty((B, k), dtype=torch.int32, device=dev)
        if n_pages is None:
            n_pages = torch.empty((B,), dtype=torch.int32, device=dev)
        self._dev(ids, torch.int64, "ids", B * k)
        self._dev(scores, torch.float32, "scores", B * k)
        self._dev(page_ids, torch.int32, "page_ids", B * k)
        self._dev(n_pages, torch.int32, "n_pages", B)
        if q_ns is None and not sort_by_time:
            _check(load_library().akashic_mem_retrieve(
                self._h, _ptr(q), B, k, float(alpha), hops, _ptr(ids), _ptr(scores),
                _ptr(page_ids), _ptr(n_pages), _stream(torch, stream, self.device)))
        else:
            if q_ns is not None:
                self._dev(q_ns, torch.int32, "q_ns", B)
            _check(load_library().akashic_mem_retrieve_scoped(
                self._h, _ptr(q), B, k, float(alpha), hops,
                None if q_ns is None else _ptr(q_ns), int(bool(sort_by_time)), _ptr(ids),
                _ptr(scores), _ptr(page_ids), _ptr(n_pages), _stream(torch, stream, self.device)))
        return ids, scores, page_ids, n_pages

    def size(self):
        n, e = ctypes.c_int64(), ctypes.c_int64()
        _check(load_library().akashic_mem_size(self._h, ctypes.byref(n), ctypes.byref(e)))
        return n.value, e.value

    def export_csr(self, stream=None):
        torch = self._torch
        n, e = ctypes.c_int64(), ctypes.c_int64()
        lib = load_library()
        st = _stream(torch, stream, self.device)
        _check(lib.akashic_mem_export_csr(self._h, ctypes.byref(n), ctypes.byref(e), None, None,
                                          None, None, st))
        dev = torch.device("cuda", self.device)
        rp = torch.empty(n.value + 1, dtype=torch.int64, device=dev)
        col = torch.empty(max(e.value, 1), dtype=torch.int32, device=dev)
        aff = torch.empty(max(e.value, 1), dtype=torch.float32, device=dev)
        w = torch.empty(max(e.value, 1), dtype=torch.float32, device=dev)
        _check(lib.akashic_mem_export_csr(self._h, ctypes.byref(n), ctypes.byref(e), _ptr(rp),
                                          _ptr(col), _ptr(aff), _ptr(w), st))
        return rp, col[:e.value], aff[:e.value], w[:e.value]

    def sync(self, stream=None):
        _check(load_library().akashic_mem_sync(self._h, _stream(self._torch, stream, self.device)))

    def check_wait_timeout(self, polls: int, stream=None):
        """Queue the bounded-wait self-check: the next sync() raises ETIMEOUT."""
        _check(load_library().akashic_mem_check_wait_timeout(
            self._h, int(polls), _stream(self._torch, stream, self.device)))

    def set_profiling(self, on: bool):
        _check(load_library().akashic_mem_set_profiling(self._h, int(bool(on))))

    def phase_times(self):
        ms = (ctypes.c_float * len(PHASES))()
        ln = (ctypes.c_int32 * len(PHASES))()
        _check(load_library().akashic_mem_phase_times(self._h, ms, ln))
        return {p: (ms[i], ln[i]) for i, p in enumerate(PHASES)}
