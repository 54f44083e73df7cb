"""CPU oracle for the Akashic MemAttention dense-surrogate hot path.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may use it; the product library never does.

Thin ctypes wrapper around ``akashic_oracle.c`` (plain single-threaded fp64
C, compiled with gcc -O2 and no fast-math).  The C file states what is
computed and which passages of arXiv 2607.05708 each step follows: the
softmax score over chunks and top-k selection of query-aware retrieval
(§4.1, Algorithm 1, in its Dense-only form, §5.5), relation propagation
along cross-chunk relations (§4.1), page resolve and distinct-page count
(FetchByID in Algorithm 1; the locality gap |P(R_t)| of §3.2) and the
relation update that selects related prior chunks for each new chunk
(Algorithm 1, compaction half).

Pins (tests/test_oracle_pins.py): a hand-worked three-chunk example
(tests/golden), dense matrix-power closed forms, mass conservation,
identity/uniform graphs, alpha=0 reduction to an argsort, permutation and
placement invariance, forced ties, page-count bounds and the relation update's
duplicate-chunk and CSR well-formedness properties.  Every function here is
pinned; none is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "akashic_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (portable flags; no -march, no fast-math)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
                        "-ffp-contract=off", "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i64, i32, f64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
            lib.ora_row_softmax.argtypes = [i64, P, P, P]
            lib.ora_row_softmax.restype = ctypes.c_int
            lib.ora_retrieve.argtypes = [P, i64, i32, P, i32, P, P, P, f64, f64, i32, i32, P,
                                         P, P, P, P, P, P, P]
            lib.ora_retrieve.restype = ctypes.c_int
            lib.ora_retrieve_scoped.argtypes = [P, i64, i32, P, i32, P, P, P, f64, f64, i32, i32,
                                                P, P, P, P, i32, P, P, P, P, P]
            lib.ora_retrieve_scoped.restype = ctypes.c_int
            lib.ora_drop_dead.argtypes = [i64, P, P, P, P, P, P, P]
            lib.ora_drop_dead.restype = ctypes.c_int
            lib.ora_update_relations.argtypes = [P, i32, i64, i64, i32, f64, i32, P, P, P, P, P, P,
                                                 P, P]
            lib.ora_update_relations.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _check(rc, what):
    if rc == 1:
        raise ValueError(f"oracle {what}: invalid argument")
    if rc == 2:
        raise MemoryError(f"oracle {what}: out of memory")
    if rc != 0:
        raise RuntimeError(f"oracle {what}: status {rc}")


def row_softmax(row_ptr: np.ndarray, aff: np.ndarray) -> np.ndarray:
    """Relation weights w = softmax of each row's edge logits (fp64)."""
    row_ptr = np.ascontiguousarray(row_ptr, dtype=np.int64)
    aff = np.ascontiguousarray(aff, dtype=np.float32)
    w = np.zeros(aff.shape[0], dtype=np.float64)
    _check(_load().ora_row_softmax(row_ptr.shape[0] - 1, _ptr(row_ptr), _ptr(aff), _ptr(w)),
           "row_softmax")
    return w


def retrieve(emb, queries, row_ptr, col, w, *, tau, alpha, hops, k, page_of=None,
             want_final=False, ns_of=None, q_ns=None, sort_by_time=False, dead=None):
    """Score -> propagate -> top-k -> page resolve for every query (fp64).

    Returns dict(ids int64[B,k], scores float64[B,k], page_ids int32[B,k],
    n_pages int32[B], z float64[B], shift float64[B], final float64[B,N] if
    want_final).  With ns_of (int32[N], a namespace tag per chunk) and q_ns
    (int32[B]) query b selects only among chunks tagged q_ns[b] (padding:
    ID -1, score 0, page -1; z and shift are then not reported); with
    sort_by_time the selected IDs come in ascending ID order (§4.1,
    Algorithm 1: namespace-scoped candidates, SortByTime).  With dead
    (bool[N]) deleted chunks get no score and are never selected."""
    if ns_of is not None or q_ns is not None or sort_by_time or dead is not None:
        return _retrieve_scoped(emb, queries, row_ptr, col, w, tau=tau, alpha=alpha, hops=hops,
                                k=k, page_of=page_of, want_final=want_final, ns_of=ns_of,
                                q_ns=q_ns, sort_by_time=sort_by_time, dead=dead)
    emb = np.ascontiguousarray(emb, dtype=np.uint16)
    queries = np.ascontiguousarray(queries, dtype=np.uint16)
    n, d = emb.shape
    b = queries.shape[0]
    if row_ptr is not None:
        row_ptr = np.ascontiguousarray(row_ptr, dtype=np.int64)
        col = np.ascontiguousarray(col, dtype=np.int32)
        w = np.ascontiguousarray(w, dtype=np.float64)
    if page_of is not None:
        page_of = np.ascontiguousarray(page_of, dtype=np.int32)
    out = dict(
        ids=np.zeros((b, k), np.int64), scores=np.zeros((b, k), np.float64),
        page_ids=np.zeros((b, k), np.int32), n_pages=np.zeros(b, np.int32),
        z=np.zeros(b, np.float64), shift=np.zeros(b, np.float64),
    )
    final = np.zeros((b, n), np.float64) if want_final else None
    rc = _load().ora_retrieve(
        _ptr(emb), n, d, _ptr(queries), b, _ptr(row_ptr), _ptr(col), _ptr(w),
        float(tau), float(alpha), int(hops), int(k), _ptr(page_of), _ptr(out["ids"]),
        _ptr(out["scores"]), _ptr(out["page_ids"]), _ptr(out["n_pages"]), _ptr(final),
        _ptr(out["z"]), _ptr(out["shift"]))
    _check(rc, "retrieve")
    if final is not None:
        out["final"] = final
    return out


def _retrieve_scoped(emb, queries, row_ptr, col, w, *, tau, alpha, hops, k, page_of, want_final,
                     ns_of, q_ns, sort_by_time, dead):
    emb = np.ascontiguousarray(emb, dtype=np.uint16)
    queries = np.ascontiguousarray(queries, dtype=np.uint16)
    n, d = emb.shape
    b = queries.shape[0]
    if row_ptr is not None:
        row_ptr = np.ascontiguousarray(row_ptr, dtype=np.int64)
        col = np.ascontiguousarray(col, dtype=np.int32)
        w = np.ascontiguousarray(w, dtype=np.float64)
    if page_of is not None:
        page_of = np.ascontiguousarray(page_of, dtype=np.int32)
    if (ns_of is None) != (q_ns is None):
        raise ValueError("ns_of and q_ns go together")
    if ns_of is not None:
        ns_of = np.ascontiguousarray(ns_of, dtype=np.int32)
        q_ns = np.ascontiguousarray(q_ns, dtype=np.int32)
    if dead is not None:
        dead = np.ascontiguousarray(dead, dtype=np.uint8)
    out = dict(ids=np.zeros((b, k), np.int64), scores=np.zeros((b, k), np.float64),
               page_ids=np.zeros((b, k), np.int32), n_pages=np.zeros(b, np.int32))
    final = np.zeros((b, n), np.float64) if want_final else None
    rc = _load().ora_retrieve_scoped(
        _ptr(emb), n, d, _ptr(queries), b, _ptr(row_ptr), _ptr(col), _ptr(w), float(tau),
        float(alpha), int(hops), int(k), _ptr(page_of), _ptr(ns_of), _ptr(q_ns), _ptr(dead),
        int(bool(sort_by_time)), _ptr(out["ids"]), _ptr(out["scores"]), _ptr(out["page_ids"]),
        _ptr(out["n_pages"]), _ptr(final))
    _check(rc, "retrieve_scoped")
    if final is not None:
        out["final"] = final
    return out


def drop_dead(row_ptr, col, aff, dead):
    """The CSR without every edge into or out of a deleted chunk (dead bool[N])."""
    row_ptr = np.ascontiguousarray(row_ptr, dtype=np.int64)
    col = np.ascontiguousarray(col, dtype=np.int32)
    aff = np.ascontiguousarray(aff, dtype=np.float32)
    dead = np.ascontiguousarray(dead, dtype=np.uint8)
    n = row_ptr.shape[0] - 1
    rp = np.zeros(n + 1, np.int64)
    c = np.zeros(max(col.shape[0], 1), np.int32)
    a = np.zeros(max(col.shape[0], 1), np.float32)
    _check(_load().ora_drop_dead(n, _ptr(row_ptr), _ptr(col), _ptr(aff), _ptr(dead), _ptr(rp),
                                 _ptr(c), _ptr(a)), "drop_dead")
    return rp, c[:rp[-1]], a[:rp[-1]]


def update_relations(emb, first, n_new, m, row_ptr, col, aff, *, scale=10.0, reciprocal=True):
    """Top-M prior neighbours of chunks [first, first+n_new) and the new CSR.

    `emb` holds at least first+n_new rows; the CSR has first+n_new rows with
    rows >= first empty.  Returns dict(row_ptr, col, aff, nbr_ids[n_new,M],
    nbr_cos[n_new,M])."""
    emb = np.ascontiguousarray(emb, dtype=np.uint16)
    d = emb.shape[1]
    row_ptr = np.ascontiguousarray(row_ptr, dtype=np.int64)
    col = np.ascontiguousarray(col, dtype=np.int32)
    aff = np.ascontiguousarray(aff, dtype=np.float32)
    n_rows = first + n_new
    if row_ptr.shape[0] != n_rows + 1:
        raise ValueError("row_ptr must have first+n_new+1 entries")
    cap = int(row_ptr[-1]) + n_new * m * (2 if reciprocal else 1)
    new_row_ptr = np.zeros(n_rows + 1, np.int64)
    new_col = np.zeros(max(cap, 1), np.int32)
    new_aff = np.zeros(max(cap, 1), np.float32)
    nbr_ids = np.zeros((n_new, m), np.int64)
    nbr_cos = np.zeros((n_new, m), np.float64)
    rc = _load().ora_update_relations(
        _ptr(emb), d, int(first), int(n_new), int(m), float(scale), int(bool(reciprocal)),
        _ptr(row_ptr), _ptr(col), _ptr(aff), _ptr(new_row_ptr), _ptr(new_col), _ptr(new_aff),
        _ptr(nbr_ids), _ptr(nbr_cos))
    _check(rc, "update_relations")
    nnz = int(new_row_ptr[-1])
    return dict(row_ptr=new_row_ptr, col=new_col[:nnz].copy(), aff=new_aff[:nnz].copy(),
                nbr_ids=nbr_ids, nbr_cos=nbr_cos)
