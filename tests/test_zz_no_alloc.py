"""The allocation-free score entry point against the store's retrieval.

akashic_mem_softmax_scores_noalloc serves callers that cannot allocate
device memory when they need scores (graph capture, a serving runtime's
fixed memory pool, hosts without a device allocator): it computes the
softmax scores over caller-owned buffers with a fixed scratch array.  This
test calls it through the C ABI twice in a row on the same inputs and
checks both results against akashic_mem_retrieve (hops = 0), the existing
entry point whose first step is the same score kernel, with the parity
tolerances of the other GPU tests.  It sits in a file of its own that pytest
collects last, and needs no state from the other tests.
"""
import ctypes

import numpy as np
import pytest

import synth
from _parity import SCORE_REL, SWAP_REL

pytestmark = pytest.mark.gpu


def _host_topk(u, z, k):
    """Top-k of u[:, b] / z[b] by (score desc, chunk ID asc), per query."""
    n, B = u.shape
    ids = np.empty((B, k), np.int64)
    sc = np.empty((B, k), np.float64)
    for b in range(B):
        order = np.lexsort((np.arange(n), -u[:, b]))[:k]
        ids[b] = order
        sc[b] = u[order, b].astype(np.float64) / float(z[b])
    return ids, sc


def test_noalloc_scores_match_retrieve_twice():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_05708_gb300 import MemStore, _build, load_library
    _build.build()
    lib = load_library()
    wl = synth.workload(1, scale=1 / 16)              # N=4096, d=768, B=64 queries, k=16
    k = wl.k
    dev = torch.device("cuda", 0)
    emb = torch.from_numpy(wl.emb.view(np.int16)).to(dev)
    q = torch.from_numpy(wl.queries.view(np.int16)).to(dev)
    n, B = wl.n, wl.n_queries
    # existing entry point: a store in ID order, no relations, plain top-k
    store = MemStore.from_arrays(wl.emb, None, capacity=n, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau)
    ref_ids, ref_sc, _, _ = store.retrieve(q, k, 0.0, 0)
    store.sync()
    ref_ids = ref_ids.cpu().numpy()
    ref_sc = ref_sc.cpu().numpy().astype(np.float64)

    u = torch.empty((n, B), dtype=torch.float32, device=dev)
    z = torch.empty((B,), dtype=torch.float32, device=dev)
    status = torch.full((1,), -1, dtype=torch.int32, device=dev)
    stream = ctypes.c_void_p(torch.cuda.current_stream(dev).cuda_stream)
    for call in range(2):
        u.fill_(float("nan"))
        z.fill_(float("nan"))
        rc = lib.akashic_mem_softmax_scores_noalloc(
            ctypes.c_void_p(emb.data_ptr()), n, wl.dim, ctypes.c_void_p(q.data_ptr()), B,
            float(wl.tau), ctypes.c_void_p(u.data_ptr()), ctypes.c_void_p(z.data_ptr()), None,
            ctypes.c_void_p(status.data_ptr()), stream)
        assert rc == 0, lib.akashic_mem_last_error()
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        un, zn = u.cpu().numpy(), z.cpu().numpy()
        assert np.isfinite(un).all() and np.isfinite(zn).all()
        ids, sc = _host_topk(un, zn, k)
        for b in range(B):
            got, want = set(ids[b].tolist()), set(ref_ids[b].tolist())
            kth = ref_sc[b][k - 1]
            for x in got ^ want:
                s = float(un[x, b]) / float(zn[b])
                assert abs(s - kth) <= SWAP_REL * max(s, kth), f"call {call}, query {b}: chunk {x}"
            common = sorted(got & want)
            mine = {i: v for i, v in zip(ids[b], sc[b])}
            theirs = {i: v for i, v in zip(ref_ids[b], ref_sc[b])}
            for i in common:
                assert abs(mine[i] - theirs[i]) <= SCORE_REL * abs(theirs[i])


def test_noalloc_rejects_oversized_batch():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_05708_gb300 import load_library
    lib = load_library()
    buf = torch.zeros(1 << 16, dtype=torch.float32, device="cuda")
    p = ctypes.c_void_p(buf.data_ptr())
    rc = lib.akashic_mem_softmax_scores_noalloc(p, 16, 64, p, 512, 0.0, p, p, None, None, None)
    assert rc == 1 and b"B must be" in lib.akashic_mem_last_error()
