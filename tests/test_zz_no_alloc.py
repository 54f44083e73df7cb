"""The allocation-free score entry point, against the oracle and against the
store's retrieval.

akashic_mem_softmax_scores_noalloc is for callers that cannot allocate
device memory at the moment they need scores: a serving runtime that works
inside a memory pool it reserved up front, code recording work into a
stream capture, or a host without a device allocator.  It computes the
softmax scores over caller-owned buffers with a fixed scratch array.  Each
case calls it through the C ABI twice in a row on the same inputs and
checks both results:
  * per element against the oracle's fp64 softmax (oracle.retrieve with
    hops = 0, want_final=True): u[j, b] / z[b] within 2e-3 relative of
    s0[b, j]; and z[b] exp(shift[b]) against the oracle's Z exp(c_b) (both
    equal the sum of exp(tau <q_b, e_j>) whatever shift each side takes),
    compared as logarithms;
  * against akashic_mem_retrieve (hops = 0), the existing entry point whose
    first step is the same score kernel, with the parity tolerances of the
    other GPU tests;
  * that the call allocates nothing: torch's allocator and the device's
    free memory are unchanged across the second call.
It sits in a file of its own that pytest collects last, and needs no state
from the other tests.
"""
import ctypes

import numpy as np
import pytest

import oracle
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


def _padded(queries, width):
    """The queries followed by zero rows up to `width` (the call takes 32,
    64, 128 or 256 queries)."""
    out = np.zeros((width, queries.shape[1]), np.uint16)
    out[:queries.shape[0]] = queries
    return out


@pytest.mark.parametrize("cfg,scale,width", [(0, 1.0, 32), (1, 1 / 16, 64)],
                         ids=["tiny-4096x256", "gmm65k-recipe-4096x768"])
def test_noalloc_scores_match_oracle_and_retrieve_twice(cfg, scale, width):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_05708_gb300 import MemStore, _build, load_library
    _build.build()
    lib = load_library()
    wl = synth.workload(cfg, scale=scale)
    k = wl.k
    n, nq = wl.n, wl.n_queries
    qpad = _padded(wl.queries, width)
    dev = torch.device("cuda", 0)
    emb = torch.from_numpy(wl.emb.view(np.int16)).to(dev)
    q = torch.from_numpy(qpad.view(np.int16)).to(dev)

    # the oracle: fp64 softmax over the store, no relations
    ref = oracle.retrieve(wl.emb, wl.queries, None, None, None, tau=wl.tau, alpha=0.0, hops=0,
                          k=k, want_final=True)
    log_total = np.log(ref["z"]) + ref["shift"]          # log sum_j exp(tau <q_b, e_j>)

    # existing entry point: a store in ID order, no relations, plain top-k
    store = MemStore.from_arrays(wl.emb, None, capacity=n, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau)
    ref_ids, ref_sc, _, _ = store.retrieve(q[:nq], k, 0.0, 0)
    store.sync()
    ref_ids = ref_ids.cpu().numpy()
    ref_sc = ref_sc.cpu().numpy().astype(np.float64)

    u = torch.empty((n, width), dtype=torch.float32, device=dev)
    z = torch.empty((width,), dtype=torch.float32, device=dev)
    shift = torch.empty((width,), dtype=torch.float32, device=dev)
    status = torch.full((1,), -1, dtype=torch.int32, device=dev)
    stream = ctypes.c_void_p(torch.cuda.current_stream(dev).cuda_stream)
    for call in range(2):
        u.fill_(float("nan"))
        z.fill_(float("nan"))
        torch.cuda.synchronize()
        alloc0, free0 = torch.cuda.memory_allocated(dev), torch.cuda.mem_get_info(dev)[0]
        rc = lib.akashic_mem_softmax_scores_noalloc(
            ctypes.c_void_p(emb.data_ptr()), n, wl.dim, ctypes.c_void_p(q.data_ptr()), width,
            float(wl.tau), ctypes.c_void_p(u.data_ptr()), ctypes.c_void_p(z.data_ptr()),
            ctypes.c_void_p(shift.data_ptr()), ctypes.c_void_p(status.data_ptr()), stream)
        assert rc == 0, lib.akashic_mem_last_error()
        torch.cuda.synchronize()
        if call == 1:
            # the first call may load kernels; the second allocates nothing
            assert torch.cuda.memory_allocated(dev) == alloc0
            assert torch.cuda.mem_get_info(dev)[0] == free0
        assert int(status.item()) == 0
        un, zn, sn = u.cpu().numpy()[:, :nq], z.cpu().numpy()[:nq], shift.cpu().numpy()[:nq]
        assert np.isfinite(un).all() and np.isfinite(zn).all()

        # 1. the oracle, element by element
        s0 = un.astype(np.float64) / zn.astype(np.float64)
        rel = np.abs(s0 - ref["final"].T) / ref["final"].T
        assert rel.max() <= SCORE_REL, f"call {call}: softmax error {rel.max():.3g}"
        dlog = np.abs(np.log(zn.astype(np.float64)) + sn.astype(np.float64) - log_total)
        assert dlog.max() <= np.log1p(SCORE_REL), f"call {call}: Z exp(c) differs by {dlog.max():.3g}"

        # 2. the store's retrieval (same score kernel): same top-k up to near-ties
        ids, sc = _host_topk(un, zn, k)
        for b in range(nq):
            got, want = set(ids[b].tolist()), set(ref_ids[b].tolist())
            kth = ref_sc[b][k - 1]
            for x in got ^ want:
                s = float(un[x, b]) / float(zn[b])
                assert abs(s - kth) <= SWAP_REL * max(s, kth), f"call {call}, query {b}: chunk {x}"
            mine = {i: v for i, v in zip(ids[b], sc[b])}
            theirs = {i: v for i, v in zip(ref_ids[b], ref_sc[b])}
            for i in sorted(got & want):
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
