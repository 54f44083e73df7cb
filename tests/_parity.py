"""Parity helpers: run a synthetic workload through the CUDA library and the
oracle on the same inputs and compare element by element.

Tolerances (written here, used by every parity test):
  * Selected IDs, page IDs and page counts are compared exactly, except that
    an ID may be swapped for another whose ORACLE score lies within the
    near-tie band |s - s_k| <= SWAP_REL * max(s, s_k) of the oracle's k-th
    score (every softmax score is about 1/N, so the band is relative; a
    relative 1e-4 is a logit difference of 1e-4), and the order inside the
    list may differ only among such near-ties.
  * Page IDs must equal the page table applied to the GPU's own IDs and the
    page count must equal the number of distinct ones: bit-exact.
  * Each GPU score is within SCORE_REL (2e-3) of the oracle's fp64 score of
    the same chunk.
  * Relation update: neighbour lists exact except swaps whose oracle cosines
    differ by < COS_ABS (1e-4) at the M-th/(M+1)-th boundary; the CSR
    (row pointers, columns) exactly equal after those swaps; logits within
    1e-5 absolute of scale * fp64 cosine; weights within 2e-3 relative.
"""
from __future__ import annotations

import numpy as np

import oracle

SWAP_REL = 1e-4
SCORE_REL = 2e-3
COS_ABS = 1e-4


# --------------------------------------------------------------------------- retrieval
def gpu_store(wl, placement, capacity=None):
    from paper_2607_05708_gb300 import MemStore
    return MemStore.from_arrays(wl.emb, wl.page_of[placement], wl.row_ptr, wl.col, wl.aff,
                                capacity=capacity or wl.n, chunks_per_page=wl.chunks_per_page,
                                temperature=wl.tau)


def gpu_retrieve(wl, placement, store=None, queries=None, k=None, alpha=None, hops=None):
    import torch
    if store is None:
        store = gpu_store(wl, placement)
    q = wl.queries if queries is None else queries
    qt = torch.from_numpy(np.ascontiguousarray(q).view(np.int16)).cuda()
    ids, sc, pg, npg = store.retrieve(qt, k or wl.k, wl.alpha if alpha is None else alpha,
                                      wl.hops if hops is None else hops)
    store.sync()
    return store, dict(ids=ids.cpu().numpy(), scores=sc.cpu().numpy(), page_ids=pg.cpu().numpy(),
                       n_pages=npg.cpu().numpy())


def oracle_weights(wl):
    # cached on the workload object itself (a dataclasses.replace copy starts
    # without it); an id()-keyed cache could hand a new object the weights of
    # a freed one whose id it reuses
    w = wl.__dict__.get("_oracle_w")
    if w is None:
        w = oracle.row_softmax(wl.row_ptr, wl.aff)
        wl.__dict__["_oracle_w"] = w
    return w


def oracle_retrieve(wl, placement, queries=None, k=None, alpha=None, hops=None):
    q = wl.queries if queries is None else queries
    return oracle.retrieve(wl.emb, q, wl.row_ptr, wl.col, oracle_weights(wl), tau=wl.tau,
                           alpha=wl.alpha if alpha is None else alpha,
                           hops=wl.hops if hops is None else hops, k=k or wl.k,
                           page_of=wl.page_of[placement], want_final=True)


def oracle_retrieve_rows(wl, placement, rows, threads=None):
    """The oracle on the query rows `rows`, a few rows per host thread (the
    oracle's C code releases the interpreter lock; each call is the plain
    single-threaded oracle on its rows).  Same dict as oracle_retrieve."""
    import os
    from concurrent.futures import ThreadPoolExecutor
    rows = list(rows)
    oracle_weights(wl)                         # once, before the threads
    threads = max(1, min(len(rows), threads or os.cpu_count() or 1))
    parts = [rows[i::threads] for i in range(threads)]
    with ThreadPoolExecutor(max_workers=threads) as ex:
        outs = list(ex.map(lambda r: oracle_retrieve(wl, placement, queries=wl.queries[r]),
                           parts))
    order = np.argsort(np.concatenate([np.asarray(p) for p in parts]), kind="stable")
    return {key: np.concatenate([o[key] for o in outs])[order] for key in outs[0]}


def assert_retrieval_parity(wl, placement, got, ref, rows=None):
    """got: GPU outputs (row r of got = query rows[r] of ref if rows is given)."""
    page_of = wl.page_of[placement]
    k = ref["ids"].shape[1]
    n_rows = got["ids"].shape[0] if rows is None else len(rows)
    for r in range(n_rows):
        b = r if rows is None else rows[r]
        gi = got["ids"][r].astype(np.int64)
        oi = ref["ids"][b]
        fin = ref["final"][b]
        assert len(set(gi.tolist())) == k, f"query {b}: repeated IDs {gi}"
        assert (gi >= 0).all() and (gi < wl.n).all(), f"query {b}: ID out of range"
        sk = ref["scores"][b][k - 1]
        band = lambda s: abs(s - sk) <= SWAP_REL * max(abs(s), abs(sk))
        for x in set(gi.tolist()) ^ set(oi.tolist()):
            assert band(fin[x]), (f"query {b}: chunk {x} (oracle score {fin[x]!r}) swapped "
                                  f"outside the near-tie band of the k-th score {sk!r}")
        s_gpu_ids = fin[gi]
        for a in range(k - 1):
            hi, lo = s_gpu_ids[a], s_gpu_ids[a + 1]
            assert hi >= lo - SWAP_REL * max(abs(hi), abs(lo)), (
                f"query {b}: order differs beyond near-ties at {a}: {hi!r} < {lo!r}")
        rel = np.abs(got["scores"][r].astype(np.float64) - fin[gi]) / np.abs(fin[gi])
        assert rel.max() <= SCORE_REL, f"query {b}: score error {rel.max():.3g} > {SCORE_REL}"
        assert (got["page_ids"][r] == page_of[gi]).all(), f"query {b}: page IDs differ"
        assert got["n_pages"][r] == len(set(page_of[gi].tolist())), f"query {b}: page count"
        assert got["n_pages"][r] == ref["n_pages"][b] or set(gi.tolist()) != set(oi.tolist())


def assert_scoped_parity(wl, placement, got, ref, ns_of, q_ns, sort_by_time):
    """Namespace-scoped retrieval: every real ID lies in the query's
    namespace, the real IDs equal the oracle's up to near-tie swaps at the
    k-th in-namespace score, padding (-1) exactly where the oracle pads, the
    order is by score (up to near-ties) or, with SortByTime, by ascending ID;
    scores, page IDs and page counts as in assert_retrieval_parity."""
    page_of = wl.page_of[placement]
    k = ref["ids"].shape[1]
    for b in range(got["ids"].shape[0]):
        gi = got["ids"][b].astype(np.int64)
        oi = ref["ids"][b]
        fin = ref["final"][b]
        nv = int((oi >= 0).sum())
        assert (gi[nv:] == -1).all() and (gi[:nv] >= 0).all(), f"query {b}: padding {gi}"
        assert (got["page_ids"][b][nv:] == -1).all(), f"query {b}: padding pages"
        g, o = gi[:nv], oi[:nv]
        assert len(set(g.tolist())) == nv, f"query {b}: repeated IDs"
        assert (ns_of[g] == q_ns[b]).all(), f"query {b}: ID outside namespace {q_ns[b]}"
        if nv:
            sk = ref["scores"][b][:nv].min()
            for x in set(g.tolist()) ^ set(o.tolist()):
                assert abs(fin[x] - sk) <= SWAP_REL * max(abs(fin[x]), abs(sk)), (
                    f"query {b}: chunk {x} swapped outside the near-tie band")
        if sort_by_time:
            assert (np.diff(g) > 0).all(), f"query {b}: not in ascending ID order {g}"
        else:
            sg = fin[g]
            for a in range(nv - 1):
                assert sg[a] >= sg[a + 1] - SWAP_REL * max(abs(sg[a]), abs(sg[a + 1])), (
                    f"query {b}: score order differs at {a}")
        if nv:
            rel = np.abs(got["scores"][b][:nv].astype(np.float64) - fin[g]) / np.abs(fin[g])
            assert rel.max() <= SCORE_REL, f"query {b}: score error {rel.max():.3g}"
        assert (got["page_ids"][b][:nv] == page_of[g]).all(), f"query {b}: page IDs differ"
        assert got["n_pages"][b] == len(set(page_of[g].tolist())), f"query {b}: page count"


# --------------------------------------------------------------------------- relation update
def check_update(wl, sample=None, M=None, seed=0, golden=None):
    """Append wl.new_emb to a store holding wl, run the update on the GPU and
    compare with the oracle: all new rows (the oracle run here, or its
    stored result `golden` = dict(nbr_ids, nbr_cos) for every new chunk),
    or a seeded sample of them."""
    import torch
    from paper_2607_05708_gb300 import MemStore
    M = M or wl.top_m
    n_old, n_new = wl.n, wl.new_emb.shape[0]
    store = MemStore.from_arrays(wl.emb, wl.page_of["clustered"], wl.row_ptr, wl.col, wl.aff,
                                 capacity=n_old + n_new, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau, relation_scale=wl.relation_scale)
    new = torch.from_numpy(np.ascontiguousarray(wl.new_emb).view(np.int16)).cuda()
    first = store.append_chunks(new)
    assert first == n_old
    store.update_relations(first, n_new, M, reciprocal=wl.reciprocal)
    store.sync()
    rp, col, aff, w = (t.cpu().numpy() for t in store.export_csr())
    if golden is not None:
        _compare_update(wl, M, rp, col, aff, w, golden, np.arange(n_new), full=True)
    elif sample is None:
        all_emb = np.concatenate([wl.emb, wl.new_emb])
        old_rp = np.concatenate([wl.row_ptr, np.full(n_new, wl.row_ptr[-1], np.int64)])
        ref = oracle.update_relations(all_emb, n_old, n_new, M, old_rp, wl.col, wl.aff,
                                      scale=wl.relation_scale, reciprocal=wl.reciprocal)
        _compare_update(wl, M, rp, col, aff, w, ref, np.arange(n_new), full=True)
    else:
        rng = np.random.default_rng(seed)
        picks = np.sort(rng.choice(n_new, size=min(sample, n_new), replace=False))
        # oracle on the sampled new chunks only (each is independent of the others)
        sub_emb = np.concatenate([wl.emb, wl.new_emb[picks]])
        old_rp = np.concatenate([wl.row_ptr, np.full(len(picks), wl.row_ptr[-1], np.int64)])
        ref = oracle.update_relations(sub_emb, n_old, len(picks), M, old_rp, wl.col, wl.aff,
                                      scale=wl.relation_scale, reciprocal=wl.reciprocal)
        _compare_update(wl, M, rp, col, aff, w, ref, picks, full=False)
    return store


def _cosines(wl, nids, cols):
    """fp64 <e_nid, e_col> of the widened stored values, pair by pair."""
    all_emb = (wl.emb, wl.new_emb)
    n_old = wl.n

    def rows(ids):
        ids = np.asarray(ids, np.int64)
        out = np.empty((ids.size, wl.dim), np.uint16)
        old = ids < n_old
        out[old] = all_emb[0][ids[old]]
        out[~old] = all_emb[1][ids[~old] - n_old]
        return oracle_free_widen(out)

    res = np.empty(len(nids), np.float64)
    for s in range(0, len(nids), 16384):
        a, b = rows(nids[s:s + 16384]), rows(cols[s:s + 16384])
        res[s:s + 16384] = np.einsum("ij,ij->i", a, b)
    return res


def _compare_update(wl, M, rp, col, aff, w, ref, picks, full):
    """The picked new rows against the oracle's selection (swaps only among
    near-ties at the M-th cosine), logits = scale * fp64 cosine, reciprocal
    edges.  With `full`, every row of the exported CSR against the oracle's
    CSR with those recorded swaps applied: the old edges of every row in
    place and bit-exact, then the reciprocal edges of the new chunks that
    chose the row, in ascending ID order; each new row its M neighbours in
    ascending ID order; row pointers equal throughout."""
    n_old, n_new = wl.n, len(wl.new_emb)
    scale = wl.relation_scale
    assert (np.diff(rp) >= 0).all()
    assert rp[-1] == wl.row_ptr[-1] + n_new * M * (2 if wl.reciprocal else 1)
    nid_all = n_old + np.asarray(picks, np.int64)
    g_nbr = np.stack([col[rp[nid]:rp[nid + 1]] for nid in nid_all]).astype(np.int64)
    assert g_nbr.shape == (len(picks), M), "a new row does not hold M neighbours"
    assert (np.diff(g_nbr, axis=1) > 0).all() and (g_nbr < n_old).all()
    swaps = 0
    for t, nid in enumerate(nid_all):
        o_ids = np.asarray(ref["nbr_ids"][t], np.int64)
        kth = float(ref["nbr_cos"][t][M - 1])
        diff = sorted(set(g_nbr[t].tolist()) ^ set(o_ids.tolist()))
        if diff:
            cx = _cosines(wl, np.full(len(diff), nid), np.array(diff))
            for x, c in zip(diff, cx):
                assert abs(c - kth) < COS_ABS, f"new chunk {nid}: neighbour {x} swapped ({c} vs {kth})"
            swaps += len(diff) // 2
    # logits of the new rows = scale * fp64 cosine; reciprocal edges carry the same
    fwd_pos = np.concatenate([np.arange(rp[nid], rp[nid + 1]) for nid in nid_all])
    cx = _cosines(wl, np.repeat(nid_all, M), g_nbr.ravel())
    lg = aff[fwd_pos].astype(np.float64)
    assert (np.abs(lg - scale * cx) <= 1e-5 * np.maximum(1.0, np.abs(scale * cx))).all(), \
        "new-row logits differ from scale * cos"
    if wl.reciprocal:
        for t, nid in enumerate(nid_all):
            for x, l in zip(g_nbr[t], aff[rp[nid]:rp[nid + 1]]):
                row = col[rp[x]:rp[x + 1]]
                pos = np.searchsorted(row, nid)
                assert pos < len(row) and row[pos] == nid, f"missing reciprocal edge {x}->{nid}"
                assert aff[rp[x] + pos] == l
    # weights: row softmax of the exported logits
    wr = oracle.row_softmax(rp, aff)
    assert np.allclose(w, wr, rtol=2e-3, atol=0)
    if not full:
        return swaps
    # the whole CSR, row by row (vectorised)
    orig_len = np.diff(wl.row_ptr)
    js = g_nbr.ravel()
    nids = np.repeat(nid_all, M)
    cnt = np.bincount(js, minlength=n_old) if wl.reciprocal else np.zeros(n_old, np.int64)
    exp_len = np.concatenate([orig_len + cnt, np.full(n_new, M, np.int64)])
    exp_rp = np.concatenate([[0], np.cumsum(exp_len)])
    assert (rp == exp_rp).all(), "row pointers differ from the oracle's CSR with its swaps"
    exp_col = np.full(exp_rp[-1], -1, np.int64)
    owner = np.repeat(np.arange(n_old), orig_len)
    old_pos = exp_rp[owner] + (np.arange(wl.row_ptr[-1]) - wl.row_ptr[owner])
    exp_col[old_pos] = wl.col
    if wl.reciprocal:
        order = np.lexsort((nids, js))
        js_s, nid_s = js[order], nids[order]
        rank = np.arange(js_s.size) - np.searchsorted(js_s, js_s, side="left")
        exp_col[exp_rp[js_s] + orig_len[js_s] + rank] = nid_s
    exp_col[fwd_pos] = js
    assert (exp_col >= 0).all()
    bad = np.nonzero(col != exp_col)[0]
    assert bad.size == 0, f"{bad.size} CSR columns differ, first at edge {bad[:5]}"
    assert (aff[old_pos] == wl.aff).all(), "old edges' logits changed"
    if swaps == 0 and "row_ptr" in ref:
        assert (ref["row_ptr"] == rp).all() and (ref["col"] == col).all()
        assert np.allclose(aff, ref["aff"], rtol=1e-5, atol=1e-5)
    return swaps


def oracle_free_widen(h):
    """fp64 values of bf16 bits (plain widening, used for the test's own checks)."""
    return ((np.ascontiguousarray(h).astype(np.uint32) << 16).view(np.float32)).astype(np.float64)
