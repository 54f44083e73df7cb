"""GPU parity: the CUDA library (through its C ABI) against the oracle on the
same seeded synthetic inputs, element by element.  Tolerances: _parity.py."""
import numpy as np
import pytest

import synth
from _parity import (assert_retrieval_parity, assert_scoped_parity, check_update, gpu_retrieve,
                     gpu_store, oracle_retrieve, oracle_retrieve_rows, oracle_weights)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_05708_gb300 import _build
    _build.build()


# --------------------------------------------------------------------------- retrieval
def test_tiny_store_full():
    """N=4096, d=256, B=4, one hop, k=8, 16 chunks per page in ID order."""
    wl = synth.workload(0)
    _, got = gpu_retrieve(wl, "id")
    ref = oracle_retrieve(wl, "id")
    assert_retrieval_parity(wl, "id", got, ref)


def test_gmm65k_scaled():
    """gmm65k recipe (exact top-16 cosine graph) at N=4096, B=64, k=16."""
    wl = synth.workload(1, scale=1 / 16)
    _, got = gpu_retrieve(wl, "component")
    ref = oracle_retrieve(wl, "component")
    assert_retrieval_parity(wl, "component", got, ref)


@pytest.mark.parametrize("placement", ["clustered", "random"])
def test_gmm1m_scaled_two_hops(placement):
    """gmm1m recipe at N=16384 (power-law in-degree: hub rows are split into
    segments), B=256, two hops, k=32, both placements."""
    wl = synth.workload(2, scale=1 / 64)
    _, got = gpu_retrieve(wl, placement)
    ref = oracle_retrieve(wl, placement)
    assert_retrieval_parity(wl, placement, got, ref)


@pytest.mark.parametrize("hops,B", [(0, 256), (2, 256), (0, 128), (2, 128), (2, 200)])
def test_pair_gemm_store(hops, B):
    """A store large enough for the score GEMM's CTA-pair form (256-row
    tiles on clusters of two, B >= 128): the gmm1m recipe at N=32768 cut to
    N=32700 (the last pair tile's odd half partly past the last row), no
    hops (the fused top-k filter in the GEMM) and two hops, query batches
    of 256, 128 and 200 (padded to 256), against the oracle."""
    base = synth.workload(2, scale=1 / 32)
    n = 32700
    keep = base.row_ptr[:n + 1]
    cols = base.col[:keep[-1]]
    ok = cols < n
    rows = np.repeat(np.arange(n), np.diff(keep))
    rp = np.concatenate([[0], np.cumsum(np.bincount(rows[ok], minlength=n))]).astype(np.int64)
    wl = synth.Workload(name="pair", dim=base.dim, emb=base.emb[:n], queries=base.queries[:B],
                        row_ptr=rp, col=cols[ok].astype(np.int32),
                        aff=base.aff[:keep[-1]][ok],
                        page_of={"clustered": base.page_of["clustered"][:n]},
                        chunks_per_page=64, alpha=base.alpha, hops=hops, k=base.k)
    assert wl.queries.shape[0] == B
    _, got = gpu_retrieve(wl, "clustered")
    ref = oracle_retrieve(wl, "clustered")
    assert_retrieval_parity(wl, "clustered", got, ref)


@pytest.mark.parametrize("B,k,hops,alpha", [
    (1, 1, 0, 0.0), (5, 64, 1, 0.5), (37, 13, 2, 0.3), (130, 32, 3, 0.7), (300, 8, 2, 0.5),
    (16, 10, 2, 0.0),
])
def test_ragged_shapes(B, k, hops, alpha):
    """Ragged N (not a tile multiple), B across padding widths and above 256
    (two batches), k from 1 to 64, hops 0..3, alpha 0."""
    base = synth.workload(2, scale=1 / 256)          # N=4096 from the gmm1m recipe
    n = 3001
    keep = base.row_ptr[:n + 1]
    cols = base.col[:keep[-1]]
    ok = cols < n
    rows = np.repeat(np.arange(n), np.diff(keep))
    rp = np.concatenate([[0], np.cumsum(np.bincount(rows[ok], minlength=n))]).astype(np.int64)
    wl = synth.Workload(name="ragged", dim=base.dim, emb=base.emb[:n],
                        queries=np.tile(base.queries, (2, 1))[:B], row_ptr=rp,
                        col=cols[ok].astype(np.int32), aff=base.aff[:keep[-1]][ok],
                        page_of={"clustered": base.page_of["clustered"][:n]},
                        chunks_per_page=64, alpha=alpha, hops=hops, k=k)
    _, got = gpu_retrieve(wl, "clustered")
    ref = oracle_retrieve(wl, "clustered")
    assert_retrieval_parity(wl, "clustered", got, ref)


def test_fused_filter_overflow_falls_back():
    """Every row with out-edges to its 8 successors (uniform weights, no
    hubs), alpha = 4, two hops, N = 16384: the last hop raises every score
    about fourfold over the previous level, so all rows clear the bound
    taken from that level's sample and the 8192-key buffer of every column
    overflows; the merge then selects from the whole final column.  The
    premise is checked on the oracle: even the k-th largest one-hop score (a
    bound at least as high as any sample's) is reached by more than 8192 rows."""
    import dataclasses
    base = synth.workload(2, scale=1 / 64)
    n = base.n
    col = np.sort((np.arange(n)[:, None] + np.arange(1, 9)[None, :]) % n, axis=1)
    wl = dataclasses.replace(base, row_ptr=np.arange(0, 8 * n + 1, 8, dtype=np.int64),
                             col=col.astype(np.int32).ravel(), aff=np.zeros(8 * n, np.float32),
                             alpha=4.0)
    q = wl.queries[:8]
    one = oracle_retrieve(wl, "clustered", queries=q, hops=1)["final"]
    ref = oracle_retrieve(wl, "clustered", queries=q)
    kth1 = -np.sort(-one, axis=1)[:, wl.k - 1]
    assert ((ref["final"] >= kth1[:, None]).sum(axis=1) > 8192).all()
    _, got = gpu_retrieve(wl, "clustered", queries=q)
    assert_retrieval_parity(wl, "clustered", got, ref)


@pytest.mark.parametrize("hops,k", [(1, 32), (2, 32), (2, 1), (3, 8), (2, 64)])
def test_last_hop_row_bounds_change_nothing(hops, k, monkeypatch):
    """The last hop skips every row whose upper bound (propagated from u's
    row extremes, widened by the fp32 rounding of each level) stays below a
    floor that every query's k-th largest final score reaches.  The selected
    IDs, pages and page counts must equal those computed without the skip,
    and the oracle's (gmm1m recipe at N = 16384, hub rows split).  Scores may
    differ in the last bits only: without the skip more rows clear the
    filter's sample bound, a query's buffer can overflow, and its column is
    then recomputed by the merge with another summation order.  The two-hop
    path from reach coefficients is switched off in both runs: it is tested
    on its own below."""
    import dataclasses
    wl = dataclasses.replace(synth.workload(2, scale=1 / 64), hops=hops, k=k)
    monkeypatch.setenv("AKASHIC_REACH", "0")
    monkeypatch.setenv("AKASHIC_HOP_PRUNE", "0")
    _, full = gpu_retrieve(wl, "clustered")
    monkeypatch.setenv("AKASHIC_HOP_PRUNE", "1")
    _, pruned = gpu_retrieve(wl, "clustered")
    for key in ("ids", "page_ids", "n_pages"):
        assert np.array_equal(full[key], pruned[key]), key
    np.testing.assert_allclose(pruned["scores"], full["scores"], rtol=1e-5, atol=0)
    assert_retrieval_parity(wl, "clustered", pruned, oracle_retrieve(wl, "clustered"))


@pytest.mark.parametrize("hops", [0, 1, 2])
def test_unfused_selection_switch(hops, monkeypatch):
    """AKASHIC_FUSE_FILTER=0 (the measurement switch that writes the last
    slab and selects from it in a separate pass, and with no hops leaves the
    score GEMM unfiltered) against the oracle (gmm1m recipe at N = 16384)."""
    import dataclasses
    wl = dataclasses.replace(synth.workload(2, scale=1 / 64), hops=hops)
    monkeypatch.setenv("AKASHIC_FUSE_FILTER", "0")
    _, got = gpu_retrieve(wl, "random")
    assert_retrieval_parity(wl, "random", got, oracle_retrieve(wl, "random"))


def test_full_transpose_switch_after_update(monkeypatch):
    """AKASHIC_FULL_TRANSPOSE=1 (the measurement switch that rebuilds the
    in-edge transpose by radix sort after an update instead of patching
    it): the update's whole CSR against the oracle, then retrieval on the
    updated store against the oracle."""
    monkeypatch.setenv("AKASHIC_FULL_TRANSPOSE", "1")
    wl = synth.workload(3, scale=1 / 64)
    store = check_update(wl)
    _retrieval_on_store(wl, store, [wl.new_emb.shape[0]])


def test_score_filter_overflow_falls_back():
    """No hops, N = 16384 chunks sharing one embedding: every score is equal,
    all rows clear the bound taken from the score's row sample and the
    8192-key buffer of every query overflows; the merge recomputes the
    query's scores and selects the k lowest IDs among the ties."""
    import dataclasses
    base = synth.workload(2, scale=1 / 64)
    emb = np.repeat(base.emb[:1], base.n, axis=0)
    wl = dataclasses.replace(base, emb=emb, row_ptr=np.zeros(base.n + 1, np.int64),
                             col=np.zeros(0, np.int32), aff=np.zeros(0, np.float32), hops=0)
    q = wl.queries[:4]
    _, got = gpu_retrieve(wl, "clustered", queries=q, k=8)
    ref = oracle_retrieve(wl, "clustered", queries=q, k=8)
    assert_retrieval_parity(wl, "clustered", got, ref)
    assert (np.sort(got["ids"], axis=1) == np.arange(8)).all()


@pytest.mark.parametrize("hops,sort_by_time", [(0, False), (2, False), (2, True), (1, True)])
def test_namespace_scoped_retrieval(hops, sort_by_time, monkeypatch):
    """Chunks tagged by component mod 6 (namespace 5 queried by no query),
    plus a namespace of only 3 chunks; each of the 256 queries scoped to a
    seeded namespace (every 17th to the small one, which pads its list);
    scores and propagation over the whole store, candidates from the
    namespace only; score order or SortByTime.  N = 16384 from the gmm1m
    recipe.  The last hop's per-namespace floors (each namespace's k-th
    largest lower bound; rows of unqueried namespaces skipped) must select
    what the unpruned hops select."""
    import oracle
    import torch
    wl = synth.workload(2, scale=1 / 64)
    rng = np.random.default_rng(11)
    ns_of = (wl.component % 6).astype(np.int32)
    ns_of[rng.choice(wl.n, 3, replace=False)] = 7
    q_ns = rng.integers(0, 5, wl.n_queries).astype(np.int32)
    q_ns[::17] = 7
    q = torch.from_numpy(np.ascontiguousarray(wl.queries).view(np.int16)).cuda()

    def run():
        store = gpu_store(wl, "clustered")
        store.set_namespace(0, torch.from_numpy(ns_of).cuda())
        ids, sc, pg, npg = store.retrieve(q, wl.k, wl.alpha, hops,
                                          q_ns=torch.from_numpy(q_ns).cuda(),
                                          sort_by_time=sort_by_time)
        store.sync()
        return dict(ids=ids.cpu().numpy(), scores=sc.cpu().numpy(), page_ids=pg.cpu().numpy(),
                    n_pages=npg.cpu().numpy())

    got = run()
    if hops >= 1:
        monkeypatch.setenv("AKASHIC_HOP_PRUNE", "0")
        full = run()
        for key in ("ids", "page_ids", "n_pages"):
            assert np.array_equal(full[key], got[key]), key
    ref = oracle.retrieve(wl.emb, wl.queries, wl.row_ptr, wl.col, oracle_weights(wl), tau=wl.tau,
                          alpha=wl.alpha, hops=hops, k=wl.k, page_of=wl.page_of["clustered"],
                          want_final=True, ns_of=ns_of, q_ns=q_ns, sort_by_time=sort_by_time)
    assert_scoped_parity(wl, "clustered", got, ref, ns_of, q_ns, sort_by_time)
    assert (got["ids"][::17][:, 3:] == -1).all()


@pytest.mark.parametrize("hops", [0, 2])
def test_delete_then_retrieve(hops):
    """Delete 600 chunks (the 20 most-pointed-at hubs among them) from the
    16384-chunk gmm1m-recipe store: the exported CSR equals the oracle's edge
    drop exactly and its weights are the row softmax of what remains, and
    retrieval (deleted chunks score nothing and are never selected) matches
    the oracle with the same tombstones."""
    import oracle
    import torch
    wl = synth.workload(2, scale=1 / 64)
    rng = np.random.default_rng(17)
    indeg = np.bincount(wl.col, minlength=wl.n)
    victims = np.unique(np.concatenate([np.argsort(-indeg)[:20],
                                        rng.choice(wl.n, 580, replace=False)]))
    dead = np.zeros(wl.n, bool)
    dead[victims] = True
    store = gpu_store(wl, "clustered")
    store.delete(torch.from_numpy(victims.astype(np.int64)).cuda())
    store.sync()
    rp, col, aff, w = (t.cpu().numpy() for t in store.export_csr())
    orp, ocol, oaff = oracle.drop_dead(wl.row_ptr, wl.col, wl.aff, dead)
    assert (rp == orp).all() and (col == ocol).all() and (aff == oaff).all()
    assert np.allclose(w, oracle.row_softmax(rp, aff), rtol=2e-3, atol=0)
    q = torch.from_numpy(np.ascontiguousarray(wl.queries).view(np.int16)).cuda()
    ids, sc, pg, npg = store.retrieve(q, wl.k, wl.alpha, hops)
    store.sync()
    got = dict(ids=ids.cpu().numpy(), scores=sc.cpu().numpy(), page_ids=pg.cpu().numpy(),
               n_pages=npg.cpu().numpy())
    assert not dead[got["ids"]].any()
    ref = oracle.retrieve(wl.emb, wl.queries, rp, col, oracle.row_softmax(rp, aff), tau=wl.tau,
                          alpha=wl.alpha, hops=hops, k=wl.k, page_of=wl.page_of["clustered"],
                          want_final=True, dead=dead)
    assert_retrieval_parity(wl, "clustered", got, ref)


@pytest.mark.parametrize("placement,B,k,must", [
    ("clustered", 256, 32, True), ("random", 256, 32, True), ("clustered", 128, 32, True),
    ("clustered", 128, 64, False),
])
def test_two_hop_scores_from_reach_coefficients(placement, B, k, must, monkeypatch):
    """Two hops without running them: when every row that can reach the
    top-k floor is one of the candidate rows with graph-only reach
    coefficients, s^(2) of those rows comes from one pass over u.  On the
    gmm1m recipe (N = 16384) that path must be taken where `must` (no
    propagation hop is launched) and select what the hops select: the same
    IDs except near-ties (scores within REACH_REL of the k-th), pages from
    the page table, scores of the common IDs within REACH_REL, and the
    oracle's selection (B = 256 and 128 queries, k = 32 and 64).  REACH_REL
    = 5e-5: the candidates' terms are split-bf16 products (each operand
    hi + lo to 2^-16, the lo x lo term dropped: at most 3 * 2^-16 = 4.6e-5
    relative per product, all products non-negative) with fp32 sums."""
    import dataclasses
    wl = dataclasses.replace(synth.workload(2, scale=1 / 64), k=k)
    wl = dataclasses.replace(wl, queries=wl.queries[:B])
    monkeypatch.setenv("AKASHIC_REACH", "0")
    _, hops_out = gpu_retrieve(wl, placement)
    monkeypatch.setenv("AKASHIC_REACH", "1")
    store = gpu_store(wl, placement)
    gpu_retrieve(wl, placement, store=store)          # builds the reach coefficients
    store.set_profiling(True)
    store.phase_times()
    _, reach_out = gpu_retrieve(wl, placement, store=store)
    ph = store.phase_times()
    store.set_profiling(False)
    if must:
        assert ph["propagate"][1] == 0, ph            # no hop launched
        assert ph["last_hop"][1] > 0, ph              # the reach scores were
    REACH_REL = 5e-5
    for b in range(B):
        hi, ri = hops_out["ids"][b].tolist(), reach_out["ids"][b].tolist()
        hs = dict(zip(hi, hops_out["scores"][b].astype(np.float64)))
        rs = dict(zip(ri, reach_out["scores"][b].astype(np.float64)))
        kth = min(hs.values())
        for x in set(hi) ^ set(ri):
            s = hs.get(x, rs.get(x))
            assert abs(s - kth) <= REACH_REL * kth, f"query {b}: chunk {x} swapped ({s} vs {kth})"
        for x in set(hi) & set(ri):
            assert abs(rs[x] - hs[x]) <= REACH_REL * hs[x], f"query {b}: chunk {x} score"
    assert_retrieval_parity(wl, placement, reach_out, oracle_retrieve(wl, placement))


def test_row_bounds_follow_graph_changes():
    """The last hop's graph-only mass levels are cached on the store and
    must be recomputed after the graph changes: retrieve (fills the cache),
    delete 300 chunks including 10 hubs, retrieve, then append 64 chunks
    without edges and retrieve again (N changes, the graph does not) - each
    retrieval against the oracle on the store's current graph."""
    import oracle
    import torch
    wl = synth.workload(2, scale=1 / 64)
    store = gpu_store(wl, "clustered", capacity=wl.n + 64)
    _, got = gpu_retrieve(wl, "clustered", store=store)
    assert_retrieval_parity(wl, "clustered", got, oracle_retrieve(wl, "clustered"))
    rng = np.random.default_rng(23)
    indeg = np.bincount(wl.col, minlength=wl.n)
    victims = np.unique(np.concatenate([np.argsort(-indeg)[:10],
                                        rng.choice(wl.n, 290, replace=False)]))
    dead = np.zeros(wl.n, bool)
    dead[victims] = True
    store.delete(torch.from_numpy(victims.astype(np.int64)).cuda())
    rp, col, aff, _ = (t.cpu().numpy() for t in store.export_csr())
    w = oracle.row_softmax(rp, aff)

    def check(n_extra):
        emb = wl.emb if n_extra == 0 else np.concatenate([wl.emb, wl.emb[:n_extra]])
        d = np.concatenate([dead, np.zeros(n_extra, bool)])
        rp2 = np.concatenate([rp, np.full(n_extra, rp[-1], np.int64)])
        pages = np.concatenate([wl.page_of["clustered"],
                                wl.page_of["clustered"].max() + 1 + np.arange(n_extra) // 64])
        q = torch.from_numpy(np.ascontiguousarray(wl.queries).view(np.int16)).cuda()
        ids, sc, pg, npg = store.retrieve(q, wl.k, wl.alpha, wl.hops)
        store.sync()
        got = dict(ids=ids.cpu().numpy(), scores=sc.cpu().numpy(), page_ids=pg.cpu().numpy(),
                   n_pages=npg.cpu().numpy())
        assert not d[got["ids"]].any()
        ref = oracle.retrieve(emb, wl.queries, rp2, col, w, tau=wl.tau, alpha=wl.alpha,
                              hops=wl.hops, k=wl.k, page_of=pages.astype(np.int32),
                              want_final=True, dead=d)
        import dataclasses
        wl2 = dataclasses.replace(wl, emb=emb, page_of={"clustered": pages.astype(np.int32)})
        assert_retrieval_parity(wl2, "clustered", got, ref)

    check(0)
    store.append_chunks(torch.from_numpy(np.ascontiguousarray(wl.emb[:64]).view(np.int16)).cuda())
    check(64)


def test_delete_then_update_skips_deleted():
    """After deletions a relation update links each new chunk to its top-M
    among the live prior chunks only: its neighbour set equals the oracle's
    on the store rebuilt without the deleted chunks (IDs mapped back), and
    retrieval on the result matches the oracle."""
    import dataclasses
    import oracle
    import torch
    from paper_2607_05708_gb300 import MemStore
    wl = synth.workload(3, scale=1 / 64)
    n_old, n_new, M = wl.n, wl.new_emb.shape[0], wl.top_m
    store = MemStore.from_arrays(wl.emb, wl.page_of["clustered"], wl.row_ptr, wl.col, wl.aff,
                                 capacity=n_old + n_new, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau, relation_scale=wl.relation_scale)
    # delete, for each new chunk, its best prior neighbour (and more at random)
    all_emb = np.concatenate([wl.emb, wl.new_emb])
    E = synth.bf16_to_f32(all_emb).astype(np.float64)
    best = np.argmax(E[n_old:] @ E[:n_old].T, axis=1)
    victims = np.unique(np.concatenate([best, np.random.default_rng(3).choice(n_old, 200, replace=False)]))
    dead = np.zeros(n_old + n_new, bool)
    dead[victims] = True
    store.delete(torch.from_numpy(victims.astype(np.int64)).cuda())
    first = store.append_chunks(torch.from_numpy(np.ascontiguousarray(wl.new_emb).view(np.int16)).cuda())
    store.update_relations(first, n_new, M, reciprocal=True)
    store.sync()
    rp, col, aff, _ = (t.cpu().numpy() for t in store.export_csr())
    live = np.nonzero(~dead[:n_old])[0]
    for a in range(n_new):
        nbrs = col[rp[n_old + a]:rp[n_old + a + 1]]
        assert len(nbrs) == M and not dead[nbrs].any()
    # oracle on the live-only prior store (edges among live chunks, re-indexed)
    orp, ocol, oaff = oracle.drop_dead(wl.row_ptr, wl.col, wl.aff, dead[:n_old])
    new_id = -np.ones(n_old, np.int64)
    new_id[live] = np.arange(live.size)
    src = np.repeat(np.arange(n_old), np.diff(orp))
    rp_l = np.concatenate([[0], np.cumsum(np.bincount(new_id[src], minlength=live.size)),
                           np.full(n_new, len(ocol))])
    ref = oracle.update_relations(np.concatenate([wl.emb[live], wl.new_emb]), live.size, n_new, M,
                                  rp_l, new_id[ocol].astype(np.int32), oaff,
                                  scale=wl.relation_scale, reciprocal=True)
    for a in range(n_new):
        g = set(col[rp[n_old + a]:rp[n_old + a + 1]].tolist())
        o = set(live[ref["nbr_ids"][a]].tolist())
        kth = ref["nbr_cos"][a][M - 1]
        for x in g ^ o:
            assert abs(float(E[x] @ E[n_old + a]) - kth) < 1e-4, f"new chunk {a}: {x} swapped"
    wl2 = dataclasses.replace(wl, emb=all_emb, row_ptr=rp, col=col, aff=aff,
                              page_of={"clustered": _pages_after_appends(wl, [n_new])})
    _, got = gpu_retrieve(wl2, "clustered", store=store)
    ref2 = oracle.retrieve(all_emb, wl.queries, rp, col, oracle.row_softmax(rp, aff), tau=wl.tau,
                           alpha=wl.alpha, hops=wl.hops, k=wl.k,
                           page_of=wl2.page_of["clustered"], want_final=True, dead=dead)
    assert_retrieval_parity(wl2, "clustered", got, ref2)


def test_delete_errors():
    """An out-of-range ID deletes nothing (EINVAL); an appended edge that
    points at a deleted chunk is rejected (EDEVICE) and nothing is appended."""
    import torch
    from paper_2607_05708_gb300 import AkashicError, MemStore
    wl = synth.workload(0)
    st = MemStore.from_arrays(wl.emb, wl.page_of["id"], wl.row_ptr, wl.col, wl.aff,
                              capacity=wl.n + 8, chunks_per_page=wl.chunks_per_page)
    before = [t.cpu().numpy() for t in st.export_csr()]
    with pytest.raises(AkashicError) as e:
        st.delete(torch.tensor([3, wl.n + 5], dtype=torch.int64, device="cuda"))
    assert e.value.code == "EINVAL"
    after = [t.cpu().numpy() for t in st.export_csr()]
    assert all((x == y).all() for x, y in zip(before, after))
    st.delete(torch.tensor([3], dtype=torch.int64, device="cuda"))
    t = lambda x, dt: torch.from_numpy(np.ascontiguousarray(x).view(dt)).cuda()
    with pytest.raises(AkashicError) as e:
        st.append_chunks(t(wl.emb[:1], np.int16), None, t(np.array([0, 1], np.int64), np.int64),
                         t(np.array([3], np.int32), np.int32), t(np.array([1.0], np.float32), np.float32))
    assert e.value.code == "EDEVICE"
    assert st.size()[0] == wl.n


def test_no_edges_and_single_chunk_pages():
    """A store without relations: propagation adds nothing."""
    wl0 = synth.workload(0)
    wl = synth.Workload(name="noedges", dim=wl0.dim, emb=wl0.emb, queries=wl0.queries,
                        row_ptr=np.zeros(wl0.n + 1, np.int64), col=np.zeros(0, np.int32),
                        aff=np.zeros(0, np.float32), page_of={"id": np.arange(wl0.n, dtype=np.int32)},
                        chunks_per_page=1, alpha=0.5, hops=2, k=8)
    _, got = gpu_retrieve(wl, "id")
    ref = oracle_retrieve(wl, "id")
    assert_retrieval_parity(wl, "id", got, ref)
    assert (got["n_pages"] == 8).all()


def test_batch_equals_single_queries():
    """Queries are independent: one batch equals per-query calls (same ids)."""
    wl = synth.workload(2, scale=1 / 128)
    store, got = gpu_retrieve(wl, "clustered")
    for b in (0, 7, 200):
        _, one = gpu_retrieve(wl, "clustered", store=store, queries=wl.queries[b:b + 1])
        assert (one["ids"][0] == got["ids"][b]).all()


def test_queries_at_any_alignment():
    """Query rows that do not start on a 16-byte boundary (a view two bytes
    into its buffer) take the element-wise load path.  Its |q| sums in
    another order, so the shift and the scores may differ in the last bits:
    both calls must match the oracle, and agree within 1e-5 wherever they
    chose the same chunk."""
    import torch
    wl = synth.workload(2, scale=1 / 128)
    store = gpu_store(wl, "clustered")
    q = np.ascontiguousarray(wl.queries).view(np.int16)
    flat = torch.empty(q.size + 1, dtype=torch.int16, device="cuda")
    flat[1:] = torch.from_numpy(q.ravel()).cuda()
    odd = flat[1:].view(q.shape)
    assert odd.data_ptr() % 16 != 0
    even = torch.from_numpy(q).cuda()
    keys = ("ids", "scores", "page_ids", "n_pages")
    a = dict(zip(keys, (t.cpu().numpy() for t in store.retrieve(even, wl.k, wl.alpha, wl.hops))))
    b = dict(zip(keys, (t.cpu().numpy() for t in store.retrieve(odd, wl.k, wl.alpha, wl.hops))))
    store.sync()
    ref = oracle_retrieve(wl, "clustered")
    assert_retrieval_parity(wl, "clustered", a, ref)
    assert_retrieval_parity(wl, "clustered", b, ref)
    same = a["ids"] == b["ids"]
    assert same.mean() > 0.99
    np.testing.assert_allclose(b["scores"][same], a["scores"][same], rtol=1e-5, atol=0)


def test_appends_in_pieces_equal_one_append():
    """Appending the store in three pieces gives the same retrieval."""
    import torch
    from paper_2607_05708_gb300 import MemStore
    wl = synth.workload(0)
    st = MemStore(wl.dim, wl.n, 16, temperature=wl.tau)
    cuts = [0, 1000, 2500, wl.n]
    for a, b in zip(cuts[:-1], cuts[1:]):
        rp = wl.row_ptr[a:b + 1]
        t = lambda x, dt: torch.from_numpy(np.ascontiguousarray(x).view(dt)).cuda()
        # edges may only point below b: keep them all (targets < N) by appending
        # rows without edges, then compare the graph-free retrieval
        first = st.append_chunks(t(wl.emb[a:b], np.int16), t(wl.page_of["id"][a:b], np.int32))
        assert first == a
    _, got = gpu_retrieve(wl, "id", store=st, hops=0)
    ref = oracle_retrieve(wl, "id", hops=0)
    assert_retrieval_parity(wl, "id", got, ref)


# --------------------------------------------------------------------------- full size
@pytest.fixture(scope="module")
def gmm1m():
    return synth.workload(2)


@pytest.mark.parametrize("placement", ["clustered", "random"])
def test_gmm1m_full_size_sampled(gmm1m, placement):
    """N=1,048,576, d=1024, B=256, two hops, k=32, both placements (the
    co-retrieval-clustered and the random page table): the whole batch runs
    in the launch configuration the benchmark times; the oracle recomputes a
    seeded sample of 3 queries."""
    wl = gmm1m
    _, got = gpu_retrieve(wl, placement)
    rows = [0, 97, 255]
    ref = oracle_retrieve_rows(wl, placement, rows)
    sub = {k: v[rows] for k, v in got.items()}
    assert_retrieval_parity(wl, placement, sub, ref)
    # properties at any size: page counts within [ceil(k/P), k]
    assert (got["n_pages"] >= int(np.ceil(wl.k / wl.chunks_per_page))).all()
    assert (got["n_pages"] <= wl.k).all()


def test_gmm65k_full_size():
    """The gmm65k workload at its stated size: N=65,536, d=768, exact top-16
    cosine graph, B=64 queries near mixture centres, one hop, alpha=0.5,
    k=16, 32 chunks per page by component; every query against the oracle."""
    wl = synth.workload(1)
    assert wl.n == 65536 and wl.n_queries == 64
    _, got = gpu_retrieve(wl, "component")
    ref = oracle_retrieve_rows(wl, "component", range(wl.n_queries))
    assert_retrieval_parity(wl, "component", got, ref)


def _streams_retrieve(wl, store, placement, per_stream, seed):
    """The workload's queries as its streams of equal slices, issued in the
    seeded arrival order and all in flight at once (each stream has its own
    scratch); returns the sampled rows (per_stream per stream) with their
    outputs, after checking every stream's page counts in [1, k]."""
    import torch
    per = wl.n_queries // wl.streams
    streams = [torch.cuda.Stream() for _ in range(wl.streams)]
    outs = {}
    for i in wl.stream_order:
        q = torch.from_numpy(np.ascontiguousarray(wl.queries[i * per:(i + 1) * per]).view(np.int16)).cuda()
        torch.cuda.current_stream().synchronize()
        outs[i] = store.retrieve(q, wl.k, wl.alpha, wl.hops, stream=streams[i]) + (q,)
    torch.cuda.synchronize()
    store.sync()
    rng = np.random.default_rng(seed)
    rows = []
    got = {"ids": [], "scores": [], "page_ids": [], "n_pages": []}
    for i in range(wl.streams):
        ids, sc, pg, npg, _ = outs[i]
        for r in sorted(rng.choice(per, size=per_stream, replace=False)):
            rows.append(i * per + r)
            got["ids"].append(ids[r].cpu().numpy())
            got["scores"].append(sc[r].cpu().numpy())
            got["page_ids"].append(pg[r].cpu().numpy())
            got["n_pages"].append(int(npg[r]))
        assert (npg.cpu().numpy() <= wl.k).all()
        assert (npg.cpu().numpy() >= 1).all()
    return rows, {k: np.array(v) for k, v in got.items()}


@pytest.mark.parametrize("placement", ["clustered", "random"])
def test_gmm4m_full_size_streams_sampled(placement):
    """The gmm4m workload at its stated size: N=4,194,304, d=768,
    16384-component mixture, 32-neighbour graph, 1024 queries as 8 streams
    of 128 in the seeded arrival order, two hops, alpha=0.4, k=64, 64 chunks
    per page; 2 sampled queries per stream against the oracle."""
    wl = _gmm4m()
    assert wl.n == 4194304 and wl.n_queries == 1024 and wl.streams == 8
    store = gpu_store(wl, placement)
    rows, got = _streams_retrieve(wl, store, placement, 2, seed=11)
    store.close()
    ref = oracle_retrieve_rows(wl, placement, rows)
    assert_retrieval_parity(wl, placement, got, ref)


_GMM4M = []


def _gmm4m():
    if not _GMM4M:
        _GMM4M.append(synth.workload(4))
    return _GMM4M[0]


# --------------------------------------------------------------------------- relation update
def test_update_scaled_full_oracle():
    """4096/256 = 16 new chunks appended to a 4096-chunk gmm1m-recipe store:
    top-32 cosine neighbours + reciprocal edges, whole CSR vs the oracle."""
    check_update(synth.workload(3, scale=1 / 256))


def test_update_mid_scale():
    """64 new chunks into a 16384-chunk store (several query batches of the
    cosine GEMM would not be exercised; this covers ragged tiles)."""
    check_update(synth.workload(3, scale=1 / 64))


def test_update_errors():
    import torch
    from paper_2607_05708_gb300 import AkashicError, MemStore
    wl = synth.workload(3, scale=1 / 256)
    st = MemStore.from_arrays(wl.emb, wl.page_of["clustered"], wl.row_ptr, wl.col, wl.aff,
                              capacity=wl.n + 64)
    with pytest.raises(AkashicError) as e:
        st.update_relations(wl.n, 1, 32)          # beyond the store
    assert e.value.code == "EINVAL"
    with pytest.raises(AkashicError) as e:
        st.update_relations(0, 10, 32)            # rows already have out-edges / M > first
    assert e.value.code == "EINVAL"


# --------------------------------------------------------------------------- error paths
def test_retrieve_argument_errors():
    import torch
    from paper_2607_05708_gb300 import AkashicError
    wl = synth.workload(0)
    st = gpu_store(wl, "id")
    q = torch.from_numpy(wl.queries.view(np.int16)).cuda()
    for kwargs, code in (({"k": 0, "alpha": 0.5, "hops": 1}, "EINVAL"),
                         ({"k": 65, "alpha": 0.5, "hops": 1}, "EINVAL"),
                         ({"k": 8, "alpha": -1.0, "hops": 1}, "EINVAL"),
                         ({"k": 8, "alpha": float("nan"), "hops": 1}, "EINVAL"),
                         ({"k": 8, "alpha": 0.5, "hops": 17}, "EINVAL")):
        with pytest.raises(AkashicError) as e:
            st.retrieve(q, **kwargs)
        assert e.value.code == code


def test_capacity_and_bad_csr():
    import torch
    from paper_2607_05708_gb300 import AkashicError, MemStore
    wl = synth.workload(0)
    t = lambda x, dt: torch.from_numpy(np.ascontiguousarray(x).view(dt)).cuda()
    st = MemStore(wl.dim, 100, 16)
    with pytest.raises(AkashicError) as e:
        st.append_chunks(t(wl.emb[:101], np.int16))
    assert e.value.code == "ECAPACITY"
    # a self-loop is rejected and nothing is committed
    rp = np.array([0, 1, 1], np.int64)
    col = np.array([0], np.int32)                 # row 0 -> itself
    aff = np.array([1.0], np.float32)
    with pytest.raises(AkashicError) as e:
        st.append_chunks(t(wl.emb[:2], np.int16), None, t(rp, np.int64), t(col, np.int32),
                         t(aff, np.float32))
    assert e.value.code == "EDEVICE"
    assert st.size() == (0, 0)
    # a valid append still works afterwards
    col = np.array([1], np.int32)
    assert st.append_chunks(t(wl.emb[:2], np.int16), None, t(rp, np.int64), t(col, np.int32),
                            t(aff, np.float32)) == 0
    assert st.size() == (2, 1)


def _pages_after_appends(wl, batches):
    """Page table of a store holding wl (clustered placement) after appends
    of the given sizes without a page table: each batch takes fresh pages
    in ID order, starting after the last page in use."""
    pages = [wl.page_of["clustered"].astype(np.int64)]
    nxt = int(pages[0].max()) + 1
    for n_b in batches:
        pages.append(nxt + np.arange(n_b) // wl.chunks_per_page)
        nxt += -(-n_b // wl.chunks_per_page)
    return np.concatenate(pages).astype(np.int32)


def _retrieval_on_store(wl, store, batches, k=None, hops=None):
    """Retrieval through the store after updates vs the oracle on the graph
    the store exports (the transpose used by propagation is checked by it)."""
    import dataclasses
    n_new = sum(batches)
    rp, col, aff, _ = (t.cpu().numpy() for t in store.export_csr())
    wl2 = dataclasses.replace(wl, emb=np.concatenate([wl.emb, wl.new_emb[:n_new]]), row_ptr=rp,
                              col=col, aff=aff,
                              page_of={"clustered": _pages_after_appends(wl, batches)})
    _, got = gpu_retrieve(wl2, "clustered", store=store, k=k, hops=hops)
    ref = oracle_retrieve(wl2, "clustered", k=k, hops=hops)
    assert_retrieval_parity(wl2, "clustered", got, ref)


def test_retrieval_after_update():
    """Retrieval on the store right after a relation update (the in-edge
    transpose is patched, not rebuilt): 64 new chunks into 16384."""
    wl = synth.workload(3, scale=1 / 64)
    store = check_update(wl)
    _retrieval_on_store(wl, store, [wl.new_emb.shape[0]])


def test_dense_only_top5():
    """The Dense-only form with the paper's top-p = 5: relation update with
    M = 5 (whole CSR against the oracle), then retrieval with k = 5 and no
    propagation on the updated store."""
    wl = synth.workload(3, scale=1 / 64)
    store = check_update(wl, M=5)
    _retrieval_on_store(wl, store, [wl.new_emb.shape[0]], k=5, hops=0)


def test_retrieval_after_two_updates():
    """Two appends + updates in a row (the second links new chunks to rows
    that gained in-edges in the first), then retrieval parity."""
    import torch
    from paper_2607_05708_gb300 import MemStore
    wl = synth.workload(3, scale=1 / 64)
    n_new = wl.new_emb.shape[0]
    store = MemStore.from_arrays(wl.emb, wl.page_of["clustered"], wl.row_ptr, wl.col, wl.aff,
                                 capacity=wl.n + n_new, chunks_per_page=wl.chunks_per_page,
                                 temperature=wl.tau, relation_scale=wl.relation_scale)
    half = n_new // 2
    for a, b in ((0, half), (half, n_new)):
        new = torch.from_numpy(np.ascontiguousarray(wl.new_emb[a:b]).view(np.int16)).cuda()
        first = store.append_chunks(new)
        assert first == wl.n + a
        store.update_relations(first, b - a, wl.top_m, reciprocal=True)
    store.sync()
    _retrieval_on_store(wl, store, [half, n_new - half])


@pytest.fixture(scope="module")
def update_full():
    return synth.workload(3)


def test_update_full_size_whole_csr(update_full):
    """4096 new chunks linked into the N=1,048,576 store in one call (the
    benchmark's update), and the whole exported CSR (every row's pointers,
    columns and logits) against the oracle's: its top-32 of every new chunk
    is stored in tests/golden/update_gmm1m_top32.npz by
    tests/golden/make_update_golden.py (oracle/ only), with the SHA-256 of
    the inputs it was computed on, checked here first."""
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "update_gmm1m_top32.npz")
    g = np.load(path)
    import importlib.util
    spec = importlib.util.spec_from_file_location(
        "make_update_golden", os.path.join(os.path.dirname(__file__), "golden",
                                           "make_update_golden.py"))
    mk = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mk)
    wl = update_full
    assert str(g["inputs_sha256"]) == mk.input_digest(wl), "generated inputs differ from the golden's"
    assert int(g["n_old"]) == wl.n and int(g["top_m"]) == wl.top_m
    check_update(wl, golden={"nbr_ids": g["nbr_ids"], "nbr_cos": g["nbr_cos"]})


def test_gmm4m_recipe_eight_concurrent_streams():
    """gmm4m recipe at N=65536 (d=768, k=64, alpha=0.4): 1024 queries issued
    as 8 streams of 128 in the seeded arrival order, all in flight at once
    (each stream has its own scratch); 2 sampled queries per stream against
    the oracle, and every stream's page counts within [1, k]."""
    wl = synth.workload(4, scale=1 / 64)
    store = gpu_store(wl, "clustered")
    rows, got = _streams_retrieve(wl, store, "clustered", 2, seed=7)
    ref = oracle_retrieve(wl, "clustered", queries=wl.queries[rows])
    assert_retrieval_parity(wl, "clustered", got, ref)


@pytest.mark.parametrize("hops", [3, 2])
def test_first_retrieves_from_two_threads(hops):
    """Two host threads, each with its own stream, make the first retrieves
    of a fresh store at the same moment (gmm1m recipe at N = 16384, 128
    queries each).  The graph-only tables of the last hop's row bounds (and,
    for two hops, the reach coefficients) are built by whichever call comes
    first; the other call's stream is ordered after that build.  Both
    threads' results must match the oracle."""
    import dataclasses
    import threading
    import torch
    wl = dataclasses.replace(synth.workload(2, scale=1 / 64), hops=hops)
    store = gpu_store(wl, "clustered")
    half = wl.n_queries // 2
    streams = [torch.cuda.Stream() for _ in range(2)]
    qs = [torch.from_numpy(np.ascontiguousarray(wl.queries[i * half:(i + 1) * half])
                           .view(np.int16)).cuda() for i in range(2)]
    torch.cuda.synchronize()
    outs, errs = [None, None], []
    gate = threading.Barrier(2)

    def run(i):
        try:
            with torch.cuda.stream(streams[i]):
                gate.wait()
                outs[i] = store.retrieve(qs[i], wl.k, wl.alpha, wl.hops, stream=streams[i])
        except Exception as e:      # re-raised on the main thread below
            errs.append(e)

    threads = [threading.Thread(target=run, args=(i,)) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    torch.cuda.synchronize()
    store.sync()
    assert not errs, errs
    got = {key: np.concatenate([o[j].cpu().numpy() for o in outs])
           for j, key in enumerate(("ids", "scores", "page_ids", "n_pages"))}
    assert_retrieval_parity(wl, "clustered", got, oracle_retrieve(wl, "clustered"))


@pytest.mark.parametrize("B", [64, 256])
def test_sixteen_hops(B):
    """The largest hop count retrieve accepts: H = 16 on the gmm1m recipe at
    N = 16384 (alpha = 0.5, k = 32), the last hop's row bounds over 16 mass
    levels; oracle parity."""
    import dataclasses
    wl = synth.workload(2, scale=1 / 64)
    wl = dataclasses.replace(wl, hops=16, queries=wl.queries[:B])
    _, got = gpu_retrieve(wl, "clustered")
    assert_retrieval_parity(wl, "clustered", got, oracle_retrieve(wl, "clustered"))


@pytest.mark.parametrize("dim", [64, 4096])
def test_embedding_width_limits(dim):
    """The narrowest and widest embeddings a store accepts, d = 64 and 4096
    (the score GEMM's K loop runs over 1 and 64 blocks of 64): the tiny
    store's graph and pages with fresh unit-length bf16 rows of that width,
    37 queries, two hops, k = 16; oracle parity."""
    import dataclasses
    base = synth.workload(0)
    rng = np.random.default_rng(dim)

    def unit(m):
        x = rng.standard_normal((m, dim)).astype(np.float32)
        return synth.to_bf16(x / np.linalg.norm(x, axis=1, keepdims=True))

    wl = dataclasses.replace(base, dim=dim, emb=unit(base.n), queries=unit(37), hops=2, k=16)
    _, got = gpu_retrieve(wl, "id")
    assert_retrieval_parity(wl, "id", got, oracle_retrieve(wl, "id"))


def test_bounded_wait_gives_up_and_the_store_stays_usable():
    """Every device-side wait in the library gives up after a bounded number
    of polls, records ETIMEOUT and lets its kernel return.  A wait that
    nothing ever releases (akashic_mem_check_wait_timeout, 1000 polls) must
    surface as ETIMEOUT at the next sync, the status must then be clear, and
    a retrieval on the same store must still match the oracle."""
    from paper_2607_05708_gb300 import AkashicError
    wl = synth.workload(0)
    store = gpu_store(wl, "id")
    store.check_wait_timeout(1000)
    with pytest.raises(AkashicError) as err:
        store.sync()
    assert err.value.code == "ETIMEOUT"
    store.sync()                                      # the word was cleared
    _, got = gpu_retrieve(wl, "id", store=store)
    assert_retrieval_parity(wl, "id", got, oracle_retrieve(wl, "id"))
    with pytest.raises(AkashicError) as err:
        store.check_wait_timeout(0)
    assert err.value.code == "EINVAL"
