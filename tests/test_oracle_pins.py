"""Pins for the CPU oracle, checked against things other than itself.

Each test names the property of the method (arXiv 2607.05708) that it pins:
a hand-worked example, a closed form, an invariant, a reduction to a
textbook/library routine, or brute force on a tiny store.  The mistakes each
is meant to catch are listed beside it.
"""
import math
import os

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------- helpers
def tiny_store(seed, n, d, deg, n_q=3, self_loops=False, empty_rows=False):
    rng = np.random.default_rng(seed)
    emb = synth.to_bf16(rng.standard_normal((n, d)).astype(np.float32) * 0.3)
    q = synth.to_bf16(rng.standard_normal((n_q, d)).astype(np.float32) * 0.3)
    cols, ptr = [], [0]
    for i in range(n):
        m = 0 if (empty_rows and i % 7 == 3) else deg
        c = rng.choice(n, size=m, replace=False) if self_loops else \
            (lambda p: np.where(p >= i, p + 1, p))(rng.choice(n - 1, size=m, replace=False))
        cols.append(np.sort(c))
        ptr.append(ptr[-1] + m)
    col = np.concatenate(cols).astype(np.int32) if cols else np.zeros(0, np.int32)
    aff = rng.standard_normal(col.shape[0]).astype(np.float32)
    return emb, q, np.array(ptr, np.int64), col, aff


def widen(h):
    return synth.bf16_to_f32(h).astype(np.float64)


def dense_R(n, row_ptr, col, w):
    R = np.zeros((n, n))
    for i in range(n):
        for e in range(row_ptr[i], row_ptr[i + 1]):
            R[i, col[e]] += w[e]
    return R


def softmax_lib(x):
    from scipy.special import softmax
    return softmax(x)


# --------------------------------------------------------------------------- golden example
def _golden():
    g = {"emb": {}, "edge": [], "hop1": {}, "hop2": {}}
    with open(os.path.join(GOLDEN, "three_chunks.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, _, rest = line.partition(" ")
            rest = rest.strip()
            if key == "emb":
                i, *v = rest.split()
                g["emb"][int(i)] = [float(x) for x in v]
            elif key == "edge":
                a, b, c = rest.split()
                g["edge"].append((int(a), int(b), float(c)))
            elif key in ("hop1", "hop2"):
                i, expr = rest.split(None, 1)
                g[key][int(i)] = eval(expr, {"__builtins__": {}}, {"exp": math.exp})
            elif key in ("Z",):
                g[key] = eval(rest, {"__builtins__": {}}, {"exp": math.exp})
            else:
                g[key] = rest
    return g


def _golden_inputs(g):
    n = len(g["emb"])
    emb = synth.to_bf16(np.array([g["emb"][i] for i in range(n)], np.float32))
    q = synth.to_bf16(np.array([[float(x) for x in g["query"].split()]], np.float32))
    edges = sorted(g["edge"])
    row_ptr = np.zeros(n + 1, np.int64)
    for a, _, _ in edges:
        row_ptr[a + 1] += 1
    row_ptr = np.cumsum(row_ptr)
    col = np.array([b for _, b, _ in edges], np.int32)
    aff = np.array([c for _, _, c in edges], np.float32)
    page_of = np.array([int(x) for x in g["page_of"].split()], np.int32)
    return emb, q, row_ptr, col, aff, page_of


@pytest.mark.parametrize("hops", [1, 2])
def test_golden_three_chunks(hops):
    """Hand-worked example: catches wrong edge direction (in/out), a dropped
    u term, alpha applied twice, wrong row normalisation, wrong shift."""
    g = _golden()
    emb, q, row_ptr, col, aff, page_of = _golden_inputs(g)
    w = oracle.row_softmax(row_ptr, aff)
    out = oracle.retrieve(emb, q, row_ptr, col, w, tau=float(g["tau"]), alpha=float(g["alpha"]),
                          hops=hops, k=2, page_of=page_of, want_final=True)
    want = g[f"hop{hops}"]
    Z = g["Z"]
    assert out["z"][0] == pytest.approx(Z, rel=1e-15)
    assert out["shift"][0] == pytest.approx(float(g["shift"]), abs=0)
    for j in range(3):
        assert out["final"][0, j] == pytest.approx(want[j] / Z, rel=1e-14)
    assert list(out["ids"][0]) == [int(x) for x in g[f"top2_hop{hops}"].split()]
    assert list(out["page_ids"][0]) == [int(x) for x in g["pages_top2"].split()]
    assert out["n_pages"][0] == int(g["npages_top2"])
    out3 = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.5, alpha=0.5, hops=hops, k=3,
                           page_of=page_of)
    assert out3["n_pages"][0] == int(g["npages_top3"])


# --------------------------------------------------------------------------- relation weights
def test_row_softmax_closed_forms():
    """Equal logits -> uniform; logits (0, ln 3) -> (1/4, 3/4); shift-invariant;
    empty rows untouched.  Catches a missing max-shift, a wrong denominator."""
    row_ptr = np.array([0, 3, 3, 5, 6], np.int64)
    aff = np.array([2.0, 2.0, 2.0, 0.0, math.log(3.0), -50.0], np.float32)
    w = oracle.row_softmax(row_ptr, aff)
    assert w[:3] == pytest.approx([1 / 3] * 3, rel=1e-15)
    assert w[3] == pytest.approx(0.25, rel=1e-7) and w[4] == pytest.approx(0.75, rel=1e-7)
    assert w[5] == 1.0
    w2 = oracle.row_softmax(row_ptr, aff + np.float32(7.0))
    assert np.allclose(w, w2, rtol=1e-6, atol=0)
    rng = np.random.default_rng(5)
    _, _, rp, col, a = tiny_store(5, 50, 8, 6)
    w = oracle.row_softmax(rp, a)
    for i in range(50):
        seg = slice(rp[i], rp[i + 1])
        assert np.allclose(w[seg], softmax_lib(a[seg].astype(np.float64)), rtol=1e-13)


# --------------------------------------------------------------------------- score
def test_score_is_library_softmax():
    """s0 = softmax(tau * E q) with tau = 1/sqrt(d): scipy softmax of a numpy
    matmul.  Catches a wrong temperature, missing exp, wrong Z."""
    emb, q, *_ = tiny_store(1, 300, 64, 4)
    tau = 1 / 8.0
    out = oracle.retrieve(emb, q, None, None, None, tau=tau, alpha=0.0, hops=0, k=10,
                          want_final=True)
    z = tau * widen(q) @ widen(emb).T
    for b in range(q.shape[0]):
        assert np.allclose(out["final"][b], softmax_lib(z[b]), rtol=1e-12, atol=0)
        assert out["final"][b].sum() == pytest.approx(1.0, abs=1e-12)
        assert out["shift"][b] == pytest.approx(z[b].max(), rel=1e-14)


def test_alpha_zero_is_argsort():
    """alpha=0 (and hops=0) reduce to the plain top-k of the scores: the
    library's lexsort of (-z, id)."""
    emb, q, row_ptr, col, aff = tiny_store(2, 400, 32, 5)
    w = oracle.row_softmax(row_ptr, aff)
    z = widen(q) @ widen(emb).T
    for alpha, hops in ((0.0, 2), (0.5, 0)):
        out = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.2, alpha=alpha, hops=hops, k=12)
        for b in range(q.shape[0]):
            ref = np.lexsort((np.arange(400), -z[b]))[:12]
            assert list(out["ids"][b]) == list(ref)


# --------------------------------------------------------------------------- propagation
@pytest.mark.parametrize("hops,alpha", [(1, 0.5), (2, 0.5), (3, 0.4), (2, 1.0), (16, 0.6)])
def test_propagation_matrix_power_closed_form(hops, alpha):
    """s^(H) = u * sum_{h=0..H} (alpha R)^h, evaluated with numpy
    matrix_power on the dense R: a different formula (power series, dense,
    gather) from the oracle's recurrence (scatter).  Catches wrong direction,
    off-by-one hop count, dropped u term."""
    n = 120
    emb, q, row_ptr, col, aff = tiny_store(3, n, 16, 7, empty_rows=True)
    w = oracle.row_softmax(row_ptr, aff)
    out = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.25, alpha=alpha, hops=hops, k=9,
                          want_final=True)
    R = dense_R(n, row_ptr, col, w)
    S = sum(np.linalg.matrix_power(alpha * R, h) for h in range(hops + 1))
    z = 0.25 * widen(q) @ widen(emb).T
    for b in range(q.shape[0]):
        s0 = softmax_lib(z[b])
        ref = s0 @ S
        assert np.allclose(out["final"][b], ref, rtol=1e-12, atol=0)
        top = np.lexsort((np.arange(n), -ref))[:9]
        assert list(out["ids"][b]) == list(top)
        assert np.allclose(out["scores"][b], ref[top], rtol=1e-12)


@pytest.mark.parametrize("hops,alpha", [(1, 0.5), (2, 0.5), (2, 0.4), (4, 0.3), (16, 0.9)])
def test_mass_conservation(hops, alpha):
    """With no empty rows each hop preserves mass: sum_j s_j = sum_h alpha^h
    (up to the largest hop count the library accepts, 16)."""
    emb, q, row_ptr, col, aff = tiny_store(4, 200, 16, 9)
    w = oracle.row_softmax(row_ptr, aff)
    out = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=alpha, hops=hops, k=5,
                          want_final=True)
    want = sum(alpha ** h for h in range(hops + 1))
    assert np.allclose(out["final"].sum(axis=1), want, rtol=1e-12)


def test_identity_graph_scales_scores():
    """R = I (self-loops, weight 1): s^(H) = s0 * sum_h alpha^h, same top-k as alpha=0."""
    n = 150
    emb, q, *_ = tiny_store(6, n, 16, 1)
    row_ptr = np.arange(n + 1, dtype=np.int64)
    col = np.arange(n, dtype=np.int32)
    w = oracle.row_softmax(row_ptr, np.zeros(n, np.float32))
    base = oracle.retrieve(emb, q, None, None, None, tau=0.3, alpha=0, hops=0, k=10,
                           want_final=True)
    out = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=0.5, hops=2, k=10,
                          want_final=True)
    assert np.allclose(out["final"], base["final"] * 1.75, rtol=1e-13)
    assert (out["ids"] == base["ids"]).all()


def test_uniform_complete_graph_adds_constant():
    """Every row links to every chunk (itself included) with equal logits:
    (sR)_j = (sum_i s_i)/N, so s1 = s0 + alpha/N and the ranking is unchanged."""
    n = 60
    emb, q, *_ = tiny_store(7, n, 16, 1)
    row_ptr = np.arange(0, n * n + 1, n, dtype=np.int64)
    col = np.tile(np.arange(n, dtype=np.int32), n)
    w = oracle.row_softmax(row_ptr, np.zeros(n * n, np.float32))
    base = oracle.retrieve(emb, q, None, None, None, tau=0.3, alpha=0, hops=0, k=8,
                           want_final=True)
    out = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=0.5, hops=1, k=8,
                          want_final=True)
    assert np.allclose(out["final"], base["final"] + 0.5 / n, rtol=1e-12)
    assert (out["ids"] == base["ids"]).all()


# --------------------------------------------------------------------------- top-k / invariances
def test_permutation_invariance():
    """Relabel chunks (rows of E, graph, pages) by a random permutation: the
    selected set maps back, the scores agree.  Catches ID/position mix-ups."""
    n = 500
    emb, q, row_ptr, col, aff = tiny_store(8, n, 32, 6)
    page_of = (np.arange(n) // 16).astype(np.int32)
    w = oracle.row_softmax(row_ptr, aff)
    a = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.2, alpha=0.5, hops=2, k=16,
                        page_of=page_of)
    perm = np.random.default_rng(9).permutation(n)       # new id of old chunk i = perm[i]
    inv = np.argsort(perm)
    emb2 = emb[inv]
    rows, cols2, aff2 = [], [], []
    ptr = [0]
    for new in range(n):
        old = inv[new]
        seg = slice(row_ptr[old], row_ptr[old + 1])
        c = perm[col[seg]]
        o = np.argsort(c)
        cols2.append(c[o])
        aff2.append(aff[seg][o])
        ptr.append(ptr[-1] + len(c))
    rp2 = np.array(ptr, np.int64)
    col2 = np.concatenate(cols2).astype(np.int32)
    aff2 = np.concatenate(aff2).astype(np.float32)
    w2 = oracle.row_softmax(rp2, aff2)
    b = oracle.retrieve(emb2, q, rp2, col2, w2, tau=0.2, alpha=0.5, hops=2, k=16,
                        page_of=page_of[inv])
    for r in range(q.shape[0]):
        assert sorted(inv[b["ids"][r]]) == sorted(a["ids"][r])
        m = dict(zip(a["ids"][r], a["scores"][r]))
        for nid, sc in zip(b["ids"][r], b["scores"][r]):
            assert sc == pytest.approx(m[inv[nid]], rel=1e-12)
        assert b["n_pages"][r] == a["n_pages"][r]


def test_placement_invariance_and_page_bounds():
    """Page placement changes only the page outputs; ceil(k/P) <= n_pages <= k;
    ID-order placement gives len(set(id // P))."""
    n, k, P = 640, 24, 16
    emb, q, row_ptr, col, aff = tiny_store(10, n, 32, 5, n_q=6)
    w = oracle.row_softmax(row_ptr, aff)
    id_pages = (np.arange(n) // P).astype(np.int32)
    rnd_pages = (np.random.default_rng(11).permutation(n) // P).astype(np.int32)
    a = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.2, alpha=0.5, hops=1, k=k,
                        page_of=id_pages)
    b = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.2, alpha=0.5, hops=1, k=k,
                        page_of=rnd_pages)
    assert (a["ids"] == b["ids"]).all() and (a["scores"] == b["scores"]).all()
    for r in range(q.shape[0]):
        assert a["n_pages"][r] == len(set((a["ids"][r] // P).tolist()))
        assert list(b["page_ids"][r]) == list(rnd_pages[b["ids"][r]])
        assert b["n_pages"][r] == len(set(rnd_pages[b["ids"][r]].tolist()))
        for x in (a, b):
            assert math.ceil(k / P) <= x["n_pages"][r] <= k


def test_ties_resolve_to_lower_id():
    """Duplicate chunks score identically: the lower ID must come first."""
    rng = np.random.default_rng(12)
    base = synth.to_bf16(rng.standard_normal((50, 16)).astype(np.float32))
    emb = np.concatenate([base, base[::-1]])              # chunk i and 99-i identical
    q = synth.to_bf16(rng.standard_normal((2, 16)).astype(np.float32))
    out = oracle.retrieve(emb, q, None, None, None, tau=0.25, alpha=0, hops=0, k=20)
    for r in range(2):
        ids, sc = out["ids"][r], out["scores"][r]
        for a in range(19):
            assert sc[a] >= sc[a + 1]
            if sc[a] == sc[a + 1]:
                assert ids[a] < ids[a + 1]
        assert all((99 - i) in set(ids.tolist()) for i in ids[:18])


def test_batching_and_duplicate_queries():
    """Queries are independent: a batch equals single calls; repeats repeat."""
    emb, q, row_ptr, col, aff = tiny_store(13, 300, 32, 6, n_q=4)
    q = np.concatenate([q, q[1:2]])
    w = oracle.row_softmax(row_ptr, aff)
    batch = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.2, alpha=0.5, hops=2, k=7)
    for r in range(q.shape[0]):
        one = oracle.retrieve(emb, q[r:r + 1], row_ptr, col, w, tau=0.2, alpha=0.5, hops=2, k=7)
        assert (one["ids"][0] == batch["ids"][r]).all()
        assert (one["scores"][0] == batch["scores"][r]).all()
    assert (batch["ids"][4] == batch["ids"][1]).all()


def test_brute_force_enumeration_tiny():
    """N=7: enumerate every chunk's final score from the dense closed form
    and compare the whole ordering, for all k."""
    n = 7
    emb, q, row_ptr, col, aff = tiny_store(14, n, 8, 3, n_q=2)
    w = oracle.row_softmax(row_ptr, aff)
    R = dense_R(n, row_ptr, col, w)
    z = 0.5 * widen(q) @ widen(emb).T
    for k in range(1, n + 1):
        out = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.5, alpha=0.5, hops=2, k=k)
        for b in range(2):
            s = softmax_lib(z[b]) @ (np.eye(n) + 0.5 * R + 0.25 * R @ R)
            order = sorted(range(n), key=lambda i: (-s[i], i))[:k]
            assert list(out["ids"][b]) == order


def test_invalid_arguments():
    emb, q, row_ptr, col, aff = tiny_store(15, 20, 8, 3)
    w = oracle.row_softmax(row_ptr, aff)
    with pytest.raises(ValueError):
        oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=0.5, hops=1, k=21)
    with pytest.raises(ValueError):
        oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=-0.1, hops=1, k=3)


# --------------------------------------------------------------------------- relation update
def _update_case(seed=16, n_old=300, n_new=12, d=32, m=8, dup_of=None):
    rng = np.random.default_rng(seed)
    emb, _, row_ptr, col, aff = tiny_store(seed, n_old, d, 5)
    new = synth.to_bf16(rng.standard_normal((n_new, d)).astype(np.float32) * 0.3)
    if dup_of is not None:
        for a, j in dup_of.items():
            new[a] = emb[j]
    all_emb = np.concatenate([emb, new])
    rp = np.concatenate([row_ptr, np.full(n_new, row_ptr[-1], np.int64)])
    return all_emb, rp, col, aff, n_old, n_new, m


def test_update_brute_force_and_csr_shape():
    """Top-M neighbours equal numpy's lexsort of (-<e_n,e_i>, i); the new CSR
    keeps every old edge, adds M out-edges per new chunk and M reciprocal
    edges, columns ascending, no self-loops or repeats, and the reciprocal
    edge carries the same logit.  Catches a wrong neighbour set, a missing
    reciprocal edge, unsorted rows."""
    emb, rp, col, aff, first, n_new, m = _update_case()
    out = oracle.update_relations(emb, first, n_new, m, rp, col, aff, scale=10.0)
    E = widen(emb)
    for a in range(n_new):
        dots = E[:first] @ E[first + a]
        ref = np.lexsort((np.arange(first), -dots))[:m]
        assert list(out["nbr_ids"][a]) == list(ref)
        assert np.allclose(out["nbr_cos"][a], dots[ref], rtol=1e-13)
    nrp, ncol, naff = out["row_ptr"], out["col"], out["aff"]
    assert nrp[-1] == rp[-1] + 2 * n_new * m
    assert (np.diff(nrp) >= 0).all()
    old = {(i, int(c)): float(a) for i in range(first) for c, a in
           zip(col[rp[i]:rp[i + 1]], aff[rp[i]:rp[i + 1]])}
    new_edges = {}
    for i in range(first + n_new):
        c = ncol[nrp[i]:nrp[i + 1]]
        assert (np.diff(c) > 0).all() and (c != i).all()
        for cc, aa in zip(c, naff[nrp[i]:nrp[i + 1]]):
            new_edges[(i, int(cc))] = float(aa)
    for e, a in old.items():
        assert new_edges[e] == a
    for a in range(n_new):
        nid = first + a
        assert nrp[nid + 1] - nrp[nid] == m
        for j, c in zip(out["nbr_ids"][a], out["nbr_cos"][a]):
            lg = np.float32(10.0 * c)
            assert new_edges[(nid, int(j))] == lg
            assert new_edges[(int(j), nid)] == lg
    w = oracle.row_softmax(nrp, naff)
    sums = np.add.reduceat(w, nrp[:-1][np.diff(nrp) > 0])
    assert np.allclose(sums, 1.0, atol=1e-12)


def test_update_duplicate_chunk_is_top_neighbour():
    """A new chunk that duplicates prior chunk j has j as its first neighbour
    with cos = |e_j|^2 (unless an equal-dot chunk with a lower ID exists)."""
    emb, rp, col, aff, first, n_new, m = _update_case(seed=17, dup_of={0: 42, 3: 7})
    out = oracle.update_relations(emb, first, n_new, m, rp, col, aff)
    E = widen(emb)
    for a, j in ((0, 42), (3, 7)):
        assert out["nbr_ids"][a][0] == j
        assert out["nbr_cos"][a][0] == pytest.approx(E[j] @ E[j], rel=1e-15)


def test_update_without_reciprocal():
    emb, rp, col, aff, first, n_new, m = _update_case(seed=18)
    out = oracle.update_relations(emb, first, n_new, m, rp, col, aff, reciprocal=False)
    assert out["row_ptr"][-1] == rp[-1] + n_new * m
    assert (out["row_ptr"][:first + 1] == rp[:first + 1]).all()


def test_update_rejects_nonempty_new_rows():
    emb, rp, col, aff, first, n_new, m = _update_case(seed=19)
    rp = rp.copy()
    col2 = np.concatenate([col, np.array([0], np.int32)])
    aff2 = np.concatenate([aff, np.array([1.0], np.float32)])
    rp[first + 1:] += 1                                   # row `first` gains an edge
    with pytest.raises(ValueError):
        oracle.update_relations(emb, first, n_new, m, rp, col2, aff2)


# --------------------------------------------------------------------------- namespaces, SortByTime
def _dense_final(emb, q, row_ptr, col, w, tau, alpha, hops):
    """Final scores from the dense power series (numpy, gather form)."""
    n = emb.shape[0]
    S = sum(np.linalg.matrix_power(alpha * dense_R(n, row_ptr, col, w), h) for h in range(hops + 1))
    z = tau * widen(q) @ widen(emb).T
    return np.stack([softmax_lib(z[b]) @ S for b in range(q.shape[0])])


@pytest.mark.parametrize("hops", [0, 2])
def test_scoped_selection_is_restricted_sort(hops):
    """Namespace scope (§4.1: candidates are the caller's (user, session)
    chunks): the selected IDs are the top-k of the whole store's final
    scores restricted to the query's namespace, from the dense closed form.
    Catches masking applied to the wrong side (query vs chunk), masks that
    leak into propagation, and the padding when a namespace is smaller than k."""
    n, k = 150, 9
    emb, q, row_ptr, col, aff = tiny_store(21, n, 16, 6, n_q=4)
    w = oracle.row_softmax(row_ptr, aff)
    rng = np.random.default_rng(5)
    ns_of = rng.integers(0, 5, n).astype(np.int32)
    ns_of[ns_of == 4] = 3
    ns_of[:4] = 4                      # namespace 4 holds only chunks 0..3 (< k)
    q_ns = np.array([0, 2, 3, 4], np.int32)
    page_of = (np.arange(n) // 10).astype(np.int32)
    out = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=0.5, hops=hops, k=k,
                          page_of=page_of, ns_of=ns_of, q_ns=q_ns, want_final=True)
    ref = _dense_final(emb, q, row_ptr, col, w, 0.3, 0.5, hops)
    for b in range(4):
        cand = np.nonzero(ns_of == q_ns[b])[0]
        top = cand[np.lexsort((cand, -ref[b][cand]))][:k]
        got = out["ids"][b]
        assert list(got[:len(top)]) == list(top)
        assert (got[len(top):] == -1).all() and (out["page_ids"][b][len(top):] == -1).all()
        assert np.allclose(out["scores"][b][:len(top)], ref[b][top], rtol=1e-12)
        assert out["n_pages"][b] == len(set(page_of[top].tolist()))
        assert np.allclose(out["final"][b], ref[b], rtol=1e-12)   # scores of the whole store


def test_sort_by_time_reorders_only():
    """SortByTime (Algorithm 1): the same chunks as the score order, returned
    in ascending chunk ID (append order), padding last; with one namespace
    holding every chunk the scoped result equals the unscoped one."""
    n, k = 120, 7
    emb, q, row_ptr, col, aff = tiny_store(22, n, 16, 5, n_q=3)
    w = oracle.row_softmax(row_ptr, aff)
    base = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=0.5, hops=1, k=k)
    one = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=0.5, hops=1, k=k,
                          ns_of=np.zeros(n, np.int32), q_ns=np.zeros(3, np.int32))
    assert (one["ids"] == base["ids"]).all()
    tm = oracle.retrieve(emb, q, row_ptr, col, w, tau=0.3, alpha=0.5, hops=1, k=k,
                         sort_by_time=True)
    for b in range(3):
        assert list(tm["ids"][b]) == sorted(base["ids"][b].tolist())
        sc = dict(zip(base["ids"][b].tolist(), base["scores"][b].tolist()))
        assert [sc[i] for i in tm["ids"][b]] == tm["scores"][b].tolist()


# --------------------------------------------------------------------------- deletion
def test_drop_dead_is_edge_filter():
    """Deleting chunks drops exactly the edges into or out of them (numpy
    filter over the edge list), rows keep their column order."""
    emb, q, row_ptr, col, aff = tiny_store(31, 90, 8, 6)
    dead = np.zeros(90, bool)
    dead[[3, 17, 40, 41, 89]] = True
    rp, c, a = oracle.drop_dead(row_ptr, col, aff, dead)
    src = np.repeat(np.arange(90), np.diff(row_ptr))
    keep = ~dead[src] & ~dead[col]
    assert (np.diff(rp) == np.bincount(src[keep], minlength=90)).all()
    assert (c == col[keep]).all() and (a == aff[keep]).all()


@pytest.mark.parametrize("hops", [0, 2])
def test_deleted_chunks_equal_removed_store(hops):
    """A store with tombstoned chunks retrieves exactly like the store
    rebuilt without them (rows removed, graph re-indexed, weights re-softmaxed):
    same IDs (mapped back), same scores.  Catches a deleted chunk still
    counted in Z, still propagating mass, or still selectable."""
    n, k = 140, 8
    emb, q, row_ptr, col, aff = tiny_store(32, n, 16, 6, n_q=3)
    rng = np.random.default_rng(9)
    dead = np.zeros(n, bool)
    dead[rng.choice(n, 25, replace=False)] = True
    rp, c, a = oracle.drop_dead(row_ptr, col, aff, dead)
    w = oracle.row_softmax(rp, a)
    out = oracle.retrieve(emb, q, rp, c, w, tau=0.3, alpha=0.5, hops=hops, k=k, dead=dead)
    live = np.nonzero(~dead)[0]
    new_id = -np.ones(n, np.int64)
    new_id[live] = np.arange(live.size)
    src = np.repeat(np.arange(n), np.diff(rp))
    rp2 = np.concatenate([[0], np.cumsum(np.bincount(new_id[src], minlength=live.size))])
    c2 = new_id[c].astype(np.int32)
    w2 = oracle.row_softmax(rp2, a)
    ref = oracle.retrieve(emb[live], q, rp2, c2, w2, tau=0.3, alpha=0.5, hops=hops, k=k)
    assert (out["ids"] == live[ref["ids"]]).all()
    assert np.allclose(out["scores"], ref["scores"], rtol=1e-12)
