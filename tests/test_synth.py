"""The seeded workload generator: determinism and the structure each
workload promises (the inputs of every parity test and of the benchmark)."""
import hashlib

import numpy as np
import pytest

import synth


def _digest(wl):
    h = hashlib.sha256()
    for a in (wl.emb, wl.queries, wl.row_ptr, wl.col, wl.aff, *wl.page_of.values()):
        h.update(np.ascontiguousarray(a).tobytes())
    return h.hexdigest()


def test_deterministic():
    assert _digest(synth.workload(0)) == _digest(synth.workload(0))
    assert _digest(synth.workload(2, scale=1 / 256)) == _digest(synth.workload(2, scale=1 / 256))


def test_bf16_rounding_ties_to_even():
    v = np.array([1.0, 1.00390625, 1.005859375, -1.00390625, 3.0e-38, 0.0], np.float32)
    assert list(synth.to_bf16(v)) == [0x3F80, 0x3F80, 0x3F81, 0xBF80, 0x0123, 0x0000]
    x = np.random.default_rng(0).standard_normal(1000).astype(np.float32)
    back = synth.bf16_to_f32(synth.to_bf16(x))
    assert np.all(np.abs(back - x) <= np.abs(x) * 2.0 ** -8)


def _check_csr(wl, deg):
    n = wl.n
    assert wl.row_ptr[0] == 0 and wl.row_ptr[-1] == wl.nnz
    assert (np.diff(wl.row_ptr) == deg).all()
    rows = np.repeat(np.arange(n), deg)
    assert (wl.col != rows).all(), "self loops"
    c = wl.col.reshape(n, deg)
    assert (np.diff(c, axis=1) > 0).all(), "columns not strictly ascending"
    assert (c >= 0).all() and (c < n).all()
    assert np.isfinite(wl.aff).all()


def test_tiny_store_shape():
    wl = synth.workload(0)
    assert (wl.n, wl.dim, wl.n_queries, wl.k, wl.hops, wl.alpha) == (4096, 256, 4, 8, 1, 0.5)
    _check_csr(wl, 8)
    assert (wl.aff <= 0).all()                         # ln U, U in (0, 1]
    assert (wl.page_of["id"] == np.arange(wl.n) // 16).all()
    norms = np.linalg.norm(synth.bf16_to_f32(wl.emb), axis=1)
    assert np.allclose(norms, 1.0, atol=1e-2)


def test_gmm65k_graph_is_exact_cosine_knn():
    """Within-component top-16 equals the global top-16 (checked on a sample
    against every chunk of the store)."""
    wl = synth.workload(1, scale=1 / 16)
    _check_csr(wl, 16)
    E = synth.bf16_to_f32(wl.emb).astype(np.float64)
    rng = np.random.default_rng(0)
    for i in rng.choice(wl.n, size=40, replace=False):
        dots = E @ E[i]
        dots[i] = -np.inf
        ref = np.lexsort((np.arange(wl.n), -dots))[:16]
        assert sorted(ref) == sorted(wl.col[wl.row_ptr[i]:wl.row_ptr[i + 1]])
        assert np.allclose(wl.aff[wl.row_ptr[i]:wl.row_ptr[i + 1]],
                           10 * dots[np.sort(ref)], atol=1e-5)


def test_gmm1m_recipe_power_law_and_placements():
    wl = synth.workload(2, scale=1 / 64)
    _check_csr(wl, 32)
    indeg = np.bincount(wl.col, minlength=wl.n)
    assert indeg.max() > 50 * np.median(indeg)        # heavy-tailed in-degree
    sizes = np.bincount(wl.component)
    assert sizes.sum() == wl.n and sizes.min() >= 1
    assert sizes.max() > 20 * np.median(sizes)        # Zipf component sizes
    for kind in ("clustered", "random"):
        pages = wl.page_of[kind]
        assert np.bincount(pages).max() <= wl.chunks_per_page
    # clustered pages hold one component each except at component boundaries
    cl = wl.page_of["clustered"]
    mixed = sum(len(set(wl.component[cl == p])) > 1 for p in range(cl.max() + 1))
    assert mixed <= wl.component.max() + 1


def test_zipf_sizes():
    s = synth.zipf_sizes(1000, 10, 1.1)
    assert s.sum() == 1000 and (s >= 1).all() and (np.diff(s) <= 0).all()


def test_update_workload():
    wl = synth.workload(3, scale=1 / 256)
    assert wl.new_emb.shape == (16, wl.dim) and wl.top_m == 32
    assert wl.new_component.max() <= wl.component.max()


def test_request_trace():
    """The Memory Manager's query trace: deterministic for a seed, unit-length
    bf16 rows, each within the noise of one of the anchor chunks, and the
    anchors' popularity falling with rank like Zipf(1.1) (the most popular
    anchor draws about 1 / H_{512, 1.1} of the queries here)."""
    wl = synth.workload(0)
    a = synth.request_trace(wl, 4000, n_topics=512)
    b = synth.request_trace(wl, 4000, n_topics=512)
    assert a.dtype == np.uint16 and a.shape == (4000, wl.dim)
    assert np.array_equal(a, b)
    assert not np.array_equal(a, synth.request_trace(wl, 4000, n_topics=512, seed=1))
    x = synth.bf16_to_f32(a).astype(np.float64)
    assert np.allclose(np.linalg.norm(x, axis=1), 1.0, atol=1e-2)
    e = synth.bf16_to_f32(wl.emb).astype(np.float64)
    e /= np.linalg.norm(e, axis=1, keepdims=True)
    nearest = (x @ e.T).argmax(axis=1)
    cos = (x @ e.T).max(axis=1)
    assert cos.min() > 0.99                     # noise 0.05 / sqrt(d) per dimension
    counts = np.bincount(nearest, minlength=wl.n)
    top = np.sort(counts)[::-1]
    h = (1.0 / np.arange(1, 513) ** 1.1).sum()
    assert abs(top[0] / 4000 - 1 / h) < 0.03
    assert (counts > 0).sum() <= 512


def test_gmm1m_edge_logits_follow_the_stated_reading():
    """gmm1m / gmm4m edge logits are 10 * [same mixture component] + ln U with
    U ~ U(0, 1] (the reading recorded for these sampled graphs, standing in for
    10 * cos: inside a component the cosine is about 0.9, across about 0): the
    remainder aff - 10 * same is <= 0, finite and spread like ln U (mean -1,
    standard deviation 1), and most edges stay inside their component (each
    draw lands there with probability 0.75, less where a component is too
    small to hold distinct targets: about 0.65 at this scale)."""
    wl = synth.workload(2, scale=1 / 64)
    src = np.repeat(np.arange(wl.n), np.diff(wl.row_ptr))
    same = wl.component[src] == wl.component[wl.col]
    rest = wl.aff.astype(np.float64) - 10.0 * same
    assert np.isfinite(rest).all() and (rest <= 0).all()
    assert abs(rest.mean() + 1.0) < 0.02            # E[ln U] = -1
    assert abs(rest.std() - 1.0) < 0.02             # Var[ln U] = 1
    assert 0.6 <= same.mean() < 0.9
    # inside a component the cosine is high, across it is near zero
    E = synth.bf16_to_f32(wl.emb).astype(np.float64)
    pick = np.random.default_rng(1).choice(src.size, 2000, replace=False)
    cos = np.einsum("ij,ij->i", E[src[pick]], E[wl.col[pick]])
    assert cos[same[pick]].mean() > 0.8 and abs(cos[~same[pick]].mean()) < 0.05
