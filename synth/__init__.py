"""Seeded synthetic memory stores shaped like the paper's workloads.

The paper (arXiv 2607.05708) evaluates on LoCoMo, SWE-bench, BrowseComp and
WebArena (§5.1); none of those suites, nor any embedding store built from
them, is available here.  This module stands in for them with seeded,
synthetic stores of the five shapes the retrieval hot path is measured on:

    tiny     N=4096, d=256, iid unit vectors, 8 random out-edges per chunk
    gmm65k   N=65536, d=768, 512-component mixture, exact top-16 cosine graph
    gmm1m    N=1,048,576, d=1024, 4096-component Zipf(1.1) mixture,
             32 sampled out-edges per chunk with power-law in-degree
    update   4096 new chunks from the gmm1m mixture appended to gmm1m
    gmm4m    N=4,194,304, d=768, 16384-component Zipf(1.1) mixture,
             queries issued as 8 streams of 128

It produces INPUTS only: bf16 chunk and query embeddings (raw uint16 bits),
the relation graph as an out-edge CSR of edge logits (`aff`), and page
placements.  It holds none of the method's arithmetic: no softmax, no
propagation, no selection, no page counting.  The oracle and the CUDA path
both consume these arrays and share nothing else.

Generation is deterministic for a given (config, scale): every random draw
comes from `numpy.random.SeedSequence(seed)` children taken in a fixed
order over fixed-size row blocks, so the thread count never changes a value.
The exact cosine neighbours of the gmm65k graph are found with float64 dot
products of the stored bf16 values; each product is exact and the partial
sums of unit vectors stay within 53 bits, so neither the neighbour choice nor
its edge logits depend on the summation order.
"""
from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "Workload", "CONFIGS", "workload", "to_bf16", "bf16_to_f32",
    "zipf_sizes", "config_names",
]

_BLOCK = 65536          # graph rows per seeded block (fixed: results never depend on threads)
_EBLOCK = 8192          # embedding rows per seeded block


def _threads() -> int:
    return max(1, min(16, os.cpu_count() or 1))


# --------------------------------------------------------------------------- bf16
def to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round to nearest, ties to even); uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    if not np.isfinite(x).all():
        raise ValueError("to_bf16 expects finite values")
    u = x.view(np.uint32)
    r = u + np.uint32(0x7FFF)          # finite patterns stay below 2^32
    r += (u >> np.uint32(16)) & np.uint32(1)
    r >>= np.uint32(16)
    return r.astype(np.uint16)


def bf16_to_f32(h: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bits to float32."""
    h = np.ascontiguousarray(h, dtype=np.uint16)
    return (h.astype(np.uint32) << np.uint32(16)).view(np.float32)


# --------------------------------------------------------------------------- workload record
@dataclass
class Workload:
    name: str
    dim: int
    emb: np.ndarray                 # uint16 [N, dim]   bf16 chunk embeddings, ID order
    queries: np.ndarray             # uint16 [B, dim]   bf16 query embeddings
    row_ptr: np.ndarray             # int64  [N+1]      out-edge CSR
    col: np.ndarray                 # int32  [nnz]      targets, ascending within a row
    aff: np.ndarray                 # float32[nnz]      edge logits (weights = row softmax)
    page_of: dict                   # placement name -> int32 [N]
    chunks_per_page: int
    alpha: float
    hops: int
    k: int
    component: np.ndarray | None = None     # int32 [N] mixture component of each chunk
    temperature: float | None = None        # None: 1/sqrt(dim)
    streams: int = 1                        # queries issued as `streams` equal slices
    stream_order: np.ndarray | None = None  # arrival order of the slices
    new_emb: np.ndarray | None = None       # uint16 [n_new, dim] (relation update only)
    new_component: np.ndarray | None = None
    top_m: int = 0
    reciprocal: bool = True
    relation_scale: float = 10.0
    recipe: str = ""
    meta: dict = field(default_factory=dict)

    @property
    def n(self) -> int:
        return int(self.emb.shape[0])

    @property
    def n_queries(self) -> int:
        return int(self.queries.shape[0])

    @property
    def nnz(self) -> int:
        return int(self.col.shape[0])

    @property
    def tau(self) -> float:
        return self.temperature if self.temperature else 1.0 / math.sqrt(self.dim)


# --------------------------------------------------------------------------- helpers
def zipf_sizes(n_items: int, n_comp: int, s: float = 1.1) -> np.ndarray:
    """Component sizes proportional to (c+1)^-s, each >= 1, summing to n_items.

    One member is given to every component first; the remaining items are
    shared in proportion to the Zipf weights by the largest-remainder rule
    (ties broken towards the lower component index)."""
    if n_items < n_comp:
        raise ValueError("need at least one item per component")
    w = np.arange(1, n_comp + 1, dtype=np.float64) ** (-s)
    rest = n_items - n_comp
    quota = rest * (w / w.sum())
    base = np.floor(quota).astype(np.int64)
    rem = int(rest - base.sum())
    frac = quota - base
    order = np.lexsort((np.arange(n_comp), -frac))
    base[order[:rem]] += 1
    return base + 1


def _unit_rows(x: np.ndarray) -> np.ndarray:
    nrm = np.sqrt(np.einsum("ij,ij->i", x, x, dtype=np.float64))
    return (x / nrm[:, None]).astype(np.float32)


def _widen64(h: np.ndarray) -> np.ndarray:
    return bf16_to_f32(h).astype(np.float64)


def _parallel(fn, n_blocks: int):
    if n_blocks <= 1:
        for b in range(n_blocks):
            fn(b)
        return
    with ThreadPoolExecutor(max_workers=_threads()) as ex:
        list(ex.map(fn, range(n_blocks)))


def _iid_unit_bf16(seed_seq: np.random.SeedSequence, n: int, d: int) -> np.ndarray:
    out = np.empty((n, d), dtype=np.uint16)
    n_blocks = (n + _EBLOCK - 1) // _EBLOCK
    kids = seed_seq.spawn(n_blocks)

    def work(b):
        r0, r1 = b * _EBLOCK, min(n, (b + 1) * _EBLOCK)
        rng = np.random.default_rng(kids[b])
        x = rng.standard_normal((r1 - r0, d), dtype=np.float32)
        out[r0:r1] = to_bf16(_unit_rows(x))

    _parallel(work, n_blocks)
    return out


def _mixture_bf16(seed_seq, centers: np.ndarray, comp: np.ndarray, sigma: float) -> np.ndarray:
    n, d = comp.shape[0], centers.shape[1]
    out = np.empty((n, d), dtype=np.uint16)
    n_blocks = (n + _EBLOCK - 1) // _EBLOCK
    kids = seed_seq.spawn(n_blocks)

    def work(b):
        r0, r1 = b * _EBLOCK, min(n, (b + 1) * _EBLOCK)
        rng = np.random.default_rng(kids[b])
        x = rng.standard_normal((r1 - r0, d), dtype=np.float32)
        x *= np.float32(sigma)
        x += centers[comp[r0:r1]]
        out[r0:r1] = to_bf16(_unit_rows(x))

    _parallel(work, n_blocks)
    return out


def _centers(rng: np.random.Generator, n_comp: int, d: int) -> np.ndarray:
    c = rng.standard_normal((n_comp, d))
    c /= np.linalg.norm(c, axis=1, keepdims=True)
    return c.astype(np.float32)


def _placements(comp: np.ndarray | None, n: int, per_page: int, rng, kinds) -> dict:
    pages = {}
    ids = np.arange(n, dtype=np.int64)
    for kind in kinds:
        if kind == "id":
            pos = ids
        elif kind in ("clustered", "component"):
            order = np.lexsort((ids, comp))          # by (component, id)
            pos = np.empty(n, dtype=np.int64)
            pos[order] = ids
        elif kind == "random":
            order = rng.permutation(n)
            pos = np.empty(n, dtype=np.int64)
            pos[order] = ids
        else:
            raise ValueError(kind)
        pages[kind] = (pos // per_page).astype(np.int32)
    return pages


def _sort_rows(row_ptr: np.ndarray, col: np.ndarray, *payload):
    """Sort each CSR row by ascending column (stable), permuting payload alike."""
    n = row_ptr.shape[0] - 1
    rows = np.repeat(np.arange(n, dtype=np.int64), np.diff(row_ptr))
    order = np.lexsort((col, rows))
    return (col[order],) + tuple(p[order] for p in payload)


# --------------------------------------------------------------------------- graphs
def _random_graph(rng, n: int, deg: int):
    """`deg` distinct uniformly random out-neighbours per chunk, never itself."""
    col = np.empty((n, deg), dtype=np.int64)
    for i0 in range(0, n, _BLOCK):
        i1 = min(n, i0 + _BLOCK)
        r = i1 - i0
        picks = np.empty((r, deg), dtype=np.int64)
        # rejection by rows: draw deg values from n-1 candidates (skip self)
        for i in range(r):
            p = rng.choice(n - 1, size=deg, replace=False)
            p[p >= i0 + i] += 1
            picks[i] = p
        col[i0:i1] = picks
    col.sort(axis=1)
    row_ptr = np.arange(0, n * deg + 1, deg, dtype=np.int64)
    return row_ptr, col.reshape(-1).astype(np.int32)


def _knn_within_components(emb: np.ndarray, comp: np.ndarray, n_comp: int, m: int):
    """Exact top-m cosine neighbours of every chunk among its own component.

    Dots are float64 over the stored bf16 values (exact).  Order: cosine
    descending, then lower chunk ID; the chunk itself is excluded."""
    n = emb.shape[0]
    col = np.empty((n, m), dtype=np.int64)
    dots = np.empty((n, m), dtype=np.float64)
    members = np.argsort(comp, kind="stable")
    bounds = np.searchsorted(comp[members], np.arange(n_comp + 1))
    for c in range(n_comp):
        mem = members[bounds[c]:bounds[c + 1]]
        if mem.shape[0] <= m:
            raise ValueError("component smaller than m+1")
        x = _widen64(emb[mem])
        g = x @ x.T
        np.fill_diagonal(g, -np.inf)
        # order by (-dot, id): lexsort keys last-major
        idx = np.lexsort((np.broadcast_to(mem, g.shape), -g), axis=1)[:, :m]
        col[mem] = mem[idx]
        dots[mem] = np.take_along_axis(g, idx, axis=1)
    order = np.argsort(col, axis=1, kind="stable")
    col = np.take_along_axis(col, order, axis=1)
    dots = np.take_along_axis(dots, order, axis=1)
    row_ptr = np.arange(0, n * m + 1, m, dtype=np.int64)
    return row_ptr, col.reshape(-1).astype(np.int32), dots.reshape(-1)


def _first_distinct(cand: np.ndarray, rows: np.ndarray, deg: int):
    """Per row, the first `deg` candidates (in draw order) that are neither the
    row's own ID nor a repeat of an earlier candidate; -1 pads short rows."""
    r, m = cand.shape
    order = np.argsort(cand, axis=1, kind="stable")
    srt = np.take_along_axis(cand, order, axis=1)
    dup = np.zeros((r, m), dtype=bool)
    np.put_along_axis(dup, order[:, 1:], srt[:, 1:] == srt[:, :-1], axis=1)
    valid = ~dup & (cand != rows[:, None])
    rank = np.cumsum(valid, axis=1)
    keep = valid & (rank <= deg)
    out = np.full((r, deg), -1, dtype=np.int64)
    rr, cc = np.nonzero(keep)
    out[rr, rank[rr, cc] - 1] = cand[rr, cc]
    return out, np.minimum(rank[:, -1], deg)


def _popularity_graph(seed_seq, comp: np.ndarray, n_comp: int, deg: int,
                      p_in: float = 0.75, exponent: float = 1.1):
    """`deg` distinct out-neighbours per chunk with power-law in-degree.

    Every chunk gets a seeded popularity rank r (a permutation of 1..N) and
    weight r^-exponent.  Each draw for chunk i picks, with probability p_in,
    a member of i's own component, else any chunk of the store, in both cases
    with probability proportional to popularity.  Self and repeated picks
    are discarded and drawing continues until `deg` distinct targets exist;
    they are kept in draw order and then sorted ascending.

    Edge logit: 10 for an edge inside a component, 0 across components (the
    cosine of two members of one component is about 0.9, of two random
    centres about 0 +- 1/sqrt(d)), plus ln(U), U~U(0,1], so that weights
    inside a row vary."""
    n = comp.shape[0]
    rng = np.random.default_rng(seed_seq.spawn(1)[0])
    rank = rng.permutation(n).astype(np.float64) + 1.0
    pop = rank ** (-exponent)
    cs_all = np.cumsum(pop)
    members = np.argsort(comp, kind="stable")
    cs_comp = np.cumsum(pop[members])
    bounds = np.searchsorted(comp[members], np.arange(n_comp + 1))
    lo = np.concatenate(([0.0], cs_comp))[bounds[:-1]]      # cumulative before component
    hi = cs_comp[bounds[1:] - 1]
    col = np.empty((n, deg), dtype=np.int64)
    aff = np.empty((n, deg), dtype=np.float32)
    n_blocks = (n + _BLOCK - 1) // _BLOCK
    kids = seed_seq.spawn(n_blocks + 1)[1:]

    def draw(rng_b, rows, n_draw):
        c = comp[rows]
        r = rows.shape[0]
        u = rng_b.random((r, n_draw))
        inside = rng_b.random((r, n_draw)) < p_in
        small = (bounds[c + 1] - bounds[c]) <= 1
        inside &= ~small[:, None]
        v_in = lo[c][:, None] + u * (hi[c] - lo[c])[:, None]
        pos = np.searchsorted(cs_comp, v_in, side="right")
        pos = np.clip(pos, bounds[c][:, None], (bounds[c + 1] - 1)[:, None])
        t_in = members[pos]
        t_all = np.searchsorted(cs_all, u * cs_all[-1], side="right")
        t_all = np.minimum(t_all, n - 1)
        return np.where(inside, t_in, t_all)

    def work(b):
        rng_b = np.random.default_rng(kids[b])
        r0, r1 = b * _BLOCK, min(n, (b + 1) * _BLOCK)
        rows = np.arange(r0, r1)
        cand = draw(rng_b, rows, 2 * deg)
        out, got = _first_distinct(cand, rows, deg)
        todo = np.nonzero(got < deg)[0]
        width = 2 * deg
        while todo.shape[0]:
            width *= 2
            prev = out[todo]
            extra = draw(rng_b, rows[todo], width)
            cand = np.concatenate([np.where(prev < 0, rows[todo][:, None], prev), extra], axis=1)
            o2, g2 = _first_distinct(cand, rows[todo], deg)
            out[todo] = o2
            todo = todo[g2 < deg]
        out.sort(axis=1)
        col[r0:r1] = out
        same = comp[out] == comp[rows][:, None]
        jitter = np.log(1.0 - rng_b.random(out.shape))
        aff[r0:r1] = (10.0 * same + jitter).astype(np.float32)

    _parallel(work, n_blocks)
    row_ptr = np.arange(0, n * deg + 1, deg, dtype=np.int64)
    return row_ptr, col.reshape(-1).astype(np.int32), aff.reshape(-1)


# --------------------------------------------------------------------------- configs
CONFIGS = {
    0: dict(name="tiny", n=4096, dim=256, n_comp=0, deg=8, queries=4, hops=1,
            alpha=0.5, k=8, per_page=16, placements=("id",), seed=0),
    1: dict(name="gmm65k", n=65536, dim=768, n_comp=512, deg=16, queries=64, hops=1,
            alpha=0.5, k=16, per_page=32, placements=("component",), seed=1),
    2: dict(name="gmm1m", n=1_048_576, dim=1024, n_comp=4096, deg=32, queries=256, hops=2,
            alpha=0.5, k=32, per_page=64, placements=("clustered", "random"), seed=2),
    3: dict(name="update", n=1_048_576, dim=1024, n_comp=4096, deg=32, queries=256, hops=2,
            alpha=0.5, k=32, per_page=64, placements=("clustered",), seed=2,
            new=4096, top_m=32, new_seed=3),
    4: dict(name="gmm4m", n=4_194_304, dim=768, n_comp=16384, deg=32, queries=1024, hops=2,
            alpha=0.4, k=64, per_page=64, placements=("clustered", "random"), seed=4,
            streams=8, order_seed=1004),
}


def config_names():
    return {i: c["name"] for i, c in CONFIGS.items()}


def workload(index: int, scale: float = 1.0, placements=None) -> Workload:
    """Build config `index` (0..4).  `scale` < 1 shrinks N and the number of
    mixture components by the same factor (dim, B, k, hops, degree and page
    size are kept), for parity cases the oracle finishes in seconds."""
    cfg = dict(CONFIGS[index])
    n = max(64, int(round(cfg["n"] * scale)))
    d = cfg["dim"]
    kinds = tuple(placements) if placements else cfg["placements"]
    ss = np.random.SeedSequence(cfg["seed"])
    s_emb, s_graph, s_query, s_place, s_misc = ss.spawn(5)
    rng_misc = np.random.default_rng(s_misc)

    if index == 0:
        emb = _iid_unit_bf16(s_emb, n, d)
        rng_g = np.random.default_rng(s_graph)
        row_ptr, col = _random_graph(rng_g, n, cfg["deg"])
        u = 1.0 - rng_g.random(col.shape[0])               # U(0,1]
        aff = np.log(u).astype(np.float32)                 # softmax(log u) = u / sum(u)
        queries = _iid_unit_bf16(s_query, cfg["queries"], d)
        comp = None
        wl_centers = None
        recipe = ("iid N(0,1) rows, L2-normalised in fp32, rounded to bf16; 8 distinct uniform "
                  "out-neighbours per chunk (never itself); edge logit ln(U), U~U(0,1], so the row "
                  "softmax equals U row-normalised; queries from the same distribution; 16 chunks "
                  "per page in ID order")
    else:
        n_comp = max(2, int(round(cfg["n_comp"] * scale)))
        rng_c = np.random.default_rng(s_misc.spawn(1)[0])
        centers = _centers(rng_c, n_comp, d)
        if index == 1:
            sizes = np.full(n_comp, n // n_comp, dtype=np.int64)
            sizes[: n - sizes.sum()] += 1
        else:
            sizes = zipf_sizes(n, n_comp, 1.1)
        comp = rng_misc.permutation(np.repeat(np.arange(n_comp, dtype=np.int32), sizes))
        sigma = 0.3 / math.sqrt(d)
        emb = _mixture_bf16(s_emb, centers, comp, sigma)
        if index == 1:
            row_ptr, col, dots = _knn_within_components(emb, comp, n_comp, cfg["deg"])
            recipe = ("512 equal components, centres uniform on the unit sphere, member = centre + "
                      "N(0, (0.3/sqrt(d))^2 I), L2-normalised, bf16; graph = exact top-16 cosine "
                      "neighbours (within the component), edge logit 10*cos; queries = centre + "
                      "N(0,(0.1/sqrt(d))^2 I) around a uniformly drawn centre; 32 chunks per page "
                      "packed by component")
        else:
            row_ptr, col, aff = _popularity_graph(s_graph, comp, n_comp, cfg["deg"])
            recipe = (f"{n_comp} components with Zipf(1.1) sizes, centres uniform on the unit sphere, "
                      "member = centre + N(0,(0.3/sqrt(d))^2 I), L2-normalised, bf16; 32 distinct "
                      "out-neighbours per chunk drawn with probability 0.75 from its component, else "
                      "from the store, proportionally to a seeded popularity rank^-1.1 (power-law "
                      "in-degree); edge logit 10*[same component] + ln U, U~U(0,1]; queries near uniformly drawn centres "
                      "(std 0.1/sqrt(d)); 64 chunks per page, clustered (by component) and random")
        if index == 1:
            aff = (10.0 * dots).astype(np.float32)
        wl_centers = centers
        rng_q = np.random.default_rng(s_query)
        qc = rng_q.integers(0, n_comp, size=cfg["queries"])
        queries = _mixture_bf16(s_query.spawn(1)[0], centers, qc.astype(np.int32), 0.1 / math.sqrt(d))

    pages = _placements(comp, n, cfg["per_page"], np.random.default_rng(s_place), kinds)
    wl = Workload(
        name=cfg["name"], dim=d, emb=emb, queries=queries, row_ptr=row_ptr, col=col, aff=aff,
        page_of=pages, chunks_per_page=cfg["per_page"], alpha=cfg["alpha"], hops=cfg["hops"],
        k=cfg["k"], component=comp, streams=cfg.get("streams", 1), recipe=recipe,
        meta=dict(index=index, scale=scale, seed=cfg["seed"], centers=wl_centers),
    )
    if "order_seed" in cfg:
        wl.stream_order = np.random.default_rng(cfg["order_seed"]).permutation(cfg["streams"])
    if "new" in cfg:
        n_new = max(16, int(round(cfg["new"] * scale)))
        ss_new = np.random.SeedSequence(cfg["new_seed"])
        a, b = ss_new.spawn(2)
        probs = sizes / sizes.sum()
        new_comp = np.random.default_rng(a).choice(n_comp, size=n_new, p=probs).astype(np.int32)
        wl.new_emb = _mixture_bf16(b, centers, new_comp, 0.3 / math.sqrt(d))
        wl.new_component = new_comp
        wl.top_m = cfg["top_m"]
        wl.recipe += ("; update: new chunks from the same mixture (component drawn in proportion "
                      "to its size), "
                      "top-32 cosine neighbours among the old store, reciprocal edges")
    return wl


def query_batches(wl: Workload, count: int, seed: int = 2026) -> list:
    """`count` further query batches of the workload's size, drawn by the
    workload's own query recipe (mixture stores: a uniformly drawn centre +
    N(0, (0.1/sqrt(d))^2 I); the iid store: iid unit rows), unit length,
    bf16, from SeedSequence(seed).  Returns a list of uint16 [B, dim]."""
    ss = np.random.SeedSequence(seed)
    out = []
    centers = wl.meta.get("centers")
    for kid in ss.spawn(count):
        if centers is None:
            out.append(_iid_unit_bf16(kid, wl.n_queries, wl.dim))
        else:
            a, b = kid.spawn(2)
            qc = np.random.default_rng(a).integers(0, centers.shape[0], size=wl.n_queries)
            out.append(_mixture_bf16(b, centers, qc.astype(np.int32), 0.1 / math.sqrt(wl.dim)))
    return out


def request_trace(wl: Workload, n_queries: int, n_topics: int = 4096, s: float = 1.1,
                  seed: int = 2607, noise: float = 0.05) -> np.ndarray:
    """A replayable query trace for the Memory Manager workload: `n_topics`
    anchor chunks drawn uniformly from the store, each query an anchor drawn
    with Zipf(s) popularity by rank plus N(0, (noise/sqrt(d))^2 I), unit
    length, bf16.  Popular anchors recur, as the memory a long-running agent
    keeps re-reading does, so the same top-p sets are retrieved again and
    again.  Returns uint16 [n_queries, dim]."""
    ss = np.random.SeedSequence(seed)
    s_anchor, s_pick, s_noise = ss.spawn(3)
    anchors = np.random.default_rng(s_anchor).choice(wl.n, size=n_topics, replace=False)
    w = 1.0 / np.arange(1, n_topics + 1, dtype=np.float64) ** s
    pick = np.random.default_rng(s_pick).choice(n_topics, size=n_queries, p=w / w.sum())
    rows = bf16_to_f32(wl.emb[anchors[pick]])
    x = np.random.default_rng(s_noise).standard_normal(rows.shape, dtype=np.float32)
    x *= np.float32(noise / math.sqrt(wl.dim))
    x += rows
    return to_bf16(_unit_rows(x))
