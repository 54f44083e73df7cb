"""GPU parity of the Memory Manager (relocation of co-retrieved chunks and
block compaction, Algorithm 2; phi(B) of §4.2) against the oracle in
oracle/memory_manager.py: the page directory and the page accounting must
be equal exactly (integer work)."""
import os

import numpy as np
import pytest

import synth
from oracle.memory_manager import MemoryManager

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "memory_manager_trace.txt")


@pytest.fixture(scope="module", autouse=True)
def _built():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_05708_gb300 import _build
    _build.build()


def _store(n, d, page_of, P, ns=None):
    import torch
    from paper_2607_05708_gb300 import MemStore
    rng = np.random.default_rng(n)
    emb = synth.to_bf16(rng.standard_normal((n, d)).astype(np.float32) / np.sqrt(d))
    st = MemStore.from_arrays(emb, page_of.astype(np.int32), np.zeros(n + 1, np.int64),
                              np.zeros(0, np.int32), np.zeros(0, np.float32), capacity=n,
                              chunks_per_page=P)
    if ns is not None:
        st.set_namespace(0, torch.from_numpy(ns.astype(np.int32)).cuda())
    return st


def _check(st, mm):
    pages = st.export_pages().cpu().numpy()
    live = ~mm.dead
    assert (pages[live] == mm.page[live]).all(), "page directory differs"
    got = st.page_stats()
    want = mm.stats()
    for key in ("pages_in_use", "slots_total", "slots_live", "chunk_writes", "appended"):
        assert got[key] == want[key], f"{key}: {got[key]} vs {want[key]}"


def test_golden_trace_on_gpu():
    """The hand-worked trace of tests/golden/memory_manager_trace.txt."""
    import torch
    g = {"request": []}
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, *v = line.split()
                v = [int(x) for x in v]
                if k == "request":
                    g["request"].append(v)
                else:
                    g[k] = v
    st = _store(8, 64, np.array(g["initial"]), 4)
    S = np.full((3, 3), -1, np.int64)
    for i, r in enumerate(g["request"]):
        S[i, :len(r)] = r
    st.relocate(torch.from_numpy(S).cuda(), 0.7)
    st.delete(torch.tensor(g["delete"], dtype=torch.int64, device="cuda"))
    assert st.compact_pages(0.75, 0.7) == len(g["released"])
    pages = st.export_pages().cpu().numpy()
    live = np.ones(8, bool)
    live[g["delete"]] = False
    assert (pages[live] == np.array(g["final"])[live]).all()
    stats = st.page_stats()
    for key in ("pages_in_use", "slots_total", "slots_live", "chunk_writes"):
        assert stats[key] == g[key][0], key


def _topic_trace(seed, n, n_req, s_len, n_topics=60, topic_size=6, loose=False, pool=None):
    """Seeded requests drawn from fixed topics (co-retrieved chunk groups)
    over the chunk IDs of `pool` (default: all).  Tight: a request retrieves
    all or all but one of its topic's chunks, so topic members reach a high
    co-retrieval affinity.  Loose: a random 2..s subset of the topic, so few
    pairs do.  Both add stray chunks, repeated IDs and -1 padding."""
    rng = np.random.default_rng(seed)
    pool = np.arange(n) if pool is None else np.asarray(pool)
    topics = [rng.choice(pool, topic_size, replace=False) for _ in range(n_topics)]
    pop = rng.zipf(1.3, n_topics).astype(np.float64)
    pop /= pop.sum()
    S = np.full((n_req, s_len), -1, np.int64)
    for r in range(n_req):
        t = topics[rng.choice(n_topics, p=pop)]
        k = rng.integers(2, s_len + 1) if loose else rng.integers(topic_size - 1, topic_size + 1)
        pick = rng.choice(t, size=min(k, t.size), replace=False)
        if rng.random() < 0.3:
            pick = np.concatenate([pick, rng.integers(0, n, 1)])
        if rng.random() < 0.1:
            pick = np.concatenate([pick, pick[:1]])
        S[r, :min(pick.size, s_len)] = pick[:s_len]
    return S


@pytest.mark.parametrize("tau", [0.5, 0.7])
def test_relocate_and_compact_match_oracle(tau):
    """4096 chunks, 16 per page, three namespaces; a loose then a tight
    batch of 400 topic-driven requests, deletions, two compactions: the
    directory and the accounting equal the oracle's after every step."""
    import torch
    n, P = 4096, 16
    page_of = np.arange(n) // P
    ns = (np.arange(n) * 7) % 3
    st = _store(n, 64, page_of, P, ns)
    mm = MemoryManager(page_of, P, ns_of=ns)
    rng = np.random.default_rng(8)
    for batch in range(2):
        S = _topic_trace(100 + batch, n, 400, 8, topic_size=12 if batch == 0 else 6,
                         loose=batch == 0)
        st.relocate(torch.from_numpy(S).cuda(), tau)
        mm.relocate(S, tau)
        _check(st, mm)
        victims = rng.choice(n, 150, replace=False)
        st.delete(torch.from_numpy(victims.astype(np.int64)).cuda())
        mm.delete(victims)
        _check(st, mm)
        rel = st.compact_pages(0.75, tau)
        assert rel == len(mm.compact(0.75, tau))
        _check(st, mm)
    assert mm.stats()["chunk_writes"] > n      # relocation and compaction did write


def test_compaction_groups_associated_chunks():
    """Block compaction with live chunks to move (§4.2, Algorithm 2): 40
    pages keep 4 survivors each and lose the other 12 (phi = 0.75), topics
    are drawn from the survivors, relocation runs at a strict threshold so
    few move, and compaction at a looser one groups the survivors by
    association (union-find by earliest chunk) within their namespaces."""
    import torch
    n, P = 4096, 16
    page_of = np.arange(n) // P
    ns = (np.arange(n) * 5) % 3
    rng = np.random.default_rng(21)
    pages = rng.choice(n // P, 40, replace=False)
    survivors, victims = [], []
    for p in pages:
        ids = rng.permutation(np.arange(p * P, (p + 1) * P))
        survivors += ids[:4].tolist()
        victims += ids[4:].tolist()
    st = _store(n, 64, page_of, P, ns)
    mm = MemoryManager(page_of, P, ns_of=ns)
    S = _topic_trace(31, n, 500, 8, n_topics=25, pool=survivors)
    st.relocate(torch.from_numpy(S).cuda(), 0.95)
    mm.relocate(S, 0.95)
    _check(st, mm)
    v = np.array(victims + rng.choice(n, 60, replace=False).tolist(), np.int64)
    st.delete(torch.from_numpy(v).cuda())
    mm.delete(v)
    _check(st, mm)
    w, first = mm.writes, mm.next_page
    rel = st.compact_pages(0.75, 0.5)
    assert rel == len(mm.compact(0.75, 0.5))
    _check(st, mm)
    assert mm.writes - w >= 100                 # survivors were moved, grouped
    # §4.2: compaction never mixes namespaces on a page; the three
    # namespaces' survivors do not fill whole pages
    pages = st.export_pages().cpu().numpy()
    moved = np.nonzero((pages >= first) & ~mm.dead)[0]
    per_ns = np.bincount(ns[moved], minlength=3)
    assert (per_ns > 0).all() and (per_ns % P != 0).any()
    for p in np.unique(pages[moved]):
        assert np.unique(ns[moved[pages[moved] == p]]).size == 1, p
    assert mm.next_page - first == sum(-(-int(v) // P) for v in per_ns)


def test_relocation_lowers_pages_per_request():
    """The point of relocation (§4.2): after the co-retrieved groups move
    together, the same requests touch fewer pages (directory from the GPU,
    page counts computed here)."""
    import torch
    n, P = 4096, 16
    page_of = np.random.default_rng(4).permutation(n) // P      # scattered layout
    st = _store(n, 64, page_of, P)
    S = _topic_trace(7, n, 600, 8)
    def pages_per_request(pages):
        return np.mean([len(set(pages[r[r >= 0]].tolist())) for r in S])
    before = pages_per_request(st.export_pages().cpu().numpy())
    st.relocate(torch.from_numpy(S).cuda(), 0.5)
    after = pages_per_request(st.export_pages().cpu().numpy())
    assert after < 0.5 * before, (before, after)
