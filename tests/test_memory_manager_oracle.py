"""Pins for the Memory Manager oracle (oracle/memory_manager.py): the hand-
worked trace of tests/golden/memory_manager_trace.txt (Algorithm 2, §4.2),
the affinity rule against a brute-force Jaccard over the request sets, and
invariants of the directory and counters on seeded random traces."""
import os

import numpy as np
import pytest

from oracle.memory_manager import MemoryManager

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "memory_manager_trace.txt")


def _golden():
    g = {"request": []}
    with open(GOLDEN) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *vals = line.split()
            vals = [int(v) for v in vals]
            if key == "request":
                g["request"].append(vals)
            else:
                g[key] = vals
    return g


def test_golden_trace():
    g = _golden()
    mm = MemoryManager(np.array(g["initial"]), g["pages_per_slot"][0])
    reqs = np.full((len(g["request"]), 3), -1)
    for i, r in enumerate(g["request"]):
        reqs[i, :len(r)] = r
    mm.relocate(reqs, 0.7)
    mm.delete(g["delete"])
    released = mm.compact(0.75, 0.7)
    assert list(mm.page) == g["final"]
    assert released == g["released"]
    st = mm.stats()
    for key in ("pages_in_use", "slots_total", "slots_live", "chunk_writes"):
        assert st[key] == g[key][0], key


def _random_trace(seed, n=300, P=8, n_req=120, s=6, n_comp=12):
    rng = np.random.default_rng(seed)
    comp = rng.integers(0, n_comp, n)
    page_of = np.arange(n) // P
    reqs = np.full((n_req, s), -1)
    for r in range(n_req):
        c = rng.integers(0, n_comp)
        members = np.nonzero(comp == c)[0]
        k = min(s, members.size)
        reqs[r, :k] = rng.choice(members, size=k, replace=False)
    return page_of, reqs, comp


def test_affinity_is_jaccard_of_request_sets():
    """affinity >= tau exactly when |A ∩ B| / |A ∪ B| >= tau for the sets of
    requests that retrieved each chunk (computed here from the sets)."""
    page_of, reqs, _ = _random_trace(1)
    mm = MemoryManager(page_of, 8)
    mm.relocate(reqs, 0.7)
    sets = {}
    for r, row in enumerate(reqs):
        for c in set(int(x) for x in row if x >= 0):
            sets.setdefault(c, set()).add(r)
    ids = sorted(sets)
    for a in ids[:60]:
        for b in ids[:60]:
            if a >= b:
                continue
            inter = len(sets[a] & sets[b])
            union = len(sets[a] | sets[b])
            for tau in (0.2, 0.3, 0.5, 0.7):
                # the decision in fp64 with tau rounded to fp32 (exact here:
                # small integers times a 24-bit fraction)
                want = inter > 0 and inter >= float(np.float32(tau)) * union
                assert mm.affinity_at_least(a, b, tau) == want


@pytest.mark.parametrize("seed", [2, 3, 4])
def test_directory_invariants(seed):
    """Every live chunk sits on exactly one page in use; per-page live
    counts match the directory; slots never fall below live chunks; writes
    add up; after compaction no page in use has phi >= theta; relocated
    groups occupy their fresh pages in chunk-ID order."""
    page_of, reqs, comp = _random_trace(seed)
    mm = MemoryManager(page_of, 8, ns_of=comp % 3)
    rng = np.random.default_rng(seed)
    for half in (reqs[:60], reqs[60:]):
        before = mm.next_page
        mm.relocate(half, 0.5)
        # fresh pages hold chunk IDs in ascending order within each page
        for p in range(before, mm.next_page):
            members = np.nonzero(mm.page == p)[0]
            assert (np.diff(members) > 0).all()
        mm.delete(rng.choice(mm.n, 10, replace=False))
        mm.compact(0.75, 0.5)
        live = ~mm.dead
        counts = np.bincount(mm.page[live], minlength=mm.next_page)
        for p in range(mm.next_page):
            assert mm.live.get(p, 0) == counts[p]
            assert mm.total.get(p, 0) >= mm.live.get(p, 0)
            tot = mm.total.get(p, 0)
            if tot > 0:
                assert (tot - mm.live[p]) < 0.75 * tot
        st = mm.stats()
        assert st["slots_live"] == int(live.sum())
        assert st["slots_total"] >= st["slots_live"]


@pytest.mark.parametrize("seed", [5, 6, 7])
def test_compaction_packs_connected_components(seed):
    """Block compaction against an independent construction: the live
    chunks of the pages whose invalid ratio reaches theta, the graph of
    their associated pairs (same namespace, Jaccard index of the two chunks'
    request sets >= tau, computed here from the trace), its connected
    components (networkx), and the packing by (namespace, earliest chunk of
    the component, chunk ID), P chunks per fresh page from the next free
    page on, each namespace starting on a page of its own (§4.2)."""
    nx = pytest.importorskip("networkx")
    # relocation at 0.5 leaves tombstones; compaction groups at 0.2, so that
    # associated pairs remain among the chunks it moves
    tau_r, tau, theta, P = 0.5, 0.2, 0.75, 8
    page_of, reqs, comp = _random_trace(seed)
    ns = comp % 3
    mm = MemoryManager(page_of, P, ns_of=ns)
    mm.relocate(reqs, tau_r)
    rng = np.random.default_rng(seed)
    mm.delete(rng.choice(mm.n, 60, replace=False))
    cand = sorted(p for p, tot in mm.total.items()
                  if tot > 0 and (tot - mm.live[p]) >= np.float32(theta) * tot)
    moving = [c for c in range(mm.n) if not mm.dead[c] and int(mm.page[c]) in set(cand)]
    sets = {}
    for r, row in enumerate(reqs):
        for c in set(int(x) for x in row if x >= 0):
            sets.setdefault(c, set()).add(r)
    g = nx.Graph()
    g.add_nodes_from(moving)
    for i, a in enumerate(moving):
        for b in moving[i + 1:]:
            if ns[a] != ns[b] or a not in sets or b not in sets:
                continue
            inter = len(sets[a] & sets[b])
            if inter and inter >= float(np.float32(tau)) * len(sets[a] | sets[b]):
                g.add_edge(a, b)
    comps = sorted((sorted(cc) for cc in nx.connected_components(g)),
                   key=lambda cc: (int(ns[cc[0]]), cc[0]))
    assert cand and max(len(cc) for cc in comps) >= 2          # not vacuous
    first = mm.next_page
    expect, base = {}, first
    for t in sorted({int(ns[c]) for c in moving}):
        members = [c for cc in comps if int(ns[cc[0]]) == t for c in cc]
        for i, c in enumerate(members):
            expect[c] = base + i // P
        base += -(-len(members) // P)
    released = mm.compact(theta, tau)
    assert released == cand
    for c, p in expect.items():
        assert mm.page[c] == p, (c, p)
    assert mm.next_page == base
    for p in cand:
        assert mm.total[p] == 0 and mm.live[p] == 0


@pytest.mark.parametrize("seed", [5, 8, 9])
def test_compaction_never_mixes_namespaces(seed):
    """§4.2: block compaction partitions the survivors by user and session
    (PartitionByUserSession, Algorithm 2), so it never mixes chunks of two
    tenants or sessions on a page.  Three namespaces whose survivor counts
    are not multiples of P: every page compaction writes holds a single
    namespace, and each namespace fills exactly ceil(survivors / P) pages.
    Packing the survivors back to back across namespaces fails this."""
    tau_r, tau, theta, P = 0.5, 0.2, 0.75, 8
    page_of, reqs, comp = _random_trace(seed)
    ns = (comp * 7 + 3) % 5 % 3
    mm = MemoryManager(page_of, P, ns_of=ns)
    mm.relocate(reqs, tau_r)
    rng = np.random.default_rng(seed + 100)
    mm.delete(rng.choice(mm.n, 60, replace=False))
    first = mm.next_page
    released = mm.compact(theta, tau)
    moved = [c for c in range(mm.n) if not mm.dead[c] and mm.page[c] >= first]
    counts = {}
    for c in moved:
        counts[int(ns[c])] = counts.get(int(ns[c]), 0) + 1
    assert released and len(counts) == 3                      # not vacuous
    assert any(v % P for v in counts.values())
    owner = {}
    for c in moved:
        assert owner.setdefault(int(mm.page[c]), int(ns[c])) == int(ns[c]), c
    for t, v in counts.items():
        assert len({int(mm.page[c]) for c in moved if ns[c] == t}) == -(-v // P)
    assert mm.next_page - first == sum(-(-v // P) for v in counts.values())
