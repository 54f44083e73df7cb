"""CPU oracle of the Memory Manager: association-driven relocation and block
compaction of the page directory (arXiv 2607.05708, §4.2 and Algorithm 2).

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle``): the tests and the
benchmark's CPU baseline may use it; the product library never does.

Plain Python over small stores.  The paper's model calls are replaced by
their dense stand-ins (the same substitution as the Dense-only form, §5.5):

  co-retrieval statistics  sel(c) = number of requests whose retrieved set
      held chunk c, co(a, b) = number that held both.  A batch of requests
      adds its counts first; its relocations then run in request order.
  affinity(a, b) = co / (sel(a) + sel(b) - co) (the Jaccard index of the two
      chunks' request sets); "high pairwise association" is
      affinity >= tau_assoc (0.7 in the paper's sensitivity study, §5.5),
      decided exactly as  co >= tau * (sel(a) + sel(b) - co)  in fp64 with
      tau rounded to fp32 first.
  LLMCoLocate(S)  the chunks of S that have a partner in S at or above the
      threshold.  If two or more, not all on one page already, they are
      written out of place, in chronological order (SortByTime: chunk ID
      order), into fresh pages of P slots; each old copy becomes an invalid
      slot of its page (a tombstone).
  Block compaction: every page B whose invalid ratio
      phi(B) = invalid / total >= theta (0.75, §4.2) is compacted: its live
      chunks are partitioned by namespace (PartitionByUserSession), grouped
      within a partition by LLMGroup's stand-in -- connected components of
      the pairs at or above the affinity threshold (both chunks live on
      compacted pages, same namespace) -- and repacked into fresh pages
      partition by partition, group by group (groups ordered by their
      earliest chunk), chunk ID order within a group, P slots per page.
      Every partition starts on a fresh page, so no page ever holds chunks
      of two namespaces (§4.2: compaction never mixes tenants or sessions).
      Within a partition the groups are packed back to back and may share a
      page: Algorithm 2 packs each group "into one or more new blocks", but
      a fresh page per group would give every singleton survivor (the
      common case) a page of its own and multiply space by up to P, against
      the reclamation §4.2 gives as compaction's first purpose.  B is
      released.
  Deleted chunks (tombstones of a delete) are invalid slots of their pages;
      they are never relocated.

Accounting: slots_total = slots of pages in use (live + invalid), slots_live
= live chunks, chunk_writes = chunks written (appends, relocations,
compaction moves); space amplification = slots_total / slots_live, write
amplification = chunk_writes / appended chunks.

Pins: tests/test_memory_manager_oracle.py (a hand-worked trace in
tests/golden, invariants of the directory and of the counters, the
affinity rule against a brute-force Jaccard over the request sets, and the
compaction's packing against the connected components of the associated
pairs built independently with networkx).
"""
from __future__ import annotations

import numpy as np


class MemoryManager:
    def __init__(self, page_of, chunks_per_page, ns_of=None, dead=None):
        page_of = np.asarray(page_of, dtype=np.int64)
        self.n = page_of.shape[0]
        self.P = int(chunks_per_page)
        self.page = page_of.copy()                      # directory: chunk ID -> page
        self.ns = (np.zeros(self.n, np.int64) if ns_of is None
                   else np.asarray(ns_of, dtype=np.int64).copy())
        self.dead = np.zeros(self.n, bool) if dead is None else np.asarray(dead, bool).copy()
        self.total = {}
        self.live = {}
        for c in range(self.n):
            p = int(self.page[c])
            self.total[p] = self.total.get(p, 0) + 1
            self.live[p] = self.live.get(p, 0) + (0 if self.dead[c] else 1)
        self.next_page = int(page_of.max()) + 1 if self.n else 0
        self.sel = np.zeros(self.n, np.int64)
        self.co = {}
        self.appended = self.n
        self.writes = self.n

    # ------------------------------------------------------------------ statistics
    @staticmethod
    def _request_set(row):
        seen = []
        for c in row:
            c = int(c)
            if c >= 0 and c not in seen:
                seen.append(c)
        return seen

    def affinity_at_least(self, a, b, tau):
        key = (min(a, b), max(a, b))
        co = self.co.get(key, 0)
        union = int(self.sel[a] + self.sel[b] - co)
        t = float(np.float32(tau))
        return co > 0 and float(co) >= t * float(union)

    def _new_pages(self, chunks):
        """Write `chunks` (already ordered) into fresh pages, P per page."""
        for i, c in enumerate(chunks):
            old = int(self.page[c])
            self.live[old] -= 1
            p = self.next_page + i // self.P
            self.page[c] = p
            self.total[p] = self.total.get(p, 0) + 1
            self.live[p] = self.live.get(p, 0) + 1
        self.next_page += -(-len(chunks) // self.P)
        self.writes += len(chunks)

    # ------------------------------------------------------------------ Algorithm 2, relocation
    def relocate(self, requests, tau):
        """requests: int array [R, s] of retrieved chunk IDs (-1 padding)."""
        sets = []
        for row in np.asarray(requests):
            s = [c for c in self._request_set(row) if c < self.n and not self.dead[c]]
            sets.append(s)
            for c in s:
                self.sel[c] += 1
            for i in range(len(s)):
                for j in range(i + 1, len(s)):
                    key = (min(s[i], s[j]), max(s[i], s[j]))
                    self.co[key] = self.co.get(key, 0) + 1
        for s in sets:
            g = [c for c in s if any(self.affinity_at_least(c, d, tau) for d in s if d != c)]
            if len(g) < 2 or len({int(self.page[c]) for c in g}) == 1:
                continue
            self._new_pages(sorted(g))

    # ------------------------------------------------------------------ Algorithm 2, block compaction
    def compact(self, theta, tau):
        t = float(np.float32(theta))
        cand = sorted(p for p, tot in self.total.items()
                      if tot > 0 and float(tot - self.live[p]) >= t * float(tot))
        cset = set(cand)
        moving = [c for c in range(self.n) if not self.dead[c] and int(self.page[c]) in cset]
        mset = set(moving)
        parent = {c: c for c in moving}

        def find(x):
            while parent[x] != x:
                x = parent[x]
            return x

        for (a, b) in sorted(self.co):
            if a in mset and b in mset and self.ns[a] == self.ns[b] and \
                    self.affinity_at_least(a, b, tau):
                ra, rb = find(a), find(b)
                if ra != rb:
                    parent[max(ra, rb)] = min(ra, rb)   # root = earliest chunk of the group
        order = sorted(moving, key=lambda c: (int(self.ns[c]), find(c), c))
        for p in cand:
            self.total[p] = 0
            self.live[p] = 0
        p, fill, prev_ns = self.next_page - 1, self.P, None
        for c in order:
            if fill == self.P or int(self.ns[c]) != prev_ns:
                p, fill = p + 1, 0            # a full page, or a new partition
            self.page[c] = p
            self.total[p] = self.total.get(p, 0) + 1
            self.live[p] = self.live.get(p, 0) + 1
            fill, prev_ns = fill + 1, int(self.ns[c])
        self.next_page = p + 1
        self.writes += len(order)
        return cand

    # ------------------------------------------------------------------ deletion (tombstones)
    def delete(self, ids):
        for c in ids:
            c = int(c)
            if not self.dead[c]:
                self.dead[c] = True
                self.live[int(self.page[c])] -= 1

    def stats(self):
        in_use = [p for p, tot in self.total.items() if tot > 0]
        slots_total = sum(self.total[p] for p in in_use)
        slots_live = sum(self.live[p] for p in in_use)
        return dict(pages_in_use=len(in_use), slots_total=slots_total, slots_live=slots_live,
                    chunk_writes=self.writes, appended=self.appended)
