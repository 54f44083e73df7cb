"""Writes tests/golden/update_gmm1m_top32.npz: the oracle's relation update of
the full-size update workload (4096 new chunks of the gmm1m mixture appended
to the N = 1,048,576 store, top-32 cosine neighbours among the prior chunks,
§4.1 / Algorithm 1 LLMSelect of related prior chunks in its Dense-only form).

Only oracle/ computes: every new chunk's top-32 prior neighbours in (cos
desc, ID asc) order and their fp64 cosines, from oracle.update_relations.
The new chunks are independent of one another (new chunks are linked only to
prior chunks), so the script runs the oracle on slices of them in a few
threads (the oracle's C code releases the interpreter lock) and
concatenates the slices; the relation graph plays no part in the
selection, so each slice passes an empty one.  Stored with the SHA-256 of
the generated inputs, which the GPU test checks before it compares.

    python tests/golden/make_update_golden.py [--threads T]

Takes about 3 CPU-hours of oracle work (about 2.7 s per new chunk on one
core)."""
from __future__ import annotations

import argparse
import hashlib
import os
import sys
import time
from concurrent.futures import ThreadPoolExecutor

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

OUT = os.path.join(HERE, "update_gmm1m_top32.npz")
SLICE = 16


def input_digest(wl) -> str:
    h = hashlib.sha256()
    for a in (wl.emb, wl.new_emb, wl.row_ptr, wl.col, wl.aff):
        h.update(np.ascontiguousarray(a).tobytes())
    return h.hexdigest()


def main():
    import oracle
    import synth
    ap = argparse.ArgumentParser()
    ap.add_argument("--threads", type=int, default=os.cpu_count() or 1)
    args = ap.parse_args()
    wl = synth.workload(3)
    n_old, n_new, m = wl.n, wl.new_emb.shape[0], wl.top_m
    ids = np.zeros((n_new, m), np.int32)
    cos = np.zeros((n_new, m), np.float64)
    no_col, no_aff = np.zeros(0, np.int32), np.zeros(0, np.float32)
    t0 = time.time()

    def work(s0):
        s1 = min(n_new, s0 + SLICE)
        emb = np.concatenate([wl.emb, wl.new_emb[s0:s1]])
        rp = np.zeros(n_old + (s1 - s0) + 1, np.int64)
        r = oracle.update_relations(emb, n_old, s1 - s0, m, rp, no_col, no_aff,
                                    scale=wl.relation_scale, reciprocal=True)
        ids[s0:s1] = r["nbr_ids"]
        cos[s0:s1] = r["nbr_cos"]
        print(f"new chunks {s0}..{s1 - 1} done at {time.time() - t0:.0f} s", flush=True)

    with ThreadPoolExecutor(max_workers=args.threads) as ex:
        list(ex.map(work, range(0, n_new, SLICE)))
    np.savez_compressed(OUT, nbr_ids=ids, nbr_cos=cos, inputs_sha256=np.array(input_digest(wl)),
                        n_old=np.int64(n_old), top_m=np.int64(m))
    print(f"wrote {OUT} in {time.time() - t0:.0f} s")


if __name__ == "__main__":
    main()
