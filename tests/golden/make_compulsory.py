"""Write compulsory_bytes.json: the bytes a decode of each full-size workload
cannot avoid moving, with the latent texels counted by the oracle.

Every query record is read once (16 B), every output row written once (4 C
bytes), every distinct latent texel that a query's taps touch read once (16 B:
8 fp16 channels; the taps are the oracle's own addressing, both mips of a
blend), and every decoder's weights read once (fp16).  The benchmark divides
these bytes by the measured time for its compulsory roofline, beside the
algorithmic one (which counts every tap of every query).

Run from the repository root:  python tests/golden/make_compulsory.py
It calls only oracle/ and the seeded input generators.
"""
import json
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2608_27888_gb300 import workloads as W  # noqa: E402

OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "compulsory_bytes.json")
# (workload, the grouping used for the record; every grouping of a workload
# shares its latents and queries, so the touched texels are the same)
WORKLOADS = [("raster-256", None), ("uniform-4m", None), ("gbuffer-1080p", "identity"),
             ("gbuffer-2160p", "128"), ("gbuffer-2160p-x4-trilinear", None)]
CHUNK = 1 << 20


def touched_texels(a, q):
    """Distinct latent texels touched by the taps of every query."""
    total = a.latents.size // a.channels
    seen = np.zeros(total, dtype=bool)
    for s in range(0, len(q), CHUNK):
        idx, _, _ = oracle.taps(a, q[s:s + CHUNK])
        idx = idx.reshape(-1)
        seen[idx[idx != np.iinfo(np.uint64).max].astype(np.int64)] = True
    return int(seen.sum()), total


def main():
    rec = {"what": "bytes a decode must move at least: queries 16 B + outputs 4 C B each, distinct latent "
                   "texels touched (oracle taps) 16 B each, every decoder's fp16 weights once",
           "written_by": "tests/golden/make_compulsory.py", "workloads": {}}
    for name, variant in WORKLOADS:
        t0 = time.time()
        w = W.named(name, "full", variant)
        a, q = w.assets, w.queries
        u, total = touched_texels(a, q)
        n, C = len(q), a.out_dim
        H, I, L = a.hidden, a.in_dim, a.num_hidden_layers
        wbytes = a.num_decoders * (I * H + (L - 1) * H * H + C * H) * 2
        comp = 16 * n + 4 * C * n + 16 * u + wbytes
        rec["workloads"][name] = {"queries": n, "out_dim": C, "latent_texels": total, "touched_texels": u,
                                  "weight_bytes_per_decoder": wbytes // a.num_decoders,
                                  "compulsory_bytes_excluding_weights": 16 * n + 4 * C * n + 16 * u,
                                  "compulsory_bytes_per_query_excluding_weights":
                                      (16 * n + 4 * C * n + 16 * u) / n,
                                  "compulsory_bytes_with_record_grouping": comp, "grouping": variant}
        print(f"{name}: {n} queries, {u} of {total} texels touched, {comp / n:.1f} B/query "
              f"({time.time() - t0:.0f} s)", flush=True)
        del w, a, q
    with open(OUT, "w") as f:
        json.dump(rec, f, indent=1)
        f.write("\n")


if __name__ == "__main__":
    main()
