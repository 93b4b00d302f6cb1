"""Write ``fullsize_oracle.json``: the oracle's results on the full-size
seeded workloads, as SHA-256 digests of every per-candidate field plus the
oracle's own top-16, keyed by workload, seed, size and the digest of the
inputs.

Calls only the oracle (``oracle/``) and the seeded input generator; nothing
here runs or reads the CUDA path.  The GPU full-size tests compare the
library's outputs with these digests and with a live oracle run on the same
inputs.  Run from the repository root:

    python tests/golden/make_fullsize_oracle.py [--threads N]
"""

from __future__ import annotations

import argparse
import json
import os
import sys
import time

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)
sys.path.insert(0, os.path.join(ROOT, "tests"))

import fullsize_common as F  # noqa: E402

OUT = os.path.join(HERE, "fullsize_oracle.json")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--threads", type=int, default=os.cpu_count() or 1)
    ap.add_argument("--only", default=None, help="one workload name")
    args = ap.parse_args()
    from oracle import oracle as O
    from paper_2609_34244_gb300 import workloads as W
    O.build()
    table = {}
    if os.path.exists(OUT):
        with open(OUT) as f:
            table = json.load(f)
    for name, n in F.FULL_SIZES:
        if args.only and name != args.only:
            continue
        t0 = time.time()
        w = W.make_workload(name, seed=F.SEED, n=n)
        ref = O.Oracle(w.cluster, w.model).price(w.cands, threads=args.threads, bounds=False)
        top = O.topk(ref, w.cands["M"], F.TOPK)
        table[F.key(name, n)] = F.record(w, ref, top)
        print("%s n=%d: %.1f s" % (name, n, time.time() - t0), flush=True)
    with open(OUT, "w") as f:
        json.dump(table, f, indent=1, sort_keys=True)
        f.write("\n")


if __name__ == "__main__":
    main()
