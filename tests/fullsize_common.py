"""Shared definitions of the full-size parity records: which workloads, and
how a record (input digest, per-field digests of the oracle's results, the
oracle's top-k) is formed.  Used by the script that writes
``golden/fullsize_oracle.json`` (oracle only) and by the GPU tests that read
it.  Holds no pricing arithmetic."""

from __future__ import annotations

import hashlib

import numpy as np

SEED = 0
TOPK = 16
# the four generated workloads at the sizes that define them (tiny is
# enumerated and compared in full by the parity suite)
FULL_SIZES = (("dense32", 100_000), ("dense80", 1_000_000), ("moe48", 1_000_000), ("stress128", 10_000_000))
FIELDS = (("T", "<i8"), ("bottleneck", "<i8"), ("n_dp", "<u2"), ("status", "u1"))


def key(name: str, n: int) -> str:
    return "%s/seed%d/n%d" % (name, SEED, n)


def digest(a, dtype) -> str:
    return hashlib.sha256(np.ascontiguousarray(np.asarray(a).astype(dtype, copy=False)).tobytes()).hexdigest()


def input_digest(cands: dict) -> str:
    h = hashlib.sha256()
    for k, dt in (("S", "u1"), ("M", "<u2"), ("code", "u1")):
        h.update(np.ascontiguousarray(np.asarray(cands[k]).astype(dt, copy=False)).tobytes())
    return h.hexdigest()


def field_digests(res: dict) -> dict:
    return {k: digest(res[k], dt) for k, dt in FIELDS}


def record(w, ref: dict, top: dict) -> dict:
    return {"workload": w.name, "seed": SEED, "n": int(w.n), "inputs_sha256": input_digest(w.cands),
            "fields_sha256": field_digests(ref),
            "status_counts": {str(s): int(c) for s, c in zip(*np.unique(ref["status"], return_counts=True))},
            "topk": {"k": TOPK, "count": int(top["count"]), "idx": [int(x) for x in top["idx"]],
                     "T": [int(x) for x in top["T"]], "nM": [int(x) for x in top["nM"]]}}
