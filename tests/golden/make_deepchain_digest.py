"""Writes deepchain_oracle_digest.txt: digests of the CPU oracle's outputs for
the whole deep-chain batch (L = 1024, 16,384 instances, seed 4), both directions.

Run from the repository root: python tests/golden/make_deepchain_digest.py
It calls only the oracle (and the input recipe in workloads.py) and takes about
20 minutes on 8 cores. The GPU test test_config_deepchain_full_batch_digest
compares the library's outputs for the same batch against these digests, chunk
by chunk, so that every instance of the batch is checked bit for bit without
running the oracle on the GPU machine.
"""
import hashlib
import os
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2101_07968_gb300 import workloads as wl  # noqa: E402

CHUNK = 256
OUT = os.path.join(os.path.dirname(os.path.abspath(__file__)), "deepchain_oracle_digest.txt")


def profile_digest(a: np.ndarray) -> str:
    return hashlib.sha256(np.ascontiguousarray(a, dtype="<i8").tobytes()).hexdigest()


def chunk_digest(out: dict, lo: int, hi: int) -> str:
    """sha256 over makespan (<i8), bits (<u4, row-major), nseg (<i4), status (<i4)."""
    h = hashlib.sha256()
    h.update(np.ascontiguousarray(out["makespan"][lo:hi], dtype="<i8").tobytes())
    h.update(np.ascontiguousarray(out["bits"][lo:hi], dtype="<u4").tobytes())
    h.update(np.ascontiguousarray(out["nseg"][lo:hi], dtype="<i4").tobytes())
    h.update(np.ascontiguousarray(out["status"][lo:hi], dtype="<i4").tobytes())
    return h.hexdigest()


def main():
    cfg = wl.config("deepchain")
    prof = oracle.profile_gen(cfg)
    B = cfg["batch"]
    lines = [
        "# Oracle outputs for the full deep-chain batch: L = 1024, 16,384 instances, seed 4",
        "# (the configuration of workloads.config('deepchain')), both directions.",
        "# Written by tests/golden/make_deepchain_digest.py, which calls only oracle/.",
        f"# profile <array> <sha256 of the [batch, L] (dt: [batch]) little-endian int64 array>",
        f"# chunk <direction 0 fwd / 1 bwd> <first instance> <end> <sha256 of makespan, bits, nseg, status>",
    ]
    for k in ("fc", "pt", "bc", "gt", "dt"):
        lines.append(f"profile {k} {profile_digest(prof[k])}")
    nthreads = os.cpu_count() or 1
    for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
        t0 = time.time()
        out = oracle.schedule_batch(d, prof[c], prof[x], prof["dt"], nthreads=nthreads)
        print(f"direction {d}: {time.time() - t0:.0f} s", flush=True)
        hist = np.bincount(out["nseg"])
        lines.append(f"# direction {d}: status counts {np.bincount(out['status']).tolist()}, "
                     f"makespan sum {int(out['makespan'].sum())}, "
                     f"nseg 1..{len(hist) - 1} counts {hist[1:].tolist()}")
        for lo in range(0, B, CHUNK):
            hi = min(B, lo + CHUNK)
            lines.append(f"chunk {d} {lo} {hi} {chunk_digest(out, lo, hi)}")
    with open(OUT, "w") as f:
        f.write("\n".join(lines) + "\n")


if __name__ == "__main__":
    main()
