"""Writes the stored oracle values of one complete 128-key block of Ktil and
Vtil for the N = 262,144 workload (B 1, H 4, N 262144, d 64, no mask, seed 4).

The block is key columns [199936, 200064) of head 1: a whole column block of
the kernels (128 keys), placed past 2^17 so that index arithmetic above that
point is covered.  Ktil_j and Vtil_j (eqs. 6-7; App. C steps 3 and 7) sum
over every query row, so the fp64 oracle runs all 262,144 rows of the head
(about an hour on 8 cores) and keeps only that block's column sums.

Only the oracle (oracle/) and the seeded input generator are called.  Usage:

    python tests/golden/make_n256k_d64_key_block.py

The output file, n256k_d64_head1_keys_199936.txt, is read by
tests/test_gpu_configs.py.
"""
from __future__ import annotations

import os
import sys
import time

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(_HERE)))

import oracle  # noqa: E402
from paper_2609_24089_gb300 import synth  # noqa: E402

WORKLOAD = "n256k_d64"
HEAD = 1
C0, C1 = 199936, 200064
OUT = os.path.join(_HERE, "n256k_d64_head1_keys_199936.txt")


def main():
    w = synth.WORKLOADS[WORKLOAD]
    bits = synth.make_inputs(w.B, w.H, w.N, w.d, w.seed, w.sigma, heads=[HEAD])
    X = [synth.to_f64(bits[n][0, 0]) for n in synth.NAMES]
    t0 = time.time()
    r = oracle.bob_head(*X, w.scale, w.causal, rows=np.arange(w.N, dtype=np.int64),
                        cols=(C0, C1), row_outputs=False, head=HEAD)
    dt = time.time() - t0
    with open(OUT + ".tmp", "w") as f:
        f.write(f"# workload {WORKLOAD}: B {w.B}, H {w.H}, N {w.N}, d {w.d}, causal {int(w.causal)},"
                f" seed {w.seed}, scale 1/sqrt({w.d})\n")
        f.write(f"# head {HEAD}, key columns [{C0}, {C1}): Ktil then Vtil, one key per line,"
                f" {w.d} values each\n")
        f.write("# Ktil_j = tau sum_i (Stil_ij q_i + dS_ij u_Q,i), Vtil_j = sum_i P_ij h_ij do_i"
                " (eqs. 6-7; App. C steps 3, 7), all rows i of the head\n")
        f.write(f"# written by tests/golden/make_n256k_d64_key_block.py (fp64 oracle,"
                f" {dt:.0f} s)\n")
        for name in ("kbar", "vbar"):
            for row in r[name]:
                f.write(" ".join(f"{x:.7e}" for x in row) + "\n")
    os.replace(OUT + ".tmp", OUT)


def load(path=OUT):
    """(kbar, vbar) of the stored block, each (C1 - C0) x d float64."""
    a = np.loadtxt(path, comments="#", dtype=np.float64)
    n = C1 - C0
    assert a.shape[0] == 2 * n, a.shape
    return a[:n], a[n:]


if __name__ == "__main__":
    main()
