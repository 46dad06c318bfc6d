"""The pins have power: each planted mistake in the oracle fails them.

The oracle source carries ten deliberately wrong variants behind the
compile-time switch FBOB_MUTANT (a dropped term, a wrong sign, a transposed
operand, a wrong index, a dropout gate left out ...).  Each is built into a
temporary directory and run through the finite-difference pin, without and
with dropout; every one must be caught.  The
default build (FBOB_MUTANT=0) is the oracle itself.
"""
import numpy as np
import pytest

import oracle
from tests import pins


@pytest.mark.parametrize("mutant", list(range(1, 11)))
def test_planted_mistake_is_caught(mutant):
    out_dir = oracle.mutant_build_dir()
    oracle.build(mutant=mutant, out_dir=out_dir)
    caught = []
    for (N, d, causal, p) in ((12, 4, True, 0.0), (10, 4, False, 0.0), (12, 4, True, 0.3)):
        rng = np.random.default_rng(mutant * 10 + N)
        X = [rng.standard_normal((N, d)) for _ in range(7)]
        tau = 1 / np.sqrt(d)
        gate = pins.dropout_gate(N, p, 5, 0) if p else None
        r = oracle.bob_head(*X, tau, causal, mutant=mutant, mutant_dir=out_dir,
                            dropout=(p, 5))
        fd = pins.bob_central_fd(*X, tau, causal, gate=gate)
        errs = [pins.rel_fro(g, r[n]) for g, n in zip(fd, ("qbar", "kbar", "vbar", "dobar"))]
        caught.append(max(errs) > 1e-6)
    assert any(caught), f"mutant {mutant} passed the finite-difference pin"
