"""The pins have power: each planted mistake in the oracle fails them.

The oracle source carries eleven deliberately wrong variants behind the
compile-time switch FBOB_MUTANT (a dropped term, a wrong sign, a transposed
operand, a wrong index, a dropout gate left out, masked blocks left in the
softmax normaliser ...).  Each is built into a temporary directory and run
through the finite-difference pin, without and with dropout and with a
block-sparse mask; every one must be caught.  The
default build (FBOB_MUTANT=0) is the oracle itself.
"""
import numpy as np
import pytest

import oracle
from tests import pins


@pytest.mark.parametrize("mutant", list(range(1, 12)))
def test_planted_mistake_is_caught(mutant):
    out_dir = oracle.mutant_build_dir()
    oracle.build(mutant=mutant, out_dir=out_dir)
    caught = []
    # (the last problem has a block-sparse mask: blocks of 3, the diagonal
    # and one off-diagonal block per block row)
    bm = np.eye(4, dtype=np.uint8) + np.eye(4, k=-1, dtype=np.uint8)
    for (N, d, causal, p, blk) in ((12, 4, True, 0.0, None), (10, 4, False, 0.0, None),
                                   (12, 4, True, 0.3, None), (12, 4, False, 0.0, (bm, 3))):
        rng = np.random.default_rng(mutant * 10 + N)
        X = [rng.standard_normal((N, d)) for _ in range(7)]
        tau = 1 / np.sqrt(d)
        gate = pins.dropout_gate(N, p, 5, 0) if p else None
        r = oracle.bob_head(*X, tau, causal, mutant=mutant, mutant_dir=out_dir,
                            dropout=(p, 5), block_mask=None if blk is None else blk[0],
                            block_size=3)
        fd = pins.bob_central_fd(*X, tau, causal, gate=gate, block=blk)
        errs = [pins.rel_fro(g, r[n]) for g, n in zip(fd, ("qbar", "kbar", "vbar", "dobar"))]
        caught.append(max(errs) > 1e-6)
    assert any(caught), f"mutant {mutant} passed the finite-difference pin"
