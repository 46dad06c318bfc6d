"""GPU parity of packed variable-length sequences (App. "Extensions"): offsets
split the N rows into sequences and a row sees only the columns of its own
sequence (intersected with the causal mask and the window).  Every kernel
runs through the C ABI and is compared with the fp64 oracle."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

CASES = [  # B, H, N, d, causal, window, offsets
    (1, 2, 500, 64, True, None, [0, 100, 237, 238, 500]),
    (1, 1, 700, 128, False, None, [0, 128, 256, 700]),
    (2, 1, 333, 128, True, (40, -1), [0, 50, 50, 333]),
    (1, 2, 300, 64, False, (20, 20), [0, 10, 20, 30, 300]),
    (1, 1, 1000, 128, True, None, [0, 64, 65, 300, 301, 777, 1000]),
    (1, 2, 400, 32, True, None, [0, 33, 200, 400]),
]


def ids(c):
    B, H, N, d, causal, win, seg = c
    return f"B{B}H{H}N{N}d{d}{'c' if causal else ''}w{win}s{len(seg) - 1}"


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_forward_and_first_backward_packed(case):
    B, H, N, d, causal, win, seg = case
    bits = G.inputs(B, H, N, d, seed=2 * N + d)
    scale = 1 / np.sqrt(d)
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    segs = G.dev_segments(seg)
    o, lse = fbob.attn_fwd(q, k, v, scale, causal, win, segs)
    dq, dk, dv, dstat = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal, win, segs)
    assert fbob.fbob_device_status() == 0
    X = [G.f64(bits[n]) for n in ("q", "k", "v", "dout")]
    O, L = oracle.fwd(*X[:3], scale, causal, window=win, segments=seg)
    G.check("O", G.host(o), O)
    assert np.abs(lse.cpu().numpy() - L).max() <= 1e-3
    dQ, dK, dV, Dv = oracle.bwd(*X, scale, causal, window=win, segments=seg)
    G.check("dQ", G.host(dq), dQ)
    G.check("dK", G.host(dk), dK)
    G.check("dV", G.host(dv), dV)
    G.check("D", dstat.cpu().numpy(), Dv)


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_bob_packed(case):
    B, H, N, d, causal, win, seg = case
    bits = G.inputs(B, H, N, d, seed=3 * N + d)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal, window=win, segments=seg)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, window=win,
                     segments=seg)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)


def test_one_sequence_matches_no_offsets_bitwise():
    B, H, N, d = 1, 2, 300, 64
    bits = G.inputs(B, H, N, d, seed=23)
    scale = 1 / np.sqrt(d)
    a = G.run_bob(bits, scale, True)
    b = G.run_bob(bits, scale, True, segments=[0, N])
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"):
        assert np.array_equal(a[n], b[n]), n
