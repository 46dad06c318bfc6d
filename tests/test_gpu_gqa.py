"""GPU parity of grouped-query attention: query head h reads key/value head
h / (H / H_kv); dK, dV, k_bar and v_bar of a key/value head sum over its query
heads.  Every kernel runs through the C ABI against the fp64 oracle."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

CASES = [  # B, H, H_kv, N, d, causal, window
    (1, 4, 2, 300, 64, True, None),
    (2, 3, 1, 257, 128, False, None),
    (1, 8, 2, 520, 128, True, (100, -1)),
    (1, 4, 1, 700, 64, False, None),
    (2, 2, 2, 200, 64, True, None),
    (1, 6, 2, 270, 32, True, None),
]


def ids(c):
    B, H, Hkv, N, d, causal, win = c
    return f"B{B}H{H}kv{Hkv}N{N}d{d}{'c' if causal else ''}w{win}"


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_forward_and_first_backward_gqa(case):
    B, H, Hkv, N, d, causal, win = case
    bits = G.inputs(B, H, N, d, seed=N + H + Hkv, kv_heads=Hkv)
    scale = 1 / np.sqrt(d)
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    o, lse = fbob.attn_fwd(q, k, v, scale, causal, win)
    dq, dk, dv, dstat = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal, win)
    assert fbob.fbob_device_status() == 0
    assert dk.shape == k.shape and dv.shape == v.shape
    X = [G.f64(bits[n]) for n in ("q", "k", "v", "dout")]
    O, L = oracle.fwd(*X[:3], scale, causal, window=win)
    G.check("O", G.host(o), O)
    assert np.abs(lse.cpu().numpy() - L).max() <= 1e-3
    dQ, dK, dV, Dv = oracle.bwd(*X, scale, causal, window=win)
    G.check("dQ", G.host(dq), dQ)
    G.check("dK", G.host(dk), dK)
    G.check("dV", G.host(dv), dV)
    G.check("D", dstat.cpu().numpy(), Dv)


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_bob_gqa(case):
    B, H, Hkv, N, d, causal, win = case
    bits = G.inputs(B, H, N, d, seed=2 * N + H + Hkv, kv_heads=Hkv)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal, window=win)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, window=win)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)
