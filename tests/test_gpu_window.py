"""GPU parity of the sliding-window band (App. "Sliding-window attention"):
row i keeps i - wl <= j <= i + wr (-1 unbounded), capped at j <= i when causal.
Every kernel runs through the C ABI and is compared with the fp64 oracle."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

CASES = [  # B, H, N, d, causal, (wl, wr)
    (1, 2, 300, 64, True, (100, -1)),
    (1, 1, 257, 128, True, (64, -1)),
    (1, 2, 333, 64, False, (70, 45)),
    (1, 1, 520, 64, False, (-1, 10)),
    (1, 1, 400, 128, True, (5, -1)),
    (1, 2, 700, 128, False, (130, 200)),
    (2, 1, 200, 128, False, (1, 1)),
    (1, 2, 330, 32, True, (90, -1)),
]


def ids(c):
    B, H, N, d, causal, (wl, wr) = c
    return f"B{B}H{H}N{N}d{d}{'c' if causal else ''}w{wl}_{wr}"


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_forward_and_first_backward_with_window(case):
    B, H, N, d, causal, win = case
    bits = G.inputs(B, H, N, d, seed=N + 3 * d)
    scale = 1 / np.sqrt(d)
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    o, lse = fbob.attn_fwd(q, k, v, scale, causal, win)
    dq, dk, dv, dstat = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal, win)
    assert fbob.fbob_device_status() == 0
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
def test_bob_with_window(case):
    B, H, N, d, causal, win = case
    bits = G.inputs(B, H, N, d, seed=5 * N + d)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal, window=win)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, window=win)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)


@pytest.mark.parametrize("d", [64, 128])
def test_diagonal_window_is_a_stack_of_single_key_problems(d):
    """wl = wr = 0: every row sees only its own key, so P = I.  Exactly:
    O = V, dV = dO, dQ = dK = 0, and the BoB is q_bar = k_bar = v_bar = 0,
    dout_bar = U_V.  The vanishing outputs cancel only up to rounding:
    * dQ_i = tau (dP_ii - D_i) k_i with dP_ii (tensor-core fp32 sum) and D_i
      (fp32 dot of do_i and o_i = v_i) the same d products summed in different
      orders, so |dQ_i| <= tau 2d 2^-24 sum_a |do_ia v_ia| max|k_i|; the test
      allows 2^-12 in place of 2d 2^-24 (d <= 128);
    * q_bar row i as in the single-key case (test_single_key_degenerate):
      tau 2^-8 (|C_ii| + |F_ii dP_ii|) max|k_i|."""
    B, H, N = 1, 2, 200
    win = (0, 0)
    bits = G.inputs(B, H, N, d, seed=40 + d)
    scale = 1 / np.sqrt(d)
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    o, lse = fbob.attn_fwd(q, k, v, scale, False, win)
    dq, dk, dv, _ = fbob.attn_bwd(q, k, v, o, lse, do, scale, False, win)
    r = G.run_bob(bits, scale, False, window=win)
    assert r["status"] == 0
    X = {n: G.f64(bits[n]) for n in synth.NAMES}
    G.check("O", G.host(o), X["v"])
    G.check("dV", G.host(dv), X["dout"])
    G.check("dobar", r["dobar"], X["gv"])
    dq_h, dk_h = G.host(dq), G.host(dk)
    for h in range(H):
        Q, K, V, dO, UQ, UK, UV = (X[n][0, h] for n in synth.NAMES)
        sdv = np.abs(dO * V).sum(-1)
        assert np.all(np.abs(dq_h[0, h]).max(-1) <= scale * 2.0 ** -12 * sdv * np.abs(K).max(-1))
        assert np.all(np.abs(dk_h[0, h]).max(-1) <= scale * 2.0 ** -12 * sdv * np.abs(Q).max(-1))
        C = (dO * UV).sum(-1)
        F = scale * ((UQ * K).sum(-1) + (Q * UK).sum(-1))
        dP = (dO * V).sum(-1)
        bound = scale * 2.0 ** -8 * (np.abs(C) + np.abs(F * dP)) * np.abs(K).max(-1)
        assert np.all(np.abs(r["qbar"][0, h]).max(-1) <= bound), h
    assert np.abs(r["kbar"]).max() <= 1e-4 * scale * np.abs(X["q"]).max() * np.abs(X["gv"]).max() * d
    assert np.abs(r["vbar"]).max() <= 1e-4 * np.abs(X["dout"]).max() * np.abs(X["gq"]).max() * d


def test_window_covering_everything_matches_no_window_bitwise():
    B, H, N, d = 1, 2, 300, 128
    bits = G.inputs(B, H, N, d, seed=17)
    scale = 1 / np.sqrt(d)
    a = G.run_bob(bits, scale, True)
    b = G.run_bob(bits, scale, True, window=(N, N))
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"):
        assert np.array_equal(a[n], b[n]), n
