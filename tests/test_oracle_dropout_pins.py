"""Pins for the oracle's attention dropout (App. "Extensions": the forward
uses a scaled keep mask sigma R on P; the BoB gates dP and C by it, and the
row scalars keep their ungated definitions).

Independent of the oracle's code: published Philox4x32-10 known-answer
vectors, a separate numpy Philox, keep-rate statistics, finite differences
of an independent numpy first backward with the mask applied, and a torch
fp64 double backward through O = (sigma R o P) V."""
import os

import numpy as np
import pytest

import oracle
from tests import pins

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def kat_rows():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                w = [int(x, 16) for x in line.split()]
                rows.append((w[:4], w[4:6], w[6:10]))
    return rows


def test_philox_known_answers():
    rows = kat_rows()
    assert len(rows) == 3
    for ctr, key, want in rows:
        assert list(oracle.philox(ctr, key)) == want
        got = pins.philox4x32_10(*([c] for c in ctr), *key)
        assert [int(x[0]) for x in got] == want


def test_oracle_philox_matches_numpy_philox():
    rng = np.random.default_rng(3)
    for _ in range(200):
        ctr = rng.integers(0, 2 ** 32, 4, dtype=np.uint64).astype(np.uint32)
        key = rng.integers(0, 2 ** 32, 2, dtype=np.uint64).astype(np.uint32)
        got = pins.philox4x32_10(*([c] for c in ctr), int(key[0]), int(key[1]))
        assert list(oracle.philox(ctr, key)) == [int(x[0]) for x in got]


@pytest.mark.parametrize("p", [0.1, 0.5, 0.9])
def test_keep_rate_and_scale(p):
    N = 512
    g = pins.dropout_gate(N, p, 0x1234_5678_9ABC_DEF0, 5)
    keep = g > 0
    n = keep.size
    pr = pins.dropout_rate(p)
    assert abs(pr - p) <= 1 / 512
    assert abs(keep.mean() - (1 - pr)) <= 5 * np.sqrt(pr * (1 - pr) / n)
    assert np.allclose(g[keep], 1 / (1 - pr))
    # the gate is unbiased: E[sigma R] = 1
    assert abs(g.mean() - 1) <= 5 * np.sqrt(pr / (1 - pr) / n)
    # neighbouring words of one Philox block and neighbouring rows are uncorrelated
    a, b = keep[:, :-1].astype(float).ravel(), keep[:, 1:].astype(float).ravel()
    assert abs(np.corrcoef(a, b)[0, 1]) <= 5 / np.sqrt(a.size)
    a, b = keep[:-1].astype(float).ravel(), keep[1:].astype(float).ravel()
    assert abs(np.corrcoef(a, b)[0, 1]) <= 5 / np.sqrt(a.size)


def test_masks_differ_across_heads_and_seeds():
    a = pins.dropout_gate(64, 0.5, 11, 0)
    assert not np.array_equal(a, pins.dropout_gate(64, 0.5, 11, 1))
    assert not np.array_equal(a, pins.dropout_gate(64, 0.5, 12, 0))
    assert not np.array_equal(a, pins.dropout_gate(64, 0.5, 11 + (1 << 32), 0))


CASES = [  # N, d, causal, p, seed, head, window, segments
    (24, 8, True, 0.2, 99, 0, None, None),
    (21, 4, False, 0.5, (7 << 32) + 5, 3, None, None),
    (30, 8, True, 0.3, 2024, 6, (9, -1), None),
    (26, 4, True, 0.4, 31, 1, None, (0, 9, 17, 26)),
]


def ids(c):
    return f"N{c[0]}d{c[1]}{'c' if c[2] else ''}p{c[3]}h{c[5]}"


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_central_fd_with_dropout_gate(case):
    N, d, causal, p, seed, head, win, seg = case
    rng = np.random.default_rng(700 + N)
    X = [rng.standard_normal((N, d)) for _ in range(7)]
    tau = 1 / np.sqrt(d)
    gate = pins.dropout_gate(N, p, seed, head)
    r = oracle.bob_head(*X, tau, causal, window=win, segments=seg, dropout=(p, seed), head=head)
    fd = pins.bob_central_fd(*X, tau, causal, window=win, segments=seg, gate=gate)
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), fd):
        assert pins.rel_fro(g, r[name]) <= 1e-6, (name, pins.rel_fro(g, r[name]))
    # the row scalars keep their definitions over the ungated P; D = dO . O
    O, _ = oracle.fwd(X[0], X[1], X[2], tau, causal, window=win, segments=seg, dropout=(p, seed))
    P = pins.softmax_probs(X[0], X[1], tau, causal, win, seg)
    assert np.allclose(r["D"], (X[3] * pins.attention(*X[:3], tau, causal, win, seg, gate)).sum(1),
                       atol=1e-12)
    F = tau * (X[4] @ X[1].T + X[0] @ X[5].T)
    assert np.allclose(r["alpha"], (P * F).sum(1), atol=1e-12)


@pytest.mark.parametrize("H,Hkv,causal,p", [(2, 2, True, 0.25), (4, 2, False, 0.5), (3, 1, True, 0.1)])
def test_torch_double_backward_with_dropout(H, Hkv, causal, p):
    torch = pytest.importorskip("torch")
    B, N, d, seed = 2, 20, 8, 424242
    rng = np.random.default_rng(50 + H + Hkv)
    q, do, gq = (rng.standard_normal((B, H, N, d)) for _ in range(3))
    k, v, gk, gv = (rng.standard_normal((B, Hkv, N, d)) for _ in range(4))
    tau = 1 / np.sqrt(d)
    G = H // Hkv
    gate = np.stack([np.stack([pins.dropout_gate(N, p, seed, b * H + h) for h in range(H)])
                     for b in range(B)])
    T = lambda x, g=True: torch.tensor(x, dtype=torch.float64, requires_grad=g)
    tq, tk, tv, tdo = T(q), T(k), T(v), T(do)
    kk = tk.repeat_interleave(G, dim=1)
    vv = tv.repeat_interleave(G, dim=1)
    s = tau * tq @ kk.transpose(-1, -2)
    if causal:
        s = s.masked_fill(torch.triu(torch.ones(N, N, dtype=torch.bool), 1), float("-inf"))
    o = (T(gate, False) * torch.softmax(s, dim=-1)) @ vv
    dq, dk, dv = torch.autograd.grad(o, (tq, tk, tv), tdo, create_graph=True)
    phi = ((dq * T(gq, False)).sum() + (dk * T(gk, False)).sum() + (dv * T(gv, False)).sum())
    grads = torch.autograd.grad(phi, (tq, tk, tv, tdo))
    ref = oracle.bob(q, k, v, do, gq, gk, gv, tau, causal, dropout=(p, seed))
    for name, g, r in zip(("qbar", "kbar", "vbar", "dobar"), grads, ref):
        assert pins.rel_fro(g.numpy(), r) <= 1e-12, name
    O, L = oracle.fwd(q, k, v, tau, causal, dropout=(p, seed))
    assert np.allclose(O, o.detach().numpy(), atol=1e-12)
    assert np.allclose(L, torch.logsumexp(s, -1).detach().numpy(), atol=1e-12)
    dQ, dK, dV, _ = oracle.bwd(q, k, v, do, tau, causal, dropout=(p, seed))
    for got, want in ((dQ, dq), (dK, dk), (dV, dv)):
        assert np.allclose(got, want.detach().numpy(), atol=1e-12)


@pytest.mark.parametrize("causal", [True, False])
@pytest.mark.parametrize("p", [0.0, 0.0019])
def test_zero_rate_is_no_dropout(causal, p):
    # rates below 1/512 round to a zero byte threshold: nothing is dropped
    rng = np.random.default_rng(8)
    X = [rng.standard_normal((1, 2, 19, 8)) for _ in range(7)]
    tau = 0.3
    a = oracle.bob(*X, tau, causal)
    b = oracle.bob(*X, tau, causal, dropout=(p, 77))
    for x, y in zip(a, b):
        assert np.array_equal(x, y)
    assert all(np.array_equal(x, y) for x, y in zip(oracle.fwd(*X[:3], tau, causal),
                                                    oracle.fwd(*X[:3], tau, causal,
                                                               dropout=(p, 77))))


def test_realised_rate_and_block_layout():
    """The mask of one 4 x 4 block comes from one Philox call: byte j mod 4
    of word i mod 4, compared with the rounded byte threshold."""
    seed, head, p = (3 << 32) + 9, 2, 0.3
    g = pins.dropout_gate(8, p, seed, head)
    t = round(256 * p)
    for I in range(2):
        for J in range(2):
            w = oracle.philox([J, I, head, 0], [seed & 0xFFFFFFFF, seed >> 32])
            for a in range(4):
                for b in range(4):
                    byte = (int(w[a]) >> (8 * b)) & 0xFF
                    assert (g[4 * I + a, 4 * J + b] > 0) == (byte >= t)
    assert pins.dropout_rate(0.3) == 77 / 256 and pins.dropout_rate(0.999) == 255 / 256
