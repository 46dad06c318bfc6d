"""Pins for the oracle's sliding-window band (App. "Sliding-window
attention": the inner column range is restricted to the window; App.
"Extensions": masked entries have zero probability).

Band: row i keeps i - wl <= j <= i + wr (a negative side is unbounded),
capped at j <= i with the causal mask.  Each check below is independent of
the oracle's code: finite differences and a torch fp64 double backward over
an explicit 0/1 band mask, an exact closed form, and invariants."""
import numpy as np
import pytest

import oracle
from tests import pins

WINDOWS = [  # N, d, causal, (wl, wr)
    (40, 8, True, (7, -1)),
    (33, 8, False, (5, 5)),
    (36, 4, False, (12, 0)),
    (30, 8, False, (0, 9)),
    (29, 8, True, (3, 3)),
]


def rand_problem(N, d, seed):
    rng = np.random.default_rng(seed)
    return [rng.standard_normal((N, d)) for _ in range(7)]


def ids(c):
    N, d, causal, (wl, wr) = c
    return f"N{N}d{d}{'c' if causal else ''}w{wl}_{wr}"


@pytest.mark.parametrize("case", WINDOWS, ids=ids)
def test_central_fd_with_band_mask(case):
    N, d, causal, win = case
    X = rand_problem(N, d, 500 + N)
    tau = 1 / np.sqrt(d)
    r = oracle.bob_head(*X, tau, causal, window=win)
    fd = pins.bob_central_fd(*X, tau, causal, window=win)
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), fd):
        assert pins.rel_fro(g, r[name]) <= 1e-6, (name, pins.rel_fro(g, r[name]))


@pytest.mark.parametrize("case", WINDOWS[:3], ids=ids)
def test_torch_double_backward_with_band_mask(case):
    torch = pytest.importorskip("torch")
    N, d, causal, win = case
    X = rand_problem(N, d, 600 + N)
    tau = 1 / np.sqrt(d)
    keep = torch.tensor(pins.mask(N, causal, win) > 0)
    q, k, v, do = (torch.tensor(x, dtype=torch.float64, requires_grad=True) for x in X[:4])
    uq, uk, uv = (torch.tensor(x, dtype=torch.float64) for x in X[4:])
    s = (tau * q @ k.T).masked_fill(~keep, float("-inf"))
    o = torch.softmax(s, dim=-1) @ v
    dq, dk, dv = torch.autograd.grad(o, (q, k, v), do, create_graph=True)
    phi = (dq * uq).sum() + (dk * uk).sum() + (dv * uv).sum()
    grads = torch.autograd.grad(phi, (q, k, v, do))
    r = oracle.bob_head(*X, tau, causal, window=win)
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), grads):
        assert pins.rel_fro(g.numpy(), r[name]) <= 1e-12, name
    # forward and first backward under the same band
    O, L = oracle.fwd(*X[:3], tau, causal, window=win)
    assert np.allclose(O[0, 0], o.detach().numpy(), atol=1e-12)
    assert np.allclose(L[0, 0], torch.logsumexp(s, -1).detach().numpy(), atol=1e-12)
    dQ, dK, dV, _ = oracle.bwd(*X[:4], tau, causal, window=win)
    for got, want in ((dQ, dq), (dK, dk), (dV, dv)):
        assert np.allclose(got[0, 0], want.detach().numpy(), atol=1e-12)


@pytest.mark.parametrize("causal", [True, False])
def test_window_covering_everything_is_no_window(causal):
    N, d = 37, 8
    X = rand_problem(N, d, 77)
    tau = 1 / np.sqrt(d)
    a = oracle.bob_head(*X, tau, causal)
    b = oracle.bob_head(*X, tau, causal, window=(N, N))
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D", "L"):
        assert np.array_equal(a[n], b[n]), n


def test_diagonal_window_closed_form():
    """wl = wr = 0: P = I, so h = F - alpha = 0, dS = 0, Stil = 0 and the BoB
    is q_bar = k_bar = v_bar = 0, dout_bar = U_V (eqs. 6-7)."""
    N, d = 20, 8
    X = rand_problem(N, d, 5)
    r = oracle.bob_head(*X, 1 / np.sqrt(d), False, window=(0, 0))
    for n in ("qbar", "kbar", "vbar"):
        assert np.abs(r[n]).max() <= 1e-12, n
    assert np.allclose(r["dobar"], X[6], atol=1e-12)


@pytest.mark.parametrize("case", WINDOWS, ids=ids)
def test_column_sums_vanish_and_sampling_agrees(case):
    """sum_j Ktil_j = sum_j Vtil_j = 0 for any mask (each row sums of Stil,
    dS and P o h vanish), and sampled rows / column ranges match the full run."""
    N, d, causal, win = case
    X = rand_problem(N, d, 900 + N)
    tau = 1 / np.sqrt(d)
    r = oracle.bob_head(*X, tau, causal, window=win)
    scale = np.abs(r["kbar"]).max() + np.abs(r["vbar"]).max()
    assert np.abs(r["kbar"].sum(0)).max() <= 1e-12 * max(1.0, scale) * N
    assert np.abs(r["vbar"].sum(0)).max() <= 1e-12 * max(1.0, scale) * N
    rows = np.array([0, N // 3, N - 1])
    s = oracle.bob_head(*X, tau, causal, rows=rows, window=win)
    for n in ("qbar", "dobar", "alpha", "E", "D"):
        assert np.allclose(s[n], r[n][rows], atol=1e-13), n
    c0, c1 = N // 4, N // 2
    wl, wr = win
    lo = max(0, c0 - (wr if wr >= 0 else N)) if not causal else c0
    hi = min(N, c1 + (wl if wl >= 0 else N))
    c = oracle.bob_head(*X, tau, causal, rows=np.arange(lo, hi), cols=(c0, c1), window=win)
    assert np.allclose(c["kbar"], r["kbar"][c0:c1], atol=1e-12)
    assert np.allclose(c["vbar"], r["vbar"][c0:c1], atol=1e-12)


# ---------------------------------------------------------------- varlen
# Packed variable-length sequences (App. "Extensions"): segment offsets split
# the N rows; a row sees only the columns of its own sequence.
SEGMENTS = [  # N, d, causal, window, offsets
    (40, 8, True, None, [0, 7, 20, 21, 40]),
    (36, 8, False, None, [0, 13, 13, 36]),
    (45, 4, True, (6, -1), [0, 30, 45]),
    (30, 8, False, (3, 2), [0, 1, 2, 17, 30]),
]


def sids(c):
    N, d, causal, win, seg = c
    return f"N{N}{'c' if causal else ''}w{win}s{len(seg) - 1}"


@pytest.mark.parametrize("case", SEGMENTS, ids=sids)
def test_central_fd_with_segment_mask(case):
    N, d, causal, win, seg = case
    X = rand_problem(N, d, 700 + N)
    tau = 1 / np.sqrt(d)
    r = oracle.bob_head(*X, tau, causal, window=win, segments=seg)
    fd = pins.bob_central_fd(*X, tau, causal, window=win, segments=seg)
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), fd):
        assert pins.rel_fro(g, r[name]) <= 1e-6, (name, pins.rel_fro(g, r[name]))


@pytest.mark.parametrize("case", SEGMENTS[:2], ids=sids)
def test_torch_double_backward_with_segment_mask(case):
    torch = pytest.importorskip("torch")
    N, d, causal, win, seg = case
    X = rand_problem(N, d, 800 + N)
    tau = 1 / np.sqrt(d)
    keep = torch.tensor(pins.mask(N, causal, win, seg) > 0)
    q, k, v, do = (torch.tensor(x, dtype=torch.float64, requires_grad=True) for x in X[:4])
    uq, uk, uv = (torch.tensor(x, dtype=torch.float64) for x in X[4:])
    s = (tau * q @ k.T).masked_fill(~keep, float("-inf"))
    o = torch.softmax(s, dim=-1) @ v
    dq, dk, dv = torch.autograd.grad(o, (q, k, v), do, create_graph=True)
    phi = (dq * uq).sum() + (dk * uk).sum() + (dv * uv).sum()
    grads = torch.autograd.grad(phi, (q, k, v, do))
    r = oracle.bob_head(*X, tau, causal, window=win, segments=seg)
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), grads):
        assert pins.rel_fro(g.numpy(), r[name]) <= 1e-12, name
    O, L = oracle.fwd(*X[:3], tau, causal, window=win, segments=seg)
    assert np.allclose(O[0, 0], o.detach().numpy(), atol=1e-12)
    dQ, dK, dV, _ = oracle.bwd(*X[:4], tau, causal, window=win, segments=seg)
    for got, want in ((dQ, dq), (dK, dk), (dV, dv)):
        assert np.allclose(got[0, 0], want.detach().numpy(), atol=1e-12)


@pytest.mark.parametrize("case", SEGMENTS, ids=sids)
def test_packed_sequences_are_independent_problems(case):
    """A block-diagonal mask decouples the sequences: the packed BoB equals
    the BoB of each sequence on its own."""
    N, d, causal, win, seg = case
    X = rand_problem(N, d, 900 + N)
    tau = 1 / np.sqrt(d)
    r = oracle.bob_head(*X, tau, causal, window=win, segments=seg)
    for a, b in zip(seg[:-1], seg[1:]):
        if b == a:
            continue
        part = oracle.bob_head(*(x[a:b] for x in X), tau, causal, window=win)
        for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D", "L"):
            assert np.allclose(r[n][a:b], part[n], rtol=0, atol=1e-12), (n, a, b)


def test_one_segment_is_no_segments():
    N, d = 33, 8
    X = rand_problem(N, d, 12)
    tau = 1 / np.sqrt(d)
    a = oracle.bob_head(*X, tau, True)
    b = oracle.bob_head(*X, tau, True, segments=[0, N])
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D", "L"):
        assert np.array_equal(a[n], b[n]), n
