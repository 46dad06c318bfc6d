"""Pins for the oracle's block-sparse masks (App. "Extensions": a sparse mask
needs only a well-defined set of allowed columns per row, masked entries
having zero probability; the streamed loops then visit only the block pairs
of V, the set of blocks with an unmasked entry).

The mask is an [nb, nb] 0/1 array over square blocks of bs rows and columns;
the pair (i, j) is kept only if its block is set (and the causal mask, the
window and the packed sequences keep it).  Every diagonal block is set, so
every row keeps its diagonal.  The checks are independent of the oracle's
code: finite differences and a torch fp64 double backward over the explicit
0/1 element mask, the equivalence of a block-diagonal block mask with packed
sequences (pinned on their own), and invariants."""
import numpy as np
import pytest

import oracle
from tests import pins


def block_mask(N, bs, density, seed, empty_rows=()):
    """Random [nb, nb] 0/1 block mask with every diagonal block set; the
    block rows in empty_rows keep only their diagonal block."""
    nb = (N + bs - 1) // bs
    rng = np.random.default_rng(seed)
    bm = (rng.random((nb, nb)) < density).astype(np.uint8)
    for r in empty_rows:
        bm[r, :] = 0
    np.fill_diagonal(bm, 1)
    return bm


CASES = [  # N, d, bs, causal, window, density, empty block rows
    (40, 8, 8, False, None, 0.4, (2,)),
    (37, 8, 5, True, None, 0.5, ()),
    (33, 4, 4, False, (9, 6), 0.6, (0, 5)),
    (30, 8, 7, True, (11, -1), 0.3, (3,)),
]


def ids(c):
    N, d, bs, causal, win, dens, er = c
    return f"N{N}d{d}b{bs}{'c' if causal else ''}w{win}p{dens}"


def rand_problem(N, d, seed):
    rng = np.random.default_rng(seed)
    return [rng.standard_normal((N, d)) for _ in range(7)]


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_central_fd_with_block_mask(case):
    N, d, bs, causal, win, dens, er = case
    X = rand_problem(N, d, 1100 + N)
    bm = block_mask(N, bs, dens, N, er)
    tau = 1 / np.sqrt(d)
    r = oracle.bob_head(*X, tau, causal, window=win, block_mask=bm, block_size=bs)
    fd = pins.bob_central_fd(*X, tau, causal, window=win, block=(bm, bs))
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), fd):
        assert pins.rel_fro(g, r[name]) <= 1e-6, (name, pins.rel_fro(g, r[name]))


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_torch_double_backward_with_block_mask(case):
    torch = pytest.importorskip("torch")
    N, d, bs, causal, win, dens, er = case
    X = rand_problem(N, d, 1200 + N)
    bm = block_mask(N, bs, dens, 2 * N, er)
    tau = 1 / np.sqrt(d)
    keep = torch.tensor(pins.mask(N, causal, win, block=(bm, bs)) > 0)
    q, k, v, do = (torch.tensor(x, dtype=torch.float64, requires_grad=True) for x in X[:4])
    uq, uk, uv = (torch.tensor(x, dtype=torch.float64) for x in X[4:])
    s = (tau * q @ k.T).masked_fill(~keep, float("-inf"))
    o = torch.softmax(s, dim=-1) @ v
    dq, dk, dv = torch.autograd.grad(o, (q, k, v), do, create_graph=True)
    phi = (dq * uq).sum() + (dk * uk).sum() + (dv * uv).sum()
    grads = torch.autograd.grad(phi, (q, k, v, do))
    r = oracle.bob_head(*X, tau, causal, window=win, block_mask=bm, block_size=bs)
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), grads):
        assert pins.rel_fro(g.numpy(), r[name]) <= 1e-12, name
    O, L = oracle.fwd(*X[:3], tau, causal, window=win, block_mask=bm, block_size=bs)
    assert np.allclose(O[0, 0], o.detach().numpy(), atol=1e-12)
    assert np.allclose(L[0, 0], torch.logsumexp(s, -1).detach().numpy(), atol=1e-12)
    dQ, dK, dV, _ = oracle.bwd(*X[:4], tau, causal, window=win, block_mask=bm, block_size=bs)
    for got, want in ((dQ, dq), (dK, dk), (dV, dv)):
        assert np.allclose(got[0, 0], want.detach().numpy(), atol=1e-12)


@pytest.mark.parametrize("causal", [True, False])
def test_full_block_mask_is_no_mask(causal):
    N, d, bs = 35, 8, 6
    X = rand_problem(N, d, 31)
    tau = 1 / np.sqrt(d)
    nb = (N + bs - 1) // bs
    a = oracle.bob_head(*X, tau, causal)
    b = oracle.bob_head(*X, tau, causal, block_mask=np.ones((nb, nb)), block_size=bs)
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D", "L"):
        assert np.array_equal(a[n], b[n]), n


@pytest.mark.parametrize("causal", [True, False])
def test_block_diagonal_mask_is_packed_sequences(causal):
    """Blocks of bs rows that see only their own block: the same problem as
    packed sequences cut at every multiple of bs (an independently pinned
    path of the oracle)."""
    N, d, bs = 38, 8, 8
    X = rand_problem(N, d, 41)
    tau = 1 / np.sqrt(d)
    nb = (N + bs - 1) // bs
    seg = list(range(0, N, bs)) + [N]
    a = oracle.bob_head(*X, tau, causal, segments=seg)
    b = oracle.bob_head(*X, tau, causal, block_mask=np.eye(nb), block_size=bs)
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D", "L"):
        assert np.allclose(a[n], b[n], rtol=0, atol=1e-13), n


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_column_sums_vanish_and_sampling_agrees(case):
    """sum_j Ktil_j = sum_j Vtil_j = 0 under any mask, and sampled rows and
    column ranges match the full run."""
    N, d, bs, causal, win, dens, er = case
    X = rand_problem(N, d, 1300 + N)
    bm = block_mask(N, bs, dens, 3 * N, er)
    tau = 1 / np.sqrt(d)
    r = oracle.bob_head(*X, tau, causal, window=win, block_mask=bm, block_size=bs)
    scale = np.abs(r["kbar"]).max() + np.abs(r["vbar"]).max()
    assert np.abs(r["kbar"].sum(0)).max() <= 1e-12 * max(1.0, scale) * N
    assert np.abs(r["vbar"].sum(0)).max() <= 1e-12 * max(1.0, scale) * N
    rows = np.array([0, N // 3, N - 1])
    s = oracle.bob_head(*X, tau, causal, rows=rows, window=win, block_mask=bm, block_size=bs)
    for n in ("qbar", "dobar", "alpha", "E", "D"):
        assert np.allclose(s[n], r[n][rows], atol=1e-13), n
    c = oracle.bob_head(*X, tau, causal, rows=np.arange(N), cols=(N // 4, N // 2), window=win,
                        block_mask=bm, block_size=bs)
    assert np.allclose(c["kbar"], r["kbar"][N // 4:N // 2], atol=1e-12)
    assert np.allclose(c["vbar"], r["vbar"][N // 4:N // 2], atol=1e-12)


def test_diagonal_only_block_of_size_one_closed_form():
    """bs = 1 with only the diagonal set: P = I, so the BoB is q_bar = k_bar =
    v_bar = 0 and dout_bar = U_V (eqs. 6-7), as for the zero-width window."""
    N, d = 18, 8
    X = rand_problem(N, d, 5)
    r = oracle.bob_head(*X, 1 / np.sqrt(d), False, block_mask=np.eye(N), block_size=1)
    for n in ("qbar", "kbar", "vbar"):
        assert np.abs(r[n]).max() <= 1e-12, n
    assert np.allclose(r["dobar"], X[6], atol=1e-12)


def test_central_fd_with_block_mask_and_packed_sequences():
    """A block mask and packed sequences at once (both restrict the same rows)."""
    N, d, bs = 36, 8, 6
    seg = [0, 10, 25, 36]
    X = rand_problem(N, d, 1400)
    bm = block_mask(N, bs, 0.5, 14, (2,))
    tau = 1 / np.sqrt(d)
    r = oracle.bob_head(*X, tau, True, segments=seg, block_mask=bm, block_size=bs)
    fd = pins.bob_central_fd(*X, tau, True, segments=seg, block=(bm, bs))
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), fd):
        assert pins.rel_fro(g, r[name]) <= 1e-6, (name, pins.rel_fro(g, r[name]))
