"""Pins for the fp64 oracle: nothing here trusts the oracle on its own word.

Each test checks the oracle against something it does not share code with:
  * central finite differences of an independent numpy first backward
    (rel. error <= 1e-6);
  * an explicit complex-step Jacobian of that first backward, J_g^T vec(U);
  * symbolic differentiation (sympy) of the first backward written from eqs. (1)-(3);
  * torch fp64 double backward (autograd through attention twice);
  * linearity in (U_Q, U_K, U_V) and in dO, and independence of dOtil from dO;
  * closed-form special cases: Lemma D.2 (forward-attention embedding),
    U_Q = U_K = 0 (reduces to an ordinary attention backward), N = 1,
    causal row 0, U = 0;
  * exact invariants: column sums of Ktil and Vtil vanish; three Euler
    identities; orthogonal equivariance.
"""
import numpy as np
import pytest

import oracle
from tests import pins

# (the last two: head dimension 256, which the GPU path runs in kernels of
# its own, at a few rows)
CASES = [(32, 16, True), (32, 8, False), (24, 4, True), (17, 8, False), (6, 256, True),
         (5, 256, False)]


def rand_problem(N, d, seed, scale_q=1.0):
    rng = np.random.default_rng(seed)
    X = [rng.standard_normal((N, d)) for _ in range(7)]
    X[0] *= scale_q
    X[1] *= scale_q
    return X


def oracle_bob(X, tau, causal):
    r = oracle.bob_head(*X, tau, causal)
    return r


@pytest.mark.parametrize("N,d,causal", CASES)
def test_central_fd_of_independent_first_backward(N, d, causal):
    """Sec. 3.1 eq. (5): BoB is grad of Phi; central differences of Phi built
    from an independent first backward agree with the oracle to <= 1e-6."""
    X = rand_problem(N, d, 100 + N + d + causal)
    tau = 1 / np.sqrt(d)
    r = oracle_bob(X, tau, causal)
    fd = pins.bob_central_fd(*X, tau, causal)
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), fd):
        ref = r[name]
        assert pins.rel_fro(g, ref) <= 1e-6, (name, pins.rel_fro(g, ref))
        assert np.max(np.abs(g - ref)) <= 1e-6 * np.max(np.abs(ref)), name


@pytest.mark.parametrize("N,d,causal", [(8, 4, True), (8, 4, False), (6, 8, True)])
def test_explicit_jacobian_transpose_product(N, d, causal):
    """Sec. 3.1: BoB = J_g^T (U_Q, U_K, U_V) with J_g the Jacobian of the first
    backward; J_g built column by column by complex step (accuracy ~1e-13)."""
    X = rand_problem(N, d, 7 + N + d)
    tau = 1 / np.sqrt(d)
    J = pins.jacobian_complex_step(*X[:4], tau, causal)
    u = np.concatenate([X[4].ravel(), X[5].ravel(), X[6].ravel()])
    bob = J.T @ u
    r = oracle_bob(X, tau, causal)
    ref = np.concatenate([r[n].ravel() for n in ("qbar", "kbar", "vbar", "dobar")])
    assert np.max(np.abs(bob - ref)) <= 1e-11 * max(1.0, np.max(np.abs(ref)))


@pytest.mark.parametrize("causal", [True, False])
def test_symbolic_differentiation(causal):
    """Symbolic reverse of eqs. (1)-(4) (sympy, 30 digits) at rational points."""
    sp = pytest.importorskip("sympy")
    N, d = 3, 2
    tau_s = 1 / sp.sqrt(d)
    rng = np.random.default_rng(11 + causal)

    def sym(name):
        return sp.Matrix(N, d, lambda i, a: sp.Symbol(f"{name}{i}_{a}"))

    def rat():
        return sp.Matrix(N, d, lambda i, a: sp.Rational(int(rng.integers(-9, 10)), 5))

    Q, K, V, dO = sym("q"), sym("k"), sym("v"), sym("o")
    U = [rat(), rat(), rat()]
    S = tau_s * Q * K.T
    P = sp.zeros(N, N)
    for i in range(N):
        js = [j for j in range(N) if (not causal or j <= i)]
        Z = sum(sp.exp(S[i, j]) for j in js)
        for j in js:
            P[i, j] = sp.exp(S[i, j]) / Z
    dP = dO * V.T
    Dv = [sum(P[i, j] * dP[i, j] for j in range(N)) for i in range(N)]
    dS = sp.Matrix(N, N, lambda i, j: P[i, j] * (dP[i, j] - Dv[i]))
    dQ, dK, dV = tau_s * dS * K, tau_s * dS.T * Q, P.T * dO
    Phi = sum(dQ[i, a] * U[0][i, a] + dK[i, a] * U[1][i, a] + dV[i, a] * U[2][i, a]
              for i in range(N) for a in range(d))
    vals = {}
    num = []
    for M in (Q, K, V, dO):
        arr = np.zeros((N, d))
        for i in range(N):
            for a in range(d):
                v = sp.Rational(int(rng.integers(-9, 10)), 5)
                vals[M[i, a]] = v
                arr[i, a] = float(v)
        num.append(arr)
    Un = [np.array(u.tolist(), dtype=float) for u in U]
    r = oracle_bob(num + Un, 1 / np.sqrt(d), causal)
    for M, name in zip((Q, K, V, dO), ("qbar", "kbar", "vbar", "dobar")):
        for i in range(N):
            for a in range(d):
                ref = float(sp.diff(Phi, M[i, a]).evalf(30, subs=vals))
                assert abs(r[name][i, a] - ref) <= 1e-12 * max(1.0, abs(ref)), (name, i, a)


@pytest.mark.parametrize("N,d,causal", [(48, 16, True), (40, 8, False), (256, 32, True),
                                         (70, 256, True), (33, 256, False)])
def test_torch_double_backward(N, d, causal):
    """The paper's math path (autograd through attention twice, App. H) in
    torch fp64 on the CPU."""
    torch = pytest.importorskip("torch")
    X = rand_problem(N, d, 31 + N)
    tau = 1 / np.sqrt(d)
    q, k, v, do = (torch.tensor(x, dtype=torch.float64, requires_grad=True) for x in X[:4])
    uq, uk, uv = (torch.tensor(x, dtype=torch.float64) for x in X[4:])
    s = tau * q @ k.T
    if causal:
        s = s.masked_fill(torch.triu(torch.ones(N, N, dtype=torch.bool), 1), float("-inf"))
    o = torch.softmax(s, dim=-1) @ v
    dq, dk, dv = torch.autograd.grad(o, (q, k, v), do, create_graph=True)
    phi = (dq * uq).sum() + (dk * uk).sum() + (dv * uv).sum()
    grads = torch.autograd.grad(phi, (q, k, v, do))
    r = oracle_bob(X, tau, causal)
    for name, g in zip(("qbar", "kbar", "vbar", "dobar"), grads):
        assert pins.rel_fro(g.numpy(), r[name]) <= 1e-12, name


@pytest.mark.parametrize("causal", [True, False])
def test_oracle_fwd_bwd_against_torch(causal):
    torch = pytest.importorskip("torch")
    N, d = 70, 16
    X = rand_problem(N, d, 3)
    tau = 1 / np.sqrt(d)
    q, k, v = (torch.tensor(x, dtype=torch.float64, requires_grad=True) for x in X[:3])
    do = torch.tensor(X[3])
    s = tau * q @ k.T
    if causal:
        s = s.masked_fill(torch.triu(torch.ones(N, N, dtype=torch.bool), 1), float("-inf"))
    lse = torch.logsumexp(s, dim=-1)
    o = torch.softmax(s, dim=-1) @ v
    dq, dk, dv = torch.autograd.grad(o, (q, k, v), do)
    O, L = oracle.fwd(X[0], X[1], X[2], tau, causal)
    assert np.allclose(O[0, 0], o.detach().numpy(), rtol=0, atol=1e-12)
    assert np.allclose(L[0, 0], lse.detach().numpy(), rtol=0, atol=1e-12)
    gQ, gK, gV, D = oracle.bwd(*X[:4], tau, causal)
    assert np.allclose(gQ[0, 0], dq.numpy(), atol=1e-12)
    assert np.allclose(gK[0, 0], dk.numpy(), atol=1e-12)
    assert np.allclose(gV[0, 0], dv.numpy(), atol=1e-12)
    # D_i = do_i . o_i (Sec. 2, below eq. 3)
    assert np.allclose(D[0, 0], (X[3] * O[0, 0]).sum(-1), atol=1e-12)


def test_linearity_in_cotangents_and_dO():
    N, d, causal = 20, 8, True
    X = rand_problem(N, d, 5)
    Y = rand_problem(N, d, 6)
    tau = 1 / np.sqrt(d)
    a, b = 0.7, -1.3
    names = ("qbar", "kbar", "vbar", "dobar")
    r1 = oracle_bob(X, tau, causal)
    r2 = oracle_bob(X[:4] + Y[4:], tau, causal)
    r12 = oracle_bob(X[:4] + [a * x + b * y for x, y in zip(X[4:], Y[4:])], tau, causal)
    for n in names:   # jointly linear in (U_Q, U_K, U_V)
        assert np.allclose(r12[n], a * r1[n] + b * r2[n], atol=1e-12, rtol=0), n
    # Qtil, Ktil, Vtil linear (additive, homogeneous) in dO; dOtil independent of dO
    rA = oracle_bob(X[:3] + [Y[3]] + X[4:], tau, causal)
    rS = oracle_bob(X[:3] + [a * X[3] + b * Y[3]] + X[4:], tau, causal)
    for n in ("qbar", "kbar", "vbar"):
        assert np.allclose(rS[n], a * r1[n] + b * rA[n], atol=1e-12, rtol=0), n
    assert np.allclose(rA["dobar"], r1["dobar"], atol=1e-13, rtol=0)
    assert np.allclose(rS["dobar"], r1["dobar"], atol=1e-13, rtol=0)


@pytest.mark.parametrize("causal", [True, False])
def test_lemma_d2_forward_attention_embedding(causal):
    """Lemma D.2: V = dO = U_Q = U_K = 0, U_V = W gives dOtil = softmax(tau Q K^T) W
    and Qtil = Ktil = Vtil = 0."""
    N, d = 33, 8
    X = rand_problem(N, d, 9)
    Z = np.zeros((N, d))
    W = X[6]
    tau = 1 / np.sqrt(d)
    r = oracle_bob([X[0], X[1], Z, Z, Z, Z, W], tau, causal)
    ref = pins.attention(X[0], X[1], W, tau, causal)
    assert np.allclose(r["dobar"], ref, atol=1e-13, rtol=0)
    for n in ("qbar", "kbar", "vbar"):
        assert np.max(np.abs(r[n])) == 0.0


@pytest.mark.parametrize("causal", [True, False])
def test_uq_uk_zero_reduces_to_attention_backward(causal):
    """U_Q = U_K = 0: Phi = <dO, P U_V>, so Vtil = 0, dOtil = P U_V and
    (Qtil, Ktil) is the ordinary backward (dQ, dK) of attention with V := U_V."""
    N, d = 29, 8
    X = rand_problem(N, d, 12)
    Z = np.zeros((N, d))
    tau = 1 / np.sqrt(d)
    r = oracle_bob(X[:4] + [Z, Z, X[6]], tau, causal)
    dQ, dK, _ = pins.first_backward(X[0], X[1], X[6], X[3], tau, causal)
    assert np.allclose(r["qbar"], dQ, atol=1e-12, rtol=0)
    assert np.allclose(r["kbar"], dK, atol=1e-12, rtol=0)
    assert np.max(np.abs(r["vbar"])) <= 1e-14
    assert np.allclose(r["dobar"], pins.attention(X[0], X[1], X[6], tau, causal), atol=1e-13)


def test_degenerate_cases():
    d = 8
    tau = 1 / np.sqrt(d)
    X = rand_problem(1, d, 13)
    r = oracle_bob(X, tau, False)          # N = 1: P = [1], everything cancels
    for n in ("qbar", "kbar", "vbar"):
        assert np.max(np.abs(r[n])) <= 1e-15
    assert np.allclose(r["dobar"], X[6], atol=1e-15)
    X = rand_problem(12, d, 14)
    r = oracle_bob(X, tau, True)           # causal row 0 sees only itself
    assert np.max(np.abs(r["qbar"][0])) <= 1e-15
    assert np.allclose(r["dobar"][0], X[6][0], atol=1e-15)
    Z = np.zeros((12, d))
    r = oracle_bob(X[:4] + [Z, Z, Z], tau, True)   # U = 0
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E"):
        assert np.max(np.abs(r[n])) == 0.0


@pytest.mark.parametrize("N,d,causal", [(64, 16, True), (50, 8, False)])
def test_exact_invariants(N, d, causal):
    X = rand_problem(N, d, 21 + N)
    tau = 1 / np.sqrt(d)
    r = oracle_bob(X, tau, causal)
    scale = max(np.abs(r[n]).max() for n in ("kbar", "vbar"))
    # Phi is invariant under K -> K + 1 c^T and V -> V + 1 c^T
    assert np.abs(r["kbar"].sum(0)).max() <= 1e-12 * N * scale
    assert np.abs(r["vbar"].sum(0)).max() <= 1e-12 * N * scale
    dQ, dK, dV = pins.first_backward(*X[:4], tau, causal)
    gq, gk, gv = X[4:]
    a, b, c = pins.inner(dQ, gq), pins.inner(dK, gk), pins.inner(dV, gv)
    phi = a + b + c
    tol = 1e-11 * max(1.0, abs(a) + abs(b) + abs(c))
    assert abs(pins.inner(r["dobar"], X[3]) - phi) <= tol            # degree 1 in dO
    assert abs(pins.inner(r["vbar"], X[2]) - (a + b)) <= tol         # V -> sV
    assert abs(pins.inner(r["qbar"], X[0]) - pins.inner(r["kbar"], X[1]) - (b - a)) <= tol
    # orthogonal equivariance: (Q,K,U_Q,U_K) R -> (Qtil,Ktil) R, Vtil and dOtil unchanged
    R, _ = np.linalg.qr(np.random.default_rng(1).standard_normal((d, d)))
    Xr = [X[0] @ R, X[1] @ R, X[2], X[3], X[4] @ R, X[5] @ R, X[6]]
    rr = oracle_bob(Xr, tau, causal)
    assert np.allclose(rr["qbar"], r["qbar"] @ R, atol=1e-11)
    assert np.allclose(rr["kbar"], r["kbar"] @ R, atol=1e-11)
    assert np.allclose(rr["vbar"], r["vbar"], atol=1e-11)
    assert np.allclose(rr["dobar"], r["dobar"], atol=1e-11)


def test_row_sampling_and_column_ranges_agree_with_full():
    """The sampled-row and column-range entry points return exactly the rows
    and columns of the full computation (used at full sizes)."""
    N, d = 90, 8
    X = rand_problem(N, d, 40)
    tau = 1 / np.sqrt(d)
    for causal in (True, False):
        full = oracle_bob(X, tau, causal)
        rows = np.array([89, 0, 45, 7])
        part = oracle.bob_head(*X, tau, causal, rows=rows)
        for n in ("qbar", "dobar", "alpha", "E", "D"):
            assert np.array_equal(part[n], full[n][rows]), n
        if causal:   # causal tail: rows >= 60 complete the columns >= 60
            tail = oracle.bob_head(*X, tau, causal, rows=np.arange(60, N), cols=(60, N))
            assert np.allclose(tail["kbar"], full["kbar"][60:], atol=1e-13)
            assert np.allclose(tail["vbar"], full["vbar"][60:], atol=1e-13)


def test_alpha_E_D_definitions():
    """Row scalars: alpha_i = sum P F, D_i = sum P dP = do_i.o_i, and
    E_i = sum P Ptil, checked against the independent numpy forms."""
    N, d, causal = 40, 8, True
    X = rand_problem(N, d, 41)
    tau = 1 / np.sqrt(d)
    r = oracle_bob(X, tau, causal)
    Q, K, V, dO, UQ, UK, UV = X
    P = pins.softmax_probs(Q, K, tau, causal)
    F = tau * (UQ @ K.T + Q @ UK.T)
    dP = dO @ V.T
    O = P @ V
    alpha = (P * F).sum(1)
    D = (dO * O).sum(1)
    Pt = dO @ UV.T + F * (dP - D[:, None]) - alpha[:, None] * dP
    E = (P * Pt).sum(1)
    assert np.allclose(r["alpha"], alpha, atol=1e-13)
    assert np.allclose(r["D"], D, atol=1e-13)
    assert np.allclose(r["E"], E, atol=1e-12)
