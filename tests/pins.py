"""Independent references used to pin the fp64 oracle.

Nothing here imports the oracle.  The first backward below is written in
matrix form from Sec. 2 eqs. (1)-(3) (numpy, batched, real or complex), so
finite differences and complex-step derivatives of

    Phi = <dQ, U_Q> + <dK, U_K> + <dV, U_V>          (eq. 4)

give backward-over-backward results that owe nothing to the oracle's
closed-form App. C walk.
"""
from __future__ import annotations

import numpy as np


def mask(N, causal, window=None, segments=None, block=None):
    """0/1 mask: causal keeps j <= i; window (wl, wr) keeps i - wl <= j <= i + wr
    (a negative side is unbounded); segments (offsets of packed sequences)
    keeps i and j in the same sequence (a block-diagonal mask); block
    (bm, bs) keeps (i, j) only where the [nb, nb] 0/1 block mask bm has its
    block (i // bs, j // bs) set (a block-sparse mask)."""
    i = np.arange(N)[:, None]
    j = np.arange(N)[None, :]
    keep = np.ones((N, N), dtype=bool)
    if block is not None:
        bm, bs = block
        keep &= np.asarray(bm)[i // bs, j // bs] != 0
    if segments is not None:
        sid = np.searchsorted(np.asarray(segments)[1:], np.arange(N), side="right")
        keep &= sid[:, None] == sid[None, :]
    if causal:
        keep &= j <= i
    if window is not None:
        wl, wr = window
        if wl >= 0:
            keep &= j >= i - wl
        if wr >= 0:
            keep &= j <= i + wr
    return keep.astype(np.float64)


def softmax_probs(Q, K, tau, causal, window=None, segments=None, block=None):
    """P = softmax_row(tau Q K^T + M) for [..., N, d] inputs (real or complex).

    The shift uses the real part of the row max so the function stays
    complex-analytic (the shift cancels exactly in the ratio)."""
    N = Q.shape[-2]
    S = tau * (Q @ np.swapaxes(K, -1, -2))
    Mk = mask(N, causal, window, segments, block)
    shift = np.max(np.where(Mk > 0, S.real, -np.inf), axis=-1, keepdims=True)
    Ex = np.exp(S - shift) * Mk
    return Ex / Ex.sum(axis=-1, keepdims=True)


def first_backward(Q, K, V, dO, tau, causal, window=None, segments=None, gate=None,
                   block=None):
    """g(Q, K, V, dO) = (dQ, dK, dV), eqs. (2)-(3), batched over leading dims.
    gate: [N, N] dropout gate sigma R of the forward O = (gate o P) V, which
    turns the derivative with respect to P into gate o (dO V^T) and dV into
    (gate o P)^T dO."""
    P = softmax_probs(Q, K, tau, causal, window, segments, block)
    g = 1.0 if gate is None else gate
    dP = g * (dO @ np.swapaxes(V, -1, -2))
    D = (P * dP).sum(axis=-1, keepdims=True)
    dS = P * (dP - D)
    dQ = tau * dS @ K
    dK = tau * np.swapaxes(dS, -1, -2) @ Q
    dV = np.swapaxes(g * P, -1, -2) @ dO
    return dQ, dK, dV


def attention(Q, K, V, tau, causal, window=None, segments=None, gate=None, block=None):
    P = softmax_probs(Q, K, tau, causal, window, segments, block)
    return (P if gate is None else gate * P) @ V


def phi(Q, K, V, dO, UQ, UK, UV, tau, causal, window=None, segments=None, gate=None,
        block=None):
    dQ, dK, dV = first_backward(Q, K, V, dO, tau, causal, window, segments, gate, block)
    return ((dQ * UQ).sum(axis=(-1, -2)) + (dK * UK).sum(axis=(-1, -2))
            + (dV * UV).sum(axis=(-1, -2)))


_M0, _M1 = np.uint64(0xD2511F53), np.uint64(0xCD9E8D57)
_W0, _W1 = np.uint32(0x9E3779B9), np.uint32(0xBB67AE85)
_LO = np.uint64(0xFFFFFFFF)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Philox4x32-10 (Salmon et al., SC'11) on arrays of uint32 counter words
    under a scalar key, vectorised in numpy: each round multiplies words 0 and
    2 by the Philox multipliers, swaps the products' halves into the four
    words, xors the key in, and raises the key by the Weyl constants."""
    c = [np.asarray(x, dtype=np.uint32) for x in (c0, c1, c2, c3)]
    k0, k1 = np.uint32(k0), np.uint32(k1)
    with np.errstate(over="ignore"):
        for r in range(10):
            if r:
                k0 = np.uint32(k0 + _W0)
                k1 = np.uint32(k1 + _W1)
            p0 = _M0 * c[0].astype(np.uint64)
            p1 = _M1 * c[2].astype(np.uint64)
            c = [((p1 >> np.uint64(32)).astype(np.uint32) ^ c[1] ^ k0),
                 (p1 & _LO).astype(np.uint32),
                 ((p0 >> np.uint64(32)).astype(np.uint32) ^ c[3] ^ k1),
                 (p0 & _LO).astype(np.uint32)]
    return c


def dropout_gate(N, p, seed, head):
    """[N, N] gate sigma R of one head.  The (query, key) pair (i, j) reads
    byte j mod 4 of word i mod 4 of Philox4x32-10(counter (j div 4, i div 4,
    head, 0), key (seed mod 2^32, seed div 2^32)); R_ij = 1 iff that byte is
    at least t = min(255, floor(256 p + 1/2)), and sigma = 256 / (256 - t)."""
    i = np.arange(N, dtype=np.uint32)[:, None]
    j = np.arange(N, dtype=np.uint32)[None, :]
    z = np.zeros((N, N), dtype=np.uint32)
    w = philox4x32_10(z + (j >> np.uint32(2)), z + (i >> np.uint32(2)), z + np.uint32(head), z,
                      seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
    word = np.choose((i & np.uint32(3)).astype(np.int64) + 0 * z, w)
    byte = (word >> (np.uint32(8) * (j & np.uint32(3)))) & np.uint32(0xFF)
    t = min(255, int(np.floor(256 * p + 0.5)))
    if t == 0:
        return np.ones((N, N))
    return (byte >= np.uint32(t)).astype(np.float64) * (256.0 / (256 - t))


def dropout_rate(p):
    """The realised drop rate t / 256 of a requested rate p."""
    return min(255, int(np.floor(256 * p + 0.5))) / 256


def _perturbed(X, which, deltas):
    """Stack of copies of the 4 primal inputs with input `which` perturbed
    entrywise: returns list of 4 arrays shaped [N*d, N, d]."""
    N, d = X[0].shape
    out = []
    for t in range(4):
        base = np.broadcast_to(X[t], (N * d, N, d)).astype(np.result_type(X[t], deltas))
        if t == which:
            base = base.copy()
            idx = np.arange(N * d)
            base[idx, idx // d, idx % d] += deltas
        out.append(base)
    return out


def bob_central_fd(Q, K, V, dO, UQ, UK, UV, tau, causal, rel_h=1e-5, window=None,
                   segments=None, gate=None, block=None):
    """grad_{Q,K,V,dO} Phi by central differences, one entry at a time."""
    X = [Q, K, V, dO]
    grads = []
    for which in range(4):
        x = X[which].reshape(-1)
        h = rel_h * np.maximum(1.0, np.abs(x))
        plus = _perturbed(X, which, h)
        minus = _perturbed(X, which, -h)
        fp = phi(*plus, UQ, UK, UV, tau, causal, window, segments, gate, block)
        fm = phi(*minus, UQ, UK, UV, tau, causal, window, segments, gate, block)
        grads.append(((fp - fm) / (2 * h)).reshape(X[which].shape))
    return grads


def jacobian_complex_step(Q, K, V, dO, tau, causal, h=1e-30, window=None):
    """Explicit Jacobian of g: rows index vec(dQ, dK, dV) (3Nd), columns index
    vec(Q, K, V, dO) (4Nd); built column by column by complex step."""
    N, d = Q.shape
    X = [Q.astype(complex), K.astype(complex), V.astype(complex), dO.astype(complex)]
    cols = []
    for which in range(4):
        pert = _perturbed(X, which, np.full(N * d, 1j * h))
        dQ, dK, dV = first_backward(*pert, tau, causal, window)
        J = np.concatenate([dQ.reshape(N * d, -1), dK.reshape(N * d, -1),
                            dV.reshape(N * d, -1)], axis=1).imag / h   # [Nd(in), 3Nd(out)]
        cols.append(J.T)
    return np.concatenate(cols, axis=1)                                 # [3Nd, 4Nd]


def inner(a, b):
    return float(np.sum(np.asarray(a) * np.asarray(b)))


def rel_fro(x, ref):
    den = np.linalg.norm(ref)
    return np.linalg.norm(x - ref) / (den if den > 0 else 1.0)
