"""Pins for the oracle's grouped-query attention (query head h reads key/value
head h // G): torch fp64 double backward through attention with the key/value
heads repeated across each group (autograd sums the group's gradients by
itself), for the forward, the first backward and the BoB."""
import numpy as np
import pytest

import oracle
from tests import pins


@pytest.mark.parametrize("H,Hkv,causal", [(4, 2, True), (3, 1, False), (4, 4, True)])
def test_gqa_against_torch_double_backward(H, Hkv, causal):
    torch = pytest.importorskip("torch")
    B, N, d = 1, 24, 8
    rng = np.random.default_rng(40 + H + Hkv)
    q, do, gq = (rng.standard_normal((B, H, N, d)) for _ in range(3))
    k, v, gk, gv = (rng.standard_normal((B, Hkv, N, d)) for _ in range(4))
    tau = 1 / np.sqrt(d)
    G = H // Hkv
    T = lambda x, g=True: torch.tensor(x, dtype=torch.float64, requires_grad=g)
    tq, tk, tv, tdo = T(q), T(k), T(v), T(do)
    kk = tk.repeat_interleave(G, dim=1)
    vv = tv.repeat_interleave(G, dim=1)
    s = tau * tq @ kk.transpose(-1, -2)
    if causal:
        s = s.masked_fill(torch.triu(torch.ones(N, N, dtype=torch.bool), 1), float("-inf"))
    o = torch.softmax(s, dim=-1) @ vv
    dq, dk, dv = torch.autograd.grad(o, (tq, tk, tv), tdo, create_graph=True)
    phi = ((dq * T(gq, False)).sum() + (dk * T(gk, False)).sum() + (dv * T(gv, False)).sum())
    grads = torch.autograd.grad(phi, (tq, tk, tv, tdo))
    ref = oracle.bob(q, k, v, do, gq, gk, gv, tau, causal)
    for name, g, r in zip(("qbar", "kbar", "vbar", "dobar"), grads, ref):
        assert r.shape == tuple(g.shape), name
        assert pins.rel_fro(g.numpy(), r) <= 1e-12, name
    O, L = oracle.fwd(q, k, v, tau, causal)
    assert np.allclose(O, o.detach().numpy(), atol=1e-12)
    dQ, dK, dV, _ = oracle.bwd(q, k, v, do, tau, causal)
    for got, want in ((dQ, dq), (dK, dk), (dV, dv)):
        assert np.allclose(got, want.detach().numpy(), atol=1e-12)
