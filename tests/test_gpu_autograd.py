"""Double backward through torch.autograd: attention(q, k, v) -> grad with
create_graph -> grad again runs fwd -> bwd -> BoB in the library's kernels and
must agree with the fp64 oracle's BoB (Sec. 3.1, eqs. 4-7)."""
import numpy as np
import pytest

import oracle
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G


@pytest.mark.gpu
@pytest.mark.parametrize("shape", [(1, 2, 200, 64, True), (1, 1, 257, 128, False),
                                   (1, 2, 150, 256, True)],
                         ids=lambda s: "B{}H{}N{}d{}{}".format(*s[:4], "c" if s[4] else ""))
def test_hessian_vector_product_through_autograd(shape):
    t = G.torch()
    from paper_2609_24089_gb300.autograd import attention
    B, H, N, d, causal = shape
    bits = G.inputs(B, H, N, d, seed=11)
    scale = 1 / np.sqrt(d)
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    for x in (q, k, v, do):
        x.requires_grad_(True)
    o = attention(q, k, v, scale, causal)
    loss = (o.float() * do.float()).sum()                      # dL/dO = dO
    dq, dk, dv = t.autograd.grad(loss, (q, k, v), create_graph=True)
    phi = ((dq.float() * gq.float()).sum() + (dk.float() * gk.float()).sum()
           + (dv.float() * gv.float()).sum())
    qb, kb, vb, dob = t.autograd.grad(phi, (q, k, v, do))
    import paper_2609_24089_gb300 as fbob
    assert fbob.fbob_device_status() == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal)
    for name, got, want in zip(("qbar", "kbar", "vbar", "dobar"), (qb, kb, vb, dob), ref):
        G.check(name, G.host(got), want)
    # the first backward itself, against the oracle
    dQ, dK, dV, _ = oracle.bwd(*(G.f64(bits[n]) for n in ("q", "k", "v", "dout")), scale, causal)
    G.check("dQ", G.host(dq.detach()), dQ)
    G.check("dK", G.host(dk.detach()), dK)
    G.check("dV", G.host(dv.detach()), dV)


@pytest.mark.gpu
def test_hessian_vector_product_with_block_mask_and_dropout():
    """The same double backward under a block-sparse mask and dropout: the mask
    and the keep mask reach the forward, the first backward and the BoB."""
    t = G.torch()
    from paper_2609_24089_gb300.autograd import attention
    B, H, N, d, causal = 1, 2, 400, 64, True
    bits = G.inputs(B, H, N, d, seed=13)
    scale = 1 / np.sqrt(d)
    nb = (N + 127) // 128
    bm = np.eye(nb, dtype=np.uint8)
    bm[2, 0] = bm[3, 1] = 1
    drop = (0.1, 77)
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    for x in (q, k, v, do):
        x.requires_grad_(True)
    o = attention(q, k, v, scale, causal, dropout_p=drop[0], seed=drop[1],
                  block_mask=G.dev_blocks(bm))
    loss = (o.float() * do.float()).sum()
    dq, dk, dv = t.autograd.grad(loss, (q, k, v), create_graph=True)
    phi = ((dq.float() * gq.float()).sum() + (dk.float() * gk.float()).sum()
           + (dv.float() * gv.float()).sum())
    qb, kb, vb, dob = t.autograd.grad(phi, (q, k, v, do))
    import paper_2609_24089_gb300 as fbob
    assert fbob.fbob_device_status() == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, dropout=drop,
                     block_mask=bm)
    for name, got, want in zip(("qbar", "kbar", "vbar", "dobar"), (qb, kb, vb, dob), ref):
        G.check(name, G.host(got), want)


def test_attention_rejects_host_tensors():
    """No CPU fallback: host or non-bf16 tensors are refused before any call."""
    torch = pytest.importorskip("torch")
    from paper_2609_24089_gb300.autograd import attention
    x = torch.zeros(1, 1, 8, 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        attention(x, x, x)
    with pytest.raises(ValueError):
        attention(x.float(), x.float(), x.float())
