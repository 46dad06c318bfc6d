"""GPU parity of attention dropout (App. "Extensions"): O = sigma (R o P) V,
and the first backward and the BoB of that forward, with the keep mask R
regenerated from Philox in every kernel.  Every kernel runs through the C
ABI and is compared with the fp64 oracle under the same (p, seed); the keep
mask itself is compared bit for bit with an independent numpy Philox."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G
from tests import pins

pytestmark = pytest.mark.gpu

CASES = [  # B, H, N, d, causal, p, seed, window, kv_heads
    (1, 2, 300, 64, True, 0.1, 1234, None, None),
    (2, 1, 257, 128, False, 0.5, (9 << 32) + 77, None, None),
    (1, 3, 200, 64, False, 0.3, 42, None, None),
    (1, 2, 390, 128, True, 0.2, 7, None, None),
    (1, 1, 333, 128, False, 0.25, 99, (60, 45), None),
    (1, 4, 260, 128, True, 0.15, 5, None, 2),
    (2, 2, 130, 64, True, 0.9, 31337, None, None),
    (1, 2, 280, 32, True, 0.3, 77, None, None),
    (1, 4, 150, 32, False, 0.2, 78, (30, 30), 2),
]


def ids(c):
    B, H, N, d, causal, p, seed, win, hkv = c
    w = "" if win is None else f"w{win[0]}_{win[1]}"
    g = "" if hkv is None else f"g{hkv}"
    return f"B{B}H{H}N{N}d{d}{'c' if causal else ''}p{p}{w}{g}"


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


def oracle_heads_fwd_bwd(bits, scale, causal, win, drop):
    X = [G.f64(bits[n]) for n in ("q", "k", "v", "dout")]
    O, L = oracle.fwd(*X[:3], scale, causal, window=win, dropout=drop)
    dQ, dK, dV, Dv = oracle.bwd(*X, scale, causal, window=win, dropout=drop)
    return O, L, dQ, dK, dV, Dv


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_forward_and_first_backward_with_dropout(case):
    B, H, N, d, causal, p, seed, win, hkv = case
    drop = (p, seed)
    bits = G.inputs(B, H, N, d, seed=N + d + 1, kv_heads=hkv)
    scale = 1 / np.sqrt(d)
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    o, lse = fbob.attn_fwd(q, k, v, scale, causal, win, None, drop)
    dq, dk, dv, dstat = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal, win, None, drop)
    assert fbob.fbob_device_status() == 0
    O, L, dQ, dK, dV, Dv = oracle_heads_fwd_bwd(bits, scale, causal, win, drop)
    G.check("O", G.host(o), O)
    assert np.abs(lse.cpu().numpy() - L).max() <= 1e-3
    G.check("dQ", G.host(dq), dQ)
    G.check("dK", G.host(dk), dK)
    G.check("dV", G.host(dv), dV)
    G.check("D", dstat.cpu().numpy(), Dv)


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_bob_with_dropout(case):
    B, H, N, d, causal, p, seed, win, hkv = case
    drop = (p, seed)
    bits = G.inputs(B, H, N, d, seed=3 * N + d, kv_heads=hkv)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal, o_l=G.oracle_o_l(bits, scale, causal, win, dropout=drop),
                  window=win, dropout=drop)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, window=win,
                     dropout=drop)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)


def test_bob_with_dropout_packed_sequences():
    seg = [0, 70, 71, 200, 333]
    B, H, N, d, causal, drop = 1, 2, 333, 128, True, (0.2, 2024)
    bits = G.inputs(B, H, N, d, seed=17)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal, segments=seg, dropout=drop)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, segments=seg,
                     dropout=drop)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)


@pytest.mark.parametrize("d", [32, 64, 128])
def test_keep_mask_bit_exact_in_both_engines(d):
    """Zeros of O and dV are the keep mask, pair by pair.  Q = 0 makes P
    uniform over each row's keys; with V rows one-hot in (j mod d) and the
    band j in [i, i + d - 1], column a of row i of O holds only the key
    j = a (mod d) of its band: O_ia = sigma R_ij P_ij (row engine).  With
    dO rows one-hot in (i mod d) and the band j in [i - d + 1, i], column a
    of key j of dV holds only query i = a (mod d): dV_ja = sigma R_ij P_ij
    (column engine)."""
    t = G.torch()
    B, H, N, p, seed = 2, 3, 1000, 0.4, 0xDEADBEEF12345
    z = t.zeros(B, H, N, d, dtype=t.bfloat16, device="cuda")
    eye = t.eye(d, dtype=t.bfloat16, device="cuda")
    onehot = eye[t.arange(N, device="cuda") % d].expand(B, H, N, d).contiguous()
    scale = 1 / np.sqrt(d)
    idx = np.arange(N)
    for engine in ("row", "col"):
        win = (0, d - 1) if engine == "row" else (d - 1, 0)
        o, lse = fbob.attn_fwd(z, z, onehot, scale, False, win, None, (p, seed))
        if engine == "col":
            _, _, dv, _ = fbob.attn_bwd(z, z, z, o, lse, onehot, scale, False, win, None, (p, seed))
        assert fbob.fbob_device_status() == 0
        got = (o if engine == "row" else dv).float().cpu().numpy() != 0
        for hh in range(B * H):
            b, h = divmod(hh, H)
            R = pins.dropout_gate(N, p, seed, hh) > 0
            a = np.arange(d)
            if engine == "row":  # key j of column a in row i's band [i, i + d - 1]
                j = idx[:, None] + ((a[None, :] - idx[:, None]) % d)
                valid = j < N
                want = np.where(valid, R[idx[:, None], np.minimum(j, N - 1)], False)
            else:                # query i of column a in key j's band [j, j + d - 1]
                i = idx[:, None] + ((a[None, :] - idx[:, None]) % d)
                valid = i < N
                want = np.where(valid, R[np.minimum(i, N - 1), idx[:, None]], False)
            assert np.array_equal(got[b, h], want), (engine, hh, int((got[b, h] != want).sum()))


@pytest.mark.parametrize("p", [0.0, 0.0015])
def test_rate_rounding_to_zero_is_no_dropout(p):
    """A rate that rounds to a zero byte threshold runs the kernels without
    dropout: results are bitwise those of the call without it."""
    B, H, N, d, causal = 1, 2, 250, 128, True
    bits = G.inputs(B, H, N, d, seed=23)
    scale = 1 / np.sqrt(d)
    a = G.run_bob(bits, scale, causal)
    b = G.run_bob(bits, scale, causal, dropout=(p, 5))
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D", "o", "lse"):
        assert np.array_equal(a[n], b[n]), n


def test_dropout_rate_out_of_range_is_rejected():
    t = G.torch()
    x = t.zeros(1, 1, 64, 64, dtype=t.bfloat16, device="cuda")
    for p in (1.0, -0.1, float("nan")):
        with pytest.raises(fbob.FbobError):
            fbob.attn_fwd(x, x, x, 0.125, False, None, None, (p, 1))


def test_hessian_vector_product_through_autograd_with_dropout():
    t = G.torch()
    from paper_2609_24089_gb300.autograd import attention
    B, H, N, d, causal, p, seed = 1, 2, 230, 64, True, 0.2, 8
    bits = G.inputs(B, H, N, d, seed=13)
    scale = 1 / np.sqrt(d)
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    for x in (q, k, v, do):
        x.requires_grad_(True)
    o = attention(q, k, v, scale, causal, dropout_p=p, seed=seed)
    loss = (o.float() * do.float()).sum()
    dq, dk, dv = t.autograd.grad(loss, (q, k, v), create_graph=True)
    phi = ((dq.float() * gq.float()).sum() + (dk.float() * gk.float()).sum()
           + (dv.float() * gv.float()).sum())
    qb, kb, vb, dob = t.autograd.grad(phi, (q, k, v, do))
    assert fbob.fbob_device_status() == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, dropout=(p, seed))
    for name, got, want in zip(("qbar", "kbar", "vbar", "dobar"), (qb, kb, vb, dob), ref):
        G.check(name, G.host(got), want)
