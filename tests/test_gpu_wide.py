"""GPU parity of the head-dimension-256 kernels (wide_engine.cuh) against the
fp64 oracle: forward, first backward and backward-over-backward at ragged N,
each pass alone, the mask and head-layout variants, dropout, determinism, and
the full-size n16k_d256_causal workload.  All calls go through the C ABI."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

D = 256
SHAPES = [  # B, H, N, causal
    (1, 1, 128, False),
    (1, 2, 17, True),
    (2, 1, 100, False),
    (1, 1, 300, True),
    (1, 2, 257, False),
    (1, 1, 1, True),
    (1, 1, 3, False),
    (1, 1, 520, True),
]


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


def ids(s):
    return "B{}H{}N{}{}".format(*s[:3], "c" if s[3] else "")


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_forward_and_first_backward(shape):
    B, H, N, causal = shape
    bits = G.inputs(B, H, N, D, seed=N + 3)
    scale = 1 / np.sqrt(D)
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    o, lse = fbob.attn_fwd(q, k, v, scale, causal)
    assert fbob.fbob_launch_count("fwd") == 1
    dq, dk, dv, dstat = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal)
    assert fbob.fbob_launch_count("bwd") == 3
    assert fbob.fbob_device_status() == 0
    X = [G.f64(bits[n]) for n in ("q", "k", "v", "dout")]
    O, L = oracle.fwd(*X[:3], scale, causal)
    G.check("O", G.host(o), O)
    assert np.abs(lse.cpu().numpy() - L).max() <= 1e-3
    dQ, dK, dV, Dv = oracle.bwd(*X, scale, causal)
    if N == 1:
        # one key: P = 1, so dS = dP - D = do . v - do . o vanishes exactly in
        # real arithmetic, and dQ = tau dS k, dK = tau dS q are zero up to
        # fp32 summation order: dP (tensor core) and D (do . o from the bf16
        # O = v) each carry at most d 2^-24 sum_a |do_a v_a| of rounding
        # (the classical bound on a d-term dot product), so
        # |dS| <= 2^-22 d sum_a |do_a v_a| with a factor 2 of margin.
        do_, v_ = X[3][..., 0, :], X[2][..., 0, :]
        ds_max = 2.0 ** -22 * D * np.abs(do_ * v_).sum(-1)
        assert np.all(np.abs(G.host(dq)[..., 0, :]) <= scale * ds_max[..., None] *
                      np.abs(X[1][..., 0, :]))
        assert np.all(np.abs(G.host(dk)[..., 0, :]) <= scale * ds_max[..., None] *
                      np.abs(X[0][..., 0, :]))
    else:
        G.check("dQ", G.host(dq), dQ)
        G.check("dK", G.host(dk), dK)
    G.check("dV", G.host(dv), dV)
    G.check("D", dstat.cpu().numpy(), Dv)


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_bob_end_to_end(shape):
    B, H, N, causal = shape
    bits = G.inputs(B, H, N, D, seed=7 * N + 5)
    scale = 1 / np.sqrt(D)
    r = G.run_bob(bits, scale, causal)
    assert r["status"] == 0
    assert fbob.fbob_launch_count("bob") == 4
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        if N == 1 and name in ("qbar", "kbar", "vbar"):
            continue  # exact zeros up to rounding: test_single_key_degenerate bounds them
        G.check(name, r[name], x)


@pytest.mark.parametrize("shape", [(1, 2, 300, True), (2, 1, 200, False)], ids=ids)
def test_each_pass_alone(shape):
    """Pass 1 (two kernels: row scalars with dOtil, then Qtil), the row
    statistics alone, the direct form (dOtil, Qtil) and Pass 2 fed the
    oracle's row state."""
    B, H, N, causal = shape
    bits = G.inputs(B, H, N, D, seed=41)
    scale = 1 / np.sqrt(D)
    X = [G.f64(bits[n]) for n in synth.NAMES]
    qb, kb, vb, dob, al, E, Dv = oracle.bob(*X, scale, causal)
    o_bits, L = G.oracle_o_l(bits, scale, causal)
    rs_ref = np.stack([al, E, Dv]).astype(np.float32)
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    o, lse = G.dev(o_bits), G.dev_f32(L)
    shp = fbob.make_shape(B, H, N, D, scale, causal)
    q_bar, dout_bar = t.empty_like(q), t.empty_like(q)
    rs = t.empty((3, B, H, N), dtype=t.float32, device="cuda")
    fbob.fbob_attn_bob_pass1(shp, q, k, v, o, lse, do, gq, gk, gv, q_bar, dout_bar, rs)
    assert fbob.fbob_launch_count("bob_pass1") == 2
    assert fbob.fbob_device_status() == 0
    got = rs.cpu().numpy().astype(np.float64)
    for i, name in enumerate(("alpha", "E", "D")):
        G.check(name, got[i], rs_ref[i])
    G.check("qbar", G.host(q_bar), qb)
    G.check("dobar", G.host(dout_bar), dob)
    rs2 = t.empty((3, B, H, N), dtype=t.float32, device="cuda")
    fbob.fbob_attn_bob_row_stats(shp, q, k, v, o, lse, do, gq, gk, gv, rs2)
    assert fbob.fbob_launch_count("bob_row_stats") == 1
    assert fbob.fbob_device_status() == 0
    assert np.array_equal(rs2.cpu().numpy(), rs.cpu().numpy())
    q2, d2 = t.empty_like(q), t.empty_like(q)
    fbob.fbob_attn_bob_pass1_direct(shp, q, k, v, lse, do, gq, gk, gv, G.dev_f32(rs_ref), q2, d2)
    assert fbob.fbob_launch_count("bob_pass1_direct") == 2
    k_bar, v_bar = t.empty_like(k), t.empty_like(v)
    fbob.fbob_attn_bob_pass2(shp, q, k, v, lse, do, gq, gk, gv, G.dev_f32(rs_ref), k_bar, v_bar)
    assert fbob.fbob_launch_count("bob_pass2") == 2
    assert fbob.fbob_device_status() == 0
    G.check("qbar(direct)", G.host(q2), qb)
    G.check("dobar(direct)", G.host(d2), dob)
    G.check("kbar", G.host(k_bar), kb)
    G.check("vbar", G.host(v_bar), vb)


def test_one_sweep_pass1_is_unsupported():
    """Four 256-column accumulators do not fit TMEM: the fused entry point
    refuses d = 256 before any launch."""
    B, H, N = 1, 1, 64
    bits = G.inputs(B, H, N, D, seed=2)
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    shp = fbob.make_shape(B, H, N, D, 1 / np.sqrt(D), True)
    lse = t.zeros((B, H, N), dtype=t.float32, device="cuda")
    rs = t.empty((3, B, H, N), dtype=t.float32, device="cuda")
    with pytest.raises(RuntimeError, match="UNSUPPORTED"):
        fbob.fbob_attn_bob_pass1_fused(shp, q, k, v, q, lse, do, gq, gk, gv, t.empty_like(q),
                                       t.empty_like(q), rs)


VARIANTS = {  # name: (B, H, N, causal, extra)
    "window": (1, 2, 333, True, dict(window=(100, -1))),
    "band": (1, 1, 300, False, dict(window=(40, 70))),
    "varlen": (1, 2, 400, True, dict(segments=[0, 37, 200, 201, 400])),
    "gqa": (1, 4, 270, True, dict(kv_heads=2)),
    "mqa": (2, 3, 150, False, dict(kv_heads=1)),
    "blocks": (1, 2, 520, True, dict(block_mask="random")),
    "dropout": (1, 2, 300, True, dict(dropout=(0.1, 12345))),
    "dropout_gqa": (1, 4, 200, False, dict(dropout=(0.25, 99), kv_heads=2)),
}


@pytest.mark.parametrize("name", list(VARIANTS))
def test_variants(name):
    """Masks (band, packed sequences, block-sparse), grouped-query heads and
    dropout at d = 256: forward, first backward and BoB against the oracle."""
    B, H, N, causal, ex = VARIANTS[name]
    kvh = ex.get("kv_heads")
    bits = G.inputs(B, H, N, D, seed=len(name) * 31 + N, kv_heads=kvh)
    scale = 1 / np.sqrt(D)
    window = ex.get("window")
    segments = ex.get("segments")
    dropout = ex.get("dropout")
    bm = None
    if ex.get("block_mask") == "random":
        nb = (N + 127) // 128
        rng = np.random.default_rng(N)
        bm = (rng.random((nb, nb)) < 0.5).astype(np.uint8)
        np.fill_diagonal(bm, 1)
    kw = dict(window=window, segments=segments, dropout=dropout, block_mask=bm)
    X = [G.f64(bits[n]) for n in synth.NAMES]
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    seg, bmk = G.dev_segments(segments), G.dev_blocks(bm)
    o, lse = fbob.attn_fwd(q, k, v, scale, causal, window, seg, dropout, bmk)
    dq, dk, dv, dstat = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal, window, seg, dropout, bmk)
    assert fbob.fbob_device_status() == 0
    O, L = oracle.fwd(X[0], X[1], X[2], scale, causal, **kw)
    G.check("O", G.host(o), O)
    assert np.abs(lse.cpu().numpy() - L).max() <= 1e-3
    dQ, dK, dV, Dv = oracle.bwd(*X[:4], scale, causal, **kw)
    G.check("dQ", G.host(dq), dQ)
    G.check("dK", G.host(dk), dK)
    G.check("dV", G.host(dv), dV)
    G.check("D", dstat.cpu().numpy(), Dv)
    r = G.run_bob(bits, scale, causal, window=window, segments=segments, dropout=dropout,
                  block_mask=bm)
    assert r["status"] == 0
    ref = oracle.bob(*X, scale, causal, **kw)
    for nm, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(nm, r[nm], x)


def test_runs_are_bitwise_identical():
    bits = G.inputs(1, 3, 555, D, seed=9)
    scale = 1 / np.sqrt(D)
    a = G.run_bob(bits, scale, True)
    b = G.run_bob(bits, scale, True)
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D", "o", "lse"):
        assert np.array_equal(a[n], b[n]), n


def sample_rows(N, seed, n=24):
    rng = np.random.default_rng(seed)
    fixed = [0, 1, 31, 32, 127, 128, N // 2, N - 129, N - 1]
    rows = set(r for r in fixed if 0 <= r < N)
    rows.update(rng.integers(0, N, n).tolist())
    return np.array(sorted(rows), dtype=np.int64)


def test_n16k_d256_causal_rows_and_tail():
    """The full-size head-dimension-256 workload in the configuration the
    benchmark times: sampled rows of two heads, and the causal tail (key
    columns >= N - 256 are complete once rows >= N - 256 are summed)."""
    w = synth.WORKLOADS["n16k_d256_causal"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal)
    assert r["status"] == 0
    N = w.N
    heads = [0, w.B * w.H - 1]
    rows = sample_rows(N, 256)
    refs = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=rows)
    for hh, ref in zip(heads, refs):
        for name in ("qbar", "dobar", "alpha", "E", "D"):
            G.check(f"{name}[head {hh}]", G.flat(r[name], hh, w.H)[rows], ref[name])
    t0 = N - 256
    tail = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=np.arange(t0, N), cols=(t0, N))
    for hh, ref in zip(heads, tail):
        G.check("kbar[tail]", G.flat(r["kbar"], hh, w.H)[t0:], ref["kbar"])
        G.check("vbar[tail]", G.flat(r["vbar"], hh, w.H)[t0:], ref["vbar"])
