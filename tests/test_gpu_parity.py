"""GPU parity against the fp64 oracle at sizes the oracle finishes in seconds:
several tiles, ragged tails, both masks, both head dims, every kernel alone
and the whole pipeline.  All calls go through the C ABI."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

SHAPES = [  # B, H, N, d, causal
    (1, 1, 128, 64, False),
    (1, 2, 17, 64, True),
    (2, 1, 100, 128, False),
    (1, 1, 129, 64, True),
    (1, 2, 300, 128, True),
    (1, 3, 257, 64, False),
    (1, 1, 2, 64, False),
    (1, 1, 3, 128, True),
    (2, 2, 384, 128, False),
    (1, 2, 520, 64, True),
    (1, 1, 128, 32, False),   # head dim 32 (in 64-wide tiles)
    (1, 2, 301, 32, True),
    (2, 1, 3, 32, False),
]


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


def ids(s):
    return "B{}H{}N{}d{}{}".format(*s[:4], "c" if s[4] else "")


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_forward_and_first_backward(shape):
    B, H, N, d, causal = shape
    bits = G.inputs(B, H, N, d, seed=N + d)
    scale = 1 / np.sqrt(d)
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    o, lse = fbob.attn_fwd(q, k, v, scale, causal)
    dq, dk, dv, dstat = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal)
    assert fbob.fbob_device_status() == 0
    X = [G.f64(bits[n]) for n in ("q", "k", "v", "dout")]
    O, L = oracle.fwd(*X[:3], scale, causal)
    G.check("O", G.host(o), O)
    assert np.abs(lse.cpu().numpy() - L).max() <= 1e-3
    dQ, dK, dV, Dv = oracle.bwd(*X, scale, causal)
    G.check("dQ", G.host(dq), dQ)
    G.check("dK", G.host(dk), dK)
    G.check("dV", G.host(dv), dV)
    G.check("D", dstat.cpu().numpy(), Dv)


@pytest.mark.parametrize("shape", SHAPES, ids=ids)
def test_bob_end_to_end(shape):
    B, H, N, d, causal = shape
    bits = G.inputs(B, H, N, d, seed=7 * N + d)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)


@pytest.mark.parametrize("shape", [(1, 2, 300, 64, True), (2, 1, 200, 128, False),
                                   (1, 1, 190, 32, True)], ids=ids)
def test_pass2_alone_on_oracle_row_state(shape):
    """Algorithm 2's second loop fed the oracle's L, D, alpha, E."""
    B, H, N, d, causal = shape
    bits = G.inputs(B, H, N, d, seed=3)
    scale = 1 / np.sqrt(d)
    X = [G.f64(bits[n]) for n in synth.NAMES]
    qb, kb, vb, dob, al, E, D = oracle.bob(*X, scale, causal)
    _, L = oracle.fwd(*X[:3], scale, causal)
    rs = np.stack([al, E, D]).astype(np.float32)
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    k_bar, v_bar = t.empty_like(k), t.empty_like(v)
    shp = fbob.make_shape(B, H, N, d, scale, causal)
    fbob.fbob_attn_bob_pass2(shp, q, k, v, G.dev_f32(L), do, gq, gk, gv, G.dev_f32(rs),
                             k_bar, v_bar)
    assert fbob.fbob_device_status() == 0
    G.check("kbar", G.host(k_bar), kb)
    G.check("vbar", G.host(v_bar), vb)


@pytest.mark.parametrize("shape", [(1, 2, 300, 64, True), (2, 1, 200, 128, False)], ids=ids)
def test_pass1_alone(shape):
    """Algorithm 2's first loop: Qtil, dOtil and the row scalars alpha, E, D."""
    B, H, N, d, causal = shape
    bits = G.inputs(B, H, N, d, seed=4)
    scale = 1 / np.sqrt(d)
    X = [G.f64(bits[n]) for n in synth.NAMES]
    qb, kb, vb, dob, al, E, D = oracle.bob(*X, scale, causal)
    o_bits, L = G.oracle_o_l(bits, scale, causal)
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    q_bar, dout_bar = t.empty_like(q), t.empty_like(q)
    rs = t.empty((3, B, H, N), dtype=t.float32, device="cuda")
    shp = fbob.make_shape(B, H, N, d, scale, causal)
    fbob.fbob_attn_bob_pass1(shp, q, k, v, G.dev(o_bits), G.dev_f32(L), do, gq, gk, gv,
                             q_bar, dout_bar, rs)
    assert fbob.fbob_device_status() == 0
    rs = rs.cpu().numpy().astype(np.float64)
    G.check("alpha", rs[0], al)
    G.check("E", rs[1], E)
    G.check("D", rs[2], D)
    G.check("qbar", G.host(q_bar), qb)
    G.check("dobar", G.host(dout_bar), dob)


@pytest.mark.parametrize("shape", [(1, 2, 300, 64, True), (2, 1, 200, 128, False),
                                   (1, 1, 129, 128, True)], ids=ids)
def test_row_stats_alone(shape):
    """The row scalars of eq. (6) from the statistics kernel alone."""
    B, H, N, d, causal = shape
    bits = G.inputs(B, H, N, d, seed=5)
    scale = 1 / np.sqrt(d)
    X = [G.f64(bits[n]) for n in synth.NAMES]
    _, _, _, _, al, E, D = oracle.bob(*X, scale, causal)
    o_bits, L = G.oracle_o_l(bits, scale, causal)
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    rs = t.empty((3, B, H, N), dtype=t.float32, device="cuda")
    shp = fbob.make_shape(B, H, N, d, scale, causal)
    fbob.fbob_attn_bob_row_stats(shp, q, k, v, G.dev(o_bits), G.dev_f32(L), do, gq, gk, gv, rs)
    assert fbob.fbob_device_status() == 0
    assert fbob.fbob_launch_count("bob_row_stats") == 1
    rs = rs.cpu().numpy().astype(np.float64)
    G.check("alpha", rs[0], al)
    G.check("E", rs[1], E)
    G.check("D", rs[2], D)


@pytest.mark.parametrize("shape", [(1, 2, 300, 64, True), (2, 1, 200, 128, False),
                                   (1, 1, 257, 128, True)], ids=ids)
def test_pass1_direct_on_oracle_row_state(shape):
    """Qtil, dOtil from eqs. (6)-(7) given the oracle's alpha, E, D and L."""
    B, H, N, d, causal = shape
    bits = G.inputs(B, H, N, d, seed=6)
    scale = 1 / np.sqrt(d)
    X = [G.f64(bits[n]) for n in synth.NAMES]
    qb, _, _, dob, al, E, D = oracle.bob(*X, scale, causal)
    _, L = oracle.fwd(*X[:3], scale, causal)
    rs = np.stack([al, E, D]).astype(np.float32)
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    q_bar, dout_bar = t.empty_like(q), t.empty_like(q)
    shp = fbob.make_shape(B, H, N, d, scale, causal)
    fbob.fbob_attn_bob_pass1_direct(shp, q, k, v, G.dev_f32(L), do, gq, gk, gv, G.dev_f32(rs),
                                    q_bar, dout_bar)
    assert fbob.fbob_device_status() == 0
    assert fbob.fbob_launch_count("bob_pass1_direct") == 1
    G.check("qbar", G.host(q_bar), qb)
    G.check("dobar", G.host(dout_bar), dob)


def test_one_sweep_and_two_kernel_pass1_agree_at_d64():
    """At d = 64 both Pass-1 schedules exist; they compute the same outputs."""
    B, H, N, d, causal = 1, 2, 333, 64, True
    bits = G.inputs(B, H, N, d, seed=8)
    scale = 1 / np.sqrt(d)
    o_bits, L = G.oracle_o_l(bits, scale, causal)
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    o, lse = G.dev(o_bits), G.dev_f32(L)
    shp = fbob.make_shape(B, H, N, d, scale, causal)
    qa, da = t.empty_like(q), t.empty_like(q)
    ra = t.empty((3, B, H, N), dtype=t.float32, device="cuda")
    fbob.fbob_attn_bob_pass1(shp, q, k, v, o, lse, do, gq, gk, gv, qa, da, ra)
    assert fbob.fbob_launch_count("bob_pass1") == 1
    qb, db = t.empty_like(q), t.empty_like(q)
    rb = t.empty((3, B, H, N), dtype=t.float32, device="cuda")
    fbob.fbob_attn_bob_row_stats(shp, q, k, v, o, lse, do, gq, gk, gv, rb)
    fbob.fbob_attn_bob_pass1_direct(shp, q, k, v, lse, do, gq, gk, gv, rb, qb, db)
    assert fbob.fbob_device_status() == 0
    G.check("row_stats", G.host(rb), G.host(ra), rel=1e-4, mx=1e-3)
    G.check("qbar", G.host(qb), G.host(qa))
    G.check("dobar", G.host(db), G.host(da))


def test_runs_are_bitwise_identical():
    bits = G.inputs(1, 4, 777, 128, seed=9)
    scale = 1 / np.sqrt(128)
    a = G.run_bob(bits, scale, True)
    b = G.run_bob(bits, scale, True)
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"):
        assert np.array_equal(a[n], b[n]), n


@pytest.mark.parametrize("d", [64, 256])
def test_lemma_d2_embedding_on_gpu(d):
    """V = dO = U_Q = U_K = 0, U_V = W: dOtil = softmax(tau Q K^T) W exactly
    (Lemma D.2) and the other outputs vanish."""
    B, H, N = 1, 2, 200
    bits = G.inputs(B, H, N, d, seed=21)
    z = np.zeros_like(bits["q"])
    for n in ("v", "dout", "gq", "gk"):
        bits[n] = z
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, True)
    O, _ = oracle.fwd(G.f64(bits["q"]), G.f64(bits["k"]), G.f64(bits["gv"]), scale, True)
    G.check("dobar", r["dobar"], O)
    for n in ("qbar", "kbar", "vbar"):
        assert np.abs(r[n]).max() == 0.0, n


@pytest.mark.parametrize("d,causal", [(64, False), (128, True), (256, True)])
def test_single_key_degenerate(d, causal):
    """N = 1: P = 1, so Qtil = Ktil = Vtil = 0 and dOtil = U_V exactly.  The
    fused form Qtil = tau (Omega - alpha R - E B) cancels to zero only up to
    the bf16 rounding of its operand tiles: with N = 1 it equals
    tau [(bf16(C) - C) - F (bf16(dP) - dP)] k, so |Qtil| is bounded by
    tau 2^-8 (|C| + |F dP|) max|k| (bf16 relative rounding <= 2^-9, factor 2
    of margin).  Ktil and Vtil cancel in fp32 (alpha and E are fp32)."""
    B, H, N = 1, 3, 1
    bits = G.inputs(B, H, N, d, seed=5 + d)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal)
    assert r["status"] == 0
    X = {n: G.f64(bits[n]) for n in synth.NAMES}
    for h in range(H):
        q, k, v, do, uq, uk, uv = (X[n][0, h, 0] for n in synth.NAMES)
        C = do @ uv
        F = scale * (uq @ k + q @ uk)
        dP = do @ v
        bound = scale * 2.0 ** -8 * (abs(C) + abs(F * dP)) * np.abs(k).max()
        assert np.abs(r["qbar"][0, h, 0]).max() <= bound, h
        G.check("dobar", r["dobar"][0, h, 0], uv)
    assert np.abs(r["kbar"]).max() <= 1e-4 * scale * np.abs(X["q"]).max() * np.abs(X["gv"]).max() * d
    assert np.abs(r["vbar"]).max() <= 1e-4 * np.abs(X["dout"]).max() * np.abs(X["gq"]).max() * d


STALL_CASES = [  # entry, d, causal, dropout
    ("bob", 64, False, None),     # one-sweep Pass 1, Pass 2 at d = 64
    ("bob", 128, True, None),     # row statistics + direct Pass 1, Pass 2 at d = 128
    ("bob", 32, True, None),      # head dim 32 in the d = 64 tiles
    ("bob", 128, True, (0.1, 5)),  # the dropout instantiations of all three
    ("bob", 64, False, (0.2, 9)),  # dropout at d = 64: statistics + direct form
    ("fwd", 64, False, None),     # forward engine (608 threads, its own barriers)
    ("fwd", 128, True, None),
    ("fwd", 128, False, (0.1, 3)),
    ("bwd", 64, True, None),      # first backward: dQ (row) and dK/dV (column) kernels
    ("bwd", 128, False, None),
    ("bwd", 128, True, (0.1, 4)),
    ("bob", 256, True, None),     # head dim 256: the five wide kernels of BoB
    ("bob", 256, False, (0.1, 6)),
    ("fwd", 256, True, None),     # the d = 256 forward (online softmax)
    ("bwd", 256, False, (0.1, 7)),  # dQ, dV and dK kernels
]


def stall_id(c):
    return "{}_d{}{}{}".format(c[0], c[1], "c" if c[2] else "", "_drop" if c[3] else "")


@pytest.mark.parametrize("case", STALL_CASES, ids=stall_id)
def test_bounded_wait_timeout_is_reported_and_context_survives(monkeypatch, case):
    """Failure detection without a GPU fault: with the producers' loads
    suppressed (FBOB_INJECT_STALL=1) every consumer wait runs into its bounded
    limit; the kernels record FBOB_ERR_DEVICE_TIMEOUT, release tensor memory
    and exit, and the next call on the same context computes correct results.
    Every kernel family is covered: the BoB passes (each Pass 1 form, with and
    without dropout), the forward and both first-backward kernels."""
    entry, d, causal, drop = case
    B, H, N = 1, 2, 300
    bits = G.inputs(B, H, N, d, seed=77 + d)
    scale = 1 / np.sqrt(d)
    X = {n: G.f64(bits[n]) for n in synth.NAMES}
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))

    def run():
        if entry == "fwd":
            o, lse = fbob.attn_fwd(q, k, v, scale, causal, dropout=drop)
            return fbob.fbob_device_status(), (o, lse)
        if entry == "bwd":
            o_l = G.oracle_o_l(bits, scale, causal, dropout=drop)
            o, lse = G.dev(o_l[0]), G.dev_f32(o_l[1])
            out = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal, dropout=drop)
            return fbob.fbob_device_status(), out
        r = G.run_bob(bits, scale, causal, o_l=G.oracle_o_l(bits, scale, causal, dropout=drop),
                      dropout=drop)
        return r["status"], r

    monkeypatch.setenv("FBOB_WAIT_LIMIT_MS", "50")
    monkeypatch.setenv("FBOB_INJECT_STALL", "1")
    status, _ = run()
    assert status == fbob.STATUS_CODES["FBOB_ERR_DEVICE_TIMEOUT"]
    monkeypatch.delenv("FBOB_INJECT_STALL")
    monkeypatch.delenv("FBOB_WAIT_LIMIT_MS")
    status, out = run()
    assert status == 0
    if entry == "fwd":
        O, _ = oracle.fwd(X["q"], X["k"], X["v"], scale, causal, dropout=drop)
        G.check("O", G.host(out[0]), O)
    elif entry == "bwd":
        ref = oracle.bwd(X["q"], X["k"], X["v"], X["dout"], scale, causal, dropout=drop)
        for name, got, x in zip(("dQ", "dK", "dV"), out[:3], ref[:3]):
            G.check(name, G.host(got), x)
    else:
        ref = oracle.bob(*(X[n] for n in synth.NAMES), scale, causal, dropout=drop)
        for name, x in zip(("qbar", "kbar", "vbar", "dobar"), ref):
            G.check(name, out[name], x)


@pytest.mark.parametrize("d,causal,rising", [(64, False, True), (128, True, True),
                                             (128, False, False), (256, True, True)])
def test_forward_running_maximum_raised_many_times(d, causal, rising):
    """Scores that ramp along the keys by about 85 log2 units: the forward's
    lazily raised row maximum goes up some ten times (and every tile's largest
    score sits in its second key half, so the first half takes it from the
    exchange); a falling ramp never raises it after the first tile."""
    B, H, N = 1, 2, 1000
    rng = np.random.default_rng(7 + d)
    e = np.full(d, 1.0 / np.sqrt(d))
    amp = np.sqrt(60.0 * np.sqrt(d))  # q . k / sqrt(d) spans about [0, 60]
    ramp = np.arange(N) / N if rising else 1.0 - np.arange(N) / N
    q = amp * e + 0.1 * rng.standard_normal((B, H, N, d))
    k = (amp * ramp)[:, None] * e + 0.1 * rng.standard_normal((B, H, N, d))
    v = rng.standard_normal((B, H, N, d))
    bits = {n: synth.bf16_bits(x.astype(np.float32)) for n, x in (("q", q), ("k", k), ("v", v))}
    scale = 1 / np.sqrt(d)
    o, lse = fbob.attn_fwd(G.dev(bits["q"]), G.dev(bits["k"]), G.dev(bits["v"]), scale, causal)
    assert fbob.fbob_device_status() == 0
    O, L = oracle.fwd(G.f64(bits["q"]), G.f64(bits["k"]), G.f64(bits["v"]), scale, causal)
    G.check("O", G.host(o), O)
    assert np.abs(lse.cpu().numpy() - L).max() <= 1e-3
    assert L.max() > 40.0  # the ramp reached the scores
