"""Parity on the five synthetic workloads, run on the GPU at full size in the
launch configuration the benchmark times.

  n128_d64               full oracle; O and L from the oracle's forward
  n4k_d64                full oracle on a seeded set of heads (all heads: FBOB_SLOW=1)
  n16k_d128_causal       full oracle on two seeded heads
  n64k_d128_causal_peaky oracle on sampled rows (row-owned outputs) and on the
                         causal tail: key columns >= N - 256 are complete once
                         rows >= N - 256 are summed
  n256k_d64              oracle on sampled rows; one 128-key block of Ktil, Vtil
                         (keys 199936..200063 of head 1) against stored oracle
                         values; every head through identities that hold at any
                         size (column sums vanish, Euler identities)
  n16k_d128_causal_swa4k sliding window w = N/4: oracle on sampled rows and on a
                         256-key block, complete once the rows whose band holds
                         it (keys j .. j + 4095) are summed
  n16k_d128_causal_varlen / _gqa4 / _drop10
                         packed sequences, grouped-query heads, dropout: sampled
                         rows plus one whole sequence or the causal tail
  n4k_d{32,64,128}_causal_b4h12
                         the head-dimension sweep's shape: two full heads each
"""
import os

import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G
from tests.golden import make_n256k_d64_key_block as key_block

pytestmark = pytest.mark.gpu

ROWS_OUT = ("qbar", "dobar", "alpha", "E", "D")


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


def sample_rows(N, seed, n=40):
    rng = np.random.default_rng(seed)
    fixed = [0, 1, 2, 63, 64, 127, 128, 129, N // 2, N - 129, N - 128, N - 2, N - 1]
    rows = set(r for r in fixed if 0 <= r < N)
    rows.update(rng.integers(0, N, n).tolist())
    return np.array(sorted(rows), dtype=np.int64)


def check_rows(r, refs, heads, H, rows):
    for hh, ref in zip(heads, refs):
        for name in ROWS_OUT:
            got = G.flat(r[name], hh, H)[rows]
            G.check(f"{name}[head {hh}]", got, ref[name])


def test_n128_d64_full_with_oracle_forward():
    w = synth.WORKLOADS["n128_d64"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal, o_l=G.oracle_o_l(bits, w.scale, w.causal))
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), w.scale, w.causal)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)


def test_n4k_d64_heads():
    w = synth.WORKLOADS["n4k_d64"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal)
    assert r["status"] == 0
    BH = w.B * w.H
    heads = list(range(BH)) if os.environ.get("FBOB_SLOW") == "1" else [0, 21, 42, 63]
    refs = G.oracle_bob_heads(bits, w.scale, w.causal, heads)
    for hh, ref in zip(heads, refs):
        for name in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"):
            G.check(f"{name}[head {hh}]", G.flat(r[name], hh, w.H), ref[name])


def test_n16k_d128_causal_two_heads():
    w = synth.WORKLOADS["n16k_d128_causal"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal)
    assert r["status"] == 0
    heads = [0, w.B * w.H - 1]
    refs = G.oracle_bob_heads(bits, w.scale, w.causal, heads)
    for hh, ref in zip(heads, refs):
        for name in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"):
            G.check(f"{name}[head {hh}]", G.flat(r[name], hh, w.H), ref[name])


def test_n64k_d128_causal_peaky_rows_and_tail():
    w = synth.WORKLOADS["n64k_d128_causal_peaky"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal)
    assert r["status"] == 0
    N = w.N
    heads = [3]
    rows = sample_rows(N, 64)
    check_rows(r, G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=rows), heads, w.H, rows)
    t0 = N - 256
    tail = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=np.arange(t0, N), cols=(t0, N))
    for hh, ref in zip(heads, tail):
        G.check("kbar[tail]", G.flat(r["kbar"], hh, w.H)[t0:], ref["kbar"])
        G.check("vbar[tail]", G.flat(r["vbar"], hh, w.H)[t0:], ref["vbar"])


def test_n256k_d64_rows_and_identities():
    w = synth.WORKLOADS["n256k_d64"]
    bits = synth.workload_inputs(w)
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    o, lse = fbob.attn_fwd(q, k, v, w.scale, w.causal)
    qb, kb, vb, dob, rs = fbob.attn_bob(q, k, v, o, lse, do, gq, gk, gv, w.scale, w.causal)
    dq, dk, dv, _ = fbob.attn_bwd(q, k, v, o, lse, do, w.scale, w.causal)
    assert fbob.fbob_device_status() == 0
    H = w.H
    heads = [1]
    rows = sample_rows(w.N, 256)
    r = {"qbar": G.host(qb), "dobar": G.host(dob), "alpha": rs[0].cpu().numpy(),
         "E": rs[1].cpu().numpy(), "D": rs[2].cpu().numpy()}
    check_rows(r, G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=rows), heads, H, rows)
    # one complete 128-key block of Ktil and Vtil past 2^17, element by element
    # against the stored fp64 oracle values (all 262,144 rows of head 1 summed;
    # tests/golden/make_n256k_d64_key_block.py wrote them)
    kref, vref = key_block.load()
    c0, c1 = key_block.C0, key_block.C1
    b, h = divmod(key_block.HEAD, H)
    G.check("kbar[head 1, keys 199936..200063]", G.host(kb[b, h, c0:c1]), kref)
    G.check("vbar[head 1, keys 199936..200063]", G.host(vb[b, h, c0:c1]), vref)
    # identities, per head, in fp64 over the bf16 outputs
    for hh in range(w.B * H):
        b, h = divmod(hh, H)
        X = {n: G.f64(bits[n][b, h]) for n in synth.NAMES}
        Kt, Vt = G.host(kb[b, h]), G.host(vb[b, h])
        Qt, dOt = G.host(qb[b, h]), G.host(dob[b, h])
        dQ, dK, dV = G.host(dq[b, h]), G.host(dk[b, h]), G.host(dv[b, h])
        for name, M in (("kbar", Kt), ("vbar", Vt)):   # shift invariance of Phi
            colsum = np.abs(M.sum(0))
            assert np.all(colsum <= 3e-2 * np.linalg.norm(M, axis=0)), name
        a = float((dQ * X["gq"]).sum())
        bk = float((dK * X["gk"]).sum())
        c = float((dV * X["gv"]).sum())
        phi = a + bk + c
        # Euler identities (degree 1 in dO; V -> sV; Q -> sQ, K -> K/s)
        sc = abs(a) + abs(bk) + abs(c)
        assert abs(float((dOt * X["dout"]).sum()) - phi) <= 2e-2 * sc
        assert abs(float((Vt * X["v"]).sum()) - (a + bk)) <= 2e-2 * (abs(a) + abs(bk))
        lhs = float((Qt * X["q"]).sum()) - float((Kt * X["k"]).sum())
        assert abs(lhs - (bk - a)) <= 2e-2 * (abs(a) + abs(bk))


def test_n16k_d128_causal_swa4k_rows_and_key_block():
    w = synth.WORKLOADS["n16k_d128_causal_swa4k"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal, window=w.window)
    assert r["status"] == 0
    N, wl = w.N, w.window[0]
    heads = [5]
    rows = sample_rows(N, 65)
    check_rows(r, G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=rows, window=w.window),
               heads, w.H, rows)
    c0, c1 = N // 2, N // 2 + 256
    blk = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=np.arange(c0, min(N, c1 + wl)),
                             cols=(c0, c1), window=w.window)
    for hh, ref in zip(heads, blk):
        G.check("kbar[block]", G.flat(r["kbar"], hh, w.H)[c0:c1], ref["kbar"])
        G.check("vbar[block]", G.flat(r["vbar"], hh, w.H)[c0:c1], ref["vbar"])


def test_n16k_d128_causal_varlen_rows_and_sequence():
    """Packed sequences at full size: sampled rows, and the key columns of one
    whole sequence (complete once that sequence's rows are summed)."""
    w = synth.WORKLOADS["n16k_d128_causal_varlen"]
    seg = list(w.segments)
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal, segments=seg)
    assert r["status"] == 0
    heads = [9]
    rows = sample_rows(w.N, 66)
    check_rows(r, G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=rows, segments=seg),
               heads, w.H, rows)
    a, b = seg[5], seg[6]
    blk = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=np.arange(a, b), cols=(a, b),
                             segments=seg)
    for hh, ref in zip(heads, blk):
        G.check("kbar[sequence]", G.flat(r["kbar"], hh, w.H)[a:b], ref["kbar"])
        G.check("vbar[sequence]", G.flat(r["vbar"], hh, w.H)[a:b], ref["vbar"])


def test_n16k_d128_causal_gqa4_rows_and_tail():
    """Grouped-query workload at full size: sampled rows of one query head,
    and the causal tail of one key/value head (its key columns >= N - 256 are
    complete once rows >= N - 256 of its four query heads are summed)."""
    w = synth.WORKLOADS["n16k_d128_causal_gqa4"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal)
    assert r["status"] == 0
    N, H, Hkv = w.N, w.H, w.kv_heads
    Gq = H // Hkv
    hq = 6  # query head 6 of batch 0 reads key/value head 1
    rows = sample_rows(N, 67)
    X = {n: G.f64(bits[n][0, hq // Gq if n in ("k", "v", "gk", "gv") else hq])
         for n in synth.NAMES}
    ref = oracle.bob_head(*(X[n] for n in synth.NAMES), w.scale, w.causal, rows=rows)
    for name in ROWS_OUT:
        G.check(f"{name}[head {hq}]", r[name][0, hq][rows], ref[name])
    t0 = N - 256
    kb = np.zeros((256, w.d))
    vb = np.zeros((256, w.d))
    for g in range(Gq):
        h = 1 * Gq + g
        Y = {n: G.f64(bits[n][0, 1 if n in ("k", "v", "gk", "gv") else h]) for n in synth.NAMES}
        t = oracle.bob_head(*(Y[n] for n in synth.NAMES), w.scale, w.causal,
                            rows=np.arange(t0, N), cols=(t0, N))
        kb += t["kbar"]
        vb += t["vbar"]
    G.check("kbar[kv head 1, tail]", r["kbar"][0, 1][t0:], kb)
    G.check("vbar[kv head 1, tail]", r["vbar"][0, 1][t0:], vb)


def test_n16k_d128_causal_drop10_rows_and_tail():
    """Dropout workload (p = 0.1) at full size: sampled rows of one head and
    its causal tail, against the oracle with the same keep mask."""
    w = synth.WORKLOADS["n16k_d128_causal_drop10"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal, dropout=w.dropout)
    assert r["status"] == 0
    N = w.N
    heads = [w.H + 3]  # batch entry 1, head 3
    rows = sample_rows(N, 68)
    check_rows(r, G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=rows,
                                     dropout=w.dropout), heads, w.H, rows)
    t0 = N - 256
    tail = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=np.arange(t0, N), cols=(t0, N),
                              dropout=w.dropout)
    for hh, ref in zip(heads, tail):
        G.check("kbar[tail]", G.flat(r["kbar"], hh, w.H)[t0:], ref["kbar"])
        G.check("vbar[tail]", G.flat(r["vbar"], hh, w.H)[t0:], ref["vbar"])


@pytest.mark.parametrize("d", [32, 64, 128])
def test_n4k_causal_b4h12_head_dim_sweep_two_heads(d):
    """The head-dimension sweep's shape (B 4, H 12, N 4096, causal): two full heads."""
    w = synth.WORKLOADS[f"n4k_d{d}_causal_b4h12"]
    bits = synth.workload_inputs(w)
    r = G.run_bob(bits, w.scale, w.causal)
    assert r["status"] == 0
    heads = [1, w.B * w.H - 2]
    refs = G.oracle_bob_heads(bits, w.scale, w.causal, heads)
    for hh, ref in zip(heads, refs):
        for name in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"):
            G.check(f"{name}[head {hh}]", G.flat(r[name], hh, w.H), ref[name])
