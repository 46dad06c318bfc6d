"""GPU parity of Pass 1 in one sweep with the affine fusion of Prop. 3.1
(eq. 8) at every head dimension, through fbob_attn_bob_pass1_fused.

At d = 128 the four Pass-1 accumulators (B, dOtil0, G, Omega) are split by
output column over two CTAs per row block; the row scalars alpha, E, D come
out of the same sweep.  Each case runs the fused Pass 1 and then Pass 2 on
its row statistics, and compares every output with the fp64 oracle: ragged
N, both masks, a window, packed sequences, grouped-query heads, and the
full-size n16k_d128_causal (two whole heads) and n64k_d128_causal_peaky
(sampled rows and the causal tail) workloads."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

CASES = [  # B, H, N, d, causal, window, segments, kv heads
    (1, 2, 300, 128, True, None, None, None),
    (2, 1, 257, 128, False, None, None, None),
    (1, 1, 129, 128, True, None, None, None),
    (1, 2, 3, 128, False, None, None, None),
    (1, 1, 777, 128, True, (200, -1), None, None),
    (1, 2, 600, 128, True, None, [0, 100, 350, 351, 600], None),
    (1, 4, 400, 128, False, None, None, 2),
    (1, 2, 520, 64, True, None, None, None),
    (1, 2, 301, 32, False, None, None, None),
]


def ids(c):
    B, H, N, d, causal, win, seg, hkv = c
    return (f"B{B}H{H}N{N}d{d}{'c' if causal else ''}w{win}"
            f"{'s' if seg else ''}{'_gqa' if hkv else ''}")


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


def run_fused(bits, scale, causal, window=None, segments=None, o_l=None):
    """Forward, then the fused Pass 1 and Pass 2 through the C ABI."""
    t = G.torch()
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    seg = G.dev_segments(segments)
    if o_l is None:
        o, lse = fbob.attn_fwd(q, k, v, scale, causal, window, seg)
    else:
        o, lse = G.dev(o_l[0]), G.dev_f32(o_l[1])
    B, H, N, d = q.shape
    shp = fbob.make_shape(B, H, N, d, scale, causal, window, seg, kv_heads=k.shape[1])
    qb, dob = t.empty_like(q), t.empty_like(q)
    kb, vb = t.empty_like(k), t.empty_like(v)
    rs = t.empty((3, B, H, N), dtype=t.float32, device="cuda")
    fbob.fbob_attn_bob_pass1_fused(shp, q, k, v, o, lse, do, gq, gk, gv, qb, dob, rs)
    assert fbob.fbob_launch_count("bob_pass1_fused") == (1 if N else 0)
    fbob.fbob_attn_bob_pass2(shp, q, k, v, lse, do, gq, gk, gv, rs, kb, vb)
    status = fbob.fbob_device_status()
    t.cuda.synchronize()
    return {"qbar": G.host(qb), "kbar": G.host(kb), "vbar": G.host(vb), "dobar": G.host(dob),
            "alpha": rs[0].cpu().numpy().astype(np.float64),
            "E": rs[1].cpu().numpy().astype(np.float64),
            "D": rs[2].cpu().numpy().astype(np.float64), "status": status}


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_fused_pass1_and_pass2(case):
    B, H, N, d, causal, win, seg, hkv = case
    bits = G.inputs(B, H, N, d, seed=11 * N + d, kv_heads=hkv)
    scale = 1 / np.sqrt(d)
    r = run_fused(bits, scale, causal, win, seg)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, window=win,
                     segments=seg)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)


def test_fused_runs_are_bitwise_identical():
    bits = G.inputs(1, 2, 700, 128, seed=5)
    a = run_fused(bits, 1 / np.sqrt(128), True)
    b = run_fused(bits, 1 / np.sqrt(128), True)
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"):
        assert np.array_equal(a[n], b[n]), n


def test_fused_rejects_dropout():
    t = G.torch()
    x = t.zeros((1, 1, 128, 128), dtype=t.bfloat16, device="cuda")
    lse = t.zeros((1, 1, 128), dtype=t.float32, device="cuda")
    rs = t.empty((3, 1, 1, 128), dtype=t.float32, device="cuda")
    shp = fbob.make_shape(1, 1, 128, 128, 0.088, True, dropout=(0.1, 1))
    with pytest.raises(fbob.FbobError) as e:
        fbob.fbob_attn_bob_pass1_fused(shp, x, x, x, x, lse, x, x, x, x,
                                       t.empty_like(x), t.empty_like(x), rs)
    assert e.value.status == fbob.STATUS_CODES["FBOB_ERR_UNSUPPORTED"]


def test_n16k_d128_causal_fused_two_heads():
    w = synth.WORKLOADS["n16k_d128_causal"]
    bits = synth.workload_inputs(w)
    r = run_fused(bits, w.scale, w.causal)
    assert r["status"] == 0
    heads = [1, w.B * w.H - 2]
    refs = G.oracle_bob_heads(bits, w.scale, w.causal, heads)
    for hh, ref in zip(heads, refs):
        for name in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"):
            G.check(f"{name}[head {hh}]", G.flat(r[name], hh, w.H), ref[name])


def test_n64k_d128_causal_peaky_fused_rows_and_tail():
    w = synth.WORKLOADS["n64k_d128_causal_peaky"]
    bits = synth.workload_inputs(w)
    r = run_fused(bits, w.scale, w.causal)
    assert r["status"] == 0
    N = w.N
    heads = [5]
    rng = np.random.default_rng(64)
    rows = np.unique(np.concatenate([[0, 1, 127, 128, N // 2, N - 1], rng.integers(0, N, 40)]))
    ref = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=rows)
    for name in ("qbar", "dobar", "alpha", "E", "D"):
        G.check(f"{name}[head 5]", G.flat(r[name], 5, w.H)[rows], ref[0][name])
    t0 = N - 256
    tail = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=np.arange(t0, N), cols=(t0, N))
    G.check("kbar[tail]", G.flat(r["kbar"], 5, w.H)[t0:], tail[0]["kbar"])
    G.check("vbar[tail]", G.flat(r["vbar"], 5, w.H)[t0:], tail[0]["vbar"])
