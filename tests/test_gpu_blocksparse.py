"""GPU parity of block-sparse masks (App. "Extensions": each row keeps a set
of allowed columns, masked entries have zero probability, and the streamed
loops visit only the block pairs with an allowed entry).

The mask is an [nb, nb] byte array over 128 x 128 (query block, key block)
tiles, every diagonal block set.  The cases below span several blocks with
ragged tails, rows of blocks that keep only their diagonal, columns of
blocks no other query block reads, the causal mask, a window, grouped-query
heads, dropout and d = 32, 64, 128.  Every kernel runs through the C ABI and
is compared with the fp64 oracle on the same mask."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu


def random_blocks(N, density, seed, empty_rows=()):
    nb = (N + 127) // 128
    rng = np.random.default_rng(seed)
    bm = (rng.random((nb, nb)) < density).astype(np.uint8)
    for r in empty_rows:
        bm[r, :] = 0
    np.fill_diagonal(bm, 1)
    return bm


CASES = [  # B, H, N, d, causal, window, density, empty block rows, kv heads, dropout
    (1, 2, 700, 64, False, None, 0.4, (1,), None, None),
    (1, 1, 1000, 128, True, None, 0.5, (3,), None, None),
    (2, 1, 520, 128, False, None, 0.3, (0, 4), None, None),
    (1, 2, 777, 32, True, None, 0.6, (), None, None),
    (1, 2, 900, 64, True, (300, -1), 0.5, (2,), None, None),
    (1, 4, 640, 128, False, None, 0.5, (), 2, None),
    (1, 2, 600, 64, True, None, 0.5, (1,), None, (0.1, 11)),
    (1, 1, 129, 128, False, None, 0.0, (), None, None),
]

SEG_CASES = [  # B, H, N, d, causal, segments, density
    (1, 2, 700, 128, True, [0, 100, 356, 357, 700], 0.5),
    (1, 1, 600, 64, False, [0, 300, 600], 0.4),
]


def ids(c):
    B, H, N, d, causal, win, dens, er, hkv, drop = c
    return (f"B{B}H{H}N{N}d{d}{'c' if causal else ''}w{win}p{dens}"
            f"{'_gqa' if hkv else ''}{'_drop' if drop else ''}")


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


def case_inputs(c, seed):
    B, H, N, d, causal, win, dens, er, hkv, drop = c
    bits = G.inputs(B, H, N, d, seed=seed, kv_heads=hkv)
    return bits, random_blocks(N, dens, seed + 1, er)


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_forward_and_first_backward_block_sparse(case):
    B, H, N, d, causal, win, dens, er, hkv, drop = case
    bits, bm = case_inputs(case, 5 * N + d)
    scale = 1 / np.sqrt(d)
    q, k, v, do = (G.dev(bits[n]) for n in ("q", "k", "v", "dout"))
    bmk = G.dev_blocks(bm)
    o, lse = fbob.attn_fwd(q, k, v, scale, causal, win, None, drop, bmk)
    dq, dk, dv, dstat = fbob.attn_bwd(q, k, v, o, lse, do, scale, causal, win, None, drop, bmk)
    assert fbob.fbob_device_status() == 0
    X = [G.f64(bits[n]) for n in ("q", "k", "v", "dout")]
    O, L = oracle.fwd(*X[:3], scale, causal, window=win, dropout=drop, block_mask=bm)
    G.check("O", G.host(o), O)
    assert np.abs(lse.cpu().numpy() - L).max() <= 1e-3
    dQ, dK, dV, Dv = oracle.bwd(*X, scale, causal, window=win, dropout=drop, block_mask=bm)
    G.check("dQ", G.host(dq), dQ)
    G.check("dK", G.host(dk), dK)
    G.check("dV", G.host(dv), dV)
    G.check("D", dstat.cpu().numpy(), Dv)


@pytest.mark.parametrize("case", CASES, ids=ids)
def test_bob_block_sparse(case):
    B, H, N, d, causal, win, dens, er, hkv, drop = case
    bits, bm = case_inputs(case, 7 * N + d)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal, window=win, dropout=drop, block_mask=bm)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, window=win,
                     dropout=drop, block_mask=bm)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)


def test_full_block_mask_is_bitwise_no_mask():
    """All blocks set: the same tiles in the same order, so the same bits."""
    B, H, N, d = 1, 2, 600, 128
    bits = G.inputs(B, H, N, d, seed=3)
    scale = 1 / np.sqrt(d)
    nb = (N + 127) // 128
    a = G.run_bob(bits, scale, True)
    b = G.run_bob(bits, scale, True, block_mask=np.ones((nb, nb), dtype=np.uint8))
    assert a["status"] == 0 and b["status"] == 0
    for n in ("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D", "o", "lse"):
        assert np.array_equal(a[n], b[n]), n


def test_n16k_d128_causal_bsparse_rows_and_key_block():
    """The block-sparse workload at full size: sampled rows of one head, and
    one key block complete once every query block that keeps it is summed."""
    w = synth.WORKLOADS["n16k_d128_causal_bsparse"]
    bits = synth.workload_inputs(w)
    bm = synth.workload_blocks(w)
    r = G.run_bob(bits, w.scale, w.causal, block_mask=bm)
    assert r["status"] == 0
    N = w.N
    heads = [w.H + 7]
    rng = np.random.default_rng(70)
    rows = np.unique(np.concatenate([[0, 127, 128, N // 2, N - 1], rng.integers(0, N, 40)]))
    ref = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=rows, block_mask=bm)
    for name in ("qbar", "dobar", "alpha", "E", "D"):
        G.check(f"{name}[head {heads[0]}]", G.flat(r[name], heads[0], w.H)[rows], ref[0][name])
    cb = 40  # key block 40: its columns take only the query blocks that keep it
    qrows = np.concatenate([np.arange(qb * 128, min(N, qb * 128 + 128))
                            for qb in range(cb, bm.shape[0]) if bm[qb, cb]])
    c0, c1 = cb * 128, cb * 128 + 128
    blk = G.oracle_bob_heads(bits, w.scale, w.causal, heads, rows=qrows, cols=(c0, c1),
                             block_mask=bm)
    G.check("kbar[block 40]", G.flat(r["kbar"], heads[0], w.H)[c0:c1], blk[0]["kbar"])
    G.check("vbar[block 40]", G.flat(r["vbar"], heads[0], w.H)[c0:c1], blk[0]["vbar"])


@pytest.mark.parametrize("case", SEG_CASES, ids=lambda c: f"N{c[2]}d{c[3]}{'c' if c[4] else ''}s{len(c[5]) - 1}")
def test_bob_block_sparse_with_packed_sequences(case):
    """A block mask together with packed sequences: each pair must pass both."""
    B, H, N, d, causal, seg, dens = case
    bits = G.inputs(B, H, N, d, seed=9 * N + d)
    bm = random_blocks(N, dens, N + d)
    scale = 1 / np.sqrt(d)
    r = G.run_bob(bits, scale, causal, segments=seg, block_mask=bm)
    assert r["status"] == 0
    ref = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal, segments=seg,
                     block_mask=bm)
    for name, x in zip(("qbar", "kbar", "vbar", "dobar", "alpha", "E", "D"), ref):
        G.check(name, r[name], x)
    O, _ = oracle.fwd(*(G.f64(bits[n]) for n in ("q", "k", "v")), scale, causal, segments=seg,
                      block_mask=bm)
    G.check("O", r["o"], O)
