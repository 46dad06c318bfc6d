"""fbob_attn_bob_host: BoB with every tensor in host memory, pipelined over
chunks of heads through a device workspace.  Its results must equal those of
fbob_attn_bob on device buffers bit for bit (the same kernels run on each
head), for any chunking the workspace forces, and agree with the oracle."""
import numpy as np
import pytest

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

CASES = [  # B, H, Hkv, N, d, causal, window, segments, dropout
    (2, 4, None, 300, 128, True, None, None, None),
    (1, 6, 2, 257, 64, False, None, None, None),
    (2, 3, None, 200, 64, True, None, None, (0.2, 99)),
    (1, 4, 4, 333, 128, True, (50, -1), [0, 100, 333], None),
    (3, 2, 1, 190, 32, True, None, None, (0.1, 5)),
    (1, 4, 2, 260, 256, True, None, None, None),       # head dimension 256: four kernels
    (2, 2, None, 150, 256, False, (60, 30), None, (0.1, 8)),
]


def ids(c):
    B, H, Hkv, N, d, causal, win, seg, drop = c
    return (f"B{B}H{H}kv{Hkv}N{N}d{d}{'c' if causal else ''}"
            f"{'w' if win else ''}{'s' if seg else ''}{'p' if drop else ''}")


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


def pinned(t):
    return t.cpu().pin_memory()


def expected_chunks(BH, G, hc):
    """Chunk count the call is documented to use: chunks of at most hc heads
    in whole groups; with more than two full chunks, first and last about a
    quarter of a full chunk and the rest even."""
    U, b = BH // G, hc // G
    if U <= 2 * b:
        return -(-U // b)
    e = -(-b // 4)
    return -(-(U - 2 * e) // b) + 2


@pytest.mark.parametrize("case", CASES, ids=ids)
@pytest.mark.parametrize("chunk", ["quarter", "one_group"])
def test_host_buffers_equal_device_buffers(case, chunk):
    torch = G.torch()
    B, H, Hkv, N, d, causal, win, seg, drop = case
    bits = G.inputs(B, H, N, d, seed=B * 100 + N + d, kv_heads=Hkv)
    scale = 1 / np.sqrt(d)
    q, k, v, do, gq, gk, gv = (G.dev(bits[n]) for n in synth.NAMES)
    segs = G.dev_segments(seg)
    o, lse = fbob.attn_fwd(q, k, v, scale, causal, win, segs, drop)
    ref = fbob.attn_bob(q, k, v, o, lse, do, gq, gk, gv, scale, causal, win, segs, drop)
    torch.cuda.synchronize()
    shp = fbob.make_shape(B, H, N, d, scale, causal, win, segs, kv_heads=Hkv, dropout=drop)
    Gq = H // (Hkv or H)
    heads = B * H // 4 if chunk == "quarter" else Gq
    ws = torch.empty(fbob.fbob_attn_bob_host_workspace(shp, max(heads, 1)), dtype=torch.uint8,
                     device="cuda")
    hin = [pinned(t) for t in (q, k, v, o, lse, do, gq, gk, gv)]
    hout = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in ref]
    fbob.fbob_attn_bob_host(shp, *hin, *hout, ws)
    torch.cuda.synchronize()
    assert fbob.fbob_device_status() == 0
    units = B * H // Gq                      # key/value groups
    u = min(-(-units // 4), -(-max(heads, 1) // Gq))  # groups per full chunk the call takes
    nchunks = expected_chunks(B * H, Gq, u * Gq)
    per_chunk = 4 if d == 256 else (1 if (d <= 64 and not drop) else 2) + 1
    assert fbob.fbob_launch_count("bob_host") == nchunks * per_chunk
    for name, got, want in zip(("qbar", "kbar", "vbar", "dobar", "row_stats"), hout, ref):
        assert torch.equal(got, want.cpu()), name


def test_host_buffers_against_the_oracle():
    torch = G.torch()
    B, H, N, d, causal = 1, 3, 230, 128, True
    bits = G.inputs(B, H, N, d, seed=7)
    scale = 1 / np.sqrt(d)
    o_bits, L = G.oracle_o_l(bits, scale, causal)
    hin = [torch.from_numpy(bits[n].view(np.int16)).view(torch.bfloat16).pin_memory()
           for n in ("q", "k", "v")]
    o = torch.from_numpy(o_bits.view(np.int16)).view(torch.bfloat16).pin_memory()
    lse = torch.from_numpy(L).pin_memory()
    rest = [torch.from_numpy(bits[n].view(np.int16)).view(torch.bfloat16).pin_memory()
            for n in ("dout", "gq", "gk", "gv")]
    outs = [torch.empty(B, H, N, d, dtype=torch.bfloat16).pin_memory() for _ in range(4)]
    rs = torch.empty(3, B, H, N, dtype=torch.float32).pin_memory()
    shp = fbob.make_shape(B, H, N, d, scale, causal)
    ws = torch.empty(fbob.fbob_attn_bob_host_workspace(shp, 1), dtype=torch.uint8, device="cuda")
    fbob.fbob_attn_bob_host(shp, *hin, o, lse, *rest, *outs, rs, ws)
    torch.cuda.synchronize()
    assert fbob.fbob_device_status() == 0
    want = oracle.bob(*(G.f64(bits[n]) for n in synth.NAMES), scale, causal)
    for name, got, w in zip(("qbar", "kbar", "vbar", "dobar"), outs, want):
        G.check(name, G.host(got), w)
    for t, name in enumerate(("alpha", "E", "D")):
        G.check(name, rs[t].numpy().astype(np.float64), want[4 + t])
