"""fbob_attn_bob_host_noalloc: the host-buffer BoB staged in the library's
fixed device array instead of a caller workspace.  Two calls in a row (with
different inputs, so the second finds the first one's data in the array)
must each equal fbob_attn_bob_host bit for bit.  Named to be collected last;
it also passes alone."""
import numpy as np
import pytest

import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth
from tests import gpu_util as G

pytestmark = pytest.mark.gpu

CASES = [  # B, H, Hkv, N, d, causal, dropout
    (2, 3, None, 8192, 128, True, None),     # 2 heads per chunk: 3 chunks
    (1, 4, 2, 3000, 64, False, (0.15, 11)),  # grouped-query heads and dropout: one chunk
]


@pytest.fixture(scope="module", autouse=True)
def built():
    fbob.build()
    fbob.load()


def host_inputs(B, H, Hkv, N, d, causal, drop, seed):
    torch = G.torch()
    bits = G.inputs(B, H, N, d, seed=seed, kv_heads=Hkv)
    scale = 1 / np.sqrt(d)
    q, k, v = (G.dev(bits[n]) for n in ("q", "k", "v"))
    o, lse = fbob.attn_fwd(q, k, v, scale, causal, None, None, drop)
    torch.cuda.synchronize()
    dev = {n: G.dev(bits[n]) for n in synth.NAMES}
    order = [dev["q"], dev["k"], dev["v"], o, lse, dev["dout"], dev["gq"], dev["gk"], dev["gv"]]
    return [t.cpu().pin_memory() for t in order], scale


@pytest.mark.parametrize("case", CASES, ids=lambda c: "B{}H{}kv{}N{}d{}".format(*c[:5]))
def test_two_calls_in_a_row_equal_the_workspace_call(case):
    torch = G.torch()
    B, H, Hkv, N, d, causal, drop = case
    shp = None
    for call in range(2):
        hin, scale = host_inputs(B, H, Hkv, N, d, causal, drop, seed=31 + 17 * call)
        shp = fbob.make_shape(B, H, N, d, scale, causal, kv_heads=Hkv, dropout=drop)
        shapes = [hin[0].shape, hin[1].shape, hin[2].shape, hin[0].shape]
        outs_a = [torch.empty(sh, dtype=torch.bfloat16).pin_memory() for sh in shapes]
        outs_b = [torch.empty(sh, dtype=torch.bfloat16).pin_memory() for sh in shapes]
        rs_a = torch.empty(3, B, H, N, dtype=torch.float32).pin_memory()
        rs_b = torch.empty(3, B, H, N, dtype=torch.float32).pin_memory()
        fbob.fbob_attn_bob_host_noalloc(shp, *hin, *outs_a, rs_a)
        torch.cuda.synchronize()
        assert fbob.fbob_device_status() == 0
        assert fbob.fbob_launch_count("bob_host_noalloc") > 0
        ws = torch.empty(fbob.fbob_attn_bob_host_workspace(shp, B * H), dtype=torch.uint8,
                         device="cuda")
        fbob.fbob_attn_bob_host(shp, *hin, *outs_b, rs_b, ws)
        torch.cuda.synchronize()
        assert fbob.fbob_device_status() == 0
        for name, a, b in zip(("qbar", "kbar", "vbar", "dobar", "row_stats"),
                              (*outs_a, rs_a), (*outs_b, rs_b)):
            assert torch.equal(a, b), (call, name)


def test_too_large_a_problem_is_refused():
    torch = G.torch()
    # one head of N = 65536 at d = 128 needs about 192 MiB of staging
    x = torch.zeros(1, 1, 65536, 128, dtype=torch.bfloat16).pin_memory()
    lse = torch.zeros(1, 1, 65536, dtype=torch.float32).pin_memory()
    outs = [torch.empty_like(x) for _ in range(4)]
    rs = torch.empty(3, 1, 1, 65536, dtype=torch.float32).pin_memory()
    shp = fbob.make_shape(1, 1, 65536, 128, 0.088, True)
    with pytest.raises(fbob.FbobError) as err:
        fbob.fbob_attn_bob_host_noalloc(shp, x, torch.zeros_like(x), torch.zeros_like(x),
                                        torch.zeros_like(x), lse, torch.zeros_like(x),
                                        torch.zeros_like(x), torch.zeros_like(x),
                                        torch.zeros_like(x), *outs, rs)
    assert err.value.status == fbob.STATUS_CODES["FBOB_ERR_SCRATCH_LIMIT"]
