"""Helpers shared by the GPU parity tests: device upload of the seeded bf16
inputs, the CUDA pipeline (forward -> backward-over-backward) through the C
ABI, and the tolerance check against the fp64 oracle.

Tolerance (per output tensor): relative Frobenius error <= 1e-2 and
max |got - ref| <= 5e-2 * max |ref|.
"""
from __future__ import annotations

import os

import numpy as np

import oracle
import paper_2609_24089_gb300 as fbob
from paper_2609_24089_gb300 import synth

REL_FRO = 1e-2
MAX_ABS = 5e-2

# every check appends (test id, tensor, rel_fro, max_abs/max|ref|); the session
# hook in conftest.py writes them out when FBOB_PARITY_REPORT names a file
RECORD = []


def torch():
    import torch as _t
    return _t


def dev(bits: np.ndarray):
    t = torch()
    return t.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(t.bfloat16).cuda()


def dev_f32(x: np.ndarray):
    t = torch()
    return t.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()


def host(t) -> np.ndarray:
    return t.float().cpu().numpy().astype(np.float64)


def check(name, got, ref, rel=REL_FRO, mx=MAX_ABS, zero_atol=1e-6):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{name}: non-finite values"
    scale = np.abs(ref).max() if ref.size else 0.0
    if scale == 0.0:
        assert np.abs(got).max(initial=0.0) <= zero_atol, f"{name}: expected zeros"
        return 0.0, 0.0
    r = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    m = np.abs(got - ref).max() / scale
    RECORD.append((os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0], name, float(r), float(m)))
    assert r <= rel and m <= mx, f"{name}: rel_fro={r:.3e} (<= {rel}) max_abs/max|ref|={m:.3e} (<= {mx})"
    return r, m


def inputs(B, H, N, d, seed, sigma=(1.0,) * 7, heads=None, kv_heads=None):
    """Seeded bf16 inputs; with kv_heads, k, v, gk, gv keep only the first
    kv_heads heads (grouped-query attention)."""
    bits = synth.make_inputs(B, H, N, d, seed, sigma, heads=heads)
    if kv_heads is not None:
        for n in ("k", "v", "gk", "gv"):
            bits[n] = np.ascontiguousarray(bits[n][:, :kv_heads])
    return bits


def f64(bits):
    return synth.to_f64(bits)


def oracle_o_l(bits, scale, causal, window=None, segments=None, dropout=None, block_mask=None):
    """O rounded to bf16 and L rounded to fp32, from the oracle's forward."""
    O, L = oracle.fwd(f64(bits["q"]), f64(bits["k"]), f64(bits["v"]), scale, causal,
                      window=window, segments=segments, dropout=dropout, block_mask=block_mask)
    return synth.bf16_bits(O.astype(np.float32)), L.astype(np.float32)


def dev_segments(segments):
    """Packed-sequence offsets as the int32 CUDA tensor the library reads."""
    if segments is None:
        return None
    t = torch()
    return t.tensor(np.asarray(segments, dtype=np.int32), device="cuda")


def dev_blocks(block_mask):
    """Block mask as the uint8 CUDA tensor the library reads."""
    if block_mask is None:
        return None
    t = torch()
    return t.tensor(np.asarray(block_mask, dtype=np.uint8), device="cuda")


def run_bob(bits, scale, causal, o_l=None, window=None, segments=None, dropout=None,
            block_mask=None):
    """Upload, (forward unless o_l is given), then backward-over-backward.
    Returns dict of host float64 arrays and the device status."""
    t = torch()
    q, k, v, do, gq, gk, gv = (dev(bits[n]) for n in synth.NAMES)
    seg = dev_segments(segments)
    bmk = dev_blocks(block_mask)
    if o_l is None:
        o, lse = fbob.attn_fwd(q, k, v, scale, causal, window, seg, dropout, bmk)
    else:
        o, lse = dev(o_l[0]), dev_f32(o_l[1])
    qb, kb, vb, dob, rs = fbob.attn_bob(q, k, v, o, lse, do, gq, gk, gv, scale, causal, window,
                                        seg, dropout, bmk)
    status = fbob.fbob_device_status()
    t.cuda.synchronize()
    return {"qbar": host(qb), "kbar": host(kb), "vbar": host(vb), "dobar": host(dob),
            "alpha": rs[0].cpu().numpy().astype(np.float64),
            "E": rs[1].cpu().numpy().astype(np.float64),
            "D": rs[2].cpu().numpy().astype(np.float64),
            "o": host(o), "lse": lse.cpu().numpy().astype(np.float64), "status": status}


def oracle_bob_heads(bits, scale, causal, heads, rows=None, cols=None, window=None,
                     segments=None, dropout=None, block_mask=None):
    """Oracle on selected flat heads of a [B,H,N,d] bit tensor set (the
    key/value side of a grouped-query set is read from head h // G)."""
    B, H, N, d = bits["q"].shape
    G = H // bits["k"].shape[1]
    out = []
    for hh in heads:
        b, h = divmod(hh, H)
        X = [f64(bits[n][b, h // G if n in ("k", "v", "gk", "gv") else h]) for n in synth.NAMES]
        out.append(oracle.bob_head(*X, scale, causal, rows=rows, cols=cols, window=window,
                                   segments=segments, dropout=dropout, head=hh,
                                   block_mask=block_mask))
    return out


def flat(x, hh, H):
    b, h = divmod(hh, H)
    return x[b, h]
