"""fp64 CPU oracle for exact attention backward-over-backward (test infrastructure).

Only tests/, ``__graft_entry__.smoke()`` and bench.py's CPU-baseline / reference
leg may import this package.  The product (paper_2609_24089_gb300) never does.

The arithmetic lives in ``fbob_oracle.c`` (plain fp64 C, OpenMP over rows); this
module only builds that file, marshals numpy float64 arrays into it and loops
over heads.  Every input is [B, H, N, d] (or [N, d] for one head) float64.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import tempfile

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fbob_oracle.c")
_LIBS = {}


def lib_path(mutant: int = 0, out_dir: str | None = None) -> str:
    name = "libfbob_oracle.so" if mutant == 0 else f"libfbob_oracle_mutant{mutant}.so"
    return os.path.join(out_dir or _HERE, name)


def build(mutant: int = 0, out_dir: str | None = None, force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP, no fast-math)."""
    path = lib_path(mutant, out_dir)
    if (not force and os.path.exists(path)
            and os.path.getmtime(path) >= os.path.getmtime(_SRC)):
        return path
    tmp = path + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-fno-fast-math", "-ffp-contract=off", f"-DFBOB_MUTANT={int(mutant)}",
           _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, path)
    return path


def _load(mutant: int = 0, out_dir: str | None = None):
    key = (mutant, out_dir)
    if key in _LIBS:
        return _LIBS[key]
    lib = ctypes.CDLL(build(mutant, out_dir))
    i64, dbl, cint = ctypes.c_int64, ctypes.c_double, ctypes.c_int
    u64, p = ctypes.c_uint64, ctypes.c_void_p
    mask = [i64, i64, dbl, cint, i64, i64, p, i64, dbl, u64, i64, p, i64]
    lib.fbob_oracle_fwd.argtypes = mask + [p, p, p, p, p, cint]
    lib.fbob_oracle_bwd.argtypes = mask + [p, p, p, p, p, p, p, p, cint]
    lib.fbob_oracle_bob.argtypes = mask + [p, p, p, p, p, p, p,
                                           p, i64, i64, i64, p, p, p, p, p, p, p, p, cint]
    for f in (lib.fbob_oracle_fwd, lib.fbob_oracle_bwd, lib.fbob_oracle_bob):
        f.restype = cint
    lib.fbob_oracle_philox.argtypes = [p, p, p]
    lib.fbob_oracle_philox.restype = None
    _LIBS[key] = lib
    return lib


def _c(x):
    return np.ascontiguousarray(x, dtype=np.float64)


def _ptr(x):
    return None if x is None else x.ctypes.data_as(ctypes.c_void_p)


def _window(window):
    """(wl, wr) of the sliding-window band i - wl <= j <= i + wr; -1 = unbounded."""
    if window is None:
        return -1, -1
    wl, wr = (int(w) for w in window)
    return wl, wr


def _segments(segments, N):
    """Segment offsets of packed variable-length sequences as an int64 array
    (seg[0] = 0, non-decreasing, seg[-1] = N), or None for one sequence."""
    if segments is None:
        return None, 0
    seg = np.ascontiguousarray(segments, dtype=np.int64)
    assert seg.ndim == 1 and seg.size >= 2 and seg[0] == 0 and seg[-1] == N
    assert np.all(np.diff(seg) >= 0)
    return seg, seg.size - 1


def _blocks(block_mask, block_size, N):
    """Block-sparse mask (App. "Extensions"): a [nb, nb] 0/1 array over square
    blocks of block_size rows and columns, nb = ceil(N / block_size), as
    uint8 bytes; None keeps every block."""
    if block_mask is None:
        return None, 0
    bs = int(block_size)
    nb = (N + bs - 1) // bs
    bm = np.ascontiguousarray(np.asarray(block_mask) != 0, dtype=np.uint8)
    assert bm.shape == (nb, nb), (bm.shape, nb)
    return bm, bs


def _dropout(dropout):
    """(p, seed) of attention dropout (App. "Extensions"); p = 0: none."""
    if dropout is None:
        return 0.0, 0
    pd, seed = dropout
    pd = float(pd)
    assert 0.0 <= pd < 1.0, pd
    return pd, int(seed) & 0xFFFFFFFFFFFFFFFF


def philox(ctr, key):
    """Philox4x32-10 of a 4-word counter under a 2-word key (four uint32)."""
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    _load().fbob_oracle_philox(_ptr(c), _ptr(k), _ptr(out))
    return out


def _group(H, Hkv):
    """Query heads per key/value head (grouped-query attention: query head h
    reads key/value head h // G)."""
    assert Hkv >= 1 and H % Hkv == 0, (H, Hkv)
    return H // Hkv


def _heads(x):
    x = np.asarray(x)
    if x.ndim == 2:
        return x[None, None]
    return x


def fwd(q, k, v, scale, causal, nthreads=0, window=None, segments=None, dropout=None,
        block_mask=None, block_size=128):
    """Forward attention (eq. 1).  Returns O [B,H,N,d] and natural-log L [B,H,N].
    window: (wl, wr) sliding-window band (default: none); segments: offsets of
    packed sequences (default: one sequence); dropout: (p, seed), the keep
    mask of query head b*H + h drawn from Philox with that head index;
    block_mask: [nb, nb] 0/1 blocks of block_size (default: none)."""
    wl, wr = _window(window)
    pd, seed = _dropout(dropout)
    q, k, v = (_c(_heads(t)) for t in (q, k, v))
    B, H, N, d = q.shape
    G = _group(H, k.shape[1])
    seg, nseg = _segments(segments, N)
    bm, bs = _blocks(block_mask, block_size, N)
    lib = _load()
    O = np.zeros_like(q)
    L = np.zeros((B, H, N))
    for b in range(B):
        for h in range(H):
            o_ = np.zeros((N, d)); l_ = np.zeros(N)
            hk = h // G
            rc = lib.fbob_oracle_fwd(N, d, float(scale), int(bool(causal)), wl, wr,
                                     _ptr(seg), nseg, pd, seed, b * H + h, _ptr(bm), bs,
                                     _ptr(_c(q[b, h])), _ptr(_c(k[b, hk])), _ptr(_c(v[b, hk])),
                                     _ptr(o_), _ptr(l_), int(nthreads))
            assert rc == 0, rc
            O[b, h], L[b, h] = o_, l_
    return O, L


def bwd(q, k, v, dout, scale, causal, nthreads=0, window=None, segments=None, dropout=None,
        block_mask=None, block_size=128):
    """First backward (eqs. 2-3).  Returns dQ [B,H,N,d], dK, dV [B,Hkv,N,d] and
    D [B,H,N]; with grouped-query attention (k, v with Hkv < H heads) dK and dV
    of a key/value head are the sums over its query heads.  dropout and
    block_mask as in fwd."""
    wl, wr = _window(window)
    pd, seed = _dropout(dropout)
    q, k, v, dout = (_c(_heads(t)) for t in (q, k, v, dout))
    B, H, N, d = q.shape
    G = _group(H, k.shape[1])
    seg, nseg = _segments(segments, N)
    bm, bs = _blocks(block_mask, block_size, N)
    lib = _load()
    outs = [np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)]
    D = np.zeros((B, H, N))
    for b in range(B):
        for h in range(H):
            hk = h // G
            dq, dk, dv, dd = np.zeros((N, d)), np.zeros((N, d)), np.zeros((N, d)), np.zeros(N)
            rc = lib.fbob_oracle_bwd(N, d, float(scale), int(bool(causal)), wl, wr,
                                     _ptr(seg), nseg, pd, seed, b * H + h, _ptr(bm), bs,
                                     _ptr(_c(q[b, h])), _ptr(_c(k[b, hk])), _ptr(_c(v[b, hk])),
                                     _ptr(_c(dout[b, h])), _ptr(dq), _ptr(dk), _ptr(dv),
                                     _ptr(dd), int(nthreads))
            assert rc == 0, rc
            outs[0][b, h], D[b, h] = dq, dd
            outs[1][b, hk] += dk
            outs[2][b, hk] += dv
    return outs[0], outs[1], outs[2], D


def bob_head(q, k, v, dout, gq, gk, gv, scale, causal, rows=None, cols=None,
             nthreads=0, mutant=0, mutant_dir=None, window=None, segments=None,
             dropout=None, head=0, row_outputs=True, block_mask=None, block_size=128):
    """Backward-over-backward of one head ([N, d] float64 arrays).

    rows: query rows whose row-owned outputs are wanted (default: all).
    cols: (c0, c1) key columns receiving the listed rows' contributions to
          Ktil, Vtil (default: all columns when rows is all rows, else none).
    Returns a dict with qbar, dobar, alpha, E, D, L (indexed like rows) and
    kbar, vbar ((c1-c0) x d; complete only if every contributing row is listed).
    window: (wl, wr) sliding-window band i - wl <= j <= i + wr (-1 = unbounded).
    segments: offsets of packed sequences; a row sees only its own sequence.
    dropout: (p, seed); head: the flat query-head index b*H + h that keys the
    head's dropout mask.
    block_mask: [nb, nb] 0/1 array over square blocks of block_size rows and
    columns (nb = ceil(N / block_size)); a pair is kept only if its block is.
    row_outputs: False skips the listed rows' qbar and dobar (left as zeros),
    for callers that want only the column block (it halves the work per row).
    """
    wl, wr = _window(window)
    pd, seed = _dropout(dropout)
    q, k, v, dout, gq, gk, gv = (_c(t) for t in (q, k, v, dout, gq, gk, gv))
    N, d = q.shape
    seg, nseg = _segments(segments, N)
    bm, bs = _blocks(block_mask, block_size, N)
    if rows is None:
        rows = np.arange(N, dtype=np.int64)
        if cols is None:
            cols = (0, N)
    rows = np.ascontiguousarray(rows, dtype=np.int64)
    if cols is None:
        cols = (0, 0)
    c0, c1 = int(cols[0]), int(cols[1])
    nr = rows.shape[0]
    nc = max(c1 - c0, 0)
    res = {
        "qbar": np.zeros((nr, d)), "dobar": np.zeros((nr, d)),
        "alpha": np.zeros(nr), "E": np.zeros(nr), "D": np.zeros(nr), "L": np.zeros(nr),
        "kbar": np.zeros((nc, d)), "vbar": np.zeros((nc, d)),
    }
    lib = _load(mutant, mutant_dir)
    rc = lib.fbob_oracle_bob(N, d, float(scale), int(bool(causal)), wl, wr, _ptr(seg), nseg,
                             pd, seed, int(head), _ptr(bm), bs,
                             _ptr(q), _ptr(k), _ptr(v), _ptr(dout), _ptr(gq), _ptr(gk), _ptr(gv),
                             _ptr(rows), nr, c0, c1,
                             _ptr(res["qbar"] if row_outputs else None),
                             _ptr(res["dobar"] if row_outputs else None), _ptr(res["alpha"]),
                             _ptr(res["E"]), _ptr(res["D"]), _ptr(res["L"]),
                             _ptr(res["kbar"]), _ptr(res["vbar"]), int(nthreads))
    assert rc == 0, rc
    return res


def bob(q, k, v, dout, gq, gk, gv, scale, causal, nthreads=0, mutant=0, mutant_dir=None,
        window=None, segments=None, dropout=None, block_mask=None, block_size=128):
    """Full backward-over-backward on [B,H,N,d] (or [N,d]) float64 arrays.

    Returns (qbar, kbar, vbar, dobar, alpha, E, D) with the input's batch shape.
    Grouped-query attention: k, v, gk, gv may have Hkv < H heads (query head h
    reads head h // (H / Hkv)).  Phi then splits into one term per query head,
    each using its key/value head's tensors, so kbar and vbar of a key/value
    head are the sums of the per-query-head results over its group.
    """
    ts = [_c(_heads(t)) for t in (q, k, v, dout, gq, gk, gv)]
    B, H, N, d = ts[0].shape
    Hkv = ts[1].shape[1]
    G = _group(H, Hkv)
    out = {n: np.zeros((B, H, N, d)) for n in ("qbar", "dobar")}
    for n in ("kbar", "vbar"):
        out[n] = np.zeros((B, Hkv, N, d))
    for n in ("alpha", "E", "D"):
        out[n] = np.zeros((B, H, N))
    kv_side = (1, 2, 5, 6)  # k, v, gk, gv
    for b in range(B):
        for h in range(H):
            args = [t[b, h // G] if i in kv_side else t[b, h] for i, t in enumerate(ts)]
            r = bob_head(*args, scale, causal, nthreads=nthreads,
                         mutant=mutant, mutant_dir=mutant_dir, window=window,
                         segments=segments, dropout=dropout, head=b * H + h,
                         block_mask=block_mask, block_size=block_size)
            for n in ("qbar", "dobar", "alpha", "E", "D"):
                out[n][b, h] = r[n]
            out["kbar"][b, h // G] += r["kbar"]
            out["vbar"][b, h // G] += r["vbar"]
    return (out["qbar"], out["kbar"], out["vbar"], out["dobar"],
            out["alpha"], out["E"], out["D"])


def mutant_build_dir():
    d = os.path.join(tempfile.gettempdir(), "fbob_oracle_mutants")
    os.makedirs(d, exist_ok=True)
    return d
