"""Python binding of libfbob (include/fbob.h): exact backward-over-backward of
softmax attention on GB300.

The functions named like the C entry points (``fbob_attn_fwd``, ...) only
marshal torch tensors into device pointers and the current CUDA stream; every
step of the computation runs in the library's kernels.  There is no fallback:
if libfbob.so is missing or a call fails, an exception is raised.
The ``attn_*`` helpers additionally allocate the outputs with torch.
"""
from __future__ import annotations

import ctypes
import os
import re

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfbob.so")
HEADER = os.path.join(os.path.dirname(_HERE), "include", "fbob.h")

FBOB_OK = 0
STATUS = {0: "FBOB_OK", 1: "FBOB_ERR_INVALID_ARGUMENT", 2: "FBOB_ERR_UNSUPPORTED",
          3: "FBOB_ERR_CUDA", 4: "FBOB_ERR_DEVICE_TIMEOUT", 5: "FBOB_ERR_DEVICE_FAULT",
          6: "FBOB_ERR_SCRATCH_LIMIT"}
STATUS_CODES = {v: k for k, v in STATUS.items()}


class FbobError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {STATUS.get(status, status)}")
        self.status = status


class fbob_shape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int64), ("H", ctypes.c_int64), ("N", ctypes.c_int64),
                ("d", ctypes.c_int64), ("scale", ctypes.c_float), ("causal", ctypes.c_int32),
                ("window_left", ctypes.c_int32), ("window_right", ctypes.c_int32),
                ("seq_offsets", ctypes.c_void_p), ("num_seqs", ctypes.c_int64),
                ("H_kv", ctypes.c_int64), ("dropout_p", ctypes.c_double),
                ("dropout_seed", ctypes.c_uint64), ("block_mask", ctypes.c_void_p)]


_lib = None


def build(force: bool = False) -> str:
    from . import buildlib
    return buildlib.build(force=force)


def load():
    """Load libfbob.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"libfbob.so not built ({LIB_PATH}); run paper_2609_24089_gb300.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P = ctypes.c_void_p
    S = ctypes.POINTER(fbob_shape)
    sig = {
        "fbob_attn_fwd": [S, P, P, P, P, P, P],
        "fbob_attn_bwd": [S, P, P, P, P, P, P, P, P, P, P, P],
        "fbob_attn_bob": [S, P, P, P, P, P, P, P, P, P, P, P, P, P, P, P],
        "fbob_attn_bob_pass1": [S, P, P, P, P, P, P, P, P, P, P, P, P, P],
        "fbob_attn_bob_pass1_fused": [S, P, P, P, P, P, P, P, P, P, P, P, P, P],
        "fbob_attn_bob_pass2": [S, P, P, P, P, P, P, P, P, P, P, P, P],
        "fbob_attn_bob_row_stats": [S, P, P, P, P, P, P, P, P, P, P, P],
        "fbob_attn_bob_pass1_direct": [S, P, P, P, P, P, P, P, P, P, P, P, P],
        "fbob_attn_bob_host": [S] + [P] * 15 + [ctypes.c_int64, P],
        "fbob_attn_bob_host_workspace": [S, ctypes.c_int64],
        "fbob_attn_bob_host_noalloc": [S] + [P] * 14 + [P],
        "fbob_device_status": [P],
        "fbob_launch_count": [ctypes.c_char_p],
        "fbob_status_string": [ctypes.c_int],
    }
    for name, argt in sig.items():
        f = getattr(lib, name)
        f.argtypes = argt
        f.restype = (ctypes.c_char_p if name == "fbob_status_string" else
                     ctypes.c_int64 if name == "fbob_attn_bob_host_workspace" else ctypes.c_int)
    _lib = lib
    return lib


def header_symbols() -> list:
    """Entry points declared in include/fbob.h."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\**\s+\**(fbob_\w+)\s*\(", text, re.M)))


def make_shape(B, H, N, d, scale, causal, window=None, segments=None,
               kv_heads=None, dropout=None, block_mask=None) -> fbob_shape:
    """window: (left, right) sliding-window band i - left <= j <= i + right;
    -1 (or None) leaves a side unbounded.  segments: contiguous int32 CUDA
    tensor of packed-sequence offsets [num_seqs + 1] (it must stay alive
    until the calls using this shape have run), or None for one sequence.
    kv_heads: key/value heads for grouped-query attention (None: H).
    dropout: (p, seed) attention dropout after the softmax (None: none); the
    realised rate is round(256 p) / 256.  block_mask: contiguous uint8 CUDA
    tensor [nb, nb] (nb = ceil(N / 128)) of 128 x 128 query-key blocks to
    keep, every diagonal block set (kept alive like segments), or None."""
    wl, wr = (-1, -1) if window is None else (int(window[0]), int(window[1]))
    if segments is None:
        seg, nseg = None, 0
    else:
        import torch
        if (not segments.is_cuda or segments.dtype != torch.int32 or segments.dim() != 1
                or not segments.is_contiguous()):
            raise ValueError("segments must be a contiguous 1-D int32 CUDA tensor")
        seg, nseg = segments.data_ptr(), segments.numel() - 1
    hkv = 0 if kv_heads is None or int(kv_heads) == int(H) else int(kv_heads)
    dp, seed = (0.0, 0) if dropout is None else (float(dropout[0]), int(dropout[1]))
    bm = None
    if block_mask is not None:
        import torch
        nb = (int(N) + 127) // 128
        if (not block_mask.is_cuda or block_mask.dtype != torch.uint8
                or tuple(block_mask.shape) != (nb, nb) or not block_mask.is_contiguous()):
            raise ValueError(f"block_mask must be a contiguous [{nb}, {nb}] uint8 CUDA tensor")
        bm = block_mask.data_ptr()
    return fbob_shape(int(B), int(H), int(N), int(d), float(scale), int(causal), wl, wr,
                      seg, nseg, hkv, dp, seed & 0xFFFFFFFFFFFFFFFF, bm)


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return t.data_ptr()


def _stream(stream):
    if stream is not None:
        return stream if isinstance(stream, int) else stream.cuda_stream
    import torch
    return torch.cuda.current_stream().cuda_stream


def _check(rc, where):
    if rc != FBOB_OK:
        raise FbobError(rc, where)


def _shape_of(q, k, scale, causal, window=None, segments=None, dropout=None, block_mask=None):
    B, H, N, d = q.shape
    return make_shape(B, H, N, d, scale, causal, window, segments, kv_heads=k.shape[1],
                      dropout=dropout, block_mask=block_mask)


# ------------------------------------------------ entry points, same names as the C ABI
def fbob_attn_fwd(shape, q, k, v, o, lse, stream=None):
    _check(load().fbob_attn_fwd(ctypes.byref(shape), *map(_ptr, (q, k, v, o, lse)),
                                _stream(stream)), "fbob_attn_fwd")


def fbob_attn_bwd(shape, q, k, v, o, lse, dout, dq, dk, dv, dstat, stream=None):
    _check(load().fbob_attn_bwd(ctypes.byref(shape),
                                *map(_ptr, (q, k, v, o, lse, dout, dq, dk, dv, dstat)),
                                _stream(stream)), "fbob_attn_bwd")


def fbob_attn_bob(shape, q, k, v, o, lse, dout, gq, gk, gv, q_bar, k_bar, v_bar, dout_bar,
                  row_stats, stream=None):
    _check(load().fbob_attn_bob(
        ctypes.byref(shape),
        *map(_ptr, (q, k, v, o, lse, dout, gq, gk, gv, q_bar, k_bar, v_bar, dout_bar, row_stats)),
        _stream(stream)), "fbob_attn_bob")


def fbob_attn_bob_pass1(shape, q, k, v, o, lse, dout, gq, gk, gv, q_bar, dout_bar, row_stats,
                        stream=None):
    _check(load().fbob_attn_bob_pass1(
        ctypes.byref(shape),
        *map(_ptr, (q, k, v, o, lse, dout, gq, gk, gv, q_bar, dout_bar, row_stats)),
        _stream(stream)), "fbob_attn_bob_pass1")


def fbob_attn_bob_pass1_fused(shape, q, k, v, o, lse, dout, gq, gk, gv, q_bar, dout_bar,
                              row_stats, stream=None):
    _check(load().fbob_attn_bob_pass1_fused(
        ctypes.byref(shape),
        *map(_ptr, (q, k, v, o, lse, dout, gq, gk, gv, q_bar, dout_bar, row_stats)),
        _stream(stream)), "fbob_attn_bob_pass1_fused")


def fbob_attn_bob_pass2(shape, q, k, v, lse, dout, gq, gk, gv, row_stats, k_bar, v_bar,
                        stream=None):
    _check(load().fbob_attn_bob_pass2(
        ctypes.byref(shape),
        *map(_ptr, (q, k, v, lse, dout, gq, gk, gv, row_stats, k_bar, v_bar)),
        _stream(stream)), "fbob_attn_bob_pass2")


def fbob_attn_bob_row_stats(shape, q, k, v, o, lse, dout, gq, gk, gv, row_stats, stream=None):
    _check(load().fbob_attn_bob_row_stats(
        ctypes.byref(shape),
        *map(_ptr, (q, k, v, o, lse, dout, gq, gk, gv, row_stats)),
        _stream(stream)), "fbob_attn_bob_row_stats")


def fbob_attn_bob_pass1_direct(shape, q, k, v, lse, dout, gq, gk, gv, row_stats, q_bar, dout_bar,
                               stream=None):
    _check(load().fbob_attn_bob_pass1_direct(
        ctypes.byref(shape),
        *map(_ptr, (q, k, v, lse, dout, gq, gk, gv, row_stats, q_bar, dout_bar)),
        _stream(stream)), "fbob_attn_bob_pass1_direct")


def fbob_attn_bob_host(shape, q, k, v, o, lse, dout, gq, gk, gv, q_bar, k_bar, v_bar, dout_bar,
                       row_stats, workspace, stream=None):
    """Host tensors (pinned for overlap) in and out; workspace: a CUDA uint8
    tensor (its size is passed as workspace_bytes)."""
    _check(load().fbob_attn_bob_host(
        ctypes.byref(shape),
        *map(_ptr, (q, k, v, o, lse, dout, gq, gk, gv, q_bar, k_bar, v_bar, dout_bar, row_stats,
                    workspace)),
        workspace.numel() * workspace.element_size(), _stream(stream)), "fbob_attn_bob_host")


def fbob_attn_bob_host_noalloc(shape, q, k, v, o, lse, dout, gq, gk, gv, q_bar, k_bar, v_bar,
                               dout_bar, row_stats, stream=None):
    """As fbob_attn_bob_host, staged in the library's fixed device array."""
    _check(load().fbob_attn_bob_host_noalloc(
        ctypes.byref(shape),
        *map(_ptr, (q, k, v, o, lse, dout, gq, gk, gv, q_bar, k_bar, v_bar, dout_bar, row_stats)),
        _stream(stream)), "fbob_attn_bob_host_noalloc")


def fbob_attn_bob_host_workspace(shape, chunk_heads) -> int:
    return load().fbob_attn_bob_host_workspace(ctypes.byref(shape), int(chunk_heads))


def fbob_device_status(stream=None) -> int:
    return load().fbob_device_status(_stream(stream))


def fbob_launch_count(entry: str) -> int:
    return load().fbob_launch_count(entry.encode())


# ------------------------------------------------ allocating helpers
def attn_fwd(q, k, v, scale, causal, window=None, segments=None, dropout=None,
             block_mask=None):
    import torch
    B, H, N, d = q.shape
    o = torch.empty_like(q)
    lse = torch.empty((B, H, N), dtype=torch.float32, device=q.device)
    fbob_attn_fwd(_shape_of(q, k, scale, causal, window, segments, dropout, block_mask),
                  q, k, v, o, lse)
    return o, lse


def attn_bwd(q, k, v, o, lse, dout, scale, causal, window=None, segments=None, dropout=None,
             block_mask=None):
    import torch
    B, H, N, d = q.shape
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    dstat = torch.empty((B, H, N), dtype=torch.float32, device=q.device)
    fbob_attn_bwd(_shape_of(q, k, scale, causal, window, segments, dropout, block_mask),
                  q, k, v, o, lse, dout, dq, dk, dv, dstat)
    return dq, dk, dv, dstat


def attn_bob(q, k, v, o, lse, dout, gq, gk, gv, scale, causal, window=None, segments=None,
             dropout=None, block_mask=None):
    """Returns (q_bar, k_bar, v_bar, dout_bar, row_stats[3,B,H,N] = alpha, E, D)."""
    import torch
    B, H, N, d = q.shape
    outs = [torch.empty_like(q), torch.empty_like(k), torch.empty_like(v), torch.empty_like(q)]
    row_stats = torch.empty((3, B, H, N), dtype=torch.float32, device=q.device)
    fbob_attn_bob(_shape_of(q, k, scale, causal, window, segments, dropout, block_mask),
                  q, k, v, o, lse, dout, gq, gk, gv, *outs, row_stats)
    return (*outs, row_stats)
