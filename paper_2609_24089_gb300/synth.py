"""Seeded synthetic inputs for attention backward-over-backward.

This module draws random numbers and rounds them to bf16; it holds none of the
method's arithmetic, so the CUDA path and the CPU oracle can both consume its
output without sharing any computation.

Recipe (the paper's isolated-kernel benchmark uses fixed-seed random inputs at
GPT-2 head shape, Sec. 4.1; the shapes below stand in for it):
  * numpy ``Generator(PCG64(seed))``;
  * draw order Q, K, V, dO, U_Q, U_K, U_V, each ``standard_normal`` in fp32
    times the tensor's standard deviation;
  * round to nearest-even bf16 on the host.  Tensors are carried as uint16
    bit patterns ([B, H, N, d], row-major) so that both sides see identical
    values; ``to_f64`` up-casts them exactly.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

NAMES = ("q", "k", "v", "dout", "gq", "gk", "gv")


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    N: int
    d: int
    causal: bool
    seed: int
    sigma: tuple  # per tensor in NAMES order
    window: tuple = (-1, -1)  # sliding-window band (left, right); -1 = unbounded
    segments: tuple = ()      # offsets of packed sequences along N; () = one sequence
    kv_heads: int = 0         # key/value heads (grouped-query attention); 0 = H
    dropout: tuple = ()       # attention dropout (p, seed); () = none
    blocks: tuple = ()        # block-sparse mask (local, sinks, density, seed); () = none

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.d)

    @property
    def shape(self) -> tuple:
        return (self.B, self.H, self.N, self.d)


def _s(*v):
    return tuple(float(x) for x in v)


# The five synthetic workloads.  Standard deviations follow each workload's
# stated distribution; seeds are the workload index minus one.
WORKLOADS = {
    "n128_d64": Workload("n128_d64", 1, 1, 128, 64, False, 0, _s(1, 1, 1, 1, 1, 1, 1)),
    "n4k_d64": Workload("n4k_d64", 4, 16, 4096, 64, False, 1, _s(1, 1, 1, 1, 1, 1, 1)),
    "n16k_d128_causal": Workload(
        "n16k_d128_causal", 2, 16, 16384, 128, True, 2,
        _s(1, 1, 1, *(4 * [1 / math.sqrt(128)]))),
    "n64k_d128_causal_peaky": Workload(
        "n64k_d128_causal_peaky", 1, 8, 65536, 128, True, 3, _s(1.5, 1.5, 1, 1, 1, 1, 1)),
    "n256k_d64": Workload("n256k_d64", 1, 4, 262144, 64, False, 4, _s(1, 1, 1, 1, 1, 1, 1)),
    # sliding-window variant of n16k_d128_causal with the window of the paper's
    # sliding-window experiment, w = N/4 keys (row i keeps i - w < j <= i)
    "n16k_d128_causal_swa4k": Workload(
        "n16k_d128_causal_swa4k", 2, 16, 16384, 128, True, 5,
        _s(1, 1, 1, *(4 * [1 / math.sqrt(128)])), (4095, -1)),
}


def packed_offsets(N: int, n: int, seed: int) -> tuple:
    """Offsets of n packed sequences filling N: seeded lengths drawn
    uniformly between N/(4n) and 7N/(4n), rescaled to sum to N."""
    rng = np.random.Generator(np.random.PCG64(seed))
    lens = rng.uniform(0.25, 1.75, n)
    cuts = np.round(np.cumsum(lens) / lens.sum() * N).astype(np.int64)
    cuts[-1] = N
    return tuple(int(x) for x in np.concatenate([[0], cuts]))


# packed variable-length variant of n16k_d128_causal: 12 causal sequences of
# seeded lengths (about 340 to 2400 tokens) in the 16K rows of each head
# grouped-query variant of n16k_d128_causal: 4 key/value heads for 16 query heads
WORKLOADS["n16k_d128_causal_gqa4"] = Workload(
    "n16k_d128_causal_gqa4", 2, 16, 16384, 128, True, 7,
    _s(1, 1, 1, *(4 * [1 / math.sqrt(128)])), kv_heads=4)

# dropout variant of n16k_d128_causal: p = 0.1 after the softmax
WORKLOADS["n16k_d128_causal_drop10"] = Workload(
    "n16k_d128_causal_drop10", 2, 16, 16384, 128, True, 8,
    _s(1, 1, 1, *(4 * [1 / math.sqrt(128)])), dropout=(0.1, (8 << 32) | 8))

# head-dimension sweep at the shape of the paper's sensitivity table
# (App. "Head-dimension sensitivity": N = 4096, B = 4, H = 12, causal)
for _d in (32, 64, 128, 256):
    WORKLOADS[f"n4k_d{_d}_causal_b4h12"] = Workload(
        f"n4k_d{_d}_causal_b4h12", 4, 12, 4096, _d, True, 9, _s(1, 1, 1, 1, 1, 1, 1))

# block-sparse variant of n16k_d128_causal (App. "Extensions"): each query
# block keeps its own and the 2 previous key blocks, the first key block, and
# random blocks with probability 0.1 (about a quarter of the causal blocks)
WORKLOADS["n16k_d128_causal_bsparse"] = Workload(
    "n16k_d128_causal_bsparse", 2, 16, 16384, 128, True, 10,
    _s(1, 1, 1, *(4 * [1 / math.sqrt(128)])), blocks=(2, 1, 0.1, 10))

# head dimension 256 (App. "Head-dimension sensitivity" names it as the next
# specialisation): the causal headline shape at one batch entry and 8 heads
WORKLOADS["n16k_d256_causal"] = Workload(
    "n16k_d256_causal", 1, 8, 16384, 256, True, 11, _s(1, 1, 1, *(4 * [1 / math.sqrt(256)])))

WORKLOADS["n16k_d128_causal_varlen"] = Workload(
    "n16k_d128_causal_varlen", 2, 16, 16384, 128, True, 6,
    _s(1, 1, 1, *(4 * [1 / math.sqrt(128)])), segments=packed_offsets(16384, 12, 6))


def block_pattern(N: int, local: int, sinks: int, density: float, seed: int,
                  block: int = 128) -> np.ndarray:
    """[nb, nb] uint8 block-sparse mask over block x block tiles (nb =
    ceil(N / block)): query block b keeps key blocks b - local .. b (its own
    and `local` before it), the first `sinks` key blocks, and every other key
    block with probability `density` (seeded); the diagonal is always set."""
    nb = (N + block - 1) // block
    rng = np.random.Generator(np.random.PCG64(seed))
    bm = (rng.random((nb, nb)) < density)
    b = np.arange(nb)
    bm |= (b[None, :] <= b[:, None]) & (b[None, :] >= b[:, None] - local)
    bm[:, :sinks] = True
    return bm.astype(np.uint8)


def workload_blocks(w: Workload):
    """The workload's block mask ([nb, nb] uint8, 128 x 128 blocks), or None."""
    if not w.blocks:
        return None
    local, sinks, density, seed = w.blocks
    return block_pattern(w.N, int(local), int(sinks), float(density), int(seed))


def band_pairs(w: Workload, rows=None) -> float:
    """Valid (i, j) pairs of the listed rows (all rows by default) under the
    workload's mask: the band i - wl <= j <= i + wr, capped at j <= i if causal."""
    r = np.arange(w.N, dtype=np.int64) if rows is None else np.asarray(rows, dtype=np.int64)
    wl, wr = w.window
    lo = np.zeros_like(r) if wl < 0 else np.maximum(0, r - wl)
    hi = np.full_like(r, w.N) if wr < 0 else np.minimum(w.N, r + wr + 1)
    if w.causal:
        hi = np.minimum(hi, r + 1)
    if w.segments:
        seg = np.asarray(w.segments, dtype=np.int64)
        s = np.searchsorted(seg[1:], r, side="right")
        lo = np.maximum(lo, seg[s])
        hi = np.minimum(hi, seg[s + 1])
    bm = workload_blocks(w)
    if bm is None:
        return float(np.sum(hi - lo))
    # with a block mask: the part of each row's [lo, hi) inside its set blocks
    total = 0.0
    for kb in range(bm.shape[1]):
        keep = bm[r // 128, kb] != 0
        a = np.maximum(lo, kb * 128)
        b = np.minimum(hi, min(w.N, (kb + 1) * 128))
        total += float(np.sum(np.where(keep, np.maximum(b - a, 0), 0)))
    return total


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (round to nearest, ties to even); return uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return rounded.astype(np.uint16)


def to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact up-cast of bf16 bit patterns to float64."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def make_inputs(B, H, N, d, seed, sigma=(1.0,) * 7, heads=None):
    """Draw the seven bf16 inputs.  ``heads`` (list of flat b*H+h indices)
    keeps only those heads after drawing, so a slice sees exactly the values
    the full tensor holds."""
    rng = np.random.Generator(np.random.PCG64(seed))
    out = {}
    for name, s in zip(NAMES, sigma):
        x = rng.standard_normal((B, H, N, d), dtype=np.float32)
        if s != 1.0:
            x *= np.float32(s)
        bits = bf16_bits(x)
        if heads is not None:
            bits = np.ascontiguousarray(bits.reshape(B * H, N, d)[list(heads)])
            bits = bits.reshape(1, len(heads), N, d)
        out[name] = bits
        del x
    return out


def workload_inputs(w: Workload, heads=None):
    """The workload's seven inputs; with kv_heads, k, v, gk, gv keep the first
    kv_heads heads of each batch entry."""
    bits = make_inputs(w.B, w.H, w.N, w.d, w.seed, w.sigma, heads=heads)
    if w.kv_heads and heads is None:
        for n in ("k", "v", "gk", "gv"):
            bits[n] = np.ascontiguousarray(bits[n][:, :w.kv_heads])
    return bits
