// dropout.cuh -- attention dropout keep mask, regenerated in every kernel that
// needs it (App. "Extensions": a counter-based generator replaces any stored
// N x N mask).
//
// Layout: one Philox4x32-10 call covers a 4 x 4 block of (query, key) pairs
// of one query head.  Block (I, J) of head h uses counter {J, I, h, 0} and key
// {seed low 32 bits, seed high 32 bits}; pair (4I + a, 4J + b) takes byte b
// (bits 8b .. 8b + 7) of output word a and is kept iff that byte is >= t.
// With t = round(256 p) the realised drop rate is t / 256 and the kept
// entries are scaled by sigma = 256 / (256 - t).
//
// The tile engines give each elementwise thread one stationary row (a query
// in the row engine, a key in the column engine) and 16 consecutive
// streamed indices aligned to 16, and lanes 4m .. 4m + 3 hold 4 consecutive
// stationary rows.  So the four lanes of such a group need exactly four
// blocks: each lane computes one and the keep bits are exchanged with three
// shuffles inside the group.
#pragma once

#include <stdint.h>

namespace fbob {

// Philox4x32-10 (Salmon, Moraes, Dror and Shaw, SC'11): ten rounds of the
// Philox S-box.  rk[2r], rk[2r + 1] is the key of round r: the seed raised r
// times by the Weyl constants 0x9E3779B9, 0xBB67AE85 (formed on the host, so
// the kernels read them from the parameter bank).
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, const uint32_t (&rk)[20]) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ rk[2 * r], lo1, hi0 ^ c.w ^ rk[2 * r + 1], lo0);
  }
  return c;
}

struct DropKey {
  const uint32_t (&rk)[20];  // round keys (kernel parameters)
  uint32_t tlow4;            // (t mod 128) in each byte
  uint32_t tmask;            // all ones if t < 128, else zero
};

// Per byte of x: most significant bit set iff the byte is >= t.  r's bytes
// (x | 0x80) - (t mod 128) compare the low seven bits without borrows; the
// top bits then decide: x >= t iff (x7 or r7) when t < 128, (x7 and r7)
// otherwise, i.e. the majority of x7, r7 and the t < 128 flag.
__device__ __forceinline__ uint32_t bytes_ge(uint32_t x, const DropKey& k) {
  const uint32_t r = (x | 0x80808080u) - k.tlow4;
  return (x & r) | (k.tmask & (x | r));
}

// Keep bits of block (I, J) of query head `head`: bit 4a + b keeps the pair
// (query 4I + a, key 4J + b).
__device__ __forceinline__ uint32_t keep_block(uint32_t I, uint32_t J, uint32_t head,
                                               const DropKey& k) {
  const uint4 w = philox4x32_10(make_uint4(J, I, head, 0u), k.rk);
  // bytes' top bits 7, 15, 23, 31 gathered to 28..31 by one multiply
  // (partial products land on distinct lower bits, so nothing carries)
  auto nib = [&](uint32_t x) -> uint32_t {
    return ((bytes_ge(x, k) & 0x80808080u) * 0x00204081u) >> 28;
  };
  return nib(w.x) | (nib(w.y) << 4) | (nib(w.z) << 8) | (nib(w.w) << 12);
}

// Row-owned tile (row engine): this thread's query i and keys j0 .. j0 + 15
// (j0 a multiple of 16; lanes 4m .. 4m + 3 hold queries 4I .. 4I + 3).
// Returns bit c = keep(i, j0 + c).  All 32 lanes must call it together.
__device__ __forceinline__ uint32_t keep_row16(int i, int j0, uint32_t head, const DropKey& k) {
  const int t = threadIdx.x & 3;
  const uint32_t mine = keep_block((uint32_t)i >> 2, ((uint32_t)j0 >> 2) + t, head, k);
  uint32_t own = 0;
#pragma unroll
  for (int s = 0; s < 4; ++s) {  // block s holds keys j0 + 4s .. + 3
    const uint32_t ms = __shfl_sync(0xffffffffu, mine, s, 4);
    own += ((ms >> (4 * t)) & 0xFu) << (4 * s);
  }
  return own;
}

// Column-owned tile (column engine): this thread's key j and queries
// i0 .. i0 + 15 (i0 a multiple of 16; lanes 4m .. 4m + 3 hold keys
// 4J .. 4J + 3).  Returns bit c = keep(i0 + c, j).  All 32 lanes must call it
// together.
__device__ __forceinline__ uint32_t keep_col16(int j, int i0, uint32_t head, const DropKey& k) {
  const int t = threadIdx.x & 3;
  const uint32_t mine = keep_block(((uint32_t)i0 >> 2) + t, (uint32_t)j >> 2, head, k);
  uint32_t own = 0;
#pragma unroll
  for (int s = 0; s < 4; ++s) {  // block s holds queries i0 + 4s .. + 3
    const uint32_t ms = __shfl_sync(0xffffffffu, mine, s, 4);
    // bits 4a + t (a = 0..3) to bits 12 + a: multiply by 2^12 + 2^9 + 2^6 + 2^3
    // (the other partial products fall on distinct bits outside 12..15)
    const uint32_t x = (ms >> t) & 0x1111u;
    own += ((x * 0x1248u) >> 12 & 0xFu) << (4 * s);
  }
  return own;
}

// The gate sigma R of columns c and c + 1 of a 16-bit keep mask.
__device__ __forceinline__ float2 gate2(uint32_t keep, int c, float sigma) {
  return make_float2((keep >> c) & 1u ? sigma : 0.f, (keep >> (c + 1)) & 1u ? sigma : 0.f);
}

}  // namespace fbob
