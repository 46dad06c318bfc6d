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
// Philox S-box; the key is raised by the Weyl constants before each round
// after the first.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

struct DropKey {
  uint32_t k0, k1;  // Philox key (the seed)
  uint32_t thr4;    // byte threshold t in each of the four bytes
};

// Keep bits of block (I, J) of query head `head`: bit 4a + b keeps the pair
// (query 4I + a, key 4J + b).
__device__ __forceinline__ uint32_t keep_block(uint32_t I, uint32_t J, uint32_t head,
                                               const DropKey& k) {
  const uint4 w = philox4x32_10(make_uint4(J, I, head, 0u), k.k0, k.k1);
  // per byte 0xFF where byte >= t; byte b's bit b, summed into the top byte
  auto nib = [&](uint32_t x) -> uint32_t {
    return ((__vcmpgeu4(x, k.thr4) & 0x08040201u) * 0x01010101u) >> 24;
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
    own |= ((ms >> (4 * t)) & 0xFu) << (4 * s);
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
    const uint32_t x = (ms >> t) & 0x1111u;  // bits 4a + t, a = 0..3
    own |= ((x | (x >> 3) | (x >> 6) | (x >> 9)) & 0xFu) << (4 * s);
  }
  return own;
}

// The gate sigma R of columns c and c + 1 of a 16-bit keep mask.
__device__ __forceinline__ float2 gate2(uint32_t keep, int c, float sigma) {
  return make_float2((keep >> c) & 1u ? sigma : 0.f, (keep >> (c + 1)) & 1u ? sigma : 0.f);
}

}  // namespace fbob
