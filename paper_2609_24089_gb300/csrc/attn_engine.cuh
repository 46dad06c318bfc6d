// attn_engine.cuh -- warp-specialised tcgen05 tile engines for softmax
// attention and its backward-over-backward on sm_103a.
//
// Two engines share one schedule skeleton:
//   * row engine: a CTA owns BM = 128 query rows (TMEM lanes) and streams key
//     tiles of BN = 64 rows.  Used by the dQ half of the first backward
//     (eqs. 2-3) and BoB Pass 1 (Alg. 2, first loop): at
//     d = 64 in one sweep with the affine fusion of Prop. 3.1 (four
//     accumulators); at d = 128 as a row-statistics kernel (alpha, E, D; stage
//     A only) followed by the direct form of eqs. (6)-(7) (two accumulators).
//   * column engine: a CTA owns BM = 128 key rows and streams query tiles of
//     BN = 64 rows, computing transposed tiles (key rows on lanes).  Used by
//     the dK/dV half of the first backward and BoB Pass 2 (Alg. 2, second loop).
// The forward (eq. 1) has its own engine with two query tiles per CTA
// (fwd_engine.cuh).
//
// Roles (352 threads):
//   warps 0-7  elementwise: two warpgroups; warp w reads TMEM lanes
//              32*(w%4) .. +31, one stationary row per thread.  Warpgroup g
//              takes columns 16g .. 16g+15 of every 32-column half tile.
//   warp 8     TMA producer: stationary tiles once, then a ring of NSTAGES
//              stream stages (mbarrier full/empty pairs).  In the column engine
//              it also stages the streamed rows' fp32 row vectors in shared memory.
//   warp 9     MMA issuer X (one lane; the warp also allocates TMEM).
//   warp 10    MMA issuer Y (one lane).
//
// Tensor memory (512 columns): accumulators at 0..255; stage-A area "SF" at
// 256..383 (scores, and F in the BoB passes), owned by issuer X; stage-A area
// "DC" at 384..511 (dP, and C in the BoB passes), owned by issuer Y.  Where
// the DC tile leaves room (the column engine at d = 64, both first-backward
// kernels) DC is double-buffered and issued two tiles ahead.
//
// Per streamed tile t:
//   X  issues SF(t+1) as soon as the elementwise warps have copied SF(t)
//      into registers, so the next tile's largest stage-A contractions run
//      while the elementwise warps still work on tile t.
//   Y  issues DC(t) (per 32-column half in the one-sweep Pass 1, for the
//      whole tile otherwise).
//   elementwise: copy SF to registers and release it; then per half read DC,
//      compute, and write the bf16 operand tiles of stage B over the DC
//      columns just read; stage B of half 0 overlaps the elementwise work on
//      half 1.
//   stage B is issued by Y, or (config flag XSHARE) split between the
//      issuers by accumulator: X then owns B and dOtil0 (Pass 1) or the value
//      gradient (column engine) and Y the rest.
// Every accumulator has one writer issuer, so it is summed in a fixed order
// (bitwise reproducible results).  With XSHARE the one cross-issuer hazard is
// that DC(t+1) overwrites operand tiles X's stage-B MMAs of tile t read: X
// commits those MMAs to bar_xb and Y waits for that before issuing DC(t+1).
//
// A single thread issues at most one tcgen05.mma about every 53 cycles and
// the tensor core needs N >= 128 per instruction to stay busy, so MMAs that
// share an operand are fused to N = 128 ([S|F] = Q [K;U_K]^T,
// [B|dOtil0] += P [K|U_V], [G|Omega] += dS [K|U_K], ...).
//
// Shared memory: stationary tensors as 128-row x 64-column swizzled boxes;
// each stream stage as, per 64-column box, 64-row tiles in tensor order.  In
// Pass 1, V and U_V are stored as 32-row chunks V_0 U_V_0 V_1 U_V_1 so that
// [V_h ; U_V_h] is one 64-row operand.
//
// Every wait is bounded (tc_ptx.cuh); on expiry the CTA records a timeout in
// the device error word, drains its own asynchronous work and exits.
#pragma once

#include "dropout.cuh"
#include "engine_params.h"
#include "tc_ptx.cuh"

namespace fbob {

constexpr uint32_t kColSF = 256;   // stage-A area of issuer X
constexpr uint32_t kColDC = 384;   // stage-A area of issuer Y
// row statistics kernel: Q and U_Q as MMA A operands in TMEM (bf16 pairs per
// column, D/2 columns each) at kColQT and kColQT + D/2; second SF buffer
constexpr uint32_t kColQT = 0;
constexpr uint32_t kColSF1 = 128;

// Shared-memory bookkeeping block (in the MISC area).
struct Misc {
  uint64_t bar_stat;
  uint64_t bar_full[kMaxStages];    // first part of a stream stage landed (all issuer X reads)
  uint64_t bar_full_b[kMaxStages];  // rest of the stage (and, column engine, the row vectors)
  uint64_t bar_empty[kMaxStages];
  uint64_t bar_sa_sf[2];   // X's stage A of a tile completed (per SF buffer)
  uint64_t bar_sf_free[2]; // elementwise warps copied SF to registers (per SF buffer)
  uint64_t bar_dc_free; // elementwise warps copied DC to registers (row statistics kernel)
  uint64_t bar_sa_dc[2];
  uint64_t bar_ew[4];   // [DC buffer][half]; a single DC buffer uses [0..1]
  uint64_t bar_xb[2];   // issuer X's stage-B MMAs completed (per half, or per DC buffer)
  uint64_t bar_acc;
  // issuer X's per-tile signal to issuer Y, per parity of the tile: its part
  // of SF(t) completed (row statistics kernel), or SF(t+1) issued (Pass 2
  // with P o h in SF)
  uint64_t bar_xsig[2];
  uint32_t tmem_base;
  uint32_t pad;
  WaitCtl wctl;
};
static_assert(sizeof(Misc) <= 256, "Misc must fit the first 256 bytes of the MISC area");

__device__ __forceinline__ uint32_t lane_base_addr(uint32_t tmem_base, int warp) {
  return tmem_base + ((uint32_t)(32 * (warp & 3)) << 16);
}

// Offset inside a stream stage of rows 32h .. 32h+31 of streamed tensor t,
// 64-column box b.  Tensors are 64-row tiles in order, except that with
// kHalvesVUV (Pass 1) tensors 2 and 3 (V, U_V) are interleaved 32-row chunks.
template <int NSTREAM, bool kHalvesVUV>
__device__ __forceinline__ uint32_t soff(int t, int h, int b) {
  constexpr int kBox = NSTREAM * BN * 128;
  if (kHalvesVUV && t >= 2)
    return (uint32_t)(b * kBox + 2 * BN * 128 + h * 2 * kChunk + (t - 2) * kChunk);
  return (uint32_t)(b * kBox + t * BN * 128 + h * kChunk);
}

// Second-chance drain used only on the abort path: waits (bounded, ignoring
// the abort flag) for asynchronous work this CTA started.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > 200000000ull) return;
  }
}

// [lo, hi) of the packed sequence holding index i: [0, N) without offsets.
// A binary search for the last s with off[s] <= i; the result is clamped to
// [0, N) and to contain i, so offsets that break the documented rules give
// wrong values but never an access outside the buffers or an empty row.
__device__ __forceinline__ void seq_bounds(const EngineParams& p, int i, int& lo, int& hi) {
  lo = 0;
  hi = p.N;
  if (p.seq_off == nullptr) return;
  int a = 0, b = p.nseq;
  while (b - a > 1) {
    const int m = (a + b) >> 1;
    if (p.seq_off[m] <= i) a = m;
    else b = m;
  }
  lo = max(0, min(p.seq_off[a], i));
  hi = min(p.N, max(p.seq_off[a + 1], i + 1));
}

// Streamed tiles of one CTA under a block-sparse mask (App. "Extensions":
// the streamed loop visits only the block pairs with an unmasked entry).
// Tiles of BN = 64 rows lie in 128-row mask blocks; tile t is visited if the
// mask entry of its block (t / 2) is set.  mb points at the stationary
// block's entry for streamed block 0 and stride steps to the next streamed
// block (1 along a mask row, nbm down a column); mb == nullptr visits every
// tile of the band t0 .. t1.
struct TileSet {
  const uint8_t* mb;
  int stride;
  int t0, t1;
  __device__ __forceinline__ bool set(int t) const {
    return mb == nullptr || mb[(size_t)(t >> 1) * stride] != 0;
  }
  // number of visited tiles
  __device__ int count() const {
    if (mb == nullptr) return t1 - t0 + 1;
    int n = 0;
    for (int b = t0 >> 1; b <= (t1 >> 1); ++b)
      if (mb[(size_t)b * stride] != 0) n += min(2 * b + 1, t1) - max(2 * b, t0) + 1;
    return n;
  }
  // first visited tile >= t (t1 + 1 if there is none)
  __device__ __forceinline__ int next(int t) const {
    if (mb == nullptr) return t;
    while (t <= t1 && mb[(size_t)(t >> 1) * stride] == 0) t = (t | 1) + 1;
    return t;
  }
};

// CTA order: heads in groups of p.head_group; within a group the blocks are
// outermost (with the causal mask the longest first) and the group's heads
// innermost.  head_group 1 is head-major (the CTAs in flight share one head's
// streamed tiles in L2); head_group >= BH puts every head's longest block
// first (the best balance, the least sharing).
__device__ __forceinline__ void cta_order(const EngineParams& p, int lin, int& rbi, int& bh) {
  const int G = p.head_group;
  const int grp = lin / (p.nblk * G);
  const int gsz = min(G, p.BH - grp * G);
  const int rem = lin - grp * p.nblk * G;
  rbi = rem / gsz;
  bh = grp * G + rem % gsz;
}

__device__ __forceinline__ float bits_f(uint32_t u) { return __uint_as_float(u); }
__device__ __forceinline__ float2 pair(const uint32_t (&r)[16], int c) {
  return make_float2(__uint_as_float(r[c]), __uint_as_float(r[c + 1]));
}
__device__ __forceinline__ float2 splat(float x) { return make_float2(x, x); }

// 16 bf16 values -> two 16-byte global stores.
__device__ __forceinline__ void store_row16(__nv_bfloat16* dst, const float (&v)[16]) {
  uint4 a, b;
  a.x = pack_bf16(v[0], v[1]);
  a.y = pack_bf16(v[2], v[3]);
  a.z = pack_bf16(v[4], v[5]);
  a.w = pack_bf16(v[6], v[7]);
  b.x = pack_bf16(v[8], v[9]);
  b.y = pack_bf16(v[10], v[11]);
  b.z = pack_bf16(v[12], v[13]);
  b.w = pack_bf16(v[14], v[15]);
  reinterpret_cast<uint4*>(dst)[0] = a;
  reinterpret_cast<uint4*>(dst)[1] = b;
}

__device__ __forceinline__ void load_row16(const __nv_bfloat16* src, float (&v)[16]) {
  const uint4 a = reinterpret_cast<const uint4*>(src)[0];
  const uint4 b = reinterpret_cast<const uint4*>(src)[1];
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
  for (int t = 0; t < 8; ++t) {
    v[2 * t] = __uint_as_float(w[t] << 16);
    v[2 * t + 1] = __uint_as_float(w[t] & 0xFFFF0000u);
  }
}

// D_i = do_i . o_i (fp32) for the 128 rows of a row block, computed by the
// 256 elementwise threads together and returned to thread r (any warpgroup)
// for row r.  Each row's DG bf16 values are read by DG / 8 consecutive lanes,
// 16 bytes each, so a warp's loads cover whole rows (coalesced); the lanes'
// partial sums are added by shuffles and passed on through s_d[128].  Every
// elementwise thread must call it (it ends in a named barrier).
template <int DG>
__device__ __forceinline__ float block_row_dots(const __nv_bfloat16* dout, const __nv_bfloat16* o,
                                                size_t head_off, int i0, int row_end, float* s_d,
                                                int ew_tid) {
  constexpr int LPR = DG / 8;     // lanes per row
  constexpr int RPI = 32 / LPR;   // rows per warp instruction
  const int warp = ew_tid >> 5, lane = ew_tid & 31;
  const int sub = lane / LPR, part = lane % LPR;
  float acc[16 / RPI];
#pragma unroll
  for (int k = 0; k < 16 / RPI; ++k) {  // this warp's 16 rows, RPI at a time
    const int r = 16 * warp + RPI * k + sub;
    acc[k] = 0.f;
    if (i0 + r < row_end) {
      const size_t off = head_off + (size_t)(i0 + r) * DG + 8 * part;
      const uint4 va = *reinterpret_cast<const uint4*>(dout + off);
      const uint4 vb = *reinterpret_cast<const uint4*>(o + off);
      const uint32_t wa[4] = {va.x, va.y, va.z, va.w};
      const uint32_t wb[4] = {vb.x, vb.y, vb.z, vb.w};
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        acc[k] = fmaf(__uint_as_float(wa[t] << 16), __uint_as_float(wb[t] << 16), acc[k]);
        acc[k] = fmaf(__uint_as_float(wa[t] & 0xFFFF0000u), __uint_as_float(wb[t] & 0xFFFF0000u),
                      acc[k]);
      }
    }
  }
#pragma unroll
  for (int k = 0; k < 16 / RPI; ++k) {
#pragma unroll
    for (int s = LPR / 2; s > 0; s >>= 1) acc[k] += __shfl_xor_sync(0xffffffffu, acc[k], s);
    if (part == 0) s_d[16 * warp + RPI * k + sub] = acc[k];
  }
  named_bar_sync(2, kEwThreads);
  return s_d[32 * (warp & 3) + lane];
}

// p = exp2(s * sl2 - L2) for a pair of scores.
__device__ __forceinline__ float2 probs2(float2 s, float2 sl2, float2 nL2) {
  const float2 a = __ffma2_rn(s, sl2, nL2);
  return make_float2(ex2(a.x), ex2(a.y));
}

// Masked columns (c < lo or c >= hi) of a thread's 16 scores set to -inf, so
// that P = 2^-inf = 0 there; only tiles that cross a band edge need it, which
// keeps the mask out of the elementwise loops.
__device__ __forceinline__ void mask16(uint32_t (&r)[16], int lo, int hi) {
#pragma unroll
  for (int c = 0; c < 16; ++c)
    if (c < lo || c >= hi) r[c] = 0xFF800000u;
}

// ============================================================== row engine
// D: head dimension of the tiles (64 or 128); DG <= D: head dimension of the
// tensors in global memory.  DG = 32 runs in the D = 64 tiles: the TMA loads
// fill columns 32..63 with zeros, which add nothing to any contraction, and
// only the first DG columns are read or written directly.
// DROP: attention dropout (App. "Extensions"); the one-sweep Pass 1 has none.
template <RowOp OP, int D, bool DROP, int DG>
__global__ void __launch_bounds__(kThreads, 1) row_engine(const __grid_constant__ EngineParams p) {
  using C = RowCfg<OP, D>;
  static_assert(DG == D || (DG == 32 && D == 64), "global head dim 32 runs in 64-wide tiles");
  static_assert(!DROP || OP != RowOp::BobPass1, "dropout Pass 1 runs as statistics + direct");
  static_assert(C::NSTAGES >= 2 && C::NSTAGES <= kMaxStages, "the stage barriers hold kMaxStages stages");
  constexpr bool kBob = OP == RowOp::BobPass1;      // Pass 1, one sweep (Prop. 3.1)
  constexpr bool kStats = OP == RowOp::BobStats;    // row scalars alpha, E, D only
  constexpr bool kDirect = OP == RowOp::BobPass1D;  // Pass 1 with alpha, E given
  constexpr bool kB4 = row_bob(OP);                 // streamed K, U_K, V, U_V
  constexpr bool kDcHalves = C::DC_HALVES;           // DC issued per 32-column half
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* s_stat = smem;
  uint8_t* s_stream = smem + C::STAT_BYTES;
  Misc* m = reinterpret_cast<Misc*>(s_stream + C::NSTAGES * C::STAGE_BYTES);
  float* s_xchg = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(m) + 256);  // 4 x BM floats
  float* s_d = s_xchg + 4 * BM;  // BM floats: the rows' D (block_row_dots)

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  if ((smem_u32(smem) & 1023u) != 0) {  // swizzle atoms need 1024-byte alignment
    if (tid == 0) atomicOr(&g_fbob_error_word, kDevErrBadLaunch);
    return;
  }

  // ---- tile decode (CTA order: cta_order).
  const int N = p.N;
  // one-sweep Pass 1 at d = 128: the C::SPLIT CTAs of a row block are
  // neighbours in launch order; hc selects this CTA's 64 output columns
  const int hc = C::SPLIT > 1 ? (int)(blockIdx.x % C::SPLIT) : 0;
  const int lin = blockIdx.x / C::SPLIT;
  int rbi, bh;
  cta_order(p, lin, rbi, bh);
  const int rb = p.causal ? (p.nblk - 1 - rbi) : rbi;
  // key/value head of this query head (grouped-query attention: h / (H / Hkv))
  const int bh_kv = p.Hkv == p.H ? bh : (bh / p.H) * p.Hkv + (bh % p.H) / (p.H / p.Hkv);
  const int i0 = rb * BM;
  const int last_row = min(i0 + BM, N) - 1;
  // streamed key tiles: those overlapping the rows' bands [i - wl, i + wr]
  // (negative w: unbounded; the causal mask has wr = 0) within their packed
  // sequences; both ends of a row's range grow with i
  int seq_lo0, seq_hi0, seq_lo1, seq_hi1;
  seq_bounds(p, i0, seq_lo0, seq_hi0);
  seq_bounds(p, last_row, seq_lo1, seq_hi1);
  const int key_lo = max(seq_lo0, p.wl < 0 ? 0 : i0 - p.wl);
  const int key_hi = min(seq_hi1, p.wr < 0 ? N : last_row + p.wr + 1);  // exclusive
  const int first_tile = key_lo / BN;
  // (with a block-sparse mask only the tiles of this row block's set blocks)
  const TileSet tiles = {p.bmask ? p.bmask + (size_t)rb * p.nbm : nullptr, 1, first_tile,
                         (key_hi - 1) / BN};
  const int nsteps = tiles.count();

  if (tid == 0) {
    m->wctl.abort = 0;
    m->wctl.limit_ns = p.wait_limit_ns;
    // stationary tiles: one TMA transaction (plus, with C::STAT_TMEM, the
    // elementwise threads' stores of Q and U_Q into TMEM)
    mbar_init(&m->bar_stat, C::STAT_TMEM ? 1 + kEwThreads : 1);
    for (int s = 0; s < C::NSTAGES; ++s) {
      mbar_init(&m->bar_full[s], 1);
      mbar_init(&m->bar_full_b[s], 1);
    }
    // released by both MMA issuers, per stage or (C::HALF_REL) per 32-key half
    for (int s = 0; s < (C::HALF_REL ? 2 : 1) * C::NSTAGES; ++s) mbar_init(&m->bar_empty[s], 2);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&m->bar_sa_sf[b], 1);
      mbar_init(&m->bar_sf_free[b], kEwThreads);
    }
    mbar_init(&m->bar_dc_free, kEwThreads);
    for (int h = 0; h < 2; ++h) {
      mbar_init(&m->bar_sa_dc[h], 1);
      mbar_init(&m->bar_xb[h], 1);
      mbar_init(&m->bar_xsig[h], 1);
    }
    for (int h = 0; h < 4; ++h) mbar_init(&m->bar_ew[h], kEwThreads);
    mbar_init(&m->bar_acc, 2);
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&m->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = m->tmem_base;
  WaitCtl* wctl = &m->wctl;
  volatile int* abort_flag = &m->wctl.abort;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------ producer
    // p.inject_stall (host-side fault injection, off by default): issue no
    // loads at all, so every consumer wait runs into its bounded limit.
    if (elect_lane0() && !p.inject_stall) {
      for (int t = 0; t < C::NSTAT + C::NSTREAM; ++t) tma_prefetch_desc(&p.tm[t]);
      // (with C::STAT_TMEM only dO, map 2, goes to shared memory)
      mbar_arrive_expect_tx(&m->bar_stat, C::STAT_BYTES);
      for (int t = C::STAT_TMEM ? 2 : 0; t < C::NSTAT; ++t)
        for (int b = 0; b < C::KB; ++b)
          tma_load_3d(s_stat + ((C::STAT_TMEM ? 0 : t) * C::KB + b) * (BM * 128), &p.tm[t],
                      &m->bar_stat, 64 * b, i0, bh);
      int issued[kMaxStages] = {-1, -1, -1, -1};
      int tile = first_tile - 1;
      bool go = true;
      for (int st = 0; go && st < nsteps; ++st) {
        const int stage = st % C::NSTAGES;
        const uint32_t epar = ((st / C::NSTAGES) - 1) & 1;
        if (st >= C::NSTAGES && !C::HALF_REL) {
          if (!mbar_wait(&m->bar_empty[stage], epar, wctl)) break;
        }
        tile = tiles.next(tile + 1);
        const int j0 = tile * BN;
        const int nt = C::NSTREAM;
        uint8_t* dst = s_stream + stage * C::STAGE_BYTES;
        // BoB: K and U_K first on bar_full (all issuer X needs), then V and
        // U_V on bar_full_b; the other operations use bar_full alone
        const int nt_a = kB4 ? 2 : nt;
        if (!kB4) {
          mbar_arrive_expect_tx(&m->bar_full[stage], nt_a * C::KB * BN * 128);
          for (int b = 0; b < C::KB; ++b)
            for (int t = 0; t < nt_a; ++t)
              tma_load_3d(dst + soff<C::NSTREAM, kB4>(t, 0, b), &p.tm[C::NSTAT + t],
                          &m->bar_full[stage], 64 * b, j0, bh_kv);
          issued[stage] = st;
        } else {
          // every streamed tensor in 32-row chunks (map box rows HB), half h
          // of the tile (keys 32 h ..) after the other; with C::HALF_REL each
          // half of the stage is refilled as soon as its own release comes.
          // The full barriers are armed only once half 0 is released: that
          // release implies the stage's previous phase completed.
          for (int h = 0; h < 2; ++h) {
            if (C::HALF_REL && st >= C::NSTAGES &&
                !mbar_wait(&m->bar_empty[2 * stage + h], epar, wctl)) {
              go = false;
              break;
            }
            if (h == 0) {
              mbar_arrive_expect_tx(&m->bar_full[stage], 2 * C::KB * BN * 128);
              mbar_arrive_expect_tx(&m->bar_full_b[stage], 2 * C::KB * BN * 128);
              issued[stage] = st;  // (a stage left half loaded drains by its time limit)
            }
            for (int b = 0; b < C::KB; ++b)
              for (int t = 0; t < 2; ++t)
                tma_load_3d(dst + soff<C::NSTREAM, kB4>(t, h, b), &p.tm[C::NSTAT + t],
                            &m->bar_full[stage], 64 * b, j0 + HB * h, bh_kv);
            for (int b = 0; b < C::KB; ++b)
              for (int t = 2; t < 4; ++t)
                tma_load_3d(dst + soff<C::NSTREAM, kB4>(t, h, b), &p.tm[C::NSTAT + t],
                            &m->bar_full_b[stage], 64 * b, j0 + HB * h, bh_kv);
          }
        }
      }
      if (*abort_flag) {  // drain loads still in flight
        for (int s = 0; s < C::NSTAGES; ++s)
          if (issued[s] >= 0) {
            drain_wait(&m->bar_full[s], (issued[s] / C::NSTAGES) & 1);
            if (kB4) drain_wait(&m->bar_full_b[s], (issued[s] / C::NSTAGES) & 1);
          }
        drain_wait(&m->bar_stat, 0);
      }
    }
  } else if (warp == kMmaWarp || warp == kMmaWarpY) {
    // ------------------------------------------------------------ MMA issuers
    if (elect_lane0()) {
      constexpr uint32_t id_n64 = idesc_bf16(128, 64, false);
      constexpr uint32_t id_n128 = idesc_bf16(128, 128, false);
      // stage B of the one-sweep Pass 1 accumulates 64 output columns per CTA
      constexpr uint32_t id_b = idesc_bf16(128, kBob ? 64 : D, true);
      constexpr uint32_t id_b2 = idesc_bf16(128, 2 * (kBob ? 64 : D), true);
      // descriptors are formed once; per MMA only the start-address field moves
      const uint64_t sd0 = sdesc_sw128(smem_u32(s_stat), 16, 1024);
      auto sd = [&](int t, int k) -> uint64_t {
        return sd0 + (uint64_t)(((t * C::KB + k / 4) * (BM * 128) + (k % 4) * 32) >> 4);
      };
      // K-major view of streamed rows 32h.. (64 of them) of tensor t, K-step k
      auto kd = [&](uint64_t kd0, int t, int h, int k) -> uint64_t {
        return kd0 + (uint64_t)((soff<C::NSTREAM, kB4>(t, h, k / 4) + (k % 4) * 32) >> 4);
      };
      // stage B of half h: K-steps s = 2h + sub, 16 streamed rows each; the
      // operand tiles of K-step s sit at DC columns written by warpgroup sub.
      // With C::XSHARE issuer X takes the MMAs into B and dOtil0 (one sweep)
      // or dOtil (direct form) (part 0) and issuer Y the rest (part 1);
      // otherwise Y takes them all (part 2).
      auto stage_b = [&](uint32_t sb, int h, int st, int part) {
        constexpr uint32_t kBoxBytes = C::NSTREAM * BN * 128;
        const uint64_t md0 = sdesc_sw128(sb, kBoxBytes, 1024);
#pragma unroll
        for (int sub = 0; sub < 2; ++sub) {
          const int s = 2 * h + sub;
          auto md = [&](int t, int bo) -> uint64_t {
            return md0 + (uint64_t)((soff<C::NSTREAM, kB4>(t, h, bo) + sub * 2048) >> 4);
          };
          const uint32_t first = (st == 0 && s == 0) ? 0u : 1u;
          if constexpr (kBob) {
            // B operands: the 64-column box hc of K, U_V, V, U_K (this CTA's
            // output columns)
            const uint32_t A = tmem + kColDC + 64 * h + 16 * sub;
            const uint32_t k_rows = sb + soff<C::NSTREAM, kB4>(0, h, hc) + sub * 2048;
            if (part != 1) {
              // [B | dOtil0] += P [K | U_V]   (second 64-wide block at U_V)
              const uint64_t fKUV = sdesc_sw128(
                  k_rows,
                  soff<C::NSTREAM, kB4>(3, h, hc) - soff<C::NSTREAM, kB4>(0, h, hc),
                  1024);
              mma_ts(tmem + 0, A + 0, fKUV, id_b2, first);
              mma_ts(tmem + 64, A + 8, md(2, hc), id_b, 1);  // dOtil0 += (P o F) V
            }
            if (part != 0) {
              // [G | Omega] += dS [K | U_K] ;  Omega += (P o Pt0) K
              const uint64_t fKUK = sdesc_sw128(
                  k_rows,
                  soff<C::NSTREAM, kB4>(1, h, hc) - soff<C::NSTREAM, kB4>(0, h, hc),
                  1024);
              mma_ts(tmem + 128, A + 40, fKUK, id_b2, first);
              mma_ts(tmem + 192, A + 32, md(0, hc), id_b, 1);
            }
          } else if constexpr (kDirect) {
            // eqs. (6)-(7): Qtil += Stil K + dS U_K (part 1) ; dOtil += P U_V +
            // (P o h) V (part 0, issuer X's share with XSHARE)
            const uint32_t A = tmem + kColDC + 64 * h + 16 * sub;
            if (part != 0) {
              mma_ts(tmem + 0, A + 32, md(0, 0), id_b, first);
              mma_ts(tmem + 0, A + 40, md(1, 0), id_b, 1);
            }
            if (part != 1) {
              mma_ts(tmem + D, A + 0, md(3, 0), id_b, first);
              mma_ts(tmem + D, A + 8, md(2, 0), id_b, 1);
            }
          } else if constexpr (OP == RowOp::BwdDQ) {
            const uint32_t dcb = C::DC2 ? 64u * (uint32_t)(st & 1) : 0u;  // dP buffer of tile st
            mma_ts(tmem + 0, tmem + kColDC + dcb + 16 * s, md(0, 0), id_b, first);  // dQ += dS K
          }
        }
      };
      if (warp == kMmaWarp) {
        // ---------------- issuer X: SF(t) = scores (and F) of tile t, and
        // with C::XSHARE its share of stage B
        // part 1: [S | F] (and S alone); part 2: F += U_Q K^T; 0: both
        auto stage_sf = [&](int st, uint32_t col, int part = 0) {
          const int stage = st % C::NSTAGES;
          const uint64_t kd0 = sdesc_sw128(smem_u32(s_stream + stage * C::STAGE_BYTES), 16, 1024);
          const uint32_t R = tmem + col;
          if constexpr (C::STAT_TMEM) {  // the same with Q and U_Q from TMEM
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // [S | F] = Q [K ; U_K]^T
              mma_ts(R + 0, tmem + kColQT + 8 * k, kd(kd0, 0, 0, k), id_n128, k > 0);
#pragma unroll
            for (int k = 0; k < D / 32; ++k)  // F += U_Q K^T, first half of the K-steps
              mma_ts(R + 64, tmem + kColQT + D / 2 + 8 * k, kd(kd0, 0, 0, k), id_n64, 1);
          } else if constexpr (kB4) {
            // stationary: 0 Q, 1 U_Q, 2 dO ; stream: 0 K, 1 U_K, 2 V, 3 U_V
            if (part != 2) {
#pragma unroll
              for (int k = 0; k < D / 16; ++k)  // [S | F] = Q [K ; U_K]^T
                mma_ss(R + 0, sd(0, k), kd(kd0, 0, 0, k), id_n128, k > 0);
            }
            if (part != 1) {
#pragma unroll
              for (int k = 0; k < D / 16; ++k)  // F += U_Q K^T
                mma_ss(R + 64, sd(1, k), kd(kd0, 0, 0, k), id_n64, 1);
            }
          } else {
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // S = Q K^T
              mma_ss(R + 0, sd(0, k), kd(kd0, 0, 0, k), id_n64, k > 0);
          }
        };
        bool ok = mbar_wait(&m->bar_stat, 0, wctl);
        if constexpr (kStats) {
          // two SF buffers (tile t in buffer t & 1), so X runs up to a tile
          // ahead of the elementwise warps; no stage B, so a stage is released
          // as soon as the MMAs reading it complete.  Issuer Y adds the second
          // half of F += U_Q K^T once X's part has completed (12 MMAs per tile
          // on each issuer), and signals SF(t)
          for (int st = 0; ok && st < nsteps; ++st) {
            const int b = st & 1;
            const int stage = st % C::NSTAGES;
            if ((st >= 2 && !mbar_wait(&m->bar_sf_free[b], ((st - 2) >> 1) & 1, wctl)) ||
                !mbar_wait(&m->bar_full[stage], (st / C::NSTAGES) & 1, wctl))
              break;
            tc_fence_after();
            stage_sf(st, b ? kColSF1 : kColSF);
            mma_commit(&m->bar_xsig[b]);
            mma_commit(&m->bar_empty[stage]);
          }
          ok = false;
        }
        ok = ok && nsteps > 0 && mbar_wait(&m->bar_full[0], 0, wctl);
        if (ok) {
          tc_fence_after();
          stage_sf(0, kColSF);
          mma_commit(&m->bar_sa_sf[0]);
        }
        for (int st = 0; ok && st < nsteps; ++st) {
          const int stage = st % C::NSTAGES;
          const bool more = st + 1 < nsteps;
          // without XSHARE, X's last read of this stage was SF(t), already
          // issued: release the stage when that completes (a commit after
          // SF(t+1) would hold it until SF(t+1) completes, a tile later)
          if (!C::XSHARE) {
            if (C::HALF_REL) {
              mma_commit(&m->bar_empty[2 * stage]);
              mma_commit(&m->bar_empty[2 * stage + 1]);
            } else {
              mma_commit(&m->bar_empty[stage]);
            }
          }
          if (more) {  // SF(t+1) once the elementwise warps hold SF(t)
            if (!mbar_wait(&m->bar_sf_free[0], st & 1, wctl) ||
                !mbar_wait(&m->bar_full[(st + 1) % C::NSTAGES], ((st + 1) / C::NSTAGES) & 1, wctl))
              break;
            tc_fence_after();
            // with XSHARE only [S | F] now: X's stage-B share of half 0 goes
            // between the two parts, so that issuer Y's next DC (which waits
            // for that share) does not queue behind all of SF(t+1)
            stage_sf(st + 1, kColSF, C::XSHARE ? 1 : 0);
            if (!C::XSHARE) mma_commit(&m->bar_sa_sf[0]);
          }
          if constexpr (C::XSHARE) {
            // V and U_V of this stage (already observed by issuer Y; the wait
            // makes the acquire explicit)
            if (!mbar_wait(&m->bar_full_b[stage], (st / C::NSTAGES) & 1, wctl)) break;
            const uint32_t sb = smem_u32(s_stream + stage * C::STAGE_BYTES);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              if (!mbar_wait(&m->bar_ew[h], st & 1, wctl)) {
                ok = false;
                break;
              }
              tc_fence_after();
              stage_b(sb, h, st, 0);
              mma_commit(&m->bar_xb[h]);
              if (h == 0 && more) {
                stage_sf(st + 1, kColSF, 2);
                mma_commit(&m->bar_sa_sf[0]);
              }
            }
            if (!ok) break;
            mma_commit(&m->bar_empty[stage]);
          }
        }
        mma_commit(&m->bar_acc);
        if (*abort_flag) drain_wait(&m->bar_acc, 0);
      } else {
        // ---------------- issuer Y: DC(t) and the remaining stage-B MMAs
        auto stage_dc = [&](uint32_t sb, int h, uint32_t dcb = 0) {
          const uint64_t kd0 = sdesc_sw128(sb, 16, 1024);
          if constexpr (kStats) {  // whole tile: [dP_0|C_0|dP_1|C_1] = dO [V_0;U_V_0;V_1;U_V_1]^T
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // (dO is the one stationary tile in shared memory)
              mma_ss(tmem + kColDC, sd(0, k), kd(kd0, 2, 0, k), id_n128, k > 0);
          } else if constexpr (kB4 && kDcHalves) {  // [dP_h | C_h] = dO [V_h ; U_V_h]^T
#pragma unroll
            for (int k = 0; k < D / 16; ++k)
              mma_ss(tmem + kColDC + 64 * h, sd(2, k), kd(kd0, 2, h, k), id_n64, k > 0);
          } else if constexpr (kB4) {  // whole tile: [dP_0|C_0|dP_1|C_1] = dO [V_0;U_V_0;V_1;U_V_1]^T
#pragma unroll
            for (int k = 0; k < D / 16; ++k)
              mma_ss(tmem + kColDC, sd(2, k), kd(kd0, 2, 0, k), id_n128, k > 0);
          } else if constexpr (OP == RowOp::BwdDQ) {  // dP = dO V^T (whole tile)
#pragma unroll
            for (int k = 0; k < D / 16; ++k)
              mma_ss(tmem + kColDC + dcb, sd(1, k), kd(kd0, 1, 0, k), id_n64, k > 0);
          }
        };
        // issuer Y reads every streamed tensor: wait for both halves of a stage
        auto wait_stage = [&](int stg, uint32_t par) {
          return mbar_wait(&m->bar_full[stg], par, wctl) &&
                 (!kB4 || mbar_wait(&m->bar_full_b[stg], par, wctl));
        };
        bool ok = mbar_wait(&m->bar_stat, 0, wctl) && nsteps > 0 && wait_stage(0, 0);
        if constexpr (kStats) {
          // tile t: the second half of F += U_Q K^T once issuer X's part of
          // SF(t) has completed (then SF(t) is whole), and DC(t), for t + 1
          // once the elementwise warps hold DC(t) in registers
          auto tile_y = [&](int t) -> bool {
            const int b = t & 1;
            if (!mbar_wait(&m->bar_xsig[b], (t >> 1) & 1, wctl)) return false;
            tc_fence_after();
            const uint32_t sb = smem_u32(s_stream + (t % C::NSTAGES) * C::STAGE_BYTES);
            const uint64_t kd0 = sdesc_sw128(sb, 16, 1024);
            const uint32_t R = tmem + (b ? kColSF1 : kColSF);
#pragma unroll
            for (int k = D / 32; k < D / 16; ++k)  // F += U_Q K^T, second half
              mma_ts(R + 64, tmem + kColQT + D / 2 + 8 * k, kd(kd0, 0, 0, k), id_n64, 1);
            mma_commit(&m->bar_sa_sf[b]);
            stage_dc(sb, 0);
            mma_commit(&m->bar_sa_dc[0]);
            mma_commit(&m->bar_empty[t % C::NSTAGES]);
            return true;
          };
          if (ok) {
            tc_fence_after();
            ok = tile_y(0);
          }
          for (int st = 0; ok && st + 1 < nsteps; ++st) {
            const int ns = (st + 1) % C::NSTAGES;
            if (!mbar_wait(&m->bar_dc_free, st & 1, wctl) ||
                !wait_stage(ns, ((st + 1) / C::NSTAGES) & 1) || !tile_y(st + 1))
              break;
          }
          ok = false;  // no stage B
        }
        if constexpr (C::DC2) {
          // dP(t) in buffer t & 1 (columns kColDC + 64 (t & 1)), two tiles
          // ahead: dP(t+2) goes into the buffer stage B(t) has just read
          for (int t = 0; ok && t < 2 && t < nsteps; ++t) {
            if (t == 1) ok = wait_stage(1 % C::NSTAGES, (1 / C::NSTAGES) & 1);
            if (!ok) break;
            tc_fence_after();
            stage_dc(smem_u32(s_stream + (t % C::NSTAGES) * C::STAGE_BYTES), 0, 64u * t);
            mma_commit(&m->bar_sa_dc[t]);
          }
          for (int st = 0; ok && st < nsteps; ++st) {
            const int b = st & 1;
            const uint32_t par = (st >> 1) & 1;
            const int stage = st % C::NSTAGES;
            const uint32_t sb = smem_u32(s_stream + stage * C::STAGE_BYTES);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              if (!mbar_wait(&m->bar_ew[2 * b + h], par, wctl)) {
                ok = false;
                break;
              }
              tc_fence_after();
              stage_b(sb, h, st, 2);
            }
            if (!ok) break;
            mma_commit(&m->bar_empty[stage]);
            const int nx = st + 2;
            if (nx < nsteps) {
              if (!wait_stage(nx % C::NSTAGES, (nx / C::NSTAGES) & 1)) break;
              tc_fence_after();
              stage_dc(smem_u32(s_stream + (nx % C::NSTAGES) * C::STAGE_BYTES), 0, 64u * b);
              mma_commit(&m->bar_sa_dc[b]);
            }
          }
          ok = false;
        }
        if (ok) {
          tc_fence_after();
          const uint32_t sb0 = smem_u32(s_stream);
          stage_dc(sb0, 0);
          mma_commit(&m->bar_sa_dc[0]);
          if (kDcHalves) {
            stage_dc(sb0, 1);
            mma_commit(&m->bar_sa_dc[1]);
          }
        }
        for (int st = 0; ok && st < nsteps; ++st) {
          const int stage = st % C::NSTAGES;
          const uint32_t sb = smem_u32(s_stream + stage * C::STAGE_BYTES);
          const int nstage = (st + 1) % C::NSTAGES;
          const uint32_t nsb = smem_u32(s_stream + nstage * C::STAGE_BYTES);
          const bool more = st + 1 < nsteps;
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            if (!mbar_wait(&m->bar_ew[h], st & 1, wctl)) {
              ok = false;
              break;
            }
            tc_fence_after();
            stage_b(sb, h, st, C::XSHARE ? 1 : 2);
            // issuer Y's last read of the stage (of its half h with C::HALF_REL)
            if (C::HALF_REL)
              mma_commit(&m->bar_empty[2 * stage + h]);
            else if (h == 1)
              mma_commit(&m->bar_empty[stage]);
            if (more && (kDcHalves || h == 1)) {
              if ((h == 0 || !kDcHalves) && !wait_stage(nstage, ((st + 1) / C::NSTAGES) & 1)) {
                ok = false;
                break;
              }
              // DC(t+1) of half h overwrites the operand tiles that issuer
              // X's stage-B MMAs of half h read; wait for their completion
              if (C::XSHARE && !mbar_wait(&m->bar_xb[h], st & 1, wctl)) {
                ok = false;
                break;
              }
              tc_fence_after();
              stage_dc(nsb, kDcHalves ? h : 0);
              mma_commit(&m->bar_sa_dc[kDcHalves ? h : 0]);
            }
          }
        }
        mma_commit(&m->bar_acc);
        if (*abort_flag) drain_wait(&m->bar_acc, 0);
      }
    }
  } else {
    // ------------------------------------------------------------ elementwise
    const int wg = warp >> 2;                    // warpgroup 0/1
    const int r = 32 * (warp & 3) + (tid & 31);  // stationary row in the block
    const int gi = i0 + r;
    const bool row_ok = gi < N;
    // this row's valid keys [jlo, jhi): its band within its sequence (none past N)
    int jlo = 0, jhi = 0;
    if (row_ok) {
      seq_bounds(p, gi, jlo, jhi);
      if (p.wl >= 0) jlo = max(jlo, gi - p.wl);
      if (p.wr >= 0) jhi = min(jhi, gi + p.wr + 1);
    }
    const uint32_t ta = lane_base_addr(tmem, warp);
    const size_t rowoff = ((size_t)bh * N + (size_t)(row_ok ? gi : 0)) * DG;
    const float tau = p.scale;
    const float sl2 = tau * kLog2e;
    // dropout: keep bits of this row's 16 keys in each half of key tile jt
    // (computed before the tile's scores are waited for); gate sigma R
    const DropKey dkey = {p.drop_rk, p.drop_tlow4, p.drop_tmask};
    const float dsig = p.drop_sigma;
    auto tile_keep = [&](int jt, uint32_t (&kb)[2]) {
#pragma unroll
      for (int h = 0; h < 2; ++h)
        kb[h] = keep_row16(gi, jt + HB * h + 16 * wg, (uint32_t)(p.head0 + bh), dkey);
    };
    // with dropout the lanes of a warp exchange keep bits, so a wait that
    // gives up makes the whole warp leave together
    auto ew_wait = [&](uint64_t* bar, uint32_t par) -> bool {
      const bool w = mbar_wait(bar, par, wctl);
      if constexpr (DROP) return __all_sync(0xffffffffu, w);
      return w;
    };
    float L2 = 0.f, Dr = 0.f, nal = 0.f, nE = 0.f;  // nal = -alpha, nE = -E (direct form)
    {
      if (row_ok) {
        const size_t ri = (size_t)bh * N + gi;
        L2 = p.lse[ri] * kLog2e;
        if constexpr (kDirect) {  // row scalars written by the statistics kernel
          nal = -p.vec_in[ri];
          nE = -p.vec_in[p.bhn + ri];
          Dr = p.vec_in[2 * p.bhn + ri];
        }
      }
    }
    // D = do . o (the statistics kernel first puts Q and U_Q into TMEM, so
    // that issuer X can start while D is summed)
    if constexpr (!kDirect && !C::STAT_TMEM)
      Dr = block_row_dots<DG>(p.dout, p.o, (size_t)bh * N * DG, i0, N, s_d, tid);
    if constexpr (C::STAT_TMEM) {
      // stationary rows straight into TMEM as MMA A operands (word c of a
      // bf16 row = elements 2c, 2c+1 = column c of its operand): warpgroup 0
      // writes Q, warpgroup 1 U_Q
      // (every load of the row first, so the CTA waits for one memory round
      // trip instead of one per 8 columns)
      auto put_row = [&](const __nv_bfloat16* row, uint32_t col) {
        const uint4* src = reinterpret_cast<const uint4*>(row);
        uint4 v[D / 8];  // the row's D bf16 values, 8 per uint4
#pragma unroll
        for (int u = 0; u < D / 8; ++u)  // zero columns past the tensor's head dim
          v[u] = (row_ok && 8 * u < DG) ? src[u] : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int c = 0; c < D / 2; c += 8) {
          const uint4 a = v[c / 4], b = v[c / 4 + 1];
          const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
          tmem_st8(ta + col + c, w);
        }
      };
      put_row((wg == 0 ? p.q : p.uq) + rowoff, kColQT + wg * (D / 2));
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&m->bar_stat);
      Dr = block_row_dots<DG>(p.dout, p.o, (size_t)bh * N * DG, i0, N, s_d, tid);
    }
    float2 acc_a = splat(0.f), acc_e = splat(0.f);  // Pass 1 partial row sums
    bool ok = true;
    int tile = first_tile - 1;
    for (int st = 0; ok && st < nsteps; ++st) {
      tile = tiles.next(tile + 1);
      const int jt = tile * BN;  // first key of the tile
      // SF buffer of this tile (the statistics kernel alternates two)
      const int sfb = kStats ? (st & 1) : 0;
      const uint32_t sfcol = sfb ? kColSF1 : kColSF;
      uint32_t kb[2];
      if constexpr (DROP) tile_keep(jt, kb);
      if (!ew_wait(&m->bar_sa_sf[sfb], kStats ? ((st >> 1) & 1) : (st & 1))) {
        ok = false;
        break;
      }
      tc_fence_after();
      // ---- copy this thread's SF columns of both halves, then release SF
      uint32_t rS[2][16], rF[2][16];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        tmem_ld16(ta + sfcol + HB * h + 16 * wg, rS[h]);
        if constexpr (kB4) tmem_ld16(ta + sfcol + 64 + HB * h + 16 * wg, rF[h]);
      }
      tmem_ld_wait(rS[0]);
      reg_dep(rS[1]);
      if constexpr (kB4) {
        reg_dep(rF[0]);
        reg_dep(rF[1]);
      }
      tc_fence_before();
      mbar_arrive(&m->bar_sf_free[sfb]);
      const float2 sl2v = splat(sl2), nL2v = splat(-L2);
      if constexpr (kStats) {
        // ---- row statistics: copy DC of the whole tile, release it, then
        // accumulate alpha = sum P F and E0 = sum P (C + F (dP - D))  (eq. 6)
        if (!ew_wait(&m->bar_sa_dc[0], st & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t rdP[2][16], rC[2][16];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          tmem_ld16(ta + kColDC + 64 * h + 16 * wg, rdP[h]);
          tmem_ld16(ta + kColDC + 64 * h + 32 + 16 * wg, rC[h]);
        }
        tmem_ld_wait(rdP[0]);
        reg_dep(rdP[1]);
        reg_dep(rC[0]);
        reg_dep(rC[1]);
        tc_fence_before();
        mbar_arrive(&m->bar_dc_free);
        const float2 tauv = splat(tau), nDv = splat(-Dr);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int j0 = jt + HB * h + 16 * wg;
          const int mlo = jlo - j0, mhi = jhi - j0;  // valid columns: mlo <= c < mhi
          if (mlo > 0 || mhi < 16) mask16(rS[h], mlo, mhi);
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            const float2 pr = probs2(pair(rS[h], c), sl2v, nL2v);
            const float2 f = __fmul2_rn(pair(rF[h], c), tauv);
            float2 dp = pair(rdP[h], c), cv = pair(rC[h], c);
            if constexpr (DROP) {  // dP -> sigma R dP, C -> sigma R C
              const float2 g = gate2(kb[h], c, dsig);
              dp = __fmul2_rn(dp, g);
              cv = __fmul2_rn(cv, g);
            }
            const float2 t = __fadd2_rn(dp, nDv);
            const float2 pt0 = __ffma2_rn(f, t, cv);  // Ptil0 = C + F (dP - D)
            acc_a = __ffma2_rn(pr, f, acc_a);
            acc_e = __ffma2_rn(pr, pt0, acc_e);
          }
        }
      } else {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          // (the dQ kernel alternates two dP buffers: buffer st & 1, phase st >> 1)
          const int dcbi = C::DC2 ? (st & 1) : 0;
          if (kDcHalves || h == 0) {
            if (!ew_wait(&m->bar_sa_dc[kDcHalves ? h : dcbi],
                         C::DC2 ? ((st >> 1) & 1) : (st & 1))) {
              ok = false;
              break;
            }
            tc_fence_after();
          }
          const int c0 = HB * h + 16 * wg;  // tile column of this thread's 16
          const int j0 = jt + c0;           // first key of this thread's 16
          const int mlo = jlo - j0, mhi = jhi - j0;  // valid columns: mlo <= c < mhi
          if (mlo > 0 || mhi < 16) mask16(rS[h], mlo, mhi);
          if constexpr (kBob) {
            const uint32_t R = ta + kColDC + 64 * h + 16 * wg;  // [dP_h | C_h] columns
            uint32_t rdP[16], rC[16];
            tmem_ld16(R + 0, rdP);
            tmem_ld16(R + 32, rC);
            tmem_ld_wait(rdP);
            reg_dep(rC);
            const float2 tauv = splat(tau), nDv = splat(-Dr);
            uint32_t oP[8], oPF[8], oPPt[8], odS[8];
#pragma unroll
            for (int c = 0; c < 16; c += 2) {
              const float2 pr = probs2(pair(rS[h], c), sl2v, nL2v);
              const float2 f = __fmul2_rn(pair(rF[h], c), tauv);
              const float2 dp = pair(rdP, c);
              const float2 t = __fadd2_rn(dp, nDv);
              const float2 pt0 = __ffma2_rn(f, t, pair(rC, c));  // Ptil0 = C + F (dP - D)
              const float2 pf = __fmul2_rn(pr, f);
              const float2 ppt = __fmul2_rn(pr, pt0);
              const float2 ds = __fmul2_rn(pr, t);
              acc_a = __fadd2_rn(acc_a, pf);
              acc_e = __fadd2_rn(acc_e, ppt);
              oP[c / 2] = pack_bf16(pr.x, pr.y);
              oPF[c / 2] = pack_bf16(pf.x, pf.y);
              oPPt[c / 2] = pack_bf16(ppt.x, ppt.y);
              odS[c / 2] = pack_bf16(ds.x, ds.y);
            }
            tmem_st8(R + 0, oP);
            tmem_st8(R + 8, oPF);
            tmem_st8(R + 32, oPPt);
            tmem_st8(R + 40, odS);
          } else if constexpr (kDirect) {
            const uint32_t R = ta + kColDC + 64 * h + 16 * wg;  // [dP_h | C_h] columns
            uint32_t rdP[16], rC[16];
            tmem_ld16(R + 0, rdP);
            tmem_ld16(R + 32, rC);
            tmem_ld_wait(rdP);
            reg_dep(rC);
            const float2 tauv = splat(tau), nDv = splat(-Dr), nalv = splat(nal), nEv = splat(nE);
            uint32_t oP[8], oPh[8], oSt[8], odS[8];
#pragma unroll
            for (int c = 0; c < 16; c += 2) {
              const float2 pr = probs2(pair(rS[h], c), sl2v, nL2v);
              const float2 f = __fmul2_rn(pair(rF[h], c), tauv);
              float2 dp = pair(rdP, c), cv = pair(rC, c), gp = pr;
              if constexpr (DROP) {  // dP, C and the dOtil operands gated by sigma R
                const float2 g = gate2(kb[h], c, dsig);
                dp = __fmul2_rn(dp, g);
                cv = __fmul2_rn(cv, g);
                gp = __fmul2_rn(pr, g);
              }
              const float2 t = __fadd2_rn(dp, nDv);
              // Ptil = C + F (dP - D) - alpha dP ; Stil = P (Ptil - E) ; h = F - alpha
              const float2 pt = __ffma2_rn(nalv, dp, __ffma2_rn(f, t, cv));
              const float2 ph = __fmul2_rn(gp, __fadd2_rn(f, nalv));
              const float2 stl = __fmul2_rn(pr, __fadd2_rn(pt, nEv));
              const float2 ds = __fmul2_rn(pr, t);
              oP[c / 2] = pack_bf16(gp.x, gp.y);
              oPh[c / 2] = pack_bf16(ph.x, ph.y);
              oSt[c / 2] = pack_bf16(stl.x, stl.y);
              odS[c / 2] = pack_bf16(ds.x, ds.y);
            }
            tmem_st8(R + 0, oP);
            tmem_st8(R + 8, oPh);
            tmem_st8(R + 32, oSt);
            tmem_st8(R + 40, odS);
          } else if constexpr (OP == RowOp::BwdDQ) {
            const uint32_t R = ta + kColDC + 64 * dcbi + c0;
            uint32_t rdP[16];
            tmem_ld16(R, rdP);
            tmem_ld_wait(rdP);
            const float2 nDv = splat(-Dr);
            uint32_t odS[8];
#pragma unroll
            for (int c = 0; c < 16; c += 2) {
              const float2 pr = probs2(pair(rS[h], c), sl2v, nL2v);
              float2 dp = pair(rdP, c);
              if constexpr (DROP) dp = __fmul2_rn(dp, gate2(kb[h], c, dsig));
              const float2 ds = __fmul2_rn(pr, __fadd2_rn(dp, nDv));
              odS[c / 2] = pack_bf16(ds.x, ds.y);
            }
            tmem_st8(R, odS);
          }
          tmem_st_wait();
          tc_fence_before();
          mbar_arrive(&m->bar_ew[C::DC2 ? 2 * dcbi + h : h]);
        }
      }
    }
    // ---------------------------------------------------------- epilogue
    if (ok) ok = mbar_wait(&m->bar_acc, 0, wctl);
    if (ok && *abort_flag) ok = false;
    tc_fence_after();
    if constexpr (kBob || kStats) {
      s_xchg[wg * BM + r] = acc_a.x + acc_a.y;
      s_xchg[(2 + wg) * BM + r] = acc_e.x + acc_e.y;
      named_bar_sync(1, kEwThreads);
    }
    if (ok) {
      if constexpr (OP == RowOp::BobPass1) {
        const float alpha = s_xchg[r] + s_xchg[BM + r];
        const float E0 = s_xchg[2 * BM + r] + s_xchg[3 * BM + r];
        const float E = E0 - alpha * Dr;  // eq. (8): E = E0 - alpha D
        const int cbase = 64 * hc + 32 * wg;  // output column of accumulator column 32 wg
#pragma unroll 1
        for (int q = 0; q < 2; ++q) {
          const int cc = 32 * wg + 16 * q;  // accumulator column (0..63)
          // accumulators: B at 0, dOtil0 at 64, G at 128, Omega at 192
          uint32_t rB[16], rO[16], rG[16], rW[16];
          tmem_ld16(ta + 0 + cc, rB);
          tmem_ld16(ta + 64 + cc, rO);
          tmem_ld16(ta + 128 + cc, rG);
          tmem_ld16(ta + 192 + cc, rW);
          tmem_ld_wait(rB);
          reg_dep(rO);
          reg_dep(rG);
          reg_dep(rW);
          if (row_ok && cbase + 16 * q < DG) {
            float ov[16], qt[16], dot[16];
            load_row16(p.o + rowoff + cbase + 16 * q, ov);
#pragma unroll
            for (int c = 0; c < 16; ++c) {
              // eq. (8) with R = G + D B (G = sum_j dS_ij k_j) and E + alpha D = E0:
              // Qtil = tau (Omega - alpha G - E0 B), dOtil = dOtil0 - alpha o
              qt[c] = tau * (bits_f(rW[c]) - alpha * bits_f(rG[c]) - E0 * bits_f(rB[c]));
              dot[c] = bits_f(rO[c]) - alpha * ov[c];
            }
            store_row16(p.out0 + rowoff + cbase + 16 * q, qt);
            store_row16(p.out1 + rowoff + cbase + 16 * q, dot);
          }
        }
        if (row_ok && wg == 0 && hc == 0) {
          const size_t ri = (size_t)bh * N + gi;
          p.vec_out[ri] = alpha;
          p.vec_out[p.bhn + ri] = E;
          p.vec_out[2 * p.bhn + ri] = Dr;
        }
      } else if constexpr (kStats) {
        if (row_ok && wg == 0) {
          const float alpha = s_xchg[r] + s_xchg[BM + r];
          const float E0 = s_xchg[2 * BM + r] + s_xchg[3 * BM + r];
          const size_t ri = (size_t)bh * N + gi;
          p.vec_out[ri] = alpha;
          p.vec_out[p.bhn + ri] = E0 - alpha * Dr;  // E = E0 - alpha D
          p.vec_out[2 * p.bhn + ri] = Dr;
        }
      } else if constexpr (kDirect) {
        // Qtil = tau * acc[0, D), dOtil = acc[D, 2D); columns [wg*D/2, +D/2)
#pragma unroll 1
        for (int q = 0; q < D / 32; ++q) {
          const int cc = wg * (D / 2) + 16 * q;
          uint32_t rQ[16], rO[16];
          tmem_ld16(ta + cc, rQ);
          tmem_ld16(ta + D + cc, rO);
          tmem_ld_wait(rQ);
          reg_dep(rO);
          if (row_ok && cc < DG) {
            float qt[16], dot[16];
#pragma unroll
            for (int c = 0; c < 16; ++c) {
              qt[c] = tau * bits_f(rQ[c]);
              dot[c] = bits_f(rO[c]);
            }
            store_row16(p.out0 + rowoff + cc, qt);
            store_row16(p.out1 + rowoff + cc, dot);
          }
        }
      } else {
        // dQ = tau * acc (first backward), columns [wg*D/2, +D/2), and D
#pragma unroll 1
        for (int q = 0; q < D / 32; ++q) {
          const int cc = wg * (D / 2) + 16 * q;
          uint32_t rA[16];
          tmem_ld16(ta + cc, rA);
          tmem_ld_wait(rA);
          if (row_ok && cc < DG) {
            float v[16];
#pragma unroll
            for (int c = 0; c < 16; ++c) v[c] = tau * bits_f(rA[c]);
            store_row16(p.out0 + rowoff + cc, v);
          }
        }
        if (row_ok && wg == 0) p.vec_out[(size_t)bh * N + gi] = Dr;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ============================================================ column engine
// D, DG as in the row engine; DROP: attention dropout (App. "Extensions")
template <ColOp OP, int D, bool DROP, int DG>
__global__ void __launch_bounds__(kThreads, 1) col_engine(const __grid_constant__ EngineParams p) {
  using C = ColCfg<OP, D>;
  static_assert(DG == D || (DG == 32 && D == 64), "global head dim 32 runs in 64-wide tiles");
  static_assert(C::NSTAGES >= 2 && C::NSTAGES <= kMaxStages, "the stage barriers hold kMaxStages stages");
  constexpr bool kBob = OP == ColOp::BobPass2;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* s_stat = smem;
  uint8_t* s_stream = smem + C::STAT_BYTES;
  Misc* m = reinterpret_cast<Misc*>(s_stream + C::NSTAGES * C::STAGE_BYTES);

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  if ((smem_u32(smem) & 1023u) != 0) {
    if (tid == 0) atomicOr(&g_fbob_error_word, kDevErrBadLaunch);
    return;
  }
  // ---- tile decode (as in the row engine); key block 0 has the most work
  // under the causal mask
  // DC buffer of tile t, and the phase parity of its per-buffer barriers
  auto dc_sel = [](int t) -> int { return C::DC2 ? (t & 1) : 0; };
  auto dc_col = [](int t) -> uint32_t { return (C::DC2 && (t & 1)) ? C::DC1_COL : kColDC; };
  auto dc_par = [](int t) -> uint32_t { return C::DC2 ? ((t >> 1) & 1) : (t & 1); };
  const int N = p.N;
  const int lin = blockIdx.x;
  int cb, bh;
  cta_order(p, lin, cb, bh);
  const int j0 = cb * BM;
  // streamed query tiles: rows whose band holds a key of this block,
  // j - wr <= i <= j + wl (negative w: unbounded; causal: wr = 0)
  // (within the keys' packed sequences)
  const int last_key = min(j0 + BM, N) - 1;
  int seq_lo0, seq_hi0, seq_lo1, seq_hi1;
  seq_bounds(p, j0, seq_lo0, seq_hi0);
  seq_bounds(p, last_key, seq_lo1, seq_hi1);
  const int q_lo = max(seq_lo0, p.wr < 0 ? 0 : j0 - p.wr);
  const int q_hi = min(seq_hi1, p.wl < 0 ? N : last_key + p.wl + 1);  // exclusive
  const int first_tile = q_lo / BN;
  // query tiles per query head (with a block-sparse mask only the tiles of
  // the query blocks set in this key block's mask column)
  const TileSet tiles = {p.bmask ? p.bmask + cb : nullptr, p.nbm, first_tile, (q_hi - 1) / BN};
  const int nsteps_h = tiles.count();
  // grouped-query attention: this key/value head's G query heads are streamed
  // one after the other (their sums accumulate in this CTA, in a fixed order)
  const int G = p.H / p.Hkv;
  const int bh_q0 = (bh / p.Hkv) * p.H + (bh % p.Hkv) * G;  // first query head
  const int nsteps = G * nsteps_h;

  if (tid == 0) {
    m->wctl.abort = 0;
    m->wctl.limit_ns = p.wait_limit_ns;
    mbar_init(&m->bar_stat, 1);
    for (int s = 0; s < C::NSTAGES; ++s) {
      mbar_init(&m->bar_full[s], 1);         // Q (and U_Q): all issuer X needs
      mbar_init(&m->bar_full_b[s], 1 + 32);  // dO + 32 producer lanes' row vectors
      mbar_init(&m->bar_empty[s], 2);        // released by both MMA issuers
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&m->bar_sa_sf[b], 1);
      mbar_init(&m->bar_sf_free[b], kEwThreads);
    }
    for (int h = 0; h < 2; ++h) {
      mbar_init(&m->bar_sa_dc[h], 1);
      mbar_init(&m->bar_xb[h], 1);
      mbar_init(&m->bar_xsig[h], 1);
    }
    for (int h = 0; h < 4; ++h) mbar_init(&m->bar_ew[h], kEwThreads);
    mbar_init(&m->bar_acc, 2);
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&m->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = m->tmem_base;
  WaitCtl* wctl = &m->wctl;
  volatile int* abort_flag = &m->wctl.abort;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------ producer
    // (p.inject_stall: no loads at all, as in the row engine)
    const int lane = tid & 31;
    const int nprod = p.inject_stall ? 0 : nsteps;
    if (lane == 0 && !p.inject_stall) {
      for (int t = 0; t < C::NSTAT + C::NSTREAM; ++t) tma_prefetch_desc(&p.tm[t]);
      mbar_arrive_expect_tx(&m->bar_stat, C::STAT_BYTES);
      for (int t = 0; t < C::NSTAT; ++t)
        for (int b = 0; b < C::KB; ++b)
          tma_load_3d(s_stat + (t * C::KB + b) * (BM * 128), &p.tm[t], &m->bar_stat, 64 * b, j0,
                      bh);
    }
    int issued[kMaxStages] = {-1, -1, -1, -1};
    // query tile and head of step st (the tile cursor restarts for each of
    // the key/value head's query heads)
    int tile = first_tile - 1;
    auto advance = [&](int st, int& ib, int& bhq) {
      if (st % nsteps_h == 0) tile = first_tile - 1;
      tile = tiles.next(tile + 1);
      ib = tile * BN;
      bhq = bh_q0 + st / nsteps_h;
    };
    // row vectors of a step's streamed query rows, two rows per lane, as
    // loaded: [0] L, [1] D, [2] alpha, [3] E (the first backward: L, D).
    // They are loaded one step ahead and only written (negated, L scaled by
    // log2 e) into the stage at the next step: no arithmetic touches them
    // here, so the loads stay in flight while the producer moves on (a use
    // right after the load would stall the producer for the whole load
    // latency every step).  Rows past N read the head's last row; the write
    // zeroes them.
    constexpr int NV = C::NVEC;
    auto load_vec = [&](int ib, int bhq, float (&v)[2][NV]) {
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const size_t ri = (size_t)bhq * N + min(ib + lane + 32 * q, N - 1);
        v[q][0] = p.lse[ri];
        if constexpr (OP == ColOp::BwdDKDV) {
          v[q][1] = p.vec_in[ri];
        } else {
          v[q][1] = p.vec_in[2 * p.bhn + ri];  // D
          v[q][2] = p.vec_in[ri];              // alpha
          v[q][3] = p.vec_in[p.bhn + ri];      // E
        }
      }
    };
    int ib_n = 0, bhq_n = 0;
    float vn[2][NV];
    if (nprod > 0) {
      advance(0, ib_n, bhq_n);
      load_vec(ib_n, bhq_n, vn);
    }
    for (int st = 0; st < nprod; ++st) {
      const int stage = st % C::NSTAGES;
      if (st >= C::NSTAGES) {
        if (!mbar_wait(&m->bar_empty[stage], ((st / C::NSTAGES) - 1) & 1, wctl)) break;
      }
      const int ib = ib_n, bhq = bhq_n;  // this step's query tile and head
      uint8_t* dst = s_stream + stage * C::STAGE_BYTES;
      if (lane == 0) {
        // Q (and U_Q) first on bar_full, dO on bar_full_b
        constexpr int na = C::NSTREAM - 1;
        mbar_arrive_expect_tx(&m->bar_full[stage], na * C::KB * BN * 128);
        for (int b = 0; b < C::KB; ++b)
          for (int t = 0; t < na; ++t)
            tma_load_3d(dst + soff<C::NSTREAM, false>(t, 0, b), &p.tm[C::NSTAT + t],
                        &m->bar_full[stage], 64 * b, ib, bhq);
        mbar_arrive_expect_tx(&m->bar_full_b[stage], C::KB * BN * 128);
        for (int b = 0; b < C::KB; ++b)
          tma_load_3d(dst + soff<C::NSTREAM, false>(na, 0, b), &p.tm[C::NSTAT + na],
                      &m->bar_full_b[stage], 64 * b, ib, bhq);
      }
      float* vec = reinterpret_cast<float*>(dst + C::TILE_BYTES);
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const bool ok = ib + lane + 32 * q < N;
#pragma unroll
        for (int k = 0; k < NV; ++k)
          vec[64 * k + lane + 32 * q] = ok ? -(k == 0 ? vn[q][k] * kLog2e : vn[q][k]) : 0.f;
      }
      mbar_arrive(&m->bar_full_b[stage]);
      issued[stage] = st;
      if (st + 1 < nprod) {  // the next step's coordinates and row vectors
        advance(st + 1, ib_n, bhq_n);
        load_vec(ib_n, bhq_n, vn);
      }
    }
    if (lane == 0 && *abort_flag) {
      for (int s = 0; s < C::NSTAGES; ++s)
        if (issued[s] >= 0) {
          drain_wait(&m->bar_full[s], (issued[s] / C::NSTAGES) & 1);
          drain_wait(&m->bar_full_b[s], (issued[s] / C::NSTAGES) & 1);
        }
      drain_wait(&m->bar_stat, 0);
    }
  } else if (warp == kMmaWarp || warp == kMmaWarpY) {
    // ------------------------------------------------------------ MMA issuers
    if (elect_lane0()) {
      constexpr uint32_t id_n64 = idesc_bf16(128, 64, false);
      constexpr uint32_t id_n128 = idesc_bf16(128, 128, false);
      constexpr uint32_t id_b = idesc_bf16(128, D, true);
      const uint64_t sd0 = sdesc_sw128(smem_u32(s_stat), 16, 1024);
      auto sd = [&](int t, int k) -> uint64_t {
        return sd0 + (uint64_t)(((t * C::KB + k / 4) * (BM * 128) + (k % 4) * 32) >> 4);
      };
      auto kd = [&](uint64_t kd0, int t, int k) -> uint64_t {
        return kd0 + (uint64_t)((soff<C::NSTREAM, false>(t, 0, k / 4) + (k % 4) * 32) >> 4);
      };
      // stage B of half h (K-steps s = 2h + sub).  With C::XSHARE issuer X
      // takes the MMAs into the value accumulator (part 0) and issuer Y those
      // into the key accumulator (part 1); otherwise Y takes them all (part 2).
      auto stage_b = [&](uint32_t sb, int h, int st, int part) {
        constexpr uint32_t kBoxBytes = C::NSTREAM * BN * 128;
        const uint32_t dcol = dc_col(st);
        const uint64_t md0 = sdesc_sw128(sb, kBoxBytes, 1024);
#pragma unroll
        for (int sub = 0; sub < 2; ++sub) {
          const int s = 2 * h + sub;
          auto md = [&](int t) -> uint64_t {
            return md0 + (uint64_t)((soff<C::NSTREAM, false>(t, h, 0) + sub * 2048) >> 4);
          };
          const uint32_t first = (st == 0 && s == 0) ? 0u : 1u;
          const uint32_t A = tmem + dcol + 16 * s;
          if constexpr (kBob) {
            if (part != 1) mma_ts(tmem + D, A + 0, md(2), id_b, first);  // Vtil += (P o h)^T dO
            if (part != 0) {
              mma_ts(tmem + 0, A + 8, md(0), id_b, first);  // Ktil += Stil^T Q
              mma_ts(tmem + 0, A + 64, md(1), id_b, 1);     //      += dS^T U_Q
            }
          } else {
            if (part != 1) mma_ts(tmem + D, A + 0, md(1), id_b, first);  // dV += P^T dO
            if (part != 0) mma_ts(tmem + 0, A + 8, md(0), id_b, first);  // dK += dS^T Q
          }
        }
      };
      if (warp == kMmaWarp) {
        // ---------------- issuer X: SF(t) = transposed scores (and F), and
        // with C::XSHARE the stage-B MMAs into the value accumulator
        auto stage_sf = [&](int st) {
          const int stage = st % C::NSTAGES;
          const uint64_t kd0 = sdesc_sw128(smem_u32(s_stream + stage * C::STAGE_BYTES), 16, 1024);
          const uint32_t R = tmem + kColSF;
          if constexpr (kBob) {
            // stationary: 0 K, 1 V, 2 U_K, 3 U_V ; stream: 0 Q, 1 U_Q, 2 dO
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // [S^T | F^T] = K [Q ; U_Q]^T
              mma_ss(R + 0, sd(0, k), kd(kd0, 0, k), id_n128, k > 0);
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // F^T += U_K Q^T
              mma_ss(R + 64, sd(2, k), kd(kd0, 0, k), id_n64, 1);
          } else {
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // S^T = K Q^T
              mma_ss(R + 0, sd(0, k), kd(kd0, 0, k), id_n64, k > 0);
          }
        };
        // with C::PH_SF: Vtil(t) += (P o h)^T dO from the operand tile the
        // elementwise warps wrote into SF (K-step s at SF column 16 s)
        auto stage_vt = [&](uint32_t sb, int st) {
          constexpr uint32_t kBoxBytes = C::NSTREAM * BN * 128;
          const uint64_t md0 = sdesc_sw128(sb, kBoxBytes, 1024);
#pragma unroll
          for (int s = 0; s < 4; ++s) {
            const uint64_t md =
                md0 + (uint64_t)((soff<C::NSTREAM, false>(2, s >> 1, 0) + (s & 1) * 2048) >> 4);
            mma_ts(tmem + D, tmem + kColSF + 16 * s, md, id_b, (st == 0 && s == 0) ? 0u : 1u);
          }
        };
        bool ok = mbar_wait(&m->bar_stat, 0, wctl) && nsteps > 0 &&
                  mbar_wait(&m->bar_full[0], 0, wctl);
        if (ok) {
          tc_fence_after();
          stage_sf(0);
          mma_commit(&m->bar_sa_sf[0]);
        }
        for (int st = 0; ok && st < nsteps; ++st) {
          const int stage = st % C::NSTAGES;
          if constexpr (C::PH_SF) {
            // the elementwise warps hold SF(t) in registers and have written
            // P o h over it: Vtil(t), then SF(t+1) (in issue order, so SF(t+1)
            // overwrites the operand tile only after Vtil(t) has read it)
            if (!mbar_wait(&m->bar_sf_free[0], st & 1, wctl) ||
                !mbar_wait(&m->bar_full_b[stage], (st / C::NSTAGES) & 1, wctl))
              break;
            tc_fence_after();
            stage_vt(smem_u32(s_stream + stage * C::STAGE_BYTES), st);
            // X's last read of this stage: release it once Vtil(t) has read it
            mma_commit(&m->bar_empty[stage]);
            if (st + 1 < nsteps) {
              if (!mbar_wait(&m->bar_full[(st + 1) % C::NSTAGES], ((st + 1) / C::NSTAGES) & 1,
                             wctl))
                break;
              tc_fence_after();
              stage_sf(st + 1);
              mma_commit(&m->bar_sa_sf[0]);
              // SF(t+1) is in the tensor pipe ahead of issuer Y's MMAs of tile t
              mbar_arrive(&m->bar_xsig[st & 1]);
            }
            continue;
          }
          // without XSHARE, X's last read of this stage was SF(t): release it
          // when that completes, not after SF(t+1) as well
          if (!C::XSHARE) mma_commit(&m->bar_empty[stage]);
          if (st + 1 < nsteps) {  // SF(t+1) once the elementwise warps hold SF(t)
            if (!mbar_wait(&m->bar_sf_free[0], st & 1, wctl) ||
                !mbar_wait(&m->bar_full[(st + 1) % C::NSTAGES], ((st + 1) / C::NSTAGES) & 1, wctl))
              break;
            tc_fence_after();
            stage_sf(st + 1);
            mma_commit(&m->bar_sa_sf[0]);
          }
          if constexpr (C::XSHARE) {
            // dO of this stage (already observed by issuer Y; explicit acquire)
            if (!mbar_wait(&m->bar_full_b[stage], (st / C::NSTAGES) & 1, wctl)) break;
            const uint32_t sb = smem_u32(s_stream + stage * C::STAGE_BYTES);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              if (!mbar_wait(&m->bar_ew[2 * dc_sel(st) + h], dc_par(st), wctl)) {
                ok = false;
                break;
              }
              tc_fence_after();
              stage_b(sb, h, st, 0);
            }
            if (!ok) break;
            mma_commit(&m->bar_xb[dc_sel(st)]);
            mma_commit(&m->bar_empty[stage]);
          }
        }
        mma_commit(&m->bar_acc);
        if (*abort_flag) drain_wait(&m->bar_acc, 0);
      } else {
        // ---------------- issuer Y: DC(t) and the key-accumulator MMAs
        // DC(t) of streamed tile t (stage buffer of tile t) into its DC buffer
        auto stage_dc = [&](int t) {
          const uint64_t kd0 =
              sdesc_sw128(smem_u32(s_stream + (t % C::NSTAGES) * C::STAGE_BYTES), 16, 1024);
          const uint32_t dcol = tmem + dc_col(t);
          if constexpr (kBob) {
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // dP^T = V dO^T
              mma_ss(dcol, sd(1, k), kd(kd0, 2, k), id_n64, k > 0);
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // C^T = U_V dO^T
              mma_ss(dcol + 64, sd(3, k), kd(kd0, 2, k), id_n64, k > 0);
          } else {
#pragma unroll
            for (int k = 0; k < D / 16; ++k)  // dP^T = V dO^T
              mma_ss(dcol, sd(1, k), kd(kd0, 1, k), id_n64, k > 0);
          }
          mma_commit(&m->bar_sa_dc[dc_sel(t)]);
        };
        auto wait_stage = [&](int stg, uint32_t par) {
          return mbar_wait(&m->bar_full[stg], par, wctl) &&
                 mbar_wait(&m->bar_full_b[stg], par, wctl);
        };
        // with two DC buffers DC runs two tiles ahead of stage B: DC(t+2) is
        // issued right after stage B(t), whose operand tiles it overwrites
        constexpr int kAhead = C::DC2 ? 2 : 1;
        bool ok = mbar_wait(&m->bar_stat, 0, wctl);
        for (int t = 0; ok && t < kAhead && t < nsteps; ++t) {
          ok = wait_stage(t % C::NSTAGES, (t / C::NSTAGES) & 1);
          if (ok) {
            tc_fence_after();
            stage_dc(t);
          }
        }
        for (int st = 0; ok && st < nsteps; ++st) {
          const int stage = st % C::NSTAGES;
          const uint32_t sb = smem_u32(s_stream + stage * C::STAGE_BYTES);
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            if (!mbar_wait(&m->bar_ew[2 * dc_sel(st) + h], dc_par(st), wctl)) {
              ok = false;
              break;
            }
            tc_fence_after();
            stage_b(sb, h, st, (C::XSHARE || C::PH_SF) ? 1 : 2);
          }
          if (!ok) break;
          mma_commit(&m->bar_empty[stage]);
          const int nx = st + kAhead;
          if (nx < nsteps) {
            // DC(nx) overwrites the operand tiles of tile st; with XSHARE wait
            // for issuer X's stage-B MMAs on them as well as for the stage
            if (!wait_stage(nx % C::NSTAGES, (nx / C::NSTAGES) & 1) ||
                (C::XSHARE && !mbar_wait(&m->bar_xb[dc_sel(st)], dc_par(st), wctl)))
              break;
            // with P o h in SF: the elementwise warps wait for SF(t+1) first and
            // DC(t+1) only after P o h, so DC(t+1) enters the pipe after SF(t+1)
            if (C::PH_SF && !mbar_wait(&m->bar_xsig[st & 1], (st >> 1) & 1, wctl)) break;
            tc_fence_after();
            stage_dc(nx);
          }
        }
        mma_commit(&m->bar_acc);
        if (*abort_flag) drain_wait(&m->bar_acc, 0);
      }
    }
  } else {
    // ------------------------------------------------------------ elementwise
    const int wg = warp >> 2;
    const int r = 32 * (warp & 3) + (tid & 31);
    const int gj = j0 + r;  // stationary key row
    const bool row_ok = gj < N;
    // query rows that see this key: [qlo, qhi), within its sequence (none past N)
    int qlo = 0, qhi = 0;
    if (row_ok) {
      seq_bounds(p, gj, qlo, qhi);
      if (p.wr >= 0) qlo = max(qlo, gj - p.wr);
      if (p.wl >= 0) qhi = min(qhi, gj + p.wl + 1);
    }
    const uint32_t ta = lane_base_addr(tmem, warp);
    const float tau = p.scale;
    const float2 sl2v = splat(tau * kLog2e), tauv = splat(tau);
    // dropout: keep bits of this key's 16 queries in each half of a query
    // tile (computed before the tile's scores are waited for); gate sigma R
    const DropKey dkey = {p.drop_rk, p.drop_tlow4, p.drop_tmask};
    const float dsig = p.drop_sigma;
    // with dropout the lanes of a warp exchange keep bits, so a wait that
    // gives up makes the whole warp leave together
    auto ew_wait = [&](uint64_t* bar, uint32_t par) -> bool {
      const bool w = mbar_wait(bar, par, wctl);
      if constexpr (DROP) return __all_sync(0xffffffffu, w);
      return w;
    };
    bool ok = true;
    int tile = first_tile - 1;
    for (int st = 0; ok && st < nsteps; ++st) {
      const int stage = st % C::NSTAGES;
      if (st % nsteps_h == 0) tile = first_tile - 1;  // next query head: from the start
      tile = tiles.next(tile + 1);
      const int it = tile * BN;  // first query row of the tile
      uint32_t kb[2];
      if constexpr (DROP) {
        const uint32_t bhq = (uint32_t)(p.head0 + bh_q0 + st / nsteps_h);
#pragma unroll
        for (int h = 0; h < 2; ++h) kb[h] = keep_col16(gj, it + HB * h + 16 * wg, bhq, dkey);
      }
      // the row vectors were written by the producer: acquire them explicitly
      if (!ew_wait(&m->bar_full_b[stage], (st / C::NSTAGES) & 1) ||
          !ew_wait(&m->bar_sa_sf[0], st & 1)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float* vec = reinterpret_cast<const float*>(s_stream + stage * C::STAGE_BYTES +
                                                        C::TILE_BYTES);
      // ---- copy this thread's SF columns of both halves, then release SF
      uint32_t rS[2][16], rF[2][16];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        tmem_ld16(ta + kColSF + HB * h + 16 * wg, rS[h]);
        if constexpr (kBob) tmem_ld16(ta + kColSF + 64 + HB * h + 16 * wg, rF[h]);
      }
      tmem_ld_wait(rS[0]);
      reg_dep(rS[1]);
      if constexpr (kBob) {
        reg_dep(rF[0]);
        reg_dep(rF[1]);
      }
      if constexpr (C::PH_SF) {
        // ---- from SF alone: P, f = tau F and the Vtil operand P o h (h = F -
        // alpha) of both halves; P o h goes over the S columns just copied
        float2 pP[2][8], pF[2][8];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int cv = HB * h + 16 * wg;
          const int lo = qlo - (it + cv), hi = qhi - (it + cv);
          if (lo > 0 || hi < 16) mask16(rS[h], lo, hi);
          uint32_t oPh[8];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            const float2 nL2 = *reinterpret_cast<const float2*>(vec + cv + c);
            const float2 nal = *reinterpret_cast<const float2*>(vec + 128 + cv + c);
            const float2 pr = probs2(pair(rS[h], c), sl2v, nL2);
            const float2 f = __fmul2_rn(pair(rF[h], c), tauv);
            float2 gp = pr;
            if constexpr (DROP) gp = __fmul2_rn(pr, gate2(kb[h], c, dsig));
            const float2 ph = __fmul2_rn(gp, __fadd2_rn(f, nal));
            pP[h][c / 2] = pr;
            pF[h][c / 2] = f;
            oPh[c / 2] = pack_bf16(ph.x, ph.y);
          }
          tmem_st8(ta + kColSF + cv, oPh);
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&m->bar_sf_free[0]);
        if (!ew_wait(&m->bar_sa_dc[dc_sel(st)], dc_par(st))) {
          ok = false;
          break;
        }
        tc_fence_after();
        // ---- with DC: Stil and dS into the DC columns just read
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int cv = HB * h + 16 * wg;
          const uint32_t R = ta + dc_col(st) + cv;
          uint32_t rdP[16], rC[16];
          tmem_ld16(R + 0, rdP);
          tmem_ld16(R + 64, rC);
          tmem_ld_wait(rdP);
          reg_dep(rC);
          uint32_t oSt[8], odS[8];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            const float2 nD = *reinterpret_cast<const float2*>(vec + 64 + cv + c);
            const float2 nal = *reinterpret_cast<const float2*>(vec + 128 + cv + c);
            const float2 nE = *reinterpret_cast<const float2*>(vec + 192 + cv + c);
            const float2 pr = pP[h][c / 2], f = pF[h][c / 2];
            float2 dp = pair(rdP, c), cc = pair(rC, c);
            if constexpr (DROP) {  // dP and C gated by sigma R
              const float2 g = gate2(kb[h], c, dsig);
              dp = __fmul2_rn(dp, g);
              cc = __fmul2_rn(cc, g);
            }
            const float2 t = __fadd2_rn(dp, nD);
            // Ptil = C + F (dP - D) - alpha dP ; Stil = P (Ptil - E)
            const float2 pt = __ffma2_rn(nal, dp, __ffma2_rn(f, t, cc));
            const float2 stl = __fmul2_rn(pr, __fadd2_rn(pt, nE));
            const float2 ds = __fmul2_rn(pr, t);
            oSt[c / 2] = pack_bf16(stl.x, stl.y);
            odS[c / 2] = pack_bf16(ds.x, ds.y);
          }
          tmem_st8(R + 8, oSt);
          tmem_st8(R + 64, odS);
          tmem_st_wait();
          tc_fence_before();
          mbar_arrive(&m->bar_ew[2 * dc_sel(st) + h]);
        }
        continue;
      }
      tc_fence_before();
      mbar_arrive(&m->bar_sf_free[0]);
      if (!ew_wait(&m->bar_sa_dc[dc_sel(st)], dc_par(st))) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t dcol = dc_col(st);
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int cv = HB * h + 16 * wg;  // tile column of this thread's first
        const int ib = it + cv;           // first query row of this thread's 16
        // valid query columns c satisfy  lo <= c < hi
        const int lo = qlo - ib, hi = qhi - ib;
        if (lo > 0 || hi < 16) mask16(rS[h], lo, hi);
        const uint32_t R = ta + dcol + cv;
        if constexpr (kBob) {
          uint32_t rdP[16], rC[16];
          tmem_ld16(R + 0, rdP);
          tmem_ld16(R + 64, rC);
          tmem_ld_wait(rdP);
          reg_dep(rC);
          uint32_t oPh[8], oSt[8], odS[8];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            const float2 nL2 = *reinterpret_cast<const float2*>(vec + cv + c);
            const float2 nD = *reinterpret_cast<const float2*>(vec + 64 + cv + c);
            const float2 nal = *reinterpret_cast<const float2*>(vec + 128 + cv + c);
            const float2 nE = *reinterpret_cast<const float2*>(vec + 192 + cv + c);
            const float2 pr = probs2(pair(rS[h], c), sl2v, nL2);
            const float2 f = __fmul2_rn(pair(rF[h], c), tauv);
            float2 dp = pair(rdP, c), cv = pair(rC, c), gp = pr;
            if constexpr (DROP) {  // dP, C and the Vtil operand gated by sigma R
              const float2 g = gate2(kb[h], c, dsig);
              dp = __fmul2_rn(dp, g);
              cv = __fmul2_rn(cv, g);
              gp = __fmul2_rn(pr, g);
            }
            const float2 t = __fadd2_rn(dp, nD);
            // Ptil = C + F (dP - D) - alpha dP ; Stil = P (Ptil - E) ; h = F - alpha
            const float2 pt = __ffma2_rn(nal, dp, __ffma2_rn(f, t, cv));
            const float2 ph = __fmul2_rn(gp, __fadd2_rn(f, nal));
            const float2 stl = __fmul2_rn(pr, __fadd2_rn(pt, nE));
            const float2 ds = __fmul2_rn(pr, t);
            oPh[c / 2] = pack_bf16(ph.x, ph.y);
            oSt[c / 2] = pack_bf16(stl.x, stl.y);
            odS[c / 2] = pack_bf16(ds.x, ds.y);
          }
          tmem_st8(R + 0, oPh);
          tmem_st8(R + 8, oSt);
          tmem_st8(R + 64, odS);
        } else {
          uint32_t rdP[16];
          tmem_ld16(R, rdP);
          tmem_ld_wait(rdP);
          uint32_t oP[8], odS[8];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            const float2 nL2 = *reinterpret_cast<const float2*>(vec + cv + c);
            const float2 nD = *reinterpret_cast<const float2*>(vec + 64 + cv + c);
            const float2 pr = probs2(pair(rS[h], c), sl2v, nL2);
            float2 dp = pair(rdP, c), gp = pr;
            if constexpr (DROP) {  // dV = (sigma R o P)^T dO, dS = P (sigma R dP - D)
              const float2 g = gate2(kb[h], c, dsig);
              dp = __fmul2_rn(dp, g);
              gp = __fmul2_rn(pr, g);
            }
            const float2 ds = __fmul2_rn(pr, __fadd2_rn(dp, nD));
            oP[c / 2] = pack_bf16(gp.x, gp.y);
            odS[c / 2] = pack_bf16(ds.x, ds.y);
          }
          tmem_st8(R + 0, oP);
          tmem_st8(R + 8, odS);
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&m->bar_ew[2 * dc_sel(st) + h]);
      }
    }
    if (ok) ok = mbar_wait(&m->bar_acc, 0, wctl);
    if (ok && *abort_flag) ok = false;
    tc_fence_after();
    if (ok) {
      const size_t rowoff = ((size_t)bh * N + (size_t)(row_ok ? gj : 0)) * DG;
#pragma unroll 1
      for (int q = 0; q < D / 32; ++q) {
        const int cc = wg * (D / 2) + 16 * q;
        uint32_t rK[16], rV[16];
        tmem_ld16(ta + cc, rK);
        tmem_ld16(ta + D + cc, rV);
        tmem_ld_wait(rK);
        reg_dep(rV);
        if (row_ok && cc < DG) {
          float kv[16], vv[16];
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            kv[c] = tau * bits_f(rK[c]);
            vv[c] = bits_f(rV[c]);
          }
          store_row16(p.out0 + rowoff + cc, kv);
          store_row16(p.out1 + rowoff + cc, vv);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace fbob
