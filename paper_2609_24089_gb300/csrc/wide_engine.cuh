// wide_engine.cuh -- tcgen05 tile kernels for head dimension 256 (App.
// "Head-dimension sensitivity": a d = 256 specialisation whose binding
// constraints are the Pass-1 accumulators and the live tiles on chip).
//
// At d = 256 one 128-row stationary tensor is 64 KB of shared memory and one
// 128 x 256 fp32 accumulator takes 256 of the 512 TMEM columns, so the row and
// column engines' plans (three or four stationary tensors in shared memory,
// two accumulators next to the stage-A tiles) do not fit an SM.  The kernels
// here keep 128 stationary rows per CTA (M = 128 MMAs, one row per TMEM lane)
// and change the rest:
//   * streamed tiles of 32 rows (one warpgroup per 16 of them), so a stream
//     stage of four tensors is 64 KB;
//   * one or two stationary operands live in TMEM as MMA A operands (128
//     columns each: bf16 pairs), written there once per CTA;
//   * one accumulator per kernel.  BoB Pass 1 runs as two kernels: the row
//     scalars alpha, E, D (eq. 6) together with dOtil (its alpha-free part
//     dOtil0 = P U_V + (P o F) V accumulated in the same sweep, dOtil =
//     dOtil0 - alpha o, eq. 8), then Qtil = tau (Stil K + dS U_K) (eqs. 6-7)
//     with those scalars known.  (The per-pass entry points also run the row
//     scalars alone and dOtil = P U_V + (P o h) V given them.)  Pass 2 runs
//     as Vtil = (P o h)^T dO and Ktil = tau (Stil^T Q + dS^T U_Q), the latter
//     over two CTAs per key block, each owning 128 output columns.
//     The forward is one sweep with an online softmax (the two warpgroups
//     share each tile's row maximum through shared memory; O in TMEM is
//     rescaled only when the running maximum grows by more than 8 in log2
//     units) and the first backward three kernels (dQ and D, dV, dK);
//   * where a kernel reads a streamed tensor only in its stage A, that tensor
//     has a ring of its own (ring B), released as soon as the stage-A MMAs
//     reading it complete.
//
// Roles (352 threads) as in attn_engine.cuh: warps 0-7 elementwise (thread =
// stationary row, warpgroup g = streamed columns 16g .. 16g+15 of a tile),
// warp 8 TMA producer (and, in the column kernels, the streamed rows' row
// vectors), warp 9 issuer X (stage A "SF": scores and F), warp 10 issuer Y
// (stage A "DC": dP and C, and stage B).  Every accumulator has one issuer,
// so results are bitwise reproducible; there are no atomics.
//
// Per tile t: X issues SF(t) into SF buffer t % NSF once the buffer is free
// (the elementwise warps copied SF(t - NSF), or, where the stage-B operands
// are written over SF, stage B(t - NSF) completed).  Y issues DC(t) NDC tiles
// ahead and stage B(t) once the elementwise warps wrote its operand tiles.
// The elementwise warps write those bf16 operand tiles over the SF or DC
// columns they have just read, each thread only over its own columns.
//
// Every wait is bounded (tc_ptx.cuh): on expiry the CTA records a timeout in
// the device error word, drains its asynchronous work and exits.
#pragma once

#include "attn_engine.cuh"
#include "wide_launch.h"

namespace fbob {

// WOp (wide_launch.h): Fwd: O and L (eq. 1).  Stats: alpha, E, D (eq.
// 6); DOut: dOtil; DQ: Qtil (eqs.
// 6-7).  StatsDO: alpha, E, D and dOtil in one sweep: dOtil0 = P U_V +
// (P o F) V needs no row scalar, and dOtil = dOtil0 - alpha o (Prop. 3.1,
// eq. 8).  BwdDQ: dQ and D; BwdDV: dV; BwdDK: dK (eqs. 2-3).  P2V: Vtil;
// P2K: Ktil (Alg. 2, second loop; eq. 7).

constexpr int WD = 256;               // head dimension of these kernels
constexpr int WKB = WD / 64;          // 64-column boxes per row
constexpr int WBN = 32;               // streamed rows per tile
constexpr int kWBox = WBN * 128;      // one 32-row x 64-column bf16 box (4 KB)
constexpr int kWStat = WKB * BM * 128;  // one stationary 128 x 256 bf16 tensor (64 KB)

// Per-kernel plan.  Stationary operands: NTT in TMEM (columns 0 and 128),
// NTS in shared memory.  Streamed tensors: NTA in ring A (NSA stages; read by
// SF and stage B), NTB in ring B (NSB stages; read only by DC).  NVEC fp32 row
// vectors of the streamed rows (column kernels).  SF: SFW columns per buffer,
// NSF buffers; DC likewise.  ACC_N accumulator columns.  SPLIT CTAs per
// stationary block (each its ACC_N output columns).
//
// PAIR (StatsDO): the four streamed tensors travel as two pairs, (K, U_K)
// read only by SF and (V, U_V) read by DC and stage B, through one ring of
// NSA 32 KB slots in the order KU(0), VU(0), KU(1), VU(1), ...; each slot is
// released by the one issuer that reads its pair last (X after SF, Y after
// stage B), so with three slots tile t+1's pairs load while tile t runs
// (KU(t+1) reuses the slot of VU(t-1), VU(t+1) that of KU(t)).
template <WOp OP>
struct WCfg {
  static constexpr bool PAIR = OP == WOp::StatsDO;
  static constexpr bool ROW = OP == WOp::Fwd || OP == WOp::Stats ||
                              OP == WOp::DOut || OP == WOp::DQ || OP == WOp::BwdDQ || PAIR;
  static constexpr int NTT = (OP == WOp::Stats || OP == WOp::P2K) ? 2 : 1;
  static constexpr int NTS = (OP == WOp::Fwd || OP == WOp::BwdDV) ? 0
                             : (OP == WOp::DQ || OP == WOp::P2K || PAIR)             ? 2
                                                                                     : 1;
  // (PAIR: tensors per slot; the maps hold K, U_K, then V, U_V)
  static constexpr int NTA = (OP == WOp::Stats || OP == WOp::DOut) ? 4
                             : OP == WOp::P2V                        ? 3
                             : (OP == WOp::Fwd || OP == WOp::DQ || OP == WOp::P2K ||
                                OP == WOp::BwdDV || PAIR)
                                 ? 2
                                 : 1;
  static constexpr int NTB = OP == WOp::DQ ? 2
                             : (OP == WOp::BwdDQ || OP == WOp::P2K || OP == WOp::BwdDK) ? 1
                                                                                          : 0;
  static constexpr int NVEC = OP == WOp::P2V   ? 2   // L, alpha
                              : OP == WOp::P2K ? 4   // L, D, alpha, E
                              : OP == WOp::BwdDV ? 1 // L
                              : OP == WOp::BwdDK ? 2 // L, D
                                                 : 0;
  static constexpr int NSA = (OP == WOp::Stats || OP == WOp::DOut || OP == WOp::DQ || OP == WOp::P2K)
                                 ? 2
                             : (OP == WOp::P2V || PAIR) ? 3
                                                        : 4;
  static constexpr int NSB = NTB == 0 ? 0 : OP == WOp::DQ ? 1 : OP == WOp::P2K ? 2 : 4;
  static constexpr int SFW = (OP == WOp::Stats || OP == WOp::DOut || OP == WOp::DQ ||
                              OP == WOp::P2V || OP == WOp::P2K || PAIR)
                                 ? 64   // [S | F]
                                 : 32;  // S
  static constexpr int NSF = (OP == WOp::DQ || OP == WOp::P2K || PAIR) ? 1 : 2;
  static constexpr int DCW = (OP == WOp::Stats || OP == WOp::DQ || OP == WOp::P2K || PAIR) ? 64  // [dP | C]
                             : (OP == WOp::BwdDQ || OP == WOp::BwdDK)              ? 32  // dP
                                                                                   : 0;
  static constexpr int NDC = DCW == 0 ? 0 : (OP == WOp::DQ || OP == WOp::P2K || PAIR) ? 1 : 2;
  static constexpr int NDC1 = NDC > 0 ? NDC : 1;  // (divisor where there is no DC)
  static constexpr int ACC_N = OP == WOp::Stats ? 0 : OP == WOp::P2K ? 128 : 256;
  static constexpr int SPLIT = OP == WOp::P2K ? 2 : 1;
  // stage-B operand tiles written over the SF columns (else over DC)
  static constexpr bool OPS_SF = OP == WOp::Fwd || OP == WOp::DOut || OP == WOp::P2V ||
                                 OP == WOp::BwdDV;
  static constexpr bool OPS_DC = OP == WOp::DQ || OP == WOp::BwdDQ || OP == WOp::P2K ||
                                 OP == WOp::BwdDK || PAIR;
  static constexpr bool HAS_B = ACC_N > 0;
  // issuer Y reads ring A (stage B, or the statistics kernel's DC); with
  // PAIR each slot has one releasing issuer
  static constexpr bool Y_READS_A = (HAS_B || OP == WOp::Stats) && !PAIR;
  // D = do . o summed in the prologue; alpha / E0 row sums (or the
  // forward's row sums) exchanged between the two warpgroups; the forward's
  // per-tile row maxima exchanged likewise (MX)
  static constexpr bool ROW_DOTS = OP == WOp::Stats || OP == WOp::BwdDQ || PAIR;
  static constexpr bool XCHG = OP == WOp::Stats || OP == WOp::Fwd || PAIR;
  static constexpr bool MX = OP == WOp::Fwd;

  // TMEM columns
  static constexpr uint32_t ACC_COL = 128u * NTT;
  static constexpr uint32_t SF_COL = ACC_COL + ACC_N;
  static constexpr uint32_t DC_COL = SF_COL + NSF * SFW;
  static_assert(DC_COL + NDC * DCW <= kTmemCols, "TMEM plan exceeds 512 columns");

  // shared memory
  static constexpr int STAT_BYTES = NTS * kWStat;
  static constexpr int STAGE_A = NTA * WKB * kWBox;
  static constexpr int STAGE_B = NTB * WKB * kWBox;
  static constexpr int VEC_BYTES = NVEC * WBN * 4;  // per ring-A stage
  static constexpr int OFF_A = STAT_BYTES;
  static constexpr int OFF_B = OFF_A + NSA * STAGE_A;
  static constexpr int OFF_VEC = OFF_B + NSB * STAGE_B;
  static constexpr int OFF_MISC = OFF_VEC + NSA * VEC_BYTES;
  static constexpr int MISC_BYTES =
      512 + (XCHG ? 4 * BM * 4 : 0) + (ROW_DOTS ? BM * 4 : 0) + (MX ? 4 * BM * 4 : 0);
  static constexpr int SMEM_BYTES = OFF_MISC + MISC_BYTES;
  static_assert(SMEM_BYTES <= 232448, "shared-memory plan exceeds 227 KB");
  static_assert(NSA <= kMaxStages && NSB <= kMaxStages, "ring bound");
};

struct WMisc {
  uint64_t bar_stat;
  uint64_t full_a[kMaxStages], empty_a[kMaxStages];
  uint64_t full_b[kMaxStages], empty_b[kMaxStages];
  uint64_t sf[2], sf_read[2];  // SF(t) completed; the elementwise warps copied it
  uint64_t dc[2], dc_read[2];
  uint64_t ew[2];  // the elementwise warps wrote the stage-B operands of tile t (t & 1)
  uint64_t sb[2];  // stage B(t) completed (per SF buffer)
  uint64_t mx[2];  // forward: both warpgroups posted tile t's row maxima (t & 1)
  uint64_t acc;
  uint32_t tmem_base;
  uint32_t pad;
  WaitCtl wctl;
};
static_assert(sizeof(WMisc) <= 512, "WMisc must fit 512 bytes");

// Streamed tiles of a CTA under a block-sparse mask over 128 x 128 blocks
// (App. "Extensions": only the block pairs with an unmasked entry are
// visited); 32-row tiles, four per block.
struct TileSet32 {
  const uint8_t* mb;
  int stride;
  int t0, t1;
  __device__ int count() const {
    if (mb == nullptr) return t1 - t0 + 1;
    int n = 0;
    for (int b = t0 >> 2; b <= (t1 >> 2); ++b)
      if (mb[(size_t)b * stride] != 0) n += min(4 * b + 3, t1) - max(4 * b, t0) + 1;
    return n;
  }
  __device__ __forceinline__ int next(int t) const {
    if (mb == nullptr) return t;
    while (t <= t1 && mb[(size_t)(t >> 2) * stride] == 0) t = (t | 3) + 1;
    return t;
  }
};

template <WOp OP, bool DROP>
__global__ void __launch_bounds__(kThreads, 1) wide_engine(const __grid_constant__ EngineParams p) {
  using C = WCfg<OP>;
  constexpr bool kRow = C::ROW;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* s_stat = smem;
  uint8_t* s_a = smem + C::OFF_A;
  uint8_t* s_b = smem + C::OFF_B;
  float* s_vec = reinterpret_cast<float*>(smem + C::OFF_VEC);
  WMisc* m = reinterpret_cast<WMisc*>(smem + C::OFF_MISC);
  float* s_xchg = reinterpret_cast<float*>(smem + C::OFF_MISC + 512);  // 4 x BM floats
  float* s_d = s_xchg + (C::XCHG ? 4 * BM : 0);                        // BM floats
  float* s_mx = s_d + (C::ROW_DOTS ? BM : 0);  // forward: [tile & 1][warpgroup][row]

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  if ((smem_u32(smem) & 1023u) != 0) {
    if (tid == 0) atomicOr(&g_fbob_error_word, kDevErrBadLaunch);
    return;
  }

  // ---- tile decode.  Row kernels: stationary query block rb of query head
  // bh, streamed key tiles of key/value head bh_kv.  Column kernels:
  // stationary key block of key/value head bh, streamed query tiles of its
  // G query heads one after the other.
  const int N = p.N;
  const int hc = C::SPLIT > 1 ? (int)(blockIdx.x % C::SPLIT) : 0;
  const int lin = blockIdx.x / C::SPLIT;
  int bi, bh;
  cta_order(p, lin, bi, bh);
  const int blk = (kRow && p.causal) ? (p.nblk - 1 - bi) : bi;  // longest first
  const int r0 = blk * BM;                                       // first stationary row
  const int last_row = min(r0 + BM, N) - 1;
  int seq_lo0, seq_hi0, seq_lo1, seq_hi1;
  seq_bounds(p, r0, seq_lo0, seq_hi0);
  seq_bounds(p, last_row, seq_lo1, seq_hi1);
  int s_lo, s_hi;  // streamed rows [s_lo, s_hi) that meet a stationary row's band
  if constexpr (kRow) {
    s_lo = max(seq_lo0, p.wl < 0 ? 0 : r0 - p.wl);
    s_hi = min(seq_hi1, p.wr < 0 ? N : last_row + p.wr + 1);
  } else {
    s_lo = max(seq_lo0, p.wr < 0 ? 0 : r0 - p.wr);
    s_hi = min(seq_hi1, p.wl < 0 ? N : last_row + p.wl + 1);
  }
  const int first_tile = s_lo / WBN;
  const TileSet32 tiles = {p.bmask ? (kRow ? p.bmask + (size_t)blk * p.nbm : p.bmask + blk) : nullptr,
                           kRow ? 1 : p.nbm, first_tile, (s_hi - 1) / WBN};
  const int nsteps_h = tiles.count();
  const int G = kRow ? 1 : p.H / p.Hkv;
  const int bh_kv = p.Hkv == p.H ? bh : (bh / p.H) * p.Hkv + (bh % p.H) / (p.H / p.Hkv);
  const int bh_q0 = (bh / p.Hkv) * p.H + (bh % p.Hkv) * G;  // column kernels: first query head
  const int nsteps = G * nsteps_h;
  // head of the stationary rows and of streamed step st
  const int bh_stat = bh;
  auto stream_head = [&](int st) -> int { return kRow ? bh_kv : bh_q0 + st / nsteps_h; };

  if (tid == 0) {
    m->wctl.abort = 0;
    m->wctl.limit_ns = p.wait_limit_ns;
    // producer's TMA transaction + the elementwise threads' TMEM operand stores
    mbar_init(&m->bar_stat, 1 + kEwThreads);
    for (int s = 0; s < C::NSA; ++s) {
      mbar_init(&m->full_a[s], C::NVEC ? 1 + 32 : 1);  // + the producer lanes' row vectors
      mbar_init(&m->empty_a[s], C::Y_READS_A ? 2 : 1);
    }
    for (int s = 0; s < C::NSB; ++s) {
      mbar_init(&m->full_b[s], 1);
      mbar_init(&m->empty_b[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&m->sf[b], 1);
      mbar_init(&m->sf_read[b], kEwThreads);
      mbar_init(&m->dc[b], 1);
      mbar_init(&m->dc_read[b], kEwThreads);
      mbar_init(&m->ew[b], kEwThreads);
      mbar_init(&m->sb[b], 1);
      mbar_init(&m->mx[b], kEwThreads);
    }
    mbar_init(&m->acc, 2);
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
    const int lane = tid & 31;
    const bool stall = p.inject_stall != 0;
    int issued_a[kMaxStages] = {-1, -1, -1, -1}, issued_b[kMaxStages] = {-1, -1, -1, -1};
    if (lane == 0 && !stall) {
      constexpr int kMaps = C::NTS + (C::PAIR ? 2 * C::NTA : C::NTA + C::NTB);
      for (int t = 0; t < kMaps; ++t) tma_prefetch_desc(&p.tm[t]);
      mbar_arrive_expect_tx(&m->bar_stat, C::STAT_BYTES);
      for (int t = 0; t < C::NTS; ++t)
        for (int b = 0; b < WKB; ++b)
          tma_load_3d(s_stat + t * kWStat + b * (BM * 128), &p.tm[t], &m->bar_stat, 64 * b, r0,
                      bh_stat);
    }
    int tile = first_tile - 1;
    for (int st = 0; !stall && st < nsteps; ++st) {
      if (st % nsteps_h == 0) tile = first_tile - 1;
      tile = tiles.next(tile + 1);
      const int row = tile * WBN;
      const int hs = stream_head(st);
      if constexpr (C::PAIR) {
        // pair pr of tile st (0: K, U_K; 1: V, U_V) at ring position 2 st + pr
        bool go = true;
        for (int pr = 0; pr < 2; ++pr) {
          const int pos = 2 * st + pr, sl = pos % C::NSA, use = pos / C::NSA;
          if (use >= 1 && !mbar_wait(&m->empty_a[sl], (use - 1) & 1, wctl)) {
            go = false;
            break;
          }
          if (lane == 0) {
            uint8_t* dst = s_a + sl * C::STAGE_A;
            mbar_arrive_expect_tx(&m->full_a[sl], C::STAGE_A);
            for (int b = 0; b < WKB; ++b)
              for (int t = 0; t < 2; ++t)
                tma_load_3d(dst + (b * 2 + t) * kWBox, &p.tm[C::NTS + 2 * pr + t], &m->full_a[sl],
                            64 * b, row, hs);
          }
          issued_a[sl] = pos;
        }
        if (!go) break;
        continue;
      }
      // ring A
      const int sa = st % C::NSA;
      if (st >= C::NSA && !mbar_wait(&m->empty_a[sa], ((st / C::NSA) - 1) & 1, wctl)) break;
      if (lane == 0) {
        uint8_t* dst = s_a + sa * C::STAGE_A;
        mbar_arrive_expect_tx(&m->full_a[sa], C::STAGE_A);
        for (int b = 0; b < WKB; ++b)
          for (int t = 0; t < C::NTA; ++t)
            tma_load_3d(dst + (b * C::NTA + t) * kWBox, &p.tm[C::NTS + t], &m->full_a[sa], 64 * b,
                        row, hs);
      }
      if constexpr (C::NVEC > 0) {
        // row vectors of the streamed rows, negated (L scaled by log2 e):
        // [0] L, then (BoB Pass 2) alpha, or D, alpha, E; (dK) D
        float* vec = s_vec + sa * (C::NVEC * WBN);
        const int ri = row + lane;
        const bool ok = ri < N;
        const size_t gi = (size_t)hs * N + (ok ? ri : 0);
        float v[4] = {0.f, 0.f, 0.f, 0.f};
        if (ok) {
          v[0] = -p.lse[gi] * kLog2e;
          if constexpr (OP == WOp::P2V) v[1] = -p.vec_in[gi];
          if constexpr (OP == WOp::P2K) {
            v[1] = -p.vec_in[2 * p.bhn + gi];
            v[2] = -p.vec_in[gi];
            v[3] = -p.vec_in[p.bhn + gi];
          }
          if constexpr (OP == WOp::BwdDK) v[1] = -p.vec_in[gi];
        }
#pragma unroll
        for (int k = 0; k < C::NVEC; ++k) vec[k * WBN + lane] = v[k];
        mbar_arrive(&m->full_a[sa]);
      }
      issued_a[sa] = st;
      // ring B
      if constexpr (C::NSB > 0) {
        const int sb = st % C::NSB;
        if (st >= C::NSB && !mbar_wait(&m->empty_b[sb], ((st / C::NSB) - 1) & 1, wctl)) break;
        if (lane == 0) {
          uint8_t* dst = s_b + sb * C::STAGE_B;
          mbar_arrive_expect_tx(&m->full_b[sb], C::STAGE_B);
          for (int b = 0; b < WKB; ++b)
            for (int t = 0; t < C::NTB; ++t)
              tma_load_3d(dst + (b * C::NTB + t) * kWBox, &p.tm[C::NTS + C::NTA + t],
                          &m->full_b[sb], 64 * b, row, hs);
        }
        issued_b[sb] = st;
      }
    }
    if (lane == 0 && *abort_flag) {  // drain loads still in flight
      for (int s = 0; s < C::NSA; ++s)
        if (issued_a[s] >= 0) drain_wait(&m->full_a[s], (issued_a[s] / C::NSA) & 1);
      if constexpr (C::NSB > 0) {
        for (int s = 0; s < C::NSB; ++s)
          if (issued_b[s] >= 0) drain_wait(&m->full_b[s], (issued_b[s] / C::NSB) & 1);
      }
      drain_wait(&m->bar_stat, 0);
    }
  } else if (warp == kMmaWarp || warp == kMmaWarpY) {
    // ------------------------------------------------------------ MMA issuers
    if (elect_lane0()) {
      // stationary shared-memory operand t, K-step k (K-major, 128 rows)
      const uint64_t sd0 = sdesc_sw128(smem_u32(s_stat), 16, 1024);
      auto sd = [&](int t, int k) -> uint64_t {
        return sd0 + (uint64_t)((t * kWStat + (k / 4) * (BM * 128) + (k % 4) * 32) >> 4);
      };
      // streamed rows (K-major, the N side of stage A) of ring tensor t, K-step k
      auto kd = [&](uint32_t stage, int nt, int t, int k) -> uint64_t {
        return sdesc_sw128(stage + ((k / 4) * nt + t) * kWBox + (k % 4) * 32, 16, 1024);
      };
      // streamed rows 16 s .. of ring tensor t as the B operand of stage B
      // (MN-major: K = streamed rows, N = output columns from box b0 on)
      auto md = [&](uint32_t stage, int nt, int t, int s, int b0) -> uint64_t {
        return sdesc_sw128(stage + (b0 * nt + t) * kWBox + s * 2048, nt * kWBox, 1024);
      };
      constexpr uint32_t id_sf = idesc_bf16(128, C::SFW, false);
      constexpr uint32_t id_n32 = idesc_bf16(128, 32, false);
      constexpr uint32_t id_dc = idesc_bf16(128, C::DCW > 0 ? C::DCW : 32, false);
      constexpr uint32_t id_b = idesc_bf16(128, C::ACC_N > 0 ? C::ACC_N : 32, true);
      const uint32_t tT0 = tmem + 0, tT1 = tmem + 128;  // TMEM operands
      const uint32_t acc = tmem + C::ACC_COL;
      bool ok = mbar_wait(&m->bar_stat, 0, wctl);
      if (warp == kMmaWarp) {
        // ---------------- issuer X: SF(t)
        for (int st = 0; ok && st < nsteps; ++st) {
          // ring slot of this tile's SF operands and its use count
          const int apos = C::PAIR ? 2 * st : st;
          const int b = st % C::NSF, sa = apos % C::NSA;
          if (st >= C::NSF) {
            uint64_t* freed = C::OPS_SF ? &m->sb[b] : &m->sf_read[b];
            if (!mbar_wait(freed, ((st / C::NSF) - 1) & 1, wctl)) break;
          }
          if (!mbar_wait(&m->full_a[sa], (apos / C::NSA) & 1, wctl)) break;
          tc_fence_after();
          const uint32_t stg = smem_u32(s_a + sa * C::STAGE_A);
          const uint32_t R = tmem + C::SF_COL + b * C::SFW;
          if constexpr (C::SFW == 32) {
#pragma unroll
            for (int k = 0; k < WD / 16; ++k)  // S = Q K^T (row) / S^T = K Q^T (column)
              mma_ts(R, tT0 + 8 * k, kd(stg, C::NTA, 0, k), id_n32, k > 0);
          } else {
#pragma unroll
            for (int k = 0; k < WD / 16; ++k)  // [S | F] = Q [K ; U_K]^T  /  K [Q ; U_Q]^T
              mma_ts(R, tT0 + 8 * k, kd(stg, C::NTA, 0, k), id_sf, k > 0);
            if constexpr (OP == WOp::Stats) {
#pragma unroll
              for (int k = 0; k < WD / 16; ++k)  // F += U_Q K^T (U_Q in TMEM)
                mma_ts(R + 32, tT1 + 8 * k, kd(stg, C::NTA, 0, k), id_n32, 1);
            } else {
#pragma unroll
              for (int k = 0; k < WD / 16; ++k)  // F += U_Q K^T  /  F^T += U_K Q^T
                mma_ss(R + 32, sd(0, k), kd(stg, C::NTA, 0, k), id_n32, 1);
            }
          }
          mma_commit(&m->sf[b]);
          mma_commit(&m->empty_a[sa]);  // X's last read of the stage
        }
      } else {
        // ---------------- issuer Y: DC(t), NDC tiles ahead, and stage B(t)
        auto issue_dc = [&](int u) -> bool {
          const int b = u % C::NDC1;
          if (!C::OPS_DC && u >= C::NDC &&
              !mbar_wait(&m->dc_read[b], ((u / C::NDC1) - 1) & 1, wctl))
            return false;
          uint32_t stg;
          int nt, t0;
          if constexpr (C::PAIR) {  // V, U_V: pair 1 of tile u
            const int pos = 2 * u + 1, sl = pos % C::NSA;
            if (!mbar_wait(&m->full_a[sl], (pos / C::NSA) & 1, wctl)) return false;
            stg = smem_u32(s_a + sl * C::STAGE_A);
            nt = 2;
            t0 = 0;
          } else if constexpr (C::NTB > 0) {
            const int sbx = u % C::NSB;
            if (!mbar_wait(&m->full_b[sbx], (u / C::NSB) & 1, wctl)) return false;
            stg = smem_u32(s_b + sbx * C::STAGE_B);
            nt = C::NTB;
            t0 = 0;
          } else {  // the statistics kernel: V, U_V are ring-A tensors 2, 3
            const int sax = u % C::NSA;
            if (!mbar_wait(&m->full_a[sax], (u / C::NSA) & 1, wctl)) return false;
            stg = smem_u32(s_a + sax * C::STAGE_A);
            nt = C::NTA;
            t0 = 2;
          }
          tc_fence_after();
          const uint32_t R = tmem + C::DC_COL + b * C::DCW;
          if constexpr (OP == WOp::P2K) {
#pragma unroll
            for (int k = 0; k < WD / 16; ++k)  // dP^T = V dO^T (V in TMEM)
              mma_ts(R, tT1 + 8 * k, kd(stg, nt, 0, k), id_n32, k > 0);
#pragma unroll
            for (int k = 0; k < WD / 16; ++k)  // C^T = U_V dO^T
              mma_ss(R + 32, sd(1, k), kd(stg, nt, 0, k), id_n32, k > 0);
          } else {
            // [dP | C] = dO [V ; U_V]^T ; dP = dO V^T ; dP^T = V dO^T
            constexpr int kA = (OP == WOp::DQ || C::PAIR) ? 1 : 0;  // stationary dO (V for dK)
#pragma unroll
            for (int k = 0; k < WD / 16; ++k) mma_ss(R, sd(kA, k), kd(stg, nt, t0, k), id_dc, k > 0);
          }
          mma_commit(&m->dc[b]);
          if constexpr (C::PAIR) {
            // (V, U_V stay for stage B, which releases them)
          } else if constexpr (C::NTB > 0) {
            mma_commit(&m->empty_b[u % C::NSB]);
          } else {
            mma_commit(&m->empty_a[u % C::NSA]);
          }
          return true;
        };
        if constexpr (C::NDC > 0) {
          for (int u = 0; ok && u < C::NDC && u < nsteps; ++u) ok = issue_dc(u);
        }
        for (int st = 0; ok && st < nsteps; ++st) {
          if constexpr (C::HAS_B) {
            if (!mbar_wait(&m->ew[st & 1], (st >> 1) & 1, wctl)) break;
            tc_fence_after();
            // (PAIR: the slot of V, U_V)
            const int sa = (C::PAIR ? 2 * st + 1 : st) % C::NSA;
            const uint32_t stg = smem_u32(s_a + sa * C::STAGE_A);
            const uint32_t A = tmem + (C::OPS_SF ? C::SF_COL + (st % C::NSF) * C::SFW
                                                 : C::DC_COL + (st % C::NDC1) * C::DCW);
#pragma unroll
            for (int s = 0; s < 2; ++s) {  // K-step s: streamed rows 16 s .. (warpgroup s)
              const uint32_t first = (st == 0 && s == 0) ? 0u : 1u;
              const uint32_t As = A + 16 * s;
              if constexpr (OP == WOp::Fwd) {  // O += P V
                mma_ts(acc, As, md(stg, C::NTA, 1, s, 0), id_b, first);
              } else if constexpr (OP == WOp::DOut) {  // dOtil += P U_V + (P o h) V
                mma_ts(acc, As, md(stg, C::NTA, 3, s, 0), id_b, first);
                mma_ts(acc, As + 8, md(stg, C::NTA, 2, s, 0), id_b, 1);
              } else if constexpr (OP == WOp::DQ) {  // Qtil += Stil K + dS U_K
                mma_ts(acc, As, md(stg, C::NTA, 0, s, 0), id_b, first);
                mma_ts(acc, As + 8, md(stg, C::NTA, 1, s, 0), id_b, 1);
              } else if constexpr (OP == WOp::BwdDQ) {  // dQ += dS K
                mma_ts(acc, As, md(stg, C::NTA, 0, s, 0), id_b, first);
              } else if constexpr (OP == WOp::P2V) {  // Vtil += (P o h)^T dO
                mma_ts(acc, As, md(stg, C::NTA, 2, s, 0), id_b, first);
              } else if constexpr (OP == WOp::P2K) {  // Ktil += Stil^T Q + dS^T U_Q (columns of hc)
                mma_ts(acc, As, md(stg, C::NTA, 0, s, 2 * hc), id_b, first);
                mma_ts(acc, As + 8, md(stg, C::NTA, 1, s, 2 * hc), id_b, 1);
              } else if constexpr (OP == WOp::BwdDV) {  // dV += P^T dO
                mma_ts(acc, As, md(stg, C::NTA, 1, s, 0), id_b, first);
              } else if constexpr (OP == WOp::BwdDK) {  // dK += dS^T Q
                mma_ts(acc, As, md(stg, C::NTA, 0, s, 0), id_b, first);
              } else if constexpr (C::PAIR) {  // dOtil0 += P U_V + (P o F) V
                mma_ts(acc, As, md(stg, 2, 1, s, 0), id_b, first);
                mma_ts(acc, As + 8, md(stg, 2, 0, s, 0), id_b, 1);
              }
            }
            if constexpr (C::OPS_SF) mma_commit(&m->sb[st % C::NSF]);
            mma_commit(&m->empty_a[sa]);  // Y's last read of the stage
          }
          if constexpr (C::NDC > 0) {
            // DC(st + NDC) overwrites the operand tiles stage B(st) reads:
            // issued after it by this thread, so it runs after it
            if (st + C::NDC < nsteps && !issue_dc(st + C::NDC)) break;
          }
        }
      }
      mma_commit(&m->acc);
      if (*abort_flag) drain_wait(&m->acc, 0);
    }
  } else {
    // ------------------------------------------------------------ elementwise
    const int wg = warp >> 2;
    const int r = 32 * (warp & 3) + (tid & 31);  // stationary row in the block
    const int gr = r0 + r;
    const bool row_ok = gr < N;
    // this row's valid streamed indices [vlo, vhi) (keys of a query row, or
    // queries of a key row), within its sequence
    int vlo = 0, vhi = 0;
    if (row_ok) {
      seq_bounds(p, gr, vlo, vhi);
      if constexpr (kRow) {
        if (p.wl >= 0) vlo = max(vlo, gr - p.wl);
        if (p.wr >= 0) vhi = min(vhi, gr + p.wr + 1);
      } else {
        if (p.wr >= 0) vlo = max(vlo, gr - p.wr);
        if (p.wl >= 0) vhi = min(vhi, gr + p.wl + 1);
      }
    }
    const uint32_t ta = lane_base_addr(tmem, warp);
    const size_t rowoff = ((size_t)bh_stat * N + (size_t)(row_ok ? gr : 0)) * WD;
    const float tau = p.scale;
    const float sl2 = tau * kLog2e;
    const float2 sl2v = splat(sl2), tauv = splat(tau);
    const DropKey dkey = {p.drop_rk, p.drop_tlow4, p.drop_tmask};
    const float dsig = p.drop_sigma;
    // every lane of a warp takes a wait's outcome together: the TMEM loads
    // and stores after it are warp-collective (and with dropout the lanes
    // exchange keep bits), so no lane may leave the loop alone
    auto ew_wait = [&](uint64_t* bar, uint32_t par) -> bool {
      const bool w = mbar_wait(bar, par, wctl);
      return __all_sync(0xffffffffu, w);
    };

    // ---- stationary operands into TMEM (bf16 pairs: word c of a row =
    // elements 2c, 2c + 1 = column c of the A operand): warpgroup g writes
    // elements 128 g .. 128 g + 127 of each, 16 columns at a time
    {
#pragma unroll 1
      for (int slot = 0; slot < C::NTT; ++slot) {
        const __nv_bfloat16* src = (slot == 0 ? p.q : p.uq) + rowoff + 128 * wg;
        const uint4* s4 = reinterpret_cast<const uint4*>(src);
        uint4 v[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) v[u] = row_ok ? s4[u] : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int c = 0; c < 64; c += 8) {
          const uint4 a = v[c / 4], b = v[c / 4 + 1];
          const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
          tmem_st8(ta + 128 * slot + 64 * wg + c, w);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&m->bar_stat);
    }

    // ---- row scalars of a stationary row (row kernels)
    float nL2 = 0.f, nal = 0.f, nE = 0.f, Dr = 0.f;
    if constexpr (kRow) {
      if (row_ok && OP != WOp::Fwd) {
        const size_t ri = (size_t)bh_stat * N + gr;
        nL2 = -p.lse[ri] * kLog2e;
        if constexpr (OP == WOp::DOut || OP == WOp::DQ) {
          nal = -p.vec_in[ri];
          nE = -p.vec_in[p.bhn + ri];
          Dr = p.vec_in[2 * p.bhn + ri];
        }
      }
    }
    if constexpr (C::ROW_DOTS)
      Dr = block_row_dots<WD>(p.dout, p.o, (size_t)bh_stat * N * WD, r0, N, s_d, tid);
    const float2 nL2v = splat(nL2), nalv = splat(nal), nEv = splat(nE), nDv = splat(-Dr);

    float2 acc_a = splat(0.f), acc_e = splat(0.f);      // row sums (statistics)
    float run_m = -INFINITY, run_l = 0.f;  // forward: running maximum (log2 units) and sum
    bool ok = true;
    int tile = first_tile - 1;
    for (int st = 0; ok && st < nsteps; ++st) {
      if (st % nsteps_h == 0) tile = first_tile - 1;
      tile = tiles.next(tile + 1);
      const int c0 = tile * WBN + 16 * wg;  // first streamed index of this thread's 16
      const int hs = stream_head(st);
      uint32_t kb = 0;
      if constexpr (DROP) {
        if constexpr (kRow) kb = keep_row16(gr, c0, (uint32_t)(p.head0 + bh_stat), dkey);
        else kb = keep_col16(gr, c0, (uint32_t)(p.head0 + hs), dkey);
      }
      const int b = st % C::NSF;
      if (!ew_wait(&m->sf[b], (st / C::NSF) & 1)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const uint32_t Rsf = ta + C::SF_COL + b * C::SFW + 16 * wg;
      uint32_t rS[16], rF[16];
      tmem_ld16(Rsf, rS);
      if constexpr (C::SFW == 64) tmem_ld16(Rsf + 32, rF);
      tmem_ld_wait(rS);
      if constexpr (C::SFW == 64) reg_dep(rF);
      if constexpr (!C::OPS_SF) {
        tc_fence_before();
        mbar_arrive(&m->sf_read[b]);
      }
      // column kernels: the streamed rows' vectors (acquire the producer's stores)
      const float* vec = s_vec + (st % C::NSA) * (C::NVEC * WBN) + 16 * wg;
      if constexpr (C::NVEC > 0) {
        if (!ew_wait(&m->full_a[st % C::NSA], (st / C::NSA) & 1)) {
          ok = false;
          break;
        }
      }
      uint32_t rdP[16], rC[16];
      const int dcb = st % C::NDC1;
      const uint32_t Rdc = ta + C::DC_COL + dcb * C::DCW + 16 * wg;
      if constexpr (C::NDC > 0) {
        if (!ew_wait(&m->dc[dcb], (st / C::NDC1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
        tmem_ld16(Rdc, rdP);
        if constexpr (C::DCW == 64) tmem_ld16(Rdc + 32, rC);
        tmem_ld_wait(rdP);
        if constexpr (C::DCW == 64) reg_dep(rC);
        if constexpr (!C::OPS_DC) {
          tc_fence_before();
          mbar_arrive(&m->dc_read[dcb]);
        }
      }
      const int mlo = vlo - c0, mhi = vhi - c0;  // valid columns: mlo <= c < mhi
      if (mlo > 0 || mhi < 16) mask16(rS, mlo, mhi);

      if constexpr (OP == WOp::Fwd) {
        // this thread's tile maximum (log2 units), shared with the other
        // warpgroup's half of the row behind mx[t & 1] (bounded wait)
        float mt = -INFINITY;
#pragma unroll
        for (int c = 0; c < 16; ++c) mt = fmaxf(mt, bits_f(rS[c]));
        mt *= sl2;
        float* mxs = s_mx + (st & 1) * 2 * BM;
        mxs[wg * BM + r] = mt;
        mbar_arrive(&m->mx[st & 1]);
        if (!ew_wait(&m->mx[st & 1], (st >> 1) & 1)) {
          ok = false;
          break;
        }
        const float mrow = fmaxf(mt, mxs[(1 - wg) * BM + r]);
        // the running maximum is raised only when a tile's exceeds it by
        // more than 8 (so P <= 2^8): then the row sum and O (once the MMAs
        // into it so far have completed) are scaled by 2^(old - new); both
        // warpgroups take the same decision from the same maxima.  The
        // TMEM loads and stores are warp-collective, so a warp rescales
        // together whenever one of its rows needs it (the others by 1)
        const bool raise = mrow > run_m + 8.f;
        const float sc = raise ? ex2(run_m - mrow) : 1.f;  // 0 while run_m is -inf
        // (a row whose maximum was -inf so far holds only zeros in O)
        if (__any_sync(0xffffffffu, raise && run_m != -INFINITY) && st > 0) {
          if (!ew_wait(&m->sb[(st - 1) % C::NSF], ((st - 1) / C::NSF) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll 1
          for (int q = 0; q < 8; ++q) {
            const uint32_t ca = ta + C::ACC_COL + 128 * wg + 16 * q;
            uint32_t rO[16];
            tmem_ld16(ca, rO);
            tmem_ld_wait(rO);
            uint32_t w0[8], w1[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) {
              w0[c] = __float_as_uint(bits_f(rO[c]) * sc);
              w1[c] = __float_as_uint(bits_f(rO[8 + c]) * sc);
            }
            tmem_st8(ca, w0);
            tmem_st8(ca + 8, w1);
          }
        }
        if (raise) {
          run_l *= sc;
          run_m = mrow;
        }
        const float2 mu = splat(run_m == -INFINITY ? 0.f : -run_m);
        uint32_t o0[8];
        float2 ls = splat(0.f);
#pragma unroll
        for (int c = 0; c < 16; c += 2) {
          const float2 pr = probs2(pair(rS, c), sl2v, mu);
          ls = __fadd2_rn(ls, pr);
          float2 gp = pr;
          if constexpr (DROP) gp = __fmul2_rn(pr, gate2(kb, c, dsig));  // O = (sigma R o P) V
          o0[c / 2] = pack_bf16(gp.x, gp.y);
        }
        run_l += ls.x + ls.y;
        tmem_st8(Rsf, o0);
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&m->ew[st & 1]);
      } else {
        uint32_t o0[8], o1[8];
#pragma unroll
        for (int c = 0; c < 16; c += 2) {
          // per-column scalars: the row's own (row kernels) or the streamed
          // rows' (column kernels, from the stage's vectors)
          float2 cL2 = nL2v, cal = nalv, cE = nEv, cD = nDv;
          if constexpr (!kRow) {
            cL2 = *reinterpret_cast<const float2*>(vec + c);
            if constexpr (OP == WOp::P2V) cal = *reinterpret_cast<const float2*>(vec + WBN + c);
            if constexpr (OP == WOp::P2K) {
              cD = *reinterpret_cast<const float2*>(vec + WBN + c);
              cal = *reinterpret_cast<const float2*>(vec + 2 * WBN + c);
              cE = *reinterpret_cast<const float2*>(vec + 3 * WBN + c);
            }
            if constexpr (OP == WOp::BwdDK) cD = *reinterpret_cast<const float2*>(vec + WBN + c);
          }
          const float2 pr = probs2(pair(rS, c), sl2v, cL2);
          float2 g = splat(1.f);
          if constexpr (DROP) g = gate2(kb, c, dsig);
          if constexpr (OP == WOp::BwdDV) {  // (sigma R o P)
            const float2 gp = DROP ? __fmul2_rn(pr, g) : pr;
            o0[c / 2] = pack_bf16(gp.x, gp.y);
          } else if constexpr (C::PAIR) {
            // alpha += P F ; E0 += P (C + F (dP - D)) (dP, C gated); the
            // dOtil0 operands sigma R o P and sigma R o P o F
            const float2 f = __fmul2_rn(pair(rF, c), tauv);
            float2 dp = pair(rdP, c), cv = pair(rC, c), gp = pr;
            if constexpr (DROP) {
              dp = __fmul2_rn(dp, g);
              cv = __fmul2_rn(cv, g);
              gp = __fmul2_rn(pr, g);
            }
            const float2 pt0 = __ffma2_rn(f, __fadd2_rn(dp, cD), cv);
            acc_a = __ffma2_rn(pr, f, acc_a);
            acc_e = __ffma2_rn(pr, pt0, acc_e);
            const float2 pf = __fmul2_rn(gp, f);
            o0[c / 2] = pack_bf16(gp.x, gp.y);
            o1[c / 2] = pack_bf16(pf.x, pf.y);
          } else if constexpr (OP == WOp::Stats) {
            // alpha += P F ; E0 += P (C + F (dP - D))  (dP, C gated)
            const float2 f = __fmul2_rn(pair(rF, c), tauv);
            float2 dp = pair(rdP, c), cv = pair(rC, c);
            if constexpr (DROP) {
              dp = __fmul2_rn(dp, g);
              cv = __fmul2_rn(cv, g);
            }
            const float2 pt0 = __ffma2_rn(f, __fadd2_rn(dp, cD), cv);
            acc_a = __ffma2_rn(pr, f, acc_a);
            acc_e = __ffma2_rn(pr, pt0, acc_e);
          } else if constexpr (OP == WOp::DOut || OP == WOp::P2V) {
            // P (gated) and P o h, h = F - alpha
            const float2 f = __fmul2_rn(pair(rF, c), tauv);
            const float2 gp = DROP ? __fmul2_rn(pr, g) : pr;
            const float2 ph = __fmul2_rn(gp, __fadd2_rn(f, cal));
            if constexpr (OP == WOp::DOut) {
              o0[c / 2] = pack_bf16(gp.x, gp.y);
              o1[c / 2] = pack_bf16(ph.x, ph.y);
            } else {
              o0[c / 2] = pack_bf16(ph.x, ph.y);
            }
          } else if constexpr (OP == WOp::DQ || OP == WOp::P2K) {
            // Ptil = C + F (dP - D) - alpha dP ; Stil = P (Ptil - E) ; dS = P (dP - D)
            const float2 f = __fmul2_rn(pair(rF, c), tauv);
            float2 dp = pair(rdP, c), cv = pair(rC, c);
            if constexpr (DROP) {
              dp = __fmul2_rn(dp, g);
              cv = __fmul2_rn(cv, g);
            }
            const float2 t = __fadd2_rn(dp, cD);
            const float2 pt = __ffma2_rn(cal, dp, __ffma2_rn(f, t, cv));
            const float2 stl = __fmul2_rn(pr, __fadd2_rn(pt, cE));
            const float2 ds = __fmul2_rn(pr, t);
            o0[c / 2] = pack_bf16(stl.x, stl.y);
            o1[c / 2] = pack_bf16(ds.x, ds.y);
          } else if constexpr (OP == WOp::BwdDQ || OP == WOp::BwdDK) {  // dS = P (dP - D)
            float2 dp = pair(rdP, c);
            if constexpr (DROP) dp = __fmul2_rn(dp, g);
            const float2 ds = __fmul2_rn(pr, __fadd2_rn(dp, cD));
            o0[c / 2] = pack_bf16(ds.x, ds.y);
          }
        }
        if constexpr (C::HAS_B) {
          // operand tiles over this thread's own SF (or dP) columns just read
          const uint32_t R = C::OPS_SF ? Rsf : Rdc;
          tmem_st8(R, o0);
          if constexpr (OP == WOp::DOut || OP == WOp::DQ || OP == WOp::P2K || C::PAIR)
            tmem_st8(R + 8, o1);
          tmem_st_wait();
          tc_fence_before();
          mbar_arrive(&m->ew[st & 1]);
        }
      }
    }
    // ---------------------------------------------------------- epilogue
    if (ok) ok = mbar_wait(&m->acc, 0, wctl);
    if (ok && *abort_flag) ok = false;
    ok = __all_sync(0xffffffffu, ok);  // (the TMEM loads below are warp-collective)
    tc_fence_after();
    if constexpr (C::XCHG) {
      if constexpr (OP == WOp::Stats || C::PAIR) {
        s_xchg[wg * BM + r] = acc_a.x + acc_a.y;
        s_xchg[(2 + wg) * BM + r] = acc_e.x + acc_e.y;
      } else {  // the forward: each warpgroup's row sum (the maxima agree)
        s_xchg[wg * BM + r] = run_l;
      }
      named_bar_sync(1, kEwThreads);
    }
    if (ok) {
      const size_t ri = (size_t)bh_stat * N + gr;
      if constexpr (OP == WOp::Fwd) {
        // O = (sum of P V) / l and the natural-log L = (m + log2 l) ln 2
        const float l = s_xchg[r] + s_xchg[BM + r];
        const float il = l > 0.f ? 1.f / l : 0.f;
        if (row_ok && wg == 0) p.vec_out[ri] = (run_m + log2f(l)) * kLn2;
#pragma unroll 1
        for (int q = 0; q < WD / 32; ++q) {
          const int cc = wg * (WD / 2) + 16 * q;
          uint32_t rA[16];
          tmem_ld16(ta + C::ACC_COL + cc, rA);
          tmem_ld_wait(rA);
          if (row_ok) {
            float v[16];
#pragma unroll
            for (int c = 0; c < 16; ++c) v[c] = bits_f(rA[c]) * il;
            store_row16(p.out0 + rowoff + cc, v);
          }
        }
      } else if constexpr (OP == WOp::Stats) {
        if (row_ok && wg == 0) {
          const float alpha = s_xchg[r] + s_xchg[BM + r];
          const float E0 = s_xchg[2 * BM + r] + s_xchg[3 * BM + r];
          p.vec_out[ri] = alpha;
          p.vec_out[p.bhn + ri] = E0 - alpha * Dr;  // E = E0 - alpha D
          p.vec_out[2 * p.bhn + ri] = Dr;
        }
      } else if constexpr (C::PAIR) {
        // eq. (8): E = E0 - alpha D, dOtil = dOtil0 - alpha o
        const float alpha = s_xchg[r] + s_xchg[BM + r];
        const float E0 = s_xchg[2 * BM + r] + s_xchg[3 * BM + r];
        if (row_ok && wg == 0) {
          p.vec_out[ri] = alpha;
          p.vec_out[p.bhn + ri] = E0 - alpha * Dr;
          p.vec_out[2 * p.bhn + ri] = Dr;
        }
#pragma unroll 1
        for (int q = 0; q < WD / 32; ++q) {
          const int cc = wg * (WD / 2) + 16 * q;
          uint32_t rA[16];
          tmem_ld16(ta + C::ACC_COL + cc, rA);
          tmem_ld_wait(rA);
          if (row_ok) {
            float ov[16], v[16];
            load_row16(p.o + rowoff + cc, ov);
#pragma unroll
            for (int c = 0; c < 16; ++c) v[c] = nsteps > 0 ? bits_f(rA[c]) - alpha * ov[c] : 0.f;
            store_row16(p.out0 + rowoff + cc, v);
          }
        }
      } else {
        // the accumulator's ACC_N columns: warpgroup g stores half of them
        // (tau for the score-gradient outputs Qtil, Ktil, dQ, dK)
        constexpr bool kTau = OP == WOp::DQ || OP == WOp::P2K || OP == WOp::BwdDQ ||
                              OP == WOp::BwdDK;
        const float sc = kTau ? tau : 1.f;
        __nv_bfloat16* out = p.out0 + rowoff + C::ACC_N * hc;
#pragma unroll 1
        for (int q = 0; q < C::ACC_N / 32; ++q) {
          const int cc = wg * (C::ACC_N / 2) + 16 * q;
          uint32_t rA[16];
          tmem_ld16(ta + C::ACC_COL + cc, rA);
          tmem_ld_wait(rA);
          if (row_ok) {
            float v[16];
#pragma unroll
            for (int c = 0; c < 16; ++c) v[c] = nsteps > 0 ? sc * bits_f(rA[c]) : 0.f;
            store_row16(out + cc, v);
          }
        }
        if constexpr (OP == WOp::BwdDQ) {
          if (row_ok && wg == 0) p.vec_out[ri] = Dr;
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
