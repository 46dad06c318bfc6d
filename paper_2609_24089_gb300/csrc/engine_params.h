// engine_params.h -- host-visible tile constants, operation kinds, kernel
// parameter block and per-kernel shared-memory plans of the tile engines.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace fbob {

// Bits of the device-side error word.
enum : uint32_t { kDevErrTimeout = 1u, kDevErrBadLaunch = 2u };

constexpr int BM = 128;          // stationary rows per CTA (TMEM lanes)
constexpr int BN = 64;           // streamed rows per tile
constexpr int HB = 32;           // streamed rows per half tile (TMA box rows of streamed maps)
constexpr int kChunk = HB * 128; // bytes of one 32-row x 64-column bf16 chunk
constexpr int kThreads = 352;
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;   // MMA issuer X (and TMEM allocator)
constexpr int kMmaWarpY = 10; // MMA issuer Y
constexpr int kEwThreads = 256;
constexpr int kMaxStages = 4;  // stream stages the barrier arrays hold
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColA = 256;  // stage-A region of half h starts at kColA + 128 h
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// BobPass1: Pass 1 in one sweep with the affine fusion of Prop. 3.1 (d = 64).
// BobStats + BobPass1D: Pass 1 in two kernels (d = 128): the row scalars
// alpha, E (and D) first, then Qtil and dOtil directly from eqs. (6)-(7).
// (Fwd names the forward for the launcher; it runs in fwd_engine.cuh.)
enum class RowOp { Fwd, BwdDQ, BobPass1, BobStats, BobPass1D };
enum class ColOp { BwdDKDV, BobPass2 };

// ---------------------------------------------------------------- parameters
struct EngineParams {
  CUtensorMap tm[7];  // stationary maps first (box rows BM), then streamed (box rows BN)
  // Q and U_Q; in the kernels that hold stationary MMA A operands in TMEM
  // (the row statistics kernel, every head-dimension-256 kernel) the sources
  // of those operands: Q, U_Q in the row kernels, K, V in the column kernels
  const __nv_bfloat16* q;
  const __nv_bfloat16* uq;
  const __nv_bfloat16* o;     // forward output O (row engine: D and dOtil)
  const __nv_bfloat16* dout;  // dO (row engine: D = do.o)
  const float* lse;           // natural-log L [BH, N]
  const float* vec_in;        // column engine: D (bwd) or row_stats (alpha,E,D) (pass 2)
  __nv_bfloat16* out0;        // O | dQ | Qtil  ||  dK | Ktil
  __nv_bfloat16* out1;        // dOtil          ||  dV | Vtil
  float* vec_out;             // lse | D | row_stats(alpha, E, D)
  int N;
  int BH;
  int nblk;  // stationary blocks per head
  int causal;
  int wl, wr;  // valid band of row i: i - wl <= j <= i + wr (-1: unbounded); causal gives wr = 0
  const int* seq_off;  // packed sequences: offsets [nseq + 1], or nullptr for one sequence
  int nseq;
  // block-sparse mask: [nbm][nbm] bytes over 128 x 128 blocks (query block,
  // key block), or nullptr; nbm = ceil(N / 128)
  const uint8_t* bmask;
  int nbm;
  int H, Hkv;  // query and key/value heads per batch entry (grouped-query attention)
  float scale;
  long long bhn;  // BH * N (row_stats plane stride)
  unsigned long long wait_limit_ns;  // bound of every device-side wait
  int inject_stall;                  // fault injection: producers issue nothing
  int head_group;                    // CTA order: heads per group (attn_engine.cuh, cta_order)
  // dropout (kernels instantiated with it): Philox round keys (the seed
  // raised r times by the Weyl constants, r = 0..9), the byte threshold t as
  // (t mod 128) in each byte and a flag (all ones if t < 128), and
  // sigma = 256 / (256 - t)
  uint32_t drop_rk[20];
  uint32_t drop_tlow4, drop_tmask;
  float drop_sigma;
  int head0;  // flat index b*H + h of the launch's first query head (dropout counter)
};

// ---------------------------------------------------------------- configs
// BoB row kernels: stationary Q, U_Q, dO; streamed K, U_K, V, U_V
constexpr bool row_bob(RowOp op) {
  return op == RowOp::BobPass1 || op == RowOp::BobStats || op == RowOp::BobPass1D;
}

template <RowOp OP, int D>
struct RowCfg {
  static constexpr int KB = D / 64;  // 64-wide boxes per row
  static constexpr int NSTAT = OP == RowOp::BwdDQ ? 2 : 3;
  static constexpr int NSTREAM = row_bob(OP) ? 4 : 2;
  // the one-sweep Pass 1 (Prop. 3.1) holds four accumulators of 64 output
  // columns next to the stage-A tiles (4 x 64 + 128 + 128 = 512 TMEM
  // columns): at d = 128 the output columns are split over SPLIT = 2 CTAs per
  // row block, each computing the whole stage A and its half of stage B
  static constexpr int SPLIT = OP == RowOp::BobPass1 ? D / 64 : 1;
  static_assert(OP != RowOp::BobPass1 || D == 64 || D == 128, "one-sweep Pass 1: d <= 128");
  // the row statistics kernel has no accumulators: Q and U_Q live in TMEM as
  // MMA A operands next to two SF buffers; only dO stays in shared memory,
  // which leaves room for another stream stage
  static constexpr bool STAT_TMEM = OP == RowOp::BobStats;
  static constexpr int STAT_BYTES = (STAT_TMEM ? 1 : NSTAT) * KB * BM * 128;
  static constexpr int STAGE_BYTES = NSTREAM * KB * BN * 128;
  static constexpr int NSTAGES = STAT_TMEM ? (D == 64 ? 4 : 3) : row_bob(OP) ? (D == 64 ? 3 : 2) : 4;
  // issuer X also issues the stage-B MMAs into B and dOtil0, between the two
  // parts of SF(t+1).  Measured faster for the one-sweep Pass 1 (d = 64); for
  // the direct form at d = 128 (dOtil on X) Y's wait for X's share before
  // each DC cost 5 % more than it saved.
  static constexpr bool XSHARE = OP == RowOp::BobPass1;
  // Pass 1's DC ([dP | C]) issued per 32-key half, so that stage B of half 0
  // overlaps the elementwise work on half 1; otherwise one N = 128 MMA per
  // K-step for the whole tile.  Measured for the direct form at d = 128:
  // whole-tile DC is 5 % faster (16 N = 64 MMAs per tile cost issuer Y more
  // than the overlap saved).
  static constexpr bool DC_HALVES = OP == RowOp::BobPass1;
  // the dQ kernel's DC tile (dP, 64 columns) leaves the other half of the DC
  // area free: two dP buffers, dP(t+2) issued right after stage B(t)
  static constexpr bool DC2 = OP == RowOp::BwdDQ;
  // the direct form's stream stages are released per 32-key half: half h of
  // tile t's stage is free once stage B(t) of half h has run, and the
  // producer refills it with half h of tile t + NSTAGES at once (with only
  // two 64 KB stages its loads otherwise land late for issuer X)
  // (d = 128; at d = 64 three stages already keep the loads ahead)
  static constexpr bool HALF_REL = OP == RowOp::BobPass1D && 2 * NSTAGES <= kMaxStages;
  // bookkeeping (256), the row-sum exchange (4 x BM floats), the rows' D (BM floats)
  static constexpr int MISC_BYTES = 2816;
  static constexpr int SMEM_BYTES = STAT_BYTES + NSTAGES * STAGE_BYTES + MISC_BYTES;
};

template <ColOp OP, int D>
struct ColCfg {
  static constexpr int KB = D / 64;
  static constexpr int NSTAT = OP == ColOp::BwdDKDV ? 2 : 4;
  static constexpr int NSTREAM = OP == ColOp::BwdDKDV ? 2 : 3;
  static constexpr int NVEC = OP == ColOp::BwdDKDV ? 2 : 4;  // L2, D (, alpha, E)
  static constexpr int STAT_BYTES = NSTAT * KB * BM * 128;
  static constexpr int TILE_BYTES = NSTREAM * KB * BN * 128;
  static constexpr int STAGE_BYTES = TILE_BYTES + 1024;  // + row vectors
  static constexpr int NSTAGES = (OP == ColOp::BobPass2 && D == 128) ? 2 : (D == 64 ? 4 : 3);
  // two DC buffers in TMEM (DC(t+1) is issued before stage B(t)): possible
  // when the accumulators (2 D columns) leave columns 128..255 free, or, in
  // the first backward, whose DC tile (dP^T) takes 64 of the DC area's 128
  // columns, in the DC area's second half
  static constexpr bool DC2 = D == 64 || OP == ColOp::BwdDKDV;
  static constexpr uint32_t DC1_COL = D == 64 ? 128u : 448u;  // second DC buffer
  // issuer X takes the value-accumulator MMAs of stage B.  With one DC buffer
  // issuer Y would have to wait for them before the next DC (measured slower);
  // with two that wait is two tiles back and off the critical path.
  static constexpr bool XSHARE = DC2;
  // BoB Pass 2 with one DC buffer (d = 128): the Vtil operand P o h needs
  // only the scores tile, so the elementwise warps write it into the SF
  // columns they have just copied, and issuer X accumulates Vtil from there
  // (before SF(t+1), in its own issue order).  Issuer Y's chain per tile is
  // then the Ktil MMAs and DC(t+1) alone, and the exponentials leave the
  // elementwise work that waits for DC.  Measured 2.5 % faster at d = 128;
  // at d = 64 (two DC buffers, XSHARE) it was 10 % slower: there SF(t+1)
  // waiting for P o h is the longer delay.
  static constexpr bool PH_SF = OP == ColOp::BobPass2 && !DC2;
  static constexpr int MISC_BYTES = 256;
  static constexpr int SMEM_BYTES = STAT_BYTES + NSTAGES * STAGE_BYTES + MISC_BYTES;
};

}  // namespace fbob
