// attn_engine.cuh -- warp-specialised tcgen05 tile engines for softmax
// attention and its backward-over-backward on sm_103a.
//
// Two engines share one schedule skeleton:
//   * row engine: a CTA owns BM = 128 query rows (TMEM lanes) and streams key
//     blocks of BN = 64 rows.  Used by the forward (eq. 1), the dQ half of the
//     first backward (eqs. 2-3) and BoB Pass 1 (Alg. 2, first loop).
//   * column engine: a CTA owns BM = 128 key rows and streams query blocks of
//     BN = 64 rows, computing transposed tiles (key rows on lanes).  Used by
//     the dK/dV half of the first backward and BoB Pass 2 (Alg. 2, second loop).
//
// Roles (320 threads):
//   warps 0-7  elementwise: two warpgroups; warp w reads TMEM lanes
//              32*(w%4) .. +31, one stationary row per thread.  Each 64-column
//              tile is processed as 4 K-steps of 16 columns, warpgroup g taking
//              K-steps 2h+g of chunk h = 0, 1.
//   warp 8     TMA producer: stationary tiles once, then a ring of NSTAGES
//              stream stages (mbarrier full/empty pairs).  In the column engine
//              it also stages the streamed rows' fp32 row vectors in shared memory.
//   warp 9     TMEM allocator and MMA issuer (one lane).
//
// Per streamed tile: stage A (scores and friends, fp32 in TMEM, A and B from
// shared memory) -> elementwise (TMEM -> registers -> bf16 operand tiles
// written back into TMEM over stage-A columns already consumed) -> stage B
// (accumulators += bf16 tile (TMEM) x streamed tile (shared memory,
// MN-major)).  Stage B of chunk 0 runs while the elementwise warps work on
// chunk 1.  Tensor-memory map (512 columns): accumulators at 0..255,
// stage-A tiles at 256..511.
//
// Every wait is bounded (tc_ptx.cuh); on expiry the CTA records a timeout in
// the device error word, drains its own asynchronous work and exits.
#pragma once

#include "engine_params.h"
#include "tc_ptx.cuh"

namespace fbob {

// Shared-memory bookkeeping block (in the MISC area).
struct Misc {
  uint64_t bar_stat;
  uint64_t bar_full[4];
  uint64_t bar_empty[4];
  uint64_t bar_sa;
  uint64_t bar_ew[2];
  uint64_t bar_acc;
  uint32_t tmem_base;
  int abort_flag;
};

__device__ __forceinline__ uint32_t lane_base_addr(uint32_t tmem_base, int warp) {
  return tmem_base + ((uint32_t)(32 * (warp & 3)) << 16);
}

// Second-chance drain used only on the abort path: waits (bounded, ignoring
// the abort flag) for asynchronous work this CTA started.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait(bar, parity)) {
    if (global_timer_ns() - t0 > 200000000ull) return;
  }
}

__device__ __forceinline__ float bits_f(uint32_t u) { return __uint_as_float(u); }

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

// fp32 dot product of one bf16 row pair of length D (D = do_i . o_i).
template <int D>
__device__ __forceinline__ float row_dot(const __nv_bfloat16* a, const __nv_bfloat16* b) {
  float acc = 0.f;
#pragma unroll
  for (int c = 0; c < D; c += 16) {
    float x[16], y[16];
    load_row16(a + c, x);
    load_row16(b + c, y);
#pragma unroll
    for (int t = 0; t < 16; ++t) acc = fmaf(x[t], y[t], acc);
  }
  return acc;
}

// ============================================================== row engine
template <RowOp OP, int D>
__global__ void __launch_bounds__(kThreads, 1) row_engine(const __grid_constant__ EngineParams p) {
  using C = RowCfg<OP, D>;
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* s_stat = smem;
  uint8_t* s_stream = smem + C::STAT_BYTES;
  Misc* m = reinterpret_cast<Misc*>(s_stream + C::NSTAGES * C::STAGE_BYTES);
  float* s_xchg = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(m) + 256);  // 4 x BM floats

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  if ((smem_u32(smem) & 1023u) != 0) {  // swizzle atoms need 1024-byte alignment
    if (tid == 0) atomicOr(&g_fbob_error_word, kDevErrBadLaunch);
    return;
  }

  // ---- tile decode: consecutive CTAs take different heads of one row block;
  // with the causal mask the longest row blocks go first.
  const int N = p.N;
  int lin = blockIdx.x;
  const int bh = lin % p.BH;
  lin /= p.BH;
  const int split = lin % C::NSPLIT;
  const int rbi = lin / C::NSPLIT;
  const int rb = p.causal ? (p.nblk - 1 - rbi) : rbi;
  const int i0 = rb * BM;
  const int last_row = min(i0 + BM, N) - 1;
  const int ntiles = p.causal ? (last_row / BN + 1) : (N + BN - 1) / BN;
  const int nsteps = OP == RowOp::Fwd ? 2 * ntiles : ntiles;

  if (tid == 0) {
    m->abort_flag = 0;
    mbar_init(&m->bar_stat, 1);
    for (int s = 0; s < C::NSTAGES; ++s) {
      mbar_init(&m->bar_full[s], 1);
      mbar_init(&m->bar_empty[s], 1);
    }
    mbar_init(&m->bar_sa, 1);
    mbar_init(&m->bar_ew[0], kEwThreads);
    mbar_init(&m->bar_ew[1], kEwThreads);
    mbar_init(&m->bar_acc, 1);
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
  volatile int* abort_flag = &m->abort_flag;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------ producer
    if (elect_lane0()) {
      for (int t = 0; t < C::NSTAT + C::NSTREAM; ++t) tma_prefetch_desc(&p.tm[t]);
      mbar_arrive_expect_tx(&m->bar_stat, C::STAT_BYTES);
      for (int t = 0; t < C::NSTAT; ++t)
        for (int b = 0; b < C::KB; ++b)
          tma_load_3d(s_stat + (t * C::KB + b) * (BM * 128), &p.tm[t], &m->bar_stat, 64 * b, i0,
                      bh);
      int issued[4] = {-1, -1, -1, -1};
      for (int st = 0; st < nsteps; ++st) {
        const int stage = st % C::NSTAGES;
        if (st >= C::NSTAGES) {
          if (!mbar_wait(&m->bar_empty[stage], ((st / C::NSTAGES) - 1) & 1, abort_flag)) break;
        }
        const int j = st % ntiles;
        const bool k_only = (OP == RowOp::Fwd) && st < ntiles;
        uint8_t* dst = s_stream + stage * C::STAGE_BYTES;
        mbar_arrive_expect_tx(&m->bar_full[stage],
                              k_only ? C::KB * BN * 128 : C::STAGE_BYTES);
        for (int t = 0; t < (k_only ? 1 : C::NSTREAM); ++t)
          for (int b = 0; b < C::KB; ++b)
            tma_load_3d(dst + (b * C::NSTREAM + t) * (BN * 128), &p.tm[C::NSTAT + t],
                        &m->bar_full[stage], 64 * b, j * BN, bh);
        issued[stage] = st;
      }
      if (*abort_flag) {  // drain loads still in flight
        for (int s = 0; s < C::NSTAGES; ++s)
          if (issued[s] >= 0) drain_wait(&m->bar_full[s], (issued[s] / C::NSTAGES) & 1);
        drain_wait(&m->bar_stat, 0);
      }
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (elect_lane0()) {
      const uint32_t id_n64 = idesc_bf16(128, 64, false);
      const uint32_t id_n128 = idesc_bf16(128, 128, false);
      const uint32_t id_b = idesc_bf16(128, C::DOUT, true);
      const uint32_t tA = tmem + kColA;
      bool ok = mbar_wait(&m->bar_stat, 0, abort_flag);
      for (int st = 0; ok && st < nsteps; ++st) {
        const int stage = st % C::NSTAGES;
        if (!mbar_wait(&m->bar_full[stage], (st / C::NSTAGES) & 1, abort_flag)) break;
        tc_fence_after();
        const uint32_t sbase = smem_u32(s_stream + stage * C::STAGE_BYTES);
        const uint32_t stat = smem_u32(s_stat);
        auto stat_desc = [&](int t, int k) {
          return sdesc_sw128(stat + (t * C::KB + k / 4) * (BM * 128) + (k % 4) * 32, 16, 1024);
        };
        auto strm_desc = [&](int t, int k) {
          return sdesc_sw128(sbase + ((k / 4) * C::NSTREAM + t) * (BN * 128) + (k % 4) * 32, 16,
                             1024);
        };
        // ---- stage A
        if constexpr (OP == RowOp::BobPass1) {
          // stationary: 0 Q, 1 U_Q, 2 dO ; stream: 0 K, 1 U_K, 2 V, 3 U_V
          for (int k = 0; k < D / 16; ++k)  // [S | F2] = Q [K ; U_K]^T
            mma_ss(tA + 0, stat_desc(0, k), strm_desc(0, k), id_n128, k > 0);
          for (int k = 0; k < D / 16; ++k)  // [dP | C] = dO [V ; U_V]^T
            mma_ss(tA + 128, stat_desc(2, k), strm_desc(2, k), id_n128, k > 0);
          for (int k = 0; k < D / 16; ++k)  // F += U_Q K^T
            mma_ss(tA + 64, stat_desc(1, k), strm_desc(0, k), id_n64, 1);
        } else if constexpr (OP == RowOp::BwdDQ) {
          // stationary: 0 Q, 1 dO ; stream: 0 K, 1 V
          for (int k = 0; k < D / 16; ++k)
            mma_ss(tA + 0, stat_desc(0, k), strm_desc(0, k), id_n64, k > 0);
          for (int k = 0; k < D / 16; ++k)
            mma_ss(tA + 64, stat_desc(1, k), strm_desc(1, k), id_n64, k > 0);
        } else {
          for (int k = 0; k < D / 16; ++k)
            mma_ss(tA + 0, stat_desc(0, k), strm_desc(0, k), id_n64, k > 0);
        }
        mma_commit(&m->bar_sa);
        // ---- stage B, per chunk, once the elementwise warps have written it
        for (int h = 0; h < 2; ++h) {
          if (!mbar_wait(&m->bar_ew[h], st & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          for (int s = 2 * h; s < 2 * h + 2; ++s) {
            const uint32_t first = (st == 0 && s == 0) ? 0u : 1u;
            auto mn_desc = [&](int t) {  // streamed tile t, output block `split`, rows 16s..
              return sdesc_sw128(
                  sbase + (split * C::NSTREAM + t) * (BN * 128) + s * 2048,
                  C::NSTREAM * BN * 128, 1024);
            };
            if constexpr (OP == RowOp::BobPass1) {
              const uint32_t aP = tA + 16 * s, aPF = tA + 16 * s + 8;
              const uint32_t aPPt = tA + 128 + 16 * s, adS = tA + 128 + 16 * s + 8;
              const uint32_t aPdP = tA + 192 + 16 * s;
              mma_ts(tmem + 0, aP, mn_desc(3), id_b, first);     // dOtil0 += P U_V
              mma_ts(tmem + 0, aPF, mn_desc(2), id_b, 1);        //        += (P o F) V
              mma_ts(tmem + 64, aPPt, mn_desc(0), id_b, first);  // Omega  += (P o Pt0) K
              mma_ts(tmem + 64, adS, mn_desc(1), id_b, 1);       //        += dS U_K
              mma_ts(tmem + 128, aP, mn_desc(0), id_b, first);   // B      += P K
              mma_ts(tmem + 192, aPdP, mn_desc(0), id_b, first); // R      += (P o dP) K
            } else if constexpr (OP == RowOp::BwdDQ) {
              mma_ts(tmem + 0, tA + 16 * s, mn_desc(0), id_b, first);  // dQ += dS K
            } else {
              if (st >= ntiles) {  // second sweep: O += P V
                const uint32_t f2 = (st == ntiles && s == 0) ? 0u : 1u;
                mma_ts(tmem + 0, tA + 16 * s, mn_desc(1), id_b, f2);
              }
            }
          }
        }
        if (!ok) break;
        mma_commit(&m->bar_empty[stage]);
      }
      mma_commit(&m->bar_acc);
      if (*abort_flag) drain_wait(&m->bar_acc, 0);
    }
  } else {
    // ------------------------------------------------------------ elementwise
    const int wg = warp >> 2;                 // warpgroup 0/1
    const int r = 32 * (warp & 3) + (tid & 31);  // stationary row in the block
    const int gi = i0 + r;
    const bool row_ok = gi < N;
    const uint32_t ta = lane_base_addr(tmem, warp);
    const uint32_t tA = ta + kColA;
    const size_t rowoff = ((size_t)bh * N + (size_t)(row_ok ? gi : 0)) * D;
    const float tau = p.scale;
    const float sl2 = tau * kLog2e;
    float L2 = 0.f, Dr = 0.f;
    if constexpr (OP != RowOp::Fwd) {
      if (row_ok) {
        L2 = p.lse[(size_t)bh * N + gi] * kLog2e;
        Dr = row_dot<D>(p.dout + rowoff, p.o + rowoff);
      }
    }
    float mrow = -INFINITY, lrow = 0.f;  // forward sweep-1 running max / sum (log2 domain)
    float a_part = 0.f, e_part = 0.f;    // Pass 1 partial row sums
    bool ok = true;
    for (int st = 0; st < nsteps; ++st) {
      if (!mbar_wait(&m->bar_sa, st & 1, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int j0 = (st % ntiles) * BN;
      const bool need_mask = (!row_ok) || (j0 + BN > N) || (p.causal && j0 + BN - 1 > gi);
      if constexpr (OP == RowOp::Fwd) {
        if (st == ntiles) {  // end of sweep 1: combine the two warpgroups' (max, sum)
          s_xchg[wg * BM + r] = mrow;
          s_xchg[(2 + wg) * BM + r] = lrow;
          named_bar_sync(1, kEwThreads);
          const float m0 = s_xchg[r], m1 = s_xchg[BM + r];
          const float l0 = s_xchg[2 * BM + r], l1 = s_xchg[3 * BM + r];
          const float mm = fmaxf(m0, m1);
          const float l = (m0 == -INFINITY ? 0.f : l0 * ex2(m0 - mm)) +
                          (m1 == -INFINITY ? 0.f : l1 * ex2(m1 - mm));
          L2 = row_ok ? mm + __log2f(l) : 0.f;
        }
      }
      for (int h = 0; h < 2; ++h) {
        const int s = 2 * h + wg;  // K-step handled by this warpgroup
        const int c0 = 16 * s;
        if constexpr (OP == RowOp::BobPass1) {
          uint32_t rS[16], rF[16], rdP[16], rC[16];
          tmem_ld16(tA + 0 + c0, rS);
          tmem_ld16(tA + 64 + c0, rF);
          tmem_ld16(tA + 128 + c0, rdP);
          tmem_ld16(tA + 192 + c0, rC);
          tmem_ld_wait(rS);
          reg_dep(rF);
          reg_dep(rdP);
          reg_dep(rC);
          uint32_t oP[8], oPF[8], oPPt[8], odS[8], oPdP[8];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            float pv[2], pf[2], ppt[2], ds[2], pdp[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int gj = j0 + c0 + c + e;
              float pr = ex2(fmaf(bits_f(rS[c + e]), sl2, -L2));
              if (need_mask && !(row_ok && gj < N && (!p.causal || gj <= gi))) pr = 0.f;
              const float f = tau * bits_f(rF[c + e]);
              const float dp = bits_f(rdP[c + e]);
              const float t = dp - Dr;
              const float pt0 = fmaf(f, t, bits_f(rC[c + e]));  // Ptil0 = C + F (dP - D)
              pv[e] = pr;
              pf[e] = pr * f;
              ppt[e] = pr * pt0;
              ds[e] = pr * t;
              pdp[e] = pr * dp;
              a_part += pf[e];
              e_part += ppt[e];
            }
            oP[c / 2] = pack_bf16(pv[0], pv[1]);
            oPF[c / 2] = pack_bf16(pf[0], pf[1]);
            oPPt[c / 2] = pack_bf16(ppt[0], ppt[1]);
            odS[c / 2] = pack_bf16(ds[0], ds[1]);
            oPdP[c / 2] = pack_bf16(pdp[0], pdp[1]);
          }
          tmem_st8(tA + 0 + c0, oP);
          tmem_st8(tA + 0 + c0 + 8, oPF);
          tmem_st8(tA + 128 + c0, oPPt);
          tmem_st8(tA + 128 + c0 + 8, odS);
          tmem_st8(tA + 192 + c0, oPdP);
        } else if constexpr (OP == RowOp::BwdDQ) {
          uint32_t rS[16], rdP[16];
          tmem_ld16(tA + 0 + c0, rS);
          tmem_ld16(tA + 64 + c0, rdP);
          tmem_ld_wait(rS);
          reg_dep(rdP);
          uint32_t odS[8];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            float ds[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int gj = j0 + c0 + c + e;
              float pr = ex2(fmaf(bits_f(rS[c + e]), sl2, -L2));
              if (need_mask && !(row_ok && gj < N && (!p.causal || gj <= gi))) pr = 0.f;
              ds[e] = pr * (bits_f(rdP[c + e]) - Dr);
            }
            odS[c / 2] = pack_bf16(ds[0], ds[1]);
          }
          tmem_st8(tA + c0, odS);
        } else {
          uint32_t rS[16];
          tmem_ld16(tA + c0, rS);
          tmem_ld_wait(rS);
          if (st < ntiles) {  // sweep 1: running max and sum in the log2 domain
            float x[16];
            float mx = mrow;
#pragma unroll
            for (int c = 0; c < 16; ++c) {
              const int gj = j0 + c0 + c;
              x[c] = bits_f(rS[c]) * sl2;
              if (need_mask && !(row_ok && gj < N && (!p.causal || gj <= gi))) x[c] = -INFINITY;
              mx = fmaxf(mx, x[c]);
            }
            if (mx != -INFINITY) {
              float l = (mrow == -INFINITY) ? 0.f : lrow * ex2(mrow - mx);
#pragma unroll
              for (int c = 0; c < 16; ++c) l += ex2(x[c] - mx);
              lrow = l;
              mrow = mx;
            }
          } else {  // sweep 2: normalised probabilities
            uint32_t oP[8];
#pragma unroll
            for (int c = 0; c < 16; c += 2) {
              float pv[2];
#pragma unroll
              for (int e = 0; e < 2; ++e) {
                const int gj = j0 + c0 + c + e;
                float pr = ex2(fmaf(bits_f(rS[c + e]), sl2, -L2));
                if (need_mask && !(row_ok && gj < N && (!p.causal || gj <= gi))) pr = 0.f;
                pv[e] = pr;
              }
              oP[c / 2] = pack_bf16(pv[0], pv[1]);
            }
            tmem_st8(tA + c0, oP);
          }
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&m->bar_ew[h]);
      }
    }
    // ---------------------------------------------------------- epilogue
    if (ok) ok = mbar_wait(&m->bar_acc, 0, abort_flag);
    tc_fence_after();
    if constexpr (OP == RowOp::BobPass1) {
      s_xchg[wg * BM + r] = a_part;
      s_xchg[(2 + wg) * BM + r] = e_part;
      named_bar_sync(1, kEwThreads);
    }
    if (ok) {
      if constexpr (OP == RowOp::BobPass1) {
        const float alpha = s_xchg[r] + s_xchg[BM + r];
        const float E0 = s_xchg[2 * BM + r] + s_xchg[3 * BM + r];
        const float E = E0 - alpha * Dr;  // eq. (8): E = E0 - alpha D
        const int cbase = split * 64 + 32 * wg;
#pragma unroll 1
        for (int q = 0; q < 2; ++q) {
          const int cc = 32 * wg + 16 * q;  // accumulator column (0..63)
          uint32_t rO[16], rW[16], rB[16], rR[16];
          tmem_ld16(ta + 0 + cc, rO);
          tmem_ld16(ta + 64 + cc, rW);
          tmem_ld16(ta + 128 + cc, rB);
          tmem_ld16(ta + 192 + cc, rR);
          tmem_ld_wait(rO);
          reg_dep(rW);
          reg_dep(rB);
          reg_dep(rR);
          if (row_ok) {
            float ov[16], qt[16], dot[16];
            load_row16(p.o + rowoff + cbase + 16 * q, ov);
#pragma unroll
            for (int c = 0; c < 16; ++c) {
              // eq. (8): Qtil = tau (Omega - alpha R - E B), dOtil = dOtil0 - alpha o
              qt[c] = tau * (bits_f(rW[c]) - alpha * bits_f(rR[c]) - E * bits_f(rB[c]));
              dot[c] = bits_f(rO[c]) - alpha * ov[c];
            }
            store_row16(p.out0 + rowoff + cbase + 16 * q, qt);
            store_row16(p.out1 + rowoff + cbase + 16 * q, dot);
          }
        }
        if (row_ok && split == 0 && wg == 0) {
          const size_t ri = (size_t)bh * N + gi;
          p.vec_out[ri] = alpha;
          p.vec_out[p.bhn + ri] = E;
          p.vec_out[2 * p.bhn + ri] = Dr;
        }
      } else {
        // O (forward) or dQ = tau * acc (first backward), columns [wg*D/2, +D/2)
        const float mul = OP == RowOp::BwdDQ ? tau : 1.f;
#pragma unroll 1
        for (int q = 0; q < D / 32; ++q) {
          const int cc = wg * (D / 2) + 16 * q;
          uint32_t rA[16];
          tmem_ld16(ta + cc, rA);
          tmem_ld_wait(rA);
          if (row_ok) {
            float v[16];
#pragma unroll
            for (int c = 0; c < 16; ++c) v[c] = mul * bits_f(rA[c]);
            store_row16(p.out0 + rowoff + cc, v);
          }
        }
        if (row_ok && wg == 0) {
          const size_t ri = (size_t)bh * N + gi;
          if constexpr (OP == RowOp::Fwd) p.vec_out[ri] = L2 * kLn2;
          else p.vec_out[ri] = Dr;
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

// ============================================================ column engine
template <ColOp OP, int D>
__global__ void __launch_bounds__(kThreads, 1) col_engine(const __grid_constant__ EngineParams p) {
  using C = ColCfg<OP, D>;
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
  const int N = p.N;
  int lin = blockIdx.x;
  const int bh = lin % p.BH;
  const int cb = lin / p.BH;  // key block; block 0 has the most work under the causal mask
  const int j0 = cb * BM;
  const int first_tile = p.causal ? (j0 / BN) : 0;
  const int ntotal = (N + BN - 1) / BN;
  const int nsteps = ntotal - first_tile;

  if (tid == 0) {
    m->abort_flag = 0;
    mbar_init(&m->bar_stat, 1);
    for (int s = 0; s < C::NSTAGES; ++s) {
      mbar_init(&m->bar_full[s], 1 + 32);  // TMA bytes + 32 producer lanes' row vectors
      mbar_init(&m->bar_empty[s], 1);
    }
    mbar_init(&m->bar_sa, 1);
    mbar_init(&m->bar_ew[0], kEwThreads);
    mbar_init(&m->bar_ew[1], kEwThreads);
    mbar_init(&m->bar_acc, 1);
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
  volatile int* abort_flag = &m->abort_flag;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------ producer
    const int lane = tid & 31;
    if (lane == 0) {
      for (int t = 0; t < C::NSTAT + C::NSTREAM; ++t) tma_prefetch_desc(&p.tm[t]);
      mbar_arrive_expect_tx(&m->bar_stat, C::STAT_BYTES);
      for (int t = 0; t < C::NSTAT; ++t)
        for (int b = 0; b < C::KB; ++b)
          tma_load_3d(s_stat + (t * C::KB + b) * (BM * 128), &p.tm[t], &m->bar_stat, 64 * b, j0,
                      bh);
    }
    int issued[4] = {-1, -1, -1, -1};
    for (int st = 0; st < nsteps; ++st) {
      const int stage = st % C::NSTAGES;
      if (st >= C::NSTAGES) {
        if (!mbar_wait(&m->bar_empty[stage], ((st / C::NSTAGES) - 1) & 1, abort_flag)) break;
      }
      const int ib = (first_tile + st) * BN;
      uint8_t* dst = s_stream + stage * C::STAGE_BYTES;
      if (lane == 0) {
        mbar_arrive_expect_tx(&m->bar_full[stage], C::TILE_BYTES);
        for (int t = 0; t < C::NSTREAM; ++t)
          for (int b = 0; b < C::KB; ++b)
            tma_load_3d(dst + (b * C::NSTREAM + t) * (BN * 128), &p.tm[C::NSTAT + t],
                        &m->bar_full[stage], 64 * b, ib, bh);
      }
      // row vectors of the streamed query rows: [0] L*log2e, [1] D, [2] alpha, [3] E
      float* vec = reinterpret_cast<float*>(dst + C::TILE_BYTES);
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const int c = lane + 32 * q;
        const int gi = ib + c;
        const bool ok = gi < N;
        const size_t ri = (size_t)bh * N + (ok ? gi : 0);
        if constexpr (OP == ColOp::BwdDKDV) {
          vec[c] = ok ? p.lse[ri] * kLog2e : 0.f;
          vec[64 + c] = ok ? p.vec_in[ri] : 0.f;
        } else {
          vec[c] = ok ? p.lse[ri] * kLog2e : 0.f;
          vec[64 + c] = ok ? p.vec_in[2 * p.bhn + ri] : 0.f;  // D
          vec[128 + c] = ok ? p.vec_in[ri] : 0.f;             // alpha
          vec[192 + c] = ok ? p.vec_in[p.bhn + ri] : 0.f;     // E
        }
      }
      mbar_arrive(&m->bar_full[stage]);
      issued[stage] = st;
    }
    if (lane == 0 && *abort_flag) {
      for (int s = 0; s < C::NSTAGES; ++s)
        if (issued[s] >= 0) drain_wait(&m->bar_full[s], (issued[s] / C::NSTAGES) & 1);
      drain_wait(&m->bar_stat, 0);
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------ MMA issuer
    if (elect_lane0()) {
      const uint32_t id_n64 = idesc_bf16(128, 64, false);
      const uint32_t id_n128 = idesc_bf16(128, 128, false);
      const uint32_t id_b = idesc_bf16(128, D, true);
      const uint32_t tA = tmem + kColA;
      bool ok = mbar_wait(&m->bar_stat, 0, abort_flag);
      for (int st = 0; ok && st < nsteps; ++st) {
        const int stage = st % C::NSTAGES;
        if (!mbar_wait(&m->bar_full[stage], (st / C::NSTAGES) & 1, abort_flag)) break;
        tc_fence_after();
        const uint32_t sbase = smem_u32(s_stream + stage * C::STAGE_BYTES);
        const uint32_t stat = smem_u32(s_stat);
        auto stat_desc = [&](int t, int k) {
          return sdesc_sw128(stat + (t * C::KB + k / 4) * (BM * 128) + (k % 4) * 32, 16, 1024);
        };
        auto strm_desc = [&](int t, int k) {
          return sdesc_sw128(sbase + ((k / 4) * C::NSTREAM + t) * (BN * 128) + (k % 4) * 32, 16,
                             1024);
        };
        if constexpr (OP == ColOp::BobPass2) {
          // stationary: 0 K, 1 V, 2 U_K, 3 U_V ; stream: 0 Q, 1 U_Q, 2 dO
          for (int k = 0; k < D / 16; ++k)  // [S^T | F1^T] = K [Q ; U_Q]^T
            mma_ss(tA + 0, stat_desc(0, k), strm_desc(0, k), id_n128, k > 0);
          for (int k = 0; k < D / 16; ++k)  // F^T += U_K Q^T
            mma_ss(tA + 64, stat_desc(2, k), strm_desc(0, k), id_n64, 1);
          for (int k = 0; k < D / 16; ++k)  // dP^T = V dO^T
            mma_ss(tA + 128, stat_desc(1, k), strm_desc(2, k), id_n64, k > 0);
          for (int k = 0; k < D / 16; ++k)  // C^T = U_V dO^T
            mma_ss(tA + 192, stat_desc(3, k), strm_desc(2, k), id_n64, k > 0);
        } else {
          // stationary: 0 K, 1 V ; stream: 0 Q, 1 dO
          for (int k = 0; k < D / 16; ++k)
            mma_ss(tA + 0, stat_desc(0, k), strm_desc(0, k), id_n64, k > 0);
          for (int k = 0; k < D / 16; ++k)
            mma_ss(tA + 64, stat_desc(1, k), strm_desc(1, k), id_n64, k > 0);
        }
        mma_commit(&m->bar_sa);
        for (int h = 0; h < 2; ++h) {
          if (!mbar_wait(&m->bar_ew[h], st & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          for (int s = 2 * h; s < 2 * h + 2; ++s) {
            const uint32_t first = (st == 0 && s == 0) ? 0u : 1u;
            auto mn_desc = [&](int t) {
              return sdesc_sw128(sbase + t * (BN * 128) + s * 2048, C::NSTREAM * BN * 128, 1024);
            };
            if constexpr (OP == ColOp::BobPass2) {
              mma_ts(tmem + D, tA + 16 * s, mn_desc(2), id_b, first);       // Vtil += (P o h)^T dO
              mma_ts(tmem + 0, tA + 16 * s + 8, mn_desc(0), id_b, first);   // Ktil += Stil^T Q
              mma_ts(tmem + 0, tA + 128 + 16 * s, mn_desc(1), id_b, 1);     //      += dS^T U_Q
            } else {
              mma_ts(tmem + D, tA + 16 * s, mn_desc(1), id_b, first);       // dV += P^T dO
              mma_ts(tmem + 0, tA + 16 * s + 8, mn_desc(0), id_b, first);   // dK += dS^T Q
            }
          }
        }
        if (!ok) break;
        mma_commit(&m->bar_empty[stage]);
      }
      mma_commit(&m->bar_acc);
      if (*abort_flag) drain_wait(&m->bar_acc, 0);
    }
  } else {
    // ------------------------------------------------------------ elementwise
    const int wg = warp >> 2;
    const int r = 32 * (warp & 3) + (tid & 31);
    const int gj = j0 + r;  // stationary key row
    const bool row_ok = gj < N;
    const uint32_t ta = lane_base_addr(tmem, warp);
    const uint32_t tA = ta + kColA;
    const float tau = p.scale;
    const float sl2 = tau * kLog2e;
    bool ok = true;
    for (int st = 0; st < nsteps; ++st) {
      const int stage = st % C::NSTAGES;
      // the row vectors were written by the producer: acquire them explicitly
      if (!mbar_wait(&m->bar_full[stage], (st / C::NSTAGES) & 1, abort_flag) ||
          !mbar_wait(&m->bar_sa, st & 1, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const float* vec = reinterpret_cast<const float*>(s_stream + stage * C::STAGE_BYTES +
                                                        C::TILE_BYTES);
      const int ib = (first_tile + st) * BN;
      const bool need_mask = (!row_ok) || (ib + BN > N) || (p.causal && ib < gj);
      for (int h = 0; h < 2; ++h) {
        const int s = 2 * h + wg;
        const int c0 = 16 * s;
        if constexpr (OP == ColOp::BobPass2) {
          uint32_t rS[16], rF[16], rdP[16], rC[16];
          tmem_ld16(tA + 0 + c0, rS);
          tmem_ld16(tA + 64 + c0, rF);
          tmem_ld16(tA + 128 + c0, rdP);
          tmem_ld16(tA + 192 + c0, rC);
          tmem_ld_wait(rS);
          reg_dep(rF);
          reg_dep(rdP);
          reg_dep(rC);
          uint32_t oPh[8], oSt[8], odS[8];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            float ph[2], stl[2], ds[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int cc = c0 + c + e;
              const int gi = ib + cc;
              float pr = ex2(fmaf(bits_f(rS[c + e]), sl2, -vec[cc]));
              if (need_mask && !(row_ok && gi < N && (!p.causal || gj <= gi))) pr = 0.f;
              const float Dv = vec[64 + cc], al = vec[128 + cc], Ev = vec[192 + cc];
              const float f = tau * bits_f(rF[c + e]);
              const float dp = bits_f(rdP[c + e]);
              const float t = dp - Dv;
              // Ptil = C + F (dP - D) - alpha dP ; Stil = P (Ptil - E) ; h = F - alpha
              const float pt = fmaf(-al, dp, fmaf(f, t, bits_f(rC[c + e])));
              ph[e] = pr * (f - al);
              stl[e] = pr * (pt - Ev);
              ds[e] = pr * t;
            }
            oPh[c / 2] = pack_bf16(ph[0], ph[1]);
            oSt[c / 2] = pack_bf16(stl[0], stl[1]);
            odS[c / 2] = pack_bf16(ds[0], ds[1]);
          }
          tmem_st8(tA + c0, oPh);
          tmem_st8(tA + c0 + 8, oSt);
          tmem_st8(tA + 128 + c0, odS);
        } else {
          uint32_t rS[16], rdP[16];
          tmem_ld16(tA + 0 + c0, rS);
          tmem_ld16(tA + 64 + c0, rdP);
          tmem_ld_wait(rS);
          reg_dep(rdP);
          uint32_t oP[8], odS[8];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            float pv[2], ds[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int cc = c0 + c + e;
              const int gi = ib + cc;
              float pr = ex2(fmaf(bits_f(rS[c + e]), sl2, -vec[cc]));
              if (need_mask && !(row_ok && gi < N && (!p.causal || gj <= gi))) pr = 0.f;
              pv[e] = pr;
              ds[e] = pr * (bits_f(rdP[c + e]) - vec[64 + cc]);
            }
            oP[c / 2] = pack_bf16(pv[0], pv[1]);
            odS[c / 2] = pack_bf16(ds[0], ds[1]);
          }
          tmem_st8(tA + c0, oP);
          tmem_st8(tA + c0 + 8, odS);
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&m->bar_ew[h]);
      }
    }
    if (ok) ok = mbar_wait(&m->bar_acc, 0, abort_flag);
    tc_fence_after();
    if (ok) {
      const size_t rowoff = ((size_t)bh * N + (size_t)(row_ok ? gj : 0)) * D;
#pragma unroll 1
      for (int q = 0; q < D / 32; ++q) {
        const int cc = wg * (D / 2) + 16 * q;
        uint32_t rK[16], rV[16];
        tmem_ld16(ta + cc, rK);
        tmem_ld16(ta + D + cc, rV);
        tmem_ld_wait(rK);
        reg_dep(rV);
        if (row_ok) {
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
