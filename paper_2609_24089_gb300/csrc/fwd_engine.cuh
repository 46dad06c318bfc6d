// fwd_engine.cuh -- forward attention (eq. 1) on sm_103a with two query
// tiles per CTA.
//
// A CTA owns 2 x 128 query rows of one head (query tiles 0 and 1) and streams
// 128-key tiles of K and V through a ring of stream stages.  Each query tile
// has its own score buffer S_q (128 TMEM columns) and accumulator O_q, and
// two softmax warpgroups, one per half of the key tile (64 keys each), whose
// thread i holds query row i.  Per key tile T and query tile q:
//   X   S_q(T) = Q_q K(T)^T                 (N = 128, issuer X)
//   WGs m, l (online softmax): each half's row maxima are exchanged through
//       shared memory, so both halves take the same running maximum; then
//       P = 2^(S tau log2 e - m) is written as bf16 over the first 64
//       columns of S_q (both halves hold their S in registers by then), or
//       at d = 64 into 64 TMEM columns of its own
//   Y   O_q += P_q(T) V(T)                  (A from TMEM, issuer Y)
// X issues S_q(T+1) once O_q += P_q(T) V(T) has completed (it overwrites
// P_q(T)); at d = 64 P_q has TMEM columns of its own, and S_q(T+1) follows
// as soon as the softmax holds S_q(T) in registers.  The two query tiles'
// chains interleave, so the tensor pipe works on one tile while the other's
// softmax runs.  The running maximum is raised lazily (by more than
// kFwdSlack, so P <= 2^kFwdSlack); O_q is then rescaled by the first half's
// warpgroup after the MMAs into it have completed.  Each half keeps the row
// sum of its own keys; the epilogue adds the two.
//
// Roles (608 threads): warps 0-7 softmax of query tile 0 (keys 0-63, then
// 64-127), warps 8-15 of tile 1 (warp w reads TMEM lanes 32 (w % 4) .. +31),
// warp 16 TMA producer, warp 17 issuer X, warp 18 issuer Y.  Every wait is
// bounded.
#pragma once

#include "attn_engine.cuh"

namespace fbob {

constexpr int kFwdRows = 2 * BM;  // query rows per CTA
constexpr int BN2 = 128;          // keys per streamed tile
constexpr float kFwdSlack = 8.f;
// warps 0-15: softmax, four warpgroups (query tile q = g / 2, key half g % 2);
// then the TMA producer and the two MMA issuers
constexpr int kFwdProducer = 16, kFwdX = 17, kFwdY = 18;
constexpr int kFwdThreads = 19 * 32;

template <int D>
struct FwdCfg {
  static constexpr int KB = D / 64;
  static constexpr int STAT_BYTES = 2 * KB * BM * 128;     // Q_0, Q_1
  static constexpr int STAGE_BYTES = 2 * KB * BN2 * 128;   // K, V
  static constexpr int NSTAGES = D == 64 ? 4 : 2;
  // d = 64 leaves TMEM room for separate P buffers (O 2 x 64, S 2 x 128, P
  // 2 x 64 columns): S_q(T+1) is then issued as soon as both softmax halves
  // hold S_q(T) in registers, instead of after O_q += P_q(T) V(T) has
  // completed, which takes the S MMA off each query tile's critical path
  static constexpr bool SEP_P = D == 64;
  // bookkeeping, then the row-maximum exchange [tile parity][q][half][row]
  // and the row-sum exchange [q][half][row]
  static constexpr int MISC_BYTES = 256 + 8 * BM * 4 + 4 * BM * 4;
  static constexpr int SMEM_BYTES = STAT_BYTES + NSTAGES * STAGE_BYTES + MISC_BYTES;
};

struct FwdMisc {
  uint64_t bar_stat;
  uint64_t full[kMaxStages];
  uint64_t empty[kMaxStages];
  uint64_t s_full[2];  // S_q(T) computed (issuer X)
  uint64_t p_full[2];  // P_q(T) written (128 softmax threads)
  uint64_t o_done[2];  // O_q += P_q(T) V(T) completed (issuer Y)
  uint64_t xq[2][2];   // [q][tile parity]: both halves posted their row maxima
  uint64_t xl[2];      // [q]: both halves posted their row sums (epilogue)
  uint64_t bar_acc;    // every MMA of both issuers completed (abort drain)
  uint32_t tmem_base;
  uint32_t pad;
  WaitCtl wctl;
};
static_assert(sizeof(FwdMisc) <= 256, "FwdMisc must fit the MISC area");

// max(a, b, c) in one three-input instruction
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float r;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
  return r;
}

// TMEM columns: O_q at q D, S_q at 256 + 128 q; with FwdCfg::SEP_P, P_q at
// 128 + 64 q (otherwise P_q is written over the first 64 columns of S_q).
constexpr uint32_t kColS2 = 256;
constexpr uint32_t kColP = 128;

template <int D, bool DROP, int DG>
__global__ void __launch_bounds__(kFwdThreads, 1) fwd_engine(const __grid_constant__ EngineParams p) {
  using C = FwdCfg<D>;
  static_assert(DG == D || (DG == 32 && D == 64), "global head dim 32 runs in 64-wide tiles");
  static_assert(C::NSTAGES >= 2 && C::NSTAGES <= kMaxStages, "the stage barriers hold kMaxStages stages");
  extern __shared__ __align__(1024) uint8_t smem[];
  uint8_t* s_stat = smem;
  uint8_t* s_stream = smem + C::STAT_BYTES;
  FwdMisc* m = reinterpret_cast<FwdMisc*>(s_stream + C::NSTAGES * C::STAGE_BYTES);
  float* s_xm = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(m) + 256);  // 8 x BM
  float* s_xl = s_xm + 8 * BM;                                                  // 4 x BM

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  if ((smem_u32(smem) & 1023u) != 0) {
    if (tid == 0) atomicOr(&g_fbob_error_word, kDevErrBadLaunch);
    return;
  }
  // ---- tile decode: 256 query rows; with the causal mask the row blocks
  // with the most keys go first
  const int N = p.N;
  const int lin = blockIdx.x;
  int rbi, bh;
  cta_order(p, lin, rbi, bh);
  const int rb = p.causal ? (p.nblk - 1 - rbi) : rbi;
  const int bh_kv = p.Hkv == p.H ? bh : (bh / p.H) * p.Hkv + (bh % p.H) / (p.H / p.Hkv);
  const int i0 = rb * kFwdRows;
  // per query tile: active, and its key tiles [tq0, tq1] (the union of its
  // rows' bands within their sequences)
  bool act[2];
  int tq0[2], tq1[2];
#pragma unroll
  for (int q = 0; q < 2; ++q) {
    const int first = i0 + BM * q;
    act[q] = first < N;
    tq0[q] = 0;
    tq1[q] = -1;
    if (act[q]) {
      const int last = min(first + BM, N) - 1;
      int s0, e0, s1, e1;
      seq_bounds(p, first, s0, e0);
      seq_bounds(p, last, s1, e1);
      const int lo = max(s0, p.wl < 0 ? 0 : first - p.wl);
      const int hi = min(e1, p.wr < 0 ? N : last + p.wr + 1);
      tq0[q] = lo / BN2;
      tq1[q] = (hi - 1) / BN2;
    }
  }
  const int T0 = act[1] ? min(tq0[0], tq0[1]) : tq0[0];
  const int T1 = act[1] ? max(tq1[0], tq1[1]) : tq1[0];
  // block-sparse mask (128 x 128 blocks: a key tile is one key block, query
  // tile q is query block 2 rb + q): query tile q takes key tile T only if
  // that block pair is set, and a key tile neither takes is not streamed
  const uint8_t* bm = p.bmask;
  auto part = [&](int q, int T) {
    return act[q] && T >= tq0[q] && T <= tq1[q] &&
           (bm == nullptr || bm[(size_t)(2 * rb + q) * p.nbm + T] != 0);
  };
  // next streamed key tile >= T (T1 + 1 if none)
  auto next_T = [&](int T) {
    if (bm != nullptr)
      while (T <= T1 && !part(0, T) && !part(1, T)) ++T;
    return T;
  };
  int nsteps = T1 - T0 + 1;
  if (bm != nullptr) {
    nsteps = 0;
    for (int T = T0; T <= T1; ++T) nsteps += (part(0, T) || part(1, T)) ? 1 : 0;
  }

  if (tid == 0) {
    m->wctl.abort = 0;
    m->wctl.limit_ns = p.wait_limit_ns;
    mbar_init(&m->bar_stat, 1);
    for (int s = 0; s < C::NSTAGES; ++s) {
      mbar_init(&m->full[s], 1);
      mbar_init(&m->empty[s], 2);  // issuers X and Y
    }
    for (int q = 0; q < 2; ++q) {
      mbar_init(&m->s_full[q], 1);
      mbar_init(&m->p_full[q], 2 * BM);  // both key halves
      mbar_init(&m->o_done[q], 1);
      mbar_init(&m->xq[q][0], 2 * BM);
      mbar_init(&m->xq[q][1], 2 * BM);
      mbar_init(&m->xl[q], 2 * BM);
    }
    mbar_init(&m->bar_acc, 2);
    fence_mbar_init();
  }
  if (warp == kFwdX) {
    tmem_alloc(&m->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = m->tmem_base;
  WaitCtl* wctl = &m->wctl;
  volatile int* abort_flag = &m->wctl.abort;

  if (warp == kFwdProducer) {
    // ------------------------------------------------------------ producer
    if (elect_lane0() && !p.inject_stall) {
      for (int t = 0; t < 3; ++t) tma_prefetch_desc(&p.tm[t]);
      mbar_arrive_expect_tx(&m->bar_stat, C::STAT_BYTES);
      for (int q = 0; q < 2; ++q)
        for (int b = 0; b < C::KB; ++b)
          tma_load_3d(s_stat + (q * C::KB + b) * (BM * 128), &p.tm[0], &m->bar_stat, 64 * b,
                      i0 + BM * q, bh);
      int issued[kMaxStages] = {-1, -1, -1, -1};
      int T = T0 - 1;
      for (int st = 0; st < nsteps; ++st) {
        const int stage = st % C::NSTAGES;
        if (st >= C::NSTAGES &&
            !mbar_wait(&m->empty[stage], ((st / C::NSTAGES) - 1) & 1, wctl))
          break;
        T = next_T(T + 1);
        const int j0 = T * BN2;
        uint8_t* dst = s_stream + stage * C::STAGE_BYTES;
        mbar_arrive_expect_tx(&m->full[stage], C::STAGE_BYTES);
        for (int t = 0; t < 2; ++t)        // K, V
          for (int b = 0; b < C::KB; ++b)
            for (int h = 0; h < 2; ++h)    // two 64-row boxes
              tma_load_3d(dst + (t * C::KB + b) * (BN2 * 128) + h * (BN * 128), &p.tm[1 + t],
                          &m->full[stage], 64 * b, j0 + BN * h, bh_kv);
        issued[stage] = st;
      }
      if (*abort_flag) {
        for (int s = 0; s < C::NSTAGES; ++s)
          if (issued[s] >= 0) drain_wait(&m->full[s], (issued[s] / C::NSTAGES) & 1);
        drain_wait(&m->bar_stat, 0);
      }
    }
  } else if (warp == kFwdX || warp == kFwdY) {
    // ------------------------------------------------------------ MMA issuers
    if (elect_lane0()) {
      constexpr uint32_t id_s = idesc_bf16(128, BN2, false);
      constexpr uint32_t id_o = idesc_bf16(128, D, true);
      bool ok = true;
      if (warp == kFwdX) {
        // ---------------- issuer X: S_q(T) = Q_q K(T)^T
        const uint64_t qd0 = sdesc_sw128(smem_u32(s_stat), 16, 1024);
        ok = mbar_wait(&m->bar_stat, 0, wctl);
        int T = T0 - 1, kq[2] = {0, 0};  // key tile; tiles each query tile has taken
        for (int st = 0; ok && st < nsteps; ++st) {
          T = next_T(T + 1);
          const int stage = st % C::NSTAGES;
          if (!mbar_wait(&m->full[stage], (st / C::NSTAGES) & 1, wctl)) break;
          const uint64_t kd0 =
              sdesc_sw128(smem_u32(s_stream + stage * C::STAGE_BYTES), 16, 1024);
          for (int q = 0; q < 2 && ok; ++q) {
            if (!part(q, T)) continue;
            const int k = kq[q]++;
            if (k >= 1) {
              // SEP_P: S_q(T) overwrites S_q(T-1): wait until both softmax
              // halves hold it (their row-maximum exchange of tile T-1);
              // otherwise S_q(T) overwrites P_q(T-1): wait for O_q += P_q(T-1) V
              const bool w = C::SEP_P
                                 ? mbar_wait(&m->xq[q][(k - 1) & 1], ((k - 1) >> 1) & 1, wctl)
                                 : mbar_wait(&m->o_done[q], (k - 1) & 1, wctl);
              if (!w) {
                ok = false;
                break;
              }
            }
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint64_t qd =
                  qd0 + (uint64_t)(((q * C::KB + kk / 4) * (BM * 128) + (kk % 4) * 32) >> 4);
              const uint64_t kd = kd0 + (uint64_t)(((kk / 4) * (BN2 * 128) + (kk % 4) * 32) >> 4);
              mma_ss(tmem + kColS2 + 128 * q, qd, kd, id_s, kk > 0);
            }
            mma_commit(&m->s_full[q]);
          }
          if (!ok) break;
          mma_commit(&m->empty[stage]);
        }
      } else {
        // ---------------- issuer Y: O_q += P_q(T) V(T)
        int T = T0 - 1, kq[2] = {0, 0};
        for (int st = 0; ok && st < nsteps; ++st) {
          T = next_T(T + 1);
          const int stage = st % C::NSTAGES;
          if (!mbar_wait(&m->full[stage], (st / C::NSTAGES) & 1, wctl)) break;
          // V of this stage: MN-major, 64-wide boxes BN2 * 128 bytes apart
          const uint64_t vd0 = sdesc_sw128(
              smem_u32(s_stream + stage * C::STAGE_BYTES) + C::KB * (BN2 * 128), BN2 * 128, 1024);
          for (int q = 0; q < 2 && ok; ++q) {
            if (!part(q, T)) continue;
            const int k = kq[q]++;
            if (!mbar_wait(&m->p_full[q], k & 1, wctl)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int ks = 0; ks < BN2 / 16; ++ks)
              mma_ts(tmem + q * D, tmem + (C::SEP_P ? kColP + 64 * q : kColS2 + 128 * q) + 8 * ks,
                     vd0 + (uint64_t)((ks * 2048) >> 4), id_o, (k == 0 && ks == 0) ? 0u : 1u);
            mma_commit(&m->o_done[q]);
          }
          if (!ok) break;
          mma_commit(&m->empty[stage]);
        }
      }
      mma_commit(&m->bar_acc);
      if (*abort_flag) drain_wait(&m->bar_acc, 0);
    }
  } else {
    // ------------------------------------------------------------ softmax
    // warpgroup g: query tile q = g / 2, key half hf = g % 2 (keys 64 hf ..
    // 64 hf + 63 of each tile); thread: one row of the tile (TMEM lane)
    const int g = warp >> 2;
    const int q = g >> 1, hf = g & 1;
    const int r = 32 * (warp & 3) + (tid & 31);
    const int gi = i0 + BM * q + r;
    const bool row_ok = gi < N;
    int jlo = 0, jhi = 0;  // this row's valid keys [jlo, jhi)
    if (row_ok) {
      seq_bounds(p, gi, jlo, jhi);
      if (p.wl >= 0) jlo = max(jlo, gi - p.wl);
      if (p.wr >= 0) jhi = min(jhi, gi + p.wr + 1);
    }
    const uint32_t ta = lane_base_addr(tmem, warp);
    const uint32_t scol = kColS2 + 128 * q, ocol = (uint32_t)(q * D);
    const float sl2 = p.scale * kLog2e;
    const DropKey dkey = {p.drop_rk, p.drop_tlow4, p.drop_tmask};
    auto ew_wait = [&](uint64_t* bar, uint32_t par) -> bool {
      const bool w = mbar_wait(bar, par, wctl);
      return __all_sync(0xffffffffu, w);  // the warp leaves together
    };
    float mrow = -INFINITY, lrow = 0.f;  // (lrow: this half's keys)
    bool ok = act[q];
    // key tiles this query tile takes (with a block-sparse mask, those of its
    // set blocks)
    int nq = act[q] ? tq1[q] - tq0[q] + 1 : 0;
    if (bm != nullptr && act[q]) {
      nq = 0;
      for (int T = tq0[q]; T <= tq1[q]; ++T) nq += part(q, T) ? 1 : 0;
    }
    int Tq = tq0[q] - 1;
    for (int k = 0; ok && k < nq; ++k) {
      ++Tq;
      if (p.bmask != nullptr) {  // the next set block of this query block (gi / 128)
        const uint8_t* bq = p.bmask + (size_t)(gi >> 7) * p.nbm;
        while (Tq < p.nbm - 1 && bq[Tq] == 0) ++Tq;
      }
      const int jt = Tq * BN2 + 64 * hf;  // first key of this half
      // dropout keep bits of the half's 4 x 16 keys, formed while S_q(T) is computed
      uint32_t kb[4];
      if constexpr (DROP) {
#pragma unroll
        for (int c = 0; c < 4; ++c)
          kb[c] = keep_row16(gi, jt + 16 * c, (uint32_t)(p.head0 + bh), dkey);
      }
      if (!ew_wait(&m->s_full[q], k & 1)) {
        ok = false;
        break;
      }
      tc_fence_after();
      uint32_t rS[4][16];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld16(ta + scol + 64 * hf + 16 * c, rS[c]);
      tmem_ld_wait(rS[0]);
#pragma unroll
      for (int c = 1; c < 4; ++c) reg_dep(rS[c]);
      float mraw = -INFINITY;
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const int mlo = jlo - (jt + 16 * c), mhi = jhi - (jt + 16 * c);
        if (mlo > 0 || mhi < 16) mask16(rS[c], mlo, mhi);
#pragma unroll
        for (int e = 0; e < 16; e += 2) mraw = fmax3(mraw, bits_f(rS[c][e]), bits_f(rS[c][e + 1]));
      }
      // the row maximum over both halves: post this half's, wait for both
      // (which also means both halves hold their S in registers, so P may be
      // written over S), read the other's
      float* xm = s_xm + ((k & 1) * 4 + q * 2) * BM;
      xm[hf * BM + r] = mraw;
      tc_fence_before();
      mbar_arrive(&m->xq[q][k & 1]);
      if (!ew_wait(&m->xq[q][k & 1], (k >> 1) & 1)) {
        ok = false;
        break;
      }
      tc_fence_after();
      mraw = fmaxf(mraw, xm[(1 - hf) * BM + r]);
      const float mt = mraw * sl2;
      const bool raise = mt > mrow + kFwdSlack;  // also the first tile with a valid key
      const bool rescale = raise && mrow != -INFINITY;
      if (__any_sync(0xffffffffu, rescale)) {  // (the same decision in both halves)
        if (hf == 0) {  // half 0 rescales O_q
          // every MMA into O_q so far (tiles before k) must have completed
          if (!ew_wait(&m->o_done[q], (k - 1) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const float f = rescale ? ex2(mrow - mt) : 1.f;
#pragma unroll 1
          for (int c = 0; c < D / 16; ++c) {
            uint32_t o[16];
            tmem_ld16(ta + ocol + 16 * c, o);
            tmem_ld_wait(o);
            uint32_t lo8[8], hi8[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              lo8[e] = __float_as_uint(bits_f(o[e]) * f);
              hi8[e] = __float_as_uint(bits_f(o[8 + e]) * f);
            }
            tmem_st8(ta + ocol + 16 * c, lo8);
            tmem_st8(ta + ocol + 16 * c + 8, hi8);
          }
          tmem_st_wait();
        }
        if (rescale) lrow *= ex2(mrow - mt);
      }
      if (raise) mrow = mt;
      // no valid key yet: every score is -inf, so any finite m gives P = 0
      const float nm = mrow == -INFINITY ? 0.f : -mrow;
      // SEP_P: P_q(T) overwrites P_q(T-1): wait for O_q += P_q(T-1) V
      if (C::SEP_P && k >= 1) {
        if (!ew_wait(&m->o_done[q], (k - 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
      }
      const uint32_t pcol = C::SEP_P ? kColP + 64 * q : scol;
      // pairs of scores through the packed f32x2 FMA and add (half the
      // instructions of scalar ones; the same roundings)
      const float2 sl2v = make_float2(sl2, sl2), nmv = make_float2(nm, nm);
      float2 ps = make_float2(0.f, 0.f);  // even and odd keys' partial sums
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t oP[8];
        const uint32_t kbc = DROP ? kb[c] : 0u;
#pragma unroll
        for (int e = 0; e < 16; e += 2) {
          const float2 x = __ffma2_rn(make_float2(bits_f(rS[c][e]), bits_f(rS[c][e + 1])), sl2v, nmv);
          float p0 = ex2(x.x);
          float p1 = ex2(x.y);
          ps = __fadd2_rn(ps, make_float2(p0, p1));  // L over the ungated P
          if constexpr (DROP) {  // O = sigma (R o P) V: sigma in the epilogue
            if (!((kbc >> e) & 1u)) p0 = 0.f;
            if (!((kbc >> (e + 1)) & 1u)) p1 = 0.f;
          }
          oP[e / 2] = pack_bf16(p0, p1);
        }
        // P of keys 64 hf + 16c .. + 15 in P columns 32 hf + 8c .. + 7
        tmem_st8(ta + pcol + 32 * hf + 8 * c, oP);
      }
      lrow += ps.x + ps.y;
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&m->p_full[q]);
    }
    // ---- epilogue: l over both halves; O = O_q / l (times sigma with
    // dropout), each half storing half of the columns; L = m + log2 l
    if (ok && nq > 0) ok = ew_wait(&m->o_done[q], (nq - 1) & 1);
    if (ok) {
      s_xl[(q * 2 + hf) * BM + r] = lrow;
      mbar_arrive(&m->xl[q]);
      ok = ew_wait(&m->xl[q], 0);
    }
    if (ok && *abort_flag) ok = false;
    tc_fence_after();
    if (ok) {
      const float lt = lrow + s_xl[(q * 2 + 1 - hf) * BM + r];
      const float inv = row_ok ? (DROP ? p.drop_sigma : 1.f) / lt : 0.f;
      const size_t rowoff = ((size_t)bh * N + (size_t)(row_ok ? gi : 0)) * DG;
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        const int cc = hf * (D / 2) + 16 * c;
        uint32_t o[16];
        tmem_ld16(ta + ocol + cc, o);
        tmem_ld_wait(o);
        if (row_ok && cc < DG) {
          float v[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) v[e] = bits_f(o[e]) * inv;
          store_row16(p.out0 + rowoff + cc, v);
        }
      }
      if (row_ok && hf == 0) p.vec_out[(size_t)bh * N + gi] = (mrow + __log2f(lt)) * kLn2;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kFwdX) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace fbob
