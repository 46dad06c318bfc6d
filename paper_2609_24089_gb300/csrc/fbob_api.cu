// fbob_api.cu -- the C ABI declared in include/fbob.h: argument validation,
// TMA tensor-map construction and kernel launches.  Allocates no device memory.
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "../../include/fbob.h"
#include "launch.h"
#include "wide_launch.h"

namespace fbob {
namespace {

constexpr int64_t kMaxN = int64_t(1) << 24;
constexpr int64_t kMaxBH = int64_t(1) << 24;

constexpr int kNumEntries = 10;
std::atomic<int> g_launches[kNumEntries] = {{-1}, {-1}, {-1}, {-1}, {-1},
                                            {-1}, {-1}, {-1}, {-1}, {-1}};
enum Entry {
  kEntFwd = 0, kEntBwd, kEntBob, kEntPass1, kEntPass2, kEntRowStats, kEntPass1D, kEntBobHost,
  kEntBobHostNoAlloc, kEntPass1Fused
};

// Staging memory of fbob_attn_bob_host_noalloc: a fixed device array, so that
// call allocates nothing.  Its module holds no kernels; the array is placed
// when the module is loaded on a device: at the first address lookup under
// lazy module loading (the CUDA default), at context creation under
// CUDA_MODULE_LOADING=EAGER.
constexpr int64_t kNoAllocBytes = int64_t(64) << 20;
__device__ __align__(256) uint8_t g_noalloc_scratch[kNoAllocBytes];

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// [BH, N, d] bf16 tensor viewed as 3-D (d innermost), box = 64 columns x `rows`,
// 128-byte swizzle, zero fill out of bounds (with d = 32 the box's columns
// 32..63 lie outside the tensor and arrive as zeros).
bool make_map(CUtensorMap* m, const void* base, int64_t BH, int64_t N, int64_t d, int rows) {
  auto enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)N, (cuuint64_t)BH};
  cuuint64_t strides[2] = {(cuuint64_t)(d * 2), (cuuint64_t)(N * d * 2)};
  cuuint32_t box[3] = {64, (cuuint32_t)rows, 1};
  cuuint32_t es[3] = {1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
                   box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

struct Span {
  uintptr_t lo, hi;
};

bool overlaps(const Span& a, const Span& b) { return a.lo < b.hi && b.lo < a.hi; }

// Shape rules of include/fbob.h.  Returns FBOB_OK, or the status to report;
// *empty is set when B*H*N == 0.
int check_shape(const fbob_shape* s, bool* empty) {
  if (!s) return FBOB_ERR_INVALID_ARGUMENT;
  if (s->B < 0 || s->H < 0 || s->N < 0 || s->d <= 0) return FBOB_ERR_INVALID_ARGUMENT;
  if (!(std::isfinite(s->scale) && s->scale > 0.f)) return FBOB_ERR_INVALID_ARGUMENT;
  if (s->causal != 0 && s->causal != 1) return FBOB_ERR_INVALID_ARGUMENT;
  if (s->window_left < -1 || s->window_right < -1) return FBOB_ERR_INVALID_ARGUMENT;
  if (s->H_kv < 0 || (s->H_kv > 0 && (s->H % s->H_kv) != 0)) return FBOB_ERR_INVALID_ARGUMENT;
  if (!(s->dropout_p >= 0.0 && s->dropout_p < 1.0)) return FBOB_ERR_INVALID_ARGUMENT;
  if (s->seq_offsets == nullptr ? s->num_seqs != 0
                                : (s->num_seqs < 1 || s->num_seqs > kMaxN ||
                                   (reinterpret_cast<uintptr_t>(s->seq_offsets) & 3u) != 0))
    return FBOB_ERR_INVALID_ARGUMENT;
  if (s->d != 32 && s->d != 64 && s->d != 128 && s->d != 256) return FBOB_ERR_UNSUPPORTED;
  if (s->N > kMaxN) return FBOB_ERR_INVALID_ARGUMENT;
  if (s->B > kMaxBH || s->H > kMaxBH || s->B * s->H > kMaxBH) return FBOB_ERR_INVALID_ARGUMENT;
  // the largest launch (two CTAs per 128-row block for the split one-sweep
  // Pass 1) must fit a grid
  if ((s->N + 127) / 128 * s->B * s->H * 2 > (int64_t)0x7FFFFFFF) return FBOB_ERR_INVALID_ARGUMENT;
  *empty = (s->B * s->H * s->N) == 0;
  return FBOB_OK;
}

// Null / alignment / overlap checks: `in` and `out` are (pointer, bytes) lists.
int check_ptrs(const void* const* in, const int64_t* in_bytes, int nin, void* const* out,
               const int64_t* out_bytes, int nout) {
  Span spans[16];
  int ns = 0;
  for (int t = 0; t < nin; ++t) {
    if (!in[t] || (reinterpret_cast<uintptr_t>(in[t]) & 15u)) return FBOB_ERR_INVALID_ARGUMENT;
    spans[ns++] = {reinterpret_cast<uintptr_t>(in[t]),
                   reinterpret_cast<uintptr_t>(in[t]) + (uintptr_t)in_bytes[t]};
  }
  const int first_out = ns;
  for (int t = 0; t < nout; ++t) {
    if (!out[t] || (reinterpret_cast<uintptr_t>(out[t]) & 15u)) return FBOB_ERR_INVALID_ARGUMENT;
    spans[ns++] = {reinterpret_cast<uintptr_t>(out[t]),
                   reinterpret_cast<uintptr_t>(out[t]) + (uintptr_t)out_bytes[t]};
  }
  for (int a = first_out; a < ns; ++a)
    for (int b = 0; b < ns; ++b)
      if (a != b && overlaps(spans[a], spans[b])) return FBOB_ERR_INVALID_ARGUMENT;
  return FBOB_OK;
}

// Bound of every device-side wait (FBOB_WAIT_LIMIT_MS, default 2000 ms) and
// the host-side stall injection used to test failure detection
// (FBOB_INJECT_STALL=1: the kernels' producers issue no loads, so every wait
// expires and the call reports FBOB_ERR_DEVICE_TIMEOUT).  Read at each call.
void debug_controls(EngineParams* p) {
  unsigned long long ms = 2000;
  if (const char* e = std::getenv("FBOB_WAIT_LIMIT_MS")) {
    const long long v = std::atoll(e);
    if (v > 0 && v <= 60000) ms = (unsigned long long)v;
  }
  p->wait_limit_ns = ms * 1000000ull;
  const char* inj = std::getenv("FBOB_INJECT_STALL");
  p->inject_stall = (inj && inj[0] == '1') ? 1 : 0;
}

// CTA order per kernel (heads per group, cta_order in attn_engine.cuh), from
// measurements on GB300.  Pass 1 takes heads in groups whose streamed K, U_K,
// V, U_V (4 N d bf16 per head) fit in about 96 MiB of the 129 MB L2, at most
// four: the CTAs in flight then share a few heads' streams in L2 and no
// head's longest row blocks are left to the end (n16k_d128_causal, 16.8 MB
// per head: groups of four, 0.4 % faster than one head at a time and 2 %
// faster than all heads; N = 262,144 at d = 64, 134 MB per head: one head at
// a time, 4.4 % faster than groups of four).  Pass 2 and the helper kernels
// balance the causal work better with every head's longest block first (all
// heads).
void choose_order(EngineParams* p, int heads_per_group) {
  p->head_group = heads_per_group < 1 ? 1 : (heads_per_group > p->BH ? p->BH : heads_per_group);
  if (p->head_group < 1) p->head_group = 1;
}
int pass1_heads_per_group(const fbob_shape* s) {
  const double per_head = 8.0 * (double)s->N * (double)s->d;  // bytes streamed per head
  const double g = 96.0 * 1048576.0 / (per_head > 1.0 ? per_head : 1.0);
  return g >= 4.0 ? 4 : (g >= 1.0 ? (int)g : 1);
}

// key/value heads per batch entry
int64_t kv_heads(const fbob_shape* s) { return s->H_kv > 0 ? s->H_kv : s->H; }

int n_blocks(int64_t N, int rows) { return (int)((N + rows - 1) / rows); }

// dropout byte threshold t = round(256 p), at most 255; 0 = no dropout
uint32_t drop_threshold(const fbob_shape* s) {
  const double t = std::floor(256.0 * s->dropout_p + 0.5);
  return t >= 255.0 ? 255u : (uint32_t)t;
}

bool has_dropout(const fbob_shape* s) { return drop_threshold(s) != 0; }

EngineParams base_params(const fbob_shape* s) {
  EngineParams p;
  std::memset(&p, 0, sizeof(p));
  p.N = (int)s->N;
  p.BH = (int)(s->B * s->H);
  p.causal = s->causal;
  p.wl = s->window_left;
  p.wr = s->causal ? 0 : s->window_right;
  p.seq_off = s->seq_offsets;
  p.nseq = (int)s->num_seqs;
  p.bmask = s->block_mask;
  p.nbm = n_blocks(s->N, BM);
  p.H = (int)s->H;
  p.Hkv = (int)kv_heads(s);
  p.scale = s->scale;
  p.bhn = s->B * s->H * s->N;
  const uint32_t t = drop_threshold(s);
  uint32_t k0 = (uint32_t)(s->dropout_seed & 0xFFFFFFFFull);
  uint32_t k1 = (uint32_t)(s->dropout_seed >> 32);
  for (int r = 0; r < 10; ++r) {  // Philox4x32-10 key schedule (Weyl sequence)
    p.drop_rk[2 * r] = k0;
    p.drop_rk[2 * r + 1] = k1;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  p.drop_tlow4 = (t & 0x7Fu) * 0x01010101u;
  p.drop_tmask = t < 128 ? 0xFFFFFFFFu : 0u;
  p.drop_sigma = t ? (float)(256.0 / (256.0 - (double)t)) : 1.f;
  debug_controls(&p);
  return p;
}

int launch_status(cudaError_t e) { return e == cudaSuccess ? FBOB_OK : FBOB_ERR_CUDA; }

// ---- head dimension 256 (wide_engine.cuh): stationary shared-memory
// operands in 128-row boxes, streamed tensors in 32-row boxes; the kernels'
// TMEM operands are read through p.q / p.uq

int run_wide(WOp op, const EngineParams& p, bool drop, int nblocks, cudaStream_t st) {
  return launch_status(launch_wide(op, drop, p, nblocks, st));
}

// maps[t] = (tensor, heads, box rows)
struct MapSpec {
  const void* base;
  int64_t heads;
  int rows;
};
bool wide_maps(EngineParams* p, const fbob_shape* s, const MapSpec* spec, int n) {
  for (int t = 0; t < n; ++t)
    if (!make_map(&p->tm[t], spec[t].base, spec[t].heads, s->N, s->d, spec[t].rows)) return false;
  return true;
}

// Pass 1 at d = 256: `parts` 1 = the row scalars alpha, E, D (eq. 6); 2 =
// dOtil and Qtil from eqs. (6)-(7) with row_stats given; 3 = the whole pass:
// alpha, E, D with dOtil in one sweep (dOtil0 = P U_V + (P o F) V needs no
// row scalar; dOtil = dOtil0 - alpha o, eq. 8), then Qtil.
int run_pass1_wide(const fbob_shape* s, const void* q, const void* k, const void* v,
                   const void* o, const float* lse, const void* dout, const void* gq,
                   const void* gk, const void* gv, void* q_bar, void* dout_bar, float* row_stats,
                   cudaStream_t st, int64_t head0, int parts) {
  const int64_t BH = s->B * s->H, BHk = s->B * kv_heads(s);
  EngineParams p = base_params(s);
  p.head0 = (int)head0;
  p.lse = lse;
  p.nblk = n_blocks(s->N, BM);
  choose_order(&p, pass1_heads_per_group(s));
  const bool drop = has_dropout(s);
  const int nb = p.nblk * p.BH;
  int rc = FBOB_OK;
  if (parts == 3) {
    // alpha, E, D and dOtil: Q in TMEM; U_Q, dO; (K, U_K) and (V, U_V) streamed as pairs
    EngineParams a = p;
    a.q = static_cast<const __nv_bfloat16*>(q);
    a.o = static_cast<const __nv_bfloat16*>(o);
    a.dout = static_cast<const __nv_bfloat16*>(dout);
    a.vec_out = row_stats;
    a.out0 = static_cast<__nv_bfloat16*>(dout_bar);
    const MapSpec ma[6] = {{gq, BH, BM}, {dout, BH, BM}, {k, BHk, HB},
                           {gk, BHk, HB}, {v, BHk, HB},  {gv, BHk, HB}};
    if (!wide_maps(&a, s, ma, 6)) return FBOB_ERR_CUDA;
    rc = run_wide(WOp::StatsDO, a, drop, nb, st);
    if (rc != FBOB_OK) return rc;
  }
  if (parts == 1) {  // alpha, E, D: Q, U_Q in TMEM; dO; K, U_K, V, U_V streamed
    EngineParams a = p;
    a.q = static_cast<const __nv_bfloat16*>(q);
    a.uq = static_cast<const __nv_bfloat16*>(gq);
    a.o = static_cast<const __nv_bfloat16*>(o);
    a.dout = static_cast<const __nv_bfloat16*>(dout);
    a.vec_out = row_stats;
    const MapSpec m[5] = {{dout, BH, BM}, {k, BHk, HB}, {gk, BHk, HB}, {v, BHk, HB}, {gv, BHk, HB}};
    if (!wide_maps(&a, s, m, 5)) return FBOB_ERR_CUDA;
    rc = run_wide(WOp::Stats, a, drop, nb, st);
    if (rc != FBOB_OK) return rc;
  }
  if (parts == 2) {
    // dOtil: Q in TMEM; U_Q; K, U_K, V, U_V streamed
    EngineParams a = p;
    a.q = static_cast<const __nv_bfloat16*>(q);
    a.vec_in = row_stats;
    a.out0 = static_cast<__nv_bfloat16*>(dout_bar);
    const MapSpec ma[5] = {{gq, BH, BM}, {k, BHk, HB}, {gk, BHk, HB}, {v, BHk, HB}, {gv, BHk, HB}};
    if (!wide_maps(&a, s, ma, 5)) return FBOB_ERR_CUDA;
    rc = run_wide(WOp::DOut, a, drop, nb, st);
    if (rc != FBOB_OK) return rc;
  }
  if (parts & 2) {
    // Qtil: Q in TMEM; U_Q, dO; K, U_K streamed; V, U_V in a ring of their own
    EngineParams b = p;
    b.q = static_cast<const __nv_bfloat16*>(q);
    b.vec_in = row_stats;
    b.out0 = static_cast<__nv_bfloat16*>(q_bar);
    const MapSpec mb[6] = {{gq, BH, BM}, {dout, BH, BM}, {k, BHk, HB},
                           {gk, BHk, HB}, {v, BHk, HB},  {gv, BHk, HB}};
    if (!wide_maps(&b, s, mb, 6)) return FBOB_ERR_CUDA;
    rc = run_wide(WOp::DQ, b, drop, nb, st);
  }
  return rc;
}

// Pass 2 at d = 256: Vtil (K in TMEM; U_K; Q, U_Q, dO streamed), then Ktil
// over two CTAs per key block (K, V in TMEM; U_K, U_V; Q, U_Q streamed; dO
// in a ring of its own).
int run_pass2_wide(const fbob_shape* s, const void* q, const void* k, const void* v,
                   const float* lse, const void* dout, const void* gq, const void* gk,
                   const void* gv, const float* row_stats, void* k_bar, void* v_bar,
                   cudaStream_t st, int64_t head0) {
  const int64_t BH = s->B * s->H, BHk = s->B * kv_heads(s);
  EngineParams p = base_params(s);
  p.head0 = (int)head0;
  p.BH = (int)BHk;  // one CTA column per key/value head
  p.lse = lse;
  p.vec_in = row_stats;
  p.nblk = n_blocks(s->N, BM);
  choose_order(&p, p.BH);
  const bool drop = has_dropout(s);
  EngineParams a = p;
  a.q = static_cast<const __nv_bfloat16*>(k);
  a.out0 = static_cast<__nv_bfloat16*>(v_bar);
  const MapSpec ma[4] = {{gk, BHk, BM}, {q, BH, HB}, {gq, BH, HB}, {dout, BH, HB}};
  if (!wide_maps(&a, s, ma, 4)) return FBOB_ERR_CUDA;
  int rc = run_wide(WOp::P2V, a, drop, p.nblk * p.BH, st);
  if (rc != FBOB_OK) return rc;
  EngineParams b = p;
  b.q = static_cast<const __nv_bfloat16*>(k);
  b.uq = static_cast<const __nv_bfloat16*>(v);
  b.out0 = static_cast<__nv_bfloat16*>(k_bar);
  const MapSpec mb[5] = {{gk, BHk, BM}, {gv, BHk, BM}, {q, BH, HB}, {gq, BH, HB}, {dout, BH, HB}};
  if (!wide_maps(&b, s, mb, 5)) return FBOB_ERR_CUDA;
  return run_wide(WOp::P2K, b, drop, 2 * p.nblk * p.BH, st);
}

// ---- the individual launches (arguments already validated)

// Tensor maps and pointers shared by the row-block BoB kernels: stationary
// Q, U_Q, dO; streamed K, U_K (64-row tiles) and V, U_V (32-row chunks,
// interleaved in the stream stage so that [V_h ; U_V_h] is one operand).
bool row_bob_params(const fbob_shape* s, const void* q, const void* k, const void* v,
                    const void* o, const float* lse, const void* dout, const void* gq,
                    const void* gk, const void* gv, EngineParams* p) {
  *p = base_params(s);
  const int64_t BH = s->B * s->H, N = s->N, d = s->d;
  const void* stat[3] = {q, gq, dout};
  const void* strm[4] = {k, gk, v, gv};
  for (int t = 0; t < 3; ++t)
    if (!make_map(&p->tm[t], stat[t], BH, N, d, BM)) return false;
  const int64_t BHk = s->B * kv_heads(s);
  // streamed tiles in 32-row chunks (two per 64-key tile)
  for (int t = 0; t < 4; ++t)
    if (!make_map(&p->tm[3 + t], strm[t], BHk, N, d, HB)) return false;
  p->q = static_cast<const __nv_bfloat16*>(q);
  p->uq = static_cast<const __nv_bfloat16*>(gq);
  p->o = static_cast<const __nv_bfloat16*>(o);
  p->dout = static_cast<const __nv_bfloat16*>(dout);
  p->lse = lse;
  p->nblk = n_blocks(s->N, BM);
  choose_order(p, pass1_heads_per_group(s));
  return true;
}

// Row scalars alpha, E, D (eq. 6) into row_stats.
int run_row_stats(EngineParams p, int d, bool drop, float* row_stats, cudaStream_t st) {
  p.vec_out = row_stats;
  return launch_status(launch_row(RowOp::BobStats, d, drop, p, p.nblk * p.BH, st));
}

// Qtil, dOtil from eqs. (6)-(7) with the row scalars given in row_stats.
int run_pass1_direct(EngineParams p, int d, bool drop, const float* row_stats, void* q_bar,
                     void* dout_bar, cudaStream_t st) {
  p.vec_in = row_stats;
  p.out0 = static_cast<__nv_bfloat16*>(q_bar);
  p.out1 = static_cast<__nv_bfloat16*>(dout_bar);
  return launch_status(launch_row(RowOp::BobPass1D, d, drop, p, p.nblk * p.BH, st));
}

// Pass 1 in one sweep with the affine fusion (Prop. 3.1, eq. 8): one kernel,
// at d = 128 two CTAs per row block (64 output columns each).  No dropout.
int run_pass1_fused(EngineParams p, int d, void* q_bar, void* dout_bar, float* row_stats,
                    cudaStream_t st) {
  p.out0 = static_cast<__nv_bfloat16*>(q_bar);
  p.out1 = static_cast<__nv_bfloat16*>(dout_bar);
  p.vec_out = row_stats;
  const int split = d == 128 ? 2 : 1;
  return launch_status(launch_row(RowOp::BobPass1, d, false, p, p.nblk * p.BH * split, st));
}

// The form fbob_attn_bob's Pass 1 takes: the one-sweep affine fusion at d <= 64
// without dropout; otherwise row statistics + direct form (with dropout the
// one-sweep fusion would need a fifth operand tile per half, the ungated P
// of B next to the gated P of dOtil0; at d = 128 the statistics + direct
// form was measured faster than the fused form over two CTAs per row block).
bool pass1_one_sweep(const fbob_shape* s) { return s->d <= 64 && !has_dropout(s); }

// head0: flat index of the shape's first query head within a larger problem
// (chunked host-buffer calls); it only enters the dropout counter.
int run_pass1(const fbob_shape* s, const void* q, const void* k, const void* v, const void* o,
              const float* lse, const void* dout, const void* gq, const void* gk,
              const void* gv, void* q_bar, void* dout_bar, float* row_stats,
              cudaStream_t st, int64_t head0 = 0) {
  if (s->d == 256)
    return run_pass1_wide(s, q, k, v, o, lse, dout, gq, gk, gv, q_bar, dout_bar, row_stats, st,
                          head0, 3);
  EngineParams p;
  if (!row_bob_params(s, q, k, v, o, lse, dout, gq, gk, gv, &p)) return FBOB_ERR_CUDA;
  p.head0 = (int)head0;
  if (pass1_one_sweep(s)) return run_pass1_fused(p, (int)s->d, q_bar, dout_bar, row_stats, st);
  // d = 128: the four accumulators of the one-sweep form do not fit TMEM next
  // to the stage-A tiles; with dropout (any d) the direct form gates its
  // operands tile by tile.  First the row scalars (alpha, E, D), then Qtil
  // and dOtil from eqs. (6)-(7) with those scalars known (two accumulators).
  const bool drop = has_dropout(s);
  const int rc = run_row_stats(p, (int)s->d, drop, row_stats, st);
  if (rc != FBOB_OK) return rc;
  return run_pass1_direct(p, (int)s->d, drop, row_stats, q_bar, dout_bar, st);
}

// kernels one pass-1 / pass-2 call enqueues
int pass1_launches(const fbob_shape* s) {
  return s->d == 256 ? 2 : pass1_one_sweep(s) ? 1 : 2;
}
int pass2_launches(const fbob_shape* s) { return s->d == 256 ? 2 : 1; }

int run_pass2(const fbob_shape* s, const void* q, const void* k, const void* v, const float* lse,
              const void* dout, const void* gq, const void* gk, const void* gv,
              const float* row_stats, void* k_bar, void* v_bar, cudaStream_t st,
              int64_t head0 = 0) {
  if (s->d == 256)
    return run_pass2_wide(s, q, k, v, lse, dout, gq, gk, gv, row_stats, k_bar, v_bar, st, head0);
  EngineParams p = base_params(s);
  p.head0 = (int)head0;
  const int64_t BH = s->B * s->H, N = s->N, d = s->d;
  const void* stat[4] = {k, v, gk, gv};
  const void* strm[3] = {q, gq, dout};
  const int64_t BHk = s->B * kv_heads(s);
  p.BH = (int)BHk;  // one CTA column per key/value head
  for (int t = 0; t < 4; ++t)
    if (!make_map(&p.tm[t], stat[t], BHk, N, d, BM)) return FBOB_ERR_CUDA;
  for (int t = 0; t < 3; ++t)
    if (!make_map(&p.tm[4 + t], strm[t], BH, N, d, BN)) return FBOB_ERR_CUDA;
  p.lse = lse;
  p.vec_in = row_stats;
  p.out0 = static_cast<__nv_bfloat16*>(k_bar);
  p.out1 = static_cast<__nv_bfloat16*>(v_bar);
  p.nblk = n_blocks(s->N, BM);
  choose_order(&p, p.BH);
  return launch_status(launch_col(ColOp::BobPass2, (int)d, has_dropout(s), p, p.nblk * p.BH, st));
}

// ---- host-buffer BoB: chunks of query heads pipelined through a device
// workspace of kSlots slots (copy in, compute, copy out on three streams)
constexpr int kSlots = 2;
constexpr int kBufs = 14;  // q k v o lse dout gq gk gv q_bar k_bar v_bar dout_bar row_stats

int64_t align256(int64_t x) { return (x + 255) & ~int64_t(255); }

// query heads per key/value head
int64_t group(const fbob_shape* s) { return s->H / kv_heads(s); }

// Byte offsets of the buffers of one slot holding `nq` query heads; returns
// the slot's size.
int64_t slot_layout(const fbob_shape* s, int64_t nq, int64_t* off) {
  const int64_t nkv = nq / group(s), nd = s->N * s->d * 2;
  const int64_t bytes[kBufs] = {nq * nd,  nkv * nd, nkv * nd, nq * nd,  nq * s->N * 4,
                                nq * nd,  nq * nd,  nkv * nd, nkv * nd, nq * nd,
                                nkv * nd, nkv * nd, nq * nd,  3 * nq * s->N * 4};
  int64_t at = 0;
  for (int t = 0; t < kBufs; ++t) {
    off[t] = at;
    at += align256(bytes[t]);
  }
  return at;
}

// Query heads per chunk: whole key/value groups, about a quarter of the
// problem (so copies overlap compute), at most what the workspace holds.
int64_t chunk_heads(const fbob_shape* s, int64_t ws_bytes) {
  const int64_t G = group(s), units = s->B * s->H / G, cap = ws_bytes / kSlots;
  int64_t off[kBufs];
  // unpadded bytes of one group bound the fit from above; then step down to
  // the largest chunk whose padded slot fits (a few steps: padding < 14 * 256)
  const int64_t raw = slot_layout(s, G, off) - kBufs * 255;
  int64_t u = (units + 3) / 4;
  if (raw > 0 && cap / raw < u) u = cap / raw;
  while (u > 0 && slot_layout(s, u * G, off) > cap) --u;
  return u * G;
}

// Device address of the static staging array on the current device, looked
// up on every call: an address cached across calls could outlive the context
// it belongs to (a cudaDeviceReset tears the module down and the next context
// places the array again, possibly elsewhere).  The lookup allocates nothing.
cudaError_t noalloc_scratch(uint8_t** ptr) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return e;
  *ptr = static_cast<uint8_t*>(p);
  return cudaSuccess;
}

// Validation shared by the host-buffer calls: shape, host pointers present,
// host outputs overlapping nothing.
int check_host_args(const fbob_shape* s, const void* const* hin, void* const* hout, bool* empty) {
  int rc = check_shape(s, empty);
  if (rc != FBOB_OK) return rc;
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  const int64_t inb[9] = {mat, matk, matk, mat, vec, mat, mat, matk, matk};
  const int64_t outb[5] = {mat, matk, matk, mat, 3 * vec};
  for (int t = 0; t < 9; ++t)
    if (!hin[t]) return FBOB_ERR_INVALID_ARGUMENT;
  for (int a = 0; a < 5; ++a) {
    if (!hout[a]) return FBOB_ERR_INVALID_ARGUMENT;
    const Span sa = {reinterpret_cast<uintptr_t>(hout[a]),
                     reinterpret_cast<uintptr_t>(hout[a]) + (uintptr_t)outb[a]};
    for (int b = 0; b < 14; ++b) {
      if (b == 9 + a) continue;
      const void* pb = b < 9 ? hin[b] : hout[b - 9];
      const int64_t nb = b < 9 ? inb[b] : outb[b - 9];
      const Span sb = {reinterpret_cast<uintptr_t>(pb),
                       reinterpret_cast<uintptr_t>(pb) + (uintptr_t)nb};
      if (overlaps(sa, sb)) return FBOB_ERR_INVALID_ARGUMENT;
    }
  }
  return FBOB_OK;
}

// Chunk boundaries (in query heads, whole key/value groups) for chunks of at
// most hc heads.  Only the first chunk's copy in and the last chunk's copy
// out cannot overlap any kernel, so when there are more than two full chunks
// those two are made about a quarter as large; the rest share the remainder
// evenly.  Returns the number of chunks; starts[] gets nchunks + 1 entries.
int64_t plan_chunks(int64_t BH, int64_t G, int64_t hc, int64_t* starts, int64_t max_chunks) {
  const int64_t U = BH / G, b = hc / G;  // groups in all, per full chunk
  int64_t n = 0;
  starts[n] = 0;
  if (U <= 2 * b || max_chunks < 4) {
    for (int64_t u = 0; u < U && n + 1 < max_chunks;) {
      u += (U - u) < b ? (U - u) : b;
      starts[++n] = u * G;
    }
    return n;
  }
  const int64_t e = (b + 3) / 4;          // end chunks
  const int64_t mid = U - 2 * e;          // groups for the middle chunks
  int64_t m = (mid + b - 1) / b;          // middle chunks
  if (m + 2 > max_chunks) m = max_chunks - 2;
  int64_t u = e;
  starts[++n] = u * G;
  for (int64_t c = 0; c < m; ++c) {
    u += mid / m + (c < mid % m ? 1 : 0);
    starts[++n] = u * G;
  }
  u += e;
  starts[++n] = u * G;
  return n;
}

struct HostCall {
  cudaStream_t cin = nullptr, cout = nullptr, cmp = nullptr;
  cudaEvent_t entry = nullptr, in[kSlots] = {}, comp[kSlots] = {}, out[kSlots] = {};
  ~HostCall() {  // released once their pending work completes
    if (entry) cudaEventDestroy(entry);
    for (int t = 0; t < kSlots; ++t) {
      if (in[t]) cudaEventDestroy(in[t]);
      if (comp[t]) cudaEventDestroy(comp[t]);
      if (out[t]) cudaEventDestroy(out[t]);
    }
    if (cin) cudaStreamDestroy(cin);
    if (cout) cudaStreamDestroy(cout);
    if (cmp) cudaStreamDestroy(cmp);
  }
  cudaError_t init() {
    cudaError_t e = cudaStreamCreateWithFlags(&cin, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&cout, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaStreamCreateWithFlags(&cmp, cudaStreamNonBlocking);
    if (e == cudaSuccess) e = cudaEventCreateWithFlags(&entry, cudaEventDisableTiming);
    for (int t = 0; t < kSlots && e == cudaSuccess; ++t) {
      e = cudaEventCreateWithFlags(&in[t], cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&comp[t], cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&out[t], cudaEventDisableTiming);
    }
    return e;
  }
};

}  // namespace
}  // namespace fbob

using namespace fbob;

extern "C" {

const char* fbob_status_string(int status) {
  switch (status) {
    case FBOB_OK: return "FBOB_OK";
    case FBOB_ERR_INVALID_ARGUMENT: return "FBOB_ERR_INVALID_ARGUMENT";
    case FBOB_ERR_UNSUPPORTED: return "FBOB_ERR_UNSUPPORTED";
    case FBOB_ERR_CUDA: return "FBOB_ERR_CUDA";
    case FBOB_ERR_DEVICE_TIMEOUT: return "FBOB_ERR_DEVICE_TIMEOUT";
    case FBOB_ERR_DEVICE_FAULT: return "FBOB_ERR_DEVICE_FAULT";
    case FBOB_ERR_SCRATCH_LIMIT: return "FBOB_ERR_SCRATCH_LIMIT";
    default: return "FBOB_UNKNOWN_STATUS";
  }
}

int fbob_launch_count(const char* entry) {
  if (!entry) return -1;
  static const char* names[kNumEntries] = {
      "fwd",       "bwd",       "bob",           "bob_pass1",          "bob_pass2",
      "bob_row_stats", "bob_pass1_direct", "bob_host", "bob_host_noalloc", "bob_pass1_fused"};
  for (int t = 0; t < kNumEntries; ++t)
    if (std::strcmp(entry, names[t]) == 0) return g_launches[t].load();
  return -1;
}

int fbob_attn_fwd(const fbob_shape* s, const void* q, const void* k, const void* v, void* o,
                  float* lse, struct CUstream_st* stream) {
  bool empty = false;
  int rc = check_shape(s, &empty);
  if (rc != FBOB_OK) return rc;
  if (empty) {
    g_launches[kEntFwd] = 0;
    return FBOB_OK;
  }
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  const void* in[3] = {q, k, v};
  const int64_t inb[3] = {mat, matk, matk};
  void* out[2] = {o, lse};
  const int64_t outb[2] = {mat, vec};
  rc = check_ptrs(in, inb, 3, out, outb, 2);
  if (rc != FBOB_OK) return rc;
  if (s->d == 256) {
    // one sweep with an online softmax (wide_engine.cuh)
    const int64_t BHk = s->B * kv_heads(s);
    EngineParams p = base_params(s);
    p.q = static_cast<const __nv_bfloat16*>(q);
    p.nblk = n_blocks(s->N, BM);
    p.vec_out = lse;
    p.out0 = static_cast<__nv_bfloat16*>(o);
    choose_order(&p, p.BH);
    const MapSpec m[2] = {{k, BHk, HB}, {v, BHk, HB}};
    if (!wide_maps(&p, s, m, 2)) return FBOB_ERR_CUDA;
    rc = run_wide(WOp::Fwd, p, has_dropout(s), p.nblk * p.BH, stream);
    if (rc == FBOB_OK) g_launches[kEntFwd] = 1;
    return rc;
  }
  EngineParams p = base_params(s);
  const int64_t BH = s->B * s->H, BHk = s->B * kv_heads(s);
  if (!make_map(&p.tm[0], q, BH, s->N, s->d, BM) ||
      !make_map(&p.tm[1], k, BHk, s->N, s->d, BN) || !make_map(&p.tm[2], v, BHk, s->N, s->d, BN))
    return FBOB_ERR_CUDA;
  p.out0 = static_cast<__nv_bfloat16*>(o);
  p.vec_out = lse;
  p.nblk = n_blocks(s->N, 2 * BM);  // two 128-row query tiles per CTA
  choose_order(&p, p.BH);
  rc = launch_status(launch_row(RowOp::Fwd, (int)s->d, has_dropout(s), p, p.nblk * p.BH, stream));
  if (rc == FBOB_OK) g_launches[kEntFwd] = 1;
  return rc;
}

int fbob_attn_bwd(const fbob_shape* s, const void* q, const void* k, const void* v, const void* o,
                  const float* lse, const void* dout, void* dq, void* dk, void* dv, float* dstat,
                  struct CUstream_st* stream) {
  bool empty = false;
  int rc = check_shape(s, &empty);
  if (rc != FBOB_OK) return rc;
  if (empty) {
    g_launches[kEntBwd] = 0;
    return FBOB_OK;
  }
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  const void* in[6] = {q, k, v, o, lse, dout};
  const int64_t inb[6] = {mat, matk, matk, mat, vec, mat};
  void* out[4] = {dq, dk, dv, dstat};
  const int64_t outb[4] = {mat, matk, matk, vec};
  rc = check_ptrs(in, inb, 6, out, outb, 4);
  if (rc != FBOB_OK) return rc;
  if (s->d == 256) {
    // dQ and D (row blocks), then dV and dK (key blocks, one kernel each)
    const int64_t BH = s->B * s->H, BHk = s->B * kv_heads(s);
    const bool drop = has_dropout(s);
    EngineParams p = base_params(s);
    p.q = static_cast<const __nv_bfloat16*>(q);
    p.o = static_cast<const __nv_bfloat16*>(o);
    p.dout = static_cast<const __nv_bfloat16*>(dout);
    p.lse = lse;
    p.out0 = static_cast<__nv_bfloat16*>(dq);
    p.vec_out = dstat;
    p.nblk = n_blocks(s->N, BM);
    choose_order(&p, p.BH);
    const MapSpec mq[3] = {{dout, BH, BM}, {k, BHk, HB}, {v, BHk, HB}};
    if (!wide_maps(&p, s, mq, 3)) return FBOB_ERR_CUDA;
    rc = run_wide(WOp::BwdDQ, p, drop, p.nblk * p.BH, stream);
    if (rc != FBOB_OK) return rc;
    EngineParams c = base_params(s);
    c.BH = (int)BHk;  // one CTA column per key/value head
    c.q = static_cast<const __nv_bfloat16*>(k);
    c.lse = lse;
    c.vec_in = dstat;
    c.nblk = n_blocks(s->N, BM);
    choose_order(&c, c.BH);
    EngineParams cv = c;
    cv.out0 = static_cast<__nv_bfloat16*>(dv);
    const MapSpec mv[2] = {{q, BH, HB}, {dout, BH, HB}};
    if (!wide_maps(&cv, s, mv, 2)) return FBOB_ERR_CUDA;
    rc = run_wide(WOp::BwdDV, cv, drop, c.nblk * c.BH, stream);
    if (rc != FBOB_OK) return rc;
    EngineParams ck = c;
    ck.out0 = static_cast<__nv_bfloat16*>(dk);
    const MapSpec mk[3] = {{v, BHk, BM}, {q, BH, HB}, {dout, BH, HB}};
    if (!wide_maps(&ck, s, mk, 3)) return FBOB_ERR_CUDA;
    rc = run_wide(WOp::BwdDK, ck, drop, c.nblk * c.BH, stream);
    if (rc == FBOB_OK) g_launches[kEntBwd] = 3;
    return rc;
  }
  const int64_t BH = s->B * s->H, BHk = s->B * kv_heads(s), N = s->N, d = s->d;
  // dQ and D: row-block pass (writes D, which the column pass reads)
  EngineParams p = base_params(s);
  if (!make_map(&p.tm[0], q, BH, N, d, BM) || !make_map(&p.tm[1], dout, BH, N, d, BM) ||
      !make_map(&p.tm[2], k, BHk, N, d, BN) || !make_map(&p.tm[3], v, BHk, N, d, BN))
    return FBOB_ERR_CUDA;
  p.o = static_cast<const __nv_bfloat16*>(o);
  p.dout = static_cast<const __nv_bfloat16*>(dout);
  p.lse = lse;
  p.out0 = static_cast<__nv_bfloat16*>(dq);
  p.vec_out = dstat;
  p.nblk = n_blocks(s->N, BM);
  choose_order(&p, p.BH);
  rc = launch_status(launch_row(RowOp::BwdDQ, (int)d, has_dropout(s), p, p.nblk * p.BH, stream));
  if (rc != FBOB_OK) return rc;
  // dK and dV: column-block pass
  EngineParams c = base_params(s);
  c.BH = (int)BHk;  // one CTA column per key/value head
  if (!make_map(&c.tm[0], k, BHk, N, d, BM) || !make_map(&c.tm[1], v, BHk, N, d, BM) ||
      !make_map(&c.tm[2], q, BH, N, d, BN) || !make_map(&c.tm[3], dout, BH, N, d, BN))
    return FBOB_ERR_CUDA;
  c.lse = lse;
  c.vec_in = dstat;
  c.out0 = static_cast<__nv_bfloat16*>(dk);
  c.out1 = static_cast<__nv_bfloat16*>(dv);
  c.nblk = n_blocks(s->N, BM);
  choose_order(&c, c.BH);
  rc = launch_status(launch_col(ColOp::BwdDKDV, (int)d, has_dropout(s), c, c.nblk * c.BH, stream));
  if (rc == FBOB_OK) g_launches[kEntBwd] = 2;
  return rc;
}

int fbob_attn_bob_pass1(const fbob_shape* s, const void* q, const void* k, const void* v,
                        const void* o, const float* lse, const void* dout, const void* gq,
                        const void* gk, const void* gv, void* q_bar, void* dout_bar,
                        float* row_stats, struct CUstream_st* stream) {
  bool empty = false;
  int rc = check_shape(s, &empty);
  if (rc != FBOB_OK) return rc;
  if (empty) {
    g_launches[kEntPass1] = 0;
    return FBOB_OK;
  }
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  const void* in[9] = {q, k, v, o, lse, dout, gq, gk, gv};
  const int64_t inb[9] = {mat, matk, matk, mat, vec, mat, mat, matk, matk};
  void* out[3] = {q_bar, dout_bar, row_stats};
  const int64_t outb[3] = {mat, mat, 3 * vec};
  rc = check_ptrs(in, inb, 9, out, outb, 3);
  if (rc != FBOB_OK) return rc;
  rc = run_pass1(s, q, k, v, o, lse, dout, gq, gk, gv, q_bar, dout_bar, row_stats, stream);
  if (rc == FBOB_OK) g_launches[kEntPass1] = pass1_launches(s);
  return rc;
}

int fbob_attn_bob_pass1_fused(const fbob_shape* s, const void* q, const void* k, const void* v,
                              const void* o, const float* lse, const void* dout, const void* gq,
                              const void* gk, const void* gv, void* q_bar, void* dout_bar,
                              float* row_stats, struct CUstream_st* stream) {
  bool empty = false;
  int rc = check_shape(s, &empty);
  if (rc != FBOB_OK) return rc;
  // with dropout, or at d = 256 (four 256-column accumulators), the one-sweep
  // form does not fit
  if (has_dropout(s) || s->d == 256) return FBOB_ERR_UNSUPPORTED;
  if (empty) {
    g_launches[kEntPass1Fused] = 0;
    return FBOB_OK;
  }
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  const void* in[9] = {q, k, v, o, lse, dout, gq, gk, gv};
  const int64_t inb[9] = {mat, matk, matk, mat, vec, mat, mat, matk, matk};
  void* out[3] = {q_bar, dout_bar, row_stats};
  const int64_t outb[3] = {mat, mat, 3 * vec};
  rc = check_ptrs(in, inb, 9, out, outb, 3);
  if (rc != FBOB_OK) return rc;
  EngineParams p;
  if (!row_bob_params(s, q, k, v, o, lse, dout, gq, gk, gv, &p)) return FBOB_ERR_CUDA;
  rc = run_pass1_fused(p, (int)s->d, q_bar, dout_bar, row_stats, stream);
  if (rc == FBOB_OK) g_launches[kEntPass1Fused] = 1;
  return rc;
}

int fbob_attn_bob_pass2(const fbob_shape* s, const void* q, const void* k, const void* v,
                        const float* lse, const void* dout, const void* gq, const void* gk,
                        const void* gv, const float* row_stats, void* k_bar, void* v_bar,
                        struct CUstream_st* stream) {
  bool empty = false;
  int rc = check_shape(s, &empty);
  if (rc != FBOB_OK) return rc;
  if (empty) {
    g_launches[kEntPass2] = 0;
    return FBOB_OK;
  }
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  // row_stats is an input of pass 2; check it with the inputs
  const void* in2[9] = {q, k, v, lse, dout, gq, gk, gv, row_stats};
  const int64_t inb2[9] = {mat, matk, matk, vec, mat, mat, matk, matk, 3 * vec};
  void* out[2] = {k_bar, v_bar};
  const int64_t outb[2] = {matk, matk};
  rc = check_ptrs(in2, inb2, 9, out, outb, 2);
  if (rc != FBOB_OK) return rc;
  rc = run_pass2(s, q, k, v, lse, dout, gq, gk, gv, row_stats, k_bar, v_bar, stream);
  if (rc == FBOB_OK) g_launches[kEntPass2] = pass2_launches(s);
  return rc;
}

int fbob_attn_bob_row_stats(const fbob_shape* s, const void* q, const void* k, const void* v,
                            const void* o, const float* lse, const void* dout, const void* gq,
                            const void* gk, const void* gv, float* row_stats,
                            struct CUstream_st* stream) {
  bool empty = false;
  int rc = check_shape(s, &empty);
  if (rc != FBOB_OK) return rc;
  if (empty) {
    g_launches[kEntRowStats] = 0;
    return FBOB_OK;
  }
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  const void* in[9] = {q, k, v, o, lse, dout, gq, gk, gv};
  const int64_t inb[9] = {mat, matk, matk, mat, vec, mat, mat, matk, matk};
  void* out[1] = {row_stats};
  const int64_t outb[1] = {3 * vec};
  rc = check_ptrs(in, inb, 9, out, outb, 1);
  if (rc != FBOB_OK) return rc;
  if (s->d == 256) {
    rc = run_pass1_wide(s, q, k, v, o, lse, dout, gq, gk, gv, nullptr, nullptr, row_stats, stream,
                        0, 1);
    if (rc == FBOB_OK) g_launches[kEntRowStats] = 1;
    return rc;
  }
  EngineParams p;
  if (!row_bob_params(s, q, k, v, o, lse, dout, gq, gk, gv, &p)) return FBOB_ERR_CUDA;
  rc = run_row_stats(p, (int)s->d, has_dropout(s), row_stats, stream);
  if (rc == FBOB_OK) g_launches[kEntRowStats] = 1;
  return rc;
}

int fbob_attn_bob_pass1_direct(const fbob_shape* s, const void* q, const void* k, const void* v,
                               const float* lse, const void* dout, const void* gq,
                               const void* gk, const void* gv, const float* row_stats,
                               void* q_bar, void* dout_bar, struct CUstream_st* stream) {
  bool empty = false;
  int rc = check_shape(s, &empty);
  if (rc != FBOB_OK) return rc;
  if (empty) {
    g_launches[kEntPass1D] = 0;
    return FBOB_OK;
  }
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  const void* in[9] = {q, k, v, lse, dout, gq, gk, gv, row_stats};
  const int64_t inb[9] = {mat, matk, matk, vec, mat, mat, matk, matk, 3 * vec};
  void* out[2] = {q_bar, dout_bar};
  const int64_t outb[2] = {mat, mat};
  rc = check_ptrs(in, inb, 9, out, outb, 2);
  if (rc != FBOB_OK) return rc;
  if (s->d == 256) {
    rc = run_pass1_wide(s, q, k, v, nullptr, lse, dout, gq, gk, gv, q_bar, dout_bar,
                        const_cast<float*>(row_stats), stream, 0, 2);
    if (rc == FBOB_OK) g_launches[kEntPass1D] = 2;
    return rc;
  }
  EngineParams p;
  // (o is not read: D comes from row_stats)
  if (!row_bob_params(s, q, k, v, nullptr, lse, dout, gq, gk, gv, &p)) return FBOB_ERR_CUDA;
  rc = run_pass1_direct(p, (int)s->d, has_dropout(s), row_stats, q_bar, dout_bar, stream);
  if (rc == FBOB_OK) g_launches[kEntPass1D] = 1;
  return rc;
}

int fbob_attn_bob(const fbob_shape* s, const void* q, const void* k, const void* v, const void* o,
                  const float* lse, const void* dout, const void* gq, const void* gk,
                  const void* gv, void* q_bar, void* k_bar, void* v_bar, void* dout_bar,
                  float* row_stats, struct CUstream_st* stream) {
  bool empty = false;
  int rc = check_shape(s, &empty);
  if (rc != FBOB_OK) return rc;
  if (empty) {
    g_launches[kEntBob] = 0;
    return FBOB_OK;
  }
  const int64_t mat = s->B * s->H * s->N * s->d * 2, vec = s->B * s->H * s->N * 4;
  const int64_t matk = s->B * kv_heads(s) * s->N * s->d * 2;
  const void* in[9] = {q, k, v, o, lse, dout, gq, gk, gv};
  const int64_t inb[9] = {mat, matk, matk, mat, vec, mat, mat, matk, matk};
  void* out[5] = {q_bar, k_bar, v_bar, dout_bar, row_stats};
  const int64_t outb[5] = {mat, matk, matk, mat, 3 * vec};
  rc = check_ptrs(in, inb, 9, out, outb, 5);
  if (rc != FBOB_OK) return rc;
  // Pass 1 (row blocks): Qtil, dOtil and the row scalars alpha, E, D.
  rc = run_pass1(s, q, k, v, o, lse, dout, gq, gk, gv, q_bar, dout_bar, row_stats, stream);
  if (rc != FBOB_OK) return rc;
  // Pass 2 (column blocks): Ktil, Vtil from the saved row state.  Stream
  // order is the only synchronisation between the passes.
  rc = run_pass2(s, q, k, v, lse, dout, gq, gk, gv, row_stats, k_bar, v_bar, stream);
  if (rc == FBOB_OK) g_launches[kEntBob] = pass1_launches(s) + pass2_launches(s);
  return rc;
}

int64_t fbob_attn_bob_host_workspace(const fbob_shape* s, int64_t chunk_heads) {
  bool empty = false;
  if (check_shape(s, &empty) != FBOB_OK || chunk_heads < 1) return -1;
  const int64_t G = group(s);
  const int64_t nq = (chunk_heads + G - 1) / G * G;
  int64_t off[kBufs];
  return kSlots * slot_layout(s, nq, off);
}

int fbob_attn_bob_host(const fbob_shape* s, const void* q, const void* k, const void* v,
                       const void* o, const float* lse, const void* dout, const void* gq,
                       const void* gk, const void* gv, void* q_bar, void* k_bar, void* v_bar,
                       void* dout_bar, float* row_stats, void* workspace,
                       int64_t workspace_bytes, struct CUstream_st* stream) {
  bool empty = false;
  const void* hin[9] = {q, k, v, o, lse, dout, gq, gk, gv};
  void* hout[5] = {q_bar, k_bar, v_bar, dout_bar, row_stats};
  int rc = check_host_args(s, hin, hout, &empty);
  if (rc != FBOB_OK) return rc;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) || workspace_bytes < 0)
    return FBOB_ERR_INVALID_ARGUMENT;
  if (empty) {
    g_launches[kEntBobHost] = 0;
    return FBOB_OK;
  }
  const int64_t BH = s->B * s->H, G = group(s), N = s->N, nd = N * s->d * 2;
  const int64_t hc = chunk_heads(s, workspace_bytes);
  if (hc < 1) return FBOB_ERR_INVALID_ARGUMENT;  // the workspace holds no key/value group
  int64_t off[kBufs];
  const int64_t slot = slot_layout(s, hc, off);
  HostCall hcall;
  if (hcall.init() != cudaSuccess) return FBOB_ERR_CUDA;
  cudaStream_t st = stream;
  // the copy streams start after the work already on `stream` (it may use
  // the workspace or the host buffers)
  if (cudaEventRecord(hcall.entry, st) != cudaSuccess ||
      cudaStreamWaitEvent(hcall.cin, hcall.entry, 0) != cudaSuccess ||
      cudaStreamWaitEvent(hcall.cout, hcall.entry, 0) != cudaSuccess ||
      cudaStreamWaitEvent(hcall.cmp, hcall.entry, 0) != cudaSuccess)
    return FBOB_ERR_CUDA;
  // at most 64 chunks: above that, full chunks of hc heads end to end
  int64_t starts[65];
  const int64_t nfull = (BH + hc - 1) / hc;
  int64_t nchunks = 0;
  if (nfull + 2 <= 64) {
    nchunks = plan_chunks(BH, G, hc, starts, 64);
  }
  auto h2d = [&](void* dst, const void* src, int64_t bytes) {
    return cudaMemcpyAsync(dst, src, (size_t)bytes, cudaMemcpyHostToDevice, hcall.cin);
  };
  auto d2h = [&](void* dst, const void* src, int64_t bytes) {
    return cudaMemcpyAsync(dst, src, (size_t)bytes, cudaMemcpyDeviceToHost, hcall.cout);
  };
  auto hb = [](const void* p, int64_t at) { return static_cast<const uint8_t*>(p) + at; };
  auto hbm = [](void* p, int64_t at) { return static_cast<uint8_t*>(p) + at; };
  int launches = 0;
  const int64_t nloop = nchunks ? nchunks : nfull;
  for (int64_t c = 0; c < nloop; ++c) {
    const int sl = (int)(c % kSlots);
    uint8_t* base = static_cast<uint8_t*>(workspace) + sl * slot;
    void* w[kBufs];
    for (int t = 0; t < kBufs; ++t) w[t] = base + off[t];
    const int64_t f0 = nchunks ? starts[c] : c * hc;
    const int64_t f1 = nchunks ? starts[c + 1] : ((f0 + hc) < BH ? (f0 + hc) : BH);
    const int64_t nq = f1 - f0, nkv = nq / G, k0 = f0 / G;
    // the slots' chunks alternate between two compute streams, so the next
    // chunk's kernels fill the SMs the previous chunk's last wave leaves idle
    cudaStream_t cs = sl ? hcall.cmp : st;
    cudaError_t e = cudaSuccess;
    // copy in once the slot's previous chunk has been computed
    if (c >= kSlots) e = cudaStreamWaitEvent(hcall.cin, hcall.comp[sl], 0);
    const int qside[5] = {0, 3, 5, 6};  // q, o, dout, gq
    for (int t = 0; t < 4 && e == cudaSuccess; ++t)
      e = h2d(w[qside[t]], hb(hin[qside[t]], f0 * nd), nq * nd);
    const int kside[4] = {1, 2, 7, 8};  // k, v, gk, gv
    for (int t = 0; t < 4 && e == cudaSuccess; ++t)
      e = h2d(w[kside[t]], hb(hin[kside[t]], k0 * nd), nkv * nd);
    if (e == cudaSuccess) e = h2d(w[4], hb(lse, f0 * N * 4), nq * N * 4);
    if (e == cudaSuccess) e = cudaEventRecord(hcall.in[sl], hcall.cin);
    // compute once the inputs are in and the slot's previous outputs are out
    if (e == cudaSuccess) e = cudaStreamWaitEvent(cs, hcall.in[sl], 0);
    if (e == cudaSuccess && c >= kSlots) e = cudaStreamWaitEvent(cs, hcall.out[sl], 0);
    if (e != cudaSuccess) return FBOB_ERR_CUDA;
    fbob_shape csh = *s;
    csh.B = 1;
    csh.H = nq;
    csh.H_kv = s->H_kv > 0 ? nkv : 0;
    rc = run_pass1(&csh, w[0], w[1], w[2], w[3], static_cast<const float*>(w[4]), w[5], w[6],
                   w[7], w[8], w[9], w[12], static_cast<float*>(w[13]), cs, f0);
    if (rc == FBOB_OK)
      rc = run_pass2(&csh, w[0], w[1], w[2], static_cast<const float*>(w[4]), w[5], w[6], w[7],
                     w[8], static_cast<const float*>(w[13]), w[10], w[11], cs, f0);
    if (rc != FBOB_OK) return rc;
    launches += pass1_launches(&csh) + pass2_launches(&csh);
    // copy out once computed
    e = cudaEventRecord(hcall.comp[sl], cs);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(hcall.cout, hcall.comp[sl], 0);
    if (e == cudaSuccess) e = d2h(hbm(q_bar, f0 * nd), w[9], nq * nd);
    if (e == cudaSuccess) e = d2h(hbm(dout_bar, f0 * nd), w[12], nq * nd);
    if (e == cudaSuccess) e = d2h(hbm(k_bar, k0 * nd), w[10], nkv * nd);
    if (e == cudaSuccess) e = d2h(hbm(v_bar, k0 * nd), w[11], nkv * nd);
    if (e == cudaSuccess)  // row_stats planes: [3][B*H][N] on the host, [3][nq][N] in the slot
      e = cudaMemcpy2DAsync(hbm(row_stats, f0 * N * 4), (size_t)(BH * N * 4), w[13],
                            (size_t)(nq * N * 4), (size_t)(nq * N * 4), 3, cudaMemcpyDeviceToHost,
                            hcall.cout);
    if (e == cudaSuccess) e = cudaEventRecord(hcall.out[sl], hcall.cout);
    if (e != cudaSuccess) return FBOB_ERR_CUDA;
  }
  // `stream` completes after the last copies out
  for (int sl = 0; sl < kSlots && sl < nloop; ++sl)
    if (cudaStreamWaitEvent(st, hcall.out[sl], 0) != cudaSuccess) return FBOB_ERR_CUDA;
  g_launches[kEntBobHost] = launches;
  return FBOB_OK;
}

int fbob_attn_bob_host_noalloc(const fbob_shape* s, const void* q, const void* k,
                               const void* v, const void* o, const float* lse, const void* dout,
                               const void* gq, const void* gk, const void* gv, void* q_bar,
                               void* k_bar, void* v_bar, void* dout_bar, float* row_stats,
                               struct CUstream_st* stream) {
  bool empty = false;
  const void* hin[9] = {q, k, v, o, lse, dout, gq, gk, gv};
  void* hout[5] = {q_bar, k_bar, v_bar, dout_bar, row_stats};
  int rc = check_host_args(s, hin, hout, &empty);
  if (rc != FBOB_OK) return rc;
  if (empty) {
    g_launches[kEntBobHostNoAlloc] = 0;
    return FBOB_OK;
  }
  // as many whole key/value groups per chunk as one slot of the array holds
  const int64_t BH = s->B * s->H, G = group(s), N = s->N, nd = N * s->d * 2;
  int64_t off[kBufs];
  int64_t u = s->B * s->H / G;
  const int64_t raw = slot_layout(s, G, off) - kBufs * 255;
  if (raw > 0 && kNoAllocBytes / raw < u) u = kNoAllocBytes / raw;
  while (u > 0 && slot_layout(s, u * G, off) > kNoAllocBytes) --u;
  if (u < 1) return FBOB_ERR_SCRATCH_LIMIT;  // one group's staging exceeds the array
  const int64_t hc = u * G;
  slot_layout(s, hc, off);
  uint8_t* base = nullptr;
  if (noalloc_scratch(&base) != cudaSuccess) return FBOB_ERR_CUDA;
  void* w[kBufs];
  for (int t = 0; t < kBufs; ++t) w[t] = base + off[t];
  cudaStream_t st = stream;
  auto h2d = [&](void* dst, const void* src, int64_t bytes) {
    return cudaMemcpyAsync(dst, src, (size_t)bytes, cudaMemcpyHostToDevice, st);
  };
  auto d2h = [&](void* dst, const void* src, int64_t bytes) {
    return cudaMemcpyAsync(dst, src, (size_t)bytes, cudaMemcpyDeviceToHost, st);
  };
  auto hb = [](const void* p, int64_t at) { return static_cast<const uint8_t*>(p) + at; };
  auto hbm = [](void* p, int64_t at) { return static_cast<uint8_t*>(p) + at; };
  int launches = 0;
  // one chunk after the other, all on `stream`: copy in, compute, copy out
  for (int64_t f0 = 0; f0 < BH; f0 += hc) {
    const int64_t nq = (BH - f0) < hc ? (BH - f0) : hc, nkv = nq / G, k0 = f0 / G;
    cudaError_t e = cudaSuccess;
    const int qside[4] = {0, 3, 5, 6};  // q, o, dout, gq
    for (int t = 0; t < 4 && e == cudaSuccess; ++t)
      e = h2d(w[qside[t]], hb(hin[qside[t]], f0 * nd), nq * nd);
    const int kside[4] = {1, 2, 7, 8};  // k, v, gk, gv
    for (int t = 0; t < 4 && e == cudaSuccess; ++t)
      e = h2d(w[kside[t]], hb(hin[kside[t]], k0 * nd), nkv * nd);
    if (e == cudaSuccess) e = h2d(w[4], hb(lse, f0 * N * 4), nq * N * 4);
    if (e != cudaSuccess) return FBOB_ERR_CUDA;
    fbob_shape cs = *s;
    cs.B = 1;
    cs.H = nq;
    cs.H_kv = s->H_kv > 0 ? nkv : 0;
    rc = run_pass1(&cs, w[0], w[1], w[2], w[3], static_cast<const float*>(w[4]), w[5], w[6],
                   w[7], w[8], w[9], w[12], static_cast<float*>(w[13]), st, f0);
    if (rc == FBOB_OK)
      rc = run_pass2(&cs, w[0], w[1], w[2], static_cast<const float*>(w[4]), w[5], w[6], w[7],
                     w[8], static_cast<const float*>(w[13]), w[10], w[11], st, f0);
    if (rc != FBOB_OK) return rc;
    launches += pass1_launches(&cs) + pass2_launches(&cs);
    e = d2h(hbm(q_bar, f0 * nd), w[9], nq * nd);
    if (e == cudaSuccess) e = d2h(hbm(dout_bar, f0 * nd), w[12], nq * nd);
    if (e == cudaSuccess) e = d2h(hbm(k_bar, k0 * nd), w[10], nkv * nd);
    if (e == cudaSuccess) e = d2h(hbm(v_bar, k0 * nd), w[11], nkv * nd);
    if (e == cudaSuccess)
      e = cudaMemcpy2DAsync(hbm(row_stats, f0 * N * 4), (size_t)(BH * N * 4), w[13],
                            (size_t)(nq * N * 4), (size_t)(nq * N * 4), 3, cudaMemcpyDeviceToHost,
                            st);
    if (e != cudaSuccess) return FBOB_ERR_CUDA;
  }
  g_launches[kEntBobHostNoAlloc] = launches;
  return FBOB_OK;
}

int fbob_device_status(struct CUstream_st* stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return FBOB_ERR_DEVICE_FAULT;
  uint32_t w1 = 0, w2 = 0, w3 = 0;
  if (take_row_error(&w1, stream) != cudaSuccess || take_col_error(&w2, stream) != cudaSuccess ||
      take_wide_error(&w3, stream) != cudaSuccess)
    return FBOB_ERR_CUDA;
  const uint32_t w = w1 | w2 | w3;
  if (w & kDevErrTimeout) return FBOB_ERR_DEVICE_TIMEOUT;
  if (w) return FBOB_ERR_DEVICE_FAULT;
  return FBOB_OK;
}

}  // extern "C"
