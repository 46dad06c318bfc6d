/*
 * fbob.h -- C ABI of libfbob: exact backward-over-backward (BoB) of softmax
 * attention on one NVIDIA GB300 (sm_103a).
 *
 * Notation follows the paper (FlashBoB, arXiv 2609.24089): per attention head
 * Q, K, V, dO, U_Q, U_K, U_V are N x d matrices, tau is the softmax scale,
 * P = softmax_row(tau Q K^T + M) (Sec. 2, eq. 1).  U_Q, U_K, U_V are the
 * cotangents on the first-backward outputs dQ, dK, dV; this header calls
 * them gq, gk, gv.
 *
 * Common conventions for every entry point
 * ----------------------------------------
 *  Layout     All matrices are contiguous row-major [B, H, N, d] bf16
 *             (element (b,h,i,a) at ((b*H + h)*N + i)*d + a).  Row vectors
 *             (lse, dstat, alpha, E, D) are contiguous fp32 [B, H, N].
 *  Pointers   Device pointers (global memory of the current device), each
 *             16-byte aligned.  Outputs must not overlap any input or each
 *             other.
 *  Shapes     d in {32, 64, 128, 256}; other head dims return
 *             FBOB_ERR_UNSUPPORTED.  (d = 32 runs in the kernels' 64-wide
 *             tiles, the missing columns loaded as zeros.  d = 256, App.
 *             "Head-dimension sensitivity", runs in kernels of its own with
 *             32-row streamed tiles and one accumulator per kernel; each
 *             entry point below states its launches there.)
 *             N >= 0 is arbitrary (tails are masked); B*H*N == 0 is a valid
 *             empty problem that launches nothing and returns FBOB_OK.
 *             N <= 2^24, B*H <= 2^24 and ceil(N/128) * B*H * 2 < 2^31 (the
 *             launch grids).  scale must be finite and > 0
 *             (1/sqrt(d) in the paper).  causal is 0 or 1; with 1 the mask
 *             keeps j <= i (square, top-left aligned, diagonal included).
 *             window_left, window_right (each -1 or >= 0) add a sliding-window
 *             band: row i keeps i - window_left <= j <= i + window_right
 *             (App. "Sliding-window attention"); -1 leaves that side
 *             unbounded.  Every row keeps its diagonal.  Both -1 (and causal 0)
 *             is the unmasked problem.
 *             seq_offsets (optional) packs variable-length sequences along N
 *             (App. "Extensions"): a device array of num_seqs + 1 int32 with
 *             seq_offsets[0] = 0, non-decreasing, seq_offsets[num_seqs] = N,
 *             the same for every (b, h).  Row i then keeps only the columns of
 *             its own sequence (intersected with the causal mask and the
 *             window); causal and the window apply within a sequence in the
 *             global index.  The contents are not checked on the host; offsets
 *             that break these rules give unspecified values but no access
 *             outside the caller's buffers.  NULL (with num_seqs 0) is one
 *             sequence.
 *             block_mask (optional) is a block-sparse mask (App.
 *             "Extensions": each row keeps a set of allowed columns and the
 *             streamed loops visit only the block pairs with an allowed
 *             entry): a device array of nb x nb bytes, nb = ceil(N / 128),
 *             row-major over (query block, key block) of 128 x 128 entries,
 *             the same for every (b, h).  Pair (i, j) is kept only if byte
 *             (i / 128) * nb + j / 128 is nonzero (and the causal mask, the
 *             window and the packed sequences keep it).  Every diagonal block
 *             must be set, so that every row keeps its diagonal; the contents
 *             are not checked on the host, and a mask that breaks the rule
 *             gives unspecified values but no access outside the caller's
 *             buffers.  It must not overlap any output.  Each CTA scans its
 *             row (or column) of the mask, O(nb) bytes.  NULL keeps every
 *             block.
 *  GQA        H_kv > 0 (a divisor of H) gives grouped-query attention: the
 *             key/value-side tensors (k, v, gk, gv and k_bar, v_bar, dk, dv)
 *             are [B, H_kv, N, d] and query head h reads key/value head
 *             h / (H / H_kv).  dK, dV, k_bar and v_bar of a key/value head are
 *             then sums over its H / H_kv query heads, summed inside one CTA in
 *             a fixed order.  Query-side tensors and row vectors keep H heads.
 *  Dropout    dropout_p in [0, 1) with dropout_seed applies attention dropout
 *             after the softmax (App. "Extensions"): O = sigma (R o P) V with a
 *             keep mask R and sigma the inverse keep rate; the first backward
 *             and the BoB differentiate that forward (dP, C, dV, Vtil and
 *             dOtil carry sigma R; L, D, alpha and E stay over the ungated P).
 *             R is regenerated in every kernel from Philox4x32-10 (Salmon et
 *             al., SC'11), never stored: the 4 x 4 block (i/4, j/4) of query
 *             head b*H + h uses counter {j/4, i/4, b*H + h, 0} and key
 *             {seed low 32 bits, seed high 32 bits}; pair (i, j) takes byte
 *             j%4 of output word i%4 and is kept iff that byte is >= t, with
 *             t = round(256 dropout_p) (at most 255).  The realised drop rate
 *             is t/256 and sigma = 256/(256 - t).  t = 0 (dropout_p < 1/512)
 *             is no dropout.  i and j are positions along N (with packed
 *             sequences, global positions).  The forward, first backward and
 *             BoB of one problem must be given the same dropout_p and seed.
 *  Stream     Every call enqueues its kernels on `stream` (NULL = legacy
 *             default stream) and returns without synchronising.
 *  Memory     The library allocates and frees no device memory.  The caller
 *             owns every buffer (fbob_attn_bob_host's device workspace
 *             included).  Library state is one device-side error word per
 *             device, cached driver entry points, and the fixed 64 MiB staging
 *             array of fbob_attn_bob_host_noalloc.  Under lazy module loading
 *             (the CUDA default) that array is placed on a device by that
 *             call's first use there; with CUDA_MODULE_LOADING=EAGER every
 *             context that loads the library reserves it at once, whether or
 *             not the call is ever made.  fbob_attn_bob_host creates three streams
 *             and seven events per call and releases them when their work is
 *             done; no other call creates any CUDA object.
 *  Errors     Host-side validation failures return immediately, before any
 *             CUDA call, and launch nothing.  A failed launch returns
 *             FBOB_ERR_CUDA.  Kernels never trap: every device-side wait is
 *             bounded, and on expiry the kernel records FBOB_ERR_DEVICE_TIMEOUT
 *             in the device error word and exits cleanly; fbob_device_status()
 *             reports it.
 *  Debug      Two environment variables, read at every call, control the
 *             bounded waits: FBOB_WAIT_LIMIT_MS (1..60000, default 2000) is the
 *             limit of each wait, and FBOB_INJECT_STALL=1 injects a stall (the
 *             kernels load nothing, every wait expires, the outputs are left
 *             unspecified and fbob_device_status() then reports
 *             FBOB_ERR_DEVICE_TIMEOUT) for testing failure detection.
 *  Determinism  No floating-point atomics; every output element has one
 *             writer, so results are bitwise reproducible run to run.
 */
#ifndef FBOB_H_
#define FBOB_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

struct CUstream_st; /* cudaStream_t == struct CUstream_st* */

typedef enum fbob_status {
    FBOB_OK = 0,
    FBOB_ERR_INVALID_ARGUMENT = 1, /* null/misaligned/overlapping pointer, bad shape, scale */
    FBOB_ERR_UNSUPPORTED = 2,      /* valid request the library does not implement (d not 32/64/128/256) */
    FBOB_ERR_CUDA = 3,             /* a CUDA runtime/driver call or launch failed */
    FBOB_ERR_DEVICE_TIMEOUT = 4,   /* a bounded device-side wait expired */
    FBOB_ERR_DEVICE_FAULT = 5,     /* the device reported an error while synchronising */
    FBOB_ERR_SCRATCH_LIMIT = 6     /* the problem needs more staging memory than the
                                      fixed array of fbob_attn_bob_host_noalloc */
} fbob_status;

typedef struct fbob_shape {
    int64_t B, H, N, d;
    float scale;          /* tau */
    int32_t causal;       /* 0 or 1 */
    int32_t window_left;  /* sliding window: row i keeps j >= i - window_left; -1 = unbounded */
    int32_t window_right; /* and j <= i + window_right; -1 = unbounded (causal caps it at 0) */
    const int32_t* seq_offsets; /* packed sequences: device int32 [num_seqs + 1], or NULL */
    int64_t num_seqs;           /* number of packed sequences (0 when seq_offsets is NULL) */
    int64_t H_kv; /* key/value heads (grouped-query attention); 0 = H */
    double dropout_p;      /* attention dropout rate in [0, 1); 0 = none */
    uint64_t dropout_seed; /* Philox key of the dropout mask */
    const uint8_t* block_mask; /* block-sparse mask: device uint8 [nb][nb], nb = ceil(N/128), or NULL */
} fbob_shape;

/*
 * Forward attention, Sec. 2 eq. (1):
 *   S = scale * Q K^T + M,  P = softmax_row(S),  O = P V,
 *   lse_i = L_i = log sum_{j valid} exp(S_ij)   (natural log, fp32).
 * In:  q, k, v  bf16 [B,H,N,d].   Out: o bf16 [B,H,N,d], lse fp32 [B,H,N].
 * One kernel (an online softmax over the key tiles).
 */
int fbob_attn_fwd(const fbob_shape* shape, const void* q, const void* k, const void* v,
                  void* o, float* lse, struct CUstream_st* stream);

/*
 * First backward, Sec. 2 eqs. (2)-(3):
 *   dP = dO V^T, dV = P^T dO, D_i = do_i . o_i, dS = P o (dP - D 1^T),
 *   dQ = scale dS K, dK = scale dS^T Q.
 * P is recomputed from q, k and lse.  D (fp32, from the given o and dout) is
 * written to dstat [B,H,N].
 * In:  q, k, v, o, dout bf16; lse fp32.   Out: dq, dk, dv bf16; dstat fp32.
 * Two kernels (dq and dstat by row blocks, dk and dv by key blocks); at
 * d = 256 three (dq and dstat, dv, dk).
 */
int fbob_attn_bwd(const fbob_shape* shape, const void* q, const void* k, const void* v,
                  const void* o, const float* lse, const void* dout,
                  void* dq, void* dk, void* dv, float* dstat, struct CUstream_st* stream);

/*
 * Backward-over-backward, Sec. 3.1 eqs. (4)-(5) and closed form eqs. (6)-(7):
 *   Phi = <dQ, U_Q> + <dK, U_K> + <dV, U_V>,
 *   (q_bar, k_bar, v_bar, dout_bar) = grad_{Q, K, V, dO} Phi,
 * computed by the row-block pass, then the column-block pass of Algorithm 1:
 * pass 1 as fbob_attn_bob_pass1 describes (one sweep with the affine fusion
 * of Prop. 3.1 / eq. (8) at d <= 64 without dropout; otherwise the row
 * scalars first, then the direct form of eqs. (6)-(7)), pass 2 as
 * fbob_attn_bob_pass2: 2 kernels at d <= 64, 3 at d = 128 or with dropout,
 * 5 at d = 256.  No N x N tensor is written to memory.
 * In:  q, k, v, o, dout, gq, gk, gv  bf16 [B,H,N,d]; lse fp32 [B,H,N] (natural
 *      log, as written by fbob_attn_fwd).
 * Out: q_bar, k_bar, v_bar, dout_bar bf16 [B,H,N,d];
 *      row_stats fp32 [3,B,H,N] = (alpha, E, D): the two BoB row scalars of
 *      eq. (6) (alpha_i = sum_j P_ij F_ij, E_i = sum_j P_ij Ptil_ij) and
 *      D_i = do_i . o_i.  Pass 1 writes it, pass 2 reads it; it is required.
 */
int fbob_attn_bob(const fbob_shape* shape, const void* q, const void* k, const void* v,
                  const void* o, const float* lse, const void* dout,
                  const void* gq, const void* gk, const void* gv,
                  void* q_bar, void* k_bar, void* v_bar, void* dout_bar,
                  float* row_stats, struct CUstream_st* stream);

/*
 * Pass 1 of Algorithm 1 alone (row-block outer; Alg. 2, first loop):
 * writes q_bar, dout_bar and row_stats (alpha, E, D).  Same arguments and
 * rules as fbob_attn_bob; k_bar/v_bar are not touched.  d <= 64 without
 * dropout runs one sweep with the affine fusion of Prop. 3.1 (one kernel);
 * d = 128, and any d with dropout, runs fbob_attn_bob_row_stats then
 * fbob_attn_bob_pass1_direct (two kernels; three at d = 256).
 */
int fbob_attn_bob_pass1(const fbob_shape* shape, const void* q, const void* k, const void* v,
                        const void* o, const float* lse, const void* dout,
                        const void* gq, const void* gk, const void* gv,
                        void* q_bar, void* dout_bar, float* row_stats,
                        struct CUstream_st* stream);

/*
 * Pass 1 in one sweep with the affine fusion of Prop. 3.1 (eq. 8) at any
 * supported d (the form fbob_attn_bob_pass1 takes at d <= 64): each row block
 * streams K, U_K, V, U_V once and accumulates B = sum_j P_ij k_j, dOtil0 =
 * sum_j P_ij (u_V,j + F_ij v_j), G = sum_j dS_ij k_j and Omega = sum_j
 * (P o Ptil0)_ij k_j + dS_ij u_K,j with the running row sums alpha and E0;
 * the epilogue forms E = E0 - alpha D, dOtil = dOtil0 - alpha o and Qtil =
 * tau (Omega - alpha G - E0 B).  At d = 128 the four accumulators are split
 * by output column over two CTAs per row block (each computes the whole
 * stage A and its 64 columns of stage B).  One kernel.  Same arguments and
 * outputs as fbob_attn_bob_pass1; dropout, and d = 256 (four 256-column
 * accumulators exceed tensor memory), return FBOB_ERR_UNSUPPORTED before any
 * CUDA call.
 */
int fbob_attn_bob_pass1_fused(const fbob_shape* shape, const void* q, const void* k,
                              const void* v, const void* o, const float* lse, const void* dout,
                              const void* gq, const void* gk, const void* gv, void* q_bar,
                              void* dout_bar, float* row_stats, struct CUstream_st* stream);

/*
 * Pass 2 of Algorithm 1 alone (column-block outer; Alg. 2, second loop):
 * reads row_stats (alpha, E, D, as pass 1 writes them) and lse, writes
 * k_bar and v_bar.  row_stats is an input here.  One kernel; at d = 256 two
 * (v_bar, then k_bar over two CTAs per key block, 128 output columns each).
 */
int fbob_attn_bob_pass2(const fbob_shape* shape, const void* q, const void* k, const void* v,
                        const float* lse, const void* dout,
                        const void* gq, const void* gk, const void* gv,
                        const float* row_stats, void* k_bar, void* v_bar,
                        struct CUstream_st* stream);

/*
 * Row scalars of BoB alone (eq. 6): writes row_stats [3,B,H,N] = (alpha, E, D)
 * with alpha_i = sum_j P_ij F_ij, E_i = sum_j P_ij Ptil_ij and D_i = do_i . o_i,
 * exactly as pass 1 writes them (stage A only; no N x d output).  At d = 128,
 * and with dropout, fbob_attn_bob_pass1 is this call followed by
 * fbob_attn_bob_pass1_direct.
 * Same arguments and rules as fbob_attn_bob_pass1.
 */
int fbob_attn_bob_row_stats(const fbob_shape* shape, const void* q, const void* k,
                            const void* v, const void* o, const float* lse, const void* dout,
                            const void* gq, const void* gk, const void* gv, float* row_stats,
                            struct CUstream_st* stream);

/*
 * Pass 1 given its row scalars: q_bar and dout_bar from eqs. (6)-(7) directly,
 *   q_bar = scale (Stil K + dS U_K),  dout_bar = P U_V + (P o h) V,
 * with alpha, E, D read from row_stats (as fbob_attn_bob_row_stats or pass 1
 * writes them; input here) and P from lse.  O is not needed.  One kernel; at
 * d = 256 two (dout_bar, then q_bar).
 * In:  q, k, v, dout, gq, gk, gv bf16; lse fp32; row_stats fp32 [3,B,H,N].
 * Out: q_bar, dout_bar bf16 [B,H,N,d].
 */
int fbob_attn_bob_pass1_direct(const fbob_shape* shape, const void* q, const void* k,
                               const void* v, const float* lse, const void* dout,
                               const void* gq, const void* gk, const void* gv,
                               const float* row_stats, void* q_bar, void* dout_bar,
                               struct CUstream_st* stream);

/*
 * fbob_attn_bob with every tensor in host memory: the same computation and
 * the same results, bit for bit.  The B*H query heads are processed in
 * chunks of whole key/value groups, and each chunk's inputs are copied in,
 * computed and copied out on separate streams through two slots of a
 * caller-owned device workspace, so copies and kernels of neighbouring
 * chunks overlap, and so do the kernels of consecutive chunks (each head is
 * an independent problem, Alg. 1).
 * In:  q, k, v, o, lse, dout, gq, gk, gv: host buffers with the layouts of
 *      fbob_attn_bob.  Page-locked memory lets the copies run asynchronously;
 *      pageable memory gives the same results, without the overlap.
 * Out: q_bar, k_bar, v_bar, dout_bar, row_stats: host buffers, as in
 *      fbob_attn_bob; they must not overlap any input or each other.
 * workspace: device memory of workspace_bytes, 256-byte aligned, owned by the
 *      caller and not used by anything else until `stream` has passed this
 *      call.  fbob_attn_bob_host_workspace() gives the bytes for a chunk size;
 *      the call takes about a quarter of the heads per chunk, or fewer when
 *      the workspace is smaller, and returns FBOB_ERR_INVALID_ARGUMENT if it
 *      cannot hold one key/value group.
 * Stream: the copies start after the work already enqueued on `stream`, and
 *      `stream` completes only after the last copy out; synchronise it before
 *      reading the outputs.  Three streams and seven events are created per
 *      call and released when their work completes.  If the call returns an
 *      error after validation (a failed CUDA call), copies and kernels it has
 *      already enqueued may still be running on its own streams: synchronise
 *      the device before reusing the buffers or the workspace.
 */
int fbob_attn_bob_host(const fbob_shape* shape, const void* q, const void* k, const void* v,
                       const void* o, const float* lse, const void* dout,
                       const void* gq, const void* gk, const void* gv,
                       void* q_bar, void* k_bar, void* v_bar, void* dout_bar, float* row_stats,
                       void* workspace, int64_t workspace_bytes, struct CUstream_st* stream);

/*
 * Device workspace bytes fbob_attn_bob_host needs to run chunks of
 * chunk_heads query heads (rounded up to whole key/value groups), or -1 for
 * an invalid shape or chunk_heads < 1.
 */
int64_t fbob_attn_bob_host_workspace(const fbob_shape* shape, int64_t chunk_heads);

/*
 * fbob_attn_bob_host for callers that cannot allocate device memory while they
 * run, such as a process that reserves its whole device footprint when it
 * starts and may not grow it later, or one that cannot spare a workspace of
 * its own.  No workspace argument and no allocation of any kind per call: the
 * chunks of heads are staged in a fixed 64 MiB device array that the library
 * declares statically.  The paper has no counterpart; it is the same
 * computation (the same kernels on each head) behind a different interface,
 * and its results equal fbob_attn_bob_host's bit for bit.
 * Arguments and layouts as fbob_attn_bob_host (host buffers; page-locked for
 * asynchronous copies).  The heads go in chunks of whole key/value groups, as
 * many as fit in the array, one chunk after the other on `stream` (copy in,
 * Pass 1, Pass 2, copy out; copies do not overlap the kernels).
 * Limit: the staging of one key/value group, about 12 N d (H / H_kv) * 2
 *      bytes, must fit in 64 MiB (for example N = 16384 at d = 128 without
 *      grouping); larger problems return FBOB_ERR_SCRATCH_LIMIT and run
 *      nothing (use fbob_attn_bob_host with a workspace).
 * Set-up: every call looks up the array's device address on the current
 *      device (cudaGetSymbolAddress, no allocation), so an address is never
 *      reused across a context teardown (cudaDeviceReset).  Under lazy module
 *      loading the first lookup on a device also places the array there; make
 *      that first call before any stream capture.
 * Nothing in the array has to start at zero: each call writes every byte it
 *      reads.  All calls on a device share the array, so calls that overlap in
 *      time (on other streams or threads) race; serialise them.
 */
int fbob_attn_bob_host_noalloc(const fbob_shape* shape, const void* q, const void* k,
                               const void* v, const void* o, const float* lse,
                               const void* dout, const void* gq, const void* gk,
                               const void* gv, void* q_bar, void* k_bar, void* v_bar,
                               void* dout_bar, float* row_stats, struct CUstream_st* stream);

/*
 * Synchronises `stream`, then returns and clears the device error word of the
 * current device: FBOB_OK, FBOB_ERR_DEVICE_TIMEOUT (a bounded wait expired in
 * some kernel since the last call), or FBOB_ERR_DEVICE_FAULT / FBOB_ERR_CUDA
 * if synchronisation itself failed.
 */
int fbob_device_status(struct CUstream_st* stream);

/* Number of kernels the last successful call of the named entry point
 * enqueued ("fwd", "bwd", "bob", "bob_pass1", "bob_pass2", "bob_row_stats",
 * "bob_pass1_direct", "bob_host", "bob_host_noalloc", "bob_pass1_fused");
 * -1 if unknown. */
int fbob_launch_count(const char* entry);

/* Static, human-readable name of a status code. */
const char* fbob_status_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* FBOB_H_ */
