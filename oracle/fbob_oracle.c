/*
 * fbob_oracle.c -- plain fp64 CPU oracle for exact attention backward-over-backward.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may load or call this
 * file: only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline /
 * reference leg use it.  It shares no code, header, table or helper with the
 * CUDA library under paper_2609_24089_gb300/csrc.
 *
 * What it computes, all per single attention head, on row-major [N x d] fp64
 * arrays (the bf16 test inputs up-cast exactly):
 *
 *   fbob_oracle_fwd : forward attention, Sec. 2 eq. (1):
 *                     S = tau Q K^T + M,  P = softmax_row(S),  O = P V,
 *                     L_i = log sum_{j in V_i} exp(S_ij)  (natural log).
 *   fbob_oracle_bwd : first backward, eqs. (2)-(3):
 *                     dP = dO V^T, dV = P^T dO, D_i = sum_j P_ij dP_ij,
 *                     dS = P o (dP - D 1^T), dQ = tau dS K, dK = tau dS^T Q.
 *   fbob_oracle_bob : backward-over-backward, eqs. (4)-(7), App. C steps 1-7
 *                     and the assembled identities closing App. C:
 *                     F = tau (U_Q K^T + Q U_K^T)           (App. C step 1)
 *                     alpha_i = sum_j P_ij F_ij              (step 2)
 *                     Vtil = (P o h)^T dO, h = F - alpha 1^T (step 3)
 *                     C = dO U_V^T,  dOtil = P U_V + (P o h) V   (step 4)
 *                     Ptil = C + F o (dP - D 1^T) - alpha o dP    (step 5)
 *                     E_i = sum_j P_ij Ptil_ij, Stil = P o (Ptil - E 1^T)  (step 6)
 *                     Qtil = tau (Stil K + dS U_K), Ktil = tau (Stil^T Q + dS^T U_Q) (step 7)
 *
 * The oracle deliberately does NOT use the affine fusion of Prop. 3.1 nor the
 * two-pass schedule of Algorithm 1: every row is materialised in full (all N
 * scores of that row), alpha and E are formed as plain row sums before they are
 * used, and every output is the plain sum its defining equation states.
 *
 * Masking (Sec. 2; sliding window, App. "Sliding-window attention"): the valid
 * column set of row i is the band V_i = {j : lo_i <= j < hi_i} with
 *   lo_i = max(0, i - wl)                    (wl < 0: lo_i = 0),
 *   hi_i = min(N, i + wr + 1)                (wr < 0: hi_i = N),
 * and the causal mask (square, top-left aligned, diagonal included) caps
 * hi_i at i + 1.  wl = wr = -1 is the plain mask.  Packed variable-length
 * sequences (App. "Extensions"): with segment offsets seg[0..nseg] (seg[0] =
 * 0, non-decreasing, seg[nseg] = N) row i also keeps only the columns of its
 * own segment [seg[s], seg[s+1]), s the segment holding i; seg = NULL is one
 * segment.  Block-sparse masks (App. "Extensions": a sparse mask only needs a
 * well-defined set of allowed columns per row, with zero probability on the
 * masked entries): with a block mask bm of nb x nb bytes over square blocks of
 * bs rows and bs columns (nb = ceil(N / bs)), the pair (i, j) is kept only if
 * also bm[(i / bs) * nb + j / bs] != 0; bm = NULL keeps every block.  Every
 * row keeps its diagonal (for the block mask: every diagonal block is set).
 * Entries outside V_i, and masked entries inside it, have P = 0 and
 * contribute nothing.
 *
 * Dropout (App. "Extensions"): with keep mask R and sigma = 1/(1 - p) the
 * forward uses sigma (R o P); the row scalars L, D, alpha, E stay defined over
 * the ungated P; the gating acts on dP -> sigma R dP, C -> sigma R C, on
 * dV = sigma (R o P)^T dO, and in the BoB on Vtil and dOtil:
 *   Vtil_j = sigma sum_i R_ij P_ij h_ij do_i,
 *   dOtil_i = sigma sum_j R_ij P_ij (u_V,j + h_ij v_j).
 * The paper asks for a counter-based generator such as Philox and leaves the
 * bit layout open.  Here one Philox4x32-10 call covers a 4 x 4 block of
 * (query, key) pairs with one random byte each: for the block (i / 4, j / 4)
 * of query head `head` the counter is {j / 4, i / 4, head, 0} and the key
 * {seed low 32 bits, seed high 32 bits}; the pair (i, j) takes byte (j mod 4)
 * (bits 8 (j mod 4) .. + 7) of output word (i mod 4).  R_ij = 1 iff that byte
 * is >= t, t = floor(256 p + 1/2) clamped to 255; the realised drop rate is
 * t / 256 and sigma = 256 / (256 - t).  t = 0 (p < 1/512) keeps everything
 * and leaves every result unchanged.
 *
 * Threads: rows are independent, so OpenMP splits rows across threads.  The
 * column-owned sums (Ktil, Vtil, dV, dK) are accumulated into one private
 * buffer per thread and reduced in thread order at the end.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Optional deliberately planted mistakes, used only by the test that checks
 * the pins have the power to catch them (tests/test_oracle_mutants.py).  The
 * default build has FBOB_MUTANT == 0 and none of these branches exist. */
#ifndef FBOB_MUTANT
#define FBOB_MUTANT 0
#endif

static double dot(const double* a, const double* b, int64_t d) {
    double s = 0.0;
    for (int64_t t = 0; t < d; ++t) s += a[t] * b[t];
    return s;
}

/* Philox4x32-10 (Salmon, Moraes, Dror and Shaw, "Parallel random numbers:
 * as easy as 1, 2, 3", SC'11): ten rounds of the Philox S-box on a 4 x 32-bit
 * counter under a 2 x 32-bit key, the key raised by the Weyl constants
 * 0x9E3779B9, 0xBB67AE85 before every round but the first. */
void fbob_oracle_philox(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
    uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    uint32_t k0 = key[0], k1 = key[1];
    for (int r = 0; r < 10; ++r) {
        if (r > 0) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        const uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)c0;
        const uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)c2;
        const uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
        const uint32_t n1 = (uint32_t)p1;
        const uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
        const uint32_t n3 = (uint32_t)p0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* dropout: the byte threshold t and the gate g_ij = sigma R_ij (1 without dropout) */
typedef struct { int on; uint32_t thr; double sigma; uint64_t seed; int64_t head; } drop_t;

static drop_t make_drop(double p, uint64_t seed, int64_t head) {
    drop_t r = {0, 0u, 1.0, seed, head};
    double t = floor(256.0 * p + 0.5);
    if (t > 255.0) t = 255.0;
    if (t >= 1.0) {
        r.on = 1;
        r.thr = (uint32_t)t;
        r.sigma = 256.0 / (256.0 - t);
    }
    return r;
}

static double gate(drop_t g, int64_t i, int64_t j) {
    if (!g.on) return 1.0;
    const uint32_t ctr[4] = {(uint32_t)(j >> 2), (uint32_t)(i >> 2), (uint32_t)g.head, 0u};
    const uint32_t key[2] = {(uint32_t)g.seed, (uint32_t)(g.seed >> 32)};
    uint32_t w[4];
    fbob_oracle_philox(ctr, key, w);
    const uint32_t byte = (w[i & 3] >> (8 * (j & 3))) & 0xFFu;
    return byte >= g.thr ? g.sigma : 0.0;
}

/* the valid columns [lo_i, hi_i) of row i (see the header comment), and the
 * block mask inside that range */
typedef struct {
    int causal; int64_t wl, wr; const int64_t* seg; int64_t nseg;
    const uint8_t* bm; int64_t bs, nb;
} band_t;

static band_t make_band(int64_t N, int causal, int64_t wl, int64_t wr, const int64_t* seg,
                        int64_t nseg, const uint8_t* bm, int64_t bs) {
    band_t m = {causal, wl, wr, seg, nseg, bm, bs, 0};
    if (bm && bs > 0) m.nb = (N + bs - 1) / bs;
    else m.bm = NULL;
    return m;
}

/* 1 if the block mask keeps the pair (i, j) (always without a block mask) */
static int block_keeps(band_t m, int64_t i, int64_t j) {
    return !m.bm || m.bm[(i / m.bs) * m.nb + j / m.bs] != 0;
}

static void valid_cols(int64_t i, int64_t N, band_t m, int64_t* lo, int64_t* hi) {
    int64_t a = m.wl < 0 ? 0 : i - m.wl;
    int64_t b = m.wr < 0 ? N : i + m.wr + 1;
    if (m.causal && b > i + 1) b = i + 1;
    if (m.seg) {  /* the segment holding row i: a plain scan */
        for (int64_t s = 0; s < m.nseg; ++s)
            if (m.seg[s] <= i && i < m.seg[s + 1]) {
                if (a < m.seg[s]) a = m.seg[s];
                if (b > m.seg[s + 1]) b = m.seg[s + 1];
                break;
            }
    }
    *lo = a < 0 ? 0 : a;
    *hi = b > N ? N : b;
}

static int pick_threads(int nthreads) {
#ifdef _OPENMP
    return nthreads > 0 ? nthreads : omp_get_max_threads();
#else
    (void)nthreads;
    return 1;
#endif
}

static int thread_id(void) {
#ifdef _OPENMP
    return omp_get_thread_num();
#else
    return 0;
#endif
}

/* Row i of S and P (eq. 1): S_ij = tau q_i.k_j for j in V_i = [lo, hi), L_i
 * the natural-log normaliser, P_ij = exp(S_ij - L_i).  S and P are indexed by
 * the absolute column j. */
static void softmax_row(int64_t i, int64_t N, int64_t d, double tau, band_t mk,
                        const double* Q, const double* K, double* S, double* P,
                        double* L_out, int64_t* lo_out, int64_t* hi_out) {
    int64_t lo, hi;
    valid_cols(i, N, mk, &lo, &hi);
    double m = -INFINITY;
    for (int64_t j = lo; j < hi; ++j) {
        S[j] = tau * dot(Q + i * d, K + j * d, d);
        if (block_keeps(mk, i, j) && S[j] > m) m = S[j];
    }
    double z = 0.0;
    for (int64_t j = lo; j < hi; ++j)
#if FBOB_MUTANT == 11 /* planted: masked blocks left in the normaliser */
        z += exp(S[j] - m);
#else
        if (block_keeps(mk, i, j)) z += exp(S[j] - m);
#endif
    const double L = m + log(z);
    /* masked entries of the block mask: zero probability */
    for (int64_t j = lo; j < hi; ++j) P[j] = block_keeps(mk, i, j) ? exp(S[j] - L) : 0.0;
    *L_out = L;
    *lo_out = lo;
    *hi_out = hi;
}

/* ---------------------------------------------------------------- forward */
int fbob_oracle_fwd(int64_t N, int64_t d, double tau, int causal, int64_t wl, int64_t wr,
                    const int64_t* seg, int64_t nseg, double p_drop, uint64_t seed,
                    int64_t head, const uint8_t* bm, int64_t bs,
                    const double* Q, const double* K, const double* V,
                    double* O, double* L, int nthreads) {
    if (N < 0 || d <= 0) return 1;
    const band_t mk = make_band(N, causal, wl, wr, seg, nseg, bm, bs);
    const drop_t dg = make_drop(p_drop, seed, head);
    const int nt = pick_threads(nthreads);
#pragma omp parallel num_threads(nt)
    {
        double* S = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
        double* P = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
#pragma omp for schedule(static)
        for (int64_t i = 0; i < N; ++i) {
            double Li;
            int64_t lo, hi;
            softmax_row(i, N, d, tau, mk, Q, K, S, P, &Li, &lo, &hi);
            L[i] = Li;
            for (int64_t a = 0; a < d; ++a) {
                double acc = 0.0;
                for (int64_t j = lo; j < hi; ++j) acc += gate(dg, i, j) * P[j] * V[j * d + a];
                O[i * d + a] = acc;
            }
        }
        free(S);
        free(P);
    }
    return 0;
}

/* ------------------------------------------------------- first backward */
int fbob_oracle_bwd(int64_t N, int64_t d, double tau, int causal, int64_t wl, int64_t wr,
                    const int64_t* seg, int64_t nseg, double p_drop, uint64_t seed,
                    int64_t head, const uint8_t* bm, int64_t bs,
                    const double* Q, const double* K, const double* V, const double* dO,
                    double* dQ, double* dK, double* dV, double* Dvec, int nthreads) {
    if (N < 0 || d <= 0) return 1;
    const band_t mk = make_band(N, causal, wl, wr, seg, nseg, bm, bs);
    const drop_t dg = make_drop(p_drop, seed, head);
    const int nt = pick_threads(nthreads);
    const size_t nd = (size_t)N * (size_t)d;
    double* part = (double*)calloc((size_t)nt * 2 * (nd > 0 ? nd : 1), sizeof(double));
    if (!part) return 2;
#pragma omp parallel num_threads(nt)
    {
        double* S = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
        double* P = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
        double* dP = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
        double* my_dK = part + (size_t)thread_id() * 2 * nd;
        double* my_dV = my_dK + nd;
#pragma omp for schedule(static)
        for (int64_t i = 0; i < N; ++i) {
            double Li;
            int64_t lo, hi;
            softmax_row(i, N, d, tau, mk, Q, K, S, P, &Li, &lo, &hi);
            double D = 0.0;                                   /* D_i = sum_j P_ij dP_ij */
            for (int64_t j = lo; j < hi; ++j) {
                /* dP = dO V^T, gated by dropout: sigma R dP */
                dP[j] = gate(dg, i, j) * dot(dO + i * d, V + j * d, d);
                D += P[j] * dP[j];
            }
            Dvec[i] = D;
            for (int64_t a = 0; a < d; ++a) dQ[i * d + a] = 0.0;
            for (int64_t j = lo; j < hi; ++j) {
                const double dS = P[j] * (dP[j] - D);         /* dS = P o (dP - D) */
                for (int64_t a = 0; a < d; ++a) {
                    dQ[i * d + a] += tau * dS * K[j * d + a];     /* dQ = tau dS K   */
                    my_dK[j * d + a] += tau * dS * Q[i * d + a];  /* dK = tau dS^T Q */
                    my_dV[j * d + a] += gate(dg, i, j) * P[j] * dO[i * d + a];  /* dV = (sigma R o P)^T dO */
                }
            }
        }
        free(S);
        free(P);
        free(dP);
    }
    for (size_t e = 0; e < nd; ++e) {
        double k = 0.0, v = 0.0;
        for (int t = 0; t < nt; ++t) {
            k += part[(size_t)t * 2 * nd + e];
            v += part[(size_t)t * 2 * nd + nd + e];
        }
        dK[e] = k;
        dV[e] = v;
    }
    free(part);
    return 0;
}

/* ----------------------------------------------- backward-over-backward
 *
 * rows[0..nrows): the query rows whose row-owned outputs are produced
 *   (Qtil, dOtil, alpha, E, D, L are written at positions 0..nrows of the
 *   corresponding output arrays, in the order of rows[]).
 * [c0, c1): the key columns whose column-owned outputs Ktil, Vtil receive the
 *   contributions of the listed rows (written as a (c1-c0) x d block).  They
 *   are the complete Ktil_j, Vtil_j only when every row i with j in V_i is
 *   listed: all rows without a mask, rows i >= j with the causal mask,
 *   rows j - wr <= i <= j + wl with a window, and only rows of j's segment.
 * Any output pointer may be NULL; c1 <= c0 skips the column-owned sums.
 */
int fbob_oracle_bob(int64_t N, int64_t d, double tau, int causal, int64_t wl, int64_t wr,
                    const int64_t* seg, int64_t nseg, double p_drop, uint64_t seed,
                    int64_t head, const uint8_t* bm, int64_t bs,
                    const double* Q, const double* K, const double* V, const double* dO,
                    const double* UQ, const double* UK, const double* UV,
                    const int64_t* rows, int64_t nrows, int64_t c0, int64_t c1,
                    double* Qt, double* dOt, double* alpha_out, double* E_out,
                    double* D_out, double* L_out, double* Kt, double* Vt, int nthreads) {
    if (N < 0 || d <= 0 || nrows < 0) return 1;
    const band_t mk = make_band(N, causal, wl, wr, seg, nseg, bm, bs);
    const drop_t dg = make_drop(p_drop, seed, head);
    for (int64_t r = 0; r < nrows; ++r)
        if (rows[r] < 0 || rows[r] >= N) return 1;
    if (c0 < 0) c0 = 0;
    if (c1 > N) c1 = N;
    const int64_t ncols = c1 > c0 ? c1 - c0 : 0;
    const int nt = pick_threads(nthreads);
    const size_t cd = (size_t)ncols * (size_t)d;
    double* part = NULL;
    if (cd > 0) {
        part = (double*)calloc((size_t)nt * 2 * cd, sizeof(double));
        if (!part) return 2;
    }
#pragma omp parallel num_threads(nt)
    {
        const size_t n1 = (size_t)(N > 0 ? N : 1);
        double* S = (double*)malloc(sizeof(double) * n1);
        double* P = (double*)malloc(sizeof(double) * n1);
        double* dP = (double*)malloc(sizeof(double) * n1);
        double* F = (double*)malloc(sizeof(double) * n1);
        double* C = (double*)malloc(sizeof(double) * n1);
        double* Pt = (double*)malloc(sizeof(double) * n1);
        double* St = (double*)malloc(sizeof(double) * n1);
        double* dS = (double*)malloc(sizeof(double) * n1);
        double* h = (double*)malloc(sizeof(double) * n1);
        double* G = (double*)malloc(sizeof(double) * n1);
        double* my_Kt = part ? part + (size_t)thread_id() * 2 * cd : NULL;
        double* my_Vt = part ? my_Kt + cd : NULL;
#pragma omp for schedule(static)
        for (int64_t r = 0; r < nrows; ++r) {
            const int64_t i = rows[r];
            const double* q = Q + i * d;
            const double* dout = dO + i * d;
            const double* uq = UQ + i * d;
            double Li;
            int64_t lo, hi;
            /* eq. (1): scores and probabilities of row i over V_i = [lo, hi) */
            softmax_row(i, N, d, tau, mk, Q, K, S, P, &Li, &lo, &hi);
            /* eq. (2): dP = dO V^T and D_i = sum_j P_ij dP_ij */
            double D = 0.0;
            for (int64_t j = lo; j < hi; ++j) {
                G[j] = gate(dg, i, j);                       /* sigma R_ij (dropout) */
                dP[j] = G[j] * dot(dout, V + j * d, d);
                D += P[j] * dP[j];
            }
            /* App. C step 1: F = tau (U_Q K^T + Q U_K^T); step 4: C = dO U_V^T */
            for (int64_t j = lo; j < hi; ++j) {
#if FBOB_MUTANT == 1 /* planted: dropped Q U_K^T term */
                F[j] = tau * dot(uq, K + j * d, d);
#elif FBOB_MUTANT == 2 /* planted: transposed operand, U_Q paired with U_K */
                F[j] = tau * (dot(uq, UK + j * d, d) + dot(q, UK + j * d, d));
#else
                F[j] = tau * (dot(uq, K + j * d, d) + dot(q, UK + j * d, d));
#endif
#if FBOB_MUTANT == 9 /* planted: C left ungated under dropout */
                C[j] = dot(dout, UV + j * d, d);
#else
                C[j] = G[j] * dot(dout, UV + j * d, d);
#endif
            }
            /* step 2: alpha_i = sum_j P_ij F_ij */
            double alpha = 0.0;
            for (int64_t j = lo; j < hi; ++j) alpha += P[j] * F[j];
            /* step 5: Ptil = C + F o (dP - D) - alpha dP */
            for (int64_t j = lo; j < hi; ++j) {
#if FBOB_MUTANT == 3 /* planted: wrong sign on the alpha term */
                Pt[j] = C[j] + F[j] * (dP[j] - D) + alpha * dP[j];
#elif FBOB_MUTANT == 4 /* planted: dropped C (the dV-child contribution) */
                Pt[j] = F[j] * (dP[j] - D) - alpha * dP[j];
#else
                Pt[j] = C[j] + F[j] * (dP[j] - D) - alpha * dP[j];
#endif
            }
            /* step 6: E_i = sum_j P_ij Ptil_ij, Stil = P o (Ptil - E) */
            double E = 0.0;
            for (int64_t j = lo; j < hi; ++j) E += P[j] * Pt[j];
            for (int64_t j = lo; j < hi; ++j) {
#if FBOB_MUTANT == 5 /* planted: E row scalar dropped */
                St[j] = P[j] * Pt[j];
#else
                St[j] = P[j] * (Pt[j] - E);
#endif
                dS[j] = P[j] * (dP[j] - D);                  /* eq. (2) */
                h[j] = F[j] - alpha;                          /* step 3 */
            }
            /* step 7: Qtil_i = tau sum_j (Stil_ij k_j + dS_ij u_K,j);
             * step 4: dOtil_i = sum_j (P_ij u_V,j + P_ij h_ij v_j) */
            if (Qt || dOt) {
                for (int64_t a = 0; a < d; ++a) {
                    double qa = 0.0, oa = 0.0;
                    for (int64_t j = lo; j < hi; ++j) {
                        qa += St[j] * K[j * d + a] + dS[j] * UK[j * d + a];
#if FBOB_MUTANT == 6 /* planted: h replaced by F (alpha dropped from h) */
                        oa += G[j] * (P[j] * UV[j * d + a] + P[j] * F[j] * V[j * d + a]);
#elif FBOB_MUTANT == 7 /* planted: wrong index, value row i used for every j */
                        oa += G[j] * (P[j] * UV[j * d + a] + P[j] * h[j] * V[i * d + a]);
#elif FBOB_MUTANT == 10 /* planted: the U_V term of dOtil left ungated */
                        oa += P[j] * UV[j * d + a] + G[j] * P[j] * h[j] * V[j * d + a];
#else
                        oa += G[j] * (P[j] * UV[j * d + a] + P[j] * h[j] * V[j * d + a]);
#endif
                    }
                    if (Qt) Qt[r * d + a] = tau * qa;
                    if (dOt) dOt[r * d + a] = oa;
                }
            }
            if (alpha_out) alpha_out[r] = alpha;
            if (E_out) E_out[r] = E;
            if (D_out) D_out[r] = D;
            if (L_out) L_out[r] = Li;
            /* step 7 / step 3: column-owned sums over the listed rows:
             * Ktil_j += tau (Stil_ij q_i + dS_ij u_Q,i),  Vtil_j += P_ij h_ij do_i */
            if (my_Kt) {
                const int64_t jbeg = lo > c0 ? lo : c0;
                const int64_t jend = hi < c1 ? hi : c1;
                for (int64_t j = jbeg; j < jend; ++j) {
                    double* kt = my_Kt + (size_t)(j - c0) * d;
                    double* vt = my_Vt + (size_t)(j - c0) * d;
                    const double ph = G[j] * P[j] * h[j];
                    for (int64_t a = 0; a < d; ++a) {
#if FBOB_MUTANT == 8 /* planted: U_Q term replaced by U_K of row i */
                        kt[a] += tau * (St[j] * q[a] + dS[j] * UK[i * d + a]);
#else
                        kt[a] += tau * (St[j] * q[a] + dS[j] * uq[a]);
#endif
                        vt[a] += ph * dout[a];
                    }
                }
            }
        }
        free(S); free(P); free(dP); free(F); free(C); free(Pt); free(St); free(dS); free(h);
        free(G);
    }
    if (part) {
        for (size_t e = 0; e < cd; ++e) {
            double k = 0.0, v = 0.0;
            for (int t = 0; t < nt; ++t) {
                k += part[(size_t)t * 2 * cd + e];
                v += part[(size_t)t * 2 * cd + cd + e];
            }
            if (Kt) Kt[e] = k;
            if (Vt) Vt[e] = v;
        }
        free(part);
    }
    return 0;
}
