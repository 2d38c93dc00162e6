/*
 * gla_oracle.c -- plain fp64 CPU oracle for the GTR token mixer (key-only gated
 * linear attention run along one spatial scan order).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  It shares
 * no code, header, table or helper with the CUDA path, and nothing here is
 * tuned: every loop follows the paper's definition as written.
 *
 * Definitions followed (paper "GTR: Gated Token Recurrence for Efficient Dense
 * Prediction"):
 *   - Sec. 3.1 "Key-only gated recurrence":
 *         S_t = Diag(gamma_t) S_{t-1} + k_t^T v_t,   S_0 = 0,
 *         o_t = q_t S_t
 *     with the value-side decay fixed to one (Sec. 3.1 and App. C.3), and
 *     gamma_t = exp(g_t), g_t the learned log-decay the operator consumes
 *     (Sec. 3.3).  The d_k^{-1/2} factor of the paper's o_t is NOT applied
 *     here: the caller folds it into k, which gives the same o_t (the scale
 *     multiplies every k_t^T v_t term of S_t alike).
 *   - Sec. 3.1 "Directional scanning": four raster orders over the grid
 *     (left-to-right, right-to-left, top-to-bottom, bottom-to-top), one
 *     sequence per image with the state carried across rows/columns, outputs
 *     written back at the token's spatial position.
 *   - Sec. 3.3, Eq. (chunk_boundary_main) and the chunk-output formula that
 *     follows it: the chunkwise schedule, implemented separately below with a
 *     free chunk size C as a second restatement of the same recurrence.
 *
 * Layouts (row-major, spatial token order t = y * grid_w + x):
 *   q, k, g : [B][T][H][Dk]      v, out : [B][T][H][Dv]
 *   final_state : [B][H][Dk][Dv]  (state after the last token in scan order)
 * All arrays are double.  g may hold -inf (gamma = 0).
 *
 * Build: gcc -O2 -ffp-contract=off -fopenmp -shared -fPIC (see __init__.py).
 */
#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORDER_ROW_FWD = 0, ORDER_ROW_REV = 1, ORDER_COL_FWD = 2, ORDER_COL_REV = 3 };

/* Spatial token index visited at scan position s (Sec. 3.1, "Directional
 * scanning").  Row orders walk rows left-to-right (or the exact reverse);
 * column orders walk columns top-to-bottom (or the exact reverse).  Returns
 * -1 for an unknown order. */
long gla_oracle_scan_token(int order, long grid_h, long grid_w, long s)
{
    long T = grid_h * grid_w;
    switch (order) {
    case ORDER_ROW_FWD: return s;
    case ORDER_ROW_REV: return T - 1 - s;
    case ORDER_COL_FWD: return (s % grid_h) * grid_w + s / grid_h;
    case ORDER_COL_REV: {
        long u = T - 1 - s;
        return (u % grid_h) * grid_w + u / grid_h;
    }
    default: return -1;
    }
}

static long idx4(long b, long t, long h, long c, long T, long H, long D)
{
    return ((b * T + t) * H + h) * D + c;
}

static int check_args(int B, int H, int grid_h, int grid_w, int Dk, int Dv, int order)
{
    if (B < 0 || H < 0 || grid_h < 0 || grid_w < 0 || Dk <= 0 || Dv <= 0) return 1;
    if (order < 0 || order > 3) return 1;
    return 0;
}

/* One (b, h) sequence of the token recurrence, Sec. 3.1. */
static void recurrence_one(const double *q, const double *k, const double *v, const double *g,
                           long b, long h, long B, long H, long grid_h, long grid_w,
                           long Dk, long Dv, int order, double *out, double *final_state,
                           double *S)
{
    long T = grid_h * grid_w;
    (void)B;
    memset(S, 0, sizeof(double) * (size_t)(Dk * Dv));          /* S_0 = 0 */
    for (long s = 0; s < T; ++s) {
        long t = gla_oracle_scan_token(order, grid_h, grid_w, s);
        const double *qt = q + idx4(b, t, h, 0, T, H, Dk);
        const double *kt = k + idx4(b, t, h, 0, T, H, Dk);
        const double *gt = g + idx4(b, t, h, 0, T, H, Dk);
        const double *vt = v + idx4(b, t, h, 0, T, H, Dv);
        /* S_t = Diag(gamma_t) S_{t-1} + k_t^T v_t : row i of S decays by gamma_{t,i} */
        for (long i = 0; i < Dk; ++i) {
            double gamma = exp(gt[i]);
            for (long j = 0; j < Dv; ++j)
                S[i * Dv + j] = gamma * S[i * Dv + j] + kt[i] * vt[j];
        }
        /* o_t = q_t S_t, written back at the token's spatial position */
        double *ot = out + idx4(b, t, h, 0, T, H, Dv);
        for (long j = 0; j < Dv; ++j) {
            double acc = 0.0;
            for (long i = 0; i < Dk; ++i) acc += qt[i] * S[i * Dv + j];
            ot[j] = acc;
        }
    }
    if (final_state) {
        double *fs = final_state + ((b * H + h) * Dk) * Dv;
        memcpy(fs, S, sizeof(double) * (size_t)(Dk * Dv));
    }
}

/* Chunkwise schedule of the same recurrence, Sec. 3.3 / Eq. (chunk_boundary_main).
 * For chunk c holding scan positions [c*C, c*C + Cc), Cc <= C:
 *   A_{c,r}  = sum_{m<=r} g_{c,m}                          (cumulative log-decay)
 *   o_{c,r}  = (q_{c,r} . exp(A_{c,r})) S_[c]
 *              + sum_{j<=r} [sum_i q_{c,r,i} k_{c,j,i} exp(A_{c,r,i} - A_{c,j,i})] v_{c,j}
 *   khat_{c,r} = k_{c,r} . exp(A_{c,Cc-1} - A_{c,r}),  U_c = sum_r khat_{c,r}^T v_{c,r}
 *   d_c      = exp(A_{c,Cc-1}),  S_[c+1] = Diag(d_c) S_[c] + U_c
 * The paper writes the intra-chunk weight as qtilde ktilde^T with
 * qtilde = q exp(A), ktilde = k exp(-A); the product of the two exponentials is
 * evaluated here as the single exponential of the difference A_r - A_j, which
 * is the same number and stays finite when exp(-A) alone would overflow. */
static void chunkwise_one(const double *q, const double *k, const double *v, const double *g,
                          long b, long h, long H, long grid_h, long grid_w, long Dk, long Dv,
                          int order, long C, double *out, double *final_state,
                          double *S, double *A, long *tok, double *U)
{
    long T = grid_h * grid_w;
    memset(S, 0, sizeof(double) * (size_t)(Dk * Dv));          /* S_[0] = 0 */
    for (long c0 = 0; c0 < T; c0 += C) {
        long Cc = (T - c0 < C) ? (T - c0) : C;
        for (long r = 0; r < Cc; ++r) tok[r] = gla_oracle_scan_token(order, grid_h, grid_w, c0 + r);
        /* A_{c,r} */
        for (long r = 0; r < Cc; ++r) {
            const double *gr = g + idx4(b, tok[r], h, 0, T, H, Dk);
            for (long i = 0; i < Dk; ++i)
                A[r * Dk + i] = gr[i] + (r > 0 ? A[(r - 1) * Dk + i] : 0.0);
        }
        /* chunk outputs from the boundary state S_[c] */
        for (long r = 0; r < Cc; ++r) {
            const double *qr = q + idx4(b, tok[r], h, 0, T, H, Dk);
            double *orow = out + idx4(b, tok[r], h, 0, T, H, Dv);
            for (long jv = 0; jv < Dv; ++jv) {
                double acc = 0.0;
                for (long i = 0; i < Dk; ++i) acc += qr[i] * exp(A[r * Dk + i]) * S[i * Dv + jv];
                orow[jv] = acc;
            }
            for (long j = 0; j <= r; ++j) {
                const double *kj = k + idx4(b, tok[j], h, 0, T, H, Dk);
                const double *vj = v + idx4(b, tok[j], h, 0, T, H, Dv);
                double w = 0.0;
                for (long i = 0; i < Dk; ++i) w += qr[i] * kj[i] * exp(A[r * Dk + i] - A[j * Dk + i]);
                for (long jv = 0; jv < Dv; ++jv) orow[jv] += w * vj[jv];
            }
        }
        /* chunk summary U_c and decay d_c, then the boundary-state update */
        memset(U, 0, sizeof(double) * (size_t)(Dk * Dv));
        for (long r = 0; r < Cc; ++r) {
            const double *kr = k + idx4(b, tok[r], h, 0, T, H, Dk);
            const double *vr = v + idx4(b, tok[r], h, 0, T, H, Dv);
            for (long i = 0; i < Dk; ++i) {
                double khat = kr[i] * exp(A[(Cc - 1) * Dk + i] - A[r * Dk + i]);
                for (long jv = 0; jv < Dv; ++jv) U[i * Dv + jv] += khat * vr[jv];
            }
        }
        for (long i = 0; i < Dk; ++i) {
            double d = exp(A[(Cc - 1) * Dk + i]);
            for (long jv = 0; jv < Dv; ++jv) S[i * Dv + jv] = d * S[i * Dv + jv] + U[i * Dv + jv];
        }
    }
    if (final_state) {
        double *fs = final_state + ((b * H + h) * Dk) * Dv;
        memcpy(fs, S, sizeof(double) * (size_t)(Dk * Dv));
    }
}

static int set_threads(int n_threads)
{
#ifdef _OPENMP
    if (n_threads > 0) return n_threads;
    return omp_get_max_threads();
#else
    (void)n_threads;
    return 1;
#endif
}

/* Token recurrence over a set of (b, h) pairs (all pairs when pair_b == NULL).
 * Pairs are independent; they are spread over n_threads OpenMP threads
 * (n_threads <= 0: the OpenMP default).  Returns 0 on success. */
int gla_oracle_recurrence(const double *q, const double *k, const double *v, const double *g,
                          int B, int H, int grid_h, int grid_w, int Dk, int Dv, int order,
                          const int *pair_b, const int *pair_h, int n_pairs,
                          double *out, double *final_state, int n_threads)
{
    if (check_args(B, H, grid_h, grid_w, Dk, Dv, order)) return 1;
    long npairs = pair_b ? n_pairs : (long)B * H;
    int nt = set_threads(n_threads);
    int fail = 0;
#pragma omp parallel num_threads(nt)
    {
        double *S = (double *)malloc(sizeof(double) * (size_t)Dk * (size_t)Dv);
        if (!S) {
#pragma omp atomic write
            fail = 1;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (long p = 0; p < npairs; ++p) {
                long b = pair_b ? pair_b[p] : p / H;
                long h = pair_b ? pair_h[p] : p % H;
                recurrence_one(q, k, v, g, b, h, B, H, grid_h, grid_w, Dk, Dv, order, out,
                               final_state, S);
            }
            free(S);
        }
    }
    return fail ? 2 : 0;
}

/* Chunkwise schedule (chunk size C >= 1) over all (b, h) pairs. */
int gla_oracle_chunkwise(const double *q, const double *k, const double *v, const double *g,
                         int B, int H, int grid_h, int grid_w, int Dk, int Dv, int order,
                         int C, double *out, double *final_state, int n_threads)
{
    if (check_args(B, H, grid_h, grid_w, Dk, Dv, order) || C < 1) return 1;
    long npairs = (long)B * H;
    int nt = set_threads(n_threads);
    int fail = 0;
#pragma omp parallel num_threads(nt)
    {
        double *S = (double *)malloc(sizeof(double) * (size_t)Dk * (size_t)Dv);
        double *U = (double *)malloc(sizeof(double) * (size_t)Dk * (size_t)Dv);
        double *A = (double *)malloc(sizeof(double) * (size_t)C * (size_t)Dk);
        long *tok = (long *)malloc(sizeof(long) * (size_t)C);
        if (!S || !U || !A || !tok) {
#pragma omp atomic write
            fail = 1;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (long p = 0; p < npairs; ++p)
                chunkwise_one(q, k, v, g, p / H, p % H, H, grid_h, grid_w, Dk, Dv, order, C,
                              out, final_state, S, A, tok, U);
        }
        free(S); free(U); free(A); free(tok);
    }
    return fail ? 2 : 0;
}

/* Number of OpenMP threads a call with n_threads <= 0 would use. */
int gla_oracle_max_threads(void) { return set_threads(0); }
