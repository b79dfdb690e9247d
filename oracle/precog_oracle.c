/*
 * PRECOG oracle: a plain, slow, sequential fp64 CPU implementation of the
 * hot path (corpus-chunk scan with final-state capture, readout, and exact
 * top-1 dot-product retrieval).
 *
 * TEST INFRASTRUCTURE ONLY. Nothing on the product path links, loads or
 * calls this file: only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg use it. It shares no code, header or constant with the
 * CUDA library.
 *
 * Every value is double precision. Inputs arrive already widened to double
 * (bf16/fp16/fp32 -> double is exact), so the oracle sees exactly the values
 * the GPU sees. Build with -ffp-contract=off so that results do not depend on
 * whether the compiler fuses multiply-adds.
 *
 * Notation follows the paper (Sec. 3, Eq. 1; Appendix A):
 *   per channel d and state index n,
 *     alpha_t[d,n] = exp(dt_t[d] * A[d,n])          (A[d,n] < 0, so |alpha| < 1)
 *     beta_t[d,n]  = B_t[n] * x_t[d] * dt_t[d]
 *     h_t[d,n]     = h_{t-1}[d,n] * alpha_t[d,n] + beta_t[d,n]
 *     y_t[d]       = sum_n C_t[n] * h_t[d,n]        (readout of the updated state)
 *   Reading of the exponent sign: Eq. 1 prints exp(-dt*A) with a negative
 *   real part for A, which would make |alpha| > 1 and contradict the
 *   stability premise |alpha(x)| < 1 of Appendix B.1; the oracle takes
 *   alpha = exp(dt*A) with A < 0 (equivalently exp(-dt*a) with rate a > 0).
 */
#include <complex.h>
#include <math.h>
#include <stddef.h>
#include <stdint.h>

/* Status codes returned by the oracle entry points. */
#define ORACLE_OK 0
#define ORACLE_BAD_ARG 1

/*
 * oracle_scan: roll the selective-SSM recurrence (Eq. 1) over every chunk of
 * one layer, from h0 (or from the zero state, Appendix B.1), and capture the
 * final state of each chunk (Sec. 4.2, offline indexing).
 *
 *   D, N        channels and state size
 *   n_chunks    number of chunks; chunk c owns rows offsets[c] .. offsets[c+1]-1
 *   offsets     [n_chunks+1], non-decreasing, offsets[0] >= 0
 *   x, dt       [T_tot][D] token-major (row = token)
 *   A           [D][N]
 *   B, C        [T_tot][N]; C may be NULL when y_out is NULL
 *   h0          [n_chunks][D][N] initial state per chunk, or NULL for zero
 *   states_out  [n_chunks][D][N] final state per chunk
 *   y_out       [T_tot][D] readout after each update, or NULL
 *
 * The rollout S(h, x_{1:T}) of Appendix A is applied token by token in the
 * order the chunk lists them; a zero-length chunk returns h0 unchanged.
 */
int oracle_scan(int64_t D, int64_t N, int64_t n_chunks, const int64_t *offsets,
                const double *x, const double *dt, const double *A,
                const double *B, const double *C, const double *h0,
                double *states_out, double *y_out)
{
    if (D <= 0 || N <= 0 || n_chunks < 0 || offsets == NULL || states_out == NULL)
        return ORACLE_BAD_ARG;
    if (y_out != NULL && C == NULL)
        return ORACLE_BAD_ARG;
    if (offsets[0] < 0)
        return ORACLE_BAD_ARG;
    for (int64_t c = 0; c < n_chunks; ++c)
        if (offsets[c + 1] < offsets[c])
            return ORACLE_BAD_ARG;

    for (int64_t c = 0; c < n_chunks; ++c) {
        for (int64_t d = 0; d < D; ++d) {
            double *h = states_out + (c * D + d) * N;
            for (int64_t n = 0; n < N; ++n)
                h[n] = (h0 != NULL) ? h0[(c * D + d) * N + n] : 0.0;

            for (int64_t t = offsets[c]; t < offsets[c + 1]; ++t) {
                const double dt_td = dt[t * D + d];
                const double x_td = x[t * D + d];
                for (int64_t n = 0; n < N; ++n) {
                    const double alpha = exp(dt_td * A[d * N + n]);
                    const double beta = B[t * N + n] * x_td * dt_td;
                    h[n] = h[n] * alpha + beta;
                }
                if (y_out != NULL) {
                    double y = 0.0;
                    for (int64_t n = 0; n < N; ++n)
                        y += C[t * N + n] * h[n];
                    y_out[t * D + d] = y;
                }
            }
        }
    }
    return ORACLE_OK;
}

/*
 * oracle_retrieve: exact top-1 retrieval by dot product (Sec. 4.2, query-time
 * injection: the best-matching chunk key for the query embedding; with
 * unit-norm keys and queries the dot product is the cosine similarity).
 *
 *   index    [M][dim] keys, queries [Q][dim]
 *   best_idx [Q]  row of the highest score; the lowest row wins ties because
 *                 only a strictly greater score replaces the current best;
 *                 a NaN score never compares greater, so it never wins; -1 if
 *                 no row has a comparable score (M == 0 or all NaN)
 *   best_score [Q] that score in double, NaN when best_idx is -1
 */
int oracle_retrieve(int64_t M, int64_t dim, const double *index, int64_t Q,
                    const double *queries, int64_t *best_idx, double *best_score)
{
    if (M < 0 || dim <= 0 || Q < 0 || best_idx == NULL || best_score == NULL)
        return ORACLE_BAD_ARG;
    if ((M > 0 && index == NULL) || (Q > 0 && queries == NULL))
        return ORACLE_BAD_ARG;

    for (int64_t q = 0; q < Q; ++q) {
        double best = -INFINITY;
        int64_t arg = -1;
        for (int64_t i = 0; i < M; ++i) {
            double s = 0.0;
            for (int64_t k = 0; k < dim; ++k)
                s += queries[q * dim + k] * index[i * dim + k];
            if (s > best) {
                best = s;
                arg = i;
            }
        }
        best_idx[q] = arg;
        best_score[q] = (arg < 0) ? NAN : best;
    }
    return ORACLE_OK;
}

/*
 * oracle_scores: every dot product <query_q, key_i> in double (Sec. 4.2;
 * the scores that top-1 and top-k retrieval rank).
 *   scores [Q][M]
 */
int oracle_scores(int64_t M, int64_t dim, const double *index, int64_t Q,
                  const double *queries, double *scores)
{
    if (M < 0 || dim <= 0 || Q < 0 || scores == NULL)
        return ORACLE_BAD_ARG;
    for (int64_t q = 0; q < Q; ++q)
        for (int64_t i = 0; i < M; ++i) {
            double s = 0.0;
            for (int64_t k = 0; k < dim; ++k)
                s += queries[q * dim + k] * index[i * dim + k];
            scores[q * M + i] = s;
        }
    return ORACLE_OK;
}

/*
 * oracle_trajectory: the K-dial trajectory of Sec. 5.2 (Eq. smc-trajectory):
 * roll each chunk from the zero state as oracle_scan does and keep the state
 * after every stride-th token, plus the final state when the chunk length is
 * not a multiple of stride. Chunk c keeps K_c = ceil(len_c / stride) states
 * (K = N_c / k in the paper's notation; stride >= len_c keeps only the final
 * state, the per-chunk PRECOG state).
 *   entry_offsets [n_chunks+1]  prefix sums of K_c
 *   traj_out      [entry_offsets[n_chunks]][D][N]; entry entry_offsets[c] + j
 *                 is the state after token min((j+1)*stride, len_c) of chunk c
 */
int oracle_trajectory(int64_t D, int64_t N, int64_t n_chunks, const int64_t *offsets,
                      const double *x, const double *dt, const double *A, const double *B,
                      int64_t stride, const int64_t *entry_offsets, double *traj_out)
{
    if (D <= 0 || N <= 0 || n_chunks < 0 || stride < 1 || offsets == NULL ||
        entry_offsets == NULL || traj_out == NULL)
        return ORACLE_BAD_ARG;
    for (int64_t c = 0; c < n_chunks; ++c) {
        const int64_t len = offsets[c + 1] - offsets[c];
        if (len < 0 || entry_offsets[c + 1] - entry_offsets[c] != (len + stride - 1) / stride)
            return ORACLE_BAD_ARG;
    }
    if (N > 64)
        return ORACLE_BAD_ARG;
    for (int64_t c = 0; c < n_chunks; ++c) {
        for (int64_t d = 0; d < D; ++d) {
            double h[64];
            for (int64_t n = 0; n < N; ++n)
                h[n] = 0.0;
            int64_t j = 0;
            for (int64_t t = offsets[c]; t < offsets[c + 1]; ++t) {
                const double dt_td = dt[t * D + d];
                const double x_td = x[t * D + d];
                for (int64_t n = 0; n < N; ++n) {
                    const double alpha = exp(dt_td * A[d * N + n]);
                    const double beta = B[t * N + n] * x_td * dt_td;
                    h[n] = h[n] * alpha + beta;
                }
                const int64_t step = t - offsets[c] + 1;
                if (step % stride == 0 || t + 1 == offsets[c + 1]) {
                    double *e = traj_out + ((entry_offsets[c] + j) * D + d) * N;
                    for (int64_t n = 0; n < N; ++n)
                        e[n] = h[n];
                    ++j;
                }
            }
        }
    }
    return ORACLE_OK;
}

/*
 * oracle_scan_complex: Eq. 1 with the complex diagonal A the paper prints
 * (A_k = -softplus(a_k) + i*pi*k, Sec. 3) and a complex state h in C^N:
 *   alpha = exp(dt * A[d,n])  (complex),   beta = B[t,n] * x[t,d] * dt[t,d]  (real)
 *   h[d,n] = h[d,n] * alpha + beta,        y[t,d] = Re(sum_n C[t,n] * h[d,n])
 * Reading: B and C stay real per (token, state index) as in the real scan, and
 * the readout is the real part. A_re, A_im [D][N]; h0 and states_out are
 * [n_chunks][D][N] double complex (re, im interleaved); h0 may be NULL.
 */
int oracle_scan_complex(int64_t D, int64_t N, int64_t n_chunks, const int64_t *offsets,
                        const double *x, const double *dt, const double *A_re, const double *A_im,
                        const double *B, const double *C, const double complex *h0,
                        double complex *states_out, double *y_out)
{
    if (D <= 0 || N <= 0 || n_chunks < 0 || offsets == NULL || states_out == NULL)
        return ORACLE_BAD_ARG;
    if (y_out != NULL && C == NULL)
        return ORACLE_BAD_ARG;
    for (int64_t c = 0; c < n_chunks; ++c)
        if (offsets[c] < 0 || offsets[c + 1] < offsets[c])
            return ORACLE_BAD_ARG;
    for (int64_t c = 0; c < n_chunks; ++c) {
        for (int64_t d = 0; d < D; ++d) {
            double complex *h = states_out + (c * D + d) * N;
            for (int64_t n = 0; n < N; ++n)
                h[n] = (h0 != NULL) ? h0[(c * D + d) * N + n] : 0.0;
            for (int64_t t = offsets[c]; t < offsets[c + 1]; ++t) {
                const double dt_td = dt[t * D + d];
                const double x_td = x[t * D + d];
                for (int64_t n = 0; n < N; ++n) {
                    const double complex a = A_re[d * N + n] + I * A_im[d * N + n];
                    const double complex alpha = cexp(dt_td * a);
                    const double beta = B[t * N + n] * x_td * dt_td;
                    h[n] = h[n] * alpha + beta;
                }
                if (y_out != NULL) {
                    double y = 0.0;
                    for (int64_t n = 0; n < N; ++n)
                        y += C[t * N + n] * creal(h[n]);
                    y_out[t * D + d] = y;
                }
            }
        }
    }
    return ORACLE_OK;
}

