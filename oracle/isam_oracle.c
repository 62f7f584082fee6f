/*
 * isam_oracle.c -- plain, slow, fp64 CPU oracle for the matrix-multiplication
 * hot path of "ISA Mapper: A Compute and Hardware Agnostic Deep Learning
 * Compiler" (Sotoudeh et al., SysML 2019).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library's product path may link,
 * load or call this file; only the tests, the smoke check and the benchmark's
 * CPU-baseline leg do.  It shares no code, header or constant with the CUDA
 * path.
 *
 * Conventions
 *   - bf16 operands arrive as their uint16 bit patterns and are widened
 *     exactly to double (the pattern is the top half of an IEEE float32).
 *   - fp32 operands are widened exactly to double.
 *   - All arithmetic is double precision, each sum taken in increasing order of
 *     its reduction index; the file is compiled with -ffp-contract=off so the
 *     compiler fuses nothing.
 *   - Matrices are row-major and packed.
 *   - Parallelism (OpenMP) is only over independent output elements; it never
 *     changes an output's arithmetic.
 *
 * Return value of every entry: 0 on success, 1 on an invalid argument.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static double bf(uint16_t bits) {
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/*
 * GEMM, Listing 1 (the matmul loop nest) and Listing 4 (its three-operand
 * form: tmp := A[i][k]; tmp *= B[k][j]; C[i][j] += tmp):
 *
 *   C_out[i][j] = alpha * sum_{k=0..K-1} opA[i][k] * opB[k][j] + beta * C_in[i][j]
 *
 * opA[i][k] = A[i*K + k] (transA = 0, A stored M x K) or A[k*M + i] (transA = 1).
 * opB[k][j] = B[k*N + j] (transB = 0, B stored K x N) or B[j*K + k] (transB = 1).
 * With beta == 0 C_in is not read (BLAS convention) and may be NULL.
 *
 * rows / nrows select which rows i of C to compute (rows == NULL: all M rows,
 * in order).  C_out has nrows x N entries (row r of C_out is row rows[r]).
 */
int oracle_gemm_rows(int M, int N, int K, int transA, int transB, double alpha,
                     const uint16_t *A, const uint16_t *B, double beta,
                     const float *C_in, int nrows, const int *rows, double *C_out) {
    if (M < 1 || N < 1 || K < 1 || !A || !B || !C_out) return 1;
    if (beta != 0.0 && !C_in) return 1;
    if (!rows) nrows = M;
    for (int r = 0; rows && r < nrows; ++r)
        if (rows[r] < 0 || rows[r] >= M) return 1;

#pragma omp parallel
    {
        double *acc = (double *)malloc(sizeof(double) * (size_t)N);
#pragma omp for schedule(dynamic, 1)
        for (int r = 0; r < nrows; ++r) {
            const int i = rows ? rows[r] : r;
            for (int j = 0; j < N; ++j) acc[j] = 0.0;
            for (int k = 0; k < K; ++k) {
                const double a = transA ? bf(A[(size_t)k * M + i]) : bf(A[(size_t)i * K + k]);
                if (transB) {
                    for (int j = 0; j < N; ++j) acc[j] += a * bf(B[(size_t)j * K + k]);
                } else {
                    const uint16_t *brow = B + (size_t)k * N;
                    for (int j = 0; j < N; ++j) acc[j] += a * bf(brow[j]);
                }
            }
            double *out = C_out + (size_t)r * N;
            for (int j = 0; j < N; ++j) {
                double v = alpha * acc[j];
                if (beta != 0.0) v += beta * (double)C_in[(size_t)i * N + j];
                out[j] = v;
            }
        }
        free(acc);
    }
    return 0;
}

/*
 * OCP FP8 E4M3 byte -> double, exactly: sign s, 4 exponent bits e (bias 7), 3
 * mantissa bits m.  e > 0: (-1)^s 2^(e-7) (1 + m/8); e == 0: (-1)^s 2^-6 (m/8);
 * e == 15 with m == 7 is NaN (the format has no infinities).
 */
double oracle_e4m3(uint8_t byte) {
    const int s = byte >> 7, e = (byte >> 3) & 15, m = byte & 7;
    double v;
    if (e == 15 && m == 7)
        v = NAN;
    else if (e == 0)
        v = ldexp((double)m / 8.0, -6);
    else
        v = ldexp(1.0 + (double)m / 8.0, e - 7);
    return s ? -v : v;
}

/*
 * C_out = alpha * A B^T + beta * C_in with A (M x K) and B (N x K) stored as
 * E4M3 bytes, row-major: the GEMM of Listing 1 on 8-bit operands, each dot
 * product summed in increasing k in double precision.
 */
int oracle_gemm_fp8(int M, int N, int K, double alpha, const uint8_t *A, const uint8_t *B, double beta,
                    const float *C_in, double *C_out) {
    if (M < 1 || N < 1 || K < 1 || !A || !B || !C_out) return 1;
    if (beta != 0.0 && !C_in) return 1;
#pragma omp parallel for schedule(dynamic, 1)
    for (int i = 0; i < M; ++i) {
        for (int j = 0; j < N; ++j) {
            double acc = 0.0;
            for (int k = 0; k < K; ++k)
                acc += oracle_e4m3(A[(size_t)i * K + k]) * oracle_e4m3(B[(size_t)j * K + k]);
            double v = alpha * acc;
            if (beta != 0.0) v += beta * (double)C_in[(size_t)i * N + j];
            C_out[(size_t)i * N + j] = v;
        }
    }
    return 0;
}

/*
 * OCP Microscaling (MX) shared scale byte, E8M0: the value 2^(e - 127) for e
 * in 0..254; e == 255 is NaN.  No sign, no mantissa.
 */
double oracle_e8m0(uint8_t e) {
    if (e == 255) return NAN;
    return ldexp(1.0, (int)e - 127);
}

/*
 * Block-scaled E4M3 GEMM (OCP MX, MXFP8): each run of 32 consecutive K
 * elements of a row of A, and of a row of B (stored N x K), shares one E8M0
 * scale, so element k of row i of A stands for SA[i][k / 32] * A[i][k]:
 *
 *   C_out[i][j] = alpha * sum_k (SA[i][k/32] A[i][k]) (SB[j][k/32] B[j][k])
 *                 + beta * C_in[i][j]
 *
 * SA is M x ceil(K / 32) and SB N x ceil(K / 32) scale bytes, row-major; a
 * last block shorter than 32 (K not a multiple of 32) has a scale of its
 * own.  Each dot product is summed in increasing k in double precision (every
 * product is exact there: a power-of-two scale times an E4M3 value).
 */
int oracle_gemm_mxfp8(int M, int N, int K, double alpha, const uint8_t *A, const uint8_t *SA,
                      const uint8_t *B, const uint8_t *SB, double beta, const float *C_in, double *C_out) {
    if (M < 1 || N < 1 || K < 1 || !A || !SA || !B || !SB || !C_out) return 1;
    if (beta != 0.0 && !C_in) return 1;
    const int KB = (K + 31) / 32;
#pragma omp parallel for schedule(dynamic, 1)
    for (int i = 0; i < M; ++i) {
        for (int j = 0; j < N; ++j) {
            double acc = 0.0;
            for (int k = 0; k < K; ++k) {
                const double a = oracle_e8m0(SA[(size_t)i * KB + k / 32]) * oracle_e4m3(A[(size_t)i * K + k]);
                const double bv = oracle_e8m0(SB[(size_t)j * KB + k / 32]) * oracle_e4m3(B[(size_t)j * K + k]);
                acc += a * bv;
            }
            double v = alpha * acc;
            if (beta != 0.0) v += beta * (double)C_in[(size_t)i * N + j];
            C_out[(size_t)i * N + j] = v;
        }
    }
    return 0;
}

int oracle_gemm(int M, int N, int K, int transA, int transB, double alpha,
                const uint16_t *A, const uint16_t *B, double beta,
                const float *C_in, double *C_out) {
    return oracle_gemm_rows(M, N, K, transA, transB, alpha, A, B, beta, C_in,
                            M, NULL, C_out);
}

static double sigmoid(double v) { return 1.0 / (1.0 + exp(-v)); }

/*
 * GRU forward over T steps (Section 3.6, recurrent scheduling; Section 5.1.2,
 * a GRU over 128 steps).  The paper names the cell but not its equations; this
 * is the gate-order (r, z, n) form whose recurrent product is one fused
 * 3H-wide matrix product per step, with the reset gate applied after that
 * product:
 *
 *   gx = W x_t + b_ih                    (3H; rows r | z | n)
 *   gh = U h_{t-1} + b_hh                (3H)
 *   r  = sigmoid(gx_r + gh_r)
 *   z  = sigmoid(gx_z + gh_z)
 *   n  = tanh(gx_n + r * gh_n)
 *   h_t = (1 - z) * n + z * h_{t-1}
 *
 * x [T][batch][H] bf16, W and U [3H][H] bf16 (row = output unit, col = input),
 * b [6H] fp32 = b_ih then b_hh, h0 [batch][H] fp32 or NULL (zeros),
 * h_out [T][batch][H] double (every step's hidden state).
 * Sequences in a batch are independent; the loop over them is parallel.
 */
int oracle_gru_forward(int T, int batch, int H, const uint16_t *x, const uint16_t *W,
                       const uint16_t *U, const float *b, const float *h0, double *h_out) {
    if (T < 1 || batch < 1 || H < 1 || !x || !W || !U || !b || !h_out) return 1;
    const int G = 3 * H;
#pragma omp parallel
    {
        double *h = (double *)malloc(sizeof(double) * (size_t)H);
        double *hn = (double *)malloc(sizeof(double) * (size_t)H);
        double *gx = (double *)malloc(sizeof(double) * (size_t)G);
        double *gh = (double *)malloc(sizeof(double) * (size_t)G);
#pragma omp for schedule(dynamic, 1)
        for (int s = 0; s < batch; ++s) {
            for (int j = 0; j < H; ++j) h[j] = h0 ? (double)h0[(size_t)s * H + j] : 0.0;
            for (int t = 0; t < T; ++t) {
                const uint16_t *xt = x + ((size_t)t * batch + s) * H;
                for (int g = 0; g < G; ++g) {
                    double ax = 0.0, ah = 0.0;
                    const uint16_t *wr = W + (size_t)g * H;
                    const uint16_t *ur = U + (size_t)g * H;
                    for (int k = 0; k < H; ++k) ax += bf(wr[k]) * bf(xt[k]);
                    for (int k = 0; k < H; ++k) ah += bf(ur[k]) * h[k];
                    gx[g] = ax + (double)b[g];
                    gh[g] = ah + (double)b[G + g];
                }
                double *ho = h_out + ((size_t)t * batch + s) * H;
                for (int j = 0; j < H; ++j) {
                    const double r = sigmoid(gx[j] + gh[j]);
                    const double z = sigmoid(gx[H + j] + gh[H + j]);
                    const double n = tanh(gx[2 * H + j] + r * gh[2 * H + j]);
                    hn[j] = (1.0 - z) * n + z * h[j];
                    ho[j] = hn[j];
                }
                double *tmp = h; h = hn; hn = tmp;
            }
        }
        free(h); free(hn); free(gx); free(gh);
    }
    return 0;
}

/*
 * The GRU with the reset gate applied before the candidate's recurrent
 * product (the cell's original form): the candidate sees U_n (r * h_{t-1}),
 * so r must be known for every unit before that product:
 *
 *   r  = sigmoid(W_r x_t + b_ir + U_r h_{t-1} + b_hr)
 *   z  = sigmoid(W_z x_t + b_iz + U_z h_{t-1} + b_hz)
 *   n  = tanh(W_n x_t + b_in + U_n (r * h_{t-1}) + b_hn)
 *   h_t = (1 - z) * n + z * h_{t-1}
 *
 * Same arguments and layouts as oracle_gru_forward.
 */
int oracle_gru_forward_reset_before(int T, int batch, int H, const uint16_t *x, const uint16_t *W,
                                    const uint16_t *U, const float *b, const float *h0, double *h_out) {
    if (T < 1 || batch < 1 || H < 1 || !x || !W || !U || !b || !h_out) return 1;
    const int G = 3 * H;
#pragma omp parallel
    {
        double *h = (double *)malloc(sizeof(double) * (size_t)H);
        double *rh = (double *)malloc(sizeof(double) * (size_t)H);
        double *z = (double *)malloc(sizeof(double) * (size_t)H);
        double *gx = (double *)malloc(sizeof(double) * (size_t)G);
#pragma omp for schedule(dynamic, 1)
        for (int s = 0; s < batch; ++s) {
            for (int j = 0; j < H; ++j) h[j] = h0 ? (double)h0[(size_t)s * H + j] : 0.0;
            for (int t = 0; t < T; ++t) {
                const uint16_t *xt = x + ((size_t)t * batch + s) * H;
                for (int g = 0; g < G; ++g) {
                    double ax = 0.0;
                    const uint16_t *wr = W + (size_t)g * H;
                    for (int k = 0; k < H; ++k) ax += bf(wr[k]) * bf(xt[k]);
                    gx[g] = ax + (double)b[g];
                }
                for (int j = 0; j < H; ++j) {  /* r and z from h_{t-1} */
                    double ar = 0.0, az = 0.0;
                    const uint16_t *ur = U + (size_t)j * H, *uz = U + (size_t)(H + j) * H;
                    for (int k = 0; k < H; ++k) {
                        ar += bf(ur[k]) * h[k];
                        az += bf(uz[k]) * h[k];
                    }
                    const double r = sigmoid(gx[j] + ar + (double)b[G + j]);
                    z[j] = sigmoid(gx[H + j] + az + (double)b[G + H + j]);
                    rh[j] = r * h[j];
                }
                double *ho = h_out + ((size_t)t * batch + s) * H;
                for (int j = 0; j < H; ++j) {  /* candidate from r * h_{t-1} */
                    double an = 0.0;
                    const uint16_t *un = U + (size_t)(2 * H + j) * H;
                    for (int k = 0; k < H; ++k) an += bf(un[k]) * rh[k];
                    const double n = tanh(gx[2 * H + j] + an + (double)b[G + 2 * H + j]);
                    ho[j] = (1.0 - z[j]) * n + z[j] * h[j];
                }
                for (int j = 0; j < H; ++j) h[j] = ho[j];
            }
        }
        free(h); free(rh); free(z); free(gx);
    }
    return 0;
}

/*
 * One GRU layer over one sequence s, for the stacked form below: the input
 * at step t is either bf16 (x16, the first layer) or double (x64, the hidden
 * states of the layer underneath, taken unrounded).  Gate order r, z, n;
 * reset_before selects U_n (r * h_{t-1}) over r * (U_n h_{t-1} + b_hn) in the
 * candidate.  h_out row (t, s) receives h_t.
 */
static void gru_layer_sequence(int T, int batch, int H, int s, int reset_before,
                               const uint16_t *x16, const double *x64, const uint16_t *W,
                               const uint16_t *U, const float *b, const float *h0,
                               double *h_out, double *h, double *xin, double *gx, double *gh,
                               double *rh) {
    const int G = 3 * H;
    for (int j = 0; j < H; ++j) h[j] = h0 ? (double)h0[(size_t)s * H + j] : 0.0;
    for (int t = 0; t < T; ++t) {
        const size_t row = ((size_t)t * batch + s) * H;
        for (int k = 0; k < H; ++k) xin[k] = x16 ? bf(x16[row + k]) : x64[row + k];
        for (int g = 0; g < G; ++g) {  /* input projection, every gate */
            double a = 0.0;
            const uint16_t *wr = W + (size_t)g * H;
            for (int k = 0; k < H; ++k) a += bf(wr[k]) * xin[k];
            gx[g] = a + (double)b[g];
        }
        for (int g = 0; g < 2 * H; ++g) {  /* recurrent product of r and z */
            double a = 0.0;
            const uint16_t *ur = U + (size_t)g * H;
            for (int k = 0; k < H; ++k) a += bf(ur[k]) * h[k];
            gh[g] = a + (double)b[G + g];
        }
        for (int j = 0; j < H; ++j) {
            const double r = sigmoid(gx[j] + gh[j]);
            rh[j] = reset_before ? r * h[j] : h[j];
            gh[j] = r;  /* r kept for the reset-after candidate */
        }
        for (int j = 0; j < H; ++j) {  /* candidate's recurrent product */
            double a = 0.0;
            const uint16_t *un = U + (size_t)(2 * H + j) * H;
            for (int k = 0; k < H; ++k) a += bf(un[k]) * rh[k];
            gh[2 * H + j] = a + (double)b[G + 2 * H + j];
        }
        double *ho = h_out + row;
        for (int j = 0; j < H; ++j) {
            const double r = gh[j];
            const double z = sigmoid(gx[H + j] + gh[H + j]);
            const double n = reset_before ? tanh(gx[2 * H + j] + gh[2 * H + j])
                                          : tanh(gx[2 * H + j] + r * gh[2 * H + j]);
            ho[j] = (1.0 - z) * n + z * h[j];
        }
        for (int j = 0; j < H; ++j) h[j] = ho[j];
    }
}

/*
 * Stacked GRU: `layers` GRU layers of width H (Section 5.1.2's cell, gate
 * order r, z, n), layer 0 reading x and layer l > 0 reading the hidden
 * states h^{l-1}_t of the layer below at the same step, in double precision
 * (no rounding between layers).
 *
 * x [T][batch][H] bf16; W, U [layers][3H][H] bf16 (layer l's input and
 * recurrent weights); b [layers][6H] fp32 (b_ih | b_hh per layer);
 * h0 [layers][batch][H] fp32 or NULL (zeros); h_out [layers][T][batch][H]
 * double, every layer's states.  Returns 0, or 1 on an invalid argument.
 */
int oracle_gru_stack(int layers, int T, int batch, int H, int reset_before, const uint16_t *x,
                     const uint16_t *W, const uint16_t *U, const float *b, const float *h0,
                     double *h_out) {
    if (layers < 1 || T < 1 || batch < 1 || H < 1 || !x || !W || !U || !b || !h_out) return 1;
    const size_t wsz = (size_t)3 * H * H, seq = (size_t)T * batch * H;
    for (int l = 0; l < layers; ++l) {
        const uint16_t *x16 = l == 0 ? x : NULL;
        const double *x64 = l == 0 ? NULL : h_out + (size_t)(l - 1) * seq;
        const float *h0l = h0 ? h0 + (size_t)l * batch * H : NULL;
#pragma omp parallel
        {
            double *h = (double *)malloc(sizeof(double) * (size_t)H);
            double *xin = (double *)malloc(sizeof(double) * (size_t)H);
            double *rh = (double *)malloc(sizeof(double) * (size_t)H);
            double *gx = (double *)malloc(sizeof(double) * (size_t)3 * H);
            double *gh = (double *)malloc(sizeof(double) * (size_t)3 * H);
#pragma omp for schedule(dynamic, 1)
            for (int s = 0; s < batch; ++s)
                gru_layer_sequence(T, batch, H, s, reset_before, x16, x64, W + (size_t)l * wsz,
                                   U + (size_t)l * wsz, b + (size_t)l * 6 * H, h0l,
                                   h_out + (size_t)l * seq, h, xin, gx, gh, rh);
            free(h); free(xin); free(rh); free(gx); free(gh);
        }
    }
    return 0;
}

/*
 * Separable depthwise convolution, Listing 3, with stride s = 1, channel
 * multiplier c = 1 (so r = 0 and P is indexed P[q][k]) and a zero border of
 * one pixel (input row i + di - 1, column j + dj - 1), taken in the factored
 * form the paper's factorisation pass produces (Section 2.3): the
 * D-weighted window sum over (di, dj) is formed first, then multiplied by P
 * and summed over q:
 *
 *   Y[b][i][j][q] = sum_{di,dj in 0..2} X[b][i+di-1][j+dj-1][q] * D[di][dj][q]
 *   C[b][i][j][k] = sum_{q} Y[b][i][j][q] * P[q][k]
 *
 * x NHWC [N][H][W][Cin] bf16, dw [3][3][Cin] bf16, pw [Cin][Cout] bf16,
 * out NHWC [N][H][W][Cout] double.  No rounding between the two stages.
 */
int oracle_dwsep(int N, int H, int W, int Cin, int Cout, const uint16_t *x,
                 const uint16_t *dw, const uint16_t *pw, double *out) {
    if (N < 1 || H < 1 || W < 1 || Cin < 1 || Cout < 1 || !x || !dw || !pw || !out) return 1;
    const long npix = (long)N * H * W;
#pragma omp parallel
    {
        double *y = (double *)malloc(sizeof(double) * (size_t)Cin);
#pragma omp for schedule(static)
        for (long p = 0; p < npix; ++p) {
            const int b = (int)(p / ((long)H * W));
            const int i = (int)((p / W) % H);
            const int j = (int)(p % W);
            for (int q = 0; q < Cin; ++q) {
                double s = 0.0;
                for (int di = 0; di < 3; ++di) {
                    const int ii = i + di - 1;
                    if (ii < 0 || ii >= H) continue;
                    for (int dj = 0; dj < 3; ++dj) {
                        const int jj = j + dj - 1;
                        if (jj < 0 || jj >= W) continue;
                        s += bf(x[(((size_t)b * H + ii) * W + jj) * Cin + q]) *
                             bf(dw[((size_t)di * 3 + dj) * Cin + q]);
                    }
                }
                y[q] = s;
            }
            double *o = out + (size_t)p * Cout;
            for (int k = 0; k < Cout; ++k) {
                double s = 0.0;
                for (int q = 0; q < Cin; ++q) s += y[q] * bf(pw[(size_t)q * Cout + k]);
                o[k] = s;
            }
        }
        free(y);
    }
    return 0;
}
