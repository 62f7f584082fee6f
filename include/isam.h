/*
 * isam.h -- C ABI of the GB300 (sm_103a) matrix-multiplication hot path
 * extracted and scheduled by the ISA Mapper (Sotoudeh et al., "ISA Mapper: A
 * Compute and Hardware Agnostic Deep Learning Compiler", SysML 2019).
 *
 * Library: libisam.so.  Plain C types only: sizes are int, scalars float,
 * bf16 tensors are passed as pointers to their 16-bit patterns (isam_bf16,
 * IEEE bfloat16, round-to-nearest-even where the caller rounds).
 *
 * Memory and ownership
 *   - Every tensor pointer is a DEVICE pointer on the current CUDA device,
 *     allocated and owned by the caller.  The library never frees or keeps
 *     them past the call's completion on the stream.
 *   - Tensors are packed row-major (no leading-dimension arguments).
 *   - The library owns small internal workspaces (an error word per device,
 *     the GRU's input-projection buffer, its hidden-state exchange buffer and
 *     step counter).  They are allocated on first use, reused, and released
 *     by isam_shutdown().
 *
 * Execution
 *   - Every compute call is asynchronous on the stream set by
 *     isam_set_stream() (default: the legacy default stream) and returns
 *     after the launch.  Argument errors are reported at once and nothing is
 *     launched.  Device-side failures (a bounded wait that ran out) are
 *     reported by the next isam_sync().
 *   - Calls run on the caller's current device.  Workspaces, the error word
 *     and each kernel's dynamic shared-memory opt-in are kept per device (the
 *     opt-in belongs to each device's context), so one process may drive
 *     several GPUs; the stream given to isam_set_stream() must belong to the
 *     device that is current at each call.
 *   - Every spin-wait inside the kernels is bounded in time (default 2 s,
 *     ISAM_WAIT_TIMEOUT_MS in the environment overrides); a wait that runs out
 *     sets the device error word and the kernel returns.
 *
 * Status codes: every entry returns one of the ISAM_* codes below;
 * isam_last_error_string() describes the last failure on the calling thread.
 */
#ifndef ISAM_H
#define ISAM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t isam_bf16;

enum {
    ISAM_OK = 0,
    ISAM_ERR_INVALID_ARG = 1, /* null pointer, non-positive size, bad flag     */
    ISAM_ERR_UNSUPPORTED = 2, /* valid but outside the supported shapes/aligns */
    ISAM_ERR_CUDA = 3,        /* a CUDA runtime or driver call failed          */
    ISAM_ERR_TIMEOUT = 4      /* a bounded device wait ran out (see isam_sync) */
};

/* Version of this ABI (major * 100 + minor). */
int isam_version(void);

/* Stream for subsequent calls from any thread: a cudaStream_t passed as
 * void*, or NULL for the legacy default stream.  Returns ISAM_OK. */
int isam_set_stream(void *stream);

/* Waits for the stream, then reads and clears the device error word.
 * ISAM_OK, ISAM_ERR_TIMEOUT (a bounded wait ran out; outputs of the failed
 * call are undefined) or ISAM_ERR_CUDA. */
int isam_sync(void);

/* Human-readable description of the last failure on this thread. */
const char *isam_last_error_string(void);

/* Releases every internal workspace on every device it was made on.  Waits
 * for the device first.  Later calls allocate again. */
int isam_shutdown(void);

/*
 * GEMM: C <- alpha * op(A) * op(B) + beta * C
 *
 * The computation of Listing 1 (C[i][j] += A[i][k] * B[k][j]) and its
 * three-operand form in Listing 4, with BLAS scaling; the paper's GEMM
 * benchmark (Section 5.1.1) runs it at DeepBench sizes.
 *
 *   op(A) is M x K: A stored M x K when transA == 0, K x M when transA == 1.
 *   op(B) is K x N: B stored K x N when transB == 0, N x K when transB == 1.
 *   A, B: bf16, C: fp32 (M x N), all row-major packed, device pointers.
 *   Products are exact in fp32 and accumulated in fp32 (tensor cores).
 *   beta == 0: C is write-only (never read, NaNs in it do not propagate).
 *
 * Supported: M, N, K >= 1; A and B 16-byte aligned; every stored row pitch a
 * multiple of 16 bytes, i.e. K % 8 == 0 when transA == 0 or transB == 1,
 * M % 8 == 0 when transA == 1, N % 8 == 0 when transB == 0; C 16-byte
 * aligned.  Otherwise ISAM_ERR_UNSUPPORTED.
 * ISAM_ERR_INVALID_ARG for null pointers, sizes < 1, trans flags not 0/1.
 */
int isam_gemm(int M, int N, int K, int transA, int transB, float alpha,
              const isam_bf16 *A, const isam_bf16 *B, float beta, float *C);

/*
 * GEMM on 8-bit float operands: C <- alpha * A * B^T + beta * C with A (M x K)
 * and B (N x K) stored row-major as OCP FP8 E4M3 bytes (1 sign bit, 4
 * exponent bits with bias 7, 3 mantissa bits; 0x7F and 0xFF are NaN, no
 * infinities, largest finite 448), C fp32 M x N row-major.  Products are
 * exact and accumulate in fp32, as in isam_gemm; half the operand bytes of
 * the bf16 call, for the bandwidth-bound skinny shapes.  The paper's
 * instruction selection (Section 2.4) chooses among instructions a program
 * maps onto; this is the same matrix multiplication on the tensor cores'
 * 8-bit operand kind.
 *   - Both operands K-major (the only layout); K a multiple of 16 (16-byte
 *     rows); A, B, C 16-byte aligned.  Otherwise ISAM_ERR_UNSUPPORTED.
 *   - Sizes < 1 or null pointers: ISAM_ERR_INVALID_ARG.
 * Asynchronous on the stream set by isam_set_stream; beta = 0 does not read C.
 */
int isam_gemm_fp8(int M, int N, int K, float alpha, const uint8_t *A, const uint8_t *B, float beta,
                  float *C);

/*
 * Block-scaled E4M3 GEMM in the OCP Microscaling (MX) form: every 32
 * consecutive K elements of a row of A, and of a row of B, share one E8M0
 * scale byte e meaning 2^(e - 127) (e = 255 is NaN):
 *   C[i][j] <- alpha * sum_k (2^(sa(i,k)-127) A[i][k]) (2^(sb(j,k)-127) B[j][k])
 *              + beta * C[i][j],
 * sa(i, k), sb(j, k) the scale bytes of the 32-element K block holding k.
 * The paper's instruction selection (Section 2.4) picks the instruction whose
 * semantics cover the computation; here the tensor cores' block-scaled
 * operand kind applies the scales inside the product.
 *   A  M x K, B  N x K: E4M3 bytes, row-major (K-major), device pointers,
 *      16-byte aligned; K a multiple of 16 (16-byte rows).
 *   SA, SB: the E8M0 bytes, device pointers, 4-byte aligned, atom-major:
 *      for each 128-element K atom a (ceil(K/128) of them) and each row,
 *      four consecutive bytes, byte t the scale of K block 4a + t of that
 *      row: SA[((a * M) + i) * 4 + t] scales A[i][k] for k in
 *      [128a + 32t, 128a + 32t + 32), and SB likewise with N rows.  Bytes of
 *      blocks past ceil(K/32) are ignored.  A last block shorter than 32
 *      (K % 32 != 0) has a scale of its own.  (This layout puts the words one
 *      K atom needs for consecutive rows next to each other.)
 *   C  M x N fp32 row-major, 16-byte aligned; beta == 0 does not read C.
 * Products of the scaled operands are exact and accumulate in fp32.  One
 * persistent launch over 128 x min(128, N rounded up to 16) tiles (no
 * split-K); asynchronous on the stream set by isam_set_stream.
 * ISAM_ERR_INVALID_ARG for sizes < 1 or null pointers, ISAM_ERR_UNSUPPORTED
 * for misaligned pointers or K % 16 != 0.
 */
int isam_gemm_mxfp8(int M, int N, int K, float alpha, const uint8_t *A, const uint8_t *SA,
                    const uint8_t *B, const uint8_t *SB, float beta, float *C);

/*
 * isam_gemm_mxfp8 for 1 <= count <= 64 independent problems in one launch
 * (host arrays of count entries; the rules of isam_gemm_grouped: no C[i] may
 * overlap another problem's operands or result).  Errors name the problem.
 */
int isam_gemm_grouped_mxfp8(int count, const int *M, const int *N, const int *K, const float *alpha,
                            const uint8_t *const *A, const uint8_t *const *SA,
                            const uint8_t *const *B, const uint8_t *const *SB,
                            const float *beta, float *const *C);

/*
 * Several independent GEMMs in one launch: problem i computes
 * C[i] <- alpha[i] * op(A[i]) * op(B[i]) + beta[i] * C[i] exactly as isam_gemm
 * would, with the same per-problem argument rules.
 *
 * The tiles of all problems are scheduled across the GPU's SMs by one
 * persistent kernel (the paper's scheduler placing compute tiles across
 * compute units, Sections 3.3-3.4, over a set of matrix multiplications), so
 * the per-launch costs are paid once for the group.  Arrays M..C are HOST
 * arrays of count entries; A[i], B[i], C[i] are device pointers.
 *   - 1 <= count <= 64 (else ISAM_ERR_INVALID_ARG).
 *   - The problems run concurrently: no C[i] may overlap any A[j], B[j] or
 *     another C[j]; results are undefined otherwise.
 *   - Tile width is min(128, N rounded up to 16) per problem; no split-K.
 * Errors name the offending problem.
 */
int isam_gemm_grouped(int count, const int *M, const int *N, const int *K, const int *transA,
                      const int *transB, const float *alpha, const isam_bf16 *const *A,
                      const isam_bf16 *const *B, const float *beta, float *const *C);

/*
 * isam_gemm_grouped for E4M3 problems: problem i computes
 * C[i] <- alpha[i] * A[i] * B[i]^T + beta[i] * C[i] exactly as isam_gemm_fp8
 * would (A[i]: M[i] x K[i], B[i]: N[i] x K[i], E4M3 bytes, K-major), with the
 * same argument rules per problem and the same group rules as
 * isam_gemm_grouped (1 <= count <= 64, host arrays, no overlapping C).
 */
int isam_gemm_grouped_fp8(int count, const int *M, const int *N, const int *K, const float *alpha,
                          const uint8_t *const *A, const uint8_t *const *B, const float *beta,
                          float *const *C);

/*
 * The tile plan isam_gemm would use for this problem, chosen by the
 * library's analytic cost model (the paper's "Approach" interface for
 * tiling and device-allocation choices, Sections 3.4 and 4).  Nothing is
 * launched.  out (host, 6 ints): tile width BN (tile height is 128), split-K
 * factor (CTAs of one cluster sharing a tile), shared-memory ring depth,
 * rasterisation group height, persistent grid size, dynamic shared memory
 * bytes.  Same argument checks as isam_gemm (pointers are not needed).
 */
int isam_gemm_plan_info(int M, int N, int K, int transA, int transB, float beta, int *out);

/*
 * isam_gemm_plan_info with two more outputs (out: host, 8 ints): out[0..5]
 * as above, out[6] tile height (128, or 256 for a CTA-pair plan), out[7] CTAs
 * whose tensor cores issue one MMA together (1, or 2: the two CTAs of a
 * cluster each hold 128 rows of A and half the tile's columns of B, and one
 * of them issues M = 256 MMAs over both; the pair's tile is 256 x BN).
 */
int isam_gemm_plan_info2(int M, int N, int K, int transA, int transB, float beta, int *out);

/*
 * isam_gemm_plan_info2's plan for a device with num_sms SMs, smem_optin
 * bytes of opt-in shared memory per CTA and cluster_caps[3] clusters of 2, 4
 * and 8 CTAs resident at once (host array); host arithmetic only, no CUDA
 * call, so it runs without a GPU.  out: 8 ints as isam_gemm_plan_info2.
 * ISAM_ERR_INVALID_ARG for a null out or cluster_caps or limits < 1, and the
 * argument checks of isam_gemm.
 */
int isam_gemm_plan_for(int M, int N, int K, int transA, int transB, float beta, int num_sms, int smem_optin,
                       const int *cluster_caps, int *out);

/*
 * GRU forward inference over T steps (input size == hidden).
 *
 * The recurrent model the paper schedules with a priming, a recursive and a
 * finish iteration over persistent weights (Section 3.6) and benchmarks over
 * 128 steps (Section 5.1.2).  The paper names the cell without equations;
 * this library computes the (r, z, n) form with the reset gate applied after
 * the recurrent product:
 *
 *   gx = W x_t + b_ih,  gh = U h_{t-1} + b_hh        (3H each, rows r|z|n)
 *   r = sigmoid(gx_r + gh_r),  z = sigmoid(gx_z + gh_z)
 *   n = tanh(gx_n + r * gh_n),  h_t = (1 - z) * n + z * h_{t-1}
 *
 *   x     [T][batch][hidden] bf16
 *   W, U  [3*hidden][hidden] bf16 (row = output unit of gate r, z, then n)
 *   b     [6*hidden] fp32: b_ih (3*hidden) then b_hh (3*hidden)
 *   h0    [batch][hidden] fp32, or NULL for zeros
 *   h_out [T][batch][hidden] fp32: every step's hidden state (h_T = h_out[T-1])
 *
 * The input projection for all T steps runs as one GEMM into a library
 * workspace; the recurrence runs in one persistent kernel that keeps U
 * resident in shared memory and multiplies bf16(h_{t-1}) on the tensor cores
 * (h itself is carried in fp32).  Gates are evaluated in fp32.
 *
 * Supported: T >= 1, 1 <= batch <= 256, hidden a multiple of 32 in
 * [32, 1024]; all pointers 16-byte aligned.  Otherwise ISAM_ERR_UNSUPPORTED.
 * Batches above 32 run with the batch padded to 64 or 128 rows (the MMA's N;
 * 128 only with 4 K splits), in chunks of that many rows, one launch per
 * chunk; the rows are independent sequences.  The recurrence runs on
 * hidden / 32 clusters of K-split CTAs, launched only after the device
 * reports that every cluster fits at once (they must all be resident): 4 splits when hidden is a multiple of 256, 2 for the other
 * multiples of 128, otherwise 1 up to hidden 448, 2 up to 896 and 4 above.
 * Each CTA keeps a 96-row slice of U over ceil(atoms / splits) 64-wide K
 * atoms in shared memory; where the last CTA's range ends past the matrix (a
 * hidden of 64 j + 32, or atoms not divisible by the splits) the tensor maps
 * read zeros on both sides of the product.
 */
int isam_gru_forward(int T, int batch, int hidden, const isam_bf16 *x,
                     const isam_bf16 *W, const isam_bf16 *U, const float *b,
                     const float *h0, float *h_out);

/*
 * GRU forward with the reset gate applied before the candidate's recurrent
 * product (the cell's original form):
 *
 *   r = sigmoid(gx_r + U_r h_{t-1} + b_hr),  z = sigmoid(gx_z + U_z h_{t-1} + b_hz)
 *   n = tanh(gx_n + U_n (r * h_{t-1}) + b_hn),  h_t = (1 - z) * n + z * h_{t-1}
 *
 * (gx = W x_t + b_ih as in isam_gru_forward.)  Same arguments, layouts and
 * support limits as isam_gru_forward.  The recurrent product is no longer one
 * fused 3H-wide product per step: U_n needs r of every unit first, so each
 * step of the persistent kernel runs two rounds (r and z from h_{t-1}, a
 * grid-wide exchange of bf16(r * h_{t-1}), then the n rows), the recurrent
 * scheduling of Section 3.6 with an intra-step dependency.
 */
int isam_gru_forward_reset_before(int T, int batch, int hidden, const isam_bf16 *x,
                                  const isam_bf16 *W, const isam_bf16 *U, const float *b,
                                  const float *h0, float *h_out);

/*
 * Stacked GRU: `layers` GRU layers of width `hidden`, layer 0 reading x and
 * layer l > 0 reading the hidden states of layer l - 1 at the same step
 * (Section 5.1.2's cell, stacked; the recurrent scheduling of Section 3.6 per
 * layer).  reset_before = 0 gives isam_gru_forward's cell, 1 that of
 * isam_gru_forward_reset_before.
 *
 *   x      [T][batch][hidden]            bf16, layer 0's input
 *   W, U   [layers][3*hidden][hidden]    bf16, each layer's input and
 *                                        recurrent weights (r, z, n rows)
 *   b      [layers][6*hidden]            fp32, b_ih | b_hh per layer
 *   h0     [layers][batch][hidden]       fp32 or NULL (zeros)
 *   h_out  [layers][T][batch][hidden]    fp32, every layer's states; layer
 *                                        layers - 1 is the stack's output
 *
 With the reset gate after the product and hidden a multiple of 256, layers
 * run in pairs in one persistent kernel: in round r it advances the lower
 * layer to step r and the upper one to step r - 1, computing the upper
 * layer's input projection from the same bf16 tile of the lower layer's
 * states (T + 1 rounds for two layers); between pairs, and for an odd last
 * layer, the states below are rounded to bf16 and projected by the GEMM.
 * Otherwise (the reset-before form, other hidden sizes) layer l's kernel
 * keeps its K quarter of layer l + 1's W resident and multiplies it by the
 * bf16(h_{t-1}) tile it loads for its own recurrent product, so layer
 * l + 1's projection is computed while layer l runs (one extra round covers
 * h_{T-1}); layer l + 1 reads it as per-K-rank partial sums (fixed order:
 * deterministic).  Either way the next layer sees bf16(h^l_t), as the
 * recurrent product sees bf16(h_{t-1}).
 *
 * Supported: as isam_gru_forward (batch up to 256, every multiple of 32
 * for hidden; the K splits are chosen so that both weight slices of the
 * per-layer chain fit).  Batches above 32 run layer by layer: the states
 * below are rounded to bf16 and projected by the GEMM, and each layer's
 * recurrence runs in chunks of padded rows.  Workspace: 2 x ks x T x batch x
 * 3*hidden fp32 (ks = 4, 2 or 1 K splits) beside isam_gru_forward's.
 */
int isam_gru_forward_stack(int layers, int T, int batch, int hidden, int reset_before,
                           const isam_bf16 *x, const isam_bf16 *W, const isam_bf16 *U,
                           const float *b, const float *h0, float *h_out);

/*
 * GRU forward that allocates nothing.  The paper has no counterpart: this is a
 * deployment variant of isam_gru_forward for callers that cannot let a library
 * call cudaMalloc -- a process whose device memory is all reserved up front by
 * its framework's caching allocator (a raw cudaMalloc would fail or fragment
 * that pool), or a latency-bound request path that forbids cudaMalloc/cudaFree
 * because they can synchronise the whole device.
 *
 * Same arguments, layouts and equations as isam_gru_forward; batch up to 32
 * only (1 <= batch <= 32, hidden a multiple of 32 in [32, 1024], any
 * T >= 1).  The
 * caller still passes every input and h_out.  The workspaces live in one
 * static 8 MiB device array inside libisam.so, which every GPU that loads the
 * library holds until the process exits; the input projection is computed in
 * chunks of time steps that fit it (20 steps at batch 32, hidden 1024), with h
 * carried between chunks through h_out.  No cudaMalloc, cudaFree or other
 * allocating routine is called.
 *
 *   - The first call on a device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current.
 *   - Every call shares the one array: calls that overlap on the GPU (other
 *     streams, other host threads) race and corrupt each other.  The call
 *     clears the parts that must start at zero (error word, step counter).
 *   - Unlike the other calls it synchronises its stream before returning
 *     (it reads the device error word back on that stream, then waits for
 *     that stream alone), so that it can report a device-side timeout
 *     itself; it must therefore not be called while the stream is being
 *     captured into a CUDA graph.  Results:
 *     ISAM_OK, ISAM_ERR_TIMEOUT (h_out undefined), ISAM_ERR_CUDA,
 *     ISAM_ERR_INVALID_ARG or ISAM_ERR_UNSUPPORTED (sizes beyond the limits
 *     above, misaligned pointers, a device other than sm_103a).
 */
int isam_gru_forward_noalloc(int T, int batch, int hidden, const isam_bf16 *x,
                             const isam_bf16 *W, const isam_bf16 *U, const float *b,
                             const float *h0, float *h_out);

/*
 * Separable depthwise convolution, NHWC: a 3x3 depthwise stage (stride 1,
 * zero border of one pixel, channel multiplier 1) followed by a pointwise
 * 1x1 stage, i.e. Listing 3 with s = 1 and c = 1, executed in the factored
 * form of Section 2.3: the depthwise sum feeds a GEMM with
 * M = N*H*W, K = Cin, N = Cout.
 *
 *   x     [N][H][W][Cin] bf16
 *   dw_w  [3][3][Cin] bf16   (D[di][dj][q])
 *   pw_w  [Cin][Cout] bf16   (P[q][k])
 *   out   [N][H][W][Cout] fp32
 *
 * The depthwise result is formed in fp32 and rounded to bf16 for the tensor
 * cores; it never leaves the chip.  The pointwise weights stay resident in
 * shared memory; where Cin x Cout of them do not fit beside the kernel's
 * other buffers (Cin = Cout = 256, for one), the output channels are split
 * into blocks of equal width (a multiple of 16), one launch per block, each
 * recomputing the depthwise stage.
 * Supported: Cin % 16 == 0, 16 <= Cin <= 256, Cout % 16 == 0,
 * 16 <= Cout <= 256; pointers 16-byte aligned.  Otherwise
 * ISAM_ERR_UNSUPPORTED.
 */
int isam_dwsep_conv(int N, int H, int W, int Cin, int Cout, const isam_bf16 *x,
                    const isam_bf16 *dw_w, const isam_bf16 *pw_w, float *out);

/*
 * The first factor of Listing 3 alone: a 3x3 depthwise convolution over an
 * NHWC tensor (stride 1, zero border of one pixel, channel multiplier 1),
 *   y[n][i][j][c] = bf16( sum_{di,dj in 0..2} x[n][i+di-1][j+dj-1][c] * D[di][dj][c] ),
 * summed in fp32 (taps in row-major order) and rounded once to bf16.
 * Followed by isam_gemm(M = N*H*W, N = Cout, K = C, transA = 0, transB = 0,
 * A = y, B = pw_w), it is the unfused schedule of the separable layer
 * (Section 2.3), which writes the intermediate to memory; isam_dwsep_conv is
 * the fused one.
 *   x [N][H][W][C] bf16, dw_w [3][3][C] bf16, y [N][H][W][C] bf16; device
 *   pointers, 16-byte aligned; C a multiple of 8.  Otherwise
 *   ISAM_ERR_UNSUPPORTED; sizes < 1 or null pointers ISAM_ERR_INVALID_ARG.
 */
int isam_depthwise_conv3x3(int N, int H, int W, int C, const isam_bf16 *x, const isam_bf16 *dw_w,
                           isam_bf16 *y);

/*
 * The plan isam_dwsep_conv takes for an image W pixels wide with Cin -> Cout
 * channels (it does not depend on N or H); nothing is launched.  out[4]:
 *   out[0]  kernel: 0 = whole image rows per tile with an input-row ring in
 *           shared memory, 1 = 128 pixels per tile, loaded per pixel
 *   out[1]  image rows per tile (kernel 0), else 0
 *   out[2]  output-channel blocks (launches)
 *   out[3]  channels per block (the last block may be narrower)
 * Returns ISAM_ERR_UNSUPPORTED for channel counts isam_dwsep_conv rejects.
 */
int isam_dwsep_plan_info(int W, int Cin, int Cout, int *out);

/*
 * isam_dwsep_plan_info's plan for a device whose CTAs may opt in to
 * smem_optin bytes of shared memory (232448 on sm_103a); host arithmetic
 * only, no CUDA call, so it runs without a GPU.  ISAM_ERR_INVALID_ARG for
 * sizes < 1 or a null out.
 */
int isam_dwsep_plan_for(int W, int Cin, int Cout, int smem_optin, int *out);

/*
 * The plan isam_gru_forward (layers = 1) or isam_gru_forward_stack takes for
 * this batch and hidden size (it does not depend on T); nothing is launched.
 * out[7]:
 *   out[0]  K splits per group of 32 hidden units (cluster size: 1, 2 or 4)
 *   out[1]  64-wide K atoms of U each CTA keeps resident
 *   out[2]  padded batch of the recurrence (the MMA's N: 32, 64 or 128)
 *   out[3]  CTAs of the recurrence (hidden / 32 x splits)
 *   out[4]  shared memory of one recurrence CTA in bytes (the largest kernel
 *           the call launches)
 *   out[5]  how layers run: 0 one layer; 1 pairs of layers in one kernel;
 *           2 one kernel per layer that also computes the next layer's input
 *           projection; 3 layer by layer, the batch in chunks of out[2] rows
 *   out[6]  recurrence launches per layer (batch chunks)
 * Returns ISAM_ERR_UNSUPPORTED (with the reason) for shapes the call rejects,
 * ISAM_ERR_INVALID_ARG for sizes < 1, reset_before not 0 or 1, or a null out.
 */
int isam_gru_plan_info(int layers, int batch, int hidden, int reset_before, int *out);

/*
 * isam_gru_plan_info's plan for a device with num_sms SMs (152 on a GB300)
 * and smem_optin bytes of shared memory per CTA; host arithmetic only, no
 * CUDA call.
 */
int isam_gru_plan_for(int layers, int batch, int hidden, int reset_before, int num_sms, int smem_optin,
                      int *out);

#ifdef __cplusplus
}
#endif
#endif /* ISAM_H */
