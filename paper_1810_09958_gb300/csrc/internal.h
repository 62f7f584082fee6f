// internal.h -- host-side declarations shared by the library's translation
// units.  Not part of the public ABI (that is include/isam.h).
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

#include "../../include/isam.h"

namespace isam {

// Device error word layout (uint32 x 4), written by kernels and read by
// isam_sync: [0] flags, [1] site of the first error, [2] blockIdx.x of that
// CTA, [3] detail (the cluster size a kernel found, for a launch-shape error).
enum : uint32_t { DEV_ERR_TIMEOUT = 1u, DEV_ERR_LAUNCH_SHAPE = 2u };

// Per-device state, created on first use with that device current.
struct DeviceState {
    int device = -1;
    int num_sms = 0;
    int max_smem_optin = 0;
    // Clusters of 2, 4 and 8 CTAs resident at once; 0 = ask the device (a
    // host-side plan for given limits fills them in).
    int cluster_cap[3] = {0, 0, 0};
    uint32_t *err_word = nullptr;  // 4 x uint32 on the device
    // GRU workspaces (grown on demand).
    float *gru_gx = nullptr;       // [T*batch][3H] fp32 input projection
    size_t gru_gx_bytes = 0;
    uint16_t *gru_hx = nullptr;    // 2 x [32][H] bf16 hidden-state exchange
    size_t gru_hx_bytes = 0;
    uint32_t *gru_counter = nullptr;  // step counter (1 x uint32, padded)
    float *gru_gxp = nullptr;      // 2 x [ks][T*batch][3H] fp32 stacked layers' projections
    size_t gru_gxp_bytes = 0;
    uint16_t *gru_xb = nullptr;    // [T*batch][H] bf16 states of a layer (next pair's input)
    size_t gru_xb_bytes = 0;
};

DeviceState *device_state(int *status);  // current device; null + status on failure
cudaStream_t current_stream();
unsigned long long wait_timeout_ns();

int set_error(int code, const char *fmt, ...);
int cuda_error(cudaError_t e, const char *what);

// Raises kernel fn's dynamic shared-memory limit to at least `bytes` on the
// current device, whose ordinal is `device`.  The attribute belongs to each
// device's context, so the record of what was set is kept per (device, kernel).
int ensure_smem_optin(const void *fn, int bytes, int device, const char *what);

// cuTensorMapEncodeTiled through the runtime's driver entry point, with a
// small cache keyed on every encoded field.
int make_tmap_2d_bf16(CUtensorMap *out, const void *base, uint64_t inner, uint64_t outer,
                      uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer);
int make_tmap_2d_f32(CUtensorMap *out, const void *base, uint64_t inner, uint64_t outer,
                     uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer);
// Same for 8-bit elements (E4M3 operands), 128-byte swizzle.
int make_tmap_2d_u8(CUtensorMap *out, const void *base, uint64_t inner, uint64_t outer,
                    uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer);
int make_tmap_3d_bf16(CUtensorMap *out, const void *base, const uint64_t dims[3],
                      const uint64_t strides_bytes[2], const uint32_t box[3]);

// GEMM C = alpha op(A) op(B) + beta C (+ bias[n] per column when bias != null).
struct GemmDesc {
    int M, N, K;
    int transA, transB;
    float alpha, beta;
    const uint16_t *A;
    const uint16_t *B;
    float *C;
    const float *bias_n;
    int fp8 = 0;  // A and B are E4M3 bytes (A: M x K, B: N x K, both K-major)
};

// Tile plan chosen by the cost model (or forced through ISAM_FORCE_TILE).
struct GemmPlan {
    int BN;       // tile width (tile height is always 128)
    int ka;       // 64-wide K atoms per pipeline stage
    int split;    // CTAs of one cluster sharing a tile along K (1, 2, 4 or 8)
    int stages;   // shared-memory ring depth
    int group_m;  // rasterisation group height (tiles)
    int grid;     // CTAs launched (persistent)
    size_t smem;  // dynamic shared memory bytes
    double est_us;
    int pair = 0; // 1: 256 x 256 tiles on CTA pairs (cta_group::2), see gemm_pair.cu
};

int gemm_validate(const GemmDesc &g);
int gemm_plan(const GemmDesc &g, const DeviceState &ds, GemmPlan *plan);
int gemm_launch(const GemmDesc &g, const GemmPlan &plan, DeviceState &ds, cudaStream_t s);
// The CTA-pair kernel: fills *plan and returns 1 when the problem suits it
// (K-major A, bf16, N % 4 == 0, at least one 256 x 256 tile per SM pair).
int gemm_pair_plan(const GemmDesc &g, const DeviceState &ds, GemmPlan *plan);
// Clusters of `size` CTAs (one per SM) resident at once on this device.
int gemm_cluster_capacity(const DeviceState &ds, int size);
int gemm_pair_launch(const GemmDesc &g, const GemmPlan &plan, DeviceState &ds, cudaStream_t s);

// Independent GEMMs in one persistent launch (1 <= count <= 64).
int gemm_grouped_launch(int count, const GemmDesc *g, DeviceState &ds, cudaStream_t s);

// Block-scaled E4M3 GEMM (OCP MX): C = alpha (SA o A)(SB o B)^T + beta C with
// A M x K and B N x K E4M3 bytes (K-major) and one E8M0 scale byte per 32 K
// elements of each row, atom-major: SA [ceil(K/128)][M][4], SB
// [ceil(K/128)][N][4] (4-byte aligned).
struct MxDesc {
    int M, N, K;
    float alpha, beta;
    const uint8_t *A;
    const uint8_t *SA;
    const uint8_t *B;
    const uint8_t *SB;
    float *C;
};
int gemm_mx_validate(const MxDesc &g);
// One persistent launch over the tiles of 1 <= count <= 64 problems.
int gemm_mx_launch(int count, const MxDesc *g, DeviceState &ds, cudaStream_t s);

// reset_before: the candidate's recurrent input is U_n (r * h) (two rounds per step).
int gru_launch(int T, int batch, int hidden, const uint16_t *x, const uint16_t *W,
               const uint16_t *U, const float *b, const float *h0, float *h_out, DeviceState &ds,
               cudaStream_t s, int reset_before = 0);
// Two stacked layers in one persistent kernel (reset gate after the
// product, hidden a multiple of 256): layer a's projection gx_a is given,
// layer b's comes from W_b and layer a's states inside the kernel.
bool gru_wave_supported(int H, int batch, const DeviceState &ds);
bool gru_wave_fits(int H, int batch, int num_sms, int smem_optin);
size_t gru_wave_smem_bytes(int H);

// How a GRU call runs on a device with num_sms SMs and smem_optin bytes of
// shared memory per CTA (host arithmetic only, no CUDA call).
struct GruPlan {
    int ks = 0;       // K splits per group of 32 units (cluster size)
    int ka = 0;       // 64-wide K atoms per CTA
    int bp = 0;       // padded batch (the MMA's N)
    int n_cta = 0;    // CTAs of the recurrence
    int smem = 0;     // shared memory of one recurrence CTA (the largest launched)
    int path = 0;     // 0 one layer, 1 layer pairs in one kernel, 2 per-layer chain, 3 layer by layer in batch chunks
    int chunks = 0;   // recurrence launches per layer
};
int gru_plan(int layers, int batch, int hidden, int reset_before, int num_sms, int smem_optin, GruPlan *g);
int gru_wave_launch(int T, int batch, int H, const float *gx_a, const uint16_t *U_a, const uint16_t *W_b,
                    const uint16_t *U_b, const float *b_a, const float *b_b, const float *h0_a,
                    const float *h0_b, float *out_a, float *out_b, uint16_t *hx_a, uint16_t *hx_b,
                    uint32_t *counter, DeviceState &ds, cudaStream_t stream);
int gru_stack_launch(int layers, int T, int batch, int hidden, int reset_before, const uint16_t *x,
                     const uint16_t *W, const uint16_t *U, const float *b, const float *h0, float *h_out,
                     DeviceState &ds, cudaStream_t stream);

int dwsep_launch(int N, int H, int W, int Cin, int Cout, const uint16_t *x, const uint16_t *dw,
                 const uint16_t *pw, float *out, DeviceState &ds, cudaStream_t s);
// The 3x3 depthwise stage alone: y (NHWC bf16) from x (NHWC bf16) and dw
// [3][3][C]; C a multiple of 8, pointers 16-byte aligned (checked by the caller).
int depthwise_launch(int N, int H, int W, int C, const uint16_t *x, const uint16_t *dw, uint16_t *y,
                     const DeviceState &ds, cudaStream_t s);
// out[4]: kernel (0 row ring, 1 per-pixel), image rows per tile, channel blocks, block width.
int dwsep_plan(int W, int Cin, int Cout, int smem_optin, int *out);

}  // namespace isam
