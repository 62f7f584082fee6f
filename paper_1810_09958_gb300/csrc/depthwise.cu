// depthwise.cu -- the first factor of Listing 3 on its own: a 3x3 depthwise
// convolution (stride 1, zero border of one pixel, channel multiplier 1) over
// an NHWC bf16 tensor, written back to memory as bf16.
//
// It exists to compare the factored layer's two forms: the fused kernel
// (dwsep.cu) keeps the depthwise result on chip and feeds the tensor cores
// from shared memory, while this kernel followed by isam_gemm (the pointwise
// factor, M = N*H*W, K = C, N = Cout) round-trips the intermediate through
// HBM -- the unfused schedule of Section 2.3's factorisation.
//
// One thread produces eight channels (16 bytes) of one output pixel: nine
// 16-byte tap loads (each input pixel is read by its nine neighbours; L1/L2
// serve the repeats), fp32 multiply-adds in tap order (row di, then column
// dj), one rounding to bf16 and one 16-byte store.  Consecutive threads take
// consecutive channel groups of a pixel, so every warp access is contiguous;
// a block works on one output row at a time (its three input rows stay in L2
// for the neighbouring rows' blocks).
#include <algorithm>
#include <cstdint>

#include "internal.h"

namespace isam {

namespace {

constexpr int kDwThreads = 256;

__device__ __forceinline__ float lo_f(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float hi_f(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
    uint32_t r;  // round-to-nearest-even of both; hi in the upper half
    asm("cvt.rn.bf16x2.f32 %0, %2, %1;" : "=r"(r) : "f"(lo), "f"(hi));
    return r;
}

// Blocks walk output rows (image n, row i); within a row, thread k takes
// pixel k / CG, channel group k % CG.  Indices are 32-bit inside a row; the
// row base is 64-bit.
__global__ void __launch_bounds__(kDwThreads) depthwise3x3_kernel(const uint4 *__restrict__ x,
                                                                  const uint4 *__restrict__ dw, uint4 *__restrict__ y,
                                                                  int N, int H, int W, int CG) {
    const int per_row = W * CG;
    for (int r = blockIdx.y; r < N * H; r += gridDim.y) {
        const int img = r / H, yq = r - img * H;
        const size_t img_base = static_cast<size_t>(img) * H * per_row;
        for (int k = blockIdx.x * kDwThreads + threadIdx.x; k < per_row; k += gridDim.x * kDwThreads) {
            const int xq = k / CG, g = k - xq * CG;
            float acc[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) acc[c] = 0.0f;
#pragma unroll
            for (int di = 0; di < 3; ++di) {
                const int yy = yq + di - 1;
                const bool row_ok = yy >= 0 && yy < H;
                const uint4 *xr = x + img_base + static_cast<size_t>(row_ok ? yy : 0) * per_row;
#pragma unroll
                for (int dj = 0; dj < 3; ++dj) {
                    const int xx = xq + dj - 1;
                    uint4 v = make_uint4(0u, 0u, 0u, 0u);
                    if (row_ok && xx >= 0 && xx < W) v = __ldg(xr + xx * CG + g);
                    const uint4 wv = __ldg(dw + (di * 3 + dj) * CG + g);
                    acc[0] = fmaf(lo_f(v.x), lo_f(wv.x), acc[0]);
                    acc[1] = fmaf(hi_f(v.x), hi_f(wv.x), acc[1]);
                    acc[2] = fmaf(lo_f(v.y), lo_f(wv.y), acc[2]);
                    acc[3] = fmaf(hi_f(v.y), hi_f(wv.y), acc[3]);
                    acc[4] = fmaf(lo_f(v.z), lo_f(wv.z), acc[4]);
                    acc[5] = fmaf(hi_f(v.z), hi_f(wv.z), acc[5]);
                    acc[6] = fmaf(lo_f(v.w), lo_f(wv.w), acc[6]);
                    acc[7] = fmaf(hi_f(v.w), hi_f(wv.w), acc[7]);
                }
            }
            y[img_base + static_cast<size_t>(yq) * per_row + k] =
                make_uint4(pack2(acc[0], acc[1]), pack2(acc[2], acc[3]), pack2(acc[4], acc[5]), pack2(acc[6], acc[7]));
        }
    }
}

}  // namespace

int depthwise_launch(int N, int H, int W, int C, const uint16_t *x, const uint16_t *dw, uint16_t *y,
                     const DeviceState &ds, cudaStream_t stream) {
    const int CG = C / 8;
    const long long per_row = static_cast<long long>(W) * CG;
    if (per_row > (1LL << 30))
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_depthwise_conv3x3: W * C / 8 must stay below 2^30");
    const int bx = static_cast<int>((per_row + kDwThreads - 1) / kDwThreads);
    const long long rows = static_cast<long long>(N) * H;
    if (rows > 0x7FFFFFFFLL) return set_error(ISAM_ERR_UNSUPPORTED, "isam_depthwise_conv3x3: N * H too large");
    // About four resident blocks per SM, each walking many rows: a block that
    // handled a single row would spend most of its life starting and ending.
    const long long want_y = std::max(1LL, 4LL * ds.num_sms / bx);
    const int by = static_cast<int>(std::min({rows, want_y, 65535LL}));
    depthwise3x3_kernel<<<dim3(static_cast<unsigned>(bx), static_cast<unsigned>(by)), kDwThreads, 0, stream>>>(
        reinterpret_cast<const uint4 *>(x), reinterpret_cast<const uint4 *>(dw), reinterpret_cast<uint4 *>(y), N, H,
        W, CG);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "launch depthwise3x3_kernel");
    return ISAM_OK;
}

}  // namespace isam
