// dwsep.cu -- separable depthwise convolution (Listing 3 with s = 1, c = 1,
// zero border of one pixel) on sm_103a, in the factored form of Section 2.3:
// the 3x3 depthwise sum is formed first and the result is multiplied by the
// pointwise weights, a GEMM with M = N*H*W pixels, K = Cin, N = Cout.
//
// One persistent kernel, one CTA per SM, 128-pixel tiles:
//   warps 0-7  depthwise producers: for two pixels at a time issue all nine
//              16-byte NHWC tap loads at once (clamped addresses, masked
//              afterwards), accumulate in fp32, round to bf16 and write the A
//              tile straight into the tensor cores' 128-byte swizzled K-major
//              layout (two-stage ring);
//   warp 8     loads the pointwise weights once (TMA, resident for the whole
//              kernel) and issues tcgen05.mma from one thread into a
//              double-buffered TMEM accumulator;
//   warps 9-12 drain TMEM, stage 32x32 fp32 blocks in swizzled shared memory
//              and write them out with TMA bulk tensor stores.
// The depthwise intermediate never leaves the chip.
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdio>
#include <type_traits>

#include "internal.h"
#include "ptx.cuh"

namespace isam {

namespace {

constexpr int kBM = 128;
constexpr int kProdWarps = 8;                 // depthwise producer warps 0-7
constexpr int kProd = kProdWarps * 32;
constexpr int kMmaWarp = kProdWarps;          // warp 8
constexpr int kEpiWarp0 = kProdWarps + 1;     // warps 9-12
constexpr int kThreads = (kProdWarps + 5) * 32;
constexpr int kAStages = 2;
constexpr int kStageBufs = 2;  // epilogue staging buffers per warp (4 KB each)

enum : uint32_t {
    SITE_DW_AEMPTY = 0x301,
    SITE_DW_AFULL = 0x302,
    SITE_DW_TEMPTY = 0x303,
    SITE_DW_TFULL = 0x304,
    SITE_DW_W = 0x305,
};

struct DwParams {
    int N, H, W, Cin, Cout;
    long long M;            // N*H*W pixels
    int tiles;
    int atoms;              // ceil(Cin / 64) K atoms of the A tile
    int kb;                 // ceil(Cin / 64) k-blocks of the pointwise weights
    int nchunks;            // ceil(Cout / 64) 64-wide column chunks of the weights
    const uint16_t *x;
    const uint16_t *dw;
    unsigned long long timeout_ns;
    uint32_t *err;
};

struct DwLayout {
    int a_stage_bytes, w_bytes, dwf_bytes;
    int off_a, off_w, off_stage, off_dwf, off_bars;
    int total;
};

__host__ __device__ inline DwLayout dw_layout(int Cin, int Cout) {
    DwLayout L;
    const int atoms = (Cin + 63) / 64;
    const int nchunks = (Cout + 63) / 64;
    L.a_stage_bytes = atoms * kBM * 128;
    L.w_bytes = atoms * nchunks * 8192;
    L.dwf_bytes = ((9 * Cin * 4) + 1023) / 1024 * 1024;
    L.off_a = 0;
    L.off_w = L.off_a + kAStages * L.a_stage_bytes;
    L.off_stage = L.off_w + L.w_bytes;
    L.off_dwf = L.off_stage + 4 * kStageBufs * 4096;
    L.off_bars = L.off_dwf + L.dwf_bytes;
    L.total = L.off_bars + 256 + 1024;
    return L;
}

__device__ __forceinline__ float bf_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;  // round-to-nearest-even of both; hi in the upper half
    asm("cvt.rn.bf16x2.f32 %0, %2, %1;" : "=r"(r) : "f"(lo), "f"(hi));
    return r;
}

// c + a * w with a and w bf16 (the lower or upper halves of x and wp) and c
// fp32: both bf16 operands widen exactly to fp32, and the multiply-add rounds
// once, as fmaf on the widened values would.
__device__ __forceinline__ float fma_bf16_lo(uint32_t x, uint32_t wp, float c) {
    float d;
    asm("{\n\t.reg .b16 xl, xh, wl, wh;\n\t"
        "mov.b32 {xl, xh}, %1;\n\t"
        "mov.b32 {wl, wh}, %2;\n\t"
        "fma.rn.f32.bf16 %0, xl, wl, %3;\n\t}"
        : "=f"(d)
        : "r"(x), "r"(wp), "f"(c));
    return d;
}

__device__ __forceinline__ float fma_bf16_hi(uint32_t x, uint32_t wp, float c) {
    float d;
    asm("{\n\t.reg .b16 xl, xh, wl, wh;\n\t"
        "mov.b32 {xl, xh}, %1;\n\t"
        "mov.b32 {wl, wh}, %2;\n\t"
        "fma.rn.f32.bf16 %0, xh, wh, %3;\n\t}"
        : "=f"(d)
        : "r"(x), "r"(wp), "f"(c));
    return d;
}

__global__ void __launch_bounds__(kThreads, 1)
    dwsep_fused_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmOut,
                       const DwParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    const DwLayout L = dw_layout(p.Cin, p.Cout);
    uint8_t *sA = smem + L.off_a;
    uint8_t *sW = smem + L.off_w;
    uint8_t *sStage = smem + L.off_stage;
    float *dwf = reinterpret_cast<float *>(smem + L.off_dwf);
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L.off_bars);
    uint64_t *a_full = bars;                 // [kAStages]
    uint64_t *a_empty = bars + kAStages;     // [kAStages]
    uint64_t *tfull = a_empty + kAStages;    // [2]
    uint64_t *tempty = tfull + 2;            // [2]
    uint64_t *wbar = tempty + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(wbar + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int Cin = p.Cin, Cout = p.Cout;
    const int ncols = Cout <= 64 ? 64 : (Cout <= 128 ? 128 : 256);  // accumulator width (pow2)
    const uint32_t tmem_cols = 2u * static_cast<uint32_t>(ncols);

    if (tid == 0) {
        for (int s = 0; s < kAStages; ++s) {
            mbar_init(&a_full[s], kProd);
            mbar_init(&a_empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        mbar_init(wbar, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    for (int i = tid; i < 9 * Cin; i += kThreads)
        dwf[i] = __uint_as_float(static_cast<uint32_t>(p.dw[i]) << 16);
    __syncwarp();
    if (warp == kMmaWarp) {
        tmem_alloc(tmem_slot, tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx w{p.timeout_ns, p.err, abort_flag};

    if (warp < kProdWarps) {
        // ------------------------------------------------ depthwise producers
        const int groups = Cin / 8;           // 16-byte channel groups per pixel
        const int items = kBM * groups;
        const int H = p.H, W = p.W, HW = p.H * p.W;
        const int M = static_cast<int>(p.M);
        const uint4 zero4 = make_uint4(0u, 0u, 0u, 0u);
        int stage = 0;
        uint32_t phase = 0;
        for (int tile = blockIdx.x; tile < p.tiles; tile += gridDim.x) {
            if (!bounded_wait(&a_empty[stage], phase ^ 1u, w, SITE_DW_AEMPTY)) break;
            uint8_t *a = sA + stage * L.a_stage_bytes;
            const int p0 = tile * kBM;
            for (int it0 = tid; it0 < items; it0 += 2 * kProd) {
                uint4 v[2][9];
                int rr[2], gg[2];
                bool live[2];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int it = it0 + u * kProd;
                    const int r = it / groups;
                    const int g = it - r * groups;
                    const int pix = p0 + r;
                    live[u] = it < items && pix < M;
                    rr[u] = r;
                    gg[u] = g;
                    const int n = live[u] ? pix / HW : 0;
                    const int rem = live[u] ? pix - n * HW : 0;
                    const int y = rem / W;
                    const int xx = rem - y * W;
                    const uint16_t *img = p.x + static_cast<size_t>(n) * HW * Cin + g * 8;
#pragma unroll
                    for (int t = 0; t < 9; ++t) {
                        const int yy = y + t / 3 - 1;
                        const int xc = xx + t % 3 - 1;
                        const bool ok = live[u] && static_cast<unsigned>(yy) < static_cast<unsigned>(H) &&
                                        static_cast<unsigned>(xc) < static_cast<unsigned>(W);
                        const uint16_t *src = ok ? img + (static_cast<size_t>(yy) * W + xc) * Cin : p.x;
                        const uint4 t4 = __ldg(reinterpret_cast<const uint4 *>(src));
                        v[u][t] = ok ? t4 : zero4;
                    }
                }
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    if (!live[u]) continue;
                    const int g = gg[u], r = rr[u];
                    float acc[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) acc[i] = 0.0f;
#pragma unroll
                    for (int t = 0; t < 9; ++t) {
                        const float *wt = dwf + t * Cin + g * 8;
                        const float4 w0 = *reinterpret_cast<const float4 *>(wt);
                        const float4 w1 = *reinterpret_cast<const float4 *>(wt + 4);
                        const uint4 q = v[u][t];
                        acc[0] = fmaf(bf_lo(q.x), w0.x, acc[0]);
                        acc[1] = fmaf(bf_hi(q.x), w0.y, acc[1]);
                        acc[2] = fmaf(bf_lo(q.y), w0.z, acc[2]);
                        acc[3] = fmaf(bf_hi(q.y), w0.w, acc[3]);
                        acc[4] = fmaf(bf_lo(q.z), w1.x, acc[4]);
                        acc[5] = fmaf(bf_hi(q.z), w1.y, acc[5]);
                        acc[6] = fmaf(bf_lo(q.w), w1.z, acc[6]);
                        acc[7] = fmaf(bf_hi(q.w), w1.w, acc[7]);
                    }
                    uint4 o;
                    o.x = pack_bf16x2(acc[0], acc[1]);
                    o.y = pack_bf16x2(acc[2], acc[3]);
                    o.z = pack_bf16x2(acc[4], acc[5]);
                    o.w = pack_bf16x2(acc[6], acc[7]);
                    // K-major, 128-byte swizzle: atom g/8, row r, 16-byte chunk (g%8) ^ (r%8).
                    const int atom = g >> 3;
                    const int chunk = (g & 7) ^ (r & 7);
                    *reinterpret_cast<uint4 *>(a + atom * (kBM * 128) + r * 128 + chunk * 16) = o;
                }
            }
            fence_proxy_async_smem();
            mbar_arrive(&a_full[stage]);
            if (++stage == kAStages) {
                stage = 0;
                phase ^= 1u;
            }
        }
        __syncwarp();
    } else if (warp == kMmaWarp) {
        // ------------------------------------------------ weights + MMA issuer
        if (lane == 0) {
            bool ok = true;
            tma_prefetch_desc(&tmW);
            mbar_arrive_expect_tx(wbar, static_cast<uint32_t>(L.w_bytes));
            for (int kb = 0; kb < p.kb; ++kb)
                for (int c = 0; c < p.nchunks; ++c)
                    tma_load_2d(&tmW, wbar, sW + (kb * p.nchunks + c) * 8192, c * 64, kb * 64);
            ok = bounded_wait(wbar, 0, w, SITE_DW_W);
            const uint32_t idesc = idesc_bf16_f32(kBM, Cout, false, true);
            const int ksteps = Cin / 16;
            int stage = 0, acc = 0;
            uint32_t phase = 0, acc_phase = 0;
            for (int tile = blockIdx.x; ok && tile < p.tiles; tile += gridDim.x) {
                if (!bounded_wait(&tempty[acc], acc_phase ^ 1u, w, SITE_DW_TEMPTY)) break;
                if (!bounded_wait(&a_full[stage], phase, w, SITE_DW_AFULL)) break;
                tc_fence_after();
                const uint32_t a0 = smem_u32(sA + stage * L.a_stage_bytes);
                const uint32_t w0 = smem_u32(sW);
                const uint32_t d = tmem_base + static_cast<uint32_t>(acc * ncols);
                for (int ks = 0; ks < ksteps; ++ks) {
                    const int atom = ks >> 2, kk = ks & 3;
                    const uint64_t ad = sdesc_sw128(a0 + atom * (kBM * 128) + kk * 32, 16, 1024);
                    const uint64_t bd = sdesc_sw128(w0 + atom * (p.nchunks * 8192) + kk * 2048, 8192, 1024);
                    umma_bf16(d, ad, bd, idesc, ks > 0 ? 1u : 0u);
                }
                umma_commit(&a_empty[stage]);
                umma_commit(&tfull[acc]);
                if (++stage == kAStages) {
                    stage = 0;
                    phase ^= 1u;
                }
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------ epilogue (warps 5-8)
        const int q = warp & 3;
        const int ew = warp - kEpiWarp0;
        uint8_t *stg = sStage + ew * (kStageBufs * 4096);
        int acc = 0, buf = 0;
        uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < p.tiles; tile += gridDim.x) {
            if (!__all_sync(0xffffffffu, bounded_wait(&tfull[acc], acc_phase, w, SITE_DW_TFULL) ? 1 : 0)) break;
            tc_fence_after();
            const uint32_t tb = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                static_cast<uint32_t>(acc * ncols);
            const int row0 = tile * kBM + q * 32;
            for (int c = 0; c < Cout; c += 32) {
                uint32_t r[32];
                if (Cout - c >= 32) {
                    tmem_ld32(tb + c, r);
                } else {
                    uint32_t h[16];
                    tmem_ld16(tb + c, h);
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        r[i] = h[i];
                        r[16 + i] = 0u;
                    }
                }
                tmem_ld_wait();
                // Reuse of this staging buffer: its previous bulk store must have read it.
                if (lane == 0) bulk_wait_read<kStageBufs - 1>();
                __syncwarp();
                uint8_t *sb = stg + buf * 4096;
#pragma unroll
                for (int ch = 0; ch < 8; ++ch) {
                    const int pos = ch ^ (lane & 7);
                    *reinterpret_cast<uint4 *>(sb + lane * 128 + pos * 16) =
                        make_uint4(r[4 * ch], r[4 * ch + 1], r[4 * ch + 2], r[4 * ch + 3]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&tmOut, sb, c, row0);
                    bulk_commit();
                }
                buf = (buf + 1) % kStageBufs;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        if (lane == 0) bulk_wait_all<0>();
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, tmem_cols);
    }
}

// ---------------------------------------------------------------- row-ring variant
// For images no wider than 128 pixels: a tile is rt = 128 / W whole image
// rows, each CTA walks a contiguous range of tiles, and the input rows live in
// a shared-memory ring filled by one TMA copy per row.  Every input element
// then leaves L2 about once per CTA, and the producers read the 3x3 taps from
// shared memory.
constexpr int kRProdWarps = 11;               // depthwise producer warps 0-10
constexpr int kRProd = kRProdWarps * 32;
constexpr int kRMmaWarp = kRProdWarps;         // warp 11: ring loader + MMA issuer
constexpr int kREpiWarp0 = kRProdWarps + 1;    // warps 12-19: epilogue, two per TMEM lane quarter
constexpr int kREpiWarps = 8;
constexpr int kRThreads = (kRProdWarps + 1 + kREpiWarps) * 32;
constexpr int kRingMax = 32;  // input rows resident per CTA: 2 * rt + 2 (this tile + halo + the next)

enum : uint32_t { SITE_DW_RING = 0x306 };

struct DwRowParams {
    int N, H, W, Cin, Cout;
    int rt;              // image rows per tile (rt * W <= 128)
    int tiles_per_img;   // ceil(H / rt)
    int tiles;           // N * tiles_per_img
    int kb, nchunks;
    const uint16_t *x;   // NHWC input: row (n * H + y) is W * Cin contiguous elements
    int row_bytes;       // one ring slot: W * Cin * 2 bytes of pixels + >= one pixel of zeros, rounded to 128
    int ring;            // input rows resident per CTA (2 * rt + 2 <= kRingMax)
    const uint16_t *dw;
    float *out;          // first output column of this launch's channel block
    int ldo;             // output row pitch in elements (all Cout channels of the layer)
    unsigned long long timeout_ns;
    uint32_t *err;
};

// The ring: a leading pad of dw_ring_lead bytes, then `ring` slots of
// dw_ring_row_bytes each.  A slot holds one input row (W pixels, written by
// TMA) followed by at least one pixel of zeros, so the left neighbour of
// pixel 0 (the previous slot's tail, or the leading pad) and the right
// neighbour of pixel W - 1 read as zero: the taps need no bounds test along x.
__host__ __device__ inline int dw_ring_lead(int Cin) { return (Cin * 2 + 127) / 128 * 128; }
__host__ __device__ inline int dw_ring_row_bytes(int W, int Cin) { return (W * Cin * 2 + Cin * 2 + 127) / 128 * 128; }

struct DwRowLayout {
    int off_ring, off_a, off_w, off_stage, off_bars, total;
};

__host__ __device__ inline DwRowLayout dw_row_layout(int W, int Cin, int Cout, int ring) {
    DwRowLayout L;
    const int atoms = (Cin + 63) / 64;
    const int nchunks = (Cout + 63) / 64;
    L.off_ring = 0;
    L.off_a = (dw_ring_lead(Cin) + ring * dw_ring_row_bytes(W, Cin) + 1023) / 1024 * 1024;
    L.off_w = L.off_a + atoms * kBM * 128;
    L.off_stage = L.off_w + atoms * nchunks * 8192;
    L.off_bars = L.off_stage + 4 * 2 * 4096;
    L.total = L.off_bars + 8 * (kRingMax + 8) + 16 + 1024;
    return L;
}

// First and last global input row (n * H + y) a tile reads.
__device__ __forceinline__ void tile_rows(const DwRowParams &p, int tile, int &n, int &y0, int &y1, int &lo,
                                          int &hi) {
    n = tile / p.tiles_per_img;
    y0 = (tile - n * p.tiles_per_img) * p.rt;
    y1 = min(p.H, y0 + p.rt) - 1;
    lo = n * p.H + max(0, y0 - 1);
    hi = n * p.H + min(p.H - 1, y1 + 1);
}

// A tile of the row-ring kernel: image n, tile row yt (image rows
// yt * rt .. yt * rt + rt - 1); it reads global input rows dw_lo .. dw_hi.
struct DwTilePos {
    int n, yt;
};

__device__ __forceinline__ DwTilePos dw_pos(const DwRowParams &p, int tile) {
    const int n = tile / p.tiles_per_img;
    return DwTilePos{n, tile - n * p.tiles_per_img};
}

__device__ __forceinline__ void dw_advance(const DwRowParams &p, DwTilePos &t) {
    if (++t.yt == p.tiles_per_img) {
        t.yt = 0;
        ++t.n;
    }
}

__device__ __forceinline__ int dw_lo(const DwRowParams &p, DwTilePos t) {
    return t.n * p.H + max(0, t.yt * p.rt - 1);
}

__device__ __forceinline__ int dw_hi(const DwRowParams &p, DwTilePos t) {
    return t.n * p.H + min(p.H - 1, min(p.H, t.yt * p.rt + p.rt));
}

__global__ void __launch_bounds__(kRThreads, 1)
    dwsep_rows_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmOut,
                      const __grid_constant__ CUtensorMap tmOut16, const __grid_constant__ CUtensorMap tmOut8,
                      const DwRowParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    const DwRowLayout L = dw_row_layout(p.W, p.Cin, p.Cout, p.ring);
    const int kRing = p.ring;
    const int lead = dw_ring_lead(p.Cin);
    uint8_t *ring = smem + L.off_ring + lead;  // slot s starts at ring + s * row_bytes
    uint8_t *sA = smem + L.off_a;
    uint8_t *sW = smem + L.off_w;
    uint8_t *sStage = smem + L.off_stage;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L.off_bars);
    uint64_t *ring_full = bars;           // [ring]
    uint64_t *a_full = ring_full + kRing;
    uint64_t *a_empty = a_full + 1;
    uint64_t *tfull = a_empty + 1;        // [2]
    uint64_t *tempty = tfull + 2;         // [2]
    uint64_t *wbar = tempty + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(wbar + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int Cin = p.Cin, Cout = p.Cout, W = p.W, H = p.H;
    const int ncols = Cout <= 64 ? 64 : (Cout <= 128 ? 128 : 256);
    const uint32_t tmem_cols = 2u * static_cast<uint32_t>(ncols);
    // This CTA's contiguous tile range.
    const int tb = static_cast<int>((static_cast<long long>(blockIdx.x) * p.tiles) / gridDim.x);
    const int te = static_cast<int>((static_cast<long long>(blockIdx.x + 1) * p.tiles) / gridDim.x);

    if (tid == 0) {
        for (int i = 0; i < kRing; ++i) mbar_init(&ring_full[i], 1);
        mbar_init(a_full, kRProdWarps);
        mbar_init(a_empty, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], kREpiWarps);
        }
        mbar_init(wbar, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    {
        // Zero the leading pad and every slot's tail (TMA never writes them).
        const int tail = p.row_bytes - W * Cin * 2;  // multiple of 16
        const int units = (lead + kRing * tail) / 16;
        for (int i = tid; i < units; i += kRThreads) {
            const int off = i * 16;
            int at;
            if (off < lead) {
                at = off;
            } else {
                const int s = (off - lead) / tail;
                at = lead + s * p.row_bytes + W * Cin * 2 + (off - lead - s * tail);
            }
            *reinterpret_cast<uint4 *>(smem + L.off_ring + at) = make_uint4(0u, 0u, 0u, 0u);
        }
    }
    __syncwarp();
    if (warp == kRMmaWarp) {
        tmem_alloc(tmem_slot, tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx w{p.timeout_ns, p.err, abort_flag};

    if (warp < kRProdWarps) {
        // ------------------------------------------------ depthwise producers
        // Thread tid owns 4 channels (group g, weights in registers); with
        // Cin = 128 the 32 lanes of a warp cover one pixel's channels, so
        // the image-edge decisions below are the same for the whole warp.
        // Tile, row and ring-slot positions advance incrementally: an integer
        // division by a run-time value costs hundreds of cycles of latency,
        // and here it would sit on the critical path of every tile.
        const int groups = Cin / 4;  // at most 64 (Cin <= 256), fewer than kRProd
        const int g = tid % groups;
        // Column segment of this thread: the kRProd / groups whole segments
        // split the W columns evenly (lengths differ by at most one); threads
        // past the last whole segment get an empty one (x from W to W: they
        // read valid columns and store nothing) and only join the barriers.
        const int nseg = kRProd / groups;
        const int seg = tid / groups;
        const bool seg_live = seg < nseg;
        const int xs = seg_live ? (seg * W) / nseg : W;
        const int xe = seg_live ? ((seg + 1) * W) / nseg : W;
        const int seg_max = (W + nseg - 1) / nseg;
        uint32_t wb[9][2];  // bf16 weights of channels 4g..4g+3, two per word
#pragma unroll
        for (int t = 0; t < 9; ++t) {
            const uint2 wv = *reinterpret_cast<const uint2 *>(p.dw + t * Cin + g * 4);
            wb[t][0] = wv.x;
            wb[t][1] = wv.y;
        }
        // Channels 4g..4g+3 in the A tile: K atom g / 16, 16-byte chunk
        // (g % 16) / 2 (swizzled by the pixel row), half g % 2 of the chunk.
        const int atom = g >> 4;
        const int chunk = (g & 15) >> 1;
        const int half = (g & 1) * 8;
        // Global input row r lives in ring slot (r - first_row) mod kRing;
        // its barrier completes phase (r - first_row) / kRing.  The MMA
        // thread loads the rows; the producers only wait for them.
        DwTilePos pos = dw_pos(p, tb);
        const int first_row = tb < te ? dw_lo(p, pos) : 0;
        int lo_prev = first_row, lo_slot = 0;  // slot and round of this tile's first row
        uint32_t lo_round = 0;
        uint32_t a_phase = 0;
        bool ok = true, a_ok = true;
        for (int tile = tb; tile < te; ++tile) {
            const int n = pos.n;
            const int y0 = pos.yt * p.rt;
            const int y1 = min(H, y0 + p.rt) - 1;
            const int base_row = n * H;
            const int lo = dw_lo(p, pos);
            const int hi = dw_hi(p, pos);
            for (int d = lo - lo_prev; d > 0; --d)
                if (++lo_slot == kRing) {
                    lo_slot = 0;
                    ++lo_round;
                }
            lo_prev = lo;
            // Lane k of each warp polls the barrier of the tile's k-th input
            // row, all at once (one after another they cost a barrier round
            // trip each); the barrier after it combines the answers (and a
            // failed A-stage wait of the previous tile) and joins the
            // producers again.  (Without it a warp whose lanes took different
            // branches stayed split for the whole first round of the tile:
            // measured 3x slower.)
            __syncwarp();
            bool wok = a_ok;
            if (lane <= hi - lo) {
                int sl = lo_slot + lane;
                uint32_t rnd = lo_round;
                if (sl >= kRing) {
                    sl -= kRing;
                    ++rnd;
                }
                wok = wok && bounded_wait(&ring_full[sl], rnd & 1u, w, SITE_DW_RING);
            }
            __syncwarp();
            ok = named_bar_and(2, kRProd, wok);
            if (!ok) break;  // the same decision in every producer
            const int rows = y1 - y0 + 1;
            // Ring slot of input row y0 - 1 (any slot when y0 == 0: that row is
            // outside the image and never used).
            int s_top = lo_slot + (base_row + y0 - 1 - lo);
            if (s_top < 0) s_top += kRing;
            // Each thread walks its column segment [xs, xe) of every pair of
            // tile rows (2rp, 2rp + 1), keeping a 4-row x 3-column window of
            // taps in registers: one new column (4 loads) per output pair.
            // Every thread runs the same number of steps (the longest
            // segment), so the lanes of a warp stay together; steps past the
            // segment read a valid column and store nothing.  Interior tiles
            // (every input row inside the image) run without row tests.
            const bool interior = y0 >= 1 && y1 + 1 <= H - 1;
            const int nrp = (rows + 1) >> 1;
            auto run = [&](auto check_rows) {
                constexpr bool kCheckRows = decltype(check_rows)::value;
                for (int rp = 0; rp < nrp; ++rp) {
                    const int ya = y0 + 2 * rp;
                    const bool two = 2 * rp + 1 < rows;
                    int sl = s_top + 2 * rp;  // input row ya - 1
                    while (sl >= kRing) sl -= kRing;
                    const uint8_t *rowp[4];
                    bool rv[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        rowp[k] = ring + sl * p.row_bytes + g * 8;
                        rv[k] = !kCheckRows || (ya - 1 + k >= 0 && ya - 1 + k < H);
                        sl = (sl + 1 == kRing) ? 0 : sl + 1;
                    }
                    auto col = [&](int k, int xc) {
                        uint2 q = *reinterpret_cast<const uint2 *>(rowp[k] + xc * (Cin * 2));
                        if (kCheckRows && !rv[k]) q = make_uint2(0u, 0u);
                        return q;
                    };
                    uint2 c0[4], c1[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        c0[k] = col(k, xs - 1);  // x = -1 reads the zero pad
                        c1[k] = col(k, xs);
                    }
                    for (int st = 0; st < seg_max; ++st) {
                        const int x = xs + st;
                        const bool act = x < xe;
                        uint2 c2[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) c2[k] = col(k, min(x + 1, W));  // x + 1 == W: zero pad
                        float acc0[4] = {0.0f, 0.0f, 0.0f, 0.0f}, acc1[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
#pragma unroll
                            for (int dj = 0; dj < 3; ++dj) {
                                const uint2 q = dj == 0 ? c0[k] : (dj == 1 ? c1[k] : c2[k]);
                                if (k <= 2) {
                                    const uint32_t *wt = wb[k * 3 + dj];
                                    acc0[0] = fma_bf16_lo(q.x, wt[0], acc0[0]);
                                    acc0[1] = fma_bf16_hi(q.x, wt[0], acc0[1]);
                                    acc0[2] = fma_bf16_lo(q.y, wt[1], acc0[2]);
                                    acc0[3] = fma_bf16_hi(q.y, wt[1], acc0[3]);
                                }
                                if (k >= 1) {
                                    const uint32_t *wt = wb[(k - 1) * 3 + dj];
                                    acc1[0] = fma_bf16_lo(q.x, wt[0], acc1[0]);
                                    acc1[1] = fma_bf16_hi(q.x, wt[0], acc1[1]);
                                    acc1[2] = fma_bf16_lo(q.y, wt[1], acc1[2]);
                                    acc1[3] = fma_bf16_hi(q.y, wt[1], acc1[3]);
                                }
                            }
                        }
                        if (rp == 0 && st == 0) {
                            // The A stage is free once the MMA of the previous
                            // tile is done; the first step is computed meanwhile.
                            a_ok = __all_sync(0xffffffffu, bounded_wait(a_empty, a_phase ^ 1u, w, SITE_DW_AEMPTY));
                        }
                        if (act && a_ok) {
                            const int pi = 2 * rp * W + x;
                            const uint2 o = make_uint2(pack_bf16x2(acc0[0], acc0[1]), pack_bf16x2(acc0[2], acc0[3]));
                            *reinterpret_cast<uint2 *>(sA + atom * (kBM * 128) + pi * 128 + ((chunk ^ (pi & 7)) << 4) +
                                                       half) = o;
                            if (two) {
                                const int pj = pi + W;
                                const uint2 o1 = make_uint2(pack_bf16x2(acc1[0], acc1[1]), pack_bf16x2(acc1[2], acc1[3]));
                                *reinterpret_cast<uint2 *>(sA + atom * (kBM * 128) + pj * 128 + ((chunk ^ (pj & 7)) << 4) +
                                                           half) = o1;
                            }
                        }
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            c0[k] = c1[k];
                            c1[k] = c2[k];
                        }
                    }
                    __syncwarp();
                }
            };
            if (interior)
                run(std::false_type{});
            else
                run(std::true_type{});
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(a_full);
            a_phase ^= 1u;
            dw_advance(p, pos);
        }
        __syncwarp();
    } else if (warp == kRMmaWarp) {
        // ------------------------------------------------ weights + MMA issuer
        if (lane == 0) {
            // Ring loader: rows go in order from the first tile's first row,
            // row r to slot (r - first_row) mod kRing.  Once the producers
            // are done with tile j, the rows below tile j + 1's first row are
            // free, and the rows tile j + 2 needs are loaded.
            const uint32_t row_tx = static_cast<uint32_t>(W * Cin * 2);
            DwTilePos cur = dw_pos(p, tb);
            const int first_row = tb < te ? dw_lo(p, cur) : 0;
            int next_issue = first_row, is_slot = 0;
            uint32_t is_round = 0;
            auto load_rows = [&](int last, int free_below) {
                while (next_issue <= last && next_issue - kRing < free_below) {
                    mbar_arrive_expect_tx(&ring_full[is_slot], row_tx);
                    bulk_load(ring + is_slot * p.row_bytes, p.x + static_cast<size_t>(next_issue) * W * Cin,
                              row_tx, &ring_full[is_slot]);
                    ++next_issue;
                    if (++is_slot == kRing) {
                        is_slot = 0;
                        ++is_round;
                    }
                }
            };
            if (tb < te) {
                DwTilePos nx = cur;
                dw_advance(p, nx);
                load_rows(tb + 1 < te ? dw_hi(p, nx) : dw_hi(p, cur), dw_lo(p, cur));
            }
            bool ok = true;
            tma_prefetch_desc(&tmW);
            mbar_arrive_expect_tx(wbar, static_cast<uint32_t>(p.kb * p.nchunks * 8192));
            for (int kb = 0; kb < p.kb; ++kb)
                for (int c = 0; c < p.nchunks; ++c)
                    tma_load_2d(&tmW, wbar, sW + (kb * p.nchunks + c) * 8192, c * 64, kb * 64);
            ok = bounded_wait(wbar, 0, w, SITE_DW_W);
            const uint32_t idesc = idesc_bf16_f32(kBM, Cout, false, true);
            const int ksteps = Cin / 16;
            int acc = 0;
            uint32_t phase = 0, acc_phase = 0;
            for (int tile = tb; ok && tile < te; ++tile) {
                if (!bounded_wait(&tempty[acc], acc_phase ^ 1u, w, SITE_DW_TEMPTY)) break;
                if (!bounded_wait(a_full, phase, w, SITE_DW_AFULL)) break;
                tc_fence_after();
                const uint32_t a0 = smem_u32(sA);
                const uint32_t w0 = smem_u32(sW);
                const uint32_t d = tmem_base + static_cast<uint32_t>(acc * ncols);
                for (int ks = 0; ks < ksteps; ++ks) {
                    const int atom = ks >> 2, kk = ks & 3;
                    const uint64_t ad = sdesc_sw128(a0 + atom * (kBM * 128) + kk * 32, 16, 1024);
                    const uint64_t bd = sdesc_sw128(w0 + atom * (p.nchunks * 8192) + kk * 2048, 8192, 1024);
                    umma_bf16(d, ad, bd, idesc, ks > 0 ? 1u : 0u);
                }
                umma_commit(a_empty);
                umma_commit(&tfull[acc]);
                phase ^= 1u;
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
                if (tile + 1 < te) {
                    DwTilePos n1 = cur;
                    dw_advance(p, n1);
                    DwTilePos n2 = n1;
                    dw_advance(p, n2);
                    load_rows(tile + 2 < te ? dw_hi(p, n2) : dw_hi(p, n1), dw_lo(p, n1));
                }
                dw_advance(p, cur);
            }
            // Let every row copy already issued land before the CTA can exit.
            int sl = is_slot;
            uint32_t rnd = is_round;
            for (int i = 0; i < kRing && next_issue - 1 - i >= first_row; ++i) {
                if (sl == 0) {
                    sl = kRing - 1;
                    --rnd;
                } else {
                    --sl;
                }
                const uint32_t a = smem_u32(&ring_full[sl]);
                const unsigned long long t0 = globaltimer();
                while (!mbar_try_wait(a, rnd & 1u))
                    if (globaltimer() - t0 > p.timeout_ns) break;
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------ epilogue (warps 12-19)
        // Two warps per TMEM lane quarter q, taking alternate 32-column
        // chunks: twice the TMEM loads in flight of one warp per quarter (a
        // warp's chain tcgen05.ld -> staging -> TMA store sets the pace), with
        // one 4 KB staging buffer each (the same 32 KB as two per warp).
        const int q = warp & 3;
        const int ew = warp - kREpiWarp0;
        const int c_first = (ew >> 2) * 32;  // this warp's first column chunk; it then takes every second
        uint8_t *sb = sStage + ew * 4096;
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int tile = tb; tile < te; ++tile) {
            bool tok = true;
            if (lane == 0) tok = bounded_wait(&tfull[acc], acc_phase, w, SITE_DW_TFULL);
            __syncwarp();
            // The epilogue warps decide together and leave the wait joined.
            if (!named_bar_and(3, 32 * kREpiWarps, tok)) break;
            tc_fence_after();
            int n, y0, y1, lo, hi;
            tile_rows(p, tile, n, y0, y1, lo, hi);
            const int npix = (y1 - y0 + 1) * W;
            const int nv = min(32, max(0, npix - q * 32));  // valid rows of this quadrant
            const long long row0 = (static_cast<long long>(n) * H + y0) * W + q * 32;
            const uint32_t tb_addr = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                     static_cast<uint32_t>(acc * ncols);
            // The TMEM load of the next chunk is issued as soon as the current
            // one sits in the staging buffer, so its latency overlaps the store.
            uint32_t r[32];
            if (nv > 0 && c_first < Cout) {
                if (Cout - c_first >= 32)
                    tmem_ld32(tb_addr + c_first, r);
                else
                    tmem_ld16(tb_addr + c_first, *reinterpret_cast<uint32_t (*)[16]>(&r[0]));
            }
            for (int c = c_first; c < Cout && nv > 0; c += 64) {
                tmem_ld_wait(r);
                if (lane == 0) bulk_wait_read<0>();  // the previous store has read the buffer
                __syncwarp();
#pragma unroll
                for (int ch = 0; ch < 8; ++ch) {
                    const int pos = ch ^ (lane & 7);
                    *reinterpret_cast<uint4 *>(sb + lane * 128 + pos * 16) =
                        make_uint4(r[4 * ch], r[4 * ch + 1], r[4 * ch + 2], r[4 * ch + 3]);
                }
                if (c + 64 < Cout) {
                    if (Cout - c - 64 >= 32)
                        tmem_ld32(tb_addr + c + 64, r);
                    else
                        tmem_ld16(tb_addr + c + 64, *reinterpret_cast<uint32_t (*)[16]>(&r[0]));
                }
                if (nv == 32) {
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_2d(&tmOut, sb, c, static_cast<int>(row0));
                        bulk_commit();
                    }
                } else {
                    // Partial quadrant (the tile ends inside it): its first
                    // 16 and/or 8 rows by TMA (boxes of 16 and 8 rows), the
                    // rest (fewer than 8) by plain coalesced row stores.
                    const int r16 = nv >= 16 ? 16 : 0;
                    const int r8 = nv - r16 >= 8 ? 8 : 0;
                    if (r16 + r8 > 0) {
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            if (r16) tma_store_2d(&tmOut16, sb, c, static_cast<int>(row0));
                            if (r8) tma_store_2d(&tmOut8, sb + r16 * 128, c, static_cast<int>(row0) + r16);
                            bulk_commit();
                        }
                    }
                    __syncwarp();
                    const int cols = min(32, Cout - c);
                    for (int rr = r16 + r8; rr < nv; ++rr) {
                        if (lane < cols) {
                            const int pos = (lane >> 2) ^ (rr & 7);
                            const float v = *reinterpret_cast<const float *>(sb + rr * 128 + pos * 16 + (lane & 3) * 4);
                            p.out[(row0 + rr) * p.ldo + c + lane] = v;
                        }
                    }
                    __syncwarp();
                }
                __syncwarp();  // joined again before the next aligned tcgen05.ld
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
            __syncwarp();
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        if (lane == 0) bulk_wait_all<0>();
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == kRMmaWarp) {
        tc_fence_after();
        tmem_dealloc(tmem_base, tmem_cols);
    }
}

// Image rows per tile of the row-ring kernel for a block of pc output
// channels, or 0 where that kernel does not apply (an image wider than one
// MMA block, a channel count its thread mapping does not divide, or no ring
// that fits shared memory beside the block's weights).
int dw_rows_per_tile(int W, int Cin, int pc, int smem_optin) {
    int rt = (W <= kBM && Cin / 4 <= kRProd) ? kBM / W : 0;
    if (rt > (kRingMax - 2) / 2) rt = (kRingMax - 2) / 2;
    while (rt > 1 && dw_row_layout(W, Cin, pc, 2 * rt + 2).total > smem_optin) --rt;
    return (rt >= 1 && dw_row_layout(W, Cin, pc, 2 * rt + 2).total <= smem_optin) ? rt : 0;
}

bool dw_block_fits(int W, int Cin, int pc, int smem_optin) {
    return dw_rows_per_tile(W, Cin, pc, smem_optin) > 0 || dw_layout(Cin, pc).total <= smem_optin;
}

// One launch for output channels c0 .. c0 + pc - 1 of a layer with Cout
// channels: the block's columns of pw_w and out, addressed with the layer's
// full row pitches.
int dwsep_block(int N, int H, int W, int Cin, int Cout, int c0, int pc, const uint16_t *x, const uint16_t *dw,
                const uint16_t *pw, float *out, DeviceState &ds, cudaStream_t stream) {
    const long long M = static_cast<long long>(N) * H * W;
    const uint16_t *pwb = pw + c0;
    float *outb = out + c0;
    int rc;
    const int rt = dw_rows_per_tile(W, Cin, pc, ds.max_smem_optin);
    if (rt > 0) {
        // Row-ring path: rt image rows per tile, 2 * rt + 2 rows resident.
        const DwRowLayout RL = dw_row_layout(W, Cin, pc, 2 * rt + 2);
        CUtensorMap tmW, tmOut, tmOut16, tmOut8;
        if ((rc = make_tmap_2d_bf16(&tmW, pwb, static_cast<uint64_t>(pc), static_cast<uint64_t>(Cin),
                                    static_cast<uint64_t>(Cout) * 2, 64, 64)))
            return rc;
        // Output boxes of 32 columns x 32, 16 and 8 rows.
        CUtensorMap *outs[3] = {&tmOut, &tmOut16, &tmOut8};
        for (int i = 0; i < 3; ++i)
            if ((rc = make_tmap_2d_f32(outs[i], outb, static_cast<uint64_t>(pc), static_cast<uint64_t>(M),
                                       static_cast<uint64_t>(Cout) * 4, 32, 32u >> i)))
                return rc;
        DwRowParams q{};
        q.N = N;
        q.H = H;
        q.W = W;
        q.Cin = Cin;
        q.Cout = pc;
        q.rt = rt;
        q.ring = 2 * rt + 2;
        q.tiles_per_img = (H + q.rt - 1) / q.rt;
        q.tiles = N * q.tiles_per_img;
        q.kb = (Cin + 63) / 64;
        q.nchunks = (pc + 63) / 64;
        q.row_bytes = dw_ring_row_bytes(W, Cin);
        q.x = x;
        q.dw = dw;
        q.out = outb;
        q.ldo = Cout;
        q.timeout_ns = wait_timeout_ns();
        q.err = ds.err_word;
        if ((rc = ensure_smem_optin(reinterpret_cast<const void *>(dwsep_rows_kernel), ds.max_smem_optin, ds.device,
                                    "cudaFuncSetAttribute(dwsep rows)")))
            return rc;
        const int grid = q.tiles < ds.num_sms ? q.tiles : ds.num_sms;
        dwsep_rows_kernel<<<grid, kRThreads, RL.total, stream>>>(tmW, tmOut, tmOut16, tmOut8, q);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return cuda_error(e, "launch dwsep_rows_kernel");
        return ISAM_OK;
    }
    const DwLayout L = dw_layout(Cin, pc);
    if (L.total > ds.max_smem_optin)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_dwsep_conv: Cin=%d with %d output channels per launch does not fit shared memory",
                         Cin, pc);
    CUtensorMap tmW, tmOut;
    if ((rc = make_tmap_2d_bf16(&tmW, pwb, static_cast<uint64_t>(pc), static_cast<uint64_t>(Cin),
                                static_cast<uint64_t>(Cout) * 2, 64, 64)))
        return rc;
    if ((rc = make_tmap_2d_f32(&tmOut, outb, static_cast<uint64_t>(pc), static_cast<uint64_t>(M),
                               static_cast<uint64_t>(Cout) * 4, 32, 32)))
        return rc;
    DwParams p{};
    p.N = N;
    p.H = H;
    p.W = W;
    p.Cin = Cin;
    p.Cout = pc;
    p.M = M;
    p.tiles = static_cast<int>((M + kBM - 1) / kBM);
    p.atoms = (Cin + 63) / 64;
    p.kb = (Cin + 63) / 64;
    p.nchunks = (pc + 63) / 64;
    p.x = x;
    p.dw = dw;
    p.timeout_ns = wait_timeout_ns();
    p.err = ds.err_word;
    if ((rc = ensure_smem_optin(reinterpret_cast<const void *>(dwsep_fused_kernel), ds.max_smem_optin, ds.device,
                                "cudaFuncSetAttribute(dwsep)")))
        return rc;
    const int grid = p.tiles < ds.num_sms ? p.tiles : ds.num_sms;
    dwsep_fused_kernel<<<grid, kThreads, L.total, stream>>>(tmW, tmOut, p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "launch dwsep_fused_kernel");
    return ISAM_OK;
}

}  // namespace

// Output channels in blocks of pc (a multiple of 16): the widest block whose
// resident pointwise weights fit shared memory beside the A tiles, the input
// ring and the epilogue staging.  Returns the block width, 0 if none fits.
int dw_block_width(int W, int Cin, int Cout, int smem_optin) {
    for (int blocks = 1; blocks <= Cout / 16; ++blocks) {
        const int pc = ((Cout + blocks - 1) / blocks + 15) / 16 * 16;
        if (dw_block_fits(W, Cin, pc, smem_optin)) return pc;
    }
    return 0;
}

int dwsep_plan(int W, int Cin, int Cout, int smem_optin, int *out) {
    if (Cin % 16 != 0 || Cin < 16 || Cin > 256 || Cout % 16 != 0 || Cout < 16 || Cout > 256)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_dwsep_plan_info: needs Cin and Cout multiples of 16 in [16, 256]");
    const int pc = dw_block_width(W, Cin, Cout, smem_optin);
    if (pc < 1) return set_error(ISAM_ERR_UNSUPPORTED, "isam_dwsep_plan_info: Cin=%d does not fit shared memory", Cin);
    const int rt = dw_rows_per_tile(W, Cin, pc, smem_optin);
    out[0] = rt > 0 ? 0 : 1;
    out[1] = rt;
    out[2] = (Cout + pc - 1) / pc;
    out[3] = pc;
    return ISAM_OK;
}

int dwsep_launch(int N, int H, int W, int Cin, int Cout, const uint16_t *x, const uint16_t *dw,
                 const uint16_t *pw, float *out, DeviceState &ds, cudaStream_t stream) {
    if (Cin % 16 != 0 || Cin < 16 || Cin > 256 || Cout % 16 != 0 || Cout < 16 || Cout > 256)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_dwsep_conv: needs Cin and Cout multiples of 16 in [16, 256] "
                         "(Cin=%d Cout=%d)",
                         Cin, Cout);
    if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(dw) |
         reinterpret_cast<uintptr_t>(pw) | reinterpret_cast<uintptr_t>(out)) & 15u)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_dwsep_conv: pointers must be 16-byte aligned");
    const long long M = static_cast<long long>(N) * H * W;
    if (M > (1ll << 31) - 256)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_dwsep_conv: N*H*W too large");
    // One channel block at the benchmark layer; wide layers (Cin = Cout =
    // 256, say) take several launches, each of which recomputes the
    // depthwise stage for its block.
    const int pc = dw_block_width(W, Cin, Cout, ds.max_smem_optin);
    if (pc < 1) return set_error(ISAM_ERR_UNSUPPORTED, "isam_dwsep_conv: Cin=%d does not fit shared memory", Cin);
    for (int c0 = 0; c0 < Cout; c0 += pc) {
        const int rc = dwsep_block(N, H, W, Cin, Cout, c0, std::min(pc, Cout - c0), x, dw, pw, out, ds, stream);
        if (rc != ISAM_OK) return rc;
    }
    return ISAM_OK;
}

}  // namespace isam
