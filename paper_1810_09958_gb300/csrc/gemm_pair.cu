// gemm_pair.cu -- large-tile GEMM on pairs of SMs (tcgen05 cta_group::2).
//
// The one-SM kernel's 128 x 256 tile streams, per K = 16 step, 4 KB of A and
// 8 KB of B out of one SM's shared memory into its tensor core.  Here the two
// CTAs of a cluster compute one 256 x 256 tile together: each keeps 128 rows
// of A and 128 of the 256 columns of B in its own shared memory (same
// offsets), and one thread of the first CTA issues M = 256 MMAs that read the
// A rows and B columns of both CTAs; each SM's 128 rows of the accumulator land
// in its own TMEM.  Per SM and K step the operands are 4 KB of A and 4 KB of B
// for the same 128 x 256 outputs, and each byte of B is loaded from L2 once
// per pair instead of twice.  This is the paper's mapping of a larger logical
// matrix instruction onto a set of physical units (Sections 2.4 and 3.3),
// with the pair as the unit.
//
// Roles in both CTAs: warp 0 TMA producer (its copies complete on the first
// CTA's stage barrier, which expects the bytes of both), warp 1 (first CTA
// only) MMA issuer whose commits arrive on the stage-free and
// accumulator-full barriers of both CTAs, warps 2-5 epilogue draining this
// CTA's half of the accumulator through swizzled staging to TMA stores (C
// prefetched when beta != 0) and releasing the accumulator on the first CTA's
// barrier.  Every wait is bounded.
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "gemm_common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace isam {

namespace {

constexpr int kPM = 256;                    // tile rows per pair
constexpr int kPN = 256;                    // tile columns per pair
constexpr int kHalf = 128;                  // rows of A / columns of B per CTA
constexpr int kBK = 64;
constexpr int kThreads = 192;
constexpr int kAStage = kHalf * kBK * 2;    // 16 KB
constexpr int kBStage = kHalf * kBK * 2;    // 16 KB
constexpr int kEpiBytes = 4 * 2 * 4096;     // per epilogue warp 2 x 32x32 fp32 staging
constexpr uint32_t kTmemCols = 2 * kPN;     // double-buffered accumulator: all 512 columns
constexpr uint16_t kBoth = 0x3;

enum : uint32_t {
    SITE_P_EMPTY = 0x501,
    SITE_P_FULL = 0x502,
    SITE_P_TEMPTY = 0x503,
    SITE_P_TFULL = 0x504,
    SITE_P_CLOAD = 0x505,
    SITE_P_DONE = 0x506,
};

struct PairParams {
    int M, N, K;
    int m_tiles, n_tiles, kb_total;
    int stages, group_m;
    float alpha, beta;
    const float *bias;
    unsigned long long timeout_ns;
    uint32_t *err;
};

__device__ __forceinline__ void pair_tile_coords(int tile, int m_tiles, int n_tiles, int group_m, int &mt,
                                                 int &nt) {
    const int per_group = group_m * n_tiles;
    const int g = tile / per_group;
    const int first_m = g * group_m;
    const int gm = min(group_m, m_tiles - first_m);
    const int local = tile - g * per_group;
    mt = first_m + local % gm;
    nt = local / gm;
}

template <bool B_MN>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ CUtensorMap tmC, const PairParams p) {
    if (!launch_shape_ok(p.err, 2u, gridDim.x, 0x5F0u)) return;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    const int ST = p.stages;
    uint8_t *sA = smem;
    uint8_t *sB = smem + static_cast<size_t>(ST) * kAStage;
    uint8_t *ebuf = sB + static_cast<size_t>(ST) * kBStage;
    uint64_t *bars = reinterpret_cast<uint64_t *>(ebuf + kEpiBytes);
    uint64_t *full = bars;              // [ST] first CTA: both CTAs' copies of a stage landed
    uint64_t *empty = full + ST;        // [ST] both: the pair's MMAs have read the stage
    uint64_t *tfull = empty + ST;       // [2] both: accumulator complete
    uint64_t *tempty = tfull + 2;       // [2] first CTA: 8 epilogue warps released it
    uint64_t *cbar = tempty + 2;        // [4 warps][2] C prefetch
    uint64_t *done = cbar + 8;          // local epilogue warps finished with TMEM
    uint64_t *mq = done + 1;            // first CTA: all its MMAs complete
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(mq + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    const int pair = blockIdx.x >> 1;
    const int num_pairs = gridDim.x >> 1;
    const int num_tiles = p.m_tiles * p.n_tiles;

    if (threadIdx.x == 0) {
        for (int i = 0; i < ST; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 8);
        }
        for (int i = 0; i < 8; ++i) mbar_init(&cbar[i], 1);
        mbar_init(done, 4);
        mbar_init(mq, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
        tma_prefetch_desc(&tmC);
    }
    __syncwarp();
    if (warp == 1) {
        tmem_alloc_pair(tmem_slot, kTmemCols);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();  // both CTAs' barriers and TMEM exist before any cross-CTA traffic
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx w{p.timeout_ns, p.err, abort_flag};

    griddep_launch_dependents();
    griddep_wait();

    bool aborted = false;
    if (warp == 0) {
        // ------------------------------------------------ TMA producer (both CTAs)
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int tile = pair; ok && tile < num_tiles; tile += num_pairs) {
                int mt, nt;
                pair_tile_coords(tile, p.m_tiles, p.n_tiles, p.group_m, mt, nt);
                const int arow = mt * kPM + static_cast<int>(rank) * kHalf;
                const int bcol = nt * kPN + static_cast<int>(rank) * kHalf;
                for (int kb = 0; kb < p.kb_total; ++kb) {
                    if (!bounded_wait<true>(&empty[stage], phase ^ 1u, w, SITE_P_EMPTY)) {
                        ok = false;
                        break;
                    }
                    if (leader) mbar_arrive_expect_tx(&full[stage], 2u * (kAStage + kBStage));
                    const uint32_t fb = mapa_shared(smem_u32(&full[stage]), 0u);
                    uint8_t *a = sA + static_cast<size_t>(stage) * kAStage;
                    uint8_t *b = sB + static_cast<size_t>(stage) * kBStage;
                    const int k0 = kb * kBK;
                    tma_load_2d_pair(&tmA, fb, a, k0, arow);
                    if (B_MN) {
                        tma_load_2d_pair(&tmB, fb, b, bcol, k0);
                        tma_load_2d_pair(&tmB, fb, b + 8192, bcol + 64, k0);
                    } else {
                        tma_load_2d_pair(&tmB, fb, b, k0, bcol);
                    }
                    if (++stage == ST) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            aborted = !ok;
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer (first CTA)
        if (lane == 0 && leader) {
            const uint32_t idesc = idesc_bf16_f32(kPM, kPN, false, B_MN);
            int stage = 0, acc = 0;
            uint32_t phase = 0, acc_phase = 0;
            bool ok = true, issued = false;
            for (int tile = pair; ok && tile < num_tiles; tile += num_pairs) {
                if (!bounded_wait<true>(&tempty[acc], acc_phase ^ 1u, w, SITE_P_TEMPTY)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(acc * kPN);
                for (int kb = 0; kb < p.kb_total; ++kb) {
                    if (!bounded_wait<true>(&full[stage], phase, w, SITE_P_FULL)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(sA + static_cast<size_t>(stage) * kAStage);
                    const uint32_t b0 = smem_u32(sB + static_cast<size_t>(stage) * kBStage);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k) {
                        const uint64_t ad = sdesc_sw128(a0 + k * 32, 16, 1024);
                        const uint64_t bd = B_MN ? sdesc_sw128(b0 + k * 2048, 8192, 1024)
                                                 : sdesc_sw128(b0 + k * 32, 16, 1024);
                        umma_bf16_pair(d, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                    }
                    issued = true;
                    umma_commit_pair(&empty[stage], kBoth);
                    if (++stage == ST) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                umma_commit_pair(&tfull[acc], kBoth);
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
            }
            // Every MMA of this thread has completed before TMEM can be freed.
            if (issued) {
                umma_commit_pair(mq, 0x1);
                drain_wait(mq, 0, p.timeout_ns);
            }
            aborted = !ok;
        }
        __syncwarp();
    } else {
        // ------------------------------------------------ epilogue (warps 2-5, both CTAs)
        const int ew = warp - 2;
        const int q = warp & 3;  // TMEM lane quadrant this warp may read
        uint8_t *stg = ebuf + ew * 8192;
        uint64_t *cb = cbar + ew * 2;
        uint32_t cpar[2] = {0u, 0u};
        bool cpend[2] = {false, false};
        const bool load_c = p.beta != 0.0f;
        int gbuf = 0, acc = 0;
        uint32_t acc_phase = 0;
        bool ok = true;
        for (int tile = pair; tile < num_tiles; tile += num_pairs) {
            int mt, nt;
            pair_tile_coords(tile, p.m_tiles, p.n_tiles, p.group_m, mt, nt);
            const int row0 = mt * kPM + static_cast<int>(rank) * kHalf + q * 32;
            const int col0 = nt * kPN;
            if (load_c) {
                // Prefetch the first C chunk of this tile while its MMAs run.
                if (lane == 0) {
                    bulk_wait_read<0>();
                    const int b = gbuf & 1;
                    mbar_arrive_expect_tx(&cb[b], 4096);
                    tma_load_2d(&tmC, &cb[b], stg + b * 4096, col0, row0);
                }
                cpend[gbuf & 1] = true;
                __syncwarp();
            }
            if (!warp_wait<true>(&tfull[acc], acc_phase, w, SITE_P_TFULL)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                   static_cast<uint32_t>(acc * kPN);
#pragma unroll 1
            for (int j = 0; j < kPN / 32; ++j) {
                const int b = gbuf & 1;
                if (load_c && j + 1 < kPN / 32) {
                    if (lane == 0) {
                        bulk_wait_read<0>();  // buffer b^1: its last store has read it
                        mbar_arrive_expect_tx(&cb[b ^ 1], 4096);
                        tma_load_2d(&tmC, &cb[b ^ 1], stg + (b ^ 1) * 4096, col0 + (j + 1) * 32, row0);
                    }
                    cpend[b ^ 1] = true;
                }
                if (!load_c && lane == 0) bulk_wait_read<1>();  // buffer b: store of 2 chunks ago
                uint32_t r[32];
                tmem_ld32(tbase + j * 32, r);
                tmem_ld_wait(r);
                if (load_c) {
                    if (!warp_wait(&cb[b], cpar[b], w, SITE_P_CLOAD)) {
                        ok = false;
                        break;
                    }
                    cpar[b] ^= 1u;
                    cpend[b] = false;
                }
                __syncwarp();
                uint8_t *sb = stg + b * 4096;
                const int cbase = col0 + j * 32;
#pragma unroll
                for (int ch = 0; ch < 8; ++ch) {
                    const int pos = ch ^ (lane & 7);
                    float4 *slot = reinterpret_cast<float4 *>(sb + lane * 128 + pos * 16);
                    float4 v = make_float4(p.alpha * __uint_as_float(r[4 * ch]), p.alpha * __uint_as_float(r[4 * ch + 1]),
                                           p.alpha * __uint_as_float(r[4 * ch + 2]),
                                           p.alpha * __uint_as_float(r[4 * ch + 3]));
                    if (p.bias != nullptr && cbase + 4 * ch < p.N) {
                        const float4 bv = __ldg(reinterpret_cast<const float4 *>(p.bias + cbase + 4 * ch));
                        v.x += bv.x;
                        v.y += bv.y;
                        v.z += bv.z;
                        v.w += bv.w;
                    }
                    if (load_c) {
                        const float4 cv = *slot;
                        v.x += p.beta * cv.x;
                        v.y += p.beta * cv.y;
                        v.z += p.beta * cv.z;
                        v.w += p.beta * cv.w;
                    }
                    *slot = v;
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&tmC, sb, cbase, row0);
                    bulk_commit();
                }
                ++gbuf;
            }
            if (!ok) break;
            // Release this accumulator on the first CTA's barrier.
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote(&tempty[acc], 0u);
            __syncwarp();
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        for (int b = 0; b < 2; ++b)
            if (cpend[b] && lane == 0) drain_wait(&cb[b], cpar[b], p.timeout_ns);
        if (lane == 0) bulk_wait_all<0>();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(done);
        __syncwarp();
        aborted = !ok;
    }

    // ---- teardown.  After an abort, copies this CTA issued may still be in
    // flight towards its shared memory and complete on the first CTA's
    // barriers: give them time to land (bounded, only on that path).
    if (__syncthreads_or(aborted ? 1 : 0) && threadIdx.x == 0) {
        const unsigned long long t0 = globaltimer();
        while (globaltimer() - t0 < 50000ull) {
        }
    }
    if (warp == 1) bounded_wait(done, 0, w, SITE_P_DONE);
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    // Both CTAs' epilogues are done reading TMEM and the first CTA's MMAs have
    // completed before the pair releases its TMEM together.
    cluster_sync_all();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem_base, kTmemCols);
    }
}

using PairKernel = void (*)(CUtensorMap, CUtensorMap, CUtensorMap, PairParams);

size_t pair_smem_bytes(int stages) {
    return 1024 + static_cast<size_t>(stages) * (kAStage + kBStage) + kEpiBytes + (2 * stages + 15) * 8 + 16;
}


}  // namespace

int gemm_pair_plan(const GemmDesc &g, const DeviceState &ds, GemmPlan *plan) {
    if (g.fp8 || g.transA != 0 || g.N % 4 != 0 || g.K < 4 * kBK) return 0;
    if (const char *s = getenv("ISAM_NO_PAIR"))
        if (s[0] == '1') return 0;
    const long long tiles = static_cast<long long>((g.M + kPM - 1) / kPM) * ((g.N + kPN - 1) / kPN);
    const int pairs = gemm_cluster_capacity(ds, 2);  // pairs resident at once
    if (pairs < 1 || tiles < pairs) return 0;  // smaller problems spread better as 128-row tiles
    int st = 8;
    while (st > 2 && pair_smem_bytes(st) > static_cast<size_t>(ds.max_smem_optin)) --st;
    GemmPlan p{};
    p.BN = kPN;
    p.ka = 1;
    p.split = 1;
    p.stages = st;
    p.group_m = 8;
    p.grid = static_cast<int>(std::min<long long>(tiles, pairs)) * 2;
    p.smem = pair_smem_bytes(st);
    p.pair = 1;
    p.est_us = 0.0;
    *plan = p;
    return 1;
}

int gemm_pair_launch(const GemmDesc &g, const GemmPlan &plan, DeviceState &ds, cudaStream_t stream) {
    const bool b_mn = g.transB == 0;
    CUtensorMap ta, tb, tc;
    int rc;
    if ((rc = make_tmap_2d_bf16(&ta, g.A, g.K, g.M, static_cast<uint64_t>(g.K) * 2, 64, kHalf))) return rc;
    if (b_mn)
        rc = make_tmap_2d_bf16(&tb, g.B, g.N, g.K, static_cast<uint64_t>(g.N) * 2, 64, 64);
    else
        rc = make_tmap_2d_bf16(&tb, g.B, g.K, g.N, static_cast<uint64_t>(g.K) * 2, 64, kHalf);
    if (rc) return rc;
    if ((rc = make_tmap_2d_f32(&tc, g.C, g.N, g.M, static_cast<uint64_t>(g.N) * 4, 32, 32))) return rc;

    PairParams p{};
    p.M = g.M;
    p.N = g.N;
    p.K = g.K;
    p.m_tiles = (g.M + kPM - 1) / kPM;
    p.n_tiles = (g.N + kPN - 1) / kPN;
    p.kb_total = (g.K + kBK - 1) / kBK;
    p.stages = plan.stages;
    p.group_m = plan.group_m;
    p.alpha = g.alpha;
    p.beta = g.beta;
    p.bias = g.bias_n;
    p.timeout_ns = wait_timeout_ns();
    p.err = ds.err_word;

    const PairKernel fn = b_mn ? gemm_pair_kernel<true> : gemm_pair_kernel<false>;
    {
        const int rc = ensure_smem_optin(reinterpret_cast<const void *>(fn), ds.max_smem_optin, ds.device,
                                         "cudaFuncSetAttribute(gemm pair)");
        if (rc) return rc;
    }
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.gridDim = dim3(static_cast<unsigned>(plan.grid), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = plan.smem;
    cfg.stream = stream;
    cfg.attrs = attr;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 2;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.numAttrs = 2;
    cudaError_t e = cudaLaunchKernelEx(&cfg, fn, ta, tb, tc, p);
    if (e != cudaSuccess) return cuda_error(e, "launch gemm_pair_kernel");
    return ISAM_OK;
}

}  // namespace isam
