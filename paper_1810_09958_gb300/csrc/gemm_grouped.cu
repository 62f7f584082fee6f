// gemm_grouped.cu -- many independent GEMMs in one persistent tcgen05 launch.
//
// The tiles of every problem form one list that the persistent CTAs walk
// round-robin (problems ordered by decreasing tile cost on the host), so the
// SMs stream the operands of several problems at once and the per-launch costs
// -- pipeline fill to the first data, the last tile's epilogue, the gap
// between kernels -- are paid once for the whole group instead of once per
// problem.  This is the paper's scheduler placing compute tiles across compute
// units (Sections 3.3-3.4) applied across a set of matrix multiplications.
//
// Per CTA: warp 0 TMA producer, warp 1 single-thread tcgen05.mma issuer into a
// double-buffered TMEM accumulator, warps 2-5 epilogue storing C straight
// from TMEM (16-byte stores, or single floats when a row of C is not 16-byte
// aligned).  Layout (NN/TN/NT/TT) and tile width are per problem; a problem's
// tensor maps travel in the kernel parameters.
#include <algorithm>
#include <cstdlib>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <numeric>

#include "gemm_common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace isam {

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kThreads = 192;
constexpr int kMaxGroup = 64;
constexpr int kBNMax = 128;
constexpr int kAStage = kBM * kBK * 2;      // 16 KB
constexpr int kBStage = kBNMax * kBK * 2;   // 16 KB (either B layout at BN = 128)

enum : uint32_t {
    SITE_G_EMPTY = 0x401,
    SITE_G_TEMPTY = 0x402,
    SITE_G_FULL = 0x403,
    SITE_G_TFULL = 0x404,
    SITE_G_CLOAD = 0x405,
    SITE_G_DONE = 0x406,
};

struct GroupProblem {
    int M, N, K;
    int m_tiles, n_tiles, kb_total;
    int a_mn, b_mn, bn;
    int panels;       // 128-row A panels per tile: 1, or 2 (256-row tiles for the heavy problems)
    int fp8;          // E4M3 operands (both K-major): 128-element K atoms
    int tile_start;   // first global tile index of this problem
    float alpha, beta;
    float *C;
};

struct GroupParams {
    int count, total_tiles, stages;
    unsigned long long timeout_ns;
    uint32_t *err;
    GroupProblem prob[kMaxGroup];
    CUtensorMap tmA[kMaxGroup];
    CUtensorMap tmB[kMaxGroup];
};

// The problem that owns `tile`, searched forward from `i` (a CTA visits its
// tiles in increasing order, so each role keeps its index and the search
// advances by at most a few entries per tile instead of rescanning the table
// in parameter space).  Each role then copies the problem's fields into
// registers for the tile: through a reference the fields are read again from
// parameter space after every inline-asm statement with a memory clobber
// (each TMA, MMA and barrier operation), on the issue path of every k-block
// -- the copy made the sweep 3.5% faster.
__device__ __forceinline__ int find_problem(const GroupParams &p, int tile, int i) {
    while (i + 1 < p.count && p.prob[i + 1].tile_start <= tile) ++i;
    return i;
}

__global__ void __launch_bounds__(kThreads, 1) gemm_group_kernel(const __grid_constant__ GroupParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    const int ST = p.stages;
    uint8_t *sA = smem;
    uint8_t *sB = smem + static_cast<size_t>(ST) * kAStage;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sB + static_cast<size_t>(ST) * kBStage);
    uint64_t *full = bars;
    uint64_t *empty = bars + ST;
    uint64_t *tfull = empty + ST;
    uint64_t *tempty = tfull + 2;
    uint64_t *done = tempty + 2;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    constexpr uint32_t kTmemCols = 4 * kBNMax;  // two accumulators of two 128-row panels

    if (threadIdx.x == 0) {
        for (int i = 0; i < ST; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        mbar_init(done, 4);
        *abort_flag = 0;
        fence_mbar_init();
    }
    __syncwarp();
    if (warp == 1) {
        tmem_alloc(tmem_slot, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx w{p.timeout_ns, p.err, abort_flag};

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0, issued = 0, pi = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < p.total_tiles; tile += gridDim.x) {
                pi = find_problem(p, tile, pi);
                const GroupProblem pr = p.prob[pi];  // a copy, see find_problem
                const int local = tile - pr.tile_start;
                const int mt = local % pr.m_tiles, nt = local / pr.m_tiles;
                const int panels = pr.panels;
                const uint32_t bbytes = pr.b_mn ? static_cast<uint32_t>((pr.bn + 63) / 64) * 8192u
                                                : static_cast<uint32_t>(pr.bn) * 128u;
                if (panels == 1) {
                    for (int kb = 0; kb < pr.kb_total; ++kb) {
                        if (!bounded_wait(&empty[stage], phase ^ 1u, w, SITE_G_EMPTY)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(&full[stage], static_cast<uint32_t>(kAStage) + bbytes);
                        uint8_t *a = sA + static_cast<size_t>(stage) * kAStage;
                        uint8_t *b = sB + static_cast<size_t>(stage) * kBStage;
                        const int k0 = kb * (pr.fp8 ? 2 * kBK : kBK);  // in elements
                        if (pr.a_mn) {
                            tma_load_2d(&p.tmA[pi], &full[stage], a, mt * kBM, k0);
                            tma_load_2d(&p.tmA[pi], &full[stage], a + 8192, mt * kBM + 64, k0);
                        } else {
                            tma_load_2d(&p.tmA[pi], &full[stage], a, k0, mt * kBM);
                        }
                        if (pr.b_mn) {
                            for (int c = 0; c < (pr.bn + 63) / 64; ++c)
                                tma_load_2d(&p.tmB[pi], &full[stage], b + c * 8192, nt * pr.bn + c * 64, k0);
                        } else {
                            tma_load_2d(&p.tmB[pi], &full[stage], b, k0, nt * pr.bn);
                        }
                        ++issued;
                        if (++stage == ST) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                    continue;
                }
                // A k-block of a 256-row tile takes two consecutive stages:
                // panel 0 and the B block in the first, panel 1 in the second.
                const int r0 = mt * 2 * kBM, r1 = r0 + kBM;
                for (int kb = 0; kb < pr.kb_total; ++kb) {
                    const int k0 = kb * (pr.fp8 ? 2 * kBK : kBK);  // in elements
                    if (!bounded_wait(&empty[stage], phase ^ 1u, w, SITE_G_EMPTY)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&full[stage], static_cast<uint32_t>(kAStage) + bbytes);
                    uint8_t *a = sA + static_cast<size_t>(stage) * kAStage;
                    uint8_t *b = sB + static_cast<size_t>(stage) * kBStage;
                    if (pr.a_mn) {
                        tma_load_2d(&p.tmA[pi], &full[stage], a, r0, k0);
                        tma_load_2d(&p.tmA[pi], &full[stage], a + 8192, r0 + 64, k0);
                    } else {
                        tma_load_2d(&p.tmA[pi], &full[stage], a, k0, r0);
                    }
                    if (pr.b_mn) {
                        for (int c = 0; c < (pr.bn + 63) / 64; ++c)
                            tma_load_2d(&p.tmB[pi], &full[stage], b + c * 8192, nt * pr.bn + c * 64, k0);
                    } else {
                        tma_load_2d(&p.tmB[pi], &full[stage], b, k0, nt * pr.bn);
                    }
                    ++issued;
                    if (++stage == ST) {
                        stage = 0;
                        phase ^= 1u;
                    }
                    if (!bounded_wait(&empty[stage], phase ^ 1u, w, SITE_G_EMPTY)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&full[stage], static_cast<uint32_t>(kAStage));
                    a = sA + static_cast<size_t>(stage) * kAStage;
                    if (pr.a_mn) {
                        tma_load_2d(&p.tmA[pi], &full[stage], a, r1, k0);
                        tma_load_2d(&p.tmA[pi], &full[stage], a + 8192, r1 + 64, k0);
                    } else {
                        tma_load_2d(&p.tmA[pi], &full[stage], a, k0, r1);
                    }
                    ++issued;
                    if (++stage == ST) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok) {
                const int pending = min(issued, ST);
                int s = stage;
                uint32_t ph = phase;
                for (int i = 0; i < pending; ++i) {
                    if (--s < 0) {
                        s = ST - 1;
                        ph ^= 1u;
                    }
                    drain_wait(&full[s], ph, p.timeout_ns);
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            int stage = 0, acc = 0, pi = 0;
            uint32_t phase = 0, acc_phase = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < p.total_tiles; tile += gridDim.x) {
                pi = find_problem(p, tile, pi);
                const GroupProblem pr = p.prob[pi];  // a copy, see find_problem
                const bool f8 = pr.fp8 != 0;
                const uint32_t idesc =
                    f8 ? idesc_e4m3_f32(kBM, pr.bn) : idesc_bf16_f32(kBM, pr.bn, pr.a_mn != 0, pr.b_mn != 0);
                if (!bounded_wait(&tempty[acc], acc_phase ^ 1u, w, SITE_G_TEMPTY)) break;
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(acc * 2 * kBNMax);
                if (pr.panels == 1) {
                    for (int kb = 0; kb < pr.kb_total; ++kb) {
                        if (!bounded_wait(&full[stage], phase, w, SITE_G_FULL)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t a0 = smem_u32(sA + static_cast<size_t>(stage) * kAStage);
                        const uint32_t b0 = smem_u32(sB + static_cast<size_t>(stage) * kBStage);
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            const uint64_t ad = pr.a_mn ? sdesc_sw128(a0 + k * 2048, 8192, 1024)
                                                        : sdesc_sw128(a0 + k * 32, 16, 1024);
                            const uint64_t bd = pr.b_mn ? sdesc_sw128(b0 + k * 2048, 8192, 1024)
                                                        : sdesc_sw128(b0 + k * 32, 16, 1024);
                            if (f8)
                                umma_f8(d, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                            else
                                umma_bf16(d, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                        }
                        umma_commit(&empty[stage]);
                        if (++stage == ST) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                } else {
                    // 256-row tile: each k-block spans two stages, panel 0
                    // with the B block, then panel 1; both panels multiply
                    // the first stage's B, so both stages are freed after
                    // the k-block's last MMA.
                    for (int kb = 0; kb < pr.kb_total; ++kb) {
                        const int s0 = stage;
                        if (!bounded_wait(&full[s0], phase, w, SITE_G_FULL)) {
                            ok = false;
                            break;
                        }
                        if (++stage == ST) {
                            stage = 0;
                            phase ^= 1u;
                        }
                        tc_fence_after();
                        const uint32_t a0 = smem_u32(sA + static_cast<size_t>(s0) * kAStage);
                        const uint32_t b0 = smem_u32(sB + static_cast<size_t>(s0) * kBStage);
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            const uint64_t ad = pr.a_mn ? sdesc_sw128(a0 + k * 2048, 8192, 1024)
                                                        : sdesc_sw128(a0 + k * 32, 16, 1024);
                            const uint64_t bd = pr.b_mn ? sdesc_sw128(b0 + k * 2048, 8192, 1024)
                                                        : sdesc_sw128(b0 + k * 32, 16, 1024);
                            if (f8)
                                umma_f8(d, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                            else
                                umma_bf16(d, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                        }
                        const int s1 = stage;
                        if (!bounded_wait(&full[s1], phase, w, SITE_G_FULL)) {
                            ok = false;
                            break;
                        }
                        if (++stage == ST) {
                            stage = 0;
                            phase ^= 1u;
                        }
                        tc_fence_after();
                        const uint32_t a1 = smem_u32(sA + static_cast<size_t>(s1) * kAStage);
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            const uint64_t ad = pr.a_mn ? sdesc_sw128(a1 + k * 2048, 8192, 1024)
                                                        : sdesc_sw128(a1 + k * 32, 16, 1024);
                            const uint64_t bd = pr.b_mn ? sdesc_sw128(b0 + k * 2048, 8192, 1024)
                                                        : sdesc_sw128(b0 + k * 32, 16, 1024);
                            if (f8)
                                umma_f8(d + kBNMax, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                            else
                                umma_bf16(d + kBNMax, ad, bd, idesc, (kb > 0 || k > 0) ? 1u : 0u);
                        }
                        umma_commit(&empty[s0]);
                        umma_commit(&empty[s1]);
                    }
                }
                if (!ok) break;
                umma_commit(&tfull[acc]);
                if (++acc == 2) {
                    acc = 0;
                    acc_phase ^= 1u;
                }
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------ epilogue (warps 2-5)
        const int q = warp & 3;
        // Straight from TMEM to C: lane i holds row i of the warp's 32 rows,
        // 32 consecutive columns per TMEM load, stored as 16-byte pieces (or
        // single floats where C's rows are not 16-byte aligned).  No staging
        // buffer: the 32 KB it took is a seventh ring stage, and the
        // epilogue, which overlaps the next tile's main loop through the
        // second accumulator, has time for the scattered stores.
        int acc = 0, pi = 0;
        uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < p.total_tiles; tile += gridDim.x) {
            pi = find_problem(p, tile, pi);
            const GroupProblem pr = p.prob[pi];  // a copy, see find_problem
            const int local = tile - pr.tile_start;
            const int mt = local % pr.m_tiles, nt = local / pr.m_tiles;
            const int col0 = nt * pr.bn;
            const int nch = (pr.bn + 31) / 32;
            const bool vec = (pr.N & 3) == 0;
            if (!warp_wait(&tfull[acc], acc_phase, w, SITE_G_TFULL)) break;
            tc_fence_after();
            for (int pn = 0; pn < pr.panels; ++pn) {
                const int grow = (mt * pr.panels + pn) * kBM + q * 32 + lane;
                const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                       static_cast<uint32_t>(acc * 2 * kBNMax + pn * kBNMax);
                for (int j = 0; j < nch; ++j) {
                    uint32_t r[32];
                    if (pr.bn - j * 32 >= 32) {
                        tmem_ld32(tbase + j * 32, r);
                    } else {
                        uint32_t h[16];
                        tmem_ld16(tbase + j * 32, h);
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            r[i] = h[i];
                            r[16 + i] = 0u;
                        }
                    }
                    tmem_ld_wait();
                    if (grow < pr.M) {
                        float *crow = pr.C + static_cast<size_t>(grow) * pr.N;
                        const int cbase = col0 + j * 32;
                        const int cend = min(pr.N, col0 + pr.bn);  // columns of this tile inside C
#pragma unroll
                        for (int ch = 0; ch < 8; ++ch) {
                            const int col = cbase + 4 * ch;
                            if (col >= cend) break;
                            float v[4];
#pragma unroll
                            for (int e = 0; e < 4; ++e) v[e] = pr.alpha * __uint_as_float(r[4 * ch + e]);
                            if (vec && col + 3 < cend) {
                                float4 *dst = reinterpret_cast<float4 *>(crow + col);
                                if (pr.beta != 0.0f) {
                                    const float4 cv = *dst;
                                    v[0] += pr.beta * cv.x;
                                    v[1] += pr.beta * cv.y;
                                    v[2] += pr.beta * cv.z;
                                    v[3] += pr.beta * cv.w;
                                }
                                *dst = make_float4(v[0], v[1], v[2], v[3]);
                            } else {
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    if (col + e >= cend) break;
                                    float x = v[e];
                                    if (pr.beta != 0.0f) x += pr.beta * crow[col + e];
                                    crow[col + e] = x;
                                }
                            }
                        }
                    }
                    __syncwarp();  // joined again before the next aligned tcgen05.ld
                }
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
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(done);
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        bounded_wait(done, 0, w, SITE_G_DONE);
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, kTmemCols);
    }
}

size_t group_smem_bytes(int stages) {
    return 1024 + static_cast<size_t>(stages) * (kAStage + kBStage) + (2 * stages + 5) * 8 + 16;
}

std::mutex g_group_mu;

}  // namespace

int gemm_grouped_launch(int count, const GemmDesc *g, DeviceState &ds, cudaStream_t stream) {
    if (count < 1 || count > kMaxGroup)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_grouped: count must be in [1, %d]", kMaxGroup);
    auto atoms = [&](int i) { return (g[i].K + (g[i].fp8 ? 2 * kBK : kBK) - 1) / (g[i].fp8 ? 2 * kBK : kBK); };
    // Tile height: 256 rows (two 128-row panels sharing each B block) for
    // problems whose 128-row panel of A is 640 KB or more, which halves the
    // tile starts a CTA pays on them; kept at 128 rows when that would leave
    // fewer than two tiles per SM.
    int panels[kMaxGroup];
    {
        long long tall_tiles = 0;
        for (int i = 0; i < count; ++i) {
            const long long eb = g[i].fp8 ? 1 : 2;
            panels[i] = (g[i].M > kBM && static_cast<long long>(kBM) * g[i].K * eb >= 640 * 1024) ? 2 : 1;
            const int bn = std::min(kBNMax, (g[i].N + 15) / 16 * 16);
            tall_tiles += static_cast<long long>((g[i].M + kBM * panels[i] - 1) / (kBM * panels[i])) *
                          ((g[i].N + bn - 1) / bn);
        }
        if (tall_tiles < 2LL * ds.num_sms)
            for (int i = 0; i < count; ++i) panels[i] = 1;
        // ISAM_GROUP_PANELS=1 or 2 forces the tile height (2: every problem
        // taller than one panel), for tests and measurements.
        const char *fe = getenv("ISAM_GROUP_PANELS");
        const int forced = fe ? atoi(fe) : 0;
        if (forced == 1 || forced == 2)
            for (int i = 0; i < count; ++i) panels[i] = (forced == 2 && g[i].M > kBM) ? 2 : 1;
    }
    // Host-side order: problems with the costliest tiles first, so the
    // round-robin walk over tiles ends with the cheap ones.
    int order[kMaxGroup];
    std::iota(order, order + count, 0);
    std::stable_sort(order, order + count,
                     [&](int a, int b) { return atoms(a) * panels[a] > atoms(b) * panels[b]; });

    static GroupParams p;  // ~29 KB: built under the lock, copied into the launch
    std::lock_guard<std::mutex> lk(g_group_mu);
    memset(&p, 0, sizeof p);
    p.count = count;
    int tiles = 0;
    for (int s = 0; s < count; ++s) {
        const GemmDesc &d = g[order[s]];
        GroupProblem &pr = p.prob[s];
        pr.M = d.M;
        pr.N = d.N;
        pr.K = d.K;
        pr.fp8 = d.fp8;
        pr.a_mn = d.fp8 ? 0 : d.transA;
        pr.b_mn = (d.fp8 || d.transB == 1) ? 0 : 1;
        pr.bn = std::min(kBNMax, (d.N + 15) / 16 * 16);
        pr.panels = panels[order[s]];
        pr.m_tiles = (d.M + kBM * pr.panels - 1) / (kBM * pr.panels);
        pr.n_tiles = (d.N + pr.bn - 1) / pr.bn;
        pr.kb_total = atoms(order[s]);
        pr.tile_start = tiles;
        pr.alpha = d.alpha;
        pr.beta = d.beta;
        pr.C = d.C;
        tiles += pr.m_tiles * pr.n_tiles;
        int rc;
        if (pr.fp8) {
            // 128-element (128-byte) K atoms of both K-major E4M3 operands.
            if ((rc = make_tmap_2d_u8(&p.tmA[s], d.A, d.K, d.M, static_cast<uint64_t>(d.K), 128, kBM))) return rc;
            if ((rc = make_tmap_2d_u8(&p.tmB[s], d.B, d.K, d.N, static_cast<uint64_t>(d.K), 128,
                                      static_cast<uint32_t>(pr.bn))))
                return rc;
        } else {
            if (pr.a_mn)
                rc = make_tmap_2d_bf16(&p.tmA[s], d.A, d.M, d.K, static_cast<uint64_t>(d.M) * 2, 64, 64);
            else
                rc = make_tmap_2d_bf16(&p.tmA[s], d.A, d.K, d.M, static_cast<uint64_t>(d.K) * 2, 64, kBM);
            if (rc) return rc;
            if (pr.b_mn)
                rc = make_tmap_2d_bf16(&p.tmB[s], d.B, d.N, d.K, static_cast<uint64_t>(d.N) * 2, 64, 64);
            else
                rc = make_tmap_2d_bf16(&p.tmB[s], d.B, d.K, d.N, static_cast<uint64_t>(d.K) * 2, 64,
                                       static_cast<uint32_t>(pr.bn));
            if (rc) return rc;
        }
    }
    p.total_tiles = tiles;
    int st = 8;
    while (st > 2 && group_smem_bytes(st) > static_cast<size_t>(ds.max_smem_optin)) --st;
    p.stages = st;
    p.timeout_ns = wait_timeout_ns();
    p.err = ds.err_word;
    const size_t smem = group_smem_bytes(st);
    if (const int rc = ensure_smem_optin(reinterpret_cast<const void *>(gemm_group_kernel), ds.max_smem_optin,
                                         ds.device, "cudaFuncSetAttribute(grouped gemm)"))
        return rc;
    const int grid = std::min(tiles, ds.num_sms);
    gemm_group_kernel<<<grid, kThreads, smem, stream>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "launch gemm_group_kernel");
    return ISAM_OK;
}

}  // namespace isam
