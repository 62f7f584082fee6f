// gemm_mx.cu -- block-scaled E4M3 GEMM (OCP Microscaling, "MX"): every 32
// consecutive K elements of a row of A, and of a row of B, share one E8M0
// scale 2^(e - 127).  C <- alpha * (SA o A) * (SB o B)^T + beta * C.
//
// The same matrix multiplication as the E4M3 kernels, mapped onto the tensor
// cores' block-scaled operand kind (tcgen05.mma kind::mxf8f6f4): the
// instruction applies the scales itself, so the scaled products never exist
// in memory -- the paper's instruction selection (Section 2.4) choosing the
// instruction whose semantics cover more of the computation.
//
// A persistent grid walks the tiles of one or more problems round-robin (as
// the grouped kernel does).  Per CTA:
//   warp 0      TMA producer: 128-row x 128-byte K atoms of A, BN x 128 of B;
//   warp 1      one thread issues the MMAs: four K = 32 instructions per atom,
//               scale-factor IDs 0..3 selecting the atom's four scale bytes;
//   warps 2-5   epilogue (TMEM -> alpha/beta -> C);
//   warps 6-9   scale writers: read the atom's E8M0 bytes from global memory
//               and store them into a ring of scale slots in tensor memory
//               (tcgen05.st; a warp reaches only its own 32-lane quarter).
//
// Scale slot layout (4 columns for A, then 4 for B; 32-bit cells whose bytes
// 0..3 are the atom's four 32-element blocks).  For B, lane 32q + r of column
// j holds row r + 32j of the tile, the same in every quarter q: each quarter
// of the tensor core multiplies its 32 rows of A by all of B's rows, from its
// own lanes.  For A, column 0 holds row m at lane m and columns 1..3 hold row
// r + 32j at lane 32q + r, which serves a quarter reading either its own rows
// at column 0 or column q.
//
// Scale bytes are taken atom-major: SA [ceil(K/128)][M][4], SB
// [ceil(K/128)][N][4], the four E8M0 bytes of a row for one 128-element K
// atom forming one 32-bit word (byte t = the atom's t-th 32-element block).
// The words of one atom for consecutive rows are consecutive, so the scale
// warps read them with coalesced 4-byte loads, one load per TMEM cell.
#include <algorithm>
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
constexpr int kAtom = 128;                 // K elements (bytes) per ring stage
constexpr int kThreads = 320;
constexpr int kMaxGroup = 64;
constexpr int kBNMax = 128;
constexpr int kAStage = kBM * kAtom;       // 16 KB
constexpr int kBStage = kBNMax * kAtom;    // 16 KB
constexpr int kEpiBytes = 4 * 2 * 4096;    // per epilogue warp 2 x 32x32 fp32
constexpr int kSfSlots = 8;                // scale ring depth, in K atoms
constexpr uint32_t kTmemCols = 512;        // 2 accumulators x 128 + scale ring
constexpr uint32_t kSfCol0 = 2 * kBNMax;   // first column of the scale ring

enum : uint32_t {
    SITE_X_EMPTY = 0x501,
    SITE_X_TEMPTY = 0x502,
    SITE_X_FULL = 0x503,
    SITE_X_SFULL = 0x504,
    SITE_X_TFULL = 0x505,
    SITE_X_CLOAD = 0x506,
    SITE_X_SEMPTY = 0x507,
    SITE_X_DONE = 0x508,
};

struct MxProblem {
    int M, N, K;
    int m_tiles, n_tiles, kb_total;  // kb_total: 128-element K atoms
    int nblk;                        // 32-element K blocks: ceil(K / 32)
    int bn;
    int tma_c;                       // C rows 16-byte aligned: TMA epilogue
    int tile_start;
    float alpha, beta;
    float *C;
    const uint32_t *SA;              // [ceil(K/128)][M] words of 4 scale bytes
    const uint32_t *SB;              // [ceil(K/128)][N]
};

struct MxParams {
    int count, total_tiles, stages;
    unsigned long long timeout_ns;
    uint32_t *err;
    MxProblem prob[kMaxGroup];
    CUtensorMap tmA[kMaxGroup];
    CUtensorMap tmB[kMaxGroup];
    CUtensorMap tmC[kMaxGroup];
};
static_assert(sizeof(MxParams) <= 32764, "kernel parameters exceed 32764 bytes");

// Each role copies the owning problem's fields into registers for the tile:
// through a reference they would be read again from parameter space after
// every inline-asm statement with a memory clobber (as in the grouped GEMM,
// where the copy made the sweep 3.5% faster).
__device__ __forceinline__ int mx_find_problem(const MxParams &p, int tile, int i) {
    while (i + 1 < p.count && p.prob[i + 1].tile_start <= tile) ++i;
    return i;
}

// The scale word of `row` for K atom `atom`, loaded into v only when the row
// exists (v keeps 0x7F7F7F7F, a scale of 1 on zero-filled operands,
// otherwise).  Nothing reads v here, so the load stays in flight while the
// warp goes on; mask_past_k applies the last atom's mask where v is used.
__device__ __forceinline__ void load_scale_word(uint32_t &v, const uint32_t *S, int rows, int row, int atom) {
    v = 0x7F7F7F7Fu;
    if (row < rows) v = __ldg(S + static_cast<size_t>(atom) * rows + row);
}

// The bytes of the last atom's blocks past K read as 127, whatever the caller
// stored there.
__device__ __forceinline__ uint32_t mask_past_k(uint32_t v, int nblk, int atom) {
    const int past = 4 * atom + 4 - nblk;  // 0..3 on the last atom
    if (past <= 0) return v;
    const uint32_t keep = 0xFFFFFFFFu >> (8 * past);
    return (v & keep) | (0x7F7F7F7Fu & ~keep);
}

__global__ void __launch_bounds__(kThreads, 1) gemm_mx_kernel(const __grid_constant__ MxParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    const int ST = p.stages;
    uint8_t *sA = smem;
    uint8_t *sB = smem + static_cast<size_t>(ST) * kAStage;
    uint8_t *ebuf = sB + static_cast<size_t>(ST) * kBStage;
    uint64_t *bars = reinterpret_cast<uint64_t *>(ebuf + kEpiBytes);
    uint64_t *full = bars;
    uint64_t *empty = bars + ST;
    uint64_t *sfull = empty + ST;
    uint64_t *sempty = sfull + kSfSlots;
    uint64_t *tfull = sempty + kSfSlots;
    uint64_t *tempty = tfull + 2;
    uint64_t *cbar = tempty + 2;  // [4 warps][2]
    uint64_t *done = cbar + 8;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < ST; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < kSfSlots; ++i) {
            mbar_init(&sfull[i], 4);
            mbar_init(&sempty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        for (int i = 0; i < 8; ++i) mbar_init(&cbar[i], 1);
        mbar_init(done, 8);  // epilogue and scale warps finished with TMEM
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
                pi = mx_find_problem(p, tile, pi);
                const MxProblem pr = p.prob[pi];  // a copy, see mx_find_problem
                const int local = tile - pr.tile_start;
                const int mt = local % pr.m_tiles, nt = local / pr.m_tiles;
                const uint32_t bytes = static_cast<uint32_t>(kAStage + pr.bn * kAtom);
                for (int kb = 0; kb < pr.kb_total; ++kb) {
                    if (!bounded_wait(&empty[stage], phase ^ 1u, w, SITE_X_EMPTY)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&full[stage], bytes);
                    tma_load_2d(&p.tmA[pi], &full[stage], sA + static_cast<size_t>(stage) * kAStage, kb * kAtom,
                                mt * kBM);
                    tma_load_2d(&p.tmB[pi], &full[stage], sB + static_cast<size_t>(stage) * kBStage, kb * kAtom,
                                nt * pr.bn);
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
            int stage = 0, acc = 0, pi = 0, slot = 0;
            uint32_t phase = 0, acc_phase = 0, sphase = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < p.total_tiles; tile += gridDim.x) {
                pi = mx_find_problem(p, tile, pi);
                const MxProblem pr = p.prob[pi];  // a copy, see mx_find_problem
                if (!bounded_wait(&tempty[acc], acc_phase ^ 1u, w, SITE_X_TEMPTY)) break;
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(acc * kBNMax);
                for (int kb = 0; kb < pr.kb_total; ++kb) {
                    if (!bounded_wait(&full[stage], phase, w, SITE_X_FULL) ||
                        !bounded_wait(&sfull[slot], sphase, w, SITE_X_SFULL)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(sA + static_cast<size_t>(stage) * kAStage);
                    const uint32_t b0 = smem_u32(sB + static_cast<size_t>(stage) * kBStage);
                    const uint32_t sfa = tmem_base + kSfCol0 + static_cast<uint32_t>(slot * 8);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        // K = 32 elements = 32 bytes of each 128-byte swizzled row
                        const uint64_t ad = sdesc_sw128(a0 + j * 32, 16, 1024);
                        const uint64_t bd = sdesc_sw128(b0 + j * 32, 16, 1024);
                        umma_mx(d, ad, bd, idesc_mx_e4m3(kBM, pr.bn, j, j), sfa, sfa + 4,
                                (kb > 0 || j > 0) ? 1u : 0u);
                    }
                    umma_commit(&empty[stage]);
                    umma_commit(&sempty[slot]);
                    if (++stage == ST) {
                        stage = 0;
                        phase ^= 1u;
                    }
                    if (++slot == kSfSlots) {
                        slot = 0;
                        sphase ^= 1u;
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
    } else if (warp >= 6) {
        // ------------------------------------------------ scale writers
        const int q = warp & 3;  // the TMEM lane quarter this warp may write
        int slot = 0, pi = 0;
        uint32_t sphase = 0;
        bool ok = true;
        for (int tile = blockIdx.x; ok && tile < p.total_tiles; tile += gridDim.x) {
            pi = mx_find_problem(p, tile, pi);
            const MxProblem pr = p.prob[pi];  // a copy, see mx_find_problem
            const int local = tile - pr.tile_start;
            const int mt = local % pr.m_tiles, nt = local / pr.m_tiles;
            const int m0 = mt * kBM, n0 = nt * pr.bn;
            // Scale words of K atom kb: this lane's rows of A (column 0: row
            // 32q + lane; columns 1..3: row lane + 32j) and of B (row lane + 32j).
            auto load_atom = [&](int kb, uint32_t (&va)[4], uint32_t (&vb)[4]) {
                load_scale_word(va[0], pr.SA, pr.M, m0 + q * 32 + lane, kb);
#pragma unroll
                for (int j = 1; j < 4; ++j) load_scale_word(va[j], pr.SA, pr.M, m0 + lane + 32 * j, kb);
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    load_scale_word(vb[j], pr.SB, lane + 32 * j < pr.bn ? pr.N : 0, n0 + lane + 32 * j, kb);
            };
            // The loads run kPf atoms ahead of the stores (a register ring
            // indexed at compile time), so their latency is paid once per tile.
            constexpr int kPf = 4;
            uint32_t pa[kPf][4], pb[kPf][4];
#pragma unroll
            for (int i = 0; i < kPf; ++i)
                if (i < pr.kb_total) load_atom(i, pa[i], pb[i]);
            for (int kb0 = 0; ok && kb0 < pr.kb_total; kb0 += kPf) {
#pragma unroll
                for (int i = 0; i < kPf; ++i) {
                    const int kb = kb0 + i;
                    if (kb >= pr.kb_total) break;
                    if (!warp_wait(&sempty[slot], sphase ^ 1u, w, SITE_X_SEMPTY)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t col = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + kSfCol0 +
                                         static_cast<uint32_t>(slot * 8);
                    if (4 * kb + 4 > pr.nblk) {
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            pa[i][j] = mask_past_k(pa[i][j], pr.nblk, kb);
                            pb[i][j] = mask_past_k(pb[i][j], pr.nblk, kb);
                        }
                    }
                    tmem_st4(col, pa[i]);
                    tmem_st4(col + 4, pb[i]);
                    tmem_st_wait();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&sfull[slot]);
                    if (++slot == kSfSlots) {
                        slot = 0;
                        sphase ^= 1u;
                    }
                    if (kb + kPf < pr.kb_total) load_atom(kb + kPf, pa[i], pb[i]);
                }
            }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(done);
        __syncwarp();
    } else {
        // ------------------------------------------------ epilogue (warps 2-5)
        const int ew = warp - 2;
        const int q = warp & 3;
        uint8_t *stg = ebuf + ew * 8192;
        uint64_t *cb = cbar + ew * 2;
        uint32_t cpar[2] = {0u, 0u};
        bool cpend[2] = {false, false};
        int gbuf = 0, acc = 0, pi = 0;
        uint32_t acc_phase = 0;
        for (int tile = blockIdx.x; tile < p.total_tiles; tile += gridDim.x) {
            pi = mx_find_problem(p, tile, pi);
            const MxProblem pr = p.prob[pi];  // a copy, see mx_find_problem
            const int local = tile - pr.tile_start;
            const int mt = local % pr.m_tiles, nt = local / pr.m_tiles;
            const int row0 = mt * kBM + q * 32;
            const int col0 = nt * pr.bn;
            const bool load_c = pr.tma_c && pr.beta != 0.0f;
            const int nch = (pr.bn + 31) / 32;
            if (load_c) {
                if (lane == 0) {
                    bulk_wait_read<0>();
                    const int b = gbuf & 1;
                    mbar_arrive_expect_tx(&cb[b], 4096);
                    tma_load_2d(&p.tmC[pi], &cb[b], stg + b * 4096, col0, row0);
                }
                cpend[gbuf & 1] = true;
                __syncwarp();
            }
            if (!warp_wait(&tfull[acc], acc_phase, w, SITE_X_TFULL)) break;
            tc_fence_after();
            const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                   static_cast<uint32_t>(acc * kBNMax);
            bool ok = true;
            for (int j = 0; j < nch; ++j) {
                const int b = gbuf & 1;
                if (load_c && j + 1 < nch) {
                    if (lane == 0) {
                        bulk_wait_read<0>();
                        mbar_arrive_expect_tx(&cb[b ^ 1], 4096);
                        tma_load_2d(&p.tmC[pi], &cb[b ^ 1], stg + (b ^ 1) * 4096, col0 + (j + 1) * 32, row0);
                    }
                    cpend[b ^ 1] = true;
                }
                if (!load_c && lane == 0) bulk_wait_read<1>();
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
                if (load_c) {
                    if (!warp_wait(&cb[b], cpar[b], w, SITE_X_CLOAD)) {
                        ok = false;
                        break;
                    }
                    cpar[b] ^= 1u;
                    cpend[b] = false;
                }
                __syncwarp();
                uint8_t *sb = stg + b * 4096;
#pragma unroll
                for (int ch = 0; ch < 8; ++ch) {
                    const int pos = ch ^ (lane & 7);
                    float4 *slot4 = reinterpret_cast<float4 *>(sb + lane * 128 + pos * 16);
                    float4 v = make_float4(pr.alpha * __uint_as_float(r[4 * ch]),
                                           pr.alpha * __uint_as_float(r[4 * ch + 1]),
                                           pr.alpha * __uint_as_float(r[4 * ch + 2]),
                                           pr.alpha * __uint_as_float(r[4 * ch + 3]));
                    if (load_c) {
                        const float4 cv = *slot4;
                        v.x += pr.beta * cv.x;
                        v.y += pr.beta * cv.y;
                        v.z += pr.beta * cv.z;
                        v.w += pr.beta * cv.w;
                    }
                    *slot4 = v;
                }
                const int cbase = col0 + j * 32;
                if (pr.tma_c) {
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_2d(&p.tmC[pi], sb, cbase, row0);
                        bulk_commit();
                    }
                } else {
                    // Rows of C not 16-byte aligned: plain stores, one row per
                    // iteration, 32 consecutive columns (coalesced).
                    __syncwarp();
                    const int col = cbase + lane;
                    for (int rr = 0; rr < 32; ++rr) {
                        const int grow = row0 + rr;
                        if (grow >= pr.M) break;
                        if (col < pr.N && lane < pr.bn - j * 32) {
                            const int pos = (lane >> 2) ^ (rr & 7);
                            float v = *reinterpret_cast<const float *>(sb + rr * 128 + pos * 16 + (lane & 3) * 4);
                            if (pr.beta != 0.0f) v += pr.beta * pr.C[static_cast<size_t>(grow) * pr.N + col];
                            pr.C[static_cast<size_t>(grow) * pr.N + col] = v;
                        }
                    }
                    __syncwarp();
                }
                ++gbuf;
            }
            if (!ok) break;
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(&tempty[acc]);
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
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        bounded_wait(done, 0, w, SITE_X_DONE);
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, kTmemCols);
    }
}

size_t mx_smem_bytes(int stages) {
    return 1024 + static_cast<size_t>(stages) * (kAStage + kBStage) + kEpiBytes +
           (2 * stages + 2 * kSfSlots + 13) * 8 + 16;
}

std::mutex g_mx_mu;

}  // namespace

int gemm_mx_validate(const MxDesc &g) {
    if (g.M < 1 || g.N < 1 || g.K < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_mxfp8: sizes must be >= 1 (M=%d N=%d K=%d)", g.M, g.N,
                         g.K);
    if (!g.A || !g.SA || !g.B || !g.SB || !g.C)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_mxfp8: null pointer");
    if ((reinterpret_cast<uintptr_t>(g.A) | reinterpret_cast<uintptr_t>(g.B) | reinterpret_cast<uintptr_t>(g.C)) &
        15u)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gemm_mxfp8: A, B and C must be 16-byte aligned");
    if (g.K % 16 != 0)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gemm_mxfp8: K (%d) must be a multiple of 16 (16-byte rows)",
                         g.K);
    if ((reinterpret_cast<uintptr_t>(g.SA) | reinterpret_cast<uintptr_t>(g.SB)) & 3u)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gemm_mxfp8: SA and SB must be 4-byte aligned");
    return ISAM_OK;
}

int gemm_mx_launch(int count, const MxDesc *g, DeviceState &ds, cudaStream_t stream) {
    if (count < 1 || count > kMaxGroup)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_grouped_mxfp8: count must be in [1, %d]", kMaxGroup);
    // Problems with the costliest tiles first (the round-robin walk ends
    // with the cheap ones).
    int order[kMaxGroup];
    std::iota(order, order + count, 0);
    auto atoms = [&](int i) { return (g[i].K + kAtom - 1) / kAtom; };
    std::stable_sort(order, order + count, [&](int a, int b) { return atoms(a) > atoms(b); });

    static MxParams p;  // ~30 KB: built under the lock, copied into the launch
    std::lock_guard<std::mutex> lk(g_mx_mu);
    memset(&p, 0, sizeof p);
    p.count = count;
    int tiles = 0;
    for (int s = 0; s < count; ++s) {
        const MxDesc &d = g[order[s]];
        MxProblem &pr = p.prob[s];
        pr.M = d.M;
        pr.N = d.N;
        pr.K = d.K;
        pr.bn = std::min(kBNMax, (d.N + 15) / 16 * 16);
        pr.m_tiles = (d.M + kBM - 1) / kBM;
        pr.n_tiles = (d.N + pr.bn - 1) / pr.bn;
        pr.kb_total = atoms(order[s]);
        pr.nblk = (d.K + 31) / 32;
        pr.tma_c = (d.N % 4 == 0) ? 1 : 0;
        pr.tile_start = tiles;
        pr.alpha = d.alpha;
        pr.beta = d.beta;
        pr.C = d.C;
        pr.SA = reinterpret_cast<const uint32_t *>(d.SA);
        pr.SB = reinterpret_cast<const uint32_t *>(d.SB);
        tiles += pr.m_tiles * pr.n_tiles;
        int rc;
        if ((rc = make_tmap_2d_u8(&p.tmA[s], d.A, d.K, d.M, static_cast<uint64_t>(d.K), kAtom, kBM))) return rc;
        if ((rc = make_tmap_2d_u8(&p.tmB[s], d.B, d.K, d.N, static_cast<uint64_t>(d.K), kAtom,
                                  static_cast<uint32_t>(pr.bn))))
            return rc;
        if (pr.tma_c &&
            (rc = make_tmap_2d_f32(&p.tmC[s], d.C, d.N, d.M, static_cast<uint64_t>(d.N) * 4, 32, 32)))
            return rc;
    }
    p.total_tiles = tiles;
    int st = 8;
    while (st > 2 && mx_smem_bytes(st) > static_cast<size_t>(ds.max_smem_optin)) --st;
    p.stages = st;
    p.timeout_ns = wait_timeout_ns();
    p.err = ds.err_word;
    const size_t smem = mx_smem_bytes(st);
    if (smem > static_cast<size_t>(ds.max_smem_optin))
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gemm_mxfp8: the pipeline does not fit shared memory");
    if (const int rc = ensure_smem_optin(reinterpret_cast<const void *>(gemm_mx_kernel), ds.max_smem_optin,
                                         ds.device, "cudaFuncSetAttribute(gemm mx)"))
        return rc;
    const int grid = std::min(tiles, ds.num_sms);
    gemm_mx_kernel<<<grid, kThreads, smem, stream>>>(p);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_error(e, "launch gemm_mx_kernel");
    return ISAM_OK;
}

}  // namespace isam
