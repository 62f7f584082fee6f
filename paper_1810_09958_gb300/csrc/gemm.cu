// gemm.cu -- tcgen05 GEMM for sm_103a:  C = alpha * op(A) * op(B) + beta * C
//
// The matrix-multiplication kernel of Listing 1 / Listing 4, scheduled the
// GB300 way:
//   * a persistent grid, one CTA (or one cluster of CTAs) per SM, walking
//     output tiles in an L2-friendly grouped order (the paper's "unrolling"
//     places compute tiles that share memory close together, Section 3.3);
//   * warp specialisation: warp 0 streams A/B tiles with TMA into a
//     multi-stage shared-memory ring, warp 1 issues tcgen05.mma from one
//     thread into a double-buffered TMEM accumulator, warps 2-5 drain TMEM
//     and apply alpha/beta/bias while the next tile is being multiplied;
//   * split-K for skinny problems: the CTAs of one thread-block cluster take
//     disjoint K ranges of the same tile and reduce their partial tiles
//     through distributed shared memory in a fixed rank order (deterministic);
//   * the tile width, split and ring depth come from a small analytic cost
//     model (the paper's "Approach" interface for tiling and device
//     allocation choices, Sections 3.4 and 4).
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "gemm_common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace isam {

namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;
constexpr int kThreads = 192;
constexpr int kABytes = kBM * kBK * 2;  // 16 KB

enum : uint32_t {
    SITE_PROD_EMPTY = 0x101,
    SITE_PROD_DRAIN = 0x102,
    SITE_MMA_TEMPTY = 0x111,
    SITE_MMA_FULL = 0x112,
    SITE_EPI_TFULL = 0x121,
    SITE_EPI_REDFREE = 0x122,
    SITE_EPI_REDFULL = 0x123,
};

struct GemmParams {
    int M, N, K;
    int m_tiles, n_tiles, kb_total;
    int split, stages, group_m;
    int ka;      // 64-wide K atoms per pipeline stage (1, 2 or 4)
    int kg_total;  // k-groups of ka atoms
    int n_vec4;  // 1 when N % 4 == 0 (16-byte stores in the split-K reduce)
    int tma_c;   // 1: epilogue moves C with TMA (N % 4 == 0, BN >= 32, no split)
    float alpha, beta;
    float *C;
    const float *bias;
    unsigned long long timeout_ns;
    uint32_t *err;
};

template <int BN, bool B_MN>
struct Cfg {
    static constexpr int kBAtom = B_MN ? ((BN + 63) / 64) * 8192 : BN * 128;  // one K atom of B
    static constexpr int kTmemCols = (2 * BN <= 32) ? 32 : (2 * BN <= 64) ? 64 : (2 * BN <= 128) ? 128 : (2 * BN <= 256) ? 256 : 512;
    static constexpr int kCW = BN < 32 ? BN : 32;  // epilogue column chunk
};

// Split-K partial rows of 128 columns go to their owner through a per-warp
// transpose (whole row segments per remote store); narrower tiles push each
// thread's row directly.
__host__ __device__ constexpr bool xpose_push(int BN) { return BN >= 128; }

// Epilogue shared memory: split-K partial tile (128 x BN fp32 received
// slices; rows padded by 4 floats for the direct push, plus a 4 KB transpose
// buffer per epilogue warp for the transposed one), or per-warp staging (TMA
// path: 2 x 4 KB per epilogue warp; plain path: a 32 x 33 fp32 transpose).
__host__ __device__ inline size_t epi_bytes(int BN, int split) {
    if (split > 1)
        return xpose_push(BN) ? static_cast<size_t>(kBM) * BN * 4 + 4 * 4096 : static_cast<size_t>(kBM) * (BN + 4) * 4;
    return BN >= 32 ? static_cast<size_t>(4) * 2 * 4096 : static_cast<size_t>(4) * 32 * 33 * 4;
}

__device__ __forceinline__ void tile_coords(int tile, int m_tiles, int n_tiles, int group_m,
                                            int &mt, int &nt) {
    const int per_group = group_m * n_tiles;
    const int g = tile / per_group;
    const int first_m = g * group_m;
    const int gm = min(group_m, m_tiles - first_m);
    const int local = tile - g * per_group;
    mt = first_m + local % gm;
    nt = local / gm;
}

// F8: E4M3 operands (K-major A and B only): a 128-byte K atom holds 128
// elements instead of 64; everything else -- tiles, stages, swizzle, epilogue
// -- is byte-for-byte the bf16 kernel.
template <int BN, bool A_MN, bool B_MN, bool F8 = false>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, const GemmParams p) {
    using C = Cfg<BN, B_MN>;
    if (p.split > 1 && !launch_shape_ok(p.err, static_cast<uint32_t>(p.split), gridDim.x, 0x1F0u)) return;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    const int S = p.split;
    const int ST = p.stages;
    const int KA = p.ka;
    const int a_stage = KA * kABytes;
    const int b_stage = KA * C::kBAtom;
    uint8_t *sA = smem;
    uint8_t *sB = smem + static_cast<size_t>(ST) * a_stage;
    float *ebuf = reinterpret_cast<float *>(sB + static_cast<size_t>(ST) * b_stage);
    uint64_t *bars = reinterpret_cast<uint64_t *>(reinterpret_cast<uint8_t *>(ebuf) + epi_bytes(BN, S));
    uint64_t *full = bars;
    uint64_t *empty = bars + ST;
    uint64_t *tfull = empty + ST;
    uint64_t *tempty = tfull + 2;
    uint64_t *red_full = tempty + 2;
    uint64_t *red_free = red_full + 1;
    uint64_t *cbar = red_free + 1;  // [4 epilogue warps][2] C-load barriers
    uint64_t *done = cbar + 8;      // epilogue warps finished with TMEM
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(done + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = S > 1 ? cluster_ctarank() : 0u;
    const int cluster_id = blockIdx.x / S;
    const int num_clusters = gridDim.x / S;

    if (threadIdx.x == 0) {
        for (int i = 0; i < ST; ++i) {
            mbar_init(&full[i], 1);
            mbar_init(&empty[i], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&tfull[i], 1);
            mbar_init(&tempty[i], 4);
        }
        // Direct push: one arrival per partial row (S sources x 128 / S rows).
        // Transposed push: one per (source CTA, epilogue warp) whose 32 rows
        // meet this CTA's slice of the tile.
        int red_arrivals = xpose_push(BN) ? 0 : kBM;
        if (S > 1 && xpose_push(BN)) {
            const int rp = kBM / S;
            for (int q = 0; q < 4; ++q)
                if (q * 32 < static_cast<int>(rank + 1) * rp && q * 32 + 32 > static_cast<int>(rank) * rp)
                    red_arrivals += S;
        }
        mbar_init(red_full, red_arrivals > 0 ? red_arrivals : 1);
        mbar_init(red_free, S);
        for (int i = 0; i < 8; ++i) mbar_init(&cbar[i], 1);
        mbar_init(done, 4);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
        if (p.tma_c) tma_prefetch_desc(&tmC);
    }
    __syncwarp();
    if (warp == 1) {
        tmem_alloc(tmem_slot, C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    if (S > 1) cluster_sync_all();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const WaitCtx w{p.timeout_ns, p.err, abort_flag};

    const int kg_begin = static_cast<int>((static_cast<long long>(rank) * p.kg_total) / S);
    const int kg_end = static_cast<int>((static_cast<long long>(rank + 1) * p.kg_total) / S);
    const int num_tiles = p.m_tiles * p.n_tiles;

    // Dependent launch: this grid's CTAs may start (barriers, TMEM, tensor
    // maps) on SMs the previous kernel on the stream leaves free, and wait
    // here until it has finished; every global load or store comes after.
    // (An L2 prefetch of the first stages issued before the wait made the
    // per-call sweep 3.8% slower: it delays the first real load of every CTA
    // that starts only after the previous kernel has drained.)
    griddep_launch_dependents();
    __syncwarp();
    griddep_wait();

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int issued = 0;
            bool ok = true;
            for (int tile = cluster_id; ok && tile < num_tiles; tile += num_clusters) {
                int mt, nt;
                tile_coords(tile, p.m_tiles, p.n_tiles, p.group_m, mt, nt);
                for (int kg = kg_begin; kg < kg_end; ++kg) {
                    if (!bounded_wait(&empty[stage], phase ^ 1u, w, SITE_PROD_EMPTY)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&full[stage], static_cast<uint32_t>(a_stage + b_stage));
                    uint8_t *a = sA + static_cast<size_t>(stage) * a_stage;
                    uint8_t *b = sB + static_cast<size_t>(stage) * b_stage;
                    for (int at = 0; at < KA; ++at) {
                        const int k0 = (kg * KA + at) * (F8 ? 2 * kBK : kBK);  // in elements
                        uint8_t *aa = a + at * kABytes;
                        uint8_t *bb = b + at * C::kBAtom;
                        if (A_MN) {
                            tma_load_2d(&tmA, &full[stage], aa, mt * kBM, k0);
                            tma_load_2d(&tmA, &full[stage], aa + 8192, mt * kBM + 64, k0);
                        } else {
                            tma_load_2d(&tmA, &full[stage], aa, k0, mt * kBM);
                        }
                        if (B_MN) {
#pragma unroll
                            for (int c = 0; c < (BN + 63) / 64; ++c)
                                tma_load_2d(&tmB, &full[stage], bb + c * 8192, nt * BN + c * 64, k0);
                        } else {
                            tma_load_2d(&tmB, &full[stage], bb, k0, nt * BN);
                        }
                    }
                    ++issued;
                    if (++stage == ST) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok) {
                // Let every copy already issued land before the CTA can exit.
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
            const uint32_t idesc = F8 ? idesc_e4m3_f32(kBM, BN) : idesc_bf16_f32(kBM, BN, A_MN, B_MN);
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true;
            for (int tile = cluster_id; ok && tile < num_tiles; tile += num_clusters) {
                if (!bounded_wait(&tempty[acc], acc_phase ^ 1u, w, SITE_MMA_TEMPTY)) break;
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(acc * BN);
                for (int kg = kg_begin; kg < kg_end; ++kg) {
                    if (!bounded_wait(&full[stage], phase, w, SITE_MMA_FULL)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(sA + static_cast<size_t>(stage) * a_stage);
                    const uint32_t b0 = smem_u32(sB + static_cast<size_t>(stage) * b_stage);
                    for (int at = 0; at < KA; ++at) {
                        const uint32_t aa = a0 + at * kABytes;
                        const uint32_t bb = b0 + at * C::kBAtom;
#pragma unroll
                        for (int k = 0; k < kBK / 16; ++k) {
                            const uint64_t ad = A_MN ? sdesc_sw128(aa + k * 2048, 8192, 1024)
                                                     : sdesc_sw128(aa + k * 32, 16, 1024);
                            const uint64_t bd = B_MN ? sdesc_sw128(bb + k * 2048, 8192, 1024)
                                                     : sdesc_sw128(bb + k * 32, 16, 1024);
                            if constexpr (F8)
                                umma_f8(d, ad, bd, idesc, (kg > kg_begin || at > 0 || k > 0) ? 1u : 0u);
                            else
                                umma_bf16(d, ad, bd, idesc, (kg > kg_begin || at > 0 || k > 0) ? 1u : 0u);
                        }
                    }
                    umma_commit(&empty[stage]);
                    if (++stage == ST) {
                        stage = 0;
                        phase ^= 1u;
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
        const int ew = warp - 2;          // 0..3
        const int q = warp & 3;           // TMEM lane quadrant this warp may read
        const bool use_tma = (S == 1) && (BN >= 32) && (p.tma_c != 0);
        const bool load_c = use_tma && (p.beta != 0.0f);
        uint8_t *stg = reinterpret_cast<uint8_t *>(ebuf) + ew * 8192;  // TMA path: 2 x 4 KB
        uint64_t *cb = cbar + ew * 2;
        uint32_t cpar[2] = {0u, 0u};
        bool cpend[2] = {false, false};
        int gbuf = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        int iter = 0;
        bool ok = true;
        for (int tile = cluster_id; tile < num_tiles; tile += num_clusters, ++iter) {
            int mt, nt;
            tile_coords(tile, p.m_tiles, p.n_tiles, p.group_m, mt, nt);
            const int row0 = mt * kBM + q * 32;
            const int col0 = nt * BN;
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
            if (!warp_wait(&tfull[acc], acc_phase, w, SITE_EPI_TFULL)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) +
                                   static_cast<uint32_t>(acc * BN);
            if (use_tma) {
                if constexpr (BN >= 32) {
#pragma unroll 1
                    for (int j = 0; j < BN / 32; ++j) {
                        const int b = gbuf & 1;
                        if (load_c && j + 1 < BN / 32) {
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
                        tmem_ld_wait();
                        if (load_c) {
                            if (!warp_wait(&cb[b], cpar[b], w, SITE_EPI_TFULL)) {
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
                            float4 v = make_float4(p.alpha * __uint_as_float(r[4 * ch]),
                                                   p.alpha * __uint_as_float(r[4 * ch + 1]),
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
                }
            } else if (S == 1) {
                float *tb = ebuf + ew * (32 * 33);
                constexpr int CW = C::kCW;
                constexpr int RPI = 32 / CW;  // rows per store iteration
                const int sub = lane / CW;
                const int col = lane % CW;
#pragma unroll 1
                for (int c = 0; c < BN; c += CW) {
                    uint32_t r[CW];
                    if constexpr (CW == 32) {
                        tmem_ld32(tbase + c, r);
                    } else {
                        tmem_ld16(tbase + c, r);
                    }
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < CW; ++j) tb[lane * 33 + j] = __uint_as_float(r[j]);
                    __syncwarp();
                    const int gcol = col0 + c + col;
                    const float bias = (p.bias != nullptr && gcol < p.N) ? p.bias[gcol] : 0.0f;
                    float cin[32 / RPI];
                    if (p.beta != 0.0f) {
#pragma unroll
                        for (int i = 0; i < 32 / RPI; ++i) {
                            const int grow = row0 + sub + i * RPI;
                            cin[i] = (grow < p.M && gcol < p.N) ? p.C[static_cast<size_t>(grow) * p.N + gcol] : 0.0f;
                        }
                    }
#pragma unroll
                    for (int i = 0; i < 32 / RPI; ++i) {
                        const int rr = sub + i * RPI;
                        const int grow = row0 + rr;
                        if (grow < p.M && gcol < p.N) {
                            float v = p.alpha * tb[rr * 33 + col] + bias;
                            if (p.beta != 0.0f) v += p.beta * cin[i];
                            p.C[static_cast<size_t>(grow) * p.N + gcol] = v;
                        }
                    }
                    __syncwarp();
                }
            } else {
                // Split-K, push style: row slice o (128 / S rows) of the tile is
                // reduced by cluster rank o.  Narrow tiles: every epilogue
                // thread stores its partial row straight into the owner's
                // shared memory and release-arrives on the owner's red_full
                // (128 arrivals per tile: S sources x 128 / S rows).  128-column
                // tiles: each epilogue warp transposes its 32 partial rows
                // through a 4 KB shared-memory buffer, 32 columns at a time, so
                // that every remote store instruction writes four 128-byte row
                // segments of the owner's slot instead of one 16-byte piece of
                // 32 rows, then release-arrives once on each owner of its rows.
                // Each owner sums the S slices it received in rank order
                // (deterministic) and stores its rows of C.
                // A wait that runs out skips the work but still reaches the
                // epilogue barrier below, which makes the decision to stop
                // uniform across the four warps.
                bool wok = true;
                if (iter > 0)
                    wok = warp_wait<true>(red_free, static_cast<uint32_t>((iter - 1) & 1), w, SITE_EPI_REDFREE);
                const int rows_per = kBM / S;
                constexpr bool kXpose = xpose_push(BN);
                constexpr int EP = kXpose ? BN : BN + 4;  // row pitch of the received slices
                if (kXpose && wok) {
                    uint8_t *sx = reinterpret_cast<uint8_t *>(ebuf) + static_cast<size_t>(kBM) * BN * 4 + ew * 4096;
                    // Piece j (16 bytes) of row r sits at slot j ^ (r & 7) of
                    // the row's 128 bytes: writes by row and reads by row
                    // segment both take the minimum of four wavefronts.
                    const int rr = lane >> 3;  // row segment of this lane in a read-back instruction
                    const int jj = lane & 7;   // its 16-byte piece
#pragma unroll 1
                    for (int c = 0; c < BN; c += 32) {
                        uint32_t r[32];
                        tmem_ld32(tbase + c, r);
                        tmem_ld_wait();
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            *reinterpret_cast<uint4 *>(sx + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                                make_uint4(r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
                        __syncwarp();
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int row = i * 4 + rr;  // 0..31 within this warp's rows
                            const uint4 v = *reinterpret_cast<const uint4 *>(sx + row * 128 + ((jj ^ (row & 7)) << 4));
                            const int rl = q * 32 + row;  // row of the tile
                            const uint32_t owner = static_cast<uint32_t>(rl / rows_per);
                            const int ro = rl - static_cast<int>(owner) * rows_per;
                            const uint32_t dst = mapa_shared(
                                smem_u32(ebuf + static_cast<size_t>(static_cast<int>(rank) * rows_per + ro) * EP + c +
                                         jj * 4),
                                owner);
                            st_dsmem_f4(dst, make_float4(__uint_as_float(v.x), __uint_as_float(v.y),
                                                         __uint_as_float(v.z), __uint_as_float(v.w)));
                        }
                        __syncwarp();  // the buffer is read back before the next chunk overwrites it
                    }
                    // The barrier orders every lane's remote stores before lane
                    // 0's release-arrive on each owner of this warp's rows.
                    if (lane == 0) {
                        const int o_first = (q * 32) / rows_per;
                        const int o_last = (q * 32 + 31) / rows_per;
                        for (int o = o_first; o <= o_last; ++o) mbar_arrive_remote(red_full, static_cast<uint32_t>(o));
                    }
                    __syncwarp();
                }
                if (!kXpose && wok) {
                    const int row_local = q * 32 + lane;
                    const uint32_t owner = static_cast<uint32_t>(row_local / rows_per);
                    const int rr = row_local - static_cast<int>(owner) * rows_per;
                    const uint32_t dst = mapa_shared(
                        smem_u32(ebuf + static_cast<size_t>(static_cast<int>(rank) * rows_per + rr) * (BN + 4)), owner);
                    // Up to 64 columns per TMEM round trip (loads issued together).
                    constexpr int CH = BN < 64 ? BN : 64;
#pragma unroll 1
                    for (int c = 0; c < BN; c += CH) {
                        uint32_t r[CH];
                        if constexpr (CH == 16) {
                            uint32_t (&r0)[16] = *reinterpret_cast<uint32_t(*)[16]>(&r[0]);
                            tmem_ld16(tbase + c, r0);
                        } else {
#pragma unroll
                            for (int h = 0; h < CH / 32; ++h) {
                                uint32_t (&rh)[32] = *reinterpret_cast<uint32_t(*)[32]>(&r[h * 32]);
                                tmem_ld32(tbase + c + h * 32, rh);
                            }
                        }
                        tmem_ld_wait();
#pragma unroll
                        for (int j = 0; j < CH; j += 4)
                            st_dsmem_f4(dst + static_cast<uint32_t>((c + j) * 4),
                                        make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]),
                                                    __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3])));
                    }
                    mbar_arrive_remote(red_full, owner);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&tempty[acc]);
                __syncwarp();
                if (wok) wok = warp_wait<true>(red_full, static_cast<uint32_t>(iter & 1), w, SITE_EPI_REDFULL);
                if (wok) {
                    const int g4 = BN / 4;
                    const int groups = rows_per * g4;
                    for (int g = ew * 32 + lane; g < groups; g += 128) {
                        const int rr = g / g4;
                        const int c4 = (g % g4) * 4;
                        const int grow = mt * kBM + static_cast<int>(rank) * rows_per + rr;
                        const int gcol = col0 + c4;
                        if (grow >= p.M) continue;
                        float *crow = p.C + static_cast<size_t>(grow) * p.N;
                        const bool vec = p.n_vec4 && gcol + 3 < p.N;
                        float4 cin = make_float4(0.f, 0.f, 0.f, 0.f);
                        if (p.beta != 0.0f && vec) cin = *reinterpret_cast<const float4 *>(crow + gcol);
                        float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
                        for (int r = 0; r < S; ++r) {
                            const float4 v = *reinterpret_cast<const float4 *>(
                                ebuf + static_cast<size_t>(r * rows_per + rr) * EP + c4);
                            s.x += v.x;
                            s.y += v.y;
                            s.z += v.z;
                            s.w += v.w;
                        }
                        float o[4] = {s.x, s.y, s.z, s.w};
                        if (vec) {
                            float4 v;
                            float *vv = reinterpret_cast<float *>(&v);
                            const float *ci = reinterpret_cast<const float *>(&cin);
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                float x = p.alpha * o[j] + (p.bias ? p.bias[gcol + j] : 0.0f);
                                if (p.beta != 0.0f) x += p.beta * ci[j];
                                vv[j] = x;
                            }
                            *reinterpret_cast<float4 *>(crow + gcol) = v;
                        } else {
                            for (int j = 0; j < 4; ++j) {
                                if (gcol + j >= p.N) break;
                                float x = p.alpha * o[j] + (p.bias ? p.bias[gcol + j] : 0.0f);
                                if (p.beta != 0.0f) x += p.beta * crow[gcol + j];
                                crow[gcol + j] = x;
                            }
                        }
                    }
                }
                __syncwarp();
                if (!named_bar_and(1, 128, wok)) {
                    ok = false;
                    break;
                }
                // Release the slot to every pusher, unless nobody pushes again
                // (after the cluster's last tile no remote arrive may target an
                // exited CTA).
                if (tile + num_clusters < num_tiles && ew == 0 && lane == 0) {
                    for (int r = 0; r < S; ++r) mbar_arrive_remote(red_free, static_cast<uint32_t>(r));
                }
                __syncwarp();
            }
            if (S == 1) {
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&tempty[acc]);
                __syncwarp();
            }
            if (++acc == 2) {
                acc = 0;
                acc_phase ^= 1u;
            }
        }
        // TMA path: C loads still in flight land, stores complete, before exit.
        if (use_tma) {
            for (int b = 0; b < 2; ++b)
                if (cpend[b] && lane == 0) drain_wait(&cb[b], cpar[b], p.timeout_ns);
            if (lane == 0) bulk_wait_all<0>();
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(done);
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        // TMEM is released only after every epilogue warp has stopped reading it.
        bounded_wait(done, 0, w, SITE_EPI_TFULL);
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, C::kTmemCols);
    }
}

// ---------------------------------------------------------------- host side
using KernelFn = void (*)(CUtensorMap, CUtensorMap, CUtensorMap, GemmParams);

template <int BN>
KernelFn pick3(bool a_mn, bool b_mn) {
    if (a_mn) return b_mn ? gemm_tc_kernel<BN, true, true> : gemm_tc_kernel<BN, true, false>;
    return b_mn ? gemm_tc_kernel<BN, false, true> : gemm_tc_kernel<BN, false, false>;
}

KernelFn pick_kernel_f8(int BN) {
    switch (BN) {
        case 16: return gemm_tc_kernel<16, false, false, true>;
        case 32: return gemm_tc_kernel<32, false, false, true>;
        case 64: return gemm_tc_kernel<64, false, false, true>;
        case 128: return gemm_tc_kernel<128, false, false, true>;
        case 256: return gemm_tc_kernel<256, false, false, true>;
        default: return nullptr;
    }
}

KernelFn pick_kernel(int BN, bool a_mn, bool b_mn) {
    switch (BN) {
        case 16: return pick3<16>(a_mn, b_mn);
        case 32: return pick3<32>(a_mn, b_mn);
        case 64: return pick3<64>(a_mn, b_mn);
        case 128: return pick3<128>(a_mn, b_mn);
        case 256: return pick3<256>(a_mn, b_mn);
        default: return nullptr;
    }
}

int b_bytes(int BN, bool b_mn) { return b_mn ? ((BN + 63) / 64) * 8192 : BN * 128; }

size_t smem_bytes(int BN, bool b_mn, int split, int stages, int ka) {
    return 1024 + static_cast<size_t>(stages) * ka * (kABytes + b_bytes(BN, b_mn)) +
           epi_bytes(BN, split) + (2 * stages + 15) * 8 + 16;
}

int max_stages(int BN, bool b_mn, int split, int ka, int smem_limit) {
    int st = 8;
    while (st > 2 && smem_bytes(BN, b_mn, split, st, ka) > static_cast<size_t>(smem_limit)) --st;
    return st;
}

int ceil_div(long long a, long long b) { return static_cast<int>((a + b - 1) / b); }

// Machine constants of the cost model, calibrated on GB300 with the
// kernel's own timeline (globaltimer stamps per CTA): ~2.3 us from launch to
// the first TMA data; TMA operand streaming saturates at ~47 GB/s per SM from
// four stages in flight (a per-SM cap, so bandwidth comes from using many
// SMs); ~1.3 us between launches; measured dense bf16 and copy peaks.
constexpr double kPeakFlops = 1.9e15;
constexpr double kHbmBw = 6.7e12;
constexpr double kSmStreamBw = 47e9;   // operand bytes/s one SM sustains
constexpr double kSmStoreBw = 30e9;    // epilogue bytes/s one SM sustains
constexpr double kClock = 1.9e9;
constexpr double kFirstDataUs = 2.3;
constexpr double kLaunchGapUs = 1.3;
constexpr double kTileOverheadUs = 0.3;
constexpr double kSplitTailUs = 1.5;   // push + owner reduce of a split tile

double estimate_us(const GemmDesc &g, int BN, int S, int num_sms, int cluster_cap, int *grid_out) {
    const int m_tiles = ceil_div(g.M, kBM);
    const int n_tiles = ceil_div(g.N, BN);
    const long long tiles = static_cast<long long>(m_tiles) * n_tiles;
    const int eb = g.fp8 ? 1 : 2;                  // bytes per operand element
    const int kb = ceil_div(g.K, kBK * 2 / eb);     // 128-byte K atoms
    const int kb_per = ceil_div(kb, S);
    // Clusters that can be resident at once: the CTAs of a cluster share one
    // GPC, so fewer clusters of 4 or 8 fit than num_sms / S; a cluster
    // beyond that would wait for a whole resident one to finish.
    const int clusters_max = std::max(1, std::min(num_sms / S, cluster_cap));
    const int clusters = static_cast<int>(std::min<long long>(tiles, clusters_max));
    *grid_out = clusters * S;
    const int tiles_per_cluster = ceil_div(tiles, clusters);
    // Tensor time of one tile slice: 128 x BN x 16 per k-step at 4096 MAC/clk,
    // or shared-memory bound at 128 B/clk for the A and B slices.
    const double cyc_k16 = std::max(BN / 2.0, (kBM * 32.0 + BN * 32.0) / 128.0);
    const double t_mma = kb_per * 4 * cyc_k16 / kClock * 1e6;
    const double bytes_unit = static_cast<double>(kBM + BN) * kb_per * kBK * 2.0;
    const double t_load = bytes_unit / kSmStreamBw * 1e6;
    const double t_unit = std::max(t_mma, t_load) + kTileOverheadUs;
    const double t_steady = tiles_per_cluster * t_unit;
    const double out_bytes = 4.0 * g.M * g.N * (g.beta != 0.0f ? 2.0 : 1.0);
    const double uniq = eb * (static_cast<double>(g.M) * g.K + static_cast<double>(g.K) * g.N) + out_bytes;
    const double t_hbm = uniq / kHbmBw * 1e6;
    const double t_flops = 2.0 * g.M * g.N * g.K / (kPeakFlops * (g.fp8 ? 2.0 : 1.0)) * 1e6;
    const double tail = (S > 1 ? kSplitTailUs : 0.0) + kBM * BN * 4.0 / S / kSmStoreBw * 1e6;
    return kFirstDataUs + std::max({t_steady, t_hbm, t_flops}) + tail + kLaunchGapUs;
}


}  // namespace

// Clusters of `size` CTAs (one CTA per SM, as every GEMM plan here uses) that
// the device keeps resident at once, from cudaOccupancyMaxActiveClusters;
// cached per device.  Falls back to num_sms / size if the query fails.
int gemm_cluster_capacity(const DeviceState &ds, int size) {
    if (size <= 1) return ds.num_sms;
    const int idx = size == 2 ? 0 : size == 4 ? 1 : size == 8 ? 2 : -1;
    if (idx >= 0 && ds.cluster_cap[idx] > 0) return ds.cluster_cap[idx];
    if (idx < 0 || ds.device < 0 || ds.device >= 64) return std::max(1, ds.num_sms / size);
    static std::mutex mu;
    static int cache[64][3] = {};
    std::lock_guard<std::mutex> lk(mu);
    int &c = cache[ds.device][idx];
    if (c > 0) return c;
    int n = 0;
    KernelFn fn = pick_kernel(128, false, false);
    if (ensure_smem_optin(reinterpret_cast<const void *>(fn), ds.max_smem_optin, ds.device, "cudaFuncSetAttribute(gemm)") == ISAM_OK) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = static_cast<unsigned>(size);
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(static_cast<unsigned>(size * std::max(1, ds.num_sms / size)), 1, 1);
        cfg.blockDim = dim3(kThreads, 1, 1);
        cfg.dynamicSmemBytes = static_cast<size_t>(ds.max_smem_optin);
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, fn, &cfg) != cudaSuccess) {
            (void)cudaGetLastError();
            n = 0;
        }
    } else {
        (void)cudaGetLastError();
    }
    c = n > 0 ? std::min(n, ds.num_sms / size) : std::max(1, ds.num_sms / size);
    return c;
}

int gemm_validate(const GemmDesc &g) {
    if (g.M < 1 || g.N < 1 || g.K < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm: sizes must be >= 1 (M=%d N=%d K=%d)",
                         g.M, g.N, g.K);
    if ((g.transA != 0 && g.transA != 1) || (g.transB != 0 && g.transB != 1))
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm: transA/transB must be 0 or 1");
    if (!g.A || !g.B || !g.C) return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm: null pointer");
    if ((reinterpret_cast<uintptr_t>(g.A) | reinterpret_cast<uintptr_t>(g.B) |
         reinterpret_cast<uintptr_t>(g.C)) & 15u)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gemm: A, B and C must be 16-byte aligned");
    if (g.fp8) {
        if (g.transA != 0 || g.transB != 1)
            return set_error(ISAM_ERR_UNSUPPORTED, "isam_gemm_fp8: A and B must both be K-major");
        if (g.K % 16 != 0)
            return set_error(ISAM_ERR_UNSUPPORTED,
                             "isam_gemm_fp8: K (%d) must be a multiple of 16 (16-byte rows)", g.K);
        return ISAM_OK;
    }
    const int a_pitch = g.transA ? g.M : g.K;
    const int b_pitch = g.transB ? g.K : g.N;
    if (a_pitch % 8 != 0 || b_pitch % 8 != 0)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_gemm: stored row pitch of A (%d) and B (%d) must be multiples of 8 "
                         "elements (16 bytes)",
                         a_pitch, b_pitch);
    return ISAM_OK;
}

int gemm_plan(const GemmDesc &g, const DeviceState &ds, GemmPlan *plan) {
    if (!getenv("ISAM_FORCE_TILE") && gemm_pair_plan(g, ds, plan)) return ISAM_OK;
    const bool b_mn = g.transB == 0;
    const int nsm = ds.num_sms;
    const int kb = ceil_div(g.K, g.fp8 ? 2 * kBK : kBK);
    double best = 1e300;
    GemmPlan bp{};
    const int bns[] = {16, 32, 64, 128, 256};
    const int splits[] = {1, 2, 4, 8};
    for (int BN : bns) {
        if (BN > 16 && BN / 2 >= g.N) continue;  // wider than needed
        for (int S : splits) {
            if (S > kb) continue;
            if (S > 1 && BN > 128) continue;
            int grid = 0;
            const double t = estimate_us(g, BN, S, nsm, gemm_cluster_capacity(ds, S), &grid);
            if (t < best * 0.999) {
                best = t;
                bp.BN = BN;
                bp.split = S;
                bp.grid = grid;
                bp.est_us = t;
            }
        }
    }
    bp.ka = 1;
    if (const char *f = getenv("ISAM_FORCE_TILE")) {
        // "BN,split[,stages[,atoms per stage]]" (0 = the model's choice).
        int fbn = 0, fs = 0, fst = 0, fka = 0;
        if (sscanf(f, "%d,%d,%d,%d", &fbn, &fs, &fst, &fka) >= 2 && pick_kernel(fbn, false, false) &&
            (fs == 1 || fs == 2 || fs == 4 || fs == 8) && !(fs > 1 && fbn > 128)) {
            const int ka = (fka == 2 || fka == 4) ? fka : 1;
            if (fs <= ceil_div(kb, ka)) {
                bp.BN = fbn;
                bp.split = fs;
                bp.ka = ka;
                estimate_us(g, fbn, fs, nsm, gemm_cluster_capacity(ds, fs), &bp.grid);
                if (fst >= 2) bp.stages = fst;
            }
        }
    }
    const int st_max = max_stages(bp.BN, b_mn, bp.split, bp.ka, ds.max_smem_optin);
    if (bp.stages < 2 || bp.stages > st_max) bp.stages = st_max;
    bp.smem = smem_bytes(bp.BN, b_mn, bp.split, bp.stages, bp.ka);
    bp.group_m = 16;
    if (bp.smem > static_cast<size_t>(ds.max_smem_optin))
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gemm: tile does not fit shared memory");
    *plan = bp;
    return ISAM_OK;
}

int gemm_launch(const GemmDesc &g, const GemmPlan &plan, DeviceState &ds, cudaStream_t stream) {
    if (plan.pair) return gemm_pair_launch(g, plan, ds, stream);
    const bool a_mn = g.transA == 1;
    const bool b_mn = g.transB == 0;
    CUtensorMap ta, tb, tc;
    memset(&tc, 0, sizeof tc);
    int rc;
    if (g.fp8) {
        // 128-element (128-byte) K atoms of both K-major operands.
        if ((rc = make_tmap_2d_u8(&ta, g.A, g.K, g.M, static_cast<uint64_t>(g.K), 128, kBM))) return rc;
        if ((rc = make_tmap_2d_u8(&tb, g.B, g.K, g.N, static_cast<uint64_t>(g.K), 128,
                                  static_cast<uint32_t>(plan.BN))))
            return rc;
    } else {
        if (a_mn)
            rc = make_tmap_2d_bf16(&ta, g.A, g.M, g.K, static_cast<uint64_t>(g.M) * 2, 64, 64);
        else
            rc = make_tmap_2d_bf16(&ta, g.A, g.K, g.M, static_cast<uint64_t>(g.K) * 2, 64, kBM);
        if (rc) return rc;
        if (b_mn)
            rc = make_tmap_2d_bf16(&tb, g.B, g.N, g.K, static_cast<uint64_t>(g.N) * 2, 64, 64);
        else
            rc = make_tmap_2d_bf16(&tb, g.B, g.K, g.N, static_cast<uint64_t>(g.K) * 2, 64,
                                   static_cast<uint32_t>(plan.BN));
        if (rc) return rc;
    }
    // The epilogue moves C with TMA when rows are 16-byte aligned (N % 4 == 0)
    // and the tile is at least one 32-column chunk wide.
    const int tma_c = (g.N % 4 == 0 && plan.BN >= 32 && plan.split == 1) ? 1 : 0;
    if (tma_c && (rc = make_tmap_2d_f32(&tc, g.C, g.N, g.M, static_cast<uint64_t>(g.N) * 4, 32, 32)))
        return rc;

    GemmParams p{};
    p.M = g.M;
    p.N = g.N;
    p.K = g.K;
    p.m_tiles = ceil_div(g.M, kBM);
    p.n_tiles = ceil_div(g.N, plan.BN);
    p.kb_total = ceil_div(g.K, g.fp8 ? 2 * kBK : kBK);
    p.ka = plan.ka;
    p.kg_total = ceil_div(p.kb_total, plan.ka);
    p.tma_c = tma_c;
    p.split = plan.split;
    p.stages = plan.stages;
    p.group_m = plan.group_m;
    p.n_vec4 = (g.N % 4 == 0) ? 1 : 0;
    p.alpha = g.alpha;
    p.beta = g.beta;
    p.C = g.C;
    p.bias = g.bias_n;
    p.timeout_ns = wait_timeout_ns();
    p.err = ds.err_word;

    KernelFn fn = g.fp8 ? pick_kernel_f8(plan.BN) : pick_kernel(plan.BN, a_mn, b_mn);
    if (!fn) return set_error(ISAM_ERR_UNSUPPORTED, "isam_gemm: no kernel for BN=%d", plan.BN);
    if ((rc = ensure_smem_optin(reinterpret_cast<const void *>(fn), static_cast<int>(plan.smem), ds.device,
                                "cudaFuncSetAttribute(gemm)")))
        return rc;

    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    cfg.gridDim = dim3(static_cast<unsigned>(plan.grid), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = plan.smem;
    cfg.stream = stream;
    cfg.attrs = attr;
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.numAttrs = 1;
    if (plan.split > 1) {
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = static_cast<unsigned>(plan.split);
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.numAttrs = 2;
    }
    cudaError_t e = cudaLaunchKernelEx(&cfg, fn, ta, tb, tc, p);
    if (e != cudaSuccess) return cuda_error(e, "launch gemm_tc_kernel");
    return ISAM_OK;
}

}  // namespace isam
