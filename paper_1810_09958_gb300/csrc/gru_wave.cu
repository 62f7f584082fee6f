// gru_wave.cu -- two stacked GRU layers in one persistent kernel.
//
// Layer b reads layer a's states, so step t of b can run as soon as step t of
// a is done: in round r the kernel advances layer a to step r and layer b to
// step r - 1, and two layers take T + 1 rounds instead of 2 T.  The grid is
// the single-layer recurrence's (hidden / 32 clusters of 4 CTAs, each CTA one
// K quarter of one group of 32 units), but every CTA keeps three weight slices
// resident: U_a, W_b and U_b (96 rows x K quarter each).  Per round it loads
// its quarter of bf16(h_a at step r - 1) and of bf16(h_b at step r - 2), and
// issues three products into three TMEM accumulators:
//
//   U_a h_a  -> layer a's recurrent term for step r
//   W_b h_a  -> layer b's input projection for step r - 1 (the same h_a tile:
//              the input projection of the upper layer comes from data the
//              lower layer already loaded, Section 5.1.2's reuse)
//   U_b h_b  -> layer b's recurrent term for step r - 1
//
// The partial rows of all three go to the CTA owning their units (DSMEM,
// st.async counted on one barrier), which sums the 4 K ranks in rank order,
// evaluates both layers' gates in fp32 and publishes both new states through
// one grid-wide step counter.  Layer a's projection x W_a^T + b_ih for all
// steps is a GEMM before the kernel.  Reset gate after the recurrent product,
// hidden a multiple of 256 (4 K splits), batch <= 32.  Every wait is bounded.
#include <cstdio>
#include <cstdlib>
#include <mutex>

#include "gru_common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace isam {

namespace {

constexpr int kKS = 4;                   // K splits = cluster size
constexpr int kGroup = 32;               // hidden units per cluster
constexpr int kUO = kGroup / kKS;        // units whose gates a CTA evaluates (8)
constexpr int kBatchPad = 32;
constexpr int kThreads = 128;
constexpr int kNP = kUO * kBatchPad / kThreads;  // (unit, batch) pairs per thread and layer (2)
constexpr int kBStep = kThreads / kUO;           // batch stride between a thread's pairs (16)
constexpr int kAtomU = 3 * kGroup * 128;  // one 64-wide K atom of a 96-row weight slice (12 KB)
constexpr int kAtomH = kBatchPad * 128;   // one K atom of h (4 KB)
constexpr int kBlocks = 9;                // partial-row blocks per source: 3 products x 3 gates
constexpr int kRecvStride = kBatchPad + 4;
constexpr int kMaxPieces = 4;

enum : uint32_t {
    SITE_WAVE_W = 0x221,
    SITE_WAVE_H = 0x222,
    SITE_WAVE_MMA = 0x223,
    SITE_WAVE_RED = 0x224,
};

struct WaveParams {
    int T, batch, H;
    int ka, n_cta, nq, qk;
    const float *gx_a;         // [T*batch][3H]: x W_a^T + b_ih_a
    const float *b_hh_a;       // [3H]
    const float *b_ih_b;       // [3H]
    const float *b_hh_b;       // [3H]
    const float *h0_a, *h0_b;  // [batch][H] or null
    float *out_a, *out_b;      // [T][batch][H]
    uint16_t *hx_a, *hx_b;     // [2][32][H] bf16 exchange of each layer's state
    uint32_t *counter;         // grid-wide round counter (zeroed before launch)
    int skip_publish_cta;      // debug: this CTA never publishes (-1: none)
    unsigned long long timeout_ns;
    uint32_t *err;
};

struct WaveLayout {
    int off_ua, off_wb, off_ub, off_ha, off_hb, off_recv, off_bars, total;
};

// U_a | W_b | U_b | h_a tile | h_b tile | partial rows | barriers.  An M = 128
// MMA over a 96-row atom reads 32 rows past it; for the last atom of each
// slice those rows belong to the next region, so every read stays inside the
// allocation.
__host__ __device__ inline WaveLayout wave_layout(int ka) {
    WaveLayout L;
    L.off_ua = 0;
    L.off_wb = ka * kAtomU;
    L.off_ub = 2 * ka * kAtomU;
    L.off_ha = 3 * ka * kAtomU;
    L.off_hb = L.off_ha + ka * kAtomH;
    L.off_recv = L.off_hb + ka * kAtomH;
    L.off_bars = L.off_recv + kKS * kBlocks * kUO * kRecvStride * 4;
    L.total = L.off_bars + 256 + 1024;
    return L;
}

__global__ void __launch_bounds__(kThreads, 1)
    gru_wave_kernel(const __grid_constant__ CUtensorMap tmUa, const __grid_constant__ CUtensorMap tmWb,
                    const __grid_constant__ CUtensorMap tmUb, const __grid_constant__ CUtensorMap tmHa0,
                    const __grid_constant__ CUtensorMap tmHa1, const __grid_constant__ CUtensorMap tmHb0,
                    const __grid_constant__ CUtensorMap tmHb1, const WaveParams p) {
    if (!launch_shape_ok(p.err, static_cast<uint32_t>(kKS), static_cast<uint32_t>(p.n_cta), 0x3E0u)) return;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    const WaveLayout L = wave_layout(p.ka);
    uint8_t *sUa = smem + L.off_ua;
    uint8_t *sWb = smem + L.off_wb;
    uint8_t *sUb = smem + L.off_ub;
    uint8_t *sHa = smem + L.off_ha;
    uint8_t *sHb = smem + L.off_hb;
    float *recv = reinterpret_cast<float *>(smem + L.off_recv);  // [src][block][unit][36]
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L.off_bars);
    uint64_t *wbar = bars;                       // weight slices landed
    uint64_t *hbar_a = bars + 1;                 // [kMaxPieces] h_a piece landed
    uint64_t *hbar_b = hbar_a + kMaxPieces;      // [kMaxPieces] h_b piece landed
    uint64_t *mma_done = hbar_b + kMaxPieces;    // the round's products complete
    uint64_t *red_full = mma_done + 1;           // all partial rows of my units arrived
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(red_full + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int H = p.H;
    const int G = 3 * H;
    const int T = p.T;
    const int group = blockIdx.x / kKS;
    const uint32_t rank = cluster_ctarank();
    const int unit0 = group * kGroup;
    const int atom0 = static_cast<int>(rank) * p.ka;
    const WaitCtx w{p.timeout_ns, p.err, abort_flag};
    // Products active in round r: U_a h_a while layer a has a step (r < T),
    // W_b h_a and U_b h_b while layer b has one (r >= 1).
    auto round_bytes = [&](int r) {
        const int nprod = (r < T ? 1 : 0) + (r >= 1 ? 2 : 0);
        return static_cast<uint32_t>(kKS * nprod * 3 * kUO * kBatchPad * 4);
    };

    if (tid == 0) {
        mbar_init(wbar, 1);
        for (int q = 0; q < kMaxPieces; ++q) {
            mbar_init(&hbar_a[q], 1);
            mbar_init(&hbar_b[q], 1);
        }
        mbar_init(mma_done, 1);
        mbar_init(red_full, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    __syncwarp();
    if (warp == 0) {  // accumulators: U_a h_a at column 0, W_b h_a at 32, U_b h_b at 64
        tmem_alloc(tmem_slot, 128);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();  // peers' barriers exist before any remote arrive
    tc_fence_after();
    const uint32_t tmem_d = *tmem_slot;
    if (tid == 0) mbar_arrive_expect_tx(red_full, round_bytes(0));

    // ---- priming: the three weight slices, and both layers' initial states.
    if (tid == 0) {
        tma_prefetch_desc(&tmUa);
        tma_prefetch_desc(&tmWb);
        tma_prefetch_desc(&tmUb);
        tma_prefetch_desc(&tmHa0);
        tma_prefetch_desc(&tmHa1);
        tma_prefetch_desc(&tmHb0);
        tma_prefetch_desc(&tmHb1);
        mbar_arrive_expect_tx(wbar, static_cast<uint32_t>(3 * p.ka * kAtomU));
        for (int a = 0; a < p.ka; ++a) {
            tma_load_3d(&tmUa, wbar, sUa + a * kAtomU, (atom0 + a) * 64, unit0, 0);
            tma_load_3d(&tmWb, wbar, sWb + a * kAtomU, (atom0 + a) * 64, unit0, 0);
            tma_load_3d(&tmUb, wbar, sUb + a * kAtomU, (atom0 + a) * 64, unit0, 0);
        }
    }
    __syncwarp();
    // This CTA evaluates both layers' gates for units unit0 + rank*8 + [0, 8);
    // thread tid takes unit ui = tid % 8 and batch rows tid / 8 + 16 k.
    const int ui = tid % kUO;
    const int j = unit0 + static_cast<int>(rank) * kUO + ui;
    const float bhA_r = p.b_hh_a[j], bhA_z = p.b_hh_a[H + j], bhA_n = p.b_hh_a[2 * H + j];
    const float biB_r = p.b_ih_b[j], biB_z = p.b_ih_b[H + j], biB_n = p.b_ih_b[2 * H + j];
    const float bhB_r = p.b_hh_b[j], bhB_z = p.b_hh_b[H + j], bhB_n = p.b_hh_b[2 * H + j];
    float ha[kNP], hb[kNP];
#pragma unroll
    for (int k = 0; k < kNP; ++k) {
        const int b = tid / kUO + k * kBStep;
        ha[k] = (p.h0_a != nullptr && b < p.batch) ? p.h0_a[static_cast<size_t>(b) * H + j] : 0.0f;
        hb[k] = (p.h0_b != nullptr && b < p.batch) ? p.h0_b[static_cast<size_t>(b) * H + j] : 0.0f;
        if (b < p.batch) {
            p.hx_a[static_cast<size_t>(b) * H + j] = f32_to_bf16_rne(ha[k]);
            p.hx_b[static_cast<size_t>(b) * H + j] = f32_to_bf16_rne(hb[k]);
        }
    }
    fence_proxy_async_global();
    __syncwarp();
    __syncthreads();
    if (tid == 0 && static_cast<int>(blockIdx.x) != p.skip_publish_cta) red_release_gpu_add(p.counter, 1u);
    bool ok = true;
    if (tid == 32) ok = bounded_wait(wbar, 0, w, SITE_WAVE_W);
    __syncwarp();

    const uint32_t idesc = idesc_bf16_f32(128, kBatchPad, false, false);
    int issued_round = -1;  // last round whose h loads were issued (for the drain)
    // Layer a's input projection of a step, loaded a round ahead of its use.
    float gxr[kNP], gxz[kNP], gxn[kNP];
    auto load_gx = [&](int t) {
#pragma unroll
        for (int k = 0; k < kNP; ++k) {
            const int b = tid / kUO + k * kBStep;
            if (b < p.batch && t < T) {
                const float *g = p.gx_a + (static_cast<size_t>(t) * p.batch + b) * G + j;
                gxr[k] = __ldg(g);
                gxz[k] = __ldg(g + H);
                gxn[k] = __ldg(g + 2 * H);
            } else {
                gxr[k] = gxz[k] = gxn[k] = 0.0f;
            }
        }
    };
    load_gx(0);
    int last_a = -1, last_b = -1;  // steps whose states still have to go to out_a / out_b
    auto write_out = [&]() {
#pragma unroll
        for (int k = 0; k < kNP; ++k) {
            const int b = tid / kUO + k * kBStep;
            if (b >= p.batch) continue;
            if (last_a >= 0) p.out_a[(static_cast<size_t>(last_a) * p.batch + b) * H + j] = ha[k];
            if (last_b >= 0) p.out_b[(static_cast<size_t>(last_b) * p.batch + b) * H + j] = hb[k];
        }
        last_a = last_b = -1;
    };

    // ---- rounds r = 0..T: layer a step r (r < T), layer b step r - 1 (r >= 1).
    for (int r = 0; r <= T; ++r) {
        const bool stepA = r < T, stepB = r >= 1;
        const uint32_t par = static_cast<uint32_t>(r & 1);
        if (tid == 0 && !*abort_flag) {
            if (wait_counter(p.counter, static_cast<uint32_t>((r + 1) * p.n_cta), w)) {
                fence_proxy_async_global();
                // h_a at step r - 1 sits in slot r & 1, h_b at step r - 2 in slot (r - 1) & 1.
                const CUtensorMap *ma = (r & 1) ? &tmHa1 : &tmHa0;
                const CUtensorMap *mb = ((r - 1) & 1) ? &tmHb1 : &tmHb0;
                for (int q = 0; q < p.nq; ++q) {
                    mbar_arrive_expect_tx(&hbar_a[q], static_cast<uint32_t>(p.qk * kAtomH));
                    tma_load_3d(ma, &hbar_a[q], sHa + q * p.qk * kAtomH, 0, 0, atom0 + q * p.qk);
                }
                if (stepB)
                    for (int q = 0; q < p.nq; ++q) {
                        mbar_arrive_expect_tx(&hbar_b[q], static_cast<uint32_t>(p.qk * kAtomH));
                        tma_load_3d(mb, &hbar_b[q], sHb + q * p.qk * kAtomH, 0, 0, atom0 + q * p.qk);
                    }
                issued_round = r;
            }
        }
        __syncwarp();
        // Off thread 0's path to the next counter poll: the states of the last
        // round to out_a / out_b and this round's projection of layer a.
        write_out();
        if (r > 0) load_gx(r);
        if (tid == 32 && ok) {
            // Products over h_a as its pieces land, then U_b h_b.
            for (int q = 0; q < p.nq && ok; ++q) {
                if (!bounded_wait(&hbar_a[q], par, w, SITE_WAVE_H)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int a = q * p.qk; a < (q + 1) * p.qk; ++a) {
                    const uint32_t ha_s = smem_u32(sHa + a * kAtomH);
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint64_t bd = sdesc_sw128(ha_s + k * 32, 16, 1024);
                        const uint32_t acc = (a > 0 || k > 0) ? 1u : 0u;
                        if (stepA) umma_bf16(tmem_d, sdesc_sw128(smem_u32(sUa + a * kAtomU) + k * 32, 16, 1024), bd, idesc, acc);
                        if (stepB) umma_bf16(tmem_d + 32, sdesc_sw128(smem_u32(sWb + a * kAtomU) + k * 32, 16, 1024), bd, idesc, acc);
                    }
                }
            }
            if (stepB)
                for (int q = 0; q < p.nq && ok; ++q) {
                    // h_b pieces land from round 1 on: their phase parity is that of r - 1.
                    if (!bounded_wait(&hbar_b[q], par ^ 1u, w, SITE_WAVE_H)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    for (int a = q * p.qk; a < (q + 1) * p.qk; ++a) {
                        const uint32_t hb_s = smem_u32(sHb + a * kAtomH);
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            umma_bf16(tmem_d + 64, sdesc_sw128(smem_u32(sUb + a * kAtomU) + k * 32, 16, 1024),
                                      sdesc_sw128(hb_s + k * 32, 16, 1024), idesc, (a > 0 || k > 0) ? 1u : 0u);
                    }
                }
            if (ok) umma_commit(mma_done);
        }
        __syncwarp();
        if (!__syncthreads_and(bounded_wait(mma_done, par, w, SITE_WAVE_MMA) ? 1 : 0)) break;
        tc_fence_after();
        // Push: warp g holds gate g's rows (TMEM lane = unit within the group)
        // of each active product; row u goes to the cluster CTA owning unit u,
        // block (product * 3 + gate) of its slot for this source rank.
        if (warp < 3) {
            const uint32_t owner = static_cast<uint32_t>(lane / kUO);
            const int oui = lane % kUO;
            const uint32_t rbar = mapa_shared(smem_u32(red_full), owner);
#pragma unroll
            for (int prod = 0; prod < 3; ++prod) {
                if (prod == 0 ? !stepA : !stepB) continue;
                uint32_t v[32];
                tmem_ld32(tmem_d + (static_cast<uint32_t>(warp * 32) << 16) + static_cast<uint32_t>(prod * 32), v);
                tmem_ld_wait(v);
                const uint32_t dst = mapa_shared(
                    smem_u32(recv + ((static_cast<int>(rank) * kBlocks + prod * 3 + warp) * kUO + oui) * kRecvStride),
                    owner);
#pragma unroll
                for (int c = 0; c < 8; ++c)
                    st_async_f4(dst + c * 16,
                                make_float4(__uint_as_float(v[4 * c]), __uint_as_float(v[4 * c + 1]),
                                            __uint_as_float(v[4 * c + 2]), __uint_as_float(v[4 * c + 3])),
                                rbar);
            }
        }
        tc_fence_before();
        __syncwarp();
        if (!__syncthreads_and(bounded_wait<true>(red_full, par, w, SITE_WAVE_RED) ? 1 : 0)) break;
        // Gates, partials summed over the 4 source ranks in rank order.
        uint16_t *hxa_next = p.hx_a + static_cast<size_t>((r + 1) & 1) * kBatchPad * H;
        uint16_t *hxb_next = p.hx_b + static_cast<size_t>(r & 1) * kBatchPad * H;
        auto part = [&](int s, int blk, int b) {
            return recv[((s * kBlocks + blk) * kUO + ui) * kRecvStride + b];
        };
#pragma unroll
        for (int k = 0; k < kNP; ++k) {
            const int b = tid / kUO + k * kBStep;
            if (b >= p.batch) continue;
            if (stepA) {
                float gr = bhA_r, gz = bhA_z, gn = bhA_n;
#pragma unroll
                for (int s = 0; s < kKS; ++s) {
                    gr += part(s, 0, b);
                    gz += part(s, 1, b);
                    gn += part(s, 2, b);
                }
                const float rg = sigmoidf_fast(gxr[k] + gr);
                const float zg = sigmoidf_fast(gxz[k] + gz);
                const float ng = tanhf_fast(gxn[k] + rg * gn);
                ha[k] = (1.0f - zg) * ng + zg * ha[k];
                hxa_next[static_cast<size_t>(b) * H + j] = f32_to_bf16_rne(ha[k]);
            }
            if (stepB) {
                float xr = biB_r, xz = biB_z, xn = biB_n;
                float gr = bhB_r, gz = bhB_z, gn = bhB_n;
#pragma unroll
                for (int s = 0; s < kKS; ++s) {
                    xr += part(s, 3, b);
                    xz += part(s, 4, b);
                    xn += part(s, 5, b);
                    gr += part(s, 6, b);
                    gz += part(s, 7, b);
                    gn += part(s, 8, b);
                }
                const float rg = sigmoidf_fast(xr + gr);
                const float zg = sigmoidf_fast(xz + gz);
                const float ng = tanhf_fast(xn + rg * gn);
                hb[k] = (1.0f - zg) * ng + zg * hb[k];
                hxb_next[static_cast<size_t>(b) * H + j] = f32_to_bf16_rne(hb[k]);
            }
        }
        if (stepA) last_a = r;
        if (stepB) last_b = r - 1;
        // Publish both states (the release waits only for the exchange-buffer
        // stores), then arm the barrier for the next round's partial rows.
        fence_proxy_async_global();
        __syncthreads();
        if (tid == 0 && static_cast<int>(blockIdx.x) != p.skip_publish_cta) red_release_gpu_add(p.counter, 1u);
        if (tid == 0) mbar_arrive_expect_tx(red_full, round_bytes(r + 1));
        __syncwarp();
        tc_fence_after();
    }
    write_out();

    // ---- teardown: let issued copies land, release TMEM.
    if (tid == 0 && issued_round >= 0 && *abort_flag) {
        const uint32_t rp = static_cast<uint32_t>(issued_round & 1);
        for (int q = 0; q < p.nq; ++q) {
            const unsigned long long t0 = globaltimer();
            while (!mbar_try_wait(smem_u32(&hbar_a[q]), rp))
                if (globaltimer() - t0 > p.timeout_ns) break;
            if (issued_round >= 1) {
                const unsigned long long t1 = globaltimer();
                while (!mbar_try_wait(smem_u32(&hbar_b[q]), rp ^ 1u))
                    if (globaltimer() - t1 > p.timeout_ns) break;
            }
        }
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    // No CTA leaves while a cluster peer may still write into its shared
    // memory; every wait above is bounded, so every CTA gets here.
    cluster_sync_all();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem_d, 128);
    }
}

}  // namespace

size_t gru_wave_smem_bytes(int H) { return static_cast<size_t>(wave_layout(H / (kKS * 64)).total); }

bool gru_wave_fits(int H, int batch, int num_sms, int smem_optin) {
    if (H % 256 != 0 || H < 256 || H > 1024 || batch < 1 || batch > kBatchPad) return false;
    if (H / kGroup * kKS > num_sms) return false;
    return gru_wave_smem_bytes(H) <= static_cast<size_t>(smem_optin);
}

bool gru_wave_supported(int H, int batch, const DeviceState &ds) {
    return gru_wave_fits(H, batch, ds.num_sms, ds.max_smem_optin);
}

namespace {

// A layer's weight slice map: [3 gates][H rows][H] with boxes of 96 rows (one
// group) over one 64-wide K atom.
int wave_weight_map(const uint16_t *Wt, int H, CUtensorMap *tm) {
    const uint64_t dims[3] = {static_cast<uint64_t>(H), static_cast<uint64_t>(H), 3};
    const uint64_t strides[2] = {static_cast<uint64_t>(H) * 2, static_cast<uint64_t>(H) * H * 2};
    const uint32_t box[3] = {64, kGroup, 3};
    return make_tmap_3d_bf16(tm, Wt, dims, strides, box);
}

// One exchange slot [32 batch rows][H] as [H/64 atoms][32][64]; box = one
// piece of qk atoms of a CTA's K quarter.
int wave_exchange_map(const uint16_t *slot, int H, int qk, CUtensorMap *tm) {
    const uint64_t dims[3] = {64, kBatchPad, static_cast<uint64_t>(H / 64)};
    const uint64_t strides[2] = {static_cast<uint64_t>(H) * 2, 128};
    const uint32_t box[3] = {64, kBatchPad, static_cast<uint32_t>(qk)};
    return make_tmap_3d_bf16(tm, slot, dims, strides, box);
}


}  // namespace

int gru_wave_launch(int T, int batch, int H, const float *gx_a, const uint16_t *U_a, const uint16_t *W_b,
                    const uint16_t *U_b, const float *b_a, const float *b_b, const float *h0_a,
                    const float *h0_b, float *out_a, float *out_b, uint16_t *hx_a, uint16_t *hx_b,
                    uint32_t *counter, DeviceState &ds, cudaStream_t stream) {
    if (!gru_wave_supported(H, batch, ds))
        return set_error(ISAM_ERR_UNSUPPORTED, "two-layer GRU kernel: hidden %d, batch %d not supported", H, batch);
    WaveParams p{};
    p.T = T;
    p.batch = batch;
    p.H = H;
    p.ka = H / (kKS * 64);
    p.nq = (p.ka % 4 == 0) ? 4 : (p.ka % 3 == 0) ? 3 : (p.ka % 2 == 0) ? 2 : 1;
    p.qk = p.ka / p.nq;
    p.n_cta = H / kGroup * kKS;
    p.gx_a = gx_a;
    p.b_hh_a = b_a + 3 * H;
    p.b_ih_b = b_b;
    p.b_hh_b = b_b + 3 * H;
    p.h0_a = h0_a;
    p.h0_b = h0_b;
    p.out_a = out_a;
    p.out_b = out_b;
    p.hx_a = hx_a;
    p.hx_b = hx_b;
    p.counter = counter;
    p.skip_publish_cta = -1;
    if (const char *s = getenv("ISAM_DEBUG_GRU_SKIP_CTA")) p.skip_publish_cta = atoi(s);
    p.timeout_ns = wait_timeout_ns();
    p.err = ds.err_word;

    CUtensorMap tmUa, tmWb, tmUb, tmHa0, tmHa1, tmHb0, tmHb1;
    const size_t slot = static_cast<size_t>(kBatchPad) * H;
    int rc;
    if ((rc = wave_weight_map(U_a, H, &tmUa)) || (rc = wave_weight_map(W_b, H, &tmWb)) ||
        (rc = wave_weight_map(U_b, H, &tmUb)) || (rc = wave_exchange_map(hx_a, H, p.qk, &tmHa0)) ||
        (rc = wave_exchange_map(hx_a + slot, H, p.qk, &tmHa1)) || (rc = wave_exchange_map(hx_b, H, p.qk, &tmHb0)) ||
        (rc = wave_exchange_map(hx_b + slot, H, p.qk, &tmHb1)))
        return rc;
    if ((rc = ensure_smem_optin(reinterpret_cast<const void *>(gru_wave_kernel), ds.max_smem_optin, ds.device,
                                "cudaFuncSetAttribute(gru wave)")))
        return rc;
    cudaError_t e = cudaMemsetAsync(counter, 0, sizeof(uint32_t), stream);
    if (e != cudaSuccess) return cuda_error(e, "clearing the GRU round counter");
    const size_t smem = gru_wave_smem_bytes(H);
    cudaLaunchConfig_t cfg = {};
    // A plain cluster launch, once every cluster is known to fit at the same
    // time (the round counter needs every CTA resident); no cooperative
    // attribute, whose combination with the cluster shape a tool's re-issue
    // of the launch can drop.
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kKS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(p.n_cta), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int max_clusters = 0;
    e = cudaOccupancyMaxActiveClusters(&max_clusters, gru_wave_kernel, &cfg);
    if (e != cudaSuccess) return cuda_error(e, "cudaOccupancyMaxActiveClusters(gru wave)");
    if (max_clusters * kKS < p.n_cta)
        return set_error(ISAM_ERR_UNSUPPORTED, "two-layer GRU kernel: %d CTAs in clusters of 4 cannot be co-resident",
                         p.n_cta);
    e = cudaLaunchKernelEx(&cfg, gru_wave_kernel, tmUa, tmWb, tmUb, tmHa0, tmHa1, tmHb0, tmHb1, p);
    if (e != cudaSuccess) return cuda_error(e, "launch gru_wave_kernel");
    return ISAM_OK;
}

}  // namespace isam
