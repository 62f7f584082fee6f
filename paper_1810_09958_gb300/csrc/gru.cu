// gru.cu -- GRU forward over T steps on sm_103a.
//
// Recurrent scheduling after Section 3.6 of the paper: the loop body is
// scheduled once as a priming iteration (load the persistent weights and the
// initial state onto the compute units), a recursive iteration run T times
// that overwrites its own inputs, and a finish iteration (the last state is
// already in place in h_out).  The paper credits its GRU speed-up to fusion
// and to keeping reused data on chip (Section 5.1.2); here:
//
//   1. gx = x W^T + b_ih for all T steps is one GEMM (isam_gemm's kernel, bias
//      fused in its epilogue), written to a library workspace;
//   2. one persistent kernel runs the recurrence.  Hidden units are taken in
//      groups of 32; a group is a cluster of KS CTAs (KS = 4 at hidden 1024)
//      that split the reduction dimension of U h: CTA r keeps the 96 rows of U
//      for the group's r, z and n gates over its K quarter resident in shared
//      memory for all T steps.  Per step each CTA TMA-loads its quarter of
//      bf16(h_{t-1}) (all batch rows), runs 16 tcgen05.mma (M = 128 with 96
//      rows used, N = 32 batch) into TMEM, and pushes the partial rows of the
//      units owned by each cluster peer straight into that peer's shared
//      memory; the owner sums the KS partials in rank order, evaluates the
//      gates in fp32 (h carried in fp32 registers), publishes bf16(h_t) to an
//      exchange buffer, signals a grid-wide step counter, then writes h_t to
//      h_out.  Splitting K keeps the per-step tensor instruction count per CTA
//      low: at this size each M = 128 instruction costs about the same
//      whatever its N, so the step time is set by instructions per CTA.
//      Every wait is bounded in time.
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <mutex>

#include <cuda_bf16.h>

#include "gru_common.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace isam {

namespace {

constexpr int kGroup = 32;               // hidden units per group (one cluster)
constexpr int kRowsG = 3 * kGroup;       // 96 U rows per group (r, z, n)
constexpr int kBatchPad = 32;            // MMA N for batch <= 32 (the path with every feature)
constexpr int kBatchMax = 256;           // larger batches run in chunks of the padded width
constexpr int kThreads = 128;
constexpr int kAtomU = kRowsG * 128;     // one 64-wide K atom of the U slice (12 KB)
constexpr int kUPad = 32 * 128;          // the M = 128 MMA reads 32 rows past an atom
// The padded batch BP (32, 64 or 128) is the MMA's N: one K atom of h is BP
// rows of 128 bytes, and a received partial row holds BP batch values padded
// to BP + 4 floats, so the 8 units a warp reads fall into different banks.
__host__ __device__ constexpr int atom_h_bytes(int bp) { return bp * 128; }
__host__ __device__ constexpr int recv_stride(int bp) { return bp + 4; }
__host__ __device__ constexpr int recv_bytes(int bp) { return kRowsG * recv_stride(bp) * 4; }
constexpr int kMaxPieces = 4;

enum : uint32_t {
    SITE_GRU_U = 0x202,
    SITE_GRU_H = 0x203,
    SITE_GRU_MMA = 0x204,
    SITE_GRU_RED = 0x205,
    SITE_GRU_W = 0x206,
};


struct GruParams {
    int T, batch, H;
    int bstride;               // batch rows between two steps of gx / h_out (the full batch; batch is this chunk's rows)
    int ks;                    // K splits per unit group = cluster size
    int ka;                    // 64-wide K atoms per CTA (all atoms of H, rounded up, / ks)
    int uo;                    // units whose gates one CTA evaluates (32 / ks)
    int n_cta;                 // (H / 32) * ks
    int nq, qk;                // h arrives in nq pieces of qk atoms (nq * qk == ka)
    int h2d;                   // hidden % 64 == 32: h maps are 2-D, one box per atom (the last half outside)
    const float *gx;           // [T*batch][3H], includes b_ih
    const float *b_hh;         // [3H]
    const float *h0;           // [batch][H] or null
    float *h_out;              // [T][batch][H]
    uint16_t *hx;              // [2][32][H] bf16 exchange of h
    uint16_t *rhx;             // [2][32][H] bf16 exchange of r * h (reset_before)
    int reset_before;          // candidate's recurrent input U_n (r * h): two rounds per step
    int gx_parts;              // slabs summed into each projection value (1: gx = x W^T + b_ih)
    size_t gx_slab;            // floats between two slabs of gx
    const float *b_ih;         // [3H], added to the slab sum when gx_parts > 1 (else null)
    int has_next;              // also multiply the next layer's W by every loaded h
    float *gxp_out;            // [ks][T*batch][3H]: the next layer's projection, one slab per K rank
    uint32_t *counter;         // step counter (zeroed before launch)
    int skip_publish_cta;      // debug: this CTA never publishes (-1: none)
    unsigned long long timeout_ns;
    uint32_t *err;
};

struct GruLayout {
    int off_u, off_w, off_h, off_recv, off_bars, total;
};

// U slice | next layer's W slice (has_next) | pad | h piece | partial rows | barriers.
__host__ __device__ inline GruLayout gru_layout(int ka, bool has_next, int bp = kBatchPad) {
    GruLayout L;
    L.off_u = 0;
    L.off_w = ka * kAtomU;
    L.off_h = L.off_w + (has_next ? ka * kAtomU : 0) + kUPad;
    L.off_recv = L.off_h + ka * atom_h_bytes(bp);
    L.off_bars = L.off_recv + recv_bytes(bp);
    L.total = L.off_bars + 128 + 1024;
    return L;
}

// Template arguments: KS, the K splits per unit group (cluster size, 4, 2 or
// 1), and BP, the padded batch (the MMA's N: 32, 64 or 128).  A CTA evaluates
// the gates of UO = 32 / KS units over BP batch rows, NP = UO * BP / 128
// (unit, batch) pairs per thread.  The next layer's product and the K-rank
// projection slabs exist for BP = 32 only.
template <int KS, int BP>
__global__ void __launch_bounds__(kThreads, 1)
    gru_recurrent_kernel(const __grid_constant__ CUtensorMap tmU,
                         const __grid_constant__ CUtensorMap tmH0,
                         const __grid_constant__ CUtensorMap tmH1,
                         const __grid_constant__ CUtensorMap tmR0,
                         const __grid_constant__ CUtensorMap tmR1,
                         const __grid_constant__ CUtensorMap tmWn, const GruParams p) {
    constexpr int UO = kGroup / KS;
    constexpr int NP = UO * BP / kThreads;
    constexpr int SL = BP == kBatchPad ? KS : 1;  // projection slabs a value can sum
    constexpr int AH = atom_h_bytes(BP);
    constexpr int RS = recv_stride(BP);
    constexpr int BSTEP = kThreads / UO;
    if (!launch_shape_ok(p.err, static_cast<uint32_t>(KS), static_cast<uint32_t>(p.n_cta), 0x3F0u))
        return;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                ~static_cast<uintptr_t>(1023));
    const bool HN = p.has_next != 0;
    const GruLayout L = gru_layout(p.ka, HN, BP);
    uint8_t *sU = smem + L.off_u;
    uint8_t *sW = smem + L.off_w;
    uint8_t *sH = smem + L.off_h;
    float *recv = reinterpret_cast<float *>(smem + L.off_recv);  // [ks src][3 gates][uo][32 batch]
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L.off_bars);
    uint64_t *ubar = bars;                  // U (and next W) slice landed
    uint64_t *hbar = bars + 1;              // [kMaxPieces] h piece landed
    uint64_t *mma_done = hbar + kMaxPieces; // MMAs of the step complete
    uint64_t *red_full = mma_done + 1;      // all partial rows of my units arrived
    uint64_t *w_done = red_full + 1;        // next layer's projection MMAs complete
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(w_done + 1);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;
    const int H = p.H;
    const int G = 3 * H;
    const int group = blockIdx.x / KS;
    const uint32_t rank = KS > 1 ? cluster_ctarank() : 0u;
    const int unit0 = group * kGroup;
    const int atom0 = static_cast<int>(rank) * p.ka;
    const WaitCtx w{p.timeout_ns, p.err, abort_flag};

    if (tid == 0) {
        mbar_init(ubar, 1);
        for (int q = 0; q < kMaxPieces; ++q) mbar_init(&hbar[q], 1);
        mbar_init(mma_done, 1);
        mbar_init(red_full, 1);  // armed with the bytes of a step's partial rows
        mbar_init(w_done, 1);
        *abort_flag = 0;
        fence_mbar_init();
    }
    __syncwarp();
    // Columns 0-31: the recurrent product; 32-95: the next layer's projection,
    // double-buffered by step parity.
    const uint32_t tmem_cols = HN ? 128u : static_cast<uint32_t>(BP);
    if (warp == 0) {
        tmem_alloc(tmem_slot, tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    if (KS > 1) cluster_sync_all();  // peers' barriers exist before any remote arrive
    tc_fence_after();
    const uint32_t tmem_d = *tmem_slot;
    // A step is one round (all three gates' rows from h_{t-1}) or, with the
    // reset gate before the product, two: round 0 takes the r and z rows from
    // h_{t-1} and publishes r * h_{t-1}; round 1 takes the n rows from it.
    // Partial rows of a round for my units: KS sources x gates x UO x 32.
    const bool RB = p.reset_before != 0;
    const int nph = RB ? 2 : 1;
    auto round_bytes = [&](int ph) {
        return static_cast<uint32_t>(KS * (RB ? (ph == 0 ? 2 : 1) : 3) * UO * BP * 4);
    };
    if (tid == 0) mbar_arrive_expect_tx(red_full, round_bytes(0));

    // ---- priming iteration: persistent weights and initial state.
    if (tid == 0) {
        tma_prefetch_desc(&tmU);
        tma_prefetch_desc(&tmH0);
        tma_prefetch_desc(&tmH1);
        if (RB) {
            tma_prefetch_desc(&tmR0);
            tma_prefetch_desc(&tmR1);
        }
        mbar_arrive_expect_tx(ubar, static_cast<uint32_t>(p.ka * kAtomU * (HN ? 2 : 1)));
        for (int a = 0; a < p.ka; ++a)
            tma_load_3d(&tmU, ubar, sU + a * kAtomU, (atom0 + a) * 64, unit0, 0);
        if (HN)
            for (int a = 0; a < p.ka; ++a)
                tma_load_3d(&tmWn, ubar, sW + a * kAtomU, (atom0 + a) * 64, unit0, 0);
    }
    __syncwarp();
    // This CTA evaluates the gates of units unit0 + rank*UO + [0, UO); thread
    // tid takes unit ui = tid % UO and batch rows b = tid / UO + k * BSTEP.
    const int ui = tid % UO;
    const int j = unit0 + static_cast<int>(rank) * UO + ui;
    const float bh_r = p.b_hh[j], bh_z = p.b_hh[H + j], bh_n = p.b_hh[2 * H + j];
    const float bi_r = p.b_ih ? p.b_ih[j] : 0.0f, bi_z = p.b_ih ? p.b_ih[H + j] : 0.0f,
                bi_n = p.b_ih ? p.b_ih[2 * H + j] : 0.0f;
    float hprev[NP];
#pragma unroll
    for (int k = 0; k < NP; ++k) {
        const int b = tid / UO + k * BSTEP;
        hprev[k] = (p.h0 != nullptr && b < p.batch) ? p.h0[static_cast<size_t>(b) * H + j] : 0.0f;
        if (b < p.batch) p.hx[static_cast<size_t>(b) * H + j] = f32_to_bf16_rne(hprev[k]);
    }
    fence_proxy_async_global();
    __syncwarp();
    __syncthreads();
    if (tid == 0 && static_cast<int>(blockIdx.x) != p.skip_publish_cta) red_release_gpu_add(p.counter, 1u);
    bool ok = true;
    if (tid == 32) ok = bounded_wait(ubar, 0, w, SITE_GRU_U);
    __syncwarp();

    const uint32_t idesc = idesc_bf16_f32(128, BP, false, false);
    int issued_phase = -1;  // last round whose h loads were issued (for the drain)
    // Input projection of a step (independent of h), loaded one step ahead so
    // its memory latency is off the recurrence's critical path: gx is one slab
    // holding x W^T + b_ih (the GEMM's output), or KS slabs of K-rank partial
    // products computed by the layer below.  The loads land in registers
    // (KS x NP = 8 per gate whatever KS) and are summed, after b_ih and in
    // rank order, only where the gates use them.
    float gxr[SL * NP], gxz[SL * NP], gxn[SL * NP];
    auto load_gx = [&](int tt) {
#pragma unroll
        for (int k = 0; k < NP; ++k) {
            const int b = tid / UO + k * BSTEP;
            const float *g = p.gx + (static_cast<size_t>(tt) * p.bstride + b) * G + j;
#pragma unroll
            for (int s = 0; s < SL; ++s) {
                const int i = k * SL + s;
                if (b < p.batch && tt < p.T && s < p.gx_parts) {
                    const float *gs = g + static_cast<size_t>(s) * p.gx_slab;
                    gxr[i] = __ldg(gs);
                    gxz[i] = __ldg(gs + H);
                    gxn[i] = __ldg(gs + 2 * H);
                } else {
                    gxr[i] = gxz[i] = gxn[i] = 0.0f;
                }
            }
        }
    };
    auto sum_gx = [&](const float (&v)[SL * NP], float bias, int k) {
        float a = bias;
#pragma unroll
        for (int s = 0; s < SL; ++s) a += v[k * SL + s];
        return a;
    };
    load_gx(0);
    int last_t = -1;  // step whose h (in hprev) still has to go to h_out

    // ---- recursive iteration, T times (in nph rounds each), then, when the
    // next layer's projection is fused in, a finish iteration that only
    // multiplies its W by h_{T-1}.  Phase 0 of step t >= 1 multiplies the
    // next layer's W by the h_{t-1} it has just loaded (the next layer's
    // projection of step t - 1 over this CTA's K range) into a second
    // accumulator, after the recurrent product: the h tile serves both.  That
    // product's A operand starts 32 rows early, so W's r, z and n rows land in
    // TMEM lanes 32-127, which warps 1-3 drain; warp 0 stays free to poll.
    float zsave[NP];  // update gate between the two rounds of a step
    bool alive = true;
    int w_pending = -1;  // parity of the last next-layer product committed to w_done
    int w_issued = -1;   // issuing thread: parity of its product not yet drained
    auto issue_w = [&](uint32_t col, uint32_t wp) {
        for (int a = 0; a < p.ka; ++a) {
            // 32 rows (4 KB) before the atom: still inside shared memory (the
            // U slice precedes W).
            const uint32_t wa = smem_u32(sW + a * kAtomU) - 32u * 128u;
            const uint32_t ha = smem_u32(sH + a * AH);
#pragma unroll
            for (int k = 0; k < 4; ++k)
                umma_bf16(tmem_d + col, sdesc_sw128(wa + k * 32, 16, 1024), sdesc_sw128(ha + k * 32, 16, 1024),
                          idesc, (a > 0 || k > 0) ? 1u : 0u);
        }
        umma_commit(w_done);
        w_issued = static_cast<int>(wp);
    };
    const int t_end = p.T + (HN ? 1 : 0);
    for (int t = 0; t < t_end && alive; ++t) {
        const bool finish = t == p.T;
        const int nround = finish ? 1 : nph;
        for (int ph = 0; ph < nround; ++ph) {
            const int round = t * nph + ph;
            const uint32_t par = static_cast<uint32_t>(round & 1);
            const bool wnow = HN && t > 0 && ph == 0;
            const uint32_t wpar = static_cast<uint32_t>((t - 1) & 1);
            const uint32_t wcol = 32u + 32u * wpar;
            if (tid == 0 && !*abort_flag) {
                // The next layer's product of the previous round still reads sH.
                if (wait_counter(p.counter, static_cast<uint32_t>((round + 1) * p.n_cta), w) &&
                    (w_pending < 0 || bounded_wait(w_done, static_cast<uint32_t>(w_pending), w, SITE_GRU_W))) {
                    fence_proxy_async_global();
                    const CUtensorMap *m = ph == 0 ? ((t & 1) ? &tmH1 : &tmH0) : ((t & 1) ? &tmR1 : &tmR0);
                    for (int q = 0; q < p.nq; ++q) {
                        mbar_arrive_expect_tx(&hbar[q], static_cast<uint32_t>(p.qk * AH));
                        if (p.h2d) {
                            // The last atom's upper 32 columns lie past the row:
                            // the 2-D box fills them with zeros (as U's map does).
                            for (int a = q * p.qk; a < (q + 1) * p.qk; ++a)
                                tma_load_2d(m, &hbar[q], sH + a * AH, (atom0 + a) * 64, 0);
                        } else {
                            tma_load_3d(m, &hbar[q], sH + q * p.qk * AH, 0, 0, atom0 + q * p.qk);
                        }
                    }
                    issued_phase = round;
                }
            }
            __syncwarp();
            if (ph == 0 && !finish) {
                // Off thread 0's path to the next counter poll: h_{t-1} to
                // h_out and this step's input projection (still ahead of its
                // use in the gates).
                if (last_t >= 0) {
#pragma unroll
                    for (int k = 0; k < NP; ++k) {
                        const int b = tid / UO + k * BSTEP;
                        if (b < p.batch)
                            p.h_out[(static_cast<size_t>(last_t) * p.bstride + b) * H + j] = hprev[k];
                    }
                    last_t = -1;
                }
                if (t > 0) load_gx(t);
            }
            if (tid == 32 && ok) {
                for (int q = 0; q < p.nq && ok; ++q) {
                    if (!bounded_wait(&hbar[q], par, w, SITE_GRU_H)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    if (finish) continue;
                    for (int a = q * p.qk; a < (q + 1) * p.qk; ++a) {
                        const uint32_t ua = smem_u32(sU + a * kAtomU);
                        const uint32_t ha = smem_u32(sH + a * AH);
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            umma_bf16(tmem_d, sdesc_sw128(ua + k * 32, 16, 1024),
                                      sdesc_sw128(ha + k * 32, 16, 1024), idesc,
                                      (a > 0 || k > 0) ? 1u : 0u);
                    }
                }
                if (ok && !finish) umma_commit(mma_done);
                if (ok && finish) issue_w(wcol, wpar);
            }
            __syncwarp();
            if (!finish) {
                // Block-uniform decision: every thread leaves at the same round.
                if (!__syncthreads_and(bounded_wait(mma_done, par, w, SITE_GRU_MMA) ? 1 : 0)) {
                    alive = false;
                    break;
                }
                tc_fence_after();
                // The next layer's product goes to the tensor pipe now that the
                // recurrent one is done, issued by warp 3, which pushes nothing.
                if (tid == 96 && wnow) issue_w(wcol, wpar);
                // Push: row gate*32 + u of the partial product (TMEM lane = row)
                // goes to the cluster CTA that owns unit u, into its slot for this
                // source rank.  Round 0 of a reset-before step sends the r and z
                // rows, round 1 the n rows.
                const bool pushes = RB ? (ph == 0 ? warp < 2 : warp == 2) : warp < 3;
                if (pushes) {
                    const uint32_t owner = static_cast<uint32_t>(lane / UO);
                    const int oui = lane % UO;
                    const uint32_t dst = mapa_shared(
                        smem_u32(recv + ((static_cast<int>(rank) * 3 + warp) * UO + oui) * RS), owner);
                    const uint32_t rbar = mapa_shared(smem_u32(red_full), owner);
#pragma unroll
                    for (int cb = 0; cb < BP / 32; ++cb) {  // 32 batch columns at a time
                        uint32_t r[32];
                        tmem_ld32(tmem_d + (static_cast<uint32_t>(warp * 32) << 16) + static_cast<uint32_t>(cb * 32), r);
                        tmem_ld_wait(r);
                        // Asynchronous remote stores: each counts its bytes on the
                        // owner's barrier, so nothing here waits for them to land.
#pragma unroll
                        for (int c = 0; c < 8; ++c)
                            st_async_f4(dst + cb * 128 + c * 16,
                                        make_float4(__uint_as_float(r[4 * c]), __uint_as_float(r[4 * c + 1]),
                                                    __uint_as_float(r[4 * c + 2]), __uint_as_float(r[4 * c + 3])),
                                        rbar);
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (!__syncthreads_and(bounded_wait<true>(red_full, par, w, SITE_GRU_RED) ? 1 : 0)) {
                    alive = false;
                    break;
                }
                uint16_t *hx_next = p.hx + static_cast<size_t>((t + 1) & 1) * BP * H;
                uint16_t *rhx_t = p.rhx + static_cast<size_t>(t & 1) * BP * H;
#pragma unroll
                for (int k = 0; k < NP; ++k) {
                    const int b = tid / UO + k * BSTEP;
                    if (b >= p.batch) continue;
                    float ghr = bh_r, ghz = bh_z, ghn = bh_n;
#pragma unroll
                    for (int s = 0; s < KS; ++s) {  // partials summed in rank order
                        const float *rs = recv + (s * 3 * UO + ui) * RS + b;
                        if (!RB || ph == 0) {
                            ghr += rs[0];
                            ghz += rs[UO * RS];
                        }
                        if (!RB || ph == 1) ghn += rs[2 * UO * RS];
                    }
                    if (!RB) {
                        const float rg = sigmoidf_fast(sum_gx(gxr, bi_r, k) + ghr);
                        const float zg = sigmoidf_fast(sum_gx(gxz, bi_z, k) + ghz);
                        const float ng = tanhf_fast(sum_gx(gxn, bi_n, k) + rg * ghn);
                        const float hn = (1.0f - zg) * ng + zg * hprev[k];
                        hprev[k] = hn;
                        hx_next[static_cast<size_t>(b) * H + j] = f32_to_bf16_rne(hn);
                    } else if (ph == 0) {
                        const float rg = sigmoidf_fast(sum_gx(gxr, bi_r, k) + ghr);
                        zsave[k] = sigmoidf_fast(sum_gx(gxz, bi_z, k) + ghz);
                        rhx_t[static_cast<size_t>(b) * H + j] = f32_to_bf16_rne(rg * hprev[k]);
                    } else {
                        const float ng = tanhf_fast(sum_gx(gxn, bi_n, k) + ghn);
                        const float hn = (1.0f - zsave[k]) * ng + zsave[k] * hprev[k];
                        hprev[k] = hn;
                        hx_next[static_cast<size_t>(b) * H + j] = f32_to_bf16_rne(hn);
                    }
                }
                if (ph == nph - 1) last_t = t;  // hprev holds h_t, not yet in h_out
                // Publish first (the release then waits only for the exchange-buffer
                // stores), then write this step's h_t to h_out.
                fence_proxy_async_global();
                __syncthreads();
                if (tid == 0 && static_cast<int>(blockIdx.x) != p.skip_publish_cta)
                    red_release_gpu_add(p.counter, 1u);
                // recv is consumed: arm the barrier for the next round's partial
                // rows (bytes that land before this are counted all the same).
                if (tid == 0) mbar_arrive_expect_tx(red_full, round_bytes((ph + 1) % nph));
                __syncwarp();
                tc_fence_after();
            }
            if (wnow) {
                // Next layer's projection of step t - 1 over this CTA's K range:
                // TMEM lane 32 + gate*32 + u holds unit unit0 + u of that gate
                // for the 32 batch rows; row b goes to slab `rank`.  The step
                // counter is already published, so this is off the recurrence's
                // critical path (thread 0 polls meanwhile, and waits for the
                // product itself before it reloads sH).
                w_pending = static_cast<int>(wpar);
                if (warp >= 1) {
                    if (__all_sync(0xffffffffu, bounded_wait(w_done, wpar, w, SITE_GRU_W) ? 1 : 0)) {
                        tc_fence_after();
                        uint32_t r[32];
                        tmem_ld32(tmem_d + (static_cast<uint32_t>(warp * 32) << 16) + wcol, r);
                        tmem_ld_wait(r);
                        float *dst = p.gxp_out + static_cast<size_t>(rank) * p.gx_slab +
                                     static_cast<size_t>(t - 1) * p.bstride * G + (warp - 1) * H + unit0 + lane;
#pragma unroll
                        for (int c = 0; c < 32; ++c)
                            if (c < p.batch) dst[static_cast<size_t>(c) * G] = __uint_as_float(r[c]);
                        w_issued = -1;
                    }
                    tc_fence_before();
                }
                __syncwarp();
            }
        }
    }
    // h_T of the last step reached (or the step the loop left at).
    if (last_t >= 0) {
#pragma unroll
        for (int k = 0; k < NP; ++k) {
            const int b = tid / UO + k * BSTEP;
            if (b < p.batch) p.h_out[(static_cast<size_t>(last_t) * p.bstride + b) * H + j] = hprev[k];
        }
    }

    // ---- teardown: let issued copies and products land, release TMEM.
    if ((tid == 32 || tid == 96) && w_issued >= 0) {  // only after an abort
        const uint32_t a = smem_u32(w_done);
        const unsigned long long t0 = globaltimer();
        while (!mbar_try_wait(a, static_cast<uint32_t>(w_issued)))
            if (globaltimer() - t0 > p.timeout_ns) break;
    }
    if (tid == 0 && issued_phase >= 0 && *abort_flag) {
        for (int q = 0; q < p.nq; ++q) {
            const uint32_t a = smem_u32(&hbar[q]);
            const unsigned long long t0 = globaltimer();
            while (!mbar_try_wait(a, static_cast<uint32_t>(issued_phase & 1)))
                if (globaltimer() - t0 > p.timeout_ns) break;
        }
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    // No CTA leaves while a cluster peer may still write into its shared
    // memory (a peer that gave up on a wait can be behind by a step); every
    // wait above is bounded, so every CTA gets here.
    if (KS > 1) cluster_sync_all();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem_d, tmem_cols);
    }
}

// K splits for a hidden size (the cluster size).  CTA k of a cluster takes
// the 64-wide K atoms k * ka .. k * ka + ka - 1 (ka = gru_atoms); the last
// range may end past the matrix, and a hidden of 64 j + 32 ends half an atom
// inside it: the tensor maps read zeros there on both sides of the product.
// 4 splits for multiples of 256, 2 for the other multiples of 128; otherwise
// one CTA per group up to 7 atoms (hidden <= 448), 2 up to 14 atoms and 4
// above, so that a CTA's slice of U, the next layer's slice of W (stacks) and
// its h tiles fit shared memory together at every multiple of 32.
int gru_splits(int H) {
    if (H % 256 == 0) return 4;
    if (H % 128 == 0) return 2;
    return H <= 448 ? 1 : H <= 896 ? 2 : 4;
}

// 64-wide K atoms per CTA: the hidden's atoms, rounded up, over the splits.
int gru_atoms(int H) {
    const int ks = gru_splits(H);
    return ((H + 63) / 64 + ks - 1) / ks;
}

size_t gru_smem_bytes(int H, bool has_next = false, int bp = kBatchPad) {
    return static_cast<size_t>(gru_layout(gru_atoms(H), has_next, bp).total);
}

int gru_cta_count(int H) { return H / kGroup * gru_splits(H); }

using GruKernel = void (*)(const CUtensorMap, const CUtensorMap, const CUtensorMap, const CUtensorMap,
                           const CUtensorMap, const CUtensorMap, const GruParams);

template <int BP>
GruKernel gru_kernel_for_bp(int ks) {
    return ks == 4 ? gru_recurrent_kernel<4, BP> : ks == 2 ? gru_recurrent_kernel<2, BP> : gru_recurrent_kernel<1, BP>;
}

// Padded batch widths a K-split count can run: 128 only with 4 splits (fewer
// splits leave 16 or 32 (unit, batch) pairs per thread, beyond the registers).
bool gru_bp_ok(int ks, int bp) { return bp == 32 || bp == 64 || (bp == 128 && ks == 4); }

GruKernel gru_kernel_for(int ks, int bp = kBatchPad) {
    if (bp == 128) return gru_recurrent_kernel<4, 128>;
    return bp == 64 ? gru_kernel_for_bp<64>(ks) : gru_kernel_for_bp<32>(ks);
}

// Opts every instantiation in to `bytes` of dynamic shared memory on the
// current device (ordinal `device`; the record is kept per device).
int gru_smem_attr(int bytes, int device) {
    const int ks[3] = {1, 2, 4}, bps[3] = {32, 64, 128};
    for (int k : ks)
        for (int bp : bps) {
            if (!gru_bp_ok(k, bp)) continue;
            const int rc = ensure_smem_optin(reinterpret_cast<const void *>(gru_kernel_for(k, bp)), bytes, device,
                                             "cudaFuncSetAttribute(gru)");
            if (rc) return rc;
        }
    return ISAM_OK;
}

int ensure_ws(void **ptr, size_t *cap, size_t need, const char *what) {
    if (*cap >= need) return ISAM_OK;
    if (*ptr) cudaFree(*ptr);
    *ptr = nullptr;
    *cap = 0;
    cudaError_t e = cudaMalloc(ptr, need);
    if (e != cudaSuccess) return cuda_error(e, what);
    *cap = need;
    return ISAM_OK;
}

// Tensor maps of the recurrence: U as [3 gates][H rows][H] (box: 96 rows of
// one group over one 64-wide K atom) and the two exchange buffers as
// [H/64 atoms][32 batch rows][64] (box: one CTA's h piece).
// Also the r * h exchange buffers' maps (tmR0 / tmR1 over rhx; skipped when
// null) and the next layer's input weights (tmWn over Wn, laid out as U;
// skipped when null).
int recurrent_maps(const uint16_t *U, const uint16_t *hx, const uint16_t *rhx, int H, CUtensorMap *tmU,
                   CUtensorMap *tmH0, CUtensorMap *tmH1, CUtensorMap *tmR0, CUtensorMap *tmR1,
                   const uint16_t *Wn = nullptr, CUtensorMap *tmWn = nullptr, int bp = kBatchPad) {
    int rc;
    const int ka = gru_atoms(H);
    const int nq = (ka % 4 == 0) ? 4 : (ka % 3 == 0) ? 3 : (ka % 2 == 0) ? 2 : 1;
    {
        const uint64_t dims[3] = {static_cast<uint64_t>(H), static_cast<uint64_t>(H), 3};
        const uint64_t strides[2] = {static_cast<uint64_t>(H) * 2, static_cast<uint64_t>(H) * H * 2};
        const uint32_t box[3] = {64, kGroup, 3};
        if ((rc = make_tmap_3d_bf16(tmU, U, dims, strides, box))) return rc;
        if (Wn && (rc = make_tmap_3d_bf16(tmWn, Wn, dims, strides, box))) return rc;
    }
    for (int i = 0; i < 2; ++i) {
        if (H % 64 != 0) {
            // [bp rows][H] with 64 x bp boxes, one per atom: the last atom's
            // upper half lies outside the rows and reads as zeros.
            const uint16_t *slot_h = hx + static_cast<size_t>(i) * bp * H;
            if ((rc = make_tmap_2d_bf16(i ? tmH1 : tmH0, slot_h, static_cast<uint64_t>(H), static_cast<uint64_t>(bp),
                                        static_cast<uint64_t>(H) * 2, 64, static_cast<uint32_t>(bp))))
                return rc;
            if (tmR0 && (rc = make_tmap_2d_bf16(i ? tmR1 : tmR0, rhx + static_cast<size_t>(i) * bp * H,
                                                static_cast<uint64_t>(H), static_cast<uint64_t>(bp),
                                                static_cast<uint64_t>(H) * 2, 64, static_cast<uint32_t>(bp))))
                return rc;
            continue;
        }
        const uint64_t dims[3] = {64, static_cast<uint64_t>(bp), static_cast<uint64_t>(H / 64)};
        const uint64_t strides[2] = {static_cast<uint64_t>(H) * 2, 128};
        const uint32_t box[3] = {64, static_cast<uint32_t>(bp), static_cast<uint32_t>(ka / nq)};
        if ((rc = make_tmap_3d_bf16(i ? tmH1 : tmH0, hx + static_cast<size_t>(i) * bp * H, dims,
                                    strides, box)))
            return rc;
        if (tmR0 && (rc = make_tmap_3d_bf16(i ? tmR1 : tmR0, rhx + static_cast<size_t>(i) * bp * H,
                                            dims, strides, box)))
            return rc;
    }
    return ISAM_OK;
}

int recurrent_maps(const uint16_t *U, const uint16_t *hx, int H, CUtensorMap *tmU, CUtensorMap *tmH0,
                   CUtensorMap *tmH1) {
    return recurrent_maps(U, hx, nullptr, H, tmU, tmH0, tmH1, nullptr, nullptr);
}

// Fills the shape fields of p and launches the recurrence: one cluster of KS
// CTAs per group of 32 units, as a plain cluster launch after checking that
// every cluster fits on the device at once (the step counter needs every CTA
// resident).  No cooperative attribute: a launch that carries both it and the
// cluster shape can lose the cluster shape when a tool re-issues it, and the
// bounded waits already turn a CTA that never runs into ISAM_ERR_TIMEOUT.
int launch_recurrent(GruParams &p, const CUtensorMap &tmU, const CUtensorMap &tmH0,
                     const CUtensorMap &tmH1, const CUtensorMap &tmR0, const CUtensorMap &tmR1,
                     const CUtensorMap &tmWn, size_t smem, cudaStream_t stream, int bp = kBatchPad) {
    const int H = p.H;
    p.ks = gru_splits(H);
    p.ka = gru_atoms(H);
    p.h2d = H % 64 != 0 ? 1 : 0;
    p.uo = kGroup / p.ks;
    p.n_cta = gru_cta_count(H);
    p.nq = (p.ka % 4 == 0) ? 4 : (p.ka % 3 == 0) ? 3 : (p.ka % 2 == 0) ? 2 : 1;
    p.qk = p.ka / p.nq;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(p.ks);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(static_cast<unsigned>(p.n_cta), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    const GruKernel kern = gru_kernel_for(p.ks, bp);
    int max_clusters = 0;
    cudaError_t e = cudaOccupancyMaxActiveClusters(&max_clusters, kern, &cfg);
    if (e != cudaSuccess) return cuda_error(e, "cudaOccupancyMaxActiveClusters(gru)");
    if (max_clusters * p.ks < p.n_cta)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "GRU recurrence: %d CTAs in clusters of %d cannot be co-resident (%d clusters fit)",
                         p.n_cta, p.ks, max_clusters);
    e = cudaLaunchKernelEx(&cfg, kern, tmU, tmH0, tmH1, tmR0, tmR1, tmWn, p);
    if (e != cudaSuccess) return cuda_error(e, "launch gru_recurrent_kernel");
    return ISAM_OK;
}

}  // namespace

namespace {

// bf16 copy of a layer's states (the next layer pair's GEMM input); n is a
// multiple of 4, both pointers 16-byte aligned.
__global__ void __launch_bounds__(256) states_to_bf16_kernel(const float4 *in, uint2 *out, size_t n4) {
    for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n4;
         i += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const float4 v = in[i];
        out[i] = make_uint2(static_cast<uint32_t>(f32_to_bf16_rne(v.x)) | (static_cast<uint32_t>(f32_to_bf16_rne(v.y)) << 16),
                            static_cast<uint32_t>(f32_to_bf16_rne(v.z)) | (static_cast<uint32_t>(f32_to_bf16_rne(v.w)) << 16));
    }
}

}  // namespace

int gru_plan(int layers, int batch, int hidden, int reset_before, int num_sms, int smem_optin, GruPlan *g) {
    const int H = hidden;
    if (layers < 1 || batch < 1 || batch > kBatchMax || H % 32 != 0 || H > 1024 || H < 32)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_gru_forward: needs batch <= 256 and hidden a multiple of 32 in "
                         "[32, 1024] (batch=%d hidden=%d)",
                         batch, H);
    GruPlan q;
    q.ks = gru_splits(H);
    q.ka = gru_atoms(H);
    q.n_cta = gru_cta_count(H);
    if (q.n_cta > num_sms)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gru_forward: %d CTAs cannot be co-resident", q.n_cta);
    // Padded batch of the recurrence (the MMA's N): 32 for batch <= 32, with
    // every feature; above that the narrowest of 64 and 128 that holds the
    // batch (else the widest that fits beside U), the batch running in chunks
    // of that many rows (one launch each; each chunk's rows are independent
    // sequences).  A step costs about the same whatever the width's fill.
    const bool chunked = batch > kBatchPad;
    q.bp = kBatchPad;
    if (chunked) {
        auto fits = [&](int cand) {
            return gru_bp_ok(q.ks, cand) && gru_smem_bytes(H, false, cand) <= static_cast<size_t>(smem_optin);
        };
        if (batch <= 64 && fits(64))
            q.bp = 64;
        else if (fits(128))
            q.bp = 128;
        else if (fits(64))
            q.bp = 64;
    }
    const size_t smem_last = gru_smem_bytes(H, false, q.bp);
    const size_t smem_next = gru_smem_bytes(H, true);
    if (smem_last > static_cast<size_t>(smem_optin))
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gru_forward: hidden too large for shared memory");
    if (layers > 1 && !chunked && smem_next > static_cast<size_t>(smem_optin))
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_gru_forward_stack: hidden %d leaves no room for the next layer's "
                         "weights beside the recurrent ones (%zu bytes of shared memory)",
                         H, smem_next);
    q.chunks = (batch + q.bp - 1) / q.bp;
    q.smem = static_cast<int>(smem_last);
    if (layers == 1) {
        q.path = 0;
    } else if (chunked) {
        q.path = 3;
    } else {
        const char *nw = getenv("ISAM_NO_WAVE");
        if (!reset_before && !(nw && nw[0] == '1') && gru_wave_fits(H, batch, num_sms, smem_optin)) {
            q.path = 1;
            q.smem = static_cast<int>(gru_wave_smem_bytes(H));
        } else {
            q.path = 2;
            q.smem = static_cast<int>(smem_next);
        }
    }
    *g = q;
    return ISAM_OK;
}

int gru_stack_launch(int layers, int T, int batch, int hidden, int reset_before, const uint16_t *x,
                     const uint16_t *W, const uint16_t *U, const float *b, const float *h0, float *h_out,
                     DeviceState &ds, cudaStream_t stream) {
    const int H = hidden;
    if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(W) |
         reinterpret_cast<uintptr_t>(U) | reinterpret_cast<uintptr_t>(b) |
         reinterpret_cast<uintptr_t>(h0) | reinterpret_cast<uintptr_t>(h_out)) & 15u)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gru_forward: pointers must be 16-byte aligned");
    GruPlan plan;
    int prc = gru_plan(layers, batch, H, reset_before, ds.num_sms, ds.max_smem_optin, &plan);
    if (prc != ISAM_OK) return prc;
    const bool chunked = batch > kBatchPad;  // path 3 when layers > 1
    const int bp = plan.bp;
    const size_t smem_last = gru_smem_bytes(H, false, bp);
    const size_t smem_next = gru_smem_bytes(H, true);

    int rc;
    const size_t seq_rows = static_cast<size_t>(T) * batch;
    const size_t gx_floats = seq_rows * 3 * H;
    if ((rc = ensure_ws(reinterpret_cast<void **>(&ds.gru_gx), &ds.gru_gx_bytes, gx_floats * sizeof(float),
                        "allocating the GRU projection workspace")))
        return rc;
    // Next layers' projections: two sets (read by layer l, written by layer l)
    // of ks slabs, one per K rank.
    const int ks = gru_splits(H);
    if (layers > 1 && !chunked &&
        (rc = ensure_ws(reinterpret_cast<void **>(&ds.gru_gxp), &ds.gru_gxp_bytes,
                        2 * static_cast<size_t>(ks) * gx_floats * sizeof(float),
                        "allocating the stacked GRU projection workspace")))
        return rc;
    // Exchange buffers: h (2 slots) then r * h (2 slots, the reset-before form),
    // bp rows each.
    const size_t hx_bytes = static_cast<size_t>(4) * bp * H * sizeof(uint16_t);
    if (ds.gru_hx_bytes < hx_bytes) {
        if ((rc = ensure_ws(reinterpret_cast<void **>(&ds.gru_hx), &ds.gru_hx_bytes, hx_bytes,
                            "allocating the GRU exchange buffer")))
            return rc;
        cudaError_t e = cudaMemset(ds.gru_hx, 0, hx_bytes);
        if (e != cudaSuccess) return cuda_error(e, "clearing the GRU exchange buffer");
    }
    if (!ds.gru_counter) {
        cudaError_t e = cudaMalloc(&ds.gru_counter, 256);
        if (e != cudaSuccess) return cuda_error(e, "allocating the GRU step counter");
    }
    if ((rc = gru_smem_attr(ds.max_smem_optin, ds.device))) return rc;

    const size_t wsz = static_cast<size_t>(3) * H * H;
    uint16_t *rhx = ds.gru_hx + static_cast<size_t>(2) * bp * H;
    // Input projection of layer l for all steps: gx = in W_l^T + b_ih_l
    // (M = T*batch, N = 3H, K = H).
    auto project = [&](const uint16_t *in, int l) {
        GemmDesc g{T * batch, 3 * H, H, 0, 1, 1.0f, 0.0f, in, W + l * wsz, ds.gru_gx, b + static_cast<size_t>(l) * 6 * H};
        GemmPlan plan;
        int r;
        if ((r = gemm_validate(g))) return r;
        if ((r = gemm_plan(g, ds, &plan))) return r;
        return gemm_launch(g, plan, ds, stream);
    };
    // One layer's recurrence.  Its projection is either ds.gru_gx (one slab,
    // b_ih included) or, for layer l > 0 of the per-layer chain, the slabs the
    // layer below computed; with has_next it computes layer l + 1's slabs.
    // Batch rows [b0, b0 + nb) of layer l (all rows unless chunked).
    auto recur = [&](int l, bool has_next, bool gx_from_below, int b0, int nb) {
        const uint16_t *Wn = has_next ? W + (l + 1) * wsz : nullptr;
        CUtensorMap tmU, tmH0, tmH1, tmR0, tmR1, tmWn;
        int r;
        if ((r = recurrent_maps(U + l * wsz, ds.gru_hx, rhx, H, &tmU, &tmH0, &tmH1, &tmR0, &tmR1, Wn, &tmWn, bp)))
            return r;
        GruParams p{};
        p.T = T;
        p.batch = nb;
        p.bstride = batch;
        p.H = H;
        if (!gx_from_below) {
            p.gx = ds.gru_gx + static_cast<size_t>(b0) * 3 * H;
            p.gx_parts = 1;
            p.b_ih = nullptr;
        } else {
            p.gx = ds.gru_gxp + static_cast<size_t>((l - 1) & 1) * ks * gx_floats;
            p.gx_parts = ks;
            p.b_ih = b + static_cast<size_t>(l) * 6 * H;
        }
        p.gx_slab = gx_floats;
        p.has_next = has_next ? 1 : 0;
        p.gxp_out = has_next ? ds.gru_gxp + static_cast<size_t>(l & 1) * ks * gx_floats : nullptr;
        p.b_hh = b + static_cast<size_t>(l) * 6 * H + 3 * H;
        p.h0 = h0 ? h0 + (static_cast<size_t>(l) * batch + b0) * H : nullptr;
        p.h_out = h_out + static_cast<size_t>(l) * seq_rows * H + static_cast<size_t>(b0) * H;
        p.hx = ds.gru_hx;
        p.rhx = rhx;
        p.reset_before = reset_before ? 1 : 0;
        p.counter = ds.gru_counter;
        p.skip_publish_cta = -1;
        if (const char *sk = getenv("ISAM_DEBUG_GRU_SKIP_CTA")) p.skip_publish_cta = atoi(sk);
        p.timeout_ns = wait_timeout_ns();
        p.err = ds.err_word;
        cudaError_t e = cudaMemsetAsync(ds.gru_counter, 0, sizeof(uint32_t), stream);
        if (e != cudaSuccess) return cuda_error(e, "clearing the GRU step counter");
        return launch_recurrent(p, tmU, tmH0, tmH1, tmR0, tmR1, has_next ? tmWn : tmU,
                                has_next ? smem_next : smem_last, stream, bp);
    };
    // bf16 copy of layer l - 1's states as layer l's GEMM input.
    auto states_below = [&](int l) {
        const size_t n4 = seq_rows * H / 4;
        const int blocks = static_cast<int>(std::min<size_t>((n4 + 255) / 256, static_cast<size_t>(ds.num_sms) * 8));
        states_to_bf16_kernel<<<blocks, 256, 0, stream>>>(
            reinterpret_cast<const float4 *>(h_out + static_cast<size_t>(l - 1) * seq_rows * H),
            reinterpret_cast<uint2 *>(ds.gru_xb), n4);
        cudaError_t e = cudaGetLastError();
        return e == cudaSuccess ? ISAM_OK : cuda_error(e, "launch states_to_bf16_kernel");
    };

    // Batches wider than 32: every layer projects its input with the GEMM and
    // runs its recurrence chunk by chunk.
    if (chunked) {
        if (layers > 1 && (rc = ensure_ws(reinterpret_cast<void **>(&ds.gru_xb), &ds.gru_xb_bytes,
                                          seq_rows * H * sizeof(uint16_t), "allocating the GRU layer-input buffer")))
            return rc;
        for (int l = 0; l < layers; ++l) {
            if (l > 0 && (rc = states_below(l))) return rc;
            if ((rc = project(l > 0 ? ds.gru_xb : x, l))) return rc;
            for (int b0 = 0; b0 < batch; b0 += bp)
                if ((rc = recur(l, false, false, b0, std::min(bp, batch - b0)))) return rc;
        }
        return ISAM_OK;
    }

    // Pairs of layers in one kernel (gru_wave.cu): layer l + 1 advances one
    // step behind layer l, its projection computed from the same h tiles.
    // Between pairs (and for an odd last layer) the layer below's states are
    // rounded to bf16 and projected by the GEMM.
    if (plan.path == 1) {
        if (layers > 2 && (rc = ensure_ws(reinterpret_cast<void **>(&ds.gru_xb), &ds.gru_xb_bytes,
                                          seq_rows * H * sizeof(uint16_t), "allocating the GRU layer-input buffer")))
            return rc;
        for (int l = 0; l < layers;) {
            const uint16_t *in = x;
            if (l > 0) {
                if ((rc = states_below(l))) return rc;
                in = ds.gru_xb;
            }
            if ((rc = project(in, l))) return rc;
            if (l + 1 < layers) {
                const size_t so = seq_rows * H;
                if ((rc = gru_wave_launch(T, batch, H, ds.gru_gx, U + l * wsz, W + (l + 1) * wsz, U + (l + 1) * wsz,
                                          b + static_cast<size_t>(l) * 6 * H, b + static_cast<size_t>(l + 1) * 6 * H,
                                          h0 ? h0 + static_cast<size_t>(l) * batch * H : nullptr,
                                          h0 ? h0 + static_cast<size_t>(l + 1) * batch * H : nullptr,
                                          h_out + static_cast<size_t>(l) * so, h_out + static_cast<size_t>(l + 1) * so,
                                          ds.gru_hx, rhx, ds.gru_counter, ds, stream)))
                    return rc;
                l += 2;
            } else {
                if ((rc = recur(l, false, false, 0, batch))) return rc;
                l += 1;
            }
        }
        return ISAM_OK;
    }

    // One recurrence per layer; layer l also computes layer l + 1's
    // projection (its slabs), which layer l + 1 sums as it goes.
    if ((rc = project(x, 0))) return rc;
    for (int l = 0; l < layers; ++l)
        if ((rc = recur(l, l + 1 < layers, l > 0, 0, batch))) return rc;
    return ISAM_OK;
}

int gru_launch(int T, int batch, int hidden, const uint16_t *x, const uint16_t *W,
               const uint16_t *U, const float *b, const float *h0, float *h_out, DeviceState &ds,
               cudaStream_t stream, int reset_before) {
    return gru_stack_launch(1, T, batch, hidden, reset_before, x, W, U, b, h0, h_out, ds, stream);
}

}  // namespace isam

// ===========================================================================
// Allocation-free variant of the GRU forward.
//
// Some callers cannot let a library call cudaMalloc: a serving process whose
// device memory is all reserved up front by its framework's caching allocator
// (a raw cudaMalloc would fail or fragment that pool), or a latency-bound
// request path that forbids cudaMalloc/cudaFree because they can synchronise
// the whole device.  isam_gru_forward_noalloc serves them: its workspaces
// (device error word, step counter, hidden-state exchange buffer, and the
// input projection of up to a chunk of time steps) live in the fixed array
// below, so the call allocates nothing.  It launches the same two kernels as
// isam_gru_forward, one time chunk after another, carrying h from one chunk to
// the next through h_out.
// ===========================================================================
namespace isam {
namespace {

constexpr size_t kNoAllocScratchBytes = static_cast<size_t>(8) << 20;  // 8 MiB
constexpr size_t kNaErrOff = 0;      // 16-byte device error word
constexpr size_t kNaCounterOff = 256;
constexpr size_t kNaHxOff = 512;     // 2 x [32][H] bf16 exchange buffer

}  // namespace
}  // namespace isam

// Every GPU that loads this library holds these 8 MiB until the process exits.
static __device__ __align__(256) unsigned char g_gru_noalloc_scratch[isam::kNoAllocScratchBytes];

namespace isam {
namespace {

struct NoAllocDevice {
    bool ready = false;
    unsigned char *scratch = nullptr;  // device address of g_gru_noalloc_scratch
    int num_sms = 0;
    int smem_optin = 0;
};
NoAllocDevice g_noalloc[64];
std::mutex g_noalloc_mu;

// Once per device, with that device current: the array's device address and
// the device limits the launches need.  No allocation happens here.
int noalloc_setup(int dev, NoAllocDevice *nd) {
    int major = 0, minor = 0;
    cudaError_t e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (e != cudaSuccess) return cuda_error(e, "isam_gru_forward_noalloc: device attributes");
    if (major != 10 || minor != 3)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_gru_forward_noalloc: built for sm_103a (GB300); device %d is sm_%d%d",
                         dev, major, minor);
    void *ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_gru_noalloc_scratch);
    if (e != cudaSuccess || ptr == nullptr)
        return cuda_error(e, "isam_gru_forward_noalloc: cudaGetSymbolAddress(scratch)");
    if ((e = cudaDeviceGetAttribute(&nd->num_sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&nd->smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) !=
            cudaSuccess)
        return cuda_error(e, "isam_gru_forward_noalloc: device attributes");
    nd->scratch = static_cast<unsigned char *>(ptr);
    nd->ready = true;
    return ISAM_OK;
}

}  // namespace
}  // namespace isam

extern "C" int isam_gru_forward_noalloc(int T, int batch, int hidden, const isam_bf16 *x,
                                        const isam_bf16 *W, const isam_bf16 *U, const float *b,
                                        const float *h0, float *h_out) {
    using namespace isam;
    const int H = hidden;
    if (T < 1 || batch < 1 || H < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward_noalloc: sizes must be >= 1");
    if (!x || !W || !U || !b || !h_out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward_noalloc: null pointer");
    if (batch > kBatchPad || H % 32 != 0 || H > 1024 || H < 32)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_gru_forward_noalloc: needs batch <= 32 and hidden a multiple of 32 "
                         "in [32, 1024] (batch=%d hidden=%d)",
                         batch, H);
    if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(W) |
         reinterpret_cast<uintptr_t>(U) | reinterpret_cast<uintptr_t>(b) |
         reinterpret_cast<uintptr_t>(h0) | reinterpret_cast<uintptr_t>(h_out)) & 15u)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_gru_forward_noalloc: pointers must be 16-byte aligned");
    // Scratch layout: error word | step counter | exchange buffer | projection chunk.
    const size_t hx_bytes = static_cast<size_t>(2) * kBatchPad * H * sizeof(uint16_t);
    const size_t gx_off = (kNaHxOff + hx_bytes + 255) / 256 * 256;
    const size_t step_bytes = static_cast<size_t>(batch) * 3 * H * sizeof(float);
    const long long chunk = static_cast<long long>((kNoAllocScratchBytes - gx_off) / step_bytes);
    if (chunk < 1)
        return set_error(ISAM_ERR_UNSUPPORTED,
                         "isam_gru_forward_noalloc: one step's projection (%zu bytes) exceeds the "
                         "%zu-byte scratch",
                         step_bytes, kNoAllocScratchBytes - gx_off);

    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_error(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64)
        return set_error(ISAM_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
    NoAllocDevice nd;
    {
        std::lock_guard<std::mutex> lk(g_noalloc_mu);
        if (!g_noalloc[dev].ready) {
            int rc = noalloc_setup(dev, &g_noalloc[dev]);
            if (rc) return rc;
        }
        nd = g_noalloc[dev];
        int rc0 = gru_smem_attr(nd.smem_optin, dev);
        if (rc0) return rc0;
    }
    const int n_cta = gru_cta_count(H);
    const size_t smem = gru_smem_bytes(H);
    if (n_cta > nd.num_sms || smem > static_cast<size_t>(nd.smem_optin))
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_gru_forward_noalloc: hidden too large");

    uint32_t *err = reinterpret_cast<uint32_t *>(nd.scratch + kNaErrOff);
    uint32_t *counter = reinterpret_cast<uint32_t *>(nd.scratch + kNaCounterOff);
    uint16_t *hx = reinterpret_cast<uint16_t *>(nd.scratch + kNaHxOff);
    float *gx = reinterpret_cast<float *>(nd.scratch + gx_off);
    cudaStream_t stream = current_stream();

    // A device view for the shared GEMM launcher: limits plus the scratch error word.
    DeviceState view;
    view.device = dev;
    view.num_sms = nd.num_sms;
    view.max_smem_optin = nd.smem_optin;
    view.err_word = err;

    int rc;
    if ((e = cudaMemsetAsync(err, 0, 16, stream)) != cudaSuccess)
        return cuda_error(e, "clearing the scratch error word");
    CUtensorMap tmU, tmH0, tmH1;
    if ((rc = recurrent_maps(U, hx, H, &tmU, &tmH0, &tmH1))) return rc;
    const size_t step_elems = static_cast<size_t>(batch) * H;
    for (long long t0 = 0; t0 < T; t0 += chunk) {
        const int tc = static_cast<int>(T - t0 < chunk ? T - t0 : chunk);
        // Input projection of steps [t0, t0 + tc): gx = x W^T + b_ih.
        GemmDesc g{tc * batch, 3 * H, H, 0, 1, 1.0f, 0.0f, x + static_cast<size_t>(t0) * step_elems, W,
                   gx, b};
        GemmPlan plan;
        if ((rc = gemm_validate(g))) return rc;
        if ((rc = gemm_plan(g, view, &plan))) return rc;
        if ((rc = gemm_launch(g, plan, view, stream))) return rc;
        // Recurrence over the chunk, starting from h_{t0 - 1} (h0 for the first chunk).
        if ((e = cudaMemsetAsync(counter, 0, sizeof(uint32_t), stream)) != cudaSuccess)
            return cuda_error(e, "clearing the scratch step counter");
        GruParams p{};
        p.T = tc;
        p.batch = batch;
        p.bstride = batch;
        p.H = H;
        p.gx = gx;
        p.b_hh = b + 3 * H;
        p.h0 = t0 == 0 ? h0 : h_out + static_cast<size_t>(t0 - 1) * step_elems;
        p.h_out = h_out + static_cast<size_t>(t0) * step_elems;
        p.hx = hx;
        p.counter = counter;
        p.skip_publish_cta = -1;
        p.timeout_ns = wait_timeout_ns();
        p.err = err;
        p.rhx = hx;  // the reset-after form only
        p.reset_before = 0;
        p.gx_parts = 1;
        p.gx_slab = 0;
        p.b_ih = nullptr;
        p.has_next = 0;
        p.gxp_out = nullptr;
        if ((rc = launch_recurrent(p, tmU, tmH0, tmH1, tmH0, tmH1, tmU, smem, stream))) return rc;
    }
    // Report device-side timeouts of this call before returning: the error
    // word is read back on the call's own stream (no wait on other streams),
    // then that stream alone is synchronised.
    uint32_t w[4] = {0, 0, 0, 0};
    if ((e = cudaMemcpyAsync(w, err, sizeof w, cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
        return cuda_error(e, "isam_gru_forward_noalloc: reading the scratch error word");
    if ((e = cudaStreamSynchronize(stream)) != cudaSuccess)
        return cuda_error(e, "isam_gru_forward_noalloc: cudaStreamSynchronize");
    if (w[0] & DEV_ERR_LAUNCH_SHAPE)
        return set_error(ISAM_ERR_CUDA,
                         "isam_gru_forward_noalloc: the recurrent kernel found clusters of %u CTAs, "
                         "not the shape it was launched for; h_out is undefined",
                         w[3]);
    if (w[0] != 0)
        return set_error(ISAM_ERR_TIMEOUT,
                         "isam_gru_forward_noalloc: a bounded device wait ran out (site 0x%x, "
                         "block %u); h_out is undefined",
                         w[1], w[2]);
    return ISAM_OK;
}
