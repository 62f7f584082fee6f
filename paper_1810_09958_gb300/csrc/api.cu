// api.cu -- the extern "C" boundary of libisam.so (declared in include/isam.h):
// argument checking, per-device state and workspaces, the stream, the device
// error word, and TMA descriptor encoding.
#include <cudaTypedefs.h>

#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "internal.h"

namespace isam {

namespace {

thread_local char t_err[512] = "no error";
std::mutex g_mu;
cudaStream_t g_stream = nullptr;
constexpr int kMaxDevices = 64;
DeviceState *g_dev[kMaxDevices] = {};

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

struct TmapEntry {
    uint64_t key[12];
    CUtensorMap map;
    bool used;
};
constexpr int kTmapCache = 128;
TmapEntry g_tmaps[kTmapCache];
int g_tmap_next = 0;
std::mutex g_tmap_mu;

int get_encoder() {
    if (g_encode) return ISAM_OK;
    void *fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                     cudaEnableDefault, &q);
    if (e != cudaSuccess || q != cudaDriverEntryPointSuccess || !fn)
        return set_error(ISAM_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable");
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    return ISAM_OK;
}

int encode(CUtensorMap *out, const uint64_t key[12], cuuint32_t rank, const void *base,
           const cuuint64_t *dims, const cuuint64_t *strides, const cuuint32_t *box,
           CUtensorMapDataType dtype = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16,
           CUtensorMapSwizzle swz = CU_TENSOR_MAP_SWIZZLE_128B) {
    {
        std::lock_guard<std::mutex> lk(g_tmap_mu);
        for (int i = 0; i < kTmapCache; ++i)
            if (g_tmaps[i].used && memcmp(g_tmaps[i].key, key, sizeof(uint64_t) * 12) == 0) {
                *out = g_tmaps[i].map;
                return ISAM_OK;
            }
    }
    int rc = get_encoder();
    if (rc) return rc;
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = g_encode(out, dtype, rank, const_cast<void *>(base), dims,
                          strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return set_error(ISAM_ERR_UNSUPPORTED, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
    std::lock_guard<std::mutex> lk(g_tmap_mu);
    TmapEntry &e = g_tmaps[g_tmap_next];
    g_tmap_next = (g_tmap_next + 1) % kTmapCache;
    memcpy(e.key, key, sizeof(uint64_t) * 12);
    e.map = *out;
    e.used = true;
    return ISAM_OK;
}

}  // namespace

int set_error(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(t_err, sizeof t_err, fmt, ap);
    va_end(ap);
    return code;
}

int cuda_error(cudaError_t e, const char *what) {
    return set_error(ISAM_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

cudaStream_t current_stream() {
    std::lock_guard<std::mutex> lk(g_mu);
    return g_stream;
}

unsigned long long wait_timeout_ns() {
    static unsigned long long v = [] {
        const char *s = getenv("ISAM_WAIT_TIMEOUT_MS");
        long ms = s ? strtol(s, nullptr, 10) : 2000;
        if (ms < 1) ms = 1;
        if (ms > 60000) ms = 60000;
        return static_cast<unsigned long long>(ms) * 1000000ull;
    }();
    return v;
}

namespace {
struct SmemOptin {
    int device;
    const void *fn;
    int bytes;
};
constexpr int kOptinCap = 256;
SmemOptin g_optin[kOptinCap];
int g_optin_n = 0;
std::mutex g_optin_mu;
}  // namespace

int ensure_smem_optin(const void *fn, int bytes, int device, const char *what) {
    std::lock_guard<std::mutex> lk(g_optin_mu);
    int slot = -1;
    for (int i = 0; i < g_optin_n; ++i)
        if (g_optin[i].device == device && g_optin[i].fn == fn) {
            if (g_optin[i].bytes >= bytes) return ISAM_OK;
            slot = i;
            break;
        }
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e != cudaSuccess) return cuda_error(e, what);
    if (slot < 0 && g_optin_n < kOptinCap) slot = g_optin_n++;
    if (slot >= 0) g_optin[slot] = SmemOptin{device, fn, bytes};
    return ISAM_OK;
}

DeviceState *device_state(int *status) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        *status = cuda_error(e, "cudaGetDevice");
        return nullptr;
    }
    if (dev < 0 || dev >= kMaxDevices) {
        *status = set_error(ISAM_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
        return nullptr;
    }
    std::lock_guard<std::mutex> lk(g_mu);
    if (g_dev[dev]) {
        *status = ISAM_OK;
        return g_dev[dev];
    }
    cudaDeviceProp prop;
    if ((e = cudaGetDeviceProperties(&prop, dev)) != cudaSuccess) {
        *status = cuda_error(e, "cudaGetDeviceProperties");
        return nullptr;
    }
    if (prop.major != 10 || prop.minor != 3) {
        *status = set_error(ISAM_ERR_UNSUPPORTED,
                            "libisam is built for sm_103a (GB300); device %d is sm_%d%d", dev,
                            prop.major, prop.minor);
        return nullptr;
    }
    auto *ds = new DeviceState();
    ds->device = dev;
    ds->num_sms = prop.multiProcessorCount;
    ds->max_smem_optin = static_cast<int>(prop.sharedMemPerBlockOptin);
    if ((e = cudaMalloc(&ds->err_word, 16)) != cudaSuccess ||
        (e = cudaMemset(ds->err_word, 0, 16)) != cudaSuccess) {
        *status = cuda_error(e, "allocating the device error word");
        delete ds;
        return nullptr;
    }
    g_dev[dev] = ds;
    *status = ISAM_OK;
    return ds;
}

int make_tmap_2d_bf16(CUtensorMap *out, const void *base, uint64_t inner, uint64_t outer,
                      uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer) {
    const uint64_t key[12] = {2, reinterpret_cast<uint64_t>(base), inner, outer, row_pitch_bytes,
                              box_inner, box_outer, 0, 0, 0, 0, 0};
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_pitch_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    return encode(out, key, 2, base, dims, strides, box);
}

int make_tmap_2d_u8(CUtensorMap *out, const void *base, uint64_t inner, uint64_t outer,
                    uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer) {
    const uint64_t key[12] = {0x8, reinterpret_cast<uint64_t>(base), inner, outer, row_pitch_bytes,
                              box_inner, box_outer, 0, 0, 0, 0, 0};
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_pitch_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    return encode(out, key, 2, base, dims, strides, box, CU_TENSOR_MAP_DATA_TYPE_UINT8);
}

int make_tmap_2d_f32(CUtensorMap *out, const void *base, uint64_t inner, uint64_t outer,
                     uint64_t row_pitch_bytes, uint32_t box_inner, uint32_t box_outer) {
    const uint64_t key[12] = {0xF32, reinterpret_cast<uint64_t>(base), inner, outer,
                              row_pitch_bytes, box_inner, box_outer, 0, 0, 0, 0, 0};
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_pitch_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    return encode(out, key, 2, base, dims, strides, box, CU_TENSOR_MAP_DATA_TYPE_FLOAT32);
}

int make_tmap_3d_bf16(CUtensorMap *out, const void *base, const uint64_t dims_in[3],
                      const uint64_t strides_bytes[2], const uint32_t box_in[3]) {
    const uint64_t key[12] = {3,           reinterpret_cast<uint64_t>(base),
                              dims_in[0],  dims_in[1],
                              dims_in[2],  strides_bytes[0],
                              strides_bytes[1], box_in[0],
                              box_in[1],   box_in[2],
                              0,           0};
    cuuint64_t dims[3] = {dims_in[0], dims_in[1], dims_in[2]};
    cuuint64_t strides[2] = {strides_bytes[0], strides_bytes[1]};
    cuuint32_t box[3] = {box_in[0], box_in[1], box_in[2]};
    return encode(out, key, 3, base, dims, strides, box);
}

}  // namespace isam

using namespace isam;

extern "C" {

int isam_version(void) { return 100; }

int isam_set_stream(void *stream) {
    std::lock_guard<std::mutex> lk(g_mu);
    g_stream = static_cast<cudaStream_t>(stream);
    return ISAM_OK;
}

const char *isam_last_error_string(void) { return t_err; }

int isam_sync(void) {
    int st;
    DeviceState *ds = device_state(&st);
    if (!ds) return st;
    cudaError_t e = cudaStreamSynchronize(current_stream());
    if (e != cudaSuccess) return cuda_error(e, "cudaStreamSynchronize");
    uint32_t w[4] = {0, 0, 0, 0};
    if ((e = cudaMemcpy(w, ds->err_word, sizeof w, cudaMemcpyDeviceToHost)) != cudaSuccess)
        return cuda_error(e, "reading the device error word");
    if (w[0] & DEV_ERR_LAUNCH_SHAPE) {
        cudaMemset(ds->err_word, 0, 16);
        return set_error(ISAM_ERR_CUDA,
                         "a cluster kernel found clusters of %u CTAs, not the shape it was launched "
                         "for (site 0x%x, block %u); it returned without computing",
                         w[3], w[1], w[2]);
    }
    if (w[0] != 0) {
        cudaMemset(ds->err_word, 0, 16);
        return set_error(ISAM_ERR_TIMEOUT,
                         "a bounded device wait ran out (site 0x%x, block %u); outputs of the "
                         "failed call are undefined",
                         w[1], w[2]);
    }
    return ISAM_OK;
}

int isam_shutdown(void) {
    std::lock_guard<std::mutex> lk(g_mu);
    int cur = -1;
    cudaGetDevice(&cur);
    for (int d = 0; d < kMaxDevices; ++d) {
        DeviceState *ds = g_dev[d];
        if (!ds) continue;
        cudaSetDevice(d);
        cudaDeviceSynchronize();
        cudaFree(ds->err_word);
        cudaFree(ds->gru_gx);
        cudaFree(ds->gru_hx);
        cudaFree(ds->gru_counter);
        cudaFree(ds->gru_gxp);
        cudaFree(ds->gru_xb);
        delete ds;
        g_dev[d] = nullptr;
    }
    if (cur >= 0) cudaSetDevice(cur);
    {
        std::lock_guard<std::mutex> lk2(g_tmap_mu);
        for (auto &e : g_tmaps) e.used = false;
    }
    return ISAM_OK;
}

int isam_gemm(int M, int N, int K, int transA, int transB, float alpha, const isam_bf16 *A,
              const isam_bf16 *B, float beta, float *C) {
    GemmDesc g{M, N, K, transA, transB, alpha, beta, A, B, C, nullptr};
    int rc = gemm_validate(g);
    if (rc) return rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    GemmPlan plan;
    if ((rc = gemm_plan(g, *ds, &plan))) return rc;
    return gemm_launch(g, plan, *ds, current_stream());
}

int isam_gemm_fp8(int M, int N, int K, float alpha, const uint8_t *A, const uint8_t *B, float beta, float *C) {
    GemmDesc g{M, N, K, 0, 1, alpha, beta, reinterpret_cast<const uint16_t *>(A),
               reinterpret_cast<const uint16_t *>(B), C, nullptr, 1};
    int rc = gemm_validate(g);
    if (rc) return rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    GemmPlan plan;
    if ((rc = gemm_plan(g, *ds, &plan))) return rc;
    return gemm_launch(g, plan, *ds, current_stream());
}

int isam_gemm_grouped(int count, const int *M, const int *N, const int *K, const int *transA,
                      const int *transB, const float *alpha, const isam_bf16 *const *A,
                      const isam_bf16 *const *B, const float *beta, float *const *C) {
    if (count < 1 || count > 64)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_grouped: count must be in [1, 64]");
    if (!M || !N || !K || !transA || !transB || !alpha || !A || !B || !beta || !C)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_grouped: null array");
    GemmDesc g[64];
    for (int i = 0; i < count; ++i) {
        g[i] = GemmDesc{M[i], N[i], K[i], transA[i], transB[i], alpha[i], beta[i], A[i], B[i], C[i], nullptr};
        int rc = gemm_validate(g[i]);
        if (rc) {
            char msg[640];  // prefix + the 512-byte error text
            snprintf(msg, sizeof msg, "isam_gemm_grouped: problem %d: %s", i, isam_last_error_string());
            return set_error(rc, "%s", msg);
        }
    }
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return gemm_grouped_launch(count, g, *ds, current_stream());
}

int isam_gemm_grouped_fp8(int count, const int *M, const int *N, const int *K, const float *alpha,
                          const uint8_t *const *A, const uint8_t *const *B, const float *beta, float *const *C) {
    if (count < 1 || count > 64)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_grouped_fp8: count must be in [1, 64]");
    if (!M || !N || !K || !alpha || !A || !B || !beta || !C)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_grouped_fp8: null array");
    GemmDesc g[64];
    for (int i = 0; i < count; ++i) {
        g[i] = GemmDesc{M[i], N[i], K[i], 0, 1, alpha[i], beta[i], reinterpret_cast<const uint16_t *>(A[i]),
                        reinterpret_cast<const uint16_t *>(B[i]), C[i], nullptr, 1};
        int rc = gemm_validate(g[i]);
        if (rc) {
            char msg[640];  // prefix + the 512-byte error text
            snprintf(msg, sizeof msg, "isam_gemm_grouped_fp8: problem %d: %s", i, isam_last_error_string());
            return set_error(rc, "%s", msg);
        }
    }
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return gemm_grouped_launch(count, g, *ds, current_stream());
}

int isam_depthwise_conv3x3(int N, int H, int W, int C, const isam_bf16 *x, const isam_bf16 *dw_w, isam_bf16 *y) {
    if (N < 1 || H < 1 || W < 1 || C < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_depthwise_conv3x3: sizes must be >= 1");
    if (!x || !dw_w || !y) return set_error(ISAM_ERR_INVALID_ARG, "isam_depthwise_conv3x3: null pointer");
    if (C % 8 != 0)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_depthwise_conv3x3: C (%d) must be a multiple of 8", C);
    if ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(dw_w) | reinterpret_cast<uintptr_t>(y)) & 15u)
        return set_error(ISAM_ERR_UNSUPPORTED, "isam_depthwise_conv3x3: pointers must be 16-byte aligned");
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return depthwise_launch(N, H, W, C, reinterpret_cast<const uint16_t *>(x), reinterpret_cast<const uint16_t *>(dw_w),
                            reinterpret_cast<uint16_t *>(y), *ds, current_stream());
}

int isam_gemm_mxfp8(int M, int N, int K, float alpha, const uint8_t *A, const uint8_t *SA, const uint8_t *B,
                    const uint8_t *SB, float beta, float *C) {
    MxDesc g{M, N, K, alpha, beta, A, SA, B, SB, C};
    int rc = gemm_mx_validate(g);
    if (rc) return rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return gemm_mx_launch(1, &g, *ds, current_stream());
}

int isam_gemm_grouped_mxfp8(int count, const int *M, const int *N, const int *K, const float *alpha,
                            const uint8_t *const *A, const uint8_t *const *SA, const uint8_t *const *B,
                            const uint8_t *const *SB, const float *beta, float *const *C) {
    if (count < 1 || count > 64)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_grouped_mxfp8: count must be in [1, 64]");
    if (!M || !N || !K || !alpha || !A || !SA || !B || !SB || !beta || !C)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_grouped_mxfp8: null array");
    MxDesc g[64];
    for (int i = 0; i < count; ++i) {
        g[i] = MxDesc{M[i], N[i], K[i], alpha[i], beta[i], A[i], SA[i], B[i], SB[i], C[i]};
        int rc = gemm_mx_validate(g[i]);
        if (rc) {
            char msg[640];  // prefix + the 512-byte error text
            snprintf(msg, sizeof msg, "isam_gemm_grouped_mxfp8: problem %d: %s", i, isam_last_error_string());
            return set_error(rc, "%s", msg);
        }
    }
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return gemm_mx_launch(count, g, *ds, current_stream());
}

// Reports the tile plan the cost model picks for a GEMM (for benchmarks and
// tests; nothing is launched).  out[0..5] = BN, split, stages, group_m, grid,
// shared-memory bytes.
int isam_gemm_plan_info(int M, int N, int K, int transA, int transB, float beta, int *out) {
    if (!out) return set_error(ISAM_ERR_INVALID_ARG, "null output");
    GemmDesc g{M, N, K, transA, transB, 1.0f, beta, reinterpret_cast<const uint16_t *>(16),
               reinterpret_cast<const uint16_t *>(16), reinterpret_cast<float *>(16), nullptr};
    int rc = gemm_validate(g);
    if (rc) return rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    GemmPlan plan;
    if ((rc = gemm_plan(g, *ds, &plan))) return rc;
    out[0] = plan.BN;
    out[1] = plan.split;
    out[2] = plan.stages;
    out[3] = plan.group_m;
    out[4] = plan.grid;
    out[5] = static_cast<int>(plan.smem);
    return ISAM_OK;
}

int isam_gemm_plan_info2(int M, int N, int K, int transA, int transB, float beta, int *out) {
    int rc = isam_gemm_plan_info(M, N, K, transA, transB, beta, out);
    if (rc) return rc;
    GemmDesc g{M, N, K, transA, transB, 1.0f, beta, reinterpret_cast<const uint16_t *>(16),
               reinterpret_cast<const uint16_t *>(16), reinterpret_cast<float *>(16), nullptr};
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    GemmPlan plan;
    if ((rc = gemm_plan(g, *ds, &plan))) return rc;
    out[6] = plan.pair ? 256 : 128;
    out[7] = plan.pair ? 2 : 1;
    return ISAM_OK;
}

int isam_gemm_plan_for(int M, int N, int K, int transA, int transB, float beta, int num_sms, int smem_optin,
                       const int *cluster_caps, int *out) {
    if (!out || !cluster_caps || num_sms < 1 || smem_optin < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_plan_for: null output or limits < 1");
    GemmDesc g{M, N, K, transA, transB, 1.0f, beta, reinterpret_cast<const uint16_t *>(16),
               reinterpret_cast<const uint16_t *>(16), reinterpret_cast<float *>(16), nullptr};
    int rc = gemm_validate(g);
    if (rc) return rc;
    DeviceState ds;  // no device: the limits come from the arguments
    ds.num_sms = num_sms;
    ds.max_smem_optin = smem_optin;
    for (int i = 0; i < 3; ++i) {
        if (cluster_caps[i] < 1)
            return set_error(ISAM_ERR_INVALID_ARG, "isam_gemm_plan_for: cluster capacities must be >= 1");
        ds.cluster_cap[i] = cluster_caps[i];
    }
    GemmPlan plan;
    if ((rc = gemm_plan(g, ds, &plan))) return rc;
    out[0] = plan.BN;
    out[1] = plan.split;
    out[2] = plan.stages;
    out[3] = plan.group_m;
    out[4] = plan.grid;
    out[5] = static_cast<int>(plan.smem);
    out[6] = plan.pair ? 256 : 128;
    out[7] = plan.pair ? 2 : 1;
    return ISAM_OK;
}

int isam_gru_forward(int T, int batch, int hidden, const isam_bf16 *x, const isam_bf16 *W,
                     const isam_bf16 *U, const float *b, const float *h0, float *h_out) {
    if (T < 1 || batch < 1 || hidden < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward: sizes must be >= 1");
    if (!x || !W || !U || !b || !h_out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward: null pointer");
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return gru_launch(T, batch, hidden, x, W, U, b, h0, h_out, *ds, current_stream());
}

int isam_gru_forward_reset_before(int T, int batch, int hidden, const isam_bf16 *x, const isam_bf16 *W,
                                  const isam_bf16 *U, const float *b, const float *h0, float *h_out) {
    if (T < 1 || batch < 1 || hidden < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward_reset_before: sizes must be >= 1");
    if (!x || !W || !U || !b || !h_out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward_reset_before: null pointer");
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return gru_launch(T, batch, hidden, x, W, U, b, h0, h_out, *ds, current_stream(), 1);
}

int isam_gru_forward_stack(int layers, int T, int batch, int hidden, int reset_before,
                          const isam_bf16 *x, const isam_bf16 *W, const isam_bf16 *U, const float *b,
                          const float *h0, float *h_out) {
    if (layers < 1 || T < 1 || batch < 1 || hidden < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward_stack: sizes must be >= 1");
    if (reset_before != 0 && reset_before != 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward_stack: reset_before must be 0 or 1");
    if (!x || !W || !U || !b || !h_out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_forward_stack: null pointer");
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return gru_stack_launch(layers, T, batch, hidden, reset_before, x, W, U, b, h0, h_out, *ds,
                            current_stream());
}

int isam_dwsep_conv(int N, int H, int W, int Cin, int Cout, const isam_bf16 *x,
                    const isam_bf16 *dw_w, const isam_bf16 *pw_w, float *out) {
    if (N < 1 || H < 1 || W < 1 || Cin < 1 || Cout < 1)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_dwsep_conv: sizes must be >= 1");
    if (!x || !dw_w || !pw_w || !out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_dwsep_conv: null pointer");
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return dwsep_launch(N, H, W, Cin, Cout, x, dw_w, pw_w, out, *ds, current_stream());
}

int isam_dwsep_plan_info(int W, int Cin, int Cout, int *out) {
    if (W < 1 || Cin < 1 || Cout < 1 || !out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_dwsep_plan_info: sizes must be >= 1, out non-null");
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return dwsep_plan(W, Cin, Cout, ds->max_smem_optin, out);
}

int isam_dwsep_plan_for(int W, int Cin, int Cout, int smem_optin, int *out) {
    if (W < 1 || Cin < 1 || Cout < 1 || smem_optin < 1 || !out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_dwsep_plan_for: sizes must be >= 1, out non-null");
    return dwsep_plan(W, Cin, Cout, smem_optin, out);
}

namespace {
int gru_plan_out(int layers, int batch, int hidden, int reset_before, int num_sms, int smem_optin, int *out) {
    GruPlan g;
    const int rc = gru_plan(layers, batch, hidden, reset_before, num_sms, smem_optin, &g);
    if (rc != ISAM_OK) return rc;
    out[0] = g.ks;
    out[1] = g.ka;
    out[2] = g.bp;
    out[3] = g.n_cta;
    out[4] = g.smem;
    out[5] = g.path;
    out[6] = g.chunks;
    return ISAM_OK;
}
}  // namespace

int isam_gru_plan_info(int layers, int batch, int hidden, int reset_before, int *out) {
    if (layers < 1 || batch < 1 || hidden < 1 || (reset_before != 0 && reset_before != 1) || !out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_plan_info: sizes must be >= 1, reset_before 0 or 1");
    int rc;
    DeviceState *ds = device_state(&rc);
    if (!ds) return rc;
    return gru_plan_out(layers, batch, hidden, reset_before, ds->num_sms, ds->max_smem_optin, out);
}

int isam_gru_plan_for(int layers, int batch, int hidden, int reset_before, int num_sms, int smem_optin, int *out) {
    if (layers < 1 || batch < 1 || hidden < 1 || (reset_before != 0 && reset_before != 1) || num_sms < 1 ||
        smem_optin < 1 || !out)
        return set_error(ISAM_ERR_INVALID_ARG, "isam_gru_plan_for: sizes must be >= 1, reset_before 0 or 1");
    return gru_plan_out(layers, batch, hidden, reset_before, num_sms, smem_optin, out);
}

}  // extern "C"
