// C ABI of the QSVD latent-attention path (declared in include/qsvd.h):
// argument validation, workspace carving and kernel launch order.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <unordered_map>
#include <vector>

#include "launch.h"
#include "prep_beta.h"
#include "qsvd.h"

namespace qsvd {

// Device error word: bit kErrRange / kErrTimeout set by kernels, read and
// cleared by qsvd_check.  It is a module-scope variable (no allocation).
__device__ int g_error_word;

namespace {

thread_local char g_msg[512];

int fail(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof(g_msg), fmt, ap);
    va_end(ap);
    return code;
}

int cuda_fail(cudaError_t e, const char *where) {
    return fail(QSVD_ECUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

constexpr int kMaxDevices = 64;
int g_arch_ok[kMaxDevices];          // 0 unknown, 1 sm_103, -1 other
int *g_err_ptr[kMaxDevices];

// Checks that the current device is an sm_103 part and returns the address
// of its error word.
int device_setup(int **err) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(QSVD_EUNSUPPORTED, "device index %d", dev);
    if (g_arch_ok[dev] == 0) {
        int major = 0, minor = 0;
        e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceGetAttribute");
        void *p = nullptr;
        if (major == 10 && minor == 3) {
            e = cudaGetSymbolAddress(&p, g_error_word);
            if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(error word)");
            g_err_ptr[dev] = static_cast<int *>(p);
            g_arch_ok[dev] = 1;
        } else {
            g_arch_ok[dev] = -1;
        }
    }
    if (g_arch_ok[dev] < 0)
        return fail(QSVD_EUNSUPPORTED, "this library is built for sm_103 (GB300) only");
    *err = g_err_ptr[dev];
    return QSVD_OK;
}

size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

int check_cache(const qsvd_cache *c) {
    if (!c || !c->codes || !c->scales) return fail(QSVD_EINVAL, "cache: null pointer");
    if (!aligned16(c->codes) || !aligned16(c->scales)) return fail(QSVD_EINVAL, "cache: pointers must be 16-byte aligned");
    if (c->bits != 8 && c->bits != 4) return fail(QSVD_EINVAL, "cache: bits must be 8 or 4");
    if (c->B <= 0 || c->Tmax <= 0 || c->r <= 0) return fail(QSVD_EINVAL, "cache: B, Tmax, r must be positive");
    if (c->r % 16) return fail(QSVD_EINVAL, "cache: r must be a multiple of 16");
    if (c->bits == 4 && c->r % 128) return fail(QSVD_EUNSUPPORTED, "cache: int4 needs r %% 128 == 0");
    return QSVD_OK;
}

CacheView view(const qsvd_cache *c) {
    return CacheView{c->codes, c->scales, c->bits, c->B, c->Tmax, c->r, nullptr, c->B};
}

// Profiling state of the calling thread (see qsvd_profile_events).
thread_local cudaEvent_t *t_prof_events = nullptr;
thread_local int t_prof_capacity = 0;
thread_local std::vector<const char *> t_prof_labels;

}  // namespace

int *error_word_for_current_device() {
    int *err = nullptr;
    return device_setup(&err) == QSVD_OK ? err : nullptr;
}

int setup_current_device(int **err) { return device_setup(err); }

int validate_cache(const qsvd_cache *c) { return check_cache(c); }

int set_last_error(int code, const char *msg) { return fail(code, "%s", msg); }

cudaError_t ensure_smem_ptr(const void *kernel, size_t bytes) {
    static std::mutex mu;
    static std::unordered_map<const void *, int> done;     // kernel -> device bitmask
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(mu);
    int &mask = done[kernel];
    if (dev < 31 && (mask >> dev) & 1) return cudaSuccess;
    // the opt-in limit covers static + dynamic shared memory of the kernel
    int optin = 0;
    e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
    if (e != cudaSuccess) return e;
    cudaFuncAttributes fa{};
    e = cudaFuncGetAttributes(&fa, kernel);
    if (e != cudaSuccess) return e;
    const int max_dyn = optin - int(fa.sharedSizeBytes);
    if (int64_t(bytes) > max_dyn) return cudaErrorInvalidValue;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, max_dyn);
    if (e == cudaSuccess && dev < 31) mask |= 1 << dev;
    return e;
}

namespace {
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
EncodeTiledFn encode_tiled() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *q = nullptr;
        cudaDriverEntryPointQueryResult res;
        if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &q, cudaEnableDefault, &res) == cudaSuccess &&
            res == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(q);
    });
    return fn;
}
}  // namespace

bool tensor_maps_available() { return encode_tiled() != nullptr; }

bool encode_map_2d(CUtensorMap *map, CUtensorMapDataType type, const void *base, uint64_t inner, uint64_t outer,
                   uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swizzle) {
    EncodeTiledFn fn = encode_tiled();
    if (!fn) return false;
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {row_bytes};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return fn(map, type, 2, const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

void prof_mark(cudaStream_t s, const char *label) {
    if (!t_prof_events || int(t_prof_labels.size()) >= t_prof_capacity) return;
    // inside a stream capture the record becomes an event-record node of the graph
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    (void)cudaStreamIsCapturing(s, &cs);
    const unsigned flags = cs == cudaStreamCaptureStatusActive ? cudaEventRecordExternal : cudaEventRecordDefault;
    if (cudaEventRecordWithFlags(t_prof_events[t_prof_labels.size()], s, flags) == cudaSuccess)
        t_prof_labels.push_back(label);
    else
        (void)cudaGetLastError();     // a bad event handle must not surface as a launch error
}

}  // namespace qsvd

using namespace qsvd;

extern "C" {

const char *qsvd_last_error(void) { return g_msg; }

int qsvd_version(void) { return 100; }

int qsvd_set_project_epilogue(int32_t mode) {
    if (mode < 0 || mode > 2) return fail(QSVD_EINVAL, "set_project_epilogue: mode must be 0, 1 or 2");
    const int prev = project_epilogue();
    set_project_epilogue(mode);
    return prev;
}

int qsvd_set_decode_attn_path(int32_t path) {
    if (path < 0 || path > 3) return fail(QSVD_EINVAL, "set_decode_attn_path: path must be 0, 1, 2 or 3");
    const int prev = attn_path();
    set_attn_path(path);
    return prev;
}

int qsvd_profile_events(void **events, int32_t capacity) {
    t_prof_labels.clear();
    if (!events || capacity <= 0) {
        t_prof_events = nullptr;
        t_prof_capacity = 0;
        return QSVD_OK;
    }
    t_prof_events = reinterpret_cast<cudaEvent_t *>(events);
    t_prof_capacity = capacity;
    t_prof_labels.reserve(size_t(capacity));
    return QSVD_OK;
}

int32_t qsvd_profile_count(void) { return int32_t(t_prof_labels.size()); }

const char *qsvd_profile_label(int32_t i) {
    return (i >= 0 && i < int32_t(t_prof_labels.size())) ? t_prof_labels[size_t(i)] : "";
}

int qsvd_check(cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    cudaError_t e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    int word = 0;
    e = cudaMemcpyFromSymbol(&word, g_error_word, sizeof(int));
    if (e != cudaSuccess) return cuda_fail(e, "read error word");
    if (word) {
        const int zero = 0;
        e = cudaMemcpyToSymbol(g_error_word, &zero, sizeof(int));
        if (e != cudaSuccess) return cuda_fail(e, "clear error word");
    }
    if (word & kErrTimeout) return fail(QSVD_ETIMEOUT, "a bounded device wait expired");
    if (word & kErrRange) return fail(QSVD_ERANGE, "a cache position, sequence index or length was out of range, or a value was saturated at the fp16 range");
    g_msg[0] = 0;
    return QSVD_OK;
}

int qsvd_selftest_wait_timeout(int32_t timeout_ms, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (timeout_ms < 1 || timeout_ms > 1000) return fail(QSVD_EINVAL, "selftest_wait_timeout: timeout_ms outside 1..1000");
    prof_mark(stream, "begin");
    cudaError_t e = launch_selftest_wait(static_cast<unsigned long long>(timeout_ms) * 1000000ull, err, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "selftest launch");
}

int qsvd_quantize_weight(const float *W_d, int32_t d, int32_t r, float clip, int8_t *codes,
                         uint16_t *codes_bf16, float *scale, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!W_d || !codes || !scale) return fail(QSVD_EINVAL, "quantize_weight: null pointer");
    if (d <= 0 || r <= 0) return fail(QSVD_EINVAL, "quantize_weight: d and r must be positive");
    if (!(clip > 0.0f && clip <= 1.0f)) return fail(QSVD_EINVAL, "quantize_weight: clip must lie in (0, 1]");
    prof_mark(stream, "begin");
    cudaError_t e = launch_quantize_weight(W_d, d, r, clip, codes, codes_bf16, scale, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "quantize_weight launch");
}

int qsvd_quantize_weight_ex(const float *W_d, int32_t d, int32_t r, float clip, int32_t bits, int32_t rot,
                            int8_t *codes, uint16_t *codes_bf16, uint8_t *codes_e4m3, float *scale,
                            cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!W_d || !codes || !scale) return fail(QSVD_EINVAL, "quantize_weight_ex: null pointer");
    if (d <= 0 || r <= 0) return fail(QSVD_EINVAL, "quantize_weight_ex: d and r must be positive");
    if (!(clip > 0.0f && clip <= 1.0f)) return fail(QSVD_EINVAL, "quantize_weight_ex: clip must lie in (0, 1]");
    if (bits != 8 && bits != 4) return fail(QSVD_EINVAL, "quantize_weight_ex: bits must be 8 or 4");
    if (codes_e4m3 && bits != 4) return fail(QSVD_EINVAL, "quantize_weight_ex: an e4m3 image needs bits 4");
    if (rot && (rot < 2 || (rot & (rot - 1)) || d % rot))
        return fail(QSVD_EINVAL, "quantize_weight_ex: rot must be 0 or a power of two >= 2 dividing d");
    if (rot && d > 6144) return fail(QSVD_EUNSUPPORTED, "quantize_weight_ex: rotation needs d <= 6144");
    prof_mark(stream, "begin");
    cudaError_t e = launch_quantize_weight(W_d, d, r, clip, codes, codes_bf16, scale, stream, rot, bits == 8 ? 127 : 7,
                                           codes_e4m3);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "quantize_weight_ex launch");
}

int qsvd_quantize_weight_rotated(const float *W_d, int32_t d, int32_t r, float clip, int32_t rot, int8_t *codes,
                                 uint16_t *codes_bf16, float *scale, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!W_d || !codes || !scale) return fail(QSVD_EINVAL, "quantize_weight_rotated: null pointer");
    if (d <= 0 || r <= 0) return fail(QSVD_EINVAL, "quantize_weight_rotated: d and r must be positive");
    if (!(clip > 0.0f && clip <= 1.0f)) return fail(QSVD_EINVAL, "quantize_weight_rotated: clip must lie in (0, 1]");
    if (rot < 2 || (rot & (rot - 1)) || d % rot) return fail(QSVD_EINVAL, "quantize_weight_rotated: rot must be a power of two >= 2 dividing d");
    if (d > 6144) return fail(QSVD_EUNSUPPORTED, "quantize_weight_rotated: d > 6144");
    prof_mark(stream, "begin");
    cudaError_t e = launch_quantize_weight(W_d, d, r, clip, codes, codes_bf16, scale, stream, rot);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "quantize_weight_rotated launch");
}

size_t qsvd_project_workspace_bytes(int64_t T, int32_t d, int32_t r) {
    if (T < 0 || d <= 0 || r <= 0) return 0;
    return 256 +                                // completion counter (zero at rest)
           align256(size_t(T) * d) +            // int8 codes of X
           align256(size_t(T) * 4) +            // s_x
           align256(size_t(T) * r * 4) +        // dequantized latent c_hat
           align256(size_t(T) * d * 2) +        // bf16 image of the X codes (tensor-core operand)
           (T * r <= kSplitMaxElems ? align256(size_t(kMaxSplitK) * T * r * 4) : 0);   // split-K partials
}

int qsvd_latent_project(const qsvd_down_weight *W, const uint16_t *X, int64_t T, float act_clip,
                        int32_t lat_bits, float lat_clip, void *lat_codes, void *lat_scales,
                        const qsvd_cache *dst, const int32_t *dst_seq, const int32_t *dst_pos,
                        int8_t *xq_out, float *xs_out, int32_t *acc_out, void *workspace,
                        size_t workspace_bytes, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!W || !W->codes || !W->scale) return fail(QSVD_EINVAL, "latent_project: null weight pointer");
    if (T < 0) return fail(QSVD_EINVAL, "latent_project: T < 0");
    const int d = W->d, r = W->r;
    if (d <= 0 || r <= 0 || d % 64 || r % 16) return fail(QSVD_EINVAL, "latent_project: need d %% 64 == 0 and r %% 16 == 0");
    if (r > 4096) return fail(QSVD_EUNSUPPORTED, "latent_project: r > 4096");
    const int rot = W->rot;
    if (rot && (rot < 2 || (rot & (rot - 1)) || d % rot))
        return fail(QSVD_EINVAL, "latent_project: W->rot must be 0 or a power of two >= 2 dividing d");
    if (lat_bits != 8 && lat_bits != 4) return fail(QSVD_EINVAL, "latent_project: lat_bits must be 8 or 4");
    if (lat_bits == 4 && r % 128) return fail(QSVD_EUNSUPPORTED, "latent_project: int4 needs r %% 128 == 0");
    const int wb = W->w_bits ? W->w_bits : 8, xb = W->x_bits ? W->x_bits : 8;
    if ((wb != 8 && wb != 4) || (xb != 8 && xb != 4)) return fail(QSVD_EINVAL, "latent_project: W->w_bits and W->x_bits must be 8 or 4");
    const int act_qmax = xb == 8 ? 127 : 7;
    if (!(act_clip > 0.0f && act_clip <= 1.0f) || !(lat_clip > 0.0f && lat_clip <= 1.0f))
        return fail(QSVD_EINVAL, "latent_project: clip ratios must lie in (0, 1]");
    const bool tok = lat_codes != nullptr || lat_scales != nullptr;
    if (tok && (!lat_codes || !lat_scales)) return fail(QSVD_EINVAL, "latent_project: give both lat_codes and lat_scales");
    if (!tok && !dst) return fail(QSVD_EINVAL, "latent_project: no destination for the latent");
    if (dst) {
        if ((st = check_cache(dst))) return st;
        if (dst->bits != lat_bits || dst->r != r) return fail(QSVD_EINVAL, "latent_project: cache format differs");
    }
    if (T == 0) return QSVD_OK;
    if (dst && (!dst_seq || !dst_pos)) return fail(QSVD_EINVAL, "latent_project: dst_seq/dst_pos required with dst");
    if (!X) return fail(QSVD_EINVAL, "latent_project: X is null");
    const void *ptrs[] = {X, W->codes, W->scale, lat_codes, lat_scales, xq_out, xs_out, acc_out, workspace};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return fail(QSVD_EINVAL, "latent_project: pointers must be 16-byte aligned");
    const size_t need = qsvd_project_workspace_bytes(T, d, r);
    if (!workspace || workspace_bytes < need)
        return fail(QSVD_ENOSPC, "latent_project: workspace needs %zu bytes", need);

    char *wsp = static_cast<char *>(workspace);
    int *counter = reinterpret_cast<int *>(wsp);
    wsp += 256;
    int8_t *xq = xq_out ? xq_out : reinterpret_cast<int8_t *>(wsp);
    wsp += align256(size_t(T) * d);
    float *xs = xs_out ? xs_out : reinterpret_cast<float *>(wsp);
    wsp += align256(size_t(T) * 4);
    float *c_hat = reinterpret_cast<float *>(wsp);
    wsp += align256(size_t(T) * r * 4);
    uint16_t *xq_bf16 = reinterpret_cast<uint16_t *>(wsp);
    CacheView dv{};
    if (dst) dv = view(dst);

    prof_mark(stream, "begin");
    cudaError_t e;
    if (T <= kPsMaxSplitTok && d <= 6144 && d % 256 == 0) {
        // one token: the quantizer fused into the projection, then the requantization
        // kernel; with H1 the rotation runs once per row in xquant instead (in every
        // CTA of the projection it measured slower)
        if (T < kPsSplitTok && !rot) {
            e = launch_proj_small(X, int(T), d, act_clip, W->codes, W->scale, r, lat_bits, lat_clip, c_hat, counter,
                                  xq_out, xs_out, acc_out, lat_codes, lat_scales, dst ? &dv : nullptr, dst_seq,
                                  dst_pos, err, stream, nullptr, nullptr, false, act_qmax);
            if (e == cudaSuccess)
                e = launch_requant(c_hat, T, r, lat_bits, lat_clip, lat_codes, lat_scales, dst ? &dv : nullptr, dst_seq,
                                   dst_pos, err, stream);
            return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "projection launch");
        }
        // each row quantized once, the dot products on the tensor cores, the rows requantized in parallel
        e = launch_xquant(X, T, d, act_clip, xq, nullptr, xs, stream, rot, act_qmax);
        if (e == cudaSuccess)
            e = launch_proj_small(X, int(T), d, act_clip, W->codes, W->scale, r, lat_bits, lat_clip, c_hat, counter,
                                  nullptr, nullptr, acc_out, lat_codes, lat_scales, dst ? &dv : nullptr, dst_seq,
                                  dst_pos, err, stream, xq, xs, false, act_qmax);
        if (e == cudaSuccess)
            e = launch_requant(c_hat, T, r, lat_bits, lat_clip, lat_codes, lat_scales, dst ? &dv : nullptr, dst_seq,
                               dst_pos, err, stream);
        return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "projection launch");
    }
    if (wb == 4 && xb == 4 && W->codes_e4m3 && gemm_f8_supported(d, r)) {
        // W4A4 on the fp8 tensor-core path: e4m3 images of the int4 codes, exact products and sums
        if (!aligned16(W->codes_e4m3)) return fail(QSVD_EINVAL, "latent_project: codes_e4m3 must be 16-byte aligned");
        uint8_t *xq_f8 = reinterpret_cast<uint8_t *>(xq_bf16);            // the image slot holds T * d bytes
        e = launch_xquant(X, T, d, act_clip, xq_out, nullptr, xs, stream, rot, act_qmax, xq_f8);
        if (e != cudaSuccess) return cuda_fail(e, "xquant launch");
        if (gemm_tc_fused_supported(T, r, lat_bits)) {
            e = launch_gemm_f8(xq_f8, T, d, W->codes_e4m3, W->scale, xs, r, lat_bits, lat_clip, lat_codes, lat_scales,
                               dst ? &dv : nullptr, dst_seq, dst_pos, nullptr, acc_out, err, stream);
            return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "fp8 tensor-core projection launch");
        }
        e = launch_gemm_f8(xq_f8, T, d, W->codes_e4m3, W->scale, xs, r, 0, lat_clip, nullptr, nullptr, nullptr,
                           nullptr, nullptr, c_hat, acc_out, err, stream);
        if (e != cudaSuccess) return cuda_fail(e, "fp8 tensor-core projection launch");
    } else if (W->codes_bf16 && gemm_tc_supported(d, r)) {
        if (!aligned16(W->codes_bf16)) return fail(QSVD_EINVAL, "latent_project: codes_bf16 must be 16-byte aligned");
        e = launch_xquant(X, T, d, act_clip, xq_out, xq_bf16, xs, stream, rot, act_qmax);
        if (e != cudaSuccess) return cuda_fail(e, "xquant launch");
        if (gemm_tc_fused_supported(T, r, lat_bits)) {
            // a2, a3 and a4 in one kernel: the latent never leaves the registers
            e = launch_gemm_tc_fused(xq_bf16, T, d, W->codes_bf16, W->scale, xs, r, lat_bits, lat_clip, lat_codes,
                                     lat_scales, dst ? &dv : nullptr, dst_seq, dst_pos, nullptr, acc_out, err,
                                     stream);
            return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "tensor-core projection launch");
        }
        const int splits = gemm_tc_splits(T, d, r);
        if (splits > 1) {
            // few tiles: split K over more CTAs; the splits' sums are added, dequantized and
            // requantized row by row
            int32_t *part = reinterpret_cast<int32_t *>(reinterpret_cast<char *>(xq_bf16) + align256(size_t(T) * d * 2));
            e = launch_gemm_tc(xq_bf16, T, d, W->codes_bf16, W->scale, xs, r, nullptr, nullptr, err, stream, splits,
                               part);
            if (e == cudaSuccess)
                e = launch_split_requant(part, splits, T, r, xs, W->scale, acc_out, lat_bits, lat_clip, lat_codes,
                                         lat_scales, dst ? &dv : nullptr, dst_seq, dst_pos, err, stream);
            return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "split-K projection launch");
        }
        e = launch_gemm_tc(xq_bf16, T, d, W->codes_bf16, W->scale, xs, r, c_hat, acc_out, err, stream);
        if (e != cudaSuccess) return cuda_fail(e, "tensor-core projection launch");
    } else {
        e = launch_xquant(X, T, d, act_clip, xq, nullptr, xs, stream, rot, act_qmax);
        if (e != cudaSuccess) return cuda_fail(e, "xquant launch");
        e = launch_proj_dp4a(xq, T, d, W->codes, W->scale, xs, r, c_hat, acc_out, stream);
        if (e != cudaSuccess) return cuda_fail(e, "projection launch");
    }
    e = launch_requant(c_hat, T, r, lat_bits, lat_clip, lat_codes, lat_scales, dst ? &dv : nullptr, dst_seq,
                       dst_pos, err, stream);
    if (e != cudaSuccess) return cuda_fail(e, "requant launch");
    return QSVD_OK;
}

int qsvd_cache_append(const qsvd_cache *cache, const int32_t *seq, const int32_t *pos, int64_t n,
                      const void *lat_codes, const void *lat_scales, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if ((st = check_cache(cache))) return st;
    if (n < 0) return fail(QSVD_EINVAL, "cache_append: n < 0");
    if (n == 0) return QSVD_OK;
    if (!seq || !pos || !lat_codes || !lat_scales) return fail(QSVD_EINVAL, "cache_append: null pointer");
    if (!aligned16(lat_codes)) return fail(QSVD_EINVAL, "cache_append: lat_codes must be 16-byte aligned");
    prof_mark(stream, "begin");
    cudaError_t e = launch_append(view(cache), seq, pos, n, lat_codes, lat_scales, err, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "cache_append launch");
}

size_t qsvd_decode_workspace_bytes(int32_t B, int32_t max_seq_len, int32_t r, int32_t H, int32_t dh) {
    if (B <= 0 || max_seq_len <= 0 || r <= 0 || H <= 0 || dh <= 0) return 0;
    return decode_workspace_bytes(B, max_seq_len, r, H, dh);
}

int qsvd_latent_decode_attn(const qsvd_cache *cache, const int32_t *seq_len, int32_t max_seq_len,
                            const uint16_t *U_q, const uint16_t *U_k, const uint16_t *U_v, int32_t H,
                            int32_t dh, float softmax_scale, float *O, void *workspace, size_t workspace_bytes,
                            cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if ((st = check_cache(cache))) return st;
    if (!seq_len || !U_q || !U_k || !U_v || !O) return fail(QSVD_EINVAL, "decode_attn: null pointer");
    if (dh != 64 && dh != 128) return fail(QSVD_EUNSUPPORTED, "decode_attn: dh must be 64 or 128");
    if (H <= 0) return fail(QSVD_EINVAL, "decode_attn: H must be positive");
    if (cache->r > 3072 || cache->r % 32) return fail(QSVD_EUNSUPPORTED, "decode_attn: need r %% 32 == 0 and r <= 3072");
    if ((H * dh) % 256 || H * dh > 6144) return fail(QSVD_EUNSUPPORTED, "decode_attn: need H*dh %% 256 == 0 and H*dh <= 6144");
    if (max_seq_len < 1 || max_seq_len > cache->Tmax) return fail(QSVD_EINVAL, "decode_attn: max_seq_len outside [1, Tmax]");
    const void *ptrs[] = {U_q, U_k, U_v, O, workspace};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return fail(QSVD_EINVAL, "decode_attn: pointers must be 16-byte aligned");
    const size_t need = qsvd_decode_workspace_bytes(cache->B, max_seq_len, cache->r, H, dh);
    if (!workspace || workspace_bytes < need)
        return fail(QSVD_ENOSPC, "decode_attn: workspace needs %zu bytes", need);
    DecodeArgs a{view(cache), seq_len, max_seq_len, UpW{U_q, nullptr, 16}, UpW{U_k, nullptr, 16},
                 UpW{U_v, nullptr, 16}, H, dh, softmax_scale, O};
    prof_mark(stream, "begin");
    cudaError_t e = launch_decode(a, workspace, workspace_bytes, err, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "decode_attn launch");
}

int qsvd_quantize_up(const uint16_t *U, int32_t r, int32_t d, int32_t bits, float clip, void *codes, float *scale,
                     cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!U || !codes || !scale) return fail(QSVD_EINVAL, "quantize_up: null pointer");
    if (r <= 0 || d <= 0 || d % 32) return fail(QSVD_EINVAL, "quantize_up: need r > 0 and d %% 32 == 0");
    if (bits != 8 && bits != 4) return fail(QSVD_EINVAL, "quantize_up: bits must be 8 or 4");
    if (!(clip > 0.0f && clip <= 1.0f)) return fail(QSVD_EINVAL, "quantize_up: clip must lie in (0, 1]");
    prof_mark(stream, "begin");
    const cudaError_t e = launch_quantize_up(U, r, d, bits, clip, codes, scale, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "quantize_up launch");
}

int qsvd_latent_decode_attn_qu(const qsvd_cache *cache, const int32_t *seq_len, int32_t max_seq_len,
                               const qsvd_up_weight *U_q, const qsvd_up_weight *U_k, const qsvd_up_weight *U_v,
                               int32_t H, int32_t dh, float softmax_scale, float *O, void *workspace,
                               size_t workspace_bytes, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if ((st = check_cache(cache))) return st;
    if (!seq_len || !U_q || !U_k || !U_v || !O) return fail(QSVD_EINVAL, "decode_attn_qu: null pointer");
    if (dh != 64 && dh != 128) return fail(QSVD_EUNSUPPORTED, "decode_attn_qu: dh must be 64 or 128");
    if (H <= 0) return fail(QSVD_EINVAL, "decode_attn_qu: H must be positive");
    if (cache->r > 3072 || cache->r % 32) return fail(QSVD_EUNSUPPORTED, "decode_attn_qu: need r %% 32 == 0 and r <= 3072");
    if ((H * dh) % 256 || H * dh > 6144) return fail(QSVD_EUNSUPPORTED, "decode_attn_qu: need H*dh %% 256 == 0 and H*dh <= 6144");
    if (max_seq_len < 1 || max_seq_len > cache->Tmax) return fail(QSVD_EINVAL, "decode_attn_qu: max_seq_len outside [1, Tmax]");
    const qsvd_up_weight *Us[3] = {U_q, U_k, U_v};
    for (const qsvd_up_weight *u : Us) {
        if (!u->codes || !u->scale) return fail(QSVD_EINVAL, "decode_attn_qu: null weight pointer");
        if (u->bits != 8 && u->bits != 4) return fail(QSVD_EINVAL, "decode_attn_qu: weight bits must be 8 or 4");
        if (u->r != cache->r || u->d != H * dh) return fail(QSVD_EINVAL, "decode_attn_qu: weight shape differs from [r, H*dh]");
        if (!aligned16(u->codes) || !aligned16(u->scale)) return fail(QSVD_EINVAL, "decode_attn_qu: pointers must be 16-byte aligned");
    }
    if (!aligned16(O) || (workspace && !aligned16(workspace)))
        return fail(QSVD_EINVAL, "decode_attn_qu: pointers must be 16-byte aligned");
    const size_t need = qsvd_decode_workspace_bytes(cache->B, max_seq_len, cache->r, H, dh);
    if (!workspace || workspace_bytes < need)
        return fail(QSVD_ENOSPC, "decode_attn_qu: workspace needs %zu bytes", need);
    DecodeArgs a{view(cache), seq_len, max_seq_len, UpW{U_q->codes, U_q->scale, U_q->bits},
                 UpW{U_k->codes, U_k->scale, U_k->bits}, UpW{U_v->codes, U_v->scale, U_v->bits}, H, dh,
                 softmax_scale, O};
    prof_mark(stream, "begin");
    const cudaError_t e = launch_decode(a, workspace, workspace_bytes, err, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "decode_attn_qu launch");
}

// Rows of one prefill group: the largest power of two up to kPrefillMaxRows
// whose decode workspace (queries and softmax partials, fp32) stays within
// kPrefillWsTarget bytes.  Larger groups measured faster all the way to 1024
// rows (fewer launches, fuller waves).
static int g_prefill_rows = 0;   // qsvd_set_prefill_group_rows; 0: automatic

static int prefill_group_rows(int64_t n, int max_len, int r, int H, int dh) {
    if (g_prefill_rows > 0) return int(std::min<int64_t>(g_prefill_rows, n));
    int rows = kPrefillMaxRows;
    while (rows > 16 && decode_workspace_bytes(rows, max_len, r, H, dh) > kPrefillWsTarget) rows /= 2;
    return int(std::min<int64_t>(rows, n));
}

int qsvd_set_prefill_group_rows(int32_t rows) {
    if (rows < 0 || rows > 65535) return fail(QSVD_EINVAL, "set_prefill_group_rows: rows outside [0, 65535]");
    const int prev = g_prefill_rows;
    g_prefill_rows = rows;
    return prev;
}

size_t qsvd_prefill_workspace_bytes(int64_t n, int32_t max_len, int32_t r, int32_t H, int32_t dh) {
    if (n <= 0 || max_len <= 0 || r <= 0 || H <= 0 || dh <= 0) return 0;
    return decode_workspace_bytes(prefill_group_rows(n, max_len, r, H, dh), max_len, r, H, dh);
}

int qsvd_latent_prefill_attn(const qsvd_cache *cache, const int32_t *q_seq, const int32_t *q_len, int64_t n,
                             int32_t max_len, const uint16_t *U_q, const uint16_t *U_k, const uint16_t *U_v,
                             int32_t H, int32_t dh, float softmax_scale, float *O, void *workspace,
                             size_t workspace_bytes, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if ((st = check_cache(cache))) return st;
    if (n < 0) return fail(QSVD_EINVAL, "prefill_attn: n < 0");
    if (n == 0) return QSVD_OK;
    if (!q_seq || !q_len || !U_q || !U_k || !U_v || !O) return fail(QSVD_EINVAL, "prefill_attn: null pointer");
    if (dh != 64 && dh != 128) return fail(QSVD_EUNSUPPORTED, "prefill_attn: dh must be 64 or 128");
    if (H <= 0) return fail(QSVD_EINVAL, "prefill_attn: H must be positive");
    if (cache->r > 3072 || cache->r % 32) return fail(QSVD_EUNSUPPORTED, "prefill_attn: need r %% 32 == 0 and r <= 3072");
    if ((H * dh) % 256 || H * dh > 6144) return fail(QSVD_EUNSUPPORTED, "prefill_attn: need H*dh %% 256 == 0 and H*dh <= 6144");
    if (max_len < 1 || max_len > cache->Tmax) return fail(QSVD_EINVAL, "prefill_attn: max_len outside [1, Tmax]");
    const void *ptrs[] = {q_seq, q_len, U_q, U_k, U_v, O, workspace};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return fail(QSVD_EINVAL, "prefill_attn: pointers must be 16-byte aligned");
    const int rows = prefill_group_rows(n, max_len, cache->r, H, dh);
    const size_t need = decode_workspace_bytes(rows, max_len, cache->r, H, dh);
    if (!workspace || workspace_bytes < need) return fail(QSVD_ENOSPC, "prefill_attn: workspace needs %zu bytes", need);
    const size_t d = size_t(H) * dh;
    prof_mark(stream, "begin");
    for (int64_t i0 = 0; i0 < n; i0 += rows) {
        // a group of rows is a decode step over a view whose row b is cache
        // sequence q_seq[i0 + b] at length q_len[i0 + b]
        CacheView v = view(cache);
        v.B = int(std::min<int64_t>(rows, n - i0));
        v.seq_map = q_seq + i0;
        DecodeArgs a{v, q_len + i0, max_len, UpW{U_q, nullptr, 16}, UpW{U_k, nullptr, 16}, UpW{U_v, nullptr, 16},
                     H, dh, softmax_scale, O + size_t(i0) * d};
        const cudaError_t e = launch_decode(a, workspace, workspace_bytes, err, stream);
        if (e != cudaSuccess) return cuda_fail(e, "prefill_attn launch");
    }
    return QSVD_OK;
}

}  // extern "C"

// Splits the (validated) host block list into launches of at most
// kPrefillMaxBlocks blocks and calls f(PrefillBlocks) for each; returns the
// first non-zero status of f.
template <typename F>
static int prefill_chunks(const qsvd_prefill_block *blocks, int32_t n_blocks, F &&f) {
    int64_t out = 0;
    for (int32_t i0 = 0; i0 < n_blocks; i0 += kPrefillMaxBlocks) {
        PrefillBlocks bl{};
        bl.n = std::min<int32_t>(kPrefillMaxBlocks, n_blocks - i0);
        int row = 0, tiles = 0;
        for (int k = 0; k < bl.n; ++k) {
            const qsvd_prefill_block &b = blocks[i0 + k];     // validated by the caller
            if (out > INT32_MAX - b.T) return fail(QSVD_EINVAL, "latent_prefill: more than 2^31 output rows");
            bl.seq[k] = b.seq;
            bl.t0[k] = b.t0;
            bl.L[k] = b.t0 + b.T;
            bl.row_off[k] = row;
            bl.out_off[k] = int(out);
            bl.qtile_off[k] = tiles;
            row += (bl.L[k] + 127) / 128 * 128;
            tiles += (b.T + 127) / 128;
            out += b.T;
        }
        bl.qtile_off[bl.n] = tiles;
        const int st = f(bl);
        if (st) return st;
    }
    return QSVD_OK;
}

extern "C" {

int qsvd_prefill_weights(const uint16_t *U_q, const uint16_t *U_k, const uint16_t *U_v, int32_t r, int32_t d,
                         uint16_t *Ut, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!U_q || !U_k || !U_v || !Ut) return fail(QSVD_EINVAL, "prefill_weights: null pointer");
    if (r <= 0 || d <= 0 || r % 64 || d % 256) return fail(QSVD_EUNSUPPORTED, "prefill_weights: need r %% 64 == 0 and d %% 256 == 0");
    const void *ptrs[] = {U_q, U_k, U_v, Ut};
    for (const void *p : ptrs)
        if (!aligned16(p)) return fail(QSVD_EINVAL, "prefill_weights: pointers must be 16-byte aligned");
    prof_mark(stream, "begin");
    const cudaError_t e = launch_prefill_weights(U_q, U_k, U_v, r, d, Ut, err, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "prefill_weights launch");
}

size_t qsvd_latent_prefill_workspace_bytes(const qsvd_prefill_block *blocks, int32_t n_blocks, int32_t r,
                                           int32_t H, int32_t dh) {
    if (!blocks || n_blocks <= 0 || r <= 0 || H <= 0 || dh <= 0) return 0;
    size_t R = 0;
    for (int32_t i0 = 0; i0 < n_blocks; i0 += kPrefillMaxBlocks) {
        size_t Rc = 0;
        for (int32_t k = i0; k < std::min<int32_t>(n_blocks, i0 + kPrefillMaxBlocks); ++k)
            Rc += size_t((int64_t(std::max(blocks[k].t0, 0)) + std::max(blocks[k].T, 0) + 127) / 128 * 128);
        R = std::max(R, Rc);
    }
    return prefill_mat_workspace_bytes(R, r, H * dh);
}

int qsvd_latent_prefill(const qsvd_cache *cache, const qsvd_prefill_block *blocks, int32_t n_blocks,
                        const uint16_t *Ut, int32_t H, int32_t dh, float softmax_scale, float *O, void *workspace,
                        size_t workspace_bytes, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if ((st = check_cache(cache))) return st;
    if (n_blocks < 0) return fail(QSVD_EINVAL, "latent_prefill: n_blocks < 0");
    if (n_blocks == 0) return QSVD_OK;
    if (!blocks || !Ut || !O) return fail(QSVD_EINVAL, "latent_prefill: null pointer");
    if (dh != 128) return fail(QSVD_EUNSUPPORTED, "latent_prefill: dh must be 128 (qsvd_latent_prefill_attn takes dh = 64)");
    if (H <= 0 || (H * dh) % 256) return fail(QSVD_EUNSUPPORTED, "latent_prefill: need H * dh %% 256 == 0");
    if (cache->r % 64) return fail(QSVD_EUNSUPPORTED, "latent_prefill: need r %% 64 == 0");
    if (!(softmax_scale > 0.0f) || !std::isfinite(softmax_scale))
        return fail(QSVD_EINVAL, "latent_prefill: softmax_scale must be positive and finite");
    const void *ptrs[] = {Ut, O, workspace};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return fail(QSVD_EINVAL, "latent_prefill: pointers must be 16-byte aligned");
    for (int32_t k = 0; k < n_blocks; ++k) {
        const qsvd_prefill_block &b = blocks[k];
        if (b.seq < 0 || b.seq >= cache->B || b.t0 < 0 || b.T < 1 || int64_t(b.t0) + b.T > cache->Tmax)
            return fail(QSVD_EINVAL, "latent_prefill: block %d (seq %d, t0 %d, T %d) outside the cache", int(k),
                        int(b.seq), int(b.t0), int(b.T));
    }
    for (int32_t i0 = 0; i0 < n_blocks; i0 += kPrefillMaxBlocks) {
        // the kernels index a launch's padded rows (and R * r / 8 prep threads) with 32-bit integers
        int64_t R = 0;
        for (int32_t k = i0; k < std::min<int32_t>(n_blocks, i0 + kPrefillMaxBlocks); ++k)
            R += (int64_t(blocks[k].t0) + blocks[k].T + 127) / 128 * 128;
        if (R * (cache->r / 8) >= (int64_t(1) << 31))
            return fail(QSVD_EUNSUPPORTED, "latent_prefill: blocks %d.. hold too many rows for one launch", int(i0));
    }
    const size_t need = qsvd_latent_prefill_workspace_bytes(blocks, n_blocks, cache->r, H, dh);
    if (!workspace || workspace_bytes < need)
        return fail(QSVD_ENOSPC, "latent_prefill: workspace needs %zu bytes", need);
    const CacheView c = view(cache);
    prof_mark(stream, "begin");
    return prefill_chunks(blocks, n_blocks, [&](const PrefillBlocks &bl) -> int {
        const cudaError_t e = launch_prefill_mat(c, bl, Ut, H, softmax_scale, O, workspace, err, stream);
        return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "latent_prefill launch");
    });
}

size_t qsvd_importance_workspace_bytes(int32_t N, int32_t m, int32_t k) {
    if (N <= 0 || m <= 0 || k <= 0) return 0;
    return align256(size_t(N) * ((size_t(m) + kImpRowTile - 1) / kImpRowTile) * k * sizeof(float));
}

size_t qsvd_rank_budget_workspace_bytes(void) { return rank_workspace_bytes(); }

int qsvd_rank_budget(const float *scores, int32_t n, int32_t k, uint8_t *keep, void *workspace,
                     size_t workspace_bytes, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!scores || !keep) return fail(QSVD_EINVAL, "rank_budget: null pointer");
    if (n <= 0 || k < 0 || k > n) return fail(QSVD_EINVAL, "rank_budget: need n > 0 and 0 <= k <= n");
    if (!workspace || workspace_bytes < rank_workspace_bytes())
        return fail(QSVD_ENOSPC, "rank_budget: workspace needs %zu bytes", rank_workspace_bytes());
    if (!aligned16(workspace)) return fail(QSVD_EINVAL, "rank_budget: workspace must be 16-byte aligned");
    prof_mark(stream, "begin");
    const cudaError_t e = launch_rank_budget(scores, n, k, keep, workspace, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "rank_budget launch");
}

int qsvd_importance_scores(const float *U, const float *sigma, const float *Vt, const float *G, int32_t N, int32_t m,
                           int32_t n, int32_t k, float *scores, void *workspace, size_t workspace_bytes,
                           cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!U || !sigma || !Vt || !G || !scores) return fail(QSVD_EINVAL, "importance_scores: null pointer");
    if (N <= 0 || m <= 0 || n <= 0 || k <= 0) return fail(QSVD_EINVAL, "importance_scores: N, m, n, k must be positive");
    if (N > 65535) return fail(QSVD_EUNSUPPORTED, "importance_scores: more than 65535 samples per call");
    const size_t need = qsvd_importance_workspace_bytes(N, m, k);
    if (!workspace || workspace_bytes < need)
        return fail(QSVD_ENOSPC, "importance_scores: workspace needs %zu bytes", need);
    prof_mark(stream, "begin");
    const cudaError_t e = launch_importance(U, sigma, Vt, G, N, m, n, k, scores, static_cast<float *>(workspace), err, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "importance_scores launch");
}

int qsvd_beta_factors(const double *Wd_r, const double *Wu_r, const double *fd, const double *fu, int32_t E,
                      int32_t r, int32_t n_out, int32_t u_bits, float u_clip, float *W_d, void *u_codes,
                      float *u_scale, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!Wd_r || !Wu_r || !fd || !fu || !W_d || !u_codes || !u_scale) return fail(QSVD_EINVAL, "beta_factors: null pointer");
    if (E <= 0 || r <= 0 || n_out <= 0 || n_out % 128)
        return fail(QSVD_EINVAL, "beta_factors: need E > 0, r > 0 and n_out %% 128 == 0");
    if (u_bits != 8 && u_bits != 4) return fail(QSVD_EINVAL, "beta_factors: u_bits must be 8 or 4");
    if (!(u_clip > 0.0f && u_clip <= 1.0f)) return fail(QSVD_EINVAL, "beta_factors: u_clip must lie in (0, 1]");
    const void *ptrs[] = {Wd_r, Wu_r, fd, fu, W_d, u_codes, u_scale};
    for (const void *p : ptrs)
        if (!aligned16(p)) return fail(QSVD_EINVAL, "beta_factors: pointers must be 16-byte aligned");
    prof_mark(stream, "begin");
    const cudaError_t e = launch_beta_factors(Wd_r, Wu_r, fd, fu, E, r, n_out, u_bits, u_clip, W_d, u_codes, u_scale,
                                              stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "beta_factors launch");
}

size_t qsvd_beta_objective_workspace_bytes(int64_t N, int32_t n_out) {
    if (N <= 0 || n_out <= 0) return 0;
    return beta_objective_partials(N, n_out) * sizeof(double);
}

int qsvd_beta_objective(const float *Y, int64_t N, int32_t n_out, const void *lat_codes, const void *lat_scales,
                        int32_t lat_bits, int32_t r, const void *u_codes, const float *u_scale, int32_t u_bits,
                        double *objective, void *workspace, size_t workspace_bytes, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if (!Y || !lat_codes || !lat_scales || !u_codes || !u_scale || !objective)
        return fail(QSVD_EINVAL, "beta_objective: null pointer");
    if (N <= 0 || N > int64_t(65535) * 64) return fail(QSVD_EINVAL, "beta_objective: need 0 < N <= 4194240");
    if (n_out <= 0 || n_out % 64) return fail(QSVD_EINVAL, "beta_objective: need n_out %% 64 == 0");
    if (lat_bits != 8 && lat_bits != 4) return fail(QSVD_EINVAL, "beta_objective: lat_bits must be 8 or 4");
    if (u_bits != 8 && u_bits != 4) return fail(QSVD_EINVAL, "beta_objective: u_bits must be 8 or 4");
    if (r <= 0 || r % 32 || (lat_bits == 4 && r % 128))
        return fail(QSVD_EINVAL, "beta_objective: need r %% 32 == 0 (r %% 128 == 0 for an int4 latent)");
    const void *ptrs[] = {Y, lat_codes, lat_scales, u_codes, u_scale, objective, workspace};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return fail(QSVD_EINVAL, "beta_objective: pointers must be 16-byte aligned");
    const size_t need = qsvd_beta_objective_workspace_bytes(N, n_out);
    if (!workspace || workspace_bytes < need)
        return fail(QSVD_ENOSPC, "beta_objective: workspace needs %zu bytes", need);
    prof_mark(stream, "begin");
    const cudaError_t e = launch_beta_objective(Y, N, n_out, lat_codes, lat_scales, lat_bits, r, u_codes, u_scale,
                                                u_bits, static_cast<double *>(workspace), objective, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "beta_objective launch");
}

// Workspace of a decode step: the projection's part (completion counter, X
// codes and scales, the new latents c_hat) followed by the attention's.
static size_t step_proj_bytes(int B, int d, int r) {
    return 256 + align256(size_t(B) * d) + align256(size_t(B) * 4) + align256(size_t(B) * r * 4);
}

size_t qsvd_decode_step_workspace_bytes(int32_t B, int32_t max_seq_len, int32_t d, int32_t r, int32_t H,
                                        int32_t dh) {
    if (B <= 0 || max_seq_len <= 0 || d <= 0 || r <= 0 || H <= 0 || dh <= 0) return 0;
    return step_proj_bytes(B, d, r) + decode_workspace_bytes(B, max_seq_len, r, H, dh);
}

int qsvd_decode_step(const qsvd_down_weight *W, const uint16_t *X, const qsvd_cache *cache, const int32_t *seq_len,
                     int32_t max_seq_len, const uint16_t *U_q, const uint16_t *U_k, const uint16_t *U_v, int32_t H,
                     int32_t dh, float act_clip, float lat_clip, float softmax_scale, float *O, void *workspace,
                     size_t workspace_bytes, cudaStream_t stream) {
    int *err = nullptr;
    int st = device_setup(&err);
    if (st) return st;
    if ((st = check_cache(cache))) return st;
    if (!W || !W->codes || !W->scale || !X || !seq_len || !U_q || !U_k || !U_v || !O)
        return fail(QSVD_EINVAL, "decode_step: null pointer");
    if (W->rot) return fail(QSVD_EUNSUPPORTED, "decode_step: rotated weights (W->rot) need qsvd_latent_project");
    if ((W->w_bits && W->w_bits != 8) || (W->x_bits && W->x_bits != 8))
        return fail(QSVD_EUNSUPPORTED, "decode_step: 4-bit settings (W->w_bits, W->x_bits) need qsvd_latent_project");
    const int d = W->d, r = W->r, B = cache->B;
    if (r != cache->r) return fail(QSVD_EINVAL, "decode_step: weight rank differs from the cache's");
    if (dh != 64 && dh != 128) return fail(QSVD_EUNSUPPORTED, "decode_step: dh must be 64 or 128");
    if (H <= 0 || H * dh != d) return fail(QSVD_EINVAL, "decode_step: H * dh must equal d");
    if (d % 256 || d > 6144) return fail(QSVD_EUNSUPPORTED, "decode_step: need d %% 256 == 0 and d <= 6144");
    if (r > 3072 || r % 32) return fail(QSVD_EUNSUPPORTED, "decode_step: need r %% 32 == 0 and r <= 3072");
    if (B > kPsMaxSplitTok) return fail(QSVD_EUNSUPPORTED, "decode_step: more than %d sequences", kPsMaxSplitTok);
    if (max_seq_len < 1 || max_seq_len > cache->Tmax)
        return fail(QSVD_EINVAL, "decode_step: max_seq_len outside [1, Tmax]");
    if (!(act_clip > 0.0f && act_clip <= 1.0f) || !(lat_clip > 0.0f && lat_clip <= 1.0f))
        return fail(QSVD_EINVAL, "decode_step: clip ratios must lie in (0, 1]");
    const void *ptrs[] = {X, W->codes, W->scale, U_q, U_k, U_v, O, workspace};
    for (const void *p : ptrs)
        if (p && !aligned16(p)) return fail(QSVD_EINVAL, "decode_step: pointers must be 16-byte aligned");
    const size_t need = qsvd_decode_step_workspace_bytes(B, max_seq_len, d, r, H, dh);
    if (!workspace || workspace_bytes < need) return fail(QSVD_ENOSPC, "decode_step: workspace needs %zu bytes", need);

    char *wsp = static_cast<char *>(workspace);
    int *counter = reinterpret_cast<int *>(wsp);
    int8_t *xq = reinterpret_cast<int8_t *>(wsp + 256);
    float *xs = reinterpret_cast<float *>(wsp + 256 + align256(size_t(B) * d));
    float *c_hat = reinterpret_cast<float *>(wsp + 256 + align256(size_t(B) * d) + align256(size_t(B) * 4));
    char *dws = wsp + step_proj_bytes(B, d, r);

    prof_mark(stream, "begin");
    // a1-a2: the decode-size projection leaves the new latents in c_hat (one
    // token: every CTA quantizes the row itself; more: each row quantized once)
    cudaError_t e = cudaSuccess;
    if (B < kPsSplitTok) {
        e = launch_proj_small(X, B, d, act_clip, W->codes, W->scale, r, cache->bits, lat_clip, c_hat, counter, nullptr,
                              nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, err, stream, nullptr,
                              nullptr, false, 127);
    } else {
        e = launch_xquant(X, B, d, act_clip, xq, nullptr, xs, stream, 0, 127);
        if (e == cudaSuccess)
            e = launch_proj_small(X, B, d, act_clip, W->codes, W->scale, r, cache->bits, lat_clip, c_hat, counter,
                                  nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, err, stream,
                                  xq, xs, false, 127);
    }
    if (e != cudaSuccess) return cuda_fail(e, "decode_step projection launch");
    // a3-a8: requantize and append the new latents, then attend
    DecodeArgs a{view(cache), seq_len, max_seq_len, UpW{U_q, nullptr, 16}, UpW{U_k, nullptr, 16},
                 UpW{U_v, nullptr, 16}, H, dh, softmax_scale, O, c_hat, lat_clip};
    e = launch_decode(a, dws, workspace_bytes - step_proj_bytes(B, d, r), err, stream);
    return e == cudaSuccess ? QSVD_OK : cuda_fail(e, "decode_step attention launch");
}

}  // extern "C"
