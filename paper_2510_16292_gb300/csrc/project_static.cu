// Allocation-free variant of the decode-size projection (qsvd_latent_project
// for T <= 16 tokens).
//
// Some callers cannot allocate device memory when they project a token: a
// serving process whose device memory was fully reserved at start-up by
// another allocator, or code that runs while a stream is being captured into
// a CUDA graph (where cudaMalloc is not allowed).  They cannot provide the
// workspace qsvd_latent_project needs either.  This entry point keeps that
// scratch (a completion counter and the fp32 latent rows, 16 x 4096 floats)
// in a file-scope device array instead.  The array is part of the library's
// module image: every GPU that loads the library holds it (264 KiB) until the
// process exits.  Nothing here calls cudaMalloc, cudaFree or any allocating
// routine.
#include <cstdio>
#include <mutex>

#include "launch.h"
#include "qsvd.h"

namespace qsvd {

constexpr int kStaticMaxT = kPsMaxTok;      // tokens per call (decode-size projection)
constexpr int kStaticMaxR = 4096;           // latent rank
constexpr size_t kStaticCounterBytes = 256;
constexpr size_t kStaticBytes = kStaticCounterBytes + size_t(kStaticMaxT) * kStaticMaxR * sizeof(float);

// [0, 256): completion counter (int); [256, ...): c_hat [kStaticMaxT][r] fp32.
static __device__ __align__(256) unsigned char g_project_scratch[kStaticBytes];

namespace {

constexpr int kMaxDev = 64;
void *g_scratch_ptr[kMaxDev];      // device address of g_project_scratch per device (set up once)
std::mutex g_scratch_mu;

int sfail(int code, const char *msg) { return set_last_error(code, msg); }

// Set-up, once per device with that device current: the host-side name of
// the array is not a device address, so ask the runtime for the real one.
int scratch_for_current_device(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev)
        return sfail(QSVD_ECUDA, "latent_project_static: no usable current device");
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_project_scratch) != cudaSuccess || !p)
            return sfail(QSVD_ECUDA, "latent_project_static: cudaGetSymbolAddress of the scratch array failed");
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return QSVD_OK;
}

}  // namespace
}  // namespace qsvd

using namespace qsvd;

extern "C" {

int qsvd_latent_project_static(const qsvd_down_weight *W, const uint16_t *X, int64_t T, float act_clip,
                               int32_t lat_bits, float lat_clip, void *lat_codes, void *lat_scales,
                               const qsvd_cache *dst, const int32_t *dst_seq, const int32_t *dst_pos,
                               cudaStream_t stream) {
    int *err = nullptr;
    int st = setup_current_device(&err);     // sm_103 check and error word, cached per device
    if (st) return st;
    void *scratch = nullptr;
    if ((st = scratch_for_current_device(&scratch))) return st;
    if (!W || !W->codes || !W->scale || !X) return sfail(QSVD_EINVAL, "latent_project_static: null pointer");
    if (W->rot) return sfail(QSVD_EUNSUPPORTED, "latent_project_static: rotated weights (W->rot) need qsvd_latent_project");
    const int xb = W->x_bits ? W->x_bits : 8, wb = W->w_bits ? W->w_bits : 8;
    if ((xb != 8 && xb != 4) || (wb != 8 && wb != 4))
        return sfail(QSVD_EINVAL, "latent_project_static: W->w_bits and W->x_bits must be 8 or 4");
    const void *ptrs[] = {X, W->codes, lat_codes, lat_scales};
    for (const void *p : ptrs)
        if (p && (reinterpret_cast<uintptr_t>(p) & 15u))
            return sfail(QSVD_EINVAL, "latent_project_static: pointers must be 16-byte aligned");
    const int d = W->d, r = W->r;
    if (T < 0) return sfail(QSVD_EINVAL, "latent_project_static: T < 0");
    if (T > kStaticMaxT)
        return sfail(QSVD_ENOSPC, "latent_project_static: T exceeds the 16-token maximum of the static scratch");
    if (r > kStaticMaxR)
        return sfail(QSVD_ENOSPC, "latent_project_static: r exceeds the 4096-channel maximum of the static scratch");
    if (d <= 0 || r <= 0 || d % 256 || d > 6144 || r % 16)
        return sfail(QSVD_EUNSUPPORTED, "latent_project_static: need d % 256 == 0, d <= 6144, r % 16 == 0");
    if (lat_bits != 8 && lat_bits != 4) return sfail(QSVD_EINVAL, "latent_project_static: lat_bits must be 8 or 4");
    if (lat_bits == 4 && r % 128) return sfail(QSVD_EUNSUPPORTED, "latent_project_static: int4 needs r % 128 == 0");
    if (!(act_clip > 0.0f && act_clip <= 1.0f) || !(lat_clip > 0.0f && lat_clip <= 1.0f))
        return sfail(QSVD_EINVAL, "latent_project_static: clip ratios must lie in (0, 1]");
    const bool tok = lat_codes || lat_scales;
    if (tok && (!lat_codes || !lat_scales)) return sfail(QSVD_EINVAL, "latent_project_static: give both lat_codes and lat_scales");
    if (!tok && !dst) return sfail(QSVD_EINVAL, "latent_project_static: no destination for the latent");
    CacheView dv{};
    if (dst) {
        if ((st = validate_cache(dst))) return st;      // null, alignment (the rows are stored as words), sizes
        if (dst->bits != lat_bits || dst->r != r)
            return sfail(QSVD_EINVAL, "latent_project_static: cache does not match the projection");
        if (T > 0 && (!dst_seq || !dst_pos)) return sfail(QSVD_EINVAL, "latent_project_static: dst_seq/dst_pos required");
        dv = CacheView{dst->codes, dst->scales, dst->bits, dst->B, dst->Tmax, dst->r};
    }
    if (T == 0) return QSVD_OK;
    char *base = static_cast<char *>(scratch);
    int *counter = reinterpret_cast<int *>(base);
    float *c_hat = reinterpret_cast<float *>(base + kStaticCounterBytes);
    // The array keeps the previous call's contents; only the completion
    // counter must start at zero (a call abandoned mid-way could leave it set).
    cudaError_t e = cudaMemsetAsync(counter, 0, sizeof(int), stream);
    if (e == cudaSuccess)
        e = launch_proj_small(X, int(T), d, act_clip, W->codes, W->scale, r, lat_bits, lat_clip, c_hat, counter,
                              nullptr, nullptr, nullptr, lat_codes, lat_scales, dst ? &dv : nullptr, dst_seq, dst_pos,
                              err, stream, nullptr, nullptr, true, xb == 8 ? 127 : 7);
    if (e != cudaSuccess) {
        char msg[160];
        snprintf(msg, sizeof(msg), "latent_project_static: %s", cudaGetErrorString(e));
        return set_last_error(QSVD_ECUDA, msg);
    }
    return QSVD_OK;
}

}  // extern "C"
