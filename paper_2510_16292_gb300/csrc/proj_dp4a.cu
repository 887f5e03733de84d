// Exact int8 x int8 -> int32 down-projection on the CUDA cores (dp4a), with
// the dequantization of Eq. 12's product fused behind it:
//   acc[t, j]   = sum_k xq[t, k] * w[j, k]          (exact: |acc| < 2^31)
//   c_hat[t, j] = fp32(fp32(fp32(acc) * s_x[t]) * s_w[j])
// This is the small-T path (decode: one token per sequence), where the GEMM
// is bound by reading W_d's int8 codes once; prefill-sized T goes to the
// tensor-core kernel.
#include "common.cuh"
#include "launch.h"

namespace qsvd {

constexpr int kPjWarps = 8;       // output channels per CTA (one per warp)
constexpr int kPjTokens = 16;     // tokens per CTA (grid.y tiles T)

__global__ void __launch_bounds__(kPjWarps * 32)
proj_dp4a_kernel(const int8_t *__restrict__ xq, int64_t T, int d, const int8_t *__restrict__ w,
                 const float *__restrict__ ws, const float *__restrict__ xs, int r,
                 float *__restrict__ c_hat, int32_t *__restrict__ acc_out) {
    const int lane = threadIdx.x & 31;
    const int j = blockIdx.x * kPjWarps + (threadIdx.x >> 5);
    if (j >= r) return;
    const int64_t t0 = int64_t(blockIdx.y) * kPjTokens;
    const int64_t t1 = (T < t0 + kPjTokens) ? T : t0 + kPjTokens;
    const int nint = d >> 2;
    const int *wrow = reinterpret_cast<const int *>(w + size_t(j) * d);
    const float sw = ws[j];
    for (int64_t t = t0; t < t1; ++t) {
        const int *xrow = reinterpret_cast<const int *>(xq + t * d);
        int acc = 0;
#pragma unroll 4
        for (int i = lane; i < nint; i += 32) acc = __dp4a(wrow[i], xrow[i], acc);
        acc = warp_sum_int(acc);
        if (lane == 0) {
            c_hat[t * r + j] = __fmul_rn(__fmul_rn(__int2float_rn(acc), xs[t]), sw);
            if (acc_out) acc_out[t * r + j] = acc;
        }
    }
}

cudaError_t launch_proj_dp4a(const int8_t *xq, int64_t T, int d, const int8_t *wcodes, const float *ws,
                             const float *xs, int r, float *c_hat, int32_t *acc_out, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    dim3 grid((r + kPjWarps - 1) / kPjWarps, unsigned((T + kPjTokens - 1) / kPjTokens));
    proj_dp4a_kernel<<<grid, kPjWarps * 32, 0, s>>>(xq, T, d, wcodes, ws, xs, r, c_hat, acc_out);
    prof_mark(s, "proj_dp4a");
    return cudaGetLastError();
}

}  // namespace qsvd
