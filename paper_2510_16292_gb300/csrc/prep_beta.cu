// Offline choice of beta (Sec. 3.3, Eq. 13-14) on the GPU.
//
// Eq. 3 splits the truncated joint SVD W_concat ~ Wd_r diag(sigma) Wu_r as
// W_d = Wd_r Sigma^beta and W^u = Sigma^(1-beta) Wu_r; beta moves the
// channel spread of Eq. 13 between the latent C = X W_d and W^u, and so the
// quantization error.  Eq. 14 picks beta to minimise the squared difference
// between the layer output without quantization, Y = X W_concat, and with
// it, Y' = Q(C) Q(W^u) (Eq. 11), over calibration tokens.  Per beta:
//
//   beta_wd_kernel     W_d = fp32(Wd_r[k, i] * sigma_i^beta), the input of
//                      the per-channel weight quantizer (qsvd_quantize_weight)
//   beta_up_kernel     Q(W^u): W^u[i, j] = sigma_i^(1-beta) Wu_r[i, j] in
//                      fp64 and its symmetric RTN per output channel j
//                      (int8 or packed int4 codes, one fp32 scale per j)
//   beta_err_kernel    sum over a 64 x 64 tile of (Y - Y')^2: the products
//                      of codes are exact integer sums (dp4a), the scales
//                      and the squares are applied in fp64
//   beta_sum_kernel    the tiles' sums added in a fixed order
//
// The latent Q(C) of the calibration tokens comes from qsvd_latent_project
// (token-major codes and scales).  Every sum runs in a fixed order, so the
// objective has the same bits on every run.
#include <algorithm>
#include <cstdint>
#include <cuda_fp16.h>

#include "common.cuh"
#include "launch.h"
#include "prep_beta.h"

namespace qsvd {

namespace {

__global__ void beta_wd_kernel(const double *__restrict__ Wd_r, const double *__restrict__ fd, int64_t n, int r,
                               float *__restrict__ W_d) {
    for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < n; i += int64_t(gridDim.x) * blockDim.x)
        W_d[i] = __double2float_rn(Wd_r[i] * fd[i % r]);
}

// CTA: kBuTx x kBuCols consecutive output channels, rows split over kBuTy
// groups (32 channels per CTA: n_out / 32 CTAs, 384 at the 7B shape).
constexpr int kBuCols = 4, kBuTx = 8, kBuTy = 32;

__global__ void __launch_bounds__(kBuTx * kBuTy)
beta_up_kernel(const double *__restrict__ Wu_r, const double *__restrict__ fu, int r, int n_out, int qmax, float clip,
               uint8_t *__restrict__ codes, float *__restrict__ scale) {
    __shared__ double red[kBuTy][kBuTx * kBuCols];
    __shared__ float s_sh[kBuTx * kBuCols];
    const int tx = threadIdx.x % kBuTx, ty = threadIdx.x / kBuTx;
    const int j0 = (blockIdx.x * kBuTx + tx) * kBuCols;
    const int per = (r + kBuTy - 1) / kBuTy, i0 = min(r, ty * per), i1 = min(r, i0 + per);
    // m_j = max_i |W^u[i, j]| (exact in fp64)
    double m[kBuCols] = {0.0, 0.0, 0.0, 0.0};
    for (int i = i0; i < i1; ++i) {
        const double f = fu[i];
        const double *row = Wu_r + size_t(i) * n_out + j0;
#pragma unroll
        for (int c = 0; c < kBuCols; ++c) m[c] = fmax(m[c], fabs(f * row[c]));
    }
#pragma unroll
    for (int c = 0; c < kBuCols; ++c) red[ty][tx * kBuCols + c] = m[c];
    __syncthreads();
    if (ty == 0) {
#pragma unroll
        for (int c = 0; c < kBuCols; ++c) {
            double mm = red[0][tx * kBuCols + c];
            for (int g = 1; g < kBuTy; ++g) mm = fmax(mm, red[g][tx * kBuCols + c]);
            // s = fp32(fp32(clip * m) / q_max): each step in fp64 (m is an fp64 value), rounded to fp32
            const float s = __double2float_rn(double(__double2float_rn(double(clip) * mm)) / double(qmax));
            s_sh[tx * kBuCols + c] = s;
            scale[j0 + c] = s;
        }
    }
    __syncthreads();
    float s[kBuCols];
#pragma unroll
    for (int c = 0; c < kBuCols; ++c) s[c] = s_sh[tx * kBuCols + c];
    for (int i = i0; i < i1; ++i) {
        const double f = fu[i];
        const double *row = Wu_r + size_t(i) * n_out + j0;
        int q[kBuCols];
#pragma unroll
        for (int c = 0; c < kBuCols; ++c) {
            // code = clamp(rne(fp32(v / s))), the quotient in fp64; 0 when s == 0
            int v = 0;
            if (s[c] != 0.0f) {
                v = __float2int_rn(__double2float_rn((f * row[c]) / double(s[c])));
                v = v < -qmax ? -qmax : (v > qmax ? qmax : v);
            }
            q[c] = v;
        }
        if (qmax == 127)
            *reinterpret_cast<uint32_t *>(codes + size_t(i) * n_out + j0) =
                uint32_t(q[0] & 0xff) | (uint32_t(q[1] & 0xff) << 8) | (uint32_t(q[2] & 0xff) << 16) |
                (uint32_t(q[3] & 0xff) << 24);
        else
            *reinterpret_cast<uint16_t *>(codes + size_t(i) * (n_out / 2) + j0 / 2) =
                uint16_t((q[0] & 0xf) | ((q[1] & 0xf) << 4) | ((q[2] & 0xf) << 8) | ((q[3] & 0xf) << 12));
    }
}

// Objective tiles: 64 calibration rows x 64 output channels per CTA, 32
// latent channels per step; thread (ty, tx) takes rows ty + 16 a and
// channels tx + 16 b (a, b < 4).  Shared rows of 36 bytes keep the 4-byte
// reads of the 16 columns of a warp on distinct banks.
constexpr int kObTile = 64, kObK = 32, kObThreads = 256, kObStride = kObK + 4;

__device__ __forceinline__ int8_t nib(uint32_t w, int e) {
    return int8_t(int32_t(w << (28 - 4 * e)) >> 28);        // nibble e, two's complement
}

__global__ void __launch_bounds__(kObThreads)
beta_err_kernel(const float *__restrict__ Y, int64_t N, int n_out, const void *__restrict__ lat_codes,
                const void *__restrict__ lat_scales, int lat_bits, int r, const uint8_t *__restrict__ u_codes,
                const float *__restrict__ u_scale, int u_bits, double *__restrict__ partial) {
    __shared__ __align__(16) int8_t a_s[kObTile * kObStride];    // latent codes [row][channel]
    __shared__ __align__(16) int8_t b_s[kObTile * kObStride];    // U codes [output channel][latent channel]
    __shared__ double red[kObThreads];
    const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
    const int64_t n0 = int64_t(blockIdx.y) * kObTile;
    const int j0 = blockIdx.x * kObTile;
    int acc[4][4];
    double yq[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            acc[a][b] = 0;
            yq[a][b] = 0.0;
        }
    for (int k0 = 0; k0 < r; k0 += kObK) {
        __syncthreads();
        {   // A: row tid / 4, latent channels k0 + 8 (tid % 4) .. + 7
            const int row = tid / 4, part = tid % 4;
            const int64_t n = n0 + row;
            uint32_t w0 = 0u, w1 = 0u;
            if (n < N) {
                if (lat_bits == 8) {
                    const uint2 w = *reinterpret_cast<const uint2 *>(static_cast<const int8_t *>(lat_codes) + n * r +
                                                                     k0 + part * 8);
                    w0 = w.x;
                    w1 = w.y;
                } else {
                    const uint32_t w = *reinterpret_cast<const uint32_t *>(
                        static_cast<const uint8_t *>(lat_codes) + n * (r / 2) + (k0 + part * 8) / 2);
                    w0 = uint32_t(uint8_t(nib(w, 0))) | (uint32_t(uint8_t(nib(w, 1))) << 8) |
                         (uint32_t(uint8_t(nib(w, 2))) << 16) | (uint32_t(uint8_t(nib(w, 3))) << 24);
                    w1 = uint32_t(uint8_t(nib(w, 4))) | (uint32_t(uint8_t(nib(w, 5))) << 8) |
                         (uint32_t(uint8_t(nib(w, 6))) << 16) | (uint32_t(uint8_t(nib(w, 7))) << 24);
                }
            }
            *reinterpret_cast<uint32_t *>(a_s + row * kObStride + part * 8) = w0;
            *reinterpret_cast<uint32_t *>(a_s + row * kObStride + part * 8 + 4) = w1;
        }
        {   // B: latent channel k0 + tid / 8, output channels j0 + 8 (tid % 8) .. + 7, stored transposed
            const int ch = tid / 8, part = tid % 8;
            int8_t v[8];
            if (u_bits == 8) {
                const uint2 w = *reinterpret_cast<const uint2 *>(u_codes + size_t(k0 + ch) * n_out + j0 + part * 8);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    v[e] = int8_t(w.x >> (8 * e));
                    v[4 + e] = int8_t(w.y >> (8 * e));
                }
            } else {
                const uint32_t w = *reinterpret_cast<const uint32_t *>(u_codes + size_t(k0 + ch) * (n_out / 2) +
                                                                       (j0 + part * 8) / 2);
#pragma unroll
                for (int e = 0; e < 8; ++e) v[e] = nib(w, e);
            }
#pragma unroll
            for (int e = 0; e < 8; ++e) b_s[(part * 8 + e) * kObStride + ch] = v[e];
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kObK; kk += 4) {
            int a4[4], b4[4];
#pragma unroll
            for (int a = 0; a < 4; ++a) a4[a] = *reinterpret_cast<const int *>(a_s + (ty + 16 * a) * kObStride + kk);
#pragma unroll
            for (int b = 0; b < 4; ++b) b4[b] = *reinterpret_cast<const int *>(b_s + (tx + 16 * b) * kObStride + kk);
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[a][b] = __dp4a(a4[a], b4[b], acc[a][b]);
        }
        if (lat_bits == 4 && (k0 + kObK) % 128 == 0) {
            // the end of a 128-channel group: its codes' sums times the row's group scale
            const int g = k0 / 128;
#pragma unroll
            for (int a = 0; a < 4; ++a) {
                const int64_t n = n0 + ty + 16 * a;
                const double sg = n < N ? double(__half2float(static_cast<const __half *>(lat_scales)[n * (r / 128) + g]))
                                        : 0.0;
#pragma unroll
                for (int b = 0; b < 4; ++b) {
                    yq[a][b] += sg * double(acc[a][b]);
                    acc[a][b] = 0;
                }
            }
        }
    }
    double err = 0.0;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const int64_t n = n0 + ty + 16 * a;
        if (n >= N) continue;
        const double sr = lat_bits == 8 ? double(static_cast<const float *>(lat_scales)[n]) : 0.0;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int j = j0 + tx + 16 * b;
            const double y = (lat_bits == 8 ? double(acc[a][b]) * sr : yq[a][b]) * double(u_scale[j]);
            const double dl = double(Y[n * n_out + j]) - y;
            err += dl * dl;
        }
    }
    red[tid] = err;
    __syncthreads();
    for (int s = kObThreads / 2; s > 0; s >>= 1) {
        if (tid < s) red[tid] += red[tid + s];
        __syncthreads();
    }
    if (tid == 0) partial[size_t(blockIdx.y) * gridDim.x + blockIdx.x] = red[0];
}

constexpr int kSumThreads = 256;

__global__ void __launch_bounds__(kSumThreads) beta_sum_kernel(const double *partial, int64_t n, double *out) {
    __shared__ double red[kSumThreads];
    pdl_wait();
    double v = 0.0;
    for (int64_t i = threadIdx.x; i < n; i += kSumThreads) v += partial[i];
    red[threadIdx.x] = v;
    __syncthreads();
    for (int s = kSumThreads / 2; s > 0; s >>= 1) {
        if (int(threadIdx.x) < s) red[threadIdx.x] += red[threadIdx.x + s];
        __syncthreads();
    }
    if (threadIdx.x == 0) *out = red[0];
}

}  // namespace

size_t beta_objective_partials(int64_t N, int n_out) {
    return size_t((N + kObTile - 1) / kObTile) * size_t(n_out / kObTile);
}

cudaError_t launch_beta_factors(const double *Wd_r, const double *Wu_r, const double *fd, const double *fu, int E,
                                int r, int n_out, int u_bits, float u_clip, float *W_d, void *u_codes, float *u_scale,
                                cudaStream_t s) {
    const int64_t n = int64_t(E) * r;
    const int blocks = int(std::min<int64_t>((n + 255) / 256, 152 * 8));
    beta_wd_kernel<<<blocks, 256, 0, s>>>(Wd_r, fd, n, r, W_d);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    beta_up_kernel<<<n_out / (kBuTx * kBuCols), kBuTx * kBuTy, 0, s>>>(Wu_r, fu, r, n_out, u_bits == 8 ? 127 : 7,
                                                                       u_clip, static_cast<uint8_t *>(u_codes),
                                                                       u_scale);
    e = cudaGetLastError();
    prof_mark(s, "beta_factors");
    return e;
}

cudaError_t launch_beta_objective(const float *Y, int64_t N, int n_out, const void *lat_codes, const void *lat_scales,
                                  int lat_bits, int r, const void *u_codes, const float *u_scale, int u_bits,
                                  double *partial, double *objective, cudaStream_t s) {
    const dim3 grid(unsigned(n_out / kObTile), unsigned((N + kObTile - 1) / kObTile));
    beta_err_kernel<<<grid, kObThreads, 0, s>>>(Y, N, n_out, lat_codes, lat_scales, lat_bits, r,
                                                static_cast<const uint8_t *>(u_codes), u_scale, u_bits, partial);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    e = launch_pdl(beta_sum_kernel, dim3(1), dim3(kSumThreads), 0, s, static_cast<const double *>(partial),
                   int64_t(grid.x) * grid.y, objective);
    prof_mark(s, "beta_objective");
    return e;
}

}  // namespace qsvd
