// Quantization, requantization and cache-append kernels.
//
//   xquant_kernel       a1: per-token symmetric int8 RTN of X (Sec. 4 setup),
//                       Q(X H1^T) of Eq. 12: H1 = I, or the block Hadamard
//                       rotation applied to the row first (rot = block size).
//   weight_quant_kernel offline per-output-channel int8 RTN of W_d.
//   weight_quant_rot_kernel  the same for H1 W_d (the rotation down each
//                       column first).
// H1 = I_{d/b} (x) H_b / sqrt(b) (H_b Sylvester, b a power of two dividing d)
// by the fast Walsh-Hadamard transform in fp32: stages h = 1, 2, ..., b/2 in
// that order, pair (i, i+h) with (i & h) == 0 -> (v_i + v_{i+h}, v_i - v_{i+h}),
// then every entry times fp32(1/sqrt(b)).  The stage order fixes every
// rounding, so the result does not depend on how threads share the pairs.
//   requant_kernel      a3/a4: Eq. 11's Q(C_qkv), per token (int8) or per
//                       128-channel group (int4), written token-major and/or
//                       straight into the latent cache.
//   append_kernel       a4: latent rows -> cache slots.
//   up_quant_kernel     offline per-output-channel RTN of an up-projection
//                       (Eq. 11's Q(W^u)), int8 or int4.
#include <algorithm>
#include <cmath>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

// ---------------------------------------------------------------------------
// a1: one CTA per token row.  The row is staged in shared memory as fp32
// (bf16 -> fp32 is exact), reduced to its absmax, then quantized.
// ---------------------------------------------------------------------------
constexpr int kXqThreads = 256;

// Fast Walsh-Hadamard transform of every length-b block of v[0 .. n) in
// shared memory (all threads of the CTA; b a power of two dividing n), then
// v *= scale.  Ends with the CTA synchronized.
__device__ __forceinline__ void fwht_smem(float *v, int n, int b, float scale) {
    __syncthreads();
    for (int h = 1; h < b; h <<= 1) {
        for (int p = threadIdx.x; p < n / 2; p += blockDim.x) {
            const int i = (p / h) * 2 * h + (p % h);          // (i & h) == 0; i + h stays in i's block
            const float a = v[i], c = v[i + h];
            v[i] = __fadd_rn(a, c);
            v[i + h] = __fsub_rn(a, c);
        }
        __syncthreads();
    }
    for (int i = threadIdx.x; i < n; i += blockDim.x) v[i] = __fmul_rn(v[i], scale);
    __syncthreads();
}

__global__ void __launch_bounds__(kXqThreads)
xquant_kernel(const uint16_t *__restrict__ X, int d, float clip, int rot, float rot_scale, int qmax,
              int8_t *__restrict__ xq, uint16_t *__restrict__ xq_bf16, uint8_t *__restrict__ xq_f8,
              float *__restrict__ xs) {
    extern __shared__ float row[];
    __shared__ float red[kXqThreads / 32];
    const int64_t t = blockIdx.x;
    const uint16_t *x = X + t * d;
    pdl_trigger();
    pdl_wait();
    float m = 0.0f;
    // with a rotation of 8 or more channels per block, the stages h = 1, 2, 4
    // run on the 8 values a thread loads (8 consecutive channels, 8-aligned)
    const bool pre = rot >= 8;
    for (int i = threadIdx.x * 8; i < d; i += kXqThreads * 8) {
        float f[8];
        unpack8_bf16(*reinterpret_cast<const uint4 *>(x + i), f);
        if (pre) fwht8_regs(f);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            row[i + e] = f[e];
            m = fmaxf(m, fabsf(f[e]));
        }
    }
    if (rot) {                                           // x H1^T, then the absmax of the rotated row
        __syncthreads();
        fwht_smem_rounds(row, d, rot, pre ? 8 : 1);
        m = 0.0f;
        for (int i = threadIdx.x; i < d; i += kXqThreads) {
            const float v = __fmul_rn(row[i], rot_scale);
            row[i] = v;
            m = fmaxf(m, fabsf(v));
        }
    }
    m = block_max<kXqThreads>(m, red);
    const float s = quant_scale(m, clip, float(qmax)), inv = quant_inv_scale(s);
    for (int i = threadIdx.x * 8; i < d; i += kXqThreads * 8) {
        uint32_t packed[2] = {0u, 0u}, f8w[2] = {0u, 0u};
        uint32_t bfw[4];
#pragma unroll
        for (int e = 0; e < 8; e += 2) {
            const int c0 = quant_code_fast(row[i + e], s, inv, qmax);
            const int c1 = quant_code_fast(row[i + e + 1], s, inv, qmax);
            packed[e >> 2] |= (uint32_t(c0 & 0xff) << ((e & 3) * 8)) |
                              (uint32_t(c1 & 0xff) << (((e & 3) + 1) * 8));
            f8w[e >> 2] |= (uint32_t(int_to_e4m3(c0)) << ((e & 3) * 8)) |
                           (uint32_t(int_to_e4m3(c1)) << (((e & 3) + 1) * 8));
            bfw[e >> 1] = uint32_t(int_to_bf16_bits(c0)) | (uint32_t(int_to_bf16_bits(c1)) << 16);
        }
        if (xq) *reinterpret_cast<uint2 *>(xq + t * d + i) = make_uint2(packed[0], packed[1]);
        if (xq_bf16)
            *reinterpret_cast<uint4 *>(xq_bf16 + t * d + i) = make_uint4(bfw[0], bfw[1], bfw[2], bfw[3]);
        if (xq_f8) *reinterpret_cast<uint2 *>(xq_f8 + t * d + i) = make_uint2(f8w[0], f8w[1]);
    }
    if (threadIdx.x == 0 && xs) xs[t] = s;
}

// a1 without a rotation, for rows of up to kXrMaxD channels: 128 threads per
// row, every 16-byte load of the row issued at once and the row kept in
// registers (no staging through shared memory), so a row needs one round trip
// to memory; at 70 registers per thread seven CTAs share an SM (xquant_kernel:
// 61 registers x 256 threads, four rows, two or three dependent loads per
// thread).  The codes are those of xquant_kernel (the same absmax, scale and
// quantizer).
constexpr int kXrThreads = 128;
constexpr int kXrLoads = 6;                              // 16-byte loads per thread
constexpr int kXrMaxD = kXrThreads * kXrLoads * 8;       // 6144 channels

__global__ void __launch_bounds__(kXrThreads, 7)
xquant_rows_kernel(const uint16_t *__restrict__ X, int64_t T, int d, float clip, int qmax, int8_t *__restrict__ xq,
                   uint16_t *__restrict__ xq_bf16, uint8_t *__restrict__ xq_f8, float *__restrict__ xs) {
    __shared__ float red[2][kXrThreads / 32];
    pdl_trigger();
    pdl_wait();
    for (int64_t t = blockIdx.x, n = 0; t < T; t += gridDim.x, ++n) {   // rows of this CTA
        const uint16_t *x = X + t * d;
        uint4 v[kXrLoads];
#pragma unroll
        for (int k = 0; k < kXrLoads; ++k) {
            const int i = (k * kXrThreads + int(threadIdx.x)) * 8;
            v[k] = i < d ? *reinterpret_cast<const uint4 *>(x + i) : make_uint4(0u, 0u, 0u, 0u);
        }
        float m = 0.0f;
#pragma unroll
        for (int k = 0; k < kXrLoads; ++k) {
            float f[8];
            unpack8_bf16(v[k], f);
#pragma unroll
            for (int e = 0; e < 8; ++e) m = fmaxf(m, fabsf(f[e]));
        }
        m = block_max<kXrThreads>(m, red[n & 1]);      // alternate buffers: no barrier between rows
        const float s = quant_scale(m, clip, float(qmax)), inv = quant_inv_scale(s);
#pragma unroll
        for (int k = 0; k < kXrLoads; ++k) {
            const int i = (k * kXrThreads + int(threadIdx.x)) * 8;
            if (i >= d) break;
            float f[8];
            unpack8_bf16(v[k], f);
            int c[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) c[e] = quant_code_fast(f[e], s, inv, qmax);
            if (xq_bf16) {
                uint32_t w[4];
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    w[e] = uint32_t(int_to_bf16_bits(c[2 * e])) | (uint32_t(int_to_bf16_bits(c[2 * e + 1])) << 16);
                *reinterpret_cast<uint4 *>(xq_bf16 + t * d + i) = make_uint4(w[0], w[1], w[2], w[3]);
            }
            if (xq) {
                uint32_t w[2] = {0u, 0u};
#pragma unroll
                for (int e = 0; e < 8; ++e) w[e >> 2] |= uint32_t(c[e] & 0xff) << ((e & 3) * 8);
                *reinterpret_cast<uint2 *>(xq + t * d + i) = make_uint2(w[0], w[1]);
            }
            if (xq_f8) {
                uint32_t w[2] = {0u, 0u};
#pragma unroll
                for (int e = 0; e < 8; ++e) w[e >> 2] |= uint32_t(int_to_e4m3(c[e])) << ((e & 3) * 8);
                *reinterpret_cast<uint2 *>(xq_f8 + t * d + i) = make_uint2(w[0], w[1]);
            }
        }
        if (threadIdx.x == 0 && xs) xs[t] = s;
    }
}

cudaError_t launch_xquant(const uint16_t *X, int64_t T, int d, float clip, int8_t *xq,
                          uint16_t *xq_bf16, float *xs, cudaStream_t s, int rot, int qmax, uint8_t *xq_f8) {
    if (T == 0) return cudaSuccess;
    if (!rot && d <= kXrMaxD && d % 8 == 0) {
        // one CTA per row up to the rows that are resident at once (seven per SM); beyond, each CTA walks
        // rows with a stride of the grid (no CTA launches per row)
        int dev = 0, sms = 148;
        if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        const int64_t grid = std::min<int64_t>(T, int64_t(sms) * 7);
        cudaError_t e = launch_pdl(xquant_rows_kernel, dim3(unsigned(grid)), dim3(kXrThreads), 0, s, X, T, d, clip,
                                   qmax, xq, xq_bf16, xq_f8, xs);
        prof_mark(s, "xquant");
        return e;
    }
    const size_t smem = size_t(d) * sizeof(float);
    if (smem > 48 * 1024) {
        cudaError_t e = ensure_smem(xquant_kernel, smem);
        if (e != cudaSuccess) return e;
    }
    const float rot_scale = rot ? float(1.0 / std::sqrt(double(rot))) : 1.0f;
    cudaError_t e = launch_pdl(xquant_kernel, dim3(unsigned(T)), dim3(kXqThreads), smem, s, X, d, clip, rot,
                               rot_scale, qmax, xq, xq_bf16, xq_f8, xs);
    prof_mark(s, "xquant");
    return e;
}

// ---------------------------------------------------------------------------
// Offline: W_d [d, r] fp32 row-major -> per-column codes [r, d] int8 (+bf16).
// CTA = 32 columns x 8 row lanes; coalesced reads along a row of W_d.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
weight_quant_kernel(const float *__restrict__ W, int d, int r, float clip, int qmax, int8_t *__restrict__ codes,
                    uint16_t *__restrict__ codes_bf16, uint8_t *__restrict__ codes_f8, float *__restrict__ scale) {
    __shared__ float red[8][33];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int j = blockIdx.x * 32 + tx;
    float m = 0.0f;
    if (j < r)
        for (int k = ty; k < d; k += 8) m = fmaxf(m, fabsf(W[size_t(k) * r + j]));
    red[ty][tx] = m;
    __syncthreads();
    if (ty == 0) {
        for (int i = 1; i < 8; ++i) m = fmaxf(m, red[i][tx]);
        red[0][tx] = quant_scale(m, clip, float(qmax));
    }
    __syncthreads();
    const float s = red[0][tx];
    if (j >= r) return;
    if (ty == 0) scale[j] = s;
    for (int k = ty; k < d; k += 8) {
        const int c = quant_code(W[size_t(k) * r + j], s, qmax);
        codes[size_t(j) * d + k] = int8_t(c);
        if (codes_bf16) codes_bf16[size_t(j) * d + k] = int_to_bf16_bits(c);
        if (codes_f8) codes_f8[size_t(j) * d + k] = int_to_e4m3(c);
    }
    // The projection kernels copy W_d's codes before they wait on their
    // producer grid: a dependent launch may begin only once the codes are
    // visible device-wide.
    __threadfence();
    pdl_trigger();
}

// Offline, rotated: kWqrCols columns of W_d per CTA, staged column-major in
// shared memory, transformed by H1 down each column, then quantized per
// column like weight_quant_kernel.
constexpr int kWqrCols = 4;

__global__ void __launch_bounds__(256)
weight_quant_rot_kernel(const float *__restrict__ W, int d, int r, float clip, int rot, float rot_scale, int qmax,
                        int8_t *__restrict__ codes, uint16_t *__restrict__ codes_bf16, uint8_t *__restrict__ codes_f8,
                        float *__restrict__ scale) {
    extern __shared__ float col[];                        // [kWqrCols][d]
    __shared__ float red[kWqrCols][8];
    __shared__ float sc[kWqrCols];
    const int j0 = blockIdx.x * kWqrCols;
    const int nc = min(kWqrCols, r - j0);
    for (int i = threadIdx.x; i < kWqrCols * d; i += blockDim.x) {
        const int c = i % kWqrCols, k = i / kWqrCols;
        col[c * d + k] = c < nc ? W[size_t(k) * r + j0 + c] : 0.0f;
    }
    fwht_smem(col, kWqrCols * d, rot, rot_scale);         // blocks of rot never cross a column (rot divides d)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int c = 0; c < kWqrCols; ++c) {
        float m = 0.0f;
        for (int k = threadIdx.x; k < d; k += blockDim.x) m = fmaxf(m, fabsf(col[c * d + k]));
        m = warp_max(m);
        if (lane == 0) red[c][warp] = m;
    }
    __syncthreads();
    if (threadIdx.x < kWqrCols) {
        float m = 0.0f;
        for (int w = 0; w < 8; ++w) m = fmaxf(m, red[threadIdx.x][w]);
        sc[threadIdx.x] = quant_scale(m, clip, float(qmax));
    }
    __syncthreads();
    for (int c = 0; c < nc; ++c) {
        const float s = sc[c];
        if (threadIdx.x == 0) scale[j0 + c] = s;
        for (int k = threadIdx.x; k < d; k += blockDim.x) {
            const int q = quant_code(col[c * d + k], s, qmax);
            codes[size_t(j0 + c) * d + k] = int8_t(q);
            if (codes_bf16) codes_bf16[size_t(j0 + c) * d + k] = int_to_bf16_bits(q);
            if (codes_f8) codes_f8[size_t(j0 + c) * d + k] = int_to_e4m3(q);
        }
    }
    __threadfence();                                      // see weight_quant_kernel
    pdl_trigger();
}

cudaError_t launch_quantize_weight(const float *W, int d, int r, float clip, int8_t *codes,
                                   uint16_t *codes_bf16, float *scale, cudaStream_t s, int rot, int qmax,
                                   uint8_t *codes_f8) {
    if (rot) {
        const size_t smem = size_t(kWqrCols) * d * sizeof(float);
        cudaError_t e = ensure_smem(weight_quant_rot_kernel, smem);
        if (e != cudaSuccess) return e;
        weight_quant_rot_kernel<<<dim3((r + kWqrCols - 1) / kWqrCols), 256, smem, s>>>(
            W, d, r, clip, rot, float(1.0 / std::sqrt(double(rot))), qmax, codes, codes_bf16, codes_f8, scale);
    } else {
        weight_quant_kernel<<<dim3((r + 31) / 32), 256, 0, s>>>(W, d, r, clip, qmax, codes, codes_bf16, codes_f8,
                                                                 scale);
    }
    prof_mark(s, "weight_quant");
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// a3/a4: requantize one latent row per CTA (requant_row_cta, common.cuh).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kRqThreads)
requant_kernel(const float *c_hat, int r, int bits, float clip,
               void *__restrict__ lat_codes, void *__restrict__ lat_scales, CacheView dst,
               const int32_t *__restrict__ dst_seq, const int32_t *__restrict__ dst_pos,
               int *err) {
    __shared__ float red[kRqThreads / 32];
    pdl_trigger();
    pdl_wait();
    requant_row_cta(c_hat, blockIdx.x, r, bits, clip, lat_codes, lat_scales, dst, dst_seq, dst_pos, err, red);
}

cudaError_t launch_requant(const float *c_hat, int64_t T, int r, int bits, float clip, void *lat_codes,
                           void *lat_scales, const CacheView *dst, const int32_t *dst_seq,
                           const int32_t *dst_pos, int *err, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    CacheView d{};
    if (dst) d = *dst;
    cudaError_t e = launch_pdl(requant_kernel, dim3(unsigned(T)), dim3(kRqThreads), 0, s, c_hat, r, bits, clip,
                               lat_codes, lat_scales, d, dst_seq, dst_pos, err);
    prof_mark(s, "requant");
    return e;
}

// The rows of a decode step: row b of c_hat is the new token of sequence b,
// stored at position seq_len[b] - 1 of the cache sequence behind b (an
// invalid slot is skipped and flagged).
__global__ void __launch_bounds__(kRqThreads)
requant_len_kernel(const float *c_hat, int r, int bits, float clip, CacheView dst,
                   const int32_t *__restrict__ seq_len, int *err) {
    __shared__ float red[kRqThreads / 32];
    __shared__ int32_t seq_s, pos_s;
    pdl_trigger();
    pdl_wait();
    if (threadIdx.x == 0) {
        const int b = int(blockIdx.x);
        seq_s = view_seq(dst, b);
        pos_s = seq_s < 0 ? -1 : seq_len[b] - 1;
    }
    __syncthreads();
    requant_row_cta(c_hat + size_t(blockIdx.x) * r, 0, r, bits, clip, nullptr, nullptr, dst, &seq_s, &pos_s, err, red);
}

cudaError_t launch_requant_len(const float *c_hat, int B, int r, int bits, float clip, const CacheView &dst,
                               const int32_t *seq_len, int *err, cudaStream_t s) {
    if (B <= 0) return cudaSuccess;
    cudaError_t e = launch_pdl(requant_len_kernel, dim3(unsigned(B)), dim3(kRqThreads), 0, s, c_hat, r, bits, clip,
                               dst, seq_len, err);
    prof_mark(s, "requant");
    return e;
}

// ---------------------------------------------------------------------------
// a2/a3/a4 after a split-K projection GEMM: one CTA per token row adds the
// splits' int32 partial sums in split order (exact: |acc| < 2^31), forms
// c_hat = (fp32(acc) s_x) s_w exactly as the GEMM epilogue does, and
// requantizes and stores the row from registers.  The partials and s_x are
// written by the grids this one waits on, so they are not read through the
// read-only path (no __restrict__): the loads stay behind the wait.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kRqThreads)
split_requant_kernel(const int32_t *part, int splits, int64_t T, int r, const float *xs,
                     const float *__restrict__ ws, int32_t *__restrict__ acc_out, int bits, float clip,
                     void *__restrict__ lat_codes, void *__restrict__ lat_scales, CacheView dst,
                     const int32_t *__restrict__ dst_seq, const int32_t *__restrict__ dst_pos, int *err) {
    __shared__ float red[kRqThreads / 32];
    pdl_trigger();
    pdl_wait();
    const int64_t t = blockIdx.x;
    const int nq = r / 4;
    const float sx = xs[t];
    int4 p4[kRqMaxQuads][kMaxSplitK];                 // every partial of the thread's quads, loads issued first
#pragma unroll
    for (int k = 0; k < kRqMaxQuads; ++k) {
        const int qi = int(threadIdx.x) + k * kRqThreads;
#pragma unroll
        for (int z = 0; z < kMaxSplitK; ++z)
            p4[k][z] = qi < nq && z < splits
                           ? reinterpret_cast<const int4 *>(part + (size_t(z) * size_t(T) + size_t(t)) * r)[qi]
                           : make_int4(0, 0, 0, 0);
    }
    float4 v[kRqMaxQuads];
#pragma unroll
    for (int k = 0; k < kRqMaxQuads; ++k) {
        const int qi = int(threadIdx.x) + k * kRqThreads;
        v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (qi < nq) {
            int4 a = p4[k][0];
#pragma unroll
            for (int z = 1; z < kMaxSplitK; ++z) {       // in split order; absent splits are zeros
                a.x += p4[k][z].x;
                a.y += p4[k][z].y;
                a.z += p4[k][z].z;
                a.w += p4[k][z].w;
            }
            if (acc_out) reinterpret_cast<int4 *>(acc_out + size_t(t) * r)[qi] = a;
            const float4 w = reinterpret_cast<const float4 *>(ws)[qi];
            v[k] = make_float4(__fmul_rn(__fmul_rn(__int2float_rn(a.x), sx), w.x),
                               __fmul_rn(__fmul_rn(__int2float_rn(a.y), sx), w.y),
                               __fmul_rn(__fmul_rn(__int2float_rn(a.z), sx), w.z),
                               __fmul_rn(__fmul_rn(__int2float_rn(a.w), sx), w.w));
        }
    }
    requant_row_values(v, t, r, bits, clip, lat_codes, lat_scales, dst, dst_seq, dst_pos, err, red);
}

cudaError_t launch_split_requant(const int32_t *part, int splits, int64_t T, int r, const float *xs, const float *ws,
                                 int32_t *acc_out, int bits, float clip, void *lat_codes, void *lat_scales,
                                 const CacheView *dst, const int32_t *dst_seq, const int32_t *dst_pos, int *err,
                                 cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    CacheView d{};
    if (dst) d = *dst;
    cudaError_t e = launch_pdl(split_requant_kernel, dim3(unsigned(T)), dim3(kRqThreads), 0, s, part, splits, T, r, xs,
                               ws, acc_out, bits, clip, lat_codes, lat_scales, d, dst_seq, dst_pos, err);
    prof_mark(s, "requant");
    return e;
}

// ---------------------------------------------------------------------------
// a4: copy rows into the cache.  One warp per row, 16-byte vectors.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
append_kernel(CacheView c, const int32_t *__restrict__ seq, const int32_t *__restrict__ pos, int64_t n,
              const uint8_t *__restrict__ codes, const uint8_t *__restrict__ scales, int *err) {
    const int64_t i = int64_t(blockIdx.x) * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    pdl_trigger();
    pdl_wait();
    if (i >= n) return;
    const int b = seq[i], p = pos[i];
    if (b < 0 || b >= c.B || p < 0 || p >= c.Tmax) {
        if (lane == 0) flag_error(err, kErrRange);
        return;
    }
    const size_t slot = size_t(b) * c.Tmax + p;
    const int row_bytes = c.bits == 8 ? c.r : c.r / 2;
    const int scale_bytes = c.bits == 8 ? 4 : 2 * (c.r / 128);
    const uint4 *src = reinterpret_cast<const uint4 *>(codes + i * row_bytes);
    uint4 *dstc = reinterpret_cast<uint4 *>(static_cast<uint8_t *>(c.codes) + slot * row_bytes);
    for (int k = lane; k < row_bytes / 16; k += 32) dstc[k] = src[k];
    uint8_t *dsts = static_cast<uint8_t *>(c.scales) + slot * scale_bytes;
    for (int k = lane; k < scale_bytes; k += 32) dsts[k] = scales[i * scale_bytes + k];
}

cudaError_t launch_append(const CacheView &c, const int32_t *seq, const int32_t *pos, int64_t n,
                          const void *lat_codes, const void *lat_scales, int *err, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    cudaError_t e = launch_pdl(append_kernel, dim3(unsigned((n + 7) / 8)), dim3(256), 0, s, c, seq, pos, n,
                               static_cast<const uint8_t *>(lat_codes), static_cast<const uint8_t *>(lat_scales), err);
    prof_mark(s, "append");
    return e;
}

// ---------------------------------------------------------------------------
// Offline Q(W^u) of Eq. 11 (H2 = I), the weight quantizer of the Sec. 4
// setup: per output channel (column c of U [r, d], bf16) symmetric RTN to
// `bits` (8: int8 codes [r, d]; 4: packed int4 [r, d/2], column 2i in the low
// nibble) with an fp32 scale per column.  CTA = 32 columns (lane) x 8 row
// groups (warp).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
up_quant_kernel(const uint16_t *__restrict__ U, int r, int d, int bits, float clip, uint8_t *__restrict__ codes,
                float *__restrict__ scale) {
    __shared__ float red[8][33];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int c = blockIdx.x * 32 + tx;        // d % 32 == 0: every lane has a column
    const int qm = bits == 8 ? 127 : 7;
    float m = 0.0f;
    for (int j = ty; j < r; j += 8) m = fmaxf(m, fabsf(bf16_to_f32(U[size_t(j) * d + c])));
    red[ty][tx] = m;
    __syncthreads();
    if (ty == 0) {
        for (int i = 1; i < 8; ++i) m = fmaxf(m, red[i][tx]);
        red[0][tx] = quant_scale(m, clip, float(qm));
        scale[c] = red[0][tx];
    }
    __syncthreads();
    const float s = red[0][tx];
    for (int j = ty; j < r; j += 8) {
        const int code = quant_code(bf16_to_f32(U[size_t(j) * d + c]), s, qm);
        if (bits == 8) {
            codes[size_t(j) * d + c] = uint8_t(int8_t(code));
        } else {
            const int hi = __shfl_down_sync(0xffffffffu, code, 1);
            if ((tx & 1) == 0) codes[(size_t(j) * d + c) / 2] = uint8_t((code & 0xF) | ((hi & 0xF) << 4));
        }
    }
}

cudaError_t launch_quantize_up(const uint16_t *U, int r, int d, int bits, float clip, void *codes, float *scale,
                               cudaStream_t s) {
    up_quant_kernel<<<dim3(unsigned(d / 32)), dim3(256), 0, s>>>(U, r, d, bits, clip, static_cast<uint8_t *>(codes),
                                                                scale);
    prof_mark(s, "up_quant");
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Failure-detection self-test: one thread waits on an mbarrier that nothing
// arrives on until `limit_ns` of globaltimer have passed, then sets the
// timeout bit of the device error word and returns, as every bounded wait of
// the library does when it expires.
// ---------------------------------------------------------------------------
__global__ void selftest_wait_kernel(unsigned long long limit_ns, int *err) {
    __shared__ __align__(8) uint64_t bar;
    mbar_init(&bar, 1);
    mbar_init_fence();
    unsigned long long t0, t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
    for (;;) {
        if (mbar_try_wait(&bar, 0)) return;                 // never: no arrival is ever made
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
        if (t - t0 > limit_ns) {
            flag_error(err, kErrTimeout);
            return;
        }
    }
}

cudaError_t launch_selftest_wait(unsigned long long limit_ns, int *err, cudaStream_t s) {
    selftest_wait_kernel<<<1, 1, 0, s>>>(limit_ns, err);
    prof_mark(s, "selftest_wait");
    return cudaGetLastError();
}

}  // namespace qsvd
