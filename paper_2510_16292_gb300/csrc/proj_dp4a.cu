// Exact int8 x int8 -> int32 down-projection on the CUDA cores (dp4a), with
// the dequantization of Eq. 12's product fused behind it:
//   acc[t, j]   = sum_k xq[t, k] * w[j, k]          (exact: |acc| < 2^31)
//   c_hat[t, j] = fp32(fp32(fp32(acc) * s_x[t]) * s_w[j])
// proj_dp4a_kernel is the general CUDA-core path; proj_small_kernel is the
// decode path: for T < 4 tokens it quantizes X itself, streams its 8 rows of
// W_d codes into shared memory with bulk copies, and the last CTA to finish
// requantizes the latent rows and stores them (a1-a4 in one launch); for up to
// kPsMaxSplitTok tokens it takes codes quantized by xquant_kernel, one
// 16-token block per grid row, and leaves the requantization to requant_kernel.
#include <algorithm>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

constexpr int kPjWarps = 8;       // output channels per CTA (one per warp)
constexpr int kPjTokens = 16;     // tokens per CTA (grid.y tiles T)

__global__ void __launch_bounds__(kPjWarps * 32)
proj_dp4a_kernel(const int8_t *xq, int64_t T, int d, const int8_t *__restrict__ w,
                 const float *__restrict__ ws, const float *xs, int r,
                 float *__restrict__ c_hat, int32_t *__restrict__ acc_out) {
    const int lane = threadIdx.x & 31;
    const int j = blockIdx.x * kPjWarps + (threadIdx.x >> 5);
    pdl_trigger();
    if (blockIdx.y == 0) prefetch_share_l2(w, size_t(r) * d, blockIdx.x, gridDim.x);
    pdl_wait();
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

// ---------------------------------------------------------------------------
// Decode path.  CTA = 8 output channels (one warp each) x one block of up to
// kPsMaxTok tokens (grid row y: tokens [16 y, 16 y + 16)); without xq_in every
// CTA quantizes its token rows itself (redundantly, they are tiny).
// ---------------------------------------------------------------------------
constexpr int kPsWarps = 8;
constexpr int kPsMaxD = 6144;          // d <= 6144: 24 x 16-byte vectors per lane
constexpr int kPsWarpTok = 4;          // from this many tokens on: tensor-core dot products, a warp per latent row

__global__ void __launch_bounds__(kPsWarps * 32, 2)
proj_small_kernel(const uint16_t *__restrict__ X, int T, int d, float act_clip, const int8_t *__restrict__ w,
                  const float *__restrict__ ws, int r, int lat_bits, float lat_clip, float *__restrict__ c_hat,
                  int *__restrict__ counter, int8_t *__restrict__ xq_out, float *__restrict__ xs_out,
                  int32_t *__restrict__ acc_out, void *__restrict__ lat_codes, void *__restrict__ lat_scales,
                  CacheView dst, const int32_t *__restrict__ dst_seq, const int32_t *__restrict__ dst_pos,
                  int *err, const int8_t *xq_in, const float *xs_in, int tail, int act_qmax) {
    extern __shared__ __align__(16) uint8_t smem[];
    __shared__ __align__(8) uint64_t bar, bar_x;
    {   // this CTA's token block
        const int tb = blockIdx.y * kPsMaxTok;
        T = min(T - tb, kPsMaxTok);
        X += size_t(tb) * d;
        c_hat += size_t(tb) * r;
        if (xq_in) xq_in += size_t(tb) * d;
        if (xs_in) xs_in += tb;
        if (xq_out) xq_out += size_t(tb) * d;
        if (xs_out) xs_out += tb;
        if (acc_out) acc_out += size_t(tb) * r;
    }
    __shared__ float xs_s[kPsMaxTok];
    __shared__ float red[kPsWarps];
    __shared__ float red4[kPsWarps][4];
    __shared__ int last;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j0 = blockIdx.x * kPsWarps;
    const int rows = min(kPsWarps, r - j0);
    const int dp = d + 16;                                           // padded row: conflict-free fragments
    int8_t *w_s = reinterpret_cast<int8_t *>(smem);                  // [kPsWarps][dp]
    int8_t *xq_s = reinterpret_cast<int8_t *>(smem) + kPsWarps * dp; // [T][dp]
    pdl_trigger();
    if (blockIdx.y == 0) prefetch_share_l2(w, size_t(r) * d, blockIdx.x, gridDim.x);
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_init(&bar_x, 1);
        mbar_init_fence();
    }
    __syncthreads();
    if (threadIdx.x == 0) {     // W_d codes: no kernel's output, copied before the wait on the producer grid
        mbar_arrive_expect_tx(&bar, uint32_t(rows) * d);
        for (int i = 0; i < rows; ++i) bulk_g2s(w_s + size_t(i) * dp, w + size_t(j0 + i) * d, uint32_t(d), &bar);
    } else if (threadIdx.x <= T && !xq_in) {
        // the token rows into L2 while the producer grid finishes (L2 is the point of
        // coherence, so a row written meanwhile is never seen stale: the reads come after the wait)
        prefetch_l2_bulk(X + size_t(threadIdx.x - 1) * d, uint32_t(d) * 2);
    } else if (tail && blockIdx.x == 0 && dst.codes && threadIdx.x >= 32 && threadIdx.x < 32 + T) {
        // the append indices the last CTA reads (inputs, same argument)
        asm volatile("prefetch.global.L2 [%0];" ::"l"(dst_seq + (threadIdx.x - 32)) : "memory");
        asm volatile("prefetch.global.L2 [%0];" ::"l"(dst_pos + (threadIdx.x - 32)) : "memory");
    }
    pdl_wait();
    // a1: per-token int8 quantization.  Codes quantized by the previous kernel
    // (xq_in): bulk copies into the padded rows.  Otherwise the whole CTA
    // quantizes, up to kQg tokens at a time: one round of loads, the per-token
    // maxima reduced together.
    constexpr int kQg = 4, kVt = kPsMaxD / 2048;    // tokens per round, 16-byte vectors per thread per token
    if (xq_in) {
        if (threadIdx.x == 0) {
            mbar_arrive_expect_tx(&bar_x, uint32_t(T) * d);
            for (int t = 0; t < T; ++t) bulk_g2s(xq_s + size_t(t) * dp, xq_in + size_t(t) * d, uint32_t(d), &bar_x);
        }
        if (threadIdx.x < T) xs_s[threadIdx.x] = xs_in[threadIdx.x];
    }
    for (int t0 = 0; t0 < T && !xq_in; t0 += kQg) {
        const int ng = min(kQg, T - t0);
        uint4 xv[kQg][kVt];
        float m[kQg];
#pragma unroll
        for (int g = 0; g < kQg; ++g) {
            m[g] = 0.0f;
#pragma unroll
            for (int k = 0; k < kVt; ++k) {
                const int col = (k * 256 + threadIdx.x) * 8;
                xv[g][k] = (g < ng && col < d) ? *reinterpret_cast<const uint4 *>(X + size_t(t0 + g) * d + col)
                                               : make_uint4(0u, 0u, 0u, 0u);
            }
        }
#pragma unroll
        for (int g = 0; g < kQg; ++g) {
#pragma unroll
            for (int k = 0; k < kVt; ++k) {
                float f[8];
                unpack8_bf16(xv[g][k], f);
#pragma unroll
                for (int e = 0; e < 8; ++e) m[g] = fmaxf(m[g], fabsf(f[e]));
            }
            m[g] = warp_max(m[g]);
        }
        if (lane == 0)
#pragma unroll
            for (int g = 0; g < kQg; ++g) red4[warp][g] = m[g];
        __syncthreads();
        if (threadIdx.x < ng) {
            float mm = red4[0][threadIdx.x];
#pragma unroll
            for (int w = 1; w < kPsWarps; ++w) mm = fmaxf(mm, red4[w][threadIdx.x]);
            const float s = quant_scale(mm, act_clip, float(act_qmax));
            xs_s[t0 + threadIdx.x] = s;
            if (xs_out && blockIdx.x == 0) xs_out[t0 + threadIdx.x] = s;
        }
        __syncthreads();
#pragma unroll
        for (int g = 0; g < kQg; ++g) {
            if (g >= ng) break;
            const float s = xs_s[t0 + g], inv = quant_inv_scale(s);
#pragma unroll
            for (int k = 0; k < kVt; ++k) {
                const int col = (k * 256 + threadIdx.x) * 8;
                if (col >= d) break;
                float f[8];
                unpack8_bf16(xv[g][k], f);
                uint32_t lo = 0, hi = 0;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    lo |= uint32_t(quant_code_fast(f[e], s, inv, act_qmax) & 0xff) << (8 * e);
                    hi |= uint32_t(quant_code_fast(f[e + 4], s, inv, act_qmax) & 0xff) << (8 * e);
                }
                *reinterpret_cast<uint2 *>(xq_s + size_t(t0 + g) * dp + col) = make_uint2(lo, hi);
                if (xq_out && blockIdx.x == 0)
                    *reinterpret_cast<uint2 *>(xq_out + size_t(t0 + g) * d + col) = make_uint2(lo, hi);
            }
        }
    }
    __syncthreads();
    mbar_wait(&bar, 0, err);
    if (xq_in) mbar_wait(&bar_x, 0, err);
    // a2 + first half of a3: exact int32 dot products, then the fp32 dequantization
    if (T >= kPsWarpTok) {
        // Tensor cores: the CTA's 16-token x 8-channel tile (m16n8k16, codes
        // exact in fp16), K split over the 8 warps.  A warp's partial sums stay
        // below d/8 * 127^2 < 2^24, so they are exact integers in fp32.
        const int g8 = lane >> 2, cq = lane & 3;
        const int kspan = d / kPsWarps, kb = warp * kspan;
        const bool live0 = g8 < T, live1 = g8 + 8 < T;
        const int8_t *xa0 = xq_s + size_t(live0 ? g8 : 0) * dp, *xa1 = xq_s + size_t(live1 ? g8 + 8 : 0) * dp;
        const int8_t *wb = w_s + size_t(g8 < rows ? g8 : 0) * dp;
        auto pair = [](const int8_t *p) {           // two int8 codes -> fp16 pair, exact
            const uint32_t u = uint32_t(*reinterpret_cast<const uint16_t *>(p)) ^ 0x8080u;
            const uint32_t a = __byte_perm(u, 0x64646464u, 0x5150);
            const __half2 h = __hsub2(*reinterpret_cast<const __half2 *>(&a), __half2half2(__ushort_as_half(0x6480)));
            return *reinterpret_cast<const uint32_t *>(&h);
        };
        float c0[4] = {0.f, 0.f, 0.f, 0.f}, c1[4] = {0.f, 0.f, 0.f, 0.f};
        for (int k0 = kb; k0 < kb + kspan; k0 += 32) {
#pragma unroll
            for (int u = 0; u < 2; ++u) {           // two independent accumulator chains
                const int k = k0 + 16 * u + 2 * cq;
                const uint32_t a0 = live0 ? pair(xa0 + k) : 0u, a1 = live1 ? pair(xa1 + k) : 0u;
                const uint32_t a2 = live0 ? pair(xa0 + k + 8) : 0u, a3 = live1 ? pair(xa1 + k + 8) : 0u;
                const uint32_t b0 = pair(wb + k), b1 = pair(wb + k + 8);
                float *cc = u ? c1 : c0;
                asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                             "{%0,%1,%2,%3};"
                             : "+f"(cc[0]), "+f"(cc[1]), "+f"(cc[2]), "+f"(cc[3])
                             : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
            }
        }
        // rows g8 / g8 + 8, channels 2cq / 2cq + 1; the warps' partials added as int32
        int *red_i = reinterpret_cast<int *>(xq_s);   // codes no longer needed: reuse [8 warps][16][8]
        __syncthreads();
        red_i[(warp * 16 + g8) * 8 + 2 * cq] = __float2int_rn(c0[0] + c1[0]);
        red_i[(warp * 16 + g8) * 8 + 2 * cq + 1] = __float2int_rn(c0[1] + c1[1]);
        red_i[(warp * 16 + g8 + 8) * 8 + 2 * cq] = __float2int_rn(c0[2] + c1[2]);
        red_i[(warp * 16 + g8 + 8) * 8 + 2 * cq + 1] = __float2int_rn(c0[3] + c1[3]);
        __syncthreads();
        if (threadIdx.x < 128) {
            const int t = threadIdx.x >> 3, jj = threadIdx.x & 7;
            if (t < T && jj < rows) {
                int acc = 0;
#pragma unroll
                for (int w = 0; w < kPsWarps; ++w) acc += red_i[(w * 16 + t) * 8 + jj];
                const int j = j0 + jj;
                c_hat[size_t(t) * r + j] = __fmul_rn(__fmul_rn(__int2float_rn(acc), xs_s[t]), ws[j]);
                if (acc_out) acc_out[size_t(t) * r + j] = acc;
            }
        }
    } else if (warp < rows) {
        const int j = j0 + warp;
        const int *wrow = reinterpret_cast<const int *>(w_s + size_t(warp) * dp);
        const float sw = ws[j];
        for (int t = 0; t < T; ++t) {
            const int *xrow = reinterpret_cast<const int *>(xq_s + size_t(t) * dp);
            int acc = 0;
#pragma unroll 8
            for (int i = lane; i < d / 4; i += 32) acc = __dp4a(wrow[i], xrow[i], acc);
            acc = warp_sum_int(acc);
            if (lane == 0) {
                c_hat[size_t(t) * r + j] = __fmul_rn(__fmul_rn(__int2float_rn(acc), xs_s[t]), sw);
                if (acc_out) acc_out[size_t(t) * r + j] = acc;
            }
        }
    }
    if (!tail || gridDim.y > 1) return;  // the rows are requantized by the next kernel
    // second half of a3 + a4: the last CTA requantizes every row of c_hat
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) last = atomicAdd(counter, 1) == int(gridDim.x) - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();
    if (T < kPsWarpTok) {
        static_assert(kRqThreads == kPsWarps * 32, "requant_row_cta expects one full CTA");
        for (int t = 0; t < T; ++t)
            requant_row_cta(c_hat, t, r, lat_bits, lat_clip, lat_codes, lat_scales, dst, dst_seq, dst_pos, err, red);
    } else {
        for (int t = warp; t < T; t += kPsWarps)     // one warp per latent row
            requant_row_warp(c_hat, t, r, lat_bits, lat_clip, lat_codes, lat_scales, dst, dst_seq, dst_pos, err);
    }
    if (threadIdx.x == 0) *counter = 0;
}

cudaError_t launch_proj_small(const uint16_t *X, int T, int d, float act_clip, const int8_t *wcodes,
                              const float *ws, int r, int lat_bits, float lat_clip, float *c_hat, int *counter,
                              int8_t *xq_out, float *xs_out, int32_t *acc_out, void *lat_codes, void *lat_scales,
                              const CacheView *dst, const int32_t *dst_seq, const int32_t *dst_pos, int *err,
                              cudaStream_t s, const int8_t *xq_in, const float *xs_in, bool tail, int act_qmax) {
    CacheView dv{};
    if (dst) dv = *dst;
    // padded rows; the tensor-core path reuses the code rows for an [8][16][8] int32 reduction
    const int tb = std::min(T, kPsMaxTok);                       // tokens per CTA
    const size_t smem = size_t(kPsWarps) * (d + 16) + std::max(size_t(tb) * (d + 16), size_t(kPsWarps) * 16 * 8 * 4);
    cudaError_t e = ensure_smem(proj_small_kernel, smem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(proj_small_kernel, dim3((r + kPsWarps - 1) / kPsWarps, (T + kPsMaxTok - 1) / kPsMaxTok),
                   dim3(kPsWarps * 32), smem, s, X, T, d,
                   act_clip, wcodes, ws, r, lat_bits, lat_clip, c_hat, counter, xq_out, xs_out, acc_out, lat_codes,
                   lat_scales, dv, dst_seq, dst_pos, err, xq_in, xs_in, int(tail), act_qmax);
    prof_mark(s, "proj_small");
    return e;
}

cudaError_t launch_proj_dp4a(const int8_t *xq, int64_t T, int d, const int8_t *wcodes, const float *ws,
                             const float *xs, int r, float *c_hat, int32_t *acc_out, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    dim3 grid((r + kPjWarps - 1) / kPjWarps, unsigned((T + kPjTokens - 1) / kPjTokens));
    cudaError_t e = launch_pdl(proj_dp4a_kernel, grid, dim3(kPjWarps * 32), 0, s, xq, T, d, wcodes, ws, xs, r,
                               c_hat, acc_out);
    prof_mark(s, "proj_dp4a");
    return e;
}

}  // namespace qsvd
