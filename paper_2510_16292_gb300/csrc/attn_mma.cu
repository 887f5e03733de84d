// Decode attention over the latent cache for small batch x length, and for
// shapes the tcgen05 kernel does not take (Eq. 5 with W^u_k absorbed into the
// query; W^u_v is applied by the combine kernel), on the warp-level
// tensor-core MMA (mma.sync m16n8k16, fp16 in, fp32 accumulate).  A CTA takes
// one sequence, 8 heads and a range of n_sub sub-tiles of TS tokens (16, 32
// or 64), walked one after another with a running softmax:
//
//   0. the fp16 query block Q~ [8 heads][r] (each head scaled by a power of
//      two so that its largest entry is just below 2^14) is built from q~.
//   per sub-tile:
//   1. the TS cache rows (int8 / packed int4, padded rows) and the scales go
//      to shared memory with 16-byte asynchronous copies.
//   2. scores S[t, h] = sum_ch C[t, ch] Q~[h, ch]: each warp takes a range of
//      16-channel steps, the warps' partial S are added in shared memory.
//      int8: the token scale multiplies the row; int4: code * group-scale is
//      accumulated group by group.
//   3. per head: the running maximum m and sum l are updated (o_lat is scaled
//      by 2^(m_old - m_new)), p = 2^(logit - m).
//   4. O^T[ch, h] += sum_t C[t, ch] P[t, h] (M = 16 channels per MMA, K =
//      tokens), the token / group scale folded into P; the accumulators of a
//      warp's channel blocks stay in registers across the sub-tiles.
//   5. the CTA's (m, l, o_lat) are written as one softmax partial.
//
// Within one score MMA the 16 channels (the reduction index) are used in the
// order {0,1,4,5,8,9,12,13, 2,3,6,7,10,11,14,15} on both operands (the sum
// does not depend on the order), so that a thread's operand fragment is one
// 32-bit (int8) or 16-bit (int4) shared-memory load.  Step 4 reloads the same
// fragments and transposes them in registers (movmatrix): its M rows are the
// channels in that order, which the final store undoes.
#include <cfloat>
#include <cuda_fp16.h>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

namespace am {

constexpr int kWarps = 16;
constexpr int kThreads = 32 * kWarps;
constexpr int kHG = 8;            // heads per CTA (one n-block)
constexpr int kMaxTS = 64;        // tokens per CTA
constexpr int kRowPad = 16;       // bytes of padding per cache row in shared memory
constexpr int kQPad = 8;          // fp16 of padding per query row

struct Params {
    CacheView c;
    const int32_t *seq_len;
    const float *qt;              // [B, H, r]
    const unsigned *qmax;         // [B, H] bits of max |q~|, or null: formed from q~ (r <= 2048)
    int H, TS, n_sub, n_split;     // sub-tile tokens, sub-tiles per split, splits per sequence
    float softmax_scale;
    float *pm, *pl, *po;          // [B, n_split, H] / [B, n_split, H, r]
    int *err;
};

__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t b0,
                                         uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
// Four int8 codes (element i in byte i) -> two fp16 pairs, exact.
__device__ __forceinline__ void i8x4_h2(uint32_t w, uint32_t &lo, uint32_t &hi) {
    const uint32_t u = w ^ 0x80808080u;
    const uint32_t a = __byte_perm(u, 0x64646464u, 0x5150);
    const uint32_t b = __byte_perm(u, 0x64646464u, 0x5352);
    const __half2 bias = __half2half2(__ushort_as_half(0x6480));      // 1152
    const __half2 ha = __hsub2(*reinterpret_cast<const __half2 *>(&a), bias);
    const __half2 hb = __hsub2(*reinterpret_cast<const __half2 *>(&b), bias);
    lo = *reinterpret_cast<const uint32_t *>(&ha);
    hi = *reinterpret_cast<const uint32_t *>(&hb);
}
// Byte k of w (two int4 codes, the even channel in the low nibble) -> their
// fp16 pair, exact: the nibbles xor 8 go into the mantissas of 1024 and of
// 1024 * 16, and one fused multiply-add maps both back to the codes.
__device__ __forceinline__ uint32_t i4pair_h2(uint32_t w, int k) {
    const uint32_t y = __byte_perm(w, 0u, uint32_t(k) | (4u << 4) | (uint32_t(k) << 8) | (4u << 12));
    const uint32_t z = (y & 0x00F0000Fu) ^ 0x64806408u;              // 1024 + (lo ^ 8), 1024 + 16 (hi ^ 8)
    const __half2 mul = __halves2half2(__ushort_as_half(0x3C00), __ushort_as_half(0x2C00));   // 1, 1/16
    const __half2 add = __halves2half2(__ushort_as_half(0xE408), __ushort_as_half(0xD480));   // -1032, -72
    const __half2 c = __hfma2(*reinterpret_cast<const __half2 *>(&z), mul, add);
    return *reinterpret_cast<const uint32_t *>(&c);
}
// Transpose of an 8 x 8 fp16 block held one pair per thread (thread t: row
// t/4, columns 2(t%4), 2(t%4)+1).
__device__ __forceinline__ uint32_t movm_t(uint32_t a) {
    uint32_t d;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
    return d;
}
// Score-operand fragment of cache row `row`, channel step k0: the fp16 pairs
// of channels (4cq, 4cq+1) and (4cq+2, 4cq+3), i.e. reduction indices
// (2cq, 2cq+1) and (2cq+8, 2cq+9) in the order above.
template <int BITS>
__device__ __forceinline__ void load_frag(const uint8_t *tile, int rstride, int row, int k0, int cq, uint32_t &lo,
                                          uint32_t &hi) {
    if (BITS == 8) {
        i8x4_h2(*reinterpret_cast<const uint32_t *>(tile + size_t(row) * rstride + k0 + 4 * cq), lo, hi);
    } else {
        const uint32_t w = *reinterpret_cast<const uint16_t *>(tile + size_t(row) * rstride + (k0 + 4 * cq) / 2);
        lo = i4pair_h2(w, 0);
        hi = i4pair_h2(w, 1);
    }
}

}  // namespace am

template <int BITS, int MB>
__global__ void __launch_bounds__(am::kThreads)
attn_mma_kernel(const am::Params p) {
    using namespace am;
    extern __shared__ __align__(16) uint8_t smem[];
    __shared__ float sred[kWarps][kMaxTS][kHG];     // per-warp partial scores
    __shared__ float tsc_s[kMaxTS];                 // int8 token scales
    __shared__ float qfac_s[kHG];
    __shared__ float m_s[kHG];
    __shared__ float alpha_s[kHG];                  // o_lat rescale of the current sub-tile
    __shared__ unsigned hmax_s[kHG];                // per-head max |q~| (bits) when p.qmax is null
    const CacheView &c = p.c;
    const int r = c.r, TS = p.TS, H = p.H;
    const int split = blockIdx.x, b = blockIdx.y, h0 = blockIdx.z * kHG;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, cq = lane & 3;
    const int row_bytes = BITS == 8 ? r : r / 2;
    const int rstride = row_bytes + kRowPad;                       // padded cache row
    const int qstride = r + kQPad;                                 // padded query row (fp16)
    uint8_t *tile = smem;                                          // [TS][rstride]
    __half *qs = reinterpret_cast<__half *>(smem + size_t(TS) * rstride);              // [kHG][qstride]
    __half *gsc = reinterpret_cast<__half *>(qs + size_t(kHG) * qstride);              // [TS][r/128] (int4)
    __half *ps = gsc + (BITS == 4 ? size_t(TS) * (r / 128) : 0);                       // [kHG][TS + 8] P
    const int pstride = TS + 8;
    // Below 5 sequences the combine kernel that follows launches only when this
    // grid exits: measured on GB300 (B = 1, whole decode steps), that is 0.4 us
    // faster per step than triggering it here, its CTAs no longer copying U_v
    // beside the attention's.  From 5 sequences on it is triggered at once.
    if (gridDim.y >= 5) pdl_trigger();
    // lengths and sequence map: call inputs, complete before this grid starts
    // (the query kernels let their dependents start only after their own wait)
    const int sq = view_seq(c, b);
    const int L = sq < 0 ? 0 : p.seq_len[b];
    const int t_split = split * TS * p.n_sub;
    if (L < 1 || L > c.Tmax || t_split >= L) return;               // invalid lengths are flagged by qproj_kernel
    const int n_sub = min(p.n_sub, (L - t_split + TS - 1) / TS);   // sub-tiles of this CTA
    if (threadIdx.x == 0) {
        // L2 prefetch of the split's cache rows while the producer grid finishes
        // (L2 is the point of coherence, so a row written meanwhile is never
        // seen stale: the shared-memory copies come after the wait)
        for (int sb = 0; sb < n_sub; ++sb) {
            const int t0 = t_split + sb * TS;
            prefetch_l2_bulk(static_cast<const uint8_t *>(c.codes) + (size_t(sq) * c.Tmax + t0) * row_bytes,
                             uint32_t(min(TS, L - t0)) * row_bytes);
        }
    }
    pdl_wait();

    // sub-tile `sb`: cache rows (zero beyond the length) by 16-byte asynchronous copies, and the scales
    auto load_tile = [&](int sb) {
        const int t_begin = t_split + sb * TS;
        const int n = min(TS, L - t_begin);
        const size_t slot0 = size_t(sq) * c.Tmax + t_begin;
        const int cpr = row_bytes / 16;                            // 16-byte chunks per row
        for (int i = threadIdx.x; i < TS * cpr; i += kThreads) {
            const int t = i / cpr, k = i - t * cpr;
            uint8_t *dst = tile + size_t(t) * rstride + k * 16;
            if (t < n) cp_async16(dst, static_cast<const uint8_t *>(c.codes) + (slot0 + t) * row_bytes + k * 16);
            else *reinterpret_cast<uint4 *>(dst) = make_uint4(0u, 0u, 0u, 0u);
        }
        if (BITS == 8) {
            if (threadIdx.x < TS)
                tsc_s[threadIdx.x] = threadIdx.x < n ? static_cast<const float *>(c.scales)[slot0 + threadIdx.x] : 0.0f;
        } else {
            for (int i = threadIdx.x; i < TS * (r / 128); i += kThreads) {
                const int t = i / (r / 128);
                gsc[i] = t < n ? static_cast<const __half *>(c.scales)[slot0 * (r / 128) + i] : __float2half(0.0f);
            }
        }
    };
    load_tile(0);                                                  // overlaps the query block below

    // ---- 0. query block: q~ loads first, the per-head scale applied once qmax is in
    {
        constexpr int kQL = 8;                                     // float4 per thread per pass (r <= 2048: one pass)
        const int nq4 = kHG * (r / 4);
        float4 v[kQL];
#pragma unroll
        for (int u = 0; u < kQL; ++u) {
            const int i = threadIdx.x + u * kThreads;
            const int hl = i / (r / 4), q4 = i - hl * (r / 4);
            v[u] = (i < nq4 && h0 + hl < H) ? reinterpret_cast<const float4 *>(p.qt + (size_t(b) * H + h0 + hl) * r)[q4]
                                           : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        if (!p.qmax) {
            // the per-head maxima from the loaded block itself (r <= 2048: one pass
            // holds every channel of the CTA's heads), as non-negative float bits
            if (threadIdx.x < kHG) hmax_s[threadIdx.x] = 0u;
            __syncthreads();
#pragma unroll
            for (int u = 0; u < kQL; ++u) {
                // a warp's 32 float4 belong to one head (r / 4 is a multiple of 32)
                const int i = threadIdx.x + u * kThreads;
                const float4 x = v[u];
                const float mx = warp_max(fmaxf(fmaxf(fabsf(x.x), fabsf(x.y)), fmaxf(fabsf(x.z), fabsf(x.w))));
                if (lane == 0 && i < nq4) atomicMax(&hmax_s[i / (r / 4)], __float_as_uint(mx));
            }
            __syncthreads();
        }
        if (threadIdx.x < kHG) {
            const int h = h0 + threadIdx.x;
            int e = 0;
            if (h < H) {
                const float m = __uint_as_float(p.qmax ? p.qmax[size_t(b) * H + h] : hmax_s[threadIdx.x]);
                if (m > 0.0f) frexpf(m, &e);
            }
            // scores -> logits in log2 units: undo the query scale, times softmax_scale * log2(e)
            qfac_s[threadIdx.x] = exp2f(float(e - 14)) * p.softmax_scale * 1.4426950408889634f;
            m_s[threadIdx.x] = exp2f(float(14 - e));               // the query scale
        }
        __syncthreads();
        auto store_q = [&](int i, const float4 &x) {
            const int hl = i / (r / 4), q4 = i - hl * (r / 4);
            const float sc = m_s[hl];
            const __half2 lo = __floats2half2_rn(x.x * sc, x.y * sc);
            const __half2 hi = __floats2half2_rn(x.z * sc, x.w * sc);
            *reinterpret_cast<uint2 *>(qs + size_t(hl) * qstride + 4 * q4) =
                make_uint2(*reinterpret_cast<const uint32_t *>(&lo), *reinterpret_cast<const uint32_t *>(&hi));
        };
#pragma unroll
        for (int u = 0; u < kQL; ++u) {
            const int i = threadIdx.x + u * kThreads;
            if (i < nq4) store_q(i, v[u]);
        }
        for (int i = threadIdx.x + kQL * kThreads; i < nq4; i += kThreads) {     // r > 2048
            const int hl = i / (r / 4), q4 = i - hl * (r / 4);
            const float4 x = h0 + hl < H ? reinterpret_cast<const float4 *>(p.qt + (size_t(b) * H + h0 + hl) * r)[q4]
                                         : make_float4(0.f, 0.f, 0.f, 0.f);
            store_q(i, x);
        }
    }

    const int MT = TS / 16, nks = r / 16;
    // running softmax state of head `warp` (warps < kHG), the same in every lane
    float m_run = -INFINITY, l_run = 0.0f;
    // o_lat^T accumulators: channel step mb = warp + kWarps j, fragment (reduction indices g, g+8; heads 2cq, 2cq+1)
    float o[MB][4];
#pragma unroll
    for (int j = 0; j < MB; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.0f;

    for (int sb = 0; sb < n_sub; ++sb) {
        const int t_begin = t_split + sb * TS;
        const int n = min(TS, L - t_begin);
        // ---- 1. cache rows and scales (sub-tile 0 was issued before the query block)
        if (sb > 0) {
            __syncthreads();                                       // the previous sub-tile's readers are done
            load_tile(sb);
        }
        cp_async_wait_all();
        __syncthreads();

        // ---- 2. scores: warp w takes 16-channel steps w, w+kWarps, ...; MT m-blocks of 16 tokens
        {
            float acc[kMaxTS / 16][4];
#pragma unroll
            for (int m = 0; m < kMaxTS / 16; ++m) acc[m][0] = acc[m][1] = acc[m][2] = acc[m][3] = 0.0f;
            float gacc[kMaxTS / 16][4];                    // int4: current group's sums; int8: second chain
#pragma unroll
            for (int m = 0; m < kMaxTS / 16; ++m) gacc[m][0] = gacc[m][1] = gacc[m][2] = gacc[m][3] = 0.0f;
            int cur_grp = -1;
            for (int ks = warp; ks < nks; ks += kWarps) {
                const int k0 = ks * 16;
                // B: Q~[head g][channels k0 + 4 cq .. + 3]
                const uint2 bw = *reinterpret_cast<const uint2 *>(qs + size_t(g) * qstride + k0 + 4 * cq);
                if (BITS == 4) {
                    const int grp = k0 / 128;
                    if (grp != cur_grp) {
                        if (cur_grp >= 0) {
#pragma unroll
                            for (int m = 0; m < kMaxTS / 16; ++m) {
                                if (m >= MT) break;
                                const float s0 = __half2float(gsc[(m * 16 + g) * (r / 128) + cur_grp]);
                                const float s1 = __half2float(gsc[(m * 16 + g + 8) * (r / 128) + cur_grp]);
                                acc[m][0] = fmaf(s0, gacc[m][0], acc[m][0]); acc[m][1] = fmaf(s0, gacc[m][1], acc[m][1]);
                                acc[m][2] = fmaf(s1, gacc[m][2], acc[m][2]); acc[m][3] = fmaf(s1, gacc[m][3], acc[m][3]);
                                gacc[m][0] = gacc[m][1] = gacc[m][2] = gacc[m][3] = 0.0f;
                            }
                        }
                        cur_grp = grp;
                    }
                }
#pragma unroll
                for (int m = 0; m < kMaxTS / 16; ++m) {
                    if (m >= MT) break;
                    uint32_t a0, a1, a2, a3;
                    load_frag<BITS>(tile, rstride, m * 16 + g, k0, cq, a0, a2);
                    load_frag<BITS>(tile, rstride, m * 16 + g + 8, k0, cq, a1, a3);
                    if (BITS == 8)
                        mma16816((ks / kWarps) & 1 ? gacc[m] : acc[m], a0, a1, a2, a3, bw.x, bw.y);   // two chains
                    else
                        mma16816(gacc[m], a0, a1, a2, a3, bw.x, bw.y);
                }
            }
            if (BITS == 8) {                           // add the second chain
#pragma unroll
                for (int m = 0; m < kMaxTS / 16; ++m) {
                    acc[m][0] += gacc[m][0]; acc[m][1] += gacc[m][1]; acc[m][2] += gacc[m][2]; acc[m][3] += gacc[m][3];
                }
            }
            if (BITS == 4 && cur_grp >= 0) {
#pragma unroll
                for (int m = 0; m < kMaxTS / 16; ++m) {
                    if (m >= MT) break;
                    const float s0 = __half2float(gsc[(m * 16 + g) * (r / 128) + cur_grp]);
                    const float s1 = __half2float(gsc[(m * 16 + g + 8) * (r / 128) + cur_grp]);
                    acc[m][0] = fmaf(s0, gacc[m][0], acc[m][0]); acc[m][1] = fmaf(s0, gacc[m][1], acc[m][1]);
                    acc[m][2] = fmaf(s1, gacc[m][2], acc[m][2]); acc[m][3] = fmaf(s1, gacc[m][3], acc[m][3]);
                }
            }
#pragma unroll
            for (int m = 0; m < kMaxTS / 16; ++m) {
                if (m >= MT) break;
                sred[warp][m * 16 + g][2 * cq] = acc[m][0];
                sred[warp][m * 16 + g][2 * cq + 1] = acc[m][1];
                sred[warp][m * 16 + g + 8][2 * cq] = acc[m][2];
                sred[warp][m * 16 + g + 8][2 * cq + 1] = acc[m][3];
            }
        }
        __syncthreads();

        // ---- 3. running softmax per head: a warp per head, thread per token
        if (warp < kHG) {
            const int hl = warp, h = h0 + hl;
            float lg[kMaxTS / 32];
            float mx = -INFINITY;
#pragma unroll
            for (int u = 0; u < kMaxTS / 32; ++u) {
                const int t = lane + 32 * u;
                float v = -INFINITY;
                if (t < n && h < H) {
                    float sacc = 0.0f;
#pragma unroll
                    for (int w = 0; w < kWarps; ++w) sacc += sred[w][t][hl];
                    v = sacc * qfac_s[hl] * (BITS == 8 ? tsc_s[t] : 1.0f);
                }
                lg[u] = v;
                mx = fmaxf(mx, v);
            }
            mx = warp_max(mx);
            const float m_new = fmaxf(m_run, mx);
            const float alpha = (h < H && m_run != -INFINITY) ? exp2f(m_run - m_new) : (h < H ? 0.0f : 1.0f);
            float l = 0.0f;
#pragma unroll
            for (int u = 0; u < kMaxTS / 32; ++u) {
                const int t = lane + 32 * u;
                const float pe = (t < n && h < H) ? exp2f(lg[u] - m_new) : 0.0f;
                l += pe;
                if (t < TS) ps[size_t(hl) * pstride + t] = __float2half_rn(BITS == 8 ? pe * tsc_s[t] : pe);
            }
            l = warp_sum(l);
            l_run = l_run * alpha + l;
            m_run = h < H ? m_new : m_run;
            if (lane == 0) alpha_s[hl] = alpha;
        }
        __syncthreads();

        // ---- 4. O^T[ch, h] += sum_t C[t, ch] P[t, h]: warp w, channel blocks w + kWarps j
        {
            const float al0 = alpha_s[2 * cq], al1 = alpha_s[2 * cq + 1];
#pragma unroll
            for (int j = 0; j < MB; ++j) {
                o[j][0] *= al0; o[j][1] *= al1; o[j][2] *= al0; o[j][3] *= al1;
            }
            for (int kt = 0; kt < MT; ++kt) {
                const int tb = kt * 16;
                // B: P[head g][tokens tb + 2cq, +1] and [tb + 8 + 2cq, +1]
                const uint32_t pw0 = *reinterpret_cast<const uint32_t *>(ps + size_t(g) * pstride + tb + 2 * cq);
                const uint32_t pw1 = *reinterpret_cast<const uint32_t *>(ps + size_t(g) * pstride + tb + 8 + 2 * cq);
#pragma unroll
                for (int j = 0; j < MB; ++j) {
                    const int mb = warp + kWarps * j;
                    if (mb >= nks) break;
                    // A: the score fragments of tokens tb.. tb + 15, channel step mb, transposed
                    uint32_t x0, x1, x2, x3;
                    load_frag<BITS>(tile, rstride, tb + g, mb * 16, cq, x0, x2);
                    load_frag<BITS>(tile, rstride, tb + g + 8, mb * 16, cq, x1, x3);
                    uint32_t b0 = pw0, b1 = pw1;
                    if (BITS == 4) {                    // int4: times the token's group scale
                        const int grp = mb / 8, ng = r / 128;
                        const __half2 s0 = __halves2half2(gsc[(tb + 2 * cq) * ng + grp], gsc[(tb + 2 * cq + 1) * ng + grp]);
                        const __half2 s1 = __halves2half2(gsc[(tb + 8 + 2 * cq) * ng + grp], gsc[(tb + 9 + 2 * cq) * ng + grp]);
                        const __half2 p0 = __hmul2(*reinterpret_cast<const __half2 *>(&pw0), s0);
                        const __half2 p1 = __hmul2(*reinterpret_cast<const __half2 *>(&pw1), s1);
                        b0 = *reinterpret_cast<const uint32_t *>(&p0);
                        b1 = *reinterpret_cast<const uint32_t *>(&p1);
                    }
                    mma16816(o[j], movm_t(x0), movm_t(x2), movm_t(x1), movm_t(x3), b0, b1);
                }
            }
        }
    }

    // ---- 5. the CTA's partial: o_lat^T fragments (reduction indices g, g+8 of the
    //         channel step, i.e. channels 4(g/2) + g%2 and that + 2; heads 2cq, 2cq+1),
    //         m and l per head.
    //         Lanes g = 2a and 2a + 1 hold channels 4a, 4a + 2 and 4a + 1, 4a + 3 of
    //         heads 2cq, 2cq + 1: one exchange gives each a float4 of 4 consecutive
    //         channels of one head (even lane: head 2cq, odd lane: head 2cq + 1).
    const size_t pb = (size_t(b) * p.n_split + split) * H + h0;
    const int odd = g & 1, hl = 2 * cq + odd, c4 = 4 * (g >> 1);
#pragma unroll
    for (int j = 0; j < MB; ++j) {
        const int mb = warp + kWarps * j;
        if (mb >= nks) break;
        const float v0 = __shfl_xor_sync(0xffffffffu, odd ? o[j][0] : o[j][1], 4);
        const float v1 = __shfl_xor_sync(0xffffffffu, odd ? o[j][2] : o[j][3], 4);
        const float4 w = odd ? make_float4(v0, o[j][1], v1, o[j][3]) : make_float4(o[j][0], v0, o[j][2], v1);
        if (h0 + hl < H) *reinterpret_cast<float4 *>(p.po + (pb + hl) * r + mb * 16 + c4) = w;
    }
    if (warp < kHG && lane == 0 && h0 + warp < H) {
        p.pm[pb + warp] = m_run * 0.6931471805599453f;        // natural-log units
        p.pl[pb + warp] = l_run;
    }
}

// ---------------------------------------------------------------------------
// Automatic choice: this kernel for small batch x length, and for every
// length it can split (<= 64 x 64 tokens) when the tcgen05 kernel cannot take
// the shape.
bool attn_mma_use(const CacheView &c, int H, int B, int max_seq_len) {
    const int path = attn_path();
    if (path == 1 || path == 2) return false;
    if (path == 3) return true;
    return int64_t(B) * max_seq_len <= mma_tokens_max(c.r) || !attn_tc_shape_ok(c.r, c.bits, H);
}

namespace {
// Dynamic shared memory of one CTA: a sub-tile of cache rows, the query
// block, int4 group scales and P.
size_t attn_mma_smem(int r, int bits, int ts) {
    const int row_bytes = bits == 8 ? r : r / 2;
    return size_t(ts) * (row_bytes + am::kRowPad) + size_t(am::kHG) * (r + am::kQPad) * 2 +
           (bits == 4 ? size_t(ts) * (r / 128) * 2 : 0) + size_t(am::kHG) * (ts + 8) * 2;
}
// Largest sub-tile whose rows fit next to the static arrays (about 33 KB of
// the 227 KB a CTA may hold).
int attn_mma_max_ts(int r, int bits) {
    constexpr size_t kBudget = 192 * 1024;
    int t = am::kMaxTS;
    while (t > 16 && attn_mma_smem(r, bits, t) > kBudget) t /= 2;
    return attn_mma_smem(r, bits, t) <= kBudget ? t : 0;
}
constexpr int kMaxRankMma = 3072;     // r / 16 / kWarps channel blocks per warp at most
}  // namespace

// Sub-tile: the smallest of 16, 32, 64 (within shared memory) whose grid fits
// one wave of the GPU; sub-tiles per split: at least enough for 64 partials
// per sequence, and more while two waves of CTAs remain (fewer partials to
// merge, fewer query-block loads).
int attn_mma_splits(const CacheView &c, int B, int H, int max_seq_len, int *ts, int *n_sub) {
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t hg = (H + am::kHG - 1) / am::kHG;
    const int tmax = attn_mma_max_ts(c.r, c.bits);
    int t = 16;
    while (t < tmax && int64_t(B) * ((max_seq_len + t - 1) / t) * hg > sms) t *= 2;
    const int tiles = (max_seq_len + t - 1) / t;
    int ns = (tiles + 63) / 64;
    while (2 * ns <= tiles && int64_t(B) * hg * ((tiles + 2 * ns - 1) / (2 * ns)) >= 2 * int64_t(sms)) ns *= 2;
    *ts = t;
    *n_sub = ns;
    return (tiles + ns - 1) / ns;
}

bool attn_mma_fits(const CacheView &c, int max_seq_len) {
    (void)max_seq_len;                // any length: a CTA walks as many sub-tiles as needed
    return c.r <= kMaxRankMma && attn_mma_max_ts(c.r, c.bits) > 0;
}

namespace {
template <int BITS>
cudaError_t launch_mma_bits(const am::Params &prm, dim3 grid, size_t smem, cudaStream_t s) {
    const int need = (prm.c.r / 16 + am::kWarps - 1) / am::kWarps;   // channel blocks per warp
    auto go = [&](auto kern) {
        cudaError_t e = ensure_smem(kern, smem);
        return e == cudaSuccess ? launch_pdl(kern, grid, dim3(am::kThreads), smem, s, prm) : e;
    };
    constexpr int kMaxMB = kMaxRankMma / 16 / am::kWarps;       // r <= kMaxRankMma
    static_assert(kMaxMB >= 12, "channel blocks per warp");
    if (need <= 4) return go(attn_mma_kernel<BITS, 4>);
    if (need <= 8) return go(attn_mma_kernel<BITS, 8>);
    if (need <= 12) return go(attn_mma_kernel<BITS, 12>);
    if (need <= 16) return go(attn_mma_kernel<BITS, (kMaxMB > 16 ? 16 : kMaxMB)>);
    return go(attn_mma_kernel<BITS, kMaxMB>);
}
}  // namespace

cudaError_t launch_attn_mma(const CacheView &c, const int32_t *seq_len, const float *qt, const unsigned *qmax, int H,
                            float softmax_scale, int ts, int n_sub, int n_split, float *pm, float *pl, float *po,
                            int *err, cudaStream_t s) {
    const size_t smem = attn_mma_smem(c.r, c.bits, ts);
    const am::Params prm{c, seq_len, qt, qmax, H, ts, n_sub, n_split, softmax_scale, pm, pl, po, err};
    const dim3 grid(n_split, c.B, (H + am::kHG - 1) / am::kHG);
    return c.bits == 8 ? launch_mma_bits<8>(prm, grid, smem, s) : launch_mma_bits<4>(prm, grid, smem, s);
}

}  // namespace qsvd
