// The per-step products with the up-projections around decode attention
// (Eq. 5 with W^u_k absorbed into the query and W^u_v applied last), for all
// B sequences of a step at once:
//
//   qproj_kernel      a5: q[b] = c_{L_b - 1} U_q
//   qabsorb_kernel    a5: q~[b, h, j] = U_k[j, h-block] . q[b, h-block], and the
//                     per-(b, h) maximum of |q~| (it scales the fp16 query of
//                     the tensor-core attention)
//   combine_uv_kernel a7/a8: merge the per-split softmax partials of every
//                     sequence and multiply by U_v[:, h-block]
//
// Each is a skinny product (B rows) that streams one up-projection once.  A
// CTA's weight tile arrives by one or two TMA boxes (or a few large bulk
// copies); all global loads of a phase are issued before the first use; each
// thread keeps the sums of NB sequences in registers (NB = the batch rounded up
// to a power of two, at most 16).  The products over the r latent channels
// (qproj, combine) are split over a cluster of kCl CTAs, whose partial results
// are added in rank order through distributed shared memory: the sums are
// deterministic and need no global scratch.
#include <cfloat>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

namespace {

constexpr int kBC = 16;          // largest NB
constexpr int kCl = 8;           // CTAs per cluster (split of the r latent rows; cluster_ld8 reads 8 ranks)
constexpr int kQaRows = 32;      // U_k rows per qabsorb CTA (one per lane)
constexpr int kMaxSplitsG = 64;  // softmax partials per sequence

__device__ __forceinline__ uint32_t cl_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void cl_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void tma_2d(void *dst, const CUtensorMap *map, int x, int y, uint64_t *bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(smem_addr(dst)), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
        : "memory");
}
__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void tma_prefetch(const CUtensorMap *map, int x, int y) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];"
                 ::"l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y)
                 : "memory");
}

__device__ __forceinline__ bool len_ok(int L, int Tmax) { return L >= 1 && L <= Tmax; }

// Rows of a weight tile per TMA box (box dimensions are at most 256).
__host__ __device__ __forceinline__ int box_rows(int rs) { return rs / ((rs + 255) / 256); }

// Up-projection weights are read in one of three formats (WB = bits per
// weight): 16 = bf16 values; 8 = int8 codes; 4 = packed int4 codes (element
// 2i in the low nibble of byte i, two's complement).  The codes of Eq. 11's
// Q(W^u) have one fp32 scale per output channel, applied by the kernels to
// the products' inputs or outputs.  The conversions below are exact: an int8
// byte b placed in the mantissa of 2^23 gives 2^23 + (b ^ 0x80) as an fp32,
// and subtracting 2^23 + 128 leaves the code; a nibble likewise with 2^23 + 8.
__device__ __forceinline__ float i8_byte(uint32_t u, int k) {       // u = word ^ 0x80808080
    return __uint_as_float(__byte_perm(u, 0x4B000000u, uint32_t(k) | (4u << 4) | (5u << 8) | (7u << 12))) -
           8388736.0f;
}
__device__ __forceinline__ float i4_nib(uint32_t x, int k) {        // x = word ^ 0x88888888
    return __uint_as_float(((x >> (4 * k)) & 0xFu) | 0x4B000000u) - 8388616.0f;
}
// Four consecutive weights of a tile row, starting at weight 4 * q4.
template <int WB>
__device__ __forceinline__ void load_w4(const uint8_t *row, int q4, float (&u)[4]) {
    if (WB == 16) {
        const uint2 w2 = *reinterpret_cast<const uint2 *>(row + 8 * q4);
        u[0] = bf16_lo(w2.x); u[1] = bf16_hi(w2.x); u[2] = bf16_lo(w2.y); u[3] = bf16_hi(w2.y);
    } else if (WB == 8) {
        const uint32_t x = *reinterpret_cast<const uint32_t *>(row + 4 * q4) ^ 0x80808080u;
#pragma unroll
        for (int e = 0; e < 4; ++e) u[e] = i8_byte(x, e);
    } else {
        const uint32_t x = uint32_t(*reinterpret_cast<const uint16_t *>(row + 2 * q4)) ^ 0x8888u;
#pragma unroll
        for (int e = 0; e < 4; ++e) u[e] = i4_nib(x, e);
    }
}
// Weight `col` of a tile row.
template <int WB>
__device__ __forceinline__ float load_w1(const uint8_t *row, int col) {
    if (WB == 16) return bf16_to_f32(reinterpret_cast<const uint16_t *>(row)[col]);
    if (WB == 8) return float(int8_t(row[col]));
    const int b = (row[col >> 1] >> (4 * (col & 1))) & 0xF;
    return float((b ^ 8) - 8);
}
// The 128 / WB weights held in 16 bytes.
template <int WB>
__device__ __forceinline__ void unpack16B(const uint4 &v, float (&f)[128 / WB]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    if (WB == 16) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            f[2 * k] = bf16_lo(w[k]);
            f[2 * k + 1] = bf16_hi(w[k]);
        }
    } else if (WB == 8) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint32_t x = w[k] ^ 0x80808080u;
#pragma unroll
            for (int e = 0; e < 4; ++e) f[4 * k + e] = i8_byte(x, e);
        }
    } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint32_t x = w[k] ^ 0x88888888u;
#pragma unroll
            for (int e = 0; e < 8; ++e) f[8 * k + e] = i4_nib(x, e);
        }
    }
}

}  // namespace

// ---------------------------------------------------------------------------
// a5 first half.  Grid (kCl, d / ncol), cluster (kCl, 1, 1), 256 threads.
// CTA k of a cluster takes rows [k rs, (k+1) rs) of U_q (rs = r / kCl) and the
// cluster's ncol columns.  Thread = (column quad, row group): it accumulates 4
// columns x NB sequences over its row group; the row groups are added in
// shared memory, then rank k adds the kCl partials of columns
// [k ncol/kCl, (k+1) ncol/kCl) in rank order.  CTA (0, 0) also clears qmax.
//
// FRESH: the current tokens' latents are not in the cache yet; c_hat holds
// them as the projection left them (fp32, row b = sequence b).  Every CTA
// requantizes each row the way requant_kernel does (Eq. 11's Q(C_qkv): the
// same quantizer on the same values gives the same codes and scales), keeps
// the dequantized values of its own rows, and the CTAs of the first cluster
// store their rows' codes, with the scales, at position L - 1 of the
// sequence (a4).  This saves a decode step the requantization launch and one
// dependent round trip; the kernels that read the cache run after this grid.
// ---------------------------------------------------------------------------
constexpr int kFreshQuads = 3;     // float4 of a latent row per thread (r <= 3072)

template <int NB>
__device__ __forceinline__ void fresh_rows(const float *c_hat, int b0, int nb, const int *L_s, const int *Q_s,
                                           const CacheView &c, float lat_clip, int j0, int rs, bool writer,
                                           float *c_s, float (*red)[8]) {
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, r = c.r, nq = r / 4;
    const int q_lo = j0 / 4, q_hi = (j0 + rs) / 4;      // this CTA's quads
    float4 v[NB][kFreshQuads];
#pragma unroll
    for (int bi = 0; bi < NB; ++bi)
#pragma unroll
        for (int k = 0; k < kFreshQuads; ++k) {
            const int qi = tid + k * 256;
            v[bi][k] = (bi < nb && L_s[bi] > 0 && qi < nq)
                           ? reinterpret_cast<const float4 *>(c_hat + size_t(b0 + bi) * r)[qi]
                           : make_float4(0.f, 0.f, 0.f, 0.f);
        }
    if (c.bits == 8) {
        // one scale per token: the maximum over all r channels
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) {
            float m = 0.0f;
#pragma unroll
            for (int k = 0; k < kFreshQuads; ++k)
                m = fmaxf(m, fmaxf(fmaxf(fabsf(v[bi][k].x), fabsf(v[bi][k].y)),
                                   fmaxf(fabsf(v[bi][k].z), fabsf(v[bi][k].w))));
            m = warp_max(m);
            if (lane == 0) red[bi][warp] = m;
        }
        __syncthreads();
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) {
            // rows without a valid slot hold zeros: zero scale, zero values, nothing stored
            const bool live = bi < nb && L_s[bi] > 0;
            float m = red[bi][0];
#pragma unroll
            for (int w = 1; w < 8; ++w) m = fmaxf(m, red[bi][w]);
            const float s = quant_scale(m, lat_clip, 127.0f), inv = quant_inv_scale(s);
            const size_t slot = live ? size_t(Q_s[bi]) * c.Tmax + (L_s[bi] - 1) : 0;
#pragma unroll
            for (int k = 0; k < kFreshQuads; ++k) {
                const int qi = tid + k * 256;
                if (qi < q_lo || qi >= q_hi) continue;
                const int c0 = quant_code_fast(v[bi][k].x, s, inv, 127), c1 = quant_code_fast(v[bi][k].y, s, inv, 127);
                const int c2 = quant_code_fast(v[bi][k].z, s, inv, 127), c3 = quant_code_fast(v[bi][k].w, s, inv, 127);
                *reinterpret_cast<float4 *>(c_s + bi * rs + 4 * qi - j0) =
                    make_float4(float(c0) * s, float(c1) * s, float(c2) * s, float(c3) * s);
                if (writer && live)
                    reinterpret_cast<uint32_t *>(static_cast<int8_t *>(c.codes) + slot * r)[qi] =
                        uint32_t(c0 & 0xff) | (uint32_t(c1 & 0xff) << 8) | (uint32_t(c2 & 0xff) << 16) |
                        (uint32_t(c3 & 0xff) << 24);
            }
            if (writer && live && j0 == 0 && tid == 0) static_cast<float *>(c.scales)[slot] = s;
        }
    } else {
        // one fp16 scale per 128-channel group: the 32 quads of a group are one warp's lanes
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) {
            const bool live = bi < nb && L_s[bi] > 0;
            const size_t slot = live ? size_t(Q_s[bi]) * c.Tmax + (L_s[bi] - 1) : 0;
#pragma unroll
            for (int k = 0; k < kFreshQuads; ++k) {
                const int qi = tid + k * 256;
                if (qi - lane >= nq) break;                 // warp-uniform
                float m = fmaxf(fmaxf(fabsf(v[bi][k].x), fabsf(v[bi][k].y)), fmaxf(fabsf(v[bi][k].z), fabsf(v[bi][k].w)));
                m = warp_max(m);
                if (qi < q_lo || qi >= q_hi) continue;
                const __half hs = int4_group_scale(m, lat_clip);
                const float s = __half2float(hs), inv = quant_inv_scale(s);
                const int c0 = quant_code_fast(v[bi][k].x, s, inv, 7), c1 = quant_code_fast(v[bi][k].y, s, inv, 7);
                const int c2 = quant_code_fast(v[bi][k].z, s, inv, 7), c3 = quant_code_fast(v[bi][k].w, s, inv, 7);
                *reinterpret_cast<float4 *>(c_s + bi * rs + 4 * qi - j0) =
                    make_float4(float(c0) * s, float(c1) * s, float(c2) * s, float(c3) * s);
                if (writer && live) {
                    reinterpret_cast<uint16_t *>(static_cast<uint8_t *>(c.codes) + slot * (r / 2))[qi] =
                        uint16_t((c0 & 0xf) | ((c1 & 0xf) << 4) | ((c2 & 0xf) << 8) | ((c3 & 0xf) << 12));
                    if (lane == 0) static_cast<__half *>(c.scales)[slot * (r / 128) + qi / 32] = hs;
                }
            }
        }
    }
}

template <int NB, int WB, bool FRESH>
__global__ void __cluster_dims__(kCl, 1, 1) __launch_bounds__(256)
qproj_kernel(const __grid_constant__ CUtensorMap map_u, const uint8_t *__restrict__ Uq, const float *__restrict__ sq,
             CacheView c, const int32_t *__restrict__ seq_len, int B, int d, int ncol, float *__restrict__ q,
             unsigned *__restrict__ qmax, int n_qmax, const float *c_hat, float lat_clip, int *err) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t bar;
    __shared__ int L_s[NB], Q_s[NB];   // length and cache sequence of each row
    const int r = c.r, rs = r / kCl, br = box_rows(rs);
    const int ncq = ncol / 4, G = 256 / ncq, rpg = rs / G;
    const int rb = ncol * WB / 8;                                                // tile row bytes
    const uint32_t rank = cl_rank();
    const int c0 = blockIdx.y * ncol, j0 = int(rank) * rs;
    uint8_t *u_s = smem;                                                         // [rs][rb] weight codes
    float *c_s = reinterpret_cast<float *>(smem + size_t(rs) * rb);              // [NB][rs]
    float *part = c_s + NB * rs;                                                 // [G][NB][ncol]
    const int tid = threadIdx.x;
    if (tid == 0) {
        for (int k = 0; k < rs / br; ++k) tma_prefetch(&map_u, WB == 16 ? c0 : c0 * WB / 8, j0 + k * br);
        mbar_init(&bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    // the U_q tile: 16-byte asynchronous copies by every thread (many small
    // rows: cheaper than bulk or tensor copies of 512-byte rows).  The weights
    // are no kernel's output, so the copies start before the wait on the
    // producer grid and overlap its tail.
    for (int i = tid; i < rs * (rb / 16); i += blockDim.x) {
        const int row = i / (rb / 16), k = i - row * (rb / 16);
        cp_async16(u_s + size_t(row) * rb + 16 * k, Uq + (size_t(j0 + row) * d + c0) * WB / 8 + 16 * k);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    pdl_wait();
    pdl_trigger();   // after the wait: the attention kernel two launches on reads the
                     // lengths before its own wait, and they are complete by then
    if (rank == 0 && blockIdx.y == 0)
        for (int i = tid; i < n_qmax; i += blockDim.x) qmax[i] = 0u;
    bool ready = false;
    const int per_rank = ncol / kCl;
    const int wpr = c.bits == 8 ? rs / 4 : rs / 8;        // 32-bit code words per latent row slice
    const int cq = tid % ncq, g = tid / ncq;
    for (int b0 = 0; b0 < B; b0 += NB) {
        const int nb = min(NB, B - b0);
        __syncthreads();
        if (tid < NB) {
            int L = tid < nb ? seq_len[b0 + tid] : 0;
            const int sq = tid < nb ? view_seq(c, b0 + tid) : 0;
            if (tid < nb && (sq < 0 || !len_ok(L, c.Tmax))) {
                if (rank == 0 && blockIdx.y == 0) flag_error(err, kErrRange);
                L = 0;
            }
            L_s[tid] = L;
            Q_s[tid] = sq;
        }
        __syncthreads();
        if constexpr (FRESH) {
            __shared__ float red_f[NB][8];
            fresh_rows<NB>(c_hat, b0, nb, L_s, Q_s, c, lat_clip, j0, rs, blockIdx.y == 0, c_s, red_f);
        } else {
        // dequantized latent rows c_{L-1}: code words and scales, every load issued first
        constexpr int kPer = (NB * 96 + 255) / 256;      // >= words per thread (rs <= 384)
        uint32_t wv[kPer];
        float sv[kPer];
#pragma unroll
        for (int k = 0; k < kPer; ++k) {
            const int w = tid + k * 256;
            wv[k] = 0u;
            sv[k] = 0.0f;
            if (w < nb * wpr) {
                const int bi = w / wpr, x = w - bi * wpr;
                const int L = L_s[bi];
                if (L > 0) {
                    const size_t slot = size_t(Q_s[bi]) * c.Tmax + (L - 1);
                    if (c.bits == 8) {
                        wv[k] = reinterpret_cast<const uint32_t *>(static_cast<const int8_t *>(c.codes) + slot * r + j0)[x];
                        sv[k] = static_cast<const float *>(c.scales)[slot];
                    } else {
                        wv[k] = reinterpret_cast<const uint32_t *>(static_cast<const uint8_t *>(c.codes) + slot * (r / 2) + j0 / 2)[x];
                        sv[k] = __half2float(static_cast<const __half *>(c.scales)[slot * (r / 128) + (j0 + 8 * x) / 128]);
                    }
                }
            }
        }
#pragma unroll
        for (int k = 0; k < kPer; ++k) {
            const int w = tid + k * 256;
            if (w >= nb * wpr) break;
            const int bi = w / wpr, x = w - bi * wpr;
            if (c.bits == 8) {
                float4 o;
                o.x = float(int8_t(wv[k] & 0xff)) * sv[k];
                o.y = float(int8_t((wv[k] >> 8) & 0xff)) * sv[k];
                o.z = float(int8_t((wv[k] >> 16) & 0xff)) * sv[k];
                o.w = float(int8_t(wv[k] >> 24)) * sv[k];
                *reinterpret_cast<float4 *>(c_s + bi * rs + 4 * x) = o;
            } else {
                float f[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) f[e] = float((int((wv[k] >> (4 * e)) & 0xf) ^ 8) - 8) * sv[k];
                *reinterpret_cast<float4 *>(c_s + bi * rs + 8 * x) = make_float4(f[0], f[1], f[2], f[3]);
                *reinterpret_cast<float4 *>(c_s + bi * rs + 8 * x + 4) = make_float4(f[4], f[5], f[6], f[7]);
            }
        }
        }
        for (int i = nb * rs + tid; i < NB * rs; i += blockDim.x) c_s[i] = 0.0f;
        if (!ready) {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
            ready = true;
        }
        __syncthreads();
        // 4 columns x NB sequences over rows [g rpg, (g+1) rpg)
        float acc[NB][4];
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) acc[bi][0] = acc[bi][1] = acc[bi][2] = acc[bi][3] = 0.0f;
        const int i0 = g * rpg, i1 = i0 + rpg;
        int i = i0;
        for (; i + 4 <= i1; i += 4) {
            float u[4][4];
#pragma unroll
            for (int k = 0; k < 4; ++k) load_w4<WB>(u_s + size_t(i + k) * rb, cq, u[k]);
#pragma unroll
            for (int bi = 0; bi < NB; ++bi) {
                const float4 cv = *reinterpret_cast<const float4 *>(c_s + bi * rs + i);
#pragma unroll
                for (int e = 0; e < 4; ++e)
                    acc[bi][e] = fmaf(cv.w, u[3][e], fmaf(cv.z, u[2][e], fmaf(cv.y, u[1][e], fmaf(cv.x, u[0][e], acc[bi][e]))));
            }
        }
        for (; i < i1; ++i) {                          // rows left over when rpg % 4 != 0
            float u4[4];
            load_w4<WB>(u_s + size_t(i) * rb, cq, u4);
            const float u0 = u4[0], u1 = u4[1], u2 = u4[2], u3 = u4[3];
#pragma unroll
            for (int bi = 0; bi < NB; ++bi) {
                const float cv = c_s[bi * rs + i];
                acc[bi][0] = fmaf(cv, u0, acc[bi][0]);
                acc[bi][1] = fmaf(cv, u1, acc[bi][1]);
                acc[bi][2] = fmaf(cv, u2, acc[bi][2]);
                acc[bi][3] = fmaf(cv, u3, acc[bi][3]);
            }
        }
#pragma unroll
        for (int bi = 0; bi < NB; ++bi)
            *reinterpret_cast<float4 *>(part + (size_t(g) * NB + bi) * ncol + 4 * cq) =
                make_float4(acc[bi][0], acc[bi][1], acc[bi][2], acc[bi][3]);
        __syncthreads();
        for (int o = tid; o < nb * ncol; o += blockDim.x) {     // row groups in order
            float v = part[o];
            for (int k = 1; k < G; ++k) v += part[size_t(k) * NB * ncol + o];
            part[o] = v;
        }
        cl_sync();                                   // every rank's partials are complete
        for (int o = tid; o < nb * per_rank; o += blockDim.x) {
            const int bi = o / per_rank, col = int(rank) * per_rank + (o - bi * per_rank);
            float pk[kCl];
            cluster_ld8(part + bi * ncol + col, pk);
            float v = 0.0f;
#pragma unroll
            for (int k = 0; k < kCl; ++k) v += pk[k];       // rank order
            if (WB != 16) v *= sq[c0 + col];         // per-output-channel scale of Q(U_q)
            q[size_t(b0 + bi) * d + c0 + col] = v;
        }
        cl_sync();                                   // partials read before they are overwritten / the CTA exits
    }
}

// ---------------------------------------------------------------------------
// a5 second half.  Grid (ceil(r / 32), H / hg), 32 * hg threads: lane = row j
// of U_k, warp = head.  The head block of the 32 rows sits in shared memory
// with rows padded by 16 bytes (conflict-free 16-byte reads).
// ---------------------------------------------------------------------------
template <int NB, int WB>
__global__ void __launch_bounds__(256)
qabsorb_kernel(const float *q, const uint8_t *__restrict__ Uk, const float *__restrict__ sk, int B, int r,
               int d, int H, int dh, int hg, float *__restrict__ qt, unsigned *__restrict__ qmax, int *err) {
    extern __shared__ __align__(16) uint8_t smem[];
    __shared__ __align__(8) uint64_t bar;
    const int w = hg * dh;
    const int wb = w * WB / 8;                                                   // weight bytes per row
    const int ustride = wb + 16;                                                 // bytes per padded row
    uint8_t *u_s = smem;                                                         // [32][ustride]
    float *q_s = reinterpret_cast<float *>(smem + size_t(kQaRows) * ustride);    // [NB][hg * dh]
    const int j0 = blockIdx.x * kQaRows, h0 = blockIdx.y * hg;
    const int rows = min(kQaRows, r - j0);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x < 32)
        for (int i = lane; i < rows; i += 32)
            prefetch_l2_bulk(Uk + (size_t(j0 + i) * d + size_t(h0) * dh) * WB / 8, uint32_t(wb));
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    if (warp == 0) {            // U_k rows: no kernel's output, copied before the wait on the producer grid
        if (lane == 0) mbar_arrive_expect_tx(&bar, uint32_t(rows) * wb);
        __syncwarp();
        for (int i = lane; i < rows; i += 32)
            bulk_g2s(u_s + size_t(i) * ustride, Uk + (size_t(j0 + i) * d + size_t(h0) * dh) * WB / 8, uint32_t(wb),
                     &bar);
    }
    pdl_wait();
    pdl_trigger();   // after the wait: the attention kernel two launches on reads the
                     // lengths before its own wait, and they are complete by then
    bool ready = false;
    const int h = h0 + warp;
    for (int b0 = 0; b0 < B; b0 += NB) {
        const int nb = min(NB, B - b0);
        __syncthreads();
        // q block of the pass, every load issued first (at most NB float4 per thread: dh <= 128)
        {
            float4 v[NB];
            const int n4 = nb * (w / 4);
#pragma unroll
            for (int k = 0; k < NB; ++k) {
                const int idx = threadIdx.x + k * blockDim.x;
                v[k] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (idx < n4) {
                    const int bi = idx / (w / 4), c4 = idx - bi * (w / 4);
                    v[k] = reinterpret_cast<const float4 *>(q + size_t(b0 + bi) * d + size_t(h0) * dh)[c4];
                }
            }
#pragma unroll
            for (int k = 0; k < NB; ++k) {
                const int idx = threadIdx.x + k * blockDim.x;
                if (idx < n4) {
                    float4 x = v[k];
                    if (WB != 16) {     // Q(U_k)'s per-output-channel scales fold into q
                        const int c4 = idx % (w / 4);
                        const float4 sc = reinterpret_cast<const float4 *>(sk + size_t(h0) * dh)[c4];
                        x.x *= sc.x; x.y *= sc.y; x.z *= sc.z; x.w *= sc.w;
                    }
                    reinterpret_cast<float4 *>(q_s)[idx] = x;
                }
            }
        }
        __syncthreads();
        if (!ready) {
            mbar_wait(&bar, 0, err);
            ready = true;
        }
        float acc[NB];
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) acc[bi] = 0.0f;
        const uint8_t *urow = u_s + size_t(lane) * ustride + size_t(warp) * dh * WB / 8;
        constexpr int kStep = 128 / WB;                  // weights per 16-byte read
        for (int i = 0; i < dh; i += kStep) {
            float f[kStep];
            unpack16B<WB>(*reinterpret_cast<const uint4 *>(urow + i * WB / 8), f);
#pragma unroll
            for (int bi = 0; bi < NB; ++bi) {
                if (bi >= nb) break;
                float a = acc[bi];
#pragma unroll
                for (int e = 0; e < kStep; e += 4) {
                    const float4 qa = *reinterpret_cast<const float4 *>(q_s + bi * w + warp * dh + i + e);
                    a = fmaf(f[e], qa.x, a); a = fmaf(f[e + 1], qa.y, a);
                    a = fmaf(f[e + 2], qa.z, a); a = fmaf(f[e + 3], qa.w, a);
                }
                acc[bi] = a;
            }
        }
        const bool live = lane < rows;
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) {
            if (bi >= nb) break;
            if (live) qt[(size_t(b0 + bi) * H + h) * r + j0 + lane] = acc[bi];
            const float m = warp_max(live ? fabsf(acc[bi]) : 0.0f);
            if (lane == 0) atomicMax(qmax + size_t(b0 + bi) * H + h, __float_as_uint(m));
        }
    }
}

// ---------------------------------------------------------------------------
// a7/a8.  Grid (kCl, H), cluster (kCl, 1, 1), 256 threads.  CTA k of head h's
// cluster merges, for every sequence, the softmax partials of latent rows
// [k rs, (k+1) rs) (weights exp(m_s - M) / l), multiplies them by those rows
// of U_v[:, h-block], and rank k adds the kCl products for its share of the
// dh output columns in rank order.
// ---------------------------------------------------------------------------
template <int NB, int WB>
__global__ void __cluster_dims__(kCl, 1, 1) __launch_bounds__(256)
combine_uv_kernel(const __grid_constant__ CUtensorMap map_v, const uint8_t *__restrict__ Uv, const float *__restrict__ sv,
                  const int32_t *__restrict__ seq_len, const int32_t *__restrict__ seq_map, int nseq, int B, int Tmax,
                  int H, int dh, int r, int chunk, int n_split, const float *pm,
                  const float *pl, const float *po, float *__restrict__ O, int *err) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ __align__(8) uint64_t bar;
    __shared__ float w_s[NB][kMaxSplitsG];
    __shared__ float inv_s[NB];
    __shared__ int ns_s[NB];
    const int rs = r / kCl, d = H * dh, h = blockIdx.y, br = box_rows(rs);
    const uint32_t rank = cl_rank();
    const int j0 = int(rank) * rs;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nsub = 256 / dh;
    const int rb = dh * WB / 8;                                                  // tile row bytes
    uint8_t *u_s = smem;                                                         // [rs][rb] weight codes
    float *ol_s = reinterpret_cast<float *>(smem + size_t(rs) * rb);             // [NB][rs]
    float *p_s = ol_s + NB * rs;                                                 // [nsub][NB][dh]
    pdl_trigger();
    if (tid == 0) {
        for (int k = 0; k < rs / br; ++k) tma_prefetch(&map_v, WB == 16 ? h * dh : h * rb, j0 + k * br);
        mbar_init(&bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    for (int i = tid; i < rs * (rb / 16); i += blockDim.x) {    // the U_v tile, 16-byte asynchronous copies
        const int row = i / (rb / 16), k = i - row * (rb / 16); // (before the wait: no kernel writes U_v)
        cp_async16(u_s + size_t(row) * rb + 16 * k, Uv + (size_t(j0 + row) * d + size_t(h) * dh) * WB / 8 + 16 * k);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    pdl_wait();
    bool ready = false;
    const int nq = rs / 4;                           // row quads (r % 32 == 0)
    const int sub = tid / dh, col = tid - sub * dh;
    const int per_rank = dh / kCl;
    constexpr int kWB = (NB + 7) / 8;                // sequences per warp in the weight phase
    constexpr int kParts = NB >= 4 ? 1 : 4 / NB;     // lanes sharing one (sequence, row quad)
    constexpr int kBatch = 16;                       // partial rows in flight per lane
    for (int b0 = 0; b0 < B; b0 += NB) {
        const int nb = min(NB, B - b0);
        __syncthreads();
        // merge weights of every sequence of the pass: warp w takes sequences w, w+8
        {
            int ns[kWB];
            float m0[kWB], m1[kWB], l0[kWB], l1[kWB];
#pragma unroll
            for (int k = 0; k < kWB; ++k) {
                const int bi = warp + 8 * k;
                const int L = bi < nb ? row_len(seq_len, seq_map, nseq, b0 + bi) : 0;
                ns[k] = len_ok(L, Tmax) ? (L + chunk - 1) / chunk : 0;
            }
#pragma unroll
            for (int k = 0; k < kWB; ++k) {
                const size_t base = size_t(b0 + warp + 8 * k) * n_split * H + h;
                m0[k] = lane < ns[k] ? pm[base + size_t(lane) * H] : -FLT_MAX;
                m1[k] = lane + 32 < ns[k] ? pm[base + size_t(lane + 32) * H] : -FLT_MAX;
                l0[k] = lane < ns[k] ? pl[base + size_t(lane) * H] : 0.0f;
                l1[k] = lane + 32 < ns[k] ? pl[base + size_t(lane + 32) * H] : 0.0f;
            }
#pragma unroll
            for (int k = 0; k < kWB; ++k) {
                const int bi = warp + 8 * k;
                if (bi >= NB) break;
                const float M = warp_max(fmaxf(m0[k], m1[k]));
                const float e0 = lane < ns[k] ? expf(m0[k] - M) : 0.0f;
                const float e1 = lane + 32 < ns[k] ? expf(m1[k] - M) : 0.0f;
                w_s[bi][lane] = e0;
                w_s[bi][lane + 32] = e1;
                const float l = warp_sum(e0 * l0[k] + e1 * l1[k]);
                if (lane == 0) {
                    inv_s[bi] = ns[k] ? 1.0f / l : 0.0f;
                    ns_s[bi] = ns[k];
                }
            }
        }
        __syncthreads();
        // merged o_lat rows: item = (sequence, row quad, part); the kParts lanes of
        // an item take every kParts-th split and are added by shuffles.  Loads are
        // branch-free (clamped split index, zero weight) so they stay in flight.
        const int items = NB * nq * kParts;
        for (int base = 0; base < items; base += 256) {
            const int it = base + tid;
            const int part = it % kParts, rest = it / kParts;
            const int bi = rest / nq, q4 = rest - bi * nq;
            const int ns = (it < items && bi < nb) ? ns_s[bi] : 0;
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            if (ns > 0) {
                const float *src = po + (size_t(b0 + bi) * n_split * H + h) * r + j0 + 4 * q4;
                for (int s0 = part; s0 < ns; s0 += kBatch * kParts) {
                    float4 v[kBatch];
                    float wk[kBatch];
#pragma unroll
                    for (int k = 0; k < kBatch; ++k) {
                        const int sk = s0 + k * kParts;
                        const int sc = sk < ns ? sk : ns - 1;
                        v[k] = *reinterpret_cast<const float4 *>(src + size_t(sc) * H * r);
                        wk[k] = sk < ns ? w_s[bi][sc] : 0.0f;
                    }
#pragma unroll
                    for (int k = 0; k < kBatch; ++k) {
                        acc.x = fmaf(wk[k], v[k].x, acc.x);
                        acc.y = fmaf(wk[k], v[k].y, acc.y);
                        acc.z = fmaf(wk[k], v[k].z, acc.z);
                        acc.w = fmaf(wk[k], v[k].w, acc.w);
                    }
                }
            }
#pragma unroll
            for (int o = 1; o < kParts; o <<= 1) {
                acc.x += __shfl_xor_sync(0xffffffffu, acc.x, o);
                acc.y += __shfl_xor_sync(0xffffffffu, acc.y, o);
                acc.z += __shfl_xor_sync(0xffffffffu, acc.z, o);
                acc.w += __shfl_xor_sync(0xffffffffu, acc.w, o);
            }
            if (it < items && part == 0) {
                const float il = bi < nb ? inv_s[bi] : 0.0f;
                *reinterpret_cast<float4 *>(ol_s + bi * rs + 4 * q4) =
                    make_float4(acc.x * il, acc.y * il, acc.z * il, acc.w * il);
            }
        }
        if (!ready) {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
            ready = true;
        }
        __syncthreads();
        // this rank's rows times U_v: thread = (row subset `sub`, output column `col`)
        float acc[NB];
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) acc[bi] = 0.0f;
        for (int i = 4 * sub; i < rs; i += 4 * nsub) {
            const float u0 = load_w1<WB>(u_s + size_t(i) * rb, col), u1 = load_w1<WB>(u_s + size_t(i + 1) * rb, col);
            const float u2 = load_w1<WB>(u_s + size_t(i + 2) * rb, col), u3 = load_w1<WB>(u_s + size_t(i + 3) * rb, col);
#pragma unroll
            for (int bi = 0; bi < NB; ++bi) {
                const float4 o = *reinterpret_cast<const float4 *>(ol_s + bi * rs + i);
                acc[bi] = fmaf(o.w, u3, fmaf(o.z, u2, fmaf(o.y, u1, fmaf(o.x, u0, acc[bi]))));
            }
        }
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) p_s[(sub * NB + bi) * dh + col] = acc[bi];
        __syncthreads();
        for (int o = tid; o < nb * dh; o += blockDim.x) {      // row subsets in order
            float v = p_s[o];
            for (int k = 1; k < nsub; ++k) v += p_s[size_t(k) * NB * dh + o];
            p_s[o] = v;
        }
        cl_sync();                                   // every rank's products are complete
        for (int o = tid; o < nb * per_rank; o += blockDim.x) {
            const int bi = o / per_rank, cc = int(rank) * per_rank + (o - bi * per_rank);
            float pk[kCl];
            cluster_ld8(p_s + bi * dh + cc, pk);
            float v = 0.0f;
#pragma unroll
            for (int k = 0; k < kCl; ++k) v += pk[k];       // rank order
            if (WB != 16) v *= sv[size_t(h) * dh + cc];     // per-output-channel scale of Q(U_v)
            O[size_t(b0 + bi) * d + size_t(h) * dh + cc] = v;
        }
        cl_sync();
    }
}

// ---------------------------------------------------------------------------
namespace {

int qproj_cols(int r) { return r <= 1536 ? 256 : 128; }

int qabsorb_hg(int H) {
    for (int g = 8; g > 1; g >>= 1)
        if (H % g == 0) return g;
    return 1;
}

// Sequences per pass: the batch rounded up to a power of two, at most kBC.
int pass_nb(int B) {
    int nb = 1;
    while (nb < B && nb < kBC) nb <<= 1;
    return nb;
}

template <int NB, int WB, bool FRESH = false>
cudaError_t qproj_nb(const CUtensorMap &map, const UpW &Uq, const CacheView &c, const int32_t *seq_len, int d, float *q,
                     unsigned *qmax, int n_qmax, int *err, cudaStream_t s, const float *c_hat = nullptr,
                     float lat_clip = 1.0f) {
    const int rs = c.r / kCl, ncol = qproj_cols(c.r), G = 256 / (ncol / 4);
    const size_t smem = size_t(rs) * ncol * WB / 8 + size_t(NB) * rs * 4 + size_t(G) * NB * ncol * 4;
    cudaError_t e = ensure_smem(qproj_kernel<NB, WB, FRESH>, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(qproj_kernel<NB, WB, FRESH>, dim3(kCl, d / ncol), dim3(256), smem, s, map,
                      static_cast<const uint8_t *>(Uq.w), Uq.scale, c, seq_len, c.B, d, ncol, q, qmax, n_qmax, c_hat,
                      lat_clip, err);
}

template <int NB, int WB>
cudaError_t qabsorb_nb(const float *q, const UpW &Uk, int B, int r, int d, int H, int dh, float *qt,
                       unsigned *qmax, int *err, cudaStream_t s) {
    const int hg = qabsorb_hg(H);
    const size_t smem = size_t(kQaRows) * (size_t(hg) * dh * WB / 8 + 16) + size_t(NB) * hg * dh * 4;
    cudaError_t e = ensure_smem(qabsorb_kernel<NB, WB>, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(qabsorb_kernel<NB, WB>, dim3((r + kQaRows - 1) / kQaRows, H / hg), dim3(32 * hg), smem, s, q,
                      static_cast<const uint8_t *>(Uk.w), Uk.scale, B, r, d, H, dh, hg, qt, qmax, err);
}

template <int NB, int WB>
cudaError_t combine_nb(const CUtensorMap &map, const UpW &Uv, const int32_t *seq_len, const int32_t *seq_map,
                       int nseq, int B, int Tmax, int H, int dh, int r,
                       int chunk, int n_split, const float *pm, const float *pl, const float *po, float *O, int *err,
                       cudaStream_t s) {
    const int rs = r / kCl;
    const size_t smem = size_t(rs) * dh * WB / 8 + size_t(NB) * rs * 4 + size_t(256 / dh) * NB * dh * 4;
    cudaError_t e = ensure_smem(combine_uv_kernel<NB, WB>, smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(combine_uv_kernel<NB, WB>, dim3(kCl, H), dim3(256), smem, s, map,
                      static_cast<const uint8_t *>(Uv.w), Uv.scale, seq_len, seq_map, nseq, B, Tmax, H, dh, r, chunk,
                      n_split, pm, pl, po, O, err);
}

// Tensor map over an up-projection [r, d] for the L2 prefetch of a CTA's
// tile: bf16 elements, or the bytes of the int8 / int4 codes.
bool up_map(CUtensorMap *map, const UpW &U, int r, int d, int box_cols, int box_r) {
    if (U.bits == 16)
        return encode_map_2d(map, CU_TENSOR_MAP_DATA_TYPE_UINT16, U.w, uint64_t(d), uint64_t(r), uint64_t(d) * 2,
                             uint32_t(box_cols), uint32_t(box_r), CU_TENSOR_MAP_SWIZZLE_NONE);
    const uint64_t rowb = uint64_t(d) * U.bits / 8;
    return encode_map_2d(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, U.w, rowb, uint64_t(r), rowb,
                         uint32_t(box_cols * U.bits / 8), uint32_t(box_r), CU_TENSOR_MAP_SWIZZLE_NONE);
}

// Dispatch on the pass size NB (the batch rounded up to a power of two, at
// most kBC) and the weight format.
template <template <int, int> class F, typename... A>
cudaError_t dispatch_nb_wb(int B, int bits, A &&...a) {
    switch (bits) {
        case 16:
            switch (pass_nb(B)) {
                case 1: return F<1, 16>::run(a...);
                case 2: return F<2, 16>::run(a...);
                case 4: return F<4, 16>::run(a...);
                case 8: return F<8, 16>::run(a...);
                default: return F<16, 16>::run(a...);
            }
        case 8:
            switch (pass_nb(B)) {
                case 1: return F<1, 8>::run(a...);
                case 2: return F<2, 8>::run(a...);
                case 4: return F<4, 8>::run(a...);
                case 8: return F<8, 8>::run(a...);
                default: return F<16, 8>::run(a...);
            }
        default:
            switch (pass_nb(B)) {
                case 1: return F<1, 4>::run(a...);
                case 2: return F<2, 4>::run(a...);
                case 4: return F<4, 4>::run(a...);
                case 8: return F<8, 4>::run(a...);
                default: return F<16, 4>::run(a...);
            }
    }
}
template <int NB, int WB> struct QprojF {
    template <typename... A> static cudaError_t run(A &&...a) { return qproj_nb<NB, WB>(a...); }
};
template <int NB, int WB> struct QabsorbF {
    template <typename... A> static cudaError_t run(A &&...a) { return qabsorb_nb<NB, WB>(a...); }
};
template <int NB, int WB> struct CombineF {
    template <typename... A> static cudaError_t run(A &&...a) { return combine_nb<NB, WB>(a...); }
};

}  // namespace

bool qproj_fresh_supported(const CacheView &c, const UpW &Uq) {
    return c.B <= kFreshMaxB && Uq.bits == 16 && c.r <= 4 * 256 * kFreshQuads;
}

cudaError_t launch_qproj(const CacheView &c, const int32_t *seq_len, const UpW &Uq, int d, float *q,
                         unsigned *qmax, int n_qmax, int *err, cudaStream_t s, const float *c_hat, float lat_clip) {
    const int rs = c.r / kCl, ncol = qproj_cols(c.r);
    if (c_hat && !qproj_fresh_supported(c, Uq)) return cudaErrorInvalidValue;
    CUtensorMap map;
    if (!up_map(&map, Uq, c.r, d, ncol, box_rows(rs))) return cudaErrorInvalidValue;
    cudaError_t e;
    if (c_hat) {
        switch (pass_nb(c.B)) {
            case 1: e = qproj_nb<1, 16, true>(map, Uq, c, seq_len, d, q, qmax, n_qmax, err, s, c_hat, lat_clip); break;
            case 2: e = qproj_nb<2, 16, true>(map, Uq, c, seq_len, d, q, qmax, n_qmax, err, s, c_hat, lat_clip); break;
            default: e = qproj_nb<4, 16, true>(map, Uq, c, seq_len, d, q, qmax, n_qmax, err, s, c_hat, lat_clip); break;
        }
    } else {
        e = dispatch_nb_wb<QprojF>(c.B, Uq.bits, map, Uq, c, seq_len, d, q, qmax, n_qmax, err, s);
    }
    prof_mark(s, "qproj");
    return e;
}

cudaError_t launch_qabsorb(const float *q, const UpW &Uk, int B, int r, int d, int H, int dh, float *qt,
                           unsigned *qmax, int *err, cudaStream_t s) {
    const cudaError_t e = dispatch_nb_wb<QabsorbF>(B, Uk.bits, q, Uk, B, r, d, H, dh, qt, qmax, err, s);
    prof_mark(s, "qabsorb");
    return e;
}

cudaError_t launch_combine_uv(const int32_t *seq_len, const int32_t *seq_map, int nseq, int B, int Tmax, int H, int dh,
                              int r, int chunk, int n_split, const float *pm, const float *pl, const float *po,
                              const UpW &Uv, float *O, int *err, cudaStream_t s) {
    const int rs = r / kCl, d = H * dh;
    CUtensorMap map;
    if (!up_map(&map, Uv, r, d, dh, box_rows(rs))) return cudaErrorInvalidValue;
    const cudaError_t e = dispatch_nb_wb<CombineF>(B, Uv.bits, map, Uv, seq_len, seq_map, nseq, B, Tmax, H, dh, r,
                                                   chunk, n_split, pm, pl, po, O, err, s);
    prof_mark(s, "combine_uv");
    return e;
}

}  // namespace qsvd
