// Tensor-core forms of the per-step up-projection products (a5, a8) for
// batches of 5 or more sequences.  The batch rows are the M dimension of
// mma.sync.m16n8k16 (16 rows per pass), the bf16 up-projection is the B
// operand, read from its shared-memory tile with ldmatrix, and fp32
// activations are split into a bf16 part and a bf16 residual (two MMAs; the
// pair carries about 16 significant bits, products are exact, sums fp32).
// Integer latent codes are exact in bf16 and their scales multiply the fp32
// sums per 128-channel group.
//
//   qproj_mma_kernel    q[b] = c_{L_b - 1} U_q             (K = r split over a cluster of 4)
//   qabsorb_mma_kernel  q~[b, h, j] = U_k[j, h-block] . q[b, h-block], and max |q~| per (b, h)
//   combine_mma_kernel  merge the split partials, o[b, h-block] = o_lat[b, h] U_v[:, h-block]
//                       (K = r split over a cluster of 8)
//
// Like the CUDA-core kernels they replace at these batch sizes, each copies
// its weight tile before waiting on the producer grid, and the cluster
// partials are added in rank order (deterministic sums).  Grid z runs the
// 16-sequence passes side by side (each pass re-reads its weight tile from L2).
#include <cfloat>
#include <cuda_bf16.h>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

namespace {

constexpr int kClQ = 4;          // qproj: CTAs per cluster (split of the r latent rows)
constexpr int kClV = 8;          // combine: CTAs per cluster
constexpr int kMaxSplitsM = 64;  // softmax partials per sequence
constexpr int kCmbRows = 64;     // combine: U_v rows per ring slot
// Ring slots (128-row groups) of the query projection's U_q stream: three
// while a third of an SM holds them beside the codes (rs <= 512), else two;
// never more than the groups.
__host__ __device__ constexpr int qp_slots(int rs) {
    const int want = rs <= 512 ? 3 : 2, groups = rs / 128;
    return groups < want ? groups : want;
}
// Ring slots of the combine's U_v stream: three while they fit beside the
// merged rows in a third of an SM's shared memory (rs <= 192), else two; never
// more than the chunks.
__host__ __device__ constexpr int cmb_slots(int rs) {
    const int want = rs <= 3 * kCmbRows ? 3 : 2, chunks = rs / kCmbRows;
    return chunks < want ? chunks : want;
}

__device__ __forceinline__ uint32_t mrank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void msync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ float mld_rank(const float *p, uint32_t rank) {
    uint32_t a;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(a) : "r"(smem_addr(p)), "r"(rank));
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
    return v;
}
__device__ __forceinline__ void mcp16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void *p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_addr(p)));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void *p) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(smem_addr(p)));
}
__device__ __forceinline__ void mma_bf16(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// (x, y) -> bf16 pair rounded to nearest, and the bf16 pair of the residuals.
__device__ __forceinline__ void split2(float x, float y, uint32_t &hi, uint32_t &lo) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
    const float2 hf = __bfloat1622float2(h);
    const __nv_bfloat162 l = __floats2bfloat162_rn(x - hf.x, y - hf.y);
    hi = *reinterpret_cast<const uint32_t *>(&h);
    lo = *reinterpret_cast<const uint32_t *>(&l);
}
__device__ __forceinline__ uint32_t bf16pair(float x, float y) {
    const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
    return *reinterpret_cast<const uint32_t *>(&h);
}
__device__ __forceinline__ bool mlen_ok(int L, int Tmax) { return L >= 1 && L <= Tmax; }

}  // namespace

// ---------------------------------------------------------------------------
// a5, q = c U_q.  Grid (kClQ, d / 64, B / 16), cluster (kClQ, 1, 1), 128 threads.
// CTA k of a cluster takes latent rows [k rs, (k+1) rs) (rs = r / kClQ, whole
// 128-channel groups) and the cluster's 64 columns; warp w computes columns
// 16w .. 16w+15 for the 16 sequences of its pass (grid z); rank k adds the kClQ
// partials of columns 16k .. 16k+15 in rank order.  CTA (0, 0) also clears
// qmax.  The U_q rows stream through a ring of qp_slots(rs) slots of one
// 128-row group each (the first slots are copied before the wait on the
// producer grid), so three CTAs share an SM at every rank up to 3072.
// ---------------------------------------------------------------------------
__global__ void __cluster_dims__(kClQ, 1, 1) __launch_bounds__(128)
qproj_mma_kernel(const uint16_t *__restrict__ Uq, CacheView c, const int32_t *__restrict__ seq_len, int B, int d,
                 float *__restrict__ q, unsigned *__restrict__ qmax, int n_qmax, int *err) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int L_s[16], Q_s[16];   // length and cache sequence of each row
    const int r = c.r, rs = r / kClQ, ngl = rs / 128;
    const uint32_t rank = mrank();
    const int c0 = blockIdx.y * 64, j0 = int(rank) * rs;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    constexpr int kUS = 72;                                                  // padded U row (bf16)
    const int kAS = rs + 8;                                                  // padded A row (bf16)
    const int n_slots = qp_slots(rs);
    uint16_t *u_s = reinterpret_cast<uint16_t *>(smem);                      // [n_slots][128][kUS]
    uint16_t *a_s = u_s + size_t(n_slots) * 128 * kUS;                       // [16][kAS]
    float *sc_s = reinterpret_cast<float *>(a_s + 16 * kAS);                 // [16][ngl]
    float *part = reinterpret_cast<float *>(smem);                           // [16][64], over the ring once it is dead
    auto load_group = [&](int g) {                   // U_q rows [j0 + 128 g, +128), the cluster's 64 columns
        uint16_t *dst = u_s + size_t(g % n_slots) * 128 * kUS;
        for (int i = tid; i < 128 * 8; i += 128) {
            const int row = i >> 3, k = i & 7;
            mcp16(dst + size_t(row) * kUS + 8 * k, Uq + size_t(j0 + g * 128 + row) * d + c0 + 8 * k);
        }
    };
    for (int g = 0; g < n_slots; ++g) {              // one commit group per slot (U_q is no kernel's output)
        load_group(g);
        asm volatile("cp.async.commit_group;" ::: "memory");
    }
    pdl_wait();
    pdl_trigger();   // after the wait: the attention kernel two launches on reads the
                     // lengths before its own wait, and they are complete by then
    if (rank == 0 && blockIdx.y == 0 && blockIdx.z == 0)
        for (int i = tid; i < n_qmax; i += 128) qmax[i] = 0u;
    {
        const int b0 = 16 * int(blockIdx.z), nb = min(16, B - b0);
        if (tid < 16) {
            int L = tid < nb ? seq_len[b0 + tid] : 0;
            const int sq = tid < nb ? view_seq(c, b0 + tid) : 0;
            if (tid < nb && (sq < 0 || !mlen_ok(L, c.Tmax))) {
                if (rank == 0 && blockIdx.y == 0) flag_error(err, kErrRange);
                L = 0;
            }
            L_s[tid] = L;
            Q_s[tid] = sq;
        }
        __syncthreads();
        // A: the codes of row c_{L-1} in bf16 (exact); rows without a token are zero
        if (c.bits == 8) {
            for (int i = tid; i < 16 * (rs / 16); i += 128) {
                const int row = i / (rs / 16), ch = i - row * (rs / 16);
                const int L = L_s[row];
                uint4 w = make_uint4(0u, 0u, 0u, 0u);
                if (L > 0)
                    w = *reinterpret_cast<const uint4 *>(static_cast<const int8_t *>(c.codes) +
                                                         (size_t(Q_s[row]) * c.Tmax + L - 1) * r + j0 + 16 * ch);
                const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
                uint32_t o[8];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    o[2 * e] = bf16pair(float(int8_t(ww[e] & 0xff)), float(int8_t((ww[e] >> 8) & 0xff)));
                    o[2 * e + 1] = bf16pair(float(int8_t((ww[e] >> 16) & 0xff)), float(int8_t(ww[e] >> 24)));
                }
                uint4 *dst = reinterpret_cast<uint4 *>(a_s + size_t(row) * kAS + 16 * ch);
                dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
                dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
            }
            for (int i = tid; i < 16 * ngl; i += 128) {
                const int row = i / ngl;
                const int L = L_s[row];
                sc_s[i] = L > 0 ? static_cast<const float *>(c.scales)[size_t(Q_s[row]) * c.Tmax + L - 1] : 0.0f;
            }
        } else {
            for (int i = tid; i < 16 * (rs / 32); i += 128) {
                const int row = i / (rs / 32), ch = i - row * (rs / 32);
                const int L = L_s[row];
                uint4 w = make_uint4(0u, 0u, 0u, 0u);
                if (L > 0)
                    w = *reinterpret_cast<const uint4 *>(static_cast<const uint8_t *>(c.codes) +
                                                         (size_t(Q_s[row]) * c.Tmax + L - 1) * (r / 2) + j0 / 2 +
                                                         16 * ch);
                const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
                uint4 *dst = reinterpret_cast<uint4 *>(a_s + size_t(row) * kAS + 32 * ch);
#pragma unroll
                for (int e = 0; e < 4; ++e) {            // 8 codes, element i in bits 4i..4i+3
                    uint32_t o[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        o[k] = bf16pair(float((int((ww[e] >> (8 * k)) & 0xf) ^ 8) - 8),
                                        float((int((ww[e] >> (8 * k + 4)) & 0xf) ^ 8) - 8));
                    dst[e] = make_uint4(o[0], o[1], o[2], o[3]);
                }
            }
            for (int i = tid; i < 16 * ngl; i += 128) {
                const int row = i / ngl, g = i - row * ngl;
                const int L = L_s[row];
                sc_s[i] = L > 0 ? __half2float(static_cast<const __half *>(c.scales)[(size_t(Q_s[row]) * c.Tmax + L - 1) *
                                                                                     (r / 128) + j0 / 128 + g])
                                : 0.0f;
            }
        }
        // 16 rows x 16 columns per warp: per 128-channel group, fp32 sums scaled by the group's scale
        float out[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
        const int g8 = lane >> 2;
        for (int g = 0; g < ngl; ++g) {
            // group g is commit group g; the n_slots - 1 younger groups may still be in flight
            if (n_slots == 3) asm volatile("cp.async.wait_group 2;" ::: "memory");
            else if (n_slots == 2) asm volatile("cp.async.wait_group 1;" ::: "memory");
            else asm volatile("cp.async.wait_group 0;" ::: "memory");
            __syncthreads();                         // the group (and, the first time, the codes) visible
            const uint16_t *us = u_s + size_t(g % n_slots) * 128 * kUS;
            float acc[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
            for (int ks = 0; ks < 8; ++ks) {
                const int k = g * 128 + ks * 16;
                uint32_t bfr[4], afr[4];
                ldsm_x4_t(bfr, us + size_t(ks * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * kUS + 16 * warp + (lane >> 4) * 8);
                ldsm_x4(afr, a_s + size_t(lane & 15) * kAS + k + (lane >> 4) * 8);
                mma_bf16(acc[0], afr, bfr[0], bfr[1]);
                mma_bf16(acc[1], afr, bfr[2], bfr[3]);
            }
            const float s_lo = sc_s[g8 * ngl + g], s_hi = sc_s[(g8 + 8) * ngl + g];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
                out[nt][0] = fmaf(s_lo, acc[nt][0], out[nt][0]);
                out[nt][1] = fmaf(s_lo, acc[nt][1], out[nt][1]);
                out[nt][2] = fmaf(s_hi, acc[nt][2], out[nt][2]);
                out[nt][3] = fmaf(s_hi, acc[nt][3], out[nt][3]);
            }
            if (g + n_slots < ngl) {
                __syncthreads();                     // every warp is done with the slot
                load_group(g + n_slots);
            }
            asm volatile("cp.async.commit_group;" ::: "memory");
        }
        __syncthreads();                             // the ring is dead: part takes its first bytes
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
            const int col = 16 * warp + 8 * nt + 2 * (lane & 3);
            *reinterpret_cast<float2 *>(part + g8 * 64 + col) = make_float2(out[nt][0], out[nt][1]);
            *reinterpret_cast<float2 *>(part + (g8 + 8) * 64 + col) = make_float2(out[nt][2], out[nt][3]);
        }
        msync();                                     // every rank's partials are complete
        for (int o = tid; o < nb * 16; o += 128) {
            const int row = o >> 4, col = int(rank) * 16 + (o & 15);
            float v = 0.0f;
#pragma unroll
            for (int k = 0; k < kClQ; ++k) v += mld_rank(part + row * 64 + col, uint32_t(k));
            q[size_t(b0 + row) * d + c0 + col] = v;
        }
        msync();                                     // partials read before the CTA exits
    }
}

// ---------------------------------------------------------------------------
// a5, q~ = U_k q.  Grid (r / 128, H, B / 16), 128 threads: CTA (x, h) computes q~[b, h, j]
// for j in [128 x, 128 x + 128), warp w the 32 columns 32w .. 32w+31.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128)
qabsorb_mma_kernel(const float *q, const uint16_t *__restrict__ Uk, int B, int r, int d, int H, int dh,
                   float *__restrict__ qt, unsigned *__restrict__ qmax) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ float mx_s[4][16];
    const int j0 = blockIdx.x * 128, h = blockIdx.y;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g8 = lane >> 2;
    const int kS = dh + 8;                                                   // padded rows (bf16)
    uint16_t *u_s = reinterpret_cast<uint16_t *>(smem);                      // [128 j][kS]
    uint16_t *ah_s = u_s + 128 * kS;                                         // [16][kS]
    uint16_t *al_s = ah_s + 16 * kS;                                         // [16][kS]
    for (int i = tid; i < 128 * (dh / 8); i += 128) {    // U_k rows: no kernel's output, copied before the wait
        const int row = i / (dh / 8), k = i - row * (dh / 8);
        mcp16(u_s + size_t(row) * kS + 8 * k, Uk + size_t(j0 + row) * d + size_t(h) * dh + 8 * k);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    pdl_wait();
    pdl_trigger();   // after the wait: the attention kernel two launches on reads the
                     // lengths before its own wait, and they are complete by then
    bool ready = false;
    for (int b0 = 16 * int(blockIdx.z); b0 < B; b0 += 16 * int(gridDim.z)) {   // grid z: 16-sequence passes
        const int nb = min(16, B - b0);
        __syncthreads();
        for (int i = tid; i < 16 * (dh / 4); i += 128) {     // A: q[b, h-block] as bf16 part + residual
            const int row = i / (dh / 4), c4 = i - row * (dh / 4);
            const float4 v = row < nb ? reinterpret_cast<const float4 *>(q + size_t(b0 + row) * d + size_t(h) * dh)[c4]
                                      : make_float4(0.f, 0.f, 0.f, 0.f);
            uint32_t h0, l0, h1, l1;
            split2(v.x, v.y, h0, l0);
            split2(v.z, v.w, h1, l1);
            *reinterpret_cast<uint2 *>(ah_s + size_t(row) * kS + 4 * c4) = make_uint2(h0, h1);
            *reinterpret_cast<uint2 *>(al_s + size_t(row) * kS + 4 * c4) = make_uint2(l0, l1);
        }
        if (!ready) {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
            ready = true;
        }
        __syncthreads();
        float acc[4][4];
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.0f;
        for (int ks = 0; ks < dh / 16; ++ks) {
            uint32_t ah[4], al[4];
            ldsm_x4(ah, ah_s + size_t(lane & 15) * kS + ks * 16 + (lane >> 4) * 8);
            ldsm_x4(al, al_s + size_t(lane & 15) * kS + ks * 16 + (lane >> 4) * 8);
#pragma unroll
            for (int p = 0; p < 2; ++p) {                    // 16 columns (two n8 tiles) per ldmatrix
                uint32_t bfr[4];
                ldsm_x4(bfr, u_s + size_t(32 * warp + 16 * p + (lane & 7) + (lane >> 4) * 8) * kS + ks * 16 +
                                 ((lane >> 3) & 1) * 8);
                mma_bf16(acc[2 * p], ah, bfr[0], bfr[1]);
                mma_bf16(acc[2 * p], al, bfr[0], bfr[1]);
                mma_bf16(acc[2 * p + 1], ah, bfr[2], bfr[3]);
                mma_bf16(acc[2 * p + 1], al, bfr[2], bfr[3]);
            }
        }
        // rows g8 / g8 + 8; columns 32w + 8nt + 2(lane%4) (+1)
        float m0 = 0.0f, m1 = 0.0f;
#pragma unroll
        for (int nt = 0; nt < 4; ++nt) {
            const int col = j0 + 32 * warp + 8 * nt + 2 * (lane & 3);
            if (g8 < nb)
                *reinterpret_cast<float2 *>(qt + (size_t(b0 + g8) * H + h) * r + col) = make_float2(acc[nt][0], acc[nt][1]);
            if (g8 + 8 < nb)
                *reinterpret_cast<float2 *>(qt + (size_t(b0 + g8 + 8) * H + h) * r + col) = make_float2(acc[nt][2], acc[nt][3]);
            m0 = fmaxf(m0, fmaxf(fabsf(acc[nt][0]), fabsf(acc[nt][1])));
            m1 = fmaxf(m1, fmaxf(fabsf(acc[nt][2]), fabsf(acc[nt][3])));
        }
        m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, 1));
        m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, 2));
        m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, 1));
        m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, 2));
        if ((lane & 3) == 0) {
            mx_s[warp][g8] = m0;
            mx_s[warp][g8 + 8] = m1;
        }
        __syncthreads();
        if (tid < nb) {
            const float m = fmaxf(fmaxf(mx_s[0][tid], mx_s[1][tid]), fmaxf(mx_s[2][tid], mx_s[3][tid]));
            atomicMax(qmax + size_t(b0 + tid) * H + h, __float_as_uint(m));
        }
    }
}

// ---------------------------------------------------------------------------
// a7/a8.  Grid (kClV, H, B / 16), cluster (kClV, 1, 1), 128 threads.  CTA k of
// head h's cluster merges, for the 16 sequences of its pass (grid z), the
// softmax partials of latent rows [k rs, (k+1) rs) (weights exp(m_s - M) / l),
// multiplies them by those rows of U_v[:, h-block] (warp w: output columns
// 32w .. 32w+31), and rank k adds the kClV products of columns k dh/kClV .. in
// rank order.  The U_v rows stream through a ring of cmb_slots(rs) slots of
// kCmbRows rows (the first slots are copied before the wait on the producer
// grid), so a CTA holds at most ~70 KB of shared memory at every rank up to
// 3072: three CTAs share an SM and the grid runs as one wave.  Every load of
// the merge is issued before its results are used (the merge weights of four
// sequences per warp, the partials of two outputs per thread).
// ---------------------------------------------------------------------------
__global__ void __cluster_dims__(kClV, 1, 1) __launch_bounds__(128)
combine_mma_kernel(const uint16_t *__restrict__ Uv, const int32_t *__restrict__ seq_len,
                   const int32_t *__restrict__ seq_map, int nseq, int B, int Tmax, int H,
                   int dh, int r, int chunk, int n_split, const float *pm, const float *pl,
                   const float *po, float *__restrict__ O) {
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ float inv_s[16];
    __shared__ int ns_s[16];
    const int rs = r / kClV, d = H * dh, h = blockIdx.y;
    const int n_ck = rs / kCmbRows, n_slots = cmb_slots(rs);
    const uint32_t rank = mrank();
    const int j0 = int(rank) * rs;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g8 = lane >> 2;
    const int kS = dh + 8, kAS = rs + 8;
    uint16_t *u_s = reinterpret_cast<uint16_t *>(smem);                      // [n_slots][kCmbRows][kS]
    uint16_t *ah_s = u_s + size_t(n_slots) * kCmbRows * kS;                  // [16][kAS]
    uint16_t *al_s = ah_s + 16 * kAS;                                        // [16][kAS]
    float *part = reinterpret_cast<float *>(al_s + 16 * kAS);                // [16][dh]
    float *w_s = part;           // [16][kMaxSplitsM] merge weights, dead before part is written
    const int b0 = 16 * int(blockIdx.z), nb = min(16, B - b0);
    auto load_chunk = [&](int ck) {                  // U_v rows [j0 + 64 ck, +64) of head h's columns
        uint16_t *dst = u_s + size_t(ck % n_slots) * kCmbRows * kS;
        const uint16_t *src = Uv + size_t(j0 + ck * kCmbRows) * d + size_t(h) * dh;
        for (int i = tid; i < kCmbRows * (dh / 8); i += 128) {
            const int row = i / (dh / 8), k = i - row * (dh / 8);
            mcp16(dst + size_t(row) * kS + 8 * k, src + size_t(row) * d + 8 * k);
        }
    };
    pdl_trigger();
    for (int ck = 0; ck < n_slots; ++ck) {           // one commit group per slot (U_v is no kernel's output)
        if (ck < n_ck) load_chunk(ck);
        asm volatile("cp.async.commit_group;" ::: "memory");
    }
    pdl_wait();
    // merge weights: warp w takes sequences w, w+4, w+8, w+12; the entries past a
    // row's splits (allocated, possibly stale) are loaded with the others and masked
    {
        int Lk[4];
        float mk[4][2], lk[4][2];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int bi = warp + 4 * k;
            const bool row = bi < nb;
            Lk[k] = row ? row_len(seq_len, seq_map, nseq, b0 + bi) : 0;
            const size_t base = size_t(b0 + (row ? bi : 0)) * n_split * H + h;
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int s = lane + 32 * u;
                const bool ok = row && s < n_split;
                mk[k][u] = ok ? pm[base + size_t(s) * H] : -FLT_MAX;
                lk[k][u] = ok ? pl[base + size_t(s) * H] : 0.0f;
            }
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int bi = warp + 4 * k;
            const int L = Lk[k];
            const int ns = mlen_ok(L, Tmax) ? min((L + chunk - 1) / chunk, n_split) : 0;
            const float m0 = lane < ns ? mk[k][0] : -FLT_MAX, m1 = lane + 32 < ns ? mk[k][1] : -FLT_MAX;
            const float M = warp_max(fmaxf(m0, m1));
            const float e0 = lane < ns ? expf(m0 - M) : 0.0f;
            const float e1 = lane + 32 < ns ? expf(m1 - M) : 0.0f;
            w_s[bi * kMaxSplitsM + lane] = e0;
            w_s[bi * kMaxSplitsM + lane + 32] = e1;
            const float l = warp_sum((lane < ns ? e0 * lk[k][0] : 0.0f) + (lane + 32 < ns ? e1 * lk[k][1] : 0.0f));
            if (lane == 0) {
                inv_s[bi] = ns ? 1.0f / l : 0.0f;
                ns_s[bi] = ns;
            }
        }
    }
    __syncthreads();
    // merged o_lat rows (this rank's channels) as bf16 part + residual, two outputs per thread
    const int nq = rs / 4;
    for (int it0 = tid; it0 < 16 * nq; it0 += 256) {
        int bi[2], q4[2], ns[2];
        float4 acc[2];
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            const int it = it0 + 128 * u;
            const bool live = it < 16 * nq;
            bi[u] = live ? it / nq : 0;
            q4[u] = live ? it - bi[u] * nq : 0;
            ns[u] = live ? ns_s[bi[u]] : 0;
            acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
        const int nsm = max(ns[0], ns[1]);
        for (int s0 = 0; s0 < nsm; s0 += 8) {
            float4 v[2][8];
            float wk[2][8];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const float *src = po + (size_t(b0 + bi[u]) * n_split * H + h) * r + j0 + 4 * q4[u];
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const int sk = s0 + k;
                    const bool ok = sk < ns[u];
                    v[u][k] = ok ? *reinterpret_cast<const float4 *>(src + size_t(sk) * H * r) : make_float4(0.f, 0.f, 0.f, 0.f);
                    wk[u][k] = ok ? w_s[bi[u] * kMaxSplitsM + sk] : 0.0f;
                }
            }
#pragma unroll
            for (int u = 0; u < 2; ++u)
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    acc[u].x = fmaf(wk[u][k], v[u][k].x, acc[u].x);
                    acc[u].y = fmaf(wk[u][k], v[u][k].y, acc[u].y);
                    acc[u].z = fmaf(wk[u][k], v[u][k].z, acc[u].z);
                    acc[u].w = fmaf(wk[u][k], v[u][k].w, acc[u].w);
                }
        }
#pragma unroll
        for (int u = 0; u < 2; ++u) {
            if (it0 + 128 * u >= 16 * nq) break;
            const float il = inv_s[bi[u]];
            uint32_t h0, l0, h1, l1;
            split2(acc[u].x * il, acc[u].y * il, h0, l0);
            split2(acc[u].z * il, acc[u].w * il, h1, l1);
            *reinterpret_cast<uint2 *>(ah_s + size_t(bi[u]) * kAS + 4 * q4[u]) = make_uint2(h0, h1);
            *reinterpret_cast<uint2 *>(al_s + size_t(bi[u]) * kAS + 4 * q4[u]) = make_uint2(l0, l1);
        }
    }
    float acc[4][4];
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.0f;
    for (int ck = 0; ck < n_ck; ++ck) {
        // chunk ck is commit group ck; the n_slots - 1 younger groups may still be in flight
        if (n_slots == 3) asm volatile("cp.async.wait_group 2;" ::: "memory");
        else if (n_slots == 2) asm volatile("cp.async.wait_group 1;" ::: "memory");
        else asm volatile("cp.async.wait_group 0;" ::: "memory");
        __syncthreads();                             // the chunk (and, the first time, the merged rows) visible
        const uint16_t *us = u_s + size_t(ck % n_slots) * kCmbRows * kS;
#pragma unroll
        for (int kl = 0; kl < kCmbRows / 16; ++kl) {
            const int ks = ck * (kCmbRows / 16) + kl;
            uint32_t ah[4], al[4];
            ldsm_x4(ah, ah_s + size_t(lane & 15) * kAS + ks * 16 + (lane >> 4) * 8);
            ldsm_x4(al, al_s + size_t(lane & 15) * kAS + ks * 16 + (lane >> 4) * 8);
#pragma unroll
            for (int p = 0; p < 2; ++p) {
                uint32_t bfr[4];
                ldsm_x4_t(bfr, us + size_t(kl * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * kS + 32 * warp + 16 * p +
                                   (lane >> 4) * 8);
                mma_bf16(acc[2 * p], ah, bfr[0], bfr[1]);
                mma_bf16(acc[2 * p], al, bfr[0], bfr[1]);
                mma_bf16(acc[2 * p + 1], ah, bfr[2], bfr[3]);
                mma_bf16(acc[2 * p + 1], al, bfr[2], bfr[3]);
            }
        }
        if (ck + n_slots < n_ck) {
            __syncthreads();                         // every warp is done with the slot
            load_chunk(ck + n_slots);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    }
    __syncthreads();                                 // the merge weights (in part) are dead
#pragma unroll
    for (int nt = 0; nt < 4; ++nt) {
        const int col = 32 * warp + 8 * nt + 2 * (lane & 3);
        *reinterpret_cast<float2 *>(part + g8 * dh + col) = make_float2(acc[nt][0], acc[nt][1]);
        *reinterpret_cast<float2 *>(part + (g8 + 8) * dh + col) = make_float2(acc[nt][2], acc[nt][3]);
    }
    msync();                                         // every rank's products are complete
    const int per_rank = dh / kClV;
    for (int o = tid; o < nb * per_rank; o += 128) {
        const int bi = o / per_rank, cc = int(rank) * per_rank + (o - bi * per_rank);
        float v = 0.0f;
#pragma unroll
        for (int k = 0; k < kClV; ++k) v += mld_rank(part + bi * dh + cc, uint32_t(k));
        O[size_t(b0 + bi) * d + size_t(h) * dh + cc] = v;
    }
    msync();                                         // partials read before the CTA exits
}

// ---------------------------------------------------------------------------
// Shapes these kernels take: 5 or more sequences, r % 512 == 0 (whole 128-channel
// groups per qproj rank), dh == 128 (four warps of 32 output columns in combine).
// From 5 sequences on they beat the CUDA-core forms (measured on GB300: whole
// decode steps at B = 5 and 6 are 12-17 % faster; at B = 4 the CUDA-core forms
// win at r = 3072 and at long caches).
bool decode_mma_supported(int B, int r, int d, int dh) {
    return B >= 5 && r % 512 == 0 && d % 64 == 0 && dh == 128;
}

cudaError_t launch_qproj_mma(const CacheView &c, const int32_t *seq_len, const uint16_t *Uq, int d, float *q,
                             unsigned *qmax, int n_qmax, int *err, cudaStream_t s) {
    const int rs = c.r / kClQ;
    const size_t smem = size_t(qp_slots(rs)) * 128 * 72 * 2 + size_t(16) * (rs + 8) * 2 + size_t(16) * (rs / 128) * 4;
    cudaError_t e = ensure_smem(qproj_mma_kernel, smem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(qproj_mma_kernel, dim3(kClQ, d / 64, (c.B + 15) / 16), dim3(128), smem, s, Uq, c, seq_len, c.B, d, q, qmax, n_qmax,
                   err);
    prof_mark(s, "qproj");
    return e;
}

cudaError_t launch_qabsorb_mma(const float *q, const uint16_t *Uk, int B, int r, int d, int H, int dh, float *qt,
                               unsigned *qmax, cudaStream_t s) {
    const size_t smem = size_t(128 + 32) * (dh + 8) * 2;
    cudaError_t e = ensure_smem(qabsorb_mma_kernel, smem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(qabsorb_mma_kernel, dim3(r / 128, H, (B + 15) / 16), dim3(128), smem, s, q, Uk, B, r, d, H, dh, qt, qmax);
    prof_mark(s, "qabsorb");
    return e;
}

cudaError_t launch_combine_mma(const int32_t *seq_len, const int32_t *seq_map, int nseq, int B, int Tmax, int H, int dh, int r, int chunk, int n_split,
                               const float *pm, const float *pl, const float *po, const uint16_t *Uv, float *O,
                               cudaStream_t s) {
    const int rs = r / kClV;
    const size_t smem = size_t(cmb_slots(rs)) * kCmbRows * (dh + 8) * 2 + size_t(32) * (rs + 8) * 2 +
                        size_t(16) * dh * 4;
    cudaError_t e = ensure_smem(combine_mma_kernel, smem);
    if (e != cudaSuccess) return e;
    e = launch_pdl(combine_mma_kernel, dim3(kClV, H, (B + 15) / 16), dim3(128), smem, s, Uv, seq_len, seq_map, nseq, B, Tmax, H, dh, r, chunk,
                   n_split, pm, pl, po, O);
    prof_mark(s, "combine_uv");
    return e;
}

}  // namespace qsvd
