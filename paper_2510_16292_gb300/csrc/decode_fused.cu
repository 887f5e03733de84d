// One decode step of the whole path (a1-a8) in a single persistent launch,
// for small batches (one new token per sequence, B <= kFuseMaxB).
//
// A cooperative grid of one CTA per SM runs five phases separated by grid
// barriers (bounded spin waits that flag a timeout and abandon the step):
//   P1  a1+a2+a3a  every CTA quantizes the B new tokens itself; CTA k computes
//                  the exact int8 dot products of its slice of W_d's output
//                  channels and the fp32 dequantized latent c_hat.
//   P2  a3b+a4+a5a every CTA requantizes the full latent rows (per-token
//                  scale, or fp16 scale per 128-channel group), stores its
//                  channel slice of each row into the cache, and computes its
//                  column slice of q = c_last U_q.
//   P3  a5b        CTA k computes q~[b, h, j] = U_k[j, h-block] . q_h for its
//                  slice of rows j.
//   P4  a6+a7      (sequence, token chunk, head pair) tasks: online-softmax pass
//                  over the chunk's cache rows -> (max, sum, sum_t p_t c_t).
//   P5  a7+a8      (head, 128-row block of U_v) tasks: merge the chunk partials,
//                  normalise, multiply by the U_v block; the last task of a
//                  head sums the blocks in order.
// Before its first barrier every CTA prefetches its share of W_d, U_q, U_k
// and U_v into L2, so the weight stream overlaps the whole dependency chain.
#include <cfloat>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

constexpr int kFuseThreads = 256;
constexpr int kFuseMaxD = 6144;
constexpr int kFuseSplits = 64;     // token chunks per sequence at most
constexpr int kFuseHG = 2;          // heads per attention task
constexpr int kFuseSub = 16;        // cache rows per attention sub-tile
constexpr int kFuseRowBlock = 128;  // U_v rows per combine task
constexpr int kFuseMaxRank = 3072;

static inline size_t f_align256(size_t x) { return (x + 255) & ~size_t(255); }

static int fuse_chunk(int max_seq_len) {
    int c = 32;
    while ((max_seq_len + c - 1) / c > kFuseSplits) c += 32;
    return c;
}

struct FuseWs {
    unsigned *bar;      // [0] arrival count, [1] generation
    int *head_count;    // [H]
    float *c_hat, *q, *qt, *pm, *pl, *po, *opart;
};

static size_t fuse_carve(int B, int max_seq_len, int d, int r, int H, int dh, char *base, FuseWs *w) {
    const int chunk = fuse_chunk(max_seq_len);
    const int ns = (max_seq_len + chunk - 1) / chunk;
    const int nrb = (r + kFuseRowBlock - 1) / kFuseRowBlock;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *p = base ? base + off : nullptr;
        off += f_align256(bytes);
        return p;
    };
    FuseWs t;
    t.bar = reinterpret_cast<unsigned *>(take(64));
    t.head_count = reinterpret_cast<int *>(take(size_t(H) * 4));
    t.c_hat = reinterpret_cast<float *>(take(size_t(B) * r * 4));
    t.q = reinterpret_cast<float *>(take(size_t(B) * d * 4));
    t.qt = reinterpret_cast<float *>(take(size_t(B) * H * r * 4));
    t.pm = reinterpret_cast<float *>(take(size_t(B) * ns * H * 4));
    t.pl = reinterpret_cast<float *>(take(size_t(B) * ns * H * 4));
    t.po = reinterpret_cast<float *>(take(size_t(B) * ns * H * r * 4));
    t.opart = reinterpret_cast<float *>(take(size_t(B) * H * nrb * dh * 4));
    if (w) *w = t;
    return off;
}

size_t fused_workspace_bytes(int B, int max_seq_len, int d, int r, int H, int dh) {
    return fuse_carve(B, max_seq_len, d, r, H, dh, nullptr, nullptr);
}

// Grid-wide barrier for a cooperative launch.  Returns false (and flags
// kErrTimeout) if the other CTAs did not arrive within the wait limit.
__device__ __forceinline__ bool grid_barrier(unsigned *bar, int *err) {
    __shared__ int ok;
    __syncthreads();
    if (threadIdx.x == 0) {
        ok = 1;
        volatile unsigned *vgen = bar + 1;
        const unsigned gen = *vgen;
        __threadfence();
        const unsigned arrived = atomicAdd(bar, 1u);
        if (arrived == gridDim.x - 1) {
            atomicExch(bar, 0u);
            __threadfence();
            atomicAdd(bar + 1, 1u);
        } else {
            long it = 0;
            while (*vgen == gen) {
                if (++it > (1L << 22)) {
                    flag_error(err, kErrTimeout);
                    ok = 0;
                    break;
                }
                __nanosleep(64);
            }
        }
        __threadfence();
    }
    __syncthreads();
    return ok != 0;
}

__device__ __forceinline__ float fcache_value(const CacheView &c, size_t slot, int j) {
    if (c.bits == 8) {
        const int8_t code = static_cast<const int8_t *>(c.codes)[slot * c.r + j];
        return float(code) * static_cast<const float *>(c.scales)[slot];
    }
    const uint8_t byte = static_cast<const uint8_t *>(c.codes)[slot * (c.r / 2) + (j >> 1)];
    int nib = (j & 1) ? (byte >> 4) : (byte & 0xf);
    nib = (nib ^ 8) - 8;
    return float(nib) * __half2float(static_cast<const __half *>(c.scales)[slot * (c.r / 128) + (j >> 7)]);
}

struct FuseArgs {
    const uint16_t *X;            // [B, d]
    const int8_t *w;              // [r, d]
    const float *ws;              // [r]
    CacheView c;
    const int32_t *seq_len;       // [B]
    const uint16_t *Uq, *Uk, *Uv; // [r, d]
    int B, d, H, dh, chunk, n_split;
    float act_clip, lat_clip, softmax_scale;
    float *O;                     // [B, d]
    FuseWs w_;
    int *err;
};

__global__ void __launch_bounds__(kFuseThreads, 1) decode_step_kernel(FuseArgs a) {
    extern __shared__ __align__(16) uint8_t smem[];
    __shared__ float red[kFuseThreads / 32];
    __shared__ float xs_s[kFuseMaxB];
    __shared__ float m_s[kFuseHG], l_s[kFuseHG], alpha_s[kFuseHG];
    __shared__ float wsp[kFuseSplits];
    __shared__ float inv_l;
    __shared__ int last;
    const CacheView &c = a.c;
    const int r = c.r, d = a.d, B = a.B, H = a.H, dh = a.dh;
    const int G = gridDim.x, k = blockIdx.x;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    int *err = a.err;

    // ---- prologue: L2 prefetch of this CTA's share of every weight ----------
    prefetch_share_l2(a.w, size_t(r) * d, k, G);
    prefetch_share_l2(a.Uq, size_t(r) * d * 2, k, G);
    prefetch_share_l2(a.Uk, size_t(r) * d * 2, k, G);
    prefetch_share_l2(a.Uv, size_t(r) * d * 2, k, G);
    pdl_wait();
    for (int b = 0; b < B; ++b) {
        const int L = a.seq_len[b];
        if (L < 1 || L > c.Tmax) {
            if (k == 0 && tid == 0) flag_error(err, kErrRange);
            return;                                   // uniform: every CTA sees the same lengths
        }
    }

    // ---- P1: quantize the tokens (every CTA), exact dot products of a channel slice
    int8_t *xq_s = reinterpret_cast<int8_t *>(smem);  // [B][d]
    for (int b = 0; b < B; ++b) {
        float f[kFuseMaxD / 2048][8];
        float m = 0.0f;
#pragma unroll
        for (int v = 0; v < kFuseMaxD / 2048; ++v) {
            const int col = (v * kFuseThreads + tid) * 8;
            if (col < d) {
                unpack8_bf16(*reinterpret_cast<const uint4 *>(a.X + size_t(b) * d + col), f[v]);
#pragma unroll
                for (int e = 0; e < 8; ++e) m = fmaxf(m, fabsf(f[v][e]));
            }
        }
        m = block_max<kFuseThreads>(m, red);
        const float s = quant_scale(m, a.act_clip, 127.0f);
#pragma unroll
        for (int v = 0; v < kFuseMaxD / 2048; ++v) {
            const int col = (v * kFuseThreads + tid) * 8;
            if (col < d) {
                uint32_t lo = 0, hi = 0;
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    lo |= uint32_t(quant_code(f[v][e], s, 127) & 0xff) << (8 * e);
                    hi |= uint32_t(quant_code(f[v][e + 4], s, 127) & 0xff) << (8 * e);
                }
                *reinterpret_cast<uint2 *>(xq_s + size_t(b) * d + col) = make_uint2(lo, hi);
            }
        }
        if (tid == 0) xs_s[b] = s;
    }
    __syncthreads();
    const int cpb = (r + G - 1) / G;                  // output channels per CTA
    for (int jj = warp; jj < cpb; jj += kFuseThreads / 32) {
        const int j = k * cpb + jj;
        if (j >= r) break;
        const int *wrow = reinterpret_cast<const int *>(a.w + size_t(j) * d);
        int wv[kFuseMaxD / 128];
#pragma unroll
        for (int v = 0; v < kFuseMaxD / 128; ++v)
            if (v * 32 + lane < d / 4) wv[v] = wrow[v * 32 + lane];
        const float sw = a.ws[j];
        for (int b = 0; b < B; ++b) {
            const int *xrow = reinterpret_cast<const int *>(xq_s + size_t(b) * d);
            int acc = 0;
#pragma unroll
            for (int v = 0; v < kFuseMaxD / 128; ++v)
                if (v * 32 + lane < d / 4) acc = __dp4a(wv[v], xrow[v * 32 + lane], acc);
            acc = warp_sum_int(acc);
            if (lane == 0) a.w_.c_hat[size_t(b) * r + j] = __fmul_rn(__fmul_rn(__int2float_rn(acc), xs_s[b]), sw);
        }
    }
    if (!grid_barrier(a.w_.bar, err)) return;

    // ---- P2: requantize every latent row, append own channel slice, q slice
    float *lat_s = reinterpret_cast<float *>(smem);    // [r] dequantized latent of the current b
    float *qred = lat_s + r;                            // [8 warps][32]
    const int ccols = ((d + G - 1) / G + 7) & ~7;      // q columns per CTA (multiple of 8)
    const int c0 = k * ccols;
    for (int b = 0; b < B; ++b) {
        const int L = a.seq_len[b];
        const size_t slot = size_t(b) * c.Tmax + (L - 1);
        const float *row = a.w_.c_hat + size_t(b) * r;
        __syncthreads();
        for (int j = tid; j < r; j += kFuseThreads) lat_s[j] = row[j];
        __syncthreads();
        if (c.bits == 8) {
            float m = 0.0f;
            for (int j = tid; j < r; j += kFuseThreads) m = fmaxf(m, fabsf(lat_s[j]));
            m = block_max<kFuseThreads>(m, red);
            const float s = quant_scale(m, a.lat_clip, 127.0f);
            for (int j = tid; j < r; j += kFuseThreads) {
                const int code = quant_code(lat_s[j], s, 127);
                if (j >= k * cpb && j < (k + 1) * cpb) static_cast<int8_t *>(c.codes)[slot * r + j] = int8_t(code);
                lat_s[j] = float(code) * s;
            }
            if (k == 0 && tid == 0) static_cast<float *>(c.scales)[slot] = s;
        } else {
            // one warp per 128-channel group: lane holds 4 consecutive channels
            for (int g = warp; g < r / 128; g += kFuseThreads / 32) {
                float4 v = *reinterpret_cast<const float4 *>(lat_s + g * 128 + lane * 4);
                float m = fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w)));
                m = warp_max(m);
                const __half hs = int4_group_scale(m, a.lat_clip);
                const float s = __half2float(hs);
                const int q0 = quant_code(v.x, s, 7), q1 = quant_code(v.y, s, 7);
                const int q2 = quant_code(v.z, s, 7), q3 = quant_code(v.w, s, 7);
                const int j = g * 128 + lane * 4;
                if (j >= k * cpb && j < (k + 1) * cpb) {
                    // the owner of channel j writes the packed pair bytes of j..j+3 it owns
                    const uint16_t w16 = uint16_t((q0 & 0xf) | ((q1 & 0xf) << 4) | ((q2 & 0xf) << 8) | ((q3 & 0xf) << 12));
                    reinterpret_cast<uint16_t *>(static_cast<uint8_t *>(c.codes) + slot * (r / 2))[j / 4] = w16;
                }
                if (k == 0 && lane == 0) static_cast<__half *>(c.scales)[slot * (r / 128) + g] = hs;
                *reinterpret_cast<float4 *>(lat_s + j) =
                    make_float4(float(q0) * s, float(q1) * s, float(q2) * s, float(q3) * s);
            }
        }
        __syncthreads();
        // q[b, c0 .. c0 + ccols): 256 threads = 64 row groups x 4 column octets
        if (c0 < d) {
            const int rg = tid >> 2, co = tid & 3;
            for (int cc = 0; cc < ccols; cc += 32) {
                const int col = c0 + cc + co * 8;
                float acc[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) acc[e] = 0.0f;
                if (col < min(d, c0 + ccols)) {
#pragma unroll 8
                    for (int j = rg; j < r; j += 64) {
                        float u[8];
                        unpack8_bf16(*reinterpret_cast<const uint4 *>(a.Uq + size_t(j) * d + col), u);
                        const float x = lat_s[j];
#pragma unroll
                        for (int e = 0; e < 8; ++e) acc[e] = fmaf(x, u[e], acc[e]);
                    }
                }
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    float v = acc[e];
                    v += __shfl_xor_sync(0xffffffffu, v, 4);
                    v += __shfl_xor_sync(0xffffffffu, v, 8);
                    v += __shfl_xor_sync(0xffffffffu, v, 16);
                    acc[e] = v;
                }
                __syncthreads();
                if (lane < 4)
#pragma unroll
                    for (int e = 0; e < 8; ++e) qred[warp * 32 + lane * 8 + e] = acc[e];
                __syncthreads();
                if (tid < 32) {
                    float s = 0.0f;
#pragma unroll
                    for (int w2 = 0; w2 < 8; ++w2) s += qred[w2 * 32 + tid];
                    const int oc = c0 + cc + tid;
                    if (oc < min(d, c0 + ccols)) a.w_.q[size_t(b) * d + oc] = s;
                }
            }
        }
    }
    if (!grid_barrier(a.w_.bar, err)) return;

    // ---- P3: q~ for a slice of rows of U_k
    float *q_s = reinterpret_cast<float *>(smem);      // [d]
    const int seg = dh / 8;
    for (int b = 0; b < B; ++b) {
        __syncthreads();
        for (int i = tid * 4; i < d; i += kFuseThreads * 4)
            *reinterpret_cast<float4 *>(q_s + i) = *reinterpret_cast<const float4 *>(a.w_.q + size_t(b) * d + i);
        __syncthreads();
        for (int jj = warp; jj < cpb; jj += kFuseThreads / 32) {
            const int j = k * cpb + jj;
            if (j >= r) break;
            const uint16_t *urow = a.Uk + size_t(j) * d;
#pragma unroll 4
            for (int base = 0; base < d; base += 256) {
                const int col = base + lane * 8;
                float f[8];
                unpack8_bf16(*reinterpret_cast<const uint4 *>(urow + col), f);
                const float4 q0 = *reinterpret_cast<const float4 *>(q_s + col);
                const float4 q1 = *reinterpret_cast<const float4 *>(q_s + col + 4);
                float p = f[0] * q0.x + f[1] * q0.y + f[2] * q0.z + f[3] * q0.w +
                          f[4] * q1.x + f[5] * q1.y + f[6] * q1.z + f[7] * q1.w;
                for (int o = seg >> 1; o; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
                if ((lane % seg) == 0) a.w_.qt[(size_t(b) * H + col / dh) * r + j] = p;
            }
        }
    }
    if (!grid_barrier(a.w_.bar, err)) return;

    // ---- P4: attention partials over (b, chunk, head pair) tasks
    {
        const int row_bytes = c.bits == 8 ? r : r / 2;
        float *qs = reinterpret_cast<float *>(smem);                 // [kFuseHG][r]
        float *ps = qs + kFuseHG * r;                                 // [kFuseHG][kFuseSub]
        float *tsc = ps + kFuseHG * kFuseSub;                         // [kFuseSub]
        uint8_t *tile = reinterpret_cast<uint8_t *>(tsc + kFuseSub);  // [kFuseSub][row_bytes]
        const int hgroups = (H + kFuseHG - 1) / kFuseHG;
        const int n_tasks = B * a.n_split * hgroups;
        constexpr int kQ = kFuseMaxRank / 4 / kFuseThreads;
        const int nq = r / 4;
        for (int task = k; task < n_tasks; task += G) {
            const int hgi = task % hgroups;
            const int split = (task / hgroups) % a.n_split;
            const int b = task / (hgroups * a.n_split);
            const int h0 = hgi * kFuseHG, hg = min(kFuseHG, H - h0);
            const int L = a.seq_len[b];
            const int t_begin = split * a.chunk;
            if (t_begin >= L) continue;
            const int n = min(L, t_begin + a.chunk) - t_begin;
            __syncthreads();
            for (int i = tid; i < hg * r; i += kFuseThreads) qs[i] = a.w_.qt[(size_t(b) * H + h0) * r + i];
            if (tid < kFuseHG) {
                m_s[tid] = -FLT_MAX;
                l_s[tid] = 0.0f;
            }
            float acc[kFuseHG][kQ][4];
#pragma unroll
            for (int h = 0; h < kFuseHG; ++h)
#pragma unroll
                for (int q = 0; q < kQ; ++q)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[h][q][e] = 0.0f;
            for (int t0 = 0; t0 < n; t0 += kFuseSub) {
                const int rows = min(kFuseSub, n - t0);
                const size_t slot0 = size_t(b) * c.Tmax + t_begin + t0;
                __syncthreads();
                const uint4 *src = reinterpret_cast<const uint4 *>(static_cast<const uint8_t *>(c.codes) + slot0 * row_bytes);
                for (int i = tid; i < rows * row_bytes / 16; i += kFuseThreads)
                    reinterpret_cast<uint4 *>(tile)[i] = src[i];
                if (c.bits == 8 && tid < rows) tsc[tid] = static_cast<const float *>(c.scales)[slot0 + tid];
                __syncthreads();
                for (int tl = warp; tl < rows; tl += kFuseThreads / 32) {
                    float dot[kFuseHG];
#pragma unroll
                    for (int h = 0; h < kFuseHG; ++h) dot[h] = 0.0f;
                    if (c.bits == 8) {
                        const int *rowp = reinterpret_cast<const int *>(tile + size_t(tl) * row_bytes);
                        for (int i = lane; i < r / 4; i += 32) {
                            const int w = rowp[i];
                            const float x0 = float(int8_t(w)), x1 = float(int8_t(w >> 8));
                            const float x2 = float(int8_t(w >> 16)), x3 = float(int8_t(w >> 24));
#pragma unroll
                            for (int h = 0; h < kFuseHG; ++h)
                                if (h < hg) {
                                    const float4 qv = *reinterpret_cast<const float4 *>(qs + h * r + 4 * i);
                                    dot[h] += x0 * qv.x + x1 * qv.y + x2 * qv.z + x3 * qv.w;
                                }
                        }
                        const float sc = tsc[tl] * a.softmax_scale;
#pragma unroll
                        for (int h = 0; h < kFuseHG; ++h) dot[h] = warp_sum(dot[h]) * sc;
                    } else {
                        const uint32_t *rowp = reinterpret_cast<const uint32_t *>(tile + size_t(tl) * row_bytes);
                        const __half *gsr = static_cast<const __half *>(c.scales) + (slot0 + tl) * (r / 128);
                        for (int i = lane; i < r / 8; i += 32) {
                            const uint32_t w = rowp[i];
                            float x[8];
#pragma unroll
                            for (int e = 0; e < 8; ++e) x[e] = float((int((w >> (4 * e)) & 0xf) ^ 8) - 8);
                            const float s = __half2float(gsr[i >> 4]);
#pragma unroll
                            for (int h = 0; h < kFuseHG; ++h)
                                if (h < hg) {
                                    const float4 qa = *reinterpret_cast<const float4 *>(qs + h * r + 8 * i);
                                    const float4 qb = *reinterpret_cast<const float4 *>(qs + h * r + 8 * i + 4);
                                    dot[h] += s * (x[0] * qa.x + x[1] * qa.y + x[2] * qa.z + x[3] * qa.w +
                                                   x[4] * qb.x + x[5] * qb.y + x[6] * qb.z + x[7] * qb.w);
                                }
                        }
#pragma unroll
                        for (int h = 0; h < kFuseHG; ++h) dot[h] = warp_sum(dot[h]) * a.softmax_scale;
                    }
                    if (lane == 0)
#pragma unroll
                        for (int h = 0; h < kFuseHG; ++h)
                            if (h < hg) ps[h * kFuseSub + tl] = dot[h];
                }
                __syncthreads();
                if (warp < hg) {
                    float m = -FLT_MAX;
                    for (int tl = lane; tl < rows; tl += 32) m = fmaxf(m, ps[warp * kFuseSub + tl]);
                    m = warp_max(m);
                    const float m_old = m_s[warp];
                    const float m_new = fmaxf(m_old, m);
                    float l = 0.0f;
                    for (int tl = lane; tl < rows; tl += 32) {
                        const float p = expf(ps[warp * kFuseSub + tl] - m_new);
                        ps[warp * kFuseSub + tl] = p;
                        l += p;
                    }
                    l = warp_sum(l);
                    if (lane == 0) {
                        const float al = expf(m_old - m_new);
                        alpha_s[warp] = al;
                        l_s[warp] = l_s[warp] * al + l;
                        m_s[warp] = m_new;
                    }
                }
                __syncthreads();
#pragma unroll
                for (int h = 0; h < kFuseHG; ++h) {
                    const float al = h < hg ? alpha_s[h] : 0.0f;
#pragma unroll
                    for (int q = 0; q < kQ; ++q)
#pragma unroll
                        for (int e = 0; e < 4; ++e) acc[h][q][e] *= al;
                }
                for (int tl = 0; tl < rows; ++tl) {
#pragma unroll
                    for (int q = 0; q < kQ; ++q) {
                        const int qi = tid + q * kFuseThreads;
                        if (qi >= nq) break;
                        float x[4];
                        if (c.bits == 8) {
                            const int w = reinterpret_cast<const int *>(tile + size_t(tl) * row_bytes)[qi];
                            const float sc = tsc[tl];
                            x[0] = float(int8_t(w)) * sc;
                            x[1] = float(int8_t(w >> 8)) * sc;
                            x[2] = float(int8_t(w >> 16)) * sc;
                            x[3] = float(int8_t(w >> 24)) * sc;
                        } else {
                            const uint32_t w = reinterpret_cast<const uint16_t *>(tile + size_t(tl) * row_bytes)[qi];
                            const float sc = __half2float(static_cast<const __half *>(c.scales)[(slot0 + tl) * (r / 128) + (qi >> 5)]);
#pragma unroll
                            for (int e = 0; e < 4; ++e) x[e] = float((int((w >> (4 * e)) & 0xf) ^ 8) - 8) * sc;
                        }
#pragma unroll
                        for (int h = 0; h < kFuseHG; ++h)
                            if (h < hg) {
                                const float p = ps[h * kFuseSub + tl];
#pragma unroll
                                for (int e = 0; e < 4; ++e) acc[h][q][e] = fmaf(p, x[e], acc[h][q][e]);
                            }
                    }
                }
            }
            const size_t pbase = (size_t(b) * a.n_split + split) * H + h0;
#pragma unroll
            for (int h = 0; h < kFuseHG; ++h) {
                if (h >= hg) break;
#pragma unroll
                for (int q = 0; q < kQ; ++q) {
                    const int qi = tid + q * kFuseThreads;
                    if (qi >= nq) break;
                    *reinterpret_cast<float4 *>(a.w_.po + (pbase + h) * r + 4 * qi) =
                        make_float4(acc[h][q][0], acc[h][q][1], acc[h][q][2], acc[h][q][3]);
                }
                if (tid == 0) {
                    a.w_.pm[pbase + h] = m_s[h];
                    a.w_.pl[pbase + h] = l_s[h];
                }
            }
        }
    }
    if (!grid_barrier(a.w_.bar, err)) return;

    // ---- P5: merge partials and apply U_v per (head, row block) task
    {
        const int nrb = (r + kFuseRowBlock - 1) / kFuseRowBlock;
        uint16_t *u_s = reinterpret_cast<uint16_t *>(smem);           // [128][dh]
        float *ol = reinterpret_cast<float *>(u_s + kFuseRowBlock * 128);  // [128]
        for (int task = k; task < H * nrb; task += G) {
            const int h = task % H, rb = task / H;
            const int j0 = rb * kFuseRowBlock, rows = min(kFuseRowBlock, r - j0);
            __syncthreads();
            for (int i = tid; i < rows * dh / 8; i += kFuseThreads) {
                const int row = i / (dh / 8), c8 = i % (dh / 8);
                reinterpret_cast<uint4 *>(u_s + row * dh)[c8] =
                    *reinterpret_cast<const uint4 *>(a.Uv + size_t(j0 + row) * d + h * dh + c8 * 8);
            }
            for (int b = 0; b < B; ++b) {
                const int L = a.seq_len[b];
                const int ns = (L + a.chunk - 1) / a.chunk;
                const size_t base = size_t(b) * a.n_split * H + h;
                __syncthreads();
                if (warp == 0) {                        // ns <= 64: two partials per lane
                    const float m0 = lane < ns ? a.w_.pm[base + size_t(lane) * H] : -FLT_MAX;
                    const float m1 = lane + 32 < ns ? a.w_.pm[base + size_t(lane + 32) * H] : -FLT_MAX;
                    const float l0 = lane < ns ? a.w_.pl[base + size_t(lane) * H] : 0.0f;
                    const float l1 = lane + 32 < ns ? a.w_.pl[base + size_t(lane + 32) * H] : 0.0f;
                    const float M = warp_max(fmaxf(m0, m1));
                    const float w0 = lane < ns ? expf(m0 - M) : 0.0f;
                    const float w1 = lane + 32 < ns ? expf(m1 - M) : 0.0f;
                    wsp[lane] = w0;
                    wsp[lane + 32] = w1;
                    const float l = warp_sum(w0 * l0 + w1 * l1);
                    if (lane == 0) inv_l = 1.0f / l;
                }
                __syncthreads();
                for (int jj = tid; jj < rows; jj += kFuseThreads) {
                    float o = 0.0f;
                    for (int s0 = 0; s0 < ns; s0 += 8) {
                        float v[8];
#pragma unroll
                        for (int q = 0; q < 8; ++q)
                            v[q] = s0 + q < ns ? a.w_.po[(base + size_t(s0 + q) * H) * r + j0 + jj] : 0.0f;
#pragma unroll
                        for (int q = 0; q < 8; ++q) o = fmaf(s0 + q < ns ? wsp[s0 + q] : 0.0f, v[q], o);
                    }
                    ol[jj] = o * inv_l;
                }
                __syncthreads();
                float *part = a.w_.opart + ((size_t(b) * H + h) * nrb + rb) * dh;
                for (int i = tid; i < dh; i += kFuseThreads) {
                    float acc = 0.0f;
#pragma unroll 8
                    for (int jj = 0; jj < rows; ++jj) acc = fmaf(ol[jj], bf16_to_f32(u_s[jj * dh + i]), acc);
                    part[i] = acc;
                }
            }
            __threadfence();
            __syncthreads();
            if (tid == 0) last = atomicAdd(&a.w_.head_count[h], 1) == nrb - 1;
            __syncthreads();
            if (last) {
                __threadfence();
                for (int b = 0; b < B; ++b) {
                    const float *all = a.w_.opart + (size_t(b) * H + h) * nrb * dh;
                    for (int i = tid; i < dh; i += kFuseThreads) {
                        float s = 0.0f;
                        for (int q = 0; q < nrb; ++q) s += all[size_t(q) * dh + i];
                        a.O[size_t(b) * d + h * dh + i] = s;
                    }
                }
                if (tid == 0) a.w_.head_count[h] = 0;
            }
        }
    }
}

static size_t fuse_smem_bytes(int B, int d, int r, int bits, int dh) {
    const int row_bytes = bits == 8 ? r : r / 2;
    size_t p1 = size_t(B) * d;
    size_t p2 = (size_t(r) + 8 * 32) * 4;
    size_t p3 = size_t(d) * 4;
    size_t p4 = (size_t(kFuseHG) * r + kFuseHG * kFuseSub + kFuseSub) * 4 + size_t(kFuseSub) * row_bytes;
    size_t p5 = size_t(kFuseRowBlock) * 128 * 2 + kFuseRowBlock * 4;
    (void)dh;
    size_t m = p1;
    for (size_t v : {p2, p3, p4, p5}) m = v > m ? v : m;
    return (m + 15) & ~size_t(15);
}

cudaError_t launch_decode_fused(const FusedArgs &f, void *ws, size_t ws_bytes, int *err, cudaStream_t s) {
    FuseArgs a;
    a.X = f.X;
    a.w = f.w_codes;
    a.ws = f.w_scale;
    a.c = f.cache;
    a.seq_len = f.seq_len;
    a.Uq = f.U_q;
    a.Uk = f.U_k;
    a.Uv = f.U_v;
    a.B = f.cache.B;
    a.d = f.d;
    a.H = f.H;
    a.dh = f.dh;
    a.chunk = fuse_chunk(f.max_seq_len);
    a.n_split = (f.max_seq_len + a.chunk - 1) / a.chunk;
    a.act_clip = f.act_clip;
    a.lat_clip = f.lat_clip;
    a.softmax_scale = f.softmax_scale;
    a.O = f.O;
    a.err = err;
    fuse_carve(a.B, f.max_seq_len, a.d, a.c.r, a.H, a.dh, static_cast<char *>(ws), &a.w_);
    (void)ws_bytes;
    const size_t smem = fuse_smem_bytes(a.B, a.d, a.c.r, a.c.bits, a.dh);
    cudaError_t e = ensure_smem(decode_step_kernel, smem);
    if (e != cudaSuccess) return e;
    // the grid barrier's arrival count and generation start at zero on every
    // call: a call whose barrier wait expired leaves some CTAs counted
    e = cudaMemsetAsync(a.w_.bar, 0, 2 * sizeof(unsigned), s);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_step_kernel, kFuseThreads, smem);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(sms);
    cfg.blockDim = dim3(kFuseThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    e = cudaLaunchKernelEx(&cfg, decode_step_kernel, a);
    prof_mark(s, "decode_step");
    return e;
}

}  // namespace qsvd
