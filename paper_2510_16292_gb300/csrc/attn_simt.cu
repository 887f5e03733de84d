// Decode attention over the latent cache, CUDA-core version (Eq. 5 with U_k
// absorbed into the query and U_v applied last):
//
//   qproj_kernel      a5: q[b] = c_{L-1} U_q          (c = dequantized cache row)
//   qabsorb_kernel    a5: qt[b, h, :] = U_k[:, h] q_h  (q~_h, length r)
//   attn_split_kernel a6/a7: per (b, token chunk, head group): scores
//                     c_t . q~_h * softmax_scale, chunk-local softmax, and the
//                     unnormalised latent sum  sum_t p_t c_t  (split-T partial)
//   combine_uv_kernel a7/a8: merge the partials (max-rescaled), divide by the
//                     softmax denominator, and apply U_v[:, h].
#include <cfloat>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

constexpr int kChunk = 256;    // tokens per split-T partial
constexpr int kHG = 8;         // heads per attention CTA
constexpr int kAtThreads = 256;
constexpr int kMaxRank = 3072; // 3 float4 quads per thread in attn_split_kernel

static inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct DecodeWs {
    float *q, *qt, *pm, *pl, *po;
};

static size_t carve(int B, int max_seq_len, int r, int H, int d, char *base, DecodeWs *w) {
    const int ns = (max_seq_len + kChunk - 1) / kChunk;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *p = base ? base + off : nullptr;
        off += align256(bytes);
        return reinterpret_cast<float *>(p);
    };
    DecodeWs t;
    t.q = take(size_t(B) * d * 4);
    t.qt = take(size_t(B) * H * r * 4);
    t.pm = take(size_t(B) * ns * H * 4);
    t.pl = take(size_t(B) * ns * H * 4);
    t.po = take(size_t(B) * ns * H * r * 4);
    if (w) *w = t;
    return off;
}

size_t decode_workspace_bytes(int B, int max_seq_len, int r, int H, int dh) {
    return carve(B, max_seq_len, r, H, H * dh, nullptr, nullptr);
}

// Dequantized channel j of cache slot `slot` (fp32 code * scale).
__device__ __forceinline__ float cache_value(const CacheView &c, size_t slot, int j) {
    if (c.bits == 8) {
        const int8_t code = static_cast<const int8_t *>(c.codes)[slot * c.r + j];
        return float(code) * static_cast<const float *>(c.scales)[slot];
    }
    const uint8_t byte = static_cast<const uint8_t *>(c.codes)[slot * (c.r / 2) + (j >> 1)];
    int nib = (j & 1) ? (byte >> 4) : (byte & 0xf);
    nib = (nib ^ 8) - 8;
    return float(nib) * __half2float(static_cast<const __half *>(c.scales)[slot * (c.r / 128) + (j >> 7)]);
}

__device__ __forceinline__ bool valid_len(int L, int Tmax) { return L >= 1 && L <= Tmax; }

// ---------------------------------------------------------------------------
// a5 (first half): q[b, :] = c_last[b] . U_q, two sequences per CTA, 64 columns.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
qproj_kernel(CacheView c, const int32_t *__restrict__ seq_len, int B, const uint16_t *__restrict__ Uq,
             int d, float *__restrict__ q, int *err) {
    extern __shared__ float sm[];
    const int r = c.r;
    float *chat = sm;               // [2][r]
    float *red = sm + 2 * r;        // [32][2][64]
    const int b0 = blockIdx.y * 2;
    for (int bb = 0; bb < 2; ++bb) {
        const int b = b0 + bb;
        int L = 0;
        if (b < B) {
            L = seq_len[b];
            if (!valid_len(L, c.Tmax)) {
                if (threadIdx.x == 0 && blockIdx.x == 0) flag_error(err, kErrRange);
                L = 0;
            }
        }
        for (int j = threadIdx.x; j < r; j += 256)
            chat[bb * r + j] = L ? cache_value(c, size_t(b) * c.Tmax + (L - 1), j) : 0.0f;
    }
    __syncthreads();
    const int rg = threadIdx.x >> 3, co = threadIdx.x & 7;
    const int c0 = blockIdx.x * 64 + co * 8;
    float acc[2][8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[0][e] = acc[1][e] = 0.0f;
    for (int j = rg; j < r; j += 32) {
        float u[8];
        unpack8_bf16(*reinterpret_cast<const uint4 *>(Uq + size_t(j) * d + c0), u);
        const float a0 = chat[j], a1 = chat[r + j];
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            acc[0][e] = fmaf(a0, u[e], acc[0][e]);
            acc[1][e] = fmaf(a1, u[e], acc[1][e]);
        }
    }
#pragma unroll
    for (int bb = 0; bb < 2; ++bb)
#pragma unroll
        for (int e = 0; e < 8; ++e) red[(rg * 2 + bb) * 64 + co * 8 + e] = acc[bb][e];
    __syncthreads();
    if (threadIdx.x < 128) {
        const int bb = threadIdx.x >> 6, col = threadIdx.x & 63;
        float s = 0.0f;
        for (int g = 0; g < 32; ++g) s += red[(g * 2 + bb) * 64 + col];
        if (b0 + bb < B) q[size_t(b0 + bb) * d + blockIdx.x * 64 + col] = s;
    }
}

// ---------------------------------------------------------------------------
// a5 (second half): qt[b, h, j] = sum_i U_k[j, h*dh + i] * q[b, h*dh + i].
// One warp per (b, j); lanes sweep row j of U_k 8 columns at a time and
// reduce within each head's lane segment.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
qabsorb_kernel(const float *__restrict__ q, const uint16_t *__restrict__ Uk, int r, int d, int H, int dh,
               float *__restrict__ qt) {
    const int lane = threadIdx.x & 31;
    const int j = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int b = blockIdx.y;
    if (j >= r) return;
    const uint16_t *urow = Uk + size_t(j) * d;
    const float *qb = q + size_t(b) * d;
    const int seg = dh / 8;
    for (int base = 0; base < d; base += 256) {
        const int col = base + lane * 8;
        float p = 0.0f;
        if (col < d) {
            float u[8];
            unpack8_bf16(*reinterpret_cast<const uint4 *>(urow + col), u);
            const float4 q0 = *reinterpret_cast<const float4 *>(qb + col);
            const float4 q1 = *reinterpret_cast<const float4 *>(qb + col + 4);
            p = u[0] * q0.x + u[1] * q0.y + u[2] * q0.z + u[3] * q0.w +
                u[4] * q1.x + u[5] * q1.y + u[6] * q1.z + u[7] * q1.w;
        }
        for (int o = seg >> 1; o; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
        if (col < d && (lane % seg) == 0) qt[(size_t(b) * H + col / dh) * r + j] = p;
    }
}

// ---------------------------------------------------------------------------
// a6/a7: one CTA per (token chunk, sequence, head group).
// ---------------------------------------------------------------------------
template <int BITS>
__global__ void __launch_bounds__(kAtThreads)
attn_split_kernel(CacheView c, const int32_t *__restrict__ seq_len, const float *__restrict__ qt, int H,
                  float softmax_scale, int n_split, float *__restrict__ pm, float *__restrict__ pl,
                  float *__restrict__ po) {
    extern __shared__ float sm[];
    __shared__ float sm_m[kHG], sm_l[kHG];
    const int r = c.r;
    const int split = blockIdx.x, b = blockIdx.y, h0 = blockIdx.z * kHG;
    const int hg = min(kHG, H - h0);
    const int L = seq_len[b];
    if (!valid_len(L, c.Tmax)) return;            // flagged by qproj_kernel
    const int t_begin = split * kChunk;
    if (t_begin >= L) return;
    const int n = min(L, t_begin + kChunk) - t_begin;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *qs = sm;                 // [kHG][r]
    float *ps = sm + kHG * r;       // [kHG][kChunk]
    for (int i = threadIdx.x; i < hg * r; i += kAtThreads) qs[i] = qt[(size_t(b) * H + h0) * r + i];
    __syncthreads();

    // scores
    for (int tl = warp; tl < n; tl += kAtThreads / 32) {
        const size_t slot = size_t(b) * c.Tmax + t_begin + tl;
        float dot[kHG];
#pragma unroll
        for (int h = 0; h < kHG; ++h) dot[h] = 0.0f;
        if (BITS == 8) {
            const int *row = reinterpret_cast<const int *>(static_cast<const int8_t *>(c.codes) + slot * r);
            for (int i = lane; i < r / 4; i += 32) {
                const int w = row[i];
                const float x0 = float(int8_t(w)), x1 = float(int8_t(w >> 8));
                const float x2 = float(int8_t(w >> 16)), x3 = float(int8_t(w >> 24));
#pragma unroll
                for (int h = 0; h < kHG; ++h) {
                    if (h < hg) {
                        const float4 qv = *reinterpret_cast<const float4 *>(qs + h * r + 4 * i);
                        dot[h] += x0 * qv.x + x1 * qv.y + x2 * qv.z + x3 * qv.w;
                    }
                }
            }
            const float sc = static_cast<const float *>(c.scales)[slot] * softmax_scale;
#pragma unroll
            for (int h = 0; h < kHG; ++h) dot[h] = warp_sum(dot[h]) * sc;
        } else {
            const uint32_t *row =
                reinterpret_cast<const uint32_t *>(static_cast<const uint8_t *>(c.codes) + slot * (r / 2));
            const __half *gs = static_cast<const __half *>(c.scales) + slot * (r / 128);
            for (int i = lane; i < r / 8; i += 32) {
                const uint32_t w = row[i];
                float x[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) x[e] = float((int((w >> (4 * e)) & 0xf) ^ 8) - 8);
                const float s = __half2float(gs[i >> 4]);
#pragma unroll
                for (int h = 0; h < kHG; ++h) {
                    if (h < hg) {
                        const float4 qa = *reinterpret_cast<const float4 *>(qs + h * r + 8 * i);
                        const float4 qb = *reinterpret_cast<const float4 *>(qs + h * r + 8 * i + 4);
                        const float part = x[0] * qa.x + x[1] * qa.y + x[2] * qa.z + x[3] * qa.w +
                                           x[4] * qb.x + x[5] * qb.y + x[6] * qb.z + x[7] * qb.w;
                        dot[h] += s * part;
                    }
                }
            }
#pragma unroll
            for (int h = 0; h < kHG; ++h) dot[h] = warp_sum(dot[h]) * softmax_scale;
        }
        if (lane == 0) {
#pragma unroll
            for (int h = 0; h < kHG; ++h)
                if (h < hg) ps[h * kChunk + tl] = dot[h];
        }
    }
    __syncthreads();

    // chunk-local softmax statistics
    if (warp < hg) {
        float m = -FLT_MAX;
        for (int tl = lane; tl < n; tl += 32) m = fmaxf(m, ps[warp * kChunk + tl]);
        m = warp_max(m);
        float l = 0.0f;
        for (int tl = lane; tl < n; tl += 32) {
            const float p = expf(ps[warp * kChunk + tl] - m);
            ps[warp * kChunk + tl] = p;
            l += p;
        }
        l = warp_sum(l);
        if (lane == 0) {
            sm_m[warp] = m;
            sm_l[warp] = l;
        }
    }
    __syncthreads();

    // latent accumulation  o[h, j] = sum_t p[h, t] c[t, j]
    constexpr int kQ = kMaxRank / 4 / kAtThreads;   // quads per thread
    float acc[kHG][kQ][4];
#pragma unroll
    for (int h = 0; h < kHG; ++h)
#pragma unroll
        for (int k = 0; k < kQ; ++k)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[h][k][e] = 0.0f;
    const int nq = r / 4;
    for (int tl = 0; tl < n; ++tl) {
        const size_t slot = size_t(b) * c.Tmax + t_begin + tl;
#pragma unroll
        for (int k = 0; k < kQ; ++k) {
            const int qi = threadIdx.x + k * kAtThreads;
            if (qi >= nq) break;
            float x[4];
            if (BITS == 8) {
                const int w = reinterpret_cast<const int *>(static_cast<const int8_t *>(c.codes) + slot * r)[qi];
                const float sc = static_cast<const float *>(c.scales)[slot];
                x[0] = float(int8_t(w)) * sc;
                x[1] = float(int8_t(w >> 8)) * sc;
                x[2] = float(int8_t(w >> 16)) * sc;
                x[3] = float(int8_t(w >> 24)) * sc;
            } else {
                const uint32_t w = reinterpret_cast<const uint16_t *>(
                    static_cast<const uint8_t *>(c.codes) + slot * (r / 2))[qi];
                const float sc = __half2float(static_cast<const __half *>(c.scales)[slot * (r / 128) + (qi >> 5)]);
#pragma unroll
                for (int e = 0; e < 4; ++e) x[e] = float((int((w >> (4 * e)) & 0xf) ^ 8) - 8) * sc;
            }
#pragma unroll
            for (int h = 0; h < kHG; ++h) {
                if (h < hg) {
                    const float p = ps[h * kChunk + tl];
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[h][k][e] = fmaf(p, x[e], acc[h][k][e]);
                }
            }
        }
    }
    const size_t pbase = (size_t(b) * n_split + split) * H + h0;
#pragma unroll
    for (int h = 0; h < kHG; ++h) {
        if (h >= hg) break;
#pragma unroll
        for (int k = 0; k < kQ; ++k) {
            const int qi = threadIdx.x + k * kAtThreads;
            if (qi >= nq) break;
            *reinterpret_cast<float4 *>(po + (pbase + h) * r + 4 * qi) =
                make_float4(acc[h][k][0], acc[h][k][1], acc[h][k][2], acc[h][k][3]);
        }
        if (threadIdx.x == 0) {
            pm[pbase + h] = sm_m[h];
            pl[pbase + h] = sm_l[h];
        }
    }
}

// ---------------------------------------------------------------------------
// a7/a8: merge split partials and apply U_v.  One CTA per (head, sequence).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128)
combine_uv_kernel(const int32_t *__restrict__ seq_len, int Tmax, int H, int dh, int r, int n_split,
                  const float *__restrict__ pm, const float *__restrict__ pl, const float *__restrict__ po,
                  const uint16_t *__restrict__ Uv, float *__restrict__ O) {
    extern __shared__ float sm[];
    float *ol = sm;           // [r]
    float *wsp = sm + r;      // [n_split]
    __shared__ float inv_l;
    const int h = blockIdx.x, b = blockIdx.y, d = H * dh;
    const int L = seq_len[b];
    if (!valid_len(L, Tmax)) {
        for (int i = threadIdx.x; i < dh; i += blockDim.x) O[size_t(b) * d + h * dh + i] = 0.0f;
        return;
    }
    const int ns = (L + kChunk - 1) / kChunk;
    const size_t base = size_t(b) * n_split * H + h;
    if (threadIdx.x == 0) {
        float M = -FLT_MAX;
        for (int s = 0; s < ns; ++s) M = fmaxf(M, pm[base + size_t(s) * H]);
        float l = 0.0f;
        for (int s = 0; s < ns; ++s) {
            const float w = expf(pm[base + size_t(s) * H] - M);
            wsp[s] = w;
            l += w * pl[base + size_t(s) * H];
        }
        inv_l = 1.0f / l;
    }
    __syncthreads();
    for (int j = threadIdx.x; j < r; j += blockDim.x) {
        float o = 0.0f;
        for (int s = 0; s < ns; ++s) o = fmaf(wsp[s], po[(base + size_t(s) * H) * r + j], o);
        ol[j] = o * inv_l;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < dh; i += blockDim.x) {
        float acc = 0.0f;
        for (int j = 0; j < r; ++j) acc = fmaf(ol[j], bf16_to_f32(Uv[size_t(j) * d + h * dh + i]), acc);
        O[size_t(b) * d + h * dh + i] = acc;
    }
}

// ---------------------------------------------------------------------------
cudaError_t launch_decode(const DecodeArgs &a, void *ws, size_t ws_bytes, int *err, cudaStream_t s) {
    const CacheView &c = a.cache;
    const int B = c.B, r = c.r, H = a.H, dh = a.dh, d = H * dh;
    DecodeWs w;
    carve(B, a.max_seq_len, r, H, d, static_cast<char *>(ws), &w);
    const int ns = (a.max_seq_len + kChunk - 1) / kChunk;
    cudaError_t e;

    const size_t smem_q = (2 * size_t(r) + 32 * 2 * 64) * sizeof(float);
    e = cudaFuncSetAttribute(qproj_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem_q));
    if (e != cudaSuccess) return e;
    qproj_kernel<<<dim3(d / 64, (B + 1) / 2), 256, smem_q, s>>>(c, a.seq_len, B, a.U_q, d, w.q, err);
    prof_mark(s, "qproj");
    qabsorb_kernel<<<dim3((r + 7) / 8, B), 256, 0, s>>>(w.q, a.U_k, r, d, H, dh, w.qt);
    prof_mark(s, "qabsorb");

    const size_t smem_a = (size_t(kHG) * r + size_t(kHG) * kChunk) * sizeof(float);
    dim3 grid_a(ns, B, (H + kHG - 1) / kHG);
    if (c.bits == 8) {
        e = cudaFuncSetAttribute(attn_split_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem_a));
        if (e != cudaSuccess) return e;
        attn_split_kernel<8><<<grid_a, kAtThreads, smem_a, s>>>(c, a.seq_len, w.qt, H, a.softmax_scale, ns,
                                                               w.pm, w.pl, w.po);
        prof_mark(s, "attn_split");
    } else {
        e = cudaFuncSetAttribute(attn_split_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem_a));
        if (e != cudaSuccess) return e;
        attn_split_kernel<4><<<grid_a, kAtThreads, smem_a, s>>>(c, a.seq_len, w.qt, H, a.softmax_scale, ns,
                                                               w.pm, w.pl, w.po);
        prof_mark(s, "attn_split");
    }
    const size_t smem_c = (size_t(r) + ns) * sizeof(float);
    if (smem_c > 48 * 1024) {
        e = cudaFuncSetAttribute(combine_uv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem_c));
        if (e != cudaSuccess) return e;
    }
    combine_uv_kernel<<<dim3(H, B), 128, smem_c, s>>>(a.seq_len, c.Tmax, H, dh, r, ns, w.pm, w.pl, w.po, a.U_v,
                                                      a.O);
    prof_mark(s, "combine_uv");
    return cudaGetLastError();
}

}  // namespace qsvd
