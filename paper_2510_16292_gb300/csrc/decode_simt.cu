// Decode attention over the latent cache (Eq. 5 with U_k absorbed into the
// query and U_v applied last) as a chain of kernels linked by programmatic
// dependent launch:
//
//   qproj_kernel, qabsorb_kernel (decode_gemv.cu)   a5: q and q~ for all B
//   attn_chunk_kernel (here, CUDA cores) or attn_tc_kernel (attn_tc.cu,
//       tensor cores)                               a6/a7: per (b, token
//       range): online-softmax pass over the cache rows, giving (max, sum,
//       unnormalised sum_t p_t c_t) per head
//   combine_uv_kernel (decode_gemv.cu)              a7/a8: merge the partials,
//       divide by the softmax denominator, multiply by U_v
#include <cfloat>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

constexpr int kMaxSplits = 64;   // token chunks per sequence
constexpr int kHG = 2;           // heads per attention CTA
constexpr int kAtThreads = 256;
constexpr int kMaxRank = 3072;   // 3 float4 quads per thread in attn_chunk_kernel
constexpr int kSubTileBytes = 24 * 1024;

static inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

static int chunk_tokens(int max_seq_len) {
    int c = 32;
    while ((max_seq_len + c - 1) / c > kMaxSplits) c += 32;
    return c;
}

struct DecodeWs {
    float *q, *qt, *pm, *pl, *po;
    unsigned *qmax;    // [B, H] max |q~| bit patterns (cleared by qproj_kernel)
};

// Partials per sequence the workspace holds: enough for either attention
// kernel (chunks of at least 16 tokens, at most kMaxSplits of them), and
// non-decreasing in max_seq_len so that a workspace sized for a bound also
// serves every shorter call.
static int split_capacity(int max_seq_len) {
    const int ns = (max_seq_len + 15) / 16;
    return ns < kMaxSplits ? ns : kMaxSplits;
}

static size_t carve(int B, int max_seq_len, int r, int H, int dh, char *base, DecodeWs *w) {
    const int ns = split_capacity(max_seq_len);
    const int d = H * dh;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *p = base ? base + off : nullptr;
        off += align256(bytes);
        return p;
    };
    DecodeWs t;
    t.q = reinterpret_cast<float *>(take(size_t(B) * d * 4));
    t.qt = reinterpret_cast<float *>(take(size_t(B) * H * r * 4));
    t.qmax = reinterpret_cast<unsigned *>(take(size_t(B) * H * 4));
    t.pm = reinterpret_cast<float *>(take(size_t(B) * ns * H * 4));
    t.pl = reinterpret_cast<float *>(take(size_t(B) * ns * H * 4));
    t.po = reinterpret_cast<float *>(take(size_t(B) * ns * H * r * 4));
    if (w) *w = t;
    return off;
}

size_t decode_workspace_bytes(int B, int max_seq_len, int r, int H, int dh) {
    return carve(B, max_seq_len, r, H, dh, nullptr, nullptr);
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
// a6/a7: one CTA per (token chunk, sequence, group of kHG heads).  The chunk
// is streamed through shared memory in sub-tiles (double-buffered bulk
// copies); scores and the latent sum use an online softmax per head.
// ---------------------------------------------------------------------------
template <int BITS>
__global__ void __launch_bounds__(kAtThreads)
attn_chunk_kernel(CacheView c, const int32_t *__restrict__ seq_len, const float *qt, int H,
                  float softmax_scale, int chunk, int sub, int n_split, float *__restrict__ pm,
                  float *__restrict__ pl, float *__restrict__ po, int *err) {
    extern __shared__ __align__(16) uint8_t smem[];
    __shared__ __align__(8) uint64_t bar[2];
    __shared__ float m_s[kHG], l_s[kHG], alpha_s[kHG];
    const int r = c.r;
    const int row_bytes = BITS == 8 ? r : r / 2;
    const int split = blockIdx.x, b = blockIdx.y, h0 = blockIdx.z * kHG;
    const int hg = min(kHG, H - h0);
    const int t_begin = split * chunk;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float *qs = reinterpret_cast<float *>(smem);                    // [kHG][r]
    float *ps = qs + kHG * r;                                       // [kHG][sub]
    float *ts = ps + kHG * sub;                                     // [2][sub] token scales (int8)
    uint8_t *tile = reinterpret_cast<uint8_t *>(ts + 2 * sub);      // [2][sub][row_bytes] codes
    const int slot_bytes = row_bytes;
    pdl_trigger();
    const int sq = view_seq(c, b);   // a call input, complete before this grid starts (see qproj)
    if (blockIdx.z == 0 && threadIdx.x == 0 && t_begin < c.Tmax && sq >= 0) {
        const int rows = min(chunk, c.Tmax - t_begin);
        const char *base = static_cast<const char *>(c.codes) + (size_t(sq) * c.Tmax + t_begin) * row_bytes;
        for (size_t o = 0; o < size_t(rows) * row_bytes; o += 65536)
            prefetch_l2_bulk(base + o, uint32_t(min(size_t(65536), size_t(rows) * row_bytes - o)));
    }
    if (threadIdx.x == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        mbar_init_fence();
    }
    __syncthreads();
    pdl_wait();
    const int L = sq < 0 ? 0 : seq_len[b];
    if (!valid_len(L, c.Tmax) || t_begin >= L) return;        // invalid lengths are flagged by qproj_kernel
    const int n = min(L, t_begin + chunk) - t_begin;
    const int n_sub = (n + sub - 1) / sub;

    auto issue = [&](int st, int buf) {                       // thread 0 only
        const int t0 = t_begin + st * sub;
        const int rows = min(sub, t_begin + n - t0);
        const size_t slot0 = size_t(sq) * c.Tmax + t0;
        uint8_t *dst = tile + size_t(buf) * sub * slot_bytes;
        const uint32_t code_bytes = uint32_t(rows) * row_bytes;
        mbar_arrive_expect_tx(&bar[buf], code_bytes);
        bulk_g2s(dst, static_cast<const uint8_t *>(c.codes) + slot0 * row_bytes, code_bytes, &bar[buf]);
    };
    if (threadIdx.x == 0) {
        issue(0, 0);
        if (n_sub > 1) issue(1, 1);
    }
    for (int i = threadIdx.x; i < hg * r; i += kAtThreads) qs[i] = qt[(size_t(b) * H + h0) * r + i];
    if (threadIdx.x < kHG) {
        m_s[threadIdx.x] = -FLT_MAX;
        l_s[threadIdx.x] = 0.0f;
    }
    constexpr int kQ = kMaxRank / 4 / kAtThreads;   // quads per thread
    float acc[kHG][kQ][4];
#pragma unroll
    for (int h = 0; h < kHG; ++h)
#pragma unroll
        for (int k = 0; k < kQ; ++k)
#pragma unroll
            for (int e = 0; e < 4; ++e) acc[h][k][e] = 0.0f;
    const int nq = r / 4;
    __syncthreads();

    for (int st = 0; st < n_sub; ++st) {
        const int buf = st & 1;
        const int rows = min(sub, n - st * sub);
        const uint8_t *tl_codes = tile + size_t(buf) * sub * slot_bytes;
        const __half *tl_gs = static_cast<const __half *>(c.scales) +
                              (size_t(sq) * c.Tmax + t_begin + st * sub) * (r / 128);   // int4 group scales
        float *tsc = ts + buf * sub;
        if (BITS == 8 && threadIdx.x < rows)
            tsc[threadIdx.x] = static_cast<const float *>(c.scales)[size_t(sq) * c.Tmax + t_begin + st * sub + threadIdx.x];
        mbar_wait(&bar[buf], uint32_t((st >> 1) & 1), err);
        __syncthreads();
        // scores of this sub-tile: one warp per token
        for (int tl = warp; tl < rows; tl += kAtThreads / 32) {
            float dot[kHG];
#pragma unroll
            for (int h = 0; h < kHG; ++h) dot[h] = 0.0f;
            if (BITS == 8) {
                const int *row = reinterpret_cast<const int *>(tl_codes + size_t(tl) * row_bytes);
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
                const float sc = tsc[tl] * softmax_scale;
#pragma unroll
                for (int h = 0; h < kHG; ++h) dot[h] = warp_sum(dot[h]) * sc;
            } else {
                const uint32_t *row = reinterpret_cast<const uint32_t *>(tl_codes + size_t(tl) * row_bytes);
                const __half *gsr = tl_gs + size_t(tl) * (r / 128);
                for (int i = lane; i < r / 8; i += 32) {
                    const uint32_t w = row[i];
                    float x[8];
#pragma unroll
                    for (int e = 0; e < 8; ++e) x[e] = float((int((w >> (4 * e)) & 0xf) ^ 8) - 8);
                    const float s = __half2float(gsr[i >> 4]);
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
                    if (h < hg) ps[h * sub + tl] = dot[h];
            }
        }
        __syncthreads();
        // online softmax update (one warp per head)
        if (warp < hg) {
            float m = -FLT_MAX;
            for (int tl = lane; tl < rows; tl += 32) m = fmaxf(m, ps[warp * sub + tl]);
            m = warp_max(m);
            const float m_old = m_s[warp];
            const float m_new = fmaxf(m_old, m);
            float l = 0.0f;
            for (int tl = lane; tl < rows; tl += 32) {
                const float p = expf(ps[warp * sub + tl] - m_new);
                ps[warp * sub + tl] = p;
                l += p;
            }
            l = warp_sum(l);
            if (lane == 0) {
                const float a = expf(m_old - m_new);
                alpha_s[warp] = a;
                l_s[warp] = l_s[warp] * a + l;
                m_s[warp] = m_new;
            }
        }
        __syncthreads();
        // latent accumulation  acc[h, j] = alpha_h acc[h, j] + sum_t p[h, t] c[t, j]
#pragma unroll
        for (int h = 0; h < kHG; ++h) {
            const float a = h < hg ? alpha_s[h] : 0.0f;
#pragma unroll
            for (int k = 0; k < kQ; ++k)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[h][k][e] *= a;
        }
        for (int tl = 0; tl < rows; ++tl) {
#pragma unroll
            for (int k = 0; k < kQ; ++k) {
                const int qi = threadIdx.x + k * kAtThreads;
                if (qi >= nq) break;
                float x[4];
                if (BITS == 8) {
                    const int w = reinterpret_cast<const int *>(tl_codes + size_t(tl) * row_bytes)[qi];
                    const float sc = tsc[tl];
                    x[0] = float(int8_t(w)) * sc;
                    x[1] = float(int8_t(w >> 8)) * sc;
                    x[2] = float(int8_t(w >> 16)) * sc;
                    x[3] = float(int8_t(w >> 24)) * sc;
                } else {
                    const uint32_t w = reinterpret_cast<const uint16_t *>(tl_codes + size_t(tl) * row_bytes)[qi];
                    const float sc = __half2float(tl_gs[size_t(tl) * (r / 128) + (qi >> 5)]);
#pragma unroll
                    for (int e = 0; e < 4; ++e) x[e] = float((int((w >> (4 * e)) & 0xf) ^ 8) - 8) * sc;
                }
#pragma unroll
                for (int h = 0; h < kHG; ++h) {
                    if (h < hg) {
                        const float p = ps[h * sub + tl];
#pragma unroll
                        for (int e = 0; e < 4; ++e) acc[h][k][e] = fmaf(p, x[e], acc[h][k][e]);
                    }
                }
            }
        }
        __syncthreads();                                     // buffer `buf` is free again
        if (threadIdx.x == 0 && st + 2 < n_sub) issue(st + 2, buf);
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
            pm[pbase + h] = m_s[h];
            pl[pbase + h] = l_s[h];
        }
    }
}

// ---------------------------------------------------------------------------
cudaError_t launch_decode(const DecodeArgs &a, void *ws, size_t ws_bytes, int *err, cudaStream_t s) {
    const CacheView &c = a.cache;
    const int B = c.B, r = c.r, H = a.H, dh = a.dh, d = H * dh;
    DecodeWs w;
    carve(B, a.max_seq_len, r, H, dh, static_cast<char *>(ws), &w);
    // the up-projection products on the tensor cores from 5 sequences on
    // (bf16 weights only: quantized up-projections take the CUDA-core forms at every batch size)
    const bool bf16_up = a.U_q.bits == 16 && a.U_k.bits == 16 && a.U_v.bits == 16;
    const bool mma = bf16_up && decode_mma_supported(B, r, d, dh);
    cudaError_t e;
    // the warp-level attention kernel can form the per-head maxima of q~ itself (r <= 2048)
    const bool mma_attn = attn_mma_use(c, H, B, a.max_seq_len) && attn_mma_fits(c, a.max_seq_len);
    const bool local_qmax = mma_attn && r <= 2048 && r % 128 == 0;
    const bool qfuse = !mma && qfuse_use(c, a.U_q, a.U_k, H, dh);
    // the step's new latents: requantized and stored by the query kernel itself
    // where it can, else by their own launch first
    const bool fresh_q = a.c_hat && !mma && !qfuse && qproj_fresh_supported(c, a.U_q);
    if (a.c_hat && !fresh_q) {
        e = launch_requant_len(a.c_hat, B, r, c.bits, a.lat_clip, c, a.seq_len, err, s);
        if (e != cudaSuccess) return e;
    }
    if (qfuse) {
        e = launch_qfuse(c, a.seq_len, a.U_q, a.U_k, H, dh, w.qt, local_qmax ? nullptr : w.qmax, err, s);
    } else {
        e = mma ? launch_qproj_mma(c, a.seq_len, static_cast<const uint16_t *>(a.U_q.w), d, w.q, w.qmax, B * H, err, s)
                : launch_qproj(c, a.seq_len, a.U_q, d, w.q, w.qmax, B * H, err, s, fresh_q ? a.c_hat : nullptr,
                               a.lat_clip);
        if (e != cudaSuccess) return e;
        e = mma ? launch_qabsorb_mma(w.q, static_cast<const uint16_t *>(a.U_k.w), B, r, d, H, dh, w.qt, w.qmax, s)
                : launch_qabsorb(w.q, a.U_k, B, r, d, H, dh, w.qt, w.qmax, err, s);
    }
    if (e != cudaSuccess) return e;

    int chunk = chunk_tokens(a.max_seq_len);
    int ns = (a.max_seq_len + chunk - 1) / chunk;
    if (attn_mma_use(c, H, B, a.max_seq_len) && attn_mma_fits(c, a.max_seq_len)) {
        // a6/a7 on the warp-level tensor-core MMA: one partial per range of ts tokens
        int ts = 16, n_sub = 1;
        ns = attn_mma_splits(c, B, H, a.max_seq_len, &ts, &n_sub);
        chunk = ts * n_sub;
        e = launch_attn_mma(c, a.seq_len, w.qt, qfuse && local_qmax ? nullptr : w.qmax, H, a.softmax_scale, ts,
                            n_sub, ns, w.pm, w.pl, w.po, err, s);
        if (e != cudaSuccess) return e;
        prof_mark(s, "attn_mma");
    } else if (attn_tc_use(c, H, a.max_seq_len)) {
        // a6/a7 on the tensor cores: splits of whole 128-token tiles
        int per = 1;
        ns = attn_tc_splits(B, c.r, a.max_seq_len, &per);
        chunk = per * 128;
        e = launch_attn_tc(c, a.seq_len, w.qt, w.qmax, H, a.softmax_scale, per, ns, w.pm, w.pl, w.po, err, s);
        if (e != cudaSuccess) return e;
        prof_mark(s, "attn_tc");
    } else {
        const int row_bytes = c.bits == 8 ? r : r / 2;
        int sub = kSubTileBytes / row_bytes;
        sub = sub < 8 ? 8 : (sub > 16 ? 16 : sub & ~7);
        if (sub > chunk) sub = chunk;
        const size_t smem_a = (size_t(kHG) * r + size_t(kHG) * sub + 2 * sub) * sizeof(float) +
                              2 * size_t(sub) * row_bytes;
        dim3 grid_a(ns, B, (H + kHG - 1) / kHG);
        if (c.bits == 8) {
            e = ensure_smem(attn_chunk_kernel<8>, smem_a);
            if (e == cudaSuccess)
                e = launch_pdl(attn_chunk_kernel<8>, grid_a, dim3(kAtThreads), smem_a, s, c, a.seq_len, w.qt, H,
                               a.softmax_scale, chunk, sub, ns, w.pm, w.pl, w.po, err);
        } else {
            e = ensure_smem(attn_chunk_kernel<4>, smem_a);
            if (e == cudaSuccess)
                e = launch_pdl(attn_chunk_kernel<4>, grid_a, dim3(kAtThreads), smem_a, s, c, a.seq_len, w.qt, H,
                               a.softmax_scale, chunk, sub, ns, w.pm, w.pl, w.po, err);
        }
        if (e != cudaSuccess) return e;
        prof_mark(s, "attn_chunk");
    }
    if (mma)
        return launch_combine_mma(a.seq_len, c.seq_map, c.nseq, B, c.Tmax, H, dh, r, chunk, ns, w.pm, w.pl, w.po,
                                  static_cast<const uint16_t *>(a.U_v.w), a.O, s);
    return launch_combine_uv(a.seq_len, c.seq_map, c.nseq, B, c.Tmax, H, dh, r, chunk, ns, w.pm, w.pl, w.po, a.U_v,
                             a.O, err, s);
}

}  // namespace qsvd
