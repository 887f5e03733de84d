// Decode attention over the latent cache on the CUDA cores (Eq. 5 with U_k
// absorbed into the query and U_v applied last), as a chain of four kernels
// linked by programmatic dependent launch.  Each kernel lets the next one
// launch immediately, prefetches its share of the weights into L2, waits for
// its predecessor, then pulls its weight tile into shared memory with bulk
// asynchronous copies (one mbarrier per CTA, bounded waits).
//
//   qproj_kernel      a5: q[b] = c_{L-1} U_q  per (64-row, 256-column) tile of
//                     U_q; the last CTA of a column block sums the row-block
//                     partials in order
//   qabsorb_kernel    a5: qt[b, h, j] = U_k[j, h-block] . q_h  per 8 rows of U_k
//   attn_chunk_kernel a6/a7: per (b, token chunk, head group): online-softmax
//                     pass over the chunk's cache rows, giving (max, sum,
//                     unnormalised sum_t p_t c_t) per head
//   combine_uv_kernel a7/a8: per (head, 128-row block of U_v): merge the chunk
//                     partials, divide by the softmax denominator, multiply by
//                     the U_v block; the last CTA of a head sums the blocks
#include <cfloat>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

constexpr int kMaxSplits = 64;   // token chunks per sequence
constexpr int kHG = 2;           // heads per attention CTA
constexpr int kAtThreads = 256;
constexpr int kMaxRank = 3072;   // 3 float4 quads per thread in attn_chunk_kernel
constexpr int kQpRows = 128;     // U_q tile rows
constexpr int kQpCols = 256;     // U_q tile columns
constexpr int kRowBlock = 128;   // U_v rows per combine CTA
constexpr int kSubTileBytes = 24 * 1024;

static inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

static int chunk_tokens(int max_seq_len) {
    int c = 32;
    while ((max_seq_len + c - 1) / c > kMaxSplits) c += 32;
    return c;
}

struct DecodeWs {
    int *counters;     // [d / kQpCols] qproj column blocks, then [H] combine heads
    float *qpart, *q, *qt, *pm, *pl, *po, *opart;
};

static size_t carve(int B, int max_seq_len, int r, int H, int dh, char *base, DecodeWs *w) {
    const int chunk = chunk_tokens(max_seq_len);
    const int ns = (max_seq_len + chunk - 1) / chunk;
    const int nrb = (r + kRowBlock - 1) / kRowBlock;
    const int nqr = (r + kQpRows - 1) / kQpRows;
    const int d = H * dh;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *p = base ? base + off : nullptr;
        off += align256(bytes);
        return p;
    };
    DecodeWs t;
    t.counters = reinterpret_cast<int *>(take(size_t(d / kQpCols + H) * 4));
    t.qpart = reinterpret_cast<float *>(take(size_t(nqr) * B * d * 4));
    t.q = reinterpret_cast<float *>(take(size_t(B) * d * 4));
    t.qt = reinterpret_cast<float *>(take(size_t(B) * H * r * 4));
    t.pm = reinterpret_cast<float *>(take(size_t(B) * ns * H * 4));
    t.pl = reinterpret_cast<float *>(take(size_t(B) * ns * H * 4));
    t.po = reinterpret_cast<float *>(take(size_t(B) * ns * H * r * 4));
    t.opart = reinterpret_cast<float *>(take(size_t(B) * H * nrb * dh * 4));
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
// a5 (first half).  CTA = tile [kQpRows rows x kQpCols columns] of U_q; 256
// threads, one column each.  Partial q of the tile -> qpart[row block]; the
// last CTA of a column block adds the row-block partials in order.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
qproj_kernel(CacheView c, const int32_t *__restrict__ seq_len, int B, const uint16_t *__restrict__ Uq, int d,
             float *__restrict__ qpart, float *__restrict__ q, int *__restrict__ counters, int *err) {
    extern __shared__ __align__(128) uint16_t u_s[];             // [kQpRows][kQpCols]  64 KiB
    __shared__ float c_s[kQpRows];
    __shared__ __align__(8) uint64_t bar;
    __shared__ int last;
    const int r = c.r;
    const int rb = blockIdx.x, cb = blockIdx.y;
    const int j0 = rb * kQpRows, c0 = cb * kQpCols;
    const int rows = min(kQpRows, r - j0);
    pdl_trigger();
    prefetch_share_l2(Uq, size_t(r) * d * 2, size_t(cb) * gridDim.x + rb, size_t(gridDim.x) * gridDim.y);
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    pdl_wait();
    if (threadIdx.x < 32) {
        if (threadIdx.x == 0) mbar_arrive_expect_tx(&bar, uint32_t(rows) * kQpCols * 2);
        __syncwarp();
        for (int i = threadIdx.x; i < rows; i += 32)
            bulk_g2s(u_s + i * kQpCols, Uq + size_t(j0 + i) * d + c0, kQpCols * 2, &bar);
    }
    mbar_wait(&bar, 0, err);
    const int col = threadIdx.x;
    const int nqr = gridDim.x;
    for (int b = 0; b < B; ++b) {
        int L = seq_len[b];
        if (!valid_len(L, c.Tmax)) {
            if (threadIdx.x == 0 && rb == 0 && cb == 0) flag_error(err, kErrRange);
            L = 0;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < rows; i += blockDim.x)
            c_s[i] = L ? cache_value(c, size_t(b) * c.Tmax + (L - 1), j0 + i) : 0.0f;
        __syncthreads();
        float acc = 0.0f;
#pragma unroll 16
        for (int i = 0; i < rows; ++i) acc = fmaf(c_s[i], bf16_to_f32(u_s[i * kQpCols + col]), acc);
        qpart[(size_t(rb) * B + b) * d + c0 + col] = acc;
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) last = atomicAdd(&counters[cb], 1) == nqr - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();
    for (int b = 0; b < B; ++b) {
        float s = 0.0f;
        for (int k0 = 0; k0 < nqr; k0 += 8) {        // 8 independent loads in flight
            float v[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) v[k] = k0 + k < nqr ? qpart[(size_t(k0 + k) * B + b) * d + c0 + col] : 0.0f;
#pragma unroll
            for (int k = 0; k < 8; ++k) s += v[k];
        }
        q[size_t(b) * d + c0 + col] = s;
    }
    if (threadIdx.x == 0) counters[cb] = 0;
}

// ---------------------------------------------------------------------------
// a5 (second half): qt[b, h, j] = sum_i U_k[j, h*dh + i] * q[b, h*dh + i].
// CTA = 8 rows of U_k (one warp each) copied to smem; q[b] staged per b.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
qabsorb_kernel(const float *__restrict__ q, const uint16_t *__restrict__ Uk, int B, int r, int d, int H, int dh,
               float *__restrict__ qt, int *err) {
    extern __shared__ __align__(16) uint8_t smem[];
    uint16_t *u_s = reinterpret_cast<uint16_t *>(smem);            // [8][d]
    float *q_s = reinterpret_cast<float *>(smem + size_t(8) * d * 2);  // [d]
    __shared__ __align__(8) uint64_t bar;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int j0 = blockIdx.x * 8;
    const int rows = min(8, r - j0);
    pdl_trigger();
    prefetch_share_l2(Uk, size_t(r) * d * 2, blockIdx.x, gridDim.x);
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    pdl_wait();
    if (threadIdx.x == 0) {
        mbar_arrive_expect_tx(&bar, uint32_t(rows) * d * 2);
        bulk_g2s(u_s, Uk + size_t(j0) * d, uint32_t(rows) * d * 2, &bar);
    }
    mbar_wait(&bar, 0, err);
    const int seg = dh / 8;
    const int j = j0 + warp;
    for (int b = 0; b < B; ++b) {
        __syncthreads();
        for (int i = threadIdx.x * 4; i < d; i += 256 * 4)
            *reinterpret_cast<float4 *>(q_s + i) = *reinterpret_cast<const float4 *>(q + size_t(b) * d + i);
        __syncthreads();
        if (warp >= rows) continue;
        for (int base = 0; base < d; base += 256) {
            const int col = base + lane * 8;
            float f[8];
            unpack8_bf16(*reinterpret_cast<const uint4 *>(u_s + size_t(warp) * d + col), f);
            const float4 q0 = *reinterpret_cast<const float4 *>(q_s + col);
            const float4 q1 = *reinterpret_cast<const float4 *>(q_s + col + 4);
            float p = f[0] * q0.x + f[1] * q0.y + f[2] * q0.z + f[3] * q0.w +
                      f[4] * q1.x + f[5] * q1.y + f[6] * q1.z + f[7] * q1.w;
            for (int o = seg >> 1; o; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
            if ((lane % seg) == 0) qt[(size_t(b) * H + col / dh) * r + j] = p;
        }
    }
}

// ---------------------------------------------------------------------------
// a6/a7: one CTA per (token chunk, sequence, group of kHG heads).  The chunk
// is streamed through shared memory in sub-tiles (double-buffered bulk
// copies); scores and the latent sum use an online softmax per head.
// ---------------------------------------------------------------------------
template <int BITS>
__global__ void __launch_bounds__(kAtThreads)
attn_chunk_kernel(CacheView c, const int32_t *__restrict__ seq_len, const float *__restrict__ qt, int H,
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
    if (blockIdx.z == 0 && threadIdx.x == 0 && t_begin < c.Tmax) {
        const int rows = min(chunk, c.Tmax - t_begin);
        const char *base = static_cast<const char *>(c.codes) + (size_t(b) * c.Tmax + t_begin) * row_bytes;
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
    const int L = seq_len[b];
    if (!valid_len(L, c.Tmax) || t_begin >= L) return;        // invalid lengths are flagged by qproj_kernel
    const int n = min(L, t_begin + chunk) - t_begin;
    const int n_sub = (n + sub - 1) / sub;

    auto issue = [&](int st, int buf) {                       // thread 0 only
        const int t0 = t_begin + st * sub;
        const int rows = min(sub, t_begin + n - t0);
        const size_t slot0 = size_t(b) * c.Tmax + t0;
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
                              (size_t(b) * c.Tmax + t_begin + st * sub) * (r / 128);   // int4 group scales
        float *tsc = ts + buf * sub;
        if (BITS == 8 && threadIdx.x < rows)
            tsc[threadIdx.x] = static_cast<const float *>(c.scales)[size_t(b) * c.Tmax + t_begin + st * sub + threadIdx.x];
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
// a7/a8: one CTA per (head, 128-row block of U_v), looping over sequences.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128)
combine_uv_kernel(const int32_t *__restrict__ seq_len, int B, int Tmax, int H, int dh, int r, int chunk, int n_split,
                  const float *__restrict__ pm, const float *__restrict__ pl, const float *__restrict__ po,
                  const uint16_t *__restrict__ Uv, float *__restrict__ opart, int *__restrict__ counters,
                  float *__restrict__ O, int *err) {
    __shared__ __align__(128) uint16_t u_s[kRowBlock * 128];    // [rows][dh]  32 KiB
    __shared__ float ol[kRowBlock];
    __shared__ float wsp[kMaxSplits];
    __shared__ float inv_l;
    __shared__ __align__(8) uint64_t bar;
    __shared__ int last;
    const int h = blockIdx.x, rb = blockIdx.y, d = H * dh;
    const int nrb = gridDim.y;
    const int j0 = rb * kRowBlock;
    const int rows = min(kRowBlock, r - j0);
    pdl_trigger();
    prefetch_share_l2(Uv, size_t(r) * d * 2, size_t(rb) * H + h, size_t(nrb) * H);
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        mbar_init_fence();
    }
    __syncthreads();
    pdl_wait();
    if (threadIdx.x == 0) mbar_arrive_expect_tx(&bar, uint32_t(rows) * dh * 2);
    __syncthreads();
    for (int i = threadIdx.x; i < rows; i += blockDim.x)
        bulk_g2s(u_s + i * dh, Uv + size_t(j0 + i) * d + h * dh, dh * 2, &bar);
    mbar_wait(&bar, 0, err);
    for (int b = 0; b < B; ++b) {
        const int L = seq_len[b];
        float *part = opart + ((size_t(b) * H + h) * nrb + rb) * dh;
        if (!valid_len(L, Tmax)) {
            for (int i = threadIdx.x; i < dh; i += blockDim.x) part[i] = 0.0f;
            continue;
        }
        const int ns = (L + chunk - 1) / chunk;
        const size_t base = size_t(b) * n_split * H + h;
        __syncthreads();
        if (threadIdx.x < 32) {                 // ns <= 64: two partials per lane
            const int lane = threadIdx.x;
            const float m0 = lane < ns ? pm[base + size_t(lane) * H] : -FLT_MAX;
            const float m1 = lane + 32 < ns ? pm[base + size_t(lane + 32) * H] : -FLT_MAX;
            const float l0 = lane < ns ? pl[base + size_t(lane) * H] : 0.0f;
            const float l1 = lane + 32 < ns ? pl[base + size_t(lane + 32) * H] : 0.0f;
            const float M = warp_max(fmaxf(m0, m1));
            const float w0 = lane < ns ? expf(m0 - M) : 0.0f;
            const float w1 = lane + 32 < ns ? expf(m1 - M) : 0.0f;
            wsp[lane] = w0;
            wsp[lane + 32] = w1;
            const float l = warp_sum(w0 * l0 + w1 * l1);
            if (lane == 0) inv_l = 1.0f / l;
        }
        __syncthreads();
        for (int jj = threadIdx.x; jj < rows; jj += blockDim.x) {
            float o = 0.0f;
            for (int s0 = 0; s0 < ns; s0 += 8) {       // 8 independent loads in flight
                float v[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) v[k] = s0 + k < ns ? po[(base + size_t(s0 + k) * H) * r + j0 + jj] : 0.0f;
#pragma unroll
                for (int k = 0; k < 8; ++k) o = fmaf(s0 + k < ns ? wsp[s0 + k] : 0.0f, v[k], o);
            }
            ol[jj] = o * inv_l;
        }
        __syncthreads();
        for (int i = threadIdx.x; i < dh; i += blockDim.x) {
            float acc = 0.0f;
#pragma unroll 8
            for (int jj = 0; jj < rows; ++jj) acc = fmaf(ol[jj], bf16_to_f32(u_s[jj * dh + i]), acc);
            part[i] = acc;
        }
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) last = atomicAdd(&counters[h], 1) == nrb - 1;
    __syncthreads();
    if (!last) return;
    __threadfence();
    for (int b = 0; b < B; ++b) {
        const float *all = opart + (size_t(b) * H + h) * nrb * dh;
        for (int i = threadIdx.x; i < dh; i += blockDim.x) {
            float s = 0.0f;
            for (int k0 = 0; k0 < nrb; k0 += 8) {
                float v[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) v[k] = k0 + k < nrb ? all[size_t(k0 + k) * dh + i] : 0.0f;
#pragma unroll
                for (int k = 0; k < 8; ++k) s += v[k];
            }
            O[size_t(b) * d + h * dh + i] = s;
        }
    }
    if (threadIdx.x == 0) counters[h] = 0;
}

// ---------------------------------------------------------------------------
cudaError_t launch_decode(const DecodeArgs &a, void *ws, size_t ws_bytes, int *err, cudaStream_t s) {
    const CacheView &c = a.cache;
    const int B = c.B, r = c.r, H = a.H, dh = a.dh, d = H * dh;
    DecodeWs w;
    carve(B, a.max_seq_len, r, H, dh, static_cast<char *>(ws), &w);
    const int chunk = chunk_tokens(a.max_seq_len);
    const int ns = (a.max_seq_len + chunk - 1) / chunk;
    const int nrb = (r + kRowBlock - 1) / kRowBlock;
    const int nqr = (r + kQpRows - 1) / kQpRows;
    cudaError_t e;

    const size_t smem_q = size_t(kQpRows) * kQpCols * 2;
    e = ensure_smem(qproj_kernel, smem_q);
    if (e != cudaSuccess) return e;
    e = launch_pdl(qproj_kernel, dim3(nqr, d / kQpCols), dim3(256), smem_q, s, c, a.seq_len, B, a.U_q, d, w.qpart,
                   w.q, w.counters, err);
    if (e != cudaSuccess) return e;
    prof_mark(s, "qproj");

    const size_t smem_k = size_t(8) * d * 2 + size_t(d) * 4;
    e = ensure_smem(qabsorb_kernel, smem_k);
    if (e != cudaSuccess) return e;
    e = launch_pdl(qabsorb_kernel, dim3((r + 7) / 8), dim3(256), smem_k, s, w.q, a.U_k, B, r, d, H, dh, w.qt, err);
    if (e != cudaSuccess) return e;
    prof_mark(s, "qabsorb");

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

    e = launch_pdl(combine_uv_kernel, dim3(H, nrb), dim3(128), 0, s, a.seq_len, B, c.Tmax, H, dh, r, chunk, ns, w.pm,
                   w.pl, w.po, a.U_v, w.opart, w.counters + d / kQpCols, a.O, err);
    if (e != cudaSuccess) return e;
    prof_mark(s, "combine_uv");
    return cudaSuccess;
}

}  // namespace qsvd
