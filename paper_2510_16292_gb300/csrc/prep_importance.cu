// Offline preparation (Sec. 3.2): importance scores of the joint SVD's
// singular values, Eq. 10:
//
//   score_i = (1/N) sum_n ( sigma_i [U^T G_n V]_{ii} )^2,
//   [U^T G V]_{ii} = sum_j U[j, i] sum_l G[j, l] V^T[i, l].
//
// diag_kernel: one CTA per (64 singular values i, 64 rows j, sample n)
// accumulates P[j, i] = sum_l G[j, l] V^T[i, l] over 32-wide chunks of l
// staged in shared memory (each thread a 4 x 4 block of (j, i)), then writes
// sum_j U[j, i] P[j, i] over its 64 rows as the partial part[n, jt, i] of row
// tile jt.  score_kernel adds the row tiles in order (the result does not
// depend on scheduling: the same bits every run), squares and averages.  fp32
// throughout on the CUDA cores: the gradients need fp32 range, and this runs
// once per layer offline.
//
// The cross-layer rank budget (the global sort of Sec. 3.2) keeps the k
// highest scores over every layer: rank_hist_kernel / rank_pick_kernel find
// the k-th smallest of the 64-bit keys (descending score, then ascending
// position in the layer-major concatenation, so ties go to the lower layer,
// then the lower index) by an 8-pass radix select over 8-bit digits with
// integer histograms; rank_keep_kernel marks every key at or below it.
#include <algorithm>

#include "common.cuh"
#include "launch.h"

namespace qsvd {

constexpr int kImpTile = 64, kImpK = 32;

__global__ void __launch_bounds__(256)
diag_kernel(const float *__restrict__ U, const float *__restrict__ Vt, const float *__restrict__ G, int m, int n,
            int k, float *__restrict__ part) {
    __shared__ float gs[kImpK][kImpTile + 1];            // [l][j]
    __shared__ float vs[kImpK][kImpTile + 1];            // [l][i]
    __shared__ float red[16][kImpTile];
    const int i0 = blockIdx.x * kImpTile, j0 = blockIdx.y * kImpTile, smp = blockIdx.z;
    const float *Gn = G + size_t(smp) * m * n;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;   // thread owns i = i0 + 4 tx + a, j = j0 + 4 ty + b
    float acc[4][4] = {};
    for (int l0 = 0; l0 < n; l0 += kImpK) {
        for (int e = threadIdx.x; e < kImpK * kImpTile; e += 256) {
            const int r = e / kImpK, l = e - r * kImpK;      // consecutive threads: consecutive l (coalesced rows)
            const int gl = l0 + l;
            gs[l][r] = (j0 + r < m && gl < n) ? Gn[size_t(j0 + r) * n + gl] : 0.0f;
            vs[l][r] = (i0 + r < k && gl < n) ? Vt[size_t(i0 + r) * n + gl] : 0.0f;
        }
        __syncthreads();
#pragma unroll 8
        for (int l = 0; l < kImpK; ++l) {
            float gv[4], vv[4];
#pragma unroll
            for (int b = 0; b < 4; ++b) gv[b] = gs[l][4 * ty + b];
#pragma unroll
            for (int a = 0; a < 4; ++a) vv[a] = vs[l][4 * tx + a];
#pragma unroll
            for (int b = 0; b < 4; ++b)
#pragma unroll
                for (int a = 0; a < 4; ++a) acc[b][a] = fmaf(gv[b], vv[a], acc[b][a]);
        }
        __syncthreads();
    }
    // sum over this CTA's rows j of U[j, i] P[j, i]
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const int i = i0 + 4 * tx + a;
        float part = 0.0f;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int j = j0 + 4 * ty + b;
            if (j < m && i < k) part = fmaf(U[size_t(j) * k + i], acc[b][a], part);
        }
        red[ty][4 * tx + a] = part;
    }
    __syncthreads();
    if (threadIdx.x < kImpTile) {
        float s = 0.0f;
        for (int y = 0; y < 16; ++y) s += red[y][threadIdx.x];
        const int i = i0 + threadIdx.x;
        if (i < k) part[(size_t(smp) * gridDim.y + blockIdx.y) * k + i] = s;
    }
}

__global__ void score_kernel(const float *__restrict__ part, const float *__restrict__ sigma, int N, int k, int jt,
                             float *__restrict__ scores) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= k) return;
    float acc = 0.0f;
    for (int smp = 0; smp < N; ++smp) {
        float t = 0.0f;
        for (int y = 0; y < jt; ++y) t += part[(size_t(smp) * jt + y) * k + i];     // row tiles in order
        const float v = sigma[i] * t;
        acc = fmaf(v, v, acc);
    }
    scores[i] = acc / float(N);
}

// ---------------------------------------------------------------------------
// Rank budget.  key(i) = (descending order of score_i) << 32 | i; k smallest keys kept.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint64_t rank_key(const float *scores, int i) {
    float f = scores[i];
    if (f == 0.0f) f = 0.0f;                                      // -0 sorts as +0
    const uint32_t u = __float_as_uint(f);
    const uint32_t asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u); // ascending with f
    return (uint64_t(~asc) << 32) | uint32_t(i);                  // descending score, then ascending i
}

struct RankState {
    unsigned long long prefix, mask;     // digits fixed so far
    unsigned long long k_rem;            // keys still to take below the fixed prefix
    unsigned int hist[256];
};

__global__ void rank_hist_kernel(const float *__restrict__ scores, int n, int shift, RankState *st) {
    __shared__ unsigned int h[256];
    for (int b = threadIdx.x; b < 256; b += blockDim.x) h[b] = 0u;
    __syncthreads();
    const uint64_t prefix = st->prefix, mask = st->mask;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
        const uint64_t key = rank_key(scores, i);
        if ((key & mask) == prefix) atomicAdd(&h[(key >> shift) & 0xFFu], 1u);
    }
    __syncthreads();
    for (int b = threadIdx.x; b < 256; b += blockDim.x)
        if (h[b]) atomicAdd(&st->hist[b], h[b]);                  // integer counts: exact in any order
}

__global__ void rank_init_kernel(RankState *st, int k) {
    st->hist[threadIdx.x] = 0u;
    if (threadIdx.x == 0) {
        st->prefix = 0ull;
        st->mask = 0ull;
        st->k_rem = (unsigned long long)k;
    }
}

// One CTA of 256 threads: the digit whose bin holds the k_rem-th key.
__global__ void rank_pick_kernel(int shift, RankState *st) {
    __shared__ unsigned long long cum[256];
    const int b = threadIdx.x;
    cum[b] = st->hist[b];
    __syncthreads();
    for (int o = 1; o < 256; o <<= 1) {                           // inclusive scan
        const unsigned long long v = b >= o ? cum[b - o] : 0ull;
        __syncthreads();
        cum[b] += v;
        __syncthreads();
    }
    const unsigned long long before = b ? cum[b - 1] : 0ull, k = st->k_rem;
    __syncthreads();
    if (before < k && k <= cum[b]) {
        st->k_rem = k - before;
        st->prefix |= (unsigned long long)b << shift;
        st->mask |= 0xFFull << shift;
    }
    st->hist[b] = 0u;
}

__global__ void rank_keep_kernel(const float *__restrict__ scores, int n, const RankState *st, int k,
                                 uint8_t *__restrict__ keep) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) keep[i] = (k > 0 && rank_key(scores, i) <= st->prefix) ? 1 : 0;
}

size_t rank_workspace_bytes() { return (sizeof(RankState) + 255) / 256 * 256; }

cudaError_t launch_rank_budget(const float *scores, int n, int k, uint8_t *keep, void *ws, cudaStream_t s) {
    RankState *st = static_cast<RankState *>(ws);
    rank_init_kernel<<<1, 256, 0, s>>>(st, k);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if (k > 0) {
        const int blocks = std::min((n + 255) / 256, 1024);
        for (int shift = 56; shift >= 0; shift -= 8) {
            rank_hist_kernel<<<blocks, 256, 0, s>>>(scores, n, shift, st);
            rank_pick_kernel<<<1, 256, 0, s>>>(shift, st);
        }
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    rank_keep_kernel<<<(n + 255) / 256, 256, 0, s>>>(scores, n, st, k, keep);
    e = cudaGetLastError();
    prof_mark(s, "rank_budget");
    return e;
}

cudaError_t launch_importance(const float *U, const float *sigma, const float *Vt, const float *G, int N, int m, int n,
                              int k, float *scores, float *part, cudaStream_t s) {
    const int jt = (m + kImpTile - 1) / kImpTile;
    diag_kernel<<<dim3((k + kImpTile - 1) / kImpTile, jt, N), 256, 0, s>>>(U, Vt, G, m, n, k, part);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    prof_mark(s, "importance_diag");
    score_kernel<<<(k + 127) / 128, 128, 0, s>>>(part, sigma, N, k, jt, scores);
    e = cudaGetLastError();
    prof_mark(s, "importance_score");
    return e;
}

}  // namespace qsvd
