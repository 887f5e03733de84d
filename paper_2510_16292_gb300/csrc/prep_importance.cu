// Offline preparation (Sec. 3.2): importance scores of the joint SVD's
// singular values, Eq. 10:
//
//   score_i = (1/N) sum_n ( sigma_i [U^T G_n V]_{ii} )^2,
//   [U^T G V]_{ii} = sum_j U[j, i] sum_l G[j, l] V^T[i, l].
//
// diag_kernel: one CTA per (64 singular values i, 64 rows j, sample n)
// accumulates P[j, i] = sum_l G[j, l] V^T[i, l] over 32-wide chunks of l
// staged in shared memory (each thread a 4 x 4 block of (j, i)), then adds
// sum_j U[j, i] P[j, i] over its 64 rows into t[n, i] (fp32 atomics: the sum
// order varies between runs).  score_kernel squares and averages.  fp32
// throughout on the CUDA cores: the gradients need fp32 range, and this runs
// once per layer offline.
#include "common.cuh"
#include "launch.h"

namespace qsvd {

constexpr int kImpTile = 64, kImpK = 32;

__global__ void __launch_bounds__(256)
diag_kernel(const float *__restrict__ U, const float *__restrict__ Vt, const float *__restrict__ G, int m, int n,
            int k, float *__restrict__ t) {
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
        if (i < k) atomicAdd(t + size_t(smp) * k + i, s);
    }
}

__global__ void score_kernel(const float *__restrict__ t, const float *__restrict__ sigma, int N, int k,
                             float *__restrict__ scores) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= k) return;
    float acc = 0.0f;
    for (int smp = 0; smp < N; ++smp) {
        const float v = sigma[i] * t[size_t(smp) * k + i];
        acc = fmaf(v, v, acc);
    }
    scores[i] = acc / float(N);
}

cudaError_t launch_importance(const float *U, const float *sigma, const float *Vt, const float *G, int N, int m, int n,
                              int k, float *scores, float *t, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(t, 0, size_t(N) * k * sizeof(float), s);
    if (e != cudaSuccess) return e;
    diag_kernel<<<dim3((k + kImpTile - 1) / kImpTile, (m + kImpTile - 1) / kImpTile, N), 256, 0, s>>>(U, Vt, G, m, n,
                                                                                                       k, t);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    prof_mark(s, "importance_diag");
    score_kernel<<<(k + 127) / 128, 128, 0, s>>>(t, sigma, N, k, scores);
    e = cudaGetLastError();
    prof_mark(s, "importance_score");
    return e;
}

}  // namespace qsvd
