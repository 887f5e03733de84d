// Offline preparation (Sec. 3.2): importance scores of the joint SVD's
// singular values, Eq. 10:
//
//   score_i = (1/N) sum_n ( sigma_i [U^T G_n V]_{ii} )^2,
//   [U^T G V]_{ii} = sum_j U[j, i] sum_l G[j, l] V^T[i, l].
//
// diag_tc_kernel (the tensor-core path): one CTA per (128 singular values i,
// 256 rows j, sample n) forms P^T[i, j] = sum_l V^T[i, l] G[j, l] with
// tcgen05.mma kind::tf32 in the 3xTF32 split: every fp32 operand x is
// x_hi + x_lo with x_hi = x with its low 13 mantissa bits cleared (exact in
// tf32) and x_lo = x - x_hi (exact in fp32), and P^T accumulates
// hi*hi + hi*lo + lo*hi in fp32 tensor memory (the dropped lo*lo term is below
// 2^-20 of each product), so the result keeps fp32-level accuracy.  TMA
// brings 32-column fp32 tiles of both operands; the raw tile is the hi
// operand as it stands (a tf32 product reads the upper 19 bits of each word),
// and four converter warps write the lo image beside it; the epilogue (thread = i)
// writes sum_j U[j, i] P^T[i, j] over the CTA's 128 rows as part[n, jt, i].
// diag_kernel (CUDA cores, for row lengths n that TMA cannot stride: n % 4
// != 0): one CTA per (64 i, 64 j, n) accumulating P[j, i] over 32-wide
// chunks of l staged in shared memory (each thread a 4 x 4 block of (j, i)).
// score_kernel adds the row tiles in order (the result does not depend on
// scheduling: the same bits every run), squares and averages.
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
#include "tcgen05.cuh"

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

namespace imp {
constexpr int kTile = 128;                                 // i per CTA (tensor-memory lanes)
constexpr int kTileJ = 256;                                // j per CTA (accumulator columns)
constexpr int kKs = 32;                                    // fp32 columns of l per stage (one 128-byte row)
constexpr int kImg = kTile * kKs * 4;                      // 16 KiB: one image of the A (V^T) tile of a stage
constexpr int kImgB = kTileJ * kKs * 4;                    // 32 KiB: one image of the B (G) tile
constexpr int kStages = 2;
constexpr int kThreads = 192;                              // TMA, MMA, 4 converter / epilogue warps
constexpr int kStage = 2 * kImg + 2 * kImgB;               // per stage: A hi, A lo, B hi, B lo
constexpr size_t kSmem = size_t(kStages) * kStage + 1024;
}  // namespace imp

__global__ void __launch_bounds__(imp::kThreads, 1)
diag_tc_kernel(const __grid_constant__ CUtensorMap map_v, const __grid_constant__ CUtensorMap map_g,
               const float *__restrict__ U, int m, int n, int k, float *__restrict__ part, int *err) {
    using namespace imp;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t full[kStages], conv[kStages], empty[kStages], acc_full;
    __shared__ uint32_t tmem_base;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int i0 = blockIdx.x * kTile, j0 = blockIdx.y * kTileJ, smp = blockIdx.z;
    const int n_k = (n + kKs - 1) / kKs;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full[s], 1);        // both raw tiles landed
            mbar_init(&conv[s], 4);        // hi / lo images written (one arrival per converter warp)
            mbar_init(&empty[s], 1);       // the stage's products completed
        }
        mbar_init(&acc_full, 1);
        mbar_init_fence();
        tc::prefetch_map(&map_v);
        tc::prefetch_map(&map_g);
    }
    if (warp == 1) tc::tmem_alloc(&tmem_base, kTileJ);
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tmem = tmem_base;

    if (warp == 0) {
        if (lane == 0) {
            for (int it = 0; it < n_k; ++it) {
                const int s = it % kStages;
                if (it >= kStages && !tc::wait(&empty[s], ((it / kStages) - 1) & 1, err)) break;
                uint8_t *st = smem + size_t(s) * kStage;
                mbar_arrive_expect_tx(&full[s], kImg + kImgB);
                tc::tma_load_2d(st, &map_v, it * kKs, i0, &full[s]);                       // V^T rows i
                tc::tma_load_2d(st + 2 * kImg, &map_g, it * kKs, smp * m + j0, &full[s]);  // G_n rows j
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_tf32f32(kTileJ);
            bool ok = true;
            for (int it = 0; it < n_k && ok; ++it) {
                const int s = it % kStages;
                if (!(ok = tc::wait(&conv[s], (it / kStages) & 1, err))) break;
                tc::fence_after();
                const uint32_t a_hi = smem_addr(smem + size_t(s) * kStage), a_lo = a_hi + kImg;
                const uint32_t b_hi = a_hi + 2 * kImg, b_lo = b_hi + kImgB;
#pragma unroll
                for (int kk = 0; kk < kKs / 8; ++kk) {
                    const uint32_t o = kk * 32;
                    tc::mma_ss_tf32(tmem, tc::desc_sw128(a_lo + o), tc::desc_sw128(b_hi + o), idesc,
                                    (it > 0 || kk > 0) ? 1u : 0u);
                    tc::mma_ss_tf32(tmem, tc::desc_sw128(a_hi + o), tc::desc_sw128(b_lo + o), idesc, 1u);
                    tc::mma_ss_tf32(tmem, tc::desc_sw128(a_hi + o), tc::desc_sw128(b_hi + o), idesc, 1u);
                }
                tc::commit(&empty[s]);
            }
            if (ok) tc::commit(&acc_full);
        }
    } else {
        // converters: the raw tile serves as the hi operand (the tf32 product
        // reads only the upper 19 bits of each fp32 word, x with its low 13
        // mantissa bits cleared); the lo image x - hi goes to the next image
        // (same byte offsets, so the swizzle carries over)
        const int ct = threadIdx.x - 64;
        bool ok = true;
        auto split = [](uint8_t *img, int img_bytes, int ct) {
#pragma unroll 4
            for (int c = ct; c < img_bytes / 16; c += 128) {
                const float4 v = *reinterpret_cast<const float4 *>(img + size_t(c) * 16);
                const float4 lo = make_float4(v.x - __uint_as_float(__float_as_uint(v.x) & 0xFFFFE000u),
                                              v.y - __uint_as_float(__float_as_uint(v.y) & 0xFFFFE000u),
                                              v.z - __uint_as_float(__float_as_uint(v.z) & 0xFFFFE000u),
                                              v.w - __uint_as_float(__float_as_uint(v.w) & 0xFFFFE000u));
                *reinterpret_cast<float4 *>(img + img_bytes + size_t(c) * 16) = lo;
            }
        };
        for (int it = 0; it < n_k; ++it) {
            const int s = it % kStages;
            if (!(ok = tc::wwait(&full[s], (it / kStages) & 1, err))) break;
            uint8_t *st = smem + size_t(s) * kStage;
            split(st, kImg, ct);
            split(st + 2 * kImg, kImgB, ct);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // generic writes -> tensor core reads
            __syncwarp();
            if (lane == 0) tc::arrive(&conv[s]);
        }
        // epilogue: thread = singular value i (tensor-memory lane), 128 columns j
        const int quad = warp & 3, i = i0 + quad * 32 + lane;
        if (ok) ok = tc::wwait(&acc_full, 0, err);
        tc::fence_after();
        if (ok) {
            float acc = 0.0f;
#pragma unroll 1
            for (int q = 0; q < kTileJ / 32; ++q) {
                uint32_t v[32];
                tc::tmem_ld32(tmem + (uint32_t(quad * 32) << 16) + q * 32, v);
                tc::tmem_wait_ld();
#pragma unroll
                for (int c = 0; c < 32; ++c) {
                    const int j = j0 + q * 32 + c;
                    if (j < m && i < k) acc = fmaf(U[size_t(j) * k + i], __uint_as_float(v[c]), acc);
                }
            }
            if (i < k) part[(size_t(smp) * gridDim.y + blockIdx.y) * k + i] = acc;
        }
    }
    tc::fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after();
        tc::tmem_free(tmem, kTileJ);
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
                              int k, float *scores, float *part, int *err, cudaStream_t s) {
    int jt;
    cudaError_t e;
    CUtensorMap mv, mg;
    // TMA needs 16-byte row strides (n % 4 == 0) and 16-byte aligned bases
    const bool tc_path = n % 4 == 0 && (reinterpret_cast<uintptr_t>(Vt) & 15) == 0 &&
                         (reinterpret_cast<uintptr_t>(G) & 15) == 0 && tensor_maps_available() &&
                         encode_map_2d(&mv, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, Vt, uint64_t(n), uint64_t(k),
                                       uint64_t(n) * 4, imp::kKs, imp::kTile, CU_TENSOR_MAP_SWIZZLE_128B) &&
                         encode_map_2d(&mg, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, G, uint64_t(n), uint64_t(N) * m,
                                       uint64_t(n) * 4, imp::kKs, imp::kTileJ, CU_TENSOR_MAP_SWIZZLE_128B);
    if (tc_path) {
        jt = (m + imp::kTileJ - 1) / imp::kTileJ;
        if ((e = ensure_smem(diag_tc_kernel, imp::kSmem)) != cudaSuccess) return e;
        diag_tc_kernel<<<dim3((k + imp::kTile - 1) / imp::kTile, jt, N), imp::kThreads, imp::kSmem, s>>>(
            mv, mg, U, m, n, k, part, err);
    } else {
        jt = (m + kImpTile - 1) / kImpTile;
        diag_kernel<<<dim3((k + kImpTile - 1) / kImpTile, jt, N), 256, 0, s>>>(U, Vt, G, m, n, k, part);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    prof_mark(s, "importance_diag");
    score_kernel<<<(k + 127) / 128, 128, 0, s>>>(part, sigma, N, k, jt, scores);
    e = cudaGetLastError();
    prof_mark(s, "importance_score");
    return e;
}

}  // namespace qsvd
