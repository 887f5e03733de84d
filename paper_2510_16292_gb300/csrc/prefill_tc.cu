// Causal prefill attention over the latent cache in the materialised form
// (Eq. 5 as written: K = C U_k, V = C U_v, Q = C U_q, then the decoder's
// causal softmax attention), on the 5th-generation tensor cores.
//
// At prefill every prompt token queries its prefix, so the work is a dense
// contraction: regrouping U_k into the query (the absorbed form the decode
// kernels use) would multiply the score and weighted-sum products by r / dh
// (12 to 16 at the LLaVA shapes).  Here the latent rows of a block are
// multiplied once by [U_q U_k U_v] and the attention runs at head size dh.
//
//   ut_kernel        offline: fp16 [3d, r] = [U_q U_k U_v]^T (bf16 in), so
//                    that both GEMM operands are K-major
// Every fp16 rounding (Ut, the int4 latent operand, Q, K, V) saturates at
// +-65504 and flags a range error instead of producing inf.
//   lat_prep_kernel  the latent rows of every block as an fp16 GEMM operand:
//                    int8 codes (exact in fp16) with the token scale kept
//                    for the epilogue, or int4 code x group scale rounded to
//                    fp16 (scale 1); rows padded to 128 per block with zeros
//   qkv_gemm_kernel  [R, r] x [r, 3d] on tcgen05 (M = 128 rows, N = 256
//                    columns, K staged 64 at a time through a TMA ring), one
//                    persistent CTA per SM with two fp32 accumulators in
//                    tensor memory (the epilogue of a tile overlaps the main
//                    loop of the next); the epilogue applies the
//                    token scale and writes Q and K row-major, V transposed
//                    ([d, R], so that a key tile of V is K-major for the
//                    attention's second product), all fp16
//   fa_kernel        one CTA per (pair of 128-query tiles A and B of a
//                    block, head), both tiles against each K/V tile the CTA
//                    loads: S_x = Q_x K^T into tensor memory, causal mask and
//                    online softmax in registers (4 warps per tile, thread =
//                    query row), P_x (fp16) over S_x's columns, O_x += P_x V
//                    with A from tensor memory.  While one tile's softmax
//                    runs, the tensor pipe works on the other tile's
//                    products.  O_x is rescaled only when a row's running
//                    maximum grows by more than 2^8 (otherwise the stale
//                    maximum keeps every p below 2^8); K and V stream through
//                    rings of 2 and 3 tiles.
//
// Every wait is bounded (kErrTimeout on expiry); each CTA frees its tensor
// memory before it exits.
#include <algorithm>
#include <cfloat>
#include <cmath>
#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>

#include "common.cuh"
#include "launch.h"
#include "tcgen05.cuh"

namespace qsvd {

namespace pf {

// Stores of the GEMM's outputs with an L2 evict-first policy: Q, K and V^T
// (3 d x R fp16, hundreds of MB at the 13B batch) would otherwise evict Ut
// (3 d x r fp16) from L2 between the waves of tiles that re-read it.
__device__ __forceinline__ uint64_t evict_first_policy() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ void st_v4_ef(void *p, uint4 v, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.v4.b32 [%0], {%1, %2, %3, %4}, %5;"
                 ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "l"(pol)
                 : "memory");
}
__device__ __forceinline__ void st_u16_ef(void *p, uint16_t v, uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.b16 [%0], %1, %2;" ::"l"(p), "h"(v), "l"(pol) : "memory");
}

// fp16 conversion with the range guard of the materialised operands: a value
// beyond +-65504 (fp16's largest finite) is saturated to it and `over` is set
// (the caller flags kErrRange once), so nothing becomes inf silently.
__device__ __forceinline__ __half2 h2_sat(float a, float b, bool &over) {
    over |= !(fabsf(a) <= 65504.0f) || !(fabsf(b) <= 65504.0f);
    return __floats2half2_rn(fminf(fmaxf(a, -65504.0f), 65504.0f), fminf(fmaxf(b, -65504.0f), 65504.0f));
}

constexpr int kRowTile = 128;           // rows per GEMM tile, queries and keys per attention tile
constexpr int kDh = 128;                // head size of the attention kernel

// ---- Q/K/V GEMM
constexpr int kGemmN = 256, kGemmK = 64;
constexpr int kGemmGroupM = 38;         // row tiles per rasterisation group of qkv_gemm
constexpr int kGemmStageA = kRowTile * kGemmK * 2;       // 16 KiB
constexpr int kGemmStageB = kGemmN * kGemmK * 2;         // 32 KiB
constexpr int kGemmStages = 4;
constexpr int kGemmEpiWarps = 8;                         // 2 x 4 lane quadrants x 128 columns
constexpr int kGemmThreads = 64 + 32 * kGemmEpiWarps;
constexpr size_t kGemmSmem = size_t(kGemmStages) * (kGemmStageA + kGemmStageB) + 1024;

// ---- attention
constexpr int kFaThreads = 384;                          // TMA (Q, K), S MMAs, TMA (V), PV MMAs, 2 x 4 softmax
constexpr int kTileBytes = kRowTile * kDh * 2;           // 32 KiB: 128 rows x 128 fp16 (two 64-column boxes)
constexpr int kBox = kRowTile * 128;                     // 16 KiB: one box (128 rows x 128 bytes)
constexpr int kRingK = 2, kRingV = 3;                    // V tiles are needed a softmax later than K tiles
constexpr size_t kFaSmem = size_t(2 + kRingK + kRingV) * kTileBytes + 1024;
// tensor memory: O_A, O_B (columns 0..255), S_A, S_B (256..511); P_x overwrites S_x's first 64 columns
constexpr uint32_t kColO = 0, kColS = 256, kFaTmemCols = 512;
constexpr float kRescale2 = 8.0f;                        // lazy rescale threshold (log2 units)

}  // namespace pf

// 2^x with the MUFU approximation (relative error about 2^-22; x = -inf and
// x below the fp32 range give +0).
__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// ---------------------------------------------------------------------------
// [U_q U_k U_v]^T in fp16: Ut[n, k] = U_{n / d}[k, n % d]
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
ut_kernel(const uint16_t *__restrict__ Uq, const uint16_t *__restrict__ Uk, const uint16_t *__restrict__ Uv, int r,
          int d, __half *__restrict__ Ut, int *err) {
    __shared__ float tile[32][33];
    const int n0 = blockIdx.x * 32, k0 = blockIdx.y * 32;
    const int part = n0 / d, c0 = n0 - part * d;
    const uint16_t *U = part == 0 ? Uq : (part == 1 ? Uk : Uv);
    for (int i = threadIdx.y; i < 32; i += 8)
        tile[i][threadIdx.x] = bf16_to_f32(U[size_t(k0 + i) * d + c0 + threadIdx.x]);
    __syncthreads();
    bool over = false;
    for (int i = threadIdx.y; i < 32; i += 8)
        Ut[size_t(n0 + i) * r + k0 + threadIdx.x] = __low2half(pf::h2_sat(tile[threadIdx.x][i], 0.0f, over));
    if (over) flag_error(err, kErrRange);
}

// ---------------------------------------------------------------------------
// latent rows of the blocks -> fp16 operand A [R, r] and row scale rs [R]
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256)
lat_prep_kernel(CacheView c, PrefillBlocks bl, int R, __half *__restrict__ A, float *__restrict__ rs, int *err) {
    pdl_wait();
    pdl_trigger();
    const int r = c.r, per_row = r / 8;                       // threads per row: 8 channels each
    const int t = int(blockIdx.x) * blockDim.x + threadIdx.x;      // R * r / 8 < 2^31 (checked by the host)
    if (t >= R * per_row) return;
    const int row = t / per_row, j = (t - row * per_row) * 8;
    int k = 0;
    while (k + 1 < bl.n && bl.row_off[k + 1] <= row) ++k;
    const int p = row - bl.row_off[k];
    const bool live = p < bl.L[k];
    const size_t slot = size_t(bl.seq[k]) * c.Tmax + p;
    uint4 o = make_uint4(0u, 0u, 0u, 0u);
    if (c.bits == 8) {
        if (j == 0) rs[row] = live ? static_cast<const float *>(c.scales)[slot] : 0.0f;
        if (live) {
            const uint2 w = *reinterpret_cast<const uint2 *>(static_cast<const int8_t *>(c.codes) + slot * r + j);
            const uint32_t ws[2] = {w.x, w.y};
            uint32_t h[4];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const __half2 a = __halves2half2(__int2half_rn(int8_t(ws[e] & 0xff)),
                                                 __int2half_rn(int8_t((ws[e] >> 8) & 0xff)));
                const __half2 b = __halves2half2(__int2half_rn(int8_t((ws[e] >> 16) & 0xff)),
                                                 __int2half_rn(int8_t(ws[e] >> 24)));
                h[2 * e] = *reinterpret_cast<const uint32_t *>(&a);
                h[2 * e + 1] = *reinterpret_cast<const uint32_t *>(&b);
            }
            o = make_uint4(h[0], h[1], h[2], h[3]);
        }
    } else {
        if (j == 0) rs[row] = live ? 1.0f : 0.0f;
        if (live) {
            // 8 codes, element i in bits 4i .. 4i+3, times the group's fp16 scale
            const uint32_t w = *reinterpret_cast<const uint32_t *>(static_cast<const uint8_t *>(c.codes) +
                                                                   slot * (r / 2) + j / 2);
            const float s = __half2float(static_cast<const __half *>(c.scales)[slot * (r / 128) + j / 128]);
            uint32_t h[4];
            bool over = false;             // |code| * s reaches 7 * 65504 at most
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int lo = int((w >> (8 * e)) & 0xf), hi = int((w >> (8 * e + 4)) & 0xf);
                const __half2 v = pf::h2_sat(float((lo ^ 8) - 8) * s, float((hi ^ 8) - 8) * s, over);
                h[e] = *reinterpret_cast<const uint32_t *>(&v);
            }
            if (over) flag_error(err, kErrRange);
            o = make_uint4(h[0], h[1], h[2], h[3]);
        }
    }
    *reinterpret_cast<uint4 *>(A + size_t(row) * r + j) = o;
}

// Tile t -> (first row m0, first column n0).  Groups of kGemmGroupM row tiles
// (the last group may be shorter); within a group the row tile runs fastest.
// With 152 CTAs in flight a wave covers about four column tiles of one group:
// ~4 MiB of Ut and the group's 19 MiB of A rows, so each A row tile is read
// from DRAM once and Ut once per group instead of once per wave.
__device__ __forceinline__ void gemm_tile(int t, int tiles_m, int tiles_n, int &m0, int &n0) {
    const int per_group = pf::kGemmGroupM * tiles_n;
    const int g = t / per_group, idx = t - g * per_group;
    const int gm = min(pf::kGemmGroupM, tiles_m - g * pf::kGemmGroupM);
    m0 = (g * pf::kGemmGroupM + idx % gm) * pf::kRowTile;
    n0 = (idx / gm) * pf::kGemmN;
}

// ---------------------------------------------------------------------------
// Q | K | V^T = (A [R, r] x Ut^T [r, 3d]) * rs[row], fp16 out
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(pf::kGemmThreads, 1)
qkv_gemm_kernel(const __grid_constant__ CUtensorMap map_a, const __grid_constant__ CUtensorMap map_b, int R, int r,
                int d, const float *rs, __half *__restrict__ Qm, __half *__restrict__ Km,
                __half *__restrict__ Vt, int *err) {
    // Persistent: CTA c takes tiles c, c + gridDim.x, ...  Tiles are numbered
    // in groups of kGemmGroupM row tiles, row fastest within a group (see
    // gemm_tile), so the CTAs in flight share a few Ut column tiles and a group's
    // A rows stay in L2 while its Ut columns stream past once.  Two
    // tensor-memory accumulators alternate between a CTA's tiles, so the
    // epilogue of one tile overlaps the main loop of the next.
    using namespace pf;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = smem;
    uint8_t *sB = smem + size_t(kGemmStages) * kGemmStageA;
    __shared__ __align__(8) uint64_t full_bar[kGemmStages], empty_bar[kGemmStages], acc_full[2], acc_empty[2];
    __shared__ uint32_t tmem_base;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_k = r / kGemmK;
    const int tiles_m = R / kRowTile, tiles_n = 3 * d / kGemmN, n_tiles = tiles_m * tiles_n;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kGemmStages; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&acc_full[b], 1);
            mbar_init(&acc_empty[b], kGemmEpiWarps);
        }
        mbar_init_fence();
        tc::prefetch_map(&map_a);
        tc::prefetch_map(&map_b);
    }
    if (warp == 1) tc::tmem_alloc(&tmem_base, 2 * kGemmN);
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tmem = tmem_base;
    pdl_wait();
    pdl_trigger();

    if (warp == 0) {
        if (lane == 0) {
            int it = 0;                                       // k-stages issued by this CTA so far
            bool ok = true;
            for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
                int m0, n0;
                gemm_tile(t, tiles_m, tiles_n, m0, n0);
                for (int i = 0; i < n_k; ++i, ++it) {
                    const int s = it % kGemmStages;
                    if (it >= kGemmStages && !(ok = tc::wait(&empty_bar[s], ((it / kGemmStages) - 1) & 1, err)))
                        break;
                    mbar_arrive_expect_tx(&full_bar[s], kGemmStageA + kGemmStageB);
                    tc::tma_load_2d(sA + size_t(s) * kGemmStageA, &map_a, i * kGemmK, m0, &full_bar[s]);
                    tc::tma_load_2d(sB + size_t(s) * kGemmStageB, &map_b, i * kGemmK, n0, &full_bar[s]);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_f16f32(kGemmN);
            bool ok = true;
            int it = 0, ti = 0;
            for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++ti) {
                const int buf = ti & 1;
                if (ti >= 2 && !(ok = tc::wait(&acc_empty[buf], ((ti >> 1) - 1) & 1, err))) break;
                tc::fence_after();
                const uint32_t acc = tmem + uint32_t(buf * kGemmN);
                for (int i = 0; i < n_k; ++i, ++it) {
                    const int s = it % kGemmStages;
                    if (!(ok = tc::wait(&full_bar[s], (it / kGemmStages) & 1, err))) break;
                    tc::fence_after();
                    const uint32_t a0 = smem_addr(sA + size_t(s) * kGemmStageA);
                    const uint32_t b0 = smem_addr(sB + size_t(s) * kGemmStageB);
#pragma unroll
                    for (int ks = 0; ks < kGemmK / 16; ++ks)
                        tc::mma_ss(acc, tc::desc_sw128(a0 + ks * 32), tc::desc_sw128(b0 + ks * 32), idesc,
                                   (i > 0 || ks > 0) ? 1u : 0u);
                    tc::commit(&empty_bar[s]);
                }
                if (ok) tc::commit(&acc_full[buf]);
            }
        }
    } else {
        const int quad = warp & 3, col0 = ((warp - 2) >> 2) * 128;
        const uint64_t pol = evict_first_policy();
        int ti = 0;
        for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++ti) {
            const int buf = ti & 1;
            int m0, n0;
            gemm_tile(t, tiles_m, tiles_n, m0, n0);
            const int row = m0 + quad * 32 + lane;
            if (!tc::wwait(&acc_full[buf], (ti >> 1) & 1, err)) break;
            tc::fence_after();
            const float sc = rs[row];
            const int part = n0 / d, cbase = n0 - part * d + col0;
            const uint32_t taddr = tmem + (uint32_t(quad * 32) << 16) + uint32_t(buf * kGemmN + col0);
#pragma unroll 1
            for (int j0 = 0; j0 < 128; j0 += 32) {
                uint32_t v[32];
                tc::tmem_ld32(taddr + j0, v);
                tc::tmem_wait_ld();
                uint32_t h[16];
                bool over = false;
#pragma unroll
                for (int j = 0; j < 16; ++j) {
                    const __half2 x = h2_sat(__uint_as_float(v[2 * j]) * sc, __uint_as_float(v[2 * j + 1]) * sc, over);
                    h[j] = *reinterpret_cast<const uint32_t *>(&x);
                }
                if (over) flag_error(err, kErrRange);
                if (part < 2) {
                    uint4 *dst = reinterpret_cast<uint4 *>((part == 0 ? Qm : Km) + size_t(row) * d + cbase + j0);
#pragma unroll
                    for (int q = 0; q < 4; ++q) st_v4_ef(dst + q, make_uint4(h[4 * q], h[4 * q + 1], h[4 * q + 2], h[4 * q + 3]), pol);
                } else {
                    // V^T: lanes hold consecutive rows, so each column's 32 stores are contiguous
                    uint16_t *dst = reinterpret_cast<uint16_t *>(Vt) + size_t(cbase + j0) * R + row;
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        st_u16_ef(dst + size_t(2 * j) * R, uint16_t(h[j] & 0xffffu), pol);
                        st_u16_ef(dst + size_t(2 * j + 1) * R, uint16_t(h[j] >> 16), pol);
                    }
                }
            }
            // this warp's columns of the accumulator are drained
            tc::fence_before();
            __syncwarp();
            if (lane == 0) tc::arrive(&acc_empty[buf]);
        }
    }
    tc::fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after();
        tc::tmem_free(tmem, 2 * kGemmN);
    }
}

// ---------------------------------------------------------------------------
// causal attention, one CTA per (pair of 128-query tiles, head)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(pf::kFaThreads, 1)
fa_kernel(const __grid_constant__ CUtensorMap map_q, const __grid_constant__ CUtensorMap map_k,
          const __grid_constant__ CUtensorMap map_vt, PrefillBlocks bl, int d, float c_log2, float *__restrict__ O,
          int *err) {
    using namespace pf;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sQ = smem;                                      // query tiles A and B
    uint8_t *sK = smem + 2 * kTileBytes;                     // [kRingK] tiles
    uint8_t *sV = sK + size_t(kRingK) * kTileBytes;          // [kRingV] tiles (V^T: dh rows x 128 keys)
    __shared__ __align__(8) uint64_t q_full, k_full[pf::kRingK], k_empty[pf::kRingK], v_full[pf::kRingV],
        v_empty[pf::kRingV], s_full[2], p_full[2], o_done[2];
    __shared__ uint32_t tmem_base;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // Work unit: query tiles 2u (A) and 2u + 1 (B, absent past the block's
    // last tile) of one block, units in reverse order (the longest causal rows first).
    int unit = int(gridDim.x) - 1 - int(blockIdx.x), k = 0;
    while (k + 1 < bl.n) {
        const int pairs = (bl.qtile_off[k + 1] - bl.qtile_off[k] + 1) >> 1;
        if (unit < pairs) break;
        unit -= pairs;
        ++k;
    }
    const int L = bl.L[k], row0 = bl.row_off[k];
    const int qs = bl.t0[k] + 2 * unit * kRowTile;                      // position of tile A's first query
    const bool has_b = 2 * unit + 1 < bl.qtile_off[k + 1] - bl.qtile_off[k];
    const int n_a = min(qs + kRowTile - 1, L - 1) / kRowTile + 1;      // key tiles of A
    const int n_b = has_b ? min(qs + 2 * kRowTile - 1, L - 1) / kRowTile + 1 : 0;   // of B (n_a <= n_b)
    const int n = max(n_a, n_b);

    if (threadIdx.x == 0) {
        mbar_init(&q_full, 1);
        for (int s = 0; s < kRingK; ++s) {
            mbar_init(&k_full[s], 1);
            mbar_init(&k_empty[s], 1);
        }
        for (int s = 0; s < kRingV; ++s) {
            mbar_init(&v_full[s], 1);
            mbar_init(&v_empty[s], 1);
        }
        for (int x = 0; x < 2; ++x) {
            mbar_init(&s_full[x], 1);     // S_x of the current key tile is in tensor memory
            mbar_init(&p_full[x], 4);     // P_x written (one arrival per softmax warp of tile x)
            mbar_init(&o_done[x], 1);     // O_x += P_x V has completed (S_x / P_x columns free again)
        }
        mbar_init_fence();
        tc::prefetch_map(&map_q);
        tc::prefetch_map(&map_k);
        tc::prefetch_map(&map_vt);
    }
    if (warp == 1) tc::tmem_alloc(&tmem_base, kFaTmemCols);
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tmem = tmem_base;
    pdl_wait();
    pdl_trigger();
    const int x0 = blockIdx.y * kDh;                         // head's first column in Q and K, row in V^T

    if (warp < 4) {                                          // warpgroup 0: TMA and MMA issue
    if (warp == 0) {
        // ---------------- TMA producer of Q and K ----------------
        if (lane == 0) {
            mbar_arrive_expect_tx(&q_full, (has_b ? 2 : 1) * kTileBytes);
            for (int x = 0; x < (has_b ? 2 : 1); ++x) {
                uint8_t *qd = sQ + size_t(x) * kTileBytes;
                tc::tma_load_2d(qd, &map_q, x0, row0 + qs + x * kRowTile, &q_full);
                tc::tma_load_2d(qd + kBox, &map_q, x0 + 64, row0 + qs + x * kRowTile, &q_full);
            }
            for (int j = 0; j < n; ++j) {
                const int ks = j % kRingK;
                if (j >= kRingK && !tc::wait(&k_empty[ks], ((j / kRingK) - 1) & 1, err)) break;
                mbar_arrive_expect_tx(&k_full[ks], kTileBytes);
                uint8_t *kd = sK + size_t(ks) * kTileBytes;
                tc::tma_load_2d(kd, &map_k, x0, row0 + j * kRowTile, &k_full[ks]);
                tc::tma_load_2d(kd + kBox, &map_k, x0 + 64, row0 + j * kRowTile, &k_full[ks]);
            }
        }
    } else if (warp == 2) {
        // ---------------- TMA producer of V ----------------
        if (lane == 0) {
            for (int j = 0; j < n; ++j) {
                const int vs = j % kRingV;
                if (j >= kRingV && !tc::wait(&v_empty[vs], ((j / kRingV) - 1) & 1, err)) break;
                mbar_arrive_expect_tx(&v_full[vs], kTileBytes);
                uint8_t *vd = sV + size_t(vs) * kTileBytes;
                tc::tma_load_2d(vd, &map_vt, row0 + j * kRowTile, x0, &v_full[vs]);
                tc::tma_load_2d(vd + kBox, &map_vt, row0 + j * kRowTile + 64, x0, &v_full[vs]);
            }
        }
    } else if (warp == 1) {
        // ---------------- S_x = Q_x K^T issuer ----------------
        // S_x of key tile j overwrites P_x of tile j - 1, so it waits for
        // O_x += P_x V of tile j - 1; the other query tile's products fill the
        // tensor pipe meanwhile.  The scores and the O products are issued
        // from two threads (one thread spends ~100 cycles per tcgen05.mma).
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_f16f32(kRowTile);
            bool ok = tc::wait(&q_full, 0, err);
            for (int j = 0; j < n && ok; ++j) {
                const int ks = j % kRingK;
                if (!(ok = tc::wait(&k_full[ks], (j / kRingK) & 1, err))) break;
                const uint32_t k0 = smem_addr(sK + size_t(ks) * kTileBytes);
                for (int x = 0; x < 2 && ok; ++x) {
                    if (j >= (x ? n_b : n_a)) continue;
                    if (j > 0 && !(ok = tc::wait(&o_done[x], (j - 1) & 1, err))) break;
                    tc::fence_after();
                    const uint32_t q0 = smem_addr(sQ + size_t(x) * kTileBytes);
#pragma unroll
                    for (int kk = 0; kk < kDh / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * kBox + (kk & 3) * 32;
                        tc::mma_ss(tmem + kColS + x * 128, tc::desc_sw128(q0 + off), tc::desc_sw128(k0 + off),
                                   idesc, kk > 0 ? 1u : 0u);
                    }
                    tc::commit(&s_full[x]);
                }
                tc::commit(&k_empty[ks]);
            }
        }
    } else if (warp == 3) {
        // ---------------- O_x += P_x V issuer ----------------
        if (lane == 0) {
            constexpr uint32_t idesc = tc::idesc_f16f32(kRowTile);
            bool ok = true;
            for (int j = 0; j < n && ok; ++j) {
                const int vs = j % kRingV;
                if (!(ok = tc::wait(&v_full[vs], (j / kRingV) & 1, err))) break;
                const uint32_t v0 = smem_addr(sV + size_t(vs) * kTileBytes);
                for (int x = 0; x < 2 && ok; ++x) {
                    if (j >= (x ? n_b : n_a)) continue;
                    if (!(ok = tc::wait(&p_full[x], j & 1, err))) break;
                    tc::fence_after();
#pragma unroll
                    for (int kk = 0; kk < kRowTile / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * kBox + (kk & 3) * 32;
                        tc::mma_ts(tmem + kColO + x * 128, tmem + kColS + x * 128 + kk * 8,
                                   tc::desc_sw128(v0 + off), idesc, (j > 0 || kk > 0) ? 1u : 0u);
                    }
                    tc::commit(&o_done[x]);
                }
                tc::commit(&v_empty[vs]);
            }
        }
    }
    } else {
        // ---------------- softmax warps: 4 per query tile, thread = query row ----------------
        // Running maximum m of s * c_log2 (c_log2 > 0); p = 2^(s c_log2 - m),
        // written as fp16 pairs over the first 64 columns of S_x (chunk c of
        // 32 keys into columns 16c .. 16c+15, which held scores already read).
        // O_x is rescaled only when m grows by more than kRescale2: it then
        // holds every product up to tile j - 1, since S_x of tile j was issued
        // after that product completed.
        const int x = (warp - 4) >> 2, quad = warp & 3;
        const int nX = x ? n_b : n_a;
        const int qrow = quad * 32 + lane;
        const int p = qs + x * kRowTile + qrow;                       // query position
        const uint32_t trow = tmem + (uint32_t(quad * 32) << 16);
        const uint32_t tS = trow + kColS + x * 128, tO = trow + kColO + x * 128;
        float m = -INFINITY, ls[4] = {0.0f, 0.0f, 0.0f, 0.0f};
        bool ok = true;
        for (int j = 0; j < nX; ++j) {
            if (!(ok = tc::wwait(&s_full[x], j & 1, err))) break;
            tc::fence_after();
            const int kmax = p - j * kRowTile;                        // keys 0 .. kmax of this tile are visible
            uint32_t v[4][32];                                        // the row's 128 scores, one load round trip
#pragma unroll
            for (int c = 0; c < 4; ++c) tc::tmem_ld32(tS + c * 32, v[c]);
            tc::tmem_wait_ld();
            if (kmax < 127) {
#pragma unroll
                for (int i = 0; i < 128; ++i)
                    if (i > kmax) v[i >> 5][i & 31] = __float_as_uint(-INFINITY);
            }
            float mx[4];
#pragma unroll
            for (int e = 0; e < 4; ++e) mx[e] = __uint_as_float(v[0][e]);
#pragma unroll
            for (int i = 4; i < 128; ++i) mx[i & 3] = fmaxf(mx[i & 3], __uint_as_float(v[i >> 5][i & 31]));
            const float mt = fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
            const float m_new = fmaxf(m, mt * c_log2);
            bool rescale = false;                                     // some row of the warp rescales O_x
            float alpha = 1.0f;
            if (j > 0) {
                const bool need = m_new > m + kRescale2;
                rescale = __any_sync(0xffffffffu, need);
                if (need) {
                    alpha = ex2_approx(m - m_new);
#pragma unroll
                    for (int e = 0; e < 4; ++e) ls[e] *= alpha;
                    m = m_new;
                }
            } else {
                m = m_new;
            }
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t pk[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    const float a = ex2_approx(fmaf(__uint_as_float(v[c][2 * i]), c_log2, -m));
                    const float b = ex2_approx(fmaf(__uint_as_float(v[c][2 * i + 1]), c_log2, -m));
                    ls[(2 * i) & 3] += a;
                    ls[(2 * i + 1) & 3] += b;
                    const __half2 hp = __floats2half2_rn(a, b);
                    pk[i] = *reinterpret_cast<const uint32_t *>(&hp);
                }
                tc::tmem_st16(tS + c * 16, pk);
            }
            if (rescale) {                                            // before O_x += P_x V of this tile
#pragma unroll 1
                for (int q = 0; q < 8; ++q) {
                    uint32_t o[16];
                    tc::tmem_ld16(tO + q * 16, o);
                    tc::tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 16; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
                    tc::tmem_st16(tO + q * 16, o);
                }
            }
            tc::tmem_wait_st();
            tc::fence_before();
            __syncwarp();
            if (lane == 0) tc::arrive(&p_full[x]);
        }
        if (nX > 0) {
            const float l = (ls[0] + ls[1]) + (ls[2] + ls[3]);
            if (ok) ok = tc::wwait(&o_done[x], (nX - 1) & 1, err);
            tc::fence_after();
            if (ok) {
                const float inv = 1.0f / l;
                const bool live = p < L;
                float *out = O + (size_t(bl.out_off[k]) + (p - bl.t0[k])) * d + x0;
#pragma unroll 1
                for (int q = 0; q < 4; ++q) {
                    uint32_t v[32];
                    tc::tmem_ld32(tO + q * 32, v);
                    tc::tmem_wait_ld();
                    if (live) {
#pragma unroll
                        for (int i = 0; i < 32; i += 4)
                            *reinterpret_cast<float4 *>(out + q * 32 + i) =
                                make_float4(__uint_as_float(v[i]) * inv, __uint_as_float(v[i + 1]) * inv,
                                            __uint_as_float(v[i + 2]) * inv, __uint_as_float(v[i + 3]) * inv);
                    }
                }
            }
        }
    }
    tc::fence_before();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after();
        tc::tmem_free(tmem, kFaTmemCols);
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
namespace {
size_t align256(size_t b) { return (b + 255) & ~size_t(255); }
}  // namespace

size_t prefill_mat_rows(const PrefillBlocks &bl) {
    size_t R = 0;
    for (int k = 0; k < bl.n; ++k) R += size_t((bl.L[k] + pf::kRowTile - 1) / pf::kRowTile) * pf::kRowTile;
    return R;
}

size_t prefill_mat_workspace_bytes(size_t R, int r, int d) {
    return align256(R * r * 2) + align256(R * 4) + 3 * align256(R * d * 2);
}

cudaError_t launch_prefill_weights(const uint16_t *Uq, const uint16_t *Uk, const uint16_t *Uv, int r, int d,
                                   uint16_t *Ut, int *err, cudaStream_t s) {
    ut_kernel<<<dim3(3 * d / 32, r / 32), dim3(32, 8), 0, s>>>(Uq, Uk, Uv, r, d, reinterpret_cast<__half *>(Ut), err);
    const cudaError_t e = cudaGetLastError();
    prof_mark(s, "ut");
    return e;
}

cudaError_t launch_prefill_mat(const CacheView &c, const PrefillBlocks &bl, const uint16_t *Ut, int H,
                               float softmax_scale, float *O, void *ws, int *err, cudaStream_t s) {
    using namespace pf;
    const int r = c.r, d = H * kDh;
    const int R = int(prefill_mat_rows(bl));
    char *p = static_cast<char *>(ws);
    __half *A = reinterpret_cast<__half *>(p);
    p += align256(size_t(R) * r * 2);
    float *rs = reinterpret_cast<float *>(p);
    p += align256(size_t(R) * 4);
    __half *Qm = reinterpret_cast<__half *>(p);
    p += align256(size_t(R) * d * 2);
    __half *Km = reinterpret_cast<__half *>(p);
    p += align256(size_t(R) * d * 2);
    __half *Vt = reinterpret_cast<__half *>(p);

    const int64_t prep_threads = int64_t(R) * (r / 8);
    cudaError_t e = launch_pdl(lat_prep_kernel, dim3(unsigned((prep_threads + 255) / 256)), dim3(256), 0, s, c, bl, R,
                               A, rs, err);
    if (e != cudaSuccess) return e;
    prof_mark(s, "lat_prep");

    CUtensorMap ma, mb;
    if (!encode_map_2d(&ma, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, A, uint64_t(r), uint64_t(R), uint64_t(r) * 2, 64,
                       kRowTile, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_map_2d(&mb, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, Ut, uint64_t(r), uint64_t(3 * d), uint64_t(r) * 2, 64,
                       kGemmN, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    if ((e = ensure_smem(qkv_gemm_kernel, kGemmSmem)) != cudaSuccess) return e;
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int gemm_tiles = (3 * d / kGemmN) * (R / kRowTile);
    e = launch_pdl(qkv_gemm_kernel, dim3(std::min(gemm_tiles, sms)), dim3(kGemmThreads), kGemmSmem, s, ma, mb, R, r, d,
                   static_cast<const float *>(rs), Qm, Km, Vt, err);
    if (e != cudaSuccess) return e;
    prof_mark(s, "qkv_gemm");

    CUtensorMap mq, mk, mv;
    if (!encode_map_2d(&mq, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, Qm, uint64_t(d), uint64_t(R), uint64_t(d) * 2, 64,
                       kRowTile, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_map_2d(&mk, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, Km, uint64_t(d), uint64_t(R), uint64_t(d) * 2, 64,
                       kRowTile, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_map_2d(&mv, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, Vt, uint64_t(R), uint64_t(d), uint64_t(R) * 2, 64,
                       kRowTile, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    if ((e = ensure_smem(fa_kernel, kFaSmem)) != cudaSuccess) return e;
    const float c_log2 = softmax_scale * 1.4426950408889634f;
    int pairs = 0;                                            // query-tile pairs over all blocks
    for (int k = 0; k < bl.n; ++k) pairs += (bl.qtile_off[k + 1] - bl.qtile_off[k] + 1) / 2;
    e = launch_pdl(fa_kernel, dim3(pairs, H), dim3(kFaThreads), kFaSmem, s, mq, mk, mv, bl, d, c_log2, O, err);
    prof_mark(s, "fa");
    return e;
}

}  // namespace qsvd
