// Exact int8 x int8 -> int32 down-projection on the 5th-generation tensor
// cores (a2 + the fp32 dequantization of a3), for prefill-sized T.
//
// sm_103a has no integer tcgen05 MMA, so the int8 codes are fed as bf16
// values (every integer in [-127, 127] is exact in bf16, every product
// |x w| <= 127^2 is exact in fp32) to tcgen05.mma.kind::f16 with an fp32
// accumulator in tensor memory.  A partial sum of up to 1024 such products
// stays below 2^24, so it is an exact integer in fp32 regardless of the
// order the tensor core adds in; the accumulator is therefore drained into
// int32 registers every kChunkK = 1024 of the reduction dimension, and the
// int32 sum over chunks is the exact integer product.
//
// CTA tile 128 (tokens) x BN (latent channels, 128 or 256), K staged 64 at
// a time.
//   warp 0      TMA producer: 2D tiles of X-codes [T, d] and W-codes [r, d]
//               (both K-major, 128-byte swizzle) into a ring of stages
//   warp 1      allocates tensor memory; lane 0 issues the MMAs (M=128,
//               N=BN, K=16) and commits stage releases / chunk completions
//   warps 2..   epilogue, BN/32 warps: warp w drains TMEM lane quadrant w%4,
//               columns 128*((w-2)/4) .. +127, of each chunk's accumulator
//               into int32 registers, then c_hat = (fp32(acc) s_x[t]) s_w[j]
// Two BN-column accumulators alternate between chunks so that the MMA of
// chunk c+1 overlaps the drain of chunk c.
//
// With LAT = 8 or 4 the per-token requantization of the latent (the rest of
// a3) and its store (a4) run in the same epilogue; c_hat never leaves the
// registers.  int4: a thread holds one token x one 128-channel group, so the
// group scale is local.  int8: the absmax of a token spans the r / BN CTAs of
// its row block, which form one cluster along N and swap their per-row maxima
// through distributed shared memory before quantizing.  A wide tile (BN=256) halves the
// number of MMA instructions per byte and cuts L2 traffic per MAC by a
// quarter; narrow tiles are kept for small T, where they give more CTAs.
#include <cuda.h>

#include "common.cuh"
#include "launch.h"
#include "tcgen05.cuh"

namespace qsvd {

constexpr int kBM = 128, kBK = 64;
constexpr int kRowB = 128;                     // bytes of K per staged tile row (one 128-byte swizzle atom)
constexpr int kChunkK = 1024;                  // <= 2^24 / 127^2 products per exact fp32 partial
constexpr int kStageA = kBM * kRowB;           // 16 KiB
constexpr int kRingBytes = 192 * 1024;         // TMA ring (stages of A + B tiles)

// OPB: operand bits.  16: the codes as bf16 (kind::f16, K = 16 per MMA, 64 per
// stage).  8: int4-valued codes as fp8 e4m3 (kind::f8f6f4, K = 32 per MMA,
// 128 per stage); every |x w| <= 49, so a partial sum stays an exact fp32
// integer for d < 2^24 / 49 and the accumulator is drained once at the end.
template <int BN, int OPB = 16> struct GemmCfg {
    static constexpr int kBKe = kRowB * 8 / OPB;      // K elements per stage
    static constexpr int kStageB = BN * kRowB;
    static constexpr int kStages = kRingBytes / (kStageA + kStageB);
    static constexpr int kEpiWarps = BN / 32;
    static constexpr int kThreads = 64 + 32 * kEpiWarps;
    static constexpr size_t kSmem = size_t(kStages) * (kStageA + kStageB) + 1024;   // + alignment slack
    // f32 accumulator, A and B K-major, M=128, N=BN; bf16 x bf16 (kind::f16) or e4m3 x e4m3 (kind::f8f6f4)
    static constexpr uint32_t kIdesc = (1u << 4) | (OPB == 16 ? (1u << 7) | (1u << 10) : 0u) |
                                       (uint32_t(BN >> 3) << 17) | (uint32_t(kBM >> 4) << 24);
};

// PTX wrappers: tcgen05.cuh (tc::); a spin on an mbarrier phase, bounded.
__device__ __forceinline__ bool spin_wait(uint64_t *bar, uint32_t parity, int *err) { return tc::wait(bar, parity, err); }

// ---------------------------------------------------------------------------
// Destinations of the fused requantization (LAT != 0).
struct LatOut {
    float clip;
    void *codes, *scales;              // token-major, or null
    CacheView dst;                     // dst.codes null: no cache store
    const int32_t *seq, *pos;
};

__device__ __forceinline__ uint32_t g_cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

template <int BN, int LAT, int OPB>
__global__ void __launch_bounds__(GemmCfg<BN, OPB>::kThreads, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap map_x, const __grid_constant__ CUtensorMap map_w, int64_t T, int d,
               int r, const float *xs, const float *__restrict__ ws, float *__restrict__ c_hat,
               int32_t *__restrict__ acc_out, const LatOut lo, int *err, int k_per, int32_t *__restrict__ part) {
    using C = GemmCfg<BN, OPB>;
    constexpr int kStages = C::kStages, kStageB = C::kStageB, kBKe = C::kBKe;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t *sA = smem;                                    // [kStages][128 x 128 B] SW128
    uint8_t *sB = smem + size_t(kStages) * kStageA;        // [kStages][BN x 128 B] SW128
    __shared__ __align__(8) uint64_t full_bar[kStages], empty_bar[kStages];
    __shared__ __align__(8) uint64_t acc_full[2], acc_empty[2];
    __shared__ uint32_t tmem_base;
    __shared__ float red_m[BN / 128][kBM];                 // per-row max of each 128-column half
    __shared__ float xmax[8][kBM];                         // per-row max of every CTA of the cluster (int8)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.y * kBM, n0 = blockIdx.x * BN;      // N fastest: a wave shares X tiles
    // K stages [kb, kb + n_k) of this CTA: all of them, or split blockIdx.z of
    // a split-K launch (part != null), whose int32 partial sums go to
    // part[blockIdx.z] and are added and requantized by split_requant_kernel
    const int kb = int(blockIdx.z) * k_per;
    const int n_k = min(d / kBKe - kb, k_per);
    const int stages_per_chunk = OPB == 16 ? kChunkK / kBKe : n_k;
    const int n_chunks = (n_k + stages_per_chunk - 1) / stages_per_chunk;

    pdl_trigger();
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&full_bar[s], 1);
            mbar_init(&empty_bar[s], 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(&acc_full[s], 1);
            mbar_init(&acc_empty[s], C::kEpiWarps);   // one arrival per epilogue warp
        }
        mbar_init_fence();
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_x)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&map_w)) : "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     ::"r"(smem_addr(&tmem_base)), "r"(2 * BN));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    const uint32_t tmem = tmem_base;
    pdl_wait();

    int32_t acc[128];                                     // epilogue: the tile row's int32 sums, then c_hat bits
    bool epi_ok = false;
    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            for (int i = 0; i < n_k; ++i) {
                const int s = i % kStages;
                if (i >= kStages && !spin_wait(&empty_bar[s], ((i / kStages) - 1) & 1, err)) break;
                mbar_arrive_expect_tx(&full_bar[s], kStageA + kStageB);
                tc::tma_load_2d(sA + size_t(s) * kStageA, &map_x, (kb + i) * kBKe, m0, &full_bar[s]);
                tc::tma_load_2d(sB + size_t(s) * kStageB, &map_w, (kb + i) * kBKe, n0, &full_bar[s]);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            bool ok = true;
            for (int c = 0; c < n_chunks && ok; ++c) {
                const int buf = c & 1;
                if (c >= 2) {
                    ok = spin_wait(&acc_empty[buf], ((c >> 1) - 1) & 1, err);
                    tc::fence_after();
                }
                const uint32_t d_tmem = tmem + uint32_t(buf * BN);
                const int i0 = c * stages_per_chunk, i1 = min(n_k, i0 + stages_per_chunk);
                for (int i = i0; i < i1 && ok; ++i) {
                    const int s = i % kStages;
                    ok = spin_wait(&full_bar[s], (i / kStages) & 1, err);
                    if (!ok) break;
                    tc::fence_after();
                    const uint32_t a0 = smem_addr(sA + size_t(s) * kStageA);
                    const uint32_t b0 = smem_addr(sB + size_t(s) * kStageB);
#pragma unroll
                    for (int ks = 0; ks < kRowB / 32; ++ks) {     // 32 bytes of K per MMA
                        if (OPB == 16)
                            tc::mma_ss(d_tmem, tc::desc_sw128(a0 + ks * 32), tc::desc_sw128(b0 + ks * 32), C::kIdesc,
                                      (i > i0 || ks > 0) ? 1u : 0u);
                        else
                            tc::mma_ss_f8(d_tmem, tc::desc_sw128(a0 + ks * 32), tc::desc_sw128(b0 + ks * 32), C::kIdesc,
                                    (i > i0 || ks > 0) ? 1u : 0u);
                    }
                    tc::commit(&empty_bar[s]);          // stage s may be refilled once these MMAs finish
                }
                if (ok) tc::commit(&acc_full[buf]);     // chunk c's partial sum is complete
            }
        }
    } else {
        // ---------------- epilogue (warps 2 .. 2 + kEpiWarps - 1) ----------------
        const int quad = warp & 3;                        // TMEM lane quadrant of this warp
        const int col0 = ((warp - 2) >> 2) * 128;         // this warp's 128 columns of the tile
        const int row = quad * 32 + lane;                 // row of the tile (token)
#pragma unroll
        for (int j = 0; j < 128; ++j) acc[j] = 0;
        bool ok = true;
        for (int c = 0; c < n_chunks && ok; ++c) {
            const int buf = c & 1;
            ok = spin_wait(&acc_full[buf], (c >> 1) & 1, err);
            tc::fence_after();
            if (!ok) break;
            const uint32_t taddr = tmem + (uint32_t(quad * 32) << 16) + uint32_t(buf * BN + col0);
#pragma unroll
            for (int j0 = 0; j0 < 128; j0 += 32) {
                uint32_t v[32];
                tc::tmem_ld32(taddr + j0, v);
                tc::tmem_wait_ld();
#pragma unroll
                for (int j = 0; j < 32; ++j) acc[j0 + j] += __float2int_rn(__uint_as_float(v[j]));
            }
            tc::fence_before();
            __syncwarp();
            if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(&acc_empty[buf])) : "memory");
        }
        epi_ok = ok;
        const int64_t t = m0 + row;
        const bool live = ok && t < T;
        const int nc = n0 + col0;
        if (LAT == 0 && part) {                           // split-K: this split's partial sums
            if (live) {
                int32_t *po = part + (size_t(blockIdx.z) * size_t(T) + size_t(t)) * r + nc;
#pragma unroll
                for (int j = 0; j < 128; j += 4)
                    *reinterpret_cast<int4 *>(po + j) = make_int4(acc[j], acc[j + 1], acc[j + 2], acc[j + 3]);
            }
        } else {
            if (live && acc_out) {
                int32_t *ao = acc_out + t * r + nc;
#pragma unroll
                for (int j = 0; j < 128; j += 4)
                    *reinterpret_cast<int4 *>(ao + j) = make_int4(acc[j], acc[j + 1], acc[j + 2], acc[j + 3]);
            }
            // c_hat = (fp32(acc) s_x[t]) s_w[j], kept in the same registers (as float bits)
            const float sx = live ? xs[t] : 0.0f;
            float m = 0.0f;
#pragma unroll
            for (int j = 0; j < 128; ++j) {
                const float v = __fmul_rn(__fmul_rn(__int2float_rn(acc[j]), sx), live ? ws[nc + j] : 0.0f);
                acc[j] = __float_as_int(v);
                m = fmaxf(m, fabsf(v));
            }
            if (live && c_hat) {
                float *out = c_hat + t * r + nc;
#pragma unroll
                for (int j = 0; j < 128; j += 4)
                    *reinterpret_cast<float4 *>(out + j) = make_float4(__int_as_float(acc[j]), __int_as_float(acc[j + 1]),
                                                                       __int_as_float(acc[j + 2]), __int_as_float(acc[j + 3]));
            }
            if (LAT == 8) {
                red_m[col0 / 128][row] = m;
                asm volatile("bar.sync 1, %0;" ::"r"(C::kEpiWarps * 32) : "memory");
                if (col0 == 0) {
                    float mc = red_m[0][row];
#pragma unroll
                    for (int k = 1; k < BN / 128; ++k) mc = fmaxf(mc, red_m[k][row]);
                    // this CTA's row maximum into slot [rank][row] of every CTA of the cluster
                    const uint32_t cs = gridDim.x, rank = g_cluster_rank();
                    const uint32_t local = smem_addr(&xmax[rank][row]);
                    for (uint32_t p = 0; p < cs; ++p) {
                        uint32_t remote;
                        asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(local), "r"(p));
                        asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(remote), "f"(mc) : "memory");
                    }
                }
            }
        }
    }
    if (LAT == 8) {
        // every thread of every CTA of the cluster (the maxima are exchanged)
        asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
    }
    if (LAT != 0 && warp >= 2) {
        const int quad = warp & 3, col0 = ((warp - 2) >> 2) * 128, row = quad * 32 + lane;
        const int64_t t = m0 + row;
        const int nc = n0 + col0;
        const bool live = epi_ok && t < T;
        if (live) {
            // destinations of row t (cache slot bounds-checked)
            uint8_t *cache_codes = nullptr;
            void *cache_scale = nullptr;
            if (lo.dst.codes) {
                const int b = lo.seq[t], p = lo.pos[t];
                if (b < 0 || b >= lo.dst.B || p < 0 || p >= lo.dst.Tmax) {
                    if (col0 == 0 && blockIdx.x == 0) flag_error(err, kErrRange);
                } else {
                    const size_t slot = size_t(b) * lo.dst.Tmax + p;
                    cache_codes = static_cast<uint8_t *>(lo.dst.codes) + slot * (LAT == 8 ? r : r / 2);
                    cache_scale = LAT == 8 ? static_cast<void *>(static_cast<float *>(lo.dst.scales) + slot)
                                           : static_cast<void *>(static_cast<__half *>(lo.dst.scales) + slot * (r / 128));
                }
            }
            uint8_t *tok_codes = lo.codes ? static_cast<uint8_t *>(lo.codes) + t * (LAT == 8 ? r : r / 2) : nullptr;
            if (LAT == 8) {
                float mt = 0.0f;
                for (uint32_t p = 0; p < gridDim.x; ++p) mt = fmaxf(mt, xmax[p][row]);
                const float s = quant_scale(mt, lo.clip, 127.0f);
                const float is = quant_inv_scale(s);
#pragma unroll
                for (int j = 0; j < 128; j += 16) {
                    uint32_t w[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        w[q] = uint32_t(quant_code_fast(__int_as_float(acc[j + 4 * q + 0]), s, is, 127) & 0xff) |
                               (uint32_t(quant_code_fast(__int_as_float(acc[j + 4 * q + 1]), s, is, 127) & 0xff) << 8) |
                               (uint32_t(quant_code_fast(__int_as_float(acc[j + 4 * q + 2]), s, is, 127) & 0xff) << 16) |
                               (uint32_t(quant_code_fast(__int_as_float(acc[j + 4 * q + 3]), s, is, 127) & 0xff) << 24);
                    const uint4 v4 = make_uint4(w[0], w[1], w[2], w[3]);
                    if (tok_codes) *reinterpret_cast<uint4 *>(tok_codes + nc + j) = v4;
                    if (cache_codes) *reinterpret_cast<uint4 *>(cache_codes + nc + j) = v4;
                }
                if (nc == 0) {                            // the CTA holding channels 0..127 writes the scale
                    if (lo.scales) static_cast<float *>(lo.scales)[t] = s;
                    if (cache_scale) *static_cast<float *>(cache_scale) = s;
                }
            } else {
                float mg = 0.0f;                          // the thread's 128 channels are one group
#pragma unroll
                for (int j = 0; j < 128; ++j) mg = fmaxf(mg, fabsf(__int_as_float(acc[j])));
                const __half hs = int4_group_scale(mg, lo.clip);
                const float s = __half2float(hs);
                const float is = quant_inv_scale(s);
#pragma unroll
                for (int j = 0; j < 128; j += 32) {
                    uint32_t w[4];
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint32_t x = 0;
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            x |= uint32_t(quant_code_fast(__int_as_float(acc[j + 8 * q + e]), s, is, 7) & 0xf) << (4 * e);
                        w[q] = x;
                    }
                    const uint4 v4 = make_uint4(w[0], w[1], w[2], w[3]);
                    if (tok_codes) *reinterpret_cast<uint4 *>(tok_codes + (nc + j) / 2) = v4;
                    if (cache_codes) *reinterpret_cast<uint4 *>(cache_codes + (nc + j) / 2) = v4;
                }
                const int g = nc / 128;
                if (lo.scales) static_cast<__half *>(lo.scales)[t * (r / 128) + g] = hs;
                if (cache_scale) static_cast<__half *>(cache_scale)[g] = hs;
            }
        }
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (warp == 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(2 * BN));
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
// Operand matrix [rows, cols] row-major (cols contiguous): bf16 (OPB 16) or
// one byte per element (OPB 8), box [box_rows x 128 bytes], 128B swizzle.
static bool make_map(CUtensorMap *map, const void *base, int64_t rows, int cols, int box_rows, int opb = 16) {
    return encode_map_2d(map, opb == 16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_UINT8, base,
                         uint64_t(cols), uint64_t(rows), uint64_t(cols) * opb / 8, uint32_t(kRowB * 8 / opb),
                         uint32_t(box_rows), CU_TENSOR_MAP_SWIZZLE_128B);
}

bool gemm_tc_supported(int d, int r) { return d % kBK == 0 && r % 128 == 0 && tensor_maps_available(); }

// Tile width and whether the per-token requantization can run in the epilogue:
// int4 always; int8 when the r / BN CTAs of a row block fit one portable
// cluster (<= 8).
static int pick_bn(int64_t T, int r, int lat_bits, bool *fuse) {
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t wide_tiles = ((T + kBM - 1) / kBM) * (r / 256);
    int bn = (r % 256 == 0 && wide_tiles >= 2 * sms) ? 256 : 128;
    if (lat_bits == 8 && r / bn > 8 && r % 256 == 0) bn = 256;
    *fuse = lat_bits == 4 || (lat_bits == 8 && r / bn <= 8);
    return bn;
}

template <int BN, int LAT, int OPB = 16>
static cudaError_t launch_bn(const void *xq_op, int64_t T, int d, const void *w_op, const float *ws,
                             const float *xs, int r, float *c_hat, int32_t *acc_out, const LatOut &lo, int *err,
                             cudaStream_t s, int splits = 1, int32_t *part = nullptr) {
    using C = GemmCfg<BN, OPB>;
    const int n_k = d / C::kBKe, k_per = (n_k + splits - 1) / splits;
    splits = (n_k + k_per - 1) / k_per;                 // no empty split
    CUtensorMap mx, mw;
    if (!make_map(&mx, xq_op, T, d, kBM, OPB) || !make_map(&mw, w_op, r, d, BN, OPB)) return cudaErrorInvalidValue;
    cudaError_t e = ensure_smem(gemm_tc_kernel<BN, LAT, OPB>, C::kSmem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(unsigned(r / BN), unsigned((T + kBM - 1) / kBM), unsigned(splits));
    cfg.blockDim = dim3(C::kThreads);
    cfg.dynamicSmemBytes = C::kSmem;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;        // int8 epilogue: one cluster per row block
    attr[1].val.clusterDim.x = LAT == 8 ? unsigned(r / BN) : 1u;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = LAT == 8 ? 2 : 1;
    e = cudaLaunchKernelEx(&cfg, gemm_tc_kernel<BN, LAT, OPB>, mx, mw, T, d, r, xs, ws, c_hat, acc_out, lo, err,
                           k_per, part);
    prof_mark(s, OPB == 16 ? "gemm_tc" : "gemm_f8");
    return e;
}

cudaError_t launch_gemm_tc(const uint16_t *xq_bf16, int64_t T, int d, const uint16_t *w_bf16, const float *ws,
                           const float *xs, int r, float *c_hat, int32_t *acc_out, int *err, cudaStream_t s,
                           int splits, int32_t *part) {
    if (T == 0) return cudaSuccess;
    bool fuse = false;
    const int bn = pick_bn(T, r, 0, &fuse);
    const LatOut lo{};
    if (splits < 2) part = nullptr;
    return bn == 256 ? launch_bn<256, 0>(xq_bf16, T, d, w_bf16, ws, xs, r, c_hat, acc_out, lo, err, s, splits, part)
                     : launch_bn<128, 0>(xq_bf16, T, d, w_bf16, ws, xs, r, c_hat, acc_out, lo, err, s, splits, part);
}

// K splits of the separate-epilogue GEMM: while its tiles fill less than half
// the GPU, split K so that about one wave of CTAs runs, each split at least 8
// stages (512 of K) long; at most kMaxSplitK.
int gemm_tc_splits(int64_t T, int d, int r) {
    if (T * r > kSplitMaxElems) return 1;
    bool fuse = false;
    const int bn = pick_bn(T, r, 0, &fuse);
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t tiles = ((T + kBM - 1) / kBM) * (r / bn);
    if (2 * tiles > sms) return 1;
    const int n_k = d / kBK;
    int64_t sp = std::min<int64_t>(int64_t(kMaxSplitK), int64_t(sms) / tiles);
    sp = std::max<int64_t>(1, std::min<int64_t>(sp, int64_t(n_k / 8)));
    const int64_t k_per = (n_k + sp - 1) / sp;
    return int((n_k + k_per - 1) / k_per);                 // the count launch_bn runs
}

namespace {
int g_epilogue_mode = 0;     // 0 automatic, 1 separate requantization kernel, 2 fused where possible
}
void set_project_epilogue(int mode) { g_epilogue_mode = mode; }
int project_epilogue() { return g_epilogue_mode; }

bool gemm_tc_fused_supported(int64_t T, int r, int lat_bits) {
    bool fuse = false;
    const int bn = pick_bn(T, r, lat_bits, &fuse);
    if (!fuse || g_epilogue_mode == 1) return false;
    if (g_epilogue_mode == 2) return true;
    if (lat_bits == 4) return true;
    // automatic, int8: clusters wider than 6 CTAs leave SMs of each GPC idle;
    // and below one wave of 256-column tiles the separate requantization with
    // 128-column tiles (twice the CTAs) is faster: measured on GB300 (cold L2),
    // 640 tokens x 4096 x 1536 49.8 us against 64.2 us for the call, 1280
    // tokens 56.0 against 68.3 us
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return r / bn <= 6 && ((T + kBM - 1) / kBM) * (r / bn) >= sms;
}

cudaError_t launch_gemm_tc_fused(const uint16_t *xq_bf16, int64_t T, int d, const uint16_t *w_bf16, const float *ws,
                                 const float *xs, int r, int lat_bits, float lat_clip, void *lat_codes,
                                 void *lat_scales, const CacheView *dst, const int32_t *dst_seq,
                                 const int32_t *dst_pos, float *c_hat, int32_t *acc_out, int *err, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    bool fuse = false;
    const int bn = pick_bn(T, r, lat_bits, &fuse);
    if (!fuse) return cudaErrorInvalidValue;
    LatOut lo{lat_clip, lat_codes, lat_scales, dst ? *dst : CacheView{}, dst_seq, dst_pos};
    if (lat_bits == 8)
        return bn == 256 ? launch_bn<256, 8>(xq_bf16, T, d, w_bf16, ws, xs, r, c_hat, acc_out, lo, err, s)
                         : launch_bn<128, 8>(xq_bf16, T, d, w_bf16, ws, xs, r, c_hat, acc_out, lo, err, s);
    return bn == 256 ? launch_bn<256, 4>(xq_bf16, T, d, w_bf16, ws, xs, r, c_hat, acc_out, lo, err, s)
                     : launch_bn<128, 4>(xq_bf16, T, d, w_bf16, ws, xs, r, c_hat, acc_out, lo, err, s);
}

// W4A4: the same GEMM on fp8 e4m3 images of int4-valued codes (every value in
// [-7, 7] is exact in e4m3), kind::f8f6f4; lat_bits 0 leaves the
// requantization to a separate kernel (c_hat written).
bool gemm_f8_supported(int d, int r) { return d % kRowB == 0 && r % 128 == 0 && d < (1 << 24) / 49 && tensor_maps_available(); }

cudaError_t launch_gemm_f8(const uint8_t *xq_f8, int64_t T, int d, const uint8_t *w_f8, const float *ws,
                           const float *xs, int r, int lat_bits, float lat_clip, void *lat_codes, void *lat_scales,
                           const CacheView *dst, const int32_t *dst_seq, const int32_t *dst_pos, float *c_hat,
                           int32_t *acc_out, int *err, cudaStream_t s) {
    if (T == 0) return cudaSuccess;
    bool fuse = false;
    const int bn = pick_bn(T, r, lat_bits, &fuse);
    LatOut lo{lat_clip, lat_codes, lat_scales, dst ? *dst : CacheView{}, dst_seq, dst_pos};
    if (lat_bits == 8 && fuse)
        return bn == 256 ? launch_bn<256, 8, 8>(xq_f8, T, d, w_f8, ws, xs, r, c_hat, acc_out, lo, err, s)
                         : launch_bn<128, 8, 8>(xq_f8, T, d, w_f8, ws, xs, r, c_hat, acc_out, lo, err, s);
    if (lat_bits == 4)
        return bn == 256 ? launch_bn<256, 4, 8>(xq_f8, T, d, w_f8, ws, xs, r, c_hat, acc_out, lo, err, s)
                         : launch_bn<128, 4, 8>(xq_f8, T, d, w_f8, ws, xs, r, c_hat, acc_out, lo, err, s);
    const LatOut none{};
    return bn == 256 ? launch_bn<256, 0, 8>(xq_f8, T, d, w_f8, ws, xs, r, c_hat, acc_out, none, err, s)
                     : launch_bn<128, 0, 8>(xq_f8, T, d, w_f8, ws, xs, r, c_hat, acc_out, none, err, s);
}

}  // namespace qsvd
