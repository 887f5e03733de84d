// Device helpers shared by the QSVD kernels: bf16 unpacking, the symmetric
// RTN quantizer, warp/block reductions and the device error word.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>

#include "launch.h"

namespace qsvd {

// Programmatic dependent launch: let the next kernel in the stream start its
// prologue now / wait until every earlier kernel in the stream has finished
// and its writes are visible.  Both are no-ops without the launch attribute.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
// Data written by the grid this one waits on is never read through a
// `const T *__restrict__` pointer (the read-only path): a dependent grid runs
// while its producer still writes, so such loads may be scheduled ahead of
// this wait and see stale values (measured: a row requantizer reading the
// GEMM's partial sums that way returned wrong codes on every run).
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Bulk prefetch of [p, p + bytes) into L2 (16-byte aligned, bytes % 16 == 0).
// A hint only: data written later by an earlier kernel is still read
// correctly, because later loads go through the coherent L2.
__device__ __forceinline__ void prefetch_l2_bulk(const void *p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// CTA `i` of `n` prefetches its 1/n share of a buffer into L2 (thread 0 only,
// in pieces of at most 64 KiB).
__device__ __forceinline__ void prefetch_share_l2(const void *base, size_t bytes, size_t i, size_t n) {
    if (threadIdx.x != 0 || bytes == 0) return;
    size_t per = ((bytes + n - 1) / n + 15) & ~size_t(15);
    size_t lo = i * per;
    if (lo >= bytes) return;
    size_t hi = lo + per < bytes ? lo + per : bytes;
    hi &= ~size_t(15);
    const char *c = static_cast<const char *>(base);
    for (size_t o = lo; o < hi; o += 65536) {
        const size_t len = hi - o < 65536 ? hi - o : 65536;
        prefetch_l2_bulk(c + o, uint32_t(len));
    }
}

// The fp32 at the same shared-memory offset in CTAs 0 .. 7 of the cluster,
// as one instruction block so that the eight remote loads are in flight
// together (the caller adds them in rank order).
__device__ __forceinline__ void cluster_ld8(const void *p, float (&v)[8]) {
    const uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(p));
    asm volatile("{\n\t.reg .b32 a<8>;\n\t"
                 "mapa.shared::cluster.u32 a0, %8, 0;\n\tmapa.shared::cluster.u32 a1, %8, 1;\n\t"
                 "mapa.shared::cluster.u32 a2, %8, 2;\n\tmapa.shared::cluster.u32 a3, %8, 3;\n\t"
                 "mapa.shared::cluster.u32 a4, %8, 4;\n\tmapa.shared::cluster.u32 a5, %8, 5;\n\t"
                 "mapa.shared::cluster.u32 a6, %8, 6;\n\tmapa.shared::cluster.u32 a7, %8, 7;\n\t"
                 "ld.shared::cluster.f32 %0, [a0];\n\tld.shared::cluster.f32 %1, [a1];\n\t"
                 "ld.shared::cluster.f32 %2, [a2];\n\tld.shared::cluster.f32 %3, [a3];\n\t"
                 "ld.shared::cluster.f32 %4, [a4];\n\tld.shared::cluster.f32 %5, [a5];\n\t"
                 "ld.shared::cluster.f32 %6, [a6];\n\tld.shared::cluster.f32 %7, [a7];\n\t}"
                 : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3]), "=f"(v[4]), "=f"(v[5]), "=f"(v[6]), "=f"(v[7])
                 : "r"(a)
                 : "memory");
}
// Split cluster barrier: arrive (release this CTA's earlier accesses) now,
// wait (acquire) later, so work in between overlaps the peers' arrival.
__device__ __forceinline__ void cluster_arrive() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory"); }

__device__ __forceinline__ void flag_error(int *err, int bit) {
    if (err) atomicOr(err, bit);
}

// ---------------------------------------------------------------------------
// mbarrier + bulk (TMA, non-tensor) copies global -> shared
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_init_fence() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
// One arrival that also announces `bytes` of transactions for this phase.
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}
// Bulk copy of `bytes` (multiple of 16; both addresses 16-byte aligned).
__device__ __forceinline__ void bulk_g2s(void *dst, const void *src, uint32_t bytes, uint64_t *bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(smem_addr(dst)), "l"(src), "r"(bytes), "r"(smem_addr(bar))
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile("{\n.reg .pred p;\nmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
                 "selp.u32 %0, 1, 0, p;\n}\n"
                 : "=r"(ok)
                 : "r"(smem_addr(bar)), "r"(parity)
                 : "memory");
    return ok != 0;
}
// Bounded wait for phase `parity`.  On expiry the error word gets
// kErrTimeout, then the wait continues (bounded again) so that copies still in
// flight land before the CTA may exit; returns whether the phase completed.
constexpr long kWaitLimit = 1L << 24;
static __device__ __noinline__ bool mbar_wait(uint64_t *bar, uint32_t parity, int *err) {
    for (long i = 0; i < kWaitLimit; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    flag_error(err, kErrTimeout);
    for (long i = 0; i < kWaitLimit; ++i)
        if (mbar_try_wait(bar, parity)) return false;
    return false;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }
__device__ __forceinline__ float bf16_to_f32(uint16_t b) { return __uint_as_float(uint32_t(b) << 16); }

// Unpack 8 bf16 values held in a 16-byte vector.
__device__ __forceinline__ void unpack8_bf16(const uint4 &v, float (&f)[8]) {
    f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
    f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
    f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z);
    f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}

// bf16 bit pattern of a small integer (|c| <= 255 is exact in bf16).
__device__ __forceinline__ uint16_t int_to_bf16_bits(int c) {
    return uint16_t(__float_as_uint(float(c)) >> 16);
}
// Four int8 codes -> two fp16 pairs, exact: the half with bits 0x64xx is
// 1024 + xx, so (code + 128) placed in the low byte gives 1152 + code.
__device__ __forceinline__ void i8x4_to_h2x2(uint32_t w, uint32_t &lo, uint32_t &hi) {
    const uint32_t u = w ^ 0x80808080u;
    const uint32_t a = __byte_perm(u, 0x64646464u, 0x5150);
    const uint32_t b = __byte_perm(u, 0x64646464u, 0x5352);
    const __half2 bias = __half2half2(__ushort_as_half(0x6480));      // 1152
    const __half2 ha = __hsub2(*reinterpret_cast<const __half2 *>(&a), bias);
    const __half2 hb = __hsub2(*reinterpret_cast<const __half2 *>(&b), bias);
    lo = *reinterpret_cast<const uint32_t *>(&ha);
    hi = *reinterpret_cast<const uint32_t *>(&hb);
}
// Eight int4 codes (element i in bits 4i..4i+3, two's complement) times an
// fp16 group scale -> four fp16 pairs (products rounded to nearest).
__device__ __forceinline__ void i4x8_to_h2x4(uint32_t w, __half2 s2, uint32_t *o) {
    const __half2 bias = __half2half2(__ushort_as_half(0x6408));      // 1032 = 1024 + 8
    const uint32_t x = w ^ 0x88888888u;                               // code + 8 in every nibble
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t n0 = (x >> (8 * k)) & 0xfu, n1 = (x >> (8 * k + 4)) & 0xfu;
        const uint32_t p = (0x6400u | n0) | ((0x6400u | n1) << 16);
        const __half2 h = __hmul2(__hsub2(*reinterpret_cast<const __half2 *>(&p), bias), s2);
        o[k] = *reinterpret_cast<const uint32_t *>(&h);
    }
}

// fp8 e4m3 byte of a small integer (|c| <= 16 is exact in e4m3: 3 mantissa bits).
__device__ __forceinline__ uint8_t int_to_e4m3(int c) {
    return uint8_t(__nv_cvt_float_to_fp8(float(c), __NV_SATFINITE, __NV_E4M3));
}

// ---------------------------------------------------------------------------
// Symmetric round-to-nearest quantizer (per token / per channel / per group):
//   s    = fp32(fp32(clip * m) / qmax)
//   code = clamp(rne(fp32(v / s)), -qmax, qmax),  0 when s == 0.
// IEEE round-to-nearest intrinsics keep every step bit-exact (no FMA).
// ---------------------------------------------------------------------------
__device__ __forceinline__ float quant_scale(float absmax, float clip, float qmax) {
    return __fdiv_rn(__fmul_rn(clip, absmax), qmax);
}

__device__ __forceinline__ int quant_code(float v, float s, int qmax) {
    if (s == 0.0f) return 0;
    int c = __float2int_rn(__fdiv_rn(v, s));     // float->int conversion saturates
    return c < -qmax ? -qmax : (c > qmax ? qmax : c);
}

// The same code from a precomputed inv_s = __frcp_rn(s).  x = fp32(v * inv_s)
// is within 2^-16 + 2^-17 < 2^-15 of fp32(v / s) for |v / s| <= 127.5, so the
// two round to the same integer unless fp32(v / s) lies within 2^-15 of a
// half-integer; inside a margin of 2^-14 around half-integers the correctly
// rounded quotient is computed instead (also whenever inv_s == 0, which the
// caller passes for scales too small for a finite reciprocal).  Results equal
// quant_code's: above |v / s| = 127.5 both clamp.
__device__ __forceinline__ float quant_inv_scale(float s) { return s > 1e-30f ? __frcp_rn(s) : 0.0f; }
__device__ __forceinline__ int quant_code_fast(float v, float s, float inv_s, int qmax) {
    if (s == 0.0f) return 0;
    float x = v * inv_s;
    const float f = x - floorf(x);
    if (inv_s == 0.0f || fabsf(f - 0.5f) < 6.103515625e-05f) x = __fdiv_rn(v, s);   // margin 2^-14
    int c = __float2int_rn(x);
    return c < -qmax ? -qmax : (c > qmax ? qmax : c);
}

// int4 group scale: fp32 scale rounded to fp16 (nearest even), saturated.
__device__ __forceinline__ __half int4_group_scale(float absmax, float clip) {
    return __float2half_rn(fminf(quant_scale(absmax, clip, 7.0f), 65504.0f));
}

// ---------------------------------------------------------------------------
// Reductions
// ---------------------------------------------------------------------------
// Block Hadamard transform of a row (the rotation H1; the stage order is the
// one fwht_smem in quant_kernels.cu follows, so results are identical).
// fwht8_regs: stages h = 1, 2, 4 on 8 consecutive, 8-aligned values.
__device__ __forceinline__ void fwht8_regs(float (&f)[8]) {
#pragma unroll
    for (int hh = 1; hh < 8; hh <<= 1)
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            if (e & hh) continue;
            const float a = f[e], c = f[e + hh];
            f[e] = __fadd_rn(a, c);
            f[e + hh] = __fsub_rn(a, c);
        }
}
// fwht_smem_rounds: the remaining stages, in rounds of up to four.  In a
// round starting at stride h0, a thread takes groups of 2^k elements spaced
// h0 apart (the group's base has zeros in the bits the round's strides
// cover), so the round's stages pair elements within a group only and run in
// registers; one barrier per round.  Every butterfly combines the same two
// values in the same stage order as fwht_smem, so the results are identical.
// `first` stages (h < first) have already been applied by the caller.
__device__ __forceinline__ void fwht_smem_rounds(float *v, int n, int b, int first) {
    for (int h0 = first; h0 < b; h0 <<= 4) {
        int ks = 0;
        while (ks < 4 && (h0 << ks) < b) ++ks;            // stages h0, 2 h0, ..., 2^(ks-1) h0
        const int gsz = 1 << ks, ngroups = n >> ks;
        for (int g = threadIdx.x; g < ngroups; g += blockDim.x) {
            const int base = (g / h0) * (gsz * h0) + (g % h0);
            float x[16];
#pragma unroll
            for (int e = 0; e < 16; ++e)
                if (e < gsz) x[e] = v[base + e * h0];
#pragma unroll
            for (int st = 0; st < 4; ++st) {
                if (st >= ks) break;
                const int hh = 1 << st;
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    if (e >= gsz || (e & hh)) continue;
                    const float a = x[e], c = x[e + hh];
                    x[e] = __fadd_rn(a, c);
                    x[e + hh] = __fsub_rn(a, c);
                }
            }
#pragma unroll
            for (int e = 0; e < 16; ++e)
                if (e < gsz) v[base + e * h0] = x[e];
        }
        __syncthreads();
    }
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ int warp_sum_int(int v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Block-wide max; `red` holds one float per warp.  All threads get the result.
template <int NT>
__device__ __forceinline__ float block_max(float v, float *red) {
    v = warp_max(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    __syncthreads();
    if (l == 0) red[w] = v;
    __syncthreads();
    float m = red[0];
#pragma unroll
    for (int i = 1; i < NT / 32; ++i) m = fmaxf(m, red[i]);
    return m;
}


// ---------------------------------------------------------------------------
// Per-token requantization of latent row t of c_hat [T, r] by one CTA of
// kRqThreads threads (Eq. 11's Q(C_qkv)): int8 with one fp32 scale per token,
// or int4 with one fp16 scale per 128-channel group (one warp row of float4).
// Writes token-major outputs and/or the cache slot (seq, pos) of row t;
// out-of-range slots are skipped and flagged.  `red` holds kRqThreads/32 floats.
// ---------------------------------------------------------------------------
constexpr int kRqThreads = 256;
constexpr int kRqMaxQuads = 4;     // r <= 4096

// The requantization of row t from its values already in registers: thread
// i holds channels 4 (i + k kRqThreads) .. + 3 in v[k] (zeros past r).
__device__ __forceinline__ void requant_row_values(const float4 (&v)[kRqMaxQuads], int64_t t, int r, int bits,
                                                   float clip, void *__restrict__ lat_codes,
                                                   void *__restrict__ lat_scales, const CacheView &dst,
                                                   const int32_t *__restrict__ dst_seq,
                                                   const int32_t *__restrict__ dst_pos, int *err, float *red) {
    const int nq = r / 4;
    // cache destination of this row (if any), bounds-checked
    uint8_t *cache_codes = nullptr;
    void *cache_scale = nullptr;
    if (dst.codes) {
        const int b = dst_seq[t], p = dst_pos[t];
        if (b < 0 || b >= dst.B || p < 0 || p >= dst.Tmax) {
            if (threadIdx.x == 0) flag_error(err, kErrRange);
        } else {
            const size_t slot = size_t(b) * dst.Tmax + p;
            if (bits == 8) {
                cache_codes = static_cast<uint8_t *>(dst.codes) + slot * r;
                cache_scale = static_cast<float *>(dst.scales) + slot;
            } else {
                cache_codes = static_cast<uint8_t *>(dst.codes) + slot * (r / 2);
                cache_scale = static_cast<__half *>(dst.scales) + slot * (r / 128);
            }
        }
    }
    uint8_t *tok_codes = lat_codes ? static_cast<uint8_t *>(lat_codes) + t * (bits == 8 ? r : r / 2)
                                   : nullptr;

    if (bits == 8) {
        float m = 0.0f;
#pragma unroll
        for (int k = 0; k < kRqMaxQuads; ++k)
            m = fmaxf(m, fmaxf(fmaxf(fabsf(v[k].x), fabsf(v[k].y)), fmaxf(fabsf(v[k].z), fabsf(v[k].w))));
        m = block_max<kRqThreads>(m, red);
        const float s = quant_scale(m, clip, 127.0f), inv = quant_inv_scale(s);
#pragma unroll
        for (int k = 0; k < kRqMaxQuads; ++k) {
            const int qi = threadIdx.x + k * kRqThreads;
            if (qi >= nq) break;
            const uint32_t w = uint32_t(quant_code_fast(v[k].x, s, inv, 127) & 0xff) |
                               (uint32_t(quant_code_fast(v[k].y, s, inv, 127) & 0xff) << 8) |
                               (uint32_t(quant_code_fast(v[k].z, s, inv, 127) & 0xff) << 16) |
                               (uint32_t(quant_code_fast(v[k].w, s, inv, 127) & 0xff) << 24);
            if (tok_codes) reinterpret_cast<uint32_t *>(tok_codes)[qi] = w;
            if (cache_codes) reinterpret_cast<uint32_t *>(cache_codes)[qi] = w;
        }
        if (threadIdx.x == 0) {
            if (lat_scales) static_cast<float *>(lat_scales)[t] = s;
            if (cache_scale) *static_cast<float *>(cache_scale) = s;
        }
    } else {
        // quad qi covers channels 4qi..4qi+3; its group is qi / 32 = one warp row
#pragma unroll
        for (int k = 0; k < kRqMaxQuads; ++k) {
            const int qi = threadIdx.x + k * kRqThreads;
            if (qi - (threadIdx.x & 31) >= nq) break;       // warp-uniform
            float m = fmaxf(fmaxf(fabsf(v[k].x), fabsf(v[k].y)), fmaxf(fabsf(v[k].z), fabsf(v[k].w)));
            m = warp_max(m);
            const __half hs = int4_group_scale(m, clip);
            const float s = __half2float(hs), inv = quant_inv_scale(s);
            const int c0 = quant_code_fast(v[k].x, s, inv, 7), c1 = quant_code_fast(v[k].y, s, inv, 7);
            const int c2 = quant_code_fast(v[k].z, s, inv, 7), c3 = quant_code_fast(v[k].w, s, inv, 7);
            const uint16_t w = uint16_t((c0 & 0xf) | ((c1 & 0xf) << 4) | ((c2 & 0xf) << 8) | ((c3 & 0xf) << 12));
            if (tok_codes) reinterpret_cast<uint16_t *>(tok_codes)[qi] = w;
            if (cache_codes) reinterpret_cast<uint16_t *>(cache_codes)[qi] = w;
            if ((threadIdx.x & 31) == 0) {
                const int g = qi >> 5;
                if (lat_scales) static_cast<__half *>(lat_scales)[t * (r / 128) + g] = hs;
                if (cache_scale) static_cast<__half *>(cache_scale)[g] = hs;
            }
        }
    }
}


__device__ __forceinline__ void requant_row_cta(const float *c_hat, int64_t t, int r, int bits,
                                                float clip, void *__restrict__ lat_codes,
                                                void *__restrict__ lat_scales, const CacheView &dst,
                                                const int32_t *__restrict__ dst_seq,
                                                const int32_t *__restrict__ dst_pos, int *err, float *red) {
    const float *row = c_hat + t * r;
    const int nq = r / 4;
    float4 v[kRqMaxQuads];
#pragma unroll
    for (int k = 0; k < kRqMaxQuads; ++k) {
        const int qi = threadIdx.x + k * kRqThreads;
        v[k] = qi < nq ? reinterpret_cast<const float4 *>(row)[qi] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    requant_row_values(v, t, r, bits, clip, lat_codes, lat_scales, dst, dst_seq, dst_pos, err, red);
}


// The same per-token requantization by one warp (no block barriers): two
// passes over the row, the second reading it back from L1/L2.  Codes and
// scales are identical to requant_row_cta's (the maximum does not depend on
// the order of reduction).
__device__ __forceinline__ void requant_row_warp(const float *c_hat, int64_t t, int r, int bits,
                                                 float clip, void *__restrict__ lat_codes,
                                                 void *__restrict__ lat_scales, const CacheView &dst,
                                                 const int32_t *__restrict__ dst_seq,
                                                 const int32_t *__restrict__ dst_pos, int *err) {
    const int lane = threadIdx.x & 31;
    const float4 *row = reinterpret_cast<const float4 *>(c_hat + t * r);
    const int nq = r / 4;
    uint8_t *cache_codes = nullptr;
    void *cache_scale = nullptr;
    if (dst.codes) {
        const int b = dst_seq[t], p = dst_pos[t];
        if (b < 0 || b >= dst.B || p < 0 || p >= dst.Tmax) {
            if (lane == 0) flag_error(err, kErrRange);
        } else {
            const size_t slot = size_t(b) * dst.Tmax + p;
            if (bits == 8) {
                cache_codes = static_cast<uint8_t *>(dst.codes) + slot * r;
                cache_scale = static_cast<float *>(dst.scales) + slot;
            } else {
                cache_codes = static_cast<uint8_t *>(dst.codes) + slot * (r / 2);
                cache_scale = static_cast<__half *>(dst.scales) + slot * (r / 128);
            }
        }
    }
    uint8_t *tok_codes = lat_codes ? static_cast<uint8_t *>(lat_codes) + t * (bits == 8 ? r : r / 2) : nullptr;
    constexpr int kRegQ = 16;                        // rows of r <= 2048 stay in registers (one round of loads)
    if (nq <= 32 * kRegQ) {
        float4 v[kRegQ];
#pragma unroll
        for (int k = 0; k < kRegQ; ++k) {
            const int qi = k * 32 + lane;
            v[k] = qi < nq ? row[qi] : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        if (bits == 8) {
            float m = 0.0f;
#pragma unroll
            for (int k = 0; k < kRegQ; ++k)
                m = fmaxf(m, fmaxf(fmaxf(fabsf(v[k].x), fabsf(v[k].y)), fmaxf(fabsf(v[k].z), fabsf(v[k].w))));
            m = warp_max(m);
            const float s = quant_scale(m, clip, 127.0f), inv = quant_inv_scale(s);
#pragma unroll
            for (int k = 0; k < kRegQ; ++k) {
                const int qi = k * 32 + lane;
                if (qi >= nq) break;
                const uint32_t w = uint32_t(quant_code_fast(v[k].x, s, inv, 127) & 0xff) |
                                   (uint32_t(quant_code_fast(v[k].y, s, inv, 127) & 0xff) << 8) |
                                   (uint32_t(quant_code_fast(v[k].z, s, inv, 127) & 0xff) << 16) |
                                   (uint32_t(quant_code_fast(v[k].w, s, inv, 127) & 0xff) << 24);
                if (tok_codes) reinterpret_cast<uint32_t *>(tok_codes)[qi] = w;
                if (cache_codes) reinterpret_cast<uint32_t *>(cache_codes)[qi] = w;
            }
            if (lane == 0) {
                if (lat_scales) static_cast<float *>(lat_scales)[t] = s;
                if (cache_scale) *static_cast<float *>(cache_scale) = s;
            }
        } else {
            // group g = quads 32 g .. 32 g + 31: quad k of every lane
#pragma unroll
            for (int k = 0; k < kRegQ; ++k) {
                if (k * 32 >= nq) break;
                float m = fmaxf(fmaxf(fabsf(v[k].x), fabsf(v[k].y)), fmaxf(fabsf(v[k].z), fabsf(v[k].w)));
                m = warp_max(m);
                const __half hs = int4_group_scale(m, clip);
                const float s = __half2float(hs), inv = quant_inv_scale(s);
                const int c0 = quant_code_fast(v[k].x, s, inv, 7), c1 = quant_code_fast(v[k].y, s, inv, 7);
                const int c2 = quant_code_fast(v[k].z, s, inv, 7), c3 = quant_code_fast(v[k].w, s, inv, 7);
                const uint16_t w = uint16_t((c0 & 0xf) | ((c1 & 0xf) << 4) | ((c2 & 0xf) << 8) | ((c3 & 0xf) << 12));
                const int qi = k * 32 + lane;
                if (tok_codes) reinterpret_cast<uint16_t *>(tok_codes)[qi] = w;
                if (cache_codes) reinterpret_cast<uint16_t *>(cache_codes)[qi] = w;
                if (lane == 0) {
                    if (lat_scales) static_cast<__half *>(lat_scales)[t * (r / 128) + k] = hs;
                    if (cache_scale) static_cast<__half *>(cache_scale)[k] = hs;
                }
            }
        }
        return;
    }
    if (bits == 8) {
        float m = 0.0f;
#pragma unroll 4
        for (int qi = lane; qi < nq; qi += 32) {
            const float4 v = row[qi];
            m = fmaxf(m, fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w))));
        }
        m = warp_max(m);
        const float s = quant_scale(m, clip, 127.0f), inv = quant_inv_scale(s);
#pragma unroll 4
        for (int qi = lane; qi < nq; qi += 32) {
            const float4 v = row[qi];
            const uint32_t w = uint32_t(quant_code_fast(v.x, s, inv, 127) & 0xff) |
                               (uint32_t(quant_code_fast(v.y, s, inv, 127) & 0xff) << 8) |
                               (uint32_t(quant_code_fast(v.z, s, inv, 127) & 0xff) << 16) |
                               (uint32_t(quant_code_fast(v.w, s, inv, 127) & 0xff) << 24);
            if (tok_codes) reinterpret_cast<uint32_t *>(tok_codes)[qi] = w;
            if (cache_codes) reinterpret_cast<uint32_t *>(cache_codes)[qi] = w;
        }
        if (lane == 0) {
            if (lat_scales) static_cast<float *>(lat_scales)[t] = s;
            if (cache_scale) *static_cast<float *>(cache_scale) = s;
        }
    } else {
        // group g = quads 32 g .. 32 g + 31: one quad per lane
#pragma unroll 4
        for (int g = 0; g < r / 128; ++g) {
            const int qi = g * 32 + lane;
            const float4 v = row[qi];
            float m = fmaxf(fmaxf(fabsf(v.x), fabsf(v.y)), fmaxf(fabsf(v.z), fabsf(v.w)));
            m = warp_max(m);
            const __half hs = int4_group_scale(m, clip);
            const float s = __half2float(hs), inv = quant_inv_scale(s);
            const int c0 = quant_code_fast(v.x, s, inv, 7), c1 = quant_code_fast(v.y, s, inv, 7);
            const int c2 = quant_code_fast(v.z, s, inv, 7), c3 = quant_code_fast(v.w, s, inv, 7);
            const uint16_t w = uint16_t((c0 & 0xf) | ((c1 & 0xf) << 4) | ((c2 & 0xf) << 8) | ((c3 & 0xf) << 12));
            if (tok_codes) reinterpret_cast<uint16_t *>(tok_codes)[qi] = w;
            if (cache_codes) reinterpret_cast<uint16_t *>(cache_codes)[qi] = w;
            if (lane == 0) {
                if (lat_scales) static_cast<__half *>(lat_scales)[t * (r / 128) + g] = hs;
                if (cache_scale) static_cast<__half *>(cache_scale)[g] = hs;
            }
        }
    }
}

}  // namespace qsvd
