// Device helpers shared by the QSVD kernels: bf16 unpacking, the symmetric
// RTN quantizer, warp/block reductions and the device error word.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda_fp16.h>

#include "launch.h"

namespace qsvd {

__device__ __forceinline__ void flag_error(int *err, int bit) {
    if (err) atomicOr(err, bit);
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

// int4 group scale: fp32 scale rounded to fp16 (nearest even), saturated.
__device__ __forceinline__ __half int4_group_scale(float absmax, float clip) {
    return __float2half_rn(fminf(quant_scale(absmax, clip, 7.0f), 65504.0f));
}

// ---------------------------------------------------------------------------
// Reductions
// ---------------------------------------------------------------------------
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

}  // namespace qsvd
