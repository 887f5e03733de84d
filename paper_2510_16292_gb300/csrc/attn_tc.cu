// Decode attention over the latent cache on the 5th-generation tensor cores
// (Eq. 5 with W^u_k absorbed into the query: scores c_t . q~_h, softmax, and
// the softmax-weighted latent sum sum_t p_t c_t; W^u_v is applied afterwards
// by combine_uv_kernel).
//
// Work unit: a cluster of CL CTAs (CL = 2 for r <= 1536, 4 up to r = 3072)
// takes a contiguous range of 128-token tiles of one sequence.  CTA k owns the
// latent channels [k r/CL, (k+1) r/CL) (at most 768).  Per tile it computes
// partial scores over its channels, sends them to every peer through
// distributed shared memory and adds all CL partials in rank order, so every
// CTA runs the identical online softmax; each then accumulates o_lat for its
// own channels.  Splitting the channels bounds the tensor-memory footprint of
// the o_lat accumulator and the bytes each SM reads.
//
// Both products take their A operand from tensor memory, so no fp16 copy of
// the cache is ever written to or read from shared memory.  Per tile the CTA
// streams its channels twice (the second stream hits L2):
//   pass 1  warp 0 loads 128-token x 128-channel chunks with TMA; warpgroups
//           1-2 (thread = token, one 64-channel half each) convert them to
//           fp16 and store them into tensor memory token-major (int4: a word
//           of 8 codes at a time, channels in the order 0,4,1,5,2,6,3,7 of
//           each 8, the query block in the same order); warp 1 issues
//              S[t, h] += C[t, ch] Q[ch, h]      (M = 128 tokens, N = heads,
//           B = the fp16 query block in shared memory).
//   softmax warpgroups 5-6 (thread = token, 16 heads each) read S, swap
//           partials with the peers, apply the token scale and 1/sqrt(dh), run
//           the online softmax (o_lat is rescaled lazily, only when the
//           running maximum of a head grows by more than kRescale2) and write
//           P (fp16, [heads x tokens]).
//   pass 2  warp 3 loads the same chunks again (and, for int4, the tile's
//           group scales); warpgroups 3-4 convert them to fp16, transpose
//           8 x 8 blocks in registers (movmatrix) and store them channel-major
//           into tensor memory; warp 2 issues
//              O^T[ch, h] += C^T[ch, t] P[t, h]  (M = 128 channels, K = tokens).
//           The transposed blocks put the 16 tokens of an MMA step in the
//           order 0,1,8,9,2,3,10,11,...; P is written in the same order.
// int8 codes are exact in fp16; the per-token scale multiplies the scores and
// is folded into P.  int4 codes are converted to code * group-scale in fp16.
// The query block is scaled per head by a power of two so that its largest
// entry sits just below 2^14 (the scale is undone on the scores).
//
// Every wait is bounded in time (on expiry the error word gets kErrTimeout and
// the CTA abandons its tiles); a CTA always drains its own copies and MMAs,
// meets its peer at the final cluster barrier, and frees its tensor memory.
#include <algorithm>
#include <cfloat>
#include <cstdint>
#include <cuda.h>
#include <cuda_fp16.h>

#include "common.cuh"
#include "launch.h"
#include "tcgen05.cuh"

namespace qsvd {

namespace atc {

constexpr int kTile = 128;        // tokens per tile
constexpr int kChunk = 128;       // channels per TMA chunk
constexpr int kThreads = 896;     // 28 warps
constexpr int kMaxN = 32;         // heads (padded to a multiple of 16)
constexpr int kHalfN = 16;        // heads per softmax warpgroup
constexpr int kMaxRc = 768;       // channels per CTA
constexpr int kMaxGroups = 24;    // int4 scale groups per token (r <= 3072)
constexpr float kRescale2 = 11.5f;  // lazy rescale threshold (log2 units, about 8 in natural-log units)
constexpr unsigned long long kWaitNs = 2000000000ull;   // 2 s per wait

// dynamic shared memory (byte offsets from a 1024-aligned base) of a cluster
// of CL CTAs: the exchange buffer holds the CL - 1 peers' partial scores, and
// a cluster of 4 pays for it with shallower TMA rings
constexpr int kQtBytes = kMaxN * kMaxRc * 2;       // query block, fp16, 128-byte swizzled, K-major
constexpr int kSlotBytes = kTile * kChunk;         // one int8 chunk (int4 uses half)
constexpr int kPBytes = kMaxN * kTile * 2;         // P, fp16, 128-byte swizzled, K-major
constexpr int kXchSlot = kTile * kMaxN * 4;        // one peer's partial scores
constexpr int kScBytes = kTile * kMaxGroups * 2;   // int4 group scales of one tile, [token][group]
template <int CL>
struct Lay {
    static constexpr int kRing1 = CL == 2 ? 4 : 3;    // pass-1 TMA slots
    static constexpr int kRing2 = CL == 2 ? 3 : 2;    // pass-2 TMA slots
    static constexpr int kOffQt = 0;
    static constexpr int kOffT1 = kOffQt + kQtBytes;
    static constexpr int kOffT2 = kOffT1 + kRing1 * kSlotBytes;
    static constexpr int kOffP = kOffT2 + kRing2 * kSlotBytes;
    static constexpr int kOffXch = kOffP + 2 * kPBytes;
    static constexpr int kOffSc = kOffXch + (CL - 1) * kXchSlot;
    static constexpr int kOffLt = kOffSc + 2 * kScBytes;   // softmax running sums, [heads][tokens] fp32
    static constexpr int kSmemBytes = kOffLt + kMaxN * kTile * 4 + 1024;
};
static_assert(Lay<2>::kSmemBytes <= 227 * 1024 - 2048 && Lay<4>::kSmemBytes <= 227 * 1024 - 2048, "shared memory");
// Cluster size for rank r: each CTA owns r / CL <= kMaxRc latent channels.
__host__ __device__ constexpr int cluster_for(int r) { return r <= 2 * kMaxRc ? 2 : 4; }

// tensor memory columns
constexpr uint32_t kColO = 0;      // o_lat^T: (r_c / 128) x Np       (<= 192)
constexpr uint32_t kColS = 192;    // scores: 2 buffers x 32
constexpr int kABufs = 4;          // scores A operand buffers (64 channels each)
constexpr uint32_t kColA = 256;    // scores A operand: kABufs x 32 columns
constexpr uint32_t kColV = 384;    // PV A operand: 2 buffers x 64 columns (128 tokens, fp16 pairs)
constexpr uint32_t kTmemCols = 512;

struct Params {
    CacheView c;
    const int32_t *seq_len;
    const float *qt;        // [B, H, r] fp32
    const unsigned *qmax;   // [B, H] bit patterns of max_j |qt[b, h, j]| (non-negative floats)
    int H, Hs, Np;          // heads in all (array stride); heads of this launch (<= 32), padded to 16
                            // (qt, qmax, pm, pl, po point at the launch's first head)
    float softmax_scale;
    int tiles_per_split, n_split;
    float *pm, *pl, *po;    // [B, n_split, H] and [B, n_split, H, r]
    int *err;
};

// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t map_peer(uint32_t local, uint32_t peer) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(peer));
    return r;
}
// Asynchronous 16-byte store into the peer's shared memory; its completion
// counts 16 bytes on the peer's mbarrier `bar` (both cluster addresses).
__device__ __forceinline__ void st_async_v4(uint32_t addr, float a, float b, float c, float d, uint32_t bar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, [%5];"
                 ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d), "r"(bar)
                 : "memory");
}
__device__ __forceinline__ void arrive_peer(uint32_t bar_cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster_addr) : "memory");
}
// Relaxed remote arrival: used where the caller's earlier accesses to the
// peer-written buffer are reads whose values it has already consumed.
__device__ __forceinline__ void arrive_peer_relaxed(uint32_t bar_cluster_addr) {
    asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster_addr) : "memory");
}
__device__ __forceinline__ void arrive_local(uint64_t *bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ bool try_wait_acq_cluster(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile("{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
                 "selp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(ok)
                 : "r"(smem_addr(bar)), "r"(parity)
                 : "memory");
    return ok != 0;
}
// Cluster-scope test without the acquire (no L1 invalidation per try); the
// caller fences once after the phase completed.
__device__ __forceinline__ bool try_wait_relaxed_cluster(uint64_t *bar, uint32_t parity) {
    uint32_t ok;
    asm volatile("{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.relaxed.cluster.shared::cta.b64 p, [%1], %2;\n\t"
                 "selp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(ok)
                 : "r"(smem_addr(bar)), "r"(parity)
                 : "memory");
    return ok != 0;
}
__device__ __forceinline__ void fence_acquire_cluster() { asm volatile("fence.acq_rel.cluster;" ::: "memory"); }
__device__ __forceinline__ unsigned long long now_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
// Wait for phase `parity` of `bar`, for at most kWaitNs.  Each try_wait
// suspends the thread in hardware until the phase completes or a short
// system-defined time passes, so the loop issues little; the clock is read
// every 64 tries.  `cluster`: the phase is completed by the peer CTA (relaxed
// tries, one cluster-scope acquire fence at the end).
__device__ __noinline__ bool wait_bar(uint64_t *bar, uint32_t parity, int *err, bool cluster) {
    const unsigned long long t0 = now_ns();
    for (uint32_t i = 1;; ++i) {
        if (cluster ? try_wait_relaxed_cluster(bar, parity) : mbar_try_wait(bar, parity)) {
            if (cluster) fence_acquire_cluster();
            return true;
        }
        if ((i & 63u) == 0 && now_ns() - t0 > kWaitNs) {
            flag_error(err, kErrTimeout);
            return false;
        }
    }
}
__device__ __forceinline__ bool wait(uint64_t *bar, uint32_t parity, int *err) {
    return mbar_try_wait(bar, parity) || wait_bar(bar, parity, err, false);
}
// Warp-uniform forms: every lane waits (and acquires); the warp agrees on the outcome.
__device__ __forceinline__ bool wwait(uint64_t *bar, uint32_t parity, int *err) {
    return __all_sync(0xffffffffu, wait(bar, parity, err));
}
__device__ __forceinline__ bool wwait_cluster(uint64_t *bar, uint32_t parity, int *err) {
    return __all_sync(0xffffffffu, try_wait_acq_cluster(bar, parity) || wait_bar(bar, parity, err, true));
}
// Named barrier `id` over the 128 threads of one softmax warpgroup, returning
// the OR of `v` over them.
__device__ __forceinline__ bool group_any(bool v, int id) {
    uint32_t r;
    asm volatile("{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\tbar.red.or.pred q, %2, 128, p;\n\t"
                 "selp.u32 %0, 1, 0, q;\n\t}"
                 : "=r"(r)
                 : "r"(uint32_t(v)), "r"(id)
                 : "memory");
    return r != 0;
}
__device__ __forceinline__ void group_sync(int id) { asm volatile("bar.sync %0, 128;" ::"r"(id) : "memory"); }
// L2 prefetch of one box of a tensor map (no shared memory, no completion).
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap *map, int x, int y) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global.tile [%0, {%1, %2}];"
                 ::"l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y)
                 : "memory");
}
// tcgen05 / TMA wrappers shared with the other tensor-core kernels (tcgen05.cuh)
using tc::commit;
using tc::fence_after;
using tc::fence_before;
using tc::mma_ss;
using tc::mma_ts;
using tc::tma_load_2d;
using tc::tmem_ld16;
using tc::tmem_ld32;
using tc::tmem_ld8;
using tc::tmem_st16;
using tc::tmem_st16x256_x2;
using tc::tmem_st32;
using tc::tmem_st8;
using tc::tmem_wait_ld;
using tc::tmem_wait_st;
// Shared-memory matrix descriptor, 128-byte swizzle, explicit leading / stride offsets.
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return tc::desc_sw128_lbo(saddr, lbo, sbo);
}
// Instruction descriptor: f16 x f16 -> f32, M = 128, N = n; a_mn: A is M-major.
__host__ __device__ constexpr uint32_t idesc_f16(int n, int a_mn) {
    return (1u << 4) | (uint32_t(a_mn) << 15) | (uint32_t(n >> 3) << 17) | (uint32_t(128 >> 4) << 24);
}
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Eight int4 codes (element i in bits 4i..4i+3, two's complement) times an
// fp16 group scale -> four fp16 pairs in the order (0,4), (1,5), (2,6), (3,7)
// (products rounded to nearest).  The nibbles xor 8 are placed in the
// mantissas of 1024 and 1024 * 16; one add or fused multiply-add maps them
// back to the codes exactly.
__device__ __forceinline__ void i4x8_h2x4_perm(uint32_t w, __half2 s2, uint32_t (&o)[4]) {
    const uint32_t y = w >> 8;
    const uint32_t z[4] = {(w & 0x000F000Fu) ^ 0x64086408u, (w & 0x00F000F0u) ^ 0x64806480u,
                           (y & 0x000F000Fu) ^ 0x64086408u, (y & 0x00F000F0u) ^ 0x64806480u};
    const __half2 b_lo = __half2half2(__ushort_as_half(0xE408));     // -1032
    const __half2 m_hi = __half2half2(__ushort_as_half(0x2C00));     // 1/16
    const __half2 b_hi = __half2half2(__ushort_as_half(0xD480));     // -72
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const __half2 zk = *reinterpret_cast<const __half2 *>(&z[k]);
        const __half2 c = (k & 1) ? __hfma2(zk, m_hi, b_hi) : __hadd2(zk, b_lo);
        const __half2 h = __hmul2(c, s2);
        o[k] = *reinterpret_cast<const uint32_t *>(&h);
    }
}
// Byte k of w (two int4 codes, the even channel in the low nibble) -> the fp16
// pair (code_even * s, code_odd * s), products rounded to nearest.  The nibbles
// (xor 8) are placed in the mantissas of 1024 and 1024 * 16, which the fused
// multiply-add maps back to the codes exactly.
__device__ __forceinline__ uint32_t i4pair_h2(uint32_t w, int k, __half2 s2) {
    const uint32_t y = __byte_perm(w, 0u, uint32_t(k) | (4u << 4) | (uint32_t(k) << 8) | (4u << 12));
    const uint32_t z = (y & 0x00F0000Fu) ^ 0x64806408u;            // 1024 + (lo ^ 8), 1024 + 16 (hi ^ 8)
    const __half2 mul = __halves2half2(__ushort_as_half(0x3C00), __ushort_as_half(0x2C00));   // 1, 1/16
    const __half2 add = __halves2half2(__ushort_as_half(0xE408), __ushort_as_half(0xD480));   // -1032, -72
    const __half2 c = __hfma2(*reinterpret_cast<const __half2 *>(&z), mul, add);
    const __half2 h = __hmul2(c, s2);
    return *reinterpret_cast<const uint32_t *>(&h);
}
// Bytes k, k+1 of u = w ^ 0x80808080 (two int8 codes) -> their fp16 pair, exact.
__device__ __forceinline__ uint32_t i8pair_h2(uint32_t u, int k) {
    const uint32_t a = __byte_perm(u, 0x64646464u, uint32_t(k) | (4u << 4) | (uint32_t(k + 1) << 8) | (4u << 12));
    const __half2 h = __hsub2(*reinterpret_cast<const __half2 *>(&a), __half2half2(__ushort_as_half(0x6480)));
    return *reinterpret_cast<const uint32_t *>(&h);
}
// Transpose of an 8 x 8 fp16 matrix held one pair per thread (thread t: row
// t/4, columns 2(t%4), 2(t%4)+1).
__device__ __forceinline__ uint32_t movm_t(uint32_t a) {
    uint32_t d;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
    return d;
}
// 4-byte asynchronous copy; src_bytes = 0 writes zeros without reading.
__device__ __forceinline__ void cp_async4(void *dst, const void *src, uint32_t src_bytes) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(smem_addr(dst)), "l"(src), "r"(src_bytes)
                 : "memory");
}
// Arrival on `bar` once this thread's earlier asynchronous copies have landed.
__device__ __forceinline__ void cp_async_arrive(uint64_t *bar) {
    asm volatile("cp.async.mbarrier.arrive.noinc.shared::cta.b64 [%0];" ::"r"(smem_addr(bar)) : "memory");
}
// Position of token u (0..15) of an MMA step in the K order of the transposed
// PV operand: u = 8h + 2m + e sits at 4m + 2h + e.
__device__ __forceinline__ int kpos16(int u) { return ((u & 6) << 1) | ((u & 8) >> 2) | (u & 1); }

// Byte offset of 16-byte chunk q of row `row` in a 128-byte-swizzled tile
// (rows of 128 bytes, tile base 1024-aligned).
__device__ __forceinline__ uint32_t sw128(uint32_t row, uint32_t q) { return row * 128u + ((q ^ (row & 7u)) << 4); }
// The same for a 64-byte-swizzled tile (rows of 64 bytes).
__device__ __forceinline__ uint32_t sw64(uint32_t row, uint32_t q) {
    return row * 64u + ((q ^ ((row >> 1) & 3u)) << 4);
}

__device__ __forceinline__ uint16_t load_group_scale(const CacheView &c, size_t slot, int group, bool live) {
    return live ? static_cast<const uint16_t *>(c.scales)[slot * (c.r / 128) + group] : uint16_t(0);
}

}  // namespace atc

// ---------------------------------------------------------------------------
template <int BITS, int CL>
__global__ void __launch_bounds__(atc::kThreads, 1)
attn_tc_kernel(const __grid_constant__ CUtensorMap map_c, const atc::Params p) {
    using namespace atc;
    using Ly = Lay<CL>;
    constexpr int kRing1 = Ly::kRing1, kRing2 = Ly::kRing2;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t t1_full[kRing1], t1_empty[kRing1], t2_full[kRing2], t2_empty[kRing2];
    __shared__ __align__(8) uint64_t a_full[kABufs], a_empty[kABufs], s_full[2], s_empty[2];
    __shared__ __align__(8) uint64_t pva_full[2], pva_empty[2], p_full[2], p_empty[2], sc_full[2], sc_empty[2];
    __shared__ __align__(8) uint64_t xch_full[2], xch_empty[2], mma_done[2];
    __shared__ uint32_t tmem_base;
    __shared__ float red_max[2][4][kHalfN];
    __shared__ float m_ref[kMaxN], alpha[kMaxN], q_exp[kMaxN], qfac[kMaxN];
    __shared__ volatile int abort_flag;

    const CacheView &c = p.c;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    const int split = blockIdx.x / CL, b = blockIdx.y;
    const int r = c.r, rc = r / CL, ch0 = int(rank) * rc;
    const int n_chunks = rc / kChunk;
    // H: this launch's heads; the arrays' head stride is p.H
    const int Np = p.Np, H = p.Hs;
    constexpr uint32_t kLoadBytes = BITS == 8 ? kTile * kChunk : kTile * kChunk / 2;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kRing1; ++i) {
            mbar_init(&t1_full[i], 1);
            mbar_init(&t1_empty[i], 8);
        }
        for (int i = 0; i < kRing2; ++i) {
            mbar_init(&t2_full[i], 1);
            mbar_init(&t2_empty[i], 8);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&s_full[i], 1);
            mbar_init(&s_empty[i], 8);
            mbar_init(&pva_full[i], 8);
            mbar_init(&pva_empty[i], 1);
            mbar_init(&p_full[i], 8);
            mbar_init(&p_empty[i], 1);
            mbar_init(&sc_full[i], 32);     // one cp.async-tracked arrival per lane of warp 3
            mbar_init(&sc_empty[i], 8);
            mbar_init(&mma_done[i], 1);
            mbar_init(&xch_full[i], 1);     // one local expect-tx arrival + the peers' st.async bytes
            mbar_init(&xch_empty[i], 128 * (CL - 1));   // every thread of each peer's warpgroup, after reading
        }
        for (int i = 0; i < kABufs; ++i) {
            mbar_init(&a_full[i], 4);
            mbar_init(&a_empty[i], 1);
        }
        mbar_init_fence();
        abort_flag = 0;
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     ::"r"(smem_addr(&tmem_base)), "r"(kTmemCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    fence_before();
    __syncthreads();
    fence_after();
    cluster_sync();                  // the peers' barriers exist before any remote arrive
    const uint32_t tmem = tmem_base;
    pdl_trigger();

    // lengths and sequence map: call inputs, complete before this grid starts
    // (the query kernels let their dependents start only after their own wait)
    const int sq = view_seq(c, b);
    const int L = sq < 0 ? 0 : p.seq_len[b];
    const bool valid = L >= 1 && L <= c.Tmax;
    const int t_begin = split * p.tiles_per_split * kTile;
    const int t_end = valid ? min(L, t_begin + p.tiles_per_split * kTile) : t_begin;
    const int n_tiles = t_end > t_begin ? (t_end - t_begin + kTile - 1) / kTile : 0;
    const size_t row0 = size_t(valid ? sq : 0) * c.Tmax;   // cache slot of token 0 of the sequence
    const int total = n_tiles * n_chunks;             // chunk loads per pass
    const int ngrp = r / 128;                         // int4 scale groups per token
    // the first two tiles' chunks into L2 while the producer grid finishes (L2
    // is the point of coherence, so a row the projection writes meanwhile is
    // never seen stale: the shared-memory copies come after the wait)
    constexpr int kPrefetchTiles = 2;
    if (warp == 0 && lane == 0)
        for (int i = 0; i < min(total, kPrefetchTiles * n_chunks); ++i)
            tma_prefetch_2d(&map_c, (ch0 + (i % n_chunks) * kChunk) * BITS / 8, int(row0) + t_begin + (i / n_chunks) * kTile);
    pdl_wait();

    // ---- query block: per-head power-of-two scale from the max over all r
    // channels (both CTAs of the pair get the same scale), then the fp16
    // block Q^T [heads][channels of this CTA], 128-byte swizzled, 64 channels
    // per 128-byte row, blocks of Np rows.  Built by warps 4-27 and awaited by
    // them and the MMA warps at named barrier 3; the TMA producers (warps 0 and
    // 3) start streaming cache chunks at once.  The q~ loads are issued before
    // the per-head scales are known.
    constexpr int kQbThreads = kThreads - 64;          // every warp but 0 and 3
    if (warp != 0 && warp != 3) {
        if (n_tiles > 0) {
            constexpr int kPer = 4;                     // items per thread: Np (rc / 8) <= 32 * 96 = kPer * 768
            const int items = Np * (rc / 8);            // 8 channels per item
            const int i0 = threadIdx.x - 128;
            float4 va[kPer], vb[kPer];
            if (warp >= 4) {
#pragma unroll
                for (int k = 0; k < kPer; ++k) {
                    const int i = i0 + k * (kThreads - 128);
                    const int h = i / (rc / 8), q8 = i % (rc / 8);
                    va[k] = vb[k] = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (i < items && h < H) {
                        const float4 *src = reinterpret_cast<const float4 *>(p.qt + (size_t(b) * p.H + h) * r + ch0 + q8 * 8);
                        va[k] = src[0];
                        vb[k] = src[1];
                    }
                }
            }
            if (warp == 4) {
                const int h = lane;
                int e = 0;
                if (h < H) {
                    const float m = __uint_as_float(p.qmax[size_t(b) * p.H + h]);   // max_j |q~[b, h, j]|
                    if (m > 0.0f) frexpf(m, &e);                                   // m < 2^e
                }
                q_exp[h] = float(14 - e);                                          // |q~| * 2^(14-e) < 2^14
                // scores -> logits in log2 units: undo the query scale, times softmax_scale * log2(e)
                qfac[h] = exp2f(float(e - 14)) * p.softmax_scale * 1.4426950408889634f;
                m_ref[h] = -INFINITY;
            }
            asm volatile("bar.sync 3, %0;" ::"n"(kQbThreads) : "memory");
            if (warp >= 4) {
#pragma unroll
                for (int k = 0; k < kPer; ++k) {
                    const int i = i0 + k * (kThreads - 128);
                    if (i >= items) break;
                    const int h = i / (rc / 8), q8 = i % (rc / 8);
                    const int kc = q8 >> 3, q = q8 & 7;
                    const float sc = exp2f(q_exp[h]);
                    const float4 a = va[k], bq = vb[k];
                    // int4: the order of the pass-1 operand, 0,4,1,5,2,6,3,7 within each 8 channels
                    const __half2 v0 = BITS == 4 ? __floats2half2_rn(a.x * sc, bq.x * sc) : __floats2half2_rn(a.x * sc, a.y * sc);
                    const __half2 v1 = BITS == 4 ? __floats2half2_rn(a.y * sc, bq.y * sc) : __floats2half2_rn(a.z * sc, a.w * sc);
                    const __half2 v2 = BITS == 4 ? __floats2half2_rn(a.z * sc, bq.z * sc) : __floats2half2_rn(bq.x * sc, bq.y * sc);
                    const __half2 v3 = BITS == 4 ? __floats2half2_rn(a.w * sc, bq.w * sc) : __floats2half2_rn(bq.z * sc, bq.w * sc);
                    *reinterpret_cast<uint4 *>(sm + Ly::kOffQt + kc * (Np * 128) + sw128(h, q)) =
                        make_uint4(*reinterpret_cast<const uint32_t *>(&v0), *reinterpret_cast<const uint32_t *>(&v1),
                                   *reinterpret_cast<const uint32_t *>(&v2), *reinterpret_cast<const uint32_t *>(&v3));
                }
                fence_async_smem();
            }
        }
        asm volatile("bar.sync 3, %0;" ::"n"(kQbThreads) : "memory");
    }

    if (warp == 0) {
        // ---------------- TMA producer, pass 1 ----------------
        if (lane == 0 && total > 0) {
            int issued = 0;
            // keep the chunks of the next two tiles streaming into L2 (the first
            // kPrefetchTiles were prefetched before the wait)
            const int ahead = 2 * n_chunks;
            int pj = min(total, kPrefetchTiles * n_chunks);  // next chunk to prefetch
            int pck = pj % n_chunks, ptile = pj / n_chunks;
            auto prefetch = [&]() {
                tma_prefetch_2d(&map_c, (ch0 + pck * kChunk) * BITS / 8, int(row0) + t_begin + ptile * kTile);
                ++pj;
                if (++pck == n_chunks) { pck = 0; ++ptile; }
            };
            while (pj < ahead && pj < total) prefetch();
            for (int i = 0, tile = 0, ck = 0; i < total && !abort_flag; ++i) {
                const int s = i % kRing1;
                if (pj < total) prefetch();
                if (i >= kRing1 && !wait(&t1_empty[s], ((i / kRing1) - 1) & 1, p.err)) { abort_flag = 1; break; }
                mbar_arrive_expect_tx(&t1_full[s], kLoadBytes);
                tma_load_2d(sm + Ly::kOffT1 + s * kSlotBytes, &map_c, (ch0 + ck * kChunk) * BITS / 8,
                            int(row0) + t_begin + tile * kTile, &t1_full[s]);
                ++issued;
                if (++ck == n_chunks) { ck = 0; ++tile; }
            }
            // every issued copy has landed before the CTA may finish
            for (int i = issued - kRing1 > 0 ? issued - kRing1 : 0; i < issued; ++i)
                wait(&t1_full[i % kRing1], (i / kRing1) & 1, p.err);
        }
    } else if (warp == 3) {
        // ---------------- TMA producer, pass 2 (+ int4 group scales) ----------------
        int issued = 0;
        for (int i = 0, tile = 0, ck = 0; i < total; ++i, ck = (ck + 1 == n_chunks) ? 0 : ck + 1, tile += (ck == 0)) {
            if (__any_sync(0xffffffffu, abort_flag != 0)) break;
            const int s = i % kRing2;
            if (BITS == 4 && ck == 0) {
                // the tile's scale rows [token][ngrp] into ring slot tile & 1 (4-byte copies;
                // tokens past the end get zeros, so dead rows contribute 0, never NaN)
                const int sl = tile & 1;
                if (tile >= 2 && !wwait(&sc_empty[sl], ((tile >> 1) - 1) & 1, p.err)) { abort_flag = 1; break; }
                uint8_t *dst = sm + Ly::kOffSc + sl * kScBytes;
                const int nw = ngrp / 2;
                for (int tt = lane; tt < kTile; tt += 32) {
                    const int tok = t_begin + tile * kTile + tt;
                    const bool live = tok < t_end;
                    const uint32_t *src = static_cast<const uint32_t *>(c.scales) + (row0 + (live ? tok : t_begin)) * nw;
                    for (int k = 0; k < nw; ++k) cp_async4(dst + size_t(tt * nw + k) * 4, src + k, live ? 4u : 0u);
                }
                cp_async_arrive(&sc_full[sl]);
            }
            bool ok = true;
            if (lane == 0) {
                if (i >= kRing2 && !wait(&t2_empty[s], ((i / kRing2) - 1) & 1, p.err)) ok = false;
                if (ok) {
                    mbar_arrive_expect_tx(&t2_full[s], kLoadBytes);
                    tma_load_2d(sm + Ly::kOffT2 + s * kSlotBytes, &map_c, (ch0 + ck * kChunk) * BITS / 8,
                                int(row0) + t_begin + tile * kTile, &t2_full[s]);
                }
            }
            if (!__shfl_sync(0xffffffffu, ok, 0)) { abort_flag = 1; break; }
            ++issued;
        }
        if (lane == 0)
            for (int i = issued - kRing2 > 0 ? issued - kRing2 : 0; i < issued; ++i)
                wait(&t2_full[i % kRing2], (i / kRing2) & 1, p.err);
        asm volatile("cp.async.wait_all;" ::: "memory");
    } else if (warp == 1) {
        // ---------------- scores MMA ----------------
        if (lane == 0 && n_tiles > 0) {
            const uint32_t idesc = idesc_f16(Np, 0);
            int half = 0;
            for (int tile = 0; tile < n_tiles && !abort_flag; ++tile) {
                const int sb = tile & 1;
                if (tile >= 2 && !wait(&s_empty[sb], ((tile >> 1) - 1) & 1, p.err)) { abort_flag = 1; break; }
                fence_after();
                bool ok = true;
                for (int hh = 0; hh < 2 * n_chunks; ++hh, ++half) {
                    const int ab = half % kABufs;
                    if (!wait(&a_full[ab], (half / kABufs) & 1, p.err)) { ok = false; break; }
                    fence_after();
                    const uint32_t qblk = smem_addr(sm + Ly::kOffQt + hh * (Np * 128));
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_ts(tmem + kColS + sb * 32, tmem + kColA + ab * 32 + k * 8, sdesc(qblk + k * 32, 16, 1024),
                               idesc, (hh > 0 || k > 0) ? 1u : 0u);
                    commit(&a_empty[ab]);
                }
                if (!ok) { abort_flag = 1; break; }
                commit(&s_full[sb]);
            }
            commit(&mma_done[0]);
            wait(&mma_done[0], 0, p.err);
        }
    } else if (warp == 2) {
        // ---------------- PV MMA: O^T += C^T P, A from tensor memory ----------------
        if (lane == 0 && n_tiles > 0) {
            const uint32_t idesc = idesc_f16(Np, 0);
            int chunk = 0;
            for (int tile = 0; tile < n_tiles && !abort_flag; ++tile) {
                const int pb = tile & 1;
                if (!wait(&p_full[pb], (tile >> 1) & 1, p.err)) { abort_flag = 1; break; }
                fence_after();
                const uint32_t pbase = smem_addr(sm + Ly::kOffP + pb * kPBytes);
                bool ok = true;
                for (int ck = 0; ck < n_chunks; ++ck, ++chunk) {
                    const int vb = chunk & 1;
                    if (!wait(&pva_full[vb], (chunk >> 1) & 1, p.err)) { ok = false; break; }
                    fence_after();
#pragma unroll
                    for (int k = 0; k < kTile / 16; ++k) {
                        // B: P^T rows = heads; 64-token blocks Np * 128 bytes apart
                        const uint64_t bb = sdesc(pbase + (k >> 2) * (Np * 128) + (k & 3) * 32, 16, 1024);
                        mma_ts(tmem + kColO + ck * Np, tmem + kColV + vb * 64 + k * 8, bb, idesc,
                               (tile > 0 || k > 0) ? 1u : 0u);
                    }
                    commit(&pva_empty[vb]);
                }
                if (!ok) { abort_flag = 1; break; }
                commit(&p_empty[pb]);
            }
            commit(&mma_done[1]);
            wait(&mma_done[1], 0, p.err);
        }
    } else if (warp < 12) {
        // ---------------- warpgroups 1-2: pass-1 converter, thread = token ----------------
        // warp (quad, hh): tokens 32 quad + lane, channels [64 hh, 64 hh + 64) of each chunk
        const int quad = warp & 3, hh = (warp - 4) >> 2, t = quad * 32 + lane;
        const uint32_t trow = tmem + (uint32_t(quad * 32) << 16);
        uint16_t scc[kMaxRc / 128], scn[kMaxRc / 128];     // this token's group scales, current / next tile
        auto load_sc = [&](int tile, uint16_t (&o)[kMaxRc / 128]) {
            const int tok = t_begin + tile * kTile + t;
#pragma unroll
            for (int k = 0; k < kMaxRc / 128; ++k)
                o[k] = (k < n_chunks) ? load_group_scale(c, row0 + tok, ch0 / 128 + k, tok < t_end) : uint16_t(0);
        };
        if (BITS == 4 && n_tiles > 0) load_sc(0, scn);
        for (int i = 0, tile = 0, ck = 0; i < total && !__any_sync(0xffffffffu, abort_flag != 0);
             ++i, ck = (ck + 1 == n_chunks) ? 0 : ck + 1, tile += (ck == 0)) {
            const int s = i % kRing1;
            if (BITS == 4 && ck == 0) {
#pragma unroll
                for (int k = 0; k < kMaxRc / 128; ++k) scc[k] = scn[k];
                if (tile + 1 < n_tiles) load_sc(tile + 1, scn);      // a tile ahead
            }
            if (!wwait(&t1_full[s], (i / kRing1) & 1, p.err)) { abort_flag = 1; break; }
            const uint8_t *slot = sm + Ly::kOffT1 + s * kSlotBytes;
            const int half = 2 * i + hh, ab = half % kABufs;
            bool ok = half < kABufs || wwait(&a_empty[ab], ((half / kABufs) - 1) & 1, p.err);
            if (ok) {
                uint16_t scv = scc[0];
#pragma unroll
                for (int k = 1; k < kMaxRc / 128; ++k)
                    if (k == ck) scv = scc[k];
                const __half2 s2 = __half2half2(__ushort_as_half(scv));
                // the half-chunk's codes (64 channels), every load issued first
                constexpr int kU = BITS == 8 ? 4 : 2;       // 16-byte units
                uint4 wl[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u)
                    wl[u] = *reinterpret_cast<const uint4 *>(slot + (BITS == 8 ? sw128(t, hh * 4 + u) : sw64(t, hh * 2 + u)));
#pragma unroll
                for (int q = 0; q < 2; ++q) {               // 32 channels per store
                    uint32_t v[16];
                    if (BITS == 8) {
#pragma unroll
                        for (int u = 0; u < 2; ++u) {       // 2 x 16 codes
                            const uint4 w = wl[q * 2 + u];
                            i8x4_to_h2x2(w.x, v[u * 8 + 0], v[u * 8 + 1]);
                            i8x4_to_h2x2(w.y, v[u * 8 + 2], v[u * 8 + 3]);
                            i8x4_to_h2x2(w.z, v[u * 8 + 4], v[u * 8 + 5]);
                            i8x4_to_h2x2(w.w, v[u * 8 + 6], v[u * 8 + 7]);
                        }
                    } else {
                        const uint32_t ww[4] = {wl[q].x, wl[q].y, wl[q].z, wl[q].w};   // 32 codes
#pragma unroll
                        for (int j = 0; j < 4; ++j) {    // channels 8j..8j+7 in the order 0,4,1,5,2,6,3,7
                            uint32_t o4[4];
                            i4x8_h2x4_perm(ww[j], s2, o4);
#pragma unroll
                            for (int k = 0; k < 4; ++k) v[j * 4 + k] = o4[k];
                        }
                    }
                    tmem_st16(trow + kColA + ab * 32 + q * 16, v);
                }
                tmem_wait_st();
                fence_before();
                __syncwarp();
                if (lane == 0) arrive_local(&a_full[ab]);
            }
            __syncwarp();
            if (lane == 0) arrive_local(&t1_empty[s]);
            if (!ok) { abort_flag = 1; break; }
        }
    } else if (warp < 20) {
        // ---------------- warpgroups 3-4: pass-2 converter, channel-major into tensor memory ----------------
        // warp (q, th): channels [32 q, 32 q + 32) of each chunk (its tensor-memory lanes),
        // tokens [64 th, 64 th + 64).  Thread t supplies, per 8 x 8 block (tokens x channels),
        // the pair of channels 2(t%4), 2(t%4)+1 of token t/4; movmatrix turns it into the pair
        // of tokens 2(t%4), 2(t%4)+1 of channel t/4, one 32-bit tensor-memory word.
        const int q = warp & 3, th = (warp - 12) >> 2, cq = lane & 3, g8 = lane >> 2;
        // The tokens this thread supplies are 64 th + 32 h32 + 8 j + g8: their row
        // swizzle depends on g8 only, so every shared-memory address below is a
        // per-thread base plus a compile-time offset.
        const uint32_t rbase = uint32_t(64 * th + g8);
        const uint32_t off4 = rbase * 64u + ((uint32_t(q) ^ ((uint32_t(g8) >> 1) & 3u)) << 4);        // int4 rows
        const uint32_t off8a = rbase * 128u + ((uint32_t(2 * q) ^ uint32_t(g8)) << 4);                 // int8 rows,
        const uint32_t off8b = rbase * 128u + ((uint32_t(2 * q + 1) ^ uint32_t(g8)) << 4);             // two units
        const int k8 = (cq & 1) * 2;
        for (int i = 0, tile = 0, ck = 0; i < total && !__any_sync(0xffffffffu, abort_flag != 0);
             ++i, ck = (ck + 1 == n_chunks) ? 0 : ck + 1, tile += (ck == 0)) {
            const int s = i % kRing2, vb = i & 1;
            if (!wwait(&t2_full[s], (i / kRing2) & 1, p.err)) { abort_flag = 1; break; }
            if (i >= 2 && !wwait(&pva_empty[vb], ((i >> 1) - 1) & 1, p.err)) { abort_flag = 1; break; }
            if (BITS == 4 && ck == 0 && !wwait(&sc_full[tile & 1], (tile >> 1) & 1, p.err)) { abort_flag = 1; break; }
            const uint8_t *src = sm + Ly::kOffT2 + s * kSlotBytes;
            // this thread's group scales: token rbase + 8 j' (j' = 4 h32 + j), group grp
            const __half *scs = reinterpret_cast<const __half *>(sm + Ly::kOffSc + (tile & 1) * kScBytes) +
                                rbase * ngrp + (ch0 / 128 + ck);
#pragma unroll 1
            for (int h32 = 0; h32 < 2; ++h32) {             // 32 tokens: two 16x256b stores of 16 columns
                // rows of the 4 tokens this thread supplies (16-token step g, 8-token block tb), loads first
                constexpr int kU = BITS == 8 ? 2 : 1;       // 16-byte units of the warp's 32 channels
                uint4 wl[4][kU];
                __half2 s2[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {               // j = 2 g + tb
                    const uint32_t dr = uint32_t(32 * h32 + 8 * j);         // token offset from rbase
                    if (BITS == 8) {
                        wl[j][0] = *reinterpret_cast<const uint4 *>(src + off8a + dr * 128u);
                        wl[j][kU - 1] = *reinterpret_cast<const uint4 *>(src + off8b + dr * 128u);
                    } else {
                        wl[j][0] = *reinterpret_cast<const uint4 *>(src + off4 + dr * 64u);
                        s2[j] = __half2half2(scs[dr * ngrp]);
                    }
                }
                uint32_t o0[8], o1[8];                       // channel blocks 0-1 and 2-3 of the warp
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int g = j >> 1, tb = j & 1;
                    uint32_t x[4];
                    if (BITS == 8) {
                        // channel block cb = bytes 8cb..8cb+7; pair 2cq, 2cq+1 sits in word 2cb + (cq >> 1)
                        const uint32_t wv[8] = {wl[j][0].x, wl[j][0].y, wl[j][0].z, wl[j][0].w,
                                                wl[j][kU - 1].x, wl[j][kU - 1].y, wl[j][kU - 1].z, wl[j][kU - 1].w};
#pragma unroll
                        for (int cb = 0; cb < 4; ++cb) {
                            const uint32_t wsel = (cq >> 1) ? wv[2 * cb + 1] : wv[2 * cb];
                            x[cb] = i8pair_h2(wsel ^ 0x80808080u, k8);
                        }
                    } else {
                        // pair 2cq, 2cq+1 of channel block cb is byte cq of word cb
                        x[0] = i4pair_h2(wl[j][0].x, cq, s2[j]);
                        x[1] = i4pair_h2(wl[j][0].y, cq, s2[j]);
                        x[2] = i4pair_h2(wl[j][0].z, cq, s2[j]);
                        x[3] = i4pair_h2(wl[j][0].w, cq, s2[j]);
                    }
                    // 16x256b registers of step g: (blk 2lh, tb 0), (2lh, tb 1), (2lh+1, tb 0), (2lh+1, tb 1)
                    o0[4 * g + tb] = movm_t(x[0]);
                    o0[4 * g + 2 + tb] = movm_t(x[1]);
                    o1[4 * g + tb] = movm_t(x[2]);
                    o1[4 * g + 2 + tb] = movm_t(x[3]);
                }
                const uint32_t col = kColV + vb * 64 + 32 * th + 16 * h32;
                tmem_st16x256_x2(tmem + (uint32_t(32 * q) << 16) + col, o0);
                tmem_st16x256_x2(tmem + (uint32_t(32 * q + 16) << 16) + col, o1);
            }
            tmem_wait_st();
            fence_before();
            __syncwarp();
            if (lane == 0) {
                arrive_local(&pva_full[vb]);
                arrive_local(&t2_empty[s]);
                if (BITS == 4 && ck == n_chunks - 1) arrive_local(&sc_empty[tile & 1]);
            }
        }
    } else {
        // ---------------- warpgroups 5-6: exchange, online softmax, P ----------------
        // Warpgroup hg takes heads [16 hg, 16 hg + 16); thread = token.  Logits
        // are kept in log2 units.  Each thread accumulates its own sums of p per
        // head over the tiles; the sums over tokens are formed once, at the end.
        // The reference maximum m_ref of a head only moves when a logit exceeds
        // it by more than kRescale2 (one vote per tile); then the tile maximum is
        // reduced through shared memory, and o_lat and the sums are rescaled.  A
        // failed wait marks the warp `bad`; the warpgroup leaves the tile loop
        // together at its next named barrier (bar.red.or), so no warp is left at
        // a barrier the others skip.
        const int quad = warp & 3, hg = (warp - 20) >> 2, t = quad * 32 + lane, wq = quad;
        const int hb = hg * kHalfN, bar_id = 1 + hg;
        const bool grp_live = hb < Np;                      // Np = 16: the second warpgroup has no heads
        const uint32_t trow = tmem + (uint32_t(quad * 32) << 16);
        // exchange buffer: slot j holds the partials of peer rank + 1 + j (mod CL) as
        // [head / 4][token][4] (conflict-free float4 rows); in slot 0, warpgroup hg's half
        // (heads 16 hg ..) is reused as [token][16] for its tile-maximum transposition
        // once its partials are consumed.  This CTA writes into slot CL - 2 - j of peer
        // rank + 1 + j.
        // (peer addresses are formed at each use: one mapa each, no live registers)
        auto peer_of = [&](int j) { return (rank + 1u + uint32_t(j)) % uint32_t(CL); };
        float *xr = reinterpret_cast<float *>(sm + Ly::kOffXch);
        const float *tscale = static_cast<const float *>(c.scales);
        float tsc_next = 0.0f;
        if (BITS == 8 && n_tiles > 0) tsc_next = t_begin + t < t_end ? tscale[row0 + t_begin + t] : 0.0f;
        // P^T position of this token: 64-token block, then the K order of the PV operand
        const int pcol = (t & 48) | kpos16(t & 15);

        // running sums of p per (head, token), kept in shared memory: [head][token]
        float *lt = reinterpret_cast<float *>(sm + Ly::kOffLt) + hb * kTile + t;
#pragma unroll
        for (int h = 0; h < kHalfN; ++h) lt[h * kTile] = 0.0f;
        bool failed = false;
        for (int tile = 0; tile < n_tiles; ++tile) {
            const int sb = tile & 1;
            const int tok = t_begin + tile * kTile + t;
            const bool live = tok < t_end;
            const float tsc = tsc_next;
            if (BITS == 8 && tile + 1 < n_tiles)
                tsc_next = tok + kTile < t_end ? tscale[row0 + tok + kTile] : 0.0f;
            bool bad = __any_sync(0xffffffffu, abort_flag != 0);
            if (!bad) bad = !wwait(&s_full[sb], (tile >> 1) & 1, p.err);
            float s[kHalfN];
            if (!bad) {
                fence_after();
                uint32_t v[16];
                tmem_ld16(trow + kColS + sb * 32 + hb, v);
                tmem_wait_ld();
#pragma unroll
                for (int h = 0; h < kHalfN; ++h) s[h] = __uint_as_float(v[h]);
                fence_before();
                __syncwarp();
                if (lane == 0) arrive_local(&s_empty[sb]);
            } else {
#pragma unroll
                for (int h = 0; h < kHalfN; ++h) s[h] = 0.0f;
            }
            // send the partial scores to every peer: asynchronous stores that
            // count their bytes on the peer's xch_full[hg], whose phase also
            // needs the peer's own expect-tx arrival
            if (t == 0 && !bad) mbar_arrive_expect_tx(&xch_full[hg], (CL - 1) * kTile * kHalfN * 4);
            if (!bad && tile > 0) bad = !wwait_cluster(&xch_empty[hg], (tile - 1) & 1, p.err);
            if (!bad) {
#pragma unroll
                for (int j = 0; j < CL - 1; ++j) {
                    const uint32_t dst = map_peer(smem_addr(sm + Ly::kOffXch + (CL - 2 - j) * kXchSlot), peer_of(j));
                    const uint32_t bar = map_peer(smem_addr(&xch_full[hg]), peer_of(j));
#pragma unroll
                    for (int h = 0; h < kHalfN; h += 4)
                        st_async_v4(dst + (((hb + h) >> 2) * kTile + t) * 16, s[h], s[h + 1], s[h + 2], s[h + 3], bar);
                }
                bad = !wwait_cluster(&xch_full[hg], tile & 1, p.err);
            }
            bool exceed = false;
            if (!bad) {
                // the partials of ranks 0, 1, .., CL - 1 added in rank order: the same sums on every CTA
#pragma unroll
                for (int h = 0; h < kHalfN; h += 4) {
                    float4 tot = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                    for (int q = 0; q < CL; ++q) {
                        float4 o;
                        if (q == int(rank)) {
                            o = make_float4(s[h], s[h + 1], s[h + 2], s[h + 3]);
                        } else {
                            const int slot = (q - int(rank) - 1 + CL) % CL;
                            o = *reinterpret_cast<const float4 *>(xr + slot * (kXchSlot / 4) + (((hb + h) >> 2) * kTile + t) * 4);
                        }
                        if (q == 0) tot = o;
                        else { tot.x += o.x; tot.y += o.y; tot.z += o.z; tot.w += o.w; }
                    }
                    s[h] = tot.x; s[h + 1] = tot.y; s[h + 2] = tot.z; s[h + 3] = tot.w;
                }
                // logits in log2 units; dead tokens and padding heads get -inf
#pragma unroll
                for (int h = 0; h < kHalfN; ++h) {
                    const float lg = s[h] * qfac[hb + h] * (BITS == 8 ? tsc : 1.0f);
                    s[h] = (live && hb + h < H) ? lg : -INFINITY;
                    exceed |= s[h] > m_ref[hb + h] + kRescale2;
                }
            }
            if (group_any(bad, bar_id)) { failed = true; break; }
            if (group_any(exceed, bar_id)) {
                // tile maximum per head: the logits, transposed through the exchange buffer
#pragma unroll
                for (int h = 0; h < kHalfN; ++h) xr[hg * (kTile * kHalfN) + t * kHalfN + (h ^ (lane & 15))] = s[h];
                group_sync(bar_id);
                {
                    // lane: head lane & 15 over tokens (lane >> 4) + 2j of the warp's 32
                    const int hl = lane & 15;
                    float m = -INFINITY;
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const int k = (lane >> 4) + 2 * j;
                        m = fmaxf(m, xr[hg * (kTile * kHalfN) + (wq * 32 + k) * kHalfN + (hl ^ (k & 15))]);
                    }
                    m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 16));
                    if (lane < 16) red_max[hg][wq][lane] = m;
                }
                group_sync(bar_id);
                if (t < kHalfN) {
                    const int h = hb + t;
                    float a = 1.0f;
                    if (h < H) {
                        const float tm = fmaxf(fmaxf(red_max[hg][0][t], red_max[hg][1][t]),
                                               fmaxf(red_max[hg][2][t], red_max[hg][3][t]));
                        const float mr = m_ref[h];
                        if (tm > mr + kRescale2) {
                            a = mr == -INFINITY ? 0.0f : exp2f(mr - tm);
                            m_ref[h] = tm;
                        }
                    }
                    alpha[h] = a;
                }
                group_sync(bar_id);
#pragma unroll
                for (int h = 0; h < kHalfN; ++h) lt[h * kTile] *= alpha[hb + h];
                if (tile > 0 && grp_live) {
                    // the PV MMAs of the previous tile must be complete before o_lat is scaled
                    bad = !wwait(&p_empty[(tile - 1) & 1], ((tile - 1) >> 1) & 1, p.err);
                    if (!bad) {
                        fence_after();
                        for (int c8 = 0; c8 < 2 * n_chunks; ++c8) {     // 8 heads at a time
                            const uint32_t col = trow + kColO + (c8 >> 1) * Np + hb + (c8 & 1) * 8;
                            uint32_t v[8];
                            tmem_ld8(col, v);
                            tmem_wait_ld();
#pragma unroll
                            for (int e = 0; e < 8; ++e) v[e] = __float_as_uint(__uint_as_float(v[e]) * alpha[hb + (c8 & 1) * 8 + e]);
                            tmem_st8(col, v);
                        }
                        tmem_wait_st();
                        fence_before();
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < CL - 1; ++j)      // this thread's reads of the exchange buffer have completed
                arrive_peer_relaxed(map_peer(smem_addr(&xch_empty[hg]), peer_of(j)));
            if (!bad && tile >= 2) bad = !wwait(&p_empty[sb], ((tile >> 1) - 1) & 1, p.err);
            // P^T [heads][tokens], 64-token blocks of Np rows x 128 bytes, swizzled
            uint8_t *pbuf = sm + Ly::kOffP + sb * kPBytes + (t >> 6) * (Np * 128);
            // three passes (loads, then read-modify-writes, then stores only) so that
            // no shared-memory load waits behind a store it might alias
#pragma unroll
            for (int h = 0; h < kHalfN; ++h) s[h] = hb + h < H ? exp2f(s[h] - m_ref[hb + h]) : 0.0f;
#pragma unroll
            for (int h = 0; h < kHalfN; ++h) lt[h * kTile] += s[h];
            if (!bad) {
#pragma unroll
                for (int h = 0; h < kHalfN; ++h) {
                    const int hh = hb + h;
                    if (hh < Np) {
                        const __half hv = __float2half_rn(BITS == 8 ? s[h] * tsc : s[h]);
                        *reinterpret_cast<__half *>(pbuf + hh * 128 + ((((pcol >> 3) ^ (hh & 7))) << 4) + (pcol & 7) * 2) = hv;
                    }
                }
            }
            fence_async_smem();
            if (group_any(bad, bar_id)) { failed = true; break; }
            __syncwarp();
            if (lane == 0) arrive_local(&p_full[sb]);
        }
        if (failed) abort_flag = 1;
        // ---- after the last PV MMA: this CTA's channel slice of o_lat, then (rank 0) m and l
        if (!failed && n_tiles > 0) {
            const int lt_last = n_tiles - 1;
            const bool ok = wwait(&p_empty[lt_last & 1], (lt_last >> 1) & 1, p.err);
            // sums over the tokens, transposed through the exchange buffer (the peer sends no more)
            group_sync(bar_id);
            {
                // lane: head lane & 15 over tokens (lane >> 4) + 2j of the warp's 32
                const float *lrow = reinterpret_cast<const float *>(sm + Ly::kOffLt) + (hb + (lane & 15)) * kTile + wq * 32;
                float sum = 0.0f;
#pragma unroll
                for (int j = 0; j < 16; ++j) sum += lrow[(lane >> 4) + 2 * j];
                sum += __shfl_xor_sync(0xffffffffu, sum, 16);
                if (lane < 16) red_max[hg][wq][lane] = sum;
            }
            group_sync(bar_id);
            if (!group_any(!ok, bar_id)) {
                if (grp_live) {
                    fence_after();
                    const size_t pb = (size_t(b) * p.n_split + split) * p.H;
                    for (int ck = 0; ck < n_chunks; ++ck) {
                        const int ch = ch0 + ck * kChunk + t;
                        uint32_t v[16];
                        tmem_ld16(trow + kColO + ck * Np + hb, v);
                        tmem_wait_ld();
#pragma unroll
                        for (int e = 0; e < 16; ++e)
                            if (hb + e < H) p.po[(pb + hb + e) * r + ch] = __uint_as_float(v[e]);
                    }
                    if (rank == 0 && t < kHalfN && hb + t < H) {
                        p.pm[pb + hb + t] = m_ref[hb + t] * 0.6931471805599453f;       // natural-log units
                        p.pl[pb + hb + t] = (red_max[hg][0][t] + red_max[hg][1][t]) + (red_max[hg][2][t] + red_max[hg][3][t]);
                    }
                }
            } else {
                abort_flag = 1;
            }
        }
    }

    fence_before();
    __syncthreads();
    cluster_sync();                  // the peer has finished every access to this CTA's shared memory
    fence_after();
    if (warp == 1) asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols));
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
namespace {

int g_attn_path = 0;     // 0 automatic, 1 CUDA cores, 2 tcgen05, 3 warp-level MMA

}  // namespace

void set_attn_path(int path) { g_attn_path = path; }
int attn_path() { return g_attn_path; }

// Heads go in launches of at most kMaxN (32); each reads the whole cache.
bool attn_tc_shape_ok(int r, int bits, int H) {
    const int Np = (std::min(H, atc::kMaxN) + 15) / 16 * 16, cl = atc::cluster_for(r);
    if (bits != 8 && bits != 4) return false;
    if (H < 1 || r % (cl * atc::kChunk) || r / cl > atc::kMaxRc || r / 128 > atc::kMaxGroups) return false;
    return (r / cl / atc::kChunk) * Np <= int(atc::kColS - atc::kColO);
}

bool attn_tc_use(const CacheView &c, int H, int max_seq_len) {
    if (g_attn_path == 1 || g_attn_path == 3 || !attn_tc_shape_ok(c.r, c.bits, H) || !tensor_maps_available()) return false;
    if (g_attn_path == 2) return true;
    return int64_t(c.B) * max_seq_len > mma_tokens_max(c.r);
}

int attn_tc_splits(int B, int r, int max_seq_len, int *tiles_per_split) {
    int dev = 0, sms = 148;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int tiles = (max_seq_len + atc::kTile - 1) / atc::kTile;
    const int64_t pairs = sms / atc::cluster_for(r); // clusters resident at once (one CTA per SM)
    // tiles per split: the fewest tile steps of the busiest cluster, counting the
    // fixed cost of a wave (set-up, pipeline fill and drain, partial stores) as
    // 3.5 tile steps, measured on GB300 (~7 us per tile step, ~26 us per wave at
    // B = 16, L = 4096); at most 64 partials per sequence
    int best = tiles;
    int64_t best_cost = INT64_MAX;
    for (int per = 1; per <= tiles; ++per) {
        const int splits = (tiles + per - 1) / per;
        if (splits > 64) continue;
        const int64_t waves = (int64_t(B) * splits + pairs - 1) / pairs;
        const int64_t cost = waves * (2 * per + 7);      // in half tile steps
        if (cost < best_cost) {
            best_cost = cost;
            best = per;
        }
    }
    *tiles_per_split = best;
    return (tiles + best - 1) / best;
}

cudaError_t launch_attn_tc(const CacheView &c, const int32_t *seq_len, const float *qt, const unsigned *qmax, int H,
                           float softmax_scale,
                           int tiles_per_split, int n_split, float *pm, float *pl, float *po, int *err,
                           cudaStream_t s) {
    // the cache as a byte matrix [B * Tmax rows, row_bytes]; a box is 128 rows
    // x one chunk (128 bytes of int8, 128-byte swizzle; 64 bytes of int4, 64-byte swizzle)
    const int row_bytes = c.bits == 8 ? c.r : c.r / 2;
    CUtensorMap map;
    if (!encode_map_2d(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, c.codes, uint64_t(row_bytes),
                       uint64_t(int64_t(c.nseq) * c.Tmax), uint64_t(row_bytes), c.bits == 8 ? 128u : 64u, 128u,
                       c.bits == 8 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B))
        return cudaErrorInvalidValue;
    atc::Params prm{c, seq_len, qt, qmax, H, 0, 0, softmax_scale, tiles_per_split, n_split, pm, pl, po, err};
    const int cl = atc::cluster_for(c.r);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cl * n_split, c.B);
    cfg.blockDim = dim3(atc::kThreads);
    cfg.dynamicSmemBytes = cl == 2 ? atc::Lay<2>::kSmemBytes : atc::Lay<4>::kSmemBytes;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cl;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    auto go = [&](auto kern) {
        cudaError_t e = ensure_smem(kern, cfg.dynamicSmemBytes);
        // one launch per group of at most 32 heads (H = 40: heads 0-31, then 32-39)
        for (int h0 = 0; h0 < H && e == cudaSuccess; h0 += atc::kMaxN) {
            prm.qt = qt + size_t(h0) * c.r;
            prm.qmax = qmax + h0;
            prm.pm = pm + h0;
            prm.pl = pl + h0;
            prm.po = po + size_t(h0) * c.r;
            prm.Hs = std::min(atc::kMaxN, H - h0);
            prm.Np = (prm.Hs + 15) / 16 * 16;
            e = cudaLaunchKernelEx(&cfg, kern, map, prm);
        }
        return e;
    };
    if (c.bits == 8) return cl == 2 ? go(attn_tc_kernel<8, 2>) : go(attn_tc_kernel<8, 4>);
    return cl == 2 ? go(attn_tc_kernel<4, 2>) : go(attn_tc_kernel<4, 4>);
}

}  // namespace qsvd
