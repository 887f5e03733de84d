// Both query-side products of a decode step (a5, Eq. 5 with W^u_k absorbed
// into the query) in one launch, for batches of up to four sequences with
// quantized up-projections (Eq. 11):
//
//   q[b, h-block]  = c_{L_b - 1} U_q[:, h-block]
//   q~[b, h, j]    = U_k[j, h-block] . q[b, h-block]        (j = 0 .. r-1)
//   qmax[b, h]     = max_j |q~[b, h, j]|
//
// A cluster of kClF CTAs serves one head: CTA k holds rows [k rs, (k+1) rs)
// (rs = r / kClF) of both U_q[:, h-block] and U_k[:, h-block] in shared
// memory, copied before the wait on the producer grid (the weights are no
// kernel's output).  After the wait each CTA multiplies its slice of the
// dequantized latent row by its U_q rows, the kClF partial products of q_h
// are exchanged through distributed shared memory and added in rank order
// (every CTA then holds the identical q_h), and each CTA forms q~ for its own
// rows of U_k.  The per-head maximum of |q~| is reduced across the cluster
// the same way.  Compared with two launches (qproj_kernel, qabsorb_kernel)
// this saves one kernel hand-over and the round trip of q through global
// memory, which is what a batch-1 step waits on.
//
// Weights in any of the decode formats (WB = 16 bf16, 8 int8, 4 int4 codes
// with per-output-channel scales); U_q and U_k in the same format.
#include "common.cuh"
#include "launch.h"

namespace qsvd {

namespace {

constexpr int kClF = 8;          // CTAs per head (cluster_ld8 reads 8 ranks)
constexpr int kQfThreads = 256;
constexpr int kQfMaxNB = 4;      // sequences per launch

__device__ __forceinline__ uint32_t qf_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void qf_cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void qf_cp16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}

// Decode weight formats (the same exact conversions as decode_gemv.cu).
__device__ __forceinline__ float qf_i8(uint32_t u, int k) {        // u = word ^ 0x80808080
    return __uint_as_float(__byte_perm(u, 0x4B000000u, uint32_t(k) | (4u << 4) | (5u << 8) | (7u << 12))) -
           8388736.0f;
}
__device__ __forceinline__ float qf_i4(uint32_t x, int k) {        // x = word ^ 0x88888888
    return __uint_as_float(((x >> (4 * k)) & 0xFu) | 0x4B000000u) - 8388616.0f;
}
template <int WB>
__device__ __forceinline__ void qf_w4(const uint8_t *row, int q4, float (&u)[4]) {
    if (WB == 16) {
        const uint2 w2 = *reinterpret_cast<const uint2 *>(row + 8 * q4);
        u[0] = bf16_lo(w2.x); u[1] = bf16_hi(w2.x); u[2] = bf16_lo(w2.y); u[3] = bf16_hi(w2.y);
    } else if (WB == 8) {
        const uint32_t x = *reinterpret_cast<const uint32_t *>(row + 4 * q4) ^ 0x80808080u;
#pragma unroll
        for (int e = 0; e < 4; ++e) u[e] = qf_i8(x, e);
    } else {
        const uint32_t x = uint32_t(*reinterpret_cast<const uint16_t *>(row + 2 * q4)) ^ 0x8888u;
#pragma unroll
        for (int e = 0; e < 4; ++e) u[e] = qf_i4(x, e);
    }
}
template <int WB>
__device__ __forceinline__ void qf_w16B(const uint4 &v, float (&f)[128 / WB]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        if (WB == 16) {
            f[2 * k] = bf16_lo(w[k]);
            f[2 * k + 1] = bf16_hi(w[k]);
        } else if (WB == 8) {
            const uint32_t x = w[k] ^ 0x80808080u;
#pragma unroll
            for (int e = 0; e < 4; ++e) f[4 * k + e] = qf_i8(x, e);
        } else {
            const uint32_t x = w[k] ^ 0x88888888u;
#pragma unroll
            for (int e = 0; e < 8; ++e) f[8 * k + e] = qf_i4(x, e);
        }
    }
}

// Shared-memory layout.  KRES: both weight tiles are copied before the wait;
// otherwise (bf16 tiles too large to leave room for the neighbouring kernels'
// CTAs) U_k is only prefetched into L2 before the wait and copied into the
// U_q buffer once the q product has read it.
struct QfLayout {
    int rs, rbq, rbk, G;
    size_t off_uk, off_c, off_part, off_qh, bytes;
};
constexpr size_t kQfResidentTiles = 64 * 1024;   // both tiles resident up to this size
__host__ __device__ inline bool qf_kres(int r, int dh, int WB) {
    return size_t(r / kClF) * (2 * (dh * WB / 8) + 16) <= kQfResidentTiles;
}
__host__ __device__ inline QfLayout qf_layout(int r, int dh, int NB, int WB, bool kres) {
    QfLayout l;
    l.rs = r / kClF;
    l.rbq = dh * WB / 8;                 // U_q tile row bytes
    l.rbk = dh * WB / 8 + 16;            // U_k tile row bytes, padded (conflict-free 16-byte row reads)
    l.G = kQfThreads / (dh / 4);         // row groups of the q product
    l.off_uk = kres ? size_t(l.rs) * l.rbq : 0;
    l.off_c = l.off_uk + size_t(l.rs) * l.rbk;
    l.off_part = l.off_c + size_t(NB) * l.rs * 4;
    l.off_qh = l.off_part + size_t(l.G) * NB * dh * 4;
    l.bytes = l.off_qh + size_t(NB) * dh * 4;
    return l;
}

}  // namespace

// Grid (kClF, H), cluster (kClF, 1, 1), 256 threads; B <= NB.
template <int NB, int WB, bool KRES>
__global__ void __cluster_dims__(kClF, 1, 1) __launch_bounds__(kQfThreads)
qfuse_kernel(const uint8_t *__restrict__ Uq, const float *__restrict__ sq, const uint8_t *__restrict__ Uk,
             const float *__restrict__ sk, CacheView c, const int32_t *__restrict__ seq_len, int B, int H, int dh,
             float *__restrict__ qt, unsigned *__restrict__ qmax, int *err) {
    // qmax == nullptr: the consumer (the warp-level attention kernel) forms the
    // per-head maxima from the q~ it loads, and no maximum is exchanged here
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int L_s[NB], Q_s[NB];
    __shared__ float red_s[kQfThreads / 32][NB];
    __shared__ float mx_s[NB];
    const int r = c.r, d = H * dh, h = blockIdx.y;
    const QfLayout ly = qf_layout(r, dh, NB, WB, KRES);
    const int rs = ly.rs, rbq = ly.rbq, rbk = ly.rbk, G = ly.G;
    const uint32_t rank = qf_rank();
    const int j0 = int(rank) * rs;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    uint8_t *uq_s = smem;
    uint8_t *uk_s = smem + ly.off_uk;
    float *c_s = reinterpret_cast<float *>(smem + ly.off_c);        // [NB][rs]
    float *part = reinterpret_cast<float *>(smem + ly.off_part);    // [G][NB][dh]
    float *qh_s = reinterpret_cast<float *>(smem + ly.off_qh);      // [NB][dh]

    // the U_q tile, then the U_k tile (or its L2 prefetch): two commit groups, U_q needed first
    const uint8_t *uk_src = Uk + (size_t(j0) * d + size_t(h) * dh) * WB / 8;
    auto copy_uk = [&]() {
        for (int i = tid; i < rs * (rbq / 16); i += kQfThreads) {
            const int row = i / (rbq / 16), k = i - row * (rbq / 16);
            qf_cp16(uk_s + size_t(row) * rbk + 16 * k, uk_src + size_t(row) * d * WB / 8 + 16 * k);
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    };
    for (int i = tid; i < rs * (rbq / 16); i += kQfThreads) {
        const int row = i / (rbq / 16), k = i - row * (rbq / 16);
        qf_cp16(uq_s + size_t(row) * rbq + 16 * k, Uq + (size_t(j0 + row) * d + size_t(h) * dh) * WB / 8 + 16 * k);
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
    if (KRES) {
        copy_uk();
    } else {
        for (int row = tid; row < rs; row += kQfThreads) prefetch_l2_bulk(uk_src + size_t(row) * d * WB / 8, uint32_t(rbq));
        asm volatile("cp.async.commit_group;" ::: "memory");       // an empty group keeps the counts alike
    }
    pdl_wait();
    pdl_trigger();   // after the wait: the attention kernel reads the call's lengths before its own wait

    const int nb = B;
    if (tid < NB) {
        int L = tid < nb ? seq_len[tid] : 0;
        const int sq_ = tid < nb ? view_seq(c, tid) : 0;
        if (tid < nb && (sq_ < 0 || L < 1 || L > c.Tmax)) {
            if (rank == 0 && h == 0) flag_error(err, kErrRange);
            L = 0;
        }
        L_s[tid] = L;
        Q_s[tid] = sq_;
    }
    __syncthreads();
    // dequantized latent rows c_{L-1}, this CTA's channels
    for (int i = tid; i < NB * rs; i += kQfThreads) {
        const int bi = i / rs, x = i - bi * rs;
        float v = 0.0f;
        const int L = bi < nb ? L_s[bi] : 0;
        if (L > 0) {
            const size_t slot = size_t(Q_s[bi]) * c.Tmax + (L - 1);
            const int ch = j0 + x;
            if (c.bits == 8) {
                v = float(static_cast<const int8_t *>(c.codes)[slot * r + ch]) * static_cast<const float *>(c.scales)[slot];
            } else {
                const uint8_t byte = static_cast<const uint8_t *>(c.codes)[slot * (r / 2) + (ch >> 1)];
                const int nib = (((ch & 1) ? (byte >> 4) : byte) & 0xF) ^ 8;
                v = float(nib - 8) * __half2float(static_cast<const __half *>(c.scales)[slot * (r / 128) + (ch >> 7)]);
            }
        }
        c_s[i] = v;
    }
    asm volatile("cp.async.wait_group 1;" ::: "memory");
    __syncthreads();

    // partial q over this CTA's rows: thread = (column quad cq, row group g), rows g, g + G, ...
    {
        const int cq = tid % (dh / 4), g = tid / (dh / 4);
        float acc[NB][4];
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) acc[bi][0] = acc[bi][1] = acc[bi][2] = acc[bi][3] = 0.0f;
        for (int i = g; i < rs; i += G) {
            float u[4];
            qf_w4<WB>(uq_s + size_t(i) * rbq, cq, u);
#pragma unroll
            for (int bi = 0; bi < NB; ++bi) {
                const float cv = c_s[bi * rs + i];
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[bi][e] = fmaf(cv, u[e], acc[bi][e]);
            }
        }
#pragma unroll
        for (int bi = 0; bi < NB; ++bi)
            *reinterpret_cast<float4 *>(part + (size_t(g) * NB + bi) * dh + 4 * cq) =
                make_float4(acc[bi][0], acc[bi][1], acc[bi][2], acc[bi][3]);
    }
    __syncthreads();
    if (!KRES) copy_uk();               // U_q has been read: its buffer takes U_k (from L2)
    for (int o = tid; o < NB * dh; o += kQfThreads) {          // row groups in order
        float v = part[o];
        for (int k = 1; k < G; ++k) v += part[size_t(k) * NB * dh + o];
        part[o] = v;
    }
    qf_cluster_sync();                                          // every rank's partial q_h is complete
    for (int o = tid; o < NB * dh; o += kQfThreads) {
        const int col = o % dh;
        float pk[kClF];
        cluster_ld8(part + o, pk);
        float v = 0.0f;
#pragma unroll
        for (int k = 0; k < kClF; ++k) v += pk[k];              // rank order
        if (WB != 16) v = (v * sq[size_t(h) * dh + col]) * sk[size_t(h) * dh + col];   // Q(U_q), Q(U_k) scales
        qh_s[o] = v;
    }
    cluster_arrive();                   // this CTA's reads of the peers' partials are done
    asm volatile("cp.async.wait_group 0;" ::: "memory");
    __syncthreads();

    // q~ for this CTA's rows of U_k: thread = row
    float lmax[NB];
#pragma unroll
    for (int bi = 0; bi < NB; ++bi) lmax[bi] = 0.0f;
    constexpr int kStep = 128 / WB;
    for (int j = tid; j < rs; j += kQfThreads) {
        float acc[NB];
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) acc[bi] = 0.0f;
        const uint8_t *urow = uk_s + size_t(j) * rbk;
        for (int i = 0; i < dh; i += kStep) {
            float f[kStep];
            qf_w16B<WB>(*reinterpret_cast<const uint4 *>(urow + i * WB / 8), f);
#pragma unroll
            for (int bi = 0; bi < NB; ++bi) {
                float a = acc[bi];
#pragma unroll
                for (int e = 0; e < kStep; e += 4) {
                    const float4 qv = *reinterpret_cast<const float4 *>(qh_s + bi * dh + i + e);
                    a = fmaf(f[e], qv.x, a); a = fmaf(f[e + 1], qv.y, a);
                    a = fmaf(f[e + 2], qv.z, a); a = fmaf(f[e + 3], qv.w, a);
                }
                acc[bi] = a;
            }
        }
#pragma unroll
        for (int bi = 0; bi < NB; ++bi) {
            if (bi < nb) qt[(size_t(bi) * H + h) * r + j0 + j] = acc[bi];
            lmax[bi] = fmaxf(lmax[bi], fabsf(acc[bi]));
        }
    }
    cluster_wait();                     // ... and so are the peers' reads of this CTA's
    if (!qmax) return;
#pragma unroll
    for (int bi = 0; bi < NB; ++bi) {
        const float m = warp_max(lmax[bi]);
        if (lane == 0) red_s[warp][bi] = m;
    }
    __syncthreads();
    if (tid < NB) {
        float m = 0.0f;
        for (int w = 0; w < kQfThreads / 32; ++w) m = fmaxf(m, red_s[w][tid]);
        mx_s[tid] = m;
    }
    qf_cluster_sync();                                          // every rank's maximum is in place
    if (rank == 0 && tid < nb) {
        float mk[kClF];
        cluster_ld8(mx_s + tid, mk);
        float m = 0.0f;
#pragma unroll
        for (int k = 0; k < kClF; ++k) m = fmaxf(m, mk[k]);
        qmax[size_t(tid) * H + h] = __float_as_uint(m);
    }
    qf_cluster_sync();                                          // peers' reads done before any CTA exits
}

namespace {

template <int NB, int WB, bool KRES>
cudaError_t qfuse_go(const UpW &Uq, const UpW &Uk, const CacheView &c, const int32_t *seq_len, int H, int dh,
                     float *qt, unsigned *qmax, int *err, cudaStream_t s) {
    const QfLayout ly = qf_layout(c.r, dh, NB, WB, KRES);
    cudaError_t e = ensure_smem(qfuse_kernel<NB, WB, KRES>, ly.bytes);
    if (e != cudaSuccess) return e;
    return launch_pdl(qfuse_kernel<NB, WB, KRES>, dim3(kClF, H), dim3(kQfThreads), ly.bytes, s,
                      static_cast<const uint8_t *>(Uq.w), Uq.scale, static_cast<const uint8_t *>(Uk.w), Uk.scale, c,
                      seq_len, c.B, H, dh, qt, qmax, err);
}
template <int NB, int WB>
cudaError_t qfuse_nb(const UpW &Uq, const UpW &Uk, const CacheView &c, const int32_t *seq_len, int H, int dh,
                     float *qt, unsigned *qmax, int *err, cudaStream_t s) {
    return qf_kres(c.r, dh, WB) ? qfuse_go<NB, WB, true>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s)
                                : qfuse_go<NB, WB, false>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s);
}

int qf_nb(int B) { return B <= 1 ? 1 : (B <= 2 ? 2 : 4); }

}  // namespace

bool qfuse_use(const CacheView &c, const UpW &Uq, const UpW &Uk, int H, int dh) {
    // measured at B = 1 (r = 1536, d = 4096): with int8 weights the fused launch saves ~0.8 us a step;
    // with bf16 weights the two kernels (qproj, qabsorb) are ~1.5 us faster, so they are kept there
    if (c.B > kQfMaxNB || Uq.bits != Uk.bits || Uq.bits == 16) return false;
    if (c.r % (kClF * 4) || (dh != 64 && dh != 128)) return false;
    // every CTA of the grid resident at once: at least two per SM, kClF * H CTAs
    const QfLayout ly = qf_layout(c.r, dh, qf_nb(c.B), Uq.bits, qf_kres(c.r, dh, Uq.bits));
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) !=
                                                      cudaSuccess)
            return false;
    }
    const size_t per_sm = 227 * 1024;
    const int fit = int(per_sm / (ly.bytes + 2048));
    return fit >= 2 && size_t(fit) * sms >= size_t(kClF) * H;
}

cudaError_t launch_qfuse(const CacheView &c, const int32_t *seq_len, const UpW &Uq, const UpW &Uk, int H, int dh,
                         float *qt, unsigned *qmax, int *err, cudaStream_t s) {
    cudaError_t e;
    const int nb = qf_nb(c.B);
    switch (Uq.bits) {
        case 16:
            e = nb == 1 ? qfuse_nb<1, 16>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s)
                : nb == 2 ? qfuse_nb<2, 16>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s)
                          : qfuse_nb<4, 16>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s);
            break;
        case 8:
            e = nb == 1 ? qfuse_nb<1, 8>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s)
                : nb == 2 ? qfuse_nb<2, 8>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s)
                          : qfuse_nb<4, 8>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s);
            break;
        default:
            e = nb == 1 ? qfuse_nb<1, 4>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s)
                : nb == 2 ? qfuse_nb<2, 4>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s)
                          : qfuse_nb<4, 4>(Uq, Uk, c, seq_len, H, dh, qt, qmax, err, s);
            break;
    }
    prof_mark(s, "qfuse");
    return e;
}

}  // namespace qsvd
