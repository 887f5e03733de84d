// Host-side launchers of the QSVD kernels (internal to the library; the
// public surface is include/qsvd.h).  Every launcher only enqueues work on
// `stream` and returns the launch status.
#pragma once

#include <cstddef>
#include <cstdint>
#include <utility>
#include <cuda.h>
#include <cuda_runtime.h>

struct qsvd_cache;   // include/qsvd.h

namespace qsvd {

// 2D tiled TMA descriptor over a row-major matrix of `outer` rows x `inner`
// elements (rows `row_bytes` apart), box = box_outer rows x box_inner
// elements.  Returns false if the driver entry point is missing or refuses
// the parameters.  Defined in api.cu.
bool encode_map_2d(CUtensorMap *map, CUtensorMapDataType type, const void *base, uint64_t inner, uint64_t outer,
                   uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swizzle);
// Whether the driver's tensor-map encoder could be resolved (api.cu).
bool tensor_maps_available();

// Raise a kernel's dynamic shared memory limit to the maximum the first time
// it needs more than the default (so that no attribute call happens while a
// stream is being captured into a graph).  Defined in api.cu.
cudaError_t ensure_smem_ptr(const void *kernel, size_t bytes);
template <typename K>
cudaError_t ensure_smem(K kernel, size_t bytes) {
    return ensure_smem_ptr(reinterpret_cast<const void *>(kernel), bytes);     // static + dynamic may pass 48 KiB
}

// Launch with programmatic stream serialization: the kernel may start while
// the previous kernel in the stream is still running; it must execute
// pdl_wait() before reading anything an earlier stream operation produced.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Bits of the device error word (read and cleared by qsvd_check).
enum : int { kErrRange = 1, kErrTimeout = 2 };

// Device address of the error word for the current device (nullptr if the
// device is unusable), and the thread's last-error message setter.
int *error_word_for_current_device();
int set_last_error(int code, const char *msg);

// Entry-point prologue shared by every C ABI call (api.cu): checks once per
// device that it is an sm_103 part and gives its error word; returns a QSVD_*
// status (the message is set on failure).
int setup_current_device(int **err);
// Checks a caller's cache description (pointers non-null and 16-byte aligned,
// bits 8 or 4, positive sizes, r % 16 == 0, int4 with r % 128 == 0).
int validate_cache(const ::qsvd_cache *c);

// Plain description of a latent cache (mirrors qsvd_cache), seen as B rows
// of queries.  Without a sequence map, row b is sequence b of the cache
// (decode: one query per sequence).  With one, row b reads cache sequence
// seq_map[b] of the nseq the cache holds, so several rows can query the same
// sequence at different lengths (causal prefill).
struct CacheView {
    void *codes;
    void *scales;
    int bits;
    int B;
    int Tmax;
    int r;
    const int32_t *seq_map;   // [B] device, nullable; an input no kernel writes
    int nseq;                 // sequences held by the cache
};

#ifdef __CUDACC__
// Cache sequence behind query row b, or -1 when the map points outside the
// cache (the row is then treated like one with an invalid length).
__device__ __forceinline__ int view_seq(const CacheView &c, int b) {
    if (!c.seq_map) return b;
    const int q = c.seq_map[b];
    return q >= 0 && q < c.nseq ? q : -1;
}

// Length of query row b for the merge kernels: 0 (no partials) when its map
// entry points outside the cache.
__device__ __forceinline__ int row_len(const int32_t *seq_len, const int32_t *seq_map, int nseq, int b) {
    if (seq_map) {
        const int q = seq_map[b];
        if (q < 0 || q >= nseq) return 0;
    }
    return seq_len[b];
}
#endif

// Profiling marker: when the calling thread has enabled profiling
// (qsvd_profile_events), records the next caller-provided event on `s` and
// remembers `label`; otherwise does nothing.  Every launcher calls it right
// after each kernel launch, and each entry point once before its first one.
void prof_mark(cudaStream_t s, const char *label);

// Per-token int8 quantization of X [T, d] bf16 (a1); rot > 0: of X H1^T,
// H1 the block Hadamard rotation with blocks of rot channels (quant_kernels.cu).
// qmax 127 (int8) or 7 (int4 codes, W4A4 / W8A4); xq_f8: optional fp8 e4m3 image of the codes.
cudaError_t launch_xquant(const uint16_t *X, int64_t T, int d, float clip,
                          int8_t *xq, uint16_t *xq_bf16, float *xs, cudaStream_t s, int rot = 0, int qmax = 127,
                          uint8_t *xq_f8 = nullptr);

// Per-output-channel int8 RTN of W_d [d, r] fp32 -> codes [r, d] (+ bf16 image);
// rot > 0: of H1 W_d.
// qmax 127 (int8) or 7 (int4-valued codes); codes_f8: optional fp8 e4m3 image.
cudaError_t launch_quantize_weight(const float *W, int d, int r, float clip, int8_t *codes,
                                   uint16_t *codes_bf16, float *scale, cudaStream_t s, int rot = 0, int qmax = 127,
                                   uint8_t *codes_f8 = nullptr);

// Per-output-channel RTN of an up-projection U [r, d] bf16 (Eq. 11's Q(W^u)):
// int8 codes [r, d] or packed int4 [r, d/2], fp32 scale [d]; d % 32 == 0.
cudaError_t launch_quantize_up(const uint16_t *U, int r, int d, int bits, float clip, void *codes, float *scale,
                               cudaStream_t s);

// Exact int8 GEMM on the CUDA cores (dp4a) with the dequant epilogue (a2, a3 first half):
// c_hat[t, j] = (fp32(acc) * xs[t]) * ws[j].
cudaError_t launch_proj_dp4a(const int8_t *xq, int64_t T, int d, const int8_t *wcodes,
                             const float *ws, const float *xs, int r, float *c_hat,
                             int32_t *acc_out, cudaStream_t s);

// Decode-size projection: with `tail`, a1, a2, a3 and a4 in one launch for
// T < 4 (the last CTA requantizes; `counter` must be zero before the first
// call, the kernel leaves it at zero); without it, the latent rows go to
// requant_kernel.  X is quantized by the kernel itself, or taken as codes from
// xquant (xq_in, xs_in) for up to kPsMaxSplitTok tokens; kPsMaxTok tokens per
// CTA row.
constexpr int kPsMaxTok = 16;
constexpr int kPsMaxSplitTok = 64;
cudaError_t launch_proj_small(const uint16_t *X, int T, int d, float act_clip, const int8_t *wcodes,
                              const float *ws, int r, int lat_bits, float lat_clip, float *c_hat, int *counter,
                              int8_t *xq_out, float *xs_out, int32_t *acc_out, void *lat_codes, void *lat_scales,
                              const CacheView *dst, const int32_t *dst_seq, const int32_t *dst_pos, int *err,
                              cudaStream_t s, const int8_t *xq_in = nullptr, const float *xs_in = nullptr,
                              bool tail = true, int act_qmax = 127);
// From this many tokens on, the decode projection runs as three kernels:
// xquant (one CTA per token), proj_small on the given codes, requant (one CTA
// per row); below it (one token), proj_small quantizes the row itself and
// requant_kernel follows.  Measured on GB300 (whole decode steps): at one token
// this is 1.3 us faster than xquant first and 1.8 us faster than the last CTA
// of proj_small requantizing; from two tokens on, xquant first is fastest.
constexpr int kPsSplitTok = 2;

// Exact int8 GEMM on the tensor cores (bf16 images of the codes, fp32 TMEM
// accumulators drained to int32 every 1024 of K) + the fp32 dequantization.
bool gemm_tc_supported(int d, int r);
// splits > 1 (with part: [splits, T, r] int32 scratch): each CTA sums its
// slice of K; split_requant adds the slices, dequantizes and requantizes.
cudaError_t launch_gemm_tc(const uint16_t *xq_bf16, int64_t T, int d, const uint16_t *w_bf16, const float *ws,
                           const float *xs, int r, float *c_hat, int32_t *acc_out, int *err, cudaStream_t s,
                           int splits = 1, int32_t *part = nullptr);
// K splits for a separate-epilogue projection of T tokens (1: none).  Splits
// are taken only while the tiles fill less than half the GPU, which needs
// T * r <= kSplitMaxElems (80 tiles of 128 x 128 at most); the projection
// workspace holds kMaxSplitK int32 partial latents up to that size.
constexpr int kMaxSplitK = 4;
constexpr int64_t kSplitMaxElems = int64_t(80) * 128 * 128;
int gemm_tc_splits(int64_t T, int d, int r);
// a2 + a3 after a split-K GEMM: per token row, the sum of the splits' int32
// partials (written to acc_out if given), c_hat = (fp32(acc) s_x) s_w, and the
// requantization and store of requant.
cudaError_t launch_split_requant(const int32_t *part, int splits, int64_t T, int r, const float *xs, const float *ws,
                                 int32_t *acc_out, int bits, float clip, void *lat_codes, void *lat_scales,
                                 const CacheView *dst, const int32_t *dst_seq, const int32_t *dst_pos, int *err,
                                 cudaStream_t s);

// W4A4: the GEMM on fp8 e4m3 images of int4-valued codes (kind::f8f6f4),
// with the requantization epilogue for lat_bits 8 / 4 (0: c_hat only).
bool gemm_f8_supported(int d, int r);
cudaError_t launch_gemm_f8(const uint8_t *xq_f8, int64_t T, int d, const uint8_t *w_f8, const float *ws,
                           const float *xs, int r, int lat_bits, float lat_clip, void *lat_codes, void *lat_scales,
                           const CacheView *dst, const int32_t *dst_seq, const int32_t *dst_pos, float *c_hat,
                           int32_t *acc_out, int *err, cudaStream_t s);

// The same GEMM with the per-token requantization and store of the latent
// (a3 second half + a4) in its epilogue; c_hat and acc_out are optional
// debug outputs (null: not written).
bool gemm_tc_fused_supported(int64_t T, int r, int lat_bits);
void set_project_epilogue(int mode);     // 0 automatic, 1 separate requantization, 2 fused where possible
int project_epilogue();
cudaError_t launch_gemm_tc_fused(const uint16_t *xq_bf16, int64_t T, int d, const uint16_t *w_bf16, const float *ws,
                                 const float *xs, int r, int lat_bits, float lat_clip, void *lat_codes,
                                 void *lat_scales, const CacheView *dst, const int32_t *dst_seq,
                                 const int32_t *dst_pos, float *c_hat, int32_t *acc_out, int *err, cudaStream_t s);

// Per-token requantization of c_hat [T, r] into the latent format (a3 second
// half), written token-major and/or into the cache (a4).
cudaError_t launch_requant(const float *c_hat, int64_t T, int r, int bits, float clip,
                           void *lat_codes, void *lat_scales, const CacheView *dst,
                           const int32_t *dst_seq, const int32_t *dst_pos, int *err,
                           cudaStream_t s);
// The same for the B rows of a decode step: row b goes to position
// seq_len[b] - 1 of the cache sequence behind b.
cudaError_t launch_requant_len(const float *c_hat, int B, int r, int bits, float clip, const CacheView &dst,
                               const int32_t *seq_len, int *err, cudaStream_t s);

// Copy token-major latent rows into the cache (a4).
cudaError_t launch_append(const CacheView &c, const int32_t *seq, const int32_t *pos, int64_t n,
                          const void *lat_codes, const void *lat_scales, int *err,
                          cudaStream_t s);

// An up-projection [r, d] as the decode kernels read it: bf16 values (bits
// 16, scale null), or Eq. 11's Q(W^u): int8 codes [r, d] (bits 8) or packed
// int4 codes [r, d/2] (bits 4) with one fp32 scale per output channel [d].
struct UpW {
    const void *w;
    const float *scale;
    int bits;
};

// Decode attention (a5-a8).
struct DecodeArgs {
    CacheView cache;
    const int32_t *seq_len;
    int max_seq_len;
    UpW U_q, U_k, U_v;
    int H, dh;
    float softmax_scale;
    float *O;
    // nullable: the step's new latents (fp32 [B, r]), requantized with lat_clip
    // and stored at position seq_len[b] - 1 before the attention reads the cache
    const float *c_hat;
    float lat_clip;
};
size_t decode_workspace_bytes(int B, int max_seq_len, int r, int H, int dh);

// Eq. 10 importance scores (prep_importance.cu); part: [N, ceil(m / 64), k] fp32 scratch.
constexpr int kImpRowTile = 64;
cudaError_t launch_importance(const float *U, const float *sigma, const float *Vt, const float *G, int N, int m, int n,
                              int k, float *scores, float *part, int *err, cudaStream_t s);
// Cross-layer rank budget: keep[i] = 1 for the k highest scores (ties: lower i).
size_t rank_workspace_bytes();
cudaError_t launch_rank_budget(const float *scores, int n, int k, uint8_t *keep, void *ws, cudaStream_t s);

// Causal prefill over the cache (qsvd_latent_prefill_attn) runs the decode
// chain on groups of query rows: at most kPrefillMaxRows rows per group, fewer
// while a group's workspace would exceed kPrefillWsTarget bytes.
// Materialised causal prefill (prefill_tc.cu): at most kPrefillMaxBlocks
// prompt blocks per launch.  Block k covers positions t0[k] .. L[k]-1 of cache
// sequence seq[k] as queries and 0 .. L[k]-1 as keys; its latent rows start
// at row row_off[k] (a multiple of 128) of the workspace matrices, its
// outputs at row out_off[k] of O, and its query tiles at qtile_off[k].
constexpr int kPrefillMaxBlocks = 64;
struct PrefillBlocks {
    int n;
    int seq[kPrefillMaxBlocks], t0[kPrefillMaxBlocks], L[kPrefillMaxBlocks];
    int row_off[kPrefillMaxBlocks], out_off[kPrefillMaxBlocks];
    int qtile_off[kPrefillMaxBlocks + 1];
};
size_t prefill_mat_rows(const PrefillBlocks &bl);
size_t prefill_mat_workspace_bytes(size_t R, int r, int d);
cudaError_t launch_prefill_weights(const uint16_t *Uq, const uint16_t *Uk, const uint16_t *Uv, int r, int d,
                                   uint16_t *Ut, int *err, cudaStream_t s);
cudaError_t launch_prefill_mat(const CacheView &c, const PrefillBlocks &bl, const uint16_t *Ut, int H,
                               float softmax_scale, float *O, void *ws, int *err, cudaStream_t s);

constexpr int kPrefillMaxRows = 1024;
constexpr size_t kPrefillWsTarget = size_t(2) << 30;

// a5 and a7/a8 for all B sequences of a step (decode_gemv.cu).
// decode_mma.cu: tensor-core forms of the three products, for 8 or more sequences
bool decode_mma_supported(int B, int r, int d, int dh);
cudaError_t launch_qproj_mma(const CacheView &c, const int32_t *seq_len, const uint16_t *Uq, int d, float *q,
                             unsigned *qmax, int n_qmax, int *err, cudaStream_t s);
cudaError_t launch_qabsorb_mma(const float *q, const uint16_t *Uk, int B, int r, int d, int H, int dh, float *qt,
                               unsigned *qmax, cudaStream_t s);
cudaError_t launch_combine_mma(const int32_t *seq_len, const int32_t *seq_map, int nseq, int B, int Tmax, int H, int dh, int r, int chunk, int n_split,
                               const float *pm, const float *pl, const float *po, const uint16_t *Uv, float *O,
                               cudaStream_t s);
// The CUDA-core forms (decode_gemv.cu); they read every weight format.
// c_hat (nullable): the step's new latents, fp32 [B, r] as the projection left
// them; qproj then requantizes them itself and stores them at position
// seq_len[b] - 1 (a3/a4), for up to kFreshMaxB sequences with bf16 U_q.
constexpr int kFreshMaxB = 4;
bool qproj_fresh_supported(const CacheView &c, const UpW &Uq);
cudaError_t launch_qproj(const CacheView &c, const int32_t *seq_len, const UpW &Uq, int d, float *q,
                         unsigned *qmax, int n_qmax, int *err, cudaStream_t s, const float *c_hat = nullptr,
                         float lat_clip = 1.0f);
cudaError_t launch_qabsorb(const float *q, const UpW &Uk, int B, int r, int d, int H, int dh, float *qt,
                           unsigned *qmax, int *err, cudaStream_t s);
cudaError_t launch_combine_uv(const int32_t *seq_len, const int32_t *seq_map, int nseq, int B, int Tmax, int H, int dh,
                              int r, int chunk, int n_split, const float *pm, const float *pl, const float *po,
                              const UpW &Uv, float *O, int *err, cudaStream_t s);

// a5 in one launch for up to four sequences (decode_qfuse.cu): q and q~ per
// head in a cluster, q_h exchanged in distributed shared memory; used when
// U_q and U_k share a format and the whole grid is resident at once.
bool qfuse_use(const CacheView &c, const UpW &Uq, const UpW &Uk, int H, int dh);
cudaError_t launch_qfuse(const CacheView &c, const int32_t *seq_len, const UpW &Uq, const UpW &Uk, int H, int dh,
                         float *qt, unsigned *qmax, int *err, cudaStream_t s);

// Tensor-core latent attention (a6/a7): choice of kernel, split of each
// sequence into partials (tiles of 128 tokens), and the launcher, which writes
// the same (m, l, o_lat) partials as the CUDA-core kernel.
void set_attn_path(int path);      // 0 automatic, 1 CUDA cores, 2 tcgen05 where the shape allows, 3 warp MMA
int attn_path();
bool attn_tc_shape_ok(int r, int bits, int H);
bool attn_tc_use(const CacheView &c, int H, int max_seq_len);
int attn_tc_splits(int B, int r, int max_seq_len, int *tiles_per_split);
// Warp-level tensor-core attention for small batch x length (attn_mma.cu).
// The automatic choice takes it while B x L (cached tokens of the step) is at
// most mma_tokens_max(r), and the tcgen05 kernel above that: the crossover
// measured on GB300 over B = 1..16, L = 512..4096, r = 1024..3072, int8 and
// int4 (whole decode steps; the tcgen05 kernel is up to 2.7x faster above it,
// the warp-level one up to 1.4x faster below it).
constexpr int64_t mma_tokens_max(int r) { return r <= 2048 ? 2048 : 1024; }
bool attn_mma_use(const CacheView &c, int H, int B, int max_seq_len);
bool attn_mma_fits(const CacheView &c, int max_seq_len);
int attn_mma_splits(const CacheView &c, int B, int H, int max_seq_len, int *ts, int *n_sub);
cudaError_t launch_attn_mma(const CacheView &c, const int32_t *seq_len, const float *qt, const unsigned *qmax, int H,
                            float softmax_scale, int ts, int n_sub, int n_split, float *pm, float *pl, float *po,
                            int *err, cudaStream_t s);
cudaError_t launch_attn_tc(const CacheView &c, const int32_t *seq_len, const float *qt, const unsigned *qmax, int H,
                           float softmax_scale,
                           int tiles_per_split, int n_split, float *pm, float *pl, float *po, int *err,
                           cudaStream_t s);

cudaError_t launch_decode(const DecodeArgs &a, void *ws, size_t ws_bytes, int *err,
                          cudaStream_t s);

// Failure-detection self-test: a bounded wait on a barrier nothing completes.
cudaError_t launch_selftest_wait(unsigned long long limit_ns, int *err, cudaStream_t s);

}  // namespace qsvd
