/*
 * qsvd.h -- C ABI of the QSVD latent-attention hot path on GB300 (sm_103a).
 *
 * QSVD (arxiv 2510.16292) factors the concatenated query/key/value weight
 * [W_q, W_k, W_v] of an attention layer into one shared down-projection W_d
 * (E x r) and three up-projections U_q, U_k, U_v (r x E each) (Sec. 3.1,
 * Eq. 2-4).  Only the latent C = X W_d of each token is cached; keys and
 * values are recomputed from it as K = C U_k, V = C U_v (Eq. 5).  With
 * quantization, C is computed from int8 X and int8 W_d and is itself stored
 * in low precision (Eq. 11-12).
 *
 * This library implements, on the caller's CUDA stream:
 *   qsvd_quantize_weight     offline per-channel int8 RTN of W_d (Sec. 4 setup)
 *   qsvd_quantize_weight_rotated  the same of H1 W_d (Eq. 12's online rotation)
 *   qsvd_importance_scores   offline Eq. 10 scores of singular values (Sec. 3.2)
 *   qsvd_rank_budget         offline cross-layer top-k of those scores (Sec. 3.2)
 *   qsvd_latent_project      C = Q(X) Q(W_d), requantized per token (Eq. 11-12)
 *   qsvd_cache_append        store latent rows in the latent cache (Fig. 2(f))
 *   qsvd_latent_decode_attn  one decode step of attention over that cache (Eq. 5)
 *   qsvd_quantize_up         offline per-channel RTN of an up-projection (Eq. 11)
 *   qsvd_latent_decode_attn_qu  the decode step with quantized up-projections
 *   qsvd_latent_prefill_attn causal attention of prompt tokens over that cache
 *   qsvd_latent_prefill      the same for whole prompt blocks, K and V materialised
 *   qsvd_decode_step         project, requantize and append, and attend in one call
 *   qsvd_beta_factors        offline Eq. 3 factors at one beta (Sec. 3.3)
 *   qsvd_beta_objective      offline Eq. 14 objective of those factors
 *   qsvd_latent_project_static  the decode-size projection without a workspace
 *
 * Conventions shared by every entry point:
 *   - Row-vector convention Y = X W, as in the paper.  E = d = H * dh.
 *   - Every pointer is device memory owned by the caller unless stated
 *     otherwise.  The library never allocates device memory; scratch space is
 *     a caller-provided workspace whose size the *_workspace_bytes calls give.
 *     A workspace must be zero-filled before its first use; every call leaves
 *     the workspace's completion counters at zero again, so a workspace can be
 *     reused by later calls on the same stream, but two calls that may run
 *     concurrently on the GPU need separate workspaces.
 *   - Kernels are launched with programmatic dependent launch: a call may
 *     begin copying its (read-only) weights W_d, U_q, U_k, U_v into shared
 *     memory and L2 while the previous kernel in the stream is still running;
 *     every read of other data produced by earlier stream work happens after
 *     that work has completed.  So the weights must not be written by a
 *     kernel that permits dependent launches early and runs just before on
 *     the same stream (ordinary kernels and copies, and
 *     qsvd_quantize_weight, are fine).
 *   - Calls are asynchronous on `stream` and never synchronize it, except
 *     qsvd_check.  A return of QSVD_OK means the work was enqueued.
 *   - bf16 buffers are passed as uint16_t bit patterns.
 *   - Every device pointer must be 16-byte aligned; row lengths in bytes must
 *     be multiples of 16.
 *   - Errors: argument problems are detected on the host before anything is
 *     enqueued and return a negative status; the message of the last failure
 *     on the calling thread is in qsvd_last_error().  Out-of-range cache
 *     positions and expired bounded waits are detected on the device: the
 *     offending write is skipped, a device error word is set, and qsvd_check
 *     reports it.  Nothing traps or aborts.
 *
 * Quantizer (all entry points; the paper says per-token symmetric for
 * activations, RTN per-channel symmetric for weights, and fixes no
 * arithmetic, so this is the library's definition):
 *   m = max|v| over the row (or channel, or int4 group);
 *   s = fp32(fp32(clip * m) / q_max),  q_max = 127 (int8) or 7 (int4);
 *   code = clamp(round_half_even(fp32(v / s)), -q_max, q_max), IEEE division;
 *   s == 0 gives all-zero codes.  int4 scales are fp16: s is rounded to fp16
 *   (nearest even, saturated at 65504) and the codes divide by that value.
 */
#ifndef QSVD_H_
#define QSVD_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

#define QSVD_OK             0
#define QSVD_EINVAL        -1  /* null pointer, bad shape, misaligned pointer */
#define QSVD_EUNSUPPORTED  -2  /* device is not sm_103, or a shape the kernels do not cover */
#define QSVD_ECUDA         -3  /* a CUDA runtime call or launch failed */
#define QSVD_ETIMEOUT      -4  /* a bounded device-side wait expired (from qsvd_check) */
#define QSVD_ERANGE        -5  /* a cache position or sequence index out of range, or a value saturated at the fp16 range of the block prefill */
#define QSVD_ENOSPC        -6  /* workspace smaller than the *_workspace_bytes figure */

/*
 * Quantized shared down-projection W^d_qkv (Eq. 3), stored per output
 * channel.  codes[j * d + k] is the int8 code of W_d[k, j] (row j of `codes`
 * is column j of W_d: the reduction dimension d is contiguous).  scale[j] is
 * its fp32 scale.  codes_bf16 holds the same integer codes as bf16 bit
 * patterns in the same layout; it is the tensor-core operand of the prefill
 * GEMM (every int8 code is exact in bf16).  All three are produced by
 * qsvd_quantize_weight.  Requirements: d % 64 == 0, r % 16 == 0.
 *
 * The quantization setting (Sec. 4 setup: W8A8, W8A4, W4A4) is part of the
 * weight: w_bits says how W_d was quantized (8: codes in [-127, 127]; 4: in
 * [-7, 7], stored one per int8 byte; 0 reads as 8) and x_bits how
 * qsvd_latent_project quantizes X per token (8 or 4; 0 reads as 8).  With
 * w_bits = x_bits = 4 the prefill GEMM runs on codes_e4m3, the codes as fp8
 * e4m3 bytes (every value in [-7, 7] is exact in e4m3), on the fp8 tensor-core
 * path; without it, or for the mixed settings, on codes_bf16.  The latent is
 * requantized to lat_bits as before (W4A4 pairs with an int4 latent cache).
 */
typedef struct qsvd_down_weight {
    const int8_t   *codes;       /* [r, d] */
    const uint16_t *codes_bf16;  /* [r, d] */
    const float    *scale;       /* [r]    */
    int32_t d;
    int32_t r;
    int32_t rot;                 /* 0: the codes quantize W_d and X is quantized as it is (H1 = I or folded
                                    offline); b > 0: they quantize H1 W_d (qsvd_quantize_weight_rotated) and
                                    qsvd_latent_project rotates every row of X by H1 before quantizing it */
    int32_t w_bits;              /* 8 (or 0) or 4: bits of the codes */
    int32_t x_bits;              /* 8 (or 0) or 4: bits X is quantized to per token */
    const uint8_t *codes_e4m3;   /* [r, d] or NULL: the codes as fp8 e4m3 (W4A4 tensor-core operand) */
} qsvd_down_weight;

/*
 * Latent cache of one layer (Fig. 2(f): the buffered C_qkv, eta = r L per
 * sequence), laid out [B, Tmax, ...]:
 *   bits == 8: codes int8 [B, Tmax, r];  scales fp32 [B, Tmax] (one per token)
 *   bits == 4: codes uint8 [B, Tmax, r/2], element 2i in the low nibble of
 *              byte i, two's complement;  scales fp16 [B, Tmax, r/128]
 *              (one per token and 128-channel group).  Requires r % 128 == 0.
 */
typedef struct qsvd_cache {
    void   *codes;
    void   *scales;
    int32_t bits;
    int32_t B;
    int32_t Tmax;
    int32_t r;
} qsvd_cache;

/*
 * Offline weight preparation (Sec. 4 setup: RTN, per-channel symmetric, with
 * a clipping ratio `clip` in (0, 1]).
 *   W_d        fp32 [d, r] row-major (W_d[k, j] at k * r + j).
 *   codes      int8 [r, d] out;  codes_bf16 bf16 [r, d] out (may be NULL);
 *   scale      fp32 [r] out.
 */
int qsvd_quantize_weight(const float *W_d, int32_t d, int32_t r, float clip,
                         int8_t *codes, uint16_t *codes_bf16, float *scale,
                         cudaStream_t stream);

/*
 * The same for any setting: bits 8 or 4 (codes in [-7, 7] for 4), rot 0 or
 * the H1 block size (as qsvd_quantize_weight_rotated), and optional images
 * codes_bf16 [r, d] and codes_e4m3 [r, d] (fp8 e4m3 bytes; needs bits 4).
 */
int qsvd_quantize_weight_ex(const float *W_d, int32_t d, int32_t r, float clip, int32_t bits, int32_t rot,
                            int8_t *codes, uint16_t *codes_bf16, uint8_t *codes_e4m3, float *scale,
                            cudaStream_t stream);

/*
 * Quantized joint down-projection with the latent requantization fused
 * behind it (Eq. 12 with H1 = H2 = I, then Eq. 11's Q(C_qkv)):
 *   1. X [T, d] bf16 is quantized per token to int8 (int4 codes when
 *      W->x_bits == 4) (clip `act_clip`);
 *   2. acc[t, j] = sum_k xq[t, k] * codes[j, k]    exact int32;
 *   3. c[t, j] = fp32(fp32(fp32(acc) * s_x[t]) * scale[j])   (no FMA);
 *   4. c[t, :] is requantized per token to `lat_bits` (8: one fp32 scale per
 *      token; 4: one fp16 scale per 128 channels), clip `lat_clip`.
 * Destinations (at least one must be given):
 *   lat_codes/lat_scales  token-major: int8 [T, r] + fp32 [T], or packed
 *                         uint8 [T, r/2] + fp16 [T, r/128];
 *   dst/dst_seq/dst_pos   fused cache append: row t goes to sequence
 *                         dst_seq[t] at position dst_pos[t] (device int32
 *                         arrays of length T); dst->bits must equal lat_bits.
 * Optional intermediates for inspection (NULL skips the write):
 *   xq_out int8 [T, d], xs_out fp32 [T], acc_out int32 [T, r].
 * workspace: at least qsvd_project_workspace_bytes(T, d, r) bytes, 256-byte
 * aligned (while T * r <= 80 * 128 * 128 it includes room for four int32
 * [T, r] partial sums: a product with few tiles splits K over more CTAs).
 * T may be 0 (nothing is enqueued).
 */
int qsvd_latent_project(const qsvd_down_weight *W, const uint16_t *X, int64_t T,
                        float act_clip, int32_t lat_bits, float lat_clip,
                        void *lat_codes, void *lat_scales,
                        const qsvd_cache *dst, const int32_t *dst_seq, const int32_t *dst_pos,
                        int8_t *xq_out, float *xs_out, int32_t *acc_out,
                        void *workspace, size_t workspace_bytes, cudaStream_t stream);

size_t qsvd_project_workspace_bytes(int64_t T, int32_t d, int32_t r);

/*
 * Offline preparation, Sec. 3.2: importance scores of a layer's singular
 * values (Eq. 10), score_i = (1/N) sum_n (sigma_i [U^T G_n V]_{ii})^2, for
 * the cross-layer rank budget (keep the k highest scores of all layers).
 *   U fp32 [m, k] (left singular vectors as columns), sigma fp32 [k],
 *   Vt fp32 [k, n] (right singular vectors as rows), G fp32 [N, m, n] (the
 *   loss gradient for each of N calibration samples), scores fp32 [k] out.
 *   workspace: qsvd_importance_workspace_bytes(N, m, k) bytes.
 * The products G_n V run on the tensor cores as three tf32 products per fp32
 * product (each operand split into a tf32 part and an fp32 remainder), which
 * keeps fp32-level accuracy; rows of G and Vt need n % 4 == 0 and 16-byte
 * aligned bases for that path, other shapes run in fp32 on the CUDA cores.
 * All sums run in a fixed order, so the result is the same bit for bit on
 * every run.  N <= 65535 per call.
 */
int qsvd_importance_scores(const float *U, const float *sigma, const float *Vt, const float *G, int32_t N, int32_t m,
                           int32_t n, int32_t k, float *scores, void *workspace, size_t workspace_bytes,
                           cudaStream_t stream);

size_t qsvd_importance_workspace_bytes(int32_t N, int32_t m, int32_t k);

/*
 * The cross-layer rank budget of Sec. 3.2 (the global sort after Eq. 10):
 * of the n singular values of all layers -- scores fp32 [n], the layers'
 * score vectors concatenated in layer order -- keep the k highest-scoring
 * ones: keep[i] = 1 for those, 0 for the rest (uint8 [n] out).  Equal scores
 * go to the lower position (the lower layer, then the lower index).  Scores
 * must not be NaN.  Exactly k entries are kept (0 <= k <= n).  workspace:
 * qsvd_rank_budget_workspace_bytes() bytes.
 */
int qsvd_rank_budget(const float *scores, int32_t n, int32_t k, uint8_t *keep, void *workspace,
                     size_t workspace_bytes, cudaStream_t stream);

size_t qsvd_rank_budget_workspace_bytes(void);

/*
 * The per-layer choice of beta (Sec. 3.3, Eq. 13-14), one beta at a time.
 * Eq. 3 splits the truncated joint SVD of W_concat = [W_q W_k W_v] (E x n_out,
 * n_out = 3E) as W_d = Wd_r Sigma^beta and W^u = Sigma^(1-beta) Wu_r; Eq. 14
 * keeps the beta whose quantized output Y' = Q(C) Q(W^u) (Eq. 11, C = X W_d
 * from Eq. 12) is closest to Y = X W_concat on calibration tokens.
 *
 * qsvd_beta_factors: the two factors at one beta from the caller's SVD
 *   Wd_r  fp64 [E, r] row-major, Wu_r fp64 [r, n_out] row-major (the SVD is
 *         the caller's, computed once per layer offline);
 *   fd, fu fp64 [r]: sigma_i^beta and sigma_i^(1-beta) (the caller's powers);
 *   W_d   fp32 [E, r] out, fp32(Wd_r[k, i] * fd[i]) (qsvd_quantize_weight's
 *         input);
 *   u_codes, u_scale out: Q(W^u) in the qsvd_up_weight layout (int8 [r, n_out]
 *         or packed int4 [r, n_out/2]; fp32 [n_out]), the weight quantizer
 *         per output channel j applied to W^u[i, j] = fu[i] * Wu_r[i, j] formed
 *         in fp64: s_j = fp32(fp32(u_clip * max_i |W^u[i, j]|) / q_max),
 *         code = clamp(rne(fp32(W^u[i, j] / s_j))), q_max 127 or 7.
 *   Requirements: n_out % 128 == 0, u_bits 8 or 4, u_clip in (0, 1].
 *
 * qsvd_beta_objective: Eq. 14's objective for the factors of one beta,
 *   sum over tokens n < N and channels j < n_out of (Y[n, j] - Y'[n, j])^2,
 *   Y' = Q(C) Q(W^u).
 *   Y          fp32 [N, n_out]: X W_concat (the caller's, once per layer);
 *   lat_codes, lat_scales: Q(C) of the N tokens as qsvd_latent_project writes
 *              them token-major (int8 [N, r] + fp32 [N], or packed int4
 *              [N, r/2] + fp16 [N, r/128]; lat_bits 8 or 4);
 *   u_codes, u_scale, u_bits: Q(W^u) as qsvd_beta_factors writes it;
 *   objective  one fp64 out (device).  Products of codes are exact integer
 *              sums; the scales and the squares are applied in fp64 and summed
 *              in a fixed order (the same bits on every run).
 *   workspace  qsvd_beta_objective_workspace_bytes(N, n_out) bytes.
 *   Requirements: 0 < N <= 4194240, n_out % 64 == 0, r % 32 == 0 (r % 128 == 0
 *   for an int4 latent).
 */
int qsvd_beta_factors(const double *Wd_r, const double *Wu_r, const double *fd, const double *fu, int32_t E,
                      int32_t r, int32_t n_out, int32_t u_bits, float u_clip, float *W_d, void *u_codes,
                      float *u_scale, cudaStream_t stream);

int qsvd_beta_objective(const float *Y, int64_t N, int32_t n_out, const void *lat_codes, const void *lat_scales,
                        int32_t lat_bits, int32_t r, const void *u_codes, const float *u_scale, int32_t u_bits,
                        double *objective, void *workspace, size_t workspace_bytes, cudaStream_t stream);

size_t qsvd_beta_objective_workspace_bytes(int64_t N, int32_t n_out);

/*
 * The rotation H1 of Eq. 11-12 applied on the fly (for models where it is not
 * folded into the previous layer): C = Q(X H1^T) Q(H1 W_d).  H1 is the
 * block-diagonal normalized Walsh-Hadamard matrix I_{d/rot} (x) H_rot /
 * sqrt(rot) (Sylvester H_rot, rot a power of two >= 2 dividing d; the
 * largest such rot spreads outliers furthest), symmetric and orthogonal, so
 * (X H1)(H1 W_d) = X W_d.  Both the weight quantizer below and
 * qsvd_latent_project compute it as the fast Walsh-Hadamard transform in fp32
 * (stages h = 1, 2, ..., rot/2 in that order, pair (i, i+h) with (i & h) == 0
 * -> (v_i + v_{i+h}, v_i - v_{i+h}), then every entry times fp32(1/sqrt(rot))),
 * so the codes are reproducible bit for bit.
 * qsvd_quantize_weight_rotated: as qsvd_quantize_weight, of H1 W_d; the
 * caller sets rot in the qsvd_down_weight it builds from the outputs.
 * Needs d <= 6144.  qsvd_decode_step and qsvd_latent_project_static refuse
 * rotated weights (QSVD_EUNSUPPORTED).
 */
int qsvd_quantize_weight_rotated(const float *W_d, int32_t d, int32_t r, float clip, int32_t rot, int8_t *codes,
                                 uint16_t *codes_bf16, float *scale, cudaStream_t stream);

/*
 * Latent cache append (the store of Fig. 2(f)): row i of the token-major
 * latent (codes + scales, in the cache's format) is copied to sequence
 * seq[i], position pos[i].  seq and pos are device int32 [n].  Rows whose
 * (seq, pos) fall outside [0, B) x [0, Tmax) are skipped and flag QSVD_ERANGE
 * for qsvd_check.
 */
int qsvd_cache_append(const qsvd_cache *cache, const int32_t *seq, const int32_t *pos,
                      int64_t n, const void *lat_codes, const void *lat_scales,
                      cudaStream_t stream);

/*
 * One decode step of attention over the latent cache (Eq. 5 and the decode
 * remark after it).  For every sequence b with L = seq_len[b] cached tokens
 * (the current token, already appended, at position L-1) and every head h
 * (columns h*dh .. h*dh+dh-1 of each up-projection):
 *   c_t  = dequantized latent of token t;     q_h = c_{L-1} U_q[:, h]
 *   o_h  = softmax_t( (c_t U_k[:, h]) . q_h * softmax_scale ) . (c_t U_v[:, h])
 * computed without forming K or V: U_k is absorbed into the query
 * (qt_h = U_k[:, h] q_h, scores c_t . qt_h) and U_v is applied after the
 * softmax-weighted sum of latent rows.
 *   seq_len      device int32 [B], 1 <= seq_len[b] <= max_seq_len <= Tmax;
 *   max_seq_len  host-side bound used to size the launch;
 *   U_q, U_k, U_v  bf16 [r, H*dh] row-major;
 *   O            fp32 [B, H*dh] out.
 * workspace: qsvd_decode_workspace_bytes(B, max_seq_len, r, H, dh) bytes.
 * Requirements: dh in {64, 128}; r % 32 == 0 and r <= 3072; H*dh % 256 == 0
 * and H*dh <= 6144.
 */
int qsvd_latent_decode_attn(const qsvd_cache *cache, const int32_t *seq_len, int32_t max_seq_len,
                            const uint16_t *U_q, const uint16_t *U_k, const uint16_t *U_v,
                            int32_t H, int32_t dh, float softmax_scale, float *O,
                            void *workspace, size_t workspace_bytes, cudaStream_t stream);

size_t qsvd_decode_workspace_bytes(int32_t B, int32_t max_seq_len, int32_t r, int32_t H, int32_t dh);

/*
 * Quantized up-projection (Eq. 11: Y' = Q(C) Q(H2 W^u) with H2 = I, the
 * rotation folded offline), for qsvd_latent_decode_attn_qu.  One of U_q, U_k,
 * U_v ([r, d] with d = H * dh; column c is output channel c) quantized per
 * output channel by symmetric RTN (the weight quantizer of the Sec. 4 setup):
 *   bits == 8: codes int8 [r, d], codes[j * d + c] the code of U[j, c];
 *   bits == 4: codes uint8 [r, d/2], column 2i in the low nibble of byte
 *              j * d/2 + i, two's complement;
 *   scale fp32 [d]: U[j, c] ~ code(j, c) * scale[c].
 */
typedef struct qsvd_up_weight {
    const void  *codes;
    const float *scale;
    int32_t bits;
    int32_t r;
    int32_t d;
} qsvd_up_weight;

/*
 * Offline Q(W^u) (Eq. 11) of one up-projection: U bf16 [r, d] row-major ->
 * codes and scale in the qsvd_up_weight layout above (the library's quantizer
 * with q_max = 127 or 7 and clipping ratio `clip` in (0, 1], per column).
 * Requirements: d % 32 == 0, bits 8 or 4.
 */
int qsvd_quantize_up(const uint16_t *U, int32_t r, int32_t d, int32_t bits, float clip, void *codes, float *scale,
                     cudaStream_t stream);

/*
 * qsvd_latent_decode_attn with quantized up-projections (Eq. 11): the same
 * decode step (Eq. 5, U_k absorbed into the query, U_v applied last) where
 * every product with an up-projection reads its int8 or int4 codes and
 * applies the per-output-channel scales (q = s_q * (c U_q codes);
 * q~_h = U_k codes (s_k * q_h); o = s_v * (o_lat U_v codes)), so a step
 * streams half (int8) or a quarter (int4) of the bf16 weight bytes.  The
 * three weights may differ in bits; each must have r = cache->r and d = H*dh.
 * Workspace and requirements as for qsvd_latent_decode_attn.
 */
int qsvd_latent_decode_attn_qu(const qsvd_cache *cache, const int32_t *seq_len, int32_t max_seq_len,
                               const qsvd_up_weight *U_q, const qsvd_up_weight *U_k, const qsvd_up_weight *U_v,
                               int32_t H, int32_t dh, float softmax_scale, float *O,
                               void *workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * Causal attention of prompt tokens over the latent cache (prefill; Fig. 2(f)
 * and Eq. 5 with the causal mask of a decoder).  Row i of the call is one
 * query: the token at position q_len[i]-1 of cache sequence q_seq[i], which
 * attends to positions 0 .. q_len[i]-1 of that sequence, exactly as
 * qsvd_latent_decode_attn does for a sequence of length q_len[i].  A prompt
 * of T tokens appended at positions t0 .. t0+T-1 of sequence b (by
 * qsvd_latent_project with dst = cache) is prefilled with q_seq[i] = b and
 * q_len[i] = t0 + i + 1; rows of several sequences may be mixed freely.
 *   q_seq, q_len  device int32 [n]; 0 <= q_seq[i] < cache->B and
 *                 1 <= q_len[i] <= max_len <= Tmax.  A row outside these
 *                 ranges is skipped, its output row is zero, and QSVD_ERANGE
 *                 is flagged for qsvd_check;
 *   max_len       host-side bound on q_len used to size the launches;
 *   U_q, U_k, U_v bf16 [r, H*dh] row-major;  O fp32 [n, H*dh] out.
 * The rows are processed in consecutive groups that reuse one workspace of
 * qsvd_prefill_workspace_bytes(n, max_len, r, H, dh) bytes; the cache is only
 * read.  n may be 0 (nothing is enqueued).  Requirements as for
 * qsvd_latent_decode_attn.
 */
int qsvd_latent_prefill_attn(const qsvd_cache *cache, const int32_t *q_seq, const int32_t *q_len,
                             int64_t n, int32_t max_len,
                             const uint16_t *U_q, const uint16_t *U_k, const uint16_t *U_v,
                             int32_t H, int32_t dh, float softmax_scale, float *O,
                             void *workspace, size_t workspace_bytes, cudaStream_t stream);

size_t qsvd_prefill_workspace_bytes(int64_t n, int32_t max_len, int32_t r, int32_t H, int32_t dh);

/*
 * Causal prefill of whole prompt blocks in the materialised form (Eq. 5 as
 * written): the latent rows of a block are multiplied by U_q, U_k and U_v on
 * the tensor cores (fp16 operands, fp32 accumulation, fp16 Q, K, V), then
 * every query attends causally to its prefix at head size dh.  At prefill
 * this needs r / dh times fewer products than qsvd_latent_prefill_attn, which
 * keeps the decode kernels' absorbed form; both compute the same attention.
 *
 * Block k: positions t0 .. t0+T-1 of cache sequence seq, already stored in
 * the cache together with positions 0 .. t0-1 (a continued prompt reads
 * them as keys), attend to positions 0 .. their own.  Its T output rows
 * follow the rows of blocks 0 .. k-1 in O (fp32 [sum T, H*dh]).  The blocks
 * array is host memory and is read before the call returns.
 *   Ut  fp16 [3*H*dh, r]: [U_q U_k U_v]^T from qsvd_prefill_weights (once per
 *       layer; U_* bf16 [r, H*dh]).
 *   workspace  qsvd_latent_prefill_workspace_bytes(blocks, n_blocks, r, H, dh)
 *       bytes: fp16 copies of the blocks' latent rows and of Q, K, V.
 * Requirements: dh == 128, H*dh % 256 == 0, r % 64 == 0, softmax_scale > 0
 * and finite; a block outside the cache (seq outside [0, B), t0 < 0, T < 1,
 * t0 + T > Tmax) returns QSVD_EINVAL before anything is enqueued; a launch of
 * 64 blocks whose padded rows R give R * r / 8 >= 2^31 returns
 * QSVD_EUNSUPPORTED.  fp16 Ut, Q, K, V (and the int4 latent operand) hold
 * magnitudes up to 65504: a larger value is saturated to +-65504 and flags
 * QSVD_ERANGE for qsvd_check (qsvd_prefill_weights likewise for |U| above
 * 65504), so no inf is produced silently.
 */
typedef struct {
    int32_t seq, t0, T;
} qsvd_prefill_block;

int qsvd_prefill_weights(const uint16_t *U_q, const uint16_t *U_k, const uint16_t *U_v, int32_t r, int32_t d,
                         uint16_t *Ut, cudaStream_t stream);

int qsvd_latent_prefill(const qsvd_cache *cache, const qsvd_prefill_block *blocks, int32_t n_blocks,
                        const uint16_t *Ut, int32_t H, int32_t dh, float softmax_scale, float *O,
                        void *workspace, size_t workspace_bytes, cudaStream_t stream);

size_t qsvd_latent_prefill_workspace_bytes(const qsvd_prefill_block *blocks, int32_t n_blocks, int32_t r,
                                           int32_t H, int32_t dh);

/*
 * One whole decode step in one call: for each of the B = cache->B sequences,
 * the new token X[b] (bf16 [B, d]) is quantized and projected (Eq. 12), its
 * latent is requantized and stored at position seq_len[b] - 1 of sequence b
 * (Eq. 11, Fig. 2(f)), and attention over positions 0 .. seq_len[b]-1 is
 * computed as in qsvd_latent_decode_attn (Eq. 5).  The result equals
 * qsvd_latent_project(dst = cache, dst_seq = b, dst_pos = seq_len[b] - 1)
 * followed by qsvd_latent_decode_attn, codes and scales bit for bit.  It
 * exists because a small-batch decode step is bound by the latency of its
 * chain of dependent launches rather than by its bytes: knowing both halves,
 * the call lets the query kernel requantize and store the new latents itself
 * (B <= 4), one launch and one dependent round trip fewer than the two calls.
 * An invalid slot (seq_len[b] outside [1, Tmax]) is skipped and flags
 * QSVD_ERANGE for qsvd_check.
 * Requirements: B <= 64; d = H*dh, d % 256 == 0, d <= 6144; r % 32 == 0,
 * r <= 3072; dh in {64, 128}; 8-bit X and W_d codes without a rotation.
 * workspace: qsvd_decode_step_workspace_bytes(...) bytes, zero-filled before
 * its first use.
 */
int qsvd_decode_step(const qsvd_down_weight *W, const uint16_t *X, const qsvd_cache *cache,
                     const int32_t *seq_len, int32_t max_seq_len,
                     const uint16_t *U_q, const uint16_t *U_k, const uint16_t *U_v,
                     int32_t H, int32_t dh, float act_clip, float lat_clip, float softmax_scale,
                     float *O, void *workspace, size_t workspace_bytes, cudaStream_t stream);

size_t qsvd_decode_step_workspace_bytes(int32_t B, int32_t max_seq_len, int32_t d, int32_t r,
                                        int32_t H, int32_t dh);

/*
 * Allocation-free variant of qsvd_latent_project for decode-size calls
 * (T <= 16 tokens, r <= 4096, d % 256 == 0, d <= 6144).  The paper has no
 * counterpart; it exists for callers that cannot allocate device memory when
 * they project a token, such as a serving process whose device memory was
 * reserved in full at start-up by another allocator, or code running while a
 * stream is captured into a graph (cudaMalloc is not allowed there), and
 * that therefore cannot supply the workspace qsvd_latent_project needs.
 * Arguments and results are those of qsvd_latent_project without the
 * inspection outputs and the workspace.  The scratch lives in a fixed
 * 264 KiB device array inside the library, held by every GPU that loads the
 * library until the process exits; the call allocates nothing.
 *   - The first call on a device looks up that array's device address, so
 *     make it before any stream capture on that device.
 *   - T > 16 or r > 4096 returns QSVD_ENOSPC with a message.
 *   - All calls share the one array: calls that may overlap on the GPU (on
 *     different streams, or on the same device from several threads without
 *     ordering) race and must not be issued.
 *   - Each call clears the array's completion counter before it launches.
 */
int qsvd_latent_project_static(const qsvd_down_weight *W, const uint16_t *X, int64_t T,
                               float act_clip, int32_t lat_bits, float lat_clip,
                               void *lat_codes, void *lat_scales,
                               const qsvd_cache *dst, const int32_t *dst_seq, const int32_t *dst_pos,
                               cudaStream_t stream);

/*
 * Where qsvd_latent_project requantizes the latent on the tensor-core path
 * (a library setting, not part of the paper's method; process-wide, not
 * thread-safe):
 *   0  automatic (default): in the GEMM epilogue for int4 latents, and for
 *      int8 latents when r / 256 <= 6 (the per-token maximum is exchanged
 *      within a cluster of r / 256 CTAs) and the 256-column tiles fill at
 *      least one wave of the GPU (ceil(T / 128) * r / 256 >= the SM count;
 *      below that the separate kernel with twice the tiles is faster);
 *   1  always a separate requantization kernel over an fp32 latent in the
 *      workspace;
 *   2  in the epilogue whenever possible (int8 needs r / 256 <= 8).
 * Codes and scales are identical either way.  Returns the previous setting,
 * or QSVD_EINVAL for another value.
 */
int qsvd_set_project_epilogue(int32_t mode);

/*
 * Choice of attention kernels for qsvd_latent_decode_attn (a library setting,
 * not part of the paper's method; process-wide, not thread-safe):
 *   0  automatic (default): the warp-level tensor-core kernel when
 *      B * max_seq_len <= 2048 (1024 for r > 2048) or the tcgen05 kernel
 *      cannot take the shape,
 *      else the tcgen05 kernel (the warp-level kernel needs r <= 3072;
 *      beyond that, the CUDA-core kernels);
 *   1  always the CUDA-core kernels;
 *   2  the tcgen05 kernel whenever the shape allows it;
 *   3  the warp-level tensor-core kernel whenever r <= 3072.
 * The tcgen05 kernel needs r <= 3072 with r % 256 == 0 up to r = 1536
 * (clusters of two CTAs) and r % 512 == 0 above (clusters of four); it takes
 * the heads in launches of up to 32.  Other shapes use the warp-level kernel
 * (r <= 3072) or the CUDA-core kernels.  All give the same results up to
 * floating-point rounding.  qsvd_latent_prefill_attn follows the same
 * setting.
 * Returns the previous setting, or QSVD_EINVAL for another value.
 */
int qsvd_set_decode_attn_path(int32_t path);

/*
 * Rows per group of qsvd_latent_prefill_attn (a library setting, not part of
 * the paper's method; process-wide, not thread-safe): 0 (default) picks the
 * largest power of two up to 1024 whose workspace stays within 2 GiB; a
 * value in [1, 65535] fixes the group size (the workspace size query follows
 * it).  Results do not depend on it.  Returns the previous setting, or
 * QSVD_EINVAL for a value outside [0, 65535].
 */
int qsvd_set_prefill_group_rows(int32_t rows);

/*
 * Synchronizes `stream`, then reads and clears the device error word.
 * Returns QSVD_OK, QSVD_ERANGE, QSVD_ETIMEOUT or QSVD_ECUDA.
 */
int qsvd_check(cudaStream_t stream);

/*
 * Failure-detection self-test (no counterpart in the paper).  Enqueues on
 * `stream` one thread that waits on an mbarrier no one arrives on for at
 * most timeout_ms milliseconds (1..1000), then sets the timeout bit of the
 * device error word and returns: the path every bounded device wait of the
 * library takes when it expires.  The next qsvd_check returns QSVD_ETIMEOUT
 * and clears the word; the CUDA context stays usable.  Returns QSVD_EINVAL
 * for a timeout outside 1..1000.
 */
int qsvd_selftest_wait_timeout(int32_t timeout_ms, cudaStream_t stream);

/* Message of the last failure on the calling thread ("" if none). */
const char *qsvd_last_error(void);

/*
 * Kernel-level timing for benchmarks (not part of the paper's method).
 * qsvd_profile_events(events, n) hands the calling thread an array of n
 * caller-created cudaEvent_t handles (passed as void*).  From then on every
 * entry point records the next event on its stream once before its first
 * kernel (label "begin") and once after each kernel it launches (label = the
 * kernel's name), until the array is full.  The elapsed time between event
 * i-1 and event i is the duration of kernel i whenever label i is not
 * "begin".  qsvd_profile_events(NULL, 0) switches recording off.  Nothing is
 * recorded while profiling is off.
 */
int qsvd_profile_events(void **events, int32_t capacity);
int32_t qsvd_profile_count(void);
const char *qsvd_profile_label(int32_t i);

/* Library version, major * 10000 + minor * 100 + patch. */
int qsvd_version(void);

#ifdef __cplusplus
}
#endif
#endif /* QSVD_H_ */
