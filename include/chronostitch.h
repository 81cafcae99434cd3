/*
 * chronostitch.h - C ABI of the ChronoStitch KV-composition hot path
 * (arxiv 2607.19547, "ChronoStitch: Training-Free Composition of Visual KV
 * Memories"), built for one NVIDIA GB300 GPU (sm_103a).
 *
 * The query-time procedure of Sec. 2 composes independently prefilled video
 * chunk KV caches: it re-bases stored post-rotary keys onto global
 * three-axis mRoPE coordinates (Eq. 3), scores each later-chunk visual token
 * by how far its fresh layer-1 key moved (Eq. 5), selects the top rho of them,
 * and recomputes those tokens with causal attention over the composed cache
 * (Eq. 1).  The four calls below are those four steps.
 *
 * Conventions shared by every call
 *   - Tensor pointers are DEVICE memory of the current CUDA device, owned by
 *     the caller; the library keeps no pointer after a call returns.  Layouts
 *     are row-major; strides are in elements.
 *   - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *     default stream).  Argument checks run on the host before any launch; a
 *     call that returns an error launched nothing.
 *   - Data-dependent failures found on the device (a bounded wait that gave
 *     up, a query position out of range) are recorded in a status word that
 *     is shared by every stream of the device (and every caller of this
 *     library in the process), and reported by cs_sync_status().
 *   - There is no CPU fallback: every computation runs in this library's own
 *     CUDA kernels.
 *   - head_dim must be 128 (CS_ERR_UNSUPPORTED otherwise).  Every tensor
 *     pointer and every row start must be 16-byte aligned.
 *   - The library owns no device allocation.  Its one piece of device state
 *     is a small static status word per device, whose address is looked up on
 *     the first call made on that device (and again after the device's
 *     context changes, e.g. after cudaDeviceReset); make that first call
 *     before capturing a stream.
 */
#ifndef CHRONOSTITCH_H
#define CHRONOSTITCH_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    CS_OK = 0,
    CS_ERR_INVALID_ARG = 1,   /* bad pointer, size, stride or alignment; nothing launched */
    CS_ERR_UNSUPPORTED = 2,   /* well-formed but not implemented (head_dim != 128, ...)  */
    CS_ERR_CUDA = 3,          /* a CUDA runtime call or a kernel launch failed            */
    CS_ERR_TIMEOUT = 4,       /* a device-side bounded wait gave up (from cs_sync_status) */
    CS_ERR_DEVICE_ARG = 5     /* device data failed a check, e.g. qpos out of range       */
} cs_status;

typedef enum {
    CS_DTYPE_F32 = 0,         /* IEEE binary32 storage, fp32 arithmetic                   */
    CS_DTYPE_BF16 = 1         /* bfloat16 storage, fp32 arithmetic (fp32 accumulators)    */
} cs_dtype;

/* Multimodal RoPE configuration (Eq. 2).  Frequency pair i (0 <= i < head_dim/2)
 * pairs elements i and i + head_dim/2 (half-split layout) and rotates by
 * p_sigma(i) * theta_i with theta_i = theta^(-2i/head_dim); sigma assigns the
 * first sections[0] pairs to the temporal axis, the next sections[1] to height
 * and the last sections[2] to width.  Qwen2.5-VL: theta 1e6, sections {16,24,24}. */
typedef struct {
    double theta;
    int32_t sections[3];
} cs_rope_cfg;

/* Version of this ABI (bumped on any incompatible change). */
int cs_abi_version(void);

/*
 * Step 1 - re-base stored post-rotary keys (Eq. 3, Sec. 2).
 *
 * For every layer l < n_layers, token t < T, kv head h < n_kv_heads and
 * frequency pair i:  (x_i, x_{i+64}) <- R(Delta_i) (x_i, x_{i+64}) with
 * Delta_i = (pos_global[t][sigma(i)] - pos_local[t][sigma(i)]) * theta_i, so a
 * key stored at its chunk-local coordinate becomes the key at its global
 * coordinate.  Values are not rotated (Sec. 2), so no V argument exists.
 *
 *   k_in, k_out   [n_layers][T][n_kv_heads][head_dim] with layer stride
 *                 `layer_stride` (>= T*n_kv_heads*head_dim); element
 *                 (l,t,h,d) at l*layer_stride + (t*n_kv_heads + h)*head_dim + d.
 *                 k_out == k_in re-bases in place (tokens with Delta = 0 are
 *                 not touched); otherwise every row of k_out is written and the
 *                 buffers must not overlap.
 *   pos_local, pos_global   int32 [T][3] (t, h, w) coordinates, device memory,
 *                 not overlapping k_out (CS_ERR_INVALID_ARG).
 *   rope          host pointer, read during the call only.
 *
 * Result: bf16 outputs are the exact rotation rounded once to bfloat16
 * (nearest, ties to even); f32 outputs are within a few units of the last
 * place of the exact rotation.  Tokens whose Delta is zero on all three axes
 * are returned unchanged bit for bit.
 */
cs_status cs_rebase_keys(const void *k_in, void *k_out, cs_dtype dtype, int n_layers,
                         int64_t layer_stride, int T, int n_kv_heads, int head_dim,
                         const int32_t *pos_local, const int32_t *pos_global,
                         const cs_rope_cfg *rope, void *stream);

/*
 * Step 2 - key-deviation score (Eq. 5, Sec. 2).
 *
 * score_out[t] = delta_t^2 = sum_j (k_fresh[t][j] - k_cached[t][j])^2 over the
 * E = n_kv_heads*head_dim elements of token t's layer-1 key, in fp32, in this
 * fixed order (so results are reproducible bit for bit):
 *   d_j = fp32(a_j - b_j), q_j = fp32(d_j*d_j) (no fused multiply-add);
 *   per block of 8 consecutive elements ((q0+q1)+(q2+q3))+((q4+q5)+(q6+q7));
 *   block sums s[0..E/8) padded with +0 to a power of two P, then for
 *   m = P/2, ..., 1: s[b] = s[b] + s[b+m] for b < m; the result is s[0].
 * delta_t itself is the square root; ranking uses delta_t^2, which orders the
 * same way without a rounding step.
 *
 *   k_fresh   row t at k_fresh + t*fresh_row_stride, E contiguous elements
 *   k_cached  row t at k_cached + t*cached_row_stride (e.g. the re-based layer-1
 *             rows of the composed cache: stride n_kv_heads*head_dim)
 *   score_out fp32 [n], not overlapping either key array (CS_ERR_INVALID_ARG)
 */
cs_status cs_score_deviation(const void *k_fresh, const void *k_cached, cs_dtype dtype, int n,
                             int n_kv_heads, int head_dim, int64_t fresh_row_stride,
                             int64_t cached_row_stride, float *score_out, void *stream);

/*
 * Steps 1 and 2 in one call (Eq. 3 then Eq. 5 at the score layer, Sec. 2):
 * exactly cs_rebase_keys(...) followed by
 *   cs_score_deviation(k_fresh, k_out + (score_layer*layer_stride + cand0*E),
 *                      dtype, n_cand, n_kv_heads, head_dim, fresh_row_stride, E,
 *                      score_out)              with E = n_kv_heads*head_dim,
 * bit for bit, where the candidates are tokens [cand0, cand0 + n_cand) of the
 * cache.  It is one kernel launch: the re-base computes the scores of the rows it
 * has just re-based (for bf16 and fp32, any supported kv head count).
 *
 *   0 <= score_layer < n_layers (when n_cand > 0);  0 <= cand0,  cand0 + n_cand <= T
 *   k_fresh    row c (token cand0 + c) at k_fresh + c*fresh_row_stride, E elements,
 *              device memory, 16-byte aligned rows, not overlapping k_out
 *   score_out  fp32 [n_cand], device memory, not overlapping the keys, k_fresh or
 *              the coordinates
 * Other arguments and errors as for cs_rebase_keys and cs_score_deviation.
 */
cs_status cs_rebase_and_score(const void *k_in, void *k_out, cs_dtype dtype, int n_layers,
                              int64_t layer_stride, int T, int n_kv_heads, int head_dim,
                              const int32_t *pos_local, const int32_t *pos_global,
                              const cs_rope_cfg *rope, int score_layer, int cand0, int n_cand,
                              const void *k_fresh, int64_t fresh_row_stride, float *score_out,
                              void *stream);

/*
 * Step 3 - top-rho selection (Sec. 2).
 *
 * Writes the k candidates with the largest score as ascending global indices
 * idx_base + i into out_idx[0..k).  Order: scores compare as fp32 values (for
 * non-negative scores, the order of their bit patterns; +inf above every
 * finite value, a positive NaN above +inf, negative values below -0 < +0);
 * equal scores (identical bit patterns) rank the lower index first.  The
 * caller picks k, e.g. k = ceil(rho * n) with rho in basis points:
 * (rho_bp*n + 9999)/10000.
 *
 *   score    fp32 [n], device memory;   0 <= k <= n;   idx_base + n <= INT32_MAX
 *   out_idx  int32 [k], device memory, not overlapping score (CS_ERR_INVALID_ARG)
 * One launch: one CTA for n <= 8192, else one thread-block cluster (up to 16 CTAs, as
 * many as the device can co-schedule; the first such call on a device queries that, so
 * make it before capturing a stream); no global memory besides score and out_idx is used.
 */
cs_status cs_select_topk(const float *score, int n, int k, int32_t idx_base, int32_t *out_idx,
                         void *stream);

/*
 * Step 4 - repair attention of the selected rows (Eq. 1, Sec. 2).
 *
 * For layer l, query row r and query head h:
 *   o[l][r][h] = softmax_j( scale * q[l][r][h] . k[l][j][h/G] ) v[l][j][h/G],
 *   j = 0 .. qpos[r]  (causal in global sequence order, the row's own key included),
 *   G = n_q_heads / n_kv_heads (grouped-query attention).
 *
 *   q, o     [n_layers][M][n_q_heads][head_dim], contiguous; o may be q itself
 *            but must not overlap k or v (CS_ERR_INVALID_ARG)
 *   k, v     [n_layers][T][n_kv_heads][head_dim] with layer stride kv_layer_stride
 *   qpos     int32 [M], strictly ascending, 0 <= qpos[r] < T (checked on the
 *            device; a violation yields CS_ERR_DEVICE_ARG at cs_sync_status and
 *            leaves o undefined); not overlapping o or lse (CS_ERR_INVALID_ARG)
 *   lse      optional fp32 [n_layers][M][n_q_heads]: the natural-log normaliser
 *            log(sum_j exp(scale * q.k_j)); NULL to skip; 4-byte aligned and
 *            not overlapping k, v or o (CS_ERR_INVALID_ARG)
 *   scale    the logit scale, 1/sqrt(head_dim) in Eq. 1
 * bf16 runs on the tensor cores (bf16 operands, fp32 accumulation); f32 runs
 * fp32 arithmetic on the CUDA cores.
 */
cs_status cs_repair_attention(const void *q, const void *k, const void *v, void *o, float *lse,
                              cs_dtype dtype, int n_layers, int M, int T, int n_q_heads,
                              int n_kv_heads, int head_dim, int64_t kv_layer_stride,
                              const int32_t *qpos, float scale, void *stream);

/*
 * Scatter-back of repaired rows (Sec. 2: the recomputed tokens' fresh keys and
 * values replace their stored ones in the composed cache before each layer's
 * attention).  For every layer l < n_layers and row r < n_rows:
 *   cache[l][idx[r]][:] = rows[l][r][:]          (row_elems elements per token)
 *
 *   cache      [n_layers][T][row_elems], layer stride cache_layer_stride
 *              (elements, >= T*row_elems), device memory, written in place
 *   rows       [n_layers][n_rows][row_elems], layer stride rows_layer_stride
 *              (>= n_rows*row_elems), device memory, read only; must not overlap cache
 *   idx        int32 [n_rows], device memory, distinct destination tokens, not
 *              overlapping cache (CS_ERR_INVALID_ARG);
 *              0 <= idx[r] < T is checked on the device: a row outside is
 *              skipped and cs_sync_status then returns CS_ERR_DEVICE_ARG
 *   row_elems  elements of one token row, e.g. n_kv_heads * head_dim; the row
 *              bytes, both layer strides in bytes and both pointers must be
 *              multiples of 16
 * Call once for the keys and once for the values.  Asynchronous on `stream`.
 */
cs_status cs_scatter_rows(void *cache, const void *rows, cs_dtype dtype, int n_layers, int T,
                          int64_t cache_layer_stride, int n_rows, int64_t rows_layer_stride,
                          int row_elems, const int32_t *idx, void *stream);

/*
 * Takes the device status record of the current device and waits for `stream`:
 * CS_ERR_TIMEOUT or CS_ERR_DEVICE_ARG if a kernel recorded an error since the
 * last take, CS_ERR_CUDA if the stream reported an error, else CS_OK.
 *
 * The record is device-wide: it holds the first error recorded by any kernel
 * of this library on the device, on any stream, until it is taken.  The take
 * runs on the device in `stream`'s order (one atomic exchange with zero), so
 * it covers every kernel issued earlier on `stream`; an error recorded
 * concurrently by a kernel on another stream is either taken by this call
 * (and reported here, against this stream) or left for the next call, never
 * lost.  Calls from several host threads are serialised.
 */
cs_status cs_sync_status(void *stream);

/* Diagnostics: launches one kernel that waits, through the same bounded wait
 * the attention kernel uses, on a barrier that nothing completes, giving up
 * after about `limit_us` microseconds.  cs_sync_status() then returns
 * CS_ERR_TIMEOUT.  Used to test failure detection without faulting a GPU. */
cs_status cs_debug_wait_timeout(uint32_t limit_us, void *stream);

/* Static description of a status code. */
const char *cs_status_string(cs_status s);

/* Detail of the last non-OK status returned on the calling host thread
 * (which argument failed, or the CUDA error string).  Never NULL. */
const char *cs_last_error_detail(void);

#ifdef __cplusplus
}
#endif

#endif /* CHRONOSTITCH_H */
