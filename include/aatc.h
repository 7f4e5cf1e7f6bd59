/*
 * aatc.h -- C ABI of the GB300 (sm_103a) hot path of Attention-Aware Transform Coding
 * (AATC, arxiv 2608.14191, "KV Cache Compression Through the Lens of Transform Coding").
 *
 * The problem the library solves (Sec. 3.2 KV cache, Sec. 5, Algorithm 1): calibrate a
 * per-layer, per-kv-head orthonormal transform and a per-channel bit allocation offline,
 * then, online, append each new key/value head-vector to a packed cache in transform
 * coordinates and run single-token decode attention directly over that packed cache.
 *
 * Conventions shared by every call:
 *   - head_dim d is 128.  A *stream* is one (layer, kv-head, K|V) triple; streams are
 *     indexed s = (layer * n_kv_heads + kv_head) * 2 + kind with kind 0 = keys, 1 = values.
 *   - Pointers documented as "device" must be CUDA device memory of the current device;
 *     "host" pointers are ordinary host memory.  The library never takes ownership of
 *     caller memory and never frees it.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).  All
 *     device work is enqueued on it asynchronously; only aatc_plan_create,
 *     aatc_plan_destroy and aatc_get_device_error synchronize.
 *   - Argument errors are detected on the host before any launch; the call then returns a
 *     non-zero status and leaves all outputs untouched.  A failed launch returns
 *     AATC_ERR_CUDA (see aatc_last_cuda_error).
 *   - No call allocates device memory except aatc_plan_create.
 */
#ifndef AATC_H
#define AATC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define AATC_HEAD_DIM 128
#define AATC_MAX_BITS 16       /* widest channel code a device plan holds; widths 0..AATC_MAX_BITS */
#define AATC_MAX_PLAN_BITS 16  /* widest width the host planner allocates (Sec. 5 allows b in 0..16) */

typedef struct aatc_plan_s* aatc_plan_t;   /* opaque; immutable after creation */

typedef enum {
  AATC_OK = 0,
  AATC_ERR_INVALID_ARG = 1,   /* null pointer, bad shape, out-of-range index            */
  AATC_ERR_BUDGET = 2,        /* bit budget not representable (e.g. > b_max * d)        */
  AATC_ERR_CAPACITY = 3,      /* token range exceeds the cache capacity                  */
  AATC_ERR_WORKSPACE = 4,     /* caller workspace smaller than the required size         */
  AATC_ERR_UNSUPPORTED = 5,   /* shape the kernels do not implement (e.g. GQA group > 8) */
  AATC_ERR_CUDA = 6,          /* a CUDA runtime call or kernel launch failed             */
  AATC_ERR_NOMEM = 7,         /* host or device allocation failed                        */
  AATC_ERR_DEVICE_FLAG = 8,   /* reserved for callers that turn device flags into status */
  AATC_ERR_IO = 9             /* plan file missing, unreadable, short, corrupt or another version */
} aatc_status_t;

/* Model dimensions.  d must be 128; n_q_heads % n_kv_heads == 0; b_max in 1..AATC_MAX_PLAN_BITS for
 * the host planner calls and in 1..AATC_MAX_BITS for aatc_plan_create (the paper's range
 * b in 0..16 of Sec. 6 for both). */
typedef struct {
  int32_t d;
  int32_t n_layers;
  int32_t n_kv_heads;
  int32_t n_q_heads;
  int32_t b_max;
} aatc_dims_t;

/* Human-readable name of a status code (static string). */
const char* aatc_status_string(aatc_status_t status);

/* cudaError_t value of the most recent AATC_ERR_CUDA on this thread (0 if none). */
int32_t aatc_last_cuda_error(void);

/* Library ABI version (major * 10000 + minor * 100 + patch). */
int32_t aatc_version(void);

/*
 * Offline calibration (host only, no GPU needed) -- Sec. 5 Steps 1-2 and the calibration
 * half of Algorithm 1, with the PCA eigenbasis of the calibration keys/values standing in
 * for the whitening-SVD transform (equivalent by the appendix Proposition).  Per stream:
 *   C = X^T X / N (uncentered second moment); C = U diag(sigma^2) U^T by cyclic Jacobi in
 *   fp64 (eigenvalues descending; each eigenvector's largest |entry| made positive, lowest
 *   index on ties); weights w^K_c = sum over the group's query heads of mean_i (u_c . q_i)^2
 *   (Eq. waterfilling-keys and its GQA remark), w^V_c = 1 (W_O = I);  g_c = w_c sigma_c^2;
 *   channels re-sorted by g descending (stable); integer reverse water-filling
 *   min sum_c g_c 4^-b_c s.t. sum_c b_c = round(avg_bits * d), b_c in 0..b_max (exact greedy;
 *   ties to the lower index); s_c = 99th percentile of |u_c . x| (linear interpolation at
 *   rank 0.99 (N - 1)).
 *
 *   calib_k, calib_v : host fp32 [n_layers][n_kv_heads][n_calib][128]
 *   calib_q          : host fp32 [n_layers][n_q_heads][n_calib_q][128], or NULL (then w^K = 1)
 *   avg_bits_k/v     : average code bits per channel; avg * 128 must be an integer
 *   weights_mode     : 0 = attention-aware (AATC), 1 = variance only (AATC var-only, Sec. 6)
 *   basis_out        : host fp32 [L][H_kv][2][128 (input dim)][128 (channel, storage order)]
 *   bits_out         : host uint8 [L][H_kv][2][128], non-increasing along storage order
 *   scales_out       : host fp32 [L][H_kv][2][128]
 *   sigma2_out, weights_out : host fp64 [L][H_kv][2][128] or NULL (diagnostics)
 *   n_threads        : host worker threads (0 = hardware concurrency)
 * Errors: AATC_ERR_INVALID_ARG (null/shape), AATC_ERR_BUDGET (avg*128 not integral or >
 * b_max*128 or < 0).
 */
aatc_status_t aatc_calibrate(const aatc_dims_t* dims, const float* calib_k, const float* calib_v,
                             int32_t n_calib, const float* calib_q, int32_t n_calib_q,
                             double avg_bits_k, double avg_bits_v, int32_t weights_mode,
                             float* basis_out, uint8_t* bits_out, float* scales_out,
                             double* sigma2_out, double* weights_out, int32_t n_threads);

/*
 * Head-group calibration (Sec. 5 Step 1, remark on multi-head attention: the heads of a group
 * share one transform).  The g_h kv-heads of a group are concatenated into vectors of width
 * d = 128 g_h; the planner computes one PCA basis over them (uncentered second moment, Jacobi,
 * descending eigenvalues, canonical signs), the weights w^K_c = sum over the group's query heads j
 * of u_c[block(j)]^T M_j u_c[block(j)] (query head j belongs to kv-head j / group and its score
 * sees only that kv-head's 128-dim block; M_j = mean q q^T of its calibration queries), or w = 1
 * for values / var-only, the exact integer reverse water-filling over the d channels with budget
 * avg_bits * d, b in {0..b_max}, and one P99 scale per channel.  Channels are returned in storage
 * order (g = w sigma^2 descending), so the widths are non-increasing.
 *   calib      : host fp32 [g_h][n_calib][128], the group's kv-heads on the same tokens
 *   calib_q    : host fp32 [g_h * group][n_calib_q][128] in kv-head order, or NULL (values)
 *   basis_out  : host fp32 [d][d] (dim x channel); bits_out uint8 [d]; scales_out fp32 [d];
 *   sigma2_out, weights_out : host fp64 [d] or NULL
 * Errors: AATC_ERR_INVALID_ARG (g_h outside 1..8, group < 1, n_calib < 2, null outputs, b_max
 * outside 1..AATC_MAX_PLAN_BITS), AATC_ERR_BUDGET (avg_bits * d not an integer in [0, b_max d]).
 * Host only.
 * aatc_group_plan_create builds the device plan from these outputs.
 */
aatc_status_t aatc_calibrate_head_group(int32_t g_h, int32_t group, const float* calib, int32_t n_calib,
                                        const float* calib_q, int32_t n_calib_q, double avg_bits, int32_t b_max,
                                        int32_t weights_mode, float* basis_out, uint8_t* bits_out,
                                        float* scales_out, double* sigma2_out, double* weights_out);

/*
 * Global cross-layer bit allocation (Sec. 5 "waterfilling problem for the keys / values" summed
 * over layers; Algorithm 1, global reverse water-filling over every (layer, channel) pair;
 * the experimental-setup paragraph on AATC for the normalisation and the protected layers).
 * Replaces the per-stream budgets of aatc_calibrate with one pool per kind (keys, values):
 *   - layers l < n_protect get a per-stream allocation with avg_bits_v * 128 bits for values and
 *     avg_bits_k * 128 + 128 (one bit per channel more, capped at b_max * 128) for keys;
 *   - the rest of the kind's total budget (avg_bits * 128 * n_layers * n_kv_heads) is allocated
 *     over all channels of all other layers and kv-heads at once, by exact integer reverse
 *     water-filling on g = (sigma2 / P95_l(sigma2)) * (w / P95_l(w)), where P95_l is the 95th
 *     percentile (linear interpolation) over layer l's channels of every kv-head;
 *   - b in {0..b_max}; marginal-gain greedy, ties to the lower (layer, kv-head, channel) index.
 *   sigma2, weights : host fp64 [L][H_kv][2][128] in storage order, as aatc_calibrate writes them
 *   bits_out        : host uint8 [L][H_kv][2][128]; per stream non-increasing (the order of g
 *                     within a stream is unchanged by the per-layer normalisation), so it can be
 *                     passed to aatc_plan_create with aatc_calibrate's basis and scales.
 * Errors: AATC_ERR_INVALID_ARG (null, negative or non-finite inputs), AATC_ERR_BUDGET (avg bits
 * not a multiple of 1/128, or the protected layers need more than the total budget, or the rest
 * exceeds b_max on every pooled channel).  Host only; no device work.
 */
aatc_status_t aatc_allocate_global(const aatc_dims_t* dims, const double* sigma2, const double* weights,
                                   double avg_bits_k, double avg_bits_v, int32_t n_protect, uint8_t* bits_out);

/*
 * Transform from the model weights (Sec. 5 Step 1 "Whitening-Based Feature Decorrelation", Eq.
 * AB-factorization; Appendix Proposition).  For one head's projection W (d_model x 128) and
 * calibration activations X (n x d_model) it returns the paper's factorization W = A B of the
 * whitened SVD W~ = L^T W = U S P^T (Sigma_X = X^T X / n = L L^T): A = L^-T U sqrt(S),
 * B = sqrt(S) P^T.  Computed without forming L: W~^T W~ = W^T Sigma_X W = K^T K / n for K = X W,
 * so P and S^2 are the eigenvectors / eigenvalues of K^T K / n (fp64 Jacobi, descending, each
 * column's largest-|entry| positive, U flipped alike) and A = W P S^-1/2 (U = W~ P S^-1).
 *   x        : host fp32 [n][d_model] calibration activations
 *   w        : host fp32 [d_model][128] one head's key or value projection
 *   a_out    : host fp32 [d_model][128] or NULL      b_out : host fp32 [128][128] or NULL
 *   s_out    : host fp64 [128] singular values (descending) or NULL
 *   p_out    : host fp32 [128 input dim][128 channel] right singular vectors or NULL
 *   ahat_out : host fp32 [d_model][128] = A sqrt(S) = W P or NULL (the hidden-state encode
 *              matrix: per-column positive rescaling leaves allocation and codes unchanged)
 * Errors: AATC_ERR_INVALID_ARG (null x or w, n < 1, d_model < 1, non-finite input, or a zero
 * singular value: W~ must have full column rank).  Host only.
 */
aatc_status_t aatc_whitening_transform(int32_t d_model, int32_t n, const float* x, const float* w,
                                       float* a_out, float* b_out, double* s_out, float* p_out,
                                       float* ahat_out);

/*
 * Encode operand for caching the coefficients straight from the hidden state (Sec. 5 Step 1:
 * H = X A is cached instead of K = X W).  With the plan's orthonormal basis U_s (= P of
 * aatc_whitening_transform for that head, in storage order) the coefficients of k = x W_s are
 * x (W_s U_s); this writes (W_s U_s)^T rounded to bf16 (round to nearest even), the K-major B
 * operand of aatc_encode_hidden.
 *   w_k, w_v : host fp32 [L][d_model][n_kv_heads * 128] key / value projections (head h owns
 *              columns 128 h .. 128 h + 127)
 *   basis    : host fp32 [L][n_kv][2][128][128] as aatc_calibrate writes it
 *   out      : host bf16 bits [L][n_kv][2][128 channel][d_model]
 * Errors: AATC_ERR_INVALID_ARG (invalid dims, d_model not a positive multiple of 64, null,
 * non-finite result).  Host only.
 */
aatc_status_t aatc_hidden_operand(const aatc_dims_t* dims, int32_t d_model, const float* w_k,
                                  const float* w_v, const float* basis, uint16_t* out);

/*
 * Plan files (calibration is offline and once per model, Algorithm 1's first half): the host
 * arrays a plan is made of, written to and read from a versioned little-endian file with a
 * checksum, so aatc_plan_create can rebuild the plan without recalibrating.
 *   aatc_plan_save      : dims (planner range, b_max up to AATC_MAX_PLAN_BITS), basis fp32
 *                         [L][H_kv][2][128][128], bits uint8 [L][H_kv][2][128] (<= b_max),
 *                         scales fp32 [L][H_kv][2][128], all host; bit-exact copies are stored.
 *   aatc_plan_file_dims : the dims of a file (to size the load buffers).
 *   aatc_plan_load      : fills caller-owned host buffers of those sizes; `dims` must equal the
 *                         file's dims.
 * Errors: AATC_ERR_INVALID_ARG (null, invalid dims, bits > b_max on save, dims that differ from
 * the file's on load), AATC_ERR_IO (file cannot be opened or written; wrong magic, version or
 * sizes; trailing bytes; checksum mismatch).  Host only; no device work.
 */
aatc_status_t aatc_plan_save(const char* path, const aatc_dims_t* dims, const float* basis, const uint8_t* bits,
                             const float* scales);
aatc_status_t aatc_plan_file_dims(const char* path, aatc_dims_t* dims_out);
aatc_status_t aatc_plan_load(const char* path, const aatc_dims_t* dims, float* basis_out, uint8_t* bits_out,
                             float* scales_out);

/*
 * Build an immutable device plan from basis / bits / scales in the layouts aatc_calibrate
 * writes (Algorithm 1 outputs).  Derives per stream: R = #{b_c >= 1}, bit offsets, the
 * record length W = ceil(max_s sum_c b_c / 32) words (plan-wide), f_c = s_c 2^(1-b_c), the
 * bf16 encode basis (round-to-nearest-even of `basis`), and uploads everything with one
 * copy on `stream`, then synchronizes it.  Host inputs are copied; the caller keeps them.
 * Errors: AATC_ERR_INVALID_ARG (null, bits > b_max, bits not non-increasing, scale <= 0 or
 * non-finite where bits > 0, non-finite basis), AATC_ERR_UNSUPPORTED (dims->b_max above
 * AATC_MAX_BITS, or a stream with more than 32 channels wider than 8 bits: the encode keeps
 * the high bytes of the first 32 stored values only), AATC_ERR_CUDA, AATC_ERR_NOMEM.
 * All argument checks run before any CUDA call.
 */
aatc_status_t aatc_plan_create(const aatc_dims_t* dims, const float* basis, const uint8_t* bits,
                               const float* scales, void* stream, aatc_plan_t* plan_out);

/*
 * Build a device plan whose streams are head groups (Sec. 5 Step 1, remark on multi-head
 * attention: the g_h kv-heads of a group share one transform; the paper's Llama setting has two
 * groups of four).  Inputs in the layouts aatc_calibrate_head_group writes, one group stream per
 * (layer, group, K|V), n = 128 g_h:
 *   basis  : host fp32 [L][H_kv / g_h][2][n][n] (dim x channel, channels in storage order)
 *   bits   : host uint8 [L][H_kv / g_h][2][n] non-increasing, each <= dims->b_max
 *   scales : host fp32 [L][H_kv / g_h][2][n]
 * A group stream is kept as g_h slice streams in the plan's and the cache's per-kv-head slots:
 * slot (layer, g g_h + s, kind) holds the group's storage channels s, s + g_h, s + 2 g_h, ...
 * (so every slice keeps non-increasing widths), and one alpha per token (the maximum over all n
 * channels, Sec. 5) is written to every slice's slot.  The cache size is the per-kv-head one for
 * the record length W of the widest slice.  aatc_encode and aatc_decode_attention (and
 * aatc_decode_workspace_bytes, aatc_cache_bytes, aatc_dequantize of the slices) take such a
 * plan: the encode projects the concatenated kv-heads of a group, h = [k_g g_h, ..., k_(g+1) g_h - 1] U,
 * and query head j (kv-head j / group of its group) is embedded at its kv-head's 128-dim block:
 * score (U_K^T q~) . h_hat / sqrt(128), output the block's rows of U_V (sum_t p_t h_hat^V_t).
 * Other entry points (prefill, the sink / window decode, the no-allocation decode, the
 * hidden-state encode) answer AATC_ERR_UNSUPPORTED for a group plan.
 * Errors: AATC_ERR_INVALID_ARG (null, invalid dims, g_h outside 2..8 or not dividing H_kv, bits
 * above b_max or increasing, scale <= 0 or non-finite where bits > 0, non-finite basis),
 * AATC_ERR_UNSUPPORTED (b_max > 8, g_h other than 2 or 4 -- the encode holds all 128 g_h channels
 * of a token tile in the 512 TMEM columns -- or more than 16 query heads per group stream),
 * AATC_ERR_CUDA, AATC_ERR_NOMEM.  All argument checks run before any CUDA call.
 */
aatc_status_t aatc_group_plan_create(const aatc_dims_t* dims, int32_t g_h, const float* basis, const uint8_t* bits,
                                     const float* scales, void* stream, aatc_plan_t* plan_out);

/* Free the plan and its device tables (synchronizes the device).  NULL is a no-op. */
aatc_status_t aatc_plan_destroy(aatc_plan_t plan);

/* Words per packed record (W) and per-stream retained channel counts R (host int32
 * [L][H_kv][2], may be NULL). */
aatc_status_t aatc_plan_info(aatc_plan_t plan, int32_t* n_words, int32_t* retained);

/*
 * Bytes of one layer's packed cache for `batch` sequences of capacity max_tokens:
 *   uint32 words [batch][H_kv][2][n_tiles][W][128], then fp32 alpha [batch][H_kv][2][n_tiles*128],
 *   n_tiles = ceil(max_tokens / 128).  Token t of a sequence lives in tile t/128, lane t%128
 *   (library-defined layout: the paper leaves the storage format open).
 */
aatc_status_t aatc_cache_bytes(aatc_plan_t plan, int32_t batch, int32_t max_tokens, size_t* bytes);

/*
 * Encode (Algorithm 1: "Project", "Append qtz(h)"; quantizer of Sec. 5): for every token and
 * stream, h = U_bf16^T x (bf16 x bf16 -> fp32 on tcgen05 tensor cores), alpha = max over
 * retained channels of |h_c| / s_c (fp32), code_c = clamp(floor(h_c / (alpha f_c) + 1/2),
 * -2^(b-1), 2^(b-1)-1), stored as u = code + 2^(b-1) in b_c-bit fields, LSB first in storage
 * channel order (fields may straddle words; unused bits are written as zero).
 *   K, V   : device bf16 [batch][n_tokens][n_kv_heads][128], contiguous
 *   cache  : device, one layer, sized by aatc_cache_bytes(batch, max_tokens); tokens are written
 *            at positions [start, start + n_tokens) of every sequence; other positions untouched.
 * A non-finite alpha sets device error flag bit 0 (aatc_get_device_error).
 * Errors: AATC_ERR_INVALID_ARG, AATC_ERR_CAPACITY (start + n_tokens > max_tokens), AATC_ERR_CUDA.
 * n_tokens == 0 is a no-op (K, V and cache may then be NULL: nothing is read or written).
 */
aatc_status_t aatc_encode(aatc_plan_t plan, int32_t layer, const void* K, const void* V,
                          int32_t batch, int32_t start, int32_t n_tokens, void* cache,
                          int32_t max_tokens, void* stream);

/*
 * Encode straight from the hidden state (Sec. 5 Step 1: the cache holds H = X A; Algorithm 1
 * "Project" + "Append qtz(h)").  For every kv-head of the layer, key and value coefficients
 * h = x A_hat_s (A_hat_s = W_s U_s from aatc_hidden_operand, so h = k U_s for k = x W_s) are
 * computed on the tensor cores (bf16 x bf16, fp32 accumulate over d_model) and quantized and
 * packed exactly as aatc_encode does, into positions [start, start + n_tokens) of `cache`.
 *   x       : device bf16 [batch][n_tokens][d_model], 16-byte aligned
 *   d_model : multiple of 64, 64 .. 65536
 *   a_hat   : device bf16 [L][n_kv][2][128][d_model] (aatc_hidden_operand's layout), 16-byte aligned
 * Asynchronous on `stream`.  Errors: AATC_ERR_INVALID_ARG (null or unaligned pointers, bad layer,
 * sizes or d_model), AATC_ERR_CAPACITY (start + n_tokens > max_tokens), AATC_ERR_UNSUPPORTED (a
 * plan with a width above 8: this kernel's epilogue packs one byte per stored value),
 * AATC_ERR_CUDA.  n_tokens == 0 is a no-op (x, a_hat and cache may then be NULL).
 */
aatc_status_t aatc_encode_hidden(aatc_plan_t plan, int32_t layer, const void* x, int32_t d_model, const void* a_hat,
                                 int32_t batch, int32_t start, int32_t n_tokens, void* cache, int32_t max_tokens,
                                 void* stream);

/*
 * Prefill attention over the packed cache (Def. sdpa for each row of a chunk of new query tokens,
 * causal; Algorithm 1's reconstruct / attend lines in the transformed space: scores
 * alpha_t (U_K^T q) . (f o code_t) / sqrt(128), output U_V (f o sum_t p_t alpha^V_t code^V_t)).
 * The chunk's own keys and values must already be in the cache (aatc_encode / aatc_encode_hidden).
 *   q         : device bf16 [batch][n_q][n_q_heads][128], the queries of positions
 *               q_start .. q_start + n_q - 1; each attends to cached tokens 0 .. its position
 *   cache     : the packed cache holding tokens [0, n_ctx), q_start + n_q <= n_ctx <= max_tokens
 *   out       : device fp32 [batch][n_q][n_q_heads][128]
 *   workspace : device, >= aatc_prefill_workspace_bytes(batch, n_ctx) (the signed codes of the
 *               context as f16, [batch][n_kv][K|V][ceil(n_ctx/128)*128][128], value tiles stored
 *               transposed as [channel][token] per 128-token tile); contents ignored
 * Query head j reads kv-head j / (n_q_heads / n_kv_heads).  Asynchronous on `stream`.
 * Errors: AATC_ERR_INVALID_ARG (null or unaligned pointers, bad layer or sizes, q_start + n_q >
 * n_ctx), AATC_ERR_CAPACITY (n_ctx > max_tokens), AATC_ERR_WORKSPACE, AATC_ERR_UNSUPPORTED (W > 32,
 * or a width above 12: the codes are tensor-core operands in f16, exact up to |code| = 2048),
 * AATC_ERR_CUDA.
 */
aatc_status_t aatc_prefill_workspace_bytes(aatc_plan_t plan, int32_t batch, int32_t n_ctx, size_t* bytes);
aatc_status_t aatc_prefill_attention(aatc_plan_t plan, int32_t layer, const void* q, int32_t q_start, int32_t n_q,
                                     const void* cache, int32_t batch, int32_t n_ctx, int32_t max_tokens, float* out,
                                     void* workspace, size_t workspace_bytes, void* stream);

/* Device workspace bytes aatc_decode_attention needs for (batch, n_ctx). */
aatc_status_t aatc_decode_workspace_bytes(aatc_plan_t plan, int32_t batch, int32_t n_ctx,
                                          size_t* bytes);

/*
 * Decode attention over the packed cache (Def. sdpa with one query row; Algorithm 1
 * reconstruct/attend lines computed without rebuilding K): per query head j (kv-head
 * j / group), q~ = U_K^T q, s_t = q~ . h_hat^K_t / sqrt(128), a = softmax(s),
 * o_hat = sum_t a_t h_hat^V_t, out = U_V o_hat, with h_hat_c = code_c * (alpha_t f_c).
 * Attends to tokens [0, n_ctx) of each sequence (no mask).  Split-K over the context with a
 * log-sum-exp combine; fp32 accumulation; fp32 output.
 *   q         : device bf16 [batch][n_q_heads][128]
 *   out       : device fp32 [batch][n_q_heads][128]
 *   workspace : device, >= aatc_decode_workspace_bytes(batch, n_ctx), contents ignored
 * Errors: AATC_ERR_INVALID_ARG (n_ctx < 1 ...), AATC_ERR_CAPACITY (n_ctx > max_tokens),
 * AATC_ERR_WORKSPACE, AATC_ERR_UNSUPPORTED (group > 8; or a layer whose record tables exceed what
 * the kernels hold: more than 2048 record entries per stream, per-kv-head tables beyond one SM's
 * 227 KB of shared memory, and for head-group plans more than 24 value tiles of 8 entries per
 * warp -- 48 per value slice at g_h = 4, 96 at g_h = 2 -- or score fragments plus a two-stage
 * record ring beyond 227 KB, about 5 bits on average at g_h = 4; all refused before any launch),
 * AATC_ERR_CUDA.
 */
aatc_status_t aatc_decode_attention(aatc_plan_t plan, int32_t layer, const void* q,
                                    const void* cache, int32_t batch, int32_t n_ctx,
                                    int32_t max_tokens, float* out, void* workspace,
                                    size_t workspace_bytes, void* stream);

/*
 * Decode attention over a packed range plus uncompressed tokens in one softmax: the paper's
 * inference policy keeps the first tokens (attention sink) and a recent window in full
 * precision and compresses the rest (Sec. 6 setup: 4 sink tokens, a 128-token window moved in
 * steps of 16).  Per query head j, the scores of the packed tokens [t_first, t_end) of each
 * sequence are computed as in aatc_decode_attention, the scores of the n_full uncompressed
 * tokens as q . k / sqrt(128), and a = softmax over both sets; out = U_V sum_packed a_t h_hat^V_t
 * + sum_full a_t v_t.  The order of the uncompressed tokens is irrelevant.
 *   q       : device bf16 [batch][n_q_heads][128]
 *   cache   : packed cache as written by aatc_encode; only [t_first, t_end) is read
 *   k_full, v_full : device bf16 [batch][full_cap][n_kv_heads][128]; the first n_full tokens of
 *             each sequence are attended (n_full may be 0; k_full/v_full may then be NULL).
 *             full_cap is the row stride between sequences, so the pointers may point at any
 *             row of a larger per-sequence buffer as long as every sequence's n_full rows lie
 *             inside it (a sink / window block kept in place inside a ring-like buffer).
 *   out     : device fp32 [batch][n_q_heads][128]
 *   workspace : as for aatc_decode_attention with n_ctx = t_end (not read when t_first == t_end)
 * Errors: AATC_ERR_INVALID_ARG (t_first > t_end, both sets empty, full_cap < n_full, unaligned
 * pointers, ...), AATC_ERR_CAPACITY (t_end > max_tokens or n_full > 8192), AATC_ERR_WORKSPACE,
 * AATC_ERR_UNSUPPORTED (group > 8), AATC_ERR_CUDA.
 */
aatc_status_t aatc_decode_attention_sw(aatc_plan_t plan, int32_t layer, const void* q, const void* cache,
                                       int32_t batch, int32_t t_first, int32_t t_end, int32_t max_tokens,
                                       const void* k_full, const void* v_full, int32_t n_full, int32_t full_cap,
                                       float* out, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Test hook: dequantized coefficients h_hat_c = fl32(code_c * fl32(alpha_t * f_c)) (zero for
 * dropped channels) of tokens [t0, t0 + n) of every sequence.
 *   coeffs_out : device fp32 [batch][n][n_kv_heads][2][128]
 */
aatc_status_t aatc_dequantize(aatc_plan_t plan, int32_t layer, const void* cache, int32_t batch,
                              int32_t t0, int32_t n, int32_t max_tokens, float* coeffs_out,
                              void* stream);

/*
 * Test hook for failure detection without a GPU fault: launches one CTA that waits on an mbarrier
 * nothing arrives on, with the bounded wait every kernel of this library uses, limited to
 * limit_us microseconds.  The wait runs out, the kernel sets bit 1 (value 2) of *dev_flags (a
 * device int32 the caller zeroes) as the library's kernels do on a timeout, and returns normally.
 * Errors: AATC_ERR_INVALID_ARG (null flags, limit outside 1 .. 2 000 000 us), AATC_ERR_CUDA.
 */
aatc_status_t aatc_selftest_bounded_wait(int32_t limit_us, int32_t* dev_flags, void* stream);

/* Sticky device error flags of the plan (bit 0: non-finite token scale seen by encode;
 * bit 1: a bounded wait inside a kernel timed out).  Synchronizes; clear != 0 resets them. */
aatc_status_t aatc_get_device_error(aatc_plan_t plan, int32_t* flags, int32_t clear);

/*
 * Size of the fixed scratch array behind aatc_decode_attention_noalloc (split partials).
 */
#define AATC_NOALLOC_SCRATCH_BYTES (4u << 20)

/*
 * aatc_decode_attention without a caller workspace.  The paper has no counterpart: this entry
 * point exists for callers that cannot allocate device memory when they call -- for example a
 * serving runtime that carves up all device memory once at start-up with its own pool and may
 * not call cudaMalloc on the request path (it would synchronize the device and stall other
 * streams), or plugin code running inside a framework that does not expose its allocator.
 * Same arguments, math and outputs as aatc_decode_attention; the split partials go to a fixed
 * scratch array of AATC_NOALLOC_SCRATCH_BYTES that the library keeps in device memory on every
 * GPU that loads it, until the process exits.  Nothing is allocated or freed by this call.
 *   - The first call on a device looks up that device's scratch address (with the device
 *     current); make that first call before any stream capture.
 *   - Call with the plan's device current: the array used is the current device's, so a call
 *     made with another device current returns AATC_ERR_INVALID_ARG before any launch.
 *   - Every call on a device shares the one array, and it keeps the previous call's contents.
 *     Nothing in it has to start at zero (each partial is written before it is read), but
 *     calls that overlap on the GPU (different streams, or concurrent host threads) race on it:
 *     serialize them.
 * Errors: as aatc_decode_attention, plus AATC_ERR_WORKSPACE when (batch, n_ctx) needs more
 * than AATC_NOALLOC_SCRATCH_BYTES of partials (see aatc_decode_workspace_bytes).
 */
aatc_status_t aatc_decode_attention_noalloc(aatc_plan_t plan, int32_t layer, const void* q,
                                            const void* cache, int32_t batch, int32_t n_ctx,
                                            int32_t max_tokens, float* out, void* stream);

/*
 * Reference point: uncompressed bf16 decode attention (Def. sdpa), split-K with the same
 * combine.  K, V: device bf16 [batch][max_tokens][n_kv_heads][128]; attends to [0, n_ctx).
 * q: device bf16 [batch][n_q_heads][128]; out: device fp32 [batch][n_q_heads][128].
 */
aatc_status_t aatc_bf16_decode_workspace_bytes(int32_t batch, int32_t n_kv_heads,
                                               int32_t n_q_heads, int32_t n_ctx, size_t* bytes);
aatc_status_t aatc_bf16_decode_attention(const void* K, const void* V, const void* q,
                                         int32_t batch, int32_t n_ctx, int32_t max_tokens,
                                         int32_t n_kv_heads, int32_t n_q_heads, float* out,
                                         void* workspace, size_t workspace_bytes, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* AATC_H */
