/*
 * avtp.h -- C ABI of the AVTP pruning stage on one NVIDIA GB300 (sm_103a).
 *
 * AVTP (Adaptive Visual Token Pruning for multi-image LVLMs) prunes visual tokens
 * once, at a chosen decoder layer, in four steps:
 *   1. score every visual token              (paper §3.3.1; attention variant §3.3.2)
 *   2. allocate per-image keep budgets       (paper §3.3.3 mean + adaptive ratio, App. A.2 clamps)
 *   3. keep each image's top-k tokens, keep all text, emit ascending positions
 *                                            (paper §3.1 subsequence, §3.3.3)
 *   4. compact the kept rows into a varlen-packed batch (paper §3.1, E_pruned = p(E_v))
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Pointers named as device pointers must point to GPU memory of the current
 *   device; the library reads and writes them only from kernels launched on the
 *   given stream. Host scalars are passed by value or in the argument structs.
 * - The caller owns every buffer. The library never allocates or frees memory:
 *   scratch lives in a caller-provided workspace of avtp_workspace_size() bytes,
 *   256-byte aligned. A workspace may be reused by calls that do not overlap on
 *   the GPU; calls that overlap need separate workspaces.
 * - All compute calls are asynchronous on `stream` (NULL = legacy default stream).
 *   Only avtp_read_device_status() synchronises.
 * - Errors the host can see (null pointers, bad sizes, misalignment, a workspace
 *   that is too small) are returned before anything is launched. Errors only the
 *   device can see (a span outside its request, an out-of-range keep ratio, a
 *   kept index outside [0, T)) are recorded in the workspace's status word; the
 *   affected kernels then skip their work (no trap, no out-of-bounds access) and
 *   avtp_read_device_status() returns the code.
 * - bf16 tensors are row-major with a contiguous last dimension; their base
 *   pointers and row strides must be multiples of 16 bytes.
 * - Layout: varlen-packed requests. Request r owns packed tokens
 *   [cu_seqlens[r], cu_seqlens[r+1]). Its images are entries img_cu[r] ..
 *   img_cu[r+1]-1 of img_start/img_len; a span [img_start, img_start+img_len)
 *   is request-local, at least 1 token long, and the spans of one request are
 *   sorted and disjoint. Every token outside the spans is text and is always kept.
 * - Limits: T < 2^31; at most 2^20 visual tokens and 4096 images per request.
 */
#ifndef AVTP_H_
#define AVTP_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define AVTP_API __attribute__((visibility("default")))
#else
#define AVTP_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t / CUstream. */
typedef struct CUstream_st* avtp_stream_t;

typedef enum {
  AVTP_OK = 0,
  AVTP_ERR_INVALID_ARG = 1,   /* null pointer, negative size, bad enum              */
  AVTP_ERR_UNSUPPORTED = 2,   /* head_dim not 64/128, misaligned rows, Hq % Hkv != 0 */
  AVTP_ERR_RANGE = 3,         /* a size above the documented limits                  */
  AVTP_ERR_CUDA = 4,          /* a CUDA runtime call failed (launch, copy)           */
  AVTP_ERR_TIMEOUT = 5,       /* a bounded device wait gave up (about one second)    */
  AVTP_ERR_DEVICE_INPUT = 6,  /* device-side data failed validation                  */
  AVTP_ERR_WORKSPACE = 7      /* workspace null, misaligned or too small             */
} avtp_status_t;

typedef enum {
  /* I_v = 1 - cos(h^l_v, h^prior_v): hidden-state variation (paper §3.3.1). */
  AVTP_CRIT_HIDDEN_VARIATION = 0,
  /* Mean over heads and text queries of the causal softmax probability that a
   * text query puts on each visual key (the per-token form of the attention
   * quantity of paper §3.3.2). Never materialises the attention matrix. */
  AVTP_CRIT_TEXT_ATTENTION = 1
} avtp_criterion_t;

/* Queries whose attention scores the visual keys under AVTP_CRIT_TEXT_ATTENTION. */
typedef enum {
  AVTP_QUERIES_TEXT = 0,  /* every text token of the request (paper §3.3.2)                     */
  AVTP_QUERIES_LAST = 1   /* the request's last token alone, the token whose output predicts the
                           * first generated token: the attention FAST-V ranks by (paper §4.1) */
} avtp_query_set_t;

/* Where AVTP_CRIT_TEXT_ATTENTION computes its logits. */
typedef enum {
  AVTP_PATH_AUTO = 0,    /* the narrow path for AVTP_QUERIES_LAST and for text query sets of
                          * at most 4 rows per KV group (queries x heads of the group),
                          * tcgen05 otherwise                                                  */
  AVTP_PATH_TENSOR = 1,  /* tcgen05 tensor cores, 256-row blocks (AVTP_QUERIES_TEXT only)     */
  AVTP_PATH_CUDA = 2     /* the narrow path: keys on the M side of warp-level mma.sync, every
                          * key read once, every logit of the request's rows kept in the
                          * workspace (Hq x queries x tokens x 4 bytes per request; more than
                          * 1 GiB in all returns AVTP_ERR_RANGE)                               */
} avtp_attn_path_t;

typedef struct {
  int32_t n_requests;         /* R >= 1 (host scalar)                         */
  int32_t n_images;           /* total images over all requests, >= 0 (host)  */
  int64_t n_tokens;           /* T = cu_seqlens[R] (host)                     */
  const int32_t* cu_seqlens;  /* device [R+1], cu_seqlens[0] = 0, non-decreasing */
  const int32_t* img_cu;      /* device [R+1], img_cu[0] = 0, img_cu[R] = n_images */
  const int32_t* img_start;   /* device [n_images], request-local first token */
  const int32_t* img_len;     /* device [n_images], >= 1                      */
} avtp_layout_t;

typedef struct {
  avtp_criterion_t criterion;
  /* AVTP_CRIT_HIDDEN_VARIATION: h_cur = hidden state at the pruning layer,
   * h_prior = hidden state after the previous pruning (or the input embedding
   * for the first pruning layer), paper §3.3.1. bf16 [T, hidden]; row strides
   * in elements. hidden must be a multiple of 8. */
  const void* h_cur;
  const void* h_prior;
  int32_t hidden;
  int64_t h_cur_stride;
  int64_t h_prior_stride;
  /* AVTP_CRIT_TEXT_ATTENTION: q bf16 [T, n_q_heads, head_dim] (only text rows
   * are read), k bf16 [T, n_kv_heads, head_dim]; token strides in elements.
   * Query head h reads KV head h / (n_q_heads / n_kv_heads). Logits are
   * softmax_scale * q.k. head_dim must be 64 or 128. */
  const void* q;
  const void* k;
  int32_t n_q_heads;
  int32_t n_kv_heads;
  int32_t head_dim;
  int64_t q_stride;
  int64_t k_stride;
  float softmax_scale;
  /* Optional fp32 [n_q_heads, T] (row stride lse_stride elements): the natural-log
   * log-sum-exp of the scaled causal logits of each text query, as kept by a
   * FlashAttention-style forward pass. NULL: the library computes it. */
  const float* lse;
  int64_t lse_stride;
  /* Optional upper bound on the number of text tokens in the whole batch, used
   * only to size the workspace of AVTP_CRIT_TEXT_ATTENTION (it holds the text
   * queries repacked by KV group). 0: n_tokens. A batch with more text tokens
   * than this reports AVTP_ERR_RANGE. */
  int64_t max_text_tokens;
  /* AVTP_CRIT_TEXT_ATTENTION: the query set (avtp_query_set_t) and the path
   * (avtp_attn_path_t); 0 and 0 give every text token and the automatic choice.
   * AVTP_PATH_TENSOR with AVTP_QUERIES_LAST returns AVTP_ERR_UNSUPPORTED. With
   * AVTP_QUERIES_LAST a supplied lse holds the last token's row of each request. */
  int32_t query_set;
  int32_t path;
} avtp_score_args_t;

typedef struct {
  const float* keep_ratio;  /* device [R]: base keep ratio r_base of each request, within
                             * [r_min, r_max] (else AVTP_ERR_DEVICE_INPUT: no shift of the
                             * ratios could meet both the clamps and the request's budget)
                             * and a multiple of 2^-32 (else AVTP_ERR_DEVICE_INPUT) */
  float alpha;              /* variance control alpha of paper §3.3.3, in [0, 1024]; paper uses 1.0 */
  float r_min;              /* ratio clamps of App. A.2: 0 <= r_min <= r_max <= 1; paper uses 0.05 */
  float r_max;              /*                                                        and 0.95.
                             * alpha, r_min and r_max must be multiples of 2^-32 (every fp32
                             * value of at least 2^-9 is one), else AVTP_ERR_RANGE: the rule is
                             * computed exactly, and this bounds its integers */
  int32_t relative;         /* 0: r_i = r_base + alpha*(Ibar_i - Ibar_avg) (paper §3.3.3)
                             * 1: r_i = r_base*(1 + alpha*(Ibar_i/Ibar_avg - 1)), for scores of
                             *    order 1/N such as the text-attention criterion */
} avtp_alloc_args_t;

/* One set of rows to gather: out[j] = in[kept_idx[j]] for j in [0, n_kept).
 * Device pointers; sizes and strides in bytes. Any row size works; rows whose
 * size, strides and pointers are 16-byte multiples take the vectorised path.
 * When n_kept is 0 nothing is read or written, and the pointers may be NULL
 * (an empty output tensor). */
typedef struct {
  const void* in;
  void* out;
  int64_t row_bytes;
  int64_t in_stride;
  int64_t out_stride;
} avtp_rows_t;

#define AVTP_MAX_ROW_SETS 8

/* Bytes of workspace the calls below need for this layout and scoring setup
 * (score_args may be NULL when no scoring call will use the workspace).
 * Returns AVTP_OK and writes *bytes, or an error for invalid arguments. */
AVTP_API avtp_status_t avtp_workspace_size(const avtp_layout_t* layout, const avtp_score_args_t* score_args,
                                  size_t* bytes);

/* Step 1 (paper §3.3.1 / §3.3.2). Writes scores[t] (device fp32 [T]) for every
 * visual token t; entries at text positions are left unchanged. Also writes
 * img_sums (device int64 [n_images]), the fixed-point per-image sums
 * S_i = sum_{t in V_i} rint(fx(scores[t]) * 2^32), fx mapping NaN to 0 and
 * clamping to +-2^10; being integers, they do not depend on summation order. */
AVTP_API avtp_status_t avtp_score(const avtp_layout_t* layout, const avtp_score_args_t* args, float* scores,
                         int64_t* img_sums, void* workspace, size_t workspace_bytes, avtp_stream_t stream);

/* The pruning layer's causal attention forward, with the text-attention criterion as
 * a side output (paper §3.2: FlashAttention-style attention keeps the natural-log
 * normaliser of every query row, which is what the criterion needs; §3.3.2 for the
 * criterion). For every token t and query head h of the batch:
 *   O[t, h]   = sum_u softmax_u(softmax_scale * q[t, h] . k[u, g(h)]) v[u, g(h)]
 *   lse[h, t] = ln sum_u exp(softmax_scale * q[t, h] . k[u, g(h)])
 * over the keys u of t's request with u <= t, g(h) = h / (n_q_heads / n_kv_heads).
 * bf16 tensor-core products with fp32 accumulation; P is rounded to bf16 before P V,
 * as in FlashAttention. */
typedef struct {
  const void* v;       /* device bf16 [T, n_kv_heads, head_dim], token stride v_stride
                        * elements (a multiple of 8), 16-byte aligned                  */
  int64_t v_stride;
  float* o;            /* device fp32 [T, n_q_heads, head_dim], token stride o_stride
                        * elements (a multiple of 4), 16-byte aligned: written          */
  int64_t o_stride;
  float* lse;          /* device fp32 [n_q_heads, T], row stride lse_stride >= T: written */
  int64_t lse_stride;
} avtp_forward_args_t;

/* Workspace bytes of avtp_attn_forward for these arguments (the same checks as the call). */
AVTP_API avtp_status_t avtp_forward_workspace_size(const avtp_layout_t* layout, const avtp_score_args_t* score_args,
                                                   const avtp_forward_args_t* fwd_args, size_t* bytes);

/* Runs the forward above for every token of the batch: q, k, the heads, head_dim,
 * strides and softmax_scale come from score_args (criterion AVTP_CRIT_TEXT_ATTENTION,
 * lse NULL: the forward writes it), v, O and the LSE from fwd_args. When scores and
 * img_sums are non-NULL it then scores the visual tokens as avtp_score does with
 * score_args' query set and path, reading the LSE the forward just wrote: criterion B
 * costs its mass pass (one more Q K^T over the query set and the visual keys) and no
 * pass of its own for the normaliser. The exact per-key mass needs each query's final
 * normaliser, so it cannot be formed inside the forward's own key loop. Both NULL: the
 * plain forward. The layout is validated as in avtp_score; asynchronous on `stream`. */
AVTP_API avtp_status_t avtp_attn_forward(const avtp_layout_t* layout, const avtp_score_args_t* score_args,
                                         const avtp_forward_args_t* fwd_args, float* scores, int64_t* img_sums,
                                         void* workspace, size_t workspace_bytes, avtp_stream_t stream);

/* Diagnostic: per-key-block clock stamps (SM cycles) of the last avtp_attn_forward call's
 * first CTA, the query tile with the most key blocks, head 0, for its first max_blocks (at
 * most 256; the rest of out is left untouched) key blocks. Available in the library's
 * timeline build (compiled with AVTP_TIMELINE); the default build returns
 * AVTP_ERR_UNSUPPORTED. out: host int64 [max_blocks][10]: per block j, from softmax warp 0
 * the loop top, S ready, the half maxima exchanged, the exponentials done and P handed
 * over, then from the MMA-issuing thread S_j's entry and issue and P_j V_j's entry,
 * operands ready and issue. Synchronises the device. */
AVTP_API avtp_status_t avtp_forward_timeline(int64_t* out, int32_t max_blocks);

/* Diagnostic: per-step clock stamps (SM cycles) of the first CTA of criterion B's tensor-core
 * pass `pass` (1: the log-sum-exp pass, 2: the mass pass) in the last avtp_score call that
 * ran it, for the first max_steps (at most 64; the rest of out is left untouched) steps of
 * that CTA's run. Timeline build only
 * (AVTP_TIMELINE); the default build returns AVTP_ERR_UNSUPPORTED. out: host int64
 * [max_steps][6]: the key tile's load issued, the MMA thread at the step, its operands and
 * accumulators ready, its MMAs issued, the step's first accumulator ready for epilogue
 * warp 0, the step's last accumulator released by it. Synchronises the device. */
AVTP_API avtp_status_t avtp_score_timeline(int32_t pass, int64_t* out, int32_t max_steps);

/* Step 2 (paper §3.3.3, App. A.2). From img_sums (device int64 [n_images]) writes
 * budgets (device int32 [n_images]) and out_cu_seqlens (device int32 [R+1]),
 * the packed offsets of the pruned batch. Per request, in exact rational arithmetic:
 *   B_r = floor(r_base*N_vis + 1/2);  Ibar_i = S_i / (2^32 n_i);  Ibar_avg = sum S / (2^32 N_vis);
 *   r_i = r_base + alpha*(Ibar_i - Ibar_avg), or with `relative`
 *   r_i = r_base*(1 + alpha*(Ibar_i/Ibar_avg - 1)) (r_base when sum S = 0);
 *   lambda with sum_i n_i*clamp(r_i + lambda, r_min, r_max) = B_r (every image at the
 *   nearer clamp when B_r lies outside [N_vis*r_min, N_vis*r_max]);
 *   x_i = n_i*clamp(r_i + lambda, r_min, r_max), k_i = floor(x_i), then largest
 *   remainder: one more token for the images with the largest x_i - floor(x_i) (ties
 *   to the lower index) until sum k_i = B_r (a surplus is taken from the smallest
 *   remainders, ties to the higher index).
 * No step rounds: the budgets are those of the exact rule.
 * Every |img_sums[i]| must be at most img_len[i]*2^42 (avtp_score's sums are), and
 * each keep ratio a multiple of 2^-32 (every fp32 value of at least 2^-9 is);
 * otherwise the request's budgets are not written and the call reports
 * AVTP_ERR_DEVICE_INPUT. */
AVTP_API avtp_status_t avtp_allocate(const avtp_layout_t* layout, const int64_t* img_sums, const avtp_alloc_args_t* args,
                            int32_t* budgets, int32_t* out_cu_seqlens, void* workspace, size_t workspace_bytes,
                            avtp_stream_t stream);

/* Step 3 (paper §3.1, §3.3.3). Keeps, in every image i, the budgets[i] visual
 * tokens ranked highest by (score descending, position ascending; NaN lowest,
 * -0 == +0), plus every text token, and writes their packed positions to
 * kept_idx (device int32, capacity n_kept >= out_cu_seqlens[R]) in ascending
 * order. scores: device fp32 [T]; budgets: device int32 [n_images], each in
 * [0, img_len]; out_cu_seqlens: device int32 [R+1] as written by avtp_allocate.
 * A request whose budgets and offsets disagree, or that would write past
 * n_kept, is skipped and recorded as AVTP_ERR_DEVICE_INPUT. */
AVTP_API avtp_status_t avtp_select(const avtp_layout_t* layout, const float* scores, const int32_t* budgets,
                          const int32_t* out_cu_seqlens, int32_t* kept_idx, int64_t n_kept, void* workspace,
                          size_t workspace_bytes, avtp_stream_t stream);

/* avtp_select without a workspace, for callers that cannot allocate device
 * memory where they call it: for example an inference engine that reserves all
 * free HBM for its KV-cache pool up front and gives plugins only their inputs
 * and outputs, or code running where allocation calls are not allowed. The
 * paper has no counterpart to this; it is a deployment convenience.
 * Same inputs, outputs and result as avtp_select. The scratch (about 145 KiB)
 * is a fixed device array inside the library, held by every GPU that loads
 * the library until the process exits. Limits: at most
 * AVTP_NOALLOC_MAX_IMAGES images and AVTP_NOALLOC_MAX_REQUESTS requests;
 * larger layouts return AVTP_ERR_RANGE before anything is launched.
 * Every call looks up the array's device address on the current device
 * (cudaGetSymbolAddress, which allocates nothing); the first call on a device may
 * load the library's GPU module, so make that first call before any stream
 * capture. All calls share the one array, so calls
 * that overlap on the GPU race and must not be issued; calls ordered on one
 * stream are fine, since each call rewrites the scratch it reads.
 * device_status (optional device int32, NULL to skip) receives the device-side
 * status word of this call (an avtp_status_t value). */
#define AVTP_NOALLOC_MAX_IMAGES 16384
#define AVTP_NOALLOC_MAX_REQUESTS 4096
AVTP_API avtp_status_t avtp_select_noalloc(const avtp_layout_t* layout, const float* scores, const int32_t* budgets,
                                           const int32_t* out_cu_seqlens, int32_t* kept_idx, int64_t n_kept,
                                           int32_t* device_status, avtp_stream_t stream);

/* Step 4 (paper §3.1). For each of the n_sets row sets (at most AVTP_MAX_ROW_SETS):
 * out[j] = in[kept_idx[j]] for j < n_kept. Indices outside [0, n_tokens) are
 * skipped and recorded as AVTP_ERR_DEVICE_INPUT. Position ids with P planes
 * (M-RoPE) are passed as P row sets of one element each. */
AVTP_API avtp_status_t avtp_compact(const int32_t* kept_idx, int64_t n_kept, int64_t n_tokens, const avtp_rows_t* sets,
                           int32_t n_sets, void* workspace, size_t workspace_bytes, avtp_stream_t stream);

/* Steps 1-4 fused on one stream. Outputs as in the single steps; scores and
 * img_sums may be NULL (then kept in the workspace). n_kept must equal
 * avtp_kept_count_host() for this layout and these keep ratios. Steps 2 and 3
 * run as one kernel here. The kernels are chained with programmatic dependent
 * launch (set AVTP_PDL=0 in the environment to launch them plainly).
 * step_events (optional, NULL to skip): 5 cudaEvent_t handles recorded on
 * `stream` before the first kernel and after validation, scoring,
 * allocation+selection and compaction, for per-step timing; recording them
 * serialises the kernels, so leave it NULL when timing the whole call. */
AVTP_API avtp_status_t avtp_prune(const avtp_layout_t* layout, const avtp_score_args_t* score_args,
                         const avtp_alloc_args_t* alloc_args, float* scores, int64_t* img_sums, int32_t* budgets,
                         int32_t* out_cu_seqlens, int32_t* kept_idx, int64_t n_kept, const avtp_rows_t* sets,
                         int32_t n_sets, void* workspace, size_t workspace_bytes, void* const* step_events,
                         avtp_stream_t stream);

/* Host-side size of the pruned batch: sum_r floor(keep_ratio[r]*N_vis,r + 0.5) + N_txt,r.
 * Host arrays: cu_seqlens [R+1], img_cu [R+1], img_len [n_images], keep_ratio [R].
 * Returns the count, or -1 for invalid arguments. */
AVTP_API int64_t avtp_kept_count_host(const int32_t* cu_seqlens, const int32_t* img_cu, const int32_t* img_len,
                             const float* keep_ratio, int32_t n_requests);

/* The layout of the batch avtp_prune produced, for running the stage again at a later
 * layer (the progressive schedule of paper §3.3.2, where the compacted hidden states of
 * this pruning point are the next one's h_prior, §3.3.1). Requests and their images
 * stay; image i of request r starts at img_start[i] - sum_{j<i in r} (img_len[j] -
 * budgets[j]) and holds budgets[i] tokens. Writes out_img_start and out_img_len
 * (device int32 [n_images]); the pruned layout is then {n_requests, n_images,
 * n_tokens = n_kept, cu_seqlens = out_cu_seqlens of avtp_prune, the same img_cu,
 * out_img_start, out_img_len}, all on the device, with no host round trip.
 * budgets: device int32 [n_images] as written by avtp_prune or avtp_allocate; a
 * budget outside [0, img_len] is recorded as AVTP_ERR_DEVICE_INPUT and its image gets
 * an empty span. An image that kept no token gets an empty span, which the next
 * stage's validation rejects (with the default clamps every image of 20 or more
 * tokens keeps at least one). Asynchronous on `stream`. */
AVTP_API avtp_status_t avtp_pruned_layout(const avtp_layout_t* layout, const int32_t* budgets, int32_t* out_img_start,
                                          int32_t* out_img_len, void* workspace, size_t workspace_bytes,
                                          avtp_stream_t stream);

/* avtp_kept_count_host from per-request visual token counts (host int32 [R]), for a
 * layout whose image lengths live on the device only, such as one from
 * avtp_pruned_layout. Returns sum_r floor(keep_ratio[r]*n_vis[r] + 0.5) + N_txt,r, or -1
 * for invalid arguments. Optionally (NULL to skip) writes the pruned batch's host
 * offsets out_cu_seqlens [R+1] and its visual counts out_n_vis [R], which are the
 * inputs of the same call for the next stage. */
AVTP_API int64_t avtp_kept_count_vis_host(const int32_t* cu_seqlens, const int32_t* n_vis, const float* keep_ratio,
                                          int32_t n_requests, int32_t* out_cu_seqlens, int32_t* out_n_vis);

/* Pruning-layer selection (paper §3.3.2): the attention a layer assigns to the visual
 * tokens of each sample, A_l^(i) = sum_j Attention(l, v_j), is the sum of the sample
 * request's fixed-point image sums of AVTP_CRIT_TEXT_ATTENTION at that layer (run
 * avtp_score with that layer's q and k). avtp_layer_attention writes that sum, for every
 * request r of the layout, to A[r * n_layers + layer] (device int64 [R, n_layers], units
 * of 2^-32); one call per layer fills one column. img_sums: device int64 [n_images] from
 * avtp_score. The layout is validated as in the other calls (workspace of
 * avtp_workspace_size(layout, NULL) bytes). Asynchronous on `stream`. */
#define AVTP_MAX_LAYERS 1024
AVTP_API avtp_status_t avtp_layer_attention(const avtp_layout_t* layout, const int64_t* img_sums, int64_t* A,
                                            int32_t n_layers, int32_t layer, void* workspace, size_t workspace_bytes,
                                            avtp_stream_t stream);

/* The layer ranking of paper §3.3.2 over n_samples samples and n_layers layers (at most
 * AVTP_MAX_LAYERS): per sample, Rank(A_l^(i)) = 1 for the layer with the most attention
 * (equal values rank the lower layer first); rank_sum[l] = sum_i Rank(A_l^(i)), so the
 * average rank is R_l = rank_sum[l] / n_samples (device int64 [n_layers]); top_layers
 * (device int32 [k], 1 <= k <= n_layers) receives the k layers with the best average
 * rank, best first, ties to the lower layer. A: device int64 [n_samples, n_layers],
 * row-major, as avtp_layer_attention writes it. Exact integer arithmetic. Asynchronous
 * on `stream`. */
AVTP_API avtp_status_t avtp_layer_select(const int64_t* A, int32_t n_samples, int32_t n_layers, int32_t k,
                                         int64_t* rank_sum, int32_t* top_layers, avtp_stream_t stream);

/* Check of the failure path every pipeline kernel takes when a wait on an mbarrier (a
 * TMA copy, a tensor-core commit, a hand-off between warps) does not complete: one CTA
 * of 64 threads waits on a fresh count-1 mbarrier with the library's bounded waits,
 * thread 0 with the single-thread form and warp 1 with the warp-wide form.
 *   arrive != 0: thread 0 arrives first, both waits complete, the status word stays
 *                AVTP_OK.
 *   arrive == 0: nothing arrives; each wait gives up after limit_ns nanoseconds of the
 *                GPU's global timer and the kernel records AVTP_ERR_TIMEOUT in the
 *                status word (detail = 0 or 1, the waiter that recorded first) and
 *                returns. Nothing traps or faults; the context stays usable.
 * The pipeline kernels use a limit of one second. limit_ns in [1000, 10^10];
 * workspace: device, 256-byte aligned, at least 16 bytes (its status word is reset
 * first). Asynchronous on `stream`; read the outcome with avtp_read_device_status(). */
AVTP_API avtp_status_t avtp_wait_selftest(int64_t limit_ns, int32_t arrive, void* workspace, size_t workspace_bytes,
                                          avtp_stream_t stream);

/* Waits for `stream`, then reads the workspace's device status word into *out
 * (an avtp_status_t value; AVTP_OK if no device-side error was recorded since the
 * last entry point reset it). */
AVTP_API avtp_status_t avtp_read_device_status(const void* workspace, avtp_stream_t stream, int32_t* out);

/* Static English text for a status code. */
AVTP_API const char* avtp_status_string(int32_t status);

/* Library version as MAJOR*10000 + MINOR*100 + PATCH. */
AVTP_API int32_t avtp_version(void);

#ifdef __cplusplus
}
#endif

#endif /* AVTP_H_ */
