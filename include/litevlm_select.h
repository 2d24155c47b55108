/*
 * litevlm_select.h -- C-ABI of the GB300 (sm_103a) token-selection library.
 *
 * The library implements the Token Selection Module of LiteVLM (arXiv
 * 2506.07416, Design section, "Token Selection Module"): before the LLM prefill,
 * every visual token is scored by the softmax attention it receives from the
 * request's text tokens in the first decoder layer (FastV-style attention-score
 * pruning, Related Work), the top-k tokens of each request are kept (ratio r,
 * Results section, "Visual Token Compression"; Table 1 token counts), and the
 * kept hidden / K / V rows are gathered, in their original order, into a
 * shorter ragged sequence for the prefill.
 *
 * Score definition (for request b with N_b visual and T_b text tokens, Hq query
 * heads, Hkv key heads, G = Hq / Hkv, head dimension d):
 *     s[h][i][j] = q_scale * k_scale * (q[i,h,:] . k[j, h / G, :]) / sqrt(d)
 *     score[j]   = (1 / (Hq * T_b)) * sum_h sum_i softmax_j(s[h][i][:])[j]
 * The softmax runs over the request's visual tokens only; every text token of
 * the request is a query; no causal mask (text follows the image).
 * Top-k order: score descending, then token index ascending (the lower index
 * wins a tie); NaN ranks below every number, -0 equals +0.
 * k_b = keep_k[b], or floor((double)keep_ratio * N_b) when no keep_k is given.
 *
 * Conventions for every call:
 *   - Pointers named *_d and all tensor pointers are DEVICE pointers; *_h are
 *     HOST pointers. The caller owns all of them; the library keeps none after
 *     the call returns.
 *   - Layouts are row-major and contiguous:
 *       q        [sum_b T_b, Hq,  d]   bf16, or e4m3 codes (uint8)
 *       k        [sum_b N_b, Hkv, d]   same element type as q
 *       offsets  int32 [batch + 1], offsets[0] = 0, non-decreasing
 *   - Work is enqueued on `stream` (a cudaStream_t) and runs asynchronously;
 *     a call returns after enqueueing. Host-side validation happens before any
 *     work is enqueued; on error nothing is enqueued.
 *   - The *_h offset arrays must hold the same values as their *_d mirrors;
 *     they are read on the host for validation and sizing, and for small
 *     batches the kernels take them by value (launch parameters) instead of
 *     loading the device arrays. Mirrors that disagree are undefined behaviour.
 *   - Every function returns a status and never aborts the process. The text
 *     of the last error of a handle is available from litevlm_select_last_error.
 *   - A handle is used by one host thread and one stream at a time.
 *   - Hot calls (score, topk, compact) allocate nothing; the workspace is
 *     allocated once by create and freed by destroy.
 */
#ifndef LITEVLM_SELECT_H
#define LITEVLM_SELECT_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st* litevlm_stream_t;

typedef enum {
    LITEVLM_OK = 0,
    LITEVLM_ERR_INVALID_ARG = 1,  /* bad pointer, size, offsets, k, ratio or scale */
    LITEVLM_ERR_UNSUPPORTED = 2,  /* valid but outside what the kernels implement */
    LITEVLM_ERR_WORKSPACE = 3,    /* batch or totals beyond the maxima given to create */
    LITEVLM_ERR_CUDA = 4,         /* a CUDA runtime/driver call failed */
    LITEVLM_ERR_TIMEOUT = 5,      /* a device-side bounded wait gave up (from check_device) */
    LITEVLM_ERR_DEVICE_BOUNDS = 6 /* a kernel found an index outside its buffer and skipped it */
} litevlm_status_t;

typedef enum {
    LITEVLM_BF16 = 0,     /* q and k are bfloat16 */
    LITEVLM_FP8_E4M3 = 1  /* q and k are OCP e4m3 codes with one float scale per tensor */
} litevlm_dtype_t;

/* Score-kernel selection (litevlm_select_config_t.flags). By default the
 * library picks the kernel and launch shape from the batch's sizes. */
#define LITEVLM_FLAG_SCORE_REREAD 1   /* always use the kernel that streams K twice per head */
#define LITEVLM_FLAG_SCORE_RESIDENT 2 /* use the TMEM-resident kernel whenever the shapes allow it */
#define LITEVLM_FLAG_SCORE_RESIDENT_ONE_BUFFER 8 /* the same, with one TMEM head buffer only (no head overlap) */
#define LITEVLM_FLAG_SCORE_RESIDENT_TWO_BUFFERS 16 /* the same, two TMEM head buffers where the shapes allow it */
#define LITEVLM_FLAG_SCORE_RESIDENT_FLAT 64 /* the same, one buffer, with the flattened (request, head) schedule
                                               whenever every request has the same token counts */
/* OR-ed with the above: resident plans for requests of more than 64 text
 * tokens run each query head's text rows as two pseudo-heads (the first
 * ceil(T/2) rows, then the rest) on the 64-row kernel, which reads the head's
 * K tiles once per half (the second time from L2). The sums over heads and
 * text rows are unchanged by the split (each text row's softmax is its own).
 * Off by default: on GB300 it measured slower than the re-read kernel on the
 * shapes tried (a 6144-token request with 128 text rows and 28 / 4 heads; a
 * ragged e4m3 batch of 32 requests). Not with LITEVLM_FLAG_QUERY_LAST_TOKEN. */
#define LITEVLM_FLAG_SCORE_SPLIT_QUERIES 128
/* OR-ed with at most one of the above: only the last text token of each request
 * is a query, T_b counts as 1 in the mean (the last-token variant of attention-
 * score pruning, Related Work / FastV). Requests may then have more than 128
 * text tokens. */
#define LITEVLM_FLAG_QUERY_LAST_TOKEN 32

typedef struct {
    int32_t max_batch;         /* largest batch any call will pass */
    int64_t max_total_visual;  /* largest sum_b N_b */
    int64_t max_total_text;    /* largest sum_b T_b */
    int32_t num_q_heads;       /* Hq */
    int32_t num_kv_heads;      /* Hkv, Hq % Hkv == 0 */
    int32_t head_dim;          /* d: 64 or 128 for bf16, 128 for e4m3 */
    litevlm_dtype_t qk_dtype;
    int32_t flags;             /* 0 or one LITEVLM_FLAG_SCORE_* kernel value, optionally
                                  | LITEVLM_FLAG_SCORE_SPLIT_QUERIES | LITEVLM_FLAG_QUERY_LAST_TOKEN */
} litevlm_select_config_t;

typedef struct litevlm_select* litevlm_select_t;

/*
 * Creates a handle on the current CUDA device and allocates its workspace
 * (partial-score buffer, error word). Limits: T_b <= 128 text tokens per request,
 * N_b <= 65536 visual tokens per request (both checked per call).
 * Errors: INVALID_ARG for a NULL pointer or an inconsistent config (non-positive
 * sizes, Hq % Hkv != 0, unknown flags); UNSUPPORTED for a head_dim / dtype pair
 * without a kernel; CUDA when the device cannot be used. *out is NULL on error.
 */
litevlm_status_t litevlm_select_create(const litevlm_select_config_t* config, litevlm_select_t* out);

/* Frees the workspace and the handle. NULL is accepted. Not stream-ordered:
 * the caller makes sure no work using the handle is still running. */
litevlm_status_t litevlm_select_destroy(litevlm_select_t handle);

/* Message of the last failed call on this handle ("" if none). Owned by the
 * handle, valid until the next call on it. NULL handle: message of the last
 * failed create in this thread. */
const char* litevlm_select_last_error(litevlm_select_t handle);

/* Number of kernels the last call on this handle enqueued (0 after an error
 * or a call with nothing to do); for counting launches (the score call runs
 * one kernel, two with the full key set). */
int32_t litevlm_select_last_launches(litevlm_select_t handle);

/* Static description of a status code. */
const char* litevlm_status_string(litevlm_status_t status);

/*
 * Visual-token importance scores (steps: logits, per-row softmax statistics,
 * head/query reduction; Design section, Token Selection Module).
 *   batch            number of requests, 0 <= batch <= max_batch
 *   q_text           device, [sum T_b, Hq, d] text-query rows
 *   text_offsets_d/h int32 [batch+1] prefix of T_b
 *   k_vis            device, [sum N_b, Hkv, d] visual key rows
 *   seq_offsets_d/h  int32 [batch+1] prefix of N_b
 *   q_scale, k_scale per-tensor dequantisation scales for e4m3 (> 0, finite);
 *                    must be 1 for bf16
 *   scores           device, float [sum N_b], written for every visual token
 * Requirements: T_b >= 1 whenever N_b >= 1; T_b <= 128; N_b <= 65536;
 * q_text and k_vis 16-byte aligned. The score matrix is never written to memory;
 * a request with N_b = 0 writes nothing.
 */
litevlm_status_t litevlm_select_score(litevlm_select_t handle, int32_t batch,
                                      const void* q_text, const int32_t* text_offsets_d,
                                      const int32_t* text_offsets_h,
                                      const void* k_vis, const int32_t* seq_offsets_d,
                                      const int32_t* seq_offsets_h,
                                      float q_scale, float k_scale, float* scores,
                                      litevlm_stream_t stream);

/*
 * The same scores with the softmax normaliser over the full causal key set of
 * the first decoder layer: the prompt is [system; image; text], so text query
 * i of request b attends to the S_b system keys, the N_b visual keys and the
 * text keys 0..i (causal mask). The probabilities of the visual keys are
 * summed as in litevlm_select_score; a request's scores then add up to its
 * visual attention share (< 1) instead of 1 (Design section, Token Selection
 * Module: self-attention of the first decoder layer).
 *     s[h][i][j] as above, for every key j of [system; visual; text 0..i]
 *     score[j]   = (1 / (Hq * T_b)) * sum_h sum_i exp(s[h][i][j]) / sum_{j'} exp(s[h][i][j']),  j visual
 * Arguments as for litevlm_select_score, plus
 *   k_sys            device, [sum S_b, Hkv, d] system-prompt key rows (may be NULL when sum S_b = 0)
 *   sys_offsets_d/h  int32 [batch+1] prefix of S_b (no limit on S_b)
 *   k_text           device, [sum T_b, Hkv, d] key rows of the text tokens (rows follow text_offsets)
 * k_sys and k_text have the element type and k_scale of k_vis and are 16-byte
 * aligned. With LITEVLM_FLAG_QUERY_LAST_TOKEN the one query (the last text
 * token) sees every system and text key. The extra statistics live in the
 * handle's workspace ([max_total_text][Hq] floats, allocated by create).
 * Errors: those of litevlm_select_score; INVALID_ARG for missing or unaligned
 * k_sys / k_text or bad sys_offsets.
 */
litevlm_status_t litevlm_select_score_full_keys(litevlm_select_t handle, int32_t batch,
                                                const void* q_text, const int32_t* text_offsets_d,
                                                const int32_t* text_offsets_h,
                                                const void* k_vis, const int32_t* seq_offsets_d,
                                                const int32_t* seq_offsets_h,
                                                const void* k_sys, const int32_t* sys_offsets_d,
                                                const int32_t* sys_offsets_h, const void* k_text,
                                                float q_scale, float k_scale, float* scores,
                                                litevlm_stream_t stream);

/*
 * Patch-selection gating, upstream of the scores (Design section, Patch
 * Selection Module: the final score of a camera view is a weighted sum of the
 * lexical-mapping score and the module's logit; the views scoring above a
 * predefined threshold are encoded; Results: 3.5 of 12 patches on average).
 * For request b and view v, in fp32 with no fused multiply-add:
 *     s[b][v] = w_lex * lexical[b][v] + w_logit * logits[b][v];  selected <=> s > threshold
 * When fewer than min_views views pass, the min_views best views are selected
 * instead (score descending, lower view index first, NaN lowest); min_views = 0
 * allows an empty selection. The selection fixes N_b for the score path.
 *   batch             requests, >= 0 (not limited by the handle's maxima)
 *   num_views         V, 1..64 (camera views per request)
 *   lexical, logits   device, float [batch, V]
 *   tokens_per_view_h host, int32 [V] visual tokens each view contributes (>= 0)
 *   w_lex, w_logit, threshold  the gating weights and threshold (threshold not NaN)
 *   view_mask         device, uint8 [batch, V]: 1 = selected
 *   view_offsets      device, int32 [batch+1]: prefix of the selected-view counts
 *   selected_views    device, int32 [sum of selected views] (at most batch*V): view
 *                     indices, ascending within each request
 *   seq_offsets       device, int32 [batch+1]: prefix of N_b = sum of tokens_per_view
 *                     over the selected views (the score path's seq_offsets)
 *   seq_offsets_h     optional host int32 [batch+1]: when given, the call copies
 *                     seq_offsets to it and synchronises the stream before returning
 * Errors: INVALID_ARG for sizes out of range, a NULL pointer, negative token
 * counts, a NaN threshold, or batch * sum(tokens_per_view) beyond int32.
 */
litevlm_status_t litevlm_select_views(litevlm_select_t handle, int32_t batch, int32_t num_views,
                                      const float* lexical, const float* logits,
                                      const int32_t* tokens_per_view_h, float w_lex, float w_logit,
                                      float threshold, int32_t min_views, uint8_t* view_mask,
                                      int32_t* view_offsets, int32_t* selected_views, int32_t* seq_offsets,
                                      int32_t* seq_offsets_h, litevlm_stream_t stream);

/*
 * Layer-0 projection that makes q and k for the scores (Design section: the
 * module is the first decoder layer of the LLM, whose queries and keys are
 * RoPE(W . RMSNorm(x))). Three calls:
 *
 * litevlm_select_fold_norm: w_folded[o][h] = bf16(w[o][h] * gamma[h]) -- the
 * RMSNorm weight folded into the projection weight, once per weight matrix.
 *   w, w_folded  device bf16 [out_features, hidden] (nn.Linear layout: out x in)
 *   gamma        device float [hidden]
 *
 * litevlm_select_rope_table: table[p][j] = (cos a, sin a), a = p * theta_j in
 * fp32 with theta_j = rope_base^(-2j / head_dim) rounded to fp32, for
 * p < max_positions, j < head_dim / 2.
 *   table        device float [max_positions][head_dim / 2][2]; head_dim 64 or 128
 *
 * litevlm_select_project: for each row r of x,
 *     s_r = 1 / sqrt(mean_h x[r][h]^2 + eps)
 *     y[r][o] = s_r * sum_h x[r][h] * w_folded[o][h] + bias[o]
 * then, when head_dim > 0, each head of head_dim outputs is rotated: element
 * j pairs with j + head_dim/2, (y1, y2) -> (y1 cos - y2 sin, y2 cos + y1 sin)
 * with (cos, sin) = table[positions[r]][j]. One tcgen05 contraction per
 * 128 x 256 (or 128) output tile; the row scale, bias and rotation are applied
 * to the fp32 accumulator, which is rounded once: to bf16, or, when
 * out_scale > 0, to the e4m3 code of y / out_scale (round to nearest even,
 * saturating to +-448: a static per-tensor scale as FP8 post-training
 * quantisation calibrates it; the e4m3 score path takes out_scale as q_scale /
 * k_scale).
 *   rows             0 .. 65535 * 128 token rows; hidden a multiple of 8; out_features a multiple of 128
 *   x                device bf16 [rows, hidden];  y device [rows, out_features] bf16, or
 *                    e4m3 codes when out_scale > 0 (= [rows, heads, head_dim], the layout
 *                    litevlm_select_score reads)
 *   out_scale        0: bf16 output; > 0 (finite): e4m3 output of y / out_scale
 *   bias             device float [out_features] or NULL
 *   eps              >= 0
 *   head_dim         0 (no rotation), 64 or 128
 *   positions        device int32 [rows] (with head_dim > 0); a position outside
 *                    [0, max_positions) uses row 0 of the table and sets DEVICE_BOUNDS
 *   rope_table       device, from litevlm_select_rope_table with the same head_dim
 * x, w_folded and y must be 16-byte aligned. Errors: INVALID_ARG / UNSUPPORTED
 * for sizes, pointers or head_dim outside the above.
 */
litevlm_status_t litevlm_select_fold_norm(litevlm_select_t handle, int32_t out_features, int32_t hidden,
                                          const void* w, const float* gamma, void* w_folded,
                                          litevlm_stream_t stream);
litevlm_status_t litevlm_select_rope_table(litevlm_select_t handle, int32_t max_positions, int32_t head_dim,
                                           float rope_base, float* table, litevlm_stream_t stream);
litevlm_status_t litevlm_select_project(litevlm_select_t handle, int64_t rows, int32_t hidden,
                                        int32_t out_features, const void* x, const void* w_folded,
                                        const float* bias, float eps, int32_t head_dim,
                                        const int32_t* positions, const float* rope_table,
                                        int32_t max_positions, float out_scale, void* y,
                                        litevlm_stream_t stream);

/*
 * Per-request top-k (Results section, ratio r of visual tokens kept; Table 1).
 *   scores           device, float [sum N_b]
 *   keep_k_d/h       int32 [batch] tokens to keep per request, 0 <= k_b <= N_b;
 *                    both NULL selects keep_ratio (then k_b = floor((double)keep_ratio * N_b));
 *                    when keep_k_d is given keep_k_h must be given too
 *   keep_ratio       0 <= r <= 1, used only when keep_k is NULL
 *   kept_idx         device, int32 [sum k_b]: global row indices (into the
 *                    sum N_b rows), ascending within each request
 *   out_offsets_d    device, int32 [batch+1] prefix of k_b
 *   out_offsets_h    optional host int32 [batch+1]; filled synchronously from
 *                    the host mirrors before the call returns (sizes the gather)
 * Ties are broken by the lower token index; the result is unique.
 */
litevlm_status_t litevlm_select_topk(litevlm_select_t handle, int32_t batch, const float* scores,
                                     const int32_t* seq_offsets_d, const int32_t* seq_offsets_h,
                                     const int32_t* keep_k_d, const int32_t* keep_k_h, float keep_ratio,
                                     int32_t* kept_idx, int32_t* out_offsets_d, int32_t* out_offsets_h,
                                     litevlm_stream_t stream);

/*
 * Kept-token counts of a batch, on the host, before any device work (Results
 * section, "Visual Token Compression": the ratio r of visual tokens kept;
 * Table 1's token counts follow from rounding r * N_b down). The same numbers
 * litevlm_select_topk writes to out_offsets_h, so a caller can size kept_idx
 * and the gather outputs before it calls topk.
 *   batch          >= 0 (not limited by any handle)
 *   seq_offsets_h  host int32 [batch+1] prefix of N_b
 *   keep_k_h       host int32 [batch] or NULL; NULL selects keep_ratio,
 *                  k_b = floor((double)keep_ratio * N_b)
 *   keep_ratio     0 <= r <= 1, used only when keep_k_h is NULL
 *   out_offsets_h  host int32 [batch+1]: out_offsets_h[b+1] = out_offsets_h[b] + k_b
 * No handle, no CUDA call, nothing enqueued; out_offsets_h is written only when
 * the call succeeds. Errors (message from litevlm_select_last_error(NULL)):
 * INVALID_ARG for a NULL pointer, bad offsets, k_b outside [0, N_b] or r
 * outside [0, 1].
 */
litevlm_status_t litevlm_select_keep_offsets(int32_t batch, const int32_t* seq_offsets_h, const int32_t* keep_k_h,
                                             float keep_ratio, int32_t* out_offsets_h);

/*
 * Gather of the kept rows into the compacted sequence (the LLM prefill input;
 * Design section: the module shortens the LLM input sequence; Speculative
 * Decoding Head: K/V rows feed the KV cache).
 *   kept_idx     device, int32 [total_kept], each in [0, src_rows)
 *   total_kept   rows to copy (out_offsets_h[batch] from topk)
 *   src_rows     rows of every source tensor (sum N_b)
 *   num_tensors  1..8 tensors gathered with the same index list
 *   src, dst     HOST arrays of num_tensors DEVICE pointers; src[t] is
 *                [src_rows, row_bytes[t]], dst[t] is [total_kept, row_bytes[t]].
 *                A src[t] may be the device view of pinned host memory
 *                (litevlm_select_host_view): the kernel then reads the kept
 *                rows over the host link, and no other row crosses it.
 *   row_bytes    HOST array of num_tensors row sizes in bytes (> 0)
 * dst[t][r] = src[t][kept_idx[r]] byte for byte. Rows whose size and pointers are
 * 16-byte aligned move with 128-bit loads and stores; others byte by byte.
 * An index outside [0, src_rows) is skipped on the device and reported by
 * litevlm_select_check_device as LITEVLM_ERR_DEVICE_BOUNDS.
 */
litevlm_status_t litevlm_select_compact(litevlm_select_t handle, int64_t total_kept, const int32_t* kept_idx,
                                        int64_t src_rows, int32_t num_tensors,
                                        const void* const* src, void* const* dst, const int64_t* row_bytes,
                                        litevlm_stream_t stream);

/*
 * Device view of pinned host memory, so that the gather can take its source
 * rows straight from the host (only the kept rows then cross the host link:
 * the score reads every K row, the gather only the kept hidden / K / V rows).
 *   host         HOST pointer into memory from cudaHostAlloc / cudaMallocHost
 *                (or registered with cudaHostRegister as mapped)
 *   device_view  out: the address a kernel uses for `host`
 *                (cudaHostGetDevicePointer; the same address where the host
 *                and the device share one address space)
 * LITEVLM_ERR_INVALID_ARG if the runtime gives the memory no device address
 * (memory that is neither pinned nor mapped, on a system whose GPU does not use
 * the host's page tables); nothing is enqueued. The view stays valid while the
 * memory stays pinned; the caller keeps the host data unchanged until the
 * gather that reads it has finished.
 */
litevlm_status_t litevlm_select_host_view(litevlm_select_t handle, const void* host, void** device_view);


/*
 * Scores and top-k in one call: the outputs of litevlm_select_score (scores)
 * followed by litevlm_select_topk on them, with the arguments of those two
 * calls. When the score launch splits the heads of a request over several
 * CTAs, the top-k kernel adds the head-group partial rows itself (in the same
 * order as the score kernel would, so the scores are bit-identical) instead of
 * the score kernel's ticketed fold, which shortens the critical path of small
 * batches. It does so when batch <= 256, N_b <= 8192 and head groups x the
 * largest N_b <= 32768 (the partial values one top-k CTA reads); otherwise it
 * runs the two calls unchanged.
 */
litevlm_status_t litevlm_select_score_topk(litevlm_select_t handle, int32_t batch,
                                           const void* q_text, const int32_t* text_offsets_d,
                                           const int32_t* text_offsets_h, const void* k_vis,
                                           const int32_t* seq_offsets_d, const int32_t* seq_offsets_h,
                                           float q_scale, float k_scale, float* scores,
                                           const int32_t* keep_k_d, const int32_t* keep_k_h, float keep_ratio,
                                           int32_t* kept_idx, int32_t* out_offsets_d, int32_t* out_offsets_h,
                                           litevlm_stream_t stream);

/*
 * Prefill sequence splice: the shortened LLM input after token selection
 * (Design section: the LLM prefills only the kept visual tokens with the
 * prompt). Request b's output rows are its S_b system rows, then its k_b kept
 * visual rows, then its T_b text rows, each copied byte for byte; its position
 * ids are the rows' positions in the unpruned sequence [system; all N_b
 * visual; text]: system row i -> i, kept visual row of local index j ->
 * S_b + j, text row t -> S_b + N_b + t (pruned tokens leave gaps, the kept ones
 * keep their original rotary positions).
 *   sys_rows         device [sum S_b, row_bytes]; sys_offsets_d/h int32 [batch+1]
 *   vis_rows         device [sum N_b, row_bytes]; seq_offsets_d/h int32 [batch+1]
 *   kept_idx         device int32 [sum k_b] global visual-row indices, ascending
 *                    within each request (litevlm_select_topk's output);
 *                    kept_offsets_d/h int32 [batch+1], k_b <= N_b
 *   txt_rows         device [sum T_b, row_bytes]; text_offsets_d/h int32 [batch+1]
 *   row_bytes        bytes per row (> 0), the same for the three sources
 *   out_rows         device [sum (S_b + k_b + T_b), row_bytes]
 *   out_offsets_d    device int32 [batch+1] = sys_offsets + kept_offsets + text_offsets
 *   out_offsets_h    optional host int32 [batch+1], filled before the call returns
 *   position_ids     device int32 [sum (S_b + k_b + T_b)]
 * Rows move with 128-bit loads and stores when row_bytes and every row
 * pointer are 16-byte aligned, byte by byte otherwise. A kept index outside
 * its request's rows is skipped and reported by litevlm_select_check_device as
 * LITEVLM_ERR_DEVICE_BOUNDS. Host-side checks as for the other calls.
 */
litevlm_status_t litevlm_select_splice(litevlm_select_t handle, int32_t batch, const void* sys_rows,
                                       const int32_t* sys_offsets_d, const int32_t* sys_offsets_h,
                                       const void* vis_rows, const int32_t* seq_offsets_d,
                                       const int32_t* seq_offsets_h, const int32_t* kept_idx,
                                       const int32_t* kept_offsets_d, const int32_t* kept_offsets_h,
                                       const void* txt_rows, const int32_t* text_offsets_d,
                                       const int32_t* text_offsets_h, int64_t row_bytes, void* out_rows,
                                       int32_t* out_offsets_d, int32_t* out_offsets_h, int32_t* position_ids,
                                       litevlm_stream_t stream);

/*
 * Launch shape litevlm_select_score would use for this batch (host only, no
 * device work; the occupancy of a kernel variant is queried once per handle).
 * plan[0] = kernel (1: K re-read per pass; 2: logits resident in tensor
 * memory, one head at a time; 3: the same with two heads in tensor memory, so
 * one head's epilogue overlaps the next head's MMAs and statistics exchange;
 * 4: as 2, with a flattened schedule, for batches whose requests all have the
 * same visual and text token counts: the batch's (request, head) pairs are
 * split evenly over every cluster that fits on the GPU at once, each cluster
 * running its share back to back across request boundaries; 5, 6, 7: as 2,
 * 3, 4 with the query split, so heads count pseudo-heads below),
 * plan[1] = CTAs per thread-block cluster, plan[2] = 128-token tiles per CTA,
 * plan[3] = query-head groups (grid y), or the number of clusters for plan[0]
 * = 4 or 7. plan holds 4 int32.
 * Errors as for litevlm_select_score's host-side checks.
 */
litevlm_status_t litevlm_select_score_plan(litevlm_select_t handle, int32_t batch, const int32_t* text_offsets_h,
                                           const int32_t* seq_offsets_h, int32_t* plan);

/*
 * Synchronises `stream`, then reads and clears the handle's device error word.
 * Returns OK, TIMEOUT (a kernel's bounded wait gave up; its outputs are not
 * valid, and the workspace's fold tickets are reset so the next call starts
 * clean), DEVICE_BOUNDS, or CUDA.
 */
litevlm_status_t litevlm_select_check_device(litevlm_select_t handle, litevlm_stream_t stream);

/*
 * Budget of every device-side wait of the kernels this handle launches, in SM
 * clock cycles (default 4e9, about 2 s at 2 GHz; 0 restores it). A wait that
 * runs past it sets LITEVLM_ERR_TIMEOUT in the handle's error word, its kernel
 * drains the copies and contractions it issued, frees its tensor memory and
 * returns; litevlm_select_check_device then reports TIMEOUT, clears the word
 * and re-arms the fold tickets, and the handle stays usable. No counterpart in
 * the paper: a failure-detection control, used by the tests to make a wait run
 * out on purpose. The results of a call that timed out are not valid.
 * Errors: INVALID_ARG for a NULL handle or cycles < 0.
 */
litevlm_status_t litevlm_select_set_wait_budget(litevlm_select_t handle, int64_t cycles);

/*
 * Debug switches of a handle, for tests of the failure path (no counterpart in
 * the paper). LITEVLM_DEBUG_STALL_SCORE: in the score launches (either score
 * kernel), the TMA producer first waits on an mbarrier that nothing completes, so that
 * wait runs out of the wait budget before any copy or contraction is issued;
 * every other wait of the launch then gives up as well. The launch writes
 * invalid scores, and litevlm_select_check_device reports LITEVLM_ERR_TIMEOUT.
 * Nothing faults, traps or hangs: each wait is bounded by the budget. flags = 0
 * restores normal operation. Errors: INVALID_ARG for a NULL handle or an
 * unknown flag.
 */
#define LITEVLM_DEBUG_STALL_SCORE 1
litevlm_status_t litevlm_select_set_debug_flags(litevlm_select_t handle, int32_t flags);

/*
 * litevlm_select_score without a handle and without allocating anything.
 * The paper has no counterpart: this is an integration entry point.
 *
 * Who needs it: callers that may not allocate device memory when they score,
 * such as an inference engine that plans every buffer when a model is built
 * and gives its plugins no allocator at run time, or a real-time pipeline that
 * forbids allocation after start-up (cudaMalloc can block, synchronise the
 * device, and fail on fragmented memory). These callers cannot create a handle
 * on the hot path.
 *
 * Same computation, arguments and host-side checks as litevlm_select_score.
 * A handle's config is replaced by num_q_heads, num_kv_heads, head_dim and
 * qk_dtype, with the same rules as in litevlm_select_create. The kernel and
 * launch shape are chosen as litevlm_select_score would choose them, except
 * that the flattened schedule (plan[0] = 4) is never used here: its partial
 * rows could exceed the static scratch.
 *
 * Scratch: two static device arrays in this library, one per device:
 * 4 MiB of partial scores and 64 KiB of fold tickets.
 *   - Limit 1: total_visual / 128 + 2 * batch + 2 <= 16384.
 *   - Limit 2: when the chosen launch splits the query heads over G > 1 CTA
 *     groups, G * total_visual <= 1048576.
 *   - A call beyond either limit returns LITEVLM_ERR_WORKSPACE and enqueues
 *     nothing. Limit 1 is checked before any CUDA call.
 *   - A call that splits the heads clears the tickets it uses with
 *     cudaMemsetAsync on `stream`, after every host-side check (a rejected
 *     call enqueues nothing).
 * Calls that overlap on one device (other streams, other host threads) share
 * this scratch and race. Serialise them.
 *
 * err_d: device int32, owned by the caller. Zero it before the first call.
 *   - Kernels OR error bits into it: 1 = a bounded wait gave up, so the scores
 *     are not valid; 4 = a request shape reached the kernel unchecked.
 *   - The library never reads or clears it.
 *
 * First call on a device: the library looks up the addresses of its static
 * arrays with cudaGetSymbolAddress while that device is current. This may
 * load the library's device code onto the device. The library also queries
 * occupancy the first time it uses each kernel variant. Make this first call,
 * with each head_dim / qk_dtype the caller will use, outside any stream
 * capture.
 *
 * Errors: status codes as for litevlm_select_score (device ordinal >= 64:
 * UNSUPPORTED). The message is available from litevlm_select_last_error(NULL)
 * in the calling thread.
 */
litevlm_status_t litevlm_select_score_noalloc(int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                              litevlm_dtype_t qk_dtype, int32_t batch,
                                              const void* q_text, const int32_t* text_offsets_d,
                                              const int32_t* text_offsets_h,
                                              const void* k_vis, const int32_t* seq_offsets_d,
                                              const int32_t* seq_offsets_h,
                                              float q_scale, float k_scale, float* scores, int32_t* err_d,
                                              litevlm_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* LITEVLM_SELECT_H */
