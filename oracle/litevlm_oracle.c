/*
 * CPU oracle for LiteVLM's Token Selection Module (arXiv 2506.07416).
 *
 * TEST INFRASTRUCTURE ONLY. Only the tests, the package smoke check and the
 * benchmark's CPU-baseline leg may load this library. It shares no code, header,
 * table or helper with the CUDA path; its inputs come from the seeded generator
 * module and from the caller.
 *
 * What it computes (Design section, "Token Selection Module"; Related Work,
 * FastV-style pruning by self-attention scores; Results, "Visual Token
 * Compression", ratio r):
 *
 *   For request b with N_b visual tokens and T_b text tokens, query heads Hq,
 *   key/value heads Hkv (G = Hq / Hkv), head dimension d:
 *     s[h][i][j] = (q[i,h,:] . k[j,g(h),:]) * q_scale * k_scale / sqrt(d),
 *                  g(h) = floor(h / G)
 *     m[h][i]    = max_j s[h][i][j]
 *     l[h][i]    = sum_j exp(s[h][i][j] - m[h][i])
 *     P[h][i][j] = exp(s[h][i][j] - m[h][i]) / l[h][i]
 *     score[j]   = (sum_h sum_i P[h][i][j]) / (Hq * T_b)      (fp64, rounded once to fp32)
 *   k_b = keep_k[b] if given, else floor((double)r * N_b) clamped to [0, N_b].
 *   The kept set is the first k_b tokens under the order (score descending,
 *   token index ascending); NaN ranks below every number and -0 equals +0.
 *   kept_idx lists the kept global row indices in ascending order;
 *   out_offsets[b+1] = out_offsets[b] + k_b.
 *   Compaction copies each kept row byte for byte.
 *
 * Readings where the paper leaves a choice open (each one is a decision of this
 * oracle, not a statement of the paper):
 *   R1  queries are all text tokens of the request;
 *   R2  the softmax normaliser runs over the request's visual tokens only;
 *   R3  no causal mask is applied (text follows the image, so every text query
 *       already sees every visual key);
 *   R4  heads and queries are reduced by their arithmetic mean, so the scores
 *       of a request sum to 1;
 *   R5  grouped-query attention maps query head h to key head floor(h / G);
 *   R6  the logit scale is 1/sqrt(d), times the per-tensor scales for e4m3;
 *   R7  finetuning changes only the weights that produce q and k, not this formula;
 *   R8  r is the fraction of visual tokens kept (text tokens are always kept);
 *   R9  k from r rounds down;
 *   R10 ties go to the lower token index;
 *   R11 kept rows stay in their original order;
 *   R12 NaN scores rank below everything, +inf above;
 *   R13 N_b = 0 or k_b = 0 give an empty output; N_b > 0 with T_b = 0 is an error.
 *
 * litevlm_oracle_select_views is the patch-selection gating upstream of the
 * path, litevlm_oracle_project the layer-0 projection that makes q and k
 * (each states its definition and readings at the function).
 *
 * litevlm_oracle_score_full is the variant without R2 and R3: the normaliser
 * runs over the system, visual and causal text keys of the first decoder
 * layer, so a request's scores sum to its visual attention share (< 1).
 *
 * Element decoding: bf16 is the top half of an IEEE binary32; e4m3 follows the
 * OCP 8-bit floating point specification (E4M3, bias 7, no infinities, the
 * all-ones code is NaN, subnormals m * 2^-9).
 *
 * Build: plain C99, -O2 -ffp-contract=off (no fused multiply-add contraction,
 * so x86 and Arm hosts give the same doubles).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_F32 0
#define OR_BF16 1
#define OR_E4M3 2

#define OR_OK 0
#define OR_ERR_ARG -1
#define OR_ERR_NOMEM -2

double litevlm_oracle_decode(int32_t dtype, const void* base, int64_t index)
{
    if (dtype == OR_F32) {
        float f;
        memcpy(&f, (const char*)base + 4 * index, 4);
        return (double)f;
    }
    if (dtype == OR_BF16) {
        uint16_t h;
        uint32_t u;
        float f;
        memcpy(&h, (const char*)base + 2 * index, 2);
        u = (uint32_t)h << 16;
        memcpy(&f, &u, 4);
        return (double)f;
    }
    if (dtype == OR_E4M3) {
        uint8_t c = ((const uint8_t*)base)[index];
        int sign = c >> 7, e = (c >> 3) & 0xF, m = c & 0x7;
        double v;
        if (e == 0xF && m == 0x7) return NAN;
        if (e == 0) v = ldexp((double)m, -9);          /* m/8 * 2^(1-7)  */
        else v = ldexp((double)(8 + m), e - 10);       /* (1+m/8) * 2^(e-7) */
        return sign ? -v : v;
    }
    return NAN;
}

/*
 * scores      [sum N_b]             fp32 result
 * scores64    [sum N_b] (nullable)  the same before the final rounding
 * row_sums    [sum_b Hq*T_b] (nullable)  sum_j P[h][i][j] per (b, h, i), h-major
 * row_lse     [sum_b Hq*T_b] (nullable)  m + ln(l) per (b, h, i)
 */
int litevlm_oracle_score(int32_t batch, const int32_t* seq_offsets, const int32_t* text_offsets,
                         int32_t hq, int32_t hkv, int32_t head_dim, int32_t dtype,
                         const void* q, const void* k, double q_scale, double k_scale,
                         float* scores, double* scores64, double* row_sums, double* row_lse)
{
    int64_t row_out = 0;
    if (batch < 0 || hq <= 0 || hkv <= 0 || head_dim <= 0 || hq % hkv != 0) return OR_ERR_ARG;
    if (dtype != OR_F32 && dtype != OR_BF16 && dtype != OR_E4M3) return OR_ERR_ARG;
    for (int32_t b = 0; b < batch; ++b) {
        if (seq_offsets[b + 1] < seq_offsets[b] || text_offsets[b + 1] < text_offsets[b]) return OR_ERR_ARG;
        if (seq_offsets[b + 1] > seq_offsets[b] && text_offsets[b + 1] == text_offsets[b]) return OR_ERR_ARG;
    }
    const int32_t group = hq / hkv;
    const double scale = q_scale * k_scale / sqrt((double)head_dim);

    for (int32_t b = 0; b < batch; ++b) {
        const int64_t n0 = seq_offsets[b], nb = seq_offsets[b + 1] - seq_offsets[b];
        const int64_t t0 = text_offsets[b], tb = text_offsets[b + 1] - text_offsets[b];
        if (nb == 0) {
            /* rows of this request still get their (empty) stats slots */
            if (row_sums) for (int64_t r = 0; r < (int64_t)hq * tb; ++r) row_sums[row_out + r] = 0.0;
            if (row_lse) for (int64_t r = 0; r < (int64_t)hq * tb; ++r) row_lse[row_out + r] = -INFINITY;
            row_out += (int64_t)hq * tb;
            continue;
        }
        double* acc = (double*)calloc((size_t)nb, sizeof(double));
        double* s = (double*)malloc((size_t)nb * sizeof(double));
        /* step 1: decode this request's q and k rows exactly into doubles */
        double* qd = (double*)malloc((size_t)(tb * hq * head_dim) * sizeof(double));
        double* kd = (double*)malloc((size_t)(nb * hkv * head_dim) * sizeof(double));
        if (!acc || !s || !qd || !kd) { free(acc); free(s); free(qd); free(kd); return OR_ERR_NOMEM; }
        for (int64_t x = 0; x < tb * hq * head_dim; ++x) qd[x] = litevlm_oracle_decode(dtype, q, t0 * hq * head_dim + x);
        for (int64_t x = 0; x < nb * hkv * head_dim; ++x) kd[x] = litevlm_oracle_decode(dtype, k, n0 * hkv * head_dim + x);

        for (int32_t h = 0; h < hq; ++h) {
            const int32_t g = h / group;
            for (int64_t i = 0; i < tb; ++i) {
                const int64_t qrow = (i * hq + h) * head_dim;
                double m = -INFINITY, l = 0.0, psum = 0.0;
                for (int64_t j = 0; j < nb; ++j) {
                    const int64_t krow = (j * hkv + g) * head_dim;
                    double dot = 0.0;
                    for (int32_t c = 0; c < head_dim; ++c) dot += qd[qrow + c] * kd[krow + c];
                    s[j] = dot * scale;
                    if (s[j] > m) m = s[j];
                }
                for (int64_t j = 0; j < nb; ++j) l += exp(s[j] - m);
                for (int64_t j = 0; j < nb; ++j) {
                    const double p = exp(s[j] - m) / l;
                    acc[j] += p;
                    psum += p;
                }
                if (row_sums) row_sums[row_out] = psum;
                if (row_lse) row_lse[row_out] = m + log(l);
                ++row_out;
            }
        }
        const double denom = (double)hq * (double)tb;
        for (int64_t j = 0; j < nb; ++j) {
            const double v = acc[j] / denom;
            scores[n0 + j] = (float)v;
            if (scores64) scores64[n0 + j] = v;
        }
        free(acc);
        free(s);
        free(qd);
        free(kd);
    }
    return OR_OK;
}

typedef struct {
    float key;
    int32_t idx;
} oracle_item;

/* score descending, index ascending; NaN after every number; -0 == +0 */
static int oracle_rank_cmp(const void* pa, const void* pb)
{
    const oracle_item* a = (const oracle_item*)pa;
    const oracle_item* b = (const oracle_item*)pb;
    const int an = isnan(a->key) != 0, bn = isnan(b->key) != 0;
    if (an != bn) return an ? 1 : -1;
    if (!an && a->key != b->key) return a->key > b->key ? -1 : 1;
    return (a->idx > b->idx) - (a->idx < b->idx);
}

static int oracle_index_cmp(const void* pa, const void* pb)
{
    const oracle_item* a = (const oracle_item*)pa;
    const oracle_item* b = (const oracle_item*)pb;
    return (a->idx > b->idx) - (a->idx < b->idx);
}

int64_t litevlm_oracle_keep_count(int32_t n, float keep_ratio)
{
    double kd = floor((double)keep_ratio * (double)n);
    if (kd < 0) kd = 0;
    if (kd > n) kd = n;
    return (int64_t)kd;
}

/*
 * keep_k may be NULL: then k_b = floor((double)keep_ratio * N_b) clamped to [0, N_b].
 * kept_idx receives sum_b k_b global indices; out_offsets has batch+1 entries.
 */
int litevlm_oracle_topk(int32_t batch, const int32_t* seq_offsets, const float* scores,
                        const int32_t* keep_k, float keep_ratio,
                        int32_t* kept_idx, int32_t* out_offsets)
{
    int64_t out = 0;
    if (batch < 0) return OR_ERR_ARG;
    if (!keep_k && !(keep_ratio >= 0.0f && keep_ratio <= 1.0f)) return OR_ERR_ARG;
    out_offsets[0] = 0;
    for (int32_t b = 0; b < batch; ++b) {
        const int64_t n0 = seq_offsets[b], nb = seq_offsets[b + 1] - seq_offsets[b];
        int64_t kb;
        if (nb < 0) return OR_ERR_ARG;
        kb = keep_k ? keep_k[b] : litevlm_oracle_keep_count((int32_t)nb, keep_ratio);
        if (kb < 0 || kb > nb) return OR_ERR_ARG;
        if (kb > 0) {
            oracle_item* it = (oracle_item*)malloc((size_t)nb * sizeof(oracle_item));
            if (!it) return OR_ERR_NOMEM;
            for (int64_t j = 0; j < nb; ++j) {
                it[j].key = scores[n0 + j];
                it[j].idx = (int32_t)j;
            }
            qsort(it, (size_t)nb, sizeof(oracle_item), oracle_rank_cmp);
            qsort(it, (size_t)kb, sizeof(oracle_item), oracle_index_cmp);
            for (int64_t r = 0; r < kb; ++r) kept_idx[out + r] = (int32_t)(n0 + it[r].idx);
            free(it);
        }
        out += kb;
        out_offsets[b + 1] = (int32_t)out;
    }
    return OR_OK;
}

/* dst[r] = src[kept_idx[r]] for rows of row_bytes bytes */
int litevlm_oracle_compact(int64_t total_kept, const int32_t* kept_idx,
                           const void* src, void* dst, int64_t row_bytes)
{
    if (total_kept < 0 || row_bytes < 0) return OR_ERR_ARG;
    for (int64_t r = 0; r < total_kept; ++r)
        memcpy((char*)dst + r * row_bytes, (const char*)src + (int64_t)kept_idx[r] * row_bytes, (size_t)row_bytes);
    return OR_OK;
}

/*
 * Prefill sequence splice (the LLM input after token selection; Design
 * section: the module shortens the sequence the LLM prefills). Request b's
 * output is its S_b system rows, then its k_b kept visual rows (kept_idx
 * holds global visual-row indices, ascending within the request), then its
 * T_b text rows, each row copied byte for byte.
 *   out_offsets[b] = sys_offsets[b] + kept_offsets[b] + text_offsets[b]
 * Position ids are the rows' positions in the unpruned sequence
 * [system; all N_b visual; text]: system row i -> i, kept visual row with
 * local index j -> S_b + j, text row t -> S_b + N_b + t (pruned tokens leave
 * gaps; the kept tokens keep their original positions).
 */
int litevlm_oracle_splice(int32_t batch, const int32_t* sys_offsets, const int32_t* seq_offsets,
                          const int32_t* kept_offsets, const int32_t* kept_idx, const int32_t* text_offsets,
                          const void* sys_rows, const void* vis_rows, const void* txt_rows, int64_t row_bytes,
                          void* out_rows, int32_t* out_offsets, int32_t* position_ids)
{
    if (batch < 0 || row_bytes <= 0) return OR_ERR_ARG;
    for (int32_t b = 0; b <= batch; ++b) out_offsets[b] = sys_offsets[b] + kept_offsets[b] + text_offsets[b];
    for (int32_t b = 0; b < batch; ++b) {
        const int32_t S = sys_offsets[b + 1] - sys_offsets[b];
        const int32_t N = seq_offsets[b + 1] - seq_offsets[b];
        const int32_t k = kept_offsets[b + 1] - kept_offsets[b];
        const int32_t T = text_offsets[b + 1] - text_offsets[b];
        int64_t r = out_offsets[b];
        for (int32_t i = 0; i < S; ++i, ++r) {
            memcpy((char*)out_rows + r * row_bytes, (const char*)sys_rows + (int64_t)(sys_offsets[b] + i) * row_bytes,
                   (size_t)row_bytes);
            position_ids[r] = i;
        }
        for (int32_t i = 0; i < k; ++i, ++r) {
            const int32_t g = kept_idx[kept_offsets[b] + i];
            if (g < seq_offsets[b] || g >= seq_offsets[b] + N) return OR_ERR_ARG;
            memcpy((char*)out_rows + r * row_bytes, (const char*)vis_rows + (int64_t)g * row_bytes, (size_t)row_bytes);
            position_ids[r] = S + (g - seq_offsets[b]);
        }
        for (int32_t t = 0; t < T; ++t, ++r) {
            memcpy((char*)out_rows + r * row_bytes, (const char*)txt_rows + (int64_t)(text_offsets[b] + t) * row_bytes,
                   (size_t)row_bytes);
            position_ids[r] = S + N + t;
        }
    }
    return OR_OK;
}

/*
 * Visual-token scores with the softmax normaliser over the full causal key
 * set of the first decoder layer (a reading of the Design section's
 * first-layer attention; the variant of litevlm_oracle_score that does not
 * restrict the keys to the visual tokens). Text query i of request b, head h,
 * attends to the S_b system keys, the N_b visual keys and the text keys
 * t' <= i (causal); with s the scaled logits over all of them,
 *     P[h][i][j] = exp(s[h][i][j] - m) / sum_{all keys} exp(s - m)
 *     score[j]   = (sum_h sum_i P[h][i][j]) / (Hq * T_b),  j visual
 * so a request's scores sum to the attention share of its visual tokens.
 * k_sys [sum S_b, Hkv, d] and k_txt [sum T_b, Hkv, d] are the system and text
 * tokens' keys, in the element type of q and k (same per-tensor k_scale).
 * visual_share [sum_b Hq*T_b] (nullable): sum_j P[h][i][j] over visual j.
 */
int litevlm_oracle_score_full(int32_t batch, const int32_t* seq_offsets, const int32_t* text_offsets,
                              const int32_t* sys_offsets, int32_t hq, int32_t hkv, int32_t head_dim, int32_t dtype,
                              const void* q, const void* k, const void* k_sys, const void* k_txt, double q_scale,
                              double k_scale, float* scores, double* scores64, double* visual_share)
{
    int64_t row_out = 0;
    if (batch < 0 || hq <= 0 || hkv <= 0 || head_dim <= 0 || hq % hkv != 0) return OR_ERR_ARG;
    if (dtype != OR_F32 && dtype != OR_BF16 && dtype != OR_E4M3) return OR_ERR_ARG;
    for (int32_t b = 0; b < batch; ++b) {
        if (seq_offsets[b + 1] < seq_offsets[b] || text_offsets[b + 1] < text_offsets[b] ||
            sys_offsets[b + 1] < sys_offsets[b])
            return OR_ERR_ARG;
        if (seq_offsets[b + 1] > seq_offsets[b] && text_offsets[b + 1] == text_offsets[b]) return OR_ERR_ARG;
    }
    const int32_t group = hq / hkv;
    const double scale = q_scale * k_scale / sqrt((double)head_dim);
    for (int32_t b = 0; b < batch; ++b) {
        const int64_t n0 = seq_offsets[b], nb = seq_offsets[b + 1] - seq_offsets[b];
        const int64_t t0 = text_offsets[b], tb = text_offsets[b + 1] - text_offsets[b];
        const int64_t s0 = sys_offsets[b], sb = sys_offsets[b + 1] - sys_offsets[b];
        if (nb == 0) {
            if (visual_share) for (int64_t r = 0; r < (int64_t)hq * tb; ++r) visual_share[row_out + r] = 0.0;
            row_out += (int64_t)hq * tb;
            continue;
        }
        const int64_t nkeys = sb + nb + tb;  /* system, visual, text keys of this request */
        double* acc = (double*)calloc((size_t)nb, sizeof(double));
        double* s = (double*)malloc((size_t)nkeys * sizeof(double));
        double* qd = (double*)malloc((size_t)(tb * hq * head_dim) * sizeof(double));
        double* kd = (double*)malloc((size_t)(nkeys * hkv * head_dim) * sizeof(double));
        if (!acc || !s || !qd || !kd) { free(acc); free(s); free(qd); free(kd); return OR_ERR_NOMEM; }
        const int64_t row = (int64_t)hkv * head_dim;
        for (int64_t x = 0; x < tb * hq * head_dim; ++x) qd[x] = litevlm_oracle_decode(dtype, q, t0 * hq * head_dim + x);
        for (int64_t x = 0; x < sb * row; ++x) kd[x] = litevlm_oracle_decode(dtype, k_sys, s0 * row + x);
        for (int64_t x = 0; x < nb * row; ++x) kd[sb * row + x] = litevlm_oracle_decode(dtype, k, n0 * row + x);
        for (int64_t x = 0; x < tb * row; ++x) kd[(sb + nb) * row + x] = litevlm_oracle_decode(dtype, k_txt, t0 * row + x);
        for (int32_t h = 0; h < hq; ++h) {
            const int32_t g = h / group;
            for (int64_t i = 0; i < tb; ++i) {
                const int64_t qrow = (i * hq + h) * head_dim;
                const int64_t nk = sb + nb + i + 1;  /* keys visible to text query i */
                double m = -INFINITY, z = 0.0, vis = 0.0;
                for (int64_t j = 0; j < nk; ++j) {
                    const int64_t krow = (j * hkv + g) * head_dim;
                    double dot = 0.0;
                    for (int32_t c = 0; c < head_dim; ++c) dot += qd[qrow + c] * kd[krow + c];
                    s[j] = dot * scale;
                    if (s[j] > m) m = s[j];
                }
                for (int64_t j = 0; j < nk; ++j) z += exp(s[j] - m);
                for (int64_t j = 0; j < nb; ++j) {
                    const double p = exp(s[sb + j] - m) / z;
                    acc[j] += p;
                    vis += p;
                }
                if (visual_share) visual_share[row_out] = vis;
                ++row_out;
            }
        }
        const double denom = (double)hq * (double)tb;
        for (int64_t j = 0; j < nb; ++j) {
            const double v = acc[j] / denom;
            scores[n0 + j] = (float)v;
            if (scores64) scores64[n0 + j] = v;
        }
        free(acc);
        free(s);
        free(qd);
        free(kd);
    }
    return OR_OK;
}

/*
 * Patch-selection gating (Design section, Patch Selection Module: the final
 * score of a camera view is a weighted sum of the lexical-mapping score and
 * the module's logit; the views scoring above a predefined threshold go on to
 * the vision encoder). For request b and view v, in fp32 arithmetic:
 *     s[b][v] = w_lex * lexical[b][v] + w_logit * logit[b][v]
 *     view v is selected when s[b][v] > threshold
 * Readings: the logit enters as is (no sigmoid); "above" is strict; when fewer
 * than min_views views pass, the min_views highest-scoring views are taken
 * instead (ties to the lower view index; NaN scores rank lowest and never pass
 * the threshold); min_views = 0 allows an empty selection.
 * Outputs: view_mask[b][v] in {0, 1}; view_offsets (prefix of the selected
 * view counts) and selected_views (view indices, ascending per request);
 * seq_offsets (prefix of the visual tokens: sum over selected v of
 * tokens_per_view[v]), the N_b of the token-selection path.
 */
static int oracle_view_before(float a, int ia, float b, int ib)
{
    /* strict order of (score desc, index asc), NaN lowest */
    const int an = a != a, bn = b != b;
    if (an != bn) return bn;
    if (!an && a != b) return a > b;
    return ia < ib;
}

int litevlm_oracle_select_views(int32_t batch, int32_t num_views, const float* lexical, const float* logits,
                                const int32_t* tokens_per_view, float w_lex, float w_logit, float threshold,
                                int32_t min_views, uint8_t* view_mask, int32_t* view_offsets,
                                int32_t* selected_views, int32_t* seq_offsets)
{
    if (batch < 0 || num_views <= 0 || num_views > 64 || min_views < 0 || min_views > num_views) return OR_ERR_ARG;
    view_offsets[0] = 0;
    seq_offsets[0] = 0;
    int64_t nsel = 0, ntok = 0;
    for (int32_t b = 0; b < batch; ++b) {
        float s[64];
        int pass = 0;
        for (int32_t v = 0; v < num_views; ++v) {
            const float a = w_lex * lexical[(int64_t)b * num_views + v];
            const float c = w_logit * logits[(int64_t)b * num_views + v];
            s[v] = a + c;
            const int sel = s[v] > threshold;
            view_mask[(int64_t)b * num_views + v] = (uint8_t)sel;
            pass += sel;
        }
        if (pass < min_views) {
            /* the min_views best views: rank each view by how many views come before it */
            for (int32_t v = 0; v < num_views; ++v) {
                int rank = 0;
                for (int32_t u = 0; u < num_views; ++u)
                    if (u != v && oracle_view_before(s[u], u, s[v], v)) ++rank;
                view_mask[(int64_t)b * num_views + v] = (uint8_t)(rank < min_views);
            }
        }
        for (int32_t v = 0; v < num_views; ++v) {
            if (view_mask[(int64_t)b * num_views + v]) {
                selected_views[nsel++] = v;
                ntok += tokens_per_view[v];
            }
        }
        if (ntok > INT32_MAX) return OR_ERR_ARG;
        view_offsets[b + 1] = (int32_t)nsel;
        seq_offsets[b + 1] = (int32_t)ntok;
    }
    return OR_OK;
}

/*
 * Layer-0 projection feeding the scores (Design section: the module is the
 * first decoder layer; its queries and keys are RoPE(W . RMSNorm(x))). For
 * token row r with hidden x_r (bf16, H values), position p_r:
 *     s_r   = 1 / sqrt(mean_h x_r[h]^2 + eps)
 *     y_r[o] = sum_h (x_r[h] * s_r * gamma[h]) * W[o][h] + bias[o]
 * then, when head_dim > 0, rotary position embedding on each head of head_dim
 * values, pairing element j with element j + head_dim/2 (rotate-half form):
 *     theta_j = rope_base^(-2j / head_dim),  a = p_r * theta_j
 *     y[j]           <- y[j] cos a - y[j + d/2] sin a
 *     y[j + d/2]     <- y[j + d/2] cos a + y[j] sin a
 * W is [O, H] bf16 (out x in); gamma [H] and bias [O] (nullable) are fp32;
 * y is [rows, O] in fp64.
 */
int litevlm_oracle_project(int64_t rows, int32_t hidden, int32_t out_features, const uint16_t* x, const float* gamma,
                           double eps, const uint16_t* w, const float* bias, int32_t head_dim,
                           const int32_t* positions, double rope_base, double* y)
{
    if (rows < 0 || hidden <= 0 || out_features <= 0 || head_dim < 0) return OR_ERR_ARG;
    if (head_dim > 0 && (head_dim % 2 != 0 || out_features % head_dim != 0)) return OR_ERR_ARG;
    double* xn = (double*)malloc((size_t)hidden * sizeof(double));
    if (!xn) return OR_ERR_NOMEM;
    for (int64_t r = 0; r < rows; ++r) {
        double ss = 0.0;
        for (int32_t h = 0; h < hidden; ++h) {
            const double v = litevlm_oracle_decode(OR_BF16, x, r * hidden + h);
            xn[h] = v;
            ss += v * v;
        }
        const double s = 1.0 / sqrt(ss / (double)hidden + eps);
        for (int32_t h = 0; h < hidden; ++h) xn[h] = xn[h] * s * (double)gamma[h];
        double* yr = y + r * out_features;
        for (int32_t o = 0; o < out_features; ++o) {
            double acc = 0.0;
            for (int32_t h = 0; h < hidden; ++h)
                acc += xn[h] * litevlm_oracle_decode(OR_BF16, w, (int64_t)o * hidden + h);
            yr[o] = acc + (bias ? (double)bias[o] : 0.0);
        }
        if (head_dim > 0) {
            const int32_t half = head_dim / 2;
            for (int32_t h0 = 0; h0 < out_features; h0 += head_dim) {
                for (int32_t j = 0; j < half; ++j) {
                    const double theta = pow(rope_base, -2.0 * (double)j / (double)head_dim);
                    const double a = (double)positions[r] * theta;
                    const double y1 = yr[h0 + j], y2 = yr[h0 + j + half];
                    yr[h0 + j] = y1 * cos(a) - y2 * sin(a);
                    yr[h0 + j + half] = y2 * cos(a) + y1 * sin(a);
                }
            }
        }
    }
    free(xn);
    return OR_OK;
}
