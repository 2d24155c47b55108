// Internal interfaces between the C-ABI layer (api.cu) and the kernel files.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "score.h"  // the score kernels' launch parameters, planner helpers and entry points

namespace lvs {

// bits of the device error word
constexpr int32_t kErrTimeout = 1;       // a bounded mbarrier / cluster wait gave up
constexpr int32_t kErrBounds = 2;        // an index outside its buffer was skipped
constexpr int32_t kErrShape = 4;         // a request shape the kernel cannot handle

// Wait budget for every device-side wait, in SM clock cycles (about 2 s).
constexpr long long kWaitBudgetCycles = 4000000000LL;

// Every kernel of the library is launched with programmatic dependent launch:
// it may be scheduled while the previous kernel of the stream is finishing,
// and it waits for that kernel to complete (griddepcontrol.wait) before its
// first global-memory access, so stream order is kept for all memory.
inline cudaLaunchAttribute pdl_attribute()
{
    cudaLaunchAttribute a;
    a.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    a.val.programmaticStreamSerializationAllowed = 1;
    return a;
}

// topk.cu
// Per-request sizes from the host mirrors, passed by value for small batches
// so the kernel needs no dependent global loads before it reads the scores
// (the mirrors equal the device arrays by contract).
constexpr int kTopkShapeMax = 256;
struct TopkShape {
    int32_t n;                      // requests described; 0: the kernel reads the device arrays
    int32_t n0[kTopkShapeMax];      // first visual row of the request
    int32_t len[kTopkShapeMax];     // N_b
    int32_t k[kTopkShapeMax];       // k_b
    int32_t out0[kTopkShapeMax];    // sum of k over earlier requests
    // Deferred fold (partials != null): the scores are the sum over `groups`
    // partial rows (stride total_vis, added in group order) divided by denom[b];
    // the kernel writes them to `scores` and selects on them.
    const float* partials;
    int32_t groups;
    int64_t total_vis;
    float denom[kTopkShapeMax];
};
cudaError_t launch_topk(int batch, float* scores, const int32_t* seq_off, const int32_t* keep_k,
                        float keep_ratio, int32_t* kept_idx, int32_t* out_off, int max_n, const TopkShape& shape,
                        cudaStream_t stream);


// compact.cu
constexpr int kMaxGatherTensors = 8;
struct GatherArgs {
    int32_t n;
    const uint8_t* src[kMaxGatherTensors];
    uint8_t* dst[kMaxGatherTensors];
    int64_t row_bytes[kMaxGatherTensors];
};
cudaError_t launch_compact(int64_t total_kept, const int32_t* kept_idx, int64_t src_rows, const GatherArgs& g,
                           bool vec16, int32_t* err, int num_sms, cudaStream_t stream);

// ctx_stats.cu: e[t][h] = log2 sum 2^(c q.k) over the system and causal text
// keys of every text query row (the full-key-set normaliser's extra terms)
struct CtxArgs {
    const uint8_t* q;         // [sum T, Hq, d]
    const uint8_t* k_sys;     // [sum S, Hkv, d]
    const uint8_t* k_txt;     // [sum T, Hkv, d]
    const int32_t* seq_off;   // device [batch+1] visual rows
    const int32_t* text_off;  // device [batch+1]
    const int32_t* sys_off;   // device [batch+1]
    float* out;               // [sum T][Hq]
    int32_t* err;
    int32_t batch, hq, hkv, query_last;
    float c_log2;
    long long wait_budget;
};
cudaError_t launch_ctx_stats(const CtxArgs& a, int row_bytes, bool fp8, cudaStream_t stream);

// views.cu: patch-selection gating (views -> N_b)
constexpr int kMaxViews = 64;
struct ViewsArgs {
    const float* lexical;     // [B, V]
    const float* logits;      // [B, V]
    float w_lex, w_logit, threshold;
    int32_t batch, num_views, min_views;
    int32_t tokens_per_view[kMaxViews];
    uint8_t* view_mask;       // [B, V]
    int32_t* view_offsets;    // [B+1]
    int32_t* selected_views;  // [sum of selected views]
    int32_t* seq_offsets;     // [B+1]
};
cudaError_t launch_views(const ViewsArgs& a, cudaStream_t stream);

// proj.cu: layer-0 projection RoPE(s_r * x W'^T + bias), W' = W * gamma
struct ProjArgs {
    int64_t rows;
    int32_t hidden, out_features, head_dim, max_positions;
    float eps;
    const float* bias;        // [O] or null
    const int32_t* positions; // [rows] (head_dim > 0)
    const float2* rope;       // [max_positions][head_dim / 2] (cos, sin)
    __nv_bfloat16* y;         // [rows, O] bf16 output, or
    uint8_t* y8;              // [rows, O] e4m3 codes of y * out_inv_scale (null: bf16 output)
    float out_inv_scale;
    int32_t* err;
    long long wait_budget;
};
struct RopeArgs {
    float2* table;            // [max_positions][half]
    int32_t max_positions, half;
    float inv_freq[128];      // rope_base^(-2j / head_dim), rounded to fp32
};
int proj_tile_cols(int out_features);
int proj_tile_rows(int64_t rows, int out_features, int num_sms);
cudaError_t launch_proj(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const ProjArgs& p, int tile_rows,
                        cudaStream_t stream);
cudaError_t launch_fold_norm(const __nv_bfloat16* w, const float* gamma, __nv_bfloat16* out, int64_t total,
                             int hidden, int num_sms, cudaStream_t stream);
cudaError_t launch_rope_table(const RopeArgs& a, int num_sms, cudaStream_t stream);

// splice.cu
struct SpliceArgs {
    const int32_t* sys_off;   // device [batch+1]
    const int32_t* seq_off;   // device [batch+1] visual rows
    const int32_t* kept_off;  // device [batch+1]
    const int32_t* kept_idx;  // device [sum k]
    const int32_t* text_off;  // device [batch+1]
    const uint8_t* sys;
    const uint8_t* vis;
    const uint8_t* txt;
    uint8_t* out;
    int32_t* out_off;         // device [batch+1]
    int32_t* pos;             // device [sum (S + k + T)]
    int64_t row_bytes;
    int32_t batch;
    int32_t* err;
};
cudaError_t launch_splice(const SpliceArgs& a, int max_rows, bool vec16, cudaStream_t stream);

}  // namespace lvs
