// Internal interfaces between the C-ABI layer (api.cu) and the kernel files.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace lvs {

// bits of the device error word
constexpr int32_t kErrTimeout = 1;       // a bounded mbarrier / cluster wait gave up
constexpr int32_t kErrBounds = 2;        // an index outside its buffer was skipped
constexpr int32_t kErrShape = 4;         // a request shape the kernel cannot handle

constexpr int kTileRows = 128;           // visual tokens per score tile (MMA M)
constexpr int kMaxText = 128;            // text tokens per request handled by the score kernel
constexpr int kMaxTilesPerCta = 32;      // score tiles one CTA may own
constexpr int kMaxCluster = 16;

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

struct ScoreLaunch {
    const int32_t* seq_off;   // device [batch+1]
    const int32_t* text_off;  // device [batch+1]
    float* out;               // scores [sum N]
    float* partials;          // [groups][sum N] when groups > 1 (workspace)
    int32_t* counters;        // one fold ticket per 128-token tile, zero between launches (workspace)
    int32_t* err;
    int64_t total_vis;        // partial-row stride
    int32_t hq, hkv;
    int32_t heads_per_group;
    int32_t groups;
    int32_t ctas_per_request; // cluster size * groups
    int32_t slot_cols;        // resident kernel: TMEM columns per slot (T rounded up to 16, max over batch)
    int32_t res_nb;           // resident kernel: TMEM head buffers, 1 or 2 (2: heads overlap)
    float c_log2;             // q_scale * k_scale / sqrt(d) * log2(e)
    long long wait_budget;
};

struct ScorePlan {
    int cluster;              // CTAs per (request, head group)
    int tiles_per_cta;
    int groups;               // head groups (grid.y); partial rows when > 1
    int res_nb = 1;           // resident kernel: TMEM head buffers
};

// Host helpers (score_tc.cu)
ScorePlan plan_score(int batch, int max_tiles, int hq, int hkv, int tile_bytes, int num_sms);
cudaError_t launch_score(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const ScoreLaunch& p,
                         const ScorePlan& plan, int batch, int row_bytes, bool fp8, int mrows, cudaStream_t stream);
bool score_shape_supported(int head_dim, bool fp8);

// score_res.cu (one contraction per K tile and head, logits resident in TMEM)
int res_max_tiles(int slot_cols, int nb);          // tiles per CTA that fit in tensor memory with nb head buffers
int res_max_cluster(int row_bytes, int slot_cols); // cluster size limit of the statistics buffer
int res_cluster_capacity(int row_bytes, bool fp8, int mrows, int cluster);
cudaError_t launch_score_resident(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const ScoreLaunch& p,
                                  const ScorePlan& plan, int batch, int row_bytes, bool fp8, int mrows,
                                  cudaStream_t stream);

// topk.cu
cudaError_t launch_topk(int batch, const float* scores, const int32_t* seq_off, const int32_t* keep_k,
                        float keep_ratio, int32_t* kept_idx, int32_t* out_off, int max_n, cudaStream_t stream);

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

}  // namespace lvs
