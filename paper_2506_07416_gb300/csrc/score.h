// The score kernels' interface: their tile constants, launch parameters,
// the planner's batch model and the launch entry points (score_tc.cu,
// score_res.cu). Included by internal.h.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace lvs {

constexpr int kTileRows = 128;           // visual tokens per score tile (MMA M)
constexpr int kMaxText = 128;            // text tokens per request handled by the score kernel
constexpr int kMaxTilesPerCta = 32;      // score tiles one CTA may own
constexpr int kMaxCluster = 16;
constexpr int kOrderMax = 2048;          // batches up to this size are launched largest request first
constexpr int kOffsetsByValue = 64;      // batches up to this size carry their offsets in the launch parameters
constexpr int kFlatMax = 160;            // clusters of a flattened resident launch (at least one per SM pair)

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
    int32_t slot_cols;        // resident kernel: TMEM columns per slot (query rows per head, rounded up to 16)
    // resident kernel: 1, or 2 when each query head's text rows run as two
    // pseudo-heads (the first ceil(T/2) rows, then the rest): heads_per_group,
    // groups and the flattened pairs count pseudo-heads, hq stays the model's
    int32_t qsplit;
    int32_t res_nb;           // resident kernel: TMEM head buffers, 1 or 2 (2: heads overlap)
    int32_t query_last;       // 1: only the last text token of each request is a query
    int32_t defer_fold;       // 1 (with groups > 1): leave the group partials; the top-k kernel adds them
    float c_log2;             // q_scale * k_scale / sqrt(d) * log2(e)
    long long wait_budget;
    int32_t stall;            // resident kernel: the producer first waits on a barrier nothing completes (tests)
    // [sum T][Hq] normaliser terms of the system and causal text keys (unit of
    // the merged statistic b, from ctx_stats.cu), or null: visual keys only
    const float* extra;
    // nv > 0 (batches of at most kOffsetsByValue requests): the seq / text
    // offsets by value, equal to seq_off / text_off (the host mirrors), so a
    // CTA knows its tiles without a global load and its first copies go out as
    // soon as its setup is done. nv == 0: read seq_off / text_off.
    int32_t nv;
    int32_t so_v[kOffsetsByValue + 1];
    int32_t to_v[kOffsetsByValue + 1];
    // Cluster k of the 1-D grid serves item k: request order[k / groups] (the
    // requests from the largest to the smallest, so the hardware starts the
    // biggest clusters first and fills in with small ones), head group
    // k % groups. order_n == 0: requests in index order.
    int32_t order_n;
    uint16_t order[kOrderMax];
    // Flattened schedule of the resident kernel (flat_n > 0; every request has
    // the same visual and text token counts): the batch's (request, head) pairs
    // in request-major order, cluster k taking pairs [flat_r[k], flat_r[k+1]);
    // a request whose heads span several clusters is folded from their partial
    // rows (part = cluster - first cluster of the request).
    int32_t flat_n;
    int32_t flat_r[kFlatMax + 1];
};

struct ScorePlan {
    int cluster;              // CTAs per (request, head group)
    int tiles_per_cta;
    int groups;               // head groups (grid.y); partial rows when > 1
    int res_nb = 1;           // resident kernel: TMEM head buffers
    int flat = 0;             // resident kernel: clusters of the flattened (request, head) schedule, 0: none
    int qsplit = 1;           // resident kernel: 2 = each head's text rows as two pseudo-heads (64-row kernel)
};

// Host helpers (score_tc.cu)
// The batch as the planners see it: 128-token tiles per request, largest first.
struct BatchTiles {
    const int* desc;  // [n] tiles per request, non-increasing
    int n;
};
// Time to run n_req * g items on `slots` cluster slots when clusters start
// largest first and each takes the slot that frees up first (the order the
// kernels are launched in); cost(tiles) is one item's time.
template <class Cost>
double makespan(const BatchTiles& bt, int g, int slots, const Cost& cost)
{
    if (bt.n <= 0 || slots <= 0) return 0.0;
    const long long items = (long long)bt.n * g;
    if (bt.desc[0] == bt.desc[bt.n - 1]) return (double)((items + slots - 1) / slots) * cost(bt.desc[0]);
    if (items > 4096) {  // bound instead of the schedule
        double total = 0.0;
        for (int i = 0; i < bt.n; ++i) total += g * cost(bt.desc[i]);
        const double mx = cost(bt.desc[0]);
        return (total / slots > mx ? total / slots : mx) + 0.5 * total / (double)items;
    }
    // binary min-heap of slot loads
    double heap[1024];
    const int ns = slots < 1024 ? slots : 1024;
    for (int i = 0; i < ns; ++i) heap[i] = 0.0;
    double mx = 0.0;
    for (int i = 0; i < bt.n; ++i) {
        const double c = cost(bt.desc[i]);
        for (int k = 0; k < g; ++k) {
            const double v = heap[0] + c;  // the slot that frees up first takes the item
            mx = v > mx ? v : mx;
            int j = 0;
            for (;;) {  // sift the new load down
                const int l = 2 * j + 1, r = l + 1;
                int m = j;
                double mv = v;
                if (l < ns && heap[l] < mv) { m = l; mv = heap[l]; }
                if (r < ns && heap[r] < mv) { m = r; mv = heap[r]; }
                if (m == j) break;
                heap[j] = heap[m];
                j = m;
            }
            heap[j] = v;
        }
    }
    return mx;
}

// cap_by_cluster[c]: CTAs of the re-read kernel resident at once with clusters of c (<= 0: unusable)
ScorePlan plan_score(const BatchTiles& bt, int hq, int hkv, int tile_bytes, const int* cap_by_cluster,
                     double* cost_out);
int tc_cluster_capacity(int row_bytes, bool fp8, int mrows, int cluster);
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

}  // namespace lvs
