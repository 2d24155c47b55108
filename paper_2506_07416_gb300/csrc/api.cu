// C-ABI of the token-selection library: handle and workspace management,
// host-side validation from the host offset mirrors, TMA descriptor encoding
// and the kernel launches. See include/litevlm_select.h for the contract.

#include <cudaTypedefs.h>
#include <math.h>
#include <stdint.h>

#include <algorithm>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <vector>

#include "../../include/litevlm_select.h"
#include "internal.h"

#ifdef LITEVLM_NVTX
#include <nvtx3/nvToolsExt.h>
#endif

struct litevlm_select {
    litevlm_select_config_t cfg;
    int device = 0;
    int num_sms = 0;
    float* partials = nullptr;  // [Hq][max_total_visual]: per-head-group partial scores
    int32_t* counters = nullptr;  // fold tickets of the score kernels, one per 128-token tile
    size_t n_counters = 0;
    int32_t* err_d = nullptr;   // device error word (bits lvs::kErr*)
    float* ctx_stats = nullptr; // [max_total_text][Hq]: normaliser terms of system + causal text keys
    PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    int res_capacity[2][17];  // resident score kernel: CTAs at once per cluster size, by pass-1 rows (64/128); -1 unknown
    int tc_capacity[2][17];   // the same for the re-read score kernel
    // last score-kernel choices, keyed by a hash of the batch shape (planning walks every plan)
    struct PlanMemo {
        uint64_t key = 0;
        bool used = false;
        bool resident = false;
        lvs::ScorePlan plan{1, 1, 1};
    } plan_memo[4];
    int plan_memo_next = 0;
    std::vector<int> tiles_desc;  // scratch of the planner for batches above 4096 requests (host)
    lvs::TopkShape topk_shape;    // per-request sizes passed to the top-k kernel by value
    std::string last_error;
    int32_t last_launches = 0;  // kernels the last call on this handle enqueued
    long long wait_budget = lvs::kWaitBudgetCycles;  // clock cycles each device-side wait may take
    int32_t debug_flags = 0;                         // LITEVLM_DEBUG_* (tests of the failure path)
    bool allow_flat = true;  // the resident kernel's flattened schedule may be chosen (not in the no-alloc path)
};

namespace {

thread_local std::string g_create_error;

litevlm_status_t fail(litevlm_select_t h, litevlm_status_t s, const std::string& msg)
{
    if (h) h->last_error = msg;
    else g_create_error = msg;
    return s;
}

litevlm_status_t cuda_fail(litevlm_select_t h, cudaError_t e, const char* where)
{
    return fail(h, LITEVLM_ERR_CUDA, std::string(where) + ": " + cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// An NVTX range around one C-ABI call, named after the call (builds with
// LITEVLM_NVTX; an empty object otherwise).
struct CallRange {
#ifdef LITEVLM_NVTX
    explicit CallRange(const char* name) { nvtxRangePushA(name); }
    ~CallRange() { nvtxRangePop(); }
#else
    explicit CallRange(const char*) {}
#endif
};

// Debug builds (LITEVLM_DEBUG): a device array must equal its host mirror.
// Checked before anything is enqueued, with a synchronous copy after the
// stream's earlier work (so not under stream capture); a mismatch is
// INVALID_ARG. Release builds check nothing here.
litevlm_status_t debug_mirror(litevlm_select_t h, const int32_t* d, const int32_t* host, int64_t n, const char* what,
                              litevlm_stream_t stream)
{
#ifdef LITEVLM_DEBUG
    if (!d || !host || n <= 0) return LITEVLM_OK;
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "debug mirror check");
    std::vector<int32_t> tmp((size_t)n);
    e = cudaMemcpy(tmp.data(), d, sizeof(int32_t) * (size_t)n, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(h, e, "debug mirror check");
    if (std::memcmp(tmp.data(), host, sizeof(int32_t) * (size_t)n) != 0)
        return fail(h, LITEVLM_ERR_INVALID_ARG,
                    std::string(what) + " on the device differs from its host mirror (debug build)");
#else
    (void)h;
    (void)d;
    (void)host;
    (void)n;
    (void)what;
    (void)stream;
#endif
    return LITEVLM_OK;
}

// Checks an offsets mirror: offs[0] = 0, non-decreasing, total within `max_total`.
litevlm_status_t check_offsets(litevlm_select_t h, const int32_t* offs, int32_t batch, int64_t max_total,
                               const char* name, int64_t* total)
{
    if (!offs) return fail(h, LITEVLM_ERR_INVALID_ARG, std::string(name) + " host mirror is NULL");
    if (offs[0] != 0) return fail(h, LITEVLM_ERR_INVALID_ARG, std::string(name) + "[0] must be 0");
    for (int32_t b = 0; b < batch; ++b)
        if (offs[b + 1] < offs[b])
            return fail(h, LITEVLM_ERR_INVALID_ARG, std::string(name) + " must be non-decreasing (request " +
                                                        std::to_string(b) + ")");
    *total = offs[batch];
    if (*total > max_total)
        return fail(h, LITEVLM_ERR_WORKSPACE, std::string(name) + " total " + std::to_string(*total) +
                                                  " exceeds the handle maximum " + std::to_string(max_total));
    return LITEVLM_OK;
}

int64_t keep_count_host(int32_t n, float ratio)
{
    double kd = floor((double)ratio * (double)n);
    if (kd < 0) kd = 0;
    if (kd > n) kd = n;
    return (int64_t)kd;
}

litevlm_status_t encode_rows_map(litevlm_select_t h, CUtensorMap* map, const void* base, int32_t head_dim,
                                 int32_t heads, int64_t rows, int box_rows, bool fp8, const char* what)
{
    const int esize = fp8 ? 1 : 2;
    const cuuint64_t dims[3] = {(cuuint64_t)head_dim, (cuuint64_t)heads, (cuuint64_t)rows};
    const cuuint64_t strides[2] = {(cuuint64_t)head_dim * esize, (cuuint64_t)heads * head_dim * esize};
    const cuuint32_t box[3] = {(cuuint32_t)(128 / esize), 1u, (cuuint32_t)box_rows};
    const cuuint32_t estride[3] = {1u, 1u, 1u};
    const CUresult r = h->encode(map, fp8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3,
                                 const_cast<void*>(base), dims, strides, box, estride,
                                 CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                 CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS)
        return fail(h, LITEVLM_ERR_CUDA, std::string("cuTensorMapEncodeTiled failed for ") + what + " (" +
                                             std::to_string((int)r) + ")");
    return LITEVLM_OK;
}

struct ScoreChoice {
    bool resident;
    lvs::ScorePlan plan;
};

// Picks the score kernel and its launch shape. Cost unit: one tile-head of
// the resident kernel with one TMEM head buffer (its MMAs, then its epilogue;
// about 1.2 us at 64 text columns on GB300). A CTA also pays ~6 units (launch,
// TMEM, pipeline fill) and, with one buffer, ~1 unit per head for the cluster
// exchange. With two buffers the MMAs and the statistics exchange overlap the
// epilogue, which then costs ~0.6 units per tile-head plus ~2.1 per head
// (measured on GB300 at 3 tiles per CTA), and a head takes at least the time
// its K tiles need at the CTA's share of HBM bandwidth. Waves of CTAs come from the measured
// cluster occupancy of the kernel. The re-read kernel streams every K tile
// twice (weight 1.6).
// True when every request has the same, non-zero, visual and text token
// counts (the resident kernel's flattened schedule needs it).
bool uniform_batch(int batch, const int32_t* seq_offsets_h, const int32_t* text_offsets_h)
{
    if (batch < 1) return false;
    const int32_t n = seq_offsets_h[1] - seq_offsets_h[0], t = text_offsets_h[1] - text_offsets_h[0];
    if (n <= 0 || t <= 0) return false;
    for (int32_t b = 1; b < batch; ++b)
        if (seq_offsets_h[b + 1] - seq_offsets_h[b] != n || text_offsets_h[b + 1] - text_offsets_h[b] != t) return false;
    return true;
}

ScoreChoice choose_score_kernel(litevlm_select_t h, int batch, const int32_t* seq_offsets_h, int max_t, int row_bytes,
                                bool fp8, bool uniform = false)
{
    const litevlm_select_config_t& c = h->cfg;
    const int hq = c.num_q_heads;
    const int mrows = max_t <= 64 ? 64 : 128;
    const int slot_cols = (max_t + 15) & ~15;
    // the batch's tiles per request, largest first; the memo key hashes them
    int td_small[4096];
    int* td = td_small;
    if (batch > 4096) {
        h->tiles_desc.resize((size_t)batch);
        td = h->tiles_desc.data();
    }
    for (int b = 0; b < batch; ++b) td[b] = (seq_offsets_h[b + 1] - seq_offsets_h[b] + lvs::kTileRows - 1) / lvs::kTileRows;
    std::sort(td, td + batch, [](int x, int y) { return x > y; });
    uint64_t key = 1469598103934665603ull;
    auto mix = [&](uint64_t v) { key = (key ^ v) * 1099511628211ull; };
    mix((uint64_t)batch);
    mix((uint64_t)max_t);
    mix((uint64_t)hq);
    mix((uint64_t)c.num_kv_heads);
    mix((uint64_t)row_bytes);
    mix((uint64_t)c.flags);
    mix((uint64_t)(uniform && h->allow_flat));
    for (int b = 0; b < batch; ++b) mix((uint64_t)td[b]);
    for (const auto& m : h->plan_memo)
        if (m.used && m.key == key) return ScoreChoice{m.resident, m.plan};
    const lvs::BatchTiles bt{td, batch};

    const int cmax = lvs::res_max_cluster(row_bytes, slot_cols);
    const double unit_s = 1.17e-6, hbm_bytes_per_s = 6.8e12;
    const double tile_bytes = (double)lvs::kTileRows * row_bytes;
    double tc_cost = 0.0;
    int* tcap = h->tc_capacity[mrows == 64 ? 0 : 1];
    for (int cl = 1; cl <= lvs::kMaxCluster; ++cl)
        if (tcap[cl] < 0) tcap[cl] = lvs::tc_cluster_capacity(row_bytes, fp8, mrows, cl);
    ScoreChoice best{false, lvs::plan_score(bt, hq, c.num_kv_heads, lvs::kTileRows * row_bytes, tcap, &tc_cost)};
    double best_cost = 1.6 * tc_cost;
    const int max_tiles = batch > 0 ? td[0] : 0;
    const bool split_queries = (c.flags & LITEVLM_FLAG_SCORE_SPLIT_QUERIES) != 0;
    const int kflags = c.flags & ~(LITEVLM_FLAG_QUERY_LAST_TOKEN | LITEVLM_FLAG_SCORE_SPLIT_QUERIES);
    if (kflags == LITEVLM_FLAG_SCORE_RESIDENT || kflags == LITEVLM_FLAG_SCORE_RESIDENT_ONE_BUFFER ||
        kflags == LITEVLM_FLAG_SCORE_RESIDENT_TWO_BUFFERS || kflags == LITEVLM_FLAG_SCORE_RESIDENT_FLAT)
        best_cost = 1e300;
    // Query split (LITEVLM_FLAG_SCORE_SPLIT_QUERIES, T > 64): the resident plans
    // run each head's text rows as two pseudo-heads of at most 64 rows on the
    // 64-row kernel (the second half re-reads the head's K tiles, from L2). The
    // partial-row workspace holds Hq rows, so a request's rows come in at most
    // Hq parts.
    const bool split = split_queries && max_t > 64 && !(c.flags & LITEVLM_FLAG_QUERY_LAST_TOKEN);
    for (int qs = split ? 2 : 1; qs <= (split ? 2 : 1) && kflags != LITEVLM_FLAG_SCORE_REREAD; ++qs) {
        const int mrows_r = qs == 2 ? 64 : mrows;
        const int slot_r = qs == 2 ? (((max_t + 1) / 2 + 15) & ~15) : slot_cols;
        const int hq_r = hq * qs;
        const int cmax = lvs::res_max_cluster(row_bytes, slot_r);
        int* rcap = h->res_capacity[mrows_r == 64 ? 0 : 1];
        for (int nb = 1; nb <= 2; ++nb) {
            if (nb == 2 && (kflags == LITEVLM_FLAG_SCORE_RESIDENT_ONE_BUFFER || kflags == LITEVLM_FLAG_SCORE_RESIDENT_FLAT))
                continue;
            if (nb == 1 && kflags == LITEVLM_FLAG_SCORE_RESIDENT_TWO_BUFFERS) continue;
            const int R = lvs::res_max_tiles(slot_r, nb);
            for (int cl = 1; cl <= cmax; ++cl) {
                const int tpc = (max_tiles + cl - 1) / cl;
                if (tpc > R) continue;
                if (cl > 1 && (cl - 1) * tpc >= max_tiles) continue;  // an idle rank on the largest request
                int& cap = rcap[cl];
                if (cap < 0) cap = lvs::res_cluster_capacity(row_bytes, fp8, mrows_r, cl);
                if (cap <= 0) continue;
                for (int g = 1; g <= hq; ++g) {
                    if (hq_r % g) continue;
                    const int hpg = hq_r / g;
                    if (nb == 2 && hpg < 2) continue;  // nothing to overlap
                    const long long ctas = (long long)batch * cl * g;
                    const double active = (double)(ctas < cap ? ctas : cap);
                    auto item_cost = [&](int tiles) {
                        if (tiles <= 0) return 1.0;
                        const int t = (tiles + cl - 1) / cl;
                        double per_head;
                        if (nb == 1) {
                            per_head = (double)t + (cl > 1 ? 1.0 : 0.25);
                        } else {
                            const double stream = t * tile_bytes * active / hbm_bytes_per_s / unit_s;
                            per_head = 0.6 * t + 2.1;
                            if (stream > per_head) per_head = stream;
                        }
                        return 6.0 + (g > 1 ? 2.0 : 0.0) + hpg * per_head;
                    };
                    const double cost = lvs::makespan(bt, g, cap / cl, item_cost);
                    if (cost < best_cost - 1e-9) {
                        best_cost = cost;
                        lvs::ScorePlan pl{cl, tpc, g};
                        pl.res_nb = nb;
                        pl.qsplit = qs;
                        best = ScoreChoice{true, pl};
                    }
                }
            }
        }
        // Flattened schedule (every request the same size, one TMEM head buffer):
        // the batch's (request, head) pairs split evenly over every cluster that
        // fits on the GPU at once, so there is no partial last wave; the clusters
        // run their pairs back to back and each request boundary costs a write of
        // the request's rows (a fold where a request spans two clusters).
        if (uniform && h->allow_flat && kflags != LITEVLM_FLAG_SCORE_RESIDENT_TWO_BUFFERS) {
            const int R = lvs::res_max_tiles(slot_r, 1);
            const long long pairs = (long long)batch * hq_r;
            for (int cl = 1; cl <= cmax; ++cl) {
                const int tpc = (max_tiles + cl - 1) / cl;
                if (tpc > R) continue;
                if (cl > 1 && (cl - 1) * tpc >= max_tiles) continue;
                int& cap = rcap[cl];
                if (cap < 0) cap = lvs::res_cluster_capacity(row_bytes, fp8, mrows_r, cl);
                if (cap <= 0) continue;
                long long nclu = cap / cl;
                if (nclu > pairs) nclu = pairs;
                if (nclu > lvs::kFlatMax) nclu = lvs::kFlatMax;
                if (nclu < 1) continue;
                // clusters a request's pairs reach (its partial rows), at most Hq
                int parts = 1;
                for (int b = 0, k0 = 0; b < batch; ++b) {
                    const long long first = (long long)b * hq_r, last = first + hq_r - 1;
                    while (k0 + 1 < nclu && pairs * (k0 + 1) / nclu <= first) ++k0;
                    int k1 = k0;
                    while (k1 + 1 < nclu && pairs * (k1 + 1) / nclu <= last) ++k1;
                    if (k1 - k0 + 1 > parts) parts = k1 - k0 + 1;
                }
                if (parts > hq) continue;
                const double per_head = (double)tpc + (cl > 1 ? 1.0 : 0.25);
                const long long per_cluster = (pairs + nclu - 1) / nclu;
                const double boundaries = (double)per_cluster / hq_r + 1.0;
                double cost = 6.0 + (double)per_cluster * per_head + 2.0 * boundaries;
                if (kflags == LITEVLM_FLAG_SCORE_RESIDENT_FLAT) cost -= 1e200;  // forced: any flat plan beats the others
                if (cost < best_cost - 1e-9) {
                    best_cost = cost;
                    lvs::ScorePlan pl{cl, tpc, 1};
                    pl.res_nb = 1;
                    pl.flat = (int)nclu;
                    pl.qsplit = qs;
                    best = ScoreChoice{true, pl};
                }
            }
        }
    }
    auto& m = h->plan_memo[h->plan_memo_next];
    h->plan_memo_next = (h->plan_memo_next + 1) & 3;
    m.key = key;
    m.used = true;
    m.resident = best.resident;
    m.plan = best.plan;
    return best;
}

}  // namespace

extern "C" {

const char* litevlm_status_string(litevlm_status_t s)
{
    const CallRange range_(__func__);
    switch (s) {
    case LITEVLM_OK: return "ok";
    case LITEVLM_ERR_INVALID_ARG: return "invalid argument";
    case LITEVLM_ERR_UNSUPPORTED: return "unsupported shape or type";
    case LITEVLM_ERR_WORKSPACE: return "beyond the handle's configured maxima";
    case LITEVLM_ERR_CUDA: return "CUDA error";
    case LITEVLM_ERR_TIMEOUT: return "device-side wait timed out";
    case LITEVLM_ERR_DEVICE_BOUNDS: return "device-side index out of bounds";
    }
    return "unknown status";
}

const char* litevlm_select_last_error(litevlm_select_t h)
{
    const CallRange range_(__func__);
    return h ? h->last_error.c_str() : g_create_error.c_str();
}

int32_t litevlm_select_last_launches(litevlm_select_t h) { return h ? h->last_launches : 0; }

litevlm_status_t litevlm_select_create(const litevlm_select_config_t* c, litevlm_select_t* out)
{
    const CallRange range_(__func__);
    g_create_error.clear();
    if (!out) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (!c) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "config is NULL");
    if (c->max_batch <= 0 || c->max_total_visual <= 0 || c->max_total_text <= 0)
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "max_batch, max_total_visual, max_total_text must be > 0");
    if (c->max_total_visual > INT32_MAX || c->max_total_text > INT32_MAX)
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "totals must fit in int32 row indices");
    if (c->num_q_heads <= 0 || c->num_kv_heads <= 0 || c->num_q_heads % c->num_kv_heads != 0)
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "num_q_heads must be a positive multiple of num_kv_heads");
    if (c->qk_dtype != LITEVLM_BF16 && c->qk_dtype != LITEVLM_FP8_E4M3)
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "qk_dtype must be LITEVLM_BF16 or LITEVLM_FP8_E4M3");
    const int kflags = c->flags & ~(LITEVLM_FLAG_QUERY_LAST_TOKEN | LITEVLM_FLAG_SCORE_SPLIT_QUERIES);
    if (c->flags < 0 || (kflags != 0 && kflags != LITEVLM_FLAG_SCORE_REREAD && kflags != LITEVLM_FLAG_SCORE_RESIDENT &&
                         kflags != LITEVLM_FLAG_SCORE_RESIDENT_ONE_BUFFER &&
                         kflags != LITEVLM_FLAG_SCORE_RESIDENT_TWO_BUFFERS && kflags != LITEVLM_FLAG_SCORE_RESIDENT_FLAT))
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "flags must be 0 or one LITEVLM_FLAG_SCORE_* value");
    if (c->head_dim <= 0) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "head_dim must be > 0");
    if (!lvs::score_shape_supported(c->head_dim, c->qk_dtype == LITEVLM_FP8_E4M3))
        return fail(nullptr, LITEVLM_ERR_UNSUPPORTED,
                    "head_dim " + std::to_string(c->head_dim) + " has no kernel for this dtype (bf16: 64, 128; e4m3: 128)");

    litevlm_select* h = new (std::nothrow) litevlm_select();
    if (!h) return fail(nullptr, LITEVLM_ERR_CUDA, "out of host memory");
    h->cfg = *c;
    for (auto& row : h->tc_capacity)
        for (int& v : row) v = -1;
    for (auto& row : h->res_capacity)
        for (int& v : row) v = -1;
    cudaError_t e = cudaGetDevice(&h->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, h->device);
    if (e == cudaSuccess) {
        int major = 0, minor = 0;
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, h->device);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, h->device);
        if (major != 10) {
            delete h;
            return fail(nullptr, LITEVLM_ERR_UNSUPPORTED,
                        "needs a Blackwell (sm_10x) GPU, found sm_" + std::to_string(major) + std::to_string(minor));
        }
    }
    if (e == cudaSuccess) {
        void* fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e == cudaSuccess && (q != cudaDriverEntryPointSuccess || !fn)) e = cudaErrorNotSupported;
        h->encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    if (e == cudaSuccess) e = cudaMalloc(&h->err_d, sizeof(int32_t));
    if (e == cudaSuccess) e = cudaMemset(h->err_d, 0, sizeof(int32_t));
    if (e == cudaSuccess && c->num_q_heads > 1)
        e = cudaMalloc(&h->partials, sizeof(float) * (size_t)c->num_q_heads * (size_t)c->max_total_visual);
    // one fold ticket per 128-token tile: index floor(n0 / 128) + t + b < total / 128 + 2 * batch + 1
    h->n_counters = (size_t)(c->max_total_visual / lvs::kTileRows) + 2 * (size_t)c->max_batch + 2;
    if (e == cudaSuccess) e = cudaMalloc(&h->counters, sizeof(int32_t) * h->n_counters);
    if (e == cudaSuccess) e = cudaMemset(h->counters, 0, sizeof(int32_t) * h->n_counters);
    if (e == cudaSuccess)
        e = cudaMalloc(&h->ctx_stats, sizeof(float) * (size_t)c->num_q_heads * (size_t)c->max_total_text);
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) {
        const std::string msg = std::string("create: ") + cudaGetErrorString(e);
        if (h->counters) cudaFree(h->counters);
        if (h->err_d) cudaFree(h->err_d);
        if (h->partials) cudaFree(h->partials);
        if (h->ctx_stats) cudaFree(h->ctx_stats);
        delete h;
        cudaGetLastError();
        return fail(nullptr, LITEVLM_ERR_CUDA, msg);
    }
    *out = h;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_destroy(litevlm_select_t h)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_OK;
    if (h->partials) cudaFree(h->partials);
    if (h->counters) cudaFree(h->counters);
    if (h->err_d) cudaFree(h->err_d);
    if (h->ctx_stats) cudaFree(h->ctx_stats);
    delete h;
    return LITEVLM_OK;
}

namespace {
struct ScoreShape {
    int64_t tot_n = 0, tot_t = 0;
    int max_tiles = 0, max_n = 0, max_t = 0;
};

litevlm_status_t check_score_shape(litevlm_select_t h, int32_t batch, const int32_t* text_offsets_h,
                                   const int32_t* seq_offsets_h, ScoreShape* sh)
{
    const litevlm_select_config_t& c = h->cfg;
    if (batch < 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "batch must be >= 0");
    if (batch > c.max_batch) return fail(h, LITEVLM_ERR_WORKSPACE, "batch exceeds max_batch");
    if (batch == 0) return LITEVLM_OK;
    litevlm_status_t s = check_offsets(h, seq_offsets_h, batch, c.max_total_visual, "seq_offsets", &sh->tot_n);
    if (s != LITEVLM_OK) return s;
    s = check_offsets(h, text_offsets_h, batch, c.max_total_text, "text_offsets", &sh->tot_t);
    if (s != LITEVLM_OK) return s;
    for (int32_t b = 0; b < batch; ++b) {
        const int32_t n = seq_offsets_h[b + 1] - seq_offsets_h[b];
        const int32_t t = text_offsets_h[b + 1] - text_offsets_h[b];
        if (n > 0 && t == 0)
            return fail(h, LITEVLM_ERR_INVALID_ARG,
                        "request " + std::to_string(b) + " has visual tokens but no text query token");
        const bool last_only = (h->cfg.flags & LITEVLM_FLAG_QUERY_LAST_TOKEN) != 0;
        if (t > lvs::kMaxText && !last_only)
            return fail(h, LITEVLM_ERR_UNSUPPORTED, "request " + std::to_string(b) + " has " + std::to_string(t) +
                                                        " text tokens; the score kernel handles at most 128");
        if (n > 65536)
            return fail(h, LITEVLM_ERR_UNSUPPORTED,
                        "request " + std::to_string(b) + " has more than 65536 visual tokens");
        const int tiles = (n + lvs::kTileRows - 1) / lvs::kTileRows;
        if (tiles > sh->max_tiles) sh->max_tiles = tiles;
        if (n > sh->max_n) sh->max_n = n;
        const int tq = last_only && t > 0 ? 1 : t;  // query rows the kernels use
        if (n > 0 && tq > sh->max_t) sh->max_t = tq;
    }
    return LITEVLM_OK;
}
}  // namespace

litevlm_status_t litevlm_select_score_plan(litevlm_select_t h, int32_t batch, const int32_t* text_offsets_h,
                                           const int32_t* seq_offsets_h, int32_t* plan)
{
    const CallRange range_(__func__);
    if (!h || !plan) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    ScoreShape sh;
    const litevlm_status_t s = check_score_shape(h, batch, text_offsets_h, seq_offsets_h, &sh);
    if (s != LITEVLM_OK) return s;
    plan[0] = plan[1] = plan[2] = plan[3] = 0;
    if (batch == 0 || sh.tot_n == 0) return LITEVLM_OK;
    const bool fp8 = h->cfg.qk_dtype == LITEVLM_FP8_E4M3;
    const ScoreChoice ch = choose_score_kernel(h, batch, seq_offsets_h, sh.max_t, h->cfg.head_dim * (fp8 ? 1 : 2), fp8,
                                               uniform_batch(batch, seq_offsets_h, text_offsets_h));
    plan[0] = !ch.resident ? 1 : (ch.plan.flat > 0 ? 4 : 1 + ch.plan.res_nb) + (ch.plan.qsplit == 2 ? 3 : 0);
    plan[1] = ch.plan.cluster;
    plan[2] = ch.plan.tiles_per_cta;
    plan[3] = ch.plan.flat > 0 ? ch.plan.flat : ch.plan.groups;
    return LITEVLM_OK;
}

namespace {
// Keys beyond the visual tokens for the full-key-set normaliser (null: none).
struct CtxKeys {
    const void* k_sys;
    const int32_t* sys_offsets_d;
    const int32_t* sys_offsets_h;
    const void* k_text;
};

litevlm_status_t score_impl(litevlm_select_t h, int32_t batch, const void* q_text, const int32_t* text_offsets_d,
                            const int32_t* text_offsets_h, const void* k_vis, const int32_t* seq_offsets_d,
                            const int32_t* seq_offsets_h, float q_scale, float k_scale, float* scores,
                            const CtxKeys* ctx, litevlm_stream_t stream, bool allow_defer = false,
                            int* deferred_groups = nullptr, size_t clear_tickets = 0)
{
    if (deferred_groups) *deferred_groups = 0;
    const litevlm_select_config_t& c = h->cfg;
    const bool fp8 = c.qk_dtype == LITEVLM_FP8_E4M3;
    ScoreShape sh;
    litevlm_status_t s = check_score_shape(h, batch, text_offsets_h, seq_offsets_h, &sh);
    if (s != LITEVLM_OK) return s;
    if (batch == 0) return LITEVLM_OK;
    const int64_t tot_n = sh.tot_n, tot_t = sh.tot_t;
    const int max_t = sh.max_t;
    if (tot_n == 0) return LITEVLM_OK;
    if (!q_text || !k_vis || !scores || !text_offsets_d || !seq_offsets_d)
        return fail(h, LITEVLM_ERR_INVALID_ARG, "a device pointer is NULL");
    if (!aligned16(q_text) || !aligned16(k_vis))
        return fail(h, LITEVLM_ERR_INVALID_ARG, "q_text and k_vis must be 16-byte aligned");
    if (fp8) {
        if (!(q_scale > 0.f) || !(k_scale > 0.f) || isinf(q_scale) || isinf(k_scale))
            return fail(h, LITEVLM_ERR_INVALID_ARG, "e4m3 scales must be finite and > 0");
    } else if (q_scale != 1.f || k_scale != 1.f) {
        return fail(h, LITEVLM_ERR_INVALID_ARG, "q_scale and k_scale must be 1 for bf16 inputs");
    }
    const int row_bytes = c.head_dim * (fp8 ? 1 : 2);
    if (ctx) {
        if (!ctx->sys_offsets_d || !ctx->sys_offsets_h)
            return fail(h, LITEVLM_ERR_INVALID_ARG, "sys_offsets_d and sys_offsets_h are required");
        int64_t tot_s = 0;
        s = check_offsets(h, ctx->sys_offsets_h, batch, INT32_MAX, "sys_offsets", &tot_s);
        if (s != LITEVLM_OK) return s;
        if (!ctx->k_text || (tot_s > 0 && !ctx->k_sys))
            return fail(h, LITEVLM_ERR_INVALID_ARG, "k_text (and k_sys when sum S_b > 0) must not be NULL");
        if (!aligned16(ctx->k_text) || (ctx->k_sys && !aligned16(ctx->k_sys)))
            return fail(h, LITEVLM_ERR_INVALID_ARG, "k_sys and k_text must be 16-byte aligned");
    }
    s = debug_mirror(h, seq_offsets_d, seq_offsets_h, (int64_t)batch + 1, "seq_offsets", stream);
    if (s == LITEVLM_OK) s = debug_mirror(h, text_offsets_d, text_offsets_h, (int64_t)batch + 1, "text_offsets", stream);
    if (s == LITEVLM_OK && ctx)
        s = debug_mirror(h, ctx->sys_offsets_d, ctx->sys_offsets_h, (int64_t)batch + 1, "sys_offsets", stream);
    if (s != LITEVLM_OK) return s;
    const ScoreChoice choice = choose_score_kernel(h, batch, seq_offsets_h, max_t, row_bytes, fp8,
                                                   uniform_batch(batch, seq_offsets_h, text_offsets_h));
    const lvs::ScorePlan& plan = choice.plan;
    if (plan.tiles_per_cta > lvs::kMaxTilesPerCta)
        return fail(h, LITEVLM_ERR_UNSUPPORTED, "request too long for one cluster");
    const bool qsplit = choice.resident && plan.qsplit == 2;
    const int mrows = max_t <= 64 || qsplit ? 64 : 128;  // text rows of a head's (pseudo-head's) MMA

    CUtensorMap tm_q, tm_k;
    s = encode_rows_map(h, &tm_q, q_text, c.head_dim, c.num_q_heads, tot_t, mrows, fp8, "q_text");
    if (s != LITEVLM_OK) return s;
    s = encode_rows_map(h, &tm_k, k_vis, c.head_dim, c.num_kv_heads, tot_n, lvs::kTileRows, fp8, "k_vis");
    if (s != LITEVLM_OK) return s;

    lvs::ScoreLaunch p{};
    p.seq_off = seq_offsets_d;
    p.text_off = text_offsets_d;
    p.out = scores;
    p.partials = h->partials;
    p.counters = h->counters;
    p.err = h->err_d;
    p.total_vis = tot_n;
    p.hq = c.num_q_heads;
    p.hkv = c.num_kv_heads;
    p.c_log2 = (float)((double)q_scale * (double)k_scale / sqrt((double)c.head_dim) * 1.4426950408889634);
    p.wait_budget = h->wait_budget;
    p.stall = (h->debug_flags & LITEVLM_DEBUG_STALL_SCORE) != 0;
    p.slot_cols = ((qsplit ? (max_t + 1) / 2 : max_t) + 15) & ~15;
    p.qsplit = qsplit ? 2 : 1;
    p.query_last = (c.flags & LITEVLM_FLAG_QUERY_LAST_TOKEN) != 0;
    p.extra = nullptr;
    // the top-k CTA of a request reads groups x N_b partial values: worth it
    // for small requests (it saves the score kernel's ticketed fold), not for
    // long ones with many groups
    p.defer_fold = allow_defer && plan.groups > 1 && (int64_t)plan.groups * sh.max_n <= 32768;
    if (p.defer_fold && deferred_groups) *deferred_groups = plan.groups;
    if (ctx) {
        lvs::CtxArgs ca{};
        ca.q = static_cast<const uint8_t*>(q_text);
        ca.k_sys = static_cast<const uint8_t*>(ctx->k_sys);
        ca.k_txt = static_cast<const uint8_t*>(ctx->k_text);
        ca.seq_off = seq_offsets_d;
        ca.text_off = text_offsets_d;
        ca.sys_off = ctx->sys_offsets_d;
        ca.out = h->ctx_stats;
        ca.err = h->err_d;
        ca.batch = batch;
        ca.hq = c.num_q_heads;
        ca.hkv = c.num_kv_heads;
        ca.query_last = p.query_last;
        ca.c_log2 = p.c_log2;
        ca.wait_budget = h->wait_budget;
        const cudaError_t ce = lvs::launch_ctx_stats(ca, row_bytes, fp8, (cudaStream_t)stream);
        if (ce != cudaSuccess) return cuda_fail(h, ce, "context-key statistics launch");
        p.extra = h->ctx_stats;
    }
    p.nv = 0;
    if (batch <= lvs::kOffsetsByValue) {
        for (int32_t b = 0; b <= batch; ++b) {
            p.so_v[b] = seq_offsets_h[b];
            p.to_v[b] = text_offsets_h[b];
        }
        p.nv = batch;
    }
    // clusters are launched largest request first (stable: ties keep index order)
    p.order_n = 0;
    if (batch > 1 && batch <= lvs::kOrderMax) {
        int maxn = 0, minn = INT32_MAX;
        for (int32_t b = 0; b < batch; ++b) {
            const int n = seq_offsets_h[b + 1] - seq_offsets_h[b];
            maxn = n > maxn ? n : maxn;
            minn = n < minn ? n : minn;
        }
        if (maxn != minn) {
            for (int32_t b = 0; b < batch; ++b) p.order[b] = (uint16_t)b;
            std::stable_sort(p.order, p.order + batch, [&](uint16_t x, uint16_t y) {
                return seq_offsets_h[x + 1] - seq_offsets_h[x] > seq_offsets_h[y + 1] - seq_offsets_h[y];
            });
            p.order_n = batch;
        }
    }
    // a caller whose tickets may not be at rest (the no-alloc entry point's
    // shared static scratch) has them cleared here, after every host-side check
    if (clear_tickets > 0 && plan.groups > 1) {
        const cudaError_t ce = cudaMemsetAsync(h->counters, 0, sizeof(int32_t) * clear_tickets, (cudaStream_t)stream);
        if (ce != cudaSuccess) return cuda_fail(h, ce, "clearing the fold tickets");
    }
    const cudaError_t e =
        choice.resident
            ? lvs::launch_score_resident(tm_q, tm_k, p, plan, batch, row_bytes, fp8, mrows, (cudaStream_t)stream)
            : lvs::launch_score(tm_q, tm_k, p, plan, batch, row_bytes, fp8, mrows, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "score launch");
    h->last_launches = ctx ? 2 : 1;
    return LITEVLM_OK;
}
}  // namespace

litevlm_status_t litevlm_select_score(litevlm_select_t h, int32_t batch, const void* q_text,
                                      const int32_t* text_offsets_d, const int32_t* text_offsets_h,
                                      const void* k_vis, const int32_t* seq_offsets_d,
                                      const int32_t* seq_offsets_h, float q_scale, float k_scale, float* scores,
                                      litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    return score_impl(h, batch, q_text, text_offsets_d, text_offsets_h, k_vis, seq_offsets_d, seq_offsets_h,
                      q_scale, k_scale, scores, nullptr, stream);
}

litevlm_status_t litevlm_select_score_full_keys(litevlm_select_t h, int32_t batch, const void* q_text,
                                                const int32_t* text_offsets_d, const int32_t* text_offsets_h,
                                                const void* k_vis, const int32_t* seq_offsets_d,
                                                const int32_t* seq_offsets_h, const void* k_sys,
                                                const int32_t* sys_offsets_d, const int32_t* sys_offsets_h,
                                                const void* k_text, float q_scale, float k_scale, float* scores,
                                                litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    const CtxKeys ctx{k_sys, sys_offsets_d, sys_offsets_h, k_text};
    return score_impl(h, batch, q_text, text_offsets_d, text_offsets_h, k_vis, seq_offsets_d, seq_offsets_h,
                      q_scale, k_scale, scores, &ctx, stream);
}

namespace {
// Host half of the top-k: validation from the host mirrors, out_offsets_h, and
// the per-request sizes the kernels take by value (h->topk_shape). *run is
// false when there is nothing to launch (batch 0).
litevlm_status_t topk_prepare(litevlm_select_t h, int32_t batch, const float* scores, const int32_t* seq_offsets_d,
                              const int32_t* seq_offsets_h, const int32_t* keep_k_d, const int32_t* keep_k_h,
                              float keep_ratio, int32_t* kept_idx, int32_t* out_offsets_d, int32_t* out_offsets_h,
                              int* max_n_out, int64_t* total_k_out, int64_t* tot_n_out, bool* run)
{
    *run = false;
    if (batch < 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "batch must be >= 0");
    if (batch > h->cfg.max_batch) return fail(h, LITEVLM_ERR_WORKSPACE, "batch exceeds max_batch");
    if ((keep_k_d == nullptr) != (keep_k_h == nullptr))
        return fail(h, LITEVLM_ERR_INVALID_ARG, "keep_k_d and keep_k_h must be both given or both NULL");
    if (!keep_k_h && !(keep_ratio >= 0.f && keep_ratio <= 1.f))
        return fail(h, LITEVLM_ERR_INVALID_ARG, "keep_ratio must be in [0, 1]");
    if (batch == 0) {
        if (out_offsets_h) out_offsets_h[0] = 0;
        return LITEVLM_OK;
    }
    int64_t tot_n = 0;
    litevlm_status_t s = check_offsets(h, seq_offsets_h, batch, h->cfg.max_total_visual, "seq_offsets", &tot_n);
    if (s != LITEVLM_OK) return s;
    int64_t total_k = 0;
    int max_n = 0;
    std::vector<int32_t> off((size_t)batch + 1, 0);
    for (int32_t b = 0; b < batch; ++b) {
        const int32_t n = seq_offsets_h[b + 1] - seq_offsets_h[b];
        if (n > max_n) max_n = n;
        int64_t k;
        if (keep_k_h) {
            k = keep_k_h[b];
            if (k < 0 || k > n)
                return fail(h, LITEVLM_ERR_INVALID_ARG, "keep_k[" + std::to_string(b) + "] = " + std::to_string(k) +
                                                            " outside [0, " + std::to_string(n) + "]");
        } else {
            k = keep_count_host(n, keep_ratio);
        }
        total_k += k;
        off[(size_t)b + 1] = (int32_t)total_k;
    }
    if (!out_offsets_d || !seq_offsets_d) return fail(h, LITEVLM_ERR_INVALID_ARG, "a device pointer is NULL");
    if (total_k > 0 && (!kept_idx || !scores)) return fail(h, LITEVLM_ERR_INVALID_ARG, "a device pointer is NULL");
    if (out_offsets_h)
        for (int32_t b = 0; b <= batch; ++b) out_offsets_h[b] = off[(size_t)b];
    lvs::TopkShape& sh = h->topk_shape;
    sh.n = batch <= lvs::kTopkShapeMax ? batch : 0;
    sh.partials = nullptr;
    sh.groups = 0;
    for (int32_t b = 0; b < sh.n; ++b) {
        sh.n0[b] = seq_offsets_h[b];
        sh.len[b] = seq_offsets_h[b + 1] - seq_offsets_h[b];
        sh.k[b] = off[(size_t)b + 1] - off[(size_t)b];
        sh.out0[b] = off[(size_t)b];
    }
    *max_n_out = max_n;
    *total_k_out = total_k;
    *tot_n_out = tot_n;
    *run = true;
    return LITEVLM_OK;
}
}  // namespace

litevlm_status_t litevlm_select_topk(litevlm_select_t h, int32_t batch, const float* scores,
                                     const int32_t* seq_offsets_d, const int32_t* seq_offsets_h,
                                     const int32_t* keep_k_d, const int32_t* keep_k_h, float keep_ratio,
                                     int32_t* kept_idx, int32_t* out_offsets_d, int32_t* out_offsets_h,
                                     litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    int max_n = 0;
    int64_t total_k = 0, tot_n = 0;
    bool run = false;
    litevlm_status_t s = topk_prepare(h, batch, scores, seq_offsets_d, seq_offsets_h, keep_k_d, keep_k_h,
                                      keep_ratio, kept_idx, out_offsets_d, out_offsets_h, &max_n, &total_k, &tot_n,
                                      &run);
    if (s != LITEVLM_OK || !run) return s;
    s = debug_mirror(h, seq_offsets_d, seq_offsets_h, (int64_t)batch + 1, "seq_offsets", stream);
    if (s == LITEVLM_OK) s = debug_mirror(h, keep_k_d, keep_k_h, batch, "keep_k", stream);
    if (s != LITEVLM_OK) return s;
    // scores are only read (no deferred fold here)
    const cudaError_t e = lvs::launch_topk(batch, const_cast<float*>(scores), seq_offsets_d, keep_k_d, keep_ratio,
                                           kept_idx, out_offsets_d, max_n, h->topk_shape, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "topk launch");
    h->last_launches = 1;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_score_topk(litevlm_select_t h, int32_t batch, const void* q_text,
                                           const int32_t* text_offsets_d, const int32_t* text_offsets_h,
                                           const void* k_vis, const int32_t* seq_offsets_d,
                                           const int32_t* seq_offsets_h, float q_scale, float k_scale, float* scores,
                                           const int32_t* keep_k_d, const int32_t* keep_k_h, float keep_ratio,
                                           int32_t* kept_idx, int32_t* out_offsets_d, int32_t* out_offsets_h,
                                           litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    int max_n = 0;
    int64_t total_k = 0, tot_n = 0;
    bool run = false;
    litevlm_status_t s = topk_prepare(h, batch, scores, seq_offsets_d, seq_offsets_h, keep_k_d, keep_k_h,
                                      keep_ratio, kept_idx, out_offsets_d, out_offsets_h, &max_n, &total_k, &tot_n,
                                      &run);
    if (s != LITEVLM_OK) return s;
    s = debug_mirror(h, keep_k_d, keep_k_h, batch, "keep_k", stream);
    if (s != LITEVLM_OK) return s;
    // the top-k kernel can take over the head-group fold when it holds the
    // request's keys in registers and has the sizes by value
    const bool can_defer = h->topk_shape.n == batch && max_n <= 16 * 512;
    int groups = 0;
    s = score_impl(h, batch, q_text, text_offsets_d, text_offsets_h, k_vis, seq_offsets_d, seq_offsets_h, q_scale,
                   k_scale, scores, nullptr, stream, can_defer, &groups);
    if (s != LITEVLM_OK || !run) return s;
    lvs::TopkShape& sh = h->topk_shape;
    if (groups > 0) {
        const bool last_only = (h->cfg.flags & LITEVLM_FLAG_QUERY_LAST_TOKEN) != 0;
        sh.partials = h->partials;
        sh.groups = groups;
        sh.total_vis = tot_n;
        for (int32_t b = 0; b < batch; ++b) {
            const int t = text_offsets_h[b + 1] - text_offsets_h[b];
            sh.denom[b] = (float)h->cfg.num_q_heads * (float)(last_only && t > 0 ? 1 : t);
        }
    }
    const cudaError_t e = lvs::launch_topk(batch, scores, seq_offsets_d, keep_k_d, keep_ratio, kept_idx,
                                           out_offsets_d, max_n, sh, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "topk launch");
    h->last_launches = 2;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_compact(litevlm_select_t h, int64_t total_kept, const int32_t* kept_idx,
                                        int64_t src_rows, int32_t num_tensors, const void* const* src,
                                        void* const* dst, const int64_t* row_bytes, litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    if (total_kept < 0 || src_rows < 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "sizes must be >= 0");
    if (num_tensors < 1 || num_tensors > lvs::kMaxGatherTensors)
        return fail(h, LITEVLM_ERR_INVALID_ARG, "num_tensors must be in [1, 8]");
    if (!src || !dst || !row_bytes) return fail(h, LITEVLM_ERR_INVALID_ARG, "src, dst and row_bytes are required");
    lvs::GatherArgs g{};
    g.n = num_tensors;
    bool vec16 = true;
    for (int t = 0; t < num_tensors; ++t) {
        if (row_bytes[t] <= 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "row_bytes must be > 0");
        if (total_kept > 0 && (!src[t] || !dst[t]))
            return fail(h, LITEVLM_ERR_INVALID_ARG, "tensor " + std::to_string(t) + " pointer is NULL");
        g.src[t] = static_cast<const uint8_t*>(src[t]);
        g.dst[t] = static_cast<uint8_t*>(dst[t]);
        g.row_bytes[t] = row_bytes[t];
        vec16 = vec16 && (row_bytes[t] % 16 == 0) && aligned16(src[t]) && aligned16(dst[t]);
    }
    if (total_kept == 0) return LITEVLM_OK;
    if (!kept_idx) return fail(h, LITEVLM_ERR_INVALID_ARG, "kept_idx is NULL");
    const cudaError_t e =
        lvs::launch_compact(total_kept, kept_idx, src_rows, g, vec16, h->err_d, h->num_sms, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "compact launch");
    h->last_launches = 1;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_splice(litevlm_select_t h, int32_t batch, const void* sys_rows,
                                       const int32_t* sys_offsets_d, const int32_t* sys_offsets_h,
                                       const void* vis_rows, const int32_t* seq_offsets_d,
                                       const int32_t* seq_offsets_h, const int32_t* kept_idx,
                                       const int32_t* kept_offsets_d, const int32_t* kept_offsets_h,
                                       const void* txt_rows, const int32_t* text_offsets_d,
                                       const int32_t* text_offsets_h, int64_t row_bytes, void* out_rows,
                                       int32_t* out_offsets_d, int32_t* out_offsets_h, int32_t* position_ids,
                                       litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    if (batch < 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "batch must be >= 0");
    if (batch > h->cfg.max_batch) return fail(h, LITEVLM_ERR_WORKSPACE, "batch exceeds max_batch");
    if (row_bytes <= 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "row_bytes must be > 0");
    int64_t tot_s = 0, tot_n = 0, tot_k = 0, tot_t = 0;
    litevlm_status_t s = check_offsets(h, sys_offsets_h, batch, INT32_MAX, "sys_offsets", &tot_s);
    if (s == LITEVLM_OK) s = check_offsets(h, seq_offsets_h, batch, h->cfg.max_total_visual, "seq_offsets", &tot_n);
    if (s == LITEVLM_OK) s = check_offsets(h, kept_offsets_h, batch, h->cfg.max_total_visual, "kept_offsets", &tot_k);
    if (s == LITEVLM_OK) s = check_offsets(h, text_offsets_h, batch, INT32_MAX, "text_offsets", &tot_t);
    if (s != LITEVLM_OK) return s;
    int max_rows = 0;
    for (int32_t b = 0; b < batch; ++b) {
        const int64_t kb = kept_offsets_h[b + 1] - kept_offsets_h[b];
        const int64_t nb = seq_offsets_h[b + 1] - seq_offsets_h[b];
        if (kb > nb)
            return fail(h, LITEVLM_ERR_INVALID_ARG, "request " + std::to_string(b) + " keeps more rows than it has");
        const int64_t L = (sys_offsets_h[b + 1] - sys_offsets_h[b]) + kb + (text_offsets_h[b + 1] - text_offsets_h[b]);
        if (L > max_rows) max_rows = (int)L;
    }
    const int64_t tot_out = tot_s + tot_k + tot_t;
    if (tot_out > INT32_MAX) return fail(h, LITEVLM_ERR_INVALID_ARG, "output rows exceed int32 indices");
    if (out_offsets_h)
        for (int32_t b = 0; b <= batch; ++b)
            out_offsets_h[b] = sys_offsets_h[b] + kept_offsets_h[b] + text_offsets_h[b];
    if (batch == 0) return LITEVLM_OK;
    if (!sys_offsets_d || !seq_offsets_d || !kept_offsets_d || !text_offsets_d || !out_offsets_d)
        return fail(h, LITEVLM_ERR_INVALID_ARG, "a device offsets pointer is NULL");
    if ((tot_s > 0 && !sys_rows) || (tot_k > 0 && (!vis_rows || !kept_idx)) || (tot_t > 0 && !txt_rows) ||
        (tot_out > 0 && (!out_rows || !position_ids)))
        return fail(h, LITEVLM_ERR_INVALID_ARG, "a device row pointer is NULL");
    const bool vec16 = row_bytes % 16 == 0 && aligned16(sys_rows) && aligned16(vis_rows) && aligned16(txt_rows) &&
                       aligned16(out_rows);
    const int64_t nb1 = (int64_t)batch + 1;
    s = debug_mirror(h, sys_offsets_d, sys_offsets_h, nb1, "sys_offsets", stream);
    if (s == LITEVLM_OK) s = debug_mirror(h, seq_offsets_d, seq_offsets_h, nb1, "seq_offsets", stream);
    if (s == LITEVLM_OK) s = debug_mirror(h, kept_offsets_d, kept_offsets_h, nb1, "kept_offsets", stream);
    if (s == LITEVLM_OK) s = debug_mirror(h, text_offsets_d, text_offsets_h, nb1, "text_offsets", stream);
    if (s != LITEVLM_OK) return s;
    lvs::SpliceArgs a{};
    a.sys_off = sys_offsets_d;
    a.seq_off = seq_offsets_d;
    a.kept_off = kept_offsets_d;
    a.kept_idx = kept_idx;
    a.text_off = text_offsets_d;
    a.sys = static_cast<const uint8_t*>(sys_rows);
    a.vis = static_cast<const uint8_t*>(vis_rows);
    a.txt = static_cast<const uint8_t*>(txt_rows);
    a.out = static_cast<uint8_t*>(out_rows);
    a.out_off = out_offsets_d;
    a.pos = position_ids;
    a.row_bytes = row_bytes;
    a.batch = batch;
    a.err = h->err_d;
    const cudaError_t e = lvs::launch_splice(a, max_rows, vec16, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "splice launch");
    h->last_launches = 1;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_views(litevlm_select_t h, int32_t batch, int32_t num_views, const float* lexical,
                                      const float* logits, const int32_t* tokens_per_view_h, float w_lex,
                                      float w_logit, float threshold, int32_t min_views, uint8_t* view_mask,
                                      int32_t* view_offsets, int32_t* selected_views, int32_t* seq_offsets,
                                      int32_t* seq_offsets_h, litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    if (batch < 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "batch must be >= 0");
    if (num_views < 1 || num_views > lvs::kMaxViews)
        return fail(h, LITEVLM_ERR_INVALID_ARG, "num_views must be in [1, 64]");
    if (min_views < 0 || min_views > num_views)
        return fail(h, LITEVLM_ERR_INVALID_ARG, "min_views must be in [0, num_views]");
    if (!tokens_per_view_h) return fail(h, LITEVLM_ERR_INVALID_ARG, "tokens_per_view_h is NULL");
    if (isnan(threshold)) return fail(h, LITEVLM_ERR_INVALID_ARG, "threshold is NaN");
    int64_t per_request = 0;
    lvs::ViewsArgs a{};
    for (int32_t v = 0; v < num_views; ++v) {
        if (tokens_per_view_h[v] < 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "tokens_per_view must be >= 0");
        per_request += tokens_per_view_h[v];
        a.tokens_per_view[v] = tokens_per_view_h[v];
    }
    if ((int64_t)batch * per_request > INT32_MAX)
        return fail(h, LITEVLM_ERR_INVALID_ARG, "batch x tokens per request could exceed int32 offsets");
    if (!view_offsets || !seq_offsets) return fail(h, LITEVLM_ERR_INVALID_ARG, "a device pointer is NULL");
    if (batch > 0 && (!lexical || !logits || !view_mask || !selected_views))
        return fail(h, LITEVLM_ERR_INVALID_ARG, "a device pointer is NULL");
    a.lexical = lexical;
    a.logits = logits;
    a.w_lex = w_lex;
    a.w_logit = w_logit;
    a.threshold = threshold;
    a.batch = batch;
    a.num_views = num_views;
    a.min_views = min_views;
    a.view_mask = view_mask;
    a.view_offsets = view_offsets;
    a.selected_views = selected_views;
    a.seq_offsets = seq_offsets;
    cudaError_t e = lvs::launch_views(a, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "views launch");
    h->last_launches = 1;
    if (seq_offsets_h) {
        e = cudaMemcpyAsync(seq_offsets_h, seq_offsets, sizeof(int32_t) * ((size_t)batch + 1), cudaMemcpyDeviceToHost,
                            (cudaStream_t)stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize((cudaStream_t)stream);
        if (e != cudaSuccess) return cuda_fail(h, e, "views: seq_offsets to host");
    }
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_fold_norm(litevlm_select_t h, int32_t out_features, int32_t hidden, const void* w,
                                          const float* gamma, void* w_folded, litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    if (out_features <= 0 || hidden <= 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "sizes must be > 0");
    if (!w || !gamma || !w_folded) return fail(h, LITEVLM_ERR_INVALID_ARG, "a device pointer is NULL");
    const cudaError_t e = lvs::launch_fold_norm(static_cast<const __nv_bfloat16*>(w), gamma,
                                                static_cast<__nv_bfloat16*>(w_folded),
                                                (int64_t)out_features * hidden, hidden, h->num_sms,
                                                (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "fold_norm launch");
    h->last_launches = 1;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_rope_table(litevlm_select_t h, int32_t max_positions, int32_t head_dim,
                                           float rope_base, float* table, litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    if (max_positions <= 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "max_positions must be > 0");
    if (head_dim != 64 && head_dim != 128) return fail(h, LITEVLM_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    if (!(rope_base > 1.f) || isinf(rope_base)) return fail(h, LITEVLM_ERR_INVALID_ARG, "rope_base must be > 1");
    if (!table) return fail(h, LITEVLM_ERR_INVALID_ARG, "table is NULL");
    lvs::RopeArgs a{};
    a.table = reinterpret_cast<float2*>(table);
    a.max_positions = max_positions;
    a.half = head_dim / 2;
    for (int j = 0; j < a.half; ++j) a.inv_freq[j] = (float)pow((double)rope_base, -2.0 * j / (double)head_dim);
    const cudaError_t e = lvs::launch_rope_table(a, h->num_sms, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "rope_table launch");
    h->last_launches = 1;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_project(litevlm_select_t h, int64_t rows, int32_t hidden, int32_t out_features,
                                        const void* x, const void* w_folded, const float* bias, float eps,
                                        int32_t head_dim, const int32_t* positions, const float* rope_table,
                                        int32_t max_positions, float out_scale, void* y, litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    h->last_launches = 0;
    if (rows < 0 || rows > 65535LL * 128) return fail(h, LITEVLM_ERR_INVALID_ARG, "rows must be in [0, 65535 * 128]");
    if (hidden <= 0 || hidden % 8 != 0)
        return fail(h, LITEVLM_ERR_INVALID_ARG, "hidden must be a positive multiple of 8 (16-byte rows)");
    if (out_features <= 0 || out_features % 128 != 0)
        return fail(h, LITEVLM_ERR_UNSUPPORTED, "out_features must be a positive multiple of 128");
    if (head_dim != 0 && head_dim != 64 && head_dim != 128)
        return fail(h, LITEVLM_ERR_UNSUPPORTED, "head_dim must be 0 (no rotation), 64 or 128");
    if (!(eps >= 0.f) || isinf(eps)) return fail(h, LITEVLM_ERR_INVALID_ARG, "eps must be finite and >= 0");
    if (!(out_scale >= 0.f) || isinf(out_scale))
        return fail(h, LITEVLM_ERR_INVALID_ARG, "out_scale must be 0 (bf16 output) or finite and > 0 (e4m3)");
    if (rows == 0) return LITEVLM_OK;
    if (!x || !w_folded || !y) return fail(h, LITEVLM_ERR_INVALID_ARG, "a device pointer is NULL");
    if (!aligned16(x) || !aligned16(w_folded) || !aligned16(y))
        return fail(h, LITEVLM_ERR_INVALID_ARG, "x, w_folded and y must be 16-byte aligned");
    if (head_dim > 0 && (!positions || !rope_table || max_positions <= 0))
        return fail(h, LITEVLM_ERR_INVALID_ARG, "positions, rope_table and max_positions are required with RoPE");
    const int bn = lvs::proj_tile_cols(out_features);
    const int bm = lvs::proj_tile_rows(rows, out_features, h->num_sms);
    CUtensorMap tm_x, tm_w;
    litevlm_status_t s = encode_rows_map(h, &tm_x, x, hidden, 1, rows, bm, false, "x");
    if (s != LITEVLM_OK) return s;
    s = encode_rows_map(h, &tm_w, w_folded, hidden, 1, out_features, bn, false, "w_folded");
    if (s != LITEVLM_OK) return s;
    lvs::ProjArgs p{};
    p.rows = rows;
    p.hidden = hidden;
    p.out_features = out_features;
    p.head_dim = head_dim;
    p.max_positions = max_positions;
    p.eps = eps;
    p.bias = bias;
    p.positions = positions;
    p.rope = reinterpret_cast<const float2*>(rope_table);
    p.y = out_scale > 0.f ? nullptr : static_cast<__nv_bfloat16*>(y);
    p.y8 = out_scale > 0.f ? static_cast<uint8_t*>(y) : nullptr;
    p.out_inv_scale = out_scale > 0.f ? 1.f / out_scale : 0.f;
    p.err = h->err_d;
    p.wait_budget = h->wait_budget;
    const cudaError_t e = lvs::launch_proj(tm_x, tm_w, p, bm, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(h, e, "project launch");
    h->last_launches = 1;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_check_device(litevlm_select_t h, litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    int32_t word = 0;
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e == cudaSuccess) e = cudaMemcpy(&word, h->err_d, sizeof(word), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && word) e = cudaMemset(h->err_d, 0, sizeof(int32_t));
    // a score kernel that gave up may have taken only some of its fold tickets
    if (e == cudaSuccess && (word & lvs::kErrTimeout)) e = cudaMemset(h->counters, 0, sizeof(int32_t) * h->n_counters);
    if (e != cudaSuccess) return cuda_fail(h, e, "check_device");
    if (word & lvs::kErrTimeout) return fail(h, LITEVLM_ERR_TIMEOUT, "a device-side wait timed out");
    if (word & lvs::kErrBounds) return fail(h, LITEVLM_ERR_DEVICE_BOUNDS, "a gather index was out of bounds");
    if (word & lvs::kErrShape) return fail(h, LITEVLM_ERR_UNSUPPORTED, "a request shape reached the kernel unchecked");
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_host_view(litevlm_select_t h, const void* host, void** device_view)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    if (!host || !device_view) return fail(h, LITEVLM_ERR_INVALID_ARG, "host and device_view must not be NULL");
    void* d = nullptr;
    const cudaError_t e = cudaHostGetDevicePointer(&d, const_cast<void*>(host), 0);
    if (e != cudaSuccess || !d) {
        (void)cudaGetLastError();  // not sticky: leave no error behind for the next call
        return fail(h, LITEVLM_ERR_INVALID_ARG, "the runtime gives this host memory no device address");
    }
    *device_view = d;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_keep_offsets(int32_t batch, const int32_t* seq_offsets_h, const int32_t* keep_k_h,
                                             float keep_ratio, int32_t* out_offsets_h)
{
    const CallRange range_(__func__);
    g_create_error.clear();
    if (batch < 0) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "batch must be >= 0");
    if (!out_offsets_h) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "out_offsets_h is NULL");
    if (!keep_k_h && !(keep_ratio >= 0.f && keep_ratio <= 1.f))
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "keep_ratio must be in [0, 1]");
    if (batch == 0) {
        out_offsets_h[0] = 0;
        return LITEVLM_OK;
    }
    int64_t tot_n = 0;
    litevlm_status_t s = check_offsets(nullptr, seq_offsets_h, batch, INT32_MAX, "seq_offsets", &tot_n);
    if (s != LITEVLM_OK) return s;
    for (int32_t b = 0; b < batch; ++b) {
        const int32_t n = seq_offsets_h[b + 1] - seq_offsets_h[b];
        const int64_t k = keep_k_h ? (int64_t)keep_k_h[b] : keep_count_host(n, keep_ratio);
        if (k < 0 || k > n)
            return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "keep_k[" + std::to_string(b) + "] = " + std::to_string(k) +
                                                              " outside [0, " + std::to_string(n) + "]");
    }
    // written only once every request is known to be valid
    out_offsets_h[0] = 0;
    int64_t run = 0;
    for (int32_t b = 0; b < batch; ++b) {
        const int32_t n = seq_offsets_h[b + 1] - seq_offsets_h[b];
        run += keep_k_h ? (int64_t)keep_k_h[b] : keep_count_host(n, keep_ratio);
        out_offsets_h[b + 1] = (int32_t)run;
    }
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_set_debug_flags(litevlm_select_t h, int32_t flags)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    if (flags & ~LITEVLM_DEBUG_STALL_SCORE) return fail(h, LITEVLM_ERR_INVALID_ARG, "unknown debug flag");
    h->debug_flags = flags;
    return LITEVLM_OK;
}

litevlm_status_t litevlm_select_set_wait_budget(litevlm_select_t h, int64_t cycles)
{
    const CallRange range_(__func__);
    if (!h) return LITEVLM_ERR_INVALID_ARG;
    h->last_error.clear();
    if (cycles < 0) return fail(h, LITEVLM_ERR_INVALID_ARG, "cycles must be >= 0 (0 restores the default)");
    h->wait_budget = cycles == 0 ? lvs::kWaitBudgetCycles : (long long)cycles;
    return LITEVLM_OK;
}

}  // extern "C"

// ----------------------------------------------------------------------------
// litevlm_select_score_noalloc: the score kernels with their scratch in
// static device arrays of this library instead of a handle's workspace.
//
// Some callers may not allocate device memory at the moment they score: an
// inference engine that plans every buffer of a model when it is built and
// hands its plugins no allocator at run time, or a real-time pipeline (such
// as an in-vehicle one) that forbids allocation after start-up because
// cudaMalloc can block, synchronise the device and fail when memory is
// fragmented. Such callers cannot create a handle on the hot path. This entry
// point needs no handle: the fold partials and tickets live in the arrays
// below (fixed size, loaded with the library's device code), the device
// error word is the caller's, and the launch path is the one
// litevlm_select_score takes, run on a handle built on the stack.
// ----------------------------------------------------------------------------
namespace {

constexpr int64_t kNoAllocPartialFloats = int64_t(1) << 20;  // 4 MiB of per-head-group partial scores
constexpr int64_t kNoAllocTickets = int64_t(1) << 14;        // 64 KiB of fold tickets
constexpr int kNoAllocMaxDevices = 64;

static __device__ __align__(256) float g_noalloc_partials[kNoAllocPartialFloats];
static __device__ __align__(256) int32_t g_noalloc_tickets[kNoAllocTickets];

struct NoAllocDevice {
    bool ready = false;
    int num_sms = 0;
    float* partials = nullptr;
    int32_t* tickets = nullptr;
    PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
    int res_capacity[3][2][17];  // by kernel family (bf16 d=128, bf16 d=64, e4m3), as in the handle
    int tc_capacity[3][2][17];
    litevlm_select::PlanMemo plan_memo[3][4];
    int plan_memo_next[3] = {0, 0, 0};
};

NoAllocDevice g_noalloc[kNoAllocMaxDevices];
std::mutex g_noalloc_mutex;

int noalloc_family(int32_t head_dim, litevlm_dtype_t dtype)
{
    if (dtype == LITEVLM_FP8_E4M3) return 2;
    return head_dim == 128 ? 0 : 1;
}

// One-time setup of a device (under g_noalloc_mutex, that device current):
// the addresses of the static arrays on it, its SM count and the TMA
// descriptor encoder. The symbol lookup may load this library's device code
// (and with it the arrays) onto the device.
litevlm_status_t noalloc_setup(int dev, NoAllocDevice& d)
{
    if (d.ready) return LITEVLM_OK;
    int major = 0;
    cudaError_t e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    if (e == cudaSuccess && major != 10) return fail(nullptr, LITEVLM_ERR_UNSUPPORTED, "needs a Blackwell (sm_10x) GPU");
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev);
    void* pp = nullptr;
    void* tp = nullptr;
    if (e == cudaSuccess) e = cudaGetSymbolAddress(&pp, g_noalloc_partials);
    if (e == cudaSuccess) e = cudaGetSymbolAddress(&tp, g_noalloc_tickets);
    void* fn = nullptr;
    if (e == cudaSuccess) {
        cudaDriverEntryPointQueryResult q;
        e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
        if (e == cudaSuccess && (q != cudaDriverEntryPointSuccess || !fn)) e = cudaErrorNotSupported;
    }
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(nullptr, LITEVLM_ERR_CUDA, std::string("score_noalloc setup: ") + cudaGetErrorString(e));
    }
    d.partials = static_cast<float*>(pp);
    d.tickets = static_cast<int32_t*>(tp);
    d.encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    for (auto& fam : d.res_capacity)
        for (auto& row : fam)
            for (int& v : row) v = -1;
    for (auto& fam : d.tc_capacity)
        for (auto& row : fam)
            for (int& v : row) v = -1;
    d.ready = true;
    return LITEVLM_OK;
}

}  // namespace

extern "C" litevlm_status_t litevlm_select_score_noalloc(int32_t num_q_heads, int32_t num_kv_heads, int32_t head_dim,
                                                         litevlm_dtype_t qk_dtype, int32_t batch, const void* q_text,
                                                         const int32_t* text_offsets_d, const int32_t* text_offsets_h,
                                                         const void* k_vis, const int32_t* seq_offsets_d,
                                                         const int32_t* seq_offsets_h, float q_scale, float k_scale,
                                                         float* scores, int32_t* err_d, litevlm_stream_t stream)
{
    const CallRange range_(__func__);
    g_create_error.clear();
    // ---- host-only checks, before any CUDA call
    if (num_q_heads <= 0 || num_kv_heads <= 0 || num_q_heads % num_kv_heads != 0)
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "num_q_heads must be a positive multiple of num_kv_heads");
    if (qk_dtype != LITEVLM_BF16 && qk_dtype != LITEVLM_FP8_E4M3)
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "qk_dtype must be LITEVLM_BF16 or LITEVLM_FP8_E4M3");
    if (head_dim <= 0) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "head_dim must be > 0");
    if (!lvs::score_shape_supported(head_dim, qk_dtype == LITEVLM_FP8_E4M3))
        return fail(nullptr, LITEVLM_ERR_UNSUPPORTED, "head_dim has no kernel for this dtype (bf16: 64, 128; e4m3: 128)");
    if (batch < 0) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "batch must be >= 0");
    if (batch == 0) return LITEVLM_OK;
    if (!seq_offsets_h || !text_offsets_h) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "an offsets host mirror is NULL");
    if (!err_d) return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "err_d is NULL");
    const int64_t tot_n = seq_offsets_h[batch];
    if (seq_offsets_h[0] != 0 || tot_n < 0)
        return fail(nullptr, LITEVLM_ERR_INVALID_ARG, "seq_offsets must start at 0 and be non-decreasing");
    // fold tickets of one launch: floor(n0 / 128) + t + b < total / 128 + 2 * batch + 1
    const int64_t n_tickets = tot_n / lvs::kTileRows + 2 * (int64_t)batch + 2;
    if (n_tickets > kNoAllocTickets)
        return fail(nullptr, LITEVLM_ERR_WORKSPACE,
                    "batch too large for the static scratch: total_visual / 128 + 2 * batch + 2 must be <= 16384");

    // ---- the device's static scratch
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(nullptr, LITEVLM_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
    if (dev < 0 || dev >= kNoAllocMaxDevices) return fail(nullptr, LITEVLM_ERR_UNSUPPORTED, "device ordinal >= 64");
    const int fam = noalloc_family(head_dim, qk_dtype);
    litevlm_select h;
    {
        std::lock_guard<std::mutex> lock(g_noalloc_mutex);
        NoAllocDevice& d = g_noalloc[dev];
        const litevlm_status_t s = noalloc_setup(dev, d);
        if (s != LITEVLM_OK) return s;
        h.device = dev;
        h.num_sms = d.num_sms;
        h.partials = d.partials;
        h.counters = d.tickets;
        h.n_counters = (size_t)kNoAllocTickets;
        h.encode = d.encode;
        for (int r = 0; r < 2; ++r)
            for (int c = 0; c < 17; ++c) {
                h.res_capacity[r][c] = d.res_capacity[fam][r][c];
                h.tc_capacity[r][c] = d.tc_capacity[fam][r][c];
            }
        for (int k = 0; k < 4; ++k) h.plan_memo[k] = d.plan_memo[fam][k];
        h.plan_memo_next = d.plan_memo_next[fam];
    }
    h.err_d = err_d;
    h.allow_flat = false;  // its partial rows could exceed the static scratch
    h.cfg.max_batch = batch;
    h.cfg.max_total_visual = tot_n;
    h.cfg.max_total_text = text_offsets_h[batch] > 0 ? text_offsets_h[batch] : 0;
    h.cfg.num_q_heads = num_q_heads;
    h.cfg.num_kv_heads = num_kv_heads;
    h.cfg.head_dim = head_dim;
    h.cfg.qk_dtype = qk_dtype;
    h.cfg.flags = 0;

    // ---- the plan litevlm_select_score will take, checked against the partials' size
    int32_t plan[4];
    litevlm_status_t s = litevlm_select_score_plan(&h, batch, text_offsets_h, seq_offsets_h, plan);
    if (s == LITEVLM_OK && plan[3] > 1 && (int64_t)plan[3] * tot_n > kNoAllocPartialFloats)
        s = fail(&h, LITEVLM_ERR_WORKSPACE,
                 "head groups x total_visual exceeds the static partial-score scratch (1048576 floats)");
    // the tickets start at zero (a launch that gave up may have left some
    // taken): score_impl clears them after all of its host-side checks, right
    // before the launch, so a rejected call enqueues nothing
    if (s == LITEVLM_OK)
        s = score_impl(&h, batch, q_text, text_offsets_d, text_offsets_h, k_vis, seq_offsets_d, seq_offsets_h,
                       q_scale, k_scale, scores, nullptr, stream, false, nullptr, (size_t)n_tickets);
    {
        std::lock_guard<std::mutex> lock(g_noalloc_mutex);
        NoAllocDevice& d = g_noalloc[dev];
        for (int r = 0; r < 2; ++r)
            for (int c = 0; c < 17; ++c) {
                d.res_capacity[fam][r][c] = h.res_capacity[r][c];
                d.tc_capacity[fam][r][c] = h.tc_capacity[r][c];
            }
        for (int k = 0; k < 4; ++k) d.plan_memo[fam][k] = h.plan_memo[k];
        d.plan_memo_next[fam] = h.plan_memo_next;
    }
    if (s != LITEVLM_OK) g_create_error = h.last_error;
    return s;
}
