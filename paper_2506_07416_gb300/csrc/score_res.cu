// Visual-token importance scores, TMEM-resident variant (sm_103a tcgen05).
//
// Same result as score_tc.cu (Design section, Token Selection Module:
// score[j] = 1/(Hq*T) * sum_h sum_i softmax_j(q_i . k_j / sqrt(d))), for the
// common case where one head's logits for all of a CTA's tiles fit in tensor
// memory (T rounded up to 16, times the CTA's tiles, at most 512 columns).
//
// One tensor-core contraction per K tile and head:
//     S^T = K_tile * Q_h^T   (M = 128 visual rows, N = T rounded up to 16, K = d)
// into a TMEM slot that stays resident for the whole head. Visual tokens are
// TMEM lanes, text tokens are columns. The epilogue reads each slot three times:
//   A  the column (text-row) maximum over the CTA's visual tokens: per thread
//      over its slots, then one warp-wide max per column (redux.sync) and a
//      max over the four lane-quadrant warps;
//   B  e = 2^(s*c - m*c) (m: the CTA's column max) is written back over the
//      logits; per-thread sums of e per column are reduced across lanes once
//      per head by a 5-step shuffle transpose (lane l ends with column l);
//   -  the per-column (m, l) go to every CTA of the cluster with st.async,
//      which writes the pair and completes bytes on the receiver's mbarrier;
//      each CTA merges the cluster's pairs in rank order (deterministic) into
//      b_i = M_i * c + log2(L_i), c = scale * log2(e), and the column weight
//      w_i = 2^(m_i * c - b_i);
//   C  each visual token adds sum_i e_ij * w_i (= sum_i 2^(s_ij * c - b_i)) to
//      its running score, and the slot goes back to the MMA warp.
// While the statistics travel, the producer keeps the next head's K tiles
// streaming into the ring. The four epilogue warpgroups split each slot's text
// columns (a quarter each, read 16 columns at a time; no cross-warpgroup merge
// of statistics), so every SM sub-partition runs four epilogue warps that hide
// one another's TMEM-load and exponential latencies; each warpgroup keeps its
// own partial score rows, added in a fixed order at the end. With several head
// groups the CTAs write partial rows and a per-tile ticket lets the last writer
// of each tile add them (fixed group order). Rows past a request's end (only in
// a CTA's last tile) get -inf logits in pass A, so B and C need no row mask.
//
// Schedules: one cluster per (request, head group), or for batches whose
// requests all have the same token counts the batch's (request, head) pairs
// split evenly over every cluster that fits at once (flat_n > 0). With the
// query split (template parameter QS) each head's text rows run as two
// pseudo-heads of at most 64 rows.
//
// Warp roles (608 threads): warp 0 = TMA producer, warp 1 = TMEM allocator
// and MMA issuer of the even tiles, warp 2 = MMA issuer of the odd tiles,
// warps 3..18 = epilogue warpgroups 0..3 (TMEM lane quadrant = warp % 4).
// Waits are bounded (clock budget) as in score_tc.cu.

#include <math.h>

#include "internal.h"
#include "pipe.cuh"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kResWG = 4;                       // epilogue warpgroups
constexpr int kResThreads = 96 + 128 * kResWG;  // producer warp, two MMA warps, epilogue
constexpr int kResChunk = 16;                   // text columns per epilogue TMEM load
constexpr int kResTmemCols = 512;
constexpr int kResMaxSlots = 16;
constexpr int kBufSlots = kResMaxSlots / 2;  // slots per buffer with two TMEM buffers
constexpr int kBufCols = kResTmemCols / 2;   // columns per buffer with two TMEM buffers
constexpr int kStatSlots = 4;                // heads whose statistics may be in flight
// Compact layout (256-byte rows, up to 64 text rows): score rows for at most 8
// tiles per CTA and a 320-column statistics buffer leave room for a fifth K
// stage. A launch whose tiles per CTA and cluster x slot columns fit takes it.
constexpr int kResCompactTiles = 8;
constexpr int kResCompactRecv = 320;

template <int ROW_BYTES, int MROWS, bool COMPACT>
struct ResLayout {
    static constexpr int KB = ROW_BYTES / 128;
    static constexpr int TILE_BYTES = kTileRows * ROW_BYTES;
    static constexpr int Q_BYTES = MROWS * ROW_BYTES;
    static constexpr int WGC = MROWS / kResWG;  // most text columns one warpgroup owns (16 or 32)
    // statistics receive buffer: [kStatSlots heads][cluster rank][column] (m, l);
    // cluster size times slot columns must fit RECV_COLS
    static constexpr int RECV_COLS = COMPACT ? kResCompactRecv : ROW_BYTES == 256 ? 640 : 1024;
    static constexpr int ACC_TILES = COMPACT ? kResCompactTiles : kResMaxSlots;  // score rows kept per warpgroup
    static constexpr int ACC_BYTES = kResWG * ACC_TILES * kTileRows * 4;
    // [max of head s & 1 (2) | sum][wg][quadrant warp][WGC columns]
    static constexpr int SCR_BYTES = 3 * kResWG * 4 * WGC * 4;
    static constexpr int NBAR_FIXED = 2 * 2 + 2 * kResMaxSlots + kStatSlots + 2;
    static constexpr int FIXED = 2 * Q_BYTES + ACC_BYTES + SCR_BYTES + kStatSlots * RECV_COLS * 8 +
                                 2 * kResWG * WGC * 4 + kResMaxSlots * 4 + (NBAR_FIXED + 2 * 10) * 8 + 64 + 1024;
    static constexpr int STAGES_FIT = (227 * 1024 - FIXED) / TILE_BYTES;
    static constexpr int kStages = STAGES_FIT > 10 ? 10 : STAGES_FIT;
    static constexpr int OFF_K = 0;
    static constexpr int OFF_Q = OFF_K + kStages * TILE_BYTES;
    static constexpr int OFF_ACC = OFF_Q + 2 * Q_BYTES;
    static constexpr int OFF_SCR = OFF_ACC + ACC_BYTES;
    static constexpr int OFF_RECV = OFF_SCR + SCR_BYTES;
    static constexpr int OFF_B2 = OFF_RECV + kStatSlots * RECV_COLS * 8;
    static constexpr int OFF_MC = OFF_B2 + kResWG * WGC * 4;     // column weights per warpgroup column
    static constexpr int OFF_FLAGS = OFF_MC + kResWG * WGC * 4;  // -(CTA column max * c) per warpgroup column
    static constexpr int OFF_BAR = OFF_FLAGS + kResMaxSlots * 4;
    static constexpr int NBAR = 2 * kStages + NBAR_FIXED;
    static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
    static constexpr int BYTES = OFF_MISC + 16;
    static constexpr int ALLOC = BYTES + 1024;
};

// Columns one epilogue warpgroup owns for n2 slot columns (n2 % 16 == 0), and
// the widest TMEM column a slot's epilogue reads relative to the slot start
// (the last warpgroup's last 16-column chunk may reach past the slot; the
// extra columns are read, never used or written).
__host__ __device__ __forceinline__ int res_wg_cols(int n2) { return n2 / kResWG; }
__host__ __device__ __forceinline__ int res_read_span(int n2)
{
    const int cpw = res_wg_cols(n2);
    return (kResWG - 1) * cpw + kResChunk * ((cpw + kResChunk - 1) / kResChunk);
}

// x[c] (c < 16, one value per lane per column) -> sum over the warp's 32 lanes
// of column (lane & 15), returned in every lane: four halving exchanges leave
// lane l with column l & 15 summed over the 16 lanes that share bit 4 of l,
// and one more exchange adds the two halves.
__device__ __forceinline__ float transpose_sum16(float (&x)[16], int lane)
{
#pragma unroll
    for (int step = 0; step < 4; ++step) {
        const int o = 8 >> step;
        const bool up = (lane & o) != 0;
#pragma unroll
        for (int k = 0; k < o; ++k) {
            const float send = up ? x[k] : x[k + o];
            const float keep = up ? x[k + o] : x[k];
            x[k] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
    }
    return x[0] + __shfl_xor_sync(0xffffffffu, x[0], 16);
}

// What a CTA serves of its request: the text rows, the tile range, and whether
// the shape fits the kernel's buffers (uniform over the cluster).
struct ResShape {
    int N, t0, T, Th, n2, n_tiles, tile_begin, mt, nb;
    bool bad;
};

template <int RECV_COLS, int ACC_TILES, bool QS>
__device__ __forceinline__ ResShape res_shape(const ScoreLaunch& p, int n0, int n1, int tq, int t1, uint32_t rank,
                                              uint32_t csize, int mrows)
{
    ResShape r;
    r.N = n1 - n0;
    r.t0 = p.query_last && t1 > tq ? t1 - 1 : tq;  // last-token queries: one row
    r.T = t1 - r.t0;
    r.Th = QS ? (r.T + 1) >> 1 : r.T;  // rows of the first (largest) pseudo-head
    r.n2 = (r.Th + 15) & ~15;
    r.n_tiles = (r.N + kTileRows - 1) / kTileRows;
    const int tpc = r.N > 0 ? (r.n_tiles + (int)csize - 1) / (int)csize : 0;
    // Shape errors are caught on the host; this only keeps the kernel within its buffers.
    const int span = res_read_span(p.slot_cols);  // columns the epilogue reads per slot
    r.nb = p.res_nb == 2 ? 2 : 1;
    const int buf_cols = r.nb == 2 ? kBufCols : kResTmemCols;
    r.bad = r.Th > mrows || r.n2 > p.slot_cols || (r.N > 0 && r.T <= 0) || (QS && (p.query_last || p.qsplit != 2)) ||
            (tpc > 0 && (tpc - 1) * p.slot_cols + span > buf_cols) ||
            tpc > (r.nb == 2 ? kBufSlots : kResMaxSlots) || tpc > ACC_TILES || (int)csize * p.slot_cols > RECV_COLS;
    r.tile_begin = min(r.n_tiles, (int)rank * tpc);
    r.mt = min(r.n_tiles, r.tile_begin + tpc) - r.tile_begin;
    return r;
}

// QS: the query split (each head's text rows as two pseudo-heads), a template
// parameter so that the kernels without it carry none of its bookkeeping.
template <int ROW_BYTES, bool FP8, int MROWS, bool COMPACT, bool QS>
__global__ void __launch_bounds__(kResThreads, 1)
    score_res_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                     const __grid_constant__ ScoreLaunch p)
{
    using L = ResLayout<ROW_BYTES, MROWS, COMPACT>;
    constexpr int KSTEPS = ROW_BYTES / 32;
    constexpr int ELEMS_PER_KB = FP8 ? 128 : 64;
    constexpr uint32_t FMT = FP8 ? 0u : 1u;
    constexpr int kStages = L::kStages;
    static_assert(kStages >= 3, "ring depth");
    static_assert(L::ALLOC > 116 * 1024, "one CTA per SM");
    static_assert(L::ALLOC <= 227 * 1024, "shared memory per CTA");
    static_assert(!COMPACT || kStages == 5, "the compact layout exists for its fifth K stage");

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (base - raw);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const uint32_t csize = cluster_nctarank();
    // This cluster's work: one (request, head group), or with a flattened
    // schedule the pairs [fr0, fr0 + nheads) of the request-major list of
    // (request, head) pairs, which may cross request boundaries (all requests
    // then have the same token counts); b is the first request.
    const int item = (int)(blockIdx.x / csize);
    const bool flat = p.flat_n > 0;
    const int fr0 = flat ? p.flat_r[item] : 0;
    const int nheads = flat ? p.flat_r[item + 1] - fr0 : p.heads_per_group;
    const int req_i = flat ? 0 : item / p.groups;
    // heads of a request as scheduled (pseudo-heads with the query split); read
    // from the parameters where it is used rather than held in a register
#define LVS_HQE (QS ? 2 * p.hq : p.hq)
    const int b = flat ? fr0 / LVS_HQE : (p.order_n > 0 ? (int)p.order[req_i] : req_i);
    const int hg = flat ? 0 : item - req_i * p.groups;

    // With the full-key-set terms (p.extra, written by the kernel launched just
    // before this one) only the threads that read them wait for that kernel,
    // right before the read: this kernel's other inputs come from kernels that
    // had completed before that one passed its own wait, so the visual-key work
    // overlaps it. Every CTA still waits before it exits, so this grid never
    // completes ahead of that one.
    if (!p.extra) griddep_wait();
    griddep_launch_dependents();
    // The request's offsets: by value for small batches; otherwise loaded here
    // and first used after the setup below (barriers, TMEM, cluster barrier),
    // so their latency overlaps it.
    const bool byv = p.nv > 0;
    const int n0 = byv ? p.so_v[b] : p.seq_off[b];
    const int n1 = byv ? p.so_v[b + 1] : p.seq_off[b + 1];
    const int tq = byv ? p.to_v[b] : p.text_off[b];
    const int t1 = byv ? p.to_v[b + 1] : p.text_off[b + 1];
    const bool multi = p.groups > 1;
    const int G = p.hq / p.hkv;
    const int hpg = p.heads_per_group;
    const float cl = p.c_log2;
    const int scols = p.slot_cols;

    const uint32_t bar0 = base + L::OFF_BAR;
    auto BAR = [&](int i) -> uint32_t { return bar0 + 8u * (uint32_t)i; };
    const int K_FULL = 0, K_EMPTY = kStages, Q_FULL = 2 * kStages, Q_EMPTY = Q_FULL + 2, S_FULL = Q_EMPTY + 2,
              S_EMPTY = S_FULL + kResMaxSlots, STATS = S_EMPTY + kResMaxSlots, DRAIN = STATS + kStatSlots,
              STALL = DRAIN + 1;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);
    float* acc_s = reinterpret_cast<float*>(smem + L::OFF_ACC);
    constexpr int WGC = L::WGC;
    float* scr_max = reinterpret_cast<float*>(smem + L::OFF_SCR);        // [head & 1][wg][warp][WGC]
    float* scr_sum = scr_max + 2 * kResWG * 4 * WGC;                      // [wg][warp][WGC]
    const float2* recv = reinterpret_cast<const float2*>(smem + L::OFF_RECV);
    float* b2_s = reinterpret_cast<float*>(smem + L::OFF_B2);
    float* mc_s = reinterpret_cast<float*>(smem + L::OFF_MC);
    volatile int* fold_flags = reinterpret_cast<volatile int*>(smem + L::OFF_FLAGS);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(BAR(K_FULL + s), 1);
            mbar_init(BAR(K_EMPTY + s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(BAR(Q_FULL + i), 1);
            mbar_init(BAR(Q_EMPTY + i), 2);  // one commit per MMA-issuing thread
        }
        for (int i = 0; i < kStatSlots; ++i) mbar_init(BAR(STATS + i), 1);  // the local arm; peers complete bytes
        for (int i = 0; i < kResMaxSlots; ++i) {
            mbar_init(BAR(S_FULL + i), 1);
            mbar_init(BAR(S_EMPTY + i), 4 * kResWG);  // one arrival per epilogue warp
        }
        mbar_init(BAR(DRAIN), 2);
        mbar_init(BAR(STALL), 1);  // nothing ever arrives (the debug stall below)
        *abort_flag = 0;
        fence_mbar_init_cluster();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_k);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kResTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // Cluster barrier, split: every thread arrives now (after its CTA's barriers
    // exist) and waits only before its first access to a peer's shared memory
    // (the epilogue, below) or before the final barrier (producer, MMA warp),
    // so the first copies and contractions do not wait for the slowest CTA of
    // the cluster to get here. The arrival needs no release: the barriers' set-up
    // is released by fence.mbarrier_init above, and no other write of this CTA
    // is read by a peer.
    cluster_arrive_relaxed();
    const uint32_t tmem = *tmem_slot;
    const Ctl ctl{abort_flag, p.err, p.wait_budget};

    const ResShape shp = res_shape<L::RECV_COLS, L::ACC_TILES, QS>(p, n0, n1, tq, t1, rank, csize, MROWS);
    const int N = shp.N, t0 = shp.t0, T = shp.T, Th = shp.Th, n2 = shp.n2, nb = shp.nb;
    const bool bad_shape = shp.bad || (flat && nb != 1);  // uniform for the whole cluster
    if (bad_shape || N <= 0) {
        if (p.extra) griddep_wait();
        if (bad_shape && threadIdx.x == 0 && rank == 0 && hg == 0) atomicOr(p.err, kErrShape);
        tc_fence_before();
        __syncthreads();
        if (warp == 1) {
            tc_fence_after();
            tmem_dealloc(tmem, kResTmemCols);
        }
        cluster_wait();
        cluster_sync_relaxed();
        return;
    }
    const int tile_begin = shp.tile_begin;
    const int tile_end = tile_begin + shp.mt;
    const int mt = shp.mt;
    // request, scheduled head (pseudo-head with the query split), query head,
    // first visual row, first query row and query rows of head s of this CTA's
    // sequence (with a flattened schedule the requests' rows follow one another
    // at equal strides). With the query split, pseudo-head 2h + u of a request
    // holds the query rows [u * Th, min((u + 1) * Th, T)) of head h.
    struct HeadRef {
        int b, ph, h, n0, t0, T;
    };
    const int t_stride = t1 - tq;
    auto head_of = [&](int s_) -> HeadRef {
        if constexpr (!QS) {
            if (!flat) return HeadRef{b, hg * hpg + s_, hg * hpg + s_, n0, t0, T};
            const int rh = fr0 + s_, bb = rh / p.hq;
            return HeadRef{bb, rh - bb * p.hq, rh - bb * p.hq, n0 + (bb - b) * N, t0 + (bb - b) * t_stride, T};
        } else {
            int bb = b, ph = hg * hpg + s_, nn0 = n0, tt0 = t0;
            if (flat) {
                const int rh = fr0 + s_;
                bb = rh / LVS_HQE;
                ph = rh - bb * LVS_HQE;
                nn0 = n0 + (bb - b) * N;
                tt0 = t0 + (bb - b) * t_stride;
            }
            const int u = ph & 1;
            return HeadRef{bb, ph, ph >> 1, nn0, tt0 + u * Th, u ? T - Th : Th};
        }
    };

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0 && mt > 0) {
            // Debug stall (p.stall, a test of the failure path): wait on a barrier
            // that nothing completes before issuing any copy, so this wait runs out
            // of budget, and every other wait of the launch runs out or sees the
            // abort flag, with no copy or contraction in flight.
            // Nothing is issued after the stall ran out.
            bool ok = !p.stall || wait_phase(BAR(STALL), 0, ctl);
            uint32_t ks = 0, kph = 0;
            int k_issued[kStages];
            int q_issued[2] = {0, 0};
            for (int s = 0; s < kStages; ++s) k_issued[s] = 0;
            for (int s = 0; s < nheads && ok; ++s) {
                const HeadRef hr = head_of(s);
                const int h = hr.h;
                const int g = h / G;
                const int qb = s & 1;
                if (!wait_phase(BAR(Q_EMPTY + qb), ((s >> 1) & 1) ^ 1, ctl)) break;
                mbar_arrive_expect_tx(BAR(Q_FULL + qb), L::Q_BYTES);
                const uint32_t qdst = base + L::OFF_Q + qb * L::Q_BYTES;
#pragma unroll
                for (int kb = 0; kb < L::KB; ++kb)
                    tma_load_3d(qdst + kb * MROWS * 128, &tm_q, BAR(Q_FULL + qb), kb * ELEMS_PER_KB, h, hr.t0);
                ++q_issued[qb];
                for (int t = tile_begin; t < tile_end; ++t) {
                    if (!wait_phase(BAR(K_EMPTY + ks), kph ^ 1, ctl)) { ok = false; break; }
                    mbar_arrive_expect_tx(BAR(K_FULL + ks), L::TILE_BYTES);
                    const uint32_t kdst = base + L::OFF_K + ks * L::TILE_BYTES;
#pragma unroll
                    for (int kb = 0; kb < L::KB; ++kb)
                        tma_load_3d(kdst + kb * kTileRows * 128, &tm_k, BAR(K_FULL + ks), kb * ELEMS_PER_KB, g,
                                    hr.n0 + t * kTileRows);
                    ++k_issued[ks];
                    if (++ks == kStages) { ks = 0; kph ^= 1; }
                }
            }
            volatile int no_abort = 0;
            const Ctl drain_ctl{&no_abort, p.err, kWaitBudgetCycles};
            for (int s = 0; s < kStages; ++s)
                if (k_issued[s] > 0) wait_phase(BAR(K_FULL + s), (uint32_t)(k_issued[s] - 1) & 1u, drain_ctl);
            for (int s = 0; s < 2; ++s)
                if (q_issued[s] > 0) wait_phase(BAR(Q_FULL + s), (uint32_t)(q_issued[s] - 1) & 1u, drain_ctl);
        }
        __syncwarp();
        cluster_wait();
    } else if (warp <= 2) {
        // ------------------------------------------------------------ MMA issuers
        // Two issuing threads (lane 0 of warps 1 and 2) take alternate tiles:
        // issuing a tile (two barrier waits, the contractions, two commits)
        // costs more time than the tensor core needs to run it, so one thread's
        // waits and commits overlap the other thread's contractions. Each
        // thread follows the global tile sequence for the ring's stage and
        // phase and commits its own contractions. The operand descriptors are
        // made once (per head for Q, per tile for K) and each K step adds a
        // constant to the start-address field (shared-memory offsets stay below
        // 256 KB, so the 14-bit field never carries).
        if (lane == 0) {
            const int who = warp - 1;  // 0: even tiles, 1: odd tiles
            if (mt > 0) {
                const uint32_t idesc = idesc_make(128, (uint32_t)n2, FMT);
                // A stage's consecutive loads can belong to different threads
                // (tiles gt and gt - kStages of opposite parity within their
                // heads). The K_FULL parity test is only sound once the stage's
                // previous load has landed, which a thread knows of its own tiles
                // but not of the other thread's: for those tiles it first waits
                // for the release of the previous load (its contraction done, so
                // its data had landed). `cross` marks them by tile.
                uint32_t cross = 0;
                for (int tl = who; tl < mt; tl += 2) {
                    const int ptl = ((tl - kStages) % mt + mt) % mt;
                    if ((ptl ^ tl) & 1) cross |= 1u << tl;
                }
                bool ok = true;
                for (int s = 0; s < nheads && ok; ++s) {
                    const int qb = s & 1;
                    const int buf = nb == 2 ? (s & 1) : 0;
                    const uint32_t use = nb == 2 ? (uint32_t)(s >> 1) : (uint32_t)s;  // earlier heads in this buffer
                    if (!wait_phase(BAR(Q_FULL + qb), (s >> 1) & 1, ctl)) break;
                    tc_fence_after();
                    const uint64_t qdesc = sdesc_k_sw128(base + L::OFF_Q + qb * L::Q_BYTES);
                    for (int tl = who; tl < mt; tl += 2) {
                        const int sl = buf * kBufSlots + tl;
                        const int gt = s * mt + tl;  // the ring runs over the tiles of all heads in order
                        const uint32_t ks = (uint32_t)(gt % kStages), kph = (uint32_t)(gt / kStages) & 1u;
                        if (((cross >> tl) & 1u) && gt >= kStages && !wait_phase(BAR(K_EMPTY + ks), kph ^ 1u, ctl)) {
                            ok = false;
                            break;
                        }
                        if (!wait_phase(BAR(K_FULL + ks), kph, ctl)) { ok = false; break; }
                        if (!wait_phase(BAR(S_EMPTY + sl), (use & 1u) ^ 1u, ctl)) { ok = false; break; }
                        tc_fence_after();
                        const uint64_t kdesc = sdesc_k_sw128(base + L::OFF_K + ks * L::TILE_BYTES);
                        const uint32_t d = tmem + (uint32_t)(buf * kBufCols + tl * scols);
#pragma unroll
                        for (int st = 0; st < KSTEPS; ++st) {
                            constexpr uint64_t kQ16 = MROWS * 128 / 16, kK16 = kTileRows * 128 / 16;
                            const uint64_t qoff = (uint64_t)(st >> 2) * kQ16 + (uint64_t)(st & 3) * 2;
                            const uint64_t koff = (uint64_t)(st >> 2) * kK16 + (uint64_t)(st & 3) * 2;
                            if (FP8) mma_f8(d, kdesc + koff, qdesc + qoff, idesc, st > 0);
                            else mma_f16(d, kdesc + koff, qdesc + qoff, idesc, st > 0);
                        }
                        mma_commit(BAR(S_FULL + sl));
                        mma_commit(BAR(K_EMPTY + ks));
                    }
                    // Q(s) is free once both threads' contractions of head s are done
                    // (one arrival each; a thread without tiles in this head arrives at once)
                    if (ok) mma_commit(BAR(Q_EMPTY + qb));
                }
            }
            mma_commit(BAR(DRAIN));
            volatile int no_abort = 0;
            const Ctl drain_ctl{&no_abort, p.err, kWaitBudgetCycles};
            wait_phase(BAR(DRAIN), 0, drain_ctl);
        }
        __syncwarp();
        cluster_wait();
    } else {
        // ------------------------------------------------------------ epilogue (kResWG warpgroups)
        cluster_wait();  // the peers' barriers and buffers exist before any statistics go out
        // Control flow is identical for every thread of a warpgroup (named
        // barriers); after an abort every wait returns at once. Warp-synchronous
        // instructions (tcgen05.ld, redux.sync, shuffles) run under branches
        // that are uniform in the CTA only: always 16 columns per chunk, columns
        // past the warpgroup's range masked arithmetically.
        // Iteration i runs A and B of head i and sends its statistics, then C of
        // head i - 1 with two TMEM buffers (the statistics of head i - 1 had a
        // whole A + B to travel, and the MMAs of head i + 1 fill the other buffer
        // while C reads it, slot by slot), or C of head i with one buffer.
        const int wg = (warp - 3) >> 2;
        const int quad = warp & 3;
        const int et = threadIdx.x - 96;               // 0 .. 128 * kResWG - 1
        const int wt = et - 128 * wg;                  // 0..127 within the warpgroup
        const int vrow = quad * 32 + lane;             // visual token of this lane within a tile
        const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
        const uint32_t wg_bar = 2u + (uint32_t)wg;
        const int cpw = res_wg_cols(n2);               // this warpgroup's columns: [c_begin, c_begin + cpw)
        const int c_begin = wg * cpw;
        const int nch = (cpw + kResChunk - 1) / kResChunk;
        float* accw = acc_s + wg * L::ACC_TILES * kTileRows;
        float* ssum = scr_sum + wg * 4 * WGC;
        float* b2w = b2_s + wg * WGC;                  // weight of column c_begin + c, 0 for c >= cpw or >= T
        float* mcw = mc_s + wg * WGC;                  // -(CTA column max * c) of column c_begin + c
        const uint32_t recv_base = base + L::OFF_RECV;
        const uint32_t tcol = tmem + lane_off;
        for (int tl = 0; tl < mt; ++tl) accw[tl * kTileRows + vrow] = 0.f;
        auto lane_valid = [&](int tl) { return tl < mt && (tile_begin + tl) * kTileRows + vrow < N; };
        const bool tail_tile = mt > 0 && (tile_begin + mt) * kTileRows > N;  // the request's last, partial tile
        // slot tl of buffer b is read by this warp: hand it back to the MMA warp
        // (one arrival per warp and slot)
        auto release = [&](int b_, int tl_) {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(BAR(S_EMPTY + b_ * kBufSlots + tl_));
        };

        // A (and the column maxima) of head s
        auto front_a = [&](const int s) {
            const int buf = nb == 2 ? (s & 1) : 0;
            const uint32_t use = nb == 2 ? (uint32_t)(s >> 1) : (uint32_t)s;
            const int slot = s & (kStatSlots - 1);
            const uint32_t tbuf = tcol + (uint32_t)(buf * kBufCols);
            float* smax = scr_max + ((s & 1) * kResWG + wg) * 4 * WGC;
            // (not after an abort: that phase would never complete, and arming it
            // again four heads later would arrive twice on it)
            if (et == 0 && !*abort_flag) mbar_arrive_expect_tx(BAR(STATS + slot), (uint32_t)(csize * n2 * 8));
            for (int ch = 0; ch < nch; ++ch) {
                const int cw = min(kResChunk, cpw - kResChunk * ch);  // 4, 8, 12 or 16
                const uint32_t col0 = (uint32_t)(c_begin + kResChunk * ch);
                // ---- A: column maxima, per thread over its slots, then over the lanes.
                // A request's last tile may hold rows past its end: their logits
                // become -inf in tensor memory (this warpgroup's columns), so that B
                // needs no per-value select (2^-inf = 0) and C adds nothing for them.
                float cm[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) cm[c] = -INFINITY;
                {
                    float va[16], vb[16];
                    if (ch == 0 && mt > 0) {  // a rank without tiles gets no MMA
                        wait_phase(BAR(S_FULL + buf * kBufSlots), use & 1u, ctl);
                        tc_fence_after();
                    }
                    tmem_ld16(tbuf + col0, va);
                    for (int tl = 0; tl < mt; tl += 2) {
                        const int t1 = min(tl + 1, mt - 1), t2 = min(tl + 2, mt - 1);
                        tmem_wait_ld();
                        if (ch == 0 && tl + 1 < mt) {
                            wait_phase(BAR(S_FULL + buf * kBufSlots + t1), use & 1u, ctl);
                            tc_fence_after();
                        }
                        tmem_ld16(tbuf + (uint32_t)(t1 * scols) + col0, vb);
                        if (lane_valid(tl)) {
#pragma unroll
                            for (int c = 0; c < 16; c += 2) {
                                cm[c] = fmaxf(cm[c], va[c]);
                                cm[c + 1] = fmaxf(cm[c + 1], va[c + 1]);
                            }
                        }
                        tmem_wait_ld();
                        if (ch == 0 && tl + 2 < mt) {
                            wait_phase(BAR(S_FULL + buf * kBufSlots + t2), use & 1u, ctl);
                            tc_fence_after();
                        }
                        tmem_ld16(tbuf + (uint32_t)(t2 * scols) + col0, va);
                        if (lane_valid(tl + 1)) {
#pragma unroll
                            for (int c = 0; c < 16; ++c) cm[c] = fmaxf(cm[c], vb[c]);
                        }
                    }
                    tmem_wait_ld();
                    // only the CTA's last tile can run past the request's end
                    if (tail_tile && !__all_sync(0xffffffffu, lane_valid(mt - 1))) {
                        const uint32_t ta = tbuf + (uint32_t)((mt - 1) * scols) + col0;
                        tmem_ld16(ta, va);
                        tmem_wait_ld();
                        const bool okv = lane_valid(mt - 1);
#pragma unroll
                        for (int c = 0; c < 16; ++c) va[c] = okv ? va[c] : -INFINITY;
                        tmem_st_cols16(ta, va, cw);
                        tmem_wait_st();  // B reads these rows
                    }
                }
#pragma unroll
                for (int c = 0; c < 16; ++c) cm[c] = warp_max_f32(cm[c]);
                if (lane == 0) {
#pragma unroll
                    for (int c = 0; c < 16; c += 4)
                        *reinterpret_cast<float4*>(smax + quad * WGC + kResChunk * ch + c) =
                            make_float4(cm[c], cm[c + 1], cm[c + 2], cm[c + 3]);
                }
                named_bar_sync(wg_bar, 128);
                // CTA-local column max * c, once per column, read back by B from shared
                // memory (keeps registers free in B)
                if (wt < kResChunk) {
                    float m = smax[kResChunk * ch + wt];
#pragma unroll
                    for (int q = 1; q < 4; ++q) m = fmaxf(m, smax[q * WGC + kResChunk * ch + wt]);
                    mcw[kResChunk * ch + wt] = -(m * cl);  // columns past cpw: garbage, never used
                }
                named_bar_sync(wg_bar, 128);
            }
        };
        // B of head s: e written back, column sums, statistics sent to the cluster
        auto front_b = [&](const int s) {
            const int buf = nb == 2 ? (s & 1) : 0;
            const int slot = s & (kStatSlots - 1);
            const uint32_t tbuf = tcol + (uint32_t)(buf * kBufCols);
            float* smax = scr_max + ((s & 1) * kResWG + wg) * 4 * WGC;
            for (int ch = 0; ch < nch; ++ch) {
                const int cw = min(kResChunk, cpw - kResChunk * ch);  // 4, 8, 12 or 16
                const uint32_t col0 = (uint32_t)(c_begin + kResChunk * ch);
                // ---- B: e = 2^(s*c - m*c) written back over the logits (this warpgroup's
                // columns only); per-thread column sums of e, then over the warp's lanes
                float sm[16], mh[16];  // column sums; the shifts -m*c, in registers for all tiles
#pragma unroll
                for (int c = 0; c < 16; ++c) sm[c] = 0.f;
#pragma unroll
                for (int c = 0; c < 16; c += 4) {
                    const float4 m4 = *reinterpret_cast<const float4*>(mcw + kResChunk * ch + c);
                    mh[c] = m4.x;
                    mh[c + 1] = m4.y;
                    mh[c + 2] = m4.z;
                    mh[c + 3] = m4.w;
                }
                for (int tl = 0; tl < mt; ++tl) {
                    float v[16];
                    const uint32_t ta = tbuf + (uint32_t)(tl * scols) + col0;
                    tmem_ld16(ta, v);
                    tmem_wait_ld();
                    const float2 cl2 = make_float2(cl, cl);
                    // rows past the request's end hold -inf (pass A), so their e is 0
#pragma unroll
                    for (int c = 0; c < 16; c += 4) {
                        const float2 x01 = ffma2(make_float2(v[c], v[c + 1]), cl2, make_float2(mh[c], mh[c + 1]));
                        const float2 x23 = ffma2(make_float2(v[c + 2], v[c + 3]), cl2, make_float2(mh[c + 2], mh[c + 3]));
                        const float e0 = ex2(x01.x);
                        const float e1 = ex2(x01.y);
                        const float e2 = ex2(x23.x);
                        const float e3 = ex2(x23.y);
                        v[c] = e0;
                        v[c + 1] = e1;
                        v[c + 2] = e2;
                        v[c + 3] = e3;
                        const float2 s01 = fadd2(make_float2(sm[c], sm[c + 1]), make_float2(e0, e1));
                        const float2 s23 = fadd2(make_float2(sm[c + 2], sm[c + 3]), make_float2(e2, e3));
                        sm[c] = s01.x;
                        sm[c + 1] = s01.y;
                        sm[c + 2] = s23.x;
                        sm[c + 3] = s23.y;
                    }
                    tmem_st_cols16(ta, v, cw);
                }
                const float colsum = transpose_sum16(sm, lane);
                if (lane < cw) ssum[quad * WGC + kResChunk * ch + lane] = colsum;
                named_bar_sync(wg_bar, 128);
                // ---- publish (m, l) of columns col0 .. col0+cw-1 to every CTA of the cluster
                // (not after an abort: the peers may not be waiting for it, and no
                // statistic is left in flight when the CTA exits)
                if (quad == 2 && lane < cw && !*abort_flag) {  // one warp of the warpgroup
                    const int c = kResChunk * ch + lane;
                    float m = smax[c], l = ssum[c];
#pragma unroll
                    for (int q = 1; q < 4; ++q) {
                        m = fmaxf(m, smax[q * WGC + c]);
                        l += ssum[q * WGC + c];
                    }
                    const int col = c_begin + c;
                    const uint32_t dst = recv_base + (uint32_t)(((slot * (int)csize + (int)rank) * scols + col) * 8);
                    const uint32_t bar = BAR(STATS + slot);
                    for (uint32_t r = 0; r < csize; ++r)
                        st_async_f2(mapa_shared(dst, r), m, l, mapa_shared(bar, r));
                }
            }
            tmem_wait_st();
        };
        // statistics merge and C of head s; slots go back to the MMA warp as they are read
        auto back = [&](const int s) {
            const int buf = nb == 2 ? (s & 1) : 0;
            const int slot = s & (kStatSlots - 1);
            const uint32_t tbuf = tcol + (uint32_t)(buf * kBufCols);
            const float* smax = scr_max + ((s & 1) * kResWG + wg) * 4 * WGC;
            // merge the cluster's statistics of this head (rank order) into the
            // column weights w = 2^(m_local*c - b), b = M*c + log2(L); 0 for unused columns
            wait_phase_cluster(BAR(STATS + slot), (uint32_t)(s / kStatSlots) & 1u, ctl);
            // query rows of head s (with the query split, pseudo-heads alternate
            // halves: the parity of the request's pseudo-head index, which is the
            // parity of its index in the schedule since a request has an even count)
            const int Ts = !QS ? T : ((((flat ? fr0 : hg * hpg) + s) & 1) ? T - Th : Th);
            if (wt < WGC) {
                const int col = c_begin + wt;
                float wval = 0.f;
                if (wt < cpw && col < Ts) {
                    const float2* rs = recv + (slot * (int)csize) * scols + col;  // rank r at rs[r * scols]
                    float M = -INFINITY;
                    for (int r = 0; r < (int)csize; ++r) M = fmaxf(M, rs[r * scols].x);
                    float Ls = 0.f;
                    for (int r = 0; r < (int)csize; ++r) {
                        const float2 v2 = rs[r * scols];
                        if (v2.y > 0.f) Ls += v2.y * ex2((v2.x - M) * cl);
                    }
                    float b = fmaf(M, cl, __log2f(Ls));
                    if (p.extra) {
                        griddep_wait();
                        const HeadRef hs = head_of(s);
                        b = log2_add(b, p.extra[(int64_t)(hs.t0 + col) * p.hq + hs.h]);
                    }
                    float mloc = smax[wt];  // this CTA's column max: the e values' reference
#pragma unroll
                    for (int q = 1; q < 4; ++q) mloc = fmaxf(mloc, smax[q * WGC + wt]);
                    wval = mloc == -INFINITY ? 0.f : ex2(fmaf(mloc, cl, -b));
                }
                b2w[wt] = wval;
            }
            named_bar_sync(wg_bar, 128);
            // ---- C: per-visual-token sums of e * w over this warpgroup's columns;
            // each slot goes back to the MMA warp after its last chunk is read
            for (int ch = 0; ch < nch; ++ch) {
                const int cw = min(kResChunk, cpw - kResChunk * ch);
                const uint32_t col0 = (uint32_t)(c_begin + kResChunk * ch);
                const bool last = ch == nch - 1;
                float wv[16];
#pragma unroll
                for (int c = 0; c < 16; c += 4) {
                    const float4 w4 = *reinterpret_cast<const float4*>(b2w + kResChunk * ch + c);
                    wv[c] = w4.x;
                    wv[c + 1] = w4.y;
                    wv[c + 2] = w4.z;
                    wv[c + 3] = w4.w;
                }
                float va[16], vb[16];
                if (mt > 0) tmem_ld16(tbuf + col0, va);
                for (int tl = 0; tl < mt; tl += 2) {
                    tmem_wait_ld();  // va: slot tl
                    if (last) release(buf, tl);
                    if (tl + 1 < mt) tmem_ld16(tbuf + (uint32_t)((tl + 1) * scols) + col0, vb);
                    float2 a01 = make_float2(0.f, 0.f);
#pragma unroll
                    for (int c = 0; c < 16; c += 2)
                        if (c < cw) a01 = ffma2(make_float2(va[c], va[c + 1]), make_float2(wv[c], wv[c + 1]), a01);
                    accw[tl * kTileRows + vrow] += a01.x + a01.y;
                    if (tl + 1 < mt) {
                        tmem_wait_ld();  // vb: slot tl + 1
                        if (last) release(buf, tl + 1);
                        if (tl + 2 < mt) tmem_ld16(tbuf + (uint32_t)((tl + 2) * scols) + col0, va);
                        a01 = make_float2(0.f, 0.f);
#pragma unroll
                        for (int c = 0; c < 16; c += 2)
                            if (c < cw) a01 = ffma2(make_float2(vb[c], vb[c + 1]), make_float2(wv[c], wv[c + 1]), a01);
                        accw[(tl + 1) * kTileRows + vrow] += a01.x + a01.y;
                    }
                }
            }
        };

        // One buffer: A, B, C of each head in turn. Two buffers: iteration i runs
        // A of head i, then C of head i - 1 (its statistics travelled during A),
        // which frees the other buffer so the MMAs of head i + 1 run under B of
        // head i.
        const float denom = (float)p.hq * (float)T;
        // Flattened schedule: the scores of request hr.b, whose last head in this
        // cluster's range has been through C. All of its heads in the range:
        // final scores; otherwise this cluster's partial rows, folded by the last
        // of the request's clusters to finish each tile (fixed part order).
        auto flush = [&](const HeadRef& hr) {
            const int first = hr.b * LVS_HQE, last = first + LVS_HQE - 1;
            const bool whole = first >= fr0 && last < fr0 + nheads;
            auto cluster_of = [&](int pair) {  // the cluster whose range holds the pair
                int lo = 0, hi = p.flat_n - 1;
                while (lo < hi) {
                    const int mid = (lo + hi + 1) >> 1;
                    if (p.flat_r[mid] <= pair) lo = mid;
                    else hi = mid - 1;
                }
                return lo;
            };
            const int cf = whole ? item : cluster_of(first);
            const int parts = whole ? 1 : cluster_of(last) - cf + 1;
            named_bar_sync(1, 128 * kResWG);  // every warpgroup's C contributions are in place
            for (int tl = wg; tl < mt; tl += kResWG) {
                const int j = (tile_begin + tl) * kTileRows + vrow;
                if (j < N) {
                    float a = acc_s[tl * kTileRows + vrow];
#pragma unroll
                    for (int g = 1; g < kResWG; ++g) a += acc_s[g * L::ACC_TILES * kTileRows + tl * kTileRows + vrow];
                    if (whole) p.out[hr.n0 + j] = a / denom;
                    else p.partials[(int64_t)(item - cf) * p.total_vis + hr.n0 + j] = a;
                }
            }
            named_bar_sync(1, 128 * kResWG);  // every row is read before it is cleared
            for (int tl = 0; tl < mt; ++tl) accw[tl * kTileRows + vrow] = 0.f;
            if (!whole) fold_tiles(p, hr.b, hr.n0, N, T, tile_begin, mt, et, 128 * kResWG, 1, fold_flags, parts);
        };
        if (nb == 2) {
            for (int it = 0; it <= nheads; ++it) {
                if (it < nheads) front_a(it);
                if (it >= 1) back(it - 1);
                if (it < nheads) front_b(it);
            }
        } else {
            for (int s = 0; s < nheads; ++s) {
                front_a(s);
                front_b(s);
                back(s);
                if (flat) {
                    const HeadRef hr = head_of(s);
                    if (s == nheads - 1 || hr.ph == LVS_HQE - 1) flush(hr);
                }
            }
        }
        // ---- results: the warpgroups' partial rows, added in a fixed order
        if (!flat) {
            named_bar_sync(1, 128 * kResWG);
            for (int tl = wg; tl < mt; tl += kResWG) {
                const int j = (tile_begin + tl) * kTileRows + vrow;
                if (j < N) {
                    float a = acc_s[tl * kTileRows + vrow];
#pragma unroll
                    for (int g = 1; g < kResWG; ++g) a += acc_s[g * L::ACC_TILES * kTileRows + tl * kTileRows + vrow];
                    if (!multi) p.out[n0 + j] = a / denom;
                    else p.partials[(int64_t)hg * p.total_vis + n0 + j] = a;
                }
            }
            if (multi && !p.defer_fold) fold_tiles(p, b, n0, N, T, tile_begin, mt, et, 128 * kResWG, 1, fold_flags);
        }
        tc_fence_before();
    }

    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kResTmemCols);
    }
    if (p.extra) griddep_wait();  // returns at once for threads that already waited
    // Every CTA stays resident until the cluster is done: the statistics a peer
    // sends land (st.async) in this CTA's shared memory, and every one of them
    // has completed on this CTA's barriers before its epilogue ends; no peer
    // reads this CTA's memory, so the arrival needs no release.
    cluster_sync_relaxed();
#undef LVS_HQE
}

template <int ROW_BYTES, bool FP8, int MROWS, bool COMPACT, bool QS>
cudaError_t res_prepare(int cluster)
{
    auto kern = score_res_kernel<ROW_BYTES, FP8, MROWS, COMPACT, QS>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         ResLayout<ROW_BYTES, MROWS, COMPACT>::ALLOC);
    if (e == cudaSuccess && cluster > 8) e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return e;
}

template <int ROW_BYTES, bool FP8, int MROWS, bool COMPACT = false, bool QS = false>
cudaError_t res_launch(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const ScoreLaunch& p, const ScorePlan& plan,
                       int batch, cudaStream_t stream)
{
    auto kern = score_res_kernel<ROW_BYTES, FP8, MROWS, COMPACT, QS>;
    cudaError_t e = res_prepare<ROW_BYTES, FP8, MROWS, COMPACT, QS>(plan.cluster);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    const int items = plan.flat > 0 ? plan.flat : plan.groups * batch;
    cfg.gridDim = dim3((unsigned)(plan.cluster * items), 1, 1);
    cfg.blockDim = dim3(kResThreads, 1, 1);
    cfg.dynamicSmemBytes = ResLayout<ROW_BYTES, MROWS, COMPACT>::ALLOC;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = plan.cluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1] = pdl_attribute();
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, tm_q, tm_k, p);
}

// Clusters of the given size that fit on the GPU at once. Both layouts take
// more than half of an SM's shared memory (one CTA per SM), so the full
// layout's answer holds for the compact one too.
template <int ROW_BYTES, bool FP8, int MROWS>
int res_capacity(int cluster)
{
    if (res_prepare<ROW_BYTES, FP8, MROWS, false, false>(cluster) != cudaSuccess) return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cluster, 64, 1);
    cfg.blockDim = dim3(kResThreads, 1, 1);
    cfg.dynamicSmemBytes = ResLayout<ROW_BYTES, MROWS, false>::ALLOC;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, score_res_kernel<ROW_BYTES, FP8, MROWS, false, false>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n * cluster;
}

}  // namespace

// Tiles per CTA: the epilogue reads 16 columns per chunk, so the last slot's
// padded read, (r - 1) * slot_cols + res_read_span(slot_cols), must stay within
// the 512 TMEM columns (256 per buffer with two head buffers).
int res_max_tiles(int slot_cols, int nb)
{
    if (slot_cols <= 0) return 0;
    const int span = res_read_span(slot_cols);
    const int cols = nb == 2 ? kBufCols : kResTmemCols;
    int r = nb == 2 ? kBufSlots : kResMaxSlots;
    while (r > 0 && (r - 1) * slot_cols + span > cols) --r;
    return r;
}

int res_max_cluster(int row_bytes, int slot_cols)
{
    if (slot_cols <= 0) return 0;
    const int recv = row_bytes == 256 ? ResLayout<256, 64, false>::RECV_COLS : ResLayout<128, 64, false>::RECV_COLS;
    const int c = recv / slot_cols;
    return c < kMaxCluster ? c : kMaxCluster;
}

int res_cluster_capacity(int row_bytes, bool fp8, int mrows, int cluster)
{
    if (fp8) return mrows == 64 ? res_capacity<128, true, 64>(cluster) : res_capacity<128, true, 128>(cluster);
    if (row_bytes == 256)
        return mrows == 64 ? res_capacity<256, false, 64>(cluster) : res_capacity<256, false, 128>(cluster);
    return mrows == 64 ? res_capacity<128, false, 64>(cluster) : res_capacity<128, false, 128>(cluster);
}

cudaError_t launch_score_resident(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const ScoreLaunch& p,
                                  const ScorePlan& plan, int batch, int row_bytes, bool fp8, int mrows,
                                  cudaStream_t stream)
{
    ScoreLaunch q = p;
    q.res_nb = plan.res_nb;
    q.groups = plan.groups;
    q.qsplit = plan.qsplit;
    q.heads_per_group = p.hq * plan.qsplit / plan.groups;
    q.ctas_per_request = plan.cluster * plan.groups;
    q.flat_n = 0;
    if (plan.flat > 0) {  // equal shares of the batch's (request, head) pairs, in request-major order
        if (plan.flat > kFlatMax || plan.res_nb != 1) return cudaErrorInvalidValue;
        const long long pairs = (long long)batch * p.hq * plan.qsplit;
        q.flat_n = plan.flat;
        for (int k = 0; k <= plan.flat; ++k) q.flat_r[k] = (int32_t)(pairs * k / plan.flat);
        q.order_n = 0;
    }
    const bool compact = plan.tiles_per_cta <= kResCompactTiles && plan.cluster * p.slot_cols <= kResCompactRecv;
    if (plan.qsplit == 2) {  // the 64-row kernels only
        if (mrows != 64) return cudaErrorInvalidValue;
        if (fp8) return res_launch<128, true, 64, false, true>(tm_q, tm_k, q, plan, batch, stream);
        if (row_bytes == 256)
            return compact ? res_launch<256, false, 64, true, true>(tm_q, tm_k, q, plan, batch, stream)
                           : res_launch<256, false, 64, false, true>(tm_q, tm_k, q, plan, batch, stream);
        return res_launch<128, false, 64, false, true>(tm_q, tm_k, q, plan, batch, stream);
    }
    if (fp8)
        return mrows == 64 ? res_launch<128, true, 64>(tm_q, tm_k, q, plan, batch, stream)
                           : res_launch<128, true, 128>(tm_q, tm_k, q, plan, batch, stream);
    if (row_bytes == 256 && mrows == 64) {
        if (compact) return res_launch<256, false, 64, true>(tm_q, tm_k, q, plan, batch, stream);
        return res_launch<256, false, 64>(tm_q, tm_k, q, plan, batch, stream);
    }
    if (row_bytes == 256) return res_launch<256, false, 128>(tm_q, tm_k, q, plan, batch, stream);
    return mrows == 64 ? res_launch<128, false, 64>(tm_q, tm_k, q, plan, batch, stream)
                       : res_launch<128, false, 128>(tm_q, tm_k, q, plan, batch, stream);
}

}  // namespace lvs
