// Visual-token importance scores on the sm_103a tensor cores.
//
// Computes, for every visual token j of request b (Design section, Token
// Selection Module: first-decoder-layer self-attention as importance, FastV
// style; scale 1/sqrt(d), softmax over the request's visual tokens, mean over
// query heads and text tokens):
//     score[j] = 1/(Hq*T) * sum_h sum_i exp(s_hij - m_hi) / l_hi
// without ever writing the logits s to memory.
//
// Work decomposition. One thread-block cluster of C CTAs serves one (request,
// head group); CTA r of the cluster owns a contiguous range of 128-token tiles
// of the request. For every query head h of the group:
//   pass 1: D1 = Q_h * K_tile^T on tcgen05 (M = 64 or 128 text rows, N = 128
//           visual columns) into TMEM; one or two epilogue threads per text row
//           keep an online (max, sum of 2^x) over the columns of all the CTA's
//           tiles;
//   exchange: each CTA publishes its per-row (m, l) in shared memory and
//           signals every CTA of the cluster by remote mbarrier arrivals; each
//           CTA merges the C partials in rank order (deterministic) into
//           b_hi = m_hi * c + log2(l_hi), c = scale * log2(e);
//   pass 2: D2 = K_tile * Q_h^T (M = 128 visual rows, N = T rounded up to 16)
//           into TMEM; one epilogue thread per visual token adds
//           sum_i 2^(s_ij * c - b_hi) to its running score.
// Software pipeline with one head of look-ahead: pass 1 of head s+1 runs while
// the statistics of head s travel across the cluster, then pass 2 of head s
// (a CTA that is its own cluster has nothing to wait for and runs the two
// passes of each head back to back).
// The K tiles stream through a TMA ring for both passes (the pass-2 re-read of
// a CTA's few tiles is normally served by L2). Scores are summed over the heads
// of the group in shared memory; with one head group they are final, with
// several the CTAs write partial rows and the last CTA of the request to finish
// (atomic ticket) adds them in a fixed order.
//
// Warp roles (448 threads): warp 0 = TMA producer, warp 1 = TMEM allocator and
// MMA issuer, warps 2..13 = epilogue in three warpgroups (TMEM lane quadrant =
// warp % 4); the contractions of both passes cycle through four 128-column
// TMEM buffers and warpgroup g takes units u with u % 3 == g.
// Every wait is bounded (clock budget); on expiry the kernel sets the error
// word, drains its own copies and MMAs, frees TMEM and returns.

#include <math.h>

#include "internal.h"
#include "pipe.cuh"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kEpiWG = 3;                    // epilogue warpgroups
constexpr int kEpiThreads = 128 * kEpiWG;
constexpr int kThreads = 64 + kEpiThreads;
constexpr int kStatSlots = 4;  // stats of heads s-3..s may be live across the cluster

// Shared-memory plan. The ring gets whatever is left of the 227 KB after the
// Q double buffer and the bookkeeping; every variant needs more than half of
// the SM's shared memory, so a single CTA (and a single 512-column TMEM
// allocation) lives on an SM at a time.
template <int ROW_BYTES, int MROWS>
struct SmemLayout {
    static constexpr int KB = ROW_BYTES / 128;             // 128-byte swizzle blocks along d
    static constexpr int TILE_BYTES = kTileRows * ROW_BYTES;
    static constexpr int Q_BYTES = MROWS * ROW_BYTES;
    // Q(s) lives from pass 1 of head s to pass 2 of head s; a third buffer lets
    // Q(s+2) load while pass 2 of head s is still reading Q(s).
    static constexpr int QBUF = MROWS == 64 ? 3 : 2;
    static constexpr int FIXED = QBUF * Q_BYTES + kMaxTilesPerCta * kTileRows * 4 + kStatSlots * kMaxText * 8 +
                                 2 * kMaxText * 4 + (kEpiWG - 1) * kMaxText * 8 + kMaxTilesPerCta * 4 + 512 + 64 +
                                 1024;
    static constexpr int STAGES_FIT = (227 * 1024 - FIXED) / TILE_BYTES;
    static constexpr int kStages = STAGES_FIT > 10 ? 10 : STAGES_FIT;
    static constexpr int OFF_K = 0;
    static constexpr int OFF_Q = OFF_K + kStages * TILE_BYTES;
    static constexpr int OFF_ACC = OFF_Q + QBUF * Q_BYTES;
    static constexpr int OFF_STATS = OFF_ACC + kMaxTilesPerCta * kTileRows * 4;
    static constexpr int OFF_B2 = OFF_STATS + kStatSlots * kMaxText * 8;
    static constexpr int OFF_XS = OFF_B2 + 2 * kMaxText * 4;  // [kEpiWG - 1][128] float2: other warpgroups' row stats
    static constexpr int OFF_FLAGS = OFF_XS + (kEpiWG - 1) * kMaxText * 8;  // [32] int, fold flags
    static constexpr int OFF_BAR = OFF_FLAGS + kMaxTilesPerCta * 4;
    // k_full[S], k_empty[S], q_full[QBUF], q_empty[QBUF], t1_full[2], t1_empty[2],
    // t2_full[2], t2_empty[2], stats[4], drain
    static constexpr int NBAR = 2 * kStages + 2 * QBUF + 2 * 4 + kStatSlots + 2;
    static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
    static constexpr int BYTES = OFF_MISC + 16;
    static constexpr int ALLOC = BYTES + 1024;  // slack for 1024-byte alignment
};

template <int ROW_BYTES, bool FP8, int MROWS>
__global__ void __launch_bounds__(kThreads, 1)
    score_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ ScoreLaunch p)
{
    using L = SmemLayout<ROW_BYTES, MROWS>;
    constexpr int KSTEPS = ROW_BYTES / 32;                 // one MMA consumes 32 bytes of d
    constexpr int ELEMS_PER_KB = FP8 ? 128 : 64;           // elements in 128 bytes
    constexpr uint32_t FMT = FP8 ? 0u : 1u;
    constexpr int kStages = L::kStages;
    constexpr int QBUF = L::QBUF;
    static_assert(kStages >= 3, "ring depth");
    static_assert(L::ALLOC > 116 * 1024, "one CTA per SM");
    static_assert(L::ALLOC <= 227 * 1024, "shared memory per CTA");

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (base - raw);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const uint32_t csize = cluster_nctarank();
    const int item = (int)(blockIdx.x / csize);  // this cluster's (request, head group)
    const int req_i = item / p.groups;
    const int b = p.order_n > 0 ? (int)p.order[req_i] : req_i;
    const int hg = item - req_i * p.groups;

    // With the full-key-set terms (p.extra, written by the kernel launched just
    // before this one) only the threads that read them wait for that kernel,
    // right before the read: this kernel's other inputs come from kernels that
    // had completed before that one passed its own wait, so the visual-key work
    // overlaps it. Every CTA still waits before it exits, so this grid never
    // completes ahead of that one.
    if (!p.extra) griddep_wait();
    griddep_launch_dependents();
    // the request's offsets: by value for small batches (no global load)
    const bool byv = p.nv > 0;
    const int n0 = byv ? p.so_v[b] : p.seq_off[b];
    const int N = (byv ? p.so_v[b + 1] : p.seq_off[b + 1]) - n0;
    const int tq = byv ? p.to_v[b] : p.text_off[b];
    const int t1 = byv ? p.to_v[b + 1] : p.text_off[b + 1];
    const int t0 = p.query_last && t1 > tq ? t1 - 1 : tq;  // last-token queries: one row
    const int T = t1 - t0;
    const bool multi = p.groups > 1;
    // Uniform for the whole cluster (same request). With several head groups
    // every CTA must still take its fold ticket, so only shape errors return.
    if (T > MROWS || (N > 0 && T <= 0) || N <= 0) {
        if (p.extra) griddep_wait();
        if (N > 0 && threadIdx.x == 0 && rank == 0 && hg == 0) atomicOr(p.err, kErrShape);
        return;
    }
    const int n_tiles = (N + kTileRows - 1) / kTileRows;
    const int tpc = (n_tiles + (int)csize - 1) / (int)csize;
    const int tile_begin = min(n_tiles, (int)rank * tpc);
    const int tile_end = min(n_tiles, tile_begin + tpc);
    const int mt = tile_end - tile_begin;
    const int n2 = (T + 15) & ~15;
    const int G = p.hq / p.hkv;
    const int hpg = p.heads_per_group;
    const float cl = p.c_log2;
    // Pass 2 of a head follows pass 1 of the next head (lag 1), so the
    // statistics exchange of the cluster overlaps a contraction; a CTA without
    // peers needs no exchange and runs both passes of a head in turn (lag 0),
    // which halves the K tiles that must stay in L2 for the re-read.
    const int lag = csize > 1 ? 1 : 0;

    const uint32_t bar0 = base + L::OFF_BAR;
    auto BAR = [&](int i) -> uint32_t { return bar0 + 8u * (uint32_t)i; };
    // U_FULL / U_EMPTY: a ring of four 128-column TMEM buffers shared by the
    // contractions of both passes, in issue order (unit u uses buffer u % 4)
    const int K_FULL = 0, K_EMPTY = kStages, Q_FULL = 2 * kStages, Q_EMPTY = Q_FULL + QBUF, U_FULL = Q_EMPTY + QBUF,
              U_EMPTY = U_FULL + 4, STATS = U_EMPTY + 4,
              DRAIN = STATS + kStatSlots, STALL = DRAIN + 1;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);
    volatile int* fold_flags = reinterpret_cast<volatile int*>(smem + L::OFF_FLAGS);
    float* acc_s = reinterpret_cast<float*>(smem + L::OFF_ACC);
    float2* stats_s = reinterpret_cast<float2*>(smem + L::OFF_STATS);
    float* b2_s = reinterpret_cast<float*>(smem + L::OFF_B2);
    float2* xs_s = reinterpret_cast<float2*>(smem + L::OFF_XS);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(BAR(K_FULL + s), 1);
            mbar_init(BAR(K_EMPTY + s), 1);
        }
        for (int i = 0; i < QBUF; ++i) {
            mbar_init(BAR(Q_FULL + i), 1);
            mbar_init(BAR(Q_EMPTY + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(BAR(U_FULL + i), 1);
            mbar_init(BAR(U_EMPTY + i), 4);   // one arrival per warp of the consuming warpgroup
            mbar_init(BAR(U_FULL + 2 + i), 1);
            mbar_init(BAR(U_EMPTY + 2 + i), 4);
        }
        for (int i = 0; i < kStatSlots; ++i) mbar_init(BAR(STATS + i), csize);
        mbar_init(BAR(DRAIN), 1);
        mbar_init(BAR(STALL), 1);  // nothing ever arrives (the debug stall below)
        *abort_flag = 0;
        fence_mbar_init_cluster();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_k);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // Cluster barrier, split: every thread arrives now (its CTA's barriers
    // exist) and waits only before its first remote arrival (the epilogue) or
    // before the final barrier (producer, MMA warp), so the first copies and
    // contractions do not wait for the slowest CTA of the cluster. The arrival
    // needs no release: the barriers' set-up is released by fence.mbarrier_init
    // above, and the statistics peers read are released by their own arrivals.
    cluster_arrive_relaxed();
    const uint32_t tmem = *tmem_slot;
    const Ctl ctl{abort_flag, p.err, p.wait_budget};

    // Pipeline step s (0..hpg): pass 1 of head s (s < hpg), then pass 2 of head s-1 (s >= 1).
    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0 && mt > 0) {
            uint32_t ks = 0, kph = 0;
            int k_issued[kStages];
            int q_issued[QBUF];
            for (int s = 0; s < QBUF; ++s) q_issued[s] = 0;
            for (int s = 0; s < kStages; ++s) k_issued[s] = 0;
            // Debug stall (p.stall, a test of the failure path): wait on a barrier
            // that nothing completes before issuing any copy, so this wait runs out
            // of budget and every other wait of the launch runs out or sees the
            // abort flag, with no copy or contraction in flight.
            bool ok = !p.stall || wait_phase(BAR(STALL), 0, ctl);
            auto load_tiles = [&](int g) {
                for (int t = tile_begin; t < tile_end && ok; ++t) {
                    if (!wait_phase(BAR(K_EMPTY + ks), kph ^ 1, ctl)) { ok = false; break; }
                    mbar_arrive_expect_tx(BAR(K_FULL + ks), L::TILE_BYTES);
                    const uint32_t kdst = base + L::OFF_K + ks * L::TILE_BYTES;
#pragma unroll
                    for (int kb = 0; kb < L::KB; ++kb)
                        tma_load_3d(kdst + kb * kTileRows * 128, &tm_k, BAR(K_FULL + ks), kb * ELEMS_PER_KB, g,
                                    n0 + t * kTileRows);
                    ++k_issued[ks];
                    if (++ks == kStages) { ks = 0; kph ^= 1; }
                }
            };
            for (int s = 0; s < hpg + lag && ok; ++s) {
                if (s < hpg) {
                    const int h = hg * hpg + s;
                    const int qb = s % QBUF;
                    if (!wait_phase(BAR(Q_EMPTY + qb), ((s / QBUF) & 1) ^ 1, ctl)) break;
                    mbar_arrive_expect_tx(BAR(Q_FULL + qb), L::Q_BYTES);
                    const uint32_t qdst = base + L::OFF_Q + qb * L::Q_BYTES;
#pragma unroll
                    for (int kb = 0; kb < L::KB; ++kb)
                        tma_load_3d(qdst + kb * MROWS * 128, &tm_q, BAR(Q_FULL + qb), kb * ELEMS_PER_KB, h, t0);
                    ++q_issued[qb];
                    load_tiles(h / G);
                }
                if (s >= lag && ok) load_tiles((hg * hpg + s - lag) / G);
            }
            // drain: the last load of every slot lands before the CTA leaves
            // (these waits ignore the abort flag)
            volatile int no_abort = 0;
            const Ctl drain_ctl{&no_abort, p.err, kWaitBudgetCycles};
            for (int s = 0; s < kStages; ++s)
                if (k_issued[s] > 0) wait_phase(BAR(K_FULL + s), (uint32_t)(k_issued[s] - 1) & 1u, drain_ctl);
            for (int s = 0; s < QBUF; ++s)
                if (q_issued[s] > 0) wait_phase(BAR(Q_FULL + s), (uint32_t)(q_issued[s] - 1) & 1u, drain_ctl);
        }
        __syncwarp();
        cluster_wait();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            if (mt > 0) {
                const uint32_t idesc1 = idesc_make(MROWS, 128, FMT);
                const uint32_t idesc2 = idesc_make(128, (uint32_t)n2, FMT);
                uint32_t ks = 0, kph = 0, ui = 0;
                bool ok = true;
                for (int s = 0; s < hpg + lag && ok; ++s) {
                    for (int pass = 0; pass < 2 && ok; ++pass) {
                        if (pass == 0 && s >= hpg) continue;
                        if (pass == 1 && s < lag) continue;
                        const int hs = pass == 0 ? s : s - lag;  // head of this unit
                        const int qb = hs % QBUF;
                        if (pass == 0) {
                            if (!wait_phase(BAR(Q_FULL + qb), (hs / QBUF) & 1, ctl)) { ok = false; break; }
                            tc_fence_after();
                        }
                        const uint32_t qaddr = base + L::OFF_Q + qb * L::Q_BYTES;
                        for (int t = tile_begin; t < tile_end; ++t) {
                            if (!wait_phase(BAR(K_FULL + ks), kph, ctl)) { ok = false; break; }
                            const uint32_t ub = ui & 3, uph = (ui >> 2) & 1;
                            if (!wait_phase(BAR(U_EMPTY + ub), uph ^ 1, ctl)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            const uint32_t kaddr = base + L::OFF_K + ks * L::TILE_BYTES;
                            const uint32_t d = tmem + ub * 128u;
#pragma unroll
                            for (int st = 0; st < KSTEPS; ++st) {
                                const uint32_t koff = (st >> 2) * (kTileRows * 128) + (st & 3) * 32;
                                const uint32_t qoff = (st >> 2) * (MROWS * 128) + (st & 3) * 32;
                                const uint64_t qd = sdesc_k_sw128(qaddr + qoff);
                                const uint64_t kd = sdesc_k_sw128(kaddr + koff);
                                if (pass == 0) {
                                    if (FP8) mma_f8(d, qd, kd, idesc1, st > 0);
                                    else mma_f16(d, qd, kd, idesc1, st > 0);
                                } else {
                                    if (FP8) mma_f8(d, kd, qd, idesc2, st > 0);
                                    else mma_f16(d, kd, qd, idesc2, st > 0);
                                }
                            }
                            mma_commit(BAR(U_FULL + ub));
                            mma_commit(BAR(K_EMPTY + ks));
                            ++ui;
                            if (++ks == kStages) { ks = 0; kph ^= 1; }
                        }
                        if (pass == 1 && ok) mma_commit(BAR(Q_EMPTY + qb));  // last reader of Q(hs)
                    }
                }
            }
            // drain: every MMA issued by this thread has completed
            mma_commit(BAR(DRAIN));
            volatile int no_abort = 0;
            const Ctl drain_ctl{&no_abort, p.err, kWaitBudgetCycles};
            wait_phase(BAR(DRAIN), 0, drain_ctl);
        }
        __syncwarp();
        cluster_wait();
    } else {
        // ------------------------------------------------------------ epilogue
        cluster_wait();  // the peers' barriers and buffers exist before any statistics go out
        // Three warpgroups (warps 2-5, 6-9, 10-13). The contractions of both
        // passes cycle through four TMEM buffers in issue order; warpgroup g
        // takes the units u with u % 3 == g, in order, so while one warpgroup
        // reads a buffer the others' units are being filled. A unit's buffer
        // was last used by unit u - 4, which belongs to another warpgroup and
        // comes earlier in that warpgroup's order, so no wait is circular. Control flow is identical within a
        // warpgroup (named barriers); after an abort every wait returns at once
        // and the steps run out.
        const int quad = warp & 3;
        const int wg = (warp - 2) >> 2;                       // 0 .. kEpiWG - 1
        const int et = threadIdx.x - 64;                      // 0..255
        const int vrow = quad * 32 + lane;                    // pass 2: TMEM lane = visual token in tile
        const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
        // pass 1 row of this thread: M=128 -> lane; M=64 -> lanes 16q..16q+15, two column halves
        const int prow = MROWS == 128 ? quad * 32 + lane : quad * 16 + (lane & 15);
        const int phalf = MROWS == 128 ? 0 : (lane >> 4);
        const bool p1_live = MROWS == 128 ? (quad * 32 < T) : (quad * 16 < T);
        for (int tl = wg; tl < mt; tl += kEpiWG) acc_s[tl * kTileRows + vrow] = 0.f;
        uint32_t ui = 0;  // contraction units in issue order (both passes)
        for (int s = 0; s < hpg + lag; ++s) {
            if (s < hpg) {
                // ---- pass 1 of head s: online row statistics over this warpgroup's tiles
                float m = -INFINITY, l = 0.f;
                for (int t = tile_begin; t < tile_end; ++t, ++ui) {
                    const uint32_t ub = ui & 3;
                    if ((int)(ui % kEpiWG) != wg) continue;
                    wait_phase(BAR(U_FULL + ub), (ui >> 2) & 1, ctl);
                    tc_fence_after();
                    const uint32_t ta = tmem + lane_off + ub * 128u;
                    // 32 columns at a time: M = 64 -> this thread's half of the row
                    // (columns 64 * phalf + [0, 64)); M = 128 -> the whole row
                    constexpr int NH = MROWS == 128 ? 4 : 2;
#pragma unroll
                    for (int hh = 0; hh < NH; ++hh) {
                        float v[32];
                        if (p1_live) {
                            if constexpr (MROWS == 128) tmem_ld32(ta + hh * 32, v);
                            else tmem_ld16x2_32<64>(ta + hh * 32, v);
                            tmem_wait_ld();
                        }
                        if (hh == NH - 1) {
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(BAR(U_EMPTY + ub));
                        }
                        if (p1_live) {
                            const int valid = N - t * kTileRows - (MROWS == 128 ? 0 : phalf * 64) - hh * 32;
                            row_stats_update<32>(v, valid, cl, m, l);
                        }
                    }
                }
                if (MROWS == 64) {
                    // merge the two column halves of each row (threads t and t ^ 16)
                    const float mo = __shfl_xor_sync(0xffffffffu, m, 16);
                    const float lo = __shfl_xor_sync(0xffffffffu, l, 16);
                    const float mm = fmaxf(m, mo);
                    if (mm != -INFINITY) {
                        l = (l > 0.f ? l * ex2((m - mm) * cl) : 0.f) + (lo > 0.f ? lo * ex2((mo - mm) * cl) : 0.f);
                        m = mm;
                    }
                }
                // ---- merge the warpgroups, publish (m, l) of head s to the cluster
                const bool writer = MROWS == 128 || lane < 16;
                if (wg > 0 && writer) xs_s[(wg - 1) * kMaxText + prow] = make_float2(m, l);
                named_bar_sync(1, kEpiThreads);
                if (wg == 0) {
                    if (writer) {
#pragma unroll
                        for (int o_wg = 1; o_wg < kEpiWG; ++o_wg) {  // fixed order: deterministic
                            const float2 o = xs_s[(o_wg - 1) * kMaxText + prow];
                            const float mm = fmaxf(m, o.x);
                            if (mm != -INFINITY) {
                                l = (l > 0.f ? l * ex2((m - mm) * cl) : 0.f) +
                                    (o.y > 0.f ? o.y * ex2((o.x - mm) * cl) : 0.f);
                                m = mm;
                            }
                        }
                        stats_s[(s % kStatSlots) * kMaxText + prow] = make_float2(m, l);
                    }
                    named_bar_sync(2, 128);
                    // one release arrival per CTA of the cluster, each from its own
                    // thread: a release at cluster scope covers the rows the other
                    // threads wrote before the named barrier, and the arrivals'
                    // fences (each waits for this SM's memory traffic to settle)
                    // overlap instead of running one after another
                    if (et < (int)csize) mbar_arrive_remote(mapa_shared(BAR(STATS + s % kStatSlots), (uint32_t)et));
                }
            }
            if (s >= lag) {
                // ---- merge the cluster's statistics of head s-1
                const int hs = s - lag;
                const int slot = hs % kStatSlots;
                float* b2 = b2_s + (hs & 1) * kMaxText;
                if (wg == 0) {
                    wait_phase_cluster(BAR(STATS + slot), (uint32_t)(hs / kStatSlots) & 1u, ctl);
                    if (et < T) {
                        float bm = merge_cluster_row(base + L::OFF_STATS + (uint32_t)(slot * kMaxText + et) * 8u, csize, cl);
                        if (p.extra) {
                            griddep_wait();
                            bm = log2_add(bm, p.extra[(int64_t)(t0 + et) * p.hq + hg * hpg + hs]);
                        }
                        b2[et] = -bm;  // stored negated: the fma addend of pass 2
                    } else {
                        b2[et] = -INFINITY;
                    }
                }
                named_bar_sync(1, kEpiThreads);
                // ---- pass 2 of head s-1: per-visual-token sums of probabilities
                for (int t = tile_begin; t < tile_end; ++t, ++ui) {
                    const uint32_t ub = ui & 3;
                    if ((int)(ui % kEpiWG) != wg) continue;
                    wait_phase(BAR(U_FULL + ub), (ui >> 2) & 1, ctl);
                    tc_fence_after();
                    const uint32_t ta = tmem + lane_off + ub * 128u;
                    float2 a01 = make_float2(0.f, 0.f), a23 = make_float2(0.f, 0.f);
                    const float2 cl2 = make_float2(cl, cl);
#pragma unroll
                    for (int hh = 0; hh < MROWS / 32; ++hh) {
                        const int c0 = hh * 32;
                        if (c0 < n2) {
                            float v[32];
                            if (c0 + 32 <= n2) tmem_ld32(ta + c0, v);
                            else tmem_ld16(ta + c0, v);
                            tmem_wait_ld();
#pragma unroll
                            for (int k = 0; k < 2; ++k) {
                                if (c0 + k * 16 < n2) {
#pragma unroll
                                    for (int e = 0; e < 16; e += 4) {
                                        const float4 bb = *reinterpret_cast<const float4*>(b2 + c0 + k * 16 + e);
                                        const float2 x01 = ffma2(make_float2(v[k * 16 + e], v[k * 16 + e + 1]), cl2,
                                                                 make_float2(bb.x, bb.y));
                                        const float2 x23 = ffma2(make_float2(v[k * 16 + e + 2], v[k * 16 + e + 3]),
                                                                 cl2, make_float2(bb.z, bb.w));
                                        a01 = fadd2(a01, make_float2(ex2(x01.x), ex2(x01.y)));
                                        a23 = fadd2(a23, make_float2(ex2(x23.x), ex2(x23.y)));
                                    }
                                }
                            }
                        }
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(BAR(U_EMPTY + ub));
                    acc_s[(t - tile_begin) * kTileRows + vrow] += (a01.x + a01.y) + (a23.x + a23.y);
                }
            }
        }
        named_bar_sync(1, kEpiThreads);  // every tile's sums are in acc_s
        // ---- results
        const float denom = (float)p.hq * (float)T;
        for (int tl = wg; tl < mt; tl += kEpiWG) {
            const int j = (tile_begin + tl) * kTileRows + vrow;
            if (j < N) {
                const float a = acc_s[tl * kTileRows + vrow];
                if (!multi) p.out[n0 + j] = a / denom;
                else p.partials[(int64_t)hg * p.total_vis + n0 + j] = a;
            }
        }
        if (multi && !p.defer_fold) fold_tiles<4>(p, b, n0, N, T, tile_begin, mt, et, kEpiThreads, 1, fold_flags);
        tc_fence_before();
    }

    // ---------------------------------------------------------------- teardown
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
    if (p.extra) griddep_wait();  // returns at once for threads that already waited
    cluster_sync_all();  // peers are done reading this CTA's statistics
}

template <int ROW_BYTES, bool FP8, int MROWS>
cudaError_t tc_prepare(int cluster)
{
    auto kern = score_tc_kernel<ROW_BYTES, FP8, MROWS>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         SmemLayout<ROW_BYTES, MROWS>::ALLOC);
    if (e == cudaSuccess && cluster > 8) e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    return e;
}

// CTAs resident at once with clusters of `cluster` CTAs (occupancy query)
template <int ROW_BYTES, bool FP8, int MROWS>
int tc_capacity(int cluster)
{
    if (tc_prepare<ROW_BYTES, FP8, MROWS>(cluster) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cluster * 64, 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = SmemLayout<ROW_BYTES, MROWS>::ALLOC;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, score_tc_kernel<ROW_BYTES, FP8, MROWS>, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return n * cluster;
}

template <int ROW_BYTES, bool FP8, int MROWS>
cudaError_t launch_variant(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const ScoreLaunch& p,
                           const ScorePlan& plan, int batch, cudaStream_t stream)
{
    auto kern = score_tc_kernel<ROW_BYTES, FP8, MROWS>;
    const int smem = SmemLayout<ROW_BYTES, MROWS>::ALLOC;
    cudaError_t e = tc_prepare<ROW_BYTES, FP8, MROWS>(plan.cluster);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(plan.cluster * plan.groups * batch), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
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

}  // namespace

int tc_cluster_capacity(int row_bytes, bool fp8, int mrows, int cluster)
{
    if (fp8) return mrows == 64 ? tc_capacity<128, true, 64>(cluster) : tc_capacity<128, true, 128>(cluster);
    if (row_bytes == 256)
        return mrows == 64 ? tc_capacity<256, false, 64>(cluster) : tc_capacity<256, false, 128>(cluster);
    return mrows == 64 ? tc_capacity<128, false, 64>(cluster) : tc_capacity<128, false, 128>(cluster);
}

bool score_shape_supported(int head_dim, bool fp8)
{
    if (fp8) return head_dim == 128;
    return head_dim == 64 || head_dim == 128;
}

// CTAs of one cluster size that run at once with one CTA per SM (GPC packing
// on a 152-SM GB300: 1, 2 -> 152; 4 -> 144; 8 -> 120; 16 -> 112).
ScorePlan plan_score(const BatchTiles& bt, int hq, int hkv, int tile_bytes, const int* cap_by_cluster,
                     double* cost_out)
{
    ScorePlan best{1, 1, 1};
    double best_cost = 1e300;
    const int max_tiles = bt.n > 0 ? bt.desc[0] : 0;
    if (max_tiles <= 0) {
        if (cost_out) *cost_out = 0.0;
        return best;
    }
    const int G = hq / hkv;
    for (int pass = 0; pass < 2 && best_cost >= 1e299; ++pass) {
        for (int c = 1; c <= kMaxCluster; ++c) {
            const int tpc = (max_tiles + c - 1) / c;
            if (tpc > kMaxTilesPerCta) continue;
            if (c > 1 && (c - 1) * tpc >= max_tiles) continue;  // an idle rank on the largest request
            const int cap = cap_by_cluster[c];
            if (cap < c) continue;
            for (int g = 1; g <= hq; ++g) {
                if (hq % g) continue;
                const long long ctas = (long long)bt.n * c * g;
                const int hpg = hq / g;
                // L2 window of the pass-2 re-read: while a CTA streams up to two
                // slices (pass 1 of the next head, rest of the current one) the
                // tiles it re-reads must survive in L2. Groups that split a GQA
                // key head share its tiles. The bound is loose (160 MB against
                // 126 MB of L2): the re-read follows pass 1 within one head, and
                // on GB300 whole-request CTAs with this nominal window measured
                // faster than clusters of two (fp8_ragged: 176 vs 201 us).
                const long long active = ctas < cap ? ctas : cap;
                const int share = hpg >= G ? 1 : G / hpg;
                const double window = 2.0 * tpc * tile_bytes * (double)active / share;
                if (pass == 0 && window > 160.0 * 1024 * 1024) continue;
                // one cluster (item): one tile-head of work per tile and head, plus
                // a fixed launch / pipeline fill cost of about 6 tile-heads and a
                // cluster exchange of about 1 tile-head per head; a fold when g > 1
                auto item_cost = [&](int tiles) {
                    const int t = (tiles + c - 1) / c;
                    return tiles <= 0 ? 1.0
                                      : (double)t * hpg + 6.0 + (c > 1 ? 1.0 : 0.25) * hpg + (g > 1 ? 2.0 : 0.0);
                };
                const double cost = makespan(bt, g, cap / c, item_cost);
                if (cost < best_cost - 1e-9) {
                    best_cost = cost;
                    best = ScorePlan{c, tpc, g};
                }
            }
        }
    }
    if (cost_out) *cost_out = best_cost;
    return best;
}

cudaError_t launch_score(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const ScoreLaunch& p,
                         const ScorePlan& plan, int batch, int row_bytes, bool fp8, int mrows, cudaStream_t stream)
{
    ScoreLaunch q = p;
    q.groups = plan.groups;
    q.heads_per_group = p.hq / plan.groups;
    q.ctas_per_request = plan.cluster * plan.groups;
    if (fp8) {
        return mrows == 64 ? launch_variant<128, true, 64>(tm_q, tm_k, q, plan, batch, stream)
                           : launch_variant<128, true, 128>(tm_q, tm_k, q, plan, batch, stream);
    }
    if (row_bytes == 256) {
        return mrows == 64 ? launch_variant<256, false, 64>(tm_q, tm_k, q, plan, batch, stream)
                           : launch_variant<256, false, 128>(tm_q, tm_k, q, plan, batch, stream);
    }
    return mrows == 64 ? launch_variant<128, false, 64>(tm_q, tm_k, q, plan, batch, stream)
                       : launch_variant<128, false, 128>(tm_q, tm_k, q, plan, batch, stream);
}

}  // namespace lvs
