// Pipeline helpers shared by the score kernels: bounded mbarrier waits and
// the online row-statistics update of the softmax normaliser.
#pragma once

#include <math.h>
#include <stdint.h>

#include "internal.h"
#include "ptx.cuh"

namespace lvs {

struct Ctl {
    volatile int* abort;
    int32_t* err;
    long long budget;
};

// Suspend-time hint of the retries (ns): a waiting thread sleeps until its
// phase completes or this much time passes, then checks the abort flag and
// the budget.
constexpr uint32_t kWaitSleepNs = 20000;

__device__ __forceinline__ bool wait_phase(uint32_t bar, uint32_t parity, const Ctl& c)
{
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    for (;;) {
        if (*c.abort) return false;  // checked before sleeping, so waits after an abort end at once
        if (mbar_try_wait_sleep(bar, parity, kWaitSleepNs)) return true;
        if (clock64() - t0 > c.budget) {
            *c.abort = 1;
            atomicOr(c.err, kErrTimeout);
            return false;
        }
    }
}

__device__ __forceinline__ bool wait_phase_cluster(uint32_t bar, uint32_t parity, const Ctl& c)
{
    if (mbar_try_wait_cluster(bar, parity)) return true;
    const long long t0 = clock64();
    for (;;) {
        if (*c.abort) return false;  // checked before sleeping, so waits after an abort end at once
        if (mbar_try_wait_cluster_sleep(bar, parity, kWaitSleepNs)) return true;
        if (clock64() - t0 > c.budget) {
            *c.abort = 1;
            atomicOr(c.err, kErrTimeout);
            return false;
        }
    }
}

// Online (max, sum 2^(x*c - max*c)) update of one row over NV columns.
template <int NV>
__device__ __forceinline__ void row_stats_update(const float* v, int valid, float cl, float& m, float& l)
{
    float mx0 = -INFINITY, mx1 = -INFINITY, mx2 = -INFINITY, mx3 = -INFINITY;
    if (valid >= NV) {
#pragma unroll
        for (int c = 0; c < NV; c += 8) {
            mx0 = fmax3(mx0, v[c], v[c + 1]);
            mx1 = fmax3(mx1, v[c + 2], v[c + 3]);
            mx2 = fmax3(mx2, v[c + 4], v[c + 5]);
            mx3 = fmax3(mx3, v[c + 6], v[c + 7]);
        }
    } else {
#pragma unroll
        for (int c = 0; c < NV; c += 4) {
            mx0 = fmaxf(mx0, c < valid ? v[c] : -INFINITY);
            mx1 = fmaxf(mx1, c + 1 < valid ? v[c + 1] : -INFINITY);
            mx2 = fmaxf(mx2, c + 2 < valid ? v[c + 2] : -INFINITY);
            mx3 = fmaxf(mx3, c + 3 < valid ? v[c + 3] : -INFINITY);
        }
    }
    const float m_new = fmaxf(m, fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)));
    if (m_new == -INFINITY) return;  // no valid column yet
    const float mc = m_new * cl;
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
    if (valid >= NV) {
        // packed pairs: the same per-column fma and sums, half the instructions
        const float2 cl2 = make_float2(cl, cl), nmc2 = make_float2(-mc, -mc);
        float2 s01 = make_float2(0.f, 0.f), s23 = make_float2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < NV; c += 4) {
            const float2 x01 = ffma2(make_float2(v[c], v[c + 1]), cl2, nmc2);
            const float2 x23 = ffma2(make_float2(v[c + 2], v[c + 3]), cl2, nmc2);
            s01 = fadd2(s01, make_float2(ex2(x01.x), ex2(x01.y)));
            s23 = fadd2(s23, make_float2(ex2(x23.x), ex2(x23.y)));
        }
        s0 = s01.x;
        s1 = s01.y;
        s2 = s23.x;
        s3 = s23.y;
    } else {
#pragma unroll
        for (int c = 0; c < NV; c += 4) {
            s0 += c < valid ? ex2(fmaf(v[c], cl, -mc)) : 0.f;
            s1 += c + 1 < valid ? ex2(fmaf(v[c + 1], cl, -mc)) : 0.f;
            s2 += c + 2 < valid ? ex2(fmaf(v[c + 2], cl, -mc)) : 0.f;
            s3 += c + 3 < valid ? ex2(fmaf(v[c + 3], cl, -mc)) : 0.f;
        }
    }
    l = l * ex2((m - m_new) * cl) + ((s0 + s1) + (s2 + s3));
    m = m_new;
}

// log2(2^x + 2^y) for the merged statistic b and a normaliser term of other
// keys in the same unit (x finite)
__device__ __forceinline__ float log2_add(float x, float y)
{
    const float mx = fmaxf(x, y), mn = fminf(x, y);
    return mx + __log2f(1.f + ex2(mn - mx));
}

// Merges the (max, sum) partials of one row from every CTA of the cluster in
// rank order and returns b = M * c + log2(L). All remote loads are issued
// before any is used, so their latencies overlap.
__device__ __forceinline__ float merge_cluster_row(uint32_t my_addr, uint32_t csize, float cl)
{
    float2 st[kMaxCluster];
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r)
        if (r < (int)csize) st[r] = ld_shared_cluster_f2(mapa_shared(my_addr, (uint32_t)r));
    float M = -INFINITY;
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r)
        if (r < (int)csize) M = fmaxf(M, st[r].x);
    float L = 0.f;
#pragma unroll
    for (int r = 0; r < kMaxCluster; ++r)
        if (r < (int)csize && st[r].y > 0.f) L += st[r].y * ex2((st[r].x - M) * cl);
    return fmaf(M, cl, __log2f(L));
}

// Ticket slot of tile t of the request starting at row n0 (request b): unique
// over the batch because floor((n0 + N) / 128) - floor(n0 / 128) >= tiles - 1.
__device__ __forceinline__ int fold_ticket_index(int b, int n0, int t) { return n0 / kTileRows + t + b; }

// After a CTA wrote its partial rows (head group hg) for tiles [tile_begin,
// tile_begin + mt): take one ticket per tile; the last of the `parts` CTAs
// (default: the head groups) that own a tile adds the partials of that tile
// in index order and writes the scores. `nthreads` threads (ids 0..nthreads-1, synchronised by
// named barrier `bar_id`) take part; `flags` is shared memory for mt ints.
// Each thread sums R rows at a time, with the loads of all R rows (up to 16
// partials each) in flight together: a CTA that folds a long request's tiles
// alone pays one L2 round trip per R rows instead of one per row.
template <int R = 1>
__device__ __forceinline__ void fold_tiles(const ScoreLaunch& p, int b, int n0, int N, int T, int tile_begin,
                                           int mt, int tid, int nthreads, uint32_t bar_id, volatile int* flags,
                                           int parts = 0)
{
    if (parts <= 0) parts = p.groups;  // partial rows of this request (head groups, or clusters of a flat launch)
    __threadfence();
    named_bar_sync(bar_id, nthreads);
    for (int tl = tid; tl < mt; tl += nthreads) {
        int* c = p.counters + fold_ticket_index(b, n0, tile_begin + tl);
        const int ticket = atomicAdd(c, 1);
        const int last = ticket == parts - 1;
        if (last) *c = 0;  // ready for the next launch
        flags[tl] = last;
    }
    named_bar_sync(bar_id, nthreads);
    __threadfence();
    const float denom = (float)p.hq * (float)T;
    if constexpr (R == 1) {
        // (tile, row) pairs spread over all threads; up to 16 group partials in
        // flight per row, added in group order
        for (int x = tid; x < mt * kTileRows; x += nthreads) {
            const int tl = x / kTileRows;
            if (!flags[tl]) continue;
            const int j = (tile_begin + tl) * kTileRows + (x - tl * kTileRows);
            if (j >= N) continue;
            const float* src = p.partials + n0 + j;
            float sum = 0.f;
            for (int g = 0; g < parts; g += 16) {
                float v[16];
#pragma unroll
                for (int q = 0; q < 16; ++q) v[q] = g + q < parts ? __ldcg(src + (int64_t)(g + q) * p.total_vis) : 0.f;
#pragma unroll
                for (int q = 0; q < 16; ++q)
                    if (g + q < parts) sum += v[q];
            }
            p.out[n0 + j] = sum / denom;
        }
    } else {
        // thread tid takes rows x = tid + k * nthreads, R of them at a time, their
        // group partials added in group order
        for (int x0 = tid; x0 < mt * kTileRows; x0 += R * nthreads) {
            int j[R];
            bool live[R];
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int x = x0 + r * nthreads;
                const int tl = x / kTileRows;
                j[r] = (tile_begin + tl) * kTileRows + (x - tl * kTileRows);
                live[r] = x < mt * kTileRows && flags[tl] && j[r] < N;
            }
            float sum[R];
#pragma unroll
            for (int r = 0; r < R; ++r) sum[r] = 0.f;
            for (int g = 0; g < parts; g += 16) {
                float v[R][16];
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int q = 0; q < 16; ++q)
                        v[r][q] = live[r] && g + q < parts
                                      ? __ldcg(p.partials + n0 + j[r] + (int64_t)(g + q) * p.total_vis)
                                      : 0.f;
#pragma unroll
                for (int r = 0; r < R; ++r)
#pragma unroll
                    for (int q = 0; q < 16; ++q)
                        if (g + q < parts) sum[r] += v[r][q];
            }
#pragma unroll
            for (int r = 0; r < R; ++r)
                if (live[r]) p.out[n0 + j[r]] = sum[r] / denom;
        }
    }
}

}  // namespace lvs
