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
// of the request. For each query head h of the group, the CTA
//   pass 1: D1 = Q_h * K_tile^T on tcgen05 (M = 128 text rows, N = 128 visual
//           columns) into TMEM; one epilogue thread per text row keeps an online
//           (max, sum of exp) over the columns of all its tiles;
//   exchange: each CTA publishes its per-row (m, l) in shared memory and
//           signals every CTA of the cluster through remote mbarrier arrivals;
//           every CTA merges the C partials in rank order (deterministic) into
//           b_hi = m_hi*log2(e)*scale + log2(l_hi);
//   pass 2: D2 = K_tile * Q_h^T (M = 128 visual rows, N = T rounded up to 16)
//           into TMEM; one epilogue thread per visual token adds
//           sum_i 2^(s_ij*c - b_hi) to its running score.
// The K tiles stream through a TMA ring twice per head (the second pass reads
// the CTA's few tiles again, normally from L2). Scores sum over the heads of
// the group in shared memory; one head group writes final scores, several
// write partial rows that a fold kernel adds in a fixed order.
//
// Warp roles (192 threads): warp 0 = TMA producer, warp 1 = TMEM allocator and
// MMA issuer, warps 2..5 = epilogue (TMEM lane quadrant = warp % 4).
// Every wait is bounded (clock budget); on expiry the kernel sets the error
// word, drains its own copies and MMAs, frees TMEM and returns.

#include <math.h>

#include "internal.h"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kThreads = 192;

// Ring depth: 4 x 32 KB tiles for 256-byte rows, 8 x 16 KB for 128-byte rows.
// Both layouts need more than half of the SM's shared memory, so a single CTA
// (and a single 512-column TMEM allocation) lives on an SM at a time.
template <int ROW_BYTES>
struct SmemLayout {
    static constexpr int kStages = ROW_BYTES == 256 ? 4 : 8;
    static constexpr int KB = ROW_BYTES / 128;             // 128-byte swizzle blocks along d
    static constexpr int TILE_BYTES = kTileRows * ROW_BYTES;
    static constexpr int Q_BYTES = kMaxText * ROW_BYTES;   // Q tile: 128 text rows
    static constexpr int OFF_K = 0;
    static constexpr int OFF_Q = OFF_K + kStages * TILE_BYTES;
    static constexpr int OFF_ACC = OFF_Q + 2 * Q_BYTES;
    static constexpr int OFF_STATS = OFF_ACC + kMaxTilesPerCta * kTileRows * 4;
    static constexpr int OFF_B2 = OFF_STATS + 2 * kMaxText * 8;
    static constexpr int OFF_BAR = OFF_B2 + kMaxText * 4;
    // barriers: k_full[S], k_empty[S], q_full[2], q_empty[2], t1_full[2], t1_empty[2],
    //           t2_full[2], t2_empty[2], stats[2], drain
    static constexpr int NBAR = 2 * kStages + 2 * 2 * 4 + 2 + 1;
    static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
    static constexpr int BYTES = OFF_MISC + 16;
    static constexpr int ALLOC = BYTES + 1024;  // slack for 1024-byte alignment
};

struct Ctl {
    volatile int* abort;
    int32_t* err;
    long long budget;
};

__device__ __forceinline__ bool wait_phase(uint32_t bar, uint32_t parity, const Ctl& c)
{
    if (mbar_try_wait(bar, parity)) return true;
    const long long t0 = clock64();
    for (;;) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*c.abort) return false;
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
        if (mbar_try_wait_cluster(bar, parity)) return true;
        if (*c.abort) return false;
        if (clock64() - t0 > c.budget) {
            *c.abort = 1;
            atomicOr(c.err, kErrTimeout);
            return false;
        }
    }
}

template <int ROW_BYTES, bool FP8>
__global__ void __launch_bounds__(kThreads, 1)
    score_tc_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                    const ScoreLaunch p)
{
    using L = SmemLayout<ROW_BYTES>;
    constexpr int KSTEPS = ROW_BYTES / 32;                 // one MMA consumes 32 bytes of d
    constexpr int ELEMS_PER_KB = FP8 ? 128 : 64;           // elements in 128 bytes
    constexpr uint32_t FMT = FP8 ? 0u : 1u;
    constexpr int kStages = L::kStages;
    static_assert(L::ALLOC > 116 * 1024, "one CTA per SM");
    static_assert(L::ALLOC <= 227 * 1024, "shared memory per CTA");

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (base - raw);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b = blockIdx.z, hg = blockIdx.y;
    const uint32_t rank = cluster_ctarank();
    const uint32_t csize = cluster_nctarank();

    const int n0 = p.seq_off[b];
    const int N = p.seq_off[b + 1] - n0;
    const int t0 = p.text_off[b];
    const int T = p.text_off[b + 1] - t0;
    // Uniform for the whole cluster (same request): nothing touched yet.
    if (N <= 0 || T <= 0 || T > kMaxText) {
        if (N > 0 && threadIdx.x == 0 && rank == 0) atomicOr(p.err, kErrShape);
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

    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::OFF_BAR);
    const uint32_t bar0 = base + L::OFF_BAR;
    auto BAR = [&](int i) -> uint32_t { return bar0 + 8u * (uint32_t)i; };
    const int K_FULL = 0, K_EMPTY = kStages, Q_FULL = 2 * kStages, Q_EMPTY = Q_FULL + 2, T1_FULL = Q_EMPTY + 2,
              T1_EMPTY = T1_FULL + 2, T2_FULL = T1_EMPTY + 2, T2_EMPTY = T2_FULL + 2, STATS = T2_EMPTY + 2,
              DRAIN = STATS + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);
    float* acc_s = reinterpret_cast<float*>(smem + L::OFF_ACC);
    float2* stats_s = reinterpret_cast<float2*>(smem + L::OFF_STATS);
    float* b2_s = reinterpret_cast<float*>(smem + L::OFF_B2);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(BAR(K_FULL + s), 1);
            mbar_init(BAR(K_EMPTY + s), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(BAR(Q_FULL + i), 1);
            mbar_init(BAR(Q_EMPTY + i), 1);
            mbar_init(BAR(T1_FULL + i), 1);
            mbar_init(BAR(T1_EMPTY + i), 128);
            mbar_init(BAR(T2_FULL + i), 1);
            mbar_init(BAR(T2_EMPTY + i), 128);
            mbar_init(BAR(STATS + i), csize);
        }
        mbar_init(BAR(DRAIN), 1);
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
    cluster_sync_all();  // every CTA's barriers exist before any remote arrival
    const uint32_t tmem = *tmem_slot;
    (void)bars;

    const Ctl ctl{abort_flag, p.err, p.wait_budget};

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0 && mt > 0) {
            uint32_t ks = 0, kph = 0;
            int k_issued[kStages];
            int q_issued[2] = {0, 0};
            for (int s = 0; s < kStages; ++s) k_issued[s] = 0;
            bool ok = true;
            for (int hi = 0; hi < hpg && ok; ++hi) {
                const int h = hg * hpg + hi;
                const int g = h / G;
                const int qb = hi & 1;
                if (!wait_phase(BAR(Q_EMPTY + qb), ((hi >> 1) & 1) ^ 1, ctl)) { ok = false; break; }
                mbar_arrive_expect_tx(BAR(Q_FULL + qb), L::Q_BYTES);
                const uint32_t qdst = base + L::OFF_Q + qb * L::Q_BYTES;
#pragma unroll
                for (int kb = 0; kb < L::KB; ++kb)
                    tma_load_3d(qdst + kb * kMaxText * 128, &tm_q, BAR(Q_FULL + qb), kb * ELEMS_PER_KB, h, t0);
                ++q_issued[qb];
                for (int pass = 0; pass < 2 && ok; ++pass) {
                    for (int t = tile_begin; t < tile_end; ++t) {
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
                }
            }
            // drain: the last load of every slot must land before the CTA leaves
            for (int s = 0; s < kStages; ++s)
                if (k_issued[s] > 0) wait_phase(BAR(K_FULL + s), (uint32_t)(k_issued[s] - 1) & 1u, ctl);
            for (int s = 0; s < 2; ++s)
                if (q_issued[s] > 0) wait_phase(BAR(Q_FULL + s), (uint32_t)(q_issued[s] - 1) & 1u, ctl);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            if (mt > 0) {
                const uint32_t idesc1 = idesc_make(128, 128, FMT);
                const uint32_t idesc2 = idesc_make(128, (uint32_t)n2, FMT);
                uint32_t ks = 0, kph = 0, t1i = 0, t2i = 0;
                bool ok = true;
                for (int hi = 0; hi < hpg && ok; ++hi) {
                    const int qb = hi & 1;
                    if (!wait_phase(BAR(Q_FULL + qb), (hi >> 1) & 1, ctl)) break;
                    tc_fence_after();
                    const uint32_t qaddr = base + L::OFF_Q + qb * L::Q_BYTES;
                    for (int pass = 0; pass < 2 && ok; ++pass) {
                        for (int t = tile_begin; t < tile_end; ++t) {
                            if (!wait_phase(BAR(K_FULL + ks), kph, ctl)) { ok = false; break; }
                            const uint32_t tb = pass == 0 ? (t1i & 1) : (t2i & 1);
                            const uint32_t tph = pass == 0 ? ((t1i >> 1) & 1) : ((t2i >> 1) & 1);
                            if (!wait_phase(BAR((pass == 0 ? T1_EMPTY : T2_EMPTY) + tb), tph ^ 1, ctl)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            const uint32_t kaddr = base + L::OFF_K + ks * L::TILE_BYTES;
                            const uint32_t d = tmem + (pass == 0 ? 0u : 256u) + tb * 128u;
#pragma unroll
                            for (int st = 0; st < KSTEPS; ++st) {
                                const uint32_t off = (st >> 2) * (kTileRows * 128) + (st & 3) * 32;
                                const uint64_t qd = sdesc_k_sw128(qaddr + off);
                                const uint64_t kd = sdesc_k_sw128(kaddr + off);
                                if (pass == 0) {
                                    if (FP8) mma_f8(d, qd, kd, idesc1, st > 0);
                                    else mma_f16(d, qd, kd, idesc1, st > 0);
                                } else {
                                    if (FP8) mma_f8(d, kd, qd, idesc2, st > 0);
                                    else mma_f16(d, kd, qd, idesc2, st > 0);
                                }
                            }
                            mma_commit(BAR((pass == 0 ? T1_FULL : T2_FULL) + tb));
                            mma_commit(BAR(K_EMPTY + ks));
                            if (pass == 0) ++t1i; else ++t2i;
                            if (++ks == kStages) { ks = 0; kph ^= 1; }
                        }
                    }
                    mma_commit(BAR(Q_EMPTY + qb));
                }
            }
            // drain: every MMA issued by this thread has completed
            mma_commit(BAR(DRAIN));
            wait_phase(BAR(DRAIN), 0, ctl);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int quad = warp & 3;
        const int row = quad * 32 + lane;                     // TMEM lane of this thread
        const uint32_t lane_off = (uint32_t)(quad * 32) << 16;
        for (int tl = 0; tl < mt; ++tl) acc_s[tl * kTileRows + row] = 0.f;
        uint32_t t1i = 0, t2i = 0;
        // Control flow here is identical for all 128 threads (named barriers);
        // after an abort every wait returns at once and the loop runs out.
        for (int hi = 0; hi < hpg; ++hi) {
            const int par = hi & 1;
            // ---- pass 1: online row statistics over this CTA's tiles
            float m = -INFINITY, l = 0.f;
            const bool warp_live = quad * 32 < T;
            for (int t = tile_begin; t < tile_end; ++t) {
                const uint32_t tb = t1i & 1;
                wait_phase(BAR(T1_FULL + tb), (t1i >> 1) & 1, ctl);
                tc_fence_after();
                float v[128];
                if (warp_live) {
                    const uint32_t ta = tmem + lane_off + tb * 128u;
                    tmem_ld32(ta + 0, v);
                    tmem_ld32(ta + 32, v + 32);
                    tmem_ld32(ta + 64, v + 64);
                    tmem_ld32(ta + 96, v + 96);
                    tmem_wait_ld();
                }
                tc_fence_before();
                mbar_arrive(BAR(T1_EMPTY + tb));
                ++t1i;
                if (warp_live) {
                    const int valid = N - t * kTileRows;
                    if (valid < kTileRows) {
#pragma unroll
                        for (int c = 0; c < 128; ++c)
                            if (c >= valid) v[c] = -INFINITY;
                    }
                    float mx0 = v[0], mx1 = v[1], mx2 = v[2], mx3 = v[3];
#pragma unroll
                    for (int c = 4; c < 128; c += 4) {
                        mx0 = fmaxf(mx0, v[c]);
                        mx1 = fmaxf(mx1, v[c + 1]);
                        mx2 = fmaxf(mx2, v[c + 2]);
                        mx3 = fmaxf(mx3, v[c + 3]);
                    }
                    const float m_new = fmaxf(m, fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)));
                    const float mc = m_new * cl;
                    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
                    for (int c = 0; c < 128; c += 4) {
                        s0 += ex2(fmaf(v[c], cl, -mc));
                        s1 += ex2(fmaf(v[c + 1], cl, -mc));
                        s2 += ex2(fmaf(v[c + 2], cl, -mc));
                        s3 += ex2(fmaf(v[c + 3], cl, -mc));
                    }
                    l = l * ex2((m - m_new) * cl) + ((s0 + s1) + (s2 + s3));
                    m = m_new;
                }
            }
            // ---- exchange (m, l) across the cluster
            stats_s[par * kMaxText + row] = make_float2(m, l);
            fence_acq_rel_cluster();
            named_bar_sync(1, 128);
            if (row == 0) {
                const uint32_t sb = BAR(STATS + par);
                for (uint32_t r = 0; r < csize; ++r) mbar_arrive_remote(mapa_shared(sb, r));
            }
            wait_phase_cluster(BAR(STATS + par), (hi >> 1) & 1, ctl);
            {
                const uint32_t my = base + L::OFF_STATS + (uint32_t)(par * kMaxText + row) * 8u;
                float M = -INFINITY;
                for (uint32_t r = 0; r < csize; ++r) M = fmaxf(M, ld_shared_cluster_f2(mapa_shared(my, r)).x);
                float Lsum = 0.f;
                for (uint32_t r = 0; r < csize; ++r) {
                    const float2 st = ld_shared_cluster_f2(mapa_shared(my, r));
                    if (st.y > 0.f) Lsum += st.y * ex2((st.x - M) * cl);
                }
                b2_s[row] = (row < T) ? fmaf(M, cl, __log2f(Lsum)) : INFINITY;
            }
            named_bar_sync(1, 128);
            // ---- pass 2: per-visual-token sums of probabilities
            for (int t = tile_begin; t < tile_end; ++t) {
                const uint32_t tb = t2i & 1;
                wait_phase(BAR(T2_FULL + tb), (t2i >> 1) & 1, ctl);
                tc_fence_after();
                float v[128];
                const uint32_t ta = tmem + lane_off + 256u + tb * 128u;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    if (k * 32 + 32 <= n2) tmem_ld32(ta + k * 32, v + k * 32);
                    else if (k * 32 + 16 <= n2) tmem_ld16(ta + k * 32, v + k * 32);
                }
                tmem_wait_ld();
                tc_fence_before();
                mbar_arrive(BAR(T2_EMPTY + tb));
                ++t2i;
                float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    if (k * 16 < n2) {
#pragma unroll
                        for (int e = 0; e < 16; e += 4) {
                            const float4 bb = *reinterpret_cast<const float4*>(b2_s + k * 16 + e);
                            a0 += ex2(fmaf(v[k * 16 + e], cl, -bb.x));
                            a1 += ex2(fmaf(v[k * 16 + e + 1], cl, -bb.y));
                            a2 += ex2(fmaf(v[k * 16 + e + 2], cl, -bb.z));
                            a3 += ex2(fmaf(v[k * 16 + e + 3], cl, -bb.w));
                        }
                    }
                }
                acc_s[(t - tile_begin) * kTileRows + row] += (a0 + a1) + (a2 + a3);
            }
            named_bar_sync(1, 128);
        }
        if (!*abort_flag) {
            const float denom = (float)p.hq * (float)T;
            for (int tl = 0; tl < mt; ++tl) {
                const int j = (tile_begin + tl) * kTileRows + row;
                if (j < N) {
                    const float a = acc_s[tl * kTileRows + row];
                    if (p.groups == 1) p.out[n0 + j] = a / denom;
                    else p.out[(int64_t)hg * p.total_vis + n0 + j] = a;
                }
            }
        }
        tc_fence_before();
    }

    // ---------------------------------------------------------------- teardown
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
    cluster_sync_all();  // peers are done reading this CTA's statistics
}

// scores[j] = (sum over head groups of partial[g][j]) / (Hq * T_b), fixed order
__global__ void fold_groups_kernel(const float* __restrict__ partials, int groups, int64_t total_vis,
                                   const int32_t* __restrict__ seq_off, const int32_t* __restrict__ text_off,
                                   int hq, float* __restrict__ scores)
{
    const int b = blockIdx.y;
    const int n0 = seq_off[b], N = seq_off[b + 1] - n0;
    const int T = text_off[b + 1] - text_off[b];
    const float denom = (float)hq * (float)T;
    for (int j = blockIdx.x * blockDim.x + threadIdx.x; j < N; j += gridDim.x * blockDim.x) {
        float s = 0.f;
        for (int g = 0; g < groups; ++g) s += partials[(int64_t)g * total_vis + n0 + j];
        scores[n0 + j] = s / denom;
    }
}

template <int ROW_BYTES, bool FP8>
cudaError_t launch_variant(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const ScoreLaunch& p,
                           const ScorePlan& plan, int batch, cudaStream_t stream)
{
    auto kern = score_tc_kernel<ROW_BYTES, FP8>;
    const int smem = SmemLayout<ROW_BYTES>::ALLOC;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    if (plan.cluster > 8) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(plan.cluster, plan.groups, batch);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = plan.cluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, tm_q, tm_k, p);
}

}  // namespace

bool score_shape_supported(int head_dim, bool fp8)
{
    if (fp8) return head_dim == 128;
    return head_dim == 64 || head_dim == 128;
}

size_t score_smem_bytes(int row_bytes)
{
    return row_bytes == 256 ? SmemLayout<256>::ALLOC : SmemLayout<128>::ALLOC;
}

ScorePlan plan_score(int batch, int max_tiles, int hq, int num_sms)
{
    ScorePlan pl{1, 1, 1};
    if (max_tiles <= 0) return pl;
    int tpc = (max_tiles + 7) / 8;
    int c = (max_tiles + tpc - 1) / tpc;
    if (tpc > kMaxTilesPerCta) {
        tpc = (max_tiles + kMaxCluster - 1) / kMaxCluster;
        c = (max_tiles + tpc - 1) / tpc;
    }
    pl.cluster = c;
    pl.tiles_per_cta = tpc;
    int groups = hq;
    for (int g = 1; g <= hq; ++g) {
        if (hq % g) continue;
        if ((long long)batch * c * g >= num_sms) { groups = g; break; }
    }
    pl.groups = groups;
    return pl;
}

cudaError_t launch_score(const CUtensorMap& tm_q, const CUtensorMap& tm_k, const ScoreLaunch& p,
                         const ScorePlan& plan, int batch, int row_bytes, bool fp8, float* partials,
                         float* scores, int max_n, cudaStream_t stream)
{
    ScoreLaunch q = p;
    q.groups = plan.groups;
    q.heads_per_group = p.hq / plan.groups;
    q.out = plan.groups == 1 ? scores : partials;
    cudaError_t e;
    if (fp8) e = launch_variant<128, true>(tm_q, tm_k, q, plan, batch, stream);
    else if (row_bytes == 256) e = launch_variant<256, false>(tm_q, tm_k, q, plan, batch, stream);
    else e = launch_variant<128, false>(tm_q, tm_k, q, plan, batch, stream);
    if (e != cudaSuccess || plan.groups == 1) return e;
    const int threads = 256;
    const int gx = (max_n + threads - 1) / threads;
    fold_groups_kernel<<<dim3(gx > 0 ? gx : 1, batch), threads, 0, stream>>>(partials, plan.groups, p.total_vis,
                                                                              p.seq_off, p.text_off, p.hq, scores);
    return cudaGetLastError();
}

}  // namespace lvs
