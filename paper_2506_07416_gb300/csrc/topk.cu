// Per-request top-k of the visual-token scores (Results section, "Visual Token
// Compression": a ratio r of the visual tokens is kept; Table 1 token counts).
//
// One CTA per request (512 threads; the register kernel below takes 1024 on
// requests of 2049 to 8192 tokens). Scores become order-preserving 32-bit keys (NaN -> 0,
// the lowest key; -0 and +0 the same key), an MSB-first radix select (4 passes
// of 8 bits, warp-aggregated shared-memory histograms) finds the k-th largest
// key K* and how many keys equal to K* must be taken, then one pass over the
// tokens in index order keeps every key > K* and the first keys == K* (lower
// index wins a tie). Two block-wide exclusive scans give each thread its place
// in the output, so the kept indices come out ascending, as global rows.
// k_b = keep_k[b], or floor((double)ratio * N_b) clamped to [0, N_b];
// out_offsets[b+1] = sum of k over requests 0..b.

#include <math.h>

#include "internal.h"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kTopkThreads = 512;      // the shared-memory kernel; register kernel up to 2048 tokens
constexpr int kTopkWideThreads = 1024; // register kernel, 2049 .. 8192 tokens
constexpr int kTopkWarps = kTopkThreads / 32;

__device__ __forceinline__ uint32_t order_key(float f)
{
    uint32_t u = __float_as_uint(f);
    if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 0u;  // NaN ranks below everything
    if (u == 0x80000000u) u = 0u;                     // -0 equals +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ int keep_count(const int32_t* seq_off, const int32_t* keep_k, float ratio, int b)
{
    const int n = seq_off[b + 1] - seq_off[b];
    if (keep_k) return keep_k[b];
    double kd = floor((double)ratio * (double)n);
    kd = kd < 0.0 ? 0.0 : (kd > (double)n ? (double)n : kd);
    return (int)kd;
}

// exclusive scan over the block; `total` receives the block sum
__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_sums, int& total)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = lane < kTopkWarps ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        if (lane < kTopkWarps) warp_sums[lane] = w;  // inclusive
    }
    __syncthreads();
    const int before = (warp > 0 ? warp_sums[warp - 1] : 0) + x - v;
    total = warp_sums[kTopkWarps - 1];
    __syncthreads();
    return before;
}

__global__ void __launch_bounds__(kTopkThreads)
    topk_kernel(const float* __restrict__ scores, const int32_t* __restrict__ seq_off,
                const int32_t* __restrict__ keep_k, float ratio, int32_t* __restrict__ kept_idx,
                int32_t* __restrict__ out_off, int smem_keys)
{
    extern __shared__ uint32_t keys_s[];
    __shared__ uint32_t hist[257];
    __shared__ int warp_sums[kTopkWarps];
    __shared__ uint32_t s_digit, s_above;
    __shared__ long long s_base;

    const int b = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    griddep_wait();
    griddep_launch_dependents();
    const int n0 = seq_off[b];
    const int N = seq_off[b + 1] - n0;

    // output base = sum of k over earlier requests
    long long part = 0;
    for (int bb = tid; bb < b; bb += kTopkThreads) part += keep_count(seq_off, keep_k, ratio, bb);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_down_sync(0xffffffffu, part, o);
    if (tid == 0) s_base = 0;
    __syncthreads();
    if (lane == 0 && part) atomicAdd(reinterpret_cast<unsigned long long*>(&s_base), (unsigned long long)part);
    __syncthreads();
    const long long out_base = s_base;
    const int k = keep_count(seq_off, keep_k, ratio, b);
    if (tid == 0) {
        out_off[b + 1] = (int32_t)(out_base + k);
        if (b == 0) out_off[0] = 0;
    }
    if (k <= 0 || N <= 0) return;
    int32_t* dst = kept_idx + out_base;
    if (k >= N) {
        for (int j = tid; j < N; j += kTopkThreads) dst[j] = n0 + j;
        return;
    }

    const bool in_smem = N <= smem_keys;
    if (in_smem) {
        for (int j = tid; j < N; j += kTopkThreads) keys_s[j] = order_key(scores[n0 + j]);
        __syncthreads();
    }
    auto key_at = [&](int j) -> uint32_t { return in_smem ? keys_s[j] : order_key(scores[n0 + j]); };

    // ---- radix select of the k-th largest key
    uint32_t prefix = 0u, mask = 0u;
    int remaining = k;
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int i = tid; i < 257; i += kTopkThreads) hist[i] = 0u;
        __syncthreads();
        for (int base = warp * 32; base < N; base += kTopkThreads) {
            const int j = base + lane;
            uint32_t bin = 256u;
            if (j < N) {
                const uint32_t u = key_at(j);
                if ((u & mask) == prefix) bin = (u >> shift) & 0xFFu;
            }
            const uint32_t peers = __match_any_sync(0xffffffffu, bin);
            if (lane == __ffs(peers) - 1) atomicAdd(&hist[bin], (uint32_t)__popc(peers));
        }
        __syncthreads();
        if (warp == 0) {
            uint32_t c[8], tot = 0;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                c[e] = hist[lane * 8 + e];
                tot += c[e];
            }
            uint32_t suf = tot;  // sum over lanes >= this lane
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_down_sync(0xffffffffu, suf, o);
                if (lane + o < 32) suf += y;
            }
            uint32_t above = suf - tot;
            if (above < (uint32_t)remaining && (uint32_t)remaining <= suf) {
#pragma unroll
                for (int e = 7; e >= 0; --e) {
                    if (above + c[e] >= (uint32_t)remaining) {
                        s_digit = (uint32_t)(lane * 8 + e);
                        s_above = above;
                        break;
                    }
                    above += c[e];
                }
            }
        }
        __syncthreads();
        prefix |= s_digit << shift;
        mask |= 0xFFu << shift;
        remaining -= (int)s_above;
        __syncthreads();
    }

    // ---- keep keys > prefix and the first `remaining` keys == prefix (index order)
    const int ipt = (N + kTopkThreads - 1) / kTopkThreads;
    const int j0 = min(N, tid * ipt), j1 = min(N, j0 + ipt);
    int n_eq = 0;
    for (int j = j0; j < j1; ++j) n_eq += key_at(j) == prefix;
    int total;
    const int eq_before = block_exclusive_scan(n_eq, warp_sums, total);
    int n_keep = 0;
    {
        int e = eq_before;
        for (int j = j0; j < j1; ++j) {
            const uint32_t u = key_at(j);
            if (u > prefix) ++n_keep;
            else if (u == prefix) n_keep += (e++ < remaining);
        }
    }
    int pos = block_exclusive_scan(n_keep, warp_sums, total);
    {
        int e = eq_before;
        for (int j = j0; j < j1; ++j) {
            const uint32_t u = key_at(j);
            const bool keep = u > prefix || (u == prefix && e++ < remaining);
            if (keep) dst[pos++] = n0 + j;
        }
    }
}


// The k largest keys of one request (0 < k < N), held KPT per thread by one CTA
// of NT threads (token j = e * NT + tid), with the request's
// smallest and largest key lo_k / hi_k. Calls emit(pos, j) once per kept token,
// pos = its place among the kept tokens in index order (0 .. k-1). hist and cnt
// are shared memory; hist[0] and hist[1] must be zero on entry.
template <int KPT, int NT, class Emit>
__device__ __forceinline__ void select_kept(const uint32_t (&key)[KPT], int N, int k, uint32_t lo_k, uint32_t hi_k,
                                            uint32_t (*hist)[256], int (*cnt)[NT / 32], Emit emit)
{
    constexpr int NW = NT / 32;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    // ---- radix select below the common high bits
    const uint32_t diff = lo_k ^ hi_k;
    uint32_t mask = diff ? ~((2u << (31 - __clz(diff))) - 1u) : 0xFFFFFFFFu;
    uint32_t prefix = lo_k & mask;
    int remaining = k;                // keys still to take from the keys matching prefix under mask
    int n_eq = N;                     // keys matching prefix under mask
    int top = diff ? 31 - __clz(diff) : -1;
    int pass = 0;
    while (top >= 0 && n_eq != remaining) {
        const int lo = top >= 7 ? top - 7 : 0;
        const uint32_t dmask = (2u << (top - lo)) - 1u;
        uint32_t* h = hist[pass % 3];
#pragma unroll
        for (int e = 0; e < KPT; ++e) {
            if (e * NT + tid < N && (key[e] & mask) == prefix) atomicAdd(&h[(key[e] >> lo) & dmask], 1u);
        }
        if (tid < 256) hist[(pass + 1) % 3][tid] = 0u;
        __syncthreads();
        // every warp: the digit d with (count above d) < remaining <= (count above d) + count(d)
        uint32_t c[8], tot = 0;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            c[e] = h[lane * 8 + e];
            tot += c[e];
        }
        uint32_t suf = tot;  // sum over lanes >= this lane
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_down_sync(0xffffffffu, suf, o);
            if (lane + o < 32) suf += y;
        }
        uint32_t above = suf - tot, digit = 0, cnt_d = 0, above_d = 0;
        const bool mine = above < (uint32_t)remaining && (uint32_t)remaining <= suf;
        if (mine) {
#pragma unroll
            for (int e = 7; e >= 0; --e) {
                if (cnt_d == 0 && above + c[e] >= (uint32_t)remaining) {
                    digit = (uint32_t)(lane * 8 + e);
                    cnt_d = c[e];
                    above_d = above;
                }
                above += c[e];
            }
        }
        const int src = __ffs(__ballot_sync(0xffffffffu, mine)) - 1;
        digit = __shfl_sync(0xffffffffu, digit, src);
        cnt_d = __shfl_sync(0xffffffffu, cnt_d, src);
        above_d = __shfl_sync(0xffffffffu, above_d, src);
        prefix |= digit << lo;
        mask |= dmask << lo;
        remaining -= (int)above_d;
        n_eq = (int)cnt_d;
        top = lo - 1;
        ++pass;
    }

    // ---- keep keys above prefix, and the first `remaining` keys equal to it in index order
    uint32_t gt = 0, eq = 0;
#pragma unroll
    for (int e = 0; e < KPT; ++e) {
        const bool valid = e * NT + tid < N;
        const uint32_t m = key[e] & mask;
        gt |= (uint32_t)(valid && m > prefix) << e;
        eq |= (uint32_t)(valid && m == prefix) << e;
    }
    const uint32_t lt_mask = (1u << lane) - 1u;
    uint32_t keep = gt | eq;
    if (n_eq != remaining) {
        // rank of each equal key among the equal keys (index order)
#pragma unroll
        for (int e = 0; e < KPT; ++e) {
            const uint32_t bal = __ballot_sync(0xffffffffu, (eq >> e) & 1u);
            if (lane == 0) cnt[e][warp] = __popc(bal);
        }
        __syncthreads();
        int run = 0;
        keep = gt;
#pragma unroll
        for (int e = 0; e < KPT; ++e) {
            int v = lane < NW ? cnt[e][lane] : 0;
#pragma unroll
            for (int o = 1; o < NW; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, v, o);
                if (lane >= o) v += y;
            }
            const int before_w = __shfl_sync(0xffffffffu, v, (warp + NW - 1) % NW);
            const int tot_e = __shfl_sync(0xffffffffu, v, NW - 1);
            const uint32_t bal = __ballot_sync(0xffffffffu, (eq >> e) & 1u);
            const int rank = run + (warp ? before_w : 0) + __popc(bal & lt_mask);
            if (((eq >> e) & 1u) && rank < remaining) keep |= 1u << e;
            run += tot_e;
        }
        __syncthreads();  // cnt is reused below
    }
#pragma unroll
    for (int e = 0; e < KPT; ++e) {
        const uint32_t bal = __ballot_sync(0xffffffffu, (keep >> e) & 1u);
        if (lane == 0) cnt[e][warp] = __popc(bal);
    }
    __syncthreads();
    int run = 0;
#pragma unroll
    for (int e = 0; e < KPT; ++e) {
        int v = lane < NW ? cnt[e][lane] : 0;
#pragma unroll
        for (int o = 1; o < NW; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, v, o);
            if (lane >= o) v += y;
        }
        const int before_w = __shfl_sync(0xffffffffu, v, (warp + NW - 1) % NW);
        const int tot_e = __shfl_sync(0xffffffffu, v, NW - 1);
        const uint32_t bal = __ballot_sync(0xffffffffu, (keep >> e) & 1u);
        if ((keep >> e) & 1u) emit(run + (warp ? before_w : 0) + __popc(bal & lt_mask), e * NT + tid);
        run += tot_e;
    }
}

// ---------------------------------------------------------------------------
// Register-resident variant for requests of at most NT * KPT tokens.
// Thread t holds the keys of tokens j = e * NT + t (e < KPT), so the
// loads are coalesced and "round e, warp w, lane l" is index order. The radix
// select starts below the bits that every key of the request shares (one
// min/max reduction finds them) and stops as soon as the bin holding the k-th
// key is taken whole. Every warp finds the selected digit from the shared
// histogram by itself, so a pass costs one barrier; histograms rotate over
// three buffers so a buffer is cleared two passes after it was last read.
// Output positions come from per-(round, warp) ballot counts.

template <int KPT, bool DEFER, int NT>
__global__ void __launch_bounds__(NT)
    topk_reg_kernel(float* __restrict__ scores, const int32_t* __restrict__ seq_off,
                    const int32_t* __restrict__ keep_k, float ratio, int32_t* __restrict__ kept_idx,
                    int32_t* __restrict__ out_off, const __grid_constant__ TopkShape sh)
{
    constexpr int NW = NT / 32;
    __shared__ uint32_t hist[3][256];
    __shared__ uint32_t wmin[NW], wmax[NW];
    __shared__ int cnt[KPT][NW];
    __shared__ long long s_base;

    const int b = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    // sizes in the parameters (read before the wait: they are not produced on
    // the device), so the scores are the kernel's first global loads
    const bool by_value = sh.n > 0;
    int n0 = 0, N = 0, k_v = 0, out0_v = 0;
    if (by_value) {
        n0 = sh.n0[b];
        N = sh.len[b];
        k_v = sh.k[b];
        out0_v = sh.out0[b];
    }
    griddep_wait();
    griddep_launch_dependents();
    if (!by_value) {
        n0 = seq_off[b];
        N = seq_off[b + 1] - n0;
    }

    uint32_t key[KPT];
    if constexpr (DEFER) {  // launched only with the sizes by value and the partials
        // the score kernel's last step: the head-group partials, added in group
        // order and divided once, as its own fold would
        const float den = sh.denom[b];
        float sum[KPT];
#pragma unroll
        for (int e = 0; e < KPT; ++e) sum[e] = 0.f;
        // loads in flight per key, within the registers (at most 64 registers a thread at 1024 threads)
        constexpr int QG = NT >= 1024 ? 16 / KPT : (KPT <= 4 ? 16 : (KPT <= 8 ? 4 : 2));
        for (int g0 = 0; g0 < sh.groups; g0 += QG) {
            float v[KPT][QG];
#pragma unroll
            for (int e = 0; e < KPT; ++e) {
                const int j = e * NT + tid;
#pragma unroll
                for (int q = 0; q < QG; ++q)
                    v[e][q] = (j < N && g0 + q < sh.groups)
                                  ? __ldcg(sh.partials + (int64_t)(g0 + q) * sh.total_vis + n0 + j) : 0.f;
            }
#pragma unroll
            for (int e = 0; e < KPT; ++e)
#pragma unroll
                for (int q = 0; q < QG; ++q)
                    if (g0 + q < sh.groups) sum[e] += v[e][q];
        }
#pragma unroll
        for (int e = 0; e < KPT; ++e) {
            const int j = e * NT + tid;
            const float sc = sum[e] / den;
            if (j < N) scores[n0 + j] = sc;
            key[e] = j < N ? order_key(sc) : 0u;
        }
    } else {
#pragma unroll
        for (int e = 0; e < KPT; ++e) {
            const int j = e * NT + tid;
            key[e] = j < N ? order_key(__ldcg(scores + n0 + j)) : 0u;
        }
    }

    // output base = sum of k over earlier requests
    long long part = 0;
    if (!by_value)
        for (int bb = tid; bb < b; bb += NT) part += keep_count(seq_off, keep_k, ratio, bb);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_down_sync(0xffffffffu, part, o);
    if (tid == 0) s_base = by_value ? (long long)out0_v : 0;
    __syncthreads();
    if (lane == 0 && part) atomicAdd(reinterpret_cast<unsigned long long*>(&s_base), (unsigned long long)part);
    const int k = by_value ? k_v : keep_count(seq_off, keep_k, ratio, b);

    // key range of the request (padding slots take part only through valid keys)
    uint32_t lo_k = 0xFFFFFFFFu, hi_k = 0u;
#pragma unroll
    for (int e = 0; e < KPT; ++e) {
        if (e * NT + tid < N) {
            lo_k = min(lo_k, key[e]);
            hi_k = max(hi_k, key[e]);
        }
    }
    lo_k = __reduce_min_sync(0xffffffffu, lo_k);
    hi_k = __reduce_max_sync(0xffffffffu, hi_k);
    if (lane == 0) {
        wmin[warp] = lo_k;
        wmax[warp] = hi_k;
    }
    for (int i = tid; i < 2 * 256; i += NT) (&hist[0][0])[i] = 0u;
    __syncthreads();
    const long long out_base = s_base;
    if (tid == 0) {
        out_off[b + 1] = (int32_t)(out_base + k);
        if (b == 0) out_off[0] = 0;
    }
    if (k <= 0 || N <= 0) return;
    int32_t* dst = kept_idx + out_base;
    if (k >= N) {
        for (int j = tid; j < N; j += NT) dst[j] = n0 + j;
        return;
    }
    lo_k = __reduce_min_sync(0xffffffffu, lane < NW ? wmin[lane] : 0xFFFFFFFFu);
    hi_k = __reduce_max_sync(0xffffffffu, lane < NW ? wmax[lane] : 0u);
    select_kept<KPT, NT>(key, N, k, lo_k, hi_k, hist, cnt, [&](int pos, int j) { dst[pos] = n0 + j; });
}

}  // namespace

constexpr int kTopkSmemKeys = 40 * 1024;  // keys staged in shared memory (160 KB)

template <typename... Args>
cudaError_t launch_pdl(void (*kern)(Args...), unsigned grid, unsigned block, size_t smem, cudaStream_t stream,
                       Args... args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid, 1, 1);
    cfg.blockDim = dim3(block, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1] = {pdl_attribute()};
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, args...);
}

cudaError_t launch_topk(int batch, float* scores, const int32_t* seq_off, const int32_t* keep_k,
                        float keep_ratio, int32_t* kept_idx, int32_t* out_off, int max_n, const TopkShape& shape,
                        cudaStream_t stream)
{
    if (batch <= 0) return cudaSuccess;
    // registers only: 512 threads up to 2048 tokens, 1024 threads up to 8192
    // (measured on GB300: the wider CTA halves each thread's chain of loads,
    // passes and ranks on long requests, and costs more than it saves on short ones)
    const bool defer = shape.partials != nullptr && shape.n == batch;
    if (max_n <= 4 * kTopkThreads) {
        auto kern = defer ? (max_n <= 2 * kTopkThreads ? topk_reg_kernel<2, true, kTopkThreads>
                                                       : topk_reg_kernel<4, true, kTopkThreads>)
                          : (max_n <= 2 * kTopkThreads ? topk_reg_kernel<2, false, kTopkThreads>
                                                       : topk_reg_kernel<4, false, kTopkThreads>);
        return launch_pdl(kern, (unsigned)batch, kTopkThreads, 0, stream, scores, seq_off, keep_k, keep_ratio,
                          kept_idx, out_off, shape);
    }
    if (max_n <= 8 * kTopkWideThreads) {
        auto kern = defer ? (max_n <= 4 * kTopkWideThreads ? topk_reg_kernel<4, true, kTopkWideThreads>
                                                           : topk_reg_kernel<8, true, kTopkWideThreads>)
                          : (max_n <= 4 * kTopkWideThreads ? topk_reg_kernel<4, false, kTopkWideThreads>
                                                           : topk_reg_kernel<8, false, kTopkWideThreads>);
        return launch_pdl(kern, (unsigned)batch, kTopkWideThreads, 0, stream, scores, seq_off, keep_k, keep_ratio,
                          kept_idx, out_off, shape);
    }
    const int keys = max_n < kTopkSmemKeys ? max_n : kTopkSmemKeys;
    const size_t smem = (size_t)keys * 4;
    cudaError_t e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    return launch_pdl(topk_kernel, (unsigned)batch, kTopkThreads, smem, stream, (const float*)scores, seq_off, keep_k,
                      keep_ratio, kept_idx, out_off, keys);
}

}  // namespace lvs
