// Patch-selection gating (Design section, Patch Selection Module): the final
// score of camera view v of request b is a weighted sum of its lexical-mapping
// score and the module's logit, and the views scoring above a threshold go on
// to the vision encoder. This decides N_b, the visual tokens the selection path
// scores.
//     s[b][v] = w_lex * lexical[b][v] + w_logit * logit[b][v]     (fp32, no contraction)
//     selected  <=>  s[b][v] > threshold
// When fewer than min_views views pass, the min_views best views are taken
// (score descending, lower view index first, NaN lowest).
// Outputs: view_mask [B, V] (0/1), view_offsets [B+1] and selected_views (view
// indices, ascending per request), seq_offsets [B+1] (prefix of the selected
// views' token counts).
//
// One CTA of 1024 threads walks the batch in chunks of 1024 requests, one
// request per thread; two block-wide scans (views, tokens) place each
// request's outputs, and the chunk totals carry into the next chunk.

#include "internal.h"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kViewsThreads = 1024;
constexpr int kViewsWarps = kViewsThreads / 32;

// (a, ia) strictly before (b, ib) under (score desc, index asc), NaN lowest
__device__ __forceinline__ bool view_before(float a, int ia, float b, int ib)
{
    const bool an = a != a, bn = b != b;
    if (an != bn) return bn;
    if (!an && a != b) return a > b;
    return ia < ib;
}

// inclusive scan over the block of two values; returns the exclusive prefix of
// each and the block totals
__device__ __forceinline__ void block_scan2(int x, int y, int* sx, int* sy, int& ex, int& ey, int& tx, int& ty)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int ix = x, iy = y;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int ux = __shfl_up_sync(0xffffffffu, ix, o);
        const int uy = __shfl_up_sync(0xffffffffu, iy, o);
        if (lane >= o) {
            ix += ux;
            iy += uy;
        }
    }
    if (lane == 31) {
        sx[warp] = ix;
        sy[warp] = iy;
    }
    __syncthreads();
    if (warp == 0) {
        int wx = sx[lane], wy = sy[lane];
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int ux = __shfl_up_sync(0xffffffffu, wx, o);
            const int uy = __shfl_up_sync(0xffffffffu, wy, o);
            if (lane >= o) {
                wx += ux;
                wy += uy;
            }
        }
        sx[lane] = wx;
        sy[lane] = wy;
    }
    __syncthreads();
    ex = (warp > 0 ? sx[warp - 1] : 0) + ix - x;
    ey = (warp > 0 ? sy[warp - 1] : 0) + iy - y;
    tx = sx[kViewsWarps - 1];
    ty = sy[kViewsWarps - 1];
    __syncthreads();  // sx / sy are reused by the next chunk
}

__global__ void __launch_bounds__(kViewsThreads) views_kernel(const ViewsArgs a)
{
    __shared__ int sx[kViewsWarps], sy[kViewsWarps];
    griddep_wait();
    griddep_launch_dependents();
    const int V = a.num_views;
    int carry_v = 0, carry_t = 0;
    if (threadIdx.x == 0) {
        a.view_offsets[0] = 0;
        a.seq_offsets[0] = 0;
    }
    for (int base = 0; base < a.batch; base += kViewsThreads) {
        const int b = base + (int)threadIdx.x;
        uint64_t sel = 0;
        int nv = 0, nt = 0;
        if (b < a.batch) {
            float s[kMaxViews];
            int pass = 0;
            for (int v = 0; v < V; ++v) {
                const int64_t i = (int64_t)b * V + v;
                s[v] = __fadd_rn(__fmul_rn(a.w_lex, a.lexical[i]), __fmul_rn(a.w_logit, a.logits[i]));
                if (s[v] > a.threshold) {
                    sel |= 1ull << v;
                    ++pass;
                }
            }
            if (pass < a.min_views) {
                sel = 0;
                for (int v = 0; v < V; ++v) {
                    int rank = 0;
                    for (int u = 0; u < V; ++u) rank += (u != v && view_before(s[u], u, s[v], v)) ? 1 : 0;
                    if (rank < a.min_views) sel |= 1ull << v;
                }
            }
            for (int v = 0; v < V; ++v) {
                const bool on = (sel >> v) & 1ull;
                a.view_mask[(int64_t)b * V + v] = on ? 1 : 0;
                if (on) {
                    ++nv;
                    nt += a.tokens_per_view[v];
                }
            }
        }
        int ev, et, tv, tt;
        block_scan2(nv, nt, sx, sy, ev, et, tv, tt);
        if (b < a.batch) {
            int pos = carry_v + ev;
            for (int v = 0; v < V; ++v)
                if ((sel >> v) & 1ull) a.selected_views[pos++] = v;
            a.view_offsets[b + 1] = carry_v + ev + nv;
            a.seq_offsets[b + 1] = carry_t + et + nt;
        }
        carry_v += tv;
        carry_t += tt;
    }
}

}  // namespace

cudaError_t launch_views(const ViewsArgs& a, cudaStream_t stream)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(1, 1, 1);
    cfg.blockDim = dim3(kViewsThreads, 1, 1);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1] = {pdl_attribute()};
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, views_kernel, a);
}

}  // namespace lvs
