// Gather of the kept rows into the compacted sequence (Design section: the
// token selection shortens the LLM input; the kept rows' K/V feed the KV cache).
//
// dst[t][r] = src[t][kept_idx[r]] for every gathered tensor t, byte for byte.
// One warp moves one kept row of every tensor: the index is read once, each
// lane copies 16-byte vectors with streaming (evict-first) loads and stores,
// up to eight vectors in flight per lane. Rows whose size or pointers are not
// 16-byte aligned go through the byte-wise kernel. Indices outside
// [0, src_rows) are skipped and flagged in the error word.

#include "internal.h"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kGatherThreads = 256;

__global__ void __launch_bounds__(kGatherThreads)
    compact_vec16_kernel(int64_t total_kept, const int32_t* __restrict__ kept_idx, int64_t src_rows,
                         const GatherArgs g, int32_t* err)
{
    griddep_wait();
    griddep_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int64_t w = ((int64_t)blockIdx.x * kGatherThreads + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * kGatherThreads) >> 5;
    for (int64_t r = w; r < total_kept; r += nw) {
        const int32_t idx = __ldg(kept_idx + r);
        if (idx < 0 || (int64_t)idx >= src_rows) {
            if (lane == 0) atomicOr(err, kErrBounds);
            continue;
        }
        for (int t = 0; t < g.n; ++t) {
            const int64_t rb = g.row_bytes[t];
            const int4* __restrict__ s = reinterpret_cast<const int4*>(g.src[t] + (int64_t)idx * rb);
            int4* __restrict__ d = reinterpret_cast<int4*>(g.dst[t] + r * rb);
            const int64_t n16 = rb >> 4;
            // up to 8 vectors per lane in flight (a 4 KB row in one round trip)
            for (int64_t c = lane; c < n16; c += 256) {
                int4 a[8];
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (c + 32 * u < n16) a[u] = __ldcs(s + c + 32 * u);
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (c + 32 * u < n16) __stcs(d + c + 32 * u, a[u]);
            }
        }
    }
}

__global__ void __launch_bounds__(kGatherThreads)
    compact_bytes_kernel(int64_t total_kept, const int32_t* __restrict__ kept_idx, int64_t src_rows,
                         const GatherArgs g, int32_t* err)
{
    griddep_wait();
    griddep_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int64_t w = ((int64_t)blockIdx.x * kGatherThreads + threadIdx.x) >> 5;
    const int64_t nw = ((int64_t)gridDim.x * kGatherThreads) >> 5;
    for (int64_t r = w; r < total_kept; r += nw) {
        const int32_t idx = kept_idx[r];
        if (idx < 0 || (int64_t)idx >= src_rows) {
            if (lane == 0) atomicOr(err, kErrBounds);
            continue;
        }
        for (int t = 0; t < g.n; ++t) {
            const int64_t rb = g.row_bytes[t];
            const uint8_t* s = g.src[t] + (int64_t)idx * rb;
            uint8_t* d = g.dst[t] + r * rb;
            for (int64_t c = lane; c < rb; c += 32) d[c] = s[c];
        }
    }
}

}  // namespace

cudaError_t launch_compact(int64_t total_kept, const int32_t* kept_idx, int64_t src_rows, const GatherArgs& g,
                           bool vec16, int32_t* err, int num_sms, cudaStream_t stream)
{
    if (total_kept <= 0) return cudaSuccess;
    const int64_t warps_per_block = kGatherThreads / 32;
    int64_t blocks = (total_kept + warps_per_block - 1) / warps_per_block;
    const int64_t cap = (int64_t)num_sms * 8;  // 2048 threads per SM
    if (blocks > cap) blocks = cap;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks, 1, 1);
    cfg.blockDim = dim3(kGatherThreads, 1, 1);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1] = {pdl_attribute()};
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, vec16 ? compact_vec16_kernel : compact_bytes_kernel, total_kept, kept_idx,
                              src_rows, g, err);
}

}  // namespace lvs
