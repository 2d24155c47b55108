// Prefill sequence splice: the LLM input after token selection (Design
// section: the selection module shortens the sequence the LLM prefills).
//
// Request b's output is its S_b system rows, then its k_b kept visual rows
// (kept_idx: global visual-row indices, ascending within the request), then
// its T_b text rows, each copied byte for byte. Position ids are the rows'
// positions in the unpruned sequence [system; all N_b visual; text]: system
// row i -> i, kept visual row with local index j -> S_b + j, text row t ->
// S_b + N_b + t, so the kept tokens keep their original (rotary) positions.
//   out_offsets[b] = sys_offsets[b] + kept_offsets[b] + text_offsets[b]
//
// Grid (batch, row chunks): a warp copies one output row with 16-byte vectors
// (streaming hints, up to eight in flight per lane; byte-wise when the row
// size or a pointer is not 16-byte aligned) and its lane 0 writes the
// position id. A kept index outside its request's rows is skipped and flagged
// in the error word.

#include "internal.h"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kSpliceThreads = 256;
constexpr int kSpliceRowsPerCta = 32;  // 8 warps x 4 rows

template <bool VEC>
__global__ void __launch_bounds__(kSpliceThreads) splice_kernel(const SpliceArgs a)
{
    griddep_wait();
    griddep_launch_dependents();
    const int b = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int s0 = a.sys_off[b], S = a.sys_off[b + 1] - s0;
    const int v0 = a.seq_off[b], N = a.seq_off[b + 1] - v0;
    const int k0 = a.kept_off[b], K = a.kept_off[b + 1] - k0;
    const int t0 = a.text_off[b], T = a.text_off[b + 1] - t0;
    const int64_t o0 = (int64_t)s0 + k0 + t0;
    const int L = S + K + T;
    if (blockIdx.y == 0 && threadIdx.x == 0) {
        a.out_off[b] = (int32_t)o0;
        if (b == (int)gridDim.x - 1) a.out_off[b + 1] = (int32_t)(o0 + L);
    }
    const int64_t rb = a.row_bytes;
    for (int r = blockIdx.y * (kSpliceThreads / 32) + warp; r < L; r += gridDim.y * (kSpliceThreads / 32)) {
        const uint8_t* src;
        int32_t pos;
        if (r < S) {
            src = a.sys + (int64_t)(s0 + r) * rb;
            pos = r;
        } else if (r < S + K) {
            const int g = a.kept_idx[k0 + r - S];
            if (g < v0 || g >= v0 + N) {  // uniform over the warp
                if (lane == 0) atomicOr(a.err, kErrBounds);
                continue;
            }
            src = a.vis + (int64_t)g * rb;
            pos = S + (g - v0);
        } else {
            const int t = r - S - K;
            src = a.txt + (int64_t)(t0 + t) * rb;
            pos = S + N + t;
        }
        uint8_t* dst = a.out + (o0 + r) * rb;
        if (VEC) {
            const int4* __restrict__ s = reinterpret_cast<const int4*>(src);
            int4* __restrict__ d = reinterpret_cast<int4*>(dst);
            const int64_t n16 = rb >> 4;
            for (int64_t c = lane; c < n16; c += 256) {
                int4 v[8];
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (c + 32 * u < n16) v[u] = __ldcs(s + c + 32 * u);
#pragma unroll
                for (int u = 0; u < 8; ++u)
                    if (c + 32 * u < n16) __stcs(d + c + 32 * u, v[u]);
            }
        } else {
            for (int64_t c = lane; c < rb; c += 32) dst[c] = src[c];
        }
        if (lane == 0) a.pos[o0 + r] = pos;
    }
}

}  // namespace

cudaError_t launch_splice(const SpliceArgs& a, int max_rows, bool vec16, cudaStream_t stream)
{
    if (a.batch <= 0) return cudaSuccess;
    int chunks = (max_rows + kSpliceRowsPerCta - 1) / kSpliceRowsPerCta;
    if (chunks < 1) chunks = 1;
    if (chunks > 65535) chunks = 65535;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)a.batch, (unsigned)chunks, 1);
    cfg.blockDim = dim3(kSpliceThreads, 1, 1);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1] = {pdl_attribute()};
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, vec16 ? splice_kernel<true> : splice_kernel<false>, a);
}

}  // namespace lvs
