// Softmax-normaliser terms of the keys that are not visual tokens, for the
// score variant whose softmax runs over the full causal key set of the first
// decoder layer (Design section, Token Selection Module: the first decoder
// layer's self-attention; the prompt is [system; image; text] under the
// LLM's causal mask).
//
// For request b, query head h and text query i (global text row t), with
// g = h / G and c = scale * log2(e) (the score kernels' logit unit):
//     e[t][h] = log2( sum_j 2^(c * q[t,h,:] . k_j[g,:]) )
// over the S_b system keys and the text keys t' <= t of the request. The score
// kernels fold e into their visual-key statistic b (same unit) as
// log2(2^b + 2^e) before they form probabilities, so each probability is
// normalised over [system; visual; causal text] while only the visual
// columns are summed into the scores.
//
// One CTA of 128 threads per (request, query head). The request's query rows
// (at most 128) are A of a tcgen05 contraction with M = 128; up to 256 keys
// (system rows, then text rows) are B; D[128 x N] = Q K^T lands in TMEM and
// thread r (TMEM lane r) reduces query row r over its causal prefix of
// S_b + i + 1 keys. Both operands are staged by 16-byte cp.async copies into
// the 128-byte-swizzled K-major layout the tensor core reads, padding rows
// zero-filled. More than 256 keys (long texts in last-token mode) loop over
// key tiles. Requests without visual tokens are skipped.

#include <math.h>

#include "internal.h"
#include "pipe.cuh"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kCtxThreads = 128;
constexpr int kCtxQRows = 128;   // MMA M: query rows
constexpr int kCtxKeys = 256;    // MMA N limit: keys per tile

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, uint32_t src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all()
{
    asm volatile("cp.async.commit_group;" ::: "memory");
    asm volatile("cp.async.wait_group 0;" ::: "memory");
}

// Byte offset of 16-byte piece u of row r in a K-major tile of `rows` rows
// stored as 128-byte swizzled blocks along d ([ROW_BYTES / 128][rows][128 B],
// 8-row groups of 1024 bytes, piece c of row r at c ^ (r % 8)).
__device__ __forceinline__ uint32_t sw128_offset(int r, int u, int rows)
{
    const int kb = u >> 3, c = u & 7;
    return (uint32_t)(kb * rows * 128 + r * 128 + ((c ^ (r & 7)) << 4));
}

template <int ROW_BYTES, bool FP8>
struct CtxLayout {
    static constexpr int A_BYTES = kCtxQRows * ROW_BYTES;
    static constexpr int B_BYTES = kCtxKeys * ROW_BYTES;
    static constexpr int OFF_BAR = A_BYTES + B_BYTES;
    static constexpr int OFF_MISC = OFF_BAR + 8;
    // slack for 1024-byte alignment; at least 77 KB so that no more than two
    // CTAs (2 x 256 TMEM columns) share an SM
    static constexpr int NEED = OFF_MISC + 16 + 1024;
    static constexpr int ALLOC = NEED > 77 * 1024 ? NEED : 77 * 1024;
};

template <int ROW_BYTES, bool FP8>
__global__ void __launch_bounds__(kCtxThreads) ctx_stats_kernel(const CtxArgs a)
{
    using L = CtxLayout<ROW_BYTES, FP8>;
    constexpr int UNITS = ROW_BYTES / 16;    // 16-byte pieces per row
    constexpr int KSTEPS = ROW_BYTES / 32;   // one MMA consumes 32 bytes of d
    constexpr uint32_t FMT = FP8 ? 0u : 1u;

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (base - raw);
    const uint32_t sA = base, sB = base + L::A_BYTES, bar = base + L::OFF_BAR;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);

    const int b = (int)blockIdx.x / a.hq;
    const int h = (int)blockIdx.x - b * a.hq;
    const int g = h / (a.hq / a.hkv);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    griddep_wait();
    griddep_launch_dependents();
    const int n_vis = a.seq_off[b + 1] - a.seq_off[b];
    const int tf0 = a.text_off[b], Tf = a.text_off[b + 1] - tf0;
    const int s0 = a.sys_off[b], S = a.sys_off[b + 1] - s0;
    if (n_vis <= 0 || Tf <= 0) return;  // no scores in this request
    const int i0 = a.query_last ? Tf - 1 : 0;  // first query row within the request's text
    const int Tq = Tf - i0;
    if (Tq > kCtxQRows) {
        if (threadIdx.x == 0 && h == 0) atomicOr(a.err, kErrShape);
        return;
    }
    const int nk = S + Tf;  // keys of the last text row; earlier rows see a prefix
    const int n_tiles = (nk + kCtxKeys - 1) / kCtxKeys;

    if (threadIdx.x == 0) {
        mbar_init(bar, 1);
        *abort_flag = 0;
        fence_mbar_init_cluster();
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(tmem_slot), kCtxKeys);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const Ctl ctl{abort_flag, a.err, a.wait_budget};
    const float cl = a.c_log2;

    // query rows i0 .. Tf-1 of head h; rows Tq..127 are zero
    const uint8_t* qbase = a.q + ((int64_t)(tf0 + i0) * a.hq + h) * ROW_BYTES;
    for (int x = threadIdx.x; x < kCtxQRows * UNITS; x += kCtxThreads) {
        const int r = x / UNITS, u = x - r * UNITS;
        const bool ok = r < Tq;
        const uint8_t* src = ok ? qbase + (int64_t)r * a.hq * ROW_BYTES + u * 16 : a.q;
        cp_async16(sA + sw128_offset(r, u, kCtxQRows), src, ok ? 16u : 0u);
    }

    const int row = warp * 32 + lane;           // TMEM lane = query row of this thread
    const bool warp_live = warp * 32 < Tq;      // warp-uniform
    const int vis_keys = S + i0 + row + 1;      // causal prefix of this row
    float m = -INFINITY, l = 0.f;
    int issued = 0;
    for (int kt = 0; kt < n_tiles; ++kt) {
        const int j0 = kt * kCtxKeys;
        const int nkt = min(kCtxKeys, nk - j0);
        const int N = (nkt + 15) & ~15;
        for (int x = threadIdx.x; x < N * UNITS; x += kCtxThreads) {
            const int r = x / UNITS, u = x - r * UNITS;
            const int j = j0 + r;
            const uint8_t* src = a.q;
            uint32_t bytes = 0;
            if (r < nkt) {
                src = j < S ? a.k_sys + ((int64_t)(s0 + j) * a.hkv + g) * ROW_BYTES
                            : a.k_txt + ((int64_t)(tf0 + j - S) * a.hkv + g) * ROW_BYTES;
                src += u * 16;
                bytes = 16;
            }
            cp_async16(sB + sw128_offset(r, u, kCtxKeys), src, bytes);
        }
        cp_async_wait_all();
        fence_proxy_async_shared();  // the copies' writes -> visible to the tensor core
        __syncthreads();
        if (threadIdx.x == 0) {
            tc_fence_after();
            const uint32_t idesc = idesc_make(kCtxQRows, (uint32_t)N, FMT);
#pragma unroll
            for (int st = 0; st < KSTEPS; ++st) {
                const uint64_t ad = sdesc_k_sw128(sA + (st >> 2) * (kCtxQRows * 128) + (st & 3) * 32);
                const uint64_t bd = sdesc_k_sw128(sB + (st >> 2) * (kCtxKeys * 128) + (st & 3) * 32);
                if (FP8) mma_f8(tmem, ad, bd, idesc, st > 0);
                else mma_f16(tmem, ad, bd, idesc, st > 0);
            }
            mma_commit(bar);
        }
        ++issued;
        wait_phase(bar, (uint32_t)kt & 1u, ctl);
        __syncthreads();
        if (*abort_flag) break;  // uniform: read after the barrier
        tc_fence_after();
        if (warp_live) {
            const uint32_t ta = tmem + ((uint32_t)(warp * 32) << 16);
            for (int c0 = 0; c0 < N; c0 += 32) {
                float v[32];
                if (c0 + 32 <= N) {
                    tmem_ld32(ta + (uint32_t)c0, v);
                } else {
#pragma unroll
                    for (int c = 16; c < 32; ++c) v[c] = 0.f;
                    tmem_ld16(ta + (uint32_t)c0, v);
                }
                tmem_wait_ld();
                const int valid = min(vis_keys, nk) - (j0 + c0);
                if (row < Tq && valid > 0) row_stats_update<32>(v, min(valid, N - c0), cl, m, l);
            }
        }
        tc_fence_before();
        __syncthreads();  // TMEM and the B tile are free for the next key tile
    }
    if (!*abort_flag && row < Tq) a.out[(int64_t)(tf0 + i0 + row) * a.hq + h] = fmaf(m, cl, __log2f(l));
    if (*abort_flag && threadIdx.x == 0 && issued > 0) {
        // the last contraction lands before its TMEM columns are released
        volatile int no_abort = 0;
        const Ctl drain{&no_abort, a.err, kWaitBudgetCycles};
        wait_phase(bar, (uint32_t)(issued - 1) & 1u, drain);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) {
        tc_fence_after();
        tmem_dealloc(tmem, kCtxKeys);
    }
}

template <int ROW_BYTES, bool FP8>
cudaError_t launch_variant(const CtxArgs& a, cudaStream_t stream)
{
    using L = CtxLayout<ROW_BYTES, FP8>;
    auto kern = ctx_stats_kernel<ROW_BYTES, FP8>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::ALLOC);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(a.batch * a.hq), 1, 1);
    cfg.blockDim = dim3(kCtxThreads, 1, 1);
    cfg.dynamicSmemBytes = L::ALLOC;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1] = {pdl_attribute()};
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

}  // namespace

cudaError_t launch_ctx_stats(const CtxArgs& a, int row_bytes, bool fp8, cudaStream_t stream)
{
    if (a.batch <= 0) return cudaSuccess;
    if (fp8) return launch_variant<128, true>(a, stream);
    if (row_bytes == 256) return launch_variant<256, false>(a, stream);
    return launch_variant<128, false>(a, stream);
}

}  // namespace lvs
