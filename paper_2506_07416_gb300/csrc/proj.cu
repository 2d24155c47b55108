// Layer-0 projection that makes the queries and keys the scores read (Design
// section: the module is the first decoder layer, whose q and k are
// RoPE(W . RMSNorm(x))):
//     s_r    = 1 / sqrt(mean_h x_r[h]^2 + eps)
//     y_r[o] = s_r * sum_h x_r[h] * W'[o][h] + bias[o],   W' = W * gamma (per input column)
// then rotary position embedding per head (rotate-half pairs j, j + d/2) with
// cos / sin from a table indexed by the row's position.
//
// The RMSNorm weight is folded into W once (fold kernel below), so the
// contraction reads the raw hidden rows; the per-row scale s_r is a sum of
// squares taken from the A tiles while they sit in shared memory for the
// tensor core, and is applied in the epilogue with the bias and the rotation.
//
// One CTA per (128 * MT) x BN output tile (BN = 256 or 128 columns, whole
// heads; MT = 2 when the grid still gives every SM two tiles): warp 0 streams
// A (128 * MT rows x 64 hidden) and B (BN rows of W' x 64) tiles by TMA into a
// 3- or 4-stage ring; warp 1 issues tcgen05.mma (M = 128 per row block,
// N = BN, K = 16, bf16, fp32 accumulators in TMEM); two epilogue warpgroups sum
// the squares of their rows of each A tile (a ring slot is free once the MMA
// and these warps are done with it), then read the accumulator (TMEM lane =
// row), scale, add the bias, rotate, round to bf16 and store. Every wait is
// bounded.

#include <math.h>

#include <cuda_fp8.h>

#include "internal.h"
#include "pipe.cuh"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kProjThreads = 320;  // producer, MMA issuer, two epilogue warpgroups
constexpr int kProjK = 64;  // hidden values per stage (128 bytes of bf16)

// MT row blocks of 128 per CTA (one accumulator each, MT * BN TMEM columns):
// MT = 2 halves the operand bytes per MMA cycle (each W' tile serves 256 rows).
template <int BN, int MT>
struct ProjLayout {
    static constexpr int A_BYTES = MT * 128 * 128;
    static constexpr int B_BYTES = BN * 128;
    static constexpr int STAGE = A_BYTES + B_BYTES;
    static constexpr int FIT = (225 * 1024) / STAGE;
    static constexpr int STAGES = FIT > 4 ? 4 : FIT;
    static constexpr int OFF_A = 0;
    static constexpr int OFF_B = OFF_A + STAGES * A_BYTES;
    static constexpr int OFF_BAR = OFF_B + STAGES * B_BYTES;  // full[S], empty[S], acc
    static constexpr int OFF_MISC = OFF_BAR + (2 * STAGES + 1) * 8;
    static constexpr int OFF_SC = OFF_MISC + 16;               // [128] row scales (MT = 1)
    static constexpr int ALLOC = OFF_SC + 128 * 4 + 1024;
    static constexpr int TMEM_COLS = MT * BN;
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}

// two e4m3 codes (round to nearest even, saturating to +-448)
__device__ __forceinline__ uint32_t pack_e4m3(float lo, float hi)
{
    return (uint32_t)__nv_cvt_float2_to_fp8x2(make_float2(lo, hi), __NV_SATFINITE, __NV_E4M3);
}

// 32 consecutive outputs of one row from 16 value pairs: bf16 (64 bytes), or
// e4m3 codes of y / scale (32 bytes) when the call asked for e4m3
__device__ __forceinline__ void store_pairs(const ProjArgs& p, int64_t elem, const float2 (&y)[16])
{
    if (p.y8) {
        uint32_t o[8];
#pragma unroll
        for (int q = 0; q < 8; ++q)
            o[q] = pack_e4m3(y[2 * q].x * p.out_inv_scale, y[2 * q].y * p.out_inv_scale) |
                   (pack_e4m3(y[2 * q + 1].x * p.out_inv_scale, y[2 * q + 1].y * p.out_inv_scale) << 16);
        uint4* d = reinterpret_cast<uint4*>(p.y8 + elem);
        d[0] = make_uint4(o[0], o[1], o[2], o[3]);
        d[1] = make_uint4(o[4], o[5], o[6], o[7]);
    } else {
        uint32_t o[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) o[q] = pack_bf16(y[q].x, y[q].y);
        uint4* d = reinterpret_cast<uint4*>(p.y + elem);
#pragma unroll
        for (int q = 0; q < 4; ++q) d[q] = make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
    }
}

// scale, bias, rotation and store (bf16 or e4m3) of columns [c_begin, c_end) of one
// accumulator row (this thread's); the range holds whole heads
__device__ __forceinline__ void proj_store_row(const ProjArgs& p, uint32_t ta, int64_t grow, int n0, int c_begin,
                                               int c_end, bool live, float sc)
{
    int pos = 0;
    if (live && p.head_dim > 0) {
        pos = p.positions[grow];
        if (pos < 0 || pos >= p.max_positions) {
            atomicOr(p.err, kErrBounds);
            pos = 0;
        }
    }
    const int64_t row0 = grow * (int64_t)p.out_features + n0;  // element index of this tile's first column
    if (p.head_dim > 0) {
        const int half = p.head_dim / 2;
        const float2* cs_row = p.rope + (int64_t)pos * half;
        for (int h0 = c_begin; h0 < c_end; h0 += p.head_dim) {
            for (int c = 0; c < half; c += 32) {
                float v1[32], v2[32];
                tmem_ld32(ta + (uint32_t)(h0 + c), v1);
                tmem_ld32(ta + (uint32_t)(h0 + half + c), v2);
                tmem_wait_ld();
                if (live) {
                    float2 a[16], b[16];
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int col1 = n0 + h0 + c + j;
                        const float y1 = fmaf(v1[j], sc, p.bias ? p.bias[col1] : 0.f);
                        const float y2 = fmaf(v2[j], sc, p.bias ? p.bias[col1 + half] : 0.f);
                        const float2 cs = cs_row[c + j];
                        const float r1 = y1 * cs.x - y2 * cs.y, r2 = y2 * cs.x + y1 * cs.y;
                        if (j & 1) {
                            a[j / 2].y = r1;
                            b[j / 2].y = r2;
                        } else {
                            a[j / 2].x = r1;
                            b[j / 2].x = r2;
                        }
                    }
                    store_pairs(p, row0 + h0 + c, a);
                    store_pairs(p, row0 + h0 + half + c, b);
                }
            }
        }
    } else {
        for (int c = c_begin; c < c_end; c += 32) {
            float v[32];
            tmem_ld32(ta + (uint32_t)c, v);
            tmem_wait_ld();
            if (live) {
                float2 o[16];
#pragma unroll
                for (int j = 0; j < 32; j += 2)
                    o[j / 2] = make_float2(fmaf(v[j], sc, p.bias ? p.bias[n0 + c + j] : 0.f),
                                           fmaf(v[j + 1], sc, p.bias ? p.bias[n0 + c + j + 1] : 0.f));
                store_pairs(p, row0 + c, o);
            }
        }
    }
}

template <int BN, int MT>
__global__ void __launch_bounds__(kProjThreads, 1)
    proj_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                const __grid_constant__ ProjArgs p)
{
    using L = ProjLayout<BN, MT>;
    constexpr int S = L::STAGES;
    static_assert(S >= 3, "ring depth");
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (base - raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // N tiles run fastest: the CTAs in flight share their A rows (read from DRAM
    // once, then from L2), and W' (all N tiles) stays in L2
    const int64_t m0 = (int64_t)blockIdx.y * (128 * MT);
    const int n0 = (int)blockIdx.x * BN;
    const int nk = (p.hidden + kProjK - 1) / kProjK;

    const uint32_t bar0 = base + L::OFF_BAR;
    auto FULL = [&](int s) -> uint32_t { return bar0 + 8u * (uint32_t)s; };
    auto EMPTY = [&](int s) -> uint32_t { return bar0 + 8u * (uint32_t)(S + s); };
    const uint32_t ACC = bar0 + 8u * (uint32_t)(2 * S);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(FULL(s), 1);
            mbar_init(EMPTY(s), 1 + 4 * MT);  // the MMA commit and the row-sum warps
        }
        mbar_init(ACC, 1);
        *abort_flag = 0;
        fence_mbar_init_cluster();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tm_x);
        tma_prefetch_desc(&tm_w);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), L::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const Ctl ctl{abort_flag, p.err, p.wait_budget};
    griddep_wait();
    griddep_launch_dependents();

    if (warp == 0) {
        // ---------------------------------------------------------------- TMA producer
        if (lane == 0) {
            int issued[S];
            for (int s = 0; s < S; ++s) issued[s] = 0;
            for (int kc = 0; kc < nk; ++kc) {
                const int s = kc % S;
                const uint32_t ph = (uint32_t)(kc / S) & 1u;
                if (!wait_phase(EMPTY(s), ph ^ 1u, ctl)) break;
                mbar_arrive_expect_tx(FULL(s), (uint32_t)(L::A_BYTES + L::B_BYTES));
                // one box of 128 * MT rows: the second row block lands 16 KB after the first
                tma_load_3d(base + L::OFF_A + s * L::A_BYTES, &tm_x, FULL(s), kc * kProjK, 0, (int32_t)m0);
                tma_load_3d(base + L::OFF_B + s * L::B_BYTES, &tm_w, FULL(s), kc * kProjK, 0, n0);
                ++issued[s];
            }
            volatile int no_abort = 0;
            const Ctl drain{&no_abort, p.err, kWaitBudgetCycles};
            for (int s = 0; s < S; ++s)
                if (issued[s] > 0) wait_phase(FULL(s), (uint32_t)(issued[s] - 1) & 1u, drain);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_make(128, BN, 1u);
            bool ok = true;
            for (int kc = 0; kc < nk && ok; ++kc) {
                const int s = kc % S;
                if (!wait_phase(FULL(s), (uint32_t)(kc / S) & 1u, ctl)) { ok = false; break; }
                tc_fence_after();
                const uint32_t a = base + L::OFF_A + s * L::A_BYTES, b = base + L::OFF_B + s * L::B_BYTES;
#pragma unroll
                for (int mt = 0; mt < MT; ++mt)
#pragma unroll
                    for (int st = 0; st < 4; ++st)
                        mma_f16(tmem + (uint32_t)(mt * BN), sdesc_k_sw128(a + mt * 128 * 128 + st * 32),
                                sdesc_k_sw128(b + st * 32), idesc, (kc | st) != 0);
                mma_commit(EMPTY(s));
            }
            mma_commit(ACC);  // every contraction above has landed once this arrives
            volatile int no_abort = 0;
            const Ctl drain{&no_abort, p.err, kWaitBudgetCycles};
            wait_phase(ACC, 0, drain);
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------------------- row sums + epilogue
        // MT = 2: warpgroup g owns row block g (its sums and its accumulator).
        // MT = 1: warpgroup 0 takes the row sums, and the two warpgroups split
        // the columns (whole heads) of the epilogue.
        const int quad = warp & 3;
        const int wg = (warp - 2) >> 2;
        const int r = quad * 32 + lane;  // row of the 128-row block = TMEM lane
        float* sc_s = reinterpret_cast<float*>(smem + L::OFF_SC);
        const bool sums = MT == 2 || wg == 0;
        float ss0 = 0.f, ss1 = 0.f;
        if (sums) {
            const int mt = MT == 2 ? wg : 0;
            for (int kc = 0; kc < nk; ++kc) {
                const int s = kc % S;
                if (!wait_phase(FULL(s), (uint32_t)(kc / S) & 1u, ctl)) break;
                const uint8_t* row = smem + L::OFF_A + s * L::A_BYTES + mt * 128 * 128 + r * 128;
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const uint4 v = *reinterpret_cast<const uint4*>(row + ((j ^ (r & 7)) << 4));
                    const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const float lo = __uint_as_float(w4[q] << 16), hi = __uint_as_float(w4[q] & 0xFFFF0000u);
                        ss0 = fmaf(lo, lo, ss0);
                        ss1 = fmaf(hi, hi, ss1);
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(EMPTY(s));
            }
        }
        float sc = rsqrtf((ss0 + ss1) / (float)p.hidden + p.eps);
        if (MT == 1) {
            if (wg == 0) sc_s[r] = sc;
            named_bar_sync(1, 256);
            sc = sc_s[r];
        }
        const bool ok = wait_phase(ACC, 0, ctl);
        tc_fence_after();
        const int mt = MT == 2 ? wg : 0;
        const int64_t grow = m0 + mt * 128 + r;
        int c_begin = 0, c_end = BN;
        if (MT == 1) {
            const int unit = p.head_dim > 32 ? p.head_dim : 32;
            if ((BN / 2) % unit == 0) {
                c_begin = wg * (BN / 2);
                c_end = c_begin + BN / 2;
            } else if (wg == 1) {
                c_end = 0;  // the columns cannot be split by whole heads: warpgroup 0 takes all
            }
        }
        proj_store_row(p, tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)(mt * BN), grow, n0, c_begin, c_end,
                       ok && grow < p.rows, sc);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, L::TMEM_COLS);
    }
}

// W'[o][h] = bf16(W[o][h] * gamma[h])
__global__ void fold_norm_kernel(const __nv_bfloat16* __restrict__ w, const float* __restrict__ gamma,
                                 __nv_bfloat16* __restrict__ out, int64_t total, int hidden)
{
    griddep_wait();
    griddep_launch_dependents();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x)
        out[i] = __float2bfloat16_rn(__bfloat162float(w[i]) * gamma[i % hidden]);
}

// table[p][j] = (cos, sin) of the fp32 angle p * inv_freq[j]
__global__ void rope_table_kernel(const RopeArgs a)
{
    griddep_wait();
    griddep_launch_dependents();
    const int64_t total = (int64_t)a.max_positions * a.half;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
        const int pos = (int)(i / a.half), j = (int)(i % a.half);
        float s, c;
        sincosf((float)pos * a.inv_freq[j], &s, &c);
        a.table[i] = make_float2(c, s);
    }
}

template <class... Args>
cudaError_t launch_plain(void (*kern)(Args...), unsigned grid, unsigned block, size_t smem, cudaStream_t stream,
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

template <int BN, int MT>
cudaError_t launch_proj_variant(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const ProjArgs& p,
                                cudaStream_t stream)
{
    using L = ProjLayout<BN, MT>;
    auto kern = proj_kernel<BN, MT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::ALLOC);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(p.out_features / BN), (unsigned)((p.rows + 128 * MT - 1) / (128 * MT)), 1);
    cfg.blockDim = dim3(kProjThreads, 1, 1);
    cfg.dynamicSmemBytes = L::ALLOC;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1] = {pdl_attribute()};
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, tm_x, tm_w, p);
}

}  // namespace

int proj_tile_cols(int out_features) { return out_features % 256 == 0 ? 256 : 128; }

// 256-row tiles when they still give every SM two tiles, else 128-row tiles
int proj_tile_rows(int64_t rows, int out_features, int num_sms)
{
    const int64_t n_tiles = out_features / proj_tile_cols(out_features);
    return ((rows + 255) / 256) * n_tiles >= 2LL * num_sms ? 256 : 128;
}

cudaError_t launch_proj(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const ProjArgs& p, int tile_rows,
                        cudaStream_t stream)
{
    if (p.rows <= 0) return cudaSuccess;
    const bool wide = proj_tile_cols(p.out_features) == 256;
    if (tile_rows == 256)
        return wide ? launch_proj_variant<256, 2>(tm_x, tm_w, p, stream)
                    : launch_proj_variant<128, 2>(tm_x, tm_w, p, stream);
    return wide ? launch_proj_variant<256, 1>(tm_x, tm_w, p, stream)
                : launch_proj_variant<128, 1>(tm_x, tm_w, p, stream);
}

cudaError_t launch_fold_norm(const __nv_bfloat16* w, const float* gamma, __nv_bfloat16* out, int64_t total,
                             int hidden, int num_sms, cudaStream_t stream)
{
    if (total <= 0) return cudaSuccess;
    const int64_t want = (total + 255) / 256;
    const unsigned grid = (unsigned)(want < 8LL * num_sms ? want : 8LL * num_sms);
    return launch_plain(fold_norm_kernel, grid, 256, 0, stream, w, gamma, out, total, hidden);
}

cudaError_t launch_rope_table(const RopeArgs& a, int num_sms, cudaStream_t stream)
{
    const int64_t total = (int64_t)a.max_positions * a.half;
    if (total <= 0) return cudaSuccess;
    const int64_t want = (total + 255) / 256;
    const unsigned grid = (unsigned)(want < 8LL * num_sms ? want : 8LL * num_sms);
    return launch_plain(rope_table_kernel, grid, 256, 0, stream, a);
}

}  // namespace lvs
