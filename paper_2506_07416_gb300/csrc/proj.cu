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
// One CTA per 128 x BN output tile (BN = 256 or 128 columns, whole heads):
// warp 0 streams A (128 rows x 64 hidden) and B (BN rows of W' x 64) tiles by
// TMA into a 4-stage ring; warp 1 issues tcgen05.mma (M = 128, N = BN, K = 16,
// bf16, fp32 accumulator in TMEM); warps 2-5 sum the squares of their rows of
// each A tile (a ring slot is free once the MMA and these four warps are done
// with it), then read the accumulator (TMEM lane = row), scale, add the bias,
// rotate, round to bf16 and store. Every wait is bounded.

#include <math.h>

#include "internal.h"
#include "pipe.cuh"
#include "ptx.cuh"

namespace lvs {

namespace {

constexpr int kProjThreads = 192;
constexpr int kProjStages = 4;
constexpr int kProjK = 64;  // hidden values per stage (128 bytes of bf16)

template <int BN>
struct ProjLayout {
    static constexpr int A_BYTES = 128 * 128;
    static constexpr int B_BYTES = BN * 128;
    static constexpr int OFF_A = 0;
    static constexpr int OFF_B = OFF_A + kProjStages * A_BYTES;
    static constexpr int OFF_BAR = OFF_B + kProjStages * B_BYTES;  // full[S], empty[S], acc
    static constexpr int OFF_MISC = OFF_BAR + (2 * kProjStages + 1) * 8;
    static constexpr int ALLOC = OFF_MISC + 16 + 1024;
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}

template <int BN>
__global__ void __launch_bounds__(kProjThreads, 1)
    proj_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_w,
                const __grid_constant__ ProjArgs p)
{
    using L = ProjLayout<BN>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (base - raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // N tiles run fastest: the CTAs in flight share their A rows (read from DRAM
    // once, then from L2), and W' (all N tiles) stays in L2
    const int64_t m0 = (int64_t)blockIdx.y * 128;
    const int n0 = (int)blockIdx.x * BN;
    const int nk = (p.hidden + kProjK - 1) / kProjK;

    const uint32_t bar0 = base + L::OFF_BAR;
    auto FULL = [&](int s) -> uint32_t { return bar0 + 8u * (uint32_t)s; };
    auto EMPTY = [&](int s) -> uint32_t { return bar0 + 8u * (uint32_t)(kProjStages + s); };
    const uint32_t ACC = bar0 + 8u * (uint32_t)(2 * kProjStages);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::OFF_MISC);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::OFF_MISC + 4);

    if (threadIdx.x == 0) {
        for (int s = 0; s < kProjStages; ++s) {
            mbar_init(FULL(s), 1);
            mbar_init(EMPTY(s), 1 + 4);  // the MMA commit and the four row-sum warps
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
        tmem_alloc(smem_u32(tmem_slot), BN);
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
            int issued[kProjStages] = {0, 0, 0, 0};
            for (int kc = 0; kc < nk; ++kc) {
                const int s = kc % kProjStages;
                const uint32_t ph = (uint32_t)(kc / kProjStages) & 1u;
                if (!wait_phase(EMPTY(s), ph ^ 1u, ctl)) break;
                mbar_arrive_expect_tx(FULL(s), (uint32_t)(L::A_BYTES + L::B_BYTES));
                tma_load_3d(base + L::OFF_A + s * L::A_BYTES, &tm_x, FULL(s), kc * kProjK, 0, (int32_t)m0);
                tma_load_3d(base + L::OFF_B + s * L::B_BYTES, &tm_w, FULL(s), kc * kProjK, 0, n0);
                ++issued[s];
            }
            volatile int no_abort = 0;
            const Ctl drain{&no_abort, p.err, kWaitBudgetCycles};
            for (int s = 0; s < kProjStages; ++s)
                if (issued[s] > 0) wait_phase(FULL(s), (uint32_t)(issued[s] - 1) & 1u, drain);
        }
        __syncwarp();
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = idesc_make(128, BN, 1u);
            bool ok = true;
            for (int kc = 0; kc < nk && ok; ++kc) {
                const int s = kc % kProjStages;
                if (!wait_phase(FULL(s), (uint32_t)(kc / kProjStages) & 1u, ctl)) { ok = false; break; }
                tc_fence_after();
                const uint32_t a = base + L::OFF_A + s * L::A_BYTES, b = base + L::OFF_B + s * L::B_BYTES;
#pragma unroll
                for (int st = 0; st < 4; ++st)
                    mma_f16(tmem, sdesc_k_sw128(a + st * 32), sdesc_k_sw128(b + st * 32), idesc, (kc | st) != 0);
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
        const int quad = warp & 3;
        const int r = quad * 32 + lane;  // row of the tile = TMEM lane
        float ss0 = 0.f, ss1 = 0.f;
        for (int kc = 0; kc < nk; ++kc) {
            const int s = kc % kProjStages;
            if (!wait_phase(FULL(s), (uint32_t)(kc / kProjStages) & 1u, ctl)) break;
            const uint8_t* row = smem + L::OFF_A + s * L::A_BYTES + r * 128;
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
        const bool ok = wait_phase(ACC, 0, ctl);
        tc_fence_after();
        const int64_t grow = m0 + r;
        const bool live = ok && grow < p.rows;
        const float sc = rsqrtf((ss0 + ss1) / (float)p.hidden + p.eps);
        int pos = 0;
        if (live && p.head_dim > 0) {
            pos = p.positions[grow];
            if (pos < 0 || pos >= p.max_positions) {
                atomicOr(p.err, kErrBounds);
                pos = 0;
            }
        }
        const uint32_t ta = tmem + ((uint32_t)(quad * 32) << 16);
        __nv_bfloat16* yrow = p.y + grow * (int64_t)p.out_features + n0;
        if (p.head_dim > 0) {
            const int half = p.head_dim / 2;
            const float2* cs_row = p.rope + (int64_t)pos * half;
            for (int h0 = 0; h0 < BN; h0 += p.head_dim) {
                for (int c = 0; c < half; c += 32) {
                    float v1[32], v2[32];
                    tmem_ld32(ta + (uint32_t)(h0 + c), v1);
                    tmem_ld32(ta + (uint32_t)(h0 + half + c), v2);
                    tmem_wait_ld();
                    if (live) {
                        uint32_t o1[16], o2[16];
#pragma unroll
                        for (int j = 0; j < 32; j += 2) {
                            float a[2], b[2];
#pragma unroll
                            for (int e = 0; e < 2; ++e) {
                                const int col1 = n0 + h0 + c + j + e;
                                const float y1 = fmaf(v1[j + e], sc, p.bias ? p.bias[col1] : 0.f);
                                const float y2 = fmaf(v2[j + e], sc, p.bias ? p.bias[col1 + half] : 0.f);
                                const float2 cs = cs_row[c + j + e];
                                a[e] = y1 * cs.x - y2 * cs.y;
                                b[e] = y2 * cs.x + y1 * cs.y;
                            }
                            o1[j / 2] = pack_bf16(a[0], a[1]);
                            o2[j / 2] = pack_bf16(b[0], b[1]);
                        }
                        uint4* d1 = reinterpret_cast<uint4*>(yrow + h0 + c);
                        uint4* d2 = reinterpret_cast<uint4*>(yrow + h0 + half + c);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            d1[q] = make_uint4(o1[4 * q], o1[4 * q + 1], o1[4 * q + 2], o1[4 * q + 3]);
                            d2[q] = make_uint4(o2[4 * q], o2[4 * q + 1], o2[4 * q + 2], o2[4 * q + 3]);
                        }
                    }
                }
            }
        } else {
            for (int c = 0; c < BN; c += 32) {
                float v[32];
                tmem_ld32(ta + (uint32_t)c, v);
                tmem_wait_ld();
                if (live) {
                    uint32_t o[16];
#pragma unroll
                    for (int j = 0; j < 32; j += 2)
                        o[j / 2] = pack_bf16(fmaf(v[j], sc, p.bias ? p.bias[n0 + c + j] : 0.f),
                                             fmaf(v[j + 1], sc, p.bias ? p.bias[n0 + c + j + 1] : 0.f));
                    uint4* d = reinterpret_cast<uint4*>(yrow + c);
#pragma unroll
                    for (int q = 0; q < 4; ++q) d[q] = make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, BN);
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

template <int BN>
cudaError_t launch_proj_variant(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const ProjArgs& p,
                                cudaStream_t stream)
{
    using L = ProjLayout<BN>;
    auto kern = proj_kernel<BN>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::ALLOC);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(p.out_features / BN), (unsigned)((p.rows + 127) / 128), 1);
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

cudaError_t launch_proj(const CUtensorMap& tm_x, const CUtensorMap& tm_w, const ProjArgs& p, cudaStream_t stream)
{
    if (p.rows <= 0) return cudaSuccess;
    return proj_tile_cols(p.out_features) == 256 ? launch_proj_variant<256>(tm_x, tm_w, p, stream)
                                                 : launch_proj_variant<128>(tm_x, tm_w, p, stream);
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
