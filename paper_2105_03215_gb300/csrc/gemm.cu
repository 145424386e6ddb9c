// gemm.cu -- implicit-GEMM convolution and dense layer on the sm_103a tensor
// cores (tcgen05), with the region's bias / folded batch norm / residual add
// / activation fused into the epilogue, so each offloaded composite
// (Section 3.1.1: a Conv2D-Add-ReLU style sequence mapped to one
// "instruction") makes one pass over HBM.
//
// Structure (one persistent CTA per SM, 192 threads):
//   warp 0     TMA producer: per k-block, one A tile (128 rows x BK) and one
//              B tile (BN rows x BK) into a STAGES-deep shared-memory ring.
//              A is a 2-D tile of a row-major matrix, or -- for convolutions --
//              an im2col tile: 128 consecutive output pixels of one filter tap
//              and channel chunk, with out-of-image taps zero-filled by TMA.
//   warp 1     allocates TMEM; one lane issues tcgen05.mma (M=128, N=BN, K=16
//              per instruction) into one of two fp32 accumulators in TMEM and
//              tcgen05.commit's the ring slots and the finished accumulator.
//   warps 2-5  epilogue: tcgen05.ld of 32 columns at a time (each thread owns
//              one output row), + bias, + residual, activation, bf16 rounding,
//              16-byte stores.  Releases the accumulator as soon as it has been
//              read, so the next tile's MMAs overlap this tile's stores.
#include "internal.h"
#include "ptx.cuh"

namespace byoc {

template <int BN, int BK>
struct GemmShape {
    static constexpr int BM = kGemmBM;
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int RING_BUDGET = 200 * 1024;
    static constexpr int STAGES_RAW = RING_BUDGET / STAGE_BYTES;
    static constexpr int STAGES = STAGES_RAW > 16 ? 16 : STAGES_RAW;
    static constexpr int TMEM_COLS = 2 * BN < 32 ? 32 : 2 * BN;
    static constexpr int NUM_BARS = 2 * STAGES + 5;
    static constexpr int CTRL_BYTES = 8 * NUM_BARS + 16;
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + CTRL_BYTES;
    static_assert(A_BYTES % 1024 == 0 && B_BYTES % 1024 == 0, "tiles must keep 1 KB alignment");
    static_assert(BN % 32 == 0 && BN >= 32 && BN <= 256, "BN");
    static_assert(BK == 16 || BK == 32 || BK == 64, "BK");
};

__device__ __forceinline__ float apply_act(float v, int act) {
    switch (act) {
        case kActRelu: return fmaxf(v, 0.0f);
        case kActRelu6: return fminf(fmaxf(v, 0.0f), 6.0f);
        case kActGelu: return 0.5f * v * (1.0f + erff(v * 0.70710678118654752f));
        default: return v;
    }
}

template <int BN, int BK, bool IM2COL>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_tcgen05_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB, const GemmArgs a) {
    using S = GemmShape<BN, BK>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (base - raw);
    const uint32_t sA = base;
    const uint32_t sB = base + S::STAGES * S::A_BYTES;
    const uint32_t bars = base + S::STAGES * S::STAGE_BYTES;
    const uint32_t tfull = bars + 8u * (2 * S::STAGES);  // 2 barriers
    const uint32_t tempty = tfull + 16u;                 // 2 barriers
    const uint32_t drain = tempty + 16u;
    uint32_t *tmem_slot =
        reinterpret_cast<uint32_t *>(smem + S::STAGES * S::STAGE_BYTES + 8 * S::NUM_BARS);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S::STAGES; ++s) {
            mbar_init(bars + 8u * s, 1);                  // full[s]: producer + TMA bytes
            mbar_init(bars + 8u * (S::STAGES + s), 1);    // empty[s]: MMA commit
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(tfull + 8u * b, 1);   // accumulator ready: MMA commit
            mbar_init(tempty + 8u * b, 4);  // accumulator drained: one arrive per epilogue warp
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), S::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------ TMA producer
            int it = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < a.num_tiles; tile += gridDim.x) {
                const int m0 = (tile / a.tiles_n) * S::BM;
                const int n0 = (tile % a.tiles_n) * BN;
                int img = 0, h0 = 0, w0 = 0;
                if (IM2COL) {
                    const int hw = a.Ho * a.Wo;
                    img = m0 / hw;
                    const int rem = m0 - img * hw;
                    const int p = rem / a.Wo;
                    const int q = rem - p * a.Wo;
                    h0 = p * a.stride_h - a.pad_t;
                    w0 = q * a.stride_w - a.pad_l;
                }
                for (int kb = 0; kb < a.num_kb; ++kb, ++it) {
                    const int s = it % S::STAGES;
                    const uint32_t ph = (uint32_t)(it / S::STAGES) & 1u;
                    if (!mbar_wait(bars + 8u * (S::STAGES + s), ph ^ 1u, abort_flag, a.err,
                                   kErrTimeoutProducer)) {
                        ok = false;
                        break;
                    }
                    const uint32_t full = bars + 8u * s;
                    mbar_arrive_expect_tx(full, S::STAGE_BYTES);
                    if (IM2COL) {
                        const int tap = kb / a.chunks;
                        const int cc = kb - tap * a.chunks;
                        const int r = tap / a.kw;
                        const int sx = tap - r * a.kw;
                        tma_load_im2col_4d(sA + s * S::A_BYTES, &tmA, full, cc * BK, w0, h0, img,
                                           (uint16_t)(sx * a.dil_w), (uint16_t)(r * a.dil_h));
                    } else {
                        tma_load_2d(sA + s * S::A_BYTES, &tmA, full, kb * BK, m0);
                    }
                    tma_load_2d(sB + s * S::B_BYTES, &tmB, full, kb * BK, n0);
                }
            }
            if (!ok) {
                // Gave up: let the copies already issued land before exiting.
                const int first = it - S::STAGES > 0 ? it - S::STAGES : 0;
                for (int j = first; j < it; ++j)
                    mbar_wait_drain(bars + 8u * (j % S::STAGES), (uint32_t)(j / S::STAGES) & 1u);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------ MMA issuer
            constexpr uint32_t idesc = make_idesc_bf16(S::BM, BN);
            int it = 0, t = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < a.num_tiles; tile += gridDim.x, ++t) {
                const int buf = t & 1;
                const uint32_t aph = (uint32_t)(t >> 1) & 1u;
                if (!mbar_wait(tempty + 8u * buf, aph ^ 1u, abort_flag, a.err, kErrTimeoutMma)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
                for (int kb = 0; kb < a.num_kb; ++kb, ++it) {
                    const int s = it % S::STAGES;
                    const uint32_t ph = (uint32_t)(it / S::STAGES) & 1u;
                    if (!mbar_wait(bars + 8u * s, ph, abort_flag, a.err, kErrTimeoutMma)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_s = sA + s * S::A_BYTES;
                    const uint32_t b_s = sB + s * S::B_BYTES;
#pragma unroll
                    for (int k = 0; k < BK / 16; ++k) {
                        mma_bf16_ss(d_tmem, make_smem_desc(a_s + 32u * k, BK * 2),
                                    make_smem_desc(b_s + 32u * k, BK * 2), idesc,
                                    (kb | k) != 0 ? 1u : 0u);
                    }
                    mma_commit(bars + 8u * (S::STAGES + s));  // frees the ring slot
                }
                if (!ok) break;
                mma_commit(tfull + 8u * buf);  // accumulator complete
            }
            // All issued MMAs must finish before TMEM is released.
            mma_commit(drain);
            mbar_wait_drain(drain, 0);
        }
    } else {
        // ---------------------------------------------------- epilogue
        const int quarter = warp & 3;  // TMEM lanes this warp may access
        int t = 0;
        for (int tile = blockIdx.x; tile < a.num_tiles; tile += gridDim.x, ++t) {
            const int buf = t & 1;
            const uint32_t aph = (uint32_t)(t >> 1) & 1u;
            if (!mbar_wait(tfull + 8u * buf, aph, abort_flag, a.err, kErrTimeoutEpilogue)) break;
            tc_fence_after();
            const int m0 = (tile / a.tiles_n) * S::BM;
            const int n0 = (tile % a.tiles_n) * BN;
            const int row = m0 + quarter * 32 + lane;
            const uint32_t tbase =
                tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * BN);
#pragma unroll 1
            for (int c0 = 0; c0 < BN; c0 += 32) {
                uint32_t v[32];
                tmem_ld_32cols(tbase + (uint32_t)c0, v);  // includes tcgen05.wait::ld
                if (c0 + 32 == BN) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(tempty + 8u * buf);
                }
                const int col0 = n0 + c0;
                if (row < a.M && col0 < a.N) {
                    float f[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) f[j] = __uint_as_float(v[j]);
                    if (a.bias) {
                        const float4 *bp = reinterpret_cast<const float4 *>(a.bias + col0);
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            const float4 b4 = __ldg(bp + j);
                            f[4 * j] += b4.x;
                            f[4 * j + 1] += b4.y;
                            f[4 * j + 2] += b4.z;
                            f[4 * j + 3] += b4.w;
                        }
                    }
                    const size_t off = (size_t)row * (size_t)a.N + (size_t)col0;
                    if (a.residual) {
                        const uint4 *rp = reinterpret_cast<const uint4 *>(a.residual + off);
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            if (col0 + 8 * q < a.N) {
                                const uint4 r4 = __ldg(rp + q);
                                const uint32_t rr[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
                                for (int e = 0; e < 4; ++e) {
                                    f[8 * q + 2 * e] += bf16lo(rr[e]);
                                    f[8 * q + 2 * e + 1] += bf16hi(rr[e]);
                                }
                            }
                        }
                    }
#pragma unroll
                    for (int j = 0; j < 32; ++j) f[j] = apply_act(f[j], a.act);
                    uint4 *op = reinterpret_cast<uint4 *>(a.out + off);
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        if (col0 + 8 * q < a.N) {
                            uint4 o;
                            o.x = pack_bf16x2(f[8 * q + 0], f[8 * q + 1]);
                            o.y = pack_bf16x2(f[8 * q + 2], f[8 * q + 3]);
                            o.z = pack_bf16x2(f[8 * q + 4], f[8 * q + 5]);
                            o.w = pack_bf16x2(f[8 * q + 6], f[8 * q + 7]);
                            op[q] = o;
                        }
                    }
                }
            }
        }
    }

    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, S::TMEM_COLS);
    }
}

// ---------------------------------------------------------------- dispatch

template <int BN, int BK, bool IM2COL>
static cudaError_t launch_t(const CUtensorMap &tmA, const CUtensorMap &tmB, const GemmArgs &a,
                            int grid, cudaStream_t st) {
    using S = GemmShape<BN, BK>;
    gemm_tcgen05_kernel<BN, BK, IM2COL><<<grid, kGemmThreads, S::SMEM_BYTES, st>>>(tmA, tmB, a);
    return cudaGetLastError();
}

template <int BN, int BK, bool IM2COL>
static cudaError_t prepare_t() {
    using S = GemmShape<BN, BK>;
    return cudaFuncSetAttribute(gemm_tcgen05_kernel<BN, BK, IM2COL>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, S::SMEM_BYTES);
}

// The instantiated (BN, BK, im2col) combinations.
#define BYOC_GEMM_CONFIGS(X) \
    X(32, 64, false)         \
    X(64, 64, false)         \
    X(128, 64, false)        \
    X(256, 64, false)        \
    X(32, 64, true)          \
    X(64, 64, true)          \
    X(128, 64, true)         \
    X(256, 64, true)         \
    X(64, 16, true)          \
    X(64, 32, true)          \
    X(128, 32, true)

bool gemm_config_supported(const GemmConfig &c) {
#define X(BN_, BK_, IM_) \
    if (c.bn == BN_ && c.bk == BK_ && c.im2col == IM_) return true;
    BYOC_GEMM_CONFIGS(X)
#undef X
    return false;
}

size_t gemm_smem_bytes(const GemmConfig &c) {
#define X(BN_, BK_, IM_) \
    if (c.bn == BN_ && c.bk == BK_) return (size_t)GemmShape<BN_, BK_>::SMEM_BYTES;
    BYOC_GEMM_CONFIGS(X)
#undef X
    return 0;
}

int gemm_stages(const GemmConfig &c) {
#define X(BN_, BK_, IM_) \
    if (c.bn == BN_ && c.bk == BK_) return GemmShape<BN_, BK_>::STAGES;
    BYOC_GEMM_CONFIGS(X)
#undef X
    return 0;
}

cudaError_t gemm_prepare(const GemmConfig &c) {
#define X(BN_, BK_, IM_) \
    if (c.bn == BN_ && c.bk == BK_ && c.im2col == IM_) return prepare_t<BN_, BK_, IM_>();
    BYOC_GEMM_CONFIGS(X)
#undef X
    return cudaErrorInvalidValue;
}

cudaError_t launch_gemm(const GemmConfig &c, const CUtensorMap &tmA, const CUtensorMap &tmB,
                        const GemmArgs &a, int grid, cudaStream_t st) {
#define X(BN_, BK_, IM_) \
    if (c.bn == BN_ && c.bk == BK_ && c.im2col == IM_) return launch_t<BN_, BK_, IM_>(tmA, tmB, a, grid, st);
    BYOC_GEMM_CONFIGS(X)
#undef X
    return cudaErrorInvalidValue;
}

}  // namespace byoc
