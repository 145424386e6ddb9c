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
//   warps 2-9  epilogue: two warps per 32-row TMEM lane quarter, taking
//              alternate 32-column chunks.  Per chunk: tcgen05.ld (one row per
//              thread), + bias, + residual, activation, bf16 rounding, then a
//              transpose through a 64-byte-swizzled shared-memory tile so that
//              the global stores are coalesced 64-byte row segments.  The
//              residual is read with the same coalesced pattern, two of the
//              warp's chunks ahead, into registers.  The accumulator is
//              released as soon as it has been read, so the next tile's MMAs
//              overlap this tile's stores.
#include "internal.h"
#include "ptx.cuh"

namespace byoc {

template <int BN, int BK>
struct GemmShape {
    static constexpr int BM = kGemmBM;
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int RING_BUDGET = 192 * 1024;
    static constexpr int STAGES_RAW = RING_BUDGET / STAGE_BYTES;
    static constexpr int STAGES = STAGES_RAW > 16 ? 16 : STAGES_RAW;
    static constexpr int TMEM_COLS = 2 * BN < 32 ? 32 : 2 * BN;
    // Epilogue staging per warp: one output and one residual 32x32 bf16 tile.
    static constexpr int EPI_TILE = 32 * 32 * 2;
    static constexpr int EPI_WARP_BYTES = 2 * EPI_TILE;
    static constexpr int EPI_BYTES = kGemmEpiWarps * EPI_WARP_BYTES;
    static constexpr int NUM_BARS = 2 * STAGES + 5;
    static constexpr int CTRL_BYTES = 8 * NUM_BARS + 16;
    static constexpr int SMEM_BYTES = 1024 + STAGES * STAGE_BYTES + EPI_BYTES + CTRL_BYTES;
    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
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
    const uint32_t sEpi = base + S::STAGES * S::STAGE_BYTES;
    const uint32_t bars = sEpi + S::EPI_BYTES;
    const uint32_t tfull = bars + 8u * (2 * S::STAGES);  // 2 barriers
    const uint32_t tempty = tfull + 16u;                 // 2 barriers
    const uint32_t drain = tempty + 16u;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(
        smem + S::STAGES * S::STAGE_BYTES + S::EPI_BYTES + 8 * S::NUM_BARS);
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
            mbar_init(tempty + 8u * b, kGemmEpiWarps);  // drained: one arrive per epilogue warp
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
            // The residual tile of the tile RES_L2_AHEAD steps ahead is pulled
            // into L2 when a tile's loads start, so the epilogue's residual
            // reads hit L2 instead of waiting on HBM.
            constexpr int RES_L2_AHEAD = 2;
            auto prefetch_residual = [&](int tile_i) {
                if (!a.residual || tile_i >= a.num_tiles) return;
                const int pm0 = (tile_i / a.tiles_n) * S::BM;
                const int pn0 = (tile_i % a.tiles_n) * BN;
                const int rows = min(S::BM, a.M - pm0);
                const int cols = min(BN, a.N - pn0);
                const __nv_bfloat16 *base = a.residual + (size_t)pm0 * a.N + pn0;
                if (cols == a.N) {
                    bulk_prefetch_l2(base, (uint32_t)rows * (uint32_t)a.N * 2u);
                } else {
                    for (int r = 0; r < rows; ++r)
                        bulk_prefetch_l2(base + (size_t)r * a.N, (uint32_t)cols * 2u);
                }
            };
            for (int d = 0; d < RES_L2_AHEAD; ++d) prefetch_residual(blockIdx.x + d * gridDim.x);
            int it = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < a.num_tiles; tile += gridDim.x) {
                prefetch_residual(tile + RES_L2_AHEAD * gridDim.x);
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
        const int e = warp - 2;            // 0..7
        const int quarter = warp & 3;      // TMEM lanes (= tile rows) this warp may access
        const int half = e >> 2;           // takes chunks ci with ci % 2 == half
        constexpr int NCH = BN / 32;       // 32-column chunks per tile
        const uint32_t stg_out = sEpi + (uint32_t)e * S::EPI_WARP_BYTES;
        const uint32_t stg_res = stg_out + S::EPI_TILE;
        const bool has_res = a.residual != nullptr;
        // 64-byte swizzle of the 32x32 bf16 staging tiles: 16-byte piece c of row
        // r sits at piece c ^ ((r >> 1) & 3), so both the row-per-thread and
        // the coalesced access patterns below are free of bank conflicts.
        const uint32_t sw_own = ((uint32_t)lane >> 1) & 3u;
        // coalesced pattern: access k (0..3) covers rows 8k + lane/4, piece lane%4
        const int cl_row = lane >> 2, cl_piece = lane & 3;

        // The warp's chunk sequence: tiles blockIdx.x + i*gridDim.x, chunks
        // half, half+2, ... of each.  The residual of the next assignment is
        // loaded (coalesced) while the current one is processed.
        auto res_load = [&](int tile_i, int ci, uint4 (&r)[4]) {
#pragma unroll
            for (int k = 0; k < 4; ++k) r[k] = make_uint4(0u, 0u, 0u, 0u);
            if (tile_i >= a.num_tiles) return;
            const int rrow0 = (tile_i / a.tiles_n) * S::BM + quarter * 32;
            const int rcol = (tile_i % a.tiles_n) * BN + ci * 32 + cl_piece * 8;
            if (rcol >= a.N) return;
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int row = rrow0 + 8 * k + cl_row;
                if (row < a.M)
                    r[k] = __ldg(reinterpret_cast<const uint4 *>(a.residual + (size_t)row * a.N + rcol));
            }
        };
        auto advance = [&](int &tile_i, int &ci) {
            ci += 2;
            if (ci >= NCH) {
                ci = half;
                tile_i += gridDim.x;
            }
        };
        uint4 rcur[4];
        int pf_tile = blockIdx.x, pf_ci = half;  // assignment whose residual rcur holds
        if (has_res && half < NCH) res_load(pf_tile, pf_ci, rcur);
        int t = 0;
        for (int tile = blockIdx.x; tile < a.num_tiles; tile += gridDim.x, ++t) {
            const int buf = t & 1;
            const uint32_t aph = (uint32_t)(t >> 1) & 1u;
            if (!mbar_wait(tfull + 8u * buf, aph, abort_flag, a.err, kErrTimeoutEpilogue)) break;
            tc_fence_after();
            const int m0 = (tile / a.tiles_n) * S::BM;
            const int n0 = (tile % a.tiles_n) * BN;
            const int row0 = m0 + quarter * 32;
            const uint32_t tbase =
                tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * BN);
            if (half >= NCH) {  // no chunk for this warp in this tile (BN = 32)
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(tempty + 8u * buf);
                continue;
            }
#pragma unroll 1
            for (int ci = half; ci < NCH; ci += 2) {
                const int col0 = n0 + ci * 32;
                uint32_t v[32];
                tmem_ld_32cols_nowait(tbase + (uint32_t)(ci * 32), v);
                uint4 rnext[4];
                if (has_res) {
                    advance(pf_tile, pf_ci);
                    res_load(pf_tile, pf_ci, rnext);
                }
                tmem_ld_wait_regs(v);
                if (ci + 2 >= NCH) {  // this warp's last read of the accumulator
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(tempty + 8u * buf);
                }
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
                if (has_res) {
                    // coalesced registers -> swizzled staging -> this thread's row
                    __syncwarp();
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint32_t r = (uint32_t)(8 * k + cl_row);
                        const uint32_t addr =
                            stg_res + r * 64u + ((((uint32_t)cl_piece) ^ ((r >> 1) & 3u)) << 4);
                        asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr),
                                     "r"(rcur[k].x), "r"(rcur[k].y), "r"(rcur[k].z), "r"(rcur[k].w)
                                     : "memory");
                    }
                    __syncwarp();
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint4 r4;
                        const uint32_t addr = stg_res + (uint32_t)lane * 64u + (((uint32_t)q ^ sw_own) << 4);
                        asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                     : "=r"(r4.x), "=r"(r4.y), "=r"(r4.z), "=r"(r4.w)
                                     : "r"(addr)
                                     : "memory");
                        const uint32_t rr[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
                        for (int e2 = 0; e2 < 4; ++e2) {
                            f[8 * q + 2 * e2] += bf16lo(rr[e2]);
                            f[8 * q + 2 * e2 + 1] += bf16hi(rr[e2]);
                        }
                    }
#pragma unroll
                    for (int k = 0; k < 4; ++k) rcur[k] = rnext[k];
                }
#pragma unroll
                for (int j = 0; j < 32; ++j) f[j] = apply_act(f[j], a.act);
                // this thread's row -> swizzled staging -> coalesced global stores
                __syncwarp();
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint32_t w0 = pack_bf16x2(f[8 * q + 0], f[8 * q + 1]);
                    const uint32_t w1 = pack_bf16x2(f[8 * q + 2], f[8 * q + 3]);
                    const uint32_t w2 = pack_bf16x2(f[8 * q + 4], f[8 * q + 5]);
                    const uint32_t w3 = pack_bf16x2(f[8 * q + 6], f[8 * q + 7]);
                    const uint32_t addr = stg_out + (uint32_t)lane * 64u + (((uint32_t)q ^ sw_own) << 4);
                    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(w0),
                                 "r"(w1), "r"(w2), "r"(w3)
                                 : "memory");
                }
                __syncwarp();
                const int gcol = col0 + cl_piece * 8;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const uint32_t r = (uint32_t)(8 * k + cl_row);
                    const uint32_t addr =
                        stg_out + r * 64u + ((((uint32_t)cl_piece) ^ ((r >> 1) & 3u)) << 4);
                    uint4 o;
                    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                 : "=r"(o.x), "=r"(o.y), "=r"(o.z), "=r"(o.w)
                                 : "r"(addr)
                                 : "memory");
                    const int row = row0 + (int)r;
                    if (row < a.M && gcol < a.N)
                        *reinterpret_cast<uint4 *>(a.out + (size_t)row * a.N + gcol) = o;
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
    if (c.bn == BN_ && c.bk == BK_ && c.im2col == IM_) \
        return launch_t<BN_, BK_, IM_>(tmA, tmB, a, grid, st);
    BYOC_GEMM_CONFIGS(X)
#undef X
    return cudaErrorInvalidValue;
}

}  // namespace byoc
