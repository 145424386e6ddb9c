// dwpw.cu -- a depthwise 3x3 conv + BN + activation fused with the 1x1 conv
// + BN (+ residual add) (+ activation) that consumes it: the two composites
// of a MobileNetV2 inverted-residual tail merged into one region and run as
// one kernel.  Merging regions is what lets a backend keep intermediates on
// chip (Section 3.1.2 merges supported operators into one function; Section
// 3.3 hands the whole function to the code generator): here the depthwise
// output never reaches HBM.  CUDA cores compute it tile by tile straight into
// the tensor-core A operand in shared memory, and tcgen05.mma multiplies it by
// the pointwise weights, resident in shared memory, into TMEM.
//
// Tile: tr output rows x the full output width (tr * Wo <= 128 pixels = the
// MMA's M).  The depthwise channels are processed in chunks of 64 (one
// 128-byte swizzled operand row per pixel), each chunk one K step group of
// the pointwise GEMM.  Warp roles (704 threads):
//   warp 0      TMA: the pointwise weights once per CTA, then one input box
//               (halo rows and columns, 64 channels, zero outside the image)
//               per (tile, chunk) into a ring of up to four buffers (loads
//               of the next chunks stay in flight while one is computed);
//   warp 1      TMEM allocation; one elected lane issues the MMAs (M = 128,
//               N = n_pad, K = 16) of every chunk into one of two
//               accumulators;
//   warps 2-5   epilogue: TMEM -> registers, + bias (+ residual), activation,
//               bf16, stores (one pixel row per thread);
//   warps 6-21  depthwise: a lane owns a channel pair of the chunk (a warp
//               reads and writes a pixel's 64 channels as one 128-byte row)
//               and a warp computes blocks of BH x 4 output pixels with packed
//               two-lane fp32 FMAs (9 folded weight pairs in registers),
//               rounds to bf16,
//               applies the activation on the packed pair and writes the
//               result into the A buffer in the 128-byte-swizzled K-major
//               layout the MMA descriptor reads; then fences the writes to
//               the async proxy and releases the buffer to the MMA warp.
// Every wait is bounded (2 s): a role that gives up raises the CTA's abort
// flag, the others stop at their next wait, copies in flight are drained and
// TMEM is freed before the CTA exits.
#include "internal.h"
#include "ptx.cuh"

namespace byoc {

namespace {
constexpr int kDpDwWarps = 16;
constexpr int kDpFirstDwWarp = 6;
constexpr int kDpBW = 4;  // depthwise outputs per thread item: BH rows x four columns
}  // namespace

template <int STRIDE, int DWACT, int BH>
__global__ void __launch_bounds__(kDpThreads, 1)
    dwpw_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmB,
                const DwPwArgs a) {
    constexpr int IC = (kDpBW - 1) * STRIDE + 3;  // input columns under a BH x kDpBW block
    constexpr int IR = (BH - 1) * STRIDE + 3;     // input rows under it
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (base - raw);
    const uint32_t sB = base;
    const uint32_t sA = base + (uint32_t)a.a_off;    // 2 x kDpABytes
    const uint32_t sIn = base + (uint32_t)a.in_off;  // in_stages x in_pitch
    const uint32_t ctrl = base + (uint32_t)a.ctrl_off;
    const uint32_t in_full = ctrl, in_empty = ctrl + 8u * kDpMaxInStages;  // in_stages each
    const uint32_t a_full = ctrl + 16u * kDpMaxInStages, a_empty = a_full + 16u;
    const uint32_t acc_full = a_empty + 16u, acc_empty = acc_full + 16u, b_full = acc_empty + 16u;
    const uint32_t drain = b_full + 8u;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + a.ctrl_off + 192);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + a.ctrl_off + 196);
    const int NS = a.in_stages;
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int b = 0; b < kDpMaxInStages; ++b) {
            mbar_init(in_full + 8u * b, 1);             // producer + box bytes
            mbar_init(in_empty + 8u * b, kDpDwWarps);   // one arrive per depthwise warp
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(a_full + 8u * b, kDpDwWarps);     // one arrive per depthwise warp
            mbar_init(a_empty + 8u * b, 1);             // MMA commit
            mbar_init(acc_full + 8u * b, 1);            // MMA commit
            mbar_init(acc_empty + 8u * b, 4);           // one arrive per epilogue warp
        }
        mbar_init(b_full, 1);
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmX);
        tma_prefetch_desc(&tmB);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), (uint32_t)a.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    pdl_launch_dependents();
    pdl_wait();

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (elect_one()) {
            bool ok = true;
            // once per CTA: the 1x1 weights (MMA operand B) and the folded
            // depthwise weights and bias (read by the depthwise warps)
            mbar_arrive_expect_tx(b_full, (uint32_t)(a.b_bytes + 10 * a.C * 4));
            for (int cc = 0; cc < a.chunks; ++cc)
                tma_load_2d(sB + (uint32_t)(cc * a.n_pad * 128), &tmB, b_full, cc * kDpChunk, 0);
            bulk_load_1d(base + (uint32_t)a.w_off, a.dw_w, (uint32_t)(9 * a.C * 4), b_full);
            bulk_load_1d(base + (uint32_t)(a.w_off + 9 * a.C * 4), a.dw_b, (uint32_t)(a.C * 4), b_full);
            int j = 0, s = 0;
            uint32_t ph = 0;
            for (int tile = blockIdx.x; ok && tile < a.num_tiles; tile += gridDim.x) {
                const int n = tile / a.tiles_per_img;
                const int p0 = (tile - n * a.tiles_per_img) * a.tr;
                for (int cc = 0; cc < a.chunks; ++cc, ++j) {
                    if (!mbar_wait(in_empty + 8u * s, ph ^ 1u, abort_flag, a.err, kErrTimeoutProducer)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(in_full + 8u * s, (uint32_t)a.in_bytes);
                    tma_load_4d(sIn + (uint32_t)(s * a.in_pitch), &tmX, in_full + 8u * s, cc * kDpChunk,
                                -a.pad, p0 * STRIDE - a.pad, n);
                    if (++s == NS) {
                        s = 0;
                        ph ^= 1u;
                    }
                }
            }
            if (!ok) {
                // gave up: the weight load and the last input loads must land before exit
                mbar_wait_drain(b_full, 0u);
                for (int k = j - NS > 0 ? j - NS : 0; k < j; ++k)
                    mbar_wait_drain(in_full + 8u * (k % NS), (uint32_t)(k / NS) & 1u);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (elect_one()) {
            auto wait = [&](uint32_t bar, uint32_t parity) -> bool {
                return mbar_wait(bar, parity, abort_flag, a.err, kErrTimeoutMma);
            };
            bool ok = wait(b_full, 0u);
            const uint32_t idesc = make_idesc_bf16(kGemmBM, a.n_pad);
            const uint64_t adesc0 = make_smem_desc(sA, 128);
            const uint64_t bdesc0 = make_smem_desc(sB, 128);
            int j = 0, t = 0;
            for (int tile = blockIdx.x; ok && tile < a.num_tiles; tile += gridDim.x, ++t) {
                const int acc = t & 1;
                if (!wait(acc_empty + 8u * acc, ((uint32_t)(t >> 1) & 1u) ^ 1u)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * a.acc_stride);
                uint32_t accumulate = 0u;
                for (int cc = 0; cc < a.chunks; ++cc, ++j) {
                    const int b = j & 1;
                    if (!wait(a_full + 8u * b, (uint32_t)(j >> 1) & 1u)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();  // A was written by other threads (generic proxy, fenced)
                    const int ch = a.C - cc * kDpChunk < kDpChunk ? a.C - cc * kDpChunk : kDpChunk;
                    const uint64_t ad = adesc0 + (uint64_t)((uint32_t)(b * kDpABytes) >> 4);
                    const uint64_t bd = bdesc0 + (uint64_t)((uint32_t)(cc * a.n_pad * 128) >> 4);
                    for (int k = 0; k < ch / 16; ++k)
                        mma_bf16_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                                    accumulate | (uint32_t)k);
                    accumulate = 1u;
                    mma_commit(a_empty + 8u * b);  // frees the A buffer
                }
                if (!ok) break;
                mma_commit(acc_full + 8u * acc);
            }
            // every issued MMA must finish before TMEM is freed
            mma_commit(drain);
            mbar_wait_drain(drain, 0u);
        }
        __syncwarp();
    } else if (warp < kDpFirstDwWarp) {
        // ------------------------------------------------------------ epilogue
        const int quarter = warp & 3;  // TMEM lanes this warp may read
        const int m = quarter * 32 + lane;
        int t = 0;
        for (int tile = blockIdx.x; tile < a.num_tiles; tile += gridDim.x, ++t) {
            const int acc = t & 1;
            if (!mbar_wait(acc_full + 8u * acc, (uint32_t)(t >> 1) & 1u, abort_flag, a.err,
                           kErrTimeoutEpilogue))
                break;
            tc_fence_after();
            const int n = tile / a.tiles_per_img;
            const int p0 = (tile - n * a.tiles_per_img) * a.tr;
            const int r = m / a.Wo;
            const int q = m - r * a.Wo;
            const bool valid = r < a.tr && p0 + r < a.Ho;
            const size_t pix = ((size_t)n * a.Ho + (size_t)(p0 + r)) * a.Wo + q;
            const uint32_t tb = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * a.acc_stride);
            for (int c0 = 0; c0 < a.n_pad; c0 += 32) {
                uint32_t v[32];
                tmem_ld_32cols(tb + (uint32_t)c0, v);
                if (c0 + 32 >= a.n_pad) {  // this warp's last read of the accumulator
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(acc_empty + 8u * acc);
                }
                if (!valid) continue;
#pragma unroll
                for (int g = 0; g < 4; ++g) {
                    const int c = c0 + 8 * g;
                    if (c >= a.Cout) break;
                    const float4 b0 = __ldg(reinterpret_cast<const float4 *>(a.pw_b + c));
                    const float4 b1 = __ldg(reinterpret_cast<const float4 *>(a.pw_b + c + 4));
                    float f[8] = {__uint_as_float(v[8 * g]) + b0.x,     __uint_as_float(v[8 * g + 1]) + b0.y,
                                  __uint_as_float(v[8 * g + 2]) + b0.z, __uint_as_float(v[8 * g + 3]) + b0.w,
                                  __uint_as_float(v[8 * g + 4]) + b1.x, __uint_as_float(v[8 * g + 5]) + b1.y,
                                  __uint_as_float(v[8 * g + 6]) + b1.z, __uint_as_float(v[8 * g + 7]) + b1.w};
                    if (a.residual) {
                        const uint4 rr = __ldg(reinterpret_cast<const uint4 *>(a.residual + pix * a.Cout + c));
                        const uint32_t rw[4] = {rr.x, rr.y, rr.z, rr.w};
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            f[2 * e] += bf16lo(rw[e]);
                            f[2 * e + 1] += bf16hi(rw[e]);
                        }
                    }
                    if (a.act == kActRelu || a.act == kActRelu6) {
#pragma unroll
                        for (int e = 0; e < 8; ++e) {
                            f[e] = fmaxf(f[e], 0.0f);
                            if (a.act == kActRelu6) f[e] = fminf(f[e], 6.0f);
                        }
                    }
                    uint4 o;
                    o.x = pack_bf16x2(f[0], f[1]);
                    o.y = pack_bf16x2(f[2], f[3]);
                    o.z = pack_bf16x2(f[4], f[5]);
                    o.w = pack_bf16x2(f[6], f[7]);
                    *reinterpret_cast<uint4 *>(a.out + pix * a.Cout + c) = o;
                }
            }
        }
    } else {
        // ------------------------------------------------------------ depthwise
        // lane = channel pair of the chunk (a warp covers the chunk's 64
        // channels of a pixel: 128-byte loads and stores); a warp computes one
        // BH x kDpBW block of output pixels at a time
        const int dwarp = warp - kDpFirstDwWarp;
        const int bcols = (a.Wo + kDpBW - 1) / kDpBW;
        const int blocks = ((a.tr + BH - 1) / BH) * bcols;
        const uint32_t col_step = kDpChunk * 2u;  // bytes per input column of a box
        const uint32_t row_step = (uint32_t)a.in_cols * col_step;
        uint64_t w[9];
        uint64_t bias2 = 0;
        int j = 0, s = 0;
        uint32_t sph = 0;
        // the depthwise weights arrive with the 1x1 weights
        bool ok = __all_sync(0xffffffffu, mbar_wait(b_full, 0u, abort_flag, a.err, kErrTimeoutEpilogue));
        const float *sw = reinterpret_cast<const float *>(smem + a.w_off);  // [9][C], then bias [C]
        for (int tile = blockIdx.x; ok && tile < a.num_tiles; tile += gridDim.x) {
            const int n = tile / a.tiles_per_img;
            const int p0 = (tile - n * a.tiles_per_img) * a.tr;
            const int nrows = a.Ho - p0 < a.tr ? a.Ho - p0 : a.tr;
            for (int cc = 0; cc < a.chunks; ++cc, ++j) {
                const int b = j & 1;  // A buffer
                const uint32_t ph = (uint32_t)(j >> 1) & 1u;
                ok = mbar_wait(in_full + 8u * s, sph, abort_flag, a.err, kErrTimeoutEpilogue) &&
                     mbar_wait(a_empty + 8u * b, ph ^ 1u, abort_flag, a.err, kErrTimeoutEpilogue);
                if (!__all_sync(0xffffffffu, ok)) {
                    ok = false;
                    break;
                }
                const int c = cc * kDpChunk + 2 * lane;  // this thread's channel pair
                const bool live = c < a.C;
                if (live) {
#pragma unroll
                    for (int tap = 0; tap < 9; ++tap) {
                        const float2 wq = *reinterpret_cast<const float2 *>(sw + tap * a.C + c);
                        w[tap] = f32x2(wq.x, wq.y);
                    }
                    const float2 bq = *reinterpret_cast<const float2 *>(sw + 9 * a.C + c);
                    bias2 = f32x2(bq.x, bq.y);
                }
                const uint8_t *in = smem + (a.in_off + s * a.in_pitch) + 4 * lane;
                uint8_t *ab = smem + (a.a_off + b * kDpABytes);
                for (int blk = dwarp; live && blk < blocks; blk += kDpDwWarps) {
                    const int r0 = (blk / bcols) * BH;
                    const int qb = (blk - (r0 / BH) * bcols) * kDpBW;
                    if (r0 >= nrows) continue;
                    uint64_t acc[BH][kDpBW];
#pragma unroll
                    for (int oy = 0; oy < BH; ++oy)
#pragma unroll
                        for (int ox = 0; ox < kDpBW; ++ox) acc[oy][ox] = bias2;
                    const uint8_t *sblk = in + (size_t)(r0 * STRIDE) * row_step + (size_t)(qb * STRIDE) * col_step;
#pragma unroll
                    for (int ir = 0; ir < IR; ++ir)
#pragma unroll
                        for (int ic = 0; ic < IC; ++ic) {
                            const uint32_t u =
                                *reinterpret_cast<const uint32_t *>(sblk + (size_t)ir * row_step + (size_t)ic * col_step);
                            const uint64_t x = f32x2_of_bf16x2(u);
#pragma unroll
                            for (int oy = 0; oy < BH; ++oy)
#pragma unroll
                                for (int ox = 0; ox < kDpBW; ++ox) {
                                    const int dy = ir - oy * STRIDE, dx = ic - ox * STRIDE;
                                    if (dy < 0 || dy > 2 || dx < 0 || dx > 2) continue;
                                    fma2(acc[oy][ox], x, w[dy * 3 + dx]);
                                }
                        }
#pragma unroll
                    for (int oy = 0; oy < BH; ++oy) {
                        if (r0 + oy >= nrows) break;
#pragma unroll
                        for (int ox = 0; ox < kDpBW; ++ox) {
                            const int q = qb + ox;
                            if (q >= a.Wo) break;
                            const int mm = (r0 + oy) * a.Wo + q;  // A row = tile pixel
                            // 128-byte swizzle: 16-byte piece p of row mm sits at p ^ (mm & 7)
                            const uint32_t off = (uint32_t)mm * 128u +
                                                 ((((uint32_t)lane >> 2) ^ ((uint32_t)mm & 7u)) << 4) +
                                                 (((uint32_t)lane & 3u) << 2);
                            *reinterpret_cast<uint32_t *>(ab + off) =
                                dw_act2<DWACT>(lane0(acc[oy][ox]), lane1(acc[oy][ox]));
                        }
                    }
                }
                fence_proxy_async_smem();  // A written by the generic proxy, read by the MMAs
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive(in_empty + 8u * s);
                    mbar_arrive(a_full + 8u * b);
                }
                if (++s == NS) {
                    s = 0;
                    sph ^= 1u;
                }
            }
        }
    }
    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, (uint32_t)a.tmem_cols);
    }
}

// ------------------------------------------------------------ host side

bool dwpw_plan(DwPwArgs &a, int num_sms) {
    if (a.C % 16 || a.Cout % 8 || a.pad != 1 || (a.stride != 1 && a.stride != 2)) return false;
    if (a.Wo > kGemmBM) return false;
    a.n_pad = (a.Cout + 15) / 16 * 16;
    if (a.n_pad > 256) return false;
    a.chunks = (a.C + kDpChunk - 1) / kDpChunk;
    a.b_bytes = a.chunks * a.n_pad * 128;
    if (a.b_bytes > kDpMaxBBytes) return false;
    a.acc_stride = (a.n_pad + 31) / 32 * 32;
    int cols = 32;
    while (cols < 2 * a.acc_stride) cols *= 2;
    a.tmem_cols = cols;
    a.w_off = (a.b_bytes + 1023) / 1024 * 1024;         // depthwise weights + bias: 10 C floats
    a.a_off = (a.w_off + 10 * a.C * 4 + 1023) / 1024 * 1024;
    a.in_off = a.a_off + 2 * kDpABytes;
    const int budget = (kDpSmemMax - 1024 - a.in_off - 256) / 2;  // per input buffer, two at least
    const int bcols = (a.Wo + kDpBW - 1) / kDpBW;
    a.in_cols = (bcols * kDpBW - 1) * a.stride + 3;
    if (a.in_cols > 256) return false;
    // rows of the input box: the tile's rows rounded up to whole BH-row blocks
    auto rows_in = [&](int t) {
        const int bh = t >= 2 ? 2 : 1;
        return ((t + bh - 1) / bh * bh - 1) * a.stride + 3;
    };
    int tr = kGemmBM / a.Wo < a.Ho ? kGemmBM / a.Wo : a.Ho;
    while (tr > 1 && rows_in(tr) * a.in_cols * kDpChunk * 2 > budget) --tr;
    a.tr = tr;
    a.bh = tr >= 2 ? 2 : 1;
    a.in_rows = rows_in(tr);
    a.in_bytes = a.in_rows * a.in_cols * kDpChunk * 2;
    if (a.in_bytes > budget || a.in_rows > 256) return false;
    a.in_pitch = (a.in_bytes + 1023) / 1024 * 1024;
    a.in_stages = (kDpSmemMax - 1024 - a.in_off - 256) / a.in_pitch;
    if (a.in_stages > kDpMaxInStages) a.in_stages = kDpMaxInStages;
    a.ctrl_off = a.in_off + a.in_stages * a.in_pitch;
    a.smem_bytes = 1024 + a.ctrl_off + 256;
    a.tiles_per_img = (a.Ho + tr - 1) / tr;
    a.num_tiles = a.N * a.tiles_per_img;
    (void)num_sms;
    return a.smem_bytes <= kDpSmemMax;
}

template <int STRIDE, int BH>
static auto dwpw_kernel_for(int act) -> decltype(&dwpw_kernel<1, kActNone, 1>) {
    switch (act) {
        case kActRelu: return dwpw_kernel<STRIDE, kActRelu, BH>;
        case kActRelu6: return dwpw_kernel<STRIDE, kActRelu6, BH>;
        default: return dwpw_kernel<STRIDE, kActNone, BH>;
    }
}

static auto dwpw_kernel_of(const DwPwArgs &a) -> decltype(&dwpw_kernel<1, kActNone, 1>) {
    if (a.bh == 2) return a.stride == 1 ? dwpw_kernel_for<1, 2>(a.dw_act) : dwpw_kernel_for<2, 2>(a.dw_act);
    return a.stride == 1 ? dwpw_kernel_for<1, 1>(a.dw_act) : dwpw_kernel_for<2, 1>(a.dw_act);
}

cudaError_t dwpw_prepare(const DwPwArgs &a) {
    return cudaFuncSetAttribute(dwpw_kernel_of(a), cudaFuncAttributeMaxDynamicSharedMemorySize, kDpSmemMax);
}

cudaError_t launch_dwpw(const CUtensorMap &tmX, const CUtensorMap &tmB, const DwPwArgs &a, int grid,
                        cudaStream_t st) {
    return launch_pdl(dwpw_kernel_of(a), dim3(grid), dim3(kDpThreads), (size_t)a.smem_bytes, st, tmX, tmB, a);
}

}  // namespace byoc
