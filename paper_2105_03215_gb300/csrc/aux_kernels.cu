// aux_kernels.cu -- the bandwidth-bound kernels of the offloaded path:
//   * depthwise 3x3 conv + folded BN + activation (MobileNetV2 composite),
//   * the layout transform of a stride-2 stem over <= 4 channels: the image
//     with 4 channels and zero padding, read by the stem's GEMM as pixel
//     pairs (a layout transformation node inserted at a region boundary,
//     Section 3.2), and the NCHW fp32 -> NHWC bf16 boundary transform,
//   * the host-graph operators of ResNet-50 (max pool, global average pool),
//     which the paper leaves on the host (Section 3.4, CUDA as the host).
// All tensors are bf16 NHWC; every thread moves 8 channels (16 bytes) at a
// time so that a warp's accesses are contiguous along C.
#include <algorithm>

#include "internal.h"
#include "ptx.cuh"

namespace byoc {

__device__ __forceinline__ void unpack8(const uint4 &v, float (&f)[8]) {
    f[0] = bf16lo(v.x); f[1] = bf16hi(v.x);
    f[2] = bf16lo(v.y); f[3] = bf16hi(v.y);
    f[4] = bf16lo(v.z); f[5] = bf16hi(v.z);
    f[6] = bf16lo(v.w); f[7] = bf16hi(v.w);
}

__device__ __forceinline__ uint4 pack8(const float (&f)[8]) {
    uint4 o;
    o.x = pack_bf16x2(f[0], f[1]);
    o.y = pack_bf16x2(f[2], f[3]);
    o.z = pack_bf16x2(f[4], f[5]);
    o.w = pack_bf16x2(f[6], f[7]);
    return o;
}

__device__ __forceinline__ uint4 ldg_v4(const void *p) {
    return __ldg(reinterpret_cast<const uint4 *>(p));
}

// ------------------------------------------------------------ depthwise 3x3
//
// Thread <-> (image n, output column q, 4-channel group, ROWS consecutive
// output rows).  The channel group varies fastest across threads, so a warp
// reads and writes one contiguous 256-byte run of an image row per access.
// One persistent CTA per SM walks the tiles (chunk slowest, so a CTA mostly
// keeps one channel chunk and its weights).  Thread t owns the 4-channel
// vector v = t % V (V = cc / 4), whose 9 x 4 folded weights stay in
// registers, and computes blocks of kDwBlockH x kDwBlockW outputs (blocks
// t / V + k * lanes): each input vector under a block is read from shared
// memory once (8 bytes), unpacked once and fed to every output of the block
// that uses it, with packed two-lane fp32 FMAs.  A 4 x 2 block reads 24 input
// vectors for 8 outputs at stride 1 and keeps a thread under 128 registers,
// so 16 warps per SM overlap the load, unpack and FMA latencies.  The
// activation is applied to the packed bf16 pairs (exact: rounding is
// monotonic and 0 and 6 are bf16 values).  The next tile's box loads (TMA)
// while this one is computed.
template <int STRIDE, int ACT>
__global__ void __launch_bounds__(kDwMaxThreads, 1)
    dwconv3x3_kernel(const __grid_constant__ CUtensorMap tmX, const DwArgs a) {
    constexpr int BH = kDwBlockH, BW = kDwBlockW;      // outputs per thread block
    constexpr int IR = (BH - 1) * STRIDE + 3;          // input rows under a block
    constexpr int IC = (BW - 1) * STRIDE + 3;          // input columns under a block
    extern __shared__ __align__(128) uint8_t smem_dw[];
    const uint32_t raw = smem_u32(smem_dw);
    const uint32_t base = (raw + 127u) & ~127u;
    uint8_t *sbase = smem_dw + (base - raw);
    const uint32_t bars = base + 2u * (uint32_t)a.buf_bytes;  // 2 full barriers
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sbase + 2 * a.buf_bytes + 16);
    const int tid = threadIdx.x;
    const int V = a.cc >> 2;
    const int lanes = a.threads / V;
    const int v = tid % V;
    const int g = tid / V;
    if (tid == 0) {
        mbar_init(bars, 1);
        mbar_init(bars + 8u, 1);
        *abort_flag = 0;
        fence_barrier_init();
        tma_prefetch_desc(&tmX);
    }
    __syncthreads();
    pdl_launch_dependents();
    pdl_wait();
    const int per_chunk = a.N * a.tiles_h * a.tiles_w;
    auto issue = [&](int tile, int b) {
        const int ch = tile / per_chunk;
        int r = tile - ch * per_chunk;
        const int n = r / (a.tiles_h * a.tiles_w);
        r -= n * a.tiles_h * a.tiles_w;
        const int ph = r / a.tiles_w;
        const int pw = r - ph * a.tiles_w;
        const uint32_t bar = bars + 8u * (uint32_t)b;
        mbar_arrive_expect_tx(bar, (uint32_t)(a.in_rows * a.in_cols * a.cc * 2));
        tma_load_4d(base + (uint32_t)(b * a.buf_bytes), &tmX, bar, ch * a.cc,
                    pw * a.tw * STRIDE - a.pad, ph * a.th * STRIDE - a.pad, n);
    };
    if (tid == 0) {
        if ((int)blockIdx.x < a.num_tiles) issue(blockIdx.x, 0);
        if ((int)(blockIdx.x + gridDim.x) < a.num_tiles) issue(blockIdx.x + gridDim.x, 1);
    }
    uint64_t w[9][2];  // folded weights, channel pairs
    float bias[4];
    int wc = -1;       // channel of the weights in registers
    const int bcols = a.tw / BW, blocks = (a.th / BH) * bcols;
    int i = 0;
    for (int tile = blockIdx.x; tile < a.num_tiles; tile += gridDim.x, ++i) {
        const int b = i & 1;
        const bool ok = mbar_wait(bars + 8u * (uint32_t)b, (uint32_t)(i >> 1) & 1u, abort_flag, a.err,
                                  kErrTimeoutProducer);
        if (__syncthreads_or(!ok)) {
            // gave up: let this CTA's copies in flight land before exiting
            if (tid == 0)
                for (int k = 0; k < 2; ++k)
                    if (tile + k * (int)gridDim.x < a.num_tiles)
                        mbar_wait_drain(bars + 8u * (uint32_t)((i + k) & 1), (uint32_t)((i + k) >> 1) & 1u);
            break;
        }
        const int ch = tile / per_chunk;
        int r = tile - ch * per_chunk;
        const int n = r / (a.tiles_h * a.tiles_w);
        r -= n * a.tiles_h * a.tiles_w;
        const int ph = r / a.tiles_w;
        const int pw = r - ph * a.tiles_w;
        const int c = ch * a.cc + v * 4;  // this thread's first channel
        if (c < a.C && c != wc) {
#pragma unroll
            for (int tap = 0; tap < 9; ++tap) {
                const float4 q = __ldg(reinterpret_cast<const float4 *>(a.w + (size_t)tap * a.C + c));
                w[tap][0] = f32x2(q.x, q.y);
                w[tap][1] = f32x2(q.z, q.w);
            }
            const float4 q = __ldg(reinterpret_cast<const float4 *>(a.bias + c));
            bias[0] = q.x; bias[1] = q.y; bias[2] = q.z; bias[3] = q.w;
            wc = c;
        }
        if (c < a.C) {
            // plain loads (not volatile asm), so the compiler can hoist them
            // ahead of the FMAs; the barrier wait above orders them after the copy
            const uint8_t *buf = sbase + (size_t)b * a.buf_bytes + (size_t)v * 8;
            const uint32_t col_step = (uint32_t)a.cc * 2u;
            const uint32_t row_step = (uint32_t)a.in_cols * col_step;
            const int p0 = ph * a.th, q0 = pw * a.tw;
            __nv_bfloat16 *yimg = a.y + (size_t)n * a.Ho * a.Wo * a.C + c;
            for (int blk = g; blk < blocks; blk += lanes) {
                const int br = blk / bcols;
                const int bc = blk - br * bcols;
                uint64_t acc[BH][BW][2];
#pragma unroll
                for (int oy = 0; oy < BH; ++oy)
#pragma unroll
                    for (int ox = 0; ox < BW; ++ox) {
                        acc[oy][ox][0] = f32x2(bias[0], bias[1]);
                        acc[oy][ox][1] = f32x2(bias[2], bias[3]);
                    }
                const uint8_t *sblk = buf + (size_t)(br * BH * STRIDE) * row_step +
                                      (size_t)(bc * BW * STRIDE) * col_step;
#pragma unroll
                for (int ir = 0; ir < IR; ++ir)
#pragma unroll
                    for (int ic = 0; ic < IC; ++ic) {
                        const uint2 u = *reinterpret_cast<const uint2 *>(
                            sblk + (size_t)ir * row_step + (size_t)ic * col_step);
                        const uint64_t x0 = f32x2_of_bf16x2(u.x), x1 = f32x2_of_bf16x2(u.y);
#pragma unroll
                        for (int oy = 0; oy < BH; ++oy)
#pragma unroll
                            for (int ox = 0; ox < BW; ++ox) {
                                const int dy = ir - oy * STRIDE, dx = ic - ox * STRIDE;
                                if (dy < 0 || dy > 2 || dx < 0 || dx > 2) continue;
                                fma2(acc[oy][ox][0], x0, w[dy * 3 + dx][0]);
                                fma2(acc[oy][ox][1], x1, w[dy * 3 + dx][1]);
                            }
                    }
                const int pb = p0 + br * BH, qb = q0 + bc * BW;
                __nv_bfloat16 *yb = yimg + ((size_t)pb * a.Wo + qb) * a.C;
#pragma unroll
                for (int oy = 0; oy < BH; ++oy) {
                    if (pb + oy >= a.Ho) break;
#pragma unroll
                    for (int ox = 0; ox < BW; ++ox) {
                        if (qb + ox >= a.Wo) break;
                        uint2 o;
                        o.x = dw_act2<ACT>(lane0(acc[oy][ox][0]), lane1(acc[oy][ox][0]));
                        o.y = dw_act2<ACT>(lane0(acc[oy][ox][1]), lane1(acc[oy][ox][1]));
                        *reinterpret_cast<uint2 *>(yb + ((size_t)oy * a.Wo + ox) * a.C) = o;
                    }
                }
            }
        }
        __syncthreads();  // buffer b consumed
        if (tid == 0 && tile + 2 * (int)gridDim.x < a.num_tiles) issue(tile + 2 * (int)gridDim.x, b);
    }
}

size_t dw_smem_bytes(const DwArgs &a) { return 128 + 2 * (size_t)a.buf_bytes + 64; }

bool dw_plan(DwArgs &a, int num_sms) {
    if (a.C % 8 || (a.stride != 1 && a.stride != 2)) return false;
    a.chunks = (a.C + 255) / 256;
    a.cc = ((a.C + a.chunks - 1) / a.chunks + 7) / 8 * 8;
    const int V = a.cc / 4;
    const int lanes = kDwMaxThreads / V;
    a.threads = V * lanes;
    // Tiles are whole kDwBlockH x kDwBlockW output blocks.  Full output width
    // (rounded up to the block) when its input columns fit one box (<= 256).
    constexpr int B = kDwBlockH, BW = kDwBlockW;
    const int tw_max = ((256 - 3) / a.stride + 1) / BW * BW;
    const size_t budget = kDwBufBudget;
    auto rows_in = [&](int th) { return (th - 1) * a.stride + 3; };
    // Narrower column tiles where even the shortest row tile of the full
    // width would overflow one buffer (wide rows of many channels).
    a.tw = std::min((a.Wo + BW - 1) / BW * BW, tw_max);
    while (a.tw > BW && (size_t)rows_in(B) * ((a.tw - 1) * a.stride + 3) * a.cc * 2 > budget)
        a.tw -= BW;
    a.tiles_w = (a.Wo + a.tw - 1) / a.tw;
    a.in_cols = (a.tw - 1) * a.stride + 3;
    const size_t row_bytes = (size_t)a.in_cols * a.cc * 2;
    const int ho_blocks = (a.Ho + B - 1) / B * B;
    int th = B;
    while (th + B <= ho_blocks && (size_t)rows_in(th + B) * row_bytes <= budget && rows_in(th + B) <= 256)
        th += B;
    // fewer rows per tile while there would be under two tiles per SM
    while (th > B && (long long)a.chunks * a.N * ((a.Ho + th - 1) / th) * a.tiles_w < 2ll * num_sms)
        th -= B;
    a.th = th;
    a.in_rows = rows_in(th);
    if ((size_t)a.in_rows * row_bytes > budget || a.in_rows > 256) return false;
    a.tiles_h = (a.Ho + th - 1) / th;
    a.num_tiles = a.chunks * a.N * a.tiles_h * a.tiles_w;
    a.buf_bytes = (int)(((size_t)a.in_rows * row_bytes + 127) / 128 * 128);
    return true;
}

template <int STRIDE>
static auto dw_kernel_for(int act) -> decltype(&dwconv3x3_kernel<1, kActNone>) {
    switch (act) {
        case kActRelu: return dwconv3x3_kernel<STRIDE, kActRelu>;
        case kActRelu6: return dwconv3x3_kernel<STRIDE, kActRelu6>;
        case kActGelu: return dwconv3x3_kernel<STRIDE, kActGelu>;
        default: return dwconv3x3_kernel<STRIDE, kActNone>;
    }
}

static auto dw_kernel(const DwArgs &a) -> decltype(&dwconv3x3_kernel<1, kActNone>) {
    return a.stride == 1 ? dw_kernel_for<1>(a.act) : dw_kernel_for<2>(a.act);
}

cudaError_t dw_prepare(const DwArgs &a) {
    DwArgs largest = a;
    largest.buf_bytes = (int)kDwBufBudget;
    return cudaFuncSetAttribute(dw_kernel(a), cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)dw_smem_bytes(largest));
}

cudaError_t launch_dwconv(const CUtensorMap &tmX, const DwArgs &a, int grid, cudaStream_t st) {
    return launch_pdl(dw_kernel(a), dim3(grid), dim3(a.threads), dw_smem_bytes(a), st, tmX, a);
}

// ------------------------------------------------------------ stem input layout
// xq[n, u, v, c] = x[n, u - pad, v - pad, c] for c < C inside x, else 0 (see
// StemArgs).  Block (u-block, n): kStemRows rows of xq.  The input rows under
// them are staged in shared memory first -- 16-byte loads when a row is a
// whole number of 16-byte pieces, all of a block's loads in flight at once,
// since the transform is bound by memory latency -- then each thread writes
// 16-byte pixel pairs (coalesced across the warp).  C is a template parameter
// so that the pair assembly unrolls.
constexpr int kStemRows = 8;

template <int C>
__global__ void __launch_bounds__(256) stem_layout_kernel(const StemArgs a, int vec) {
    pdl_launch_dependents();
    pdl_wait();
    extern __shared__ __align__(16) unsigned short srow[];  // [kStemRows][W * C]
    const int n = blockIdx.y;
    const int u0 = blockIdx.x * kStemRows;
    const int row_elems = a.W * C;
    const unsigned short *xs = reinterpret_cast<const unsigned short *>(a.x) + (size_t)n * a.H * row_elems;
    if (vec) {
        const int pieces = row_elems >> 3;
        for (int i = threadIdx.x; i < kStemRows * pieces; i += blockDim.x) {
            const int r = i / pieces, q = i - r * pieces;
            const int h = u0 + r - a.pad;
            if (u0 + r < a.Hq && h >= 0 && h < a.H)
                reinterpret_cast<uint4 *>(srow + (size_t)r * row_elems)[q] =
                    __ldg(reinterpret_cast<const uint4 *>(xs + (size_t)h * row_elems) + q);
        }
    } else {
        for (int i = threadIdx.x; i < kStemRows * row_elems; i += blockDim.x) {
            const int r = i / row_elems, q = i - r * row_elems;
            const int h = u0 + r - a.pad;
            if (u0 + r < a.Hq && h >= 0 && h < a.H) srow[(size_t)r * row_elems + q] = __ldg(xs + (size_t)h * row_elems + q);
        }
    }
    __syncthreads();
    const int pairs = a.Wq >> 1;
    for (int i = threadIdx.x; i < kStemRows * pairs; i += blockDim.x) {
        const int r = i / pairs, j = i - r * pairs;
        const int u = u0 + r;
        if (u >= a.Hq) break;  // i grows with r: the rest of this thread's items are past Hq too
        const int h = u - a.pad;
        const bool row_in = h >= 0 && h < a.H;
        const unsigned short *sr = srow + (size_t)r * row_elems;
        uint32_t v[8];
#pragma unroll
        for (int dx = 0; dx < 2; ++dx) {
            const int w = 2 * j + dx - a.pad;
            const bool in = row_in && w >= 0 && w < a.W;
#pragma unroll
            for (int c = 0; c < 4; ++c) v[dx * 4 + c] = (in && c < C) ? (uint32_t)sr[w * C + c] : 0u;
        }
        reinterpret_cast<uint4 *>(a.xq + ((size_t)n * a.Hq + u) * a.Wq * 4)[j] =
            make_uint4(v[0] | v[1] << 16, v[2] | v[3] << 16, v[4] | v[5] << 16, v[6] | v[7] << 16);
    }
}

size_t stem_layout_smem_bytes(const StemArgs &a) { return (size_t)kStemRows * a.W * a.C * 2; }

cudaError_t launch_stem_layout(const StemArgs &a, cudaStream_t st) {
    const size_t smem = stem_layout_smem_bytes(a);
    if (a.Hq < 1 || a.N < 1 || a.N > 65535 || (a.Wq & 1) || a.Wq < 2 || a.C < 1 || a.C > 4 ||
        smem > kStemLayoutMaxSmem)
        return cudaErrorInvalidValue;
    // 16-byte staging loads when every input row starts on a 16-byte boundary
    const int vec = (a.W * a.C) % 8 == 0 && (reinterpret_cast<uintptr_t>(a.x) & 15) == 0;
    const dim3 grid((unsigned)((a.Hq + kStemRows - 1) / kStemRows), (unsigned)a.N);
    switch (a.C) {
        case 1: return launch_pdl(stem_layout_kernel<1>, grid, dim3(256), smem, st, a, vec);
        case 2: return launch_pdl(stem_layout_kernel<2>, grid, dim3(256), smem, st, a, vec);
        case 3: return launch_pdl(stem_layout_kernel<3>, grid, dim3(256), smem, st, a, vec);
        default: return launch_pdl(stem_layout_kernel<4>, grid, dim3(256), smem, st, a, vec);
    }
}

// ------------------------------------------------------------ boundary layout transform
// y[n, h, w, c] = bf16_rne(x[n, c, h, w]) for c < C, 0 for C <= c < Cp: the
// NCHW fp32 layout of the framework side to the NHWC bf16 layout the regions
// use (a layout transformation at a region boundary, Section 3.2).  Block
// (row group, n) converts `rows` image rows: it reads C planes' rows of W
// floats (coalesced along w), stages the rows x W x Cp bf16 output in shared
// memory and writes it with 16-byte stores (output rows of one image are
// contiguous).  HBM-bound: 4 C + 2 Cp bytes per pixel.
__global__ void __launch_bounds__(256) nchw_to_nhwc_kernel(const float *x, __nv_bfloat16 *y, int C, int H,
                                                           int W, int Cp, int rows) {
    pdl_launch_dependents();
    pdl_wait();
    extern __shared__ __align__(16) unsigned short sxf[];
    const int n = blockIdx.y;
    const int h0 = blockIdx.x * rows;
    const int nr = H - h0 < rows ? H - h0 : rows;
    const size_t plane = (size_t)H * W;
    const float *xn = x + (size_t)n * C * plane + (size_t)h0 * W;
    const int per_row = W * Cp;
    const int elems = nr * per_row;
    if (Cp > C)  // padded channels are zero
        for (int i = threadIdx.x; i < elems; i += blockDim.x) sxf[i] = 0;
    __syncthreads();
    // the nr rows of one plane are one contiguous run of nr * W floats
    const int run = nr * W;
    if ((W & 3) == 0) {
        const int run4 = run >> 2;
        for (int c = 0; c < C; ++c) {
            const float4 *src = reinterpret_cast<const float4 *>(xn + (size_t)c * plane);
#pragma unroll 4
            for (int i = threadIdx.x; i < run4; i += blockDim.x) {
                const float4 v = __ldg(src + i);
                unsigned short *d = sxf + (size_t)(4 * i) * Cp + c;  // pixel 4i of the run
                __nv_bfloat16 b0 = __float2bfloat16_rn(v.x), b1 = __float2bfloat16_rn(v.y);
                __nv_bfloat16 b2 = __float2bfloat16_rn(v.z), b3 = __float2bfloat16_rn(v.w);
                d[0] = *reinterpret_cast<unsigned short *>(&b0);
                d[Cp] = *reinterpret_cast<unsigned short *>(&b1);
                d[2 * Cp] = *reinterpret_cast<unsigned short *>(&b2);
                d[3 * Cp] = *reinterpret_cast<unsigned short *>(&b3);
            }
        }
    } else {
        for (int c = 0; c < C; ++c) {
            const float *src = xn + (size_t)c * plane;
            for (int i = threadIdx.x; i < run; i += blockDim.x) {
                __nv_bfloat16 b = __float2bfloat16_rn(__ldg(src + i));
                sxf[(size_t)i * Cp + c] = *reinterpret_cast<unsigned short *>(&b);
            }
        }
    }
    __syncthreads();
    unsigned short *yo = reinterpret_cast<unsigned short *>(y) + ((size_t)n * H + h0) * per_row;
    if ((per_row & 7) == 0) {  // rows of 16-byte multiples: the run starts 16-byte aligned
        const uint4 *src = reinterpret_cast<const uint4 *>(sxf);
        uint4 *dst = reinterpret_cast<uint4 *>(yo);
        for (int i = threadIdx.x; i < (elems >> 3); i += blockDim.x) dst[i] = src[i];
    } else {
        for (int i = threadIdx.x; i < elems; i += blockDim.x) yo[i] = sxf[i];
    }
}

int nchw_rows_per_block(int W, int Cp) {
    const int r = kNchwStageElems / (W * Cp);
    return r < 1 ? 1 : (r > 32 ? 32 : r);
}

cudaError_t launch_nchw_to_nhwc(const float *x, __nv_bfloat16 *y, int N, int C, int H, int W, int Cp,
                                cudaStream_t st) {
    const int rows = nchw_rows_per_block(W, Cp);
    const size_t smem = (size_t)rows * W * Cp * 2;
    const dim3 grid((unsigned)((H + rows - 1) / rows), (unsigned)N);
    return launch_pdl(nchw_to_nhwc_kernel, grid, dim3(256), smem, st, x, y, C, H, W, Cp, rows);
}

// ------------------------------------------------------------ max pool
__global__ void maxpool_kernel(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                               int k, int s, int p, int Ho, int Wo) {
    pdl_launch_dependents();
    pdl_wait();
    const int CV = C >> 3;
    const long long total = (long long)N * Ho * Wo * CV;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int cv = (int)(idx % CV);
    long long t = idx / CV;
    const int q = (int)(t % Wo);
    t /= Wo;
    const int pp = (int)(t % Ho);
    const int n = (int)(t / Ho);
    // Positions outside the image are replaced by the nearest in-image
    // position of the same window (padding < k keeps it inside the window),
    // which leaves the maximum unchanged and makes every load unconditional.
    float m[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) m[j] = -INFINITY;
    const __nv_bfloat16 *xn = x + (size_t)n * H * W * C + cv * 8;
    for (int r = 0; r < k; ++r) {
        const int h = min(max(pp * s - p + r, 0), H - 1);
        for (int c = 0; c < k; ++c) {
            const int w = min(max(q * s - p + c, 0), W - 1);
            float f[8];
            unpack8(ldg_v4(xn + ((size_t)h * W + w) * C), f);
#pragma unroll
            for (int j = 0; j < 8; ++j) m[j] = fmaxf(m[j], f[j]);
        }
    }
    *reinterpret_cast<uint4 *>(y + (((size_t)n * Ho + pp) * Wo + q) * C + cv * 8) = pack8(m);
}

// 3x3 window (stride s, padding p): a thread computes two horizontally
// adjacent outputs of one 8-channel vector; their windows share a column at
// stride 2, so 15 loads (all issued before the first max) serve both.  The
// max of bf16 values is one of them, so it is taken on the packed pairs
// (max.bf16x2), with no conversion.  Out-of-image positions are clamped to
// the nearest in-window position (the padding never wins).
__device__ __forceinline__ uint4 max8(const uint4 &a, const uint4 &b) {
    uint4 r;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r.x) : "r"(a.x), "r"(b.x));
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r.y) : "r"(a.y), "r"(b.y));
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r.z) : "r"(a.z), "r"(b.z));
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r.w) : "r"(a.w), "r"(b.w));
    return r;
}

__global__ void maxpool3_kernel(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                                int s, int p, int Ho, int Wo) {
    pdl_launch_dependents();
    pdl_wait();
    const int CV = C >> 3;
    const int Wq = (Wo + 1) >> 1;  // output column pairs
    const int total = N * Ho * Wq * CV;
    const int idx = (int)(blockIdx.x * blockDim.x + threadIdx.x);
    if (idx >= total) return;
    const int cv = idx % CV;
    int t = idx / CV;
    const int qp = t % Wq;
    t /= Wq;
    const int pp = t % Ho;
    const int n = t / Ho;
    const int q0 = 2 * qp;
    const bool two = q0 + 1 < Wo;
    const __nv_bfloat16 *xn = x + (size_t)n * H * W * C + cv * 8;
    // columns of the two windows: q0*s - p + {0, 1, 2} and (q0+1)*s - p + {0, 1, 2}
    int col[6];
#pragma unroll
    for (int c = 0; c < 3; ++c) {
        col[c] = min(max(q0 * s - p + c, 0), W - 1);
        col[3 + c] = min(max((two ? q0 + 1 : q0) * s - p + c, 0), W - 1);
    }
    uint4 m0 = make_uint4(0, 0, 0, 0), m1 = m0;
#pragma unroll
    for (int r = 0; r < 3; ++r) {
        const int h = min(max(pp * s - p + r, 0), H - 1);  // nearest in-window row
        const __nv_bfloat16 *row = xn + (size_t)h * W * C;
        uint4 v[6];
#pragma unroll
        for (int c = 0; c < 6; ++c) {
            // at stride 2 the second window's first column is the first window's last
            if (c == 3 && s == 2) continue;
            v[c] = ldg_v4(row + (size_t)col[c] * C);
        }
        if (s == 2) v[3] = v[2];
        const uint4 a = max8(max8(v[0], v[1]), v[2]);
        const uint4 b = max8(max8(v[3], v[4]), v[5]);
        m0 = r == 0 ? a : max8(m0, a);
        m1 = r == 0 ? b : max8(m1, b);
    }
    __nv_bfloat16 *yo = y + (((size_t)n * Ho + pp) * Wo + q0) * C + cv * 8;
    *reinterpret_cast<uint4 *>(yo) = m0;
    if (two) *reinterpret_cast<uint4 *>(yo + C) = m1;
}

// 3x3 stride-2 windows, a 2 x 2 block of outputs per thread: rows
// 2pp-p .. 2pp-p+4 and columns 2q0-p .. 2q0-p+4 of the input cover all four
// windows (25 loads of 8 channels instead of 36).  Out-of-image positions
// are clamped to the nearest in-window pixel, as in maxpool3_kernel.
__global__ void maxpool3s2_kernel(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C, int p,
                                  int Ho, int Wo) {
    pdl_launch_dependents();
    pdl_wait();
    const int CV = C >> 3;
    const int Wq = (Wo + 1) >> 1, Hq = (Ho + 1) >> 1;  // output column / row pairs
    const int total = N * Hq * Wq * CV;
    const int idx = (int)(blockIdx.x * blockDim.x + threadIdx.x);
    if (idx >= total) return;
    const int cv = idx % CV;
    int t = idx / CV;
    const int qp = t % Wq;
    t /= Wq;
    const int ph = t % Hq;
    const int n = t / Hq;
    const int q0 = 2 * qp, p0 = 2 * ph;
    const __nv_bfloat16 *xn = x + (size_t)n * H * W * C + cv * 8;
    // window (i, j) covers input rows 2(p0+i)-p + {0,1,2}, columns 2(q0+j)-p + {0,1,2}; a
    // second row / column of windows past the output clamps onto the first
    const int qj = q0 + 1 < Wo ? 1 : 0, pi = p0 + 1 < Ho ? 1 : 0;
    int col[5];
#pragma unroll
    for (int c = 0; c < 5; ++c) {
        const int cc = c < 3 ? c : 2 * qj + (c - 2);  // 3, 4 -> window 1's columns 1, 2 (or window 0's)
        col[c] = min(max(2 * q0 - p + cc, 0), W - 1);
    }
    uint4 m00 = make_uint4(0, 0, 0, 0), m01 = m00, m10 = m00, m11 = m00;
#pragma unroll
    for (int r = 0; r < 5; ++r) {
        const int rr = r < 3 ? r : 2 * pi + (r - 2);
        const int h = min(max(2 * p0 - p + rr, 0), H - 1);
        const __nv_bfloat16 *row = xn + (size_t)h * W * C;
        uint4 v[5];
#pragma unroll
        for (int c = 0; c < 5; ++c) v[c] = ldg_v4(row + (size_t)col[c] * C);
        const uint4 a = max8(max8(v[0], v[1]), v[2]);  // window column 0
        const uint4 b = max8(max8(v[2], v[3]), v[4]);  // window column 1
        if (r < 3) {
            m00 = r == 0 ? a : max8(m00, a);
            m01 = r == 0 ? b : max8(m01, b);
        }
        if (r >= 2) {
            m10 = r == 2 ? a : max8(m10, a);
            m11 = r == 2 ? b : max8(m11, b);
        }
    }
    __nv_bfloat16 *yo = y + (((size_t)n * Ho + p0) * Wo + q0) * C + cv * 8;
    *reinterpret_cast<uint4 *>(yo) = m00;
    if (qj) *reinterpret_cast<uint4 *>(yo + C) = m01;
    if (pi) {
        *reinterpret_cast<uint4 *>(yo + (size_t)Wo * C) = m10;
        if (qj) *reinterpret_cast<uint4 *>(yo + (size_t)Wo * C + C) = m11;
    }
}

cudaError_t launch_maxpool(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                           int k, int s, int p, cudaStream_t st) {
    if (k == 3 && s == 2) {
        const int Ho = (H + 2 * p - 3) / 2 + 1;
        const int Wo = (W + 2 * p - 3) / 2 + 1;
        const long long total = (long long)N * ((Ho + 1) / 2) * ((Wo + 1) / 2) * (C / 8);
        if (total < (1ll << 31))
            return launch_pdl(maxpool3s2_kernel, dim3((unsigned)((total + 255) / 256)), dim3(256), 0, st, x, y,
                              N, H, W, C, p, Ho, Wo);
    }
    if (k == 3) {
        const int Ho = (H + 2 * p - 3) / s + 1;
        const int Wo = (W + 2 * p - 3) / s + 1;
        const long long total = (long long)N * Ho * ((Wo + 1) / 2) * (C / 8);
        if (total < (1ll << 31))
            return launch_pdl(maxpool3_kernel, dim3((unsigned)((total + 255) / 256)), dim3(256), 0, st, x, y,
                              N, H, W, C, s, p, Ho, Wo);
    }
    const int Ho = (H + 2 * p - k) / s + 1;
    const int Wo = (W + 2 * p - k) / s + 1;
    const long long total = (long long)N * Ho * Wo * (C / 8);
    return launch_pdl(maxpool_kernel, dim3((unsigned)((total + 255) / 256)), dim3(256), 0, st, x, y, N,
                      H, W, C, k, s, p, Ho, Wo);
}

// ------------------------------------------------------------ global average pool
// Block (channel block, image): 32 groups of 8 channels x 8 pixel slices.
// Thread (g, sl) sums pixels sl, sl + 8, ... of its group in fp32 (a warp
// reads 512 contiguous bytes per pixel); the slices are then added in slice
// order through shared memory (deterministic), scaled by 1 / (H W) and
// rounded to bf16 once.  64 x 7 x 7 x 2048 (ResNet-50): 512 blocks of 256
// threads, about six loads in flight per thread.
constexpr int kAvgGroups = 32, kAvgSlices = 8;

__global__ void __launch_bounds__(kAvgGroups * kAvgSlices)
    avgpool_kernel(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C) {
    pdl_launch_dependents();
    pdl_wait();
    __shared__ float red[kAvgSlices][kAvgGroups][8];
    const int CV = C >> 3;
    const int cblocks = (CV + kAvgGroups - 1) / kAvgGroups;
    const int n = blockIdx.x / cblocks;
    const int cv = (blockIdx.x - n * cblocks) * kAvgGroups + (int)(threadIdx.x % kAvgGroups);
    const int sl = (int)(threadIdx.x / kAvgGroups);
    float acc[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = 0.0f;
    if (cv < CV) {
        const __nv_bfloat16 *xn = x + (size_t)n * H * W * C + cv * 8;
        for (int i = sl; i < H * W; i += kAvgSlices) {
            float f[8];
            unpack8(ldg_v4(xn + (size_t)i * C), f);
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] += f[j];
        }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) red[sl][threadIdx.x % kAvgGroups][j] = acc[j];
    __syncthreads();
    if (sl == 0 && cv < CV) {
        const int g = (int)threadIdx.x;
        for (int k = 1; k < kAvgSlices; ++k)
#pragma unroll
            for (int j = 0; j < 8; ++j) acc[j] += red[k][g][j];
        const float inv = 1.0f / (float)(H * W);
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] *= inv;
        *reinterpret_cast<uint4 *>(y + (size_t)n * C + cv * 8) = pack8(acc);
    }
}

cudaError_t launch_avgpool(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                           cudaStream_t st) {
    const long long blocks = (long long)N * ((C / 8 + kAvgGroups - 1) / kAvgGroups);
    if (blocks >= (1ll << 31)) return cudaErrorInvalidValue;
    return launch_pdl(avgpool_kernel, dim3((unsigned)blocks), dim3(kAvgGroups * kAvgSlices), 0, st, x, y, N,
                      H, W, C);
}

}  // namespace byoc

namespace byoc {

// ------------------------------------------------------------ Q node (Section 3.2)
// Eight elements per thread per 16-byte piece: one load of bf16, eight fp32
// products with 1/S, four paired conversions to E4M3, one 8-byte store.  A
// thread issues the loads of four pieces (a grid stride apart) before
// converting any, so that each SM keeps enough bytes in flight to stream HBM.
__global__ void __launch_bounds__(256) quantize_e4m3_kernel(const __nv_bfloat16 *__restrict__ x,
                                                            uint8_t *__restrict__ q, size_t n8, float inv) {
    pdl_launch_dependents();
    pdl_wait();
    constexpr int U = 4;
    const size_t stride = (size_t)gridDim.x * blockDim.x;
    for (size_t i0 = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i0 < n8; i0 += U * stride) {
        uint4 v[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const size_t i = i0 + (size_t)u * stride;
            v[u] = i < n8 ? __ldg(reinterpret_cast<const uint4 *>(x) + i) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const size_t i = i0 + (size_t)u * stride;
            if (i >= n8) break;
            const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
            uint32_t p[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) p[k] = cvt_e4m3x2(bf16lo(w[k]) * inv, bf16hi(w[k]) * inv);
            uint2 o;
            o.x = p[0] | (p[1] << 16);
            o.y = p[2] | (p[3] << 16);
            reinterpret_cast<uint2 *>(q)[i] = o;
        }
    }
}

// One wave: up to 8 CTAs of 256 threads per SM, each thread 4 pieces per pass.
cudaError_t launch_quantize_e4m3(const __nv_bfloat16 *x, uint8_t *q, size_t n, float inv_scale, int num_sms,
                                 cudaStream_t st) {
    const size_t n8 = n / 8;
    const size_t blocks = (n8 + 4 * 256 - 1) / (4 * 256);
    const int grid = (int)(blocks < (size_t)num_sms * 8 ? blocks : (size_t)num_sms * 8);
    return launch_pdl(quantize_e4m3_kernel, dim3(grid > 0 ? grid : 1), dim3(256), 0, st, x, q, n8, inv_scale);
}

}  // namespace byoc
