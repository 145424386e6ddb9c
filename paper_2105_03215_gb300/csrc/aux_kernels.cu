// aux_kernels.cu -- the bandwidth-bound kernels of the offloaded path:
//   * depthwise 3x3 conv + folded BN + activation (MobileNetV2 composite),
//   * the space-to-depth boundary transform that turns a stride-2 stem over
//     3 channels into a stride-1 convolution over 16 channels (a layout
//     transformation node inserted at a region boundary, Section 3.2),
//   * the host-graph operators of ResNet-50 (max pool, global average pool),
//     which the paper leaves on the host (Section 3.4, CUDA as the host).
// All tensors are bf16 NHWC; every thread moves 8 channels (16 bytes) at a
// time so that a warp's accesses are contiguous along C.
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
// The 3 x 3 input window lives in registers as fp32 and slides down the
// column: each output row loads one new input row (stride 1; two for stride
// 2), and the next row is loaded before the current one is computed, so two
// rows of loads are in flight per thread.  Registers stay under 80, so a
// multiprocessor holds enough warps to keep HBM busy.
template <int STRIDE, int ROWS>
__global__ void __launch_bounds__(256, 2) dwconv3x3_kernel(const DwArgs a) {
    const int CG = a.C >> 2;  // 4-channel groups
    const int PB = (a.Ho + ROWS - 1) / ROWS;
    const long long total = (long long)a.N * PB * a.Wo * CG;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int cg = (int)(idx % CG);
    long long t = idx / CG;
    const int q = (int)(t % a.Wo);
    t /= a.Wo;
    const int pb = (int)(t % PB);
    const int n = (int)(t / PB);
    const int c0 = cg * 4;

    float w[9][4];
#pragma unroll
    for (int tap = 0; tap < 9; ++tap) {
        const float4 v = __ldg(reinterpret_cast<const float4 *>(a.w + (size_t)tap * a.C + c0));
        w[tap][0] = v.x; w[tap][1] = v.y; w[tap][2] = v.z; w[tap][3] = v.w;
    }
    const float4 b4 = __ldg(reinterpret_cast<const float4 *>(a.bias + c0));

    const int wc0 = q * STRIDE - a.pad;
    const __nv_bfloat16 *xn = a.x + (size_t)n * a.H * a.W * a.C + c0;
    // one input row under the filter: 3 columns x 4 channels, zero outside the image
    // Loads are unconditional (from a clamped, in-image address) and zeroed by
    // a select afterwards, so they can all be in flight at once.
    auto load_row = [&](int h, uint2 (&r)[3]) {
        const bool hv = h >= 0 && h < a.H;
        const int hc = min(max(h, 0), a.H - 1);
#pragma unroll
        for (int s = 0; s < 3; ++s) {
            const int wc = wc0 + s;
            const int wcc = min(max(wc, 0), a.W - 1);
            const uint2 v = __ldg(reinterpret_cast<const uint2 *>(xn + ((size_t)hc * a.W + wcc) * a.C));
            const bool ok = hv && wc >= 0 && wc < a.W;
            r[s] = make_uint2(ok ? v.x : 0u, ok ? v.y : 0u);
        }
    };
    auto unpack_row = [&](const uint2 (&r)[3], float (&f)[3][4]) {
#pragma unroll
        for (int s = 0; s < 3; ++s) {
            f[s][0] = bf16lo(r[s].x); f[s][1] = bf16hi(r[s].x);
            f[s][2] = bf16lo(r[s].y); f[s][3] = bf16hi(r[s].y);
        }
    };

    const int p0 = pb * ROWS;
    float win[3][3][4];
    uint2 raw[3], nxt[3];
    load_row(p0 * STRIDE - a.pad, raw);
    unpack_row(raw, win[0]);
    load_row(p0 * STRIDE - a.pad + 1, raw);
    unpack_row(raw, win[1]);
    load_row(p0 * STRIDE - a.pad + 2, nxt);
#pragma unroll
    for (int i = 0; i < ROWS; ++i) {
        const int p = p0 + i;
        if (p >= a.Ho) break;
        const int hb = p * STRIDE - a.pad;
        unpack_row(nxt, win[2]);
        // prefetch what the next output row needs beyond the rows kept
        uint2 mid[3];
        if (i + 1 < ROWS) {
            if (STRIDE == 1) {
                load_row(hb + 3, nxt);
            } else {
                load_row(hb + 3, mid);
                load_row(hb + 4, nxt);
            }
        }
        float acc[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
        for (int r = 0; r < 3; ++r)
#pragma unroll
            for (int s = 0; s < 3; ++s)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[j] = fmaf(win[r][s][j], w[r * 3 + s][j], acc[j]);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            float v = acc[j];
            if (a.act == kActRelu) v = fmaxf(v, 0.0f);
            else if (a.act == kActRelu6) v = fminf(fmaxf(v, 0.0f), 6.0f);
            else if (a.act == kActGelu) v = 0.5f * v * (1.0f + erff(v * 0.70710678118654752f));
            acc[j] = v;
        }
        uint2 o;
        o.x = pack_bf16x2(acc[0], acc[1]);
        o.y = pack_bf16x2(acc[2], acc[3]);
        *reinterpret_cast<uint2 *>(a.y + (((size_t)n * a.Ho + p) * a.Wo + q) * a.C + c0) = o;
        // slide the window
        if (STRIDE == 1) {
#pragma unroll
            for (int s = 0; s < 3; ++s)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    win[0][s][j] = win[1][s][j];
                    win[1][s][j] = win[2][s][j];
                }
        } else {
#pragma unroll
            for (int s = 0; s < 3; ++s)
#pragma unroll
                for (int j = 0; j < 4; ++j) win[0][s][j] = win[2][s][j];
            if (i + 1 < ROWS) unpack_row(mid, win[1]);
        }
    }
}

cudaError_t launch_dwconv(const DwArgs &a, int num_sms, cudaStream_t st) {
    (void)num_sms;
    const int CG = a.C / 4;
    const int threads = 256;
    if (a.stride == 1) {
        constexpr int R = 8;
        const long long total = (long long)a.N * ((a.Ho + R - 1) / R) * a.Wo * CG;
        dwconv3x3_kernel<1, R><<<(unsigned)((total + threads - 1) / threads), threads, 0, st>>>(a);
    } else {
        constexpr int R = 4;
        const long long total = (long long)a.N * ((a.Ho + R - 1) / R) * a.Wo * CG;
        dwconv3x3_kernel<2, R><<<(unsigned)((total + threads - 1) / threads), threads, 0, st>>>(a);
    }
    return cudaGetLastError();
}

// ------------------------------------------------------------ space-to-depth
// z[n, p, j, a*16 + (dy*2+dx)*C + c] = x[n, 2(p+a)+dy-pad, 2j+dx-pad, c]; one
// thread per 16-channel group (a) of one output pixel, writing 32 bytes.
// Block (p, n): output row p of image n.  Its input rows 2p-pad ..
// 2p-pad+2*taps-1 are one contiguous run of x; the block stages them in
// shared memory (zero rows outside the image; 16-byte loads, four in flight
// per thread), assembles the output row there -- per (column j, stacked
// tap) one 16-channel group -- and writes it out with coalesced 16-byte
// stores.  Staged rows are padded by 8 elements so that the stacked taps of
// one column fall in different banks.
// C is a template parameter so that the 16 channel values stay in registers.
template <int C>
__global__ void __launch_bounds__(256) s2d_kernel(const S2dArgs a) {
    extern __shared__ __align__(16) unsigned short smem_s2d[];
    const int p = blockIdx.x;
    const int n = blockIdx.y;
    const int rows = 2 * a.taps;
    const int row_elems = a.W * C;
    const int pitch = ((row_elems + 7) & ~7) + 8;  // staged row pitch (elements, 16-byte multiple)
    unsigned short *srows = smem_s2d;
    uint4 *sout = reinterpret_cast<uint4 *>(smem_s2d + (size_t)rows * pitch);
    const int h0 = 2 * p - a.pad;
    const unsigned short *xs = reinterpret_cast<const unsigned short *>(a.x);
    if ((row_elems & 7) == 0) {
        const int vec_row = row_elems >> 3;
        const int total = rows * vec_row;
        for (int base = threadIdx.x; base < total; base += 4 * blockDim.x) {
            uint4 v[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int i = base + k * (int)blockDim.x;
                const int r = i / vec_row;
                const int h = h0 + r;
                v[k] = make_uint4(0u, 0u, 0u, 0u);
                if (i < total && h >= 0 && h < a.H)
                    v[k] = __ldg(reinterpret_cast<const uint4 *>(xs + ((size_t)n * a.H + h) * row_elems) +
                                 (i - r * vec_row));
            }
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int i = base + k * (int)blockDim.x;
                const int r = i / vec_row;
                if (i < total)
                    *reinterpret_cast<uint4 *>(srows + (size_t)r * pitch + 8 * (i - r * vec_row)) = v[k];
            }
        }
    } else {
        for (int i = threadIdx.x; i < rows * row_elems; i += blockDim.x) {
            const int r = i / row_elems;
            const int h = h0 + r;
            srows[(size_t)r * pitch + (i - r * row_elems)] =
                (h >= 0 && h < a.H) ? __ldg(xs + ((size_t)n * a.H + h) * row_elems + (i - r * row_elems))
                                    : (unsigned short)0;
        }
    }
    __syncthreads();
    const int groups = a.Wz * a.taps;
    for (int idx = threadIdx.x; idx < groups; idx += blockDim.x) {
        const int j = idx / a.taps;
        const int tap = idx - j * a.taps;
        uint32_t v[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) v[k] = 0u;
#pragma unroll
        for (int dy = 0; dy < 2; ++dy) {
            const unsigned short *row = srows + (size_t)(2 * tap + dy) * pitch;
#pragma unroll
            for (int dx = 0; dx < 2; ++dx) {
                const int w = 2 * j + dx - a.pad;
                if (w < 0 || w >= a.W) continue;
#pragma unroll
                for (int c = 0; c < C; ++c) v[(dy * 2 + dx) * C + c] = row[w * C + c];
            }
        }
        sout[2 * idx] = make_uint4(v[0] | v[1] << 16, v[2] | v[3] << 16, v[4] | v[5] << 16,
                                   v[6] | v[7] << 16);
        sout[2 * idx + 1] = make_uint4(v[8] | v[9] << 16, v[10] | v[11] << 16,
                                       v[12] | v[13] << 16, v[14] | v[15] << 16);
    }
    __syncthreads();
    uint4 *zrow = reinterpret_cast<uint4 *>(a.z + ((size_t)n * a.Hz + p) * (size_t)groups * 16);
    for (int i = threadIdx.x; i < 2 * groups; i += blockDim.x) zrow[i] = sout[i];
}

size_t s2d_smem_bytes(const S2dArgs &a) {
    return (size_t)2 * a.taps * (((a.W * a.C + 7) & ~7) + 8) * 2 + (size_t)a.Wz * a.taps * 32;
}

cudaError_t launch_s2d(const S2dArgs &a, cudaStream_t st) {
    const size_t smem = s2d_smem_bytes(a);
    if (smem > kS2dMaxSmem) return cudaErrorInvalidValue;
    if (smem > 48 * 1024) {
        const void *fns[4] = {(const void *)s2d_kernel<1>, (const void *)s2d_kernel<2>,
                              (const void *)s2d_kernel<3>, (const void *)s2d_kernel<4>};
        for (const void *f : fns) {
            cudaError_t e =
                cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kS2dMaxSmem);
            if (e != cudaSuccess) return e;
        }
    }
    const dim3 grid((unsigned)a.Hz, (unsigned)a.N);
    switch (a.C) {
        case 1: s2d_kernel<1><<<grid, 256, smem, st>>>(a); break;
        case 2: s2d_kernel<2><<<grid, 256, smem, st>>>(a); break;
        case 3: s2d_kernel<3><<<grid, 256, smem, st>>>(a); break;
        case 4: s2d_kernel<4><<<grid, 256, smem, st>>>(a); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

// ------------------------------------------------------------ max pool
__global__ void maxpool_kernel(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                               int k, int s, int p, int Ho, int Wo) {
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

// 3x3 window, fully unrolled: all nine loads issue before the first max.
__global__ void maxpool3_kernel(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                                int s, int p, int Ho, int Wo) {
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
    const __nv_bfloat16 *xn = x + (size_t)n * H * W * C + cv * 8;
    uint4 v[9];
#pragma unroll
    for (int r = 0; r < 3; ++r) {
        const int h = min(max(pp * s - p + r, 0), H - 1);  // nearest in-window position
#pragma unroll
        for (int c = 0; c < 3; ++c) {
            const int w = min(max(q * s - p + c, 0), W - 1);
            v[r * 3 + c] = ldg_v4(xn + ((size_t)h * W + w) * C);
        }
    }
    float m[8];
    unpack8(v[0], m);
#pragma unroll
    for (int i = 1; i < 9; ++i) {
        float f[8];
        unpack8(v[i], f);
#pragma unroll
        for (int j = 0; j < 8; ++j) m[j] = fmaxf(m[j], f[j]);
    }
    *reinterpret_cast<uint4 *>(y + (((size_t)n * Ho + pp) * Wo + q) * C + cv * 8) = pack8(m);
}

cudaError_t launch_maxpool(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                           int k, int s, int p, cudaStream_t st) {
    if (k == 3) {
        const int Ho = (H + 2 * p - 3) / s + 1;
        const int Wo = (W + 2 * p - 3) / s + 1;
        const long long total = (long long)N * Ho * Wo * (C / 8);
        maxpool3_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(x, y, N, H, W, C, s, p, Ho, Wo);
        return cudaGetLastError();
    }
    const int Ho = (H + 2 * p - k) / s + 1;
    const int Wo = (W + 2 * p - k) / s + 1;
    const long long total = (long long)N * Ho * Wo * (C / 8);
    maxpool_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(x, y, N, H, W, C, k, s, p, Ho, Wo);
    return cudaGetLastError();
}

// ------------------------------------------------------------ global average pool
__global__ void avgpool_kernel(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W,
                               int C) {
    const int CV = C >> 3;
    const long long total = (long long)N * CV;
    const long long idx = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int cv = (int)(idx % CV);
    const int n = (int)(idx / CV);
    float acc[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = 0.0f;
    const __nv_bfloat16 *xn = x + (size_t)n * H * W * C + cv * 8;
    for (int i = 0; i < H * W; ++i) {
        float f[8];
        unpack8(ldg_v4(xn + (size_t)i * C), f);
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[j] += f[j];
    }
    const float inv = 1.0f / (float)(H * W);
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] *= inv;
    *reinterpret_cast<uint4 *>(y + (size_t)n * C + cv * 8) = pack8(acc);
}

cudaError_t launch_avgpool(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                           cudaStream_t st) {
    const long long total = (long long)N * (C / 8);
    avgpool_kernel<<<(unsigned)((total + 255) / 256), 256, 0, st>>>(x, y, N, H, W, C);
    return cudaGetLastError();
}

}  // namespace byoc
