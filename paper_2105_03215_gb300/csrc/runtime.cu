// runtime.cu -- the C ABI of include/byoc.h and include/byoc_plan.h.
//
// byoc_compile = plan (host only) + materialise (device):
//   plan        validate the region descriptor; group its ops into launches
//               (a conv2d / dense absorbs the bias_add, batch_norm, add and
//               activation that follow it: the composite of Section 3.1.1
//               runs as one kernel); fold batch norm and bias into a
//               per-channel scale and shift in fp64; scale the weights,
//               round them to bf16 (RNE) and pack them K-major; pick tiles;
//               lay out the workspace for the region's intermediates, which
//               are not data entries (Section 3.4).
//   materialise cudaMalloc + copy of the constants (the metadata module's
//               one-time load, Section 3.4), TMA descriptors of the weights,
//               kernel attributes.  The handle is the cached engine.
// byoc_run = the external call: patch activation pointers into cached TMA
// descriptors and launch the region's kernels on the caller's stream.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <type_traits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <new>
#include <string>
#include <type_traits>
#include <vector>

#include "byoc.h"
#include "byoc_plan.h"
#include "internal.h"

using byoc::GemmArgs;
using byoc::GemmConfig;

namespace {

thread_local std::string g_err;

byoc_status fail(byoc_status st, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_err = buf;
    return st;
}

byoc_status cuda_fail(cudaError_t e, const char *what) {
    return fail(e == cudaErrorMemoryAllocation ? BYOC_ERR_OOM : BYOC_ERR_CUDA, "%s: %s (%s)", what,
                cudaGetErrorName(e), cudaGetErrorString(e));
}

// ------------------------------------------------------------ driver entry points

PFN_cuTensorMapEncodeTiled_v12000 p_encode_tiled = nullptr;
PFN_cuTensorMapEncodeIm2col_v12000 p_encode_im2col = nullptr;
std::once_flag g_driver_once;
cudaError_t g_driver_err = cudaSuccess;

cudaError_t load_driver() {
    std::call_once(g_driver_once, [] {
        cudaDriverEntryPointQueryResult q1, q2;
        cudaError_t e = cudaGetDriverEntryPointByVersion(
            "cuTensorMapEncodeTiled", reinterpret_cast<void **>(&p_encode_tiled), 12000,
            cudaEnableDefault, &q1);
        if (e == cudaSuccess)
            e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeIm2col",
                                                 reinterpret_cast<void **>(&p_encode_im2col),
                                                 12000, cudaEnableDefault, &q2);
        if (e == cudaSuccess && (q1 != cudaDriverEntryPointSuccess ||
                                 q2 != cudaDriverEntryPointSuccess || !p_encode_tiled ||
                                 !p_encode_im2col))
            e = cudaErrorSymbolNotFound;
        g_driver_err = e;
    });
    return g_driver_err;
}

CUtensorMapSwizzle swizzle_for(int bk) {
    return bk == 64 ? CU_TENSOR_MAP_SWIZZLE_128B
                    : (bk == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B);
}

// 2-D row-major bf16 matrix [rows, cols]; box = [box_cols, box_rows].
CUresult encode_2d(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                   uint32_t box_cols, int bk) {
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t es[2] = {1, 1};
    return p_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims,
                          strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for(bk),
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// 2-D row-major E4M3 (1-byte) matrix [rows, cols]; box = [box_cols, box_rows].
CUresult encode_2d_u8(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                      uint32_t box_cols, CUtensorMapSwizzle swz) {
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t es[2] = {1, 1};
    return p_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(ptr), dims, strides, box, es,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// Geometry of an im2col-read convolution input.
struct Im2colGeom {
    int N, H, W, C;
    int kh, kw, sh, sw, pt, pl, pb, pr, dh, dw;
};

// im2col map over an NHWC bf16 tensor; 128 pixels x bk channels per load.
// The bounding box of filter origins runs, per spatial dimension, from -pad_before
// to (dim - 1) + pad_after - (k - 1) * dilation; corner and offset arrays list
// the spatial dimensions innermost first (W, then H), like the tensor's dims.
CUresult encode_im2col(CUtensorMap *m, const void *ptr, const Im2colGeom &g, int bk, bool e4m3 = false) {
    const cuuint64_t es_b = e4m3 ? 1 : 2;
    cuuint64_t dims[4] = {(cuuint64_t)g.C, (cuuint64_t)g.W, (cuuint64_t)g.H, (cuuint64_t)g.N};
    cuuint64_t strides[3] = {(cuuint64_t)g.C * es_b, (cuuint64_t)g.W * g.C * es_b,
                             (cuuint64_t)g.H * g.W * g.C * es_b};
    int lower[2] = {-g.pl, -g.pt};
    int upper[2] = {g.pr - (g.kw - 1) * g.dw, g.pb - (g.kh - 1) * g.dh};
    cuuint32_t es[4] = {1, (cuuint32_t)g.sw, (cuuint32_t)g.sh, 1};
    // E4M3: 128 codes per pixel fill the same 128-byte swizzled row as 64 bf16
    return p_encode_im2col(m, e4m3 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4,
                           const_cast<void *>(ptr), dims, strides, lower, upper, (cuuint32_t)(e4m3 ? 2 * bk : bk),
                           (cuuint32_t)byoc::kGemmBM, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for(bk),
                           CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// Tiled 4-D map over an NHWC tensor for slab loads: box = {bk channels, wp
// columns, rows rows, 1 image}; out-of-image elements read as zero.
CUresult encode_slab(CUtensorMap *m, const void *ptr, int N, int H, int W, int C, int wp, int rows,
                     int bk) {
    cuuint64_t dims[4] = {(cuuint64_t)C, (cuuint64_t)W, (cuuint64_t)H, (cuuint64_t)N};
    cuuint64_t strides[3] = {(cuuint64_t)C * 2, (cuuint64_t)W * C * 2, (cuuint64_t)H * W * C * 2};
    cuuint32_t box[4] = {(cuuint32_t)bk, (cuuint32_t)wp, (cuuint32_t)rows, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return p_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(ptr), dims,
                          strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for(bk),
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// Stem slab over the pixel-pair layout xq [N, Hq, Wq, 4] (StemArgs): dims
// {8 G values (G pixel pairs), wp / G pair groups, E position rows, R image
// rows, N} with E = (Hq - R) / 2 + 1.  A position row is two image rows on,
// so the position-row and image-row dimensions overlap, and every in-range
// element stays inside its image's Hq rows.  Box {8 G, wp / G, rows, R, 1}
// at (0, 0, p, 0, n), without swizzle, lands in shared memory as R planes
// [image row r][slab position (p + y, j)][16 bytes]; position rows past E
// read as zeros.  (A 16-byte-wide operand row cannot be swizzled in place:
// a 16-byte inner box under 128-byte swizzle is laid out at the 128-byte
// span per row, hence the unswizzled planes.)
CUresult encode_stem_slab(CUtensorMap *m, const void *ptr, int N, int Hq, int Wq, int R, int wp, int rows,
                          int G) {
    const cuuint64_t row = (cuuint64_t)Wq * 4 * 2;
    const cuuint64_t E = (cuuint64_t)(Hq - R) / 2 + 1;
    cuuint64_t dims[5] = {(cuuint64_t)8 * G, (cuuint64_t)(wp / G), E, (cuuint64_t)R, (cuuint64_t)N};
    cuuint64_t strides[4] = {(cuuint64_t)16 * G, 2 * row, row, (cuuint64_t)Hq * row};
    cuuint32_t box[5] = {(cuuint32_t)(8 * G), (cuuint32_t)(wp / G), (cuuint32_t)rows, (cuuint32_t)R, 1};
    cuuint32_t es[5] = {1, 1, 1, 1, 1};
    return p_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void *>(ptr), dims,
                          strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// Depthwise input box: in_rows x in_cols pixels x cc channels, no swizzle
// (the kernel reads it with plain 16-byte shared-memory loads).
CUresult encode_dw(CUtensorMap *m, const void *ptr, const byoc::DwArgs &a) {
    cuuint64_t dims[4] = {(cuuint64_t)a.C, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.N};
    cuuint64_t strides[3] = {(cuuint64_t)a.C * 2, (cuuint64_t)a.W * a.C * 2,
                             (cuuint64_t)a.H * a.W * a.C * 2};
    cuuint32_t box[4] = {(cuuint32_t)a.cc, (cuuint32_t)a.in_cols, (cuuint32_t)a.in_rows, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return p_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(ptr), dims,
                          strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// Input boxes of the fused depthwise -> 1x1 kernel: 64 channels x in_cols x
// in_rows of one image, no swizzle (read by CUDA cores), zero outside.
CUresult encode_dwpw_input(CUtensorMap *m, const void *ptr, const byoc::DwPwArgs &a) {
    cuuint64_t dims[4] = {(cuuint64_t)a.C, (cuuint64_t)a.W, (cuuint64_t)a.H, (cuuint64_t)a.N};
    cuuint64_t strides[3] = {(cuuint64_t)a.C * 2, (cuuint64_t)a.W * a.C * 2,
                             (cuuint64_t)a.H * a.W * a.C * 2};
    cuuint32_t box[4] = {(cuuint32_t)byoc::kDpChunk, (cuuint32_t)a.in_cols, (cuuint32_t)a.in_rows, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return p_encode_tiled(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(ptr), dims,
                          strides, box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// ------------------------------------------------------------ bf16 rounding (host)

uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    std::memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u) return (uint16_t)((u >> 16) | ((u & 0xFFFFu) ? 0x40u : 0u));
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Nearest FP8 E4M3 code of v: 1 sign bit, 4 exponent bits (bias 7), 3
// mantissa bits; a value in [2^e, 2^(e+1)) with e >= -6 is a multiple of
// 2^(e-3), below 2^-6 the values are the multiples of 2^-9 (exponent field
// 0).  Ties to even (nearbyint in the default rounding mode); magnitudes past
// 448, the largest finite value, saturate to it.
uint8_t e4m3_code(double v) {
    const uint8_t sign = std::signbit(v) ? 0x80 : 0x00;
    const double a = std::fabs(v);
    if (!(a == a)) return 0x7F;
    int ex = 0;
    std::frexp(a, &ex);  // a = m 2^ex, 1/2 <= m < 1
    int e = std::max(ex - 1, -6);
    double q = std::nearbyint(std::ldexp(a, 3 - e));  // a / 2^(e-3)
    if (q >= 16.0) {  // rounded up into the next binade
        q = 8.0;
        e += 1;
    }
    if (q < 8.0) return sign | (uint8_t)q;                    // exponent field 0 (e == -6)
    if (e > 8 || (e == 8 && q > 14.0)) return sign | 0x7E;   // saturate at 448 = 1.75 x 2^8
    return sign | (uint8_t)((e + 7) << 3) | (uint8_t)(q - 8.0);
}

// Per-output-channel scale of FP8 weights: the smallest power of two S with
// max |w'| / S <= 448 (1 for an all-zero channel).
double e4m3_weight_scale(double maxabs) {
    if (!(maxabs > 0.0)) return 1.0;
    int ex = 0;
    const double f = std::frexp(maxabs / 448.0, &ex);
    return std::ldexp(1.0, f == 0.5 ? ex - 1 : ex);
}

// ------------------------------------------------------------ plan structures

struct TensorInfo {
    int ndim = 0;
    int dtype = BYOC_BF16;  // BYOC_BF16 or BYOC_E4M3
    int64_t shape[4] = {0, 0, 0, 0};
    size_t elems() const {
        size_t e = 1;
        for (int i = 0; i < ndim; ++i) e *= (size_t)shape[i];
        return e;
    }
    size_t bytes() const { return elems() * (dtype == BYOC_E4M3 ? 1 : 2); }
    int64_t channels() const { return shape[ndim - 1]; }
};

struct LaunchPlan {
    int kind = BYOC_LAUNCH_GEMM;
    int first_op = -1, n_ops = 0;
    int x = -1, y = -1, res = -1;  // tensor ids (may index internal scratch tensors)
    size_t x_off = 0, y_off = 0;   // byte offsets into tensors x and y (image chunks)
    int act = byoc::kActNone;
    // GEMM
    GemmConfig cfg{64, 64, byoc::kAModeTile, false};
    GemmArgs args{};
    int grid = 0;
    int n_pad = 0, k_pack = 0;
    // A operand geometry
    Im2colGeom geo{};
    int64_t aM = 0, aK = 0;
    int slab_rows = 0;  // slab mode: padded input rows per slab
    // split-K scratch (handle workspace): fp32 partials and arrival counters
    size_t part_off = 0, part_bytes = 0, cnt_off = 0, cnt_bytes = 0;
    // constants: byte offsets into the constant blob
    size_t w_off = 0, w_bytes = 0, b_off = 0, b_bytes = 0;
    // depthwise / stem layout transform / fused depthwise -> 1x1
    byoc::DwArgs dw{};
    byoc::StemArgs stem{};
    int stem_R = 0;  // stem GEMM: row taps per slab position (StemArgs layout), else 0
    int stem_G = 0;  // stem GEMM: pixel pairs per innermost tensor-map box row
    byoc::DwPwArgs dp{};
    size_t w2_off = 0, w2_bytes = 0, b2_off = 0, b2_bytes = 0;  // fused: the 1x1 conv's constants
    // region kernel (BYOC_LAUNCH_CHAIN): per stage, the GEMM launch it replaces
    int chain_bn = 0;
    int cx[byoc::kChainMaxStages] = {}, cy[byoc::kChainMaxStages] = {}, cres[byoc::kChainMaxStages] = {};
    Im2colGeom cgeo[byoc::kChainMaxStages] = {};
    int64_t caM[byoc::kChainMaxStages] = {}, caK[byoc::kChainMaxStages] = {};
    int c_npad[byoc::kChainMaxStages] = {}, c_kpack[byoc::kChainMaxStages] = {};
    size_t cw_off[byoc::kChainMaxStages] = {}, cb_off[byoc::kChainMaxStages] = {};
    size_t order_off = 0, dep_off_off = 0, dep_list_off = 0;  // constant blob: int32 unit order, dependencies
    size_t cta_off_off = 0, cta_rec_off = 0;                  // constant blob: int32 per-CTA unit records
    size_t c_dq_off[byoc::kChainMaxStages] = {};
    // FP8 GEMM (cfg.bk = kF8BK, or a region-kernel stage): A and B are E4M3 codes; dq = [n_pad] fp32
    // dequantization scales S_x S_w[n] in the constant blob
    int fp8 = 0;
    size_t dq_off = 0;
    // a Q node fused into the epilogue: the output is E4M3 codes of x fp32(1/S)
    int out8 = 0;
    float out_inv = 0.0f;
    // BYOC_LAUNCH_QUANT: y = e4m3(x fp32(1/S))
    float q_inv = 0.0f;
    size_t flags_off = 0, flags_bytes = 0;     // workspace: unit flags + control words
    byoc::ChainArgs chain{};
    double flops = 0, bytes = 0;
};

struct Plan {
    std::vector<TensorInfo> tensors;  // region tensors, then internal scratch tensors
    int n_region_tensors = 0;
    std::vector<int> inputs, outputs;
    std::vector<LaunchPlan> launches;
    std::vector<uint8_t> blob;  // packed constants (device image)
    std::vector<size_t> ws_off;  // per tensor: workspace offset, or SIZE_MAX for boundary
    size_t ws_bytes = 0;
    double flops = 0, bytes = 0;
    int num_sms = 148;
};

size_t blob_append(std::vector<uint8_t> &blob, const void *src, size_t bytes) {
    size_t off = align_up(blob.size(), 256);
    blob.resize(off + bytes);
    std::memcpy(blob.data() + off, src, bytes);
    return off;
}

// ------------------------------------------------------------ validation

byoc_status validate(const byoc_region_desc *d, Plan &P) {
    if (!d) return fail(BYOC_ERR_INVALID_ARG, "null region descriptor");
    if (d->abi_version != BYOC_ABI_VERSION)
        return fail(BYOC_ERR_INVALID_ARG, "abi_version %u, expected %u", d->abi_version,
                    BYOC_ABI_VERSION);
    if (d->n_tensors <= 0 || !d->tensors) return fail(BYOC_ERR_INVALID_ARG, "no tensors");
    if (d->n_ops <= 0 || !d->ops) return fail(BYOC_ERR_INVALID_ARG, "no ops");
    if (d->n_inputs <= 0 || !d->input_ids || d->n_outputs <= 0 || !d->output_ids)
        return fail(BYOC_ERR_INVALID_ARG, "region needs at least one input and one output");
    const int nt = d->n_tensors;
    P.tensors.resize(nt);
    P.n_region_tensors = nt;
    for (int i = 0; i < nt; ++i) {
        const byoc_tensor &t = d->tensors[i];
        if (t.ndim != 2 && t.ndim != 4)
            return fail(BYOC_ERR_INVALID_ARG, "tensor %d: ndim %d (2 or 4 expected)", i, t.ndim);
        if ((t.ndim == 4) != (t.layout == BYOC_LAYOUT_NHWC))
            return fail(BYOC_ERR_INVALID_ARG, "tensor %d: layout %d does not match ndim %d", i,
                        t.layout, t.ndim);
        if (t.dtype != BYOC_BF16 && t.dtype != BYOC_E4M3)
            return fail(BYOC_ERR_UNSUPPORTED, "tensor %d: activations must be bf16 or E4M3 codes", i);
        P.tensors[i].ndim = t.ndim;
        P.tensors[i].dtype = t.dtype;
        for (int k = 0; k < t.ndim; ++k) {
            if (t.shape[k] <= 0 || t.shape[k] > (int64_t)1 << 31)
                return fail(BYOC_ERR_INVALID_ARG, "tensor %d: bad extent %lld", i,
                            (long long)t.shape[k]);
            P.tensors[i].shape[k] = t.shape[k];
        }
        if (P.tensors[i].elems() >= ((size_t)1 << 40))
            return fail(BYOC_ERR_INVALID_ARG, "tensor %d too large", i);
    }
    std::vector<int> producer(nt, -1), is_input(nt, 0), is_output(nt, 0);
    for (int i = 0; i < d->n_inputs; ++i) {
        int id = d->input_ids[i];
        if (id < 0 || id >= nt) return fail(BYOC_ERR_INVALID_ARG, "input id %d out of range", id);
        if (is_input[id]) return fail(BYOC_ERR_INVALID_ARG, "input id %d repeated", id);
        is_input[id] = 1;
        P.inputs.push_back(id);
    }
    for (int i = 0; i < d->n_outputs; ++i) {
        int id = d->output_ids[i];
        if (id < 0 || id >= nt) return fail(BYOC_ERR_INVALID_ARG, "output id %d out of range", id);
        if (is_output[id]) return fail(BYOC_ERR_INVALID_ARG, "output id %d repeated", id);
        if (is_input[id]) return fail(BYOC_ERR_INVALID_ARG, "tensor %d is both input and output", id);
        is_output[id] = 1;
        P.outputs.push_back(id);
    }
    for (int o = 0; o < d->n_ops; ++o) {
        const byoc_op &op = d->ops[o];
        if (op.kind < BYOC_OP_CONV2D || op.kind > BYOC_OP_QUANTIZE)
            return fail(BYOC_ERR_INVALID_ARG, "op %d: unknown kind %d", o, op.kind);
        const int want_in = op.kind == BYOC_OP_ADD ? 2 : 1;
        if (op.n_in != want_in)
            return fail(BYOC_ERR_INVALID_ARG, "op %d: %d inputs, expected %d", o, op.n_in, want_in);
        for (int k = 0; k < op.n_in; ++k) {
            int id = op.in[k];
            if (id < 0 || id >= nt) return fail(BYOC_ERR_INVALID_ARG, "op %d: input id %d", o, id);
            if (!is_input[id] && producer[id] < 0)
                return fail(BYOC_ERR_INVALID_ARG,
                            "op %d reads tensor %d before any op produces it (ops must be in "
                            "topological order)",
                            o, id);
        }
        if (op.out < 0 || op.out >= nt) return fail(BYOC_ERR_INVALID_ARG, "op %d: output id", o);
        if (is_input[op.out] || producer[op.out] >= 0)
            return fail(BYOC_ERR_INVALID_ARG, "op %d: tensor %d produced twice", o, op.out);
        producer[op.out] = o;
        const TensorInfo &X = P.tensors[op.in[0]];
        const TensorInfo &Y = P.tensors[op.out];
        auto same_shape = [](const TensorInfo &a, const TensorInfo &b) {
            if (a.ndim != b.ndim) return false;
            for (int k = 0; k < a.ndim; ++k)
                if (a.shape[k] != b.shape[k]) return false;
            return true;
        };
        // E4M3 tensors come from Q nodes and feed conv2d / dense only
        if ((Y.dtype == BYOC_E4M3) != (op.kind == BYOC_OP_QUANTIZE))
            return fail(BYOC_ERR_INVALID_ARG, "op %d: only a quantize op writes an E4M3 tensor", o);
        for (int k = 0; k < op.n_in; ++k)
            if (P.tensors[op.in[k]].dtype == BYOC_E4M3 &&
                !(k == 0 && (op.kind == BYOC_OP_CONV2D || op.kind == BYOC_OP_DENSE)))
                return fail(BYOC_ERR_UNSUPPORTED, "op %d: E4M3 tensors feed conv2d / dense data inputs only", o);
        if (op.kind == BYOC_OP_CONV2D && X.dtype == BYOC_E4M3 && op.groups != 1)
            return fail(BYOC_ERR_UNSUPPORTED, "op %d: grouped conv2d on E4M3 codes", o);
        switch (op.kind) {
            case BYOC_OP_QUANTIZE: {
                if (X.dtype != BYOC_BF16 || !same_shape(X, Y))
                    return fail(BYOC_ERR_INVALID_ARG, "op %d: quantize needs a bf16 input of its output's shape", o);
                if (!op.consts[0] || !op.consts[1])
                    return fail(BYOC_ERR_INVALID_ARG, "op %d: quantize needs its scale and zero point", o);
                const float S = op.consts[0][0], Z = op.consts[1][0];
                if (!(S > 0.0f) || !std::isfinite(S) || !std::isfinite(1.0 / (double)S))
                    return fail(BYOC_ERR_INVALID_ARG, "op %d: quantize scale %g", o, (double)S);
                if (Z != 0.0f)
                    return fail(BYOC_ERR_UNSUPPORTED, "op %d: E4M3 is symmetric: zero point must be 0", o);
                if (X.channels() % 8)
                    return fail(BYOC_ERR_UNSUPPORTED, "op %d: quantize needs channels % 8 == 0", o);
                break;
            }
            case BYOC_OP_CONV2D: {
                if (X.ndim != 4 || Y.ndim != 4)
                    return fail(BYOC_ERR_INVALID_ARG, "op %d: conv2d needs NHWC tensors", o);
                if (!op.consts[0]) return fail(BYOC_ERR_INVALID_ARG, "op %d: conv2d weight is null", o);
                if (op.kernel[0] < 1 || op.kernel[1] < 1 || op.stride[0] < 1 || op.stride[1] < 1 ||
                    op.dilation[0] < 1 || op.dilation[1] < 1 || op.groups < 1 || op.pad[0] < 0 ||
                    op.pad[1] < 0 || op.pad[2] < 0 || op.pad[3] < 0)
                    return fail(BYOC_ERR_INVALID_ARG, "op %d: bad conv2d attributes", o);
                const int64_t C = X.shape[3], K = Y.shape[3];
                if (C % op.groups || K % op.groups)
                    return fail(BYOC_ERR_INVALID_ARG, "op %d: channels not divisible by groups", o);
                const int64_t Ho = (X.shape[1] + op.pad[0] + op.pad[2] -
                                    (int64_t)op.dilation[0] * (op.kernel[0] - 1) - 1) /
                                       op.stride[0] + 1;
                const int64_t Wo = (X.shape[2] + op.pad[1] + op.pad[3] -
                                    (int64_t)op.dilation[1] * (op.kernel[1] - 1) - 1) /
                                       op.stride[1] + 1;
                if (Y.shape[0] != X.shape[0] || Y.shape[1] != Ho || Y.shape[2] != Wo || Ho < 1 ||
                    Wo < 1)
                    return fail(BYOC_ERR_INVALID_ARG,
                                "op %d: conv2d output shape [%lld,%lld,%lld,%lld] does not match "
                                "[%lld,%lld,%lld,%lld]",
                                o, (long long)Y.shape[0], (long long)Y.shape[1],
                                (long long)Y.shape[2], (long long)Y.shape[3], (long long)X.shape[0],
                                (long long)Ho, (long long)Wo, (long long)K);
                break;
            }
            case BYOC_OP_DENSE:
                if (X.ndim != 2 || Y.ndim != 2 || X.shape[0] != Y.shape[0])
                    return fail(BYOC_ERR_INVALID_ARG, "op %d: dense needs [M,I] -> [M,U]", o);
                if (!op.consts[0]) return fail(BYOC_ERR_INVALID_ARG, "op %d: dense weight is null", o);
                break;
            case BYOC_OP_BIAS_ADD:
                if (!op.consts[0]) return fail(BYOC_ERR_INVALID_ARG, "op %d: bias is null", o);
                if (!same_shape(X, Y)) return fail(BYOC_ERR_INVALID_ARG, "op %d: shape mismatch", o);
                break;
            case BYOC_OP_BATCH_NORM:
                for (int k = 0; k < 4; ++k)
                    if (!op.consts[k])
                        return fail(BYOC_ERR_INVALID_ARG, "op %d: batch_norm constant %d is null", o, k);
                if (!(op.eps >= 0.0f)) return fail(BYOC_ERR_INVALID_ARG, "op %d: eps < 0", o);
                if (!same_shape(X, Y)) return fail(BYOC_ERR_INVALID_ARG, "op %d: shape mismatch", o);
                for (int64_t c = 0; c < X.channels(); ++c)
                    if (!((double)op.consts[3][c] + op.eps > 0.0))
                        return fail(BYOC_ERR_INVALID_ARG, "op %d: var + eps <= 0 at channel %lld", o,
                                    (long long)c);
                break;
            case BYOC_OP_ADD:
                if (!same_shape(X, Y) || !same_shape(P.tensors[op.in[1]], Y))
                    return fail(BYOC_ERR_INVALID_ARG, "op %d: add operands differ in shape", o);
                break;
            default:
                if (!same_shape(X, Y)) return fail(BYOC_ERR_INVALID_ARG, "op %d: shape mismatch", o);
        }
    }
    for (int id : P.outputs)
        if (producer[id] < 0)
            return fail(BYOC_ERR_INVALID_ARG, "output tensor %d is produced by no op", id);
    for (int id : P.inputs)
        if (P.tensors[id].dtype != BYOC_BF16)
            return fail(BYOC_ERR_UNSUPPORTED, "input tensor %d: region inputs are bf16", id);
    for (int id : P.outputs)
        if (P.tensors[id].dtype != BYOC_BF16)
            return fail(BYOC_ERR_UNSUPPORTED, "output tensor %d: region outputs are bf16", id);
    return BYOC_OK;
}

// ------------------------------------------------------------ planning

int pick_bk(int64_t C) {
    if (C <= 16) return 16;
    if (C <= 32) return 32;
    return 64;
}

// Choose the output-channel tile among the compiled configurations by a
// makespan estimate of the persistent grid, in SM cycles, fitted to GB300
// traces of this kernel.  A k-block (bk channels of one filter tap) costs the
// largest of
//   * the tensor-core time of its bk / 16 MMAs (M = 128, N = bn: 40 / 48 /
//     64 / 128 cycles at bn = 32 / 64 / 128 / 256);
//   * its shared-memory traffic: every K16 MMA reads A (4 KB) and B (bn x 32
//     bytes) from shared memory, and TMA writes the k-block's operands into
//     it (A 128 x bk and B bn x bk; slab mode: B and the k-block's share of
//     the slab).  Operand reads and TMA writes share the SM's shared-memory
//     bandwidth, ~145 bytes/cycle in tile and im2col mode and ~118 in slab
//     mode (traced per 64-wide k-block: 427 / 690 cycles at bn = 128 / 256 in
//     tile mode, 316 / 420 at bn = 64 / 128 in slab mode; sharing each
//     weight tile between two SMs by multicast, which halves L2 reads but not
//     these bytes, measured no faster);
//   * in tile and im2col mode, ~450 cycles of TMA round trip and per-k-block
//     overhead, whatever bk (a k-block of 16 channels costs as much: the
//     MobileNetV2 112x112 16 -> 96 layer, measured in the whole network).
// epilogue per tile = ~600 cycles per pair of 32-column chunks (two warps per
// accumulator row block work in parallel), ~3x that with GELU (traced).
// A CTA overlaps one tile's epilogue with the next tile's mainloop, so its
// time is rounds x max(mainloop, epilogue) + min(mainloop, epilogue).
//   split-K (tile mode, no residual, one wave of units only): S splits of
//                        kblocks / S each.  Through global memory: every
//                        split writes and fences its fp32 partial (~26 bn
//                        cycles, traced) and the last one reads the other
//                        S - 1 back (~10 bn cycles each) before the epilogue.
//                        As one cluster (BN <= 128, S <= 4): the partials move
//                        through distributed shared memory (~2000 + 10 bn
//                        cycles) and each CTA runs the epilogue of its 1 / S
//                        of the tile's chunks.
// slab_kb_bytes: slab mode, the bytes of one channel chunk's slab / taps.
// *cluster_out: whether the chosen split is the cluster one.
int pick_bn(int64_t tiles_m, int64_t N, int64_t kblocks, int bk, int amode, bool res, int num_sms,
            int *splits_out = nullptr, double slab_kb_bytes = 0.0, bool gelu = false, bool *cluster_out = nullptr) {
    int best = -1, best_s = 1;
    bool best_cl = false;
    double best_cost = 1e300;
    for (int bn : {256, 128, 64, 32}) {
        GemmConfig c{bn, bk, amode, res};
        if (!byoc::gemm_config_supported(c)) continue;
        const int64_t tiles = tiles_m * ((N + bn - 1) / bn);
        // bytes of one operand row of a k-block: an FP8 k-block (128 codes)
        // is as many bytes, MMAs (K = 32 each, at twice the K16 rate) and
        // cycles as a bf16 one of 64 values
        const int kbytes = bk == byoc::kF8BK ? bk : 2 * bk;
        const double steps = kbytes / 32.0;  // MMAs per k-block
        const double mma = steps * (bn <= 32 ? 40.0 : bn <= 64 ? 48.0 : bn <= 128 ? 64.0 : 128.0);
        const double reads = steps * (4096.0 + 32.0 * bn);
        const bool slab = amode == byoc::kAModeSlab;
        const double writes = slab ? (double)kbytes * bn + slab_kb_bytes : (double)kbytes * (128.0 + bn);
        const double kb = slab ? std::max(mma, (reads + writes) / 118.0)
                               : std::max({mma, (reads + writes) / 145.0, 450.0});
        const double epilogue = 600.0 * std::max(1, bn / 64) * (gelu ? 3.0 : 1.0);
        for (int S = 1; S <= 4; ++S) {
            const bool global_ok =
                byoc::gemm_config_supported(GemmConfig{bn, bk, byoc::kAModeTileSplit, false});
            const bool cl_ok = cluster_out && byoc::cl_split_fits(bn, S) &&
                               byoc::gemm_config_supported(GemmConfig{bn, bk, byoc::kAModeTileSplitCl, false});
            if (S > 1 && (!splits_out || amode != byoc::kAModeTile || res || kblocks < 4 * S ||
                          tiles * S > num_sms || !(global_ok || cl_ok)))
                continue;
            const int64_t units = tiles * S;
            const int64_t grid = std::min<int64_t>(units, num_sms);
            const int64_t rounds = (units + grid - 1) / grid;
            const double mainloop = 300.0 + (double)((kblocks + S - 1) / S) * kb;
            const int nch = bn / 32;
            const double cost_global = mainloop + 26.0 * bn + 10.0 * bn * (S - 1) + epilogue;
            const double cost_cl = mainloop + 2000.0 + 10.0 * bn + epilogue * ((nch + S - 1) / S) / nch;
            const bool cl = S > 1 && cl_ok && (!global_ok || cost_cl < cost_global);
            const double cost =
                S == 1 ? (double)rounds * std::max(mainloop, epilogue) + std::min(mainloop, epilogue)
                       : (cl ? cost_cl : cost_global);
            if (cost < best_cost - 1e-9) {
                best_cost = cost;
                best = bn;
                best_s = S;
                best_cl = cl;
            }
        }
    }
    if (splits_out) *splits_out = best_s;
    if (cluster_out) *cluster_out = best_cl;
    return best;
}

// Slab-mode geometry of a stride-1 convolution: output rows per tile, padded
// width, slab rows, slab bytes.  Returns false when the slab mode does not fit
// (padded width over 128, under 70% of the 128 MMA rows carrying outputs, or a
// slab larger than its buffer).
struct SlabGeom {
    int wp, t, rows, bytes;
};
bool slab_geometry(int H, int W, int Ho, int Wo, int kh, int kw, int pt, int pl, int pr, int bk,
                   SlabGeom &g) {
    (void)H;
    g.wp = W + pl + pr;
    if (g.wp > 128 || g.wp > 256) return false;
    g.t = std::min(128 / g.wp, Ho);
    if (g.t < 1 || g.t * Wo < 90) return false;
    const int dmax = (kh - 1) * g.wp + (kw - 1);
    g.rows = (128 + dmax + g.wp - 1) / g.wp;
    g.bytes = g.rows * g.wp * bk * 2;
    (void)pt;
    return g.rows <= 256 && g.bytes <= byoc::slab_max_bytes(bk);
}

// Pair-unit slab (kAModeSlab2 / kAModeSlabRes2): the rows under two
// vertically adjacent tiles of t output rows each.  The second tile's MMA
// rows start t * wp slab rows in.
bool slab_pair_geometry(int kh, int kw, int bk, const SlabGeom &g, SlabGeom &pg) {
    pg = g;
    const int dmax = (kh - 1) * g.wp + (kw - 1);
    pg.rows = (g.t * g.wp + 128 + dmax + g.wp - 1) / g.wp;
    pg.bytes = pg.rows * g.wp * bk * 2;
    return pg.rows <= 256 && pg.bytes <= byoc::slab_max_bytes(bk, true);
}

// Makespan estimate (SM cycles) of a slab-mode launch: `units` m-units of
// `halves` tiles each, times tiles_n column tiles, over the persistent grid.
// A k-block costs the larger of its MMA time (halves x bk/16 MMAs of
// M=128, N=bn: 40 / 48 / 64 / 128 cycles for bn = 32 / 64 / 128 / 256) and
// the time to bring in its operand bytes (ring weights + its share of the
// slab) at ~40 B/cycle per SM -- what the GB300 traces of the 28x28 and
// 14x14 ResNet-50 3x3 layers deliver; plus ~300 cycles per unit.
double slab_makespan(int64_t units, int64_t tiles_n, int64_t kblocks, int taps, int bn, int bk, int halves,
                     bool wres, int slab_bytes, int num_sms) {
    const double mma = bn <= 32 ? 40.0 : bn <= 64 ? 48.0 : bn <= 128 ? 64.0 : 128.0;
    const double kb_bytes = (wres ? 0.0 : (double)bn * bk * 2) + (double)slab_bytes / std::max(1, taps);
    const double per_kb = std::max(halves * (bk / 16) * mma, kb_bytes / 40.0);
    const int64_t u = units * tiles_n;
    const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(u, num_sms));
    const int64_t rounds = (u + grid - 1) / grid;
    return (double)rounds * (300.0 + (double)kblocks * per_kb);
}

struct Affine {
    std::vector<double> scale, shift;
};

// Builds the launch list (no device work).  chain_bn > 0: plan every GEMM
// composite for the region kernel (tile or im2col mode, 64-wide k-blocks,
// BN = chain_bn, no split-K); plan_region then collapses them (make_chain).
byoc_status plan_region_impl(const byoc_region_desc *d, int num_sms, Plan &P, int chain_bn) {
    P = Plan();
    P.num_sms = num_sms > 0 ? num_sms : 148;
    byoc_status st = validate(d, P);
    if (st != BYOC_OK) return st;
    const int nt = d->n_tensors;
    std::vector<int> consumers(nt, 0), is_output(nt, 0), is_input(nt, 0);
    for (int o = 0; o < d->n_ops; ++o)
        for (int k = 0; k < d->ops[o].n_in; ++k) consumers[d->ops[o].in[k]]++;
    for (int id : P.outputs) is_output[id] = 1;
    for (int id : P.inputs) is_input[id] = 1;

    int o = 0;
    while (o < d->n_ops) {
        const byoc_op &op = d->ops[o];
        if (op.kind == BYOC_OP_QUANTIZE) {
            // a Q node that no epilogue absorbed (it reads a region input or
            // a tensor with other readers): its own launch
            if ((int)P.launches.size() >= BYOC_PLAN_MAX_LAUNCHES - 1)
                return fail(BYOC_ERR_UNSUPPORTED, "region needs more than %d launches", BYOC_PLAN_MAX_LAUNCHES - 1);
            LaunchPlan Q{};
            Q.kind = BYOC_LAUNCH_QUANT;
            Q.first_op = o;
            Q.n_ops = 1;
            Q.x = op.in[0];
            Q.y = op.out;
            Q.q_inv = (float)(1.0 / (double)op.consts[0][0]);
            Q.bytes = (double)P.tensors[op.in[0]].bytes() + (double)P.tensors[op.out].bytes();
            P.launches.push_back(Q);
            ++o;
            continue;
        }
        if (op.kind != BYOC_OP_CONV2D && op.kind != BYOC_OP_DENSE)
            return fail(BYOC_ERR_UNSUPPORTED,
                        "op %d (kind %d) is not preceded by a conv2d/dense it can fuse into; "
                        "standalone elementwise ops stay on the host",
                        o, op.kind);
        if ((int)P.launches.size() >= BYOC_PLAN_MAX_LAUNCHES - 1)
            return fail(BYOC_ERR_UNSUPPORTED, "region needs more than %d launches",
                        BYOC_PLAN_MAX_LAUNCHES - 1);
        const TensorInfo X = P.tensors[op.in[0]];
        const TensorInfo Yp = P.tensors[op.out];
        const int64_t Cout = Yp.channels();
        // ---------------- epilogue chain
        // Epilogue chain of the conv2d/dense at op `first`: the bias / batch
        // norm (folded into af), residual add and activation ops that follow
        // it, each the single consumer of the previous one.  Returns the index
        // of the first op after the chain.
        int out8 = 0;
        float out_inv = 0.0f;
        // a Q node right after the chain is fused: the epilogue writes E4M3
        // codes (region kernel: after any conv2d / dense; per-composite
        // kernel: after an FP8 one)
        const bool fuse_q = chain_bn > 0 ? (op.kind == BYOC_OP_DENSE || op.groups == 1)
                                         : X.dtype == BYOC_E4M3;
        auto walk_chain = [&](int first, Affine &af, int &cur, int &res, int &act) -> int {
            const int64_t Co = P.tensors[d->ops[first].out].channels();
            af.scale.assign(Co, 1.0);
            af.shift.assign(Co, 0.0);
            cur = d->ops[first].out;
            res = -1;
            act = byoc::kActNone;
            int stage = 0, jj = first + 1;
            for (; jj < d->n_ops; ++jj) {
                const byoc_op &nx = d->ops[jj];
                const bool reads_cur = nx.in[0] == cur || (nx.kind == BYOC_OP_ADD && nx.in[1] == cur);
                if (!reads_cur || consumers[cur] != 1 || is_output[cur]) break;
                if (nx.kind == BYOC_OP_BIAS_ADD && stage == 0) {
                    for (int64_t c = 0; c < Co; ++c) af.shift[c] += (double)nx.consts[0][c];
                } else if (nx.kind == BYOC_OP_BATCH_NORM && stage == 0) {
                    for (int64_t c = 0; c < Co; ++c) {
                        const double s = (double)nx.consts[0][c] /
                                         std::sqrt((double)nx.consts[3][c] + (double)nx.eps);
                        af.scale[c] *= s;
                        af.shift[c] = af.shift[c] * s + ((double)nx.consts[1][c] - s * (double)nx.consts[2][c]);
                    }
                } else if (nx.kind == BYOC_OP_ADD && stage == 0) {
                    const int r2 = nx.in[0] == cur ? nx.in[1] : nx.in[0];
                    if (r2 == cur) break;  // x + x: not a residual pattern
                    res = r2;
                    stage = 1;
                } else if (nx.kind == BYOC_OP_QUANTIZE && fuse_q && first == o) {
                    out8 = 1;
                    out_inv = (float)(1.0 / (double)nx.consts[0][0]);
                    cur = nx.out;
                    ++jj;
                    break;
                } else if ((nx.kind == BYOC_OP_RELU || nx.kind == BYOC_OP_RELU6 ||
                            nx.kind == BYOC_OP_GELU) && stage <= 1) {
                    act = nx.kind == BYOC_OP_RELU ? byoc::kActRelu
                                                  : (nx.kind == BYOC_OP_RELU6 ? byoc::kActRelu6
                                                                              : byoc::kActGelu);
                    stage = 2;
                } else {
                    break;
                }
                cur = nx.out;
            }
            return jj;
        };
        Affine af;
        int cur, res, act;
        const int j = walk_chain(o, af, cur, res, act);
        const TensorInfo Y = P.tensors[cur];
        LaunchPlan L{};
        L.first_op = o;
        L.n_ops = j - o;
        L.x = op.in[0];
        L.y = cur;
        L.res = res;
        L.act = act;
        if (Cout % 8)
            return fail(BYOC_ERR_UNSUPPORTED, "op %d: %lld output channels (multiple of 8 needed)",
                        o, (long long)Cout);
        if (X.dtype == BYOC_E4M3 && X.channels() % byoc::kF8BK)
            return fail(BYOC_ERR_UNSUPPORTED, "op %d: FP8 on %lld input channels (whole k-blocks of %d codes)",
                        o, (long long)X.channels(), byoc::kF8BK);

        if (op.kind == BYOC_OP_CONV2D && op.groups > 1) {
            // ---------------- depthwise
            const int64_t C = X.channels();
            if (op.groups != C || Cout != C)
                return fail(BYOC_ERR_UNSUPPORTED, "op %d: grouped conv other than depthwise", o);
            if (op.kernel[0] != 3 || op.kernel[1] != 3 || op.dilation[0] != 1 ||
                op.dilation[1] != 1 || op.stride[0] != op.stride[1] ||
                (op.stride[0] != 1 && op.stride[0] != 2) || op.pad[0] != op.pad[1] ||
                op.pad[0] != op.pad[2] || op.pad[1] != op.pad[3])
                return fail(BYOC_ERR_UNSUPPORTED,
                            "op %d: depthwise supports 3x3, stride 1|2, symmetric padding", o);
            if (res >= 0) return fail(BYOC_ERR_UNSUPPORTED, "op %d: residual add after depthwise", o);
            std::vector<float> w(9 * C), b(C);
            for (int64_t c = 0; c < C; ++c) {
                for (int t = 0; t < 9; ++t)
                    w[t * C + c] = (float)((double)op.consts[0][c * 9 + t] * af.scale[c]);
                b[c] = (float)af.shift[c];
            }
            // Depthwise -> 1x1 conv in one launch (dwpw.cu) when the 1x1 conv
            // is the depthwise output's only consumer: the intermediate stays
            // in shared memory (the gain of merging the two composites into
            // one region).
            if ((d->options & BYOC_OPT_FUSE_DW_PW) && j < d->n_ops && consumers[cur] == 1 && !is_output[cur] &&
                act != byoc::kActGelu) {
                const byoc_op &pw = d->ops[j];
                if (pw.kind == BYOC_OP_CONV2D && pw.in[0] == cur && pw.groups == 1 && pw.kernel[0] == 1 &&
                    pw.kernel[1] == 1 && pw.stride[0] == 1 && pw.stride[1] == 1 && pw.dilation[0] == 1 &&
                    pw.dilation[1] == 1 && pw.pad[0] == 0 && pw.pad[1] == 0 && pw.pad[2] == 0 && pw.pad[3] == 0) {
                    Affine af2;
                    int cur2, res2, act2;
                    const int j2 = walk_chain(j, af2, cur2, res2, act2);
                    const TensorInfo Y2 = P.tensors[cur2];
                    const int64_t Cout2 = Y2.channels();
                    byoc::DwPwArgs dp{};
                    dp.N = (int)X.shape[0];
                    dp.H = (int)X.shape[1];
                    dp.W = (int)X.shape[2];
                    dp.C = (int)C;
                    dp.Ho = (int)Y.shape[1];
                    dp.Wo = (int)Y.shape[2];
                    dp.stride = op.stride[0];
                    dp.pad = op.pad[0];
                    dp.dw_act = act;
                    dp.act = act2;
                    dp.Cout = (int)Cout2;
                    if (act2 != byoc::kActGelu && byoc::dwpw_plan(dp, P.num_sms)) {
                        L.kind = BYOC_LAUNCH_DWPW;
                        L.n_ops = j2 - o;
                        L.y = cur2;
                        L.res = res2;
                        L.act = act2;
                        L.w_off = blob_append(P.blob, w.data(), w.size() * 4);
                        L.w_bytes = w.size() * 4;
                        L.b_off = blob_append(P.blob, b.data(), b.size() * 4);
                        L.b_bytes = b.size() * 4;
                        // 1x1 weights: folded, bf16 RNE, [n_pad][chunks * 64] K-major, zero padded
                        L.n_pad = dp.n_pad;
                        L.k_pack = dp.chunks * byoc::kDpChunk;
                        std::vector<uint16_t> w2((size_t)L.n_pad * L.k_pack, 0);
                        for (int64_t k = 0; k < Cout2; ++k)
                            for (int64_t c = 0; c < C; ++c)
                                w2[(size_t)k * L.k_pack + c] =
                                    f32_to_bf16_rne((float)((double)pw.consts[0][k * C + c] * af2.scale[k]));
                        std::vector<float> b2((size_t)L.n_pad, 0.0f);
                        for (int64_t k = 0; k < Cout2; ++k) b2[k] = (float)af2.shift[k];
                        L.w2_off = blob_append(P.blob, w2.data(), w2.size() * 2);
                        L.w2_bytes = w2.size() * 2;
                        L.b2_off = blob_append(P.blob, b2.data(), b2.size() * 4);
                        L.b2_bytes = b2.size() * 4;
                        L.dp = dp;
                        L.grid = std::min(dp.num_tiles, P.num_sms);
                        L.flops = 2.0 * (double)Y.elems() * 9.0 + 2.0 * (double)Y2.elems() * (double)C;
                        L.bytes = (double)X.bytes() + (double)Y2.bytes() +
                                  (res2 >= 0 ? (double)P.tensors[res2].bytes() : 0.0) +
                                  (double)(w.size() + b.size()) * 4 + (double)Cout2 * C * 2 + (double)Cout2 * 4;
                        P.launches.push_back(L);
                        o = j2;
                        continue;
                    }
                }
            }
            L.kind = BYOC_LAUNCH_DEPTHWISE;
            L.w_off = blob_append(P.blob, w.data(), w.size() * 4);
            L.w_bytes = w.size() * 4;
            L.b_off = blob_append(P.blob, b.data(), b.size() * 4);
            L.b_bytes = b.size() * 4;
            L.dw.N = (int)X.shape[0];
            L.dw.H = (int)X.shape[1];
            L.dw.W = (int)X.shape[2];
            L.dw.C = (int)C;
            L.dw.Ho = (int)Y.shape[1];
            L.dw.Wo = (int)Y.shape[2];
            L.dw.stride = op.stride[0];
            L.dw.pad = op.pad[0];
            L.dw.act = act;
            if (!byoc::dw_plan(L.dw, P.num_sms))
                return fail(BYOC_ERR_UNSUPPORTED, "op %d: depthwise tile does not fit shared memory", o);
            L.grid = std::min(L.dw.num_tiles, P.num_sms);
            L.flops = 2.0 * (double)Y.elems() * 9.0;
            L.bytes = (double)X.bytes() + (double)Y.bytes() + (double)(w.size() + b.size()) * 4;
            P.launches.push_back(L);
            o = j;
            continue;
        }

        // ---------------- GEMM (conv2d groups=1, or dense)
        int64_t M, Kreal;
        int64_t stem_k = 0;     // > 0: the stem conv's reduction length (before the pixel-pair layout)
        int kh = 1, kw = 1, taps = 1, chunks, bk;
        int64_t C;
        std::vector<double> wsrc;  // weights as [Cout][kh][kw][C] (channel innermost)
        bool im2col = false;
        bool slab = false;
        SlabGeom sgeo{};
        if (op.kind == BYOC_OP_DENSE) {
            C = X.shape[1];
            M = X.shape[0];
            if (C % 8)
                return fail(BYOC_ERR_UNSUPPORTED, "op %d: dense input width %lld (multiple of 8)", o,
                            (long long)C);
            wsrc.assign(op.consts[0], op.consts[0] + Cout * C);
            L.aM = M;
            L.aK = C;
        } else {
            C = X.channels();
            kh = op.kernel[0];
            kw = op.kernel[1];
            M = Y.shape[0] * Y.shape[1] * Y.shape[2];
            const bool square = kh == kw && op.stride[0] == op.stride[1] &&
                                op.dilation[0] == op.dilation[1] && op.pad[0] == op.pad[1] &&
                                op.pad[2] == op.pad[3];
            if (C % 8) {
                // Few-channel stride-2 stem (k x k, k odd <= 7, C <= 4), run
                // as a stride-1 convolution over pixel pairs.  Output pixel
                // (p, q), filter tap (r, s = 2b + dx) reads input pixel
                // (2p + r - pad, 2q + 2b + dx - pad): with R >= k row taps
                // (4 or 8) and k2 = (k + 1) / 2 column taps b, the operand
                // row of slab position (p, j) is the R pixel pairs
                //   xq[2p + r][2j], xq[2p + r][2j + 1]   (r = 0 .. R-1)
                // of the boundary layout xq (4 channels, `pad` zero rows and
                // columns in front; StemArgs): 8R values in the order
                // r*8 + dx*4 + c, and tap b is that row read b positions on.
                // The GEMM loads it with a 5-D tensor map {8 values, R rows,
                // wp pairs, position rows (2 image rows apart), images}, so
                // the layout is the image's size (no stacked copy), and
                //   w'[k][b][r*8 + dx*4 + c] = w[k][c][r][2b + dx]   (0 outside the filter).
                if (!(square && op.stride[0] == 2 && op.dilation[0] == 1 && C <= 4 && (kh % 2) == 1 &&
                      kh <= 7))
                    return fail(BYOC_ERR_UNSUPPORTED,
                                "op %d: %lld input channels: only a stride-2 odd square stem (k <= 7) with "
                                "<= 4 channels is supported",
                                o, (long long)C);
                const int k2 = (kh + 1) / 2;
                const int R = kh <= 3 ? 4 : 8;
                const int Cz = 8 * R;
                if (X.shape[0] > 65535)
                    return fail(BYOC_ERR_UNSUPPORTED, "op %d: stem batch above 65535", o);
                // slab positions per output row: at least Wo + k2 - 1, and a
                // multiple of a group of G <= 32 pairs (G >= 16 where one
                // fits), so that the tensor map's innermost box dimension is
                // G contiguous pairs (16 G bytes), not one
                int64_t wpz = Y.shape[2] + k2 - 1;
                int G = (int)std::min<int64_t>(wpz, 32);
                if (wpz > 32) {
                    G = 0;
                    for (int64_t w = wpz; G == 0 && w <= wpz + 16; ++w)
                        for (int d = 32; d >= 16; --d)
                            if (w % d == 0) {
                                G = d;
                                wpz = w;
                                break;
                            }
                }
                if (wpz > 128)
                    return fail(BYOC_ERR_UNSUPPORTED,
                                "op %d: stem output %lld wide: a slab tile covers at most 128 positions "
                                "of one output row",
                                o, (long long)Y.shape[2]);
                // position rows the tensor map spans: the output rows and one
                // more, or a whole slab (single or pair) if that is more
                const int64_t tz = std::max<int64_t>(1, std::min<int64_t>(128 / wpz, Y.shape[1]));
                const int64_t pos_rows = std::max<int64_t>(
                    Y.shape[1] + 1, (tz * wpz + 128 + k2 - 1 + wpz - 1) / wpz);
                const int64_t Hq = 2 * (pos_rows - 1) + R;  // image rows they reach
                const int64_t Wq = 2 * wpz;
                if ((int64_t)X.shape[0] * Hq > INT32_MAX)
                    return fail(BYOC_ERR_UNSUPPORTED, "op %d: stem layout too large", o);
                TensorInfo Z{};
                Z.ndim = 4;
                Z.shape[0] = X.shape[0];
                Z.shape[1] = Hq;
                Z.shape[2] = Wq;
                Z.shape[3] = 4;
                const int zid = (int)P.tensors.size();
                P.tensors.push_back(Z);
                LaunchPlan S{};
                S.kind = BYOC_LAUNCH_S2D;
                S.x = op.in[0];
                S.y = zid;
                S.stem.N = (int)X.shape[0];
                S.stem.H = (int)X.shape[1];
                S.stem.W = (int)X.shape[2];
                S.stem.C = (int)C;
                S.stem.Hq = (int)Hq;
                S.stem.Wq = (int)Wq;
                S.stem.pad = op.pad[0];
                S.bytes = (double)X.bytes();  // xq is internal: not algorithmic traffic
                if (byoc::stem_layout_smem_bytes(S.stem) > byoc::kStemLayoutMaxSmem)
                    return fail(BYOC_ERR_UNSUPPORTED, "op %d: stem rows too wide (%lld x %lld)", o,
                                (long long)X.shape[2], (long long)C);
                P.launches.push_back(S);
                wsrc.assign((size_t)Cout * k2 * Cz, 0.0);
                for (int64_t k = 0; k < Cout; ++k)
                    for (int b = 0; b < k2; ++b)
                        for (int r = 0; r < kh; ++r)
                            for (int dx = 0; dx < 2; ++dx)
                                for (int64_t c = 0; c < C; ++c) {
                                    const int sx = 2 * b + dx;
                                    if (sx >= kw) continue;
                                    wsrc[((size_t)k * k2 + b) * Cz + r * 8 + dx * 4 + c] =
                                        op.consts[0][((k * C + c) * kh + r) * kw + sx];
                                }
                stem_k = (int64_t)kh * kw * C;  // the conv's own reduction length
                L.x = zid;
                L.stem_R = R;
                L.stem_G = G;
                C = Cz;
                kh = 1;
                kw = k2;
                im2col = true;
                // a 1 x k2 stride-1 conv over rows of wpz positions: tiles of
                // t output rows, slabs of `rows` position rows
                sgeo.wp = (int)wpz;
                sgeo.t = (int)tz;
                sgeo.rows = (int)((128 + k2 - 1 + wpz - 1) / wpz);
                sgeo.bytes = sgeo.rows * sgeo.wp * Cz * 2;
                slab = true;
                if (sgeo.bytes > byoc::slab_max_bytes(Cz))
                    return fail(BYOC_ERR_UNSUPPORTED, "op %d: stem slab of %d bytes", o, sgeo.bytes);
                L.geo = Im2colGeom{(int)X.shape[0], (int)Hq, (int)Wq, 4, 1, k2, 1, 1, 0, 0, 0, 0, 1, 1};
                L.args.stride_h = L.args.stride_w = 1;
                L.args.pad_t = L.args.pad_l = 0;
                L.args.dil_h = L.args.dil_w = 1;
            } else {
                wsrc.assign((size_t)Cout * kh * kw * C, 0.0);
                for (int64_t k = 0; k < Cout; ++k)
                    for (int r = 0; r < kh; ++r)
                        for (int s = 0; s < kw; ++s)
                            for (int64_t c = 0; c < C; ++c)
                                wsrc[((k * kh + r) * kw + s) * C + c] =
                                    op.consts[0][((k * C + c) * kh + r) * kw + s];
                const bool plain = kh == 1 && kw == 1 && op.stride[0] == 1 && op.stride[1] == 1 &&
                                   op.pad[0] == 0 && op.pad[1] == 0 && op.pad[2] == 0 &&
                                   op.pad[3] == 0;
                if (plain) {
                    L.aM = M;
                    L.aK = C;
                } else {
                    // im2col bounding-box corners must fit the 8-bit range of a
                    // 4-D map; filter-tap offsets the 16-bit instruction field
                    const int up_h = op.pad[2] - (kh - 1) * op.dilation[0];
                    const int up_w = op.pad[3] - (kw - 1) * op.dilation[1];
                    if (op.pad[0] > 128 || op.pad[1] > 128 || up_h < -128 || up_h > 127 ||
                        up_w < -128 || up_w > 127 || (kh - 1) * op.dilation[0] > 65535 ||
                        (kw - 1) * op.dilation[1] > 65535)
                        return fail(BYOC_ERR_UNSUPPORTED, "op %d: padding outside TMA im2col range", o);
                    im2col = true;
                    L.geo = Im2colGeom{(int)X.shape[0], (int)X.shape[1], (int)X.shape[2], (int)C,
                                       kh, kw, op.stride[0], op.stride[1], op.pad[0], op.pad[1],
                                       op.pad[2], op.pad[3], op.dilation[0], op.dilation[1]};
                    slab = chain_bn == 0 && X.dtype != BYOC_E4M3 && op.stride[0] == 1 && op.stride[1] == 1 && op.dilation[0] == 1 &&
                           op.dilation[1] == 1 && res < 0 &&
                           slab_geometry((int)X.shape[1], (int)X.shape[2], (int)Y.shape[1],
                                         (int)Y.shape[2], kh, kw, op.pad[0], op.pad[1], op.pad[3],
                                         pick_bk(C), sgeo);
                    L.args.stride_h = op.stride[0];
                    L.args.stride_w = op.stride[1];
                    L.args.pad_t = op.pad[0];
                    L.args.pad_l = op.pad[1];
                    L.args.dil_h = op.dilation[0];
                    L.args.dil_w = op.dilation[1];
                }
            }
        }
        taps = kh * kw;
        bk = op.kind == BYOC_OP_DENSE || chain_bn > 0 ? 64 : pick_bk(C);
        // an E4M3 input makes an FP8 layer; its k-blocks hold 128 codes (128
        // bytes, like 64 bf16 values).  The per-composite kernel takes them
        // as BK = kF8BK configurations (the region kernel keeps bk = 64 and
        // switches per stage).
        const bool fp8 = X.dtype == BYOC_E4M3;
        if (fp8 && chain_bn == 0) bk = byoc::kF8BK;
        const int kel = fp8 ? byoc::kF8BK : bk;
        chunks = (int)((C + kel - 1) / kel);
        const bool has_res = res >= 0;
        const int amode = slab ? byoc::kAModeSlab : (im2col ? byoc::kAModeIm2col : byoc::kAModeTile);
        const int64_t tiles_per_img = slab ? (Y.shape[1] + sgeo.t - 1) / sgeo.t : 0;
        const int64_t tiles_m = slab ? X.shape[0] * tiles_per_img : (M + 127) / 128;
        int splits = 1;
        bool cl_split = false;
        const int bn = chain_bn > 0 ? chain_bn
                                    : pick_bn(tiles_m, Cout, (int64_t)taps * chunks, bk, amode, has_res, P.num_sms,
                                              &splits, slab ? (double)sgeo.bytes / taps : 0.0, act == byoc::kActGelu,
                                              (d->options & BYOC_OPT_CLUSTER_SPLIT_K) ? &cl_split : nullptr);
        if (bn < 0)
            return fail(BYOC_ERR_UNSUPPORTED, "op %d: no compiled tile for BK=%d mode=%d residual=%d",
                        o, bk, amode, (int)has_res);
        L.cfg = GemmConfig{bn, bk,
                           splits > 1 ? (cl_split ? byoc::kAModeTileSplitCl : byoc::kAModeTileSplit) : amode,
                           has_res};
        if (slab && Cout <= bn) {
            // one column tile: keep the whole weight matrix in shared memory
            // when it fits beside two slabs
            const GemmConfig rc{bn, bk, byoc::kAModeSlabRes, false};
            if (byoc::gemm_config_supported(rc) && byoc::gemm_slab_res_fits(rc, taps * chunks, sgeo.bytes))
                L.cfg = rc;
        }
        // Cluster multicast of the weight tiles, on request (tile, im2col and
        // ringed slab modes without split-K; at least two m-tiles to pair)
        if (chain_bn == 0 && !fp8 && (d->options & BYOC_OPT_MULTICAST) && tiles_m >= 2 && P.num_sms >= 2 &&
            (L.cfg.amode == byoc::kAModeTile || L.cfg.amode == byoc::kAModeIm2col ||
             L.cfg.amode == byoc::kAModeSlab)) {
            GemmConfig mc = L.cfg;
            mc.mc = true;
            if (byoc::gemm_config_supported(mc)) L.cfg = mc;
        }
        int64_t units_m = tiles_m;  // m-units of the launch: tiles, or pairs of tiles
        if (slab && L.cfg.amode == byoc::kAModeSlabRes && (int64_t)taps * chunks * (bk / 16) <= 16) {
            // Pair units (two adjacent tiles sharing each weight k-block and
            // one slab) for resident-weight slabs with few MMAs per tile (the
            // stem's 16): they halve the per-unit cost of waits, commits and
            // descriptor set-up, which is a large part of such a tile.  With
            // more MMAs per tile the MMA rate is bound by the shared-memory
            // reads of its operands (A and B are read for every MMA), which
            // pairs do not reduce: measured on GB300, the 56x56 / 28x28 /
            // 14x14 ResNet-50 3x3 layers ran as fast or slower in pairs.
            // The estimate still rules out pairs that leave SMs idle.
            SlabGeom pg;
            const int64_t tn = (Cout + bn - 1) / bn;
            const int64_t pair_m = X.shape[0] * ((tiles_per_img + 1) / 2);
            if (slab_pair_geometry(kh, kw, bk, sgeo, pg)) {
                const GemmConfig pc{bn, bk, byoc::kAModeSlabRes2, false};
                const double single = slab_makespan(tiles_m, tn, (int64_t)taps * chunks, taps, bn, bk, 1, true,
                                                    sgeo.bytes, P.num_sms);
                const double pair = slab_makespan(pair_m, tn, (int64_t)taps * chunks, taps, bn, bk, 2, true,
                                                  pg.bytes, P.num_sms);
                if (byoc::gemm_config_supported(pc) && byoc::gemm_slab_res_fits(pc, taps * chunks, pg.bytes) &&
                    pair < single) {
                    L.cfg = pc;
                    units_m = pair_m;
                    sgeo = pg;
                }
            }
        }
        if (slab) {
            L.slab_rows = sgeo.rows;
            L.args.wp = sgeo.wp;
            L.args.slab_t = sgeo.t;
            L.args.tiles_per_img = (int)tiles_per_img;
            L.args.slab_bytes = sgeo.bytes;
        }
        L.n_pad = (int)((Cout + bn - 1) / bn * bn);
        L.k_pack = taps * chunks * kel;
        Kreal = stem_k > 0 ? stem_k : (int64_t)taps * C;
        if (fp8) {
            // FP8: the folded weights of output channel k quantized with the
            // power-of-two scale S_w[k] to E4M3 codes, K-major [n_pad][k_pack];
            // the epilogue multiplies by dq[k] = fp32(S_x S_w[k]), S_x the scale
            // of the Q node that wrote the input
            double sx = 0.0;
            for (int q = 0; q < o; ++q)
                if (d->ops[q].kind == BYOC_OP_QUANTIZE && d->ops[q].out == op.in[0]) sx = d->ops[q].consts[0][0];
            if (!(sx > 0.0)) return fail(BYOC_ERR_INVALID_ARG, "op %d: E4M3 input without a quantize op", o);
            std::vector<uint8_t> w8((size_t)L.n_pad * L.k_pack, 0);
            std::vector<float> dq((size_t)L.n_pad, 0.0f);
            for (int64_t k = 0; k < Cout; ++k) {
                double m = 0.0;
                for (size_t i = 0; i < (size_t)taps * C; ++i)
                    m = std::max(m, std::fabs(wsrc[(size_t)k * taps * C + i] * af.scale[k]));
                const double sw = e4m3_weight_scale(m);
                for (int t = 0; t < taps; ++t)
                    for (int64_t c = 0; c < C; ++c) {
                        const double v = wsrc[((size_t)k * taps + t) * C + c] * af.scale[k];
                        const size_t col = ((size_t)t * chunks + c / kel) * kel + c % kel;
                        w8[(size_t)k * L.k_pack + col] = e4m3_code(v / sw);
                    }
                dq[k] = (float)(sx * sw);
            }
            L.w_off = blob_append(P.blob, w8.data(), w8.size());
            L.w_bytes = w8.size();
            L.dq_off = blob_append(P.blob, dq.data(), dq.size() * 4);
            L.fp8 = 1;
        } else {
            // Folded, bf16-rounded, K-major packed weights [n_pad][k_pack].
            std::vector<uint16_t> wp((size_t)L.n_pad * L.k_pack, 0);
            for (int64_t k = 0; k < Cout; ++k)
                for (int t = 0; t < taps; ++t)
                    for (int64_t c = 0; c < C; ++c) {
                        const double v = wsrc[((size_t)k * taps + t) * C + c] * af.scale[k];
                        const size_t col = ((size_t)t * chunks + c / bk) * bk + c % bk;
                        wp[(size_t)k * L.k_pack + col] = f32_to_bf16_rne((float)v);
                    }
            L.w_off = blob_append(P.blob, wp.data(), wp.size() * 2);
            L.w_bytes = wp.size() * 2;
        }
        L.out8 = out8;
        L.out_inv = out_inv;
        std::vector<float> bias((size_t)L.n_pad, 0.0f);
        for (int64_t k = 0; k < Cout; ++k) bias[k] = (float)af.shift[k];
        L.b_off = blob_append(P.blob, bias.data(), bias.size() * 4);
        L.b_bytes = bias.size() * 4;

        GemmArgs &A = L.args;
        A.M = (int)M;
        A.N = (int)Cout;
        A.num_kb = taps * chunks;
        A.chunks = chunks;
        A.kw = kw;
        if (!im2col) {
            A.dil_h = A.dil_w = 1;
            A.stride_h = A.stride_w = 1;
        }
        A.Ho = op.kind == BYOC_OP_DENSE ? 1 : (int)Y.shape[1];
        A.Wo = op.kind == BYOC_OP_DENSE ? 1 : (int)Y.shape[2];
        A.tiles_n = L.n_pad / bn;
        A.num_tiles = (int)(units_m * A.tiles_n);
        A.taps = taps;
        A.stem_rows = L.stem_R;
        // a pair unit's k-block is twice the MMA work of a tile's
        A.group = byoc::gemm_group(byoc::amode_pair(L.cfg.amode) ? 2 * bn : bn, fp8 ? 64 : bk,
                                   amode == byoc::kAModeSlab ? taps : (A.num_kb + splits - 1) / splits);
        byoc::gemm_slab_pool(L.cfg, A);
        A.splits = splits;
        A.m_pad = (int)(tiles_m * byoc::kGemmBM);
        A.n_pad = L.n_pad;
        if (splits > 1 && !cl_split) {  // global split-K: partials and counters in the workspace
            L.part_bytes = (size_t)splits * A.m_pad * A.n_pad * 4;
            L.cnt_bytes = (size_t)A.num_tiles * 8 * 4;
        }
        L.grid = std::min(A.num_tiles * splits, P.num_sms);
        // Short reductions over several rounds of tiles: a grid that is a
        // multiple of the column tiles keeps every CTA in one column tile, so
        // the kernel keeps its weight k-blocks in the ring (gemm.cu) -- at most
        // tiles_n - 1 SMs idle (none for 2, 4 or 8 column tiles)
        if (splits == 1 && !L.cfg.mc && !slab && !has_res && A.tiles_n > 1 && A.tiles_n <= 8 && A.num_kb <= 4 &&
            A.num_tiles >= 3 * P.num_sms && P.num_sms >= A.tiles_n)
            L.grid = P.num_sms / A.tiles_n * A.tiles_n;
        if (L.cfg.mc)  // whole clusters: one per pair of m-tiles of a column tile, at most num_sms / 2
            L.grid = 2 * (int)std::min<int64_t>((units_m + 1) / 2 * A.tiles_n, P.num_sms / 2);
        A.act = act;
        L.flops = 2.0 * (double)M * (double)Kreal * (double)Cout;
        const double in_bytes = stem_k > 0 ? 0.0  // xq: the image is counted by the layout transform
                                : L.x < P.n_region_tensors ? (double)X.bytes()
                                                           : (double)P.tensors[L.x].bytes();
        L.bytes = in_bytes + (double)Y.bytes() + (double)Cout * Kreal * (fp8 ? 1 : 2) + (double)Cout * 4 +
                  (res >= 0 ? (double)P.tensors[res].bytes() : 0.0);
        P.launches.push_back(L);
        o = j;
    }
    // Workspace: every tensor that is neither a region input nor output.
    P.ws_off.assign(P.tensors.size(), SIZE_MAX);
    size_t ws = 256;  // [0, 256): device error word
    for (size_t t = 0; t < P.tensors.size(); ++t) {
        const bool boundary = (int)t < nt && (is_input[t] || is_output[t]);
        if (boundary) continue;
        bool used = false;
        for (const LaunchPlan &L : P.launches) used |= (L.x == (int)t || L.y == (int)t || L.res == (int)t);
        if (!used) continue;
        P.ws_off[t] = ws;
        ws = align_up(ws + P.tensors[t].bytes(), 256);
    }
    for (LaunchPlan &L : P.launches) {
        if (L.part_bytes) {
            L.part_off = ws;
            ws = align_up(ws + L.part_bytes, 256);
            L.cnt_off = ws;
            ws = align_up(ws + L.cnt_bytes, 256);
        }
    }
    P.ws_bytes = ws;
    for (const LaunchPlan &L : P.launches) {
        P.flops += L.flops;
        P.bytes += L.bytes;
    }
    return BYOC_OK;
}

// Region kernel: collapse a plan of 2 .. kChainMaxStages GEMM launches, made
// by plan_region_impl with chain_bn = bn, into one BYOC_LAUNCH_CHAIN launch.
// Returns false, leaving P unchanged, when the region does not qualify.
//
// Dependencies of a unit (stage s, m-tile mt) on the stage p that wrote its A
// operand: tile mode reads rows [m0, m1] of p's output, the same pixels p
// computed as its rows [m0, m1]; im2col mode reads, for output pixels
// (n0, oh0) .. (n1, oh1), input rows oh0 * sh - pt .. oh1 * sh - pt + (kh - 1)
// * dh of images n0 .. n1 (clamped to the image), which lie in the contiguous
// range of p's rows from (n0, first row, 0) to (n1, last row, W - 1).  On the
// stage that wrote its residual: rows [m0, m1].  Either way the unit waits
// for the completion counters of p's m-tiles over those rows (every column
// tile of p).
bool make_chain(Plan &P, int bn) {
    // leading Q nodes on region inputs stay launches of their own
    int q0 = 0;
    while (q0 < (int)P.launches.size() && P.launches[q0].kind == BYOC_LAUNCH_QUANT) ++q0;
    std::vector<LaunchPlan> quants(P.launches.begin(), P.launches.begin() + q0);
    P.launches.erase(P.launches.begin(), P.launches.begin() + q0);
    const int ns = (int)P.launches.size();
    bool any8 = false;
    for (const LaunchPlan &L : P.launches) any8 |= L.fp8 != 0;
    // a single bf16 GEMM stays with the per-composite kernel
    auto undo = [&]() {
        P.launches.insert(P.launches.begin(), quants.begin(), quants.end());
        return false;
    };
    if (ns < (any8 ? 1 : 2) || ns > byoc::kChainMaxStages) return undo();
    for (const LaunchPlan &L : P.launches) {
        if (L.kind != BYOC_LAUNCH_GEMM || L.cfg.bk != 64 || L.cfg.bn != bn || L.stem_R != 0 || L.x_off ||
            L.y_off)
            return undo();
        if (L.cfg.amode != byoc::kAModeTile && L.cfg.amode != byoc::kAModeIm2col) return undo();
        // whole 128-byte k-blocks: 64 bf16 channels, or 128 E4M3 channels
        if ((L.cfg.amode == byoc::kAModeTile ? L.aK : (int64_t)L.geo.C) % (L.fp8 ? 128 : 64)) return undo();
        if (L.args.N % 32) return undo();  // the epilogue reads residual rows in 32-column pieces
        if (L.res >= 0 && P.tensors[L.res].dtype != BYOC_BF16) return undo();
        if (L.args.num_tiles != (L.args.M + byoc::kGemmBM - 1) / byoc::kGemmBM * L.args.tiles_n) return undo();
    }
    LaunchPlan C{};
    C.kind = BYOC_LAUNCH_CHAIN;
    C.chain_bn = bn;
    C.first_op = P.launches[0].first_op;
    C.x = P.launches[0].x;
    C.y = P.launches.back().y;
    C.res = P.launches.back().res;
    C.act = P.launches.back().act;
    byoc::ChainArgs &A = C.chain;
    A.n_stages = ns;
    int units = 0;
    double wbytes = 0;
    for (int s = 0; s < ns; ++s) {
        const LaunchPlan &L = P.launches[s];
        byoc::ChainStage &cs = A.st[s];
        cs.mode = L.cfg.amode == byoc::kAModeIm2col ? byoc::kChainIm2col : byoc::kChainTile;
        cs.M = L.args.M;
        cs.N = L.args.N;
        cs.num_kb = L.args.num_kb;
        cs.chunks = L.args.chunks;
        cs.kw = L.args.kw;
        cs.dil_h = L.args.dil_h;
        cs.dil_w = L.args.dil_w;
        cs.Ho = L.args.Ho;
        cs.Wo = L.args.Wo;
        cs.stride_h = L.args.stride_h;
        cs.stride_w = L.args.stride_w;
        cs.pad_t = L.args.pad_t;
        cs.pad_l = L.args.pad_l;
        cs.tiles_n = L.args.tiles_n;
        cs.num_tiles = L.args.num_tiles;
        cs.unit0 = units;
        units += cs.num_tiles;
        cs.act = L.act;
        cs.fp8 = L.fp8;
        cs.out8 = L.out8;
        cs.out_inv = L.out_inv;
        C.c_dq_off[s] = L.dq_off;
        C.n_ops += L.n_ops;
        C.cx[s] = L.x;
        C.cy[s] = L.y;
        C.cres[s] = L.res;
        C.cgeo[s] = L.geo;
        C.caM[s] = L.aM;
        C.caK[s] = L.aK;
        C.c_npad[s] = L.n_pad;
        C.c_kpack[s] = L.k_pack;
        C.cw_off[s] = L.w_off;
        C.cb_off[s] = L.b_off;
        C.flops += L.flops;
        // weights once: 2 M N K flops -> N K bf16 (E4M3) weights, N fp32 biases
        wbytes += L.flops / (2.0 * cs.M) * (L.fp8 ? 1.0 : 2.0) + (double)cs.N * (L.fp8 ? 8.0 : 4.0);
    }
    A.total_units = units;
    int ncnt = 0;
    for (int s = 0; s < ns; ++s) {
        A.st[s].cbase = ncnt;
        ncnt += (A.st[s].M + byoc::kGemmBM - 1) / byoc::kGemmBM;
    }
    A.n_counters = ncnt;
    auto producer = [&](int tensor, int before) -> int {
        for (int p = 0; p < before; ++p)
            if (C.cy[p] == tensor) return p;
        return -1;
    };
    // Dependencies in the stages' own numbering (unit = unit0 + tile), as
    // (counter, count per launch).
    std::vector<std::vector<std::pair<int32_t, int32_t>>> udeps(units);
    std::vector<int> ustage(units), utile(units);
    for (int s = 0; s < ns; ++s) {
        byoc::ChainStage &cs = A.st[s];
        const int pa = producer(C.cx[s], s), pr = C.cres[s] >= 0 ? producer(C.cres[s], s) : -1;
        if (pa >= 0) A.st[pa].consumed = 1;
        if (pr >= 0) A.st[pr].consumed = 1;
        cs.res_dep = pr >= 0 ? 1 : 0;
        for (int tile = 0; tile < cs.num_tiles; ++tile) {
            const int u = cs.unit0 + tile;
            ustage[u] = s;
            utile[u] = tile;
            const int mt = tile / cs.tiles_n, nt = tile % cs.tiles_n;
            const int64_t m0 = (int64_t)mt * byoc::kGemmBM;
            const int64_t m1 = std::min<int64_t>(m0 + byoc::kGemmBM, cs.M) - 1;
            std::vector<std::pair<int32_t, int32_t>> &d = udeps[u];
            auto add_rows = [&](int p, int64_t lo, int64_t hi) {
                const byoc::ChainStage &ps = A.st[p];
                hi = std::min<int64_t>(hi, (int64_t)ps.M - 1);
                for (int64_t pm = lo / byoc::kGemmBM; pm <= hi / byoc::kGemmBM; ++pm)
                    d.emplace_back(ps.cbase + (int)pm, byoc::kGemmEpiWarps * ps.tiles_n);
            };
            if (pa >= 0) {
                int64_t lo = m0, hi = m1;
                if (cs.mode == byoc::kChainIm2col) {
                    const Im2colGeom &g = C.cgeo[s];
                    const int64_t hw = (int64_t)cs.Ho * cs.Wo;
                    const int64_t n0 = m0 / hw, oh0 = (m0 % hw) / cs.Wo;
                    const int64_t n1 = m1 / hw, oh1 = (m1 % hw) / cs.Wo;
                    const int64_t ih0 = std::max<int64_t>(0, oh0 * g.sh - g.pt);
                    const int64_t ih1 =
                        std::max<int64_t>(0, std::min<int64_t>(g.H - 1, oh1 * g.sh - g.pt + (int64_t)(g.kh - 1) * g.dh));
                    lo = n0 * g.H * g.W + ih0 * g.W;
                    hi = std::max(lo, n1 * g.H * g.W + ih1 * g.W + g.W - 1);
                }
                add_rows(pa, lo, hi);
            }
            if (pr >= 0) {
                if (A.st[pr].M != cs.M) return false;
                add_rows(pr, m0, m1);
            }
            std::sort(d.begin(), d.end());
            d.erase(std::unique(d.begin(), d.end()), d.end());
        }
    }
    // The order units are handed out in: a list schedule of the launch on
    // the grid's CTAs with estimated durations (SM cycles).  A unit's
    // mainloop costs per k-block the larger of its MMA time (4 x 64 cycles
    // at BN = 128, 4 x 128 at BN = 256) and its operand bytes at ~60 B per
    // cycle into the SM; its epilogue ~400 cycles per two 32-column chunks
    // (+ 300 with a residual).  Repeatedly, the CTA that frees first takes
    // the unit that can start earliest among those whose dependencies are all
    // scheduled (ties: stage-major order); it frees again when the unit's
    // loads are issued (the epilogue overlaps the next unit).
    const int grid = std::min(units, P.num_sms);
    std::vector<double> main_c(ns), epi_c(ns);
    for (int s = 0; s < ns; ++s) {
        const double mma = 4.0 * (bn == 256 ? 128.0 : 64.0);
        const double ingest = (double)(byoc::kGemmBM * 64 * 2 + bn * 64 * 2) / 60.0;
        main_c[s] = 300.0 + A.st[s].num_kb * std::max(mma, ingest);
        epi_c[s] = 400.0 * (double)((bn / 32 + 1) / 2) + (C.cres[s] >= 0 ? 300.0 : 0.0);
    }
    std::vector<int> remaining(ncnt, 0);
    std::vector<double> cnt_done(ncnt, 0.0);
    for (int u = 0; u < units; ++u) {
        const byoc::ChainStage &cs = A.st[ustage[u]];
        remaining[cs.cbase + utile[u] / cs.tiles_n]++;
    }
    std::vector<double> cta_free(grid, 0.0);
    std::vector<char> taken(units, 0);
    std::vector<int> ord, ord_cta;
    ord.reserve(units);
    ord_cta.reserve(units);
    for (int i = 0; i < units; ++i) {
        const int c = (int)(std::min_element(cta_free.begin(), cta_free.end()) - cta_free.begin());
        const double f = cta_free[c];
        int best = -1;
        double best_start = 0;
        for (int u = 0; u < units; ++u) {
            if (taken[u]) continue;
            double ready = 0;
            bool ok = true;
            for (const auto &dp : udeps[u]) {
                if (remaining[dp.first] > 0) {
                    ok = false;
                    break;
                }
                ready = std::max(ready, cnt_done[dp.first]);
            }
            if (!ok) continue;
            const double st0 = std::max(f, ready);
            if (best < 0 || st0 < best_start - 1e-9) {
                best = u;
                best_start = st0;
            }
            if (st0 <= f) break;  // cannot start any earlier: keep stage-major order
        }
        taken[best] = 1;
        ord.push_back(best);
        ord_cta.push_back(c);
        const int sb = ustage[best];
        const int cnt = A.st[sb].cbase + utile[best] / A.st[sb].tiles_n;
        remaining[cnt]--;
        cnt_done[cnt] = std::max(cnt_done[cnt], best_start + main_c[sb] + epi_c[sb]);
        cta_free[c] = best_start + main_c[sb];
    }
    std::vector<int32_t> order(units), off(1, 0), list;
    for (int i = 0; i < units; ++i) {
        const int u = ord[i];
        order[i] = (ustage[u] << 24) | utile[u];
        for (const auto &c : udeps[u]) {
            list.push_back(c.first);
            list.push_back(c.second);
        }
        off.push_back((int32_t)(list.size() / 2));
    }
    if (list.empty()) list.assign(2, 0);  // keeps the blob offset valid; never read
    // each CTA's units, in the global order, as records (unit, code,
    // dependency count, first dependency, the first kChainRecDeps pairs)
    std::vector<int32_t> cta_off(grid + 1, 0), cta_rec((size_t)units * byoc::kChainRecInts, 0);
    for (int i = 0; i < units; ++i) cta_off[ord_cta[i] + 1]++;
    for (int b = 0; b < grid; ++b) cta_off[b + 1] += cta_off[b];
    {
        std::vector<int32_t> fill(cta_off.begin(), cta_off.end() - 1);
        for (int i = 0; i < units; ++i) {
            int32_t *r = &cta_rec[(size_t)fill[ord_cta[i]]++ * byoc::kChainRecInts];
            r[0] = i;
            r[1] = order[i];
            r[2] = off[i + 1] - off[i];
            r[3] = off[i];
            for (int k = 0; k < std::min(r[2], byoc::kChainRecDeps); ++k) {
                r[4 + 2 * k] = list[2 * (off[i] + k)];
                r[5 + 2 * k] = list[2 * (off[i] + k) + 1];
            }
        }
    }
    C.cta_off_off = blob_append(P.blob, cta_off.data(), cta_off.size() * 4);
    C.cta_rec_off = blob_append(P.blob, cta_rec.data(), cta_rec.size() * 4);
    C.order_off = blob_append(P.blob, order.data(), order.size() * 4);
    C.dep_off_off = blob_append(P.blob, off.data(), off.size() * 4);
    C.dep_list_off = blob_append(P.blob, list.data(), list.size() * 4);
    // algorithmic bytes: what the stages read from outside the chain (region
    // inputs, quantized inputs) and the region's outputs once, the weights once
    double io = 0;
    std::vector<int> seen_in;
    for (int s = 0; s < ns; ++s)
        for (int t : {C.cx[s], C.cres[s]}) {
            if (t < 0 || producer(t, ns) >= 0 || std::find(seen_in.begin(), seen_in.end(), t) != seen_in.end())
                continue;
            seen_in.push_back(t);
            io += (double)P.tensors[t].bytes();
        }
    for (int t : P.outputs) io += (double)P.tensors[t].bytes();
    C.bytes = io + wbytes;
    C.grid = grid;
    // workspace: 4 control words, then one completion counter per m-tile
    C.flags_off = P.ws_bytes;
    C.flags_bytes = align_up(16 + 4 * (size_t)ncnt, 256);
    P.ws_bytes += C.flags_bytes;
    P.launches = quants;
    P.launches.push_back(C);
    P.flops = C.flops;
    P.bytes = C.bytes;
    for (const LaunchPlan &Q : quants) P.bytes += Q.bytes;
    return true;
}

byoc_status plan_region(const byoc_region_desc *d, int num_sms, Plan &P) {
    if (d && d->abi_version == BYOC_ABI_VERSION && (d->options & BYOC_OPT_REGION_KERNEL)) {
        Plan C;
        if (plan_region_impl(d, num_sms, C, 128) == BYOC_OK && make_chain(C, 128)) {
            P = std::move(C);
            return BYOC_OK;
        }
    }
    return plan_region_impl(d, num_sms, P, 0);
}

void fill_report(const Plan &P, byoc_plan_report *r) {
    std::memset(r, 0, sizeof *r);
    r->n_launches = (int32_t)P.launches.size();
    for (size_t i = 0; i < P.launches.size(); ++i) {
        const LaunchPlan &L = P.launches[i];
        r->kind[i] = L.kind;
        r->first_op[i] = L.first_op;
        r->n_ops[i] = L.n_ops;
        r->act[i] = L.act;
        r->residual[i] = L.res;
        const bool dp = L.kind == BYOC_LAUNCH_DWPW;
        r->gemm_m[i] = L.kind == BYOC_LAUNCH_GEMM ? L.args.M : (dp ? L.dp.N * L.dp.Ho * L.dp.Wo : 0);
        r->gemm_n[i] = L.kind == BYOC_LAUNCH_GEMM ? L.args.N : (dp ? L.dp.Cout : 0);
        r->gemm_k[i] = L.kind == BYOC_LAUNCH_GEMM ? L.k_pack : (dp ? L.dp.C : 0);
        r->tile_n[i] = L.kind == BYOC_LAUNCH_GEMM ? L.cfg.bn : (dp ? L.dp.n_pad : 0);
        r->tile_k[i] = L.kind == BYOC_LAUNCH_GEMM ? L.cfg.bk : (dp ? byoc::kDpChunk : 0);
        r->im2col[i] = L.kind != BYOC_LAUNCH_GEMM || byoc::amode_split(L.cfg.amode)
                           ? 0
                           : std::min(L.cfg.amode, (int)byoc::kAModeSlab);
        r->splits[i] = L.kind == BYOC_LAUNCH_GEMM ? std::max(1, L.args.splits) : 0;
        r->grid[i] = L.grid;
        const bool gm = L.kind == BYOC_LAUNCH_GEMM;
        r->resident_b[i] = gm && byoc::amode_wres(L.cfg.amode) ? 1 : 0;
        r->slab_slots[i] = !gm || !byoc::amode_slab(L.cfg.amode) ? 0
                           : byoc::amode_wres(L.cfg.amode)      ? L.args.slab_slots
                                                                : 2;
        r->pair_units[i] = gm && byoc::amode_pair(L.cfg.amode) ? 1 : 0;
        r->multicast[i] = gm && L.cfg.mc ? 1 : 0;
        r->stages[i] = 1;
        r->fp8[i] = L.kind == BYOC_LAUNCH_GEMM ? L.fp8 : 0;
        if (L.kind == BYOC_LAUNCH_CHAIN) {
            r->fp8[i] = 0;
            for (int k = 0; k < L.chain.n_stages; ++k) r->fp8[i] += L.chain.st[k].fp8;
            const byoc::ChainStage &s0 = L.chain.st[0];
            r->stages[i] = L.chain.n_stages;
            r->units[i] = L.chain.total_units;
            r->gemm_m[i] = s0.M;
            r->gemm_n[i] = s0.N;
            r->gemm_k[i] = L.c_kpack[0];
            r->tile_n[i] = L.chain_bn;
            r->tile_k[i] = 64;
            r->im2col[i] = s0.mode == byoc::kChainIm2col ? 1 : 0;
            r->splits[i] = 1;
        }
    }
    r->flops = P.flops;
    r->bytes = P.bytes;
    r->const_bytes = P.blob.size();
    r->workspace_bytes = P.ws_bytes;
}

}  // namespace

namespace byoc {
void set_last_error(const char *msg) { g_err = msg ? msg : ""; }
}  // namespace byoc

// ------------------------------------------------------------ the handle

struct byoc_handle {
    Plan P;
    int sms = 0;  // SMs of the device the handle was instantiated on
    uint8_t *d_const = nullptr;
    uint8_t *d_ws = nullptr;
    int *d_err = nullptr;
    int device = 0;
    std::vector<CUtensorMap> tmB;         // per launch (GEMM only)
    std::vector<CUtensorMap> tmA;         // per launch, cached
    std::vector<const void *> tmA_ptr;    // pointer each cached A map encodes
    std::vector<CUtensorMap> tmR;         // per launch: residual map, cached
    std::vector<const void *> tmR_ptr;
    std::vector<CUtensorMap> tmO;         // per launch: output map (tile mode), cached
    std::vector<const void *> tmO_ptr;
    std::vector<byoc::ChainMaps> cmaps;   // per launch: region kernel maps (A, O cached; B fixed)
    std::vector<std::vector<const void *>> cptr;  // per launch: pointers the A [0, 4) and O [4, 8) maps encode
    std::vector<void *> ptrs;             // scratch: resolved tensor pointers
};

extern "C" {

const char *byoc_last_error(void) { return g_err.c_str(); }

byoc_status byoc_plan(const byoc_region_desc *desc, int32_t num_sms, byoc_plan_report *rep) {
    if (!rep) return fail(BYOC_ERR_INVALID_ARG, "null report");
    Plan P;
    byoc_status st = plan_region(desc, num_sms, P);
    if (st != BYOC_OK) return st;
    fill_report(P, rep);
    return BYOC_OK;
}

byoc_status byoc_plan_constants(const byoc_region_desc *desc, int32_t num_sms, int32_t launch,
                                int32_t what, void *dst, size_t dst_bytes, size_t *needed) {
    Plan P;
    byoc_status st = plan_region(desc, num_sms, P);
    if (st != BYOC_OK) return st;
    if (launch < 0 || launch >= (int)P.launches.size())
        return fail(BYOC_ERR_INVALID_ARG, "launch %d out of range", launch);
    const LaunchPlan &L = P.launches[launch];
    if (L.kind == BYOC_LAUNCH_S2D || L.kind == BYOC_LAUNCH_CHAIN)
        return fail(BYOC_ERR_INVALID_ARG, "launch %d has no constants of its own", launch);
    if ((what < 0 || what > 3) || (what > 1 && L.kind != BYOC_LAUNCH_DWPW))
        return fail(BYOC_ERR_INVALID_ARG, "launch %d has no constants of kind %d", launch, what);
    const size_t off = what == 0 ? L.w_off : what == 1 ? L.b_off : what == 2 ? L.w2_off : L.b2_off;
    const size_t n = what == 0 ? L.w_bytes : what == 1 ? L.b_bytes : what == 2 ? L.w2_bytes : L.b2_bytes;
    if (needed) *needed = n;
    if (!dst) return BYOC_OK;
    if (dst_bytes < n) return fail(BYOC_ERR_INVALID_ARG, "destination too small (%zu < %zu)", dst_bytes, n);
    std::memcpy(dst, P.blob.data() + off, n);
    return BYOC_OK;
}

byoc_status byoc_device_info(int32_t *num_sms, int32_t *cc_major, int32_t *cc_minor) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    int v = 0;
    if (num_sms) {
        if ((e = cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
            return cuda_fail(e, "cudaDeviceGetAttribute");
        *num_sms = v;
    }
    if (cc_major) {
        if ((e = cudaDeviceGetAttribute(&v, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess)
            return cuda_fail(e, "cudaDeviceGetAttribute");
        *cc_major = v;
    }
    if (cc_minor) {
        if ((e = cudaDeviceGetAttribute(&v, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess)
            return cuda_fail(e, "cudaDeviceGetAttribute");
        *cc_minor = v;
    }
    return BYOC_OK;
}

void byoc_release(byoc_handle *h) {
    if (!h) return;
    int cur = -1;
    cudaGetDevice(&cur);
    if (cur != h->device) cudaSetDevice(h->device);
    if (h->d_const) cudaFree(h->d_const);
    if (h->d_ws) cudaFree(h->d_ws);
    if (cur >= 0 && cur != h->device) cudaSetDevice(cur);
    delete h;
}

}  // extern "C"

namespace {

// The current device must be an sm_103 GPU; returns its SM count.
byoc_status check_device(int32_t *sms) {
    int32_t ccM = 0, ccm = 0;
    byoc_status st = byoc_device_info(sms, &ccM, &ccm);
    if (st != BYOC_OK) return st;
    if (ccM != 10 || ccm != 3)
        return fail(BYOC_ERR_UNSUPPORTED, "device is sm_%d%d; this library is built for sm_103a", ccM, ccm);
    cudaError_t e = load_driver();
    if (e != cudaSuccess) return cuda_fail(e, "driver entry points for TMA descriptors");
    return BYOC_OK;
}

// Device half of byoc_compile / byoc_deserialize: h->P is a complete plan.
// Uploads the constants, allocates the workspace, binds the device pointers
// into the launch arguments, encodes the weight TMA descriptors and raises
// the kernels' shared-memory limits.  Releases h on failure.
byoc_status instantiate(byoc_handle *h, byoc_handle **out) {
    cudaError_t e;
    cudaGetDevice(&h->device);
    if ((e = cudaDeviceGetAttribute(&h->sms, cudaDevAttrMultiProcessorCount, h->device)) != cudaSuccess) {
        byoc_release(h);
        return cuda_fail(e, "cudaDeviceGetAttribute");
    }
    Plan &P = h->P;
    if (!P.blob.empty()) {
        if ((e = cudaMalloc(&h->d_const, P.blob.size())) != cudaSuccess) {
            byoc_release(h);
            return cuda_fail(e, "cudaMalloc(constants)");
        }
        if ((e = cudaMemcpy(h->d_const, P.blob.data(), P.blob.size(), cudaMemcpyHostToDevice)) !=
            cudaSuccess) {
            byoc_release(h);
            return cuda_fail(e, "cudaMemcpy(constants)");
        }
    }
    if ((e = cudaMalloc(&h->d_ws, P.ws_bytes)) != cudaSuccess) {
        byoc_release(h);
        return cuda_fail(e, "cudaMalloc(workspace)");
    }
    if ((e = cudaMemset(h->d_ws, 0, 256)) != cudaSuccess) {
        byoc_release(h);
        return cuda_fail(e, "cudaMemset(error word)");
    }
    h->d_err = reinterpret_cast<int *>(h->d_ws);
    const size_t nl = P.launches.size();
    h->tmB.resize(nl);
    h->tmA.resize(nl);
    h->tmA_ptr.assign(nl, nullptr);
    h->tmR.resize(nl);
    h->tmR_ptr.assign(nl, nullptr);
    h->tmO.resize(nl);
    h->tmO_ptr.assign(nl, nullptr);
    h->cmaps.resize(nl);
    h->cptr.assign(nl, std::vector<const void *>(2 * byoc::kChainMaxStages, nullptr));
    h->ptrs.assign(P.tensors.size(), nullptr);
    for (size_t i = 0; i < nl; ++i) {
        LaunchPlan &L = P.launches[i];
        if (L.kind == BYOC_LAUNCH_GEMM) {
            L.args.bias = reinterpret_cast<const float *>(h->d_const + L.b_off);
            L.args.err = h->d_err;
            L.args.w = h->d_const + L.w_off;
            L.args.k_pack = L.k_pack;
            L.args.dq = L.fp8 ? reinterpret_cast<const float *>(h->d_const + L.dq_off) : nullptr;
            L.args.out8 = L.out8;
            L.args.out_inv = L.out_inv;
            if (L.part_bytes) {
                L.args.partial = reinterpret_cast<float *>(h->d_ws + L.part_off);
                L.args.counters = reinterpret_cast<unsigned *>(h->d_ws + L.cnt_off);
                if ((e = cudaMemset(h->d_ws + L.cnt_off, 0, L.cnt_bytes)) != cudaSuccess) {
                    byoc_release(h);
                    return cuda_fail(e, "cudaMemset(split-K counters)");
                }
            }
            // multicast: each CTA of a cluster loads half of a weight tile's
            // rows; FP8: E4M3 codes, 128 per k-block row
            CUresult r = L.fp8 ? encode_2d_u8(&h->tmB[i], h->d_const + L.w_off, (uint64_t)L.n_pad,
                                              (uint64_t)L.k_pack, (uint32_t)L.cfg.bn, byoc::kF8BK,
                                              CU_TENSOR_MAP_SWIZZLE_128B)
                               : encode_2d(&h->tmB[i], h->d_const + L.w_off, (uint64_t)L.n_pad,
                                           (uint64_t)L.k_pack, (uint32_t)(L.cfg.mc ? L.cfg.bn / 2 : L.cfg.bn),
                                           (uint32_t)L.cfg.bk, L.cfg.bk);
            if (r != CUDA_SUCCESS) {
                byoc_release(h);
                return fail(BYOC_ERR_CUDA, "launch %zu: cuTensorMapEncodeTiled(weights) = %d", i, (int)r);
            }
            if ((e = byoc::gemm_prepare(L.cfg)) != cudaSuccess) {
                byoc_release(h);
                return cuda_fail(e, "cudaFuncSetAttribute");
            }
        } else if (L.kind == BYOC_LAUNCH_DWPW) {
            L.dp.dw_w = reinterpret_cast<const float *>(h->d_const + L.w_off);
            L.dp.dw_b = reinterpret_cast<const float *>(h->d_const + L.b_off);
            L.dp.pw_b = reinterpret_cast<const float *>(h->d_const + L.b2_off);
            L.dp.err = h->d_err;
            // the 1x1 weights: 64-channel x n_pad boxes, 128-byte swizzle (the MMA's B operand)
            CUresult r = encode_2d(&h->tmB[i], h->d_const + L.w2_off, (uint64_t)L.n_pad, (uint64_t)L.k_pack,
                                   (uint32_t)L.n_pad, (uint32_t)byoc::kDpChunk, byoc::kDpChunk);
            if (r != CUDA_SUCCESS) {
                byoc_release(h);
                return fail(BYOC_ERR_CUDA, "launch %zu: cuTensorMapEncodeTiled(1x1 weights) = %d", i, (int)r);
            }
            if ((e = byoc::dwpw_prepare(L.dp)) != cudaSuccess) {
                byoc_release(h);
                return cuda_fail(e, "cudaFuncSetAttribute");
            }
        } else if (L.kind == BYOC_LAUNCH_CHAIN) {
            byoc::ChainArgs &A = L.chain;
            for (int st = 0; st < A.n_stages; ++st) {
                A.st[st].bias = reinterpret_cast<const float *>(h->d_const + L.cb_off[st]);
                A.st[st].dq = A.st[st].fp8 ? reinterpret_cast<const float *>(h->d_const + L.c_dq_off[st]) : nullptr;
                CUresult r = A.st[st].fp8
                                 ? encode_2d_u8(&h->cmaps[i].B[st], h->d_const + L.cw_off[st], (uint64_t)L.c_npad[st],
                                                (uint64_t)L.c_kpack[st], (uint32_t)L.chain_bn, 128,
                                                CU_TENSOR_MAP_SWIZZLE_128B)
                                 : encode_2d(&h->cmaps[i].B[st], h->d_const + L.cw_off[st], (uint64_t)L.c_npad[st],
                                             (uint64_t)L.c_kpack[st], (uint32_t)L.chain_bn, 64, 64);
                if (r != CUDA_SUCCESS) {
                    byoc_release(h);
                    return fail(BYOC_ERR_CUDA, "launch %zu stage %d: cuTensorMapEncodeTiled(weights) = %d", i,
                                st, (int)r);
                }
            }
            // every CTA of a region kernel must be resident at once (one per SM)
            if (L.grid > h->sms) {
                byoc_release(h);
                return fail(BYOC_ERR_UNSUPPORTED, "region kernel of %d CTAs planned for more SMs than the device has",
                            L.grid);
            }
            A.order = reinterpret_cast<const int *>(h->d_const + L.order_off);
            A.cta_off = reinterpret_cast<const int *>(h->d_const + L.cta_off_off);
            A.cta_rec = reinterpret_cast<const int *>(h->d_const + L.cta_rec_off);
            A.dep_off = reinterpret_cast<const int *>(h->d_const + L.dep_off_off);
            A.dep_list = reinterpret_cast<const int *>(h->d_const + L.dep_list_off);
            A.ctl = reinterpret_cast<unsigned *>(h->d_ws + L.flags_off);
            A.flags = A.ctl + 4;
            A.err = h->d_err;
            if ((e = cudaMemset(h->d_ws + L.flags_off, 0, L.flags_bytes)) != cudaSuccess) {
                byoc_release(h);
                return cuda_fail(e, "cudaMemset(region kernel flags)");
            }
            if ((e = byoc::chain_prepare(L.chain_bn)) != cudaSuccess) {
                byoc_release(h);
                return cuda_fail(e, "cudaFuncSetAttribute");
            }
        } else if (L.kind == BYOC_LAUNCH_DEPTHWISE) {
            L.dw.w = reinterpret_cast<const float *>(h->d_const + L.w_off);
            L.dw.bias = reinterpret_cast<const float *>(h->d_const + L.b_off);
            L.dw.err = h->d_err;
            if ((e = byoc::dw_prepare(L.dw)) != cudaSuccess) {
                byoc_release(h);
                return cuda_fail(e, "cudaFuncSetAttribute");
            }
        }
    }
    *out = h;
    return BYOC_OK;
}

// ------------------------------------------------------------ serialised plans
//
// Section 3.3, codegen option 3: the backend's output serialised so that
// deployment loads it without compiling.  Layout (host byte order):
//   magic "BYOCPLN1" | u32 format | u32 abi_version | u64 layout tag |
//   i32 num_sms | i32 n_region_tensors | u32 tensors, inputs, outputs,
//   launches | u64 blob bytes | u64 workspace bytes | f64 flops, bytes |
//   TensorInfo[] | i32 inputs[] | i32 outputs[] | LaunchPlan[] |
//   u64 ws_off[] | blob | u64 FNV-1a 64 of everything before it.
// Launch records are stored as this build's structs; the layout tag (the
// sizes of the structs, the format and ABI versions) rejects bytes written by
// a build with a different layout.  Device pointers inside the records are
// rebound when the plan is instantiated.

static_assert(std::is_trivially_copyable<LaunchPlan>::value && std::is_trivially_copyable<TensorInfo>::value,
              "launch records are stored byte for byte");
constexpr char kPlanMagic[8] = {'B', 'Y', 'O', 'C', 'P', 'L', 'N', '1'};
constexpr uint32_t kPlanFormat = 3;

uint64_t fnv1a(const uint8_t *p, size_t n, uint64_t h = 1469598103934665603ull) {
    for (size_t i = 0; i < n; ++i) {
        h ^= p[i];
        h *= 1099511628211ull;
    }
    return h;
}

uint64_t layout_tag() {
    const uint64_t sizes[] = {sizeof(TensorInfo), sizeof(LaunchPlan), sizeof(GemmArgs),
                              sizeof(byoc::DwArgs), sizeof(byoc::StemArgs), sizeof(Im2colGeom),
                              kPlanFormat, BYOC_ABI_VERSION};
    return fnv1a(reinterpret_cast<const uint8_t *>(sizes), sizeof(sizes));
}

struct PlanHeader {
    char magic[8];
    uint32_t format, abi_version;
    uint64_t tag;
    int32_t num_sms, n_region_tensors;
    uint32_t n_tensors, n_inputs, n_outputs, n_launches;
    uint64_t blob_bytes, ws_bytes;
    double flops, bytes;
};

// Records are written with their padding zeroed, so that the bytes depend
// only on the plan (no stray host memory in a serialised region).
// The objects' bytes as they are: every plan object is value-initialised
// (T x{}, vector resize), so its padding bytes are zero and copies keep them.
// (__builtin_clear_padding is not used: GCC 13 cleared array elements of
// LaunchPlan as if they were padding -- a region kernel's c_npad[1] read
// back as 0 once the struct's layout changed.)
template <typename T>
void put(std::vector<uint8_t> &out, const T *v, size_t n) {
    static_assert(std::is_trivially_copyable<T>::value, "plans are serialised byte for byte");
    const uint8_t *b = reinterpret_cast<const uint8_t *>(v);
    out.insert(out.end(), b, b + n * sizeof(T));
}

void serialize_plan(const Plan &P, std::vector<uint8_t> &out) {
    PlanHeader hd{};
    std::memcpy(hd.magic, kPlanMagic, 8);
    hd.format = kPlanFormat;
    hd.abi_version = BYOC_ABI_VERSION;
    hd.tag = layout_tag();
    hd.num_sms = P.num_sms;
    hd.n_region_tensors = P.n_region_tensors;
    hd.n_tensors = (uint32_t)P.tensors.size();
    hd.n_inputs = (uint32_t)P.inputs.size();
    hd.n_outputs = (uint32_t)P.outputs.size();
    hd.n_launches = (uint32_t)P.launches.size();
    hd.blob_bytes = P.blob.size();
    hd.ws_bytes = P.ws_bytes;
    hd.flops = P.flops;
    hd.bytes = P.bytes;
    out.clear();
    put(out, &hd, 1);
    put(out, P.tensors.data(), P.tensors.size());
    put(out, P.inputs.data(), P.inputs.size());
    put(out, P.outputs.data(), P.outputs.size());
    put(out, P.launches.data(), P.launches.size());
    std::vector<uint64_t> ws(P.ws_off.begin(), P.ws_off.end());
    put(out, ws.data(), ws.size());
    put(out, P.blob.data(), P.blob.size());
    const uint64_t sum = fnv1a(out.data(), out.size());
    put(out, &sum, 1);
}

// A deserialised region-kernel launch stays within the plan: stage tensors,
// constants, dependency lists (each unit waits only for units before it, so
// every wait of the kernel can end) and workspace flags.
int g_chain_bad = 0;  // which consistency check failed (for the error message)
bool chain_plan_ok(const Plan &P, const LaunchPlan &L) {
    const byoc::ChainArgs &A = L.chain;
    const int nt = (int)P.tensors.size();
    if ((L.chain_bn != 128 && L.chain_bn != 256) || A.n_stages < 1 || A.n_stages > byoc::kChainMaxStages ||
        (A.n_stages == 1 && !A.st[0].fp8))
        { g_chain_bad = 1; return false; }
    int units = 0, ncnt = 0;
    for (int s = 0; s < A.n_stages; ++s) {
        const byoc::ChainStage &cs = A.st[s];
        if (L.cx[s] < 0 || L.cx[s] >= nt || L.cy[s] < 0 || L.cy[s] >= nt || L.cres[s] >= nt) { g_chain_bad = 2; return false; }
        if (cs.M < 1 || cs.N < 32 || cs.N % 32) { g_chain_bad = 3; return false; }
        if (cs.tiles_n != L.c_npad[s] / L.chain_bn || L.c_npad[s] % L.chain_bn) { g_chain_bad = 13; return false; }
        if (cs.num_tiles != (cs.M + byoc::kGemmBM - 1) / byoc::kGemmBM * cs.tiles_n || cs.num_tiles >= (1 << 24))
            { g_chain_bad = 14; return false; }
        if (cs.cbase != ncnt || cs.unit0 != units) { g_chain_bad = 15; return false; }
        if (cs.num_kb < 1 || (size_t)cs.num_kb * (cs.fp8 ? 128 : 64) > (size_t)L.c_kpack[s]) { g_chain_bad = 16; return false; }
        if (P.tensors[L.cy[s]].elems() != (size_t)cs.M * cs.N) { g_chain_bad = 4; return false; }
        if ((P.tensors[L.cy[s]].dtype == BYOC_E4M3) != (cs.out8 != 0) ||
            (P.tensors[L.cx[s]].dtype == BYOC_E4M3) != (cs.fp8 != 0))
            { g_chain_bad = 21; return false; }
        if (L.cw_off[s] + (size_t)L.c_npad[s] * L.c_kpack[s] * (cs.fp8 ? 1 : 2) > P.blob.size() ||
            L.cb_off[s] + (size_t)L.c_npad[s] * 4 > P.blob.size() ||
            (cs.fp8 && L.c_dq_off[s] + (size_t)L.c_npad[s] * 4 > P.blob.size()))
            { g_chain_bad = 5; return false; }
        units += cs.num_tiles;
        ncnt += (cs.M + byoc::kGemmBM - 1) / byoc::kGemmBM;
    }
    if (units != A.total_units || ncnt != A.n_counters || L.flags_off + 16 + 4 * (size_t)ncnt > P.ws_bytes ||
        L.order_off + 4 * (size_t)units > P.blob.size() || L.dep_off_off + 4 * ((size_t)units + 1) > P.blob.size())
        { g_chain_bad = 6; return false; }
    const int32_t *order = reinterpret_cast<const int32_t *>(P.blob.data() + L.order_off);
    const int32_t *off = reinterpret_cast<const int32_t *>(P.blob.data() + L.dep_off_off);
    const int32_t *list = reinterpret_cast<const int32_t *>(P.blob.data() + L.dep_list_off);
    const size_t pairs = L.dep_list_off < P.blob.size() ? (P.blob.size() - L.dep_list_off) / 8 : 0;
    // the order is a permutation of the units; every counter a unit waits
    // for is completed by units earlier in the order only
    std::vector<char> seen(units, 0);
    if (off[0] != 0) { g_chain_bad = 7; return false; }
    for (int i = 0; i < units; ++i) {
        const int s = order[i] >> 24, tile = order[i] & 0xFFFFFF;
        if (s < 0 || s >= A.n_stages || tile >= A.st[s].num_tiles) { g_chain_bad = 8; return false; }
        const int nat = A.st[s].unit0 + tile;
        if (seen[nat]) { g_chain_bad = 9; return false; }
        seen[nat] = 1;
        if (off[i + 1] < off[i] || (size_t)off[i + 1] > pairs) { g_chain_bad = 10; return false; }
        for (int j = off[i]; j < off[i + 1]; ++j) {
            const int c = list[2 * j];
            if (c < 0 || c >= ncnt || list[2 * j + 1] <= 0) { g_chain_bad = 11; return false; }
        }
    }
    // a counter may only be waited for once all its units are before the waiter
    std::vector<int> done_at(ncnt, -1);
    for (int i = 0; i < units; ++i) {
        const int s = order[i] >> 24;
        const int c = A.st[s].cbase + (order[i] & 0xFFFFFF) / A.st[s].tiles_n;
        done_at[c] = std::max(done_at[c], i);
    }
    for (int i = 0; i < units; ++i)
        for (int j = off[i]; j < off[i + 1]; ++j)
            if (done_at[list[2 * j]] >= i) { g_chain_bad = 12; return false; }
    // per-CTA records: a partition of the units, each CTA's in the global
    // order, each record a copy of its unit's code and dependencies
    if (L.grid < 1 || L.grid > units || L.cta_off_off + 4 * ((size_t)L.grid + 1) > P.blob.size() ||
        L.cta_rec_off % 16 || L.cta_rec_off + 4 * (size_t)units * byoc::kChainRecInts > P.blob.size())
        { g_chain_bad = 17; return false; }
    const int32_t *coff = reinterpret_cast<const int32_t *>(P.blob.data() + L.cta_off_off);
    const int32_t *crec = reinterpret_cast<const int32_t *>(P.blob.data() + L.cta_rec_off);
    if (coff[0] != 0 || coff[L.grid] != units) { g_chain_bad = 18; return false; }
    std::fill(seen.begin(), seen.end(), 0);
    for (int b = 0; b < L.grid; ++b) {
        if (coff[b + 1] < coff[b]) { g_chain_bad = 19; return false; }
        for (int k = coff[b]; k < coff[b + 1]; ++k) {
            const int32_t *r = crec + (size_t)k * byoc::kChainRecInts;
            const int i = r[0];
            if (i < 0 || i >= units || seen[i] || (k > coff[b] && r[-byoc::kChainRecInts] >= i)) { g_chain_bad = 20; return false; }
            seen[i] = 1;
            if (r[1] != order[i] || r[2] != off[i + 1] - off[i] || r[3] != off[i]) { g_chain_bad = 22; return false; }
            for (int q = 0; q < std::min(r[2], byoc::kChainRecDeps); ++q)
                if (r[4 + 2 * q] != list[2 * (off[i] + q)] || r[5 + 2 * q] != list[2 * (off[i] + q) + 1])
                    { g_chain_bad = 22; return false; }
        }
    }
    return true;
}

byoc_status deserialize_plan(const void *src, size_t n, Plan &P) {
    if (!src) return fail(BYOC_ERR_INVALID_ARG, "null serialised plan");
    const uint8_t *b = static_cast<const uint8_t *>(src);
    PlanHeader hd;
    if (n < sizeof(hd) + 8) return fail(BYOC_ERR_INVALID_ARG, "serialised plan truncated (%zu bytes)", n);
    std::memcpy(&hd, b, sizeof(hd));
    if (std::memcmp(hd.magic, kPlanMagic, 8) != 0) return fail(BYOC_ERR_INVALID_ARG, "not a serialised plan");
    if (hd.format != kPlanFormat || hd.abi_version != BYOC_ABI_VERSION || hd.tag != layout_tag())
        return fail(BYOC_ERR_UNSUPPORTED, "serialised plan from another library build (format %u, abi %u)",
                    hd.format, hd.abi_version);
    const uint64_t limit = (uint64_t)1 << 40;
    if (hd.n_tensors > 4096 || hd.n_inputs > hd.n_tensors || hd.n_outputs > hd.n_tensors ||
        hd.n_launches > 4096 || hd.blob_bytes > limit || hd.ws_bytes > limit ||
        hd.n_region_tensors < 0 || (uint32_t)hd.n_region_tensors > hd.n_tensors)
        return fail(BYOC_ERR_INVALID_ARG, "serialised plan: counts out of range");
    const uint64_t body = (uint64_t)hd.n_tensors * sizeof(TensorInfo) +
                          (uint64_t)(hd.n_inputs + hd.n_outputs) * sizeof(int) +
                          (uint64_t)hd.n_launches * sizeof(LaunchPlan) + (uint64_t)hd.n_tensors * 8 +
                          hd.blob_bytes;
    if ((uint64_t)n != sizeof(hd) + body + 8)
        return fail(BYOC_ERR_INVALID_ARG, "serialised plan: %zu bytes, header describes %llu", n,
                    (unsigned long long)(sizeof(hd) + body + 8));
    uint64_t sum;
    std::memcpy(&sum, b + n - 8, 8);
    if (sum != fnv1a(b, n - 8)) return fail(BYOC_ERR_INVALID_ARG, "serialised plan: checksum mismatch");
    size_t off = sizeof(hd);
    auto take = [&](void *dst, size_t bytes) {
        if (bytes) std::memcpy(dst, b + off, bytes);
        off += bytes;
    };
    P = Plan();
    P.num_sms = hd.num_sms;
    P.n_region_tensors = hd.n_region_tensors;
    P.tensors.resize(hd.n_tensors);
    take(P.tensors.data(), P.tensors.size() * sizeof(TensorInfo));
    P.inputs.resize(hd.n_inputs);
    take(P.inputs.data(), P.inputs.size() * sizeof(int));
    P.outputs.resize(hd.n_outputs);
    take(P.outputs.data(), P.outputs.size() * sizeof(int));
    P.launches.resize(hd.n_launches);
    take(P.launches.data(), P.launches.size() * sizeof(LaunchPlan));
    std::vector<uint64_t> ws(hd.n_tensors);
    take(ws.data(), ws.size() * 8);
    P.ws_off.assign(ws.begin(), ws.end());
    P.blob.resize(hd.blob_bytes);
    take(P.blob.data(), P.blob.size());
    P.ws_bytes = hd.ws_bytes;
    P.flops = hd.flops;
    P.bytes = hd.bytes;
    // references inside the records must stay within the plan
    const int nt = (int)hd.n_tensors;
    for (int id : P.inputs)
        if (id < 0 || id >= nt) return fail(BYOC_ERR_INVALID_ARG, "serialised plan: bad input id");
    for (int id : P.outputs)
        if (id < 0 || id >= nt) return fail(BYOC_ERR_INVALID_ARG, "serialised plan: bad output id");
    for (int t = 0; t < nt; ++t)
        if (P.ws_off[t] != SIZE_MAX && P.ws_off[t] + P.tensors[t].bytes() > P.ws_bytes)
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: workspace layout out of range");
    for (const LaunchPlan &L : P.launches) {
        if (L.kind != BYOC_LAUNCH_GEMM && L.kind != BYOC_LAUNCH_DEPTHWISE && L.kind != BYOC_LAUNCH_S2D &&
            L.kind != BYOC_LAUNCH_DWPW && L.kind != BYOC_LAUNCH_CHAIN && L.kind != BYOC_LAUNCH_QUANT)
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: bad launch kind");
        if (L.kind == BYOC_LAUNCH_CHAIN && !chain_plan_ok(P, L))
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: inconsistent region kernel (check %d)", g_chain_bad);
        if (L.x < 0 || L.x >= nt || L.y < 0 || L.y >= nt || L.res >= nt)
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: bad tensor id in a launch");
        if (L.w_off + L.w_bytes > P.blob.size() || L.b_off + L.b_bytes > P.blob.size() ||
            L.w2_off + L.w2_bytes > P.blob.size() || L.b2_off + L.b2_bytes > P.blob.size())
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: constants out of range");
        if (L.part_off + L.part_bytes > P.ws_bytes || L.cnt_off + L.cnt_bytes > P.ws_bytes)
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: split-K scratch out of range");
        if (L.kind == BYOC_LAUNCH_GEMM && !byoc::gemm_config_supported(L.cfg))
            return fail(BYOC_ERR_UNSUPPORTED, "serialised plan: tile configuration not in this build");
        if (L.kind == BYOC_LAUNCH_GEMM && L.cfg.amode == byoc::kAModeTileSplit &&
            (L.args.splits < 2 ||
             L.part_bytes < (size_t)L.args.splits * (size_t)L.args.m_pad * (size_t)L.args.n_pad * 4 ||
             L.cnt_bytes < (size_t)L.args.num_tiles * 8 * 4))
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: split-K scratch too small");
        if (L.kind == BYOC_LAUNCH_GEMM && L.cfg.amode == byoc::kAModeTileSplitCl &&
            (!byoc::cl_split_fits(L.cfg.bn, L.args.splits) || L.grid != L.args.num_tiles * L.args.splits))
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: inconsistent cluster split-K");
        if (L.kind == BYOC_LAUNCH_GEMM && L.cfg.mc && (L.grid < 2 || L.grid % 2))
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: multicast launch of an odd grid");
        if (L.kind == BYOC_LAUNCH_GEMM &&
            ((L.fp8 != 0) != (L.cfg.bk == byoc::kF8BK) ||
             (P.tensors[L.x].dtype == BYOC_E4M3) != (L.fp8 != 0) ||
             (P.tensors[L.y].dtype == BYOC_E4M3) != (L.out8 != 0) ||
             (L.out8 && !L.fp8) ||
             (L.fp8 && (L.dq_off + (size_t)L.n_pad * 4 > P.blob.size() ||
                        L.w_bytes < (size_t)L.n_pad * L.k_pack || L.k_pack % byoc::kF8BK))))
            return fail(BYOC_ERR_INVALID_ARG, "serialised plan: inconsistent FP8 launch");
        if (L.kind == BYOC_LAUNCH_DEPTHWISE) {
            const byoc::DwArgs &w = L.dw;
            const size_t box = (size_t)w.in_rows * w.in_cols * w.cc * 2;
            if (w.cc < 8 || w.cc > 256 || w.in_rows < 1 || w.in_rows > 256 || w.in_cols < 1 || w.in_cols > 256 ||
                (size_t)w.buf_bytes < box || (size_t)w.buf_bytes > byoc::kDwBufBudget)
                return fail(BYOC_ERR_INVALID_ARG, "serialised plan: inconsistent depthwise tiling");
        }
    }
    return BYOC_OK;
}

}  // namespace

extern "C" {

byoc_status byoc_compile(const byoc_region_desc *desc, byoc_handle **out) {
    if (!out) return fail(BYOC_ERR_INVALID_ARG, "null output handle pointer");
    *out = nullptr;
    int32_t sms = 0;
    byoc_status st = check_device(&sms);
    if (st != BYOC_OK) return st;
    byoc_handle *h = new (std::nothrow) byoc_handle();
    if (!h) return fail(BYOC_ERR_OOM, "host allocation");
    st = plan_region(desc, sms, h->P);
    if (st != BYOC_OK) {
        delete h;
        return st;
    }
    return instantiate(h, out);
}

byoc_status byoc_serialize(const byoc_handle *h, void *dst, size_t dst_bytes, size_t *needed) {
    if (!h || !needed) return fail(BYOC_ERR_INVALID_ARG, "null handle or size pointer");
    std::vector<uint8_t> buf;
    serialize_plan(h->P, buf);
    *needed = buf.size();
    if (!dst) return BYOC_OK;
    if (dst_bytes < buf.size())
        return fail(BYOC_ERR_INVALID_ARG, "buffer of %zu bytes, %zu needed", dst_bytes, buf.size());
    std::memcpy(dst, buf.data(), buf.size());
    return BYOC_OK;
}

byoc_status byoc_deserialize(const void *src, size_t src_bytes, byoc_handle **out) {
    if (!out) return fail(BYOC_ERR_INVALID_ARG, "null output handle pointer");
    *out = nullptr;
    int32_t sms = 0;
    byoc_status st = check_device(&sms);
    if (st != BYOC_OK) return st;
    byoc_handle *h = new (std::nothrow) byoc_handle();
    if (!h) return fail(BYOC_ERR_OOM, "host allocation");
    st = deserialize_plan(src, src_bytes, h->P);
    if (st != BYOC_OK) {
        delete h;
        return st;
    }
    return instantiate(h, out);
}

byoc_status byoc_plan_serialize(const byoc_region_desc *desc, int32_t num_sms, void *dst,
                                size_t dst_bytes, size_t *needed) {
    if (!needed) return fail(BYOC_ERR_INVALID_ARG, "null size pointer");
    Plan P;
    byoc_status st = plan_region(desc, num_sms, P);
    if (st != BYOC_OK) return st;
    std::vector<uint8_t> buf;
    serialize_plan(P, buf);
    *needed = buf.size();
    if (!dst) return BYOC_OK;
    if (dst_bytes < buf.size())
        return fail(BYOC_ERR_INVALID_ARG, "buffer of %zu bytes, %zu needed", dst_bytes, buf.size());
    std::memcpy(dst, buf.data(), buf.size());
    return BYOC_OK;
}

byoc_status byoc_plan_deserialize(const void *src, size_t src_bytes, byoc_plan_report *rep) {
    if (!rep) return fail(BYOC_ERR_INVALID_ARG, "null report");
    Plan P;
    byoc_status st = deserialize_plan(src, src_bytes, P);
    if (st != BYOC_OK) return st;
    fill_report(P, rep);
    return BYOC_OK;
}

// Kernel trace (byoc_trace_begin): the buffer, its capacity in slots and the
// next free slot.
namespace {
unsigned long long *g_trace = nullptr;
int g_trace_cap = 0, g_trace_next = 0;
}  // namespace

byoc_status byoc_trace_begin(void *buf, int32_t capacity) {
    if (!buf || (reinterpret_cast<uintptr_t>(buf) & 15u) || capacity < 1)
        return fail(BYOC_ERR_INVALID_ARG, "trace: null or misaligned buffer, or capacity < 1");
    g_trace = static_cast<unsigned long long *>(buf);
    g_trace_cap = capacity;
    g_trace_next = 0;
    return BYOC_OK;
}

int32_t byoc_trace_end(void) {
    const int n = g_trace_next;
    g_trace = nullptr;
    g_trace_cap = g_trace_next = 0;
    return n;
}

byoc_status byoc_run(byoc_handle *h, const void *const *inputs, void *const *outputs,
                     void *cuda_stream) {
    if (!h) return fail(BYOC_ERR_INVALID_ARG, "null handle");
    Plan &P = h->P;
    if (!inputs || !outputs) return fail(BYOC_ERR_INVALID_ARG, "null input/output array");
    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    for (size_t i = 0; i < P.inputs.size(); ++i) {
        const void *p = inputs[i];
        if (!p || (reinterpret_cast<uintptr_t>(p) & 15u))
            return fail(BYOC_ERR_INVALID_ARG, "input %zu: null or not 16-byte aligned", i);
        h->ptrs[P.inputs[i]] = const_cast<void *>(p);
    }
    for (size_t i = 0; i < P.outputs.size(); ++i) {
        void *p = outputs[i];
        if (!p || (reinterpret_cast<uintptr_t>(p) & 15u))
            return fail(BYOC_ERR_INVALID_ARG, "output %zu: null or not 16-byte aligned", i);
        h->ptrs[P.outputs[i]] = p;
    }
    for (size_t t = 0; t < P.tensors.size(); ++t)
        if (P.ws_off[t] != SIZE_MAX) h->ptrs[t] = h->d_ws + P.ws_off[t];

    for (size_t i = 0; i < P.launches.size(); ++i) {
        LaunchPlan &L = P.launches[i];
        cudaError_t e = cudaSuccess;
        if (L.kind == BYOC_LAUNCH_GEMM) {
            const void *xa = static_cast<const char *>(h->ptrs[L.x]) + L.x_off;
            if (h->tmA_ptr[i] != xa) {
                CUresult r;
                if (byoc::amode_slab(L.cfg.amode) && L.stem_R > 0)
                    r = encode_stem_slab(&h->tmA[i], xa, L.geo.N, L.geo.H, L.geo.W, L.stem_R, L.args.wp,
                                         L.slab_rows, L.stem_G);
                else if (byoc::amode_slab(L.cfg.amode))
                    r = encode_slab(&h->tmA[i], xa, L.geo.N, L.geo.H, L.geo.W, L.geo.C, L.args.wp,
                                    L.slab_rows, L.cfg.bk);
                else if (L.cfg.amode == byoc::kAModeIm2col)
                    r = L.fp8 ? encode_im2col(&h->tmA[i], xa, L.geo, 64, true)  // 128 codes per pixel
                              : encode_im2col(&h->tmA[i], xa, L.geo, L.cfg.bk);
                else if (L.fp8)
                    r = encode_2d_u8(&h->tmA[i], xa, (uint64_t)L.aM, (uint64_t)L.aK, byoc::kGemmBM,
                                     byoc::kF8BK, CU_TENSOR_MAP_SWIZZLE_128B);
                else
                    r = encode_2d(&h->tmA[i], xa, (uint64_t)L.aM, (uint64_t)L.aK, byoc::kGemmBM,
                                  (uint32_t)L.cfg.bk, L.cfg.bk);
                if (r != CUDA_SUCCESS)
                    return fail(BYOC_ERR_CUDA, "launch %zu: encoding the activation TMA map failed (%d)",
                                i, (int)r);
                h->tmA_ptr[i] = xa;
            }
            GemmArgs a = L.args;
            a.trace = g_trace && g_trace_next < g_trace_cap ? g_trace + 2 * g_trace_next++ : nullptr;
            a.out = reinterpret_cast<__nv_bfloat16 *>(static_cast<char *>(h->ptrs[L.y]) + L.y_off);
            a.residual = L.res >= 0 ? static_cast<const __nv_bfloat16 *>(h->ptrs[L.res]) : nullptr;
            if (a.residual && h->tmR_ptr[i] != a.residual) {
                // residual [M, N]: 64-column x 128-row boxes, 128-byte swizzle
                CUresult r = encode_2d(&h->tmR[i], a.residual, (uint64_t)a.M, (uint64_t)a.N,
                                       byoc::kGemmBM, 64, 64);
                if (r != CUDA_SUCCESS)
                    return fail(BYOC_ERR_CUDA, "launch %zu: encoding the residual TMA map failed (%d)",
                                i, (int)r);
                h->tmR_ptr[i] = a.residual;
            }
            // tile mode (and FP8) stores its output with TMA: [M, N] in 32 x
            // 32 boxes, 64-byte swizzle (the layout of the epilogue's staging
            // tiles); E4M3 codes of a fused Q node: 32 x 32 bytes, unswizzled
            const bool tstore = byoc::gemm_tstore(L.cfg.amode, L.cfg.bk);
            if (tstore && h->tmO_ptr[i] != a.out) {
                CUresult r = a.out8 ? encode_2d_u8(&h->tmO[i], a.out, (uint64_t)a.M, (uint64_t)a.N, 32, 32,
                                                   CU_TENSOR_MAP_SWIZZLE_NONE)
                                    : encode_2d(&h->tmO[i], a.out, (uint64_t)a.M, (uint64_t)a.N, 32, 32, 32);
                if (r != CUDA_SUCCESS)
                    return fail(BYOC_ERR_CUDA, "launch %zu: encoding the output TMA map failed (%d)", i,
                                (int)r);
                h->tmO_ptr[i] = a.out;
            }
            e = byoc::launch_gemm(L.cfg, h->tmA[i], h->tmB[i], a.residual ? h->tmR[i] : h->tmA[i],
                                  tstore ? h->tmO[i] : h->tmA[i], a, L.grid, st);
        } else if (L.kind == BYOC_LAUNCH_CHAIN) {
            byoc::ChainArgs a = L.chain;
            byoc::ChainMaps &mp = h->cmaps[i];
            std::vector<const void *> &cp = h->cptr[i];
            for (int sg = 0; sg < a.n_stages; ++sg) {
                const void *xa = h->ptrs[L.cx[sg]];
                if (cp[sg] != xa) {
                    const bool f8 = a.st[sg].fp8 != 0;
                    CUresult r = a.st[sg].mode == byoc::kChainIm2col
                                     ? encode_im2col(&mp.A[sg], xa, L.cgeo[sg], 64, f8)
                                     : f8 ? encode_2d_u8(&mp.A[sg], xa, (uint64_t)L.caM[sg], (uint64_t)L.caK[sg],
                                                         byoc::kGemmBM, 128, CU_TENSOR_MAP_SWIZZLE_128B)
                                          : encode_2d(&mp.A[sg], xa, (uint64_t)L.caM[sg], (uint64_t)L.caK[sg],
                                                      byoc::kGemmBM, 64, 64);
                    if (r != CUDA_SUCCESS)
                        return fail(BYOC_ERR_CUDA, "launch %zu stage %d: encoding the A map failed (%d)", i, sg,
                                    (int)r);
                    cp[sg] = xa;
                }
                void *ya = h->ptrs[L.cy[sg]];
                if (cp[byoc::kChainMaxStages + sg] != ya) {
                    // bf16: 32 x 32 boxes, 64-byte swizzle; E4M3 codes: 32 x 32 bytes, unswizzled
                    CUresult r = a.st[sg].out8
                                     ? encode_2d_u8(&mp.O[sg], ya, (uint64_t)a.st[sg].M, (uint64_t)a.st[sg].N, 32, 32,
                                                    CU_TENSOR_MAP_SWIZZLE_NONE)
                                     : encode_2d(&mp.O[sg], ya, (uint64_t)a.st[sg].M, (uint64_t)a.st[sg].N, 32, 32, 32);
                    if (r != CUDA_SUCCESS)
                        return fail(BYOC_ERR_CUDA, "launch %zu stage %d: encoding the output map failed (%d)", i,
                                    sg, (int)r);
                    cp[byoc::kChainMaxStages + sg] = ya;
                }
                a.st[sg].residual =
                    L.cres[sg] >= 0 ? static_cast<const __nv_bfloat16 *>(h->ptrs[L.cres[sg]]) : nullptr;
            }
            a.trace = g_trace && g_trace_next < g_trace_cap ? g_trace + 2 * g_trace_next++ : nullptr;
            e = byoc::launch_chain(L.chain_bn, mp, a, L.grid, st);
        } else if (L.kind == BYOC_LAUNCH_QUANT) {
            e = byoc::launch_quantize_e4m3(static_cast<const __nv_bfloat16 *>(h->ptrs[L.x]),
                                           static_cast<uint8_t *>(h->ptrs[L.y]), P.tensors[L.x].elems(), L.q_inv,
                                           h->sms, st);
        } else if (L.kind == BYOC_LAUNCH_DEPTHWISE) {
            const void *xa = static_cast<const char *>(h->ptrs[L.x]) + L.x_off;
            if (h->tmA_ptr[i] != xa) {
                CUresult r = encode_dw(&h->tmA[i], xa, L.dw);
                if (r != CUDA_SUCCESS)
                    return fail(BYOC_ERR_CUDA, "launch %zu: encoding the depthwise TMA map failed (%d)",
                                i, (int)r);
                h->tmA_ptr[i] = xa;
            }
            byoc::DwArgs a = L.dw;
            a.y = reinterpret_cast<__nv_bfloat16 *>(static_cast<char *>(h->ptrs[L.y]) + L.y_off);
            e = byoc::launch_dwconv(h->tmA[i], a, L.grid, st);
        } else if (L.kind == BYOC_LAUNCH_DWPW) {
            const void *xa = h->ptrs[L.x];
            if (h->tmA_ptr[i] != xa) {
                CUresult r = encode_dwpw_input(&h->tmA[i], xa, L.dp);
                if (r != CUDA_SUCCESS)
                    return fail(BYOC_ERR_CUDA, "launch %zu: encoding the depthwise input TMA map failed (%d)",
                                i, (int)r);
                h->tmA_ptr[i] = xa;
            }
            byoc::DwPwArgs a = L.dp;
            a.out = static_cast<__nv_bfloat16 *>(h->ptrs[L.y]);
            a.residual = L.res >= 0 ? static_cast<const __nv_bfloat16 *>(h->ptrs[L.res]) : nullptr;
            e = byoc::launch_dwpw(h->tmA[i], h->tmB[i], a, L.grid, st);
        } else {
            byoc::StemArgs a = L.stem;
            a.x = reinterpret_cast<const __nv_bfloat16 *>(static_cast<const char *>(h->ptrs[L.x]) +
                                                           L.x_off);
            a.xq = reinterpret_cast<__nv_bfloat16 *>(static_cast<char *>(h->ptrs[L.y]) + L.y_off);
            e = byoc::launch_stem_layout(a, st);
        }
        if (e != cudaSuccess) return cuda_fail(e, "kernel launch");
    }
    return BYOC_OK;
}

byoc_status byoc_check(byoc_handle *h) {
    if (!h) return static_cast<byoc_status>(byoc::noalloc_check());
    int v = 0;
    cudaError_t e = cudaMemcpy(&v, h->d_err, sizeof v, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "reading the error word");
    if (v != 0) {
        cudaMemset(h->d_err, 0, sizeof v);
        // a region kernel that gave up left its unit counter and flags
        // mid-launch: start them again from zero
        for (const LaunchPlan &L : h->P.launches)
            if (L.kind == BYOC_LAUNCH_CHAIN) cudaMemset(h->d_ws + L.flags_off, 0, L.flags_bytes);
        return fail(BYOC_ERR_TIMEOUT, "a kernel's bounded wait expired (code %d)", v);
    }
    return BYOC_OK;
}

byoc_status byoc_query(const byoc_handle *h, byoc_info *info) {
    if (!h || !info) return fail(BYOC_ERR_INVALID_ARG, "null handle or info");
    const Plan &P = h->P;
    info->flops = P.flops;
    info->bytes = P.bytes;
    info->workspace_bytes = P.ws_bytes;
    info->const_bytes = P.blob.size();
    info->n_launches = (int32_t)P.launches.size();
    info->n_inputs = (int32_t)P.inputs.size();
    info->n_outputs = (int32_t)P.outputs.size();
    return BYOC_OK;
}

byoc_status byoc_max_pool2d_nhwc(const void *x, void *y, int32_t N, int32_t H, int32_t W, int32_t C,
                                 int32_t k, int32_t s, int32_t p, void *cuda_stream) {
    if (!x || !y || ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15u))
        return fail(BYOC_ERR_INVALID_ARG, "max_pool2d: null or misaligned pointer");
    if (N < 1 || H < 1 || W < 1 || C < 8 || C % 8 || k < 1 || s < 1 || p < 0 || p >= k ||
        H + 2 * p < k || W + 2 * p < k)
        return fail(BYOC_ERR_INVALID_ARG, "max_pool2d: bad shape");
    cudaError_t e = byoc::launch_maxpool(static_cast<const __nv_bfloat16 *>(x),
                                         static_cast<__nv_bfloat16 *>(y), N, H, W, C, k, s, p,
                                         static_cast<cudaStream_t>(cuda_stream));
    return e == cudaSuccess ? BYOC_OK : cuda_fail(e, "max_pool2d launch");
}

byoc_status byoc_global_avg_pool_nhwc(const void *x, void *y, int32_t N, int32_t H, int32_t W,
                                      int32_t C, void *cuda_stream) {
    if (!x || !y || ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15u))
        return fail(BYOC_ERR_INVALID_ARG, "global_avg_pool: null or misaligned pointer");
    if (N < 1 || H < 1 || W < 1 || C < 8 || C % 8)
        return fail(BYOC_ERR_INVALID_ARG, "global_avg_pool: bad shape");
    cudaError_t e = byoc::launch_avgpool(static_cast<const __nv_bfloat16 *>(x),
                                         static_cast<__nv_bfloat16 *>(y), N, H, W, C,
                                         static_cast<cudaStream_t>(cuda_stream));
    return e == cudaSuccess ? BYOC_OK : cuda_fail(e, "global_avg_pool launch");
}

byoc_status byoc_nchw_to_nhwc_bf16(const void *x, void *y, int32_t N, int32_t C, int32_t H, int32_t W,
                                   int32_t c_pad, void *cuda_stream) {
    if (!x || !y || ((reinterpret_cast<uintptr_t>(x) | reinterpret_cast<uintptr_t>(y)) & 15u))
        return fail(BYOC_ERR_INVALID_ARG, "nchw_to_nhwc: null or misaligned pointer");
    if (N < 1 || C < 1 || H < 1 || W < 1 || c_pad < C || (int64_t)W * c_pad > byoc::kNchwStageElems)
        return fail(BYOC_ERR_INVALID_ARG, "nchw_to_nhwc: bad shape (need c_pad >= C, W * c_pad <= %d)",
                    byoc::kNchwStageElems);
    cudaError_t e = byoc::launch_nchw_to_nhwc(static_cast<const float *>(x), static_cast<__nv_bfloat16 *>(y),
                                              N, C, H, W, c_pad, static_cast<cudaStream_t>(cuda_stream));
    return e == cudaSuccess ? BYOC_OK : cuda_fail(e, "nchw_to_nhwc launch");
}

}  // extern "C"
