// noalloc.cu -- an allocation-free entry point for the two-layer dense chain
//   y = (GELU(x . w1^T + b1)) . w2^T + b2
// for callers that cannot allocate device memory: code that runs inside a
// memory pool or arena it does not control (a serving runtime that hands out
// only pre-sized buffers), callers that must not trigger a device
// synchronisation or allocator lock on the inference path, and embedded
// integrations that forbid cudaMalloc after start-up.  Such callers cannot use
// byoc_compile, which allocates the packed weights and the region workspace.
//
// The hidden activation H = GELU(x . w1^T + b1) lives in a file-scope device
// array of fixed size instead of a workspace: every GPU that loads this
// library reserves it until the process exits.  Host code may not use the
// array's name as a device address (it is a host-side stand-in), so the first
// call on each device, with that device current, looks the address up with
// cudaGetSymbolAddress and caches it; that first call also raises the GEMM
// kernel's shared-memory limit and loads the TMA descriptor encoder.  A set-up
// that fails is retried by the next call; one that succeeded is kept for the
// life of the process (it does not survive cudaDeviceReset of that device).
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cstdio>
#include <cstring>
#include <mutex>

#include "byoc.h"
#include "internal.h"

namespace {

constexpr size_t kHeaderBytes = 256;                  // [0, 4): device error word
constexpr size_t kHiddenMaxElems = (size_t)8 << 20;   // 8 Mi bf16 = 16 MiB
constexpr int kMaxDevices = 64;
constexpr int kTileN = 128;

static __device__ __align__(256) unsigned char g_ffn_scratch[kHeaderBytes + kHiddenMaxElems * 2];

struct DeviceState {
    bool ready = false;                // set only by a set-up that succeeded
    unsigned char *scratch = nullptr;  // device address of g_ffn_scratch
    int num_sms = 0;
};
DeviceState g_devices[kMaxDevices];
std::mutex g_devices_mutex;

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;
cudaError_t g_encode_err = cudaSuccess;

byoc_status fail(byoc_status st, const char *msg) {
    byoc::set_last_error(msg);
    return st;
}

byoc_status cuda_fail(cudaError_t e, const char *what) {
    char buf[256];
    snprintf(buf, sizeof buf, "%s: %s", what, cudaGetErrorString(e));
    byoc::set_last_error(buf);
    return BYOC_ERR_CUDA;
}

// Per-device set-up, with that device current.  Returns the first failing
// call's error; the state is marked ready only when every step succeeded.
cudaError_t setup_device(DeviceState &d, int dev) {
    std::lock_guard<std::mutex> lock(g_devices_mutex);
    if (d.ready) return cudaSuccess;
    unsigned char *p = nullptr;
    int sms = 0;
    cudaError_t e = cudaGetSymbolAddress(reinterpret_cast<void **>(&p), g_ffn_scratch);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e == cudaSuccess) e = byoc::gemm_prepare(byoc::GemmConfig{kTileN, 64, byoc::kAModeTile, false});
    if (e != cudaSuccess) return e;
    d.scratch = p;
    d.num_sms = sms;
    d.ready = true;
    return cudaSuccess;
}

CUresult encode(CUtensorMap *m, const void *ptr, uint64_t rows, uint64_t cols, uint32_t box_rows) {
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {64, box_rows};
    cuuint32_t es[2] = {1, 1};
    return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ptr), dims, strides,
                    box, es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

// Output [rows, cols] bf16 in 32 x 32 boxes, 64-byte swizzle: the map the
// GEMM's plain tile mode stores its output through.
CUresult encode_out(CUtensorMap *m, void *ptr, uint64_t rows, uint64_t cols) {
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {cols * 2};
    cuuint32_t box[2] = {32, 32};
    cuuint32_t es[2] = {1, 1};
    return g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, ptr, dims, strides, box, es,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
}

bool misaligned(const void *p) { return !p || (reinterpret_cast<uintptr_t>(p) & 15u); }

}  // namespace

extern "C" byoc_status byoc_ffn_noalloc(const void *x, int32_t M, int32_t D, int32_t F,
                                        const void *w1, const float *b1, const void *w2,
                                        const float *b2, void *y, void *cuda_stream) {
    if (M < 1 || D < 128 || F < 128 || D % kTileN || F % kTileN)
        return fail(BYOC_ERR_INVALID_ARG,
                    "byoc_ffn_noalloc: need M >= 1 and D, F positive multiples of 128");
    if ((size_t)M * (size_t)F > kHiddenMaxElems)
        return fail(BYOC_ERR_INVALID_ARG,
                    "byoc_ffn_noalloc: M * F exceeds the 8,388,608-element (16 MiB) scratch; split "
                    "the rows into several calls");
    if (misaligned(x) || misaligned(w1) || misaligned(w2) || misaligned(y) || misaligned(b1) ||
        misaligned(b2))
        return fail(BYOC_ERR_INVALID_ARG,
                    "byoc_ffn_noalloc: null or not 16-byte aligned pointer");
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "byoc_ffn_noalloc: cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(BYOC_ERR_UNSUPPORTED, "byoc_ffn_noalloc: device ordinal");
    std::call_once(g_encode_once, [] {
        cudaDriverEntryPointQueryResult q;
        g_encode_err = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled",
                                                        reinterpret_cast<void **>(&g_encode), 12000,
                                                        cudaEnableDefault, &q);
        if (g_encode_err == cudaSuccess && (q != cudaDriverEntryPointSuccess || !g_encode))
            g_encode_err = cudaErrorSymbolNotFound;
    });
    if (g_encode_err != cudaSuccess) return cuda_fail(g_encode_err, "byoc_ffn_noalloc: TMA encoder");
    DeviceState &d = g_devices[dev];
    if ((e = setup_device(d, dev)) != cudaSuccess) return cuda_fail(e, "byoc_ffn_noalloc: per-device set-up");

    cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
    int *err_word = reinterpret_cast<int *>(d.scratch);
    __nv_bfloat16 *hidden = reinterpret_cast<__nv_bfloat16 *>(d.scratch + kHeaderBytes);
    // The error word must start each call at zero; the hidden buffer is fully
    // overwritten by the first GEMM before the second reads it.
    if ((e = cudaMemsetAsync(err_word, 0, sizeof(int), st)) != cudaSuccess)
        return cuda_fail(e, "byoc_ffn_noalloc: clearing the error word");

    CUtensorMap a1, b1m, a2, b2m, o1, o2;
    if (encode(&a1, x, (uint64_t)M, (uint64_t)D, byoc::kGemmBM) != CUDA_SUCCESS ||
        encode(&b1m, w1, (uint64_t)F, (uint64_t)D, kTileN) != CUDA_SUCCESS ||
        encode(&a2, hidden, (uint64_t)M, (uint64_t)F, byoc::kGemmBM) != CUDA_SUCCESS ||
        encode(&b2m, w2, (uint64_t)D, (uint64_t)F, kTileN) != CUDA_SUCCESS ||
        encode_out(&o1, hidden, (uint64_t)M, (uint64_t)F) != CUDA_SUCCESS ||
        encode_out(&o2, y, (uint64_t)M, (uint64_t)D) != CUDA_SUCCESS)
        return fail(BYOC_ERR_CUDA, "byoc_ffn_noalloc: encoding a TMA descriptor failed");

    const byoc::GemmConfig cfg{kTileN, 64, byoc::kAModeTile, false};
    const int tiles_m = (M + byoc::kGemmBM - 1) / byoc::kGemmBM;
    byoc::GemmArgs g{};
    g.M = M;
    g.N = F;
    g.num_kb = D / 64;
    g.chunks = g.num_kb;
    g.kw = 1;
    g.dil_h = g.dil_w = 1;
    g.Ho = g.Wo = 1;
    g.stride_h = g.stride_w = 1;
    g.tiles_n = F / kTileN;
    g.num_tiles = tiles_m * g.tiles_n;
    g.group = byoc::gemm_group(kTileN, 64, g.num_kb);
    g.act = byoc::kActGelu;
    g.bias = b1;
    g.residual = nullptr;
    g.out = hidden;
    g.err = err_word;
    if ((e = byoc::launch_gemm(cfg, a1, b1m, a1, o1, g, g.num_tiles < d.num_sms ? g.num_tiles : d.num_sms, st)) !=
        cudaSuccess)
        return cuda_fail(e, "byoc_ffn_noalloc: first GEMM launch");
    g.N = D;
    g.num_kb = F / 64;
    g.chunks = g.num_kb;
    g.tiles_n = D / kTileN;
    g.num_tiles = tiles_m * g.tiles_n;
    g.group = byoc::gemm_group(kTileN, 64, g.num_kb);
    g.act = byoc::kActNone;
    g.bias = b2;
    g.out = static_cast<__nv_bfloat16 *>(y);
    if ((e = byoc::launch_gemm(cfg, a2, b2m, a2, o2, g, g.num_tiles < d.num_sms ? g.num_tiles : d.num_sms, st)) !=
        cudaSuccess)
        return cuda_fail(e, "byoc_ffn_noalloc: second GEMM launch");
    return BYOC_OK;
}

namespace byoc {

// byoc_check(NULL): read and clear the allocation-free entry point's error
// word on the current device (the first word of g_ffn_scratch).  Before any
// call on this device there is nothing to report.
int noalloc_check() {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "byoc_check: cudaGetDevice");
    if (dev < 0 || dev >= kMaxDevices) return fail(BYOC_ERR_UNSUPPORTED, "byoc_check: device ordinal");
    DeviceState &d = g_devices[dev];
    {
        std::lock_guard<std::mutex> lock(g_devices_mutex);
        if (!d.ready) return BYOC_OK;
    }
    int v = 0;
    if ((e = cudaMemcpy(&v, d.scratch, sizeof v, cudaMemcpyDeviceToHost)) != cudaSuccess)
        return cuda_fail(e, "byoc_check: reading the allocation-free error word");
    if (v != 0) {
        if ((e = cudaMemset(d.scratch, 0, sizeof v)) != cudaSuccess)
            return cuda_fail(e, "byoc_check: clearing the allocation-free error word");
        char buf[128];
        snprintf(buf, sizeof buf, "byoc_ffn_noalloc: a kernel's bounded wait expired (code %d)", v);
        return fail(BYOC_ERR_TIMEOUT, buf);
    }
    return BYOC_OK;
}

}  // namespace byoc
