/*
 * byoc.h -- C ABI of the GB300 (sm_103a) execution engine for partitioned,
 * offloaded regions ("Bring Your Own Codegen", arXiv 2105.03215).
 *
 * The paper's flow (Section 3) partitions a model graph, encapsulates every
 * offloadable region as a function with a target attribute (Section 3.1.3),
 * hands that function to the accelerator's code generator (Section 3.3), and
 * at run time calls it as an external function that reads its inputs from,
 * and writes its outputs to, pre-allocated data entries (Section 3.4,
 * "Execute the graph nodes on the accelerator").  Constants live in the
 * metadata module and are loaded once at initialisation; the accelerator's
 * execution engine is built once and cached (Section 3.4).
 *
 * This header is that boundary:
 *   byoc_compile  -- the per-region code generation + engine initialisation:
 *                    validates the op list, folds batch norm into the weights
 *                    and bias, rounds and packs the weights, uploads them, and
 *                    picks a kernel plan.  Run once; the handle is the cache.
 *   byoc_run      -- the external call F1(...): enqueues the region's kernels
 *                    on a CUDA stream; reads inputs / writes outputs in
 *                    caller-owned device memory (the data entries).
 *   byoc_release  -- frees what byoc_compile allocated.
 *
 * Conventions shared by every entry point:
 *   - Activations are bf16, NHWC for 4-D tensors and row-major [rows, features]
 *     for 2-D tensors (Section 3.2: the accelerator fixes its layout; the
 *     caller transforms at the region boundary).  Constants are fp32, host
 *     memory, copied during byoc_compile (the caller may free them after it
 *     returns).
 *   - Device pointers passed to byoc_run must be 16-byte aligned and point to
 *     contiguous tensors of the shapes given at compile time.
 *   - Every call that can fail returns a byoc_status; on failure a thread-local
 *     message is available from byoc_last_error().  Nothing falls back to the
 *     CPU: an op chain the kernels cannot run is rejected at compile time with
 *     BYOC_ERR_UNSUPPORTED (the paper's cost/annotation rules keep such ops on
 *     the host, Section 3.1.2-3.1.3).
 *   - Device-side waits are bounded; a kernel whose wait expires records
 *     BYOC_ERR_TIMEOUT in a per-handle error word that byoc_check() reports.
 */
#ifndef BYOC_H_
#define BYOC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define BYOC_ABI_VERSION 2u

typedef struct byoc_handle byoc_handle; /* opaque: packed constants, workspace, plans */

typedef enum {
    BYOC_OK = 0,
    BYOC_ERR_INVALID_ARG = 1, /* malformed descriptor, null/misaligned pointer, bad shape */
    BYOC_ERR_UNSUPPORTED = 2, /* valid op chain that no kernel here implements */
    BYOC_ERR_CUDA = 3,        /* a CUDA runtime/driver call failed */
    BYOC_ERR_OOM = 4,         /* device or host allocation failed */
    BYOC_ERR_TIMEOUT = 5      /* a kernel's bounded wait expired (reported by byoc_check) */
} byoc_status;

typedef enum {
    BYOC_BF16 = 0,
    BYOC_FP32 = 1,
    BYOC_E4M3 = 2  /* FP8 E4M3 codes (1 byte): the output of a BYOC_OP_QUANTIZE */
} byoc_dtype;

typedef enum {
    BYOC_LAYOUT_NHWC = 0, /* 4-D activation [N, H, W, C] */
    BYOC_LAYOUT_NC = 1    /* 2-D activation [rows, features] */
} byoc_layout;

/* Operators of the composite patterns (Section 3.1.1: Conv2D, Add/bias, ReLU;
 * Section 4 models add batch norm, ReLU6, GELU and residual add). */
typedef enum {
    BYOC_OP_CONV2D = 0,     /* in[0]=data; consts[0]=weight OIHW [K, C/groups, kh, kw] */
    BYOC_OP_DENSE = 1,      /* in[0]=data [M, I]; consts[0]=weight [units, I] */
    BYOC_OP_BIAS_ADD = 2,   /* in[0]; consts[0]=bias [C] (channel = innermost axis) */
    BYOC_OP_BATCH_NORM = 3, /* in[0]; consts = gamma, beta, moving_mean, moving_var [C]; eps */
    BYOC_OP_RELU = 4,
    BYOC_OP_RELU6 = 5,      /* clip(x, 0, 6) */
    BYOC_OP_GELU = 6,       /* 0.5 x (1 + erf(x / sqrt 2)) */
    BYOC_OP_ADD = 7,        /* in[0] + in[1], same shape */
    BYOC_OP_QUANTIZE = 8    /* Section 3.2 Q node: in[0] bf16 -> out BYOC_E4M3,
                               out = e4m3(in * fp32(1 / S)) rounded to nearest even,
                               saturating at +-448; consts[0] = &S (1 float > 0),
                               consts[1] = &Z (1 float, must be 0: E4M3 is symmetric).
                               A conv2d / dense reading an E4M3 tensor runs in FP8
                               (kind::f8f6f4 tensor cores, fp32 accumulation): its
                               weights, folded with the batch norm that follows, are
                               quantized per output channel with power-of-two scales
                               S_w[k] = 2^ceil(log2(max |w'[k]| / 448)) at compile time,
                               and its output is dequantized (x S S_w[k]) in the epilogue.
                               A QUANTIZE right after the epilogue chain of an FP8
                               conv2d / dense (with BYOC_OPT_REGION_KERNEL: of any
                               conv2d / dense) is fused into that epilogue, which then
                               writes the E4M3 codes; one on a region input, or on a
                               tensor with other readers, is its own launch.  FP8
                               layers need C % 128 == 0. */
} byoc_op_kind;

typedef struct {
    int32_t ndim;     /* 4 (NHWC) or 2 (NC) */
    int64_t shape[4]; /* unused trailing entries ignored */
    int32_t dtype;    /* byoc_dtype; activations must be BYOC_BF16 */
    int32_t layout;   /* byoc_layout */
} byoc_tensor;

typedef struct {
    int32_t kind;        /* byoc_op_kind */
    int32_t n_in;        /* 1, or 2 for BYOC_OP_ADD */
    int32_t in[3];       /* tensor ids (indices into byoc_region_desc.tensors) */
    int32_t out;         /* tensor id of the result */
    int32_t kernel[2];   /* conv2d: kh, kw */
    int32_t stride[2];   /* conv2d: sh, sw */
    int32_t pad[4];      /* conv2d: top, left, bottom, right */
    int32_t dilation[2]; /* conv2d: dh, dw */
    int32_t groups;      /* conv2d: 1, or C for depthwise */
    float eps;           /* batch_norm epsilon */
    const float *consts[4]; /* host fp32 constants, see byoc_op_kind */
} byoc_op;

/* One partitioned region: the function the partitioner encapsulates
 * (Section 3.1.3) in the JSON-like graph form of codegen Option 1
 * (Section 3.3): tensors, ops in topological order, boundary tensor ids. */
typedef struct {
    uint32_t abi_version;         /* must equal BYOC_ABI_VERSION */
    const char *name;             /* region / composite name, informational */
    int32_t n_tensors;
    const byoc_tensor *tensors;
    int32_t n_ops;
    const byoc_op *ops;           /* topological order */
    int32_t n_inputs;
    const int32_t *input_ids;     /* order of byoc_run's inputs[] */
    int32_t n_outputs;
    const int32_t *output_ids;    /* order of byoc_run's outputs[] */
    uint32_t options;             /* BYOC_OPT_* bits: code-generation choices for this region */
} byoc_region_desc;

/* Code-generation options of one region (byoc_region_desc.options).  They
 * choose between kernel plans that compute the same values; the choice is
 * made at compile time and kept in the compiled (and serialised) plan.
 *   BYOC_OPT_FUSE_DW_PW: a depthwise composite and the 1x1 composite that
 *     consumes it run as one kernel whose depthwise output stays in shared
 *     memory (the data-transfer saving that motivates merging operators into
 *     one region, Section 3.1.2).  Off by default: on GB300 the depthwise
 *     arithmetic, not HBM, bounds that kernel, and two launches are faster
 *     on the MobileNetV2 shapes.  Results are bit-identical either way. */
#define BYOC_OPT_FUSE_DW_PW 0x1u
/*   BYOC_OPT_REGION_KERNEL: a region whose composites are all conv2d / dense
 *     (1x1 or k x k, no stem layout) and number two to four (one to four
 *     when FP8) runs as one persistent kernel after its leading quantize
 *     launches: the intermediates are written once and read back from L2,
 *     and a composite's output tiles start as soon as the tiles of the
 *     earlier composites they read are done (no launch boundary between
 *     composites).  Regions that do not qualify get the per-composite plan.
 *     Off by default: measured on GB300 it is slower than the per-composite
 *     plan on the BERT FFN and the ResNet-50 bottleneck. */
#define BYOC_OPT_REGION_KERNEL 0x2u
/*   BYOC_OPT_MULTICAST: a GEMM launch whose weights are streamed through its
 *     ring (tile, im2col or ringed slab mode, no split-K, at least two
 *     m-tiles) runs in clusters of two CTAs that take adjacent m-tiles of one
 *     column tile together and share each weight tile by TMA multicast,
 *     halving the weight bytes each SM reads from L2.  Off by default:
 *     measured on GB300 it is slower on every ResNet-50 / BERT layer here
 *     (the tensor cores' shared-memory operand reads, not L2, bound these
 *     layers, and the CTA pairs wait for each other at every ring stage).
 *     Results are bit-identical either way. */
#define BYOC_OPT_MULTICAST 0x4u
/*   BYOC_OPT_CLUSTER_SPLIT_K: a GEMM launch that splits each tile's k-blocks
 *     over several CTAs (deep reductions over few tiles; tiles at most 128
 *     wide, at most 4 splits) runs each tile's CTAs as one thread-block
 *     cluster that exchanges the fp32 partial accumulators through
 *     distributed shared memory, each CTA summing and storing its share of
 *     the tile's 32-column chunks.  Off by default: the partials then go
 *     through the handle's workspace in global memory, which measured as fast
 *     or faster on GB300 (clusters of three CTAs are much slower).  The
 *     partials are summed in split order either way: results are
 *     bit-identical. */
#define BYOC_OPT_CLUSTER_SPLIT_K 0x8u

/* Figures describing a compiled region. */
typedef struct {
    double flops;           /* algorithmic 2 x MACs per byoc_run (conv2d + dense only) */
    double bytes;           /* algorithmic HBM bytes per byoc_run: every launch reads its
                               inputs and weights once and writes its output once */
    size_t workspace_bytes; /* device workspace owned by the handle (region intermediates) */
    size_t const_bytes;     /* device bytes of packed constants */
    int32_t n_launches;     /* kernel launches one byoc_run enqueues */
    int32_t n_inputs;
    int32_t n_outputs;
} byoc_info;

/* Compile one region (Section 3.3 code generation + Section 3.4 engine
 * initialisation).  Validates the descriptor, folds batch norm and bias into
 * per-channel weight scales and biases in fp64, rounds the folded weights to
 * bf16 (round to nearest even), packs them K-major for the tensor cores,
 * copies all constants to the current CUDA device, and allocates the
 * region's workspace.  Launches no kernel.
 *   desc : read only during the call.
 *   out  : receives the new handle (NULL on failure).
 * Errors: INVALID_ARG (malformed), UNSUPPORTED (chain not implemented),
 *         OOM, CUDA. */
byoc_status byoc_compile(const byoc_region_desc *desc, byoc_handle **out);

/* Run a compiled region: the external function call of Section 3.4.
 *   inputs[i]  : device pointer of the tensor desc->input_ids[i]
 *   outputs[i] : device pointer of the tensor desc->output_ids[i]
 *   cuda_stream: a cudaStream_t (NULL = legacy default stream)
 * Asynchronous: enqueues the kernels and returns.  Pointers must be non-null,
 * 16-byte aligned, and stay valid until the stream reaches the end of the
 * region.  A handle's workspace is shared by its runs, so two runs of one
 * handle must not overlap on the GPU.
 * Errors: INVALID_ARG (null handle / pointer, misalignment), CUDA (launch). */
byoc_status byoc_run(byoc_handle *h, const void *const *inputs, void *const *outputs,
                     void *cuda_stream);

/* Read and clear the handle's device error word.  Call after the stream that
 * ran the handle has been synchronised; returns BYOC_ERR_TIMEOUT if a kernel
 * gave up on a bounded wait since the previous check, else BYOC_OK.
 * With h == NULL it does the same for the error word of byoc_ffn_noalloc on
 * the current device (BYOC_OK before the first such call there).
 * Synchronous (one 4-byte device-to-host copy). */
byoc_status byoc_check(byoc_handle *h);

/* Free everything byoc_compile allocated.  NULL-safe.  The caller must make
 * sure no run of this handle is still in flight. */
void byoc_release(byoc_handle *h);

/* Thread-local message describing the last non-OK status of this thread. */
const char *byoc_last_error(void);

/* Describe a compiled region (see byoc_info). */
byoc_status byoc_query(const byoc_handle *h, byoc_info *info);

/* ---------------------------------------------------------------------------
 * Serialised regions: codegen option 3 of Section 3.3, where the backend's
 * output is serialised into the module so that deployment loads it instead
 * of running the code generator again (the paper's TensorRT engines and
 * Vitis-AI artifacts).  Here the output is the compiled plan: the launch
 * list with its tile choices and arguments, the folded, rounded and packed
 * constants, and the workspace layout.  Host byte order; a layout tag ties
 * the bytes to the library build that wrote them.
 * ------------------------------------------------------------------------- */

/* Write the compiled region h into dst (host memory).
 *   dst       : buffer of dst_bytes bytes, or NULL to query the size only.
 *   needed    : receives the serialised size (always set on success and on a
 *               too-small buffer).
 * Synchronous, touches no device memory.
 * Errors: INVALID_ARG (null handle / size pointer, buffer too small). */
byoc_status byoc_serialize(const byoc_handle *h, void *dst, size_t dst_bytes, size_t *needed);

/* Rebuild a handle from byoc_serialize's bytes on the current CUDA device:
 * uploads the constants, allocates the workspace and encodes the weight
 * descriptors -- no validation of a graph, no batch-norm folding, no packing.
 * src is read only during the call; the new handle behaves exactly like the
 * one that was serialised (same kernels, same results bit for bit).
 * Errors: INVALID_ARG (truncated, corrupted -- checksum -- or inconsistent
 *         bytes), UNSUPPORTED (bytes from another library build; device not
 *         sm_103), OOM, CUDA. */
byoc_status byoc_deserialize(const void *src, size_t src_bytes, byoc_handle **out);

/* ---------------------------------------------------------------------------
 * Host-side operators.  In the paper, operators that stay outside every
 * region run on the host through the compiler's own code generation, and CUDA
 * may serve as the host (Section 3.4, footnote on the metadata module;
 * Section 4.1).  These are the ones the ResNet-50 host graph needs, written
 * here as CUDA kernels so that no step of the graph leaves this library.
 * All are asynchronous on cuda_stream; bf16 NHWC; C must be a multiple of 8;
 * pointers 16-byte aligned.  Errors: INVALID_ARG, CUDA.
 * ------------------------------------------------------------------------- */

/* max_pool2d, window k x k, stride s, symmetric zero-cost padding p (padded
 * positions never win).  x [N,H,W,C] -> y [N,Ho,Wo,C], Ho = (H+2p-k)/s+1. */
byoc_status byoc_max_pool2d_nhwc(const void *x, void *y, int32_t N, int32_t H, int32_t W,
                                 int32_t C, int32_t k, int32_t s, int32_t p, void *cuda_stream);

/* global_avg_pool2d: x [N,H,W,C] -> y [N,C] (fp32 sum, bf16 result). */
byoc_status byoc_global_avg_pool_nhwc(const void *x, void *y, int32_t N, int32_t H, int32_t W,
                                      int32_t C, void *cuda_stream);

/* Layout transformation at a region boundary (Section 3.2): the framework's
 * NCHW fp32 tensor x [N,C,H,W] -> the NHWC bf16 tensor y [N,H,W,c_pad] the
 * regions read, y[n,h,w,c] = x[n,c,h,w] rounded to nearest even, and 0 for
 * C <= c < c_pad.  Requires c_pad >= C and W * c_pad <= 16384; pointers
 * 16-byte aligned.  Asynchronous on cuda_stream.  Errors: INVALID_ARG, CUDA. */
byoc_status byoc_nchw_to_nhwc_bf16(const void *x, void *y, int32_t N, int32_t C, int32_t H, int32_t W,
                                   int32_t c_pad, void *cuda_stream);

/* ---------------------------------------------------------------------------
 * Allocation-free entry point.  The paper has no counterpart: it exists for
 * callers that cannot allocate device memory -- code running inside a memory
 * pool or arena it does not own, or an inference path that must not take an
 * allocator lock or trigger the implicit synchronisation of cudaMalloc.
 * byoc_compile allocates; this call does not.
 *
 * Computes y = GELU(x . w1^T + b1) . w2^T + b2 (the dense + bias + GELU ->
 * dense + bias chain) with the same tcgen05 kernel byoc_run uses:
 *   x  [M, D] bf16, w1 [F, D] bf16, b1 [F] fp32, w2 [D, F] bf16, b2 [D] fp32,
 *   y  [M, D] bf16; all device pointers, row-major, 16-byte aligned.
 *   D and F must be multiples of 128; M * F must not exceed 8,388,608
 *   (the hidden activation goes to a fixed 16 MiB device array that every GPU
 *   loading the library reserves until exit); larger problems fail with
 *   BYOC_ERR_INVALID_ARG -- split the rows over several calls.
 * The first call on each device, with that device current, looks up the
 * array's device address and raises the kernel's shared-memory limit; make
 * that first call before any stream capture.  Every call shares the array,
 * so calls that overlap on the GPU (for example on two streams) race; order
 * them on one stream.  The call enqueues work on cuda_stream and returns; a
 * bounded-wait timeout inside its kernels is recorded in the array and
 * reported by byoc_check(NULL) once the stream has been synchronised (the
 * next call clears it).  A set-up that fails is retried by the next call; a
 * successful one is kept for the life of the process and is not valid after
 * cudaDeviceReset of that device.  It calls no cudaMalloc, cudaFree or other
 * allocating routine.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
byoc_status byoc_ffn_noalloc(const void *x, int32_t M, int32_t D, int32_t F, const void *w1,
                             const float *b1, const void *w2, const float *b2, void *y,
                             void *cuda_stream);

/* ---------------------------------------------------------------------------
 * Kernel trace, for measurement.  Not part of the paper's flow: it lets a
 * benchmark see how long the tensor-core GEMM kernel runs inside a forward
 * pass without putting events between the launches (which would stop each
 * kernel from overlapping its set-up with the previous kernel's tail).
 *
 * byoc_trace_begin(buf, capacity): until byoc_trace_end, every GEMM launch
 * that byoc_run enqueues (also into a CUDA graph being captured) gets the
 * next slot k of buf, a device array of capacity x 2 uint64:
 *   buf[2k]     earliest %globaltimer (ns) at which a CTA of the launch had
 *               finished waiting for the previous kernel (atomic min),
 *   buf[2k + 1] latest %globaltimer at which a CTA of it exited (atomic max).
 * The caller sets buf[2k] = UINT64_MAX and buf[2k + 1] = 0 before each run
 * of the traced launches.  Launches past capacity are not traced.  The trace
 * state is process-wide: begin and end on one thread, with no other thread
 * calling byoc_run meanwhile.
 * byoc_trace_end() returns the number of slots handed out (>= 0) and stops
 * tracing; launches enqueued afterwards (and graphs captured afterwards) are
 * not traced.  Errors (begin): INVALID_ARG for a null or misaligned buf or a
 * capacity < 1. */
byoc_status byoc_trace_begin(void *buf, int32_t capacity);
int32_t byoc_trace_end(void);

/* Number of SMs and the device's compute capability, for host-side planning
 * (current device).  Errors: CUDA. */
byoc_status byoc_device_info(int32_t *num_sms, int32_t *cc_major, int32_t *cc_minor);

#ifdef __cplusplus
}
#endif

#endif /* BYOC_H_ */
