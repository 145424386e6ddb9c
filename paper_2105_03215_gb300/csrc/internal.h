// internal.h -- declarations shared by the translation units of libbyoc.so.
// Not part of the public ABI (include/byoc.h is).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace byoc {

enum Act : int { kActNone = 0, kActRelu = 1, kActRelu6 = 2, kActGelu = 3 };

// Every kernel of the library is launched with programmatic stream
// serialisation: it may be scheduled while the previous kernel in the stream
// is still running.  Each kernel signals pdl_launch_dependents() as it starts
// and calls pdl_wait() -- which returns once the previous grid has completed
// and its memory operations are visible -- before its first global memory
// access, so only set-up work (barrier init, TMEM allocation, descriptor
// prefetch) overlaps the previous kernel's tail.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                      cudaStream_t st, int cluster_x, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cluster_x > 1) {  // thread-block clusters of cluster_x CTAs along x
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = (unsigned)cluster_x;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.numAttrs = 2;
    }
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, Args... args) {
    return launch_pdl_cluster(kernel, grid, block, smem, st, 1, args...);
}

// Implicit-GEMM problem: out[M, N] = act(A[M, K] . B[N, K]^T + bias [+ residual]).
//  A is either a row-major [M, K] matrix (dense, 1x1 stride-1 conv) read with a
//  2-D tiled tensor map, or the implicit im2col matrix of an NHWC activation
//  read with an im2col tensor map: row m = output pixel (n, p, q), column
//  k = (tap r*kw+s, channel chunk, channel).  B is the packed weight matrix.
struct GemmArgs {
    int M;          // output rows
    int N;          // output channels = row stride of out / residual (elements)
    int num_kb;     // k-blocks per tile (taps * chunks)
    int chunks;     // channel chunks (of BK channels) per filter tap
    int kw;         // filter width
    int dil_h, dil_w;
    int Ho, Wo;     // output spatial size (im2col)
    int stride_h, stride_w;
    int pad_t, pad_l;
    int tiles_n;    // number of BN-wide column tiles
    int num_tiles;  // tiles_m * tiles_n
    // slab mode (stride-1 convolution): a tile is slab_t output rows of one
    // image; tile row v = y * wp + x indexes the padded width wp, and filter
    // tap (r, s) reads the slab from row r * wp + s on.  Pair modes: a unit
    // is tiles 2u and 2u + 1 of an image (the second one absent at the end of
    // an image with an odd tiles_per_img), and num_tiles counts units
    int wp;             // padded input width (W + pad_l + pad_r)
    int slab_t;         // output rows per tile
    int tiles_per_img;  // ceil(Ho / slab_t)
    int slab_bytes;     // bytes of one slab (one channel chunk)
    int taps;           // kh * kw
    // resident-weight slab mode: the packed weights (every k-block, one
    // column tile) sit at the start of the shared-memory pool, loaded once
    // per CTA; the slabs take the rest, set by gemm_slab_pool()
    int slab_off;       // bytes from the start of the pool to the first slab slot
    int slab_pitch;     // bytes per slot, a multiple of 1024
    int slab_slots;     // 2 .. kMaxSlabSlots
    // split-K (kAModeTileSplit): fp32 partials [splits][m_pad][n_pad] and one
    // arrival counter per (tile, epilogue warp slot), zeroed once, counted
    // modulo `splits`
    int splits, m_pad, n_pad;
    float *partial;
    unsigned *counters;
    int group;      // k-blocks (slab mode: filter taps) per ring stage, >= 1; the
                    // kernel lowers it so that at least two stages fit the ring
    // packed weights [n_pad][k_pack] (bf16), or null: before waiting for the
    // previous kernel, a CTA prefetches its first tile's weight rows into L2
    const void *w;
    int k_pack;
    int act;        // Act
    const float *bias;                // [tiles_n * BN], zero padded; required
    const __nv_bfloat16 *residual;    // [M, N] or null
    __nv_bfloat16 *out;               // [M, N]
    int *err;                         // device error word
    // FP8 GEMM (bk = kF8BK): the accumulator counts code products; column n
    // is dequantized by dq[n] = S_x S_w[n] before the bias (dq [tiles_n * BN],
    // zero padded).  out8: a fused Q node -- the output is E4M3 codes of
    // value x out_inv, written through the byte output map.
    const float *dq;
    int out8;
    float out_inv;
    // measurement only (byoc_trace_begin), else null: [0] earliest CTA's
    // %globaltimer once its wait for the previous kernel returned (atomic
    // min), [1] latest CTA's at exit (atomic max)
    unsigned long long *trace;
    // > 0: the slab comes from a stem layout (StemArgs) through a 5-D map,
    // box {8 values, wp positions, slab rows, stem_rows image rows, 1} at
    // (0, 0, first output row, 0, image), unswizzled: in shared memory
    // stem_rows planes of slab_bytes / stem_rows, one 16-byte piece per
    // slab position (the MMA reads them as no-swizzle core matrices)
    int stem_rows;
};

enum AMode : int {
    kAModeTile = 0,    // A is a row-major [M, K] matrix (2-D tiled TMA)
    kAModeIm2col = 1,  // A through an im2col TMA map: one load per filter tap and chunk
    kAModeSlab = 2,    // stride-1 conv: one 4-D tiled slab per chunk, taps by row shift
    kAModeSlabRes = 3,  // slab mode, one column tile, all weights resident in shared memory
    kAModeTileSplit = 4,  // tile mode with the k-blocks of every tile split over `splits` CTAs
    // kAModeSlabRes in pair units: two vertically adjacent slab tiles of one
    // image (2 x 128 MMA rows, two accumulators) share one slab load and the
    // per-unit waits and commits
    kAModeSlabRes2 = 5,
    // kAModeTileSplit with the `splits` CTAs of a tile forming one thread-block
    // cluster: the partial accumulators are summed through distributed shared
    // memory (each CTA owns every splits-th 32-column chunk of the tile)
    // instead of fp32 partials in global memory.  BN <= 128, splits <= 4,
    // at most kClRecvBlocks received 128 x 32 blocks per CTA.
    kAModeTileSplitCl = 6
};

constexpr bool amode_slab(int m) { return m == kAModeSlab || m == kAModeSlabRes || m == kAModeSlabRes2; }
constexpr bool amode_split(int m) { return m == kAModeTileSplit || m == kAModeTileSplitCl; }
constexpr int kClMaxSplits = 4;
constexpr int kClRecvBlocks = 4;  // 128 x 32 fp32 blocks (16 KB each) a CTA receives
// whether a cluster split of `splits` CTAs fits the receive buffer at tile width bn
constexpr bool cl_split_fits(int bn, int splits) {
    return splits >= 2 && splits <= kClMaxSplits && bn <= 128 &&
           ((bn / 32 + splits - 1) / splits) * (splits - 1) <= kClRecvBlocks;
}
constexpr bool amode_pair(int m) { return m == kAModeSlabRes2; }
constexpr bool amode_wres(int m) { return m == kAModeSlabRes || m == kAModeSlabRes2; }
// FP8 GEMM (E4M3 A and B, kind::f8f6f4): a k-block of 128 codes (128 bytes,
// the row of one 128-byte swizzle atom, like 64 bf16 values)
constexpr int kF8BK = 128;
// whether the epilogue stores its output with TMA (a map over [M, N] in
// 32 x 32 boxes): tile mode, and every FP8 row-tiled mode (tile, im2col,
// split-K), whose fused Q node writes E4M3 codes through a byte map
constexpr bool gemm_tstore(int amode, int bk) {
    return amode == kAModeTile || (bk == kF8BK && (amode == kAModeIm2col || amode == kAModeTileSplit));
}

struct GemmConfig {
    int bn;      // tile width in output channels: 32, 64, 128, 256
    int bk;      // k-block width in elements: 16, 32, 64 bf16 (sets the swizzle: 32/64/128 B),
                 // or kF8BK: an FP8 GEMM (E4M3 operands, 128-byte swizzle)
    int amode;   // AMode
    bool res;    // epilogue adds a residual tile (bn 64 or 128)
    // clusters of two CTAs sharing each weight tile by TMA multicast (tile,
    // im2col and ringed slab modes); the launch grid is even and the weight
    // map's box is bn / 2 rows
    bool mc = false;
};

// Largest slab (one channel chunk) the slab mode holds, per buffer; a pair
// unit's slab covers both tiles' rows.
constexpr int slab_max_bytes(int bk, bool pair = false) {
    return pair ? (bk == 64 ? 56 * 1024 : 28 * 1024) : (bk == 64 ? 48 * 1024 : 24 * 1024);
}
constexpr int kMaxSlabSlots = 8;

constexpr int kGemmBM = 128;
constexpr int kGemmEpiWarps = 8;
// warp 0 mainloop TMA, warp 1 MMA, warps 2-9 epilogue, warp 10 epilogue operands
constexpr int kGemmOperandWarp = 2 + kGemmEpiWarps;
constexpr int kGemmThreads = 32 * (kGemmOperandWarp + 1);

// k-blocks per ring stage for a run of `n` k-blocks (slab mode: the taps of
// one channel chunk): enough MMA work per barrier handshake (bn * bk * group
// >= 256 * 64, about 600 tensor-core cycles at M = 128) that the single
// issuing thread stays ahead of the tensor pipe, then evened out over n.
inline int gemm_group(int bn, int bk, int n) {
    int g = (256 * 64 + bn * bk - 1) / (bn * bk);
    if (g > 8) g = 8;
    if (n < 1) return 1;
    const int stages = (n + g - 1) / g;
    return (n + stages - 1) / stages;
}

bool gemm_config_supported(const GemmConfig &cfg);
size_t gemm_smem_bytes(const GemmConfig &cfg);
int gemm_stages(const GemmConfig &cfg);
// Resident-weight slab mode: whether num_kb weight k-blocks and two slabs of
// slab_bytes fit the configuration's pool, and the split of the pool
// (a.slab_off, slab_pitch, slab_slots from a.num_kb and a.slab_bytes).
bool gemm_slab_res_fits(const GemmConfig &cfg, int num_kb, int slab_bytes);
void gemm_slab_pool(const GemmConfig &cfg, GemmArgs &a);
cudaError_t gemm_prepare(const GemmConfig &cfg);  // raises the dynamic smem limit
// tmR: the residual [M, N] bf16 in 64-column x 128-row boxes, 128-byte
// swizzle (read only when cfg.res).  tmO: where gemm_tstore(amode, bk), the
// OUTPUT a.out [M, N] bf16 in 32-column x 32-row boxes, 64-byte swizzle
// (a.out8: E4M3 codes in 32 x 32-byte boxes, unswizzled), which the epilogue
// stores through (required: any other map is written through); unused in the
// other modes.  a.bias (and, FP8, a.dq) must cover tiles_n * bn floats.
cudaError_t launch_gemm(const GemmConfig &cfg, const CUtensorMap &tmA, const CUtensorMap &tmB,
                        const CUtensorMap &tmR, const CUtensorMap &tmO, const GemmArgs &a, int grid,
                        cudaStream_t st);

// Depthwise conv (groups = C), square kernel k in {3}, NHWC bf16, folded
// weights fp32 [k*k][C] (tap-major), bias fp32 [C], fused activation.
// Depthwise 3x3 convolution + folded BN/bias + activation, NHWC.  A tile is
// th output rows x tw output columns x cc channels of one image; its input
// (in_rows x in_cols x cc, halo included, zero outside the image) is one TMA
// box.  Persistent CTAs loop over the tiles with two input buffers.
struct DwArgs {
    const float *w;      // [9][C] folded weights, fp32
    const float *bias;   // [C]
    __nv_bfloat16 *y;    // [N, Ho, Wo, C]
    int N, H, W, C, Ho, Wo;
    int stride, pad;
    int act;
    int th, tw, cc;               // output tile rows, columns; channels per chunk (multiple of 8)
    int in_rows, in_cols;         // input box: (th-1)*stride+3, (tw-1)*stride+3
    int tiles_h, tiles_w, chunks;
    int num_tiles;                // chunks * N * tiles_h * tiles_w (chunk slowest)
    int buf_bytes;                // one input buffer, 128-byte multiple
    int threads;                  // (cc / 4) * lanes, <= kDwMaxThreads
    int *err;                     // device error word
};
constexpr int kDwMaxThreads = 512;
constexpr int kDwBlockH = 4, kDwBlockW = 2;  // outputs a thread computes (tiles are multiples)
constexpr size_t kDwBufBudget = 108 * 1024;   // bytes per input buffer; two buffers per CTA
// Tiling for the depthwise kernel; false when no tile fits shared memory.
bool dw_plan(DwArgs &a, int num_sms);
size_t dw_smem_bytes(const DwArgs &a);
// Raises the kernel's dynamic smem limit to the largest size dw_plan can
// choose: the limit belongs to the kernel, not the launch, so several regions
// sharing one instantiation must all fit under it.
cudaError_t dw_prepare(const DwArgs &a);
cudaError_t launch_dwconv(const CUtensorMap &tmX, const DwArgs &a, int grid, cudaStream_t st);

// Layout transform at the region boundary for a stride-2 stem with few
// input channels (Section 3.2): the image with 4 channels and `pad` zero rows
// and columns before it (zero after it up to Hq x Wq),
//   xq[n, u, v, c] = x[n, u - pad, v - pad, c]   (c < C, inside x), else 0,
// so that a pair of pixels is one aligned 16-byte piece.  The stem's GEMM
// reads it through a 5-D tensor map (runtime.cu, encode_stem_slab).
struct StemArgs {
    const __nv_bfloat16 *x;  // [N, H, W, C], C <= 4
    __nv_bfloat16 *xq;       // [N, Hq, Wq, 4]
    int N, H, W, C;
    int Hq, Wq;              // N * Hq <= 2^31 - 1; Wq even
    int pad;
};
// The transform stages kStemRows input rows (W * C bf16 each) in shared
// memory; the planner rejects stems whose rows need more than this.
constexpr size_t kStemLayoutMaxSmem = 48 * 1024;
size_t stem_layout_smem_bytes(const StemArgs &a);
cudaError_t launch_stem_layout(const StemArgs &a, cudaStream_t st);

cudaError_t launch_maxpool(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                           int k, int s, int p, cudaStream_t st);
// Sets the thread-local message byoc_last_error() returns.
void set_last_error(const char *msg);
// The allocation-free entry point's error word on the current device: read,
// clear, BYOC_ERR_TIMEOUT if a wait expired (noalloc.cu).
int noalloc_check();

// Depthwise 3x3 (pad 1, stride 1|2) + folded BN + activation fused with the
// 1x1 conv + folded BN (+ residual) (+ activation) that consumes it (dwpw.cu).
struct DwPwArgs {
    const float *dw_w;                // [9][C] folded depthwise weights, tap-major
    const float *dw_b;                // [C]
    const float *pw_b;                // [n_pad] folded pointwise bias, zero padded
    const __nv_bfloat16 *residual;    // [N, Ho, Wo, Cout] or null
    __nv_bfloat16 *out;               // [N, Ho, Wo, Cout]
    int *err;
    int N, H, W, C, Ho, Wo, stride, pad;
    int dw_act, act;                  // activations after the depthwise and after the pointwise
    int Cout, n_pad, chunks;          // n_pad: Cout rounded up to 16 (the MMA's N); chunks of 64 channels
    int tr;                           // output rows per tile (tr * Wo <= 128)
    int bh;                           // depthwise output rows per thread block (1 or 2)
    int tiles_per_img, num_tiles;
    int in_rows, in_cols, in_bytes, in_pitch;  // input box per (tile, chunk) and its buffer
    int in_stages;                    // input buffers in the ring (2 .. kDpMaxInStages)
    int b_bytes, w_off, a_off, in_off, ctrl_off, smem_bytes;  // shared-memory layout (bytes)
    int acc_stride, tmem_cols;        // TMEM columns per accumulator (>= 32) and allocated
};
constexpr int kDpThreads = 704;
constexpr int kDpMaxInStages = 4;
constexpr int kDpChunk = 64;
constexpr int kDpABytes = 128 * 128;  // A operand: 128 pixels x 64 channels bf16
constexpr int kDpMaxBBytes = 96 * 1024;
constexpr int kDpSmemMax = 232448;
bool dwpw_plan(DwPwArgs &a, int num_sms);  // false: the pair does not fit this kernel
cudaError_t dwpw_prepare(const DwPwArgs &a);
cudaError_t launch_dwpw(const CUtensorMap &tmX, const CUtensorMap &tmB, const DwPwArgs &a, int grid,
                        cudaStream_t st);

// Region kernel (chain.cu): a region's chain of conv2d / dense composites in
// one persistent launch.  Stage s computes out_s[M, N] = act(A_s . B_s^T +
// bias_s [+ residual_s]); A_s is a row-major matrix (tile mode: dense, 1x1
// stride-1 conv) or the im2col matrix of an NHWC tensor, read through maps.A[s];
// B_s through maps.B[s] (BN x 64 boxes); out_s is stored through maps.O[s]
// (32 x 32 boxes, 64-byte swizzle).  A unit is one 128 x BN output tile of one
// stage; order[u] = (stage << 24) | tile gives the u-th unit handed out, tile
// = m-tile * tiles_n + n-tile.  Every 128-row m-tile of a stage has a
// completion counter (counters[cbase + m-tile]) to which each of the 8
// epilogue warps of each of its units adds 1 per launch.
constexpr int kChainMaxStages = 4;
enum : int { kChainTile = 0, kChainIm2col = 1 };
// A CTA's schedule entry (cta_rec): kChainRecInts int32 -- the unit u, its
// code order[u], its dependency count n, its first dependency pair
// dep_off[u], then its first min(n, kChainRecDeps) (counter, count per
// launch) pairs -- so that the scheduler reads one self-contained, 16-byte
// aligned record per unit instead of a chain of dependent loads.
constexpr int kChainRecDeps = 4;
constexpr int kChainRecInts = 4 + 2 * kChainRecDeps;
// (Both structs are laid out without implicit padding: plans are serialised
// byte for byte.)
struct ChainStage {
    const float *bias;       // [tiles_n * BN], zero padded
    const __nv_bfloat16 *residual;  // [M, N] or null (a region input or an earlier stage's output)
    const float *dq;         // FP8 stage: [tiles_n * BN] dequantization scales S_x S_w[n], else null
    int mode;                // kChainTile | kChainIm2col
    int M, N;                // output rows; output channels (row stride of out and residual)
    int num_kb, chunks, kw;  // k-blocks of 128 bytes (im2col: taps x chunks), chunks per tap, filter width
    int dil_h, dil_w, Ho, Wo, stride_h, stride_w, pad_t, pad_l;  // im2col geometry
    int tiles_n, num_tiles;
    int unit0;               // first unit of this stage in stage-major numbering (host bookkeeping)
    int cbase;               // first completion counter of this stage (one per m-tile)
    int act;
    int consumed;            // a later stage reads this stage's output: its units count into the counters
    int res_dep;             // the residual is an earlier stage's output
    int fp8;                 // A and B are E4M3 codes (kind::f8f6f4); a k-block is 128 elements, not 64
    int out8;                // the output is quantized to E4M3 codes with out_inv (a fused Q node)
    float out_inv;           // fp32(1 / S) of that Q node
    int reserved[2];
};
struct ChainArgs {
    ChainStage st[kChainMaxStages];
    const int *order;        // [total_units]: (stage << 24) | tile of the u-th unit
    const int *cta_off;      // [grid + 1]: CTA b runs the units of records cta_off[b] .. cta_off[b+1]), in order
    const int *cta_rec;      // [total_units * kChainRecInts]: the records, CTA after CTA
    const int *dep_off;      // [total_units + 1]: unit u's dependencies are the pairs
    const int *dep_list;     //   (counter, count per launch) at dep_list[2 j], j in [dep_off[u], dep_off[u+1])
    unsigned *flags;         // [n_counters] completion counters, zeroed at compile
    unsigned *ctl;           // [4]: unused, CTAs finished, launches completed, unused
    int *err;
    unsigned long long *trace;  // as GemmArgs::trace
    int n_stages, total_units, n_counters, reserved;
};
// every field counted: 3 pointers and 26 4-byte fields, so no padding byte
static_assert(sizeof(ChainStage) == 3 * 8 + 26 * 4 && offsetof(ChainStage, reserved) + 8 == sizeof(ChainStage) &&
                  sizeof(ChainArgs) == kChainMaxStages * sizeof(ChainStage) + 9 * 8 + 16,
              "region kernel arguments without padding");
struct ChainMaps {
    CUtensorMap A[kChainMaxStages], B[kChainMaxStages], O[kChainMaxStages];
};
size_t chain_smem_bytes(int bn);
int chain_stages(int bn);
cudaError_t chain_prepare(int bn);  // bn: 128 or 256
cudaError_t launch_chain(int bn, const ChainMaps &maps, const ChainArgs &a, int grid, cudaStream_t st);

// Section 3.2 Q node on a region input: q[i] = e4m3(x[i] * inv_scale) (the
// product in fp32, nearest even, saturating at +-448); n a multiple of 8,
// both pointers 16-byte aligned.
cudaError_t launch_quantize_e4m3(const __nv_bfloat16 *x, uint8_t *q, size_t n, float inv_scale, int num_sms,
                                 cudaStream_t st);

// NCHW fp32 -> NHWC bf16 (channels zero-padded to Cp) at a region boundary.
// Requires W * Cp <= kNchwStageElems; y 16-byte aligned when its rows are.
constexpr int kNchwStageElems = 16384;
int nchw_rows_per_block(int W, int Cp);
cudaError_t launch_nchw_to_nhwc(const float *x, __nv_bfloat16 *y, int N, int C, int H, int W, int Cp,
                                cudaStream_t st);
cudaError_t launch_avgpool(const __nv_bfloat16 *x, __nv_bfloat16 *y, int N, int H, int W, int C,
                           cudaStream_t st);

}  // namespace byoc
