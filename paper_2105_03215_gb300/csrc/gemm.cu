// gemm.cu -- implicit-GEMM convolution and dense layer on the sm_103a tensor
// cores (tcgen05), with the region's bias / folded batch norm / residual add
// / activation fused into the epilogue, so each offloaded composite
// (Section 3.1.1: a Conv2D-Add-ReLU style sequence mapped to one
// "instruction") makes one pass over HBM.
//
// Structure (one persistent CTA per SM, 352 threads).  Every role that waits
// on a barrier has a warp of its own: a lane suspended in mbarrier.try_wait
// holds up the divergent paths of the other lanes of its warp.
//   warp 0     TMA producer of the mainloop (one elected lane issues).  The A
//              operand (activations) comes in one of three ways (AMODE):
//                tile   a 128 x BK tile of a row-major [M, K] matrix;
//                im2col 128 consecutive output pixels of one filter tap and
//                       channel chunk (out-of-image taps zero-filled by TMA);
//                slab   stride-1 convolutions: for each channel chunk one
//                       4-D tiled box of the padded input rows under the tile
//                       (the "slab"); each filter tap (r, s) is the same slab
//                       read from row r * Wp + s on, by shifting the MMA's
//                       shared-memory descriptor -- one load per chunk instead
//                       of one per tap.
//              The B operand (packed weights) is one BN x BK tile per k-block;
//              a ring stage holds G k-blocks.
//   warp 1     allocates TMEM; one elected lane issues tcgen05.mma (M=128,
//              N=BN, K=16 per instruction) into one of two fp32 accumulators
//              in TMEM and tcgen05.commit's the ring stages and the finished
//              accumulator.
//   warps 2-9  epilogue: two groups of four warps (one per 32-row TMEM lane
//              quarter).  For BN <= 64 the groups take alternate tiles, so
//              that two tiles' epilogues overlap; for wider tiles they split
//              each tile's 32-column chunks.  Per chunk: tcgen05.ld (one row per
//              thread), + bias and + residual from shared memory, activation,
//              bf16 rounding, then a transpose through a 64-byte-swizzled
//              shared-memory tile so that the global stores are coalesced
//              64-byte row segments.  The accumulator is released as soon as
//              it has been read, so the next tile's MMAs overlap this tile's
//              stores.
//   warp 10    producer of the epilogue operands: per tile, the tile's bias
//              slice (bulk copy) and, when the region adds a residual, the
//              128 x BN residual tile (TMA) into a ring of OPB buffers.
//
// FP8 (BK = kF8BK; Section 3.2's partial quantization): A holds the E4M3
// codes a Q node wrote, B the weights quantized per output channel; a k-block
// is 128 codes (128 bytes, the same swizzled rows as 64 bf16 values), one
// kind::f8f6f4 MMA per 32 of them.  The epilogue dequantizes with one fma
// (accumulator x S_x S_w[n] + bias[n]) and, when a Q node follows the
// composite, writes E4M3 codes instead of bf16 (TMA store of 32 x 32 bytes).
//
// Cluster multicast (MC, on request: BYOC_OPT_MULTICAST): the kernel runs in
// clusters of two CTAs that take
// the m-tiles 2i and 2i + 1 of the same column tile together, k-block by
// k-block.  Both need the same weight tile, so each CTA loads half of its
// rows and multicasts them to both; a ring stage is refilled once both CTAs'
// MMAs have read it (each MMA commit arrives on the stage's empty barrier in
// both CTAs).  This halves the weight bytes each SM pulls from L2 -- the
// operand traffic that bounds the layers whose weights are re-read by every
// m-tile.  With an odd number of m-tiles the last cluster's second CTA runs a
// phantom m-tile past the end: its loads fall outside the tensors and read
// zeros, its stores are clipped or skipped.
#include "internal.h"
#include "ptx.cuh"

namespace byoc {

template <int BN, int BK, int AMODE, bool RES, bool MC>
struct GemmShape {
    static constexpr int BM = kGemmBM;
    static constexpr bool SLAB = amode_slab(AMODE);
    static constexpr bool WRES = amode_wres(AMODE);  // weights resident
    static constexpr bool PAIR = amode_pair(AMODE);  // two tiles (halves) per unit
    static constexpr int HALVES = PAIR ? 2 : 1;
    static_assert(!PAIR || WRES, "pair units keep their weights resident");
    // FP8: E4M3 operands, 128 codes per k-block (kind::f8f6f4, K = 32 per MMA)
    static constexpr bool F8 = BK == kF8BK;
    static constexpr int ROW_BYTES = F8 ? BK : BK * 2;  // one K-major operand row (= swizzle width)
    static constexpr int A_BYTES = SLAB ? 0 : BM * ROW_BYTES;
    static constexpr int B_BYTES = BN * ROW_BYTES;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int SLAB_BYTES = SLAB ? slab_max_bytes(BK, PAIR) : 0;
    // slab barriers: two slots beside a weight ring; up to kMaxSlabSlots
    // beside resident weights (the ring and the two largest slabs form one
    // pool, split at run time)
    static constexpr int SLOTS_MAX = WRES ? kMaxSlabSlots : 2;
    // two accumulators (double buffer), each HALVES x BN columns
    static constexpr int ACC_COLS = HALVES * BN;
    static constexpr int TMEM_COLS = 2 * ACC_COLS < 32 ? 32 : 2 * ACC_COLS;
    // residual tile: BN/64 boxes of 64 columns x 128 rows, 128-byte swizzle
    static constexpr int RES_BOX = BM * 64 * 2;
    static constexpr int RES_TILE = RES ? BM * BN * 2 : 0;
    // epilogue-operand buffers (bias slice, residual tile): residual regions
    // are HBM-bound and keep more residual tiles in flight; bias-only slices
    // are small, and eight in flight keep their L2 latency off short tiles
    static constexpr int OPB = RES ? (BN >= 128 ? 3 : 4) : 8;
    static constexpr int BIAS_BYTES = BN * 4 * (F8 ? 2 : 1);  // bias slice (FP8: then the dq slice)
    static constexpr int BIAS_REGION = (OPB * BIAS_BYTES + 1023) / 1024 * 1024;
    // epilogue staging: one 32x32 bf16 output tile per epilogue warp
    static constexpr int EPI_TILE = 32 * 32 * 2;
    // tile mode (and FP8) stores its output with TMA from each warp's
    // staging tile; the others read the staging tile back for coalesced stores
    static constexpr bool TSTORE = gemm_tstore(AMODE, BK);
    static constexpr int CTRL_BYTES = 1024;
    // cluster split-K: the blocks of partial sums the other CTAs send
    static constexpr bool CLSPLIT = AMODE == kAModeTileSplitCl;
    static constexpr int RECV_BLOCK = BM * 32 * 4;  // 128 rows x 32 fp32
    static constexpr int RECV_BYTES = CLSPLIT ? kClRecvBlocks * RECV_BLOCK : 0;
    static constexpr int RECV_BARS = CLSPLIT ? 2 : 0;  // one per chunk this CTA owns (BN <= 128)
    // TMA-store mode keeps a second staging tile per warp (one store in
    // flight while the next chunk is staged) where the weight ring still
    // has 8 stages with it: short-k-block configs (BK 16 / 32)
    static constexpr int FIXED1 = 1024 + 2 * SLAB_BYTES + RECV_BYTES + OPB * RES_TILE + BIAS_REGION + CTRL_BYTES;
    static constexpr int EPI_BUFS =
        TSTORE && (232448 - FIXED1 - 2 * kGemmEpiWarps * EPI_TILE) / STAGE_BYTES >= 8 ? 2 : 1;
    static constexpr int EPI_BYTES = kGemmEpiWarps * EPI_TILE * EPI_BUFS;
    static constexpr int FIXED = FIXED1 + EPI_BYTES;
    static constexpr int STAGES_RAW = (232448 - FIXED) / STAGE_BYTES;
    static constexpr int STAGES = STAGES_RAW > 32 ? 32 : STAGES_RAW;  // ring slots (k-blocks)
    static constexpr int POOL_BYTES = STAGES * STAGE_BYTES + 2 * SLAB_BYTES;
    static constexpr int NUM_BARS = 2 * STAGES + 5 + 2 * SLOTS_MAX + 2 * OPB + RECV_BARS;
    static constexpr int SMEM_BYTES = FIXED + STAGES * STAGE_BYTES;
    static_assert(8 * NUM_BARS + 16 <= CTRL_BYTES, "control block");
    static_assert(STAGES >= 2, "ring depth");
    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
    static_assert(A_BYTES % 1024 == 0 && B_BYTES % 1024 == 0 && SLAB_BYTES % 1024 == 0,
                  "buffers must keep 1 KB alignment");
    static_assert(BN % 32 == 0 && BN >= 32 && BN <= 256, "BN");
    static_assert(TMEM_COLS <= 512, "TMEM: two accumulators of HALVES x BN columns");
    static_assert(!RES || BN % 64 == 0, "residual tiles are loaded in 64-column boxes");
    static_assert(!(RES && SLAB), "slab tiles skip pad columns; no residual tile");
    static_assert(BK == 16 || BK == 32 || BK == 64 || F8, "BK");
    static_assert(!F8 || (AMODE == kAModeTile || AMODE == kAModeIm2col || AMODE == kAModeTileSplit),
                  "FP8: tile, im2col and split-K modes");
    static_assert(!CLSPLIT || (BN <= 128 && !RES), "cluster split-K: BN <= 128, no residual");
    static_assert(!MC || (!WRES && !PAIR && !amode_split(AMODE)),
                  "multicast: weights streamed through the ring, one tile per unit");
    static constexpr int B_HALF = B_BYTES / 2;  // multicast: the rows one CTA loads
    static_assert(!MC || B_HALF % 1024 == 0, "a multicast half keeps the swizzle's 1 KB alignment");
};

// Slab modes: image, first output row and tile count (halves) of m-unit mt.
// Single-tile modes: tile mt of tiles_per_img per image.  Pair modes: tiles
// 2u and 2u + 1 of an image, the second absent past the image's last tile.
struct SlabUnit {
    int img, p0, nh;
};
template <bool PAIR>
__device__ __forceinline__ SlabUnit slab_unit(const GemmArgs &a, int mt) {
    SlabUnit u;
    if constexpr (PAIR) {
        const int upi = (a.tiles_per_img + 1) >> 1;
        u.img = mt / upi;
        const int pu = mt - u.img * upi;
        u.p0 = 2 * pu * a.slab_t;
        u.nh = 2 * pu + 1 < a.tiles_per_img ? 2 : 1;
    } else {
        u.img = mt / a.tiles_per_img;
        u.p0 = (mt - u.img * a.tiles_per_img) * a.slab_t;
        u.nh = 1;
    }
    return u;
}

// ReLU, ReLU6 or none; GELU is applied to lane pairs (gelu2) by the caller.
__device__ __forceinline__ float apply_act(float v, int act) {
    switch (act) {
        case kActRelu: return fmaxf(v, 0.0f);
        case kActRelu6: return fminf(fmaxf(v, 0.0f), 6.0f);
        default: return v;
    }
}

template <int BN, int BK, int AMODE, bool RES, bool MC>
// 168 registers: 11 warps put three on some SM sub-partitions, and three
// warps x 32 lanes x 168 fit a sub-partition's 16384 registers.
__global__ void __maxnreg__(168)
    gemm_tcgen05_kernel(const __grid_constant__ CUtensorMap tmA,
                        const __grid_constant__ CUtensorMap tmB,
                        const __grid_constant__ CUtensorMap tmR,
                        const __grid_constant__ CUtensorMap tmO, const GemmArgs a) {
    using S = GemmShape<BN, BK, AMODE, RES, MC>;
    constexpr bool PAIR = S::PAIR;
    // The two epilogue warp groups take alternate tiles (all chunks each) for
    // narrow tiles, and for launches of one column tile whose tiles hold an
    // odd number of 32-column chunks (a 2 + 1 chunk split would leave one
    // group idle half the time); otherwise both take every tile, splitting
    // its chunks (pair units: one half each).  Epilogue warps that read each
    // accumulator: four when alternating, else eight.
    // (the run-time choice only where it occurs: 128-wide plain tiles)
    constexpr bool ALT_RT = BN == 128 && AMODE == kAModeTile && !RES;
    const bool alt = (BN <= 64 && !PAIR) ||
                     (ALT_RT && a.tiles_n == 1 && ((min(BN / 32, (a.N + 31) >> 5)) & 1));
    const int epi_arrivals = alt ? kGemmEpiWarps / 2 : kGemmEpiWarps;
    // split-K: a work unit is (tile, split); split sp covers k-blocks
    // [sp * num_kb / SPL, (sp + 1) * num_kb / SPL)
    constexpr bool SPLITK = AMODE == kAModeTileSplit || AMODE == kAModeTileSplitCl;
    constexpr bool CLSPLIT = S::CLSPLIT;  // a tile's splits form one cluster (rank = split)
    const int SPL = SPLITK ? a.splits : 1;
    const int num_units = a.num_tiles * SPL;
    // The loop over work units, the same in every role: unit u_first,
    // u_first + u_step, ... below num_loop.  MC: a unit is the pair of
    // m-tiles (2i, 2i + 1) of one column tile, this CTA taking m-tile
    // 2i + crank; tile_of() gives the tile (split-K: the unit's tile).
    const int crank = MC ? (int)cluster_ctarank() : 0;
    const int num_loop = MC ? ((a.num_tiles / a.tiles_n + 1) >> 1) * a.tiles_n : num_units;
    const int u_first = MC ? (int)(blockIdx.x >> 1) : (int)blockIdx.x;
    const int u_step = MC ? (int)(gridDim.x >> 1) : (int)gridDim.x;
    auto tile_of = [&](int u) -> int {
        if constexpr (MC) {
            const int mp = u / a.tiles_n;
            return (2 * mp + crank) * a.tiles_n + (u - mp * a.tiles_n);
        } else {
            return u / SPL;
        }
    };
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (base - raw);
    const uint32_t sA = base;
    const uint32_t sB = sA + S::STAGES * S::A_BYTES;
    const uint32_t sPoolEnd = sB + S::STAGES * S::B_BYTES + 2 * S::SLAB_BYTES;
    // slabs: 2 x SLAB_BYTES after the ring, or (resident weights) slab_slots x slab_pitch
    const uint32_t sSlab = S::WRES ? sB + (uint32_t)a.slab_off : sB + S::STAGES * S::B_BYTES;
    const uint32_t sRecv = sPoolEnd;                       // RECV_BYTES (cluster split-K)
    const uint32_t sRes = sRecv + S::RECV_BYTES;           // OPB x RES_TILE
    const uint32_t sEpi = sRes + S::OPB * S::RES_TILE;     // EPI_BYTES
    const uint32_t sBias = sEpi + S::EPI_BYTES;            // 2 x BIAS_BYTES
    const uint32_t ctrl = sBias + S::BIAS_REGION;
    const uint32_t bars = ctrl;                            // full[S], empty[S]
    const uint32_t tfull = bars + 8u * (2 * S::STAGES);    // 2: accumulator ready
    const uint32_t tempty = tfull + 16u;                   // 2: accumulator drained
    const uint32_t ofull = tempty + 16u;                   // OPB: epilogue operands loaded
    const uint32_t oempty = ofull + 8u * S::OPB;           // OPB: epilogue operands consumed
    const uint32_t sfull = oempty + 8u * S::OPB;           // SLOTS_MAX: slab loaded
    const uint32_t sempty = sfull + 8u * S::SLOTS_MAX;     // SLOTS_MAX: slab consumed
    const uint32_t drain = sempty + 8u * S::SLOTS_MAX;
    const uint32_t recv_bar = drain + 8u;                  // RECV_BARS: a received chunk complete
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + (ctrl - base) + 8 * S::NUM_BARS);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S::STAGES; ++s) {
            mbar_init(bars + 8u * s, 1);                  // full[s]: producer + TMA bytes
            mbar_init(bars + 8u * (S::STAGES + s), MC ? 2 : 1);  // empty[s]: MMA commit (MC: both CTAs')
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(tfull + 8u * b, 1);                 // MMA commit
            mbar_init(tempty + 8u * b, epi_arrivals);     // one arrive per epilogue warp of the tile
        }
        for (int b = 0; b < S::SLOTS_MAX; ++b) {
            mbar_init(sfull + 8u * b, 1);                 // producer + slab bytes
            mbar_init(sempty + 8u * b, 1);                // MMA commit
        }
        for (int b = 0; b < S::OPB; ++b) {
            mbar_init(ofull + 8u * b, 1);                 // operand producer + bytes
            mbar_init(oempty + 8u * b, epi_arrivals);     // one arrive per epilogue warp of the tile
        }
        mbar_init(drain, 1);
        // every lane of the four warps that read a chunk, in each other CTA
        for (int b = 0; b < S::RECV_BARS; ++b) mbar_init(recv_bar + 8u * b, 128u * (uint32_t)(a.splits - 1));
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
        if (RES) tma_prefetch_desc(&tmR);
        if (S::TSTORE) tma_prefetch_desc(&tmO);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), S::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if constexpr (MC || CLSPLIT) cluster_sync();  // the cluster's barriers initialised
    const uint32_t tmem_base = *tmem_slot;
    // Set-up done: the next kernel may be scheduled; global memory is touched
    // only after the previous kernel has completed -- except for the packed
    // weights, constant for the handle's lifetime: the operand warp
    // prefetches its share of its first tile's weight rows into L2, and the
    // producer loads the first ring stages' weights (resident-weight mode:
    // all of them) into shared memory, while the previous kernel finishes;
    // the producer waits for it only before its first activation load.
    pdl_launch_dependents();
    if (!SPLITK && warp == kGemmOperandWarp && a.w != nullptr && u_first < num_loop) {
        if (elect_one()) {
            // The CTAs whose first unit is in column tile j (units j,
            // j + tiles_n, ...) share its weight rows (MC: this CTA's half of
            // them): each prefetches its own part, so L2 sees every byte
            // requested once.
            constexpr int PF_ROWS = MC ? BN / 2 : BN;
            const size_t row_bytes = (size_t)a.k_pack * (S::F8 ? 1 : 2);
            const int j = u_first % a.tiles_n, q = u_first / a.tiles_n;
            const int users = (min(u_step, num_loop) - 1 - j) / a.tiles_n + 1;
            const size_t slice = (size_t)PF_ROWS * row_bytes;
            const size_t part = (slice / (size_t)users + 15) / 16 * 16;
            const size_t lo = min(slice, (size_t)q * part);
            const uint8_t *src = static_cast<const uint8_t *>(a.w) +
                                 ((size_t)j * BN + (size_t)crank * PF_ROWS) * row_bytes + lo;
            const size_t bytes = min(slice, lo + part) - lo;
            for (size_t off = 0; off < bytes; off += 32768)
                bulk_prefetch_l2(src + off, (uint32_t)(bytes - off < 32768 ? bytes - off : 32768));
        }
        __syncwarp();
    }
    if (warp != 0) pdl_wait();
    if (a.trace != nullptr && threadIdx.x == 32) atomicMin(a.trace, globaltimer_ns());
    // Ring stages of G k-blocks each; at least two stages.
    const int G = a.group < 1 ? 1 : (a.group > S::STAGES / 2 ? S::STAGES / 2 : a.group);
    const int nst = S::STAGES / G;

    if (warp == 0) {
        // -------------------------------------------------- mainloop producer
        // Like the MMA warp, one lane chosen by elect.sync runs the whole
        // loop.  A ring stage holds G consecutive k-blocks (slab mode: G
        // filter taps of one channel chunk): one barrier handshake per stage.
        if (elect_one()) {
            auto wait = [&](uint32_t bar, uint32_t parity) -> bool {
                return mbar_wait(bar, parity, abort_flag, a.err, kErrTimeoutProducer);
            };
            int stage = 0, slot0 = 0, sl = 0, issued = 0;
            uint32_t phase = 0;
            bool ok = true;
            // Wait for `stage` to be free and announce `bytes` on its full barrier.
            auto claim = [&](uint32_t bytes) -> bool {
                if (!wait(bars + 8u * (S::STAGES + stage), phase ^ 1u)) return false;
                mbar_arrive_expect_tx(bars + 8u * stage, bytes);
                return true;
            };
            auto advance = [&]() {
                ++issued;
                slot0 += G;
                if (++stage == nst) {
                    stage = 0;
                    slot0 = 0;
                    phase ^= 1u;
                }
            };
            int ss = 0;        // resident weights: slab slot of slab sl, and its phase
            uint32_t sph = 0;
            // one weight tile (BN rows at n0, k-block column kx) into ring slot
            // dst; MC: this CTA's half of the rows, to both CTAs
            auto load_b = [&](uint32_t dst, uint32_t bar, int kx, int n0) {
                if constexpr (MC)
                    tma_load_2d_mc(dst + (uint32_t)(crank * S::B_HALF), &tmB, bar, kx, n0 + crank * (BN / 2),
                                   (uint16_t)0x3);
                else
                    tma_load_2d(dst, &tmB, bar, kx, n0);
            };
            if constexpr (S::WRES) {
                // the whole weight matrix once, on ring stage 0
                if (claim((uint32_t)(a.num_kb * S::B_BYTES))) {
                    for (int kb = 0; kb < a.num_kb; ++kb)
                        tma_load_2d(sB + kb * S::B_BYTES, &tmB, bars, kb * BK, 0);
                    advance();
                } else {
                    ok = false;
                }
            }
            // Where all of this CTA's units are in one column tile (tiles_n == 1,
            // or a grid that is a multiple of tiles_n: units u_first + k u_step
            // share u_first % tiles_n) they read the same weight k-blocks, and
            // where a unit's ring stages (spu of them) divide the ring, ring
            // slot s holds the same k-blocks on every pass.  After the first
            // pass over the ring the weights are in place and only A is loaded:
            // one TMA copy per k-block instead of two (measured on MobileNetV2's
            // short-K 1x1 layers: the 112x112 32 -> 16 layer 37.4 -> 29.2 us;
            // their rate is set by the per-tile copy chain).
            const int spu = (a.num_kb + G - 1) / G;
            // (several column tiles: not with a residual, where the same-box
            // A/B on ResNet-50's conv3 layers measured ~3 us slower per step)
            const bool b_keep = !SPLITK && !MC && !S::SLAB &&
                                (a.tiles_n == 1 || (!RES && u_step % a.tiles_n == 0)) && nst % spu == 0;
            // Tile / im2col / split modes: claim the first unit's first ring
            // stages and load their weights before waiting for the previous
            // kernel; their activations follow the wait (same stage barriers).
            // (measured: the same for the ringed slab mode's first chunk costs
            // ~2 us on the ResNet-50 step, so that mode waits first)
            int pre = 0;
            if constexpr (!S::SLAB) {
                if (u_first < num_loop) {
                    const int t0 = tile_of(u_first);
                    const int sp0 = SPLITK ? u_first - t0 * SPL : 0;
                    const int n00 = (t0 % a.tiles_n) * BN;
                    const int lo = SPLITK ? sp0 * a.num_kb / SPL : 0;
                    const int hi = SPLITK ? (sp0 + 1) * a.num_kb / SPL : a.num_kb;
                    for (int kb = lo; kb < hi && pre < nst; kb += G, ++pre) {
                        const int gn = hi - kb < G ? hi - kb : G;
                        // fresh ring: stage pre is free; the full barrier expects A and B
                        mbar_arrive_expect_tx(bars + 8u * pre, (uint32_t)(gn * S::STAGE_BYTES));
                        for (int g = 0; g < gn; ++g)
                            load_b(sB + (pre * G + g) * S::B_BYTES, bars + 8u * pre, (kb + g) * BK, n00);
                    }
                }
            }
            pdl_wait();
            for (int unit = u_first; ok && unit < num_loop; unit += u_step) {
                const int tile = tile_of(unit);
                const int sp = SPLITK ? unit - tile * SPL : 0;
                const int mt = tile / a.tiles_n;
                const int n0 = (tile % a.tiles_n) * BN;
                if constexpr (S::WRES) {
                    const SlabUnit su = slab_unit<PAIR>(a, mt);
                    const int img = su.img, p0 = su.p0;
                    for (int cc = 0; cc < a.chunks; ++cc, ++sl) {
                        if (!wait(sempty + 8u * ss, sph ^ 1u)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(sfull + 8u * ss, (uint32_t)a.slab_bytes);
                        if (a.stem_rows > 0)  // stem layout: one chunk
                            tma_load_5d(sSlab + (uint32_t)(ss * a.slab_pitch), &tmA, sfull + 8u * ss, 0, 0, p0, 0,
                                        img);
                        else
                            tma_load_4d(sSlab + (uint32_t)(ss * a.slab_pitch), &tmA, sfull + 8u * ss,
                                        cc * BK, -a.pad_l, p0 - a.pad_t, img);
                        if (++ss == a.slab_slots) {
                            ss = 0;
                            sph ^= 1u;
                        }
                    }
                } else if constexpr (S::SLAB) {
                    const SlabUnit su = slab_unit<PAIR>(a, mt);
                    const int img = su.img, p0 = su.p0;
                    for (int cc = 0; ok && cc < a.chunks; ++cc, ++sl) {
                        const int ss = sl & 1;
                        const uint32_t sph = (uint32_t)(sl >> 1) & 1u;
                        if (!wait(sempty + 8u * ss, sph ^ 1u)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(sfull + 8u * ss, (uint32_t)a.slab_bytes);
                        if (a.stem_rows > 0)  // stem layout: one chunk
                            tma_load_5d(sSlab + ss * S::SLAB_BYTES, &tmA, sfull + 8u * ss, 0, 0, p0, 0, img);
                        else
                            tma_load_4d(sSlab + ss * S::SLAB_BYTES, &tmA, sfull + 8u * ss, cc * BK,
                                        -a.pad_l, p0 - a.pad_t, img);
                        for (int tap = 0, kb = cc; tap < a.taps; tap += G) {
                            const int gn = a.taps - tap < G ? a.taps - tap : G;
                            if (!claim((uint32_t)(gn * S::B_BYTES))) {
                                ok = false;
                                break;
                            }
                            for (int g = 0; g < gn; ++g)
                                load_b(sB + (slot0 + g) * S::B_BYTES, bars + 8u * stage, (kb + g * a.chunks) * BK,
                                       n0);
                            kb += gn * a.chunks;
                            advance();
                        }
                    }
                } else {
                    const int m0 = mt * S::BM;
                    int img = 0, h0 = 0, w0 = 0;
                    if constexpr (AMODE == kAModeIm2col) {
                        const int hw = a.Ho * a.Wo;
                        img = m0 / hw;
                        const int rem = m0 - img * hw;
                        const int p = rem / a.Wo;
                        const int q = rem - p * a.Wo;
                        h0 = p * a.stride_h - a.pad_t;
                        w0 = q * a.stride_w - a.pad_l;
                    }
                    int cc = 0, r = 0, sx = 0;  // (tap r, s; chunk cc) of k-block kb, im2col mode
                    const int kb_lo = SPLITK ? sp * a.num_kb / SPL : 0;
                    const int kb_hi = SPLITK ? (sp + 1) * a.num_kb / SPL : a.num_kb;
                    for (int kb = kb_lo; kb < kb_hi; kb += G) {
                        const int gn = kb_hi - kb < G ? kb_hi - kb : G;
                        const bool preloaded = pre > 0;  // claimed, weights issued before the wait
                        // weights already in this ring slot (b_keep, below): A only
                        const bool skip_b = b_keep && issued >= nst;
                        if (preloaded) {
                            --pre;
                        } else if (!claim((uint32_t)(gn * (skip_b ? S::A_BYTES : S::STAGE_BYTES)))) {
                            ok = false;
                            break;
                        }
                        const uint32_t full = bars + 8u * stage;
                        for (int g = 0; g < gn; ++g) {
                            const uint32_t dA = sA + (slot0 + g) * S::A_BYTES;
                            if constexpr (AMODE == kAModeIm2col) {
                                tma_load_im2col_4d(dA, &tmA, full, cc * BK, w0, h0, img,
                                                   (uint16_t)(sx * a.dil_w), (uint16_t)(r * a.dil_h));
                                if (++cc == a.chunks) {
                                    cc = 0;
                                    if (++sx == a.kw) {
                                        sx = 0;
                                        ++r;
                                    }
                                }
                            } else {
                                tma_load_2d(dA, &tmA, full, (kb + g) * BK, m0);
                            }
                            if (!preloaded && !skip_b) load_b(sB + (slot0 + g) * S::B_BYTES, full, (kb + g) * BK, n0);
                        }
                        advance();
                    }
                }
            }
            if (!ok) {
                // Gave up: let the copies already issued land before exiting.
                for (int j = issued - nst > 0 ? issued - nst : 0; j < issued; ++j)
                    mbar_wait_drain(bars + 8u * (j % nst), (uint32_t)(j / nst) & 1u);
                const int nsl = S::WRES ? a.slab_slots : 2;
                for (int j = sl - nsl > 0 ? sl - nsl : 0; j < sl; ++j)
                    mbar_wait_drain(sfull + 8u * (j % nsl), (uint32_t)(j / nsl) & 1u);
            }
        }
        __syncwarp();
    } else if (warp == kGemmOperandWarp) {
        if (elect_one()) {
            // ------------------------------------------------ epilogue-operand producer
            int t = 0;
            for (int unit = u_first; unit < num_loop; unit += u_step, ++t) {
                const int tile = tile_of(unit);
                const int ob = t % S::OPB;
                const uint32_t oph = (uint32_t)(t / S::OPB) & 1u;
                if (!mbar_wait(oempty + 8u * ob, oph ^ 1u, abort_flag, a.err, kErrTimeoutProducer))
                    break;
                const int m0 = (tile / a.tiles_n) * S::BM;
                const int n0 = (tile % a.tiles_n) * BN;
                mbar_arrive_expect_tx(ofull + 8u * ob, S::BIAS_BYTES + S::RES_TILE);
                if constexpr (S::F8) {  // bias slice, then the dequantization scales
                    bulk_load_1d(sBias + ob * S::BIAS_BYTES, a.bias + n0, BN * 4, ofull + 8u * ob);
                    bulk_load_1d(sBias + ob * S::BIAS_BYTES + BN * 4, a.dq + n0, BN * 4, ofull + 8u * ob);
                } else {
                    bulk_load_1d(sBias + ob * S::BIAS_BYTES, a.bias + n0, S::BIAS_BYTES, ofull + 8u * ob);
                }
                if constexpr (RES) {
#pragma unroll
                    for (int j = 0; j < BN / 64; ++j)
                        tma_load_2d(sRes + ob * S::RES_TILE + j * S::RES_BOX, &tmR, ofull + 8u * ob,
                                    n0 + 64 * j, m0);
                }
            }
            // Let the last operand loads land before the CTA can exit.
            for (int j = t - S::OPB > 0 ? t - S::OPB : 0; j < t; ++j)
                mbar_wait_drain(ofull + 8u * (j % S::OPB), (uint32_t)(j / S::OPB) & 1u);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer
        // One lane chosen by elect.sync runs the whole loop: waits, MMAs and
        // commits.  Issued this way tcgen05.mma keeps the tensor pipe fed
        // (measured: a voted wait or a __syncwarp per stage starves it), and
        // the compiler knows that a single lane issues.  The path per
        // k-block is kept lean: the ring position advances by
        // compare-and-wrap, descriptors advance by adding (byte offset >> 4)
        // to their 14-bit address field, and filter taps are walked without
        // division.
        if (elect_one()) {
            auto wait = [&](uint32_t bar, uint32_t parity) -> bool {
                return mbar_wait(bar, parity, abort_flag, a.err, kErrTimeoutMma);
            };
            constexpr uint32_t idesc = S::F8 ? make_idesc_e4m3(S::BM, BN) : make_idesc_bf16(S::BM, BN);
            // Slab operands, in descriptor units (16 bytes): pos_u per slab
            // position (= operand row) and k_u per K16 slice.  TMA-swizzled
            // slabs: rows of ROW_BYTES, a slice 32 bytes on.  Stem slabs (row
            // planes, no swizzle): rows 16 bytes apart, a slice two planes on.
            const bool planes = S::SLAB && a.stem_rows > 0;
            const uint32_t plane = planes ? (uint32_t)a.slab_bytes / (uint32_t)a.stem_rows : 0u;
            const uint32_t pos_u = planes ? 1u : (uint32_t)(S::ROW_BYTES >> 4);
            const uint32_t k_u = planes ? 2u * (plane >> 4) : 2u;
            const uint64_t adesc0 = planes ? make_smem_desc_planes(sSlab, plane)
                                           : make_smem_desc(S::SLAB ? sSlab : sA, S::ROW_BYTES);
            const uint64_t bdesc0 = make_smem_desc(sB, S::ROW_BYTES);
            int stage = 0, slot0 = 0;
            uint32_t phase = 0;
            int sl = 0, t = 0;
            int ss = 0;        // resident weights: slab slot and its phase
            uint32_t sph = 0;
            bool ok = true;
            // pair units: the second half's rows start slab_t padded rows
            // further into the slab; its accumulator BN columns further on
            const uint64_t hoff = PAIR ? (uint64_t)((uint32_t)(a.slab_t * a.wp) * pos_u) : 0;
            if constexpr (S::WRES) {  // the resident weights, once per CTA
                ok = wait(bars, 0u);
                tc_fence_after();
            }
            auto advance = [&]() {
                slot0 += G;
                if (++stage == nst) {
                    stage = 0;
                    slot0 = 0;
                    phase ^= 1u;
                }
            };
            // a ring stage's MMAs are done (MC: in both CTAs' empty barriers)
            auto free_stage = [&](int st) {
                if constexpr (MC)
                    mma_commit_mc(bars + 8u * (S::STAGES + st), (uint16_t)0x3);
                else
                    mma_commit(bars + 8u * (S::STAGES + st));
            };
            for (int unit = u_first; ok && unit < num_loop; unit += u_step, ++t) {
                const int sp = SPLITK ? unit - (unit / SPL) * SPL : 0;
                const int buf = t & 1;
                const uint32_t aph = (uint32_t)(t >> 1) & 1u;
                if (!wait(tempty + 8u * buf, aph ^ 1u)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(buf * S::ACC_COLS);
                uint32_t acc = 0u;
                bool two = false;  // pair unit with both halves present
                if constexpr (PAIR) two = slab_unit<true>(a, unit / a.tiles_n).nh == 2;
                if constexpr (S::WRES) {
                    // k-block of filter tap t and chunk cc sits at t * chunks + cc
                    const uint64_t bstep = (uint64_t)((uint32_t)(a.chunks * S::B_BYTES) >> 4);
                    for (int cc = 0; ok && cc < a.chunks; ++cc) {
                        if (!wait(sfull + 8u * ss, sph)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint64_t slab_desc =
                            adesc0 + (uint64_t)((uint32_t)(ss * a.slab_pitch) >> 4);
                        uint32_t rpos = 0;  // r * wp: first slab position of filter row r
                        int sx = 0;
                        uint64_t bd = bdesc0 + (uint64_t)((uint32_t)(cc * S::B_BYTES) >> 4);
                        for (int tap = 0; tap < a.taps; ++tap, bd += bstep) {
                            const uint64_t ad = slab_desc + (uint64_t)((rpos + (uint32_t)sx) * pos_u);
#pragma unroll
                            for (int k = 0; k < BK / 16; ++k)
                                mma_bf16_ss(d_tmem, ad + (uint64_t)(k * k_u), bd + (uint64_t)(2 * k), idesc,
                                            acc | (uint32_t)k);
                            if (PAIR && two) {
#pragma unroll
                                for (int k = 0; k < BK / 16; ++k)
                                    mma_bf16_ss(d_tmem + (uint32_t)BN, ad + hoff + (uint64_t)(k * k_u),
                                                bd + (uint64_t)(2 * k), idesc, acc | (uint32_t)k);
                            }
                            acc = 1u;
                            if (++sx == a.kw) {
                                sx = 0;
                                rpos += (uint32_t)a.wp;
                            }
                        }
                        mma_commit(sempty + 8u * ss);  // frees the slab
                        if (++ss == a.slab_slots) {
                            ss = 0;
                            sph ^= 1u;
                        }
                    }
                } else if constexpr (S::SLAB) {
                    for (int cc = 0; ok && cc < a.chunks; ++cc, ++sl) {
                        const int ss = sl & 1;
                        if (!wait(sfull + 8u * ss, (uint32_t)(sl >> 1) & 1u)) {
                            ok = false;
                            break;
                        }
                        const uint64_t slab_desc = adesc0 + (uint64_t)((ss * S::SLAB_BYTES) >> 4);
                        uint32_t rpos = 0;  // r * wp: first slab position of filter row r
                        int sx = 0;
                        for (int tap = 0; tap < a.taps; tap += G) {
                            const int gn = a.taps - tap < G ? a.taps - tap : G;
                            if (!wait(bars + 8u * stage, phase)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            uint64_t bd = bdesc0 + (uint64_t)((slot0 * S::B_BYTES) >> 4);
                            for (int g = 0; g < gn; ++g, bd += (uint64_t)(S::B_BYTES >> 4)) {
                                const uint64_t ad = slab_desc + (uint64_t)((rpos + (uint32_t)sx) * pos_u);
#pragma unroll
                                for (int k = 0; k < BK / 16; ++k)
                                    mma_bf16_ss(d_tmem, ad + (uint64_t)(k * k_u), bd + (uint64_t)(2 * k),
                                                idesc, acc | (uint32_t)k);
                                acc = 1u;
                                if (++sx == a.kw) {
                                    sx = 0;
                                    rpos += (uint32_t)a.wp;
                                }
                            }
                            free_stage(stage);
                            advance();
                        }
                        if (!ok) break;
                        mma_commit(sempty + 8u * ss);  // frees the slab
                    }
                } else {
                    const int kb_lo = SPLITK ? sp * a.num_kb / SPL : 0;
                    const int kb_hi = SPLITK ? (sp + 1) * a.num_kb / SPL : a.num_kb;
                    for (int kb = kb_lo; kb < kb_hi; kb += G) {
                        const int gn = kb_hi - kb < G ? kb_hi - kb : G;
                        if (!wait(bars + 8u * stage, phase)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        uint64_t ad = adesc0 + (uint64_t)((slot0 * S::A_BYTES) >> 4);
                        uint64_t bd = bdesc0 + (uint64_t)((slot0 * S::B_BYTES) >> 4);
                        for (int g = 0; g < gn; ++g, ad += (uint64_t)(S::A_BYTES >> 4),
                                 bd += (uint64_t)(S::B_BYTES >> 4)) {
                            // one MMA per 32 bytes of the k-block row: K = 16
                            // bf16 values or K = 32 E4M3 codes
#pragma unroll
                            for (int k = 0; k < S::ROW_BYTES / 32; ++k) {
                                if constexpr (S::F8)
                                    mma_f8_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                                              acc | (uint32_t)k);
                                else
                                    mma_bf16_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc,
                                                acc | (uint32_t)k);
                            }
                            acc = 1u;
                        }
                        free_stage(stage);
                        advance();
                    }
                }
                if (!ok) break;
                mma_commit(tfull + 8u * buf);  // accumulator complete
            }
            // All issued MMAs must finish before TMEM is released.
            mma_commit(drain);
            mbar_wait_drain(drain, 0);
        }
        __syncwarp();
    } else {
        // ---------------------------------------------------- epilogue
        const int e = warp - 2;            // 0..7
        const int quarter = warp & 3;      // TMEM lanes (= tile rows) this warp may access
        constexpr int NCH = BN / 32;       // 32-column chunks per tile
        // alt: the two groups take alternate tiles (accumulator t % 2), all
        // chunks each.  Otherwise both groups take every tile, group `grp`
        // the chunks ci with ci % 2 == grp, so that a tile's accumulator is
        // read, and released to the MMAs, twice as fast.  Pair units: group
        // `grp` takes half `grp` of every unit, all chunks.  (Split-K keeps
        // the compile-time choice ALT: its partial layout depends on it.)
        constexpr bool ALT = BN <= 64 && !PAIR;
        const int grp = e >> 2;
        const uint32_t stg0 = sEpi + (uint32_t)(e * S::EPI_BUFS) * S::EPI_TILE;
        int sb = 0;  // staging tile of the next chunk (TMA-store mode with two)
        const int trow = quarter * 32 + lane;  // this thread's row within the tile
        // 64-byte swizzle of the 32x32 bf16 staging tile: 16-byte piece c of
        // row r sits at piece c ^ ((r >> 1) & 3), so both the row-per-thread
        // writes and the coalesced reads below are free of bank conflicts.
        const uint32_t sw_own = ((uint32_t)lane >> 1) & 3u;
        const int cl_row = lane >> 2, cl_piece = lane & 3;  // coalesced: rows 8k + lane/4
        const int t_first = alt ? grp : 0, t_step = alt ? 2 : 1;
        const int c_first = alt || PAIR ? 0 : grp, c_step = alt || PAIR ? 1 : 2;
        const int half = PAIR ? grp : 0;
        for (int unit = u_first + t_first * u_step, t = t_first; unit < num_loop;
             unit += t_step * u_step, t += t_step) {
            const int tile = tile_of(unit);
            const int buf = t & 1;
            const uint32_t aph = (uint32_t)(t >> 1) & 1u;
            if (!mbar_wait(tfull + 8u * buf, aph, abort_flag, a.err, kErrTimeoutEpilogue)) break;
            const int ob = t % S::OPB;  // epilogue-operand buffer
            if (!mbar_wait(ofull + 8u * ob, (uint32_t)(t / S::OPB) & 1u, abort_flag, a.err,
                           kErrTimeoutEpilogue))
                break;
            tc_fence_after();
            const int mt = tile / a.tiles_n;
            const int n0 = (tile % a.tiles_n) * BN;
            int img = 0, p0 = 0;
            if constexpr (S::SLAB) {
                const SlabUnit su = slab_unit<PAIR>(a, mt);
                if (PAIR && half >= su.nh) {
                    // single tile at the end of an image: nothing for this
                    // group; its arrivals still count the unit in
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        mbar_arrive(tempty + 8u * buf);
                        mbar_arrive(oempty + 8u * ob);
                    }
                    continue;
                }
                img = su.img;
                p0 = su.p0 + half * a.slab_t;
            }
            // output pixel (row of out / residual) of the 4 rows this lane stores, or -1
            int orow[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int v = quarter * 32 + 8 * k + cl_row;
                if constexpr (S::SLAB) {
                    const int y = v / a.wp;
                    const int x = v - y * a.wp;
                    const int row = (img * a.Ho + p0 + y) * a.Wo + x;
                    const bool ok = y < a.slab_t && x < a.Wo && p0 + y < a.Ho && row < a.M;
                    orow[k] = ok ? row : -1;
                } else {
                    const int row = mt * S::BM + v;
                    orow[k] = row < a.M ? row : -1;
                }
            }
            const uint32_t tbase = tmem_base + ((uint32_t)(quarter * 32) << 16) +
                                   (uint32_t)(buf * S::ACC_COLS + half * BN);
            const uint32_t bias_s = sBias + (uint32_t)(ob * S::BIAS_BYTES);
            const uint32_t res_s = sRes + (uint32_t)(ob * S::RES_TILE);
            // split-K: every split writes its fp32 partial of this warp's rows
            // and columns, then counts itself in on the tile's counter for this
            // warp's slot; the split that completes the count sums all partials
            // in split order (the same bits whichever split finishes last) and
            // runs the epilogue.  No split waits for another.
            const int sp = SPLITK ? unit - tile * SPL : 0;
            // Partials are laid out the way the warp reads TMEM, not as the
            // output matrix: per (tile, warp slot, chunk) 32 x 32 fp32 with
            // the 16-byte piece q of lane l at (q * 32 + l) * 16 bytes, so
            // every store (and every load of the last split) is a contiguous
            // 512-byte run.  Only the same (slot, lane) of another split ever
            // reads it.
            const int slot = ALT ? quarter : quarter * 2 + grp;
            constexpr int kSlotFloats = (ALT ? NCH : NCH / 2) * 1024;
            const size_t pbase = SPLITK ? (size_t)tile * (size_t)(S::BM * BN) + (size_t)slot * kSlotFloats +
                                              (size_t)lane * 4
                                        : 0;
            const size_t pstride = SPLITK ? (size_t)a.num_tiles * (size_t)(S::BM * BN) : 0;  // one split
            if constexpr (CLSPLIT) {
                // Cluster split-K (one tile per cluster, split = rank): chunk ci
                // belongs to rank ci % splits.  Each chunk of this warp that
                // another rank owns goes to that rank's receive block (block
                // (ci / splits) * (splits - 1) + the sender's place among the
                // other ranks; row r at r * 128 bytes, 16-byte piece q at
                // q ^ (r & 7)), then each lane arrives on the owner's barrier
                // for it, releasing its stores.  Every send comes before any
                // wait, so no rank waits on a rank that is itself waiting.
                int owned = 0;
#pragma unroll 1
                for (int ci = c_first; ci < NCH; ci += c_step) {
                    const int owner = ci % SPL;
                    if (owner == sp) {
                        ++owned;
                        continue;
                    }
                    uint32_t v[32];
                    tmem_ld_32cols(tbase + (uint32_t)(ci * 32), v);
                    const int blk = (ci / SPL) * (SPL - 1) + (sp < owner ? sp : sp - 1);
                    const uint32_t dst =
                        mapa_shared(sRecv + (uint32_t)(blk * S::RECV_BLOCK) + (uint32_t)trow * 128u, (uint32_t)owner);
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        st_cluster_v4(dst + ((((uint32_t)q) ^ ((uint32_t)trow & 7u)) << 4), v[4 * q], v[4 * q + 1],
                                      v[4 * q + 2], v[4 * q + 3]);
                    mbar_arrive_remote(mapa_shared(recv_bar + 8u * (uint32_t)(ci / SPL), (uint32_t)owner));
                }
                if (owned == 0) {  // no more reads of the accumulator by this warp
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(tempty + 8u * buf);
                }
            } else if constexpr (SPLITK) {
#pragma unroll 1
                for (int ci = c_first, k = 0; ci < NCH; ci += c_step, ++k) {
                    uint32_t v[32];
                    tmem_ld_32cols(tbase + (uint32_t)(ci * 32), v);
                    float *dst = a.partial + (size_t)sp * pstride + pbase + (size_t)k * 1024;
#pragma unroll
                    for (int q = 0; q < 8; ++q)
                        *reinterpret_cast<uint4 *>(dst + q * 128) =
                            make_uint4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
                }
                __threadfence();
                __syncwarp();
                unsigned old = 0u;
                if (lane == 0) old = atomicAdd(a.counters + (size_t)tile * 8 + slot, 1u);
                old = __shfl_sync(0xffffffffu, old, 0);
                if (old % (unsigned)SPL != (unsigned)(SPL - 1)) {
                    // not the last split of this tile: release the accumulator and operands
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) {
                        mbar_arrive(tempty + 8u * buf);
                        mbar_arrive(oempty + 8u * ob);
                    }
                    continue;
                }
                __threadfence();  // the other splits' partials are read after the count
            }
            // chunks holding output columns: the 32-column chunks of a ragged
            // last column tile that lie wholly past N are neither read nor
            // stored (split-K partials cover every chunk)
            const int nch = SPLITK ? NCH : min(NCH, (a.N - n0 + 31) >> 5);
            if (c_first >= nch) {  // nothing of this tile for this warp
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(tempty + 8u * buf);
            }
#pragma unroll 1
            for (int ci = c_first, kk = 0; ci < nch; ci += c_step, ++kk) {
                if (CLSPLIT && ci % SPL != sp) continue;  // sent to its owner above
                const int col0 = n0 + ci * 32;
                uint32_t v[32];
                tmem_ld_32cols(tbase + (uint32_t)(ci * 32), v);  // includes tcgen05.wait::ld
                int next = ci + c_step;  // this warp's next chunk (cluster split-K: that this rank owns)
                if constexpr (CLSPLIT)
                    while (next < nch && next % SPL != sp) next += c_step;
                if (next >= nch) {  // this warp's last read of the accumulator
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(tempty + 8u * buf);
                }
                if constexpr (CLSPLIT) {
                    // the other ranks' blocks of this chunk, summed in split
                    // order with this rank's own (the bits of the global split-K)
                    mbar_wait_cluster(recv_bar + 8u * (uint32_t)(ci / SPL), 0u, abort_flag, a.err,
                                      kErrTimeoutEpilogue);
                    float sum[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) sum[j] = 0.0f;
                    for (int s2 = 0; s2 < SPL; ++s2) {
                        if (s2 == sp) {
#pragma unroll
                            for (int j = 0; j < 32; ++j) sum[j] += __uint_as_float(v[j]);
                        } else {
                            const int blk = (ci / SPL) * (SPL - 1) + (s2 < sp ? s2 : s2 - 1);
                            const uint32_t src = sRecv + (uint32_t)(blk * S::RECV_BLOCK) + (uint32_t)trow * 128u;
#pragma unroll
                            for (int q = 0; q < 8; ++q) {
                                float4 p4;
                                asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                                             : "=f"(p4.x), "=f"(p4.y), "=f"(p4.z), "=f"(p4.w)
                                             : "r"(src + ((((uint32_t)q) ^ ((uint32_t)trow & 7u)) << 4)));
                                sum[4 * q] += p4.x;
                                sum[4 * q + 1] += p4.y;
                                sum[4 * q + 2] += p4.z;
                                sum[4 * q + 3] += p4.w;
                            }
                        }
                    }
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = __float_as_uint(sum[j]);
                } else if constexpr (SPLITK) {
                    float sum[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) sum[j] = 0.0f;
                    for (int s2 = 0; s2 < SPL; ++s2) {
                        if (s2 == sp) {
#pragma unroll
                            for (int j = 0; j < 32; ++j) sum[j] += __uint_as_float(v[j]);
                        } else {
                            const float *src = a.partial + (size_t)s2 * pstride + pbase + (size_t)kk * 1024;
#pragma unroll
                            for (int q = 0; q < 8; ++q) {
                                // L2: written by other CTAs
                                const float4 p4 = __ldcg(reinterpret_cast<const float4 *>(src + q * 128));
                                sum[4 * q] += p4.x;
                                sum[4 * q + 1] += p4.y;
                                sum[4 * q + 2] += p4.z;
                                sum[4 * q + 3] += p4.w;
                            }
                        }
                    }
#pragma unroll
                    for (int j = 0; j < 32; ++j) v[j] = __float_as_uint(sum[j]);
                }
                float f[32];
#pragma unroll
                for (int j = 0; j < 8; ++j) {  // bias: same address in every lane (broadcast)
                    float4 b4;
                    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                                 : "=f"(b4.x), "=f"(b4.y), "=f"(b4.z), "=f"(b4.w)
                                 : "r"(bias_s + (uint32_t)(ci * 32 + 4 * j) * 4u));
                    if constexpr (S::F8) {
                        // the accumulator is in units of S_x S_w[n]: one fma
                        // dequantizes and adds the bias
                        float4 d4;
                        asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                                     : "=f"(d4.x), "=f"(d4.y), "=f"(d4.z), "=f"(d4.w)
                                     : "r"(bias_s + (uint32_t)(BN + ci * 32 + 4 * j) * 4u));
                        f[4 * j] = fmaf(__uint_as_float(v[4 * j]), d4.x, b4.x);
                        f[4 * j + 1] = fmaf(__uint_as_float(v[4 * j + 1]), d4.y, b4.y);
                        f[4 * j + 2] = fmaf(__uint_as_float(v[4 * j + 2]), d4.z, b4.z);
                        f[4 * j + 3] = fmaf(__uint_as_float(v[4 * j + 3]), d4.w, b4.w);
                    } else {
                        f[4 * j] = __uint_as_float(v[4 * j]) + b4.x;
                        f[4 * j + 1] = __uint_as_float(v[4 * j + 1]) + b4.y;
                        f[4 * j + 2] = __uint_as_float(v[4 * j + 2]) + b4.z;
                        f[4 * j + 3] = __uint_as_float(v[4 * j + 3]) + b4.w;
                    }
                }
                if constexpr (RES) {
                    // residual row `trow`, columns ci*32.. of the 128B-swizzled box ci/2
                    const uint32_t rbox =
                        res_s + (uint32_t)((ci >> 1) * S::RES_BOX) + (uint32_t)trow * 128u;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const uint32_t piece = (uint32_t)((ci & 1) * 4 + q) ^ ((uint32_t)trow & 7u);
                        uint4 r4;
                        asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                     : "=r"(r4.x), "=r"(r4.y), "=r"(r4.z), "=r"(r4.w)
                                     : "r"(rbox + (piece << 4)));
                        const uint32_t rr[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
                        for (int e2 = 0; e2 < 4; ++e2) {
                            f[8 * q + 2 * e2] += bf16lo(rr[e2]);
                            f[8 * q + 2 * e2 + 1] += bf16hi(rr[e2]);
                        }
                    }
                }
                if (a.act == kActGelu) {
#pragma unroll
                    for (int j = 0; j < 16; ++j) {
                        const uint64_t g = gelu2(f32x2(f[2 * j], f[2 * j + 1]));
                        f[2 * j] = lane0(g);
                        f[2 * j + 1] = lane1(g);
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < 32; ++j) f[j] = apply_act(f[j], a.act);
                }
                // this thread's row -> swizzled staging -> coalesced global stores
                // (TMA-store mode: one bulk tensor store of the 32 x 32 tile;
                // the staging layout is the 64-byte swizzle TMA reads)
                const uint32_t stg = stg0 + (uint32_t)(sb * S::EPI_TILE);
                if constexpr (S::TSTORE) {
                    // the store that last used this staging tile has read it
                    if (lane == 0) bulk_wait_group_read<S::EPI_BUFS - 1>();
                }
                __syncwarp();
                if (S::F8 && a.out8) {
                    // a fused Q node: E4M3 codes of f x fp32(1/S), 32 bytes per
                    // row, rows 32 bytes apart (the unswizzled box of the byte map)
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        uint32_t w[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const float *g = f + 16 * h + 4 * k;
                            w[k] = cvt_e4m3x2(g[0] * a.out_inv, g[1] * a.out_inv) |
                                   (cvt_e4m3x2(g[2] * a.out_inv, g[3] * a.out_inv) << 16);
                        }
                        const uint32_t addr = stg + (uint32_t)lane * 32u + (uint32_t)h * 16u;
                        asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(w[0]),
                                     "r"(w[1]), "r"(w[2]), "r"(w[3])
                                     : "memory");
                    }
                } else {
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        const uint32_t w0 = pack_bf16x2(f[8 * q + 0], f[8 * q + 1]);
                        const uint32_t w1 = pack_bf16x2(f[8 * q + 2], f[8 * q + 3]);
                        const uint32_t w2 = pack_bf16x2(f[8 * q + 4], f[8 * q + 5]);
                        const uint32_t w3 = pack_bf16x2(f[8 * q + 6], f[8 * q + 7]);
                        const uint32_t addr = stg + (uint32_t)lane * 64u + (((uint32_t)q ^ sw_own) << 4);
                        asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(w0),
                                     "r"(w1), "r"(w2), "r"(w3)
                                     : "memory");
                    }
                }
                if constexpr (S::TSTORE) {
                    // rows past M and columns past N are not written by TMA
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        // (a box wholly past M -- the ragged or phantom m-tile's -- is skipped)
                        if (mt * S::BM + quarter * 32 < a.M) tma_store_2d(&tmO, stg, col0, mt * S::BM + quarter * 32);
                        bulk_commit_group();
                    }
                    if (S::EPI_BUFS == 2) sb ^= 1;
                    continue;
                }
                __syncwarp();
                const int gcol = col0 + cl_piece * 8;
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const uint32_t r = (uint32_t)(8 * k + cl_row);
                    const uint32_t addr =
                        stg + r * 64u + ((((uint32_t)cl_piece) ^ ((r >> 1) & 3u)) << 4);
                    uint4 o;
                    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                 : "=r"(o.x), "=r"(o.y), "=r"(o.z), "=r"(o.w)
                                 : "r"(addr)
                                 : "memory");
                    if (orow[k] >= 0 && gcol < a.N)
                        *reinterpret_cast<uint4 *>(a.out + (size_t)orow[k] * a.N + gcol) = o;
                }
            }
            // bias / residual reads of this tile are done (ordered by __syncwarp)
            __syncwarp();
            if (lane == 0) mbar_arrive(oempty + 8u * ob);
        }
        if constexpr (S::TSTORE) {
            // the output is written before the CTA exits (and its staging
            // tiles stay valid until TMA has read them)
            if (lane == 0) bulk_wait_group<0>();
            __syncwarp();
        }
    }

    __syncwarp();
    tc_fence_before();
    __syncthreads();
    // MC: the peer's multicast copies into this CTA and its MMA commits on
    // this CTA's barriers are complete once it has passed its own waits
    if constexpr (MC || CLSPLIT) cluster_sync();
    if (a.trace != nullptr && threadIdx.x == 0) atomicMax(a.trace + 1, globaltimer_ns());
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, S::TMEM_COLS);
    }
}

// ---------------------------------------------------------------- dispatch

template <int BN, int BK, int AMODE, bool RES, bool MC>
static cudaError_t launch_t(const CUtensorMap &tmA, const CUtensorMap &tmB, const CUtensorMap &tmR,
                            const CUtensorMap &tmO, const GemmArgs &a, int grid, cudaStream_t st) {
    using S = GemmShape<BN, BK, AMODE, RES, MC>;
    return launch_pdl_cluster(gemm_tcgen05_kernel<BN, BK, AMODE, RES, MC>, dim3(grid), dim3(kGemmThreads),
                      (size_t)S::SMEM_BYTES, st, MC ? 2 : (S::CLSPLIT ? a.splits : 1), tmA, tmB, tmR, tmO, a);
}

template <int BN, int BK, int AMODE, bool RES, bool MC>
static cudaError_t prepare_t() {
    using S = GemmShape<BN, BK, AMODE, RES, MC>;
    return cudaFuncSetAttribute(gemm_tcgen05_kernel<BN, BK, AMODE, RES, MC>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, S::SMEM_BYTES);
}

// The instantiated (BN, BK, A mode, residual, cluster multicast)
// combinations; BK = kF8BK (128) are the FP8 ones.
#define BYOC_GEMM_CONFIGS(X)                 \
    X(32, 64, kAModeTile, false, false)      \
    X(64, 64, kAModeTile, false, false)      \
    X(128, 64, kAModeTile, false, false)     \
    X(256, 64, kAModeTile, false, false)     \
    X(64, 64, kAModeTile, true, false)       \
    X(32, 16, kAModeTile, false, false)      \
    X(64, 16, kAModeTile, false, false)      \
    X(128, 16, kAModeTile, false, false)     \
    X(32, 32, kAModeTile, false, false)      \
    X(64, 32, kAModeTile, false, false)      \
    X(128, 32, kAModeTile, false, false)     \
    X(128, 64, kAModeTile, true, false)      \
    X(32, 64, kAModeIm2col, false, false)    \
    X(64, 64, kAModeIm2col, false, false)    \
    X(128, 64, kAModeIm2col, false, false)   \
    X(256, 64, kAModeIm2col, false, false)   \
    X(64, 64, kAModeIm2col, true, false)     \
    X(128, 64, kAModeIm2col, true, false)    \
    X(64, 16, kAModeIm2col, false, false)    \
    X(64, 32, kAModeIm2col, false, false)    \
    X(128, 32, kAModeIm2col, false, false)   \
    X(64, 64, kAModeSlab, false, false)      \
    X(128, 64, kAModeSlab, false, false)     \
    X(256, 64, kAModeSlab, false, false)     \
    X(64, 16, kAModeSlab, false, false)      \
    X(64, 32, kAModeSlab, false, false)      \
    X(64, 64, kAModeTileSplit, false, false) \
    X(128, 64, kAModeTileSplit, false, false) \
    X(256, 64, kAModeTileSplit, false, false) \
    X(64, 64, kAModeTileSplitCl, false, false) \
    X(128, 64, kAModeTileSplitCl, false, false) \
    X(64, 64, kAModeSlabRes, false, false)   \
    X(128, 64, kAModeSlabRes, false, false)  \
    X(64, 16, kAModeSlabRes, false, false)   \
    X(64, 32, kAModeSlabRes, false, false)   \
    X(64, 64, kAModeSlabRes2, false, false)  \
    X(128, 64, kAModeSlabRes2, false, false) \
    X(64, 32, kAModeSlabRes2, false, false)  \
    X(64, 64, kAModeTile, false, true)       \
    X(128, 64, kAModeTile, false, true)      \
    X(256, 64, kAModeTile, false, true)      \
    X(64, 64, kAModeTile, true, true)        \
    X(128, 64, kAModeTile, true, true)       \
    X(64, 64, kAModeIm2col, false, true)     \
    X(128, 64, kAModeIm2col, false, true)    \
    X(256, 64, kAModeIm2col, false, true)    \
    X(128, 64, kAModeIm2col, true, true)     \
    X(64, 64, kAModeSlab, false, true)       \
    X(128, 64, kAModeSlab, false, true)      \
    X(256, 64, kAModeSlab, false, true)       \
    X(64, 128, kAModeTile, false, false)      \
    X(128, 128, kAModeTile, false, false)     \
    X(256, 128, kAModeTile, false, false)     \
    X(64, 128, kAModeTile, true, false)       \
    X(128, 128, kAModeTile, true, false)      \
    X(64, 128, kAModeIm2col, false, false)    \
    X(128, 128, kAModeIm2col, false, false)   \
    X(256, 128, kAModeIm2col, false, false)   \
    X(128, 128, kAModeIm2col, true, false)    \
    X(64, 128, kAModeTileSplit, false, false) \
    X(128, 128, kAModeTileSplit, false, false) \
    X(256, 128, kAModeTileSplit, false, false)

#define BYOC_GEMM_MATCH(c, BN_, BK_, AM_, RES_, MC_) \
    ((c).bn == BN_ && (c).bk == BK_ && (c).amode == AM_ && (c).res == RES_ && (c).mc == MC_)

bool gemm_config_supported(const GemmConfig &c) {
#define X(BN_, BK_, AM_, RES_, MC_) \
    if (BYOC_GEMM_MATCH(c, BN_, BK_, AM_, RES_, MC_)) return true;
    BYOC_GEMM_CONFIGS(X)
#undef X
    return false;
}

static void slab_pool_shape(const GemmConfig &c, int &pool, int &bbytes) {
    pool = bbytes = 0;
#define X(BN_, BK_, AM_, RES_, MC_)                                  \
    if (BYOC_GEMM_MATCH(c, BN_, BK_, AM_, RES_, MC_)) {              \
        pool = GemmShape<BN_, BK_, AM_, RES_, MC_>::POOL_BYTES;      \
        bbytes = GemmShape<BN_, BK_, AM_, RES_, MC_>::B_BYTES;       \
    }
    BYOC_GEMM_CONFIGS(X)
#undef X
}

bool gemm_slab_res_fits(const GemmConfig &c, int num_kb, int slab_bytes) {
    int pool, bbytes;
    slab_pool_shape(c, pool, bbytes);
    const int pitch = (slab_bytes + 1023) / 1024 * 1024;
    return amode_wres(c.amode) && pool > 0 && num_kb * bbytes + 2 * pitch <= pool;
}

void gemm_slab_pool(const GemmConfig &c, GemmArgs &a) {
    a.slab_off = a.slab_pitch = a.slab_slots = 0;
    if (!amode_wres(c.amode)) return;
    int pool, bbytes;
    slab_pool_shape(c, pool, bbytes);
    a.slab_pitch = (a.slab_bytes + 1023) / 1024 * 1024;
    a.slab_off = a.num_kb * bbytes;
    const int slots = (pool - a.slab_off) / a.slab_pitch;
    a.slab_slots = slots > kMaxSlabSlots ? kMaxSlabSlots : slots;
}

size_t gemm_smem_bytes(const GemmConfig &c) {
#define X(BN_, BK_, AM_, RES_, MC_)                     \
    if (BYOC_GEMM_MATCH(c, BN_, BK_, AM_, RES_, MC_)) \
        return (size_t)GemmShape<BN_, BK_, AM_, RES_, MC_>::SMEM_BYTES;
    BYOC_GEMM_CONFIGS(X)
#undef X
    return 0;
}

int gemm_stages(const GemmConfig &c) {
#define X(BN_, BK_, AM_, RES_, MC_)                     \
    if (BYOC_GEMM_MATCH(c, BN_, BK_, AM_, RES_, MC_)) \
        return GemmShape<BN_, BK_, AM_, RES_, MC_>::STAGES;
    BYOC_GEMM_CONFIGS(X)
#undef X
    return 0;
}

cudaError_t gemm_prepare(const GemmConfig &c) {
#define X(BN_, BK_, AM_, RES_, MC_)                     \
    if (BYOC_GEMM_MATCH(c, BN_, BK_, AM_, RES_, MC_)) \
        return prepare_t<BN_, BK_, AM_, RES_, MC_>();
    BYOC_GEMM_CONFIGS(X)
#undef X
    return cudaErrorInvalidValue;
}

cudaError_t launch_gemm(const GemmConfig &c, const CUtensorMap &tmA, const CUtensorMap &tmB,
                        const CUtensorMap &tmR, const CUtensorMap &tmO, const GemmArgs &a, int grid,
                        cudaStream_t st) {
    if (c.mc && (grid < 2 || grid % 2)) return cudaErrorInvalidValue;  // whole clusters of two
    // cluster split-K: one cluster of `splits` CTAs per tile, every tile in the grid
    if (c.amode == kAModeTileSplitCl && (!cl_split_fits(c.bn, a.splits) || grid != a.num_tiles * a.splits))
        return cudaErrorInvalidValue;
#define X(BN_, BK_, AM_, RES_, MC_)                     \
    if (BYOC_GEMM_MATCH(c, BN_, BK_, AM_, RES_, MC_)) \
        return launch_t<BN_, BK_, AM_, RES_, MC_>(tmA, tmB, tmR, tmO, a, grid, st);
    BYOC_GEMM_CONFIGS(X)
#undef X
    return cudaErrorInvalidValue;
}

}  // namespace byoc
