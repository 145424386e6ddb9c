// chain.cu -- one persistent kernel for a whole region whose composites form
// a chain of convolutions / dense layers.  Section 3.1.2 merges consecutive
// supported operators into one region so that the accelerator saves the data
// movement and the kernel launches between them, and Section 3.4 keeps a
// region's intermediates out of the runtime's data entries.  The ResNet-50 bottleneck (1x1 -> 3x3 -> 1x1 +
// residual, optionally with its downsample 1x1) and the BERT FFN (dense +
// GELU -> dense) each run as one launch: the intermediates t1 / t2 / H are
// written once to the region's workspace and read back while still in L2,
// and a stage's tiles start as soon as the tiles they read are done, instead
// of after the whole previous launch.
//
// Work is cut into units: one 128-row x BN-column output tile of one stage.
// The host schedules the units on the grid's CTAs (a list schedule with
// estimated durations), so that the stages interleave across the machine like
// a pipeline instead of running one after the other; each CTA runs its list
// in that global order.  A unit only ever depends on units earlier in the
// global order, and every CTA is resident (one per SM, grid <= SMs), so every
// wait ends (and every wait is bounded anyway).  A
// unit's dependencies -- the 128-row m-tiles of earlier stages that its A
// operand (and its residual) reads -- are listed on the host
// (ChainArgs::dep_*).  Each m-tile of a stage that later stages read has a
// completion counter; each of a unit's 8 epilogue warps adds 1 to it once
// its stores have completed, so a consumer waits for 8 x (column tiles) x
// (run + 1), where run counts this region's completed launches.
//
// Roles (one CTA of 352 threads per SM, as in gemm.cu):
//   warp 0     TMA producer: per k-block A (a 128 x 64 tile, or an im2col
//              box for a k x k convolution) and B;
//   warp 1     TMEM allocation and the tcgen05.mma issuer (M=128, N=BN, K=16,
//              two fp32 accumulators);
//   warps 2-9  epilogue: + bias and + residual (global loads, one 32-column
//              chunk ahead), activation, bf16, TMA store of 32 x 32 pieces,
//              then the m-tile's completion counter;
//   warp 10    scheduler: walks the CTA's unit list (one elected lane),
//              waits for each unit's dependencies and publishes it to the CTA
//              through a 4-slot ring in shared memory.
#include "internal.h"
#include "ptx.cuh"

namespace byoc {

template <int BN>
struct ChainShape {
    static constexpr int BM = kGemmBM;
    static constexpr int BK = 64;
    static constexpr int ROW_BYTES = 128;
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = BN * BK * 2;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int NCH = BN / 32;
    static constexpr int EPI_TILE = 32 * 32 * 2;
    static constexpr int CTRL_BYTES = 1024;
    static constexpr int FIXED1 = 1024 + CTRL_BYTES;
    // a second staging tile per epilogue warp where the ring keeps 4 stages with it
    static constexpr int EPI_BUFS =
        (232448 - FIXED1 - 2 * kGemmEpiWarps * EPI_TILE) / STAGE_BYTES >= 4 ? 2 : 1;
    static constexpr int EPI_BYTES = kGemmEpiWarps * EPI_TILE * EPI_BUFS;
    static constexpr int FIXED = FIXED1 + EPI_BYTES;
    static constexpr int STAGES_RAW = (232448 - FIXED) / STAGE_BYTES;
    static constexpr int STAGES = STAGES_RAW > 16 ? 16 : STAGES_RAW;
    static constexpr int SMEM_BYTES = FIXED + STAGES * STAGE_BYTES;
    static constexpr int USLOTS = 4;  // unit broadcast ring
    static constexpr int NUM_BARS = 2 * STAGES + 4 + 2 * USLOTS + 1;
    static constexpr int TMEM_COLS = 2 * BN;
    static_assert(8 * NUM_BARS + 16 + 8 * USLOTS <= CTRL_BYTES && USLOTS <= 4, "control block");
    static_assert(STAGES >= 2, "ring depth");
    static_assert(SMEM_BYTES <= 232448, "shared memory budget");
    static_assert(BN == 128 || BN == 256, "BN");
};

template <bool B>
struct BoolTag {
    static constexpr bool value = B;
};

// readers of a unit broadcast slot: the producer lane, the MMA lane, 8
// epilogue warps
constexpr uint32_t kChainUnitReaders = 1 + kGemmEpiWarps + 1;

__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned *p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Polling load: relaxed, so a poll does not pay for an acquire each time; a
// single fence_acquire_gpu after the last poll orders what follows after
// every release the polls observed (measured on GB300: an ld.acquire.gpu per
// poll costs ~0.5 us on an SM with TMA traffic in flight, so a unit with 24
// dependencies saw them ~12 us late).
__device__ __forceinline__ unsigned ld_relaxed_gpu(const unsigned *p) {
    unsigned v;
    asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void fence_acquire_gpu() { asm volatile("fence.acq_rel.gpu;" ::: "memory"); }

__device__ __forceinline__ void red_release_gpu_add(unsigned *p, unsigned v) {
    asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Order this thread's async-proxy global accesses (TMA) with its generic ones.
__device__ __forceinline__ void fence_proxy_async_global() {
    asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ uint4 ld_cg_v4(const void *p) {
    uint4 r;
    asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
    return r;
}

// Wait until every dependency counter of unit u has reached its count for
// this launch (count per launch x (run + 1), modulo 2^32), polling them all
// together with relaxed loads; bounded like mbar_wait.  The caller issues
// fence_acquire_gpu afterwards.
__device__ __forceinline__ bool wait_deps(const ChainArgs &a, int u, unsigned run, volatile int *abort_flag) {
    const int j0 = a.dep_off[u], j1 = a.dep_off[u + 1];
    unsigned long long t0 = 0;
    for (uint32_t it = 0;; ++it) {
        bool all = true;
        for (int j = j0; j < j1; ++j) {
            const unsigned target = (unsigned)a.dep_list[2 * j + 1] * (run + 1u);
            if ((int)(ld_relaxed_gpu(a.flags + a.dep_list[2 * j]) - target) < 0) all = false;
        }
        if (all) return true;
        if (it == 0) t0 = globaltimer_ns();
        __nanosleep(64);
        if ((it & 15u) == 15u) {
            if (*abort_flag) return false;
            if (globaltimer_ns() - t0 > kWaitLimitNs) {
                *abort_flag = 1;
                if (a.err) atomicCAS(a.err, 0, kErrTimeoutDependency);
                return false;
            }
        }
    }
}

template <int BN>
__global__ void __maxnreg__(168)
    chain_tcgen05_kernel(const __grid_constant__ ChainMaps maps, const ChainArgs a) {
    using S = ChainShape<BN>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *smem = smem_raw + (base - raw);
    const uint32_t sA = base;
    const uint32_t sB = sA + S::STAGES * S::A_BYTES;
    const uint32_t sEpi = sB + S::STAGES * S::B_BYTES;
    const uint32_t ctrl = sEpi + S::EPI_BYTES;
    const uint32_t bars = ctrl;                          // full[S], empty[S]
    const uint32_t tfull = bars + 8u * (2 * S::STAGES);  // 2
    const uint32_t tempty = tfull + 16u;                 // 2
    const uint32_t ufull = tempty + 16u;                 // USLOTS
    const uint32_t uempty = ufull + 8u * S::USLOTS;      // USLOTS
    const uint32_t drain = uempty + 8u * S::USLOTS;
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(smem + (ctrl - base) + 8 * S::NUM_BARS);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
    volatile int *unit_ids = reinterpret_cast<volatile int *>(tmem_slot + 4);    // USLOTS
    volatile int *unit_codes = reinterpret_cast<volatile int *>(tmem_slot + 8);  // USLOTS: order[u]

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S::STAGES; ++s) {
            mbar_init(bars + 8u * s, 1);
            mbar_init(bars + 8u * (S::STAGES + s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(tfull + 8u * b, 1);
            mbar_init(tempty + 8u * b, kGemmEpiWarps);
        }
        for (int b = 0; b < S::USLOTS; ++b) {
            mbar_init(ufull + 8u * b, 1);
            mbar_init(uempty + 8u * b, kChainUnitReaders);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        for (int s = 0; s < a.n_stages; ++s) {
            tma_prefetch_desc(&maps.A[s]);
            tma_prefetch_desc(&maps.B[s]);
            tma_prefetch_desc(&maps.O[s]);
        }
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), S::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    pdl_launch_dependents();
    pdl_wait();
    if (a.trace != nullptr && threadIdx.x == 32) atomicMin(a.trace, globaltimer_ns());

    // Wait for a unit broadcast slot t and read its unit id (-1: no more
    // units) and code (stage << 24 | tile); every reader arrives on the
    // slot's empty barrier once.
    auto read_unit = [&](int t, int err_code, bool &ok, int &ucode) -> int {
        const int slot = t % S::USLOTS;
        ok = mbar_wait(ufull + 8u * slot, (uint32_t)(t / S::USLOTS) & 1u, abort_flag, a.err, err_code);
        if (!ok) return -1;
        ucode = unit_codes[slot];
        return unit_ids[slot];
    };

    if (warp == 0) {
        // ------------------------------------------------------ scheduler + producer
        if (elect_one()) {
            auto wait = [&](uint32_t bar, uint32_t parity) -> bool {
                return mbar_wait(bar, parity, abort_flag, a.err, kErrTimeoutProducer);
            };
            int stage = 0, issued = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int t = 0; ok; ++t) {
                int code = 0;
                const int u = read_unit(t, kErrTimeoutProducer, ok, code);
                if (ok) mbar_arrive(uempty + 8u * (t % S::USLOTS));
                if (u < 0) break;
                const int si = code >> 24;
                const ChainStage &cs = a.st[si];
                const int tile = code & 0xFFFFFF;
                const int m0 = (tile / cs.tiles_n) * S::BM;
                const int n0 = (tile % cs.tiles_n) * BN;
                int img = 0, h0 = 0, w0 = 0;
                if (cs.mode == kChainIm2col) {
                    const int hw = cs.Ho * cs.Wo;
                    img = m0 / hw;
                    const int rem = m0 - img * hw;
                    const int p = rem / cs.Wo;
                    const int q = rem - p * cs.Wo;
                    h0 = p * cs.stride_h - cs.pad_t;
                    w0 = q * cs.stride_w - cs.pad_l;
                }
                int cc = 0, r = 0, sx = 0;
                const int kel = cs.fp8 ? 2 * S::BK : S::BK;  // elements per 128-byte k-block
                for (int kb = 0; kb < cs.num_kb; ++kb) {
                    if (!wait(bars + 8u * (S::STAGES + stage), phase ^ 1u)) {
                        ok = false;
                        break;
                    }
                    const uint32_t full = bars + 8u * stage;
                    mbar_arrive_expect_tx(full, (uint32_t)S::STAGE_BYTES);
                    const uint32_t dA = sA + stage * S::A_BYTES;
                    if (cs.mode == kChainIm2col) {
                        tma_load_im2col_4d(dA, &maps.A[si], full, cc * kel, w0, h0, img,
                                           (uint16_t)(sx * cs.dil_w), (uint16_t)(r * cs.dil_h));
                        if (++cc == cs.chunks) {
                            cc = 0;
                            if (++sx == cs.kw) {
                                sx = 0;
                                ++r;
                            }
                        }
                    } else {
                        tma_load_2d(dA, &maps.A[si], full, kb * kel, m0);
                    }
                    tma_load_2d(sB + stage * S::B_BYTES, &maps.B[si], full, kb * kel, n0);
                    ++issued;
                    if (++stage == S::STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok) {
                // Gave up: let the copies already issued land before exiting.
                for (int j = issued - S::STAGES > 0 ? issued - S::STAGES : 0; j < issued; ++j)
                    mbar_wait_drain(bars + 8u * (j % S::STAGES), (uint32_t)(j / S::STAGES) & 1u);
            }
        }
        __syncwarp();
    } else if (warp == kGemmOperandWarp) {
        // ------------------------------------------------------ scheduler
        // Takes units from the counter, waits until the rows each one reads
        // are complete and acquired, and only then publishes it to the CTA.
        // The acquire happens here, on a thread with no copies of its own in
        // flight: on the producer thread the fence also waited for the
        // previous unit's TMA loads (measured: ~2 us per unit).  The producer's
        // loads, the MMAs and the epilogue's residual reads all come after
        // the publication (mbarrier release / acquire), so after the acquire.
        if (elect_one()) {
            const unsigned run = ld_acquire_gpu(a.ctl + 2);
            // This CTA's unit records are read one ahead (the record after
            // the current unit loads while the current one is handled), and
            // a unit's dependency counters are polled (loads issued) as soon
            // as the unit before it is published, so that neither latency
            // adds to every unit.  Record: {u, code, n, dep_off[u]},
            // {counter, count} x kChainRecDeps.
            static_assert(kChainRecInts == 12 && kChainRecDeps == 4, "record layout");
            const int r0 = a.cta_off[blockIdx.x], r1 = a.cta_off[blockIdx.x + 1];
            const int4 *recs = reinterpret_cast<const int4 *>(a.cta_rec);
            int4 cur[3], nxt[3];
            auto load_rec = [&](int k, int4 (&r)[3]) {
                if (r0 + k < r1) {
#pragma unroll
                    for (int q = 0; q < 3; ++q) r[q] = __ldg(recs + (size_t)(r0 + k) * 3 + q);
                } else {
                    r[0] = make_int4(-1, 0, 0, 0);
                    r[1] = r[2] = make_int4(0, 0, 0, 0);
                }
            };
            unsigned pv[kChainRecDeps];
            auto issue_polls = [&](const int4 (&r)[3]) {
                const int n = r[0].z;
                if (r[0].x < 0 || n <= 0) return;
                pv[0] = ld_relaxed_gpu(a.flags + r[1].x);
                if (n > 1) pv[1] = ld_relaxed_gpu(a.flags + r[1].z);
                if (n > 2) pv[2] = ld_relaxed_gpu(a.flags + r[2].x);
                if (n > 3) pv[3] = ld_relaxed_gpu(a.flags + r[2].z);
            };
            // every polled counter has reached its count for this launch
            // (units with more dependencies than a record holds: wait_deps)
            auto polled_ready = [&](const int4 (&r)[3]) -> bool {
                const int n = r[0].z;
                if (n > kChainRecDeps) return false;
                const unsigned k1 = run + 1u;
                bool ready = (int)(pv[0] - (unsigned)r[1].y * k1) >= 0;
                if (n > 1) ready = ready && (int)(pv[1] - (unsigned)r[1].w * k1) >= 0;
                if (n > 2) ready = ready && (int)(pv[2] - (unsigned)r[2].y * k1) >= 0;
                if (n > 3) ready = ready && (int)(pv[3] - (unsigned)r[2].w * k1) >= 0;
                return ready;
            };
            load_rec(0, cur);
            load_rec(1, nxt);
            issue_polls(cur);
            int t = 0;
            bool ok = true;
            for (;; ++t) {
                const int slot = t % S::USLOTS;
                if (!mbar_wait(uempty + 8u * slot, ((uint32_t)(t / S::USLOTS) & 1u) ^ 1u, abort_flag, a.err,
                               kErrTimeoutProducer)) {
                    ok = false;
                    break;
                }
                const int u = cur[0].x;
                if (u >= 0 && cur[0].z > 0) {
                    if (!polled_ready(cur) && !wait_deps(a, u, run, abort_flag)) {
                        ok = false;
                        break;
                    }
                    fence_acquire_gpu();
                    fence_proxy_async_global();
                }
                unit_ids[slot] = u;
                unit_codes[slot] = cur[0].y;
                mbar_arrive(ufull + 8u * slot);
                if (u < 0) break;
#pragma unroll
                for (int q = 0; q < 3; ++q) cur[q] = nxt[q];
                issue_polls(cur);
                load_rec(t + 2, nxt);
            }
            (void)ok;
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------ MMA issuer
        if (elect_one()) {
            auto wait = [&](uint32_t bar, uint32_t parity) -> bool {
                return mbar_wait(bar, parity, abort_flag, a.err, kErrTimeoutMma);
            };
            constexpr uint32_t idesc16 = make_idesc_bf16(S::BM, BN);
            constexpr uint32_t idesc8 = make_idesc_e4m3(S::BM, BN);
            const uint64_t adesc0 = make_smem_desc(sA, S::ROW_BYTES);
            const uint64_t bdesc0 = make_smem_desc(sB, S::ROW_BYTES);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int t = 0; ok; ++t) {
                int code = 0;
                const int u = read_unit(t, kErrTimeoutMma, ok, code);
                if (ok) mbar_arrive(uempty + 8u * (t % S::USLOTS));
                if (u < 0) break;
                const ChainStage &cs = a.st[code >> 24];
                const int buf = t & 1;
                if (!wait(tempty + 8u * buf, (((uint32_t)(t >> 1)) & 1u) ^ 1u)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
                const bool f8 = cs.fp8 != 0;
                uint32_t acc = 0u;
                for (int kb = 0; kb < cs.num_kb; ++kb) {
                    if (!wait(bars + 8u * stage, phase)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t ad = adesc0 + (uint64_t)((stage * S::A_BYTES) >> 4);
                    const uint64_t bd = bdesc0 + (uint64_t)((stage * S::B_BYTES) >> 4);
                    // four MMAs per 128-byte k-block: K = 16 bf16 or K = 32 E4M3
                    // values, 32 bytes each either way
                    if (f8) {
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            mma_f8_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc8, acc | (uint32_t)k);
                    } else {
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            mma_bf16_ss(d_tmem, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), idesc16,
                                        acc | (uint32_t)k);
                    }
                    acc = 1u;
                    mma_commit(bars + 8u * (S::STAGES + stage));  // frees the stage
                    if (++stage == S::STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                mma_commit(tfull + 8u * buf);
            }
            mma_commit(drain);
            mbar_wait_drain(drain, 0);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------ epilogue
        const int e = warp - 2;          // 0..7
        const int quarter = warp & 3;    // TMEM lane quarter = rows of the tile
        const int grp = e >> 2;          // chunks ci with ci % 2 == grp
        const uint32_t stg0 = sEpi + (uint32_t)(e * S::EPI_BUFS) * S::EPI_TILE;
        int sb = 0;
        const uint32_t sw_own = ((uint32_t)lane >> 1) & 3u;
        for (int t = 0;; ++t) {
            bool ok;
            int code = 0;
            int u = read_unit(t, kErrTimeoutEpilogue, ok, code);
            __syncwarp();
            if (ok && lane == 0) mbar_arrive(uempty + 8u * (t % S::USLOTS));
            if (u < 0) break;
            const int si = code >> 24;
            const ChainStage &cs = a.st[si];
            const int tile = code & 0xFFFFFF;
            const int m0 = (tile / cs.tiles_n) * S::BM;
            const int n0 = (tile % cs.tiles_n) * BN;
            const int buf = t & 1;
            const int nch = min(S::NCH, (cs.N - n0 + 31) >> 5);
            const bool has_res = cs.residual != nullptr;
            // The residual of this warp's 32 rows x 32 columns of its next
            // chunk is loaded one chunk ahead, the first before the
            // accumulator is ready (a residual written by earlier stages was
            // acquired before the unit was published): coalesced, lane l
            // reading 16-byte piece l % 4 of row 8k + l / 4, so that each load
            // instruction covers eight 64-byte row segments rather than 32
            // (measured: one row per lane left ~1.7 us of latency on a
            // chunk); the chunk's staging tile turns it into one row per lane.
            const int rrow = lane >> 2, rpiece = lane & 3;
            uint4 rn[4];
            auto load_res = [&](int ci) {
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const int rw = m0 + quarter * 32 + 8 * k + rrow;
                    rn[k] = rw < cs.M ? ld_cg_v4(cs.residual + (size_t)rw * cs.N + (n0 + ci * 32 + rpiece * 8))
                                      : make_uint4(0u, 0u, 0u, 0u);
                }
            };
            if (has_res && grp < nch) load_res(grp);
            // this warp's chunks' bias (and FP8 dequantization scales), one
            // column per lane, loaded before the accumulator is ready; lane j
            // hands column j to the others by shuffle (both arrays are zero
            // padded to tiles_n x BN)
            constexpr int KC = S::NCH / 2;  // chunks per warp
            float bl[KC], dl[KC];
#pragma unroll
            for (int k = 0; k < KC; ++k) {
                const int c = n0 + (grp + 2 * k) * 32 + lane;
                bl[k] = __ldg(cs.bias + c);
                dl[k] = cs.fp8 ? __ldg(cs.dq + c) : 0.0f;
            }
            if (!mbar_wait(tfull + 8u * buf, ((uint32_t)(t >> 1)) & 1u, abort_flag, a.err, kErrTimeoutEpilogue))
                break;
            tc_fence_after();
            const uint32_t tbase = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(buf * BN);
            if (grp >= nch) {  // nothing of this unit for this warp
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(tempty + 8u * buf);
            }
            // the chunks, compiled once with and once without the residual
            // (one copy for both measured ~1 us slower on the BERT FFN's GELU stage)
            auto chunks = [&](auto res_tag) {
                constexpr bool RESID = decltype(res_tag)::value;
#pragma unroll
                for (int k = 0; k < KC; ++k) {
                    const int ci = grp + 2 * k;
                    if (ci >= nch) break;
                    const int col0 = n0 + ci * 32;
                    uint4 rc[4];  // this chunk's residual pieces (coalesced layout)
#pragma unroll
                    for (int q = 0; q < 4; ++q) rc[q] = rn[q];
                    if (RESID && ci + 2 < nch) load_res(ci + 2);
                    uint32_t v[32];
                    tmem_ld_32cols(tbase + (uint32_t)(ci * 32), v);
                    if (ci + 2 >= nch) {  // this warp's last read of the accumulator
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(tempty + 8u * buf);
                    }
                    float f[32];
                    if (cs.fp8) {
                        // FP8: the accumulator is in units of S_x S_w[n]
#pragma unroll
                        for (int j = 0; j < 32; ++j)
                            f[j] = fmaf(__uint_as_float(v[j]), __shfl_sync(0xffffffffu, dl[k], j),
                                        __shfl_sync(0xffffffffu, bl[k], j));
                    } else {
#pragma unroll
                        for (int j = 0; j < 32; ++j) f[j] = __uint_as_float(v[j]) + __shfl_sync(0xffffffffu, bl[k], j);
                    }
                    const uint32_t stg = stg0 + (uint32_t)(sb * S::EPI_TILE);
                    if constexpr (RESID) {
                        // the store that last used this staging tile has read it
                        if (lane == 0) bulk_wait_group_read<S::EPI_BUFS - 1>();
                        __syncwarp();
                        // residual pieces -> staging tile (64-byte swizzle, as the
                        // output below) -> this lane's row
#pragma unroll
                        for (int p = 0; p < 4; ++p) {
                            const uint32_t r = (uint32_t)(8 * p + rrow);
                            const uint32_t addr = stg + r * 64u + ((((uint32_t)rpiece) ^ ((r >> 1) & 3u)) << 4);
                            asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(rc[p].x),
                                         "r"(rc[p].y), "r"(rc[p].z), "r"(rc[p].w)
                                         : "memory");
                        }
                        __syncwarp();
                        uint4 rr[4];
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                         : "=r"(rr[q].x), "=r"(rr[q].y), "=r"(rr[q].z), "=r"(rr[q].w)
                                         : "r"(stg + (uint32_t)lane * 64u + ((((uint32_t)q) ^ sw_own) << 4))
                                         : "memory");
                        __syncwarp();  // every row read before the output overwrites the tile
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const uint32_t w4[4] = {rr[q].x, rr[q].y, rr[q].z, rr[q].w};
#pragma unroll
                            for (int e2 = 0; e2 < 4; ++e2) {
                                f[8 * q + 2 * e2] += bf16lo(w4[e2]);
                                f[8 * q + 2 * e2 + 1] += bf16hi(w4[e2]);
                            }
                        }
                    }
                    if (cs.act == kActGelu) {
#pragma unroll
                        for (int j = 0; j < 16; ++j) {
                            const uint64_t g = gelu2(f32x2(f[2 * j], f[2 * j + 1]));
                            f[2 * j] = lane0(g);
                            f[2 * j + 1] = lane1(g);
                        }
                    } else if (cs.act == kActRelu) {
#pragma unroll
                        for (int j = 0; j < 32; ++j) f[j] = fmaxf(f[j], 0.0f);
                    } else if (cs.act == kActRelu6) {
#pragma unroll
                        for (int j = 0; j < 32; ++j) f[j] = fminf(fmaxf(f[j], 0.0f), 6.0f);
                    }
                    if constexpr (!RESID) {  // (with a residual: waited for above)
                        if (lane == 0) bulk_wait_group_read<S::EPI_BUFS - 1>();
                        __syncwarp();
                    }
                    if (cs.out8) {
                        // a fused Q node: E4M3 codes of f x fp32(1/S), 32 bytes per
                        // row, rows 32 bytes apart (the unswizzled box of the map)
#pragma unroll
                        for (int h = 0; h < 2; ++h) {
                            uint32_t w[4];
#pragma unroll
                            for (int k = 0; k < 4; ++k) {
                                const float *g = f + 16 * h + 4 * k;
                                w[k] = cvt_e4m3x2(g[0] * cs.out_inv, g[1] * cs.out_inv) |
                                       (cvt_e4m3x2(g[2] * cs.out_inv, g[3] * cs.out_inv) << 16);
                            }
                            const uint32_t addr = stg + (uint32_t)lane * 32u + (uint32_t)h * 16u;
                            asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(w[0]), "r"(w[1]),
                                         "r"(w[2]), "r"(w[3])
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
                            asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(w0), "r"(w1),
                                         "r"(w2), "r"(w3)
                                         : "memory");
                        }
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_2d(&maps.O[si], stg, col0, m0 + quarter * 32);
                        bulk_commit_group();
                    }
                    if (S::EPI_BUFS == 2) sb ^= 1;
                }
            };
            if (has_res)
                chunks(BoolTag<true>{});
            else
                chunks(BoolTag<false>{});
            __syncwarp();
            if (cs.consumed) {
                // the unit's rows are read by later stages: count this warp's
                // part in once its stores are complete and visible
                if (lane == 0) {
                    bulk_wait_group<0>();
                    fence_proxy_async_global();
                    red_release_gpu_add(a.flags + cs.cbase + m0 / S::BM, 1u);
                }
                __syncwarp();
            }
        }
        if (lane == 0) bulk_wait_group<0>();
        __syncwarp();
    }

    __syncwarp();
    tc_fence_before();
    __syncthreads();
    if (a.trace != nullptr && threadIdx.x == 0) atomicMax(a.trace + 1, globaltimer_ns());
    if (threadIdx.x == 0) {
        // the last CTA to finish counts this launch in (every CTA read the
        // run count at its start)
        __threadfence();
        const unsigned done = atomicAdd(a.ctl + 1, 1u);
        if (done == gridDim.x - 1) {
            a.ctl[1] = 0u;
            __threadfence();
            atomicAdd(a.ctl + 2, 1u);
        }
    }
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem_base, S::TMEM_COLS);
    }
}

size_t chain_smem_bytes(int bn) {
    return bn == 256 ? (size_t)ChainShape<256>::SMEM_BYTES : (size_t)ChainShape<128>::SMEM_BYTES;
}

int chain_stages(int bn) { return bn == 256 ? ChainShape<256>::STAGES : ChainShape<128>::STAGES; }

cudaError_t chain_prepare(int bn) {
    if (bn == 256)
        return cudaFuncSetAttribute(chain_tcgen05_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    ChainShape<256>::SMEM_BYTES);
    if (bn == 128)
        return cudaFuncSetAttribute(chain_tcgen05_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    ChainShape<128>::SMEM_BYTES);
    return cudaErrorInvalidValue;
}

cudaError_t launch_chain(int bn, const ChainMaps &maps, const ChainArgs &a, int grid, cudaStream_t st) {
    if (bn == 256)
        return launch_pdl(chain_tcgen05_kernel<256>, dim3(grid), dim3(kGemmThreads),
                          (size_t)ChainShape<256>::SMEM_BYTES, st, maps, a);
    if (bn == 128)
        return launch_pdl(chain_tcgen05_kernel<128>, dim3(grid), dim3(kGemmThreads),
                          (size_t)ChainShape<128>::SMEM_BYTES, st, maps, a);
    return cudaErrorInvalidValue;
}

}  // namespace byoc
