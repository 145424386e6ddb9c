/*
 * byoc_plan.h -- host-only inspection of what byoc_compile would build.
 *
 * byoc_compile (byoc.h) runs in two phases: a pure host phase that validates
 * the region, groups its ops into kernel launches (each conv2d / dense
 * absorbs the bias_add / batch_norm / add / activation that follow it -- the
 * composite of Section 3.1.1 becoming one kernel), folds batch norm in fp64,
 * and packs the bf16 weights; and a device phase that uploads them.  These
 * entry points run the host phase only, so the planning logic can be checked
 * on a machine without a GPU.  They never touch CUDA.
 */
#ifndef BYOC_PLAN_H_
#define BYOC_PLAN_H_

#include "byoc.h"

#ifdef __cplusplus
extern "C" {
#endif

/* launches of one region (a whole ResNet-50 body plans to 61) */
#define BYOC_PLAN_MAX_LAUNCHES 128

typedef enum {
    BYOC_LAUNCH_GEMM = 0,      /* tcgen05 implicit-GEMM conv2d / dense + fused epilogue */
    BYOC_LAUNCH_DEPTHWISE = 1, /* depthwise 3x3 conv + fused epilogue */
    BYOC_LAUNCH_S2D = 2,       /* layout transform of a stride-2 few-channel stem (4-channel, zero-padded pixel pairs) */
    BYOC_LAUNCH_DWPW = 3,      /* depthwise 3x3 + epilogue fused with the 1x1 conv + epilogue after it */
    BYOC_LAUNCH_CHAIN = 4,     /* region kernel: 1-4 conv2d / dense composites in one persistent launch */
    BYOC_LAUNCH_QUANT = 5      /* bf16 -> FP8 E4M3 quantization of a region input (Section 3.2 Q node) */
} byoc_launch_kind;

typedef struct {
    int32_t n_launches;
    int32_t kind[BYOC_PLAN_MAX_LAUNCHES];       /* byoc_launch_kind */
    int32_t first_op[BYOC_PLAN_MAX_LAUNCHES];   /* index of the launch's conv2d/dense op (-1: S2D) */
    int32_t n_ops[BYOC_PLAN_MAX_LAUNCHES];      /* region ops folded into the launch */
    int32_t act[BYOC_PLAN_MAX_LAUNCHES];        /* 0 none, 1 relu, 2 relu6, 3 gelu */
    int32_t residual[BYOC_PLAN_MAX_LAUNCHES];   /* tensor id added in the epilogue, or -1 */
    int32_t gemm_m[BYOC_PLAN_MAX_LAUNCHES];     /* GEMM rows (output pixels / dense rows) */
    int32_t gemm_n[BYOC_PLAN_MAX_LAUNCHES];     /* output channels */
    int32_t gemm_k[BYOC_PLAN_MAX_LAUNCHES];     /* packed reduction length */
    int32_t tile_n[BYOC_PLAN_MAX_LAUNCHES];     /* BN */
    int32_t tile_k[BYOC_PLAN_MAX_LAUNCHES];     /* BK */
    int32_t im2col[BYOC_PLAN_MAX_LAUNCHES];     /* 1 if A is read through an im2col map */
    int32_t grid[BYOC_PLAN_MAX_LAUNCHES];       /* CTAs launched */
    int32_t resident_b[BYOC_PLAN_MAX_LAUNCHES]; /* 1: the weights are loaded once per CTA (slab mode) */
    int32_t slab_slots[BYOC_PLAN_MAX_LAUNCHES]; /* slab buffers in flight (slab mode), else 0 */
    int32_t splits[BYOC_PLAN_MAX_LAUNCHES];     /* GEMM: CTAs sharing each tile's k-blocks (split-K), else 0 */
    int32_t pair_units[BYOC_PLAN_MAX_LAUNCHES]; /* 1: slab-mode units of two adjacent 128-row tiles
                                                   sharing each weight k-block, else 0 */
    int32_t stages[BYOC_PLAN_MAX_LAUNCHES];     /* region kernel: composites it runs (gemm_* fields
                                                   describe the first), else 1 */
    int32_t units[BYOC_PLAN_MAX_LAUNCHES];      /* region kernel: output tiles over all its composites */
    int32_t fp8[BYOC_PLAN_MAX_LAUNCHES];        /* region kernel: composites computed in FP8 */
    int32_t multicast[BYOC_PLAN_MAX_LAUNCHES];  /* GEMM: 1 if clusters of two CTAs share each
                                                   weight tile by TMA multicast (grid even) */
    double flops;
    double bytes;
    size_t const_bytes;
    size_t workspace_bytes;
} byoc_plan_report;

/* Plan a region for a device with `num_sms` SMs without touching the GPU.
 * Same validation and errors as byoc_compile. */
byoc_status byoc_plan(const byoc_region_desc *desc, int32_t num_sms, byoc_plan_report *rep);

/* Copy the packed constants of launch `launch` of that plan into dst:
 *   what = 0: weights.  GEMM: bf16 [n_pad][gemm_k], row n = output channel,
 *             column k = (filter tap, channel) K-major, zero padded;
 *             depthwise: fp32 [9][C] tap-major.
 *   what = 1: bias (fp32, folded batch norm shift), zero padded.
 *   what = 2, 3 (fused depthwise -> 1x1 launches only): the 1x1 conv's
 *             weights, bf16 [n_pad][64 * ceil(C / 64)] K-major, and bias.
 * *needed receives the byte size; dst may be NULL to query it. */
byoc_status byoc_plan_constants(const byoc_region_desc *desc, int32_t num_sms, int32_t launch,
                                int32_t what, void *dst, size_t dst_bytes, size_t *needed);

/* The host halves of byoc_serialize / byoc_deserialize, for tests without a
 * GPU: plan the region for `num_sms` SMs and serialise the plan (dst NULL:
 * size query), or parse serialised bytes and report the plan they hold.
 * Same formats and errors as byoc_serialize / byoc_deserialize. */
byoc_status byoc_plan_serialize(const byoc_region_desc *desc, int32_t num_sms, void *dst,
                                size_t dst_bytes, size_t *needed);
byoc_status byoc_plan_deserialize(const void *src, size_t src_bytes, byoc_plan_report *rep);

#ifdef __cplusplus
}
#endif

#endif /* BYOC_PLAN_H_ */
