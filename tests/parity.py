"""Helpers shared by the GPU parity tests: run a region through the C ABI on
cuda:0 and compare with the fp64 oracle on the same seeded inputs.

Tolerance (bf16 inputs, fp32 accumulation; max relative error 2e-2, max
absolute error 1e-2).  Those two terms are the stated bar; on top of them
every element may differ by what bf16 storage itself costs at that element:

  every element:        |gpu - ref| <= ATOL + RTOL |ref| + LAM * s
  every output channel: ||gpu - ref||_2 <= RTOL ||ref||_2 + ATOL sqrt(n) + 3 ||s||_2

s is the oracle's per-element error scale (oracle.graph.
evaluate_with_error_scale): under the probabilistic model of rounding-error
analysis (independent roundings with mean-zero relative errors, Hoeffding's
inequality) an implementation that rounds weights and stored activations to
bf16 and accumulates in fp32 misses the exact value by more than LAM * s with
probability at most 2 exp(-LAM^2 / 2) = 2.5e-14 per element.  A CPU emulation
of that arithmetic stays within 4 s on every workload here (tests/
test_oracle_pins.py).  s is small where the values an output is computed from
are small, so small outputs are checked at their own scale.  Systematic
errors of one channel (a wrong batch-norm fold or bias) add up linearly over
the channel's elements while rounding errors add in quadrature, which the
channel test catches.  Index and layout errors are pinned separately by the
bit-exact small-integer cases.
"""
from __future__ import annotations

import numpy as np

from oracle import graph as ograph
from oracle import ops as oops
from paper_2105_03215_gb300 import inputs as I

RTOL = 2e-2
ATOL = 1e-2
LAM = 8.0


def oracle(graph, inputs, nodes=None, keep=None):
    """(values, error scales) of the oracle for ``nodes`` of ``graph``."""
    return ograph.evaluate_with_error_scale(graph, inputs, nodes=nodes, keep=keep)


def sampled_conv_scale(x, w, pix, ks, attrs, out_scale, value):
    """Error scale of a single conv2d composite at sampled (output pixel,
    channel) pairs: the weight rounding and fp32 sum of the conv
    (oracle.graph._spread_node), times the per-channel factor ``out_scale``
    of a batch norm that follows (1 without one), plus the bf16 rounding of
    the stored ``value``."""
    x = np.asarray(x, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    a = attrs
    K = w.shape[1] * w.shape[2] * w.shape[3]
    f = lambda t, ww: oops.conv2d_nhwc_sampled(t, ww, pix, ks, a["strides"], a["padding"],
                                              a["dilation"], a["groups"])
    acc = np.sqrt(K) * ograph.U_FP32 * f(np.abs(x), np.abs(w))
    sq = ograph.U_BF16 ** 2 * f(x * x, w * w) + acc * acc
    return np.sqrt(sq * np.asarray(out_scale, np.float64) ** 2 + (ograph.U_BF16 * np.asarray(value)) ** 2)


def to_dev(a):
    import torch
    # the values are bf16-exact already; the conversion is exact
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16).cuda()


def run_region(region, inputs, poison=True, compiled=None):
    """Compile (unless ``compiled`` is given) and run ``region`` once; returns
    ({output name: float32 array}, the compiled region)."""
    import torch
    cr = compiled if compiled is not None else region.compile()
    try:
        ins = [to_dev(inputs[n]) for n in region.inputs]
        outs = []
        for n in region.outputs:
            t = torch.empty(region.graph.shape_of(n), dtype=torch.bfloat16, device="cuda")
            if poison:
                t.fill_(float("nan"))
            outs.append(t)
        cr.run(ins, outs)
        torch.cuda.synchronize()
        cr.check()
        return {n: o.float().cpu().numpy() for n, o in zip(region.outputs, outs)}, cr
    except Exception:
        cr.release()
        raise


def assert_close(got, ref, scale, what="", rtol=RTOL, atol=ATOL, lam=LAM):
    """Element and channel tests above; ``scale`` is the oracle's error scale
    (same shape as ``ref``).  Returns (max abs error, max relative error over
    |ref| > 1e-2, fraction of elements within atol + rtol |ref| alone)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    scale = np.broadcast_to(np.asarray(scale, dtype=np.float64), ref.shape)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    diff = np.abs(got - ref)
    bad = ~(diff <= atol + rtol * np.abs(ref) + lam * scale)
    if bad.any():
        idx = np.argwhere(bad)[:8]
        n_nan = int(np.isnan(got).sum())
        raise AssertionError(
            f"{what}: {int(bad.sum())}/{bad.size} elements out of tolerance "
            f"(nan {n_nan}); max abs {np.nanmax(diff):.4g}; first bad {idx.tolist()} "
            f"got {[float(got[tuple(i)]) for i in idx]} ref {[float(ref[tuple(i)]) for i in idx]} "
            f"scale {[float(scale[tuple(i)]) for i in idx]}")
    C = ref.shape[-1] if ref.ndim else 1
    d2 = (got - ref).reshape(-1, C)
    r2 = ref.reshape(-1, C)
    s2 = scale.reshape(-1, C)
    err_c = np.sqrt((d2 ** 2).sum(axis=0))
    lim_c = (rtol * np.sqrt((r2 ** 2).sum(axis=0)) + atol * np.sqrt(d2.shape[0])
             + 3.0 * np.sqrt((s2 ** 2).sum(axis=0)))
    badc = ~(err_c <= lim_c)
    if badc.any():
        ch = np.argwhere(badc).ravel()[:8]
        raise AssertionError(f"{what}: {int(badc.sum())}/{C} channels out of tolerance; first "
                             f"{ch.tolist()} err {err_c[ch].tolist()} limit {lim_c[ch].tolist()}")
    big = np.abs(ref) > 1e-2
    rel = float(np.max(diff[big] / np.abs(ref[big]))) if big.any() else 0.0
    literal = float(np.mean(diff <= atol + rtol * np.abs(ref))) if ref.size else 1.0
    return float(diff.max()) if diff.size else 0.0, rel, literal


def assert_bit_exact(got, ref, what=""):
    """GPU bf16 output == bf16 rounding (RNE) of the exact oracle value."""
    g = I.bf16_bits(np.asarray(got, dtype=np.float32))
    r = I.bf16_bits(np.asarray(ref, dtype=np.float64).astype(np.float32))
    neq = g != r
    if neq.any():
        idx = np.argwhere(neq)[:8]
        raise AssertionError(f"{what}: {int(neq.sum())}/{neq.size} bf16 mismatches; first {idx.tolist()} "
                             f"got {[float(np.asarray(got)[tuple(i)]) for i in idx]} "
                             f"ref {[float(np.asarray(ref)[tuple(i)]) for i in idx]}")
