"""Helpers shared by the GPU parity tests: run a region through the C ABI on
cuda:0 and compare with the fp64 oracle on the same seeded inputs.

Tolerance (bf16 inputs, fp32 accumulation; max relative error 2e-2, max
absolute error 1e-2).  The absolute bound is stated for unit-scale outputs;
the rounding floor of a bf16 result grows with the magnitude of the values it
is computed from, so the absolute term is scaled by the tensor's dynamic range:

  every element:        |gpu - ref| <= ATOL * max(1, max|ref|) + RTOL * |ref|
  every output channel: ||gpu - ref||_2 <= RTOL * ||ref||_2 + ATOL * max(1, rms(ref)) * sqrt(n)

For outputs bounded by 1 in magnitude the element test is exactly
|gpu - ref| <= 1e-2 + 2e-2 |ref|.  The channel test catches per-channel
errors (a wrong batch-norm fold, a wrong bias) that small elements could hide.
Index and layout errors are pinned separately by the bit-exact small-integer
cases.
"""
from __future__ import annotations

import numpy as np

from paper_2105_03215_gb300 import inputs as I

RTOL = 2e-2
ATOL = 1e-2


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


def assert_close(got, ref, what="", rtol=RTOL, atol=ATOL):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    diff = np.abs(got - ref)
    scale = max(1.0, float(np.max(np.abs(ref)))) if ref.size else 1.0
    bad = ~(diff <= atol * scale + rtol * np.abs(ref))
    if bad.any():
        idx = np.argwhere(bad)[:8]
        n_nan = int(np.isnan(got).sum())
        raise AssertionError(
            f"{what}: {int(bad.sum())}/{bad.size} elements out of tolerance "
            f"(nan {n_nan}); max abs {np.nanmax(diff):.4g}; first bad {idx.tolist()} "
            f"got {[float(got[tuple(i)]) for i in idx]} ref {[float(ref[tuple(i)]) for i in idx]}")
    C = ref.shape[-1] if ref.ndim else 1
    d2 = (got - ref).reshape(-1, C)
    r2 = ref.reshape(-1, C)
    err_c = np.sqrt((d2 ** 2).sum(axis=0))
    rms = max(1.0, float(np.sqrt(np.mean(ref ** 2)))) if ref.size else 1.0
    lim_c = rtol * np.sqrt((r2 ** 2).sum(axis=0)) + atol * rms * np.sqrt(d2.shape[0])
    badc = ~(err_c <= lim_c)
    if badc.any():
        ch = np.argwhere(badc).ravel()[:8]
        raise AssertionError(f"{what}: {int(badc.sum())}/{C} channels out of tolerance; first "
                             f"{ch.tolist()} err {err_c[ch].tolist()} limit {lim_c[ch].tolist()}")
    big = np.abs(ref) > 1e-2
    rel = float(np.max(diff[big] / np.abs(ref[big]))) if big.any() else 0.0
    return float(diff.max()), rel


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
