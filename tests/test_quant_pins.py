"""Pins of the partial-quantization oracle (oracle/quant.py; Section 3.2):
the E4M3 codebook and its rounding, checked from the format's definition and
against torch's float8_e4m3fn cast (a library routine), the 8-bit integer Q/DQ
with zero point, the per-channel power-of-two weight scales, and the FP8
layers of oracle/graph.py against an independent computation."""
import numpy as np
import pytest

from oracle import graph as ograph
from oracle import quant as Q
from paper_2105_03215_gb300 import inputs as I


def test_e4m3_codebook_from_the_format():
    v = Q.e4m3_values()
    assert len(v) == 127                      # codes 0x00 .. 0x7E
    assert v[0] == 0.0 and v[1] == 2.0 ** -9 and v[8] == 2.0 ** -6 and v[-1] == 448.0
    assert np.all(np.diff(v) > 0)
    # every value is its own rounding, and so is its negative
    assert np.array_equal(Q.round_e4m3(v), v)
    assert np.array_equal(Q.round_e4m3(-v), -v)


def test_e4m3_ties_go_to_the_even_code():
    v = Q.e4m3_values()
    mid = (v[:-1] + v[1:]) / 2                 # exact in fp64
    want = np.where(np.arange(len(mid)) % 2 == 0, v[:-1], v[1:])  # code i even -> v[i]
    assert np.array_equal(Q.round_e4m3(mid), want)
    # just off the midpoint goes to the nearer value
    eps = (v[1:] - v[:-1]) * 1e-6
    assert np.array_equal(Q.round_e4m3(mid - eps), v[:-1])
    assert np.array_equal(Q.round_e4m3(mid + eps), v[1:])


def test_e4m3_saturates_and_keeps_nan():
    assert Q.round_e4m3(1e6) == 448.0 and Q.round_e4m3(-1e6) == -448.0
    assert Q.round_e4m3(463.99) == 448.0 and Q.round_e4m3(464.0) == 448.0 and Q.round_e4m3(470.0) == 448.0
    assert np.isnan(Q.round_e4m3(np.nan))
    assert Q.round_e4m3(2.0 ** -10) == 0.0 and Q.round_e4m3(3 * 2.0 ** -10) == 2.0 ** -8


def test_e4m3_rounding_matches_torch_float8_cast_in_range():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("no float8_e4m3fn in this torch")
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(20000) * s for s in (1e-3, 0.05, 1.0, 30.0, 150.0)])
    v = Q.e4m3_values()
    x = np.concatenate([x, (v[:-1] + v[1:]) / 2, -(v[:-1] + v[1:]) / 2]).astype(np.float32)
    x = x[np.abs(x) <= 448.0]
    t = torch.from_numpy(x).to(torch.float8_e4m3fn).to(torch.float64).numpy()
    assert np.array_equal(Q.round_e4m3(x.astype(np.float64)), t)


def test_quantize_e4m3_forms_the_product_in_fp32():
    # S = 0.5: x / S = 2.125 is a tie between 2.0 and 2.25 -> 2.0 (even code)
    assert Q.quantize_e4m3(np.float32(1.0625), 0.5) == 2.0
    # the decision is taken on fp32(x * fp32(1/S)), not on the exact quotient
    S = 3.0
    x = np.float32(0.6875)                     # x / 3 = 0.22916..; fp32(1/3) x x rounds in fp32
    prod = np.float32(x * np.float32(1.0 / 3.0))
    assert Q.quantize_e4m3(x, S) == Q.round_e4m3(np.float64(prod))
    # round trip of a representable value
    assert Q.dequantize_e4m3(Q.quantize_e4m3(np.float32(1.5 * 0.25), 0.25), 0.25) == 0.375


def test_int8_quantize_with_zero_point():
    assert Q.quantize_int8(0.25, 0.5, 0) == 0          # 0.5 -> 0 (ties to even)
    assert Q.quantize_int8(0.75, 0.5, 0) == 2          # 1.5 -> 2
    assert Q.quantize_int8(-0.75, 0.5, 0) == -2
    assert Q.quantize_int8(0.0, 0.1, 10) == 10
    assert Q.quantize_int8(1000.0, 0.5, 0) == 127 and Q.quantize_int8(-1000.0, 0.5, 3) == -128
    x = np.linspace(-6.0, 6.0, 1001)
    q = Q.quantize_int8(x, 0.05, -7)
    assert np.all(np.abs(Q.dequantize_int8(q, 0.05, -7) - x) <= 0.025 + 1e-12)


def test_weight_scales_are_the_smallest_powers_of_two_that_fit():
    rng = np.random.default_rng(1)
    w = rng.standard_normal((64, 3, 3, 16)) * rng.uniform(1e-3, 10.0, (64, 1, 1, 1))
    w[5] = 0.0
    wq, s = Q.quantize_weights_e4m3(w)
    assert s[5] == 1.0 and np.all(wq[5] == 0)
    e = np.log2(s)
    assert np.array_equal(e, np.round(e))                      # powers of two
    m = np.max(np.abs(w.reshape(64, -1)), axis=1)
    live = m > 0
    assert np.all(m[live] / s[live] <= 448.0) and np.all(m[live] / s[live] > 224.0)
    # dequantized weights are the codes times the scale, within half a step
    deq = wq * s[:, None, None, None]
    assert np.all(np.abs(deq - w) <= np.abs(w) * 2.0 ** -4 + s[:, None, None, None] * 2.0 ** -10)
    assert np.array_equal(Q.round_e4m3(wq), wq)


def test_fp8_layer_with_representable_values_is_exact():
    # small integers are E4M3 values, and with unit-scale folding the
    # quantized layer equals the full-precision one
    g, _ = I.fp8_conv(N=1, H=6, W=7, C=16, K=8, k=3, act="none")
    rng = np.random.default_rng(3)
    conv, bn = g.nodes[1], g.nodes[2]
    conv.consts["weight"] = rng.integers(-2, 3, conv.attrs["weight_shape"]).astype(np.float32)
    bn.consts.update(gamma=np.ones(8, np.float32), beta=np.zeros(8, np.float32),
                     moving_mean=np.zeros(8, np.float32), moving_var=np.full(8, 1.0 - 1e-5, np.float32))
    g.nodes[0].attrs["scale"] = 1.0
    x = rng.integers(-8, 9, (1, 6, 7, 16)).astype(np.float32)
    from oracle import ops
    exact = ops.conv2d_nhwc(x, conv.consts["weight"], (1, 1), (1, 1, 1, 1))
    got = ograph.evaluate(g, {"x": x})[g.outputs[0]]
    # the folded weights w s (s = 1 + ~1e-8) quantize back to the integers w,
    # so the layer computes the integer convolution itself
    np.testing.assert_allclose(got, exact, rtol=1e-12, atol=1e-9)


def test_fp8_dense_against_torch_float8_route():
    torch = pytest.importorskip("torch")
    if not hasattr(torch, "float8_e4m3fn"):
        pytest.skip("no float8_e4m3fn in this torch")
    g, inp = I.fp8_dense(M=24, D=64, F=40)
    x = inp["x"]
    dense, bias = g.nodes[1], g.nodes[2]
    S = g.nodes[0].attrs["scale"]
    # independent route: torch's float8 cast of fp32(x * fp32(1/S)) and of w / S_w
    xq = torch.from_numpy((x.astype(np.float32) * np.float32(1.0 / S)).astype(np.float32)).to(
        torch.float8_e4m3fn).to(torch.float64).numpy() * S
    w = dense.consts["weight"].astype(np.float64)
    m = np.abs(w).max(axis=1)
    sw = 2.0 ** np.ceil(np.log2(m / 448.0))
    wq = torch.from_numpy(w / sw[:, None]).to(torch.float8_e4m3fn).to(torch.float64).numpy() * sw[:, None]
    pre = xq @ wq.T + bias.consts["bias"].astype(np.float64)
    from math import erf, sqrt
    want = np.vectorize(lambda v: 0.5 * v * (1.0 + erf(v / sqrt(2.0))))(pre)
    got = ograph.evaluate(g, inp)[g.outputs[0]]
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


def test_fp8_error_scale_is_zero_where_the_codes_are_exact():
    # Q of an exact input decides the same codes on both sides; the scale of
    # an FP8 layer's output then only carries the fp32 sum and the bf16 store
    g, inp = I.fp8_conv(N=1, H=6, W=6, C=32, K=16, k=1)
    ref, sc = ograph.evaluate_with_error_scale(g, inp, keep=[g.nodes[0].name, g.outputs[0]])
    assert np.all(sc[g.nodes[0].name] == 0)
    o = g.outputs[0]
    assert np.all(sc[o] <= 2.0 ** -9 * np.abs(ref[o]) + 1e-5)
