"""Pins of the fp64 oracle against facts fixed outside it.

Each test checks the oracle against a hand computation, a closed form, an
invariant, a special case that reduces to a library routine, or brute force on
tiny inputs, so that a dropped term, a wrong sign or index, or a transposed
operand in any oracle routine fails at least one of them.
"""
import math
import os

import numpy as np
import pytest

from oracle import ops
from oracle import graph as ograph
from paper_2105_03215_gb300 import inputs as I

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *nums = line.split()
            vals[key] = np.array([float(v) for v in nums])
    return vals


def brute_conv(x, w, stride, pad, dil, groups):
    """Pure-Python conv2d on tiny inputs (no numpy arithmetic)."""
    N, H, W, C = x.shape
    K, Cg, R, S = w.shape
    sh, sw = stride
    pt, pl, pb, pr = pad
    dh, dw = dil
    Ho = (H + pt + pb - dh * (R - 1) - 1) // sh + 1
    Wo = (W + pl + pr - dw * (S - 1) - 1) // sw + 1
    Kg = K // groups
    y = np.zeros((N, Ho, Wo, K))
    for n in range(N):
        for p in range(Ho):
            for q in range(Wo):
                for k in range(K):
                    g = k // Kg
                    acc = 0.0
                    for ci in range(Cg):
                        for r in range(R):
                            for s in range(S):
                                h = p * sh + r * dh - pt
                                ww = q * sw + s * dw - pl
                                if 0 <= h < H and 0 <= ww < W:
                                    acc += float(x[n, h, ww, g * Cg + ci]) * float(w[k, ci, r, s])
                    y[n, p, q, k] = acc
    return y


# ---------------------------------------------------------------- conv2d

def test_conv_hand_case_golden():
    g = _read_golden("conv3x3_ones_pad1.txt")
    x = g["input"].reshape(1, 3, 3, 1)
    w = g["weight"].reshape(1, 1, 3, 3)
    y = ops.conv2d_nhwc(x, w, (1, 1), (1, 1, 1, 1))
    assert np.array_equal(y.reshape(-1), g["expected"])


def test_conv_identity_1x1():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((2, 5, 7, 6))
    w = np.eye(6).reshape(6, 6, 1, 1)
    assert np.array_equal(ops.conv2d_nhwc(x, w), x)


def test_conv_centre_delta_3x3_is_identity():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((1, 6, 5, 4))
    w = np.zeros((4, 4, 3, 3))
    for c in range(4):
        w[c, c, 1, 1] = 1.0
    assert np.array_equal(ops.conv2d_nhwc(x, w, (1, 1), (1, 1, 1, 1)), x)


def test_conv_delta_input_reads_back_flipped_kernel():
    """x = delta at (2,3): y[2-1+a, 3-1+b] = w[2-a, 2-b] (cross-correlation
    orientation, not convolution)."""
    x = np.zeros((1, 5, 7, 1))
    x[0, 2, 3, 0] = 1.0
    w = np.arange(1, 10, dtype=np.float64).reshape(1, 1, 3, 3)
    y = ops.conv2d_nhwc(x, w, (1, 1), (1, 1, 1, 1))[0, :, :, 0]
    patch = y[1:4, 2:5]
    assert np.array_equal(patch, w[0, 0, ::-1, ::-1])
    assert np.count_nonzero(y) == 9


@pytest.mark.parametrize("stride,pad,dil,groups", [
    ((1, 1), (0, 0, 0, 0), (1, 1), 1),
    ((2, 2), (1, 2, 0, 1), (1, 1), 1),
    ((1, 2), (2, 1, 2, 0), (2, 1), 1),
    ((2, 1), (1, 1, 1, 1), (1, 1), 3),
])
def test_conv_matches_pure_python_brute_force(stride, pad, dil, groups):
    rng = np.random.default_rng(2)
    x = rng.standard_normal((2, 5, 6, 6))
    w = rng.standard_normal((6, 6 // groups, 3, 2))
    y = ops.conv2d_nhwc(x, w, stride, pad, dil, groups)
    ref = brute_conv(x, w, stride, pad, dil, groups)
    assert y.shape == ref.shape
    np.testing.assert_allclose(y, ref, rtol=1e-13, atol=1e-13)


def _im2col(x, R, S, stride, pad, dil):
    """Test-only explicit im2col: rows (n,p,q), columns (r,s,c)."""
    N, H, W, C = x.shape
    pt, pl, pb, pr = pad
    xp = np.zeros((N, H + pt + pb, W + pl + pr, C))
    xp[:, pt:pt + H, pl:pl + W, :] = x
    Ho = (H + pt + pb - dil[0] * (R - 1) - 1) // stride[0] + 1
    Wo = (W + pl + pr - dil[1] * (S - 1) - 1) // stride[1] + 1
    cols = np.zeros((N, Ho, Wo, R, S, C))
    for r in range(R):
        for s in range(S):
            h0, w0 = r * dil[0], s * dil[1]
            cols[:, :, :, r, s, :] = xp[:, h0:h0 + stride[0] * (Ho - 1) + 1:stride[0],
                                        w0:w0 + stride[1] * (Wo - 1) + 1:stride[1], :]
    return cols.reshape(N * Ho * Wo, R * S * C), (N, Ho, Wo)


@pytest.mark.parametrize("R,stride,pad", [(3, (1, 1), (1, 1, 1, 1)), (1, (2, 2), (0, 0, 0, 0)),
                                          (7, (2, 2), (3, 3, 3, 3)), (3, (2, 2), (1, 1, 1, 1))])
def test_conv_equals_im2col_times_gemm(R, stride, pad):
    rng = np.random.default_rng(3)
    x = rng.standard_normal((2, 13, 11, 8))
    w = rng.standard_normal((10, 8, R, R))
    A, (N, Ho, Wo) = _im2col(x, R, R, stride, pad, (1, 1))
    B = w.transpose(0, 2, 3, 1).reshape(10, -1)  # [K, (r,s,c)]
    ref = (A @ B.T).reshape(N, Ho, Wo, 10)
    y = ops.conv2d_nhwc(x, w, stride, pad)
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


def test_conv_matches_torch_float64_library_route():
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    rng = np.random.default_rng(4)
    for (C, K, groups, R, stride, pad, dil) in [(8, 12, 1, 3, 1, (1, 1, 1, 1), 1),
                                                 (16, 16, 16, 3, 2, (1, 1, 1, 1), 1),
                                                 (6, 4, 2, 3, 1, (0, 2, 1, 0), 2),
                                                 (3, 5, 1, 7, 2, (3, 3, 3, 3), 1)]:
        x = rng.standard_normal((2, 15, 14, C))
        w = rng.standard_normal((K, C // groups, R, R))
        y = ops.conv2d_nhwc(x, w, (stride, stride), pad, (dil, dil), groups)
        xt = torch.from_numpy(x).permute(0, 3, 1, 2)
        xt = F.pad(xt, (pad[1], pad[3], pad[0], pad[2]))
        ref = F.conv2d(xt, torch.from_numpy(w), stride=stride, dilation=dil, groups=groups)
        np.testing.assert_allclose(y, ref.permute(0, 2, 3, 1).numpy(), rtol=1e-12, atol=1e-12)


def test_conv_sampled_matches_brute_force():
    rng = np.random.default_rng(5)
    x = rng.standard_normal((2, 6, 7, 4))
    w = rng.standard_normal((6, 2, 3, 3))
    stride, pad, dil, groups = (2, 1), (1, 0, 2, 1), (1, 2), 2
    ref = brute_conv(x, w, stride, pad, dil, groups)
    N, Ho, Wo, K = ref.shape
    pix = rng.integers(0, N * Ho * Wo, size=40)
    ks = rng.integers(0, K, size=40)
    got = ops.conv2d_nhwc_sampled(x, w, pix, ks, stride, pad, dil, groups)
    np.testing.assert_allclose(got, ref.reshape(-1, K)[pix, ks], rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------- dense

def test_dense_identity_input_reads_back_transposed_weight():
    rng = np.random.default_rng(6)
    w = rng.standard_normal((5, 3))  # [units, in], not square
    y = ops.dense(np.eye(3), w)
    assert np.array_equal(y, w.T)


def test_dense_brute_force():
    x = np.array([[1.0, 2.0, 3.0], [-1.0, 0.5, 4.0]])
    w = np.array([[1.0, 0.0, -1.0], [2.0, 1.0, 0.0]])
    # hand: row0 . w0 = 1-3 = -2 ; row0 . w1 = 2+2 = 4 ; row1 . w0 = -1-4 = -5 ; row1 . w1 = -2+0.5 = -1.5
    assert np.array_equal(ops.dense(x, w), np.array([[-2.0, 4.0], [-5.0, -1.5]]))


def test_dense_matches_numpy_matmul():
    rng = np.random.default_rng(7)
    x = rng.standard_normal((33, 70))
    w = rng.standard_normal((21, 70))
    np.testing.assert_allclose(ops.dense(x, w), x @ w.T, rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------- elementwise

def test_bias_add_on_channel_axis():
    y = np.zeros((2, 2, 3))
    out = ops.bias_add(y, np.array([1.0, -2.0, 0.5]))
    assert np.array_equal(out[1, 1], [1.0, -2.0, 0.5]) and np.array_equal(out[0, 0], out[1, 1])


def test_batch_norm_closed_form():
    # gamma=2, beta=1, mean=3, var+eps=4  ->  y = 2*(x-3)/2 + 1 = x - 2
    x = np.array([[0.0, 5.0], [3.0, -1.0]])
    eps = 1e-5
    y = ops.batch_norm(x, np.array([2.0, 2.0]), np.array([1.0, 1.0]), np.array([3.0, 3.0]),
                       np.array([4.0 - eps, 4.0 - eps]), eps)
    np.testing.assert_allclose(y, x - 2.0, rtol=0, atol=1e-15)
    # per-channel: the second channel must use its own statistics
    y2 = ops.batch_norm(np.ones((1, 2)), np.array([1.0, 3.0]), np.array([0.0, -1.0]),
                        np.array([0.0, 1.0]), np.array([1.0, 1.0]), 0.0)
    assert np.array_equal(y2, [[1.0, -1.0]])


def test_relu_relu6_special_values():
    v = np.array([-1.0, 0.0, 3.0, 6.0, 7.0])
    assert np.array_equal(ops.relu(v), [0.0, 0.0, 3.0, 6.0, 7.0])
    assert np.array_equal(ops.relu6(v), [0.0, 0.0, 3.0, 6.0, 6.0])


def test_gelu_is_x_times_normal_cdf():
    xs = np.array([-5.0, -1.5, -0.3, 0.0, 0.2, 1.0, 2.5, 8.0])
    y = ops.gelu(xs)
    phi = np.array([0.5 * math.erfc(-v / math.sqrt(2.0)) for v in xs])  # Phi via erfc
    np.testing.assert_allclose(y, xs * phi, rtol=1e-14, atol=1e-15)
    assert y[3] == 0.0
    assert abs(y[-1] - 8.0) < 1e-12 and abs(y[0]) < 1e-5
    # gelu(x) - gelu(-x) = x  (odd part of x*Phi(x))
    np.testing.assert_allclose(ops.gelu(xs) - ops.gelu(-xs), xs, rtol=0, atol=1e-14)


def test_add_elementwise():
    a = np.arange(6.0).reshape(2, 3)
    assert np.array_equal(ops.add(a, -2 * a), -a)


# ---------------------------------------------------------------- pools

def test_max_pool_padding_never_wins():
    x = -np.arange(1, 17, dtype=np.float64).reshape(1, 4, 4, 1)  # all negative
    y = ops.max_pool2d_nhwc(x, (3, 3), (2, 2), (1, 1, 1, 1))[0, :, :, 0]
    # x[h,w] = -(4h+w+1).  Output (p,q) covers rows 2p-1..2p+1, cols 2q-1..2q+1;
    # its max is the in-image element nearest the top-left:
    # (0,0)->x[0,0]=-1, (0,1)->x[0,1]=-2, (1,0)->x[1,0]=-5, (1,1)->x[1,1]=-6.
    # A pad value of 0 winning would give 0 in the first row and column.
    assert np.array_equal(y, np.array([[-1.0, -2.0], [-5.0, -6.0]]))


def test_global_avg_pool_closed_form():
    x = np.arange(2 * 3 * 4 * 2, dtype=np.float64).reshape(2, 3, 4, 2)
    y = ops.global_avg_pool_nhwc(x)
    # mean of an arithmetic progression over (h,w) for fixed (n,c)
    assert np.allclose(y, x.mean(axis=(1, 2)), rtol=0, atol=1e-12)
    assert y[0, 0] == (0 + 22) / 2.0


# ---------------------------------------------------------------- chains

def test_bn_fold_equals_unfolded_chain():
    """conv -> bias_add -> batch_norm equals conv with w*s and folded bias
    (fold computed here in fp64; the oracle itself never folds)."""
    rng = np.random.default_rng(8)
    x = rng.standard_normal((1, 6, 6, 5))
    w = rng.standard_normal((7, 5, 3, 3))
    b = rng.standard_normal(7)
    gamma, beta = rng.uniform(0.5, 1.5, 7), rng.standard_normal(7) * 0.1
    mean, var, eps = rng.standard_normal(7) * 0.1, rng.uniform(0.5, 1.5, 7), 1e-5
    chain = ops.batch_norm(ops.bias_add(ops.conv2d_nhwc(x, w, (1, 1), (1, 1, 1, 1)), b),
                           gamma, beta, mean, var, eps)
    s = gamma / np.sqrt(var + eps)
    folded = ops.bias_add(ops.conv2d_nhwc(x, w * s[:, None, None, None], (1, 1), (1, 1, 1, 1)),
                          (b - mean) * s + beta)
    np.testing.assert_allclose(chain, folded, rtol=1e-12, atol=1e-12)


def test_graph_evaluator_on_workload_matches_direct_ops():
    g, inp = I.conv_bias_relu(N=1, H=6, W=5, C=8, K=4, seed=0)
    out = ograph.evaluate(g, inp)[g.outputs[0]]
    conv, bias = g.nodes[0], g.nodes[1]
    ref = np.maximum(brute_conv(inp["x"].astype(np.float64), conv.consts["weight"].astype(np.float64),
                                (1, 1), (1, 1, 1, 1), (1, 1), 1) + bias.consts["bias"], 0.0)
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_bf16_rounding_is_round_to_nearest_even():
    # 1 + 2^-8 is halfway between bf16 neighbours 1 and 1+2^-7: ties to even (1.0)
    # 1 + 3*2^-8 is halfway between 1+2^-7 and 1+2^-6: ties to even (1+2^-6)
    v = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, 1.0 + 2 ** -8 + 2 ** -20, -2.5],
                 dtype=np.float32)
    r = I.bf16_round(v)
    assert list(r) == [1.0, 1.0, 1.0 + 2 ** -6, 1.0 + 2 ** -7, -2.5]


# ------------------------------------------------------------ bf16 rounding (boundary cast)

def test_round_bf16_ties_to_even_and_keeps_representable_values():
    from oracle import ops
    one = 1.0
    # spacing at 1 is 2^-7; midpoints go to the even neighbour
    assert ops.round_bf16(np.array([one + 2.0 ** -8]))[0] == 1.0
    assert ops.round_bf16(np.array([one + 3 * 2.0 ** -8]))[0] == 1.0 + 2.0 ** -6
    assert ops.round_bf16(np.array([-(one + 3 * 2.0 ** -8)]))[0] == -(1.0 + 2.0 ** -6)
    assert ops.round_bf16(np.array([one + 2.0 ** -8 + 2.0 ** -20]))[0] == 1.0 + 2.0 ** -7
    rep = np.array([0.0, 1.0, -2.5, 3.0 * 2.0 ** 100, 2.0 ** -126, 1.5 * 2.0 ** -130])
    assert np.array_equal(ops.round_bf16(rep), rep)
    assert np.isinf(ops.round_bf16(np.array([3.5e38]))[0])


def test_round_bf16_is_the_nearest_bf16_value():
    # brute force: the result carries at most 8 significant bits and no other
    # such value at the same binade spacing is closer
    from oracle import ops
    rng = np.random.default_rng(5)
    x = rng.standard_normal(20000) * np.exp2(rng.integers(-20, 20, 20000))
    r = ops.round_bf16(x)
    m, e = np.frexp(r)
    assert np.all(np.ldexp(m, 8) == np.rint(np.ldexp(m, 8)))     # 8 significant bits
    ulp = np.ldexp(1.0, np.frexp(x)[1] - 8)
    assert np.all(np.abs(x - r) <= ulp / 2)
    for d in (-1, 1):
        assert np.all(np.abs(x - r) <= np.abs(x - (r + d * ulp)))


def test_nchw_to_nhwc_moves_every_value_and_pads_with_zeros():
    from oracle import ops
    x = np.arange(2 * 3 * 4 * 5, dtype=np.float64).reshape(2, 3, 4, 5)   # small integers: exact in bf16
    y = ops.nchw_to_nhwc(x, 8)
    assert y.shape == (2, 4, 5, 8)
    for n, c, h, w in [(0, 0, 0, 0), (1, 2, 3, 4), (0, 1, 2, 3)]:
        assert y[n, h, w, c] == x[n, c, h, w]
    assert not y[..., 3:].any()
