"""GPU parity: every offloaded composite, run through the C ABI on cuda:0,
against the fp64 oracle on the same seeded inputs.

Small-integer cases must match bit for bit (every fp32 partial sum is an
exact integer, so the GPU's bf16 output equals the bf16 rounding of the exact
result); float cases must satisfy |gpu - ref| <= 1e-2 + 2e-2 |ref|.
"""
import numpy as np
import pytest

from oracle import graph as ograph
from paper_2105_03215_gb300 import abi
from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import region as R

from .parity import assert_bit_exact, assert_close, oracle, run_region, sampled_conv_scale

pytestmark = pytest.mark.gpu


def _check_graph(g, inp, bit_exact=False, what="", options=0):
    reg = R.whole_graph_region(g, options=options)
    got, cr = run_region(reg, inp)
    ref, sc = oracle(g, inp)
    for name in g.outputs:
        if bit_exact:
            assert_bit_exact(got[name], ref[name], what or g.name)
        else:
            assert_close(got[name], ref[name], sc[name], what or g.name)
    cr.release()
    return got, ref


# ------------------------------------------------------------ exact (small integers)

@pytest.mark.parametrize("M,Iw,U", [(200, 192, 320), (128, 64, 64), (37, 136, 24), (300, 768, 1000)])
def test_dense_small_int_bit_exact(M, Iw, U):
    g, inp = I.small_int_dense(M=M, I=Iw, U=U)
    _check_graph(g, inp, bit_exact=True)


@pytest.mark.parametrize("N,H,W,C,K,k,stride,pad", [
    (2, 9, 11, 64, 64, 3, 1, 1),      # im2col, ragged M = 198
    (1, 7, 7, 64, 128, 1, 1, 0),      # 1x1 as plain GEMM, M < 128
    (2, 13, 10, 128, 96, 3, 2, 1),    # stride-2 3x3
    (2, 14, 14, 64, 256, 1, 2, 0),    # stride-2 1x1 (downsample)
    (1, 12, 12, 144, 32, 3, 1, 1),    # 144 channels: zero-filled tail chunk in im2col
    (1, 8, 9, 32, 64, 3, 1, 1),       # 32 channels: 64-byte swizzle
])
def test_conv_small_int_bit_exact(N, H, W, C, K, k, stride, pad):
    g, inp = I.small_int_conv(N=N, H=H, W=W, C=C, K=K, k=k, stride=stride, pad=pad)
    _check_graph(g, inp, bit_exact=True)


@pytest.mark.parametrize("kernel,strides,padding,dilation", [
    ((1, 3), (1, 1), (0, 1, 0, 1), (1, 1)),   # non-square: W taps only
    ((3, 1), (1, 1), (1, 0, 1, 0), (1, 1)),   # non-square: H taps only
    ((3, 3), (2, 1), (1, 0, 1, 2), (1, 1)),   # per-dimension stride, asymmetric padding
    ((3, 3), (1, 1), (2, 2, 2, 2), (2, 2)),   # dilation 2
    ((1, 4), (1, 1), (0, 0, 0, 0), (1, 1)),   # the shape the stem's GEMM uses
])
def test_conv_general_small_int_bit_exact(kernel, strides, padding, dilation):
    g, inp = I.conv_general(kernel=kernel, strides=strides, padding=padding, dilation=dilation,
                            small_int=True)
    _check_graph(g, inp, bit_exact=True)


@pytest.mark.parametrize("N,H,W,C,K", [
    (32, 24, 100, 64, 64),    # 1x4 conv over 64 channels (the stem GEMM's shape), 24 tiles per image
    (32, 25, 100, 64, 48),    # 25 tiles per image: a single tile ends each image; 48 of 64 columns
])
def test_slab_pair_units_small_int_bit_exact(N, H, W, C, K):
    # resident-weight slabs the planner runs as pair units: two adjacent
    # tiles of an image share one slab load and the per-unit waits
    g, inp = I.conv_general(kernel=(1, 4), strides=(1, 1), padding=(0, 0, 0, 0), dilation=(1, 1),
                            N=N, H=H, W=W, C=C, K=K, small_int=True)
    rep = R.whole_graph_region(g).plan(152)
    assert rep.pair_units[0] == 1 and rep.im2col[0] == 2 and rep.resident_b[0] == 1
    _check_graph(g, inp, bit_exact=True)


# ------------------------------------------------------------ float parity

def test_conv3x3_bias_relu_56x56():
    g, inp = I.conv_bias_relu(N=1, H=56, W=56, C=64, K=64, seed=0)
    _check_graph(g, inp)


@pytest.mark.parametrize("act", ["relu6", "gelu", "none"])
def test_conv_epilogue_activations(act):
    g, inp = I.conv_bias_relu(N=2, H=10, W=10, C=64, K=64, seed=5, act=act)
    _check_graph(g, inp)


def test_bert_ffn_small():
    g, inp = I.bert_ffn(M=256, D=256, F=512, seed=1)
    _check_graph(g, inp)


def test_bert_ffn_full():
    g, inp = I.bert_ffn(seed=1)
    _check_graph(g, inp)


def test_mbv2_dw_pw_small():
    g, inp = I.mbv2_dw_pw(N=2, H=20, W=17, C=144, Cout=24, seed=2)
    _check_graph(g, inp)


def test_mbv2_dw_pw_full():
    g, inp = I.mbv2_dw_pw(seed=2)
    _check_graph(g, inp)


@pytest.mark.parametrize("N,H,W,C,stride", [
    (2, 9, 7, 960, 1),     # channels in 4 chunks of 240
    (1, 11, 13, 264, 2),   # 2 chunks of 136, the last one ragged
    (1, 5, 300, 16, 1),    # output wider than one box: column tiles
    (1, 6, 190, 24, 2),    # stride 2, column tiles
    (3, 1, 1, 8, 1),       # 1 x 1 image, 8 channels
    (2, 2, 3, 32, 2),      # output 1 x 2
    (1, 57, 56, 144, 1),   # ragged last row tile
    (1, 112, 112, 96, 2),  # full-width tile overflows a buffer: narrowed column tiles
])
def test_depthwise_tiles(N, H, W, C, stride):
    g, inp = I.depthwise(N=N, H=H, W=W, C=C, stride=stride, seed=N * 7 + C)
    _check_graph(g, inp, what=f"depthwise {N}x{H}x{W}x{C} s{stride}")


def test_depthwise_stride2():
    g, inp = I.mbv2_dw_pw(N=2, H=21, W=20, C=96, Cout=32, seed=9, stride=2)
    _check_graph(g, inp)


def test_bottleneck_small():
    g, inp = I.resnet_bottleneck(N=2, H=14, W=14, C=256, width=64, seed=3)
    _check_graph(g, inp)


def test_bottleneck_downsample_stride2():
    g, inp = I.resnet_bottleneck(N=2, H=14, W=14, C=256, width=128, stride=2, seed=3)
    _check_graph(g, inp)


def test_bottleneck_full():
    g, inp = I.resnet_bottleneck(seed=3)
    _check_graph(g, inp)


def test_resnet50_stem_region():
    g, inp = I.resnet50(N=2, H=64, W=48, seed=4)
    stem = [n.name for n in g.nodes[:3]]  # conv 7x7/2 + bn + relu
    reg = R.Region(g, stem, "stem")
    got, cr = run_region(reg, inp)
    ref, sc = oracle(g, inp, nodes=stem, keep=reg.outputs)
    assert_close(got[reg.outputs[0]], ref[reg.outputs[0]], sc[reg.outputs[0]], "stem")
    cr.release()


@pytest.mark.parametrize("k,cout,C", [(7, 64, 3), (3, 32, 3), (5, 48, 4), (7, 64, 1)])
def test_stem_variants(k, cout, C):
    g, inp = I.stem(k=k, cout=cout, C=C)
    _check_graph(g, inp, what=f"stem{k}x{k}")


@pytest.mark.parametrize("N,H,W,C,K,k,pair", [
    (3, 30, 30, 3, 64, 7, 0),     # the ResNet-50 stem's filter on a small image
    (2, 17, 23, 4, 32, 3, 0),     # odd sizes, 4 channels, 4 row taps (32-element k-blocks)
    (2, 20, 24, 1, 48, 5, 0),     # one channel, 6 of 8 row taps used
    (40, 64, 64, 2, 64, 7, 0),    # 11 tiles of 3 output rows per image
    (64, 112, 112, 3, 64, 7, 1),  # pair units, 28 tiles of 2 output rows per image
    (48, 90, 118, 3, 64, 7, 1),   # pair units, 23 tiles per image: a single tile ends each image
])
def test_stem_small_int_bit_exact(N, H, W, C, K, k, pair):
    # stride-2 few-channel stems through the pixel-pair layout (every filter
    # tap lands in one (r, dx, c) slot of its column tap b)
    g, inp = I.conv_general(kernel=(k, k), strides=(2, 2), padding=(k // 2,) * 4, dilation=(1, 1),
                            N=N, H=H, W=W, C=C, K=K, small_int=True)
    rep = R.whole_graph_region(g).plan(152)
    assert rep.kind[0] == abi.LAUNCH_S2D and rep.im2col[1] == 2 and rep.pair_units[1] == pair
    _check_graph(g, inp, bit_exact=True)


def test_stem_at_full_size_sampled():
    # 83 images of 224 x 224 through the pixel-pair layout and one GEMM in
    # pair units (5-D tensor-map slabs); the oracle checks 3000 sampled
    # outputs, half of them in the last 20 images and the image borders
    from oracle import ops
    g, inp = I.stem(N=83, H=224, W=224, seed=17)
    reg = R.whole_graph_region(g)
    rep = reg.plan(152)
    assert rep.n_launches == 2 and rep.gemm_m[1] == 83 * 112 * 112 and rep.pair_units[1] == 1
    got, cr = run_region(reg, inp)
    y = got[g.outputs[0]].reshape(-1, 64)
    rng = np.random.default_rng(3)
    border = np.array([(n * 112 + p) * 112 + q for n in (0, 82) for p in (0, 1, 110, 111)
                       for q in (0, 1, 55, 110, 111)])
    pix = np.concatenate([rng.integers(0, 63 * 112 * 112, 1460), rng.integers(63 * 112 * 112, 83 * 112 * 112, 1500),
                          border])
    ks = rng.integers(0, 64, pix.size)
    conv, bn = g.nodes[0], g.nodes[1]
    a = conv.attrs
    v = ops.conv2d_nhwc_sampled(inp["data"], conv.consts["weight"], pix, ks, a["strides"], a["padding"],
                                a["dilation"], a["groups"]).reshape(1, -1)
    v = ops.batch_norm(v, bn.consts["gamma"][ks], bn.consts["beta"][ks], bn.consts["moving_mean"][ks],
                       bn.consts["moving_var"][ks], bn.attrs.get("epsilon", 1e-5))
    ref = ops.relu(v).ravel()
    bscale = np.abs(bn.consts["gamma"][ks]) / np.sqrt(bn.consts["moving_var"][ks].astype(np.float64) + 1e-5)
    sc = sampled_conv_scale(inp["data"], conv.consts["weight"], pix, ks, a, bscale, ref)
    assert_close(y[pix, ks], ref, sc, "stem chunks (sampled)")
    cr.release()


def test_gelu_epilogue_within_one_bf16_ulp():
    # identity weights and zero bias: the region computes GELU(x) of bf16
    # inputs swept over [-8, 8], so the epilogue's GELU is compared with the
    # exact one (oracle, erf in fp64) after rounding both to bf16
    import numpy as np
    b = I._Builder("gelu_sweep")
    x = b.input("x", (128, 128))
    y = b.gelu(b.bias_add(b.dense(x, 128)))
    g, _ = I._finish(b, [y], seed=3)
    g.nodes[0].consts["weight"] = np.eye(128, dtype=np.float32)
    g.nodes[1].consts["bias"] = np.zeros(128, dtype=np.float32)
    xs = I.bf16_round(np.linspace(-8.0, 8.0, 128 * 128, dtype=np.float32).reshape(128, 128))
    inp = {"x": xs}
    reg = R.whole_graph_region(g)
    got, cr = run_region(reg, inp)
    ref = ograph.evaluate(g, inp)[g.outputs[0]]
    gv = got[g.outputs[0]].astype(np.float64)
    got_b = I.bf16_bits(gv.astype(np.float32)).astype(np.int32)
    ref_b = I.bf16_bits(ref.astype(np.float32)).astype(np.int32)
    # where |GELU| >= 1e-3 the bf16 results agree to one ulp (bf16 patterns are
    # ordered like their values within one sign); below that, 1 + erf(z)
    # cancels in fp32 for large negative inputs, so compare absolutely
    big = np.abs(ref) >= 1e-3
    assert ((got_b < 0x8000) == (ref_b < 0x8000))[big].all()
    assert np.abs(got_b - ref_b)[big].max() <= 1
    assert np.abs(gv - ref)[~big].max() <= 1e-5
    cr.release()


def test_region_can_run_twice_with_new_pointers():
    import torch
    from .parity import to_dev
    g, inp = I.conv_bias_relu(N=1, H=16, W=16, C=64, K=64, seed=11)
    reg = R.whole_graph_region(g)
    cr = reg.compile()
    ref, sc = oracle(g, inp)
    ref, sc = ref[g.outputs[0]], sc[g.outputs[0]]
    for _ in range(2):
        x = to_dev(inp["x"])
        y = torch.full(g.shape_of(g.outputs[0]), float("nan"), dtype=torch.bfloat16, device="cuda")
        cr.run([x], [y])
        torch.cuda.synchronize()
        cr.check()
        assert_close(y.float().cpu().numpy(), ref, sc, "rerun")
    cr.release()


def test_depthwise_regions_sharing_a_kernel_run_in_any_compile_order():
    # The dynamic shared-memory limit belongs to the kernel, not the launch:
    # compiling a region with a small tile after one with a large tile must
    # not shrink the limit the first one launches under.
    import torch
    from .parity import to_dev
    big_g, big_inp = I.depthwise(N=1, H=57, W=56, C=144, stride=1, seed=4)
    small_g, small_inp = I.depthwise(N=3, H=1, W=1, C=8, stride=1, seed=5)
    big = R.whole_graph_region(big_g).compile()
    small = R.whole_graph_region(small_g).compile()
    for g, inp, cr in [(big_g, big_inp, big), (small_g, small_inp, small)]:
        x = to_dev(inp["x"])
        y = torch.full(g.shape_of(g.outputs[0]), float("nan"), dtype=torch.bfloat16, device="cuda")
        cr.run([x], [y])
        torch.cuda.synchronize()
        cr.check()
        ref, sc = oracle(g, inp)
        assert_close(y.float().cpu().numpy(), ref[g.outputs[0]], sc[g.outputs[0]], g.name)
    big.release()
    small.release()


@pytest.mark.parametrize("make", [
    lambda: I.resnet_bottleneck(N=2, H=14, W=14, C=256, width=64, seed=5),
    lambda: I.mbv2_dw_pw(N=2, H=12, W=12, C=96, Cout=32, seed=6),
    lambda: I.bert_ffn(M=96, D=128, F=256, seed=7),
])
def test_deserialized_region_runs_bit_identically(make):
    # Section 3.3 option 3: a region rebuilt from its serialised bytes runs the
    # same kernels on the same constants as the compiled one
    g, inp = make()
    reg = R.whole_graph_region(g)
    got, cr = run_region(reg, inp)
    blob = cr.serialize()
    cr.release()
    cr2 = reg.load(blob)
    assert cr2.serialize() == blob
    got2, _ = run_region(reg, inp, compiled=cr2)
    for name in g.outputs:
        assert np.array_equal(got[name].view(np.uint32), got2[name].view(np.uint32)), name
    ref, sc = oracle(g, inp)
    assert_close(got2[g.outputs[0]], ref[g.outputs[0]], sc[g.outputs[0]], g.name)
    cr2.release()


@pytest.mark.parametrize("N,C,H,W,Cp", [
    (2, 3, 37, 224, 3),    # ResNet-50 input rows; 24-row blocks and a ragged last block
    (1, 3, 9, 224, 8),     # channels zero-padded to 8
    (3, 3, 4, 5, 3),       # rows of 15 values: the unvectorised store path
    (1, 16, 7, 1024, 16),  # one row per block (W * Cp = 16384)
])
def test_nchw_fp32_to_nhwc_bf16_boundary_transform_bit_exact(N, C, H, W, Cp):
    # Section 3.2: the layout transformation and cast at a region boundary;
    # every output is one rounding of one input, so the comparison is exact
    import torch
    from oracle import ops
    from paper_2105_03215_gb300 import abi
    rng = np.random.default_rng(N * 100 + C + W)
    x = (rng.standard_normal((N, C, H, W)) * np.exp2(rng.integers(-8, 8, (N, C, H, W)))).astype(np.float32)
    xd = torch.from_numpy(x).cuda()
    y = torch.full((N, H, W, Cp), float("nan"), dtype=torch.bfloat16, device="cuda")
    abi.check(abi.lib().byoc_nchw_to_nhwc_bf16(xd.data_ptr(), y.data_ptr(), N, C, H, W, Cp, None))
    torch.cuda.synchronize()
    ref = ops.nchw_to_nhwc(x, Cp)
    assert np.array_equal(y.float().cpu().numpy().astype(np.float64), ref)


def test_nchw_boundary_rejects_bad_shapes_on_the_host():
    import torch
    from paper_2105_03215_gb300 import abi
    x = torch.zeros(1, 4, 2, 2, device="cuda")
    y = torch.zeros(1, 2, 2, 8, dtype=torch.bfloat16, device="cuda")
    assert abi.lib().byoc_nchw_to_nhwc_bf16(x.data_ptr(), y.data_ptr(), 1, 4, 2, 2, 3, None) == abi.ERR_INVALID_ARG
    assert abi.lib().byoc_nchw_to_nhwc_bf16(x.data_ptr(), y.data_ptr(), 1, 4, 2, 20000, 8, None) == abi.ERR_INVALID_ARG


def _dw_pw_graph(N, H, W, C, Cout, stride, residual, seed, small_int=False):
    b = I._Builder("dw_pw_case")
    x = b.input("x", (N, H, W, C))
    d = b.relu6(b.batch_norm(b.conv2d(x, C, 3, stride=stride, groups=C)))
    y = b.batch_norm(b.conv2d(d, Cout, 1))
    if residual:
        Ho, Wo = (H - 1) // stride + 1, (W - 1) // stride + 1
        r = b.input("r", (N, Ho, Wo, Cout))
        y = b.add(y, r)
    return I._finish(b, [y], seed)


@pytest.mark.parametrize("N,H,W,C,Cout,stride,residual", [
    (2, 13, 9, 48, 16, 1, False),     # fewer than 64 channels, ragged row tile
    (1, 30, 30, 160, 40, 2, False),   # three channel chunks (64, 64, 32), stride 2, N padded to 48
    (3, 7, 7, 96, 8, 1, True),        # 7x7 maps, one tile per image, residual, N padded to 16
    (1, 112, 112, 32, 16, 1, False),  # 112-wide rows: one output row per tile
    (2, 28, 28, 192, 64, 2, False),   # stride 2 at 28x28 (MobileNetV2 block 3 shape)
    (2, 14, 14, 384, 64, 1, True),    # 6 chunks, 64 outputs, residual
])
def test_fused_depthwise_pointwise(N, H, W, C, Cout, stride, residual):
    # depthwise + BN + ReLU6 -> 1x1 + BN (+ residual) in one kernel against the
    # oracle of the unfused chain
    from paper_2105_03215_gb300 import abi
    g, inp = _dw_pw_graph(N, H, W, C, Cout, stride, residual, seed=N + C + Cout)
    rep = R.whole_graph_region(g, options=abi.OPT_FUSE_DW_PW).plan(152)
    assert rep.n_launches == 1 and rep.kind[0] == abi.LAUNCH_DWPW
    _check_graph(g, inp, what=f"dw_pw {N}x{H}x{W}x{C}->{Cout} s{stride} res{residual}",
                 options=abi.OPT_FUSE_DW_PW)


def test_fused_depthwise_pointwise_equals_the_two_launches_bit_for_bit():
    # the fused kernel rounds the depthwise output to bf16 and accumulates the
    # 1x1 conv's K steps in the same order as the two separate launches, so the
    # outputs agree bit for bit (separate launches: the depthwise output is
    # also a region output, which keeps it out of the fusion)
    import torch
    from .parity import to_dev
    g, inp = I.mbv2_dw_pw(N=4, H=28, W=28, C=144, Cout=24, seed=12)
    fused = R.whole_graph_region(g, options=abi.OPT_FUSE_DW_PW)
    split = R.Region(g, [n.name for n in g.nodes], "split", outputs=[g.nodes[2].name, g.outputs[0]],
                     options=abi.OPT_FUSE_DW_PW)
    got_f, cf = run_region(fused, inp)
    got_s, cs = run_region(split, inp)
    assert cf.n_launches == 1 and cs.n_launches == 2
    a, b = got_f[g.outputs[0]], got_s[g.outputs[0]]
    assert np.array_equal(a.view(np.uint32), b.view(np.uint32))
    cf.release()
    cs.release()


@pytest.mark.parametrize("M,Iw,U", [(100, 3072, 256), (1024, 3072, 768), (64, 2048, 1000), (7, 1024, 40)])
def test_split_k_dense_matches_and_is_deterministic(M, Iw, U):
    # deep reductions over few tiles run split-K: every split writes an fp32
    # partial, the last to arrive sums them in split order -- within tolerance
    # of the oracle, and the same bits on every run
    import torch
    from .parity import to_dev
    b = I._Builder("dense_deep")
    x = b.input("x", (M, Iw))
    y = b.bias_add(b.dense(x, U))
    g, inp = I._finish(b, [y], seed=M + U)
    reg = R.whole_graph_region(g)
    rep = reg.plan(152)
    got, cr = run_region(reg, inp)
    ref, sc = oracle(g, inp)
    assert_close(got[g.outputs[0]], ref[g.outputs[0]], sc[g.outputs[0]], f"dense {M}x{Iw}->{U}")
    out = torch.empty(g.shape_of(g.outputs[0]), dtype=torch.bfloat16, device="cuda")
    xs = [to_dev(inp["x"])]
    ref_bits = None
    for _ in range(3):
        cr.run(xs, [out])
        torch.cuda.synchronize()
        bits = out.view(torch.int16).cpu().numpy().copy()
        ref_bits = bits if ref_bits is None else ref_bits
        assert np.array_equal(bits, ref_bits)
    cr.check()
    cr.release()
    if (M, Iw, U) == (1024, 3072, 768):
        assert rep.splits[0] == 3


@pytest.mark.parametrize("N,H,W,C,s", [(2, 15, 13, 64, 2), (1, 9, 10, 16, 1), (3, 112, 112, 64, 2), (1, 7, 1, 8, 2)])
def test_max_pool_3x3_host_operator_bit_exact(N, H, W, C, s):
    # the host max pool (padding 1): two outputs per thread, packed bf16 max --
    # the max of bf16 values is one of them, so the result is exact
    import torch
    from oracle import ops
    from paper_2105_03215_gb300 import abi
    from .parity import to_dev
    rng = np.random.default_rng(N * 31 + W)
    x = I.bf16_round(rng.standard_normal((N, H, W, C)).astype(np.float32))
    Ho, Wo = (H + 2 - 3) // s + 1, (W + 2 - 3) // s + 1
    xd = to_dev(x)
    y = torch.full((N, Ho, Wo, C), float("nan"), dtype=torch.bfloat16, device="cuda")
    abi.check(abi.lib().byoc_max_pool2d_nhwc(xd.data_ptr(), y.data_ptr(), N, H, W, C, 3, s, 1, None))
    torch.cuda.synchronize()
    ref = ops.max_pool2d_nhwc(x, (3, 3), (s, s), (1, 1, 1, 1))
    assert_bit_exact(y.float().cpu().numpy(), ref, f"maxpool {N}x{H}x{W}x{C} s{s}")


@pytest.mark.parametrize("N,H,W,C", [(64, 7, 7, 2048), (3, 5, 9, 24), (2, 1, 1, 8), (5, 14, 14, 264)])
def test_global_avg_pool_host_operator(N, H, W, C):
    # the host average pool: fp32 sums of pixel slices added in a fixed order,
    # one bf16 rounding -- within one bf16 rounding of the exact mean
    import torch
    from oracle import ops
    from .parity import to_dev
    rng = np.random.default_rng(N * 7 + C)
    x = I.bf16_round(rng.standard_normal((N, H, W, C)).astype(np.float32))
    y = torch.full((N, C), float("nan"), dtype=torch.bfloat16, device="cuda")
    abi.check(abi.lib().byoc_global_avg_pool_nhwc(to_dev(x).data_ptr(), y.data_ptr(), N, H, W, C, None))
    torch.cuda.synchronize()
    ref = ops.global_avg_pool_nhwc(x)
    got = y.float().cpu().numpy().astype(np.float64)
    # bf16 keeps 8 significant bits: |got - ref| <= 2^-8 |ref| + fp32 summation error
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 1e-5), f"avgpool {N}x{H}x{W}x{C}"
