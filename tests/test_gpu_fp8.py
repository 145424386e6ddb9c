"""Partial quantization (Section 3.2): regions with Q nodes run their
convolutions / dense layers in FP8 (E4M3 codes on kind::f8f6f4 tensor cores,
fp32 accumulation), as per-composite GEMM launches (the default) or in the
region kernel (BYOC_OPT_REGION_KERNEL), against the oracle's definition of
the quantized chain (oracle/quant.py, oracle/graph.py)."""
import numpy as np
import pytest

from oracle import graph as ograph
from paper_2105_03215_gb300 import abi
from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import region as R

from .parity import assert_bit_exact, assert_close, oracle, run_region


def _identity_fp8_conv(N=2, H=9, W=11, C=256, seed=5):
    """FP8 1x1 conv with identity weights and a unit-scale batch norm: the
    output is the dequantized input, code x S, rounded once to bf16."""
    g, inp = I.fp8_conv(N=N, H=H, W=W, C=C, K=C, k=1, act="none", seed=seed)
    conv, bn = g.nodes[1], g.nodes[2]
    conv.consts["weight"] = np.eye(C, dtype=np.float32).reshape(C, C, 1, 1)
    bn.consts.update(gamma=np.ones(C, np.float32), beta=np.zeros(C, np.float32),
                     moving_mean=np.zeros(C, np.float32), moving_var=np.full(C, 1.0 - 1e-5, np.float32))
    # a power-of-two scale: code x S is exact in fp32 and in bf16
    g.nodes[0].attrs["scale"] = 1.0 / 32.0
    rng = np.random.default_rng(seed)
    # values over the whole E4M3 range of the scale, ties and saturation included
    x = rng.standard_normal((N, H, W, C)).astype(np.float32) * np.float32(3.0)
    x.reshape(-1)[:64] = np.float32(500.0 / 32.0)  # 500 / 32 quantizes to the saturated 448
    inp["x"] = I.bf16_round(x)
    return g, inp


RK = abi.OPT_REGION_KERNEL
PLANS = {"per_composite": 0, "region_kernel": RK}


def _int_fp8(g, seed):
    """Small-integer weights and inputs, unit-scale batch norm and Q scales of
    1/16: every code, code product and fp32 sum is exact (multiples of a power
    of two far below 2^24 ulps), so any correct plan gives the same bits."""
    rng = np.random.Generator(np.random.PCG64(seed))
    for n in g.nodes:
        if n.op in ("nn.conv2d", "nn.dense"):
            n.consts["weight"] = rng.integers(-1, 2, size=n.attrs["weight_shape"]).astype(np.float32)
        elif n.op == "nn.batch_norm":
            C = n.shape[-1]
            n.consts.update(gamma=np.ones(C, np.float32), beta=rng.integers(-4, 5, C).astype(np.float32),
                            moving_mean=np.zeros(C, np.float32), moving_var=np.full(C, 1.0 - 1e-5, np.float32))
        elif n.op == "nn.bias_add":
            n.consts["bias"] = rng.integers(-4, 5, n.shape[-1]).astype(np.float32)
        elif n.op == "qnn.quantize":
            n.attrs["scale"] = 1.0 / 16.0
    return {k: rng.integers(-2, 3, size=g.shape_of(k)).astype(np.float32) for k in g.inputs}


# ------------------------------------------------------------ plans (CPU)

@pytest.mark.parametrize("make,stages", [(lambda: I.fp8_conv(N=1), 1), (lambda: I.fp8_dense(M=64), 1),
                                         (lambda: I.fp8_bottleneck(N=2), 3)])
def test_fp8_region_kernel_plan_is_a_quantize_launch_and_a_region_kernel(make, stages):
    g, _ = make()
    rep = R.whole_graph_region(g, options=RK).plan(152)
    kinds = [rep.kind[i] for i in range(rep.n_launches)]
    assert kinds == [abi.LAUNCH_QUANT, abi.LAUNCH_CHAIN]
    assert rep.stages[1] == stages and rep.fp8[1] == stages
    blob = R.whole_graph_region(g, options=RK).plan_serialized(152)
    assert [R.load_plan_report(blob).kind[i] for i in range(2)] == kinds


@pytest.mark.parametrize("make,gemms", [(lambda: I.fp8_conv(N=1), 1), (lambda: I.fp8_dense(M=64), 1),
                                        (lambda: I.fp8_bottleneck(N=2), 3)])
def test_fp8_per_composite_plan_is_a_quantize_launch_and_fp8_gemms(make, gemms):
    # the leading Q node on the region input is a launch of its own; the Q
    # nodes after the first two bottleneck convolutions are fused into their
    # epilogues (E4M3 outputs)
    g, _ = make()
    rep = R.whole_graph_region(g).plan(152)
    assert [rep.kind[i] for i in range(rep.n_launches)] == [abi.LAUNCH_QUANT] + [abi.LAUNCH_GEMM] * gemms
    for i in range(1, rep.n_launches):
        assert rep.fp8[i] == 1 and rep.tile_k[i] == 128 and rep.multicast[i] == 0
    blob = R.whole_graph_region(g).plan_serialized(152)
    back = R.load_plan_report(blob)
    assert [back.fp8[i] for i in range(back.n_launches)] == [rep.fp8[i] for i in range(rep.n_launches)]


def test_fp8_short_k_plans_a_grid_of_whole_column_tiles():
    g, _ = I.fp8_dense(M=16384, D=256, F=512)
    rep = R.whole_graph_region(g).plan(152)
    assert rep.fp8[1] == 1 and rep.tile_n[1] == 64 and rep.grid[1] % (512 // 64) == 0


def test_fp8_split_k_plans_for_few_tiles():
    # 2 m-tiles x 12 column tiles of a 3072-deep reduction: the k-blocks are
    # split over CTAs (global split-K on FP8 k-blocks)
    g, _ = I.fp8_dense(M=256, D=3072, F=768)
    rep = R.whole_graph_region(g).plan(152)
    assert rep.kind[1] == abi.LAUNCH_GEMM and rep.fp8[1] == 1 and rep.splits[1] > 1


def test_fp8_regions_the_kernels_do_not_cover_are_rejected_on_the_host():
    # a zero point on E4M3, and E4M3 codes read by an elementwise op
    g, _ = I.fp8_conv(N=1, H=4, W=4, C=128, K=128)
    g.nodes[0].attrs["zero_point"] = 3
    with pytest.raises(abi.ByocError) as e:
        R.whole_graph_region(g).plan(152)
    assert e.value.status == abi.ERR_UNSUPPORTED
    b = I._Builder("q_relu")
    x = b.input("x", (1, 4, 4, 128))
    y = b.relu(b.quantize(x, 0.1))
    g2, _ = I._finish(b, [y], 1)
    with pytest.raises(abi.ByocError) as e:
        R.whole_graph_region(g2).plan(152)
    assert e.value.status == abi.ERR_UNSUPPORTED
    # FP8 on fewer than 128 channels per k-block
    g3, _ = I.fp8_conv(N=1, H=4, W=4, C=64, K=64)
    with pytest.raises(abi.ByocError):
        R.whole_graph_region(g3).plan(152)


# ------------------------------------------------------------ GPU parity

@pytest.mark.gpu
@pytest.mark.parametrize("plan", sorted(PLANS))
@pytest.mark.parametrize("N,H,W,C", [(2, 9, 11, 256), (1, 7, 7, 128), (3, 14, 14, 512)])
def test_fp8_identity_conv_reproduces_the_quantized_input_bit_for_bit(N, H, W, C, plan):
    g, inp = _identity_fp8_conv(N=N, H=H, W=W, C=C)
    got, cr = run_region(R.whole_graph_region(g, options=PLANS[plan]), inp)
    ref = ograph.evaluate(g, inp)[g.outputs[0]]
    assert_bit_exact(got[g.outputs[0]], ref, f"fp8 identity {N}x{H}x{W}x{C}")
    cr.release()


FP8_LAYERS = {
    "conv3x3": lambda: I.fp8_conv(N=2, H=14, W=14, C=256, K=256, k=3),
    "conv1x1_ragged": lambda: I.fp8_conv(N=3, H=9, W=10, C=128, K=96, k=1),
    "dense": lambda: I.fp8_dense(M=200, D=768, F=1024),
    "dense_split_k": lambda: I.fp8_dense(M=256, D=3072, F=768),
    # two k-blocks per tile, 1024 tiles over a grid that is a multiple of the
    # 8 column tiles: every CTA keeps its weight k-blocks in the ring
    "dense_short_k_weight_reuse": lambda: I.fp8_dense(M=16384, D=256, F=512),
    # the BERT FFN with Q nodes before both dense layers (config 2 in FP8):
    # the hidden codes come from the first epilogue, the second dense splits K
    "ffn": lambda: I.fp8_ffn(),
}


@pytest.mark.gpu
@pytest.mark.parametrize("plan", sorted(PLANS))
@pytest.mark.parametrize("name", sorted(FP8_LAYERS))
def test_fp8_layer_matches_the_oracle(name, plan):
    g, inp = FP8_LAYERS[name]()
    got, cr = run_region(R.whole_graph_region(g, options=PLANS[plan]), inp)
    ref, sc = oracle(g, inp)
    o = g.outputs[0]
    assert_close(got[o], ref[o], sc[o], g.name)
    cr.release()


@pytest.mark.gpu
@pytest.mark.parametrize("plan", sorted(PLANS))
@pytest.mark.parametrize("N", [2, 32])
def test_fp8_bottleneck_matches_the_oracle(N, plan):
    # config 4 with Q nodes before each convolution: the intermediates t1, t2
    # leave their epilogues as E4M3 codes (fused Q nodes)
    g, inp = I.fp8_bottleneck(N=N)
    got, cr = run_region(R.whole_graph_region(g, options=PLANS[plan]), inp)
    assert cr.n_launches == (2 if plan == "region_kernel" else 4)
    ref, sc = oracle(g, inp)
    o = g.outputs[0]
    _, _, literal = assert_close(got[o], ref[o], sc[o], g.name)
    # re-rounded codes rarely land on the other side of a rounding boundary:
    # nearly every element also meets the stated bar alone
    assert literal > 0.98, literal
    # quantization error of the whole region against the bf16 model (reported)
    gb, _ = I.resnet_bottleneck(N=N, seed=3)
    full = ograph.evaluate(gb, inp)[gb.outputs[0]]
    rel = np.linalg.norm(got[o] - full) / np.linalg.norm(full)
    print(f"fp8 bottleneck N={N}: relative L2 error against the unquantized region {rel:.4f}")
    assert rel < 0.1
    cr.release()


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["bottleneck"] + sorted(n for n in FP8_LAYERS if n != "ffn"))
def test_fp8_per_composite_equals_the_region_kernel_on_small_integers(name):
    # the two kernels issue different tile shapes (and split-K) over the same
    # codes; with exact sums and the same epilogue arithmetic the bits agree.
    # (Not the FFN: its second dense reads GELU outputs, whose codes are not
    # multiples of one power of two, so its fp32 sums are not exact and the
    # split-K order of the per-composite plan changes their rounding.)
    g, _ = I.fp8_bottleneck(N=2) if name == "bottleneck" else FP8_LAYERS[name]()
    inp = _int_fp8(g, seed=len(name))
    pc, c1 = run_region(R.whole_graph_region(g), inp)
    rk, c2 = run_region(R.whole_graph_region(g, options=RK), inp)
    for o in g.outputs:
        assert np.array_equal(pc[o].view(np.uint32), rk[o].view(np.uint32)), o
    c1.release()
    c2.release()


# ------------------------------------------------------------ more FP8 shapes

def _fp8_conv_residual(N=2, H=14, W=14, C=128, seed=41):
    """Q(x) -> 3x3 conv -> BN -> + x -> ReLU: the im2col mode with a bf16 residual tile."""
    b = I._Builder("fp8_conv3x3_residual")
    x = b.input("x", (N, H, W, C))
    y = b.relu(b.add(b.batch_norm(b.conv2d(b.quantize(x, I.FP8_SCALE_INPUT), C, 3)), x))
    return I._finish(b, [y], seed)


def _fp8_conv_stride2(N=2, H=15, W=15, C=256, K=128, seed=42):
    """Q(x) -> 3x3 stride-2 conv -> BN -> ReLU (im2col with a stride, ragged last m-tile)."""
    b = I._Builder("fp8_conv3x3_s2")
    x = b.input("x", (N, H, W, C))
    y = b.relu(b.batch_norm(b.conv2d(b.quantize(x, I.FP8_SCALE_INPUT), K, 3, stride=2)))
    return I._finish(b, [y], seed)


def _fp8_mlp(M=256, D=3072, F=768, U=256, seed=43):
    """Q(x) -> dense (split-K) + bias + ReLU -> Q -> dense + bias: the first
    layer's split-K epilogue writes the E4M3 codes the second one reads."""
    b = I._Builder("fp8_mlp")
    x = b.input("x", (M, D))
    h = b.relu(b.bias_add(b.dense(b.quantize(x, I.FP8_SCALE_INPUT), F)))
    y = b.bias_add(b.dense(b.quantize(h, I.FP8_SCALE_HIDDEN), U))
    return I._finish(b, [y], seed)


def _fp8_two_readers(N=2, H=9, W=11, C=128, seed=44):
    """t = ReLU(BN(conv1x1(Q(x)))) is a region output and also feeds Q -> conv:
    its Q node cannot be fused into the producing epilogue (a quantize launch)."""
    b = I._Builder("fp8_two_readers")
    x = b.input("x", (N, H, W, C))
    t = b.relu(b.batch_norm(b.conv2d(b.quantize(x, I.FP8_SCALE_INPUT), C, 1)))
    y = b.batch_norm(b.conv2d(b.quantize(t, I.FP8_SCALE_HIDDEN), C, 1))
    return I._finish(b, [t, y], seed)


MORE = {"conv3x3_residual": _fp8_conv_residual, "conv3x3_stride2": _fp8_conv_stride2,
        "mlp_split_k_q": _fp8_mlp, "two_readers": _fp8_two_readers}


def test_fp8_more_plans():
    rep = R.whole_graph_region(_fp8_conv_residual()[0]).plan(152)
    assert [rep.kind[i] for i in range(rep.n_launches)] == [abi.LAUNCH_QUANT, abi.LAUNCH_GEMM]
    assert rep.im2col[1] == 1 and rep.residual[1] >= 0 and rep.fp8[1] == 1
    rep = R.whole_graph_region(_fp8_conv_stride2()[0]).plan(152)
    assert rep.im2col[1] == 1 and rep.fp8[1] == 1
    # the hidden Q node is fused into the split-K layer's epilogue: no second quantize launch
    rep = R.whole_graph_region(_fp8_mlp()[0]).plan(152)
    assert [rep.kind[i] for i in range(rep.n_launches)] == [abi.LAUNCH_QUANT, abi.LAUNCH_GEMM, abi.LAUNCH_GEMM]
    assert rep.splits[1] > 1 and rep.fp8[1] == 1 and rep.fp8[2] == 1
    # t is an output: its Q node is a launch of its own
    rep = R.whole_graph_region(_fp8_two_readers()[0]).plan(152)
    assert [rep.kind[i] for i in range(rep.n_launches)] == [abi.LAUNCH_QUANT, abi.LAUNCH_GEMM, abi.LAUNCH_QUANT,
                                                            abi.LAUNCH_GEMM]


@pytest.mark.gpu
@pytest.mark.parametrize("name", sorted(MORE))
def test_fp8_more_shapes_match_the_oracle(name):
    g, inp = MORE[name]()
    got, cr = run_region(R.whole_graph_region(g), inp)
    ref, sc = oracle(g, inp)
    for o in g.outputs:
        assert_close(got[o], ref[o], sc[o], f"{name} {o}")
    cr.release()


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["conv3x3_residual", "conv3x3_stride2", "mlp_split_k_q"])
def test_fp8_more_shapes_per_composite_equals_the_region_kernel_on_small_integers(name):
    g, _ = MORE[name]()
    inp = _int_fp8(g, seed=len(name))
    pc, c1 = run_region(R.whole_graph_region(g), inp)
    rk, c2 = run_region(R.whole_graph_region(g, options=RK), inp)
    assert c2.n_launches == 2  # the quantize launch and one region kernel
    for o in g.outputs:
        assert np.array_equal(pc[o].view(np.uint32), rk[o].view(np.uint32)), o
    c1.release()
    c2.release()


@pytest.mark.gpu
def test_fp8_ffn_quantization_error_against_the_bf16_region():
    # config 2 with Q nodes before both dense layers, against the unquantized
    # FFN of the same constants (reported; a loose bound)
    g, inp = I.fp8_ffn()
    got, cr = run_region(R.whole_graph_region(g), inp)
    gb, _ = I.bert_ffn(seed=1)
    full = ograph.evaluate(gb, inp)[gb.outputs[0]]
    o = g.outputs[0]
    rel = np.linalg.norm(got[o] - full) / np.linalg.norm(full)
    print(f"fp8 FFN: relative L2 error against the unquantized region {rel:.4f}")
    assert rel < 0.1
    cr.release()
