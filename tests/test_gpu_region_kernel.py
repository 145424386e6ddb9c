"""The region kernel (BYOC_OPT_REGION_KERNEL): a region's whole chain of
conv2d / dense composites -- the ResNet-50 bottleneck with or without its
downsample branch, the BERT FFN -- in one persistent launch, against the fp64
oracle and against the per-composite plan of the same region."""
import numpy as np
import pytest

from paper_2105_03215_gb300 import abi
from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import region as R

from .parity import assert_close, oracle, run_region

OPT = abi.OPT_REGION_KERNEL

CASES = {
    "bottleneck_2x14x14x256": lambda: I.resnet_bottleneck(N=2, H=14, W=14, C=256, width=64, seed=3),
    "bottleneck_stride2_downsample": lambda: I.resnet_bottleneck(N=2, H=14, W=14, C=256, width=128, stride=2,
                                                                 seed=4),
    "bottleneck_28x28_ragged": lambda: I.resnet_bottleneck(N=3, H=28, W=28, C=256, width=64, seed=5),
    "ffn_small": lambda: I.bert_ffn(M=256, D=256, F=512, seed=1),
    "ffn_ragged_rows": lambda: I.bert_ffn(M=200, D=128, F=384, seed=2),
}


def _int_consts(g, seed):
    """Small-integer weights and inputs, batch norm with unit scale: every
    fp32 sum is an exact integer, so any correct plan gives the same bits."""
    rng = np.random.Generator(np.random.PCG64(seed))
    for n in g.nodes:
        if n.op in ("nn.conv2d", "nn.dense"):
            n.consts["weight"] = rng.integers(-1, 2, size=n.attrs["weight_shape"]).astype(np.float32)
        elif n.op == "nn.batch_norm":
            C = n.shape[-1]
            n.consts.update(gamma=np.ones(C, np.float32), beta=rng.integers(-4, 5, C).astype(np.float32),
                            moving_mean=np.zeros(C, np.float32), moving_var=np.ones(C, np.float32))
        elif n.op == "nn.bias_add":
            n.consts["bias"] = rng.integers(-4, 5, n.shape[-1]).astype(np.float32)
    return {k: rng.integers(-2, 3, size=g.shape_of(k)).astype(np.float32) for k in g.inputs}


# ------------------------------------------------------------ plans (CPU)

@pytest.mark.parametrize("name,stages,units", [
    ("bottleneck_2x14x14x256", 3, 4 * 1 + 4 * 1 + 4 * 2),
    ("bottleneck_stride2_downsample", 4, 4 + 1 + 1 * 4 + 1 * 4),
    ("ffn_small", 2, 2 * 4 + 2 * 2),
])
def test_region_kernel_plan_is_one_launch(name, stages, units):
    g, _ = CASES[name]()
    rep = R.whole_graph_region(g, options=OPT).plan(152)
    assert rep.n_launches == 1 and rep.kind[0] == abi.LAUNCH_CHAIN
    assert rep.stages[0] == stages and rep.units[0] == units and rep.tile_n[0] == 128
    base = R.whole_graph_region(g).plan(152)
    assert abs(rep.flops - base.flops) < 1e-6 * base.flops
    # the region's intermediates stay out of the algorithmic bytes: inputs,
    # outputs and weights once
    assert rep.bytes < base.bytes


def test_region_kernel_plan_serialises():
    g, _ = CASES["bottleneck_stride2_downsample"]()
    reg = R.whole_graph_region(g, options=OPT)
    blob = reg.plan_serialized(152)
    rep = R.load_plan_report(blob)
    assert rep.n_launches == 1 and rep.kind[0] == abi.LAUNCH_CHAIN and rep.stages[0] == 4


def test_regions_the_kernel_does_not_cover_keep_the_per_composite_plan():
    # a stem (3 input channels) and a depthwise region fall back
    g, _ = I.mbv2_dw_pw(N=1, H=8, W=8)
    rep = R.whole_graph_region(g, options=OPT).plan(152)
    assert abi.LAUNCH_CHAIN not in [rep.kind[i] for i in range(rep.n_launches)]
    g, _ = I.stem(N=1, H=32, W=32)
    rep = R.whole_graph_region(g, options=OPT).plan(152)
    assert abi.LAUNCH_CHAIN not in [rep.kind[i] for i in range(rep.n_launches)]
    # a single composite is not a chain
    g, _ = I.conv_bias_relu(N=1, H=8, W=8, C=64, K=64)
    rep = R.whole_graph_region(g, options=OPT).plan(152)
    assert rep.kind[0] == abi.LAUNCH_GEMM


# ------------------------------------------------------------ GPU parity

@pytest.mark.gpu
@pytest.mark.parametrize("name", sorted(CASES))
def test_region_kernel_matches_the_oracle(name):
    g, inp = CASES[name]()
    reg = R.whole_graph_region(g, options=OPT)
    got, cr = run_region(reg, inp)
    assert cr.n_launches == 1
    ref, sc = oracle(g, inp)
    for o in g.outputs:
        assert_close(got[o], ref[o], sc[o], name)
    cr.release()


@pytest.mark.gpu
@pytest.mark.parametrize("make", [I.resnet_bottleneck, I.bert_ffn])
def test_region_kernel_at_the_workload_size(make):
    # config 4 (N=32, 14x14, 1024 -> 256 -> 1024) and config 2 (1024 x 768 -> 3072 -> 768)
    g, inp = make(seed=3 if make is I.resnet_bottleneck else 1)
    reg = R.whole_graph_region(g, options=OPT)
    got, cr = run_region(reg, inp)
    assert cr.n_launches == 1
    ref, sc = oracle(g, inp)
    assert_close(got[g.outputs[0]], ref[g.outputs[0]], sc[g.outputs[0]], g.name)
    cr.release()


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["bottleneck_2x14x14x256", "bottleneck_stride2_downsample", "ffn_small"])
def test_region_kernel_equals_the_per_composite_plan_on_small_integers(name):
    g, _ = CASES[name]()
    inp = _int_consts(g, seed=len(name))
    fused, cf = run_region(R.whole_graph_region(g, options=OPT), inp)
    split, cs = run_region(R.whole_graph_region(g), inp)
    assert cf.n_launches == 1 and cs.n_launches > 1
    for o in g.outputs:
        assert np.array_equal(fused[o].view(np.uint32), split[o].view(np.uint32)), o
    cf.release()
    cs.release()


@pytest.mark.gpu
def test_region_kernel_repeats_and_replays_in_a_graph():
    # every launch counts its units' flags one run further: eager runs, then
    # a captured graph replayed, give the same bits each time
    import torch
    from .parity import to_dev
    g, inp = CASES["bottleneck_stride2_downsample"]()
    cr = R.whole_graph_region(g, options=OPT).compile()
    x = to_dev(inp["x"])
    y = torch.empty(g.shape_of(g.outputs[0]), dtype=torch.bfloat16, device="cuda")
    outs = []
    for _ in range(3):
        y.fill_(float("nan"))
        cr.run([x], [y])
        torch.cuda.synchronize()
        cr.check()
        outs.append(y.clone())
    graph = torch.cuda.CUDAGraph()
    st = torch.cuda.Stream()
    with torch.cuda.graph(graph, stream=st):
        cr.run([x], [y], st)
    for _ in range(3):
        y.fill_(float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        cr.check()
        outs.append(y.clone())
    for o in outs[1:]:
        assert torch.equal(o, outs[0])
    ref, sc = oracle(g, inp)
    assert_close(outs[0].float().cpu().numpy(), ref[g.outputs[0]], sc[g.outputs[0]], "repeat")
    cr.release()


@pytest.mark.gpu
def test_resnet50_bottleneck_regions_as_region_kernels_teacher_forced():
    # ResNet-50 cut at most 4 composites per region (one region per
    # bottleneck): every qualifying region runs as one region kernel; each
    # region's outputs against the oracle fed the GPU's own inputs
    import torch
    from oracle import graph as ograph  # noqa: F401
    from paper_2105_03215_gb300 import executor as E
    res, inp = E.build_resnet50(N=2, H=64, W=64, max_ops=4)
    ex = E.Executor(res, options=OPT)
    n_chain = sum(c.n_launches == 1 and len(r.nodes) > 5 for c, r in zip(ex.compiled, ex.regions))
    assert n_chain >= 8, n_chain
    ex.set_input("data", torch.from_numpy(inp["data"]).to(torch.bfloat16).cuda())
    ex.run_steps()
    torch.cuda.synchronize()
    ex.check()
    g = ex.graph
    for r in ex.regions:
        feed = {n: ex.entries[n].float().cpu().numpy().astype(np.float64) for n in r.inputs}
        ref, sc = oracle(g, feed, nodes=[n.name for n in r.nodes], keep=r.outputs)
        for o in r.outputs:
            assert_close(ex.entries[o].float().cpu().numpy(), ref[o], sc[o], f"{r.name}:{o}")
    ex.release()
