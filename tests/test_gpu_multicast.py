"""Cluster multicast of the weight tiles (BYOC_OPT_MULTICAST): clusters of
two CTAs take adjacent m-tiles of one column tile and share each weight tile
by TMA multicast.  The same MMAs run
in the same order either way, so the two plans must give identical bits; and
both must match the fp64 oracle.  Cases cover every multicast mode (tile,
tile + residual, im2col, ringed slab, dense) and odd m-tile counts, where the
last cluster's second CTA runs a phantom m-tile past the end."""
import numpy as np
import pytest

from paper_2105_03215_gb300 import abi
from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import region as R

from .parity import assert_close, oracle, run_region

MC = abi.OPT_MULTICAST

CASES = {
    # 1x1 conv, tile mode, M = 320: three m-tiles (one phantom)
    "tile_1x1_odd_m": lambda: I.conv_bias_relu(N=1, H=16, W=20, C=64, K=256, k=1, pad=0, seed=21),
    # bottleneck: 1x1, 3x3 slab and 1x1 + residual (tile mode with a residual tile)
    "bottleneck_n1": lambda: I.resnet_bottleneck(N=1, H=14, W=14, C=256, width=64, seed=22),
    # stride-2 3x3 (im2col mode) and the strided 1x1 downsample branch
    "bottleneck_stride2": lambda: I.resnet_bottleneck(N=2, H=14, W=14, C=256, width=128, stride=2, seed=23),
    # 3x3 slab mode, 7 slab tiles per image (odd)
    "slab_3x3_odd_units": lambda: I.conv_bias_relu(N=1, H=28, W=28, C=128, K=128, k=3, seed=24),
    # dense layers, M = 384: three m-tiles
    "ffn_odd_m": lambda: I.bert_ffn(M=384, D=256, F=512, seed=25),
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

@pytest.mark.parametrize("name", sorted(CASES))
def test_multicast_plans_pair_ctas_on_request(name):
    g, _ = CASES[name]()
    on = R.whole_graph_region(g, options=MC).plan(152)
    off = R.whole_graph_region(g).plan(152)
    assert on.n_launches == off.n_launches
    n_mc = 0
    for i in range(on.n_launches):
        assert off.multicast[i] == 0
        if on.multicast[i]:
            n_mc += 1
            assert on.kind[i] == abi.LAUNCH_GEMM and on.splits[i] == 1 and on.resident_b[i] == 0
            assert on.grid[i] % 2 == 0 and 2 <= on.grid[i] <= 152
            assert on.tile_n[i] == off.tile_n[i]
    assert n_mc >= 1


def test_multicast_grid_covers_the_tile_pairs():
    # FFN first layer: 8 m-tiles (4 pairs) x 3072 / BN column tiles, at most
    # 76 clusters of two on 152 SMs
    g, _ = I.bert_ffn()
    rep = R.whole_graph_region(g, options=MC).plan(152)
    assert rep.multicast[0] == 1 and rep.grid[0] == 2 * min(4 * (3072 // rep.tile_n[0]), 76)
    # three m-tiles pair up as (0, 1) and (2, phantom): 2 pairs x 4 column tiles of 64
    g, _ = CASES["tile_1x1_odd_m"]()
    rep = R.whole_graph_region(g, options=MC).plan(152)
    if rep.multicast[0]:
        tiles_n = -(-256 // rep.tile_n[0])
        assert rep.grid[0] == 2 * min(2 * tiles_n, 76)


# ------------------------------------------------------------ GPU parity

@pytest.mark.gpu
@pytest.mark.parametrize("name", sorted(CASES))
def test_multicast_equals_the_unshared_plan_bit_for_bit(name):
    g, _ = CASES[name]()
    inp = _int_consts(g, seed=len(name))
    on, con = run_region(R.whole_graph_region(g, options=MC), inp)
    off, coff = run_region(R.whole_graph_region(g), inp)
    for o in g.outputs:
        assert np.array_equal(on[o].view(np.uint32), off[o].view(np.uint32)), o
    con.release()
    coff.release()


@pytest.mark.gpu
@pytest.mark.parametrize("name", sorted(CASES))
def test_multicast_matches_the_oracle(name):
    g, inp = CASES[name]()
    got, cr = run_region(R.whole_graph_region(g, options=MC), inp)
    ref, sc = oracle(g, inp)
    for o in g.outputs:
        assert_close(got[o], ref[o], sc[o], name)
    cr.release()


@pytest.mark.gpu
def test_multicast_repeats_in_a_graph():
    # clusters are launched again on every replay: same bits each time
    import torch
    from .parity import to_dev
    g, inp = CASES["bottleneck_stride2"]()
    cr = R.whole_graph_region(g, options=MC).compile()
    x = to_dev(inp["x"])
    y = torch.empty(g.shape_of(g.outputs[0]), dtype=torch.bfloat16, device="cuda")
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        cr.run([x], [y], st)
    torch.cuda.synchronize()
    first = y.clone()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=st):
        cr.run([x], [y], st)
    for _ in range(3):
        y.fill_(float("nan"))
        graph.replay()
        torch.cuda.synchronize()
        cr.check()
        assert torch.equal(y, first)
    cr.release()
