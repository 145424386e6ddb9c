"""Split-K through a thread-block cluster (BYOC_OPT_CLUSTER_SPLIT_K): the CTAs
that share a tile's k-blocks form one cluster and exchange their fp32 partial
accumulators through distributed shared memory; each CTA sums the partials of
the 32-column chunks it owns in split order and runs their epilogue.  Against
the default split-K (partials through the workspace), which sums in the same
order, the bits must be identical; with small-integer data both
must equal the bf16 rounding of the exact result; with general data both must
match the fp64 oracle."""
import numpy as np
import pytest

from paper_2105_03215_gb300 import abi
from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import region as R

from .parity import assert_close, oracle, run_region

CLUSTER = abi.OPT_CLUSTER_SPLIT_K

# (M, K, N): the BERT FFN's second dense (3 splits of 128-wide tiles), the
# ResNet-50 classifier (4 splits of 64-wide tiles, ragged N), ragged M, a
# single row tile, and a 2-way split
SHAPES = [(1024, 3072, 768), (64, 2048, 1000), (200, 2048, 384), (7, 1024, 40), (1024, 2048, 1024)]


def _dense(M, K, N, seed):
    b = I._Builder(f"dense_{M}x{K}x{N}")
    x = b.input("x", (M, K))
    y = b.bias_add(b.dense(x, N))
    return I._finish(b, [y], seed=seed)


def _int_data(g, seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    for n in g.nodes:
        if n.op == "nn.dense":
            n.consts["weight"] = rng.integers(-1, 2, size=n.attrs["weight_shape"]).astype(np.float32)
        elif n.op == "nn.bias_add":
            n.consts["bias"] = rng.integers(-4, 5, n.shape[-1]).astype(np.float32)
    return {k: rng.integers(-2, 3, size=g.shape_of(k)).astype(np.float32) for k in g.inputs}


@pytest.mark.parametrize("M,K,N", SHAPES)
def test_deep_reductions_plan_a_cluster_split_on_request(M, K, N):
    g, _ = _dense(M, K, N, seed=1)
    cl = R.whole_graph_region(g, options=CLUSTER).plan(152)
    gl = R.whole_graph_region(g).plan(152)
    assert cl.splits[0] > 1 and cl.tile_n[0] <= 128
    assert cl.grid[0] <= 152 and cl.grid[0] % cl.splits[0] == 0
    # no fp32 partials in the workspace
    assert cl.workspace_bytes < gl.workspace_bytes
    assert gl.splits[0] > 1


@pytest.mark.gpu
@pytest.mark.parametrize("M,K,N", SHAPES)
def test_cluster_split_small_integers_exact_and_equal_to_global_split(M, K, N):
    g, _ = _dense(M, K, N, seed=2)
    inp = _int_data(g, seed=M + N)
    cl, ccl = run_region(R.whole_graph_region(g, options=CLUSTER), inp)
    gl, cgl = run_region(R.whole_graph_region(g), inp)
    o = g.outputs[0]
    exact = inp["x"].astype(np.float64) @ g.nodes[0].consts["weight"].astype(np.float64).T + \
        g.nodes[1].consts["bias"].astype(np.float64)
    want = I.bf16_round(exact.astype(np.float32))
    assert np.array_equal(cl[o], want)
    assert np.array_equal(cl[o].view(np.uint32), gl[o].view(np.uint32))
    ccl.release()
    cgl.release()


@pytest.mark.gpu
@pytest.mark.parametrize("M,K,N", SHAPES)
def test_cluster_split_matches_the_oracle_and_repeats(M, K, N):
    import torch
    from .parity import to_dev
    g, inp = _dense(M, K, N, seed=3)
    reg = R.whole_graph_region(g, options=CLUSTER)
    got, cr = run_region(reg, inp)
    ref, sc = oracle(g, inp)
    o = g.outputs[0]
    assert_close(got[o], ref[o], sc[o], f"dense {M}x{K}->{N}")
    out = torch.empty(g.shape_of(o), dtype=torch.bfloat16, device="cuda")
    xs = [to_dev(inp["x"])]
    for _ in range(3):
        cr.run(xs, [out])
        torch.cuda.synchronize()
        assert np.array_equal(out.float().cpu().numpy(), got[o])
    cr.check()
    cr.release()
