"""Weight tiles kept in the ring: a GEMM launch of one column tile whose
units' ring stages divide the ring loads the weights on the first pass over
the ring only (every later unit finds the same k-blocks in the same slots).
Checked bit for bit with small-integer data on launches with enough units per
CTA for many passes, over k-block counts that give 1, 2 and 3 k-blocks per
stage and units of two stages."""
import numpy as np
import pytest

from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import region as R

from .parity import run_region

# (K, N, tiles per CTA wanted): K = 64 / 128 / 192 / 320 channels, N <= the
# tile width; and two or three column tiles with a grid that is a multiple of
# them (every CTA stays in one column tile)
CASES = [(64, 24, 20), (128, 64, 12), (192, 24, 8), (320, 32, 6), (64, 144, 24), (128, 256, 16)]


def _dense_int(M, K, N, seed):
    b = I._Builder(f"dense_{M}x{K}x{N}")
    x = b.input("x", (M, K))
    y = b.bias_add(b.dense(x, N))
    g, _ = I._finish(b, [y], seed=seed, draw=False)
    rng = np.random.Generator(np.random.PCG64(seed))
    g.nodes[0].consts["weight"] = rng.integers(-1, 2, size=(N, K)).astype(np.float32)
    g.nodes[1].consts["bias"] = rng.integers(-4, 5, N).astype(np.float32)
    x = rng.integers(-2, 3, size=(M, K)).astype(np.float32)
    return g, {"x": x}


@pytest.mark.gpu
@pytest.mark.parametrize("K,N,per_cta", CASES)
def test_single_column_tile_launches_reuse_their_weights_bit_exact(K, N, per_cta):
    M = 128 * 152 * per_cta // max(1, -(-N // 64)) + 77  # a ragged last tile
    g, inp = _dense_int(M, K, N, seed=K + N)
    reg = R.whole_graph_region(g)
    rep = reg.plan(152)
    tiles_n = -(-N // rep.tile_n[0])
    assert rep.splits[0] == 1 and rep.grid[0] % tiles_n == 0  # every CTA in one column tile
    got, cr = run_region(reg, inp)
    exact = inp["x"] @ g.nodes[0].consts["weight"].T + g.nodes[1].consts["bias"]  # integers, exact in fp32
    want = I.bf16_round(exact.astype(np.float32))
    assert np.array_equal(got[g.outputs[0]], want)
    cr.release()
