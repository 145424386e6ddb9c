"""The parity rule of tests/parity.py, checked on the CPU.

An emulation of bf16-storage arithmetic -- every conv2d / dense weight folded
with the batch norm that follows it and rounded to bf16 (depthwise weights to
fp32, as the depthwise kernel keeps them), every tensor the oracle's error
model stores rounded to bf16, exact sums -- must stay within the oracle's
error scale on the workloads' shapes, and plausible mistakes (a wrong scale on
one channel, one wrong element, a flipped filter, a dropped bias) must fail
the rule."""
import copy

import numpy as np
import pytest

from oracle import graph as ograph
from oracle import ops
from paper_2105_03215_gb300 import inputs as I

from .parity import LAM, assert_close, oracle


def _emulate(g, inp):
    g = copy.deepcopy(g)
    readers = {}
    for n in g.nodes:
        for i in n.inputs:
            readers.setdefault(i, []).append(n)
    for n in g.nodes:
        if n.op not in ("nn.conv2d", "nn.dense"):
            continue
        w = n.consts["weight"].astype(np.float64)
        s = np.ones(w.shape[0])
        cur = n.name
        while len(readers.get(cur, [])) == 1 and readers[cur][0].op in ("nn.bias_add", "nn.batch_norm"):
            nx = readers[cur][0]
            if nx.op == "nn.batch_norm":
                s = s * nx.consts["gamma"] / np.sqrt(nx.consts["moving_var"].astype(np.float64) + 1e-5)
            cur = nx.name
        shp = (-1,) + (1,) * (w.ndim - 1)
        folded = w * s.reshape(shp)
        if n.op == "nn.conv2d" and n.attrs["groups"] > 1:
            folded = folded.astype(np.float32).astype(np.float64)
        else:
            folded = ops.round_bf16(folded)
        n.consts["weight"] = folded / s.reshape(shp)
    env = {k: np.asarray(v, np.float64) for k, v in inp.items()}
    for n in g.nodes:
        v = ograph.eval_node(n, [env[i] for i in n.inputs])
        rd = readers.get(n.name, [])
        if n.name in g.outputs or len(rd) != 1 or rd[0].op in ("nn.conv2d", "nn.dense", "nn.max_pool2d",
                                                                 "nn.global_avg_pool2d"):
            v = ops.round_bf16(v)
        env[n.name] = v
    return {o: env[o] for o in g.outputs}


CASES = {
    "conv3x3_bias_relu": lambda: I.conv_bias_relu(N=1, H=28, W=28, C=64, K=64, seed=0),
    "bert_ffn": lambda: I.bert_ffn(M=64, D=256, F=512, seed=1),
    "mbv2_dw_pw": lambda: I.mbv2_dw_pw(N=1, H=28, W=28, C=144, Cout=24, seed=2),
    "bottleneck": lambda: I.resnet_bottleneck(N=1, H=14, W=14, C=256, width=64, seed=3),
    "bottleneck_stride2": lambda: I.resnet_bottleneck(N=1, H=14, W=14, C=256, width=64, stride=2, seed=3),
    "gelu_conv": lambda: I.conv_bias_relu(N=1, H=10, W=10, C=64, K=64, seed=5, act="gelu"),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_bf16_storage_emulation_stays_within_the_error_scale(name):
    g, inp = CASES[name]()
    ref, sc = oracle(g, inp)
    emu = _emulate(g, inp)
    for o in g.outputs:
        ratio = np.abs(emu[o] - ref[o]) / np.maximum(sc[o], 1e-300)
        assert ratio.max() <= LAM / 2, (name, float(ratio.max()))
        assert_close(emu[o], ref[o], sc[o], name)


def _planted(kind, g, inp):
    out = dict(_emulate(g, inp))
    o = g.outputs[0]
    y = out[o].copy()
    if kind == "channel_scale":      # one channel's fold off by 10%
        y[..., 5] *= 1.10
    elif kind == "one_element":      # one output wrong by 0.2
        y.reshape(-1)[y.size // 3] += 0.2
    elif kind == "flipped_filter":   # filter read back to front (orientation)
        g2 = copy.deepcopy(g)
        g2.nodes[0].consts["weight"] = g2.nodes[0].consts["weight"][:, :, ::-1, ::-1].copy()
        y = _emulate(g2, inp)[o]
    elif kind == "dropped_bias":     # bias not added to one channel
        b = g.nodes[1].consts["bias"]
        y[..., 7] = ops.round_bf16(np.maximum(ref_pre(g, inp)[..., 7] - b[7], 0.0))
    out[o] = y
    return out


def ref_pre(g, inp):
    # the oracle's pre-activation value (conv + bias) of the conv_bias_relu graph
    return ograph.evaluate(g, inp, keep=[g.nodes[1].name])[g.nodes[1].name]


@pytest.mark.parametrize("kind", ["channel_scale", "one_element", "flipped_filter", "dropped_bias"])
def test_planted_mistakes_fail_the_rule(kind):
    g, inp = I.conv_bias_relu(N=1, H=28, W=28, C=64, K=64, seed=7)
    ref, sc = oracle(g, inp)
    bad = _planted(kind, g, inp)
    o = g.outputs[0]
    with pytest.raises(AssertionError):
        assert_close(bad[o], ref[o], sc[o], kind)


def test_resnet50_end_to_end_bf16_storage_error_is_small():
    # End to end through 54 regions the per-element error scale outgrows the
    # values themselves (the random-init network amplifies every rounding), so
    # the end-to-end logits are gated by relative L2 instead: bf16-storage
    # arithmetic lands within 1.5% of the fp64 oracle here (measured 0.60%),
    # the number the GPU end-to-end test's 3% gate is set from
    from paper_2105_03215_gb300 import executor as E
    res, inp = E.build_resnet50(N=2, H=64, W=64)
    g = res.graph
    ref = ograph.evaluate(g, inp)[g.outputs[0]]
    em = _emulate(g, inp)[g.outputs[0]]
    rel = np.linalg.norm(em - ref) / np.linalg.norm(ref)
    assert 1e-4 < rel < 0.015, rel


def test_mobilenet_v2_end_to_end_bf16_storage_error():
    # The same for MobileNetV2 (N=2, 96x96): this random-init network
    # amplifies rounding far more (ReLU6 clipping, depthwise layers) --
    # bf16-storage arithmetic lands 11.7% from the fp64 oracle end to end,
    # the figure the GPU end-to-end test's 20% gate is set from
    from paper_2105_03215_gb300 import executor as E
    res, inp = E.build_mobilenet_v2(N=2, H=96, W=96)
    g = res.graph
    ref = ograph.evaluate(g, inp)[g.outputs[0]]
    em = _emulate(g, inp)[g.outputs[0]]
    rel = np.linalg.norm(em - ref) / np.linalg.norm(ref)
    assert 0.01 < rel < 0.15, rel
