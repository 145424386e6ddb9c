"""MobileNetV2 1.0 partitioned into 53 regions (conv2d composites with
stride-1 and stride-2 depthwise convolutions, linear projections with a fused
residual add, and the classifier), global average pool on the host, run by the
executor.  Parity per region, teacher-forced, as for ResNet-50."""
import numpy as np
import pytest

from oracle import graph as ograph
from paper_2105_03215_gb300 import executor as E

from .parity import assert_close, oracle

pytestmark = pytest.mark.gpu


def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


def test_mobilenet_v2_small_image_every_region_teacher_forced():
    import torch
    res, inp = E.build_mobilenet_v2(N=2, H=96, W=96)
    assert len(res.regions) == 53
    ex = E.Executor(res)
    ex.set_input("data", torch.from_numpy(inp["data"]).to(torch.bfloat16).cuda())
    ex.run_steps()
    torch.cuda.synchronize()
    ex.check()
    g = ex.graph
    for r in ex.regions:
        feed = {n: _f64(ex.entries[n]) for n in r.inputs}
        ref, sc = oracle(g, feed, nodes=[n.name for n in r.nodes], keep=r.outputs)
        for o in r.outputs:
            assert_close(_f64(ex.entries[o]), ref[o], sc[o], f"{r.name}:{o}")
    # end to end: a CPU emulation of bf16 storage lands 11.7% (relative L2)
    # from the fp64 oracle on this random-init network (tests/test_tolerance.py)
    full = ograph.evaluate(g, inp)[g.outputs[0]]
    got = _f64(ex.output())
    rel = np.linalg.norm(got - full) / np.linalg.norm(full)
    print(f"mobilenet_v2 N=2 96x96 end-to-end logits relative L2 error {rel:.4f}")
    assert rel < 0.2
    ex.release()


def test_mobilenet_v2_graph_replay_equals_eager():
    import torch
    res, inp = E.build_mobilenet_v2(N=2, H=96, W=96)
    ex = E.Executor(res)
    ex.set_input("data", torch.from_numpy(inp["data"]).to(torch.bfloat16).cuda())
    ex.run_steps()
    torch.cuda.synchronize()
    eager = ex.output().clone()
    ex.output().fill_(float("nan"))
    ex.capture()
    ex.replay()
    torch.cuda.synchronize()
    ex.check()
    assert torch.equal(ex.output(), eager)
    ex.release()


def test_mobilenet_v2_fused_regions_match_one_composite_per_region_bit_for_bit():
    # the whole network as one region (+ the classifier): 11 of the 17
    # depthwise -> 1x1 pairs run as fused kernels, and the logits are the same
    # bits as with every composite in a region of its own
    import torch
    from paper_2105_03215_gb300 import abi
    outs = []
    for mo in (1, None):
        res, inp = E.build_mobilenet_v2(N=2, H=96, W=96, max_ops=mo)
        ex = E.Executor(res, options=abi.OPT_FUSE_DW_PW)
        ex.set_input("data", torch.from_numpy(inp["data"]).to(torch.bfloat16).cuda())
        ex.run_steps()
        torch.cuda.synchronize()
        ex.check()
        outs.append((ex.n_launches, ex.output().clone()))
        ex.release()
    assert outs[1][0] < outs[0][0]
    assert torch.equal(outs[0][1], outs[1][1])
