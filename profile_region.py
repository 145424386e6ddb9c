"""Run one offloaded region repeatedly, for profilers (ncu) and quick timing.

  python profile_region.py --workload resnet50 --batch 64 --region 5
  python profile_region.py --workload mbv2_dw_pw --reps 5 --time
  python profile_region.py --workload fp8_bottleneck --reps 5 --time

``--region i`` picks the i-th region of ResNet-50 partitioned one composite
per region; the other workloads run as a single region.  Inputs are random
bf16 tensors of the region's boundary shapes.  With ``--time`` the median
CUDA-event time of each run (L2 flushed before each) and the region's
algorithmic TFLOP/s and GB/s are printed.
"""
from __future__ import annotations

import argparse
import os
import statistics
import sys

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="resnet50",
                    choices=["resnet50", "conv3x3", "bert_ffn", "mbv2_dw_pw", "mbv2_dw", "bottleneck",
                             "fp8_bottleneck"])
    ap.add_argument("--batch", type=int, default=64)
    ap.add_argument("--n", type=int, default=None,
                    help="batch of the other workloads (default: the workload's own)")
    ap.add_argument("--region", type=int, default=0)
    ap.add_argument("--reps", type=int, default=3)
    ap.add_argument("--warmup", type=int, default=2)
    ap.add_argument("--time", action="store_true")
    ap.add_argument("--list", action="store_true", help="list ResNet-50 regions and exit")
    ap.add_argument("--fuse-dw-pw", action="store_true",
                    help="compile with the fused depthwise -> 1x1 kernel (region option)")
    ap.add_argument("--region-kernel", action="store_true",
                    help="compile a chain of conv / dense composites as one region kernel (region option)")
    args = ap.parse_args()

    import torch

    from paper_2105_03215_gb300 import abi
    from paper_2105_03215_gb300 import inputs as I
    from paper_2105_03215_gb300 import partition as P
    from paper_2105_03215_gb300 import region as R

    if args.workload == "resnet50":
        g, _ = I.resnet50(N=args.batch, draw=False)
        res = P.partition(g, P.PATTERN_TABLE, target=P.TARGET, max_ops=1)
        if args.list:
            for i in range(len(res.regions)):
                nodes = res.region_nodes(i)
                c = g.node(nodes[0])
                print(i, nodes[0], g.shape_of(c.inputs[0]), "->", g.shape_of(nodes[-1]),
                      c.attrs.get("kernel_size"), c.attrs.get("strides"))
            return
        # draw constants only for the chosen region's nodes
        import numpy as np
        rng = np.random.default_rng(0)
        names = res.region_nodes(args.region)
        for n in g.nodes:
            if n.name not in names:
                continue
            if "weight_shape" in n.attrs:
                n.consts["weight"] = (rng.standard_normal(n.attrs["weight_shape"]) * 0.05).astype("float32")
            if n.op == "nn.bias_add":
                n.consts["bias"] = rng.uniform(-0.1, 0.1, n.shape[-1]).astype("float32")
            if n.op == "nn.batch_norm":
                C = n.shape[-1]
                n.consts.update(gamma=np.ones(C, "float32"), beta=np.zeros(C, "float32"),
                                moving_mean=np.zeros(C, "float32"), moving_var=np.ones(C, "float32"))
        reg = R.Region(g, names, f"resnet50_region{args.region}")
    else:
        nk = {} if args.n is None else {"N": args.n}
        g, _ = {"conv3x3": lambda: I.conv_bias_relu(seed=0, **nk),
                "bert_ffn": lambda: I.bert_ffn(seed=1),
                "mbv2_dw_pw": lambda: I.mbv2_dw_pw(seed=2, **nk),
                "mbv2_dw": lambda: I.mbv2_dw_pw(seed=2, **nk),
                "bottleneck": lambda: I.resnet_bottleneck(seed=3, **nk),
                "fp8_bottleneck": lambda: I.fp8_bottleneck(seed=3, **nk)}[args.workload]()
        if args.workload == "mbv2_dw":
            reg = R.Region(g, [n.name for n in g.nodes[:3]], "mbv2_dw")
        else:
            reg = R.whole_graph_region(g, options=(abi.OPT_FUSE_DW_PW if args.fuse_dw_pw else 0) |
                                       (abi.OPT_REGION_KERNEL if args.region_kernel else 0))
    cr = reg.compile()
    ins = [torch.randn(g.shape_of(n), device="cuda").to(torch.bfloat16) for n in reg.inputs]
    outs = [torch.empty(g.shape_of(n), dtype=torch.bfloat16, device="cuda") for n in reg.outputs]
    for _ in range(args.warmup):
        cr.run(ins, outs)
    torch.cuda.synchronize()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda") if args.time else None
    times = []
    for _ in range(args.reps):
        if flush is not None:
            flush.zero_()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
        cr.run(ins, outs)
        if flush is not None:
            b.record()
            torch.cuda.synchronize()
            times.append(a.elapsed_time(b) * 1e-3)
    torch.cuda.synchronize()
    cr.check()
    if times:
        t = statistics.median(times)
        print(f"{reg.name}: {t * 1e6:.1f} us  {cr.flops / t / 1e12:.1f} TFLOP/s  "
              f"{cr.bytes / t / 1e9:.0f} GB/s  ({cr.flops / 1e9:.3f} GFLOP, {cr.bytes / 1e6:.2f} MB, "
              f"{cr.n_launches} launches)")
    cr.release()


if __name__ == "__main__":
    main()
