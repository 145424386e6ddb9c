"""Evaluate an op list in fp64, node by node, with the oracle's operators.

TEST INFRASTRUCTURE.  The chain is evaluated exactly as written: batch norm
stays a separate operator with the original fp32 statistics, weights keep
their fp32 values (no folding, no bf16 rounding), and intermediates stay
fp64.  Only graph inputs arrive bf16-rounded (the generator rounds them),
which is the "partial quantization" cast at the offload boundary
(Section 3.2, Q nodes: here an fp32 -> bf16 cast).
"""
from __future__ import annotations

from typing import Dict, Iterable, Optional

import numpy as np

from . import ops


def eval_node(node, args):
    op, a, c = node.op, node.attrs, node.consts
    if op == "nn.conv2d":
        return ops.conv2d_nhwc(args[0], c["weight"], tuple(a["strides"]), tuple(a["padding"]),
                               tuple(a["dilation"]), int(a["groups"]))
    if op == "nn.dense":
        return ops.dense(args[0], c["weight"])
    if op == "nn.bias_add":
        return ops.bias_add(args[0], c["bias"])
    if op == "nn.batch_norm":
        return ops.batch_norm(args[0], c["gamma"], c["beta"], c["moving_mean"], c["moving_var"],
                              float(a.get("epsilon", 1e-5)))
    if op == "nn.relu":
        return ops.relu(args[0])
    if op == "clip":
        if float(a["a_min"]) == 0.0 and float(a["a_max"]) == 6.0:
            return ops.relu6(args[0])
        return np.clip(np.asarray(args[0], dtype=np.float64), float(a["a_min"]), float(a["a_max"]))
    if op == "nn.gelu":
        return ops.gelu(args[0])
    if op == "add":
        return ops.add(args[0], args[1])
    if op == "nn.max_pool2d":
        return ops.max_pool2d_nhwc(args[0], tuple(a["pool_size"]), tuple(a["strides"]),
                                   tuple(a["padding"]))
    if op == "nn.global_avg_pool2d":
        return ops.global_avg_pool_nhwc(args[0])
    raise NotImplementedError(op)


def evaluate(graph, inputs: Dict[str, np.ndarray], nodes: Optional[Iterable[str]] = None,
             keep: Optional[Iterable[str]] = None) -> Dict[str, np.ndarray]:
    """Evaluate ``nodes`` (default: all) of ``graph`` in graph order.

    ``inputs`` maps tensor names (graph inputs, or boundary tensors of a
    region) to arrays.  Returns every computed tensor named in ``keep``
    (default: the graph outputs that were computed)."""
    env = {k: np.asarray(v, dtype=np.float64) for k, v in inputs.items()}
    wanted = set(nodes) if nodes is not None else None
    for n in graph.nodes:
        if wanted is not None and n.name not in wanted:
            continue
        env[n.name] = eval_node(n, [env[i] for i in n.inputs])
    names = list(keep) if keep is not None else [o for o in graph.outputs if o in env]
    return {k: env[k] for k in names}
