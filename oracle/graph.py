"""Evaluate an op list in fp64, node by node, with the oracle's operators.

TEST INFRASTRUCTURE.  The chain is evaluated exactly as written: batch norm
stays a separate operator with the original fp32 statistics, weights keep
their fp32 values (no folding, no bf16 rounding), and intermediates stay
fp64.  Only graph inputs arrive bf16-rounded (the generator rounds them),
which is the "partial quantization" cast at the offload boundary
(Section 3.2, Q nodes: here an fp32 -> bf16 cast).
"""
from __future__ import annotations

from typing import Dict, Iterable, Optional, Tuple

import numpy as np

from . import ops
from . import quant

# Rounding-error model of an implementation that stores activations and
# weights in bf16 and accumulates in fp32 (the arithmetic the method's
# offloaded regions run in; Section 3.2 casts to the accelerator's type at the
# region boundary).  Each rounding of a value v is v (1 + d) with d in
# [-u, u]; the probabilistic model of rounding-error analysis takes the d of
# different roundings as independent with mean zero, so that an error
# sum_j a_j d_j has, by Hoeffding's inequality (1963),
#   P(|sum_j a_j d_j| >= lam * sqrt(sum_j a_j^2 u_j^2)) <= 2 exp(-lam^2 / 2).
# evaluate_with_error_scale propagates s^2 = sum_j a_j^2 u_j^2 per element.
U_BF16 = 2.0 ** -9   # |bf16_rne(v) - v| <= U_BF16 |v|   (8 significant bits)
U_FP32 = 2.0 ** -24  # |fp32_rne(v) - v| <= U_FP32 |v|
GELU_LIPSCHITZ = 1.13  # max |d/dx x Phi(x)| = 1.1289 (at x = sqrt 2)


def eval_node(node, args, weight=None):
    """Value of ``node`` from its inputs' values.  ``weight`` replaces the
    node's weight (the effective weights of an FP8 layer, fp8_weights)."""
    op, a, c = node.op, node.attrs, node.consts
    w = c.get("weight") if weight is None else weight
    if op == "nn.conv2d":
        return ops.conv2d_nhwc(args[0], w, tuple(a["strides"]), tuple(a["padding"]),
                               tuple(a["dilation"]), int(a["groups"]))
    if op == "nn.dense":
        return ops.dense(args[0], w)
    if op == "qnn.quantize":
        # Section 3.2 Q node: the value the next operator reads is the
        # quantized tensor's real value (code x scale)
        if a.get("dtype", "e4m3") == "e4m3":
            return quant.dequantize_e4m3(quant.quantize_e4m3(args[0], float(a["scale"])), float(a["scale"]))
        zp = int(a.get("zero_point", 0))
        return quant.dequantize_int8(quant.quantize_int8(args[0], float(a["scale"]), zp), float(a["scale"]), zp)
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


def fp8_weights(graph, nodes=None):
    """Effective weights of the FP8 layers: a conv2d / dense whose input is an
    E4M3 Q node's output computes with its weights quantized per output
    channel after folding the batch norms of its epilogue chain into them
    (oracle.quant.quantize_weights_e4m3): w_eff = w_q S_w / s, so that the
    unfolded chain conv(w_eff) -> batch norm (x s) computes with w_q S_w."""
    by = {n.name: n for n in graph.nodes}
    readers: Dict[str, list] = {}
    for n in graph.nodes:
        for i in n.inputs:
            readers.setdefault(i, []).append(n)
    out = {}
    wanted = set(nodes) if nodes is not None else None
    for n in graph.nodes:
        if n.op not in ("nn.conv2d", "nn.dense") or (wanted is not None and n.name not in wanted):
            continue
        src = by.get(n.inputs[0])
        if src is None or src.op != "qnn.quantize" or src.attrs.get("dtype", "e4m3") != "e4m3":
            continue
        w = np.asarray(n.consts["weight"], dtype=np.float64)
        s = np.ones(w.shape[0])
        cur = n.name
        while len(readers.get(cur, [])) == 1 and readers[cur][0].op in ("nn.bias_add", "nn.batch_norm"):
            nx = readers[cur][0]
            if nx.op == "nn.batch_norm":
                # epsilon as the compiled region carries it (fp32): the rounding
                # decisions below are then taken on the same folded weights
                eps = float(np.float32(nx.attrs.get("epsilon", 1e-5)))
                s = s * np.asarray(nx.consts["gamma"], np.float64) / np.sqrt(
                    np.asarray(nx.consts["moving_var"], np.float64) + eps)
            cur = nx.name
        shape = (-1,) + (1,) * (w.ndim - 1)
        wq, sw = quant.quantize_weights_e4m3(w * s.reshape(shape))
        out[n.name] = wq * sw.reshape(shape) / s.reshape(shape)
    return out


U_E4M3 = 2.0 ** -3  # one E4M3 step, relative: the most a re-rounded code can move


def _spread_node(node, args, sq, weight=None):
    """s^2 of ``node``'s output (before it is rounded for storage), given the
    inputs' values ``args`` and their s^2 ``sq``:

      conv2d / dense   sum_i sq_i w_i^2 + U_BF16^2 sum_i (x_i w_i)^2
                       + (sqrt(K) U_FP32 sum_i |x_i w_i|)^2
                       (input errors carried through the weights; each
                       weight rounded to bf16 once -- after any batch norm is
                       folded into it, which scales w_i and s alike; a K-term
                       fp32 sum, in the sqrt(K) form of the probabilistic
                       analysis of recursive summation)
      batch_norm       sq (gamma / sqrt(var + eps))^2
      bias_add, relu, clip   sq   (1-Lipschitz)
      gelu             1.13^2 sq
      add              sq_a + sq_b
      max_pool         the window's largest sq
      global_avg_pool  the window's mean sq
    """
    op, a, c = node.op, node.attrs, node.consts
    if op == "qnn.quantize":
        # an exact input is quantized identically on both sides (the same
        # fp32 product decides the code); a computed one can land on the
        # other side of a rounding boundary: one step
        return np.where(sq[0] > 0, sq[0] + (U_E4M3 * args[0]) ** 2, 0.0)
    if op in ("nn.conv2d", "nn.dense"):
        fp8 = weight is not None
        w = np.asarray(c["weight"] if weight is None else weight, dtype=np.float64)
        x = args[0]
        if op == "nn.conv2d":
            K = w.shape[1] * w.shape[2] * w.shape[3]
            lin = lambda t, ww: ops.conv2d_nhwc(t, ww, tuple(a["strides"]), tuple(a["padding"]),
                                                tuple(a["dilation"]), int(a["groups"]))
        else:
            K = w.shape[1]
            lin = ops.dense
        acc = np.sqrt(K) * U_FP32 * lin(np.abs(x), np.abs(w))
        if fp8:  # the quantized weights are the same on both sides
            return lin(sq[0], w * w) + acc * acc
        return lin(sq[0], w * w) + U_BF16 ** 2 * lin(x * x, w * w) + acc * acc
    if op == "nn.batch_norm":
        sc = np.asarray(c["gamma"], np.float64) ** 2 / (
            np.asarray(c["moving_var"], np.float64) + float(a.get("epsilon", 1e-5)))
        return sq[0] * sc
    if op in ("nn.bias_add", "nn.relu", "clip"):
        return sq[0]
    if op == "nn.gelu":
        return GELU_LIPSCHITZ ** 2 * sq[0]
    if op == "add":
        return sq[0] + sq[1]
    if op == "nn.max_pool2d":
        return ops.max_pool2d_nhwc(sq[0], tuple(a["pool_size"]), tuple(a["strides"]),
                                   tuple(a["padding"]))
    if op == "nn.global_avg_pool2d":
        return ops.global_avg_pool_nhwc(sq[0])
    raise NotImplementedError(op)


_GEMM_OR_POOL = ("nn.conv2d", "nn.dense", "nn.max_pool2d", "nn.global_avg_pool2d")


def evaluate_with_error_scale(graph, inputs: Dict[str, np.ndarray], nodes: Optional[Iterable[str]] = None,
                              keep: Optional[Iterable[str]] = None
                              ) -> Tuple[Dict[str, np.ndarray], Dict[str, np.ndarray]]:
    """``evaluate`` plus, for every kept tensor, the per-element error scale
    s = sqrt(sum_j a_j^2 u_j^2) of an implementation with bf16 storage and
    fp32 accumulation under the probabilistic rounding model (module
    comment): its error exceeds lam * s with probability at most
    2 exp(-lam^2 / 2).  Inputs count as exact (they arrive bf16-rounded).  A
    tensor is stored in bf16 -- adding (U_BF16 v)^2 to its s^2 -- where such
    an implementation must materialise it: when it is read by a conv2d,
    dense or pool, by more than one operator, by an operator outside
    ``nodes``, or is kept / a graph output.  The elementwise chains in
    between (bias, batch norm, residual add, activation) are fused and not
    rounded.  Returns (values, scales)."""
    env = {k: np.asarray(v, dtype=np.float64) for k, v in inputs.items()}
    sq = {k: np.zeros_like(v) for k, v in env.items()}
    wanted = set(nodes) if nodes is not None else None
    names = list(keep) if keep is not None else None
    kept = set(names) if names is not None else set(graph.outputs)
    readers: Dict[str, list] = {}
    for n in graph.nodes:
        for i in n.inputs:
            readers.setdefault(i, []).append(n)
    w8 = fp8_weights(graph, nodes)
    for n in graph.nodes:
        if wanted is not None and n.name not in wanted:
            continue
        args = [env[i] for i in n.inputs]
        v = eval_node(n, args, w8.get(n.name))
        q = _spread_node(n, args, [sq[i] for i in n.inputs], w8.get(n.name))
        rd = readers.get(n.name, [])
        stored = (n.name in kept or len(rd) != 1 or rd[0].op in _GEMM_OR_POOL
                  or (wanted is not None and rd[0].name not in wanted))
        # a quantizer's output is stored as its codes, exactly; a tensor a
        # quantizer reads is never stored in bf16 (the quantizer takes it)
        if n.op == "qnn.quantize" or (len(rd) == 1 and rd[0].op == "qnn.quantize" and n.name not in kept):
            stored = False
        if stored:
            q = q + (U_BF16 * v) ** 2
        env[n.name], sq[n.name] = v, q
    if names is None:
        names = [o for o in graph.outputs if o in env]
    return {k: env[k] for k in names}, {k: np.sqrt(sq[k]) for k in names}


def evaluate(graph, inputs: Dict[str, np.ndarray], nodes: Optional[Iterable[str]] = None,
             keep: Optional[Iterable[str]] = None) -> Dict[str, np.ndarray]:
    """Evaluate ``nodes`` (default: all) of ``graph`` in graph order.

    ``inputs`` maps tensor names (graph inputs, or boundary tensors of a
    region) to arrays.  Returns every computed tensor named in ``keep``
    (default: the graph outputs that were computed)."""
    env = {k: np.asarray(v, dtype=np.float64) for k, v in inputs.items()}
    wanted = set(nodes) if nodes is not None else None
    w8 = fp8_weights(graph, nodes)
    for n in graph.nodes:
        if wanted is not None and n.name not in wanted:
            continue
        env[n.name] = eval_node(n, [env[i] for i in n.inputs], w8.get(n.name))
    names = list(keep) if keep is not None else [o for o in graph.outputs if o in env]
    return {k: env[k] for k in names}
