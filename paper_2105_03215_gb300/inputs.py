"""Seeded synthetic inputs and workload graphs.

This module is pure data: random draws, the bf16 rounding of those draws, and
op lists describing the image-classification and transformer graphs whose
offloaded regions the library runs.  It holds none of the operators'
arithmetic and imports nothing else from this package, so both the fp64
oracle (test infrastructure) and the CUDA path may use it.

Graph format.  A ``Graph`` is a list of ``Node``s in topological order.  Each
node produces one tensor named after the node; ``inputs`` name graph inputs or
earlier nodes.  Operator names follow the high-level IR names the paper
partitions on (Section 3.1: operator name plus attributes such as stride,
padding and dilation):

  nn.conv2d          attrs strides=(sh,sw) padding=(t,l,b,r) dilation=(dh,dw)
                     groups; const weight OIHW fp32
  nn.dense           const weight [units, in] fp32
  nn.bias_add        const bias [C]
  nn.batch_norm      consts gamma, beta, moving_mean, moving_var; attr epsilon
  nn.relu, clip (a_min, a_max), nn.gelu (erf form), add
  nn.max_pool2d      attrs pool_size, strides, padding
  nn.global_avg_pool2d  NHWC [N,H,W,C] -> [N,C]

Activations are NHWC (Section 3.2, layout transformation); dense operands
are row-major [rows, features].

Seeds and draw order: one ``numpy.random.PCG64(seed)`` stream per workload,
drawn as: graph inputs, then every weight in node order, then every bias and
batch-norm statistic in node order.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Sequence, Tuple

import numpy as np

# ----------------------------------------------------------------------------
# bf16 helpers (round-to-nearest-even of the fp32 draws; data preparation)
# ----------------------------------------------------------------------------


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """fp32 values -> uint16 bf16 bit patterns, round to nearest even."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = (u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)
    return r.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """uint16 bf16 bit patterns -> fp32 values (exact)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32)


def bf16_round(a: np.ndarray) -> np.ndarray:
    """fp32 values rounded to the nearest bf16 value, returned as fp32."""
    return bf16_to_f32(bf16_bits(a))


# ----------------------------------------------------------------------------
# Graph data structures
# ----------------------------------------------------------------------------


@dataclasses.dataclass
class Node:
    name: str
    op: str
    inputs: List[str]
    attrs: Dict = dataclasses.field(default_factory=dict)
    consts: Dict[str, np.ndarray] = dataclasses.field(default_factory=dict)
    shape: Tuple[int, ...] = ()
    dtype: str = "bfloat16"


@dataclasses.dataclass
class Graph:
    inputs: Dict[str, Tuple[int, ...]]
    nodes: List[Node]
    outputs: List[str]
    name: str = ""

    def node(self, name: str) -> Node:
        for n in self.nodes:
            if n.name == name:
                return n
        raise KeyError(name)

    def shape_of(self, name: str) -> Tuple[int, ...]:
        if name in self.inputs:
            return tuple(self.inputs[name])
        return tuple(self.node(name).shape)


def conv_out(h: int, k: int, s: int, p0: int, p1: int, d: int = 1) -> int:
    return (h + p0 + p1 - d * (k - 1) - 1) // s + 1


class _Builder:
    """Appends nodes with inferred NHWC shapes; constants are drawn later."""

    def __init__(self, name: str):
        self.g = Graph(inputs={}, nodes=[], outputs=[], name=name)
        self._count: Dict[str, int] = {}

    def _name(self, op: str) -> str:
        base = op.split(".")[-1]
        i = self._count.get(base, 0)
        self._count[base] = i + 1
        return f"{base}_{i}"

    def input(self, name: str, shape: Sequence[int]) -> str:
        self.g.inputs[name] = tuple(int(s) for s in shape)
        return name

    def _add(self, op, inputs, shape, attrs=None, consts=None) -> str:
        n = Node(self._name(op), op, list(inputs), dict(attrs or {}), dict(consts or {}),
                 tuple(int(s) for s in shape))
        self.g.nodes.append(n)
        return n.name

    def conv2d(self, x, cout, k, stride=1, pad=None, groups=1, dilation=1, init="kaiming"):
        N, H, W, C = self.g.shape_of(x)
        if pad is None:
            pad = (k - 1) // 2 * dilation
        Ho = conv_out(H, k, stride, pad, pad, dilation)
        Wo = conv_out(W, k, stride, pad, pad, dilation)
        return self._add("nn.conv2d", [x], (N, Ho, Wo, cout),
                         dict(strides=(stride, stride), padding=(pad, pad, pad, pad),
                              dilation=(dilation, dilation), groups=groups,
                              kernel_size=(k, k), channels=cout, init=init,
                              weight_shape=(cout, C // groups, k, k)))

    def dense(self, x, units, init="normal", std=0.02):
        M, I = self.g.shape_of(x)
        return self._add("nn.dense", [x], (M, units),
                         dict(units=units, init=init, std=std, weight_shape=(units, I)))

    def bias_add(self, x):
        return self._add("nn.bias_add", [x], self.g.shape_of(x), dict(axis=-1))

    def batch_norm(self, x, eps=1e-5):
        return self._add("nn.batch_norm", [x], self.g.shape_of(x), dict(epsilon=eps, axis=-1))

    def relu(self, x):
        return self._add("nn.relu", [x], self.g.shape_of(x))

    def relu6(self, x):
        return self._add("clip", [x], self.g.shape_of(x), dict(a_min=0.0, a_max=6.0))

    def gelu(self, x):
        return self._add("nn.gelu", [x], self.g.shape_of(x))

    def add(self, a, b):
        assert self.g.shape_of(a) == self.g.shape_of(b)
        return self._add("add", [a, b], self.g.shape_of(a))

    def quantize(self, x, scale, dtype="e4m3", zero_point=0):
        """A Q node of Section 3.2 (scale S, zero point Z fixed at compile time)."""
        # the scale as a float32 value: the compiled region carries it in fp32
        return self._add("qnn.quantize", [x], self.g.shape_of(x),
                         dict(scale=float(np.float32(scale)), zero_point=int(zero_point), dtype=dtype))

    def max_pool2d(self, x, k, stride, pad):
        N, H, W, C = self.g.shape_of(x)
        return self._add("nn.max_pool2d", [x], (N, conv_out(H, k, stride, pad, pad),
                                              conv_out(W, k, stride, pad, pad), C),
                         dict(pool_size=(k, k), strides=(stride, stride),
                              padding=(pad, pad, pad, pad)))

    def global_avg_pool2d(self, x):
        N, H, W, C = self.g.shape_of(x)
        return self._add("nn.global_avg_pool2d", [x], (N, C))

    def batch_flatten(self, x):
        shp = self.g.shape_of(x)
        return self._add("nn.batch_flatten", [x], (shp[0], int(np.prod(shp[1:]))))


def _draw_constants(g: Graph, rng: np.random.Generator) -> None:
    """Weights in node order, then biases / BN statistics in node order."""
    for n in g.nodes:
        if n.op == "nn.conv2d":
            ws = n.attrs["weight_shape"]
            fan_in = ws[1] * ws[2] * ws[3]
            std = n.attrs.get("std") or math.sqrt(2.0 / fan_in)  # Kaiming-normal (fan_in, ReLU gain)
            n.consts["weight"] = (rng.standard_normal(ws, dtype=np.float32) * np.float32(std))
        elif n.op == "nn.dense":
            ws = n.attrs["weight_shape"]
            if n.attrs.get("init") == "kaiming":
                std = math.sqrt(2.0 / ws[1])
            else:
                std = n.attrs.get("std", 0.02)
            n.consts["weight"] = rng.standard_normal(ws, dtype=np.float32) * np.float32(std)
    for n in g.nodes:
        if n.op == "nn.bias_add":
            C = n.shape[-1]
            n.consts["bias"] = rng.uniform(-0.1, 0.1, size=C).astype(np.float32)
        elif n.op == "nn.batch_norm":
            C = n.shape[-1]
            n.consts["gamma"] = rng.uniform(0.5, 1.5, size=C).astype(np.float32)
            n.consts["beta"] = (rng.standard_normal(C, dtype=np.float32) * np.float32(0.1))
            n.consts["moving_mean"] = (rng.standard_normal(C, dtype=np.float32) * np.float32(0.1))
            n.consts["moving_var"] = rng.uniform(0.5, 1.5, size=C).astype(np.float32)


def _draw_inputs(g: Graph, rng: np.random.Generator) -> Dict[str, np.ndarray]:
    out = {}
    for name, shape in g.inputs.items():
        out[name] = bf16_round(rng.standard_normal(shape, dtype=np.float32))
    return out


def _finish(b: _Builder, outputs: List[str], seed: int, draw: bool = True):
    b.g.outputs = list(outputs)
    if not draw:
        return b.g, {}
    rng = np.random.Generator(np.random.PCG64(seed))
    inputs = _draw_inputs(b.g, rng)
    _draw_constants(b.g, rng)
    return b.g, inputs


# ----------------------------------------------------------------------------
# Workloads (shapes of the paper's edge-inference models)
# ----------------------------------------------------------------------------


def conv_bias_relu(N=1, H=56, W=56, C=64, K=64, k=3, stride=1, pad=None, seed=0,
                   act="relu", dilation=1):
    """Single composite region conv2d + bias_add + ReLU (the Conv2D-Add-ReLU
    pattern of Section 3.1.1), NHWC."""
    b = _Builder(f"conv{k}x{k}_bias_{act}")
    x = b.input("x", (N, H, W, C))
    y = b.conv2d(x, K, k, stride=stride, pad=pad, dilation=dilation)
    y = b.bias_add(y)
    if act == "relu":
        y = b.relu(y)
    elif act == "relu6":
        y = b.relu6(y)
    elif act == "gelu":
        y = b.gelu(y)
    return _finish(b, [y], seed)


def bert_ffn(M=1024, D=768, F=3072, seed=1):
    """Dense + bias + GELU followed by dense + bias (BERT-base FFN shapes:
    128 tokens x batch 8, 768 -> 3072 -> 768)."""
    b = _Builder("bert_ffn")
    x = b.input("x", (M, D))
    h = b.gelu(b.bias_add(b.dense(x, F, std=0.02)))
    y = b.bias_add(b.dense(h, D, std=0.02))
    return _finish(b, [y], seed)


def mbv2_dw_pw(N=32, H=56, W=56, C=144, Cout=24, seed=2, stride=1):
    """MobileNetV2 depthwise-separable block tail: depthwise 3x3 + BN + ReLU6,
    then pointwise 1x1 + BN (no activation)."""
    b = _Builder("mbv2_dw_pw")
    x = b.input("x", (N, H, W, C))
    d = b.relu6(b.batch_norm(b.conv2d(x, C, 3, stride=stride, groups=C)))
    y = b.batch_norm(b.conv2d(d, Cout, 1))
    return _finish(b, [y], seed)


def _bottleneck(b: _Builder, x: str, width: int, stride: int, downsample: bool) -> str:
    """ResNet-50 v1b bottleneck: stride on the 3x3; conv3 + BN -> add -> ReLU."""
    cout = 4 * width
    t = b.relu(b.batch_norm(b.conv2d(x, width, 1)))
    t = b.relu(b.batch_norm(b.conv2d(t, width, 3, stride=stride)))
    t = b.batch_norm(b.conv2d(t, cout, 1))
    sc = b.batch_norm(b.conv2d(x, cout, 1, stride=stride, pad=0)) if downsample else x
    return b.relu(b.add(t, sc))


def resnet_bottleneck(N=32, H=14, W=14, C=1024, width=256, stride=1, seed=3):
    """One ResNet-50 stage-3 bottleneck with identity residual."""
    b = _Builder("resnet50_bottleneck")
    x = b.input("x", (N, H, W, C))
    downsample = stride != 1 or C != 4 * width
    y = _bottleneck(b, x, width, stride, downsample)
    return _finish(b, [y], seed)


RESNET50_STAGES = ((3, 64, 1), (4, 128, 2), (6, 256, 2), (3, 512, 2))


def resnet50(N=64, H=224, W=224, num_classes=1000, seed=4, stages=RESNET50_STAGES, draw=True):
    """ResNet-50 v1b backbone + classifier: 53 convolutions, 1 dense."""
    b = _Builder("resnet50_v1b")
    x = b.input("data", (N, H, W, 3))
    t = b.relu(b.batch_norm(b.conv2d(x, 64, 7, stride=2, pad=3)))
    t = b.max_pool2d(t, 3, 2, 1)
    cin = 64
    for nblocks, width, stride in stages:
        for i in range(nblocks):
            s = stride if i == 0 else 1
            t = _bottleneck(b, t, width, s, downsample=(i == 0))
            cin = 4 * width
    p = b.global_avg_pool2d(t)
    y = b.bias_add(b.dense(p, num_classes, init="kaiming"))
    return _finish(b, [y], seed, draw)


def resnet18(N=1, H=224, W=224, num_classes=1000, seed=5, draw=False):
    """ResNet-18: basic blocks (3x3 conv-BN-ReLU, 3x3 conv-BN, add, ReLU)."""
    b = _Builder("resnet18")
    x = b.input("data", (N, H, W, 3))
    t = b.max_pool2d(b.relu(b.batch_norm(b.conv2d(x, 64, 7, stride=2, pad=3))), 3, 2, 1)
    cin = 64
    for i, width in enumerate((64, 128, 256, 512)):
        for j in range(2):
            s = 2 if (i > 0 and j == 0) else 1
            u = b.relu(b.batch_norm(b.conv2d(t, width, 3, stride=s)))
            u = b.batch_norm(b.conv2d(u, width, 3))
            sc = b.batch_norm(b.conv2d(t, width, 1, stride=s, pad=0)) if (s != 1 or cin != width) else t
            t = b.relu(b.add(u, sc))
            cin = width
    y = b.bias_add(b.dense(b.global_avg_pool2d(t), num_classes))
    return _finish(b, [y], seed, draw)


def vgg19(N=1, H=224, W=224, num_classes=1000, seed=6, draw=False):
    """VGG19: 16 conv3x3 + bias + ReLU in five stages, then three dense layers."""
    b = _Builder("vgg19")
    t = b.input("data", (N, H, W, 3))
    for nconv, width in ((2, 64), (2, 128), (4, 256), (4, 512), (4, 512)):
        for _ in range(nconv):
            t = b.relu(b.bias_add(b.conv2d(t, width, 3)))
        t = b.max_pool2d(t, 2, 2, 0)
    t = b.batch_flatten(t)
    t = b.relu(b.bias_add(b.dense(t, 4096)))
    t = b.relu(b.bias_add(b.dense(t, 4096)))
    y = b.bias_add(b.dense(t, num_classes))
    return _finish(b, [y], seed, draw)


MOBILENET_V2_BLOCKS = ((1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2), (6, 96, 3, 1),
                       (6, 160, 3, 2), (6, 320, 1, 1))


def depthwise(N=2, H=20, W=17, C=144, stride=1, seed=3):
    """Depthwise 3x3 conv (pad 1) + BN + ReLU6 alone."""
    b = _Builder(f"depthwise{C}s{stride}")
    x = b.input("x", (N, H, W, C))
    y = b.relu6(b.batch_norm(b.conv2d(x, C, 3, stride=stride, groups=C)))
    return _finish(b, [y], seed)


def mobilenet_v2(N=1, H=224, W=224, num_classes=1000, seed=7, draw=False):
    """MobileNetV2 1.0: inverted residual blocks (expand 1x1, depthwise 3x3,
    project 1x1, residual add when shapes allow), ReLU6 activations."""
    b = _Builder("mobilenet_v2")
    x = b.input("data", (N, H, W, 3))
    t = b.relu6(b.batch_norm(b.conv2d(x, 32, 3, stride=2)))
    cin = 32
    for tt, c, n, s in MOBILENET_V2_BLOCKS:
        for i in range(n):
            stride = s if i == 0 else 1
            u = t
            if tt != 1:
                u = b.relu6(b.batch_norm(b.conv2d(u, cin * tt, 1)))
            u = b.relu6(b.batch_norm(b.conv2d(u, cin * tt, 3, stride=stride, groups=cin * tt)))
            u = b.batch_norm(b.conv2d(u, c, 1))
            t = b.add(u, t) if (stride == 1 and cin == c) else u
            cin = c
    t = b.relu6(b.batch_norm(b.conv2d(t, 1280, 1)))
    y = b.bias_add(b.dense(b.global_avg_pool2d(t), num_classes))
    return _finish(b, [y], seed, draw)


def conv_general(N=2, H=11, W=13, C=64, K=32, kernel=(1, 3), strides=(1, 1), padding=(0, 1, 0, 1),
                 dilation=(1, 1), seed=12, small_int=False, act="relu"):
    """conv2d + bias_add + activation with any kernel shape, per-dimension
    strides / dilations and asymmetric padding (top, left, bottom, right)."""
    b = _Builder("conv_general")
    x = b.input("x", (N, H, W, C))
    kh, kw = kernel
    Ho = conv_out(H, kh, strides[0], padding[0], padding[2], dilation[0])
    Wo = conv_out(W, kw, strides[1], padding[1], padding[3], dilation[1])
    y = b._add("nn.conv2d", [x], (N, Ho, Wo, K),
               dict(strides=tuple(strides), padding=tuple(padding), dilation=tuple(dilation),
                    groups=1, kernel_size=(kh, kw), channels=K, init="kaiming",
                    weight_shape=(K, C, kh, kw)))
    y = b.bias_add(y)
    if act == "relu":
        y = b.relu(y)
    g, inp = _finish(b, [y], seed)
    if small_int:
        rng = np.random.Generator(np.random.PCG64(seed + 1000))
        inp = {"x": rng.integers(-4, 5, size=(N, H, W, C)).astype(np.float32)}
        g.nodes[0].consts["weight"] = rng.integers(-2, 3, size=(K, C, kh, kw)).astype(np.float32)
        g.nodes[1].consts["bias"] = rng.integers(-8, 9, size=K).astype(np.float32)
    return g, inp


# Scales of the FP8 workloads, fixed from the known distributions of the
# synthetic data (a stand-in for the calibration data of Section 3.2): region
# inputs ~N(0, 1) are quantized over +-8 (8 standard deviations); the
# intermediates after batch norm + ReLU (gamma ~ U(0.5, 1.5), Kaiming weights,
# unit-variance outputs) over +-16.
FP8_SCALE_INPUT = 8.0 / 448.0
FP8_SCALE_HIDDEN = 16.0 / 448.0


def fp8_conv(N=2, H=14, W=14, C=256, K=256, k=3, seed=31, act="relu"):
    """conv2d + BN + activation computed in FP8: Q(x) -> conv -> BN -> act."""
    b = _Builder(f"fp8_conv{k}x{k}")
    x = b.input("x", (N, H, W, C))
    y = b.batch_norm(b.conv2d(b.quantize(x, FP8_SCALE_INPUT), K, k))
    y = b.relu(y) if act == "relu" else y
    return _finish(b, [y], seed)


def fp8_dense(M=256, D=768, F=1024, seed=32):
    """dense + bias + GELU computed in FP8: Q(x) -> dense -> bias -> GELU."""
    b = _Builder("fp8_dense")
    x = b.input("x", (M, D))
    y = b.gelu(b.bias_add(b.dense(b.quantize(x, FP8_SCALE_INPUT), F)))
    return _finish(b, [y], seed)


# the BERT FFN's hidden activation GELU(x W1^T + b1): pre-activations of
# standard deviation sqrt(768) x 0.02 = 0.55, quantized over +-4
FP8_SCALE_FFN_HIDDEN = 4.0 / 448.0


def fp8_ffn(M=1024, D=768, F=3072, seed=1):
    """The BERT FFN of bert_ffn (same seed, same constants) with partial
    quantization (Section 3.2): Q nodes before both dense layers, each dense
    in FP8; the hidden activation leaves the first epilogue as E4M3 codes."""
    b = _Builder("fp8_ffn")
    x = b.input("x", (M, D))
    h = b.gelu(b.bias_add(b.dense(b.quantize(x, FP8_SCALE_INPUT), F, std=0.02)))
    y = b.bias_add(b.dense(b.quantize(h, FP8_SCALE_FFN_HIDDEN), D, std=0.02))
    return _finish(b, [y], seed)


def fp8_bottleneck(N=32, H=14, W=14, C=1024, width=256, seed=3):
    """The ResNet-50 stage-3 bottleneck of resnet_bottleneck (same seed, same
    constants) with partial quantization (Section 3.2): Q nodes before each
    convolution, each convolution in FP8; the residual stays bf16."""
    b = _Builder("fp8_bottleneck")
    x = b.input("x", (N, H, W, C))
    t = b.relu(b.batch_norm(b.conv2d(b.quantize(x, FP8_SCALE_INPUT), width, 1)))
    t = b.relu(b.batch_norm(b.conv2d(b.quantize(t, FP8_SCALE_HIDDEN), width, 3)))
    t = b.batch_norm(b.conv2d(b.quantize(t, FP8_SCALE_HIDDEN), 4 * width, 1))
    y = b.relu(b.add(t, x))
    return _finish(b, [y], seed)


def stem(N=2, H=32, W=30, k=7, cout=64, seed=13, C=3):
    """A stride-2 k x k stem conv + BN + ReLU over an image with C (<= 4) channels."""
    b = _Builder(f"stem{k}x{k}")
    x = b.input("data", (N, H, W, C))
    y = b.relu(b.batch_norm(b.conv2d(x, cout, k, stride=2, pad=k // 2)))
    return _finish(b, [y], seed)


def small_int_conv(N=2, H=9, W=11, C=64, K=64, k=3, stride=1, pad=1, seed=7, act="relu"):
    """Conv + bias + act with small-integer data (|v| <= 4), exact in bf16 and
    accumulated exactly in fp32: the GPU output must equal the bf16 rounding
    of the exact result bit for bit."""
    g, _ = conv_bias_relu(N=N, H=H, W=W, C=C, K=K, k=k, stride=stride, pad=pad, seed=seed, act=act)
    rng = np.random.Generator(np.random.PCG64(seed + 1000))
    x = rng.integers(-4, 5, size=(N, H, W, C)).astype(np.float32)
    for n in g.nodes:
        if n.op == "nn.conv2d":
            n.consts["weight"] = rng.integers(-2, 3, size=n.attrs["weight_shape"]).astype(np.float32)
        if n.op == "nn.bias_add":
            n.consts["bias"] = rng.integers(-8, 9, size=n.shape[-1]).astype(np.float32)
    return g, {"x": x}


def small_int_dense(M=200, I=192, U=320, seed=8, act="relu"):
    b = _Builder("dense_int")
    x = b.input("x", (M, I))
    y = b.bias_add(b.dense(x, U))
    if act == "relu":
        y = b.relu(y)
    g, _ = _finish(b, [y], seed)
    rng = np.random.Generator(np.random.PCG64(seed + 1000))
    xs = rng.integers(-4, 5, size=(M, I)).astype(np.float32)
    for n in g.nodes:
        if n.op == "nn.dense":
            n.consts["weight"] = rng.integers(-2, 3, size=n.attrs["weight_shape"]).astype(np.float32)
        if n.op == "nn.bias_add":
            n.consts["bias"] = rng.integers(-8, 9, size=n.shape[-1]).astype(np.float32)
    return g, {"x": xs}


def region_flops(g: Graph) -> float:
    """Multiply-accumulate count x 2 over conv2d and dense nodes (the only
    operators with MACs, Section 4.1 footnote)."""
    f = 0.0
    for n in g.nodes:
        if n.op == "nn.conv2d":
            o, ci, kh, kw = n.attrs["weight_shape"]
            f += 2.0 * np.prod(n.shape[:-1]) * o * ci * kh * kw
        elif n.op == "nn.dense":
            u, i = n.attrs["weight_shape"]
            f += 2.0 * n.shape[0] * u * i
    return float(f)
