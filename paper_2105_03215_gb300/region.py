"""Regions: encapsulated partitioned functions (Section 3.1.3) and their
compiled engines (Section 3.4).

``Region`` turns a set of graph nodes into the C descriptor of include/byoc.h
(its boundary inputs are the tensors the nodes read but do not produce; its
outputs are the tensors read outside it or listed as graph outputs).
``Region.compile()`` returns a ``CompiledRegion`` whose ``run`` is the
external function call of Section 3.4: it enqueues the region's CUDA kernels
on a stream, reading and writing caller-owned device tensors.
"""
from __future__ import annotations

import ctypes
from typing import Dict, List, Optional, Sequence

import numpy as np

from . import abi
from .inputs import Graph, Node

_OP_KIND = {
    "nn.conv2d": abi.OP_CONV2D,
    "nn.dense": abi.OP_DENSE,
    "nn.bias_add": abi.OP_BIAS_ADD,
    "nn.batch_norm": abi.OP_BATCH_NORM,
    "nn.relu": abi.OP_RELU,
    "nn.gelu": abi.OP_GELU,
    "add": abi.OP_ADD,
    "qnn.quantize": abi.OP_QUANTIZE,
}

OFFLOADABLE_OPS = frozenset(list(_OP_KIND) + ["clip"])


def op_kind(node: Node) -> int:
    if node.op == "clip":
        if float(node.attrs.get("a_min", 0.0)) == 0.0 and float(node.attrs.get("a_max", 6.0)) == 6.0:
            return abi.OP_RELU6
        raise abi.ByocError(abi.ERR_UNSUPPORTED, f"clip({node.attrs}) other than ReLU6")
    try:
        return _OP_KIND[node.op]
    except KeyError:
        raise abi.ByocError(abi.ERR_UNSUPPORTED, f"operator {node.op} cannot be offloaded") from None


class Region:
    """A set of nodes of ``graph`` encapsulated as one offloaded function."""

    def __init__(self, graph: Graph, node_names: Sequence[str], name: str = "region",
                 outputs: Optional[Sequence[str]] = None, options: int = 0):
        """``options``: abi.OPT_* bits passed to the code generator
        (byoc_region_desc.options); they pick among kernel plans that compute
        the same values."""
        self.graph = graph
        self.options = int(options)
        members = set(node_names)
        # ops keep the given order (the descriptor's op order, which decides
        # what the engine fuses); it must be topological within the region
        by_name = {n.name: n for n in graph.nodes}
        if len(members) != len(node_names) or not members <= by_name.keys():
            raise KeyError(f"unknown or repeated nodes in region {name}")
        self.nodes: List[Node] = [by_name[m] for m in node_names]
        seen = set()
        for n in self.nodes:
            if any(i in members and i not in seen for i in n.inputs):
                raise ValueError(f"region {name}: {n.name} comes before one of its inputs")
            seen.add(n.name)
        self.name = name
        produced = {n.name for n in self.nodes}
        ins: List[str] = []
        for n in self.nodes:
            for i in n.inputs:
                if i not in produced and i not in ins:
                    ins.append(i)
        self.inputs = ins
        if outputs is None:
            consumed_outside = set()
            for n in graph.nodes:
                if n.name in members:
                    continue
                consumed_outside.update(i for i in n.inputs if i in produced)
            outputs = [n.name for n in self.nodes
                       if n.name in consumed_outside or n.name in graph.outputs]
        self.outputs = list(outputs)

    # -------------------------------------------------------------- descriptor
    def to_desc(self):
        """Build the C descriptor.  Returns (desc, keepalive)."""
        g = self.graph
        names = list(self.inputs) + [n.name for n in self.nodes]
        tid = {nm: i for i, nm in enumerate(names)}
        by_name = {n.name for n in g.nodes}
        tensors = (abi.Tensor * len(names))()
        for i, nm in enumerate(names):
            shp = g.shape_of(nm)
            tensors[i].ndim = len(shp)
            for k, s in enumerate(shp):
                tensors[i].shape[k] = int(s)
            src = g.node(nm) if nm in by_name else None
            tensors[i].dtype = abi.E4M3 if src is not None and src.op == "qnn.quantize" else abi.BF16
            tensors[i].layout = abi.LAYOUT_NHWC if len(shp) == 4 else abi.LAYOUT_NC
        keep: list = [tensors]
        ops = (abi.Op * len(self.nodes))()
        for j, n in enumerate(self.nodes):
            o = ops[j]
            o.kind = op_kind(n)
            o.n_in = len(n.inputs)
            for k, i in enumerate(n.inputs):
                o.in_[k] = tid[i]
            o.out = tid[n.name]
            if n.op == "nn.conv2d":
                kh, kw = n.attrs["kernel_size"]
                o.kernel[0], o.kernel[1] = kh, kw
                o.stride[0], o.stride[1] = n.attrs["strides"]
                for k in range(4):
                    o.pad[k] = n.attrs["padding"][k]
                o.dilation[0], o.dilation[1] = n.attrs["dilation"]
                o.groups = n.attrs["groups"]
                consts = [n.consts["weight"]]
            elif n.op == "nn.dense":
                consts = [n.consts["weight"]]
            elif n.op == "nn.bias_add":
                consts = [n.consts["bias"]]
            elif n.op == "nn.batch_norm":
                consts = [n.consts["gamma"], n.consts["beta"], n.consts["moving_mean"],
                          n.consts["moving_var"]]
                o.eps = float(n.attrs.get("epsilon", 1e-5))
            elif n.op == "qnn.quantize":
                if n.attrs.get("dtype", "e4m3") != "e4m3":
                    raise abi.ByocError(abi.ERR_UNSUPPORTED, f"{n.name}: only E4M3 quantization runs here")
                consts = [np.array([n.attrs["scale"]], np.float32),
                          np.array([n.attrs.get("zero_point", 0)], np.float32)]
            else:
                consts = []
            for k, c in enumerate(consts):
                arr = np.ascontiguousarray(c, dtype=np.float32)
                keep.append(arr)
                o.consts[k] = arr.ctypes.data
        keep.append(ops)
        in_ids = (ctypes.c_int32 * len(self.inputs))(*[tid[i] for i in self.inputs])
        out_ids = (ctypes.c_int32 * len(self.outputs))(*[tid[i] for i in self.outputs])
        cname = self.name.encode()
        keep += [in_ids, out_ids, cname]
        desc = abi.RegionDesc(abi.ABI_VERSION, cname, len(names), tensors, len(self.nodes), ops,
                              len(self.inputs), in_ids, len(self.outputs), out_ids, self.options)
        return desc, keep

    # -------------------------------------------------------------- planning / compile
    def plan(self, num_sms: int = 148) -> abi.PlanReport:
        desc, keep = self.to_desc()
        rep = abi.PlanReport()
        abi.check(abi.lib().byoc_plan(ctypes.byref(desc), num_sms, ctypes.byref(rep)))
        return rep

    def plan_constants(self, launch: int, what: int, num_sms: int = 148) -> bytes:
        desc, keep = self.to_desc()
        need = ctypes.c_size_t()
        L = abi.lib()
        abi.check(L.byoc_plan_constants(ctypes.byref(desc), num_sms, launch, what, None, 0,
                                        ctypes.byref(need)))
        buf = ctypes.create_string_buffer(need.value)
        abi.check(L.byoc_plan_constants(ctypes.byref(desc), num_sms, launch, what, buf, need.value,
                                        ctypes.byref(need)))
        return buf.raw

    def compile(self) -> "CompiledRegion":
        desc, keep = self.to_desc()
        h = ctypes.c_void_p()
        abi.check(abi.lib().byoc_compile(ctypes.byref(desc), ctypes.byref(h)))
        return CompiledRegion(h, self)

    def plan_serialized(self, num_sms: int = 148) -> bytes:
        """The serialised plan of this region for ``num_sms`` SMs, made on the
        host (no GPU); ``load_plan_report`` parses it back."""
        desc, keep = self.to_desc()
        need = ctypes.c_size_t()
        L = abi.lib()
        abi.check(L.byoc_plan_serialize(ctypes.byref(desc), num_sms, None, 0, ctypes.byref(need)))
        buf = ctypes.create_string_buffer(need.value)
        abi.check(L.byoc_plan_serialize(ctypes.byref(desc), num_sms, buf, need.value,
                                        ctypes.byref(need)))
        return buf.raw

    def load(self, blob: bytes) -> "CompiledRegion":
        """A compiled region rebuilt from ``CompiledRegion.serialize()`` bytes
        (Section 3.3, option 3): no planning, folding or packing."""
        h = ctypes.c_void_p()
        buf = ctypes.create_string_buffer(bytes(blob), len(blob))
        abi.check(abi.lib().byoc_deserialize(buf, len(blob), ctypes.byref(h)))
        return CompiledRegion(h, self)


def load_plan_report(blob: bytes) -> abi.PlanReport:
    """Parse serialised region bytes on the host and report the plan they hold."""
    rep = abi.PlanReport()
    buf = ctypes.create_string_buffer(bytes(blob), len(blob))
    abi.check(abi.lib().byoc_plan_deserialize(buf, len(blob), ctypes.byref(rep)))
    return rep


class CompiledRegion:
    """A compiled, cached engine for one region (owns device constants)."""

    def __init__(self, handle: ctypes.c_void_p, region: Region):
        self._h = handle
        self.region = region
        self.name = region.name
        info = abi.Info()
        abi.check(abi.lib().byoc_query(self._h, ctypes.byref(info)))
        self.flops = info.flops
        self.bytes = info.bytes
        self.n_launches = info.n_launches
        self.workspace_bytes = info.workspace_bytes
        self.const_bytes = info.const_bytes
        n_in, n_out = len(region.inputs), len(region.outputs)
        self._in = (ctypes.c_void_p * n_in)()
        self._out = (ctypes.c_void_p * n_out)()

    def run(self, inputs: Sequence, outputs: Sequence, stream=None) -> None:
        """Enqueue the region on ``stream`` (default: torch's current stream).
        ``inputs`` / ``outputs`` are contiguous bf16 CUDA tensors (or raw
        device addresses) in the region's boundary order."""
        for k, t in enumerate(inputs):
            self._in[k] = t if isinstance(t, int) else t.data_ptr()
        for k, t in enumerate(outputs):
            self._out[k] = t if isinstance(t, int) else t.data_ptr()
        abi.check(abi.lib().byoc_run(self._h, self._in, self._out, abi._stream_ptr(stream)))

    def check(self) -> None:
        """Raise if a kernel of this region hit a bounded-wait timeout."""
        abi.check(abi.lib().byoc_check(self._h))

    def serialize(self) -> bytes:
        """The compiled region as bytes (``Region.load`` rebuilds it)."""
        need = ctypes.c_size_t()
        L = abi.lib()
        abi.check(L.byoc_serialize(self._h, None, 0, ctypes.byref(need)))
        buf = ctypes.create_string_buffer(need.value)
        abi.check(L.byoc_serialize(self._h, buf, need.value, ctypes.byref(need)))
        return buf.raw

    def release(self) -> None:
        if self._h:
            abi.lib().byoc_release(self._h)
            self._h = None

    def __del__(self):
        try:
            self.release()
        except Exception:
            pass


def whole_graph_region(graph: Graph, name: Optional[str] = None, options: int = 0) -> Region:
    """All nodes of ``graph`` as one region (the offload-everything case)."""
    return Region(graph, [n.name for n in graph.nodes], name or graph.name or "region",
                  outputs=graph.outputs, options=options)
