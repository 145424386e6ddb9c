"""Graph executor for a partitioned model (Section 3.4, runtime).

Initialisation compiles every region once (the cached execution engines) and
pre-allocates the data entries: one device buffer for every tensor that
crosses a step boundary (graph inputs and outputs, region inputs and
outputs, host-operator inputs and outputs).  Region intermediates are not
data entries; they live in each region's workspace.  ``run`` then visits the
steps in a topological order of the partitioned graph: host operators run
through this library's host kernels (CUDA serving as the host), regions
through their external call ``byoc_run``.  All work is enqueued on one CUDA
stream; ``capture()`` records the whole sequence as a CUDA graph so a forward
pass costs one launch.
"""
from __future__ import annotations

import heapq
from typing import Dict, List, Optional, Sequence, Tuple

from . import abi
from .inputs import Graph, Node
from .partition import PartitionResult

HOST_OPS = ("nn.max_pool2d", "nn.global_avg_pool2d", "nn.batch_flatten")


class Executor:
    def __init__(self, result: PartitionResult, serialized: Optional[List[bytes]] = None,
                 options: int = 0):
        """Compile every region of ``result`` with the code-generation
        ``options`` (abi.OPT_* bits) -- or, given ``serialized`` (one
        ``CompiledRegion.serialize()`` blob per region, from ``serialize()``),
        load them without compiling (Section 3.3, option 3).  ``init_s`` is
        the wall time of that step (the engine initialisation of Section 4.1)."""
        import time
        import torch
        self.torch = torch
        self.result = result
        self.graph: Graph = result.graph
        g = self.graph
        self.by_name = {n.name: n for n in g.nodes}
        # steps: ("region", index) or ("host", node name), in a topological order
        self.regions = result.region_objects()
        for r in self.regions:
            r.options = int(options)
        t0 = time.perf_counter()
        if serialized is None:
            self.compiled = [r.compile() for r in self.regions]
        else:
            if len(serialized) != len(self.regions):
                raise ValueError(f"{len(serialized)} serialised regions for {len(self.regions)} regions")
            self.compiled = [r.load(b) for r, b in zip(self.regions, serialized)]
        self.init_s = time.perf_counter() - t0
        self.steps = self._order_steps()
        # data entries
        needed = set(g.outputs) | set(g.inputs)
        for r in self.regions:
            needed.update(r.inputs)
            needed.update(r.outputs)
        for kind, x in self.steps:
            if kind == "host":
                n = self.by_name[x]
                needed.update(n.inputs)
                needed.add(n.name)
        self.entries: Dict[str, "torch.Tensor"] = {}
        for name in sorted(needed, key=self._order_key):
            node = self.by_name.get(name)
            if node is not None and node.op == "nn.batch_flatten":
                continue  # a view of its input, made below
            self.entries[name] = torch.empty(g.shape_of(name), dtype=torch.bfloat16, device="cuda")
        for name in needed:
            node = self.by_name.get(name)
            if node is not None and node.op == "nn.batch_flatten":
                src = self.entries[node.inputs[0]]
                self.entries[name] = src.view(node.shape)
        self._graph = None
        self._pipe = None
        self.n_launches = sum(c.n_launches for c in self.compiled) + sum(
            1 for k, x in self.steps if k == "host" and self.by_name[x].op != "nn.batch_flatten")

    def serialize(self) -> List[bytes]:
        """Every compiled region as bytes, in region order."""
        return [c.serialize() for c in self.compiled]

    # ------------------------------------------------------------------ planning
    def _order_key(self, name: str) -> int:
        for i, n in enumerate(self.graph.nodes):
            if n.name == name:
                return i + 1
        return 0

    def _order_steps(self) -> List[Tuple[str, object]]:
        """Kahn's algorithm over regions and host nodes (regions are convex,
        so collapsing each into one step keeps the graph acyclic); ties are
        broken by the position of the step's first node."""
        g = self.graph
        pos = {n.name: i for i, n in enumerate(g.nodes)}
        step_of: Dict[str, int] = {}
        steps: List[Tuple[str, object]] = []
        first: List[int] = []
        for ri, r in enumerate(self.regions):
            for n in r.nodes:
                step_of[n.name] = len(steps)
            steps.append(("region", ri))
            first.append(min(pos[n.name] for n in r.nodes))
        for n in g.nodes:
            if n.name not in step_of:
                if n.op not in HOST_OPS:
                    raise abi.ByocError(abi.ERR_UNSUPPORTED,
                                        f"{n.name} ({n.op}) is neither offloaded nor a host operator")
                step_of[n.name] = len(steps)
                steps.append(("host", n.name))
                first.append(pos[n.name])
        preds = [set() for _ in steps]
        for n in g.nodes:
            s = step_of[n.name]
            for i in n.inputs:
                if i in step_of and step_of[i] != s:
                    preds[s].add(step_of[i])
        indeg = [len(p) for p in preds]
        succ = [[] for _ in steps]
        for s, ps in enumerate(preds):
            for p in ps:
                succ[p].append(s)
        heap = [(first[s], s) for s in range(len(steps)) if indeg[s] == 0]
        heapq.heapify(heap)
        order = []
        while heap:
            _, s = heapq.heappop(heap)
            order.append(steps[s])
            for t in succ[s]:
                indeg[t] -= 1
                if indeg[t] == 0:
                    heapq.heappush(heap, (first[t], t))
        if len(order) != len(steps):
            raise abi.ByocError(abi.ERR_INVALID_ARG, "partition is not convex: step graph has a cycle")
        return order

    # ------------------------------------------------------------------ running
    def _host(self, node: Node, stream) -> None:
        x = self.entries[node.inputs[0]]
        y = self.entries[node.name]
        if node.op == "nn.max_pool2d":
            k = node.attrs["pool_size"][0]
            s = node.attrs["strides"][0]
            p = node.attrs["padding"][0]
            abi.max_pool2d_nhwc(x, y, k, s, p, stream)
        elif node.op == "nn.global_avg_pool2d":
            abi.global_avg_pool_nhwc(x, y, stream)
        # nn.batch_flatten: a view, nothing to run

    def run_steps(self, stream=None, hooks=None) -> None:
        """Enqueue one forward pass.  ``hooks(kind, index, 'pre'|'post')`` is
        called around every step (used to record timing events)."""
        st = abi._stream_ptr(stream)
        for i, (kind, x) in enumerate(self.steps):
            if hooks:
                hooks(kind, i, "pre")
            if kind == "region":
                r = self.regions[x]
                self.compiled[x].run([self.entries[n] for n in r.inputs],
                                     [self.entries[n] for n in r.outputs], st)
            else:
                self._host(self.by_name[x], st)
            if hooks:
                hooks(kind, i, "post")

    def set_input(self, name: str, src, non_blocking: bool = True) -> None:
        self.entries[name].copy_(src, non_blocking=non_blocking)

    def set_input_nchw(self, name: str, x, stream=None) -> None:
        """Fill the NHWC bf16 data entry ``name`` from a framework-layout
        NCHW fp32 CUDA tensor, through the boundary layout transformation
        (Section 3.2) of this library; channels beyond x's are zero."""
        dst = self.entries[name]
        N, H, W, Cp = dst.shape
        if x.dtype != self.torch.float32 or not x.is_cuda or not x.is_contiguous():
            raise ValueError("x must be a contiguous fp32 CUDA tensor")
        if tuple(x.shape) != (N, x.shape[1], H, W) or x.shape[1] > Cp:
            raise ValueError(f"x {tuple(x.shape)} does not match entry {tuple(dst.shape)} as NCHW")
        abi.check(abi.lib().byoc_nchw_to_nhwc_bf16(x.data_ptr(), dst.data_ptr(), N, x.shape[1], H, W, Cp,
                                                   abi._stream_ptr(stream)))

    def output(self, name: Optional[str] = None):
        return self.entries[name or self.graph.outputs[0]]

    def capture(self) -> None:
        """Record one forward pass as a CUDA graph (after one eager warm-up)."""
        torch = self.torch
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.run_steps(s)
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run_steps()
        self._graph = g

    def replay(self) -> None:
        if self._graph is None:
            raise RuntimeError("capture() first")
        self._graph.replay()

    def capture_double_buffered(self, name: str = "data") -> None:
        """Record two CUDA graphs of the forward pass that read the input entry
        ``name`` from two different device buffers, for run_from_host: while
        one pass runs, the next pass's input is uploaded into the other."""
        torch = self.torch
        self.capture()  # warm-up and the first graph, on the entry's own buffer
        first = self.entries[name]
        second = torch.empty_like(first)
        self.entries[name] = second
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.run_steps()
        self.entries[name] = first
        self._pipe = {"name": name, "bufs": [first, second], "graphs": [self._graph, g],
                      "copy": torch.cuda.Stream(),
                      "in_ready": [torch.cuda.Event(), torch.cuda.Event()],
                      "in_free": [torch.cuda.Event(), torch.cuda.Event()]}

    def run_from_host(self, host_inputs: Sequence, host_outputs: Sequence) -> None:
        """Forward passes over a sequence of batches in (pinned) host memory:
        pass i reads host_inputs[i] and writes its output to host_outputs[i].
        Inputs are uploaded on a copy stream into alternating device buffers,
        each as soon as the pass that last read that buffer has finished, so
        pass i + 1's upload overlaps pass i; passes run in order on the current
        stream, each followed by the read-back of its output.  Returns once
        every output is in host memory."""
        if getattr(self, "_pipe", None) is None:
            raise RuntimeError("capture_double_buffered() first")
        torch = self.torch
        p = self._pipe
        cs = torch.cuda.current_stream()
        cp = p["copy"]
        n = len(host_inputs)
        if len(host_outputs) != n:
            raise ValueError("one output buffer per input batch")

        def upload(i):
            b = i & 1
            cp.wait_event(p["in_free"][b])  # the pass that last read buffer b is done
            with torch.cuda.stream(cp):
                p["bufs"][b].copy_(host_inputs[i], non_blocking=True)
            p["in_ready"][b].record(cp)

        if n:
            upload(0)
        for i in range(n):
            if i + 1 < n:
                upload(i + 1)
            b = i & 1
            cs.wait_event(p["in_ready"][b])
            p["graphs"][b].replay()
            p["in_free"][b].record(cs)
            host_outputs[i].copy_(self.output(), non_blocking=True)
        cs.synchronize()

    def check(self) -> None:
        for c in self.compiled:
            c.check()

    def release(self) -> None:
        for c in self.compiled:
            c.release()
        self.compiled = []
        self._graph = None
        self._pipe = None
        self.entries = {}


def build_resnet50(N: int = 64, H: int = 224, W: int = 224, seed: int = 4, max_ops: Optional[int] = 1,
                   graph=None):
    """ResNet-50 v1b partitioned for this library (pools on the host); with
    ``max_ops=1`` every conv2d / dense composite is its own region (54)."""
    from . import inputs as I
    from . import partition as P
    if graph is None:
        graph, inp = I.resnet50(N=N, H=H, W=W, seed=seed)
    else:
        inp = None
    res = P.partition(graph, P.PATTERN_TABLE, target=P.TARGET, max_ops=max_ops)
    return res, inp


def build_mobilenet_v2(N: int = 64, H: int = 224, W: int = 224, seed: int = 7,
                       max_ops: Optional[int] = 1):
    """MobileNetV2 1.0 partitioned for this library (global average pool on the
    host); with ``max_ops=1`` every conv2d / dense composite is its own region
    (52 conv composites, depthwise included, + the classifier)."""
    from . import inputs as I
    from . import partition as P
    graph, inp = I.mobilenet_v2(N=N, H=H, W=W, seed=seed, draw=True)
    res = P.partition(graph, P.PATTERN_TABLE, target=P.TARGET, max_ops=max_ops)
    return res, inp
