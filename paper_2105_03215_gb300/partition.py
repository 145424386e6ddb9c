"""Graph partitioning (Section 3.1): pattern-based grouping into composites,
annotation of supported operators, greedy merging into regions, cost-based
splitting and host fallback, and encapsulation of each region as a function
with a target attribute.

Readings of points the paper leaves open:
  * ``optional`` matches the sequence with and without the optional node; at
    one root the longer match is taken.
  * The pattern table is applied in order; each pattern is tried at every
    node in reverse topological order (outputs first) before the next
    pattern is tried.
  * A match is valid only if none of its nodes already belongs to a
    composite and no non-root node of the match is read outside the match
    (or is a graph output).
  * "Consecutive supported operators" (Section 3.1.2): units -- composites
    count as one unit -- are visited in topological order; a supported unit
    joins the regions of its supported producers, one region at a time in
    region-id order, whenever the union stays convex (no path leaves the
    union and re-enters it).  Region ids follow each region's first unit.
  * The operator cap of the cost-based split (Section 3.1.3) counts a
    composite as one operator; regions are cut greedily in topological order,
    closing a region when the next unit would exceed the cap.
  * The fallback criterion of Section 4.1 keeps a region on the host when it
    has no multiply-accumulates; only conv2d and dense have MACs.
"""
from __future__ import annotations

import dataclasses
from typing import Callable, Dict, Iterable, List, Optional, Sequence, Set, Tuple

from .inputs import Graph, Node

# ---------------------------------------------------------------- pattern language


class Pattern:
    def optional(self, fn: Callable[["Pattern"], "Pattern"]) -> "Pattern":
        """The pattern with and without the node(s) ``fn`` wraps around it."""
        return Alt(fn(self), self)


class Wildcard(Pattern):
    def __repr__(self):
        return "*"


class IsOp(Pattern):
    def __init__(self, op: str, args: Sequence[Pattern] = ()):
        self.op = op
        self.args = list(args)

    def __call__(self, *args: Pattern) -> "IsOp":
        return IsOp(self.op, args)

    def __repr__(self):
        return f"{self.op}({', '.join(map(repr, self.args))})"


class Alt(Pattern):
    """First alternative preferred (the longer one for ``optional``)."""

    def __init__(self, *alts: Pattern):
        self.alts = list(alts)

    def __repr__(self):
        return " | ".join(map(repr, self.alts))


def wildcard() -> Wildcard:
    return Wildcard()


def is_op(op: str) -> IsOp:
    return IsOp(op)


# ---------------------------------------------------------------- annotation registry

_ANNOTATIONS: Dict[str, Dict[str, Callable[[Node], bool]]] = {}


def register_op_attr(op: str, attr: str):
    """``@register_op_attr("nn.conv2d", "codegen.byoc")`` registers a
    predicate deciding whether a node of that operator may be offloaded to
    the target named after ``codegen.`` (Section 3.1.2)."""
    if not attr.startswith("codegen."):
        raise ValueError("attribute must be codegen.<target>")
    target = attr[len("codegen."):]

    def deco(fn):
        _ANNOTATIONS.setdefault(target, {})[op] = fn
        return fn

    return deco


def annotations(target: str) -> Dict[str, Callable[[Node], bool]]:
    return dict(_ANNOTATIONS.get(target, {}))


# ---------------------------------------------------------------- results


@dataclasses.dataclass
class Composite:
    name: str              # pattern name
    root: str              # node whose output is the composite's output
    members: List[str]     # node names, graph order


@dataclasses.dataclass
class PartitionResult:
    graph: Graph
    units: List[List[str]]          # topological list of units (composite members or single nodes)
    unit_name: List[str]            # pattern name or operator name per unit
    composites: List[Composite]
    supported: List[bool]           # per unit
    regions: List[List[int]]        # region -> unit indices (topological)
    target: str
    host_units: List[int]

    def region_nodes(self, r: int) -> List[str]:
        names = set()
        for u in self.regions[r]:
            names.update(self.units[u])
        return [n.name for n in self.graph.nodes if n.name in names]

    def region_nodes_by_unit(self, r: int) -> List[str]:
        """The nodes of region r unit by unit (units in topological order,
        each composite's members together in graph order): the op order of
        the region's descriptor, so that the engine fuses exactly the
        composites the patterns found, whatever the region's size."""
        order = {n.name: i for i, n in enumerate(self.graph.nodes)}
        return [m for u in self.regions[r] for m in sorted(self.units[u], key=order.__getitem__)]

    def region_objects(self):
        from .region import Region
        return [Region(self.graph, self.region_nodes_by_unit(r), f"{self.target}_{r}")
                for r in range(len(self.regions))]

    def offload_ratio(self) -> Tuple[float, float]:
        """(node ratio, MAC ratio) of Tables 1, 3 and 4."""
        off = set()
        for r in range(len(self.regions)):
            off.update(self.region_nodes(r))
        total_nodes = len(self.graph.nodes)
        macs_total = sum(node_macs(n) for n in self.graph.nodes)
        macs_off = sum(node_macs(n) for n in self.graph.nodes if n.name in off)
        return (len(off) / total_nodes if total_nodes else 0.0,
                macs_off / macs_total if macs_total else 0.0)


def node_macs(n: Node) -> float:
    """Multiply-accumulates of a node: conv2d and dense only (Section 4.1)."""
    if n.op == "nn.conv2d":
        o, ci, kh, kw = n.attrs["weight_shape"]
        N, Ho, Wo, _ = n.shape
        return float(N * Ho * Wo) * o * ci * kh * kw
    if n.op == "nn.dense":
        u, i = n.attrs["weight_shape"]
        return float(n.shape[0]) * u * i
    return 0.0


# ---------------------------------------------------------------- matching


class _Graph:
    def __init__(self, g: Graph):
        self.g = g
        self.by_name = {n.name: n for n in g.nodes}
        self.order = {n.name: i for i, n in enumerate(g.nodes)}
        self.consumers: Dict[str, List[str]] = {n.name: [] for n in g.nodes}
        for n in g.nodes:
            for i in n.inputs:
                if i in self.consumers:
                    self.consumers[i].append(n.name)
        self.outputs = set(g.outputs)


def _match(G: _Graph, p: Pattern, tensor: str, taken: Set[str]) -> Optional[List[str]]:
    """Nodes matched by ``p`` rooted at the producer of ``tensor``, or None."""
    if isinstance(p, Wildcard):
        return []
    if isinstance(p, Alt):
        for a in p.alts:
            m = _match(G, a, tensor, taken)
            if m is not None:
                return m
        return None
    assert isinstance(p, IsOp)
    node = G.by_name.get(tensor)
    if node is None or node.op != p.op or node.name in taken:
        return None
    if len(p.args) < len(node.inputs):
        return None
    if any(not isinstance(a, Wildcard) for a in p.args[len(node.inputs):]):
        return None  # extra pattern arguments may only stand for constants
    got = [node.name]
    for a, t in zip(p.args, node.inputs):
        m = _match(G, a, t, taken)
        if m is None:
            return None
        got.extend(m)
    return got


def merge_composite(g: Graph, pattern_table: Sequence[Tuple]) -> List[Composite]:
    """Pattern-based grouping (Section 3.1.1).  ``pattern_table`` entries are
    (name, pattern_fn) or (name, pattern_fn, check_fn)."""
    G = _Graph(g)
    taken: Set[str] = set()
    comps: List[Composite] = []
    for entry in pattern_table:
        name, pat_fn = entry[0], entry[1]
        check = entry[2] if len(entry) > 2 else None
        pat = pat_fn()
        for node in reversed(g.nodes):
            if node.name in taken:
                continue
            m = _match(G, pat, node.name, taken)
            if not m or len(set(m)) != len(m):
                continue
            mset = set(m)
            ok = True
            for nm in m:
                if nm == node.name:
                    continue
                if nm in G.outputs or any(c not in mset for c in G.consumers[nm]):
                    ok = False
                    break
            if not ok:
                continue
            members = sorted(m, key=G.order.__getitem__)
            if check is not None and not check([G.by_name[x] for x in members]):
                continue
            comps.append(Composite(name, node.name, members))
            taken.update(m)
    comps.sort(key=lambda c: G.order[c.root])
    return comps


# ---------------------------------------------------------------- partition


def _units(g: Graph, comps: List[Composite]):
    G = _Graph(g)
    owner: Dict[str, int] = {}
    units: List[List[str]] = []
    names: List[str] = []
    comp_of_unit: Dict[int, Composite] = {}
    emitted: Set[int] = set()
    comp_index = {}
    for ci, c in enumerate(comps):
        for m in c.members:
            comp_index[m] = ci
    # a composite is placed at the position of its root (its last node)
    for n in g.nodes:
        ci = comp_index.get(n.name)
        if ci is None:
            owner[n.name] = len(units)
            units.append([n.name])
            names.append(n.op)
        elif n.name == comps[ci].root and ci not in emitted:
            emitted.add(ci)
            u = len(units)
            for m in comps[ci].members:
                owner[m] = u
            units.append(list(comps[ci].members))
            names.append(comps[ci].name)
            comp_of_unit[u] = comps[ci]
    # unit-level edges
    preds: List[Set[int]] = [set() for _ in units]
    for u, members in enumerate(units):
        ms = set(members)
        for m in members:
            for i in G.by_name[m].inputs:
                if i in owner and i not in ms:
                    preds[u].add(owner[i])
    return units, names, comp_of_unit, preds, owner


def _convex(union: Set[int], succs: List[Set[int]]) -> bool:
    """No path leaves ``union`` and re-enters it."""
    frontier = [v for u in union for v in succs[u] if v not in union]
    seen = set(frontier)
    while frontier:
        v = frontier.pop()
        for w in succs[v]:
            if w in union:
                return False
            if w not in seen:
                seen.add(w)
                frontier.append(w)
    return True


def partition(g: Graph, pattern_table: Sequence[Tuple], target: str = "byoc",
              max_ops: Optional[int] = None, fallback_no_mac: bool = True,
              annotators: Optional[Dict[str, Callable[[Node], bool]]] = None) -> PartitionResult:
    """Partition ``g`` for ``target``: composites, annotation, greedy merge,
    cost-based split (``max_ops`` units per region), MAC-free fallback."""
    comps = merge_composite(g, pattern_table)
    units, unames, comp_of_unit, preds, owner = _units(g, comps)
    ann = annotations(target) if annotators is None else annotators
    G = _Graph(g)

    def unit_supported(u: int) -> bool:
        if u in comp_of_unit:
            return all(G.by_name[m].op in ann and ann[G.by_name[m].op](G.by_name[m])
                       for m in units[u])
        n = G.by_name[units[u][0]]
        return n.op in ann and bool(ann[n.op](n))

    supported = [unit_supported(u) for u in range(len(units))]
    succs: List[Set[int]] = [set() for _ in units]
    for u, ps in enumerate(preds):
        for p in ps:
            succs[p].add(u)

    # greedy merge (Section 3.1.2)
    region_of: Dict[int, int] = {}
    regions: Dict[int, Set[int]] = {}
    next_id = 0
    for u in range(len(units)):
        if not supported[u]:
            continue
        cur = {u}
        cand = sorted({region_of[p] for p in preds[u] if p in region_of})
        absorbed = []
        for r in cand:
            union = cur | regions[r]
            if _convex(union, succs):
                cur = union
                absorbed.append(r)
        if absorbed:
            rid = min(absorbed)
            for r in absorbed:
                del regions[r]
        else:
            rid = next_id
            next_id += 1
        regions[rid] = cur
        for x in cur:
            region_of[x] = rid
    ordered = sorted(regions.values(), key=min)

    # cost-based split (Section 3.1.3)
    split: List[List[int]] = []
    for reg in ordered:
        us = sorted(reg)
        if max_ops is None:
            split.append(us)
            continue
        chunk: List[int] = []
        for u in us:
            if len(chunk) + 1 > max_ops:
                split.append(chunk)
                chunk = []
            chunk.append(u)
        if chunk:
            split.append(chunk)

    # fallback of MAC-free regions (Section 4.1: CalcMAC(graph) > 0)
    final: List[List[int]] = []
    host: List[int] = [u for u in range(len(units)) if not supported[u]]
    for reg in split:
        macs = sum(node_macs(G.by_name[m]) for u in reg for m in units[u])
        if fallback_no_mac and macs <= 0:
            host.extend(reg)
        else:
            final.append(reg)
    final.sort(key=min)
    return PartitionResult(g, units, unames, comps, supported, final, target, sorted(host))


# ---------------------------------------------------------------- this library's target

TARGET = "byoc"


def _bf16_activations(n: Node) -> bool:
    return n.dtype == "bfloat16"


@register_op_attr("nn.conv2d", "codegen.byoc")
def _conv2d(n: Node) -> bool:
    if not _bf16_activations(n):
        return False
    g = n.attrs["groups"]
    o, ci, kh, kw = n.attrs["weight_shape"]
    if g == 1:
        return o % 8 == 0
    return g == o and ci == 1 and kh == kw == 3 and o % 8 == 0


@register_op_attr("nn.dense", "codegen.byoc")
def _dense(n: Node) -> bool:
    u, i = n.attrs["weight_shape"]
    return _bf16_activations(n) and u % 8 == 0 and i % 8 == 0


for _op in ("nn.bias_add", "nn.batch_norm", "nn.relu", "nn.gelu", "add"):
    register_op_attr(_op, "codegen.byoc")(_bf16_activations)


@register_op_attr("clip", "codegen.byoc")
def _clip(n: Node) -> bool:
    return float(n.attrs.get("a_min")) == 0.0 and float(n.attrs.get("a_max")) == 6.0


def _conv_bn():
    return is_op("nn.batch_norm")(
        is_op("nn.conv2d")(wildcard(), wildcard()).optional(
            lambda x: is_op("nn.bias_add")(x, wildcard())),
        wildcard(), wildcard(), wildcard(), wildcard())


def conv2d_bn_add_relu_pattern():
    return is_op("nn.relu")(is_op("add")(_conv_bn(), wildcard()))


def conv2d_bn_add_pattern():
    """A linear projection conv + BN whose output is added to a residual
    (MobileNetV2's inverted-residual blocks)."""
    return is_op("add")(_conv_bn(), wildcard())


def conv2d_bn_act_pattern():
    return Alt(is_op("nn.relu")(_conv_bn()), is_op("clip")(_conv_bn()))


def conv2d_bn_pattern():
    return _conv_bn()


def conv2d_bias_act_pattern():
    """The listing of Section 3.1.1: conv2d, optional bias_add, ReLU."""
    conv = is_op("nn.conv2d")(wildcard(), wildcard())
    return is_op("nn.relu")(conv.optional(lambda x: is_op("nn.bias_add")(x, wildcard())))


def dense_bias_act_pattern():
    d = is_op("nn.bias_add")(is_op("nn.dense")(wildcard(), wildcard()), wildcard())
    return d.optional(lambda x: Alt(is_op("nn.gelu")(x), is_op("nn.relu")(x)))


PATTERN_TABLE = [
    ("conv2d_bn_add_relu", conv2d_bn_add_relu_pattern),
    ("conv2d_bn_add", conv2d_bn_add_pattern),
    ("conv2d_bn_act", conv2d_bn_act_pattern),
    ("conv2d_bn", conv2d_bn_pattern),
    ("conv2d_bias_act", conv2d_bias_act_pattern),
    ("dense_bias_act", dense_bias_act_pattern),
]
