"""Reference partitioning bookkeeping (Section 3.1), written independently of
the product partitioner.

TEST INFRASTRUCTURE.  It follows the paper's steps in order -- pattern-based
grouping (3.1.1), annotation and greedy merging of consecutive supported
operators (3.1.2), cost-based splitting and host fallback (3.1.3) -- under
the same readings of what the paper leaves open, but by different means:

* patterns are given as explicit operator sequences along the data path
  (input 0 of each operator, bottom-up from the root) instead of pattern
  objects; ``optional`` nodes are expanded into separate sequences, longest
  first;
* regions are kept in a union-find structure; convexity is checked against a
  precomputed transitive closure of the unit graph;
* splitting and fallback walk the regions' units in topological order.
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence, Set, Tuple

# name -> list of op sequences (root first, following input 0 downwards)
REF_PATTERNS: List[Tuple[str, List[List[str]]]] = [
    ("conv2d_bn_add_relu", [["nn.relu", "add", "nn.batch_norm", "nn.bias_add", "nn.conv2d"],
                            ["nn.relu", "add", "nn.batch_norm", "nn.conv2d"]]),
    ("conv2d_bn_add", [["add", "nn.batch_norm", "nn.bias_add", "nn.conv2d"],
                       ["add", "nn.batch_norm", "nn.conv2d"]]),
    ("conv2d_bn_act", [["nn.relu", "nn.batch_norm", "nn.bias_add", "nn.conv2d"],
                       ["nn.relu", "nn.batch_norm", "nn.conv2d"],
                       ["clip", "nn.batch_norm", "nn.bias_add", "nn.conv2d"],
                       ["clip", "nn.batch_norm", "nn.conv2d"]]),
    ("conv2d_bn", [["nn.batch_norm", "nn.bias_add", "nn.conv2d"], ["nn.batch_norm", "nn.conv2d"]]),
    ("conv2d_bias_act", [["nn.relu", "nn.bias_add", "nn.conv2d"], ["nn.relu", "nn.conv2d"]]),
    ("dense_bias_act", [["nn.gelu", "nn.bias_add", "nn.dense"], ["nn.relu", "nn.bias_add", "nn.dense"],
                        ["nn.bias_add", "nn.dense"]]),
]


class _UF:
    def __init__(self, n):
        self.p = list(range(n))

    def find(self, a):
        while self.p[a] != a:
            self.p[a] = self.p[self.p[a]]
            a = self.p[a]
        return a

    def union(self, a, b):
        a, b = self.find(a), self.find(b)
        if a != b:
            self.p[max(a, b)] = min(a, b)


def composites(graph, patterns=REF_PATTERNS):
    """[(pattern name, [member names in graph order])] in root order."""
    nodes = graph.nodes
    pos = {n.name: i for i, n in enumerate(nodes)}
    by = {n.name: n for n in nodes}
    users: Dict[str, List[str]] = {n.name: [] for n in nodes}
    for n in nodes:
        for i in n.inputs:
            if i in users:
                users[i].append(n.name)
    outs = set(graph.outputs)
    taken: Set[str] = set()
    found = []
    for pname, seqs in patterns:
        for root in reversed(nodes):
            if root.name in taken:
                continue
            for seq in seqs:  # longest first
                chain, cur, ok = [], root.name, True
                for k, op in enumerate(seq):
                    n = by.get(cur)
                    if n is None or n.op != op or n.name in taken:
                        ok = False
                        break
                    chain.append(n.name)
                    if k + 1 < len(seq):
                        if not n.inputs:
                            ok = False
                            break
                        cur = n.inputs[0]
                if not ok:
                    continue
                inner = set(chain)
                if any(c in outs or any(u not in inner for u in users[c]) for c in chain[1:]):
                    continue
                found.append((pname, sorted(chain, key=pos.__getitem__)))
                taken.update(chain)
                break
    found.sort(key=lambda c: pos[c[1][-1]])
    return found


def partition(graph, supported_ops, max_ops: Optional[int] = None, fallback_no_mac=True,
              patterns=REF_PATTERNS, node_supported=None):
    """Regions as lists of node names (graph order), sorted by first node."""
    nodes = graph.nodes
    pos = {n.name: i for i, n in enumerate(nodes)}
    comps = composites(graph, patterns)
    member_of = {}
    for ci, (_, mem) in enumerate(comps):
        for m in mem:
            member_of[m] = ci
    # units in topological order: a composite sits at its last member
    units: List[List[str]] = []
    for n in nodes:
        if n.name in member_of:
            mem = comps[member_of[n.name]][1]
            if n.name == mem[-1]:
                units.append(list(mem))
        else:
            units.append([n.name])
    uid = {m: u for u, mem in enumerate(units) for m in mem}
    nu = len(units)
    by = {n.name: n for n in nodes}
    edges = set()
    for u, mem in enumerate(units):
        for m in mem:
            for i in by[m].inputs:
                if i in uid and uid[i] != u:
                    edges.add((uid[i], u))
    # transitive closure (reach[a] = units reachable from a)
    succ = [[] for _ in range(nu)]
    for a, b in edges:
        succ[a].append(b)
    reach = [set() for _ in range(nu)]
    for a in reversed(range(nu)):
        for b in succ[a]:
            reach[a].add(b)
            reach[a] |= reach[b]

    def ok(n):
        if node_supported is not None:
            return node_supported(n)
        return n.op in supported_ops

    sup = [all(ok(by[m]) for m in mem) for mem in units]
    uf = _UF(nu)
    members: Dict[int, Set[int]] = {}

    def convex(s: Set[int]) -> bool:
        for a in s:
            for b in reach[a]:
                if b in s:
                    continue
                if reach[b] & s:
                    return False
        return True

    for u in range(nu):
        if not sup[u]:
            continue
        members[u] = {u}
        producers = sorted({uf.find(a) for (a, b) in edges if b == u and sup[a]})
        cur = u
        for r in sorted(producers, key=lambda r: min(members[r])):
            cand = members[uf.find(cur)] | members[r]
            if convex(cand):
                a, b = uf.find(cur), r
                merged = members.pop(a) | members.pop(b)
                uf.union(a, b)
                members[uf.find(a)] = merged
                cur = uf.find(a)
    regions = sorted((sorted(s) for s in members.values()), key=lambda s: s[0])
    if max_ops is not None:
        cut = []
        for r in regions:
            for k in range(0, len(r), max_ops):
                cut.append(r[k:k + max_ops])
        regions = cut

    def macs(u):
        t = 0
        for m in units[u]:
            n = by[m]
            if n.op in ("nn.conv2d", "nn.dense"):
                t += 1
        return t

    if fallback_no_mac:
        regions = [r for r in regions if sum(macs(u) for u in r) > 0]
    out = []
    for r in sorted(regions, key=lambda s: s[0]):
        names = set(m for u in r for m in units[u])
        out.append([n.name for n in nodes if n.name in names])
    return out


def is_convex(graph, region_nodes: Sequence[str]) -> bool:
    """Brute force: no path from the region to itself through outside nodes."""
    s = set(region_nodes)
    users: Dict[str, List[str]] = {n.name: [] for n in graph.nodes}
    for n in graph.nodes:
        for i in n.inputs:
            if i in users:
                users[i].append(n.name)
    for start in s:
        stack = [u for u in users[start] if u not in s]
        seen = set(stack)
        while stack:
            v = stack.pop()
            for w in users[v]:
                if w in s:
                    return False
                if w not in seen:
                    seen.add(w)
                    stack.append(w)
    return True
