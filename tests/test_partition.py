"""Partitioning bookkeeping (Section 3.1) -- bit-exact against hand-worked
expectations, the paper's Table 2 region counts, and an independently written
reference (oracle/partition_ref.py)."""
import random

import pytest

from oracle import partition_ref as ref
from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import partition as P
from paper_2105_03215_gb300.inputs import Graph, Node


def _all_supported(g):
    return {n.op: (lambda _n: True) for n in g.nodes}


def _regions(res):
    return [res.region_nodes(r) for r in range(len(res.regions))]


# ------------------------------------------------------------ pattern language

def _tiny(bias: bool, extra_consumer=False):
    b = I._Builder("tiny")
    x = b.input("x", (1, 4, 4, 8))
    c = b.conv2d(x, 8, 3)
    t = b.bias_add(c) if bias else c
    y = b.relu(t)
    outs = [y]
    if extra_consumer:
        outs.append(b.relu(t))
    g, _ = I._finish(b, outs, 0, draw=False)
    return g


def test_listing_pattern_matches_with_and_without_optional_bias():
    """The Conv2D-(bias)-ReLU listing of Section 3.1.1: both sequences match."""
    table = [("conv2d_pattern", P.conv2d_bias_act_pattern)]
    for bias in (False, True):
        g = _tiny(bias)
        comps = P.merge_composite(g, table)
        assert len(comps) == 1 and comps[0].name == "conv2d_pattern"
        assert comps[0].members == [n.name for n in g.nodes]


def test_longer_optional_match_wins():
    g = _tiny(True)
    comps = P.merge_composite(g, [("p", P.conv2d_bias_act_pattern)])
    assert "bias_add_0" in comps[0].members


def test_match_rejected_when_inner_node_escapes():
    g = _tiny(True, extra_consumer=True)  # bias_add output also read by a second relu
    comps = P.merge_composite(g, [("p", P.conv2d_bias_act_pattern)])
    assert comps == []
    assert ref.composites(g, [("p", [["nn.relu", "nn.bias_add", "nn.conv2d"]])]) == []


def test_composites_match_reference_on_resnet50():
    g, _ = I.resnet50(N=1, draw=False)
    mine = [(c.name, c.members) for c in P.merge_composite(g, P.PATTERN_TABLE)]
    assert mine == ref.composites(g)
    names = [c[0] for c in mine]
    assert names.count("conv2d_bn_add_relu") == 16      # one per bottleneck
    assert names.count("conv2d_bn") == 4                # downsample branches
    assert names.count("conv2d_bn_act") == 33
    assert names.count("dense_bias_act") == 1


def test_mobilenet_v2_composites_and_regions_match_reference():
    # every inverted-residual block with a shortcut ends in conv + BN + add
    g, _ = I.mobilenet_v2(draw=False)
    mine = [(c.name, c.members) for c in P.merge_composite(g, P.PATTERN_TABLE)]
    assert mine == ref.composites(g)
    names = [c[0] for c in mine]
    assert names.count("conv2d_bn_add") == 10
    res = P.partition(g, P.PATTERN_TABLE, target=P.TARGET, max_ops=1)
    regs = _regions(res)
    assert regs == ref.partition(g, set(P.annotations(P.TARGET)), max_ops=1)
    assert len(regs) == 53  # 52 conv composites + the classifier; global avg pool on the host
    on_host = [n.op for n in g.nodes if not any(n.name in r for r in regs)]
    assert on_host == ["nn.global_avg_pool2d"]


# ------------------------------------------------------------ Table 2 pins

@pytest.mark.parametrize("builder", [I.resnet18, I.resnet50, I.mobilenet_v2, I.vgg19])
@pytest.mark.parametrize("fallback", [False, True])
def test_classification_cnns_partition_into_one_region(builder, fallback):
    """Table 2: with every operator supported, each classification CNN is one
    subgraph, with and without the cost-based rule."""
    g, _ = builder(draw=False) if builder is not I.resnet50 else builder(N=1, draw=False)
    res = P.partition(g, P.PATTERN_TABLE, annotators=_all_supported(g), fallback_no_mac=fallback)
    assert len(res.regions) == 1
    assert res.offload_ratio() == (1.0, 1.0)
    assert _regions(res) == ref.partition(g, {n.op for n in g.nodes}, fallback_no_mac=fallback)


def test_resnet50_on_this_target_keeps_pools_on_host():
    g, _ = I.resnet50(N=1, draw=False)
    res = P.partition(g, P.PATTERN_TABLE, target=P.TARGET)
    regs = _regions(res)
    assert len(regs) == 3  # stem | body | classifier ; max/avg pool stay on the host
    node_ratio, mac_ratio = res.offload_ratio()
    assert mac_ratio == 1.0 and node_ratio == (len(g.nodes) - 2) / len(g.nodes)
    supported = set(P.annotations(P.TARGET))
    assert regs == ref.partition(g, supported)


def test_resnet50_one_composite_per_region_gives_54_regions():
    g, _ = I.resnet50(N=1, draw=False)
    res = P.partition(g, P.PATTERN_TABLE, target=P.TARGET, max_ops=1)
    regs = _regions(res)
    assert len(regs) == 54
    convs = [sum(g.node(m).op == "nn.conv2d" for m in r) for r in regs]
    dens = [sum(g.node(m).op == "nn.dense" for m in r) for r in regs]
    assert sum(convs) == 53 and sum(dens) == 1 and all(c + d == 1 for c, d in zip(convs, dens))
    assert regs == ref.partition(g, set(P.annotations(P.TARGET)), max_ops=1)
    for r in regs:
        assert ref.is_convex(g, r)


def test_bottleneck_cap_three_gives_one_region_per_block():
    g, _ = I.resnet50(N=1, draw=False)
    res = P.partition(g, P.PATTERN_TABLE, target=P.TARGET, max_ops=4)
    assert _regions(res) == ref.partition(g, set(P.annotations(P.TARGET)), max_ops=4)


@pytest.mark.parametrize("max_ops,count", [(16, 6), (None, 3)])
def test_resnet50_granularities_of_the_partition_study(max_ops, count):
    # the region counts the granularity study runs: every cut matches the
    # reference checker and keeps every region convex
    g, _ = I.resnet50(N=1, draw=False)
    res = P.partition(g, P.PATTERN_TABLE, target=P.TARGET, max_ops=max_ops)
    regs = _regions(res)
    assert regs == ref.partition(g, set(P.annotations(P.TARGET)), max_ops=max_ops)
    assert len(regs) == count
    for r in regs:
        assert ref.is_convex(g, r)


# ------------------------------------------------------------ Fig. 3 reconstruction

def test_figure3_counts_reconstruction():
    """Reconstruction of the Section 3.1 example (its figure is not available):
    Region 1 holds 4N+1 supported operators, an unsupported operator follows,
    Region 2 holds K operators plus one composite; a cap of 3N operators splits
    Region 1 into two regions."""
    N, K = 2, 3
    b = I._Builder("fig3")
    t = b.input("x", (1, 8, 8, 8))
    for _ in range(4 * N + 1):
        t = b.relu(t)
    t = b._add("nn.unsupported", [t], (1, 8, 8, 8))
    for _ in range(K):
        t = b.relu(t)
    t = b.relu(b.bias_add(b.conv2d(t, 8, 3)))
    g, _ = I._finish(b, [t], 0, draw=False)
    table = [("conv2d_pattern", P.conv2d_bias_act_pattern)]
    ann = {op: (lambda n: True) for op in ("nn.relu", "nn.conv2d", "nn.bias_add")}
    res = P.partition(g, table, annotators=ann, fallback_no_mac=False)
    assert [len(r) for r in res.regions] == [4 * N + 1, K + 1]   # units; composite = 1
    res = P.partition(g, table, annotators=ann, fallback_no_mac=False, max_ops=3 * N)
    assert [len(r) for r in res.regions] == [3 * N, N + 1, K + 1]
    # with the MAC rule, the two conv-free regions fall back to the host
    res = P.partition(g, table, annotators=ann, fallback_no_mac=True, max_ops=3 * N)
    assert [len(r) for r in res.regions] == [K + 1]
    rp = [("conv2d_pattern", [["nn.relu", "nn.bias_add", "nn.conv2d"]])]
    assert _regions(res) == ref.partition(g, set(ann), max_ops=3 * N, patterns=rp)


# ------------------------------------------------------------ random DAGs

def _random_dag(seed, n=10):
    rnd = random.Random(seed)
    nodes = []
    names = ["in"]
    for i in range(n):
        k = 1 if rnd.random() < 0.6 or len(names) < 2 else 2
        ins = rnd.sample(names, k)
        op = "nn.relu" if rnd.random() < 0.65 else "host_op"
        nodes.append(Node(f"n{i}", op, ins, shape=(1, 2, 2, 8)))
        names.append(f"n{i}")
    users = {nm: 0 for nm in names}
    for nd in nodes:
        for i in nd.inputs:
            users[i] += 1
    outs = [nd.name for nd in nodes if users[nd.name] == 0]
    return Graph({"in": (1, 2, 2, 8)}, nodes, outs, "rand")


@pytest.mark.parametrize("seed", range(60))
def test_random_dags_match_reference_and_are_convex(seed):
    g = _random_dag(seed)
    ann = {"nn.relu": lambda n: True}
    for cap in (None, 2):
        res = P.partition(g, [], annotators=ann, fallback_no_mac=False, max_ops=cap)
        regs = _regions(res)
        assert regs == ref.partition(g, {"nn.relu"}, max_ops=cap, fallback_no_mac=False, patterns=[])
        covered = sorted(m for r in regs for m in r)
        assert covered == sorted(nd.name for nd in g.nodes if nd.op == "nn.relu")
        for r in regs:
            assert ref.is_convex(g, r)


# ------------------------------------------------------------ brute-force maximality

def _dense_dag(seed, n=10):
    """Random DAG with one- to three-input nodes, about three quarters of
    them supported."""
    rnd = random.Random(1000 + seed)
    nodes, names = [], ["in"]
    for i in range(n):
        k = 1 if rnd.random() < 0.45 or len(names) < 2 else min(len(names), rnd.choice([2, 3]))
        ins = rnd.sample(names, k)
        op = "nn.relu" if rnd.random() < 0.75 else "host_op"
        nodes.append(Node(f"n{i}", op, ins, shape=(1, 2, 2, 8)))
        names.append(f"n{i}")
    users = {nm: 0 for nm in names}
    for nd in nodes:
        for i in nd.inputs:
            users[i] += 1
    outs = [nd.name for nd in nodes if users[nd.name] == 0]
    return Graph({"in": (1, 2, 2, 8)}, nodes, outs, "rand")


def _weakly_connected(g, names):
    s = set(names)
    adj = {m: set() for m in s}
    for nd in g.nodes:
        if nd.name in s:
            for i in nd.inputs:
                if i in s:
                    adj[nd.name].add(i)
                    adj[i].add(nd.name)
    start = next(iter(s))
    seen, stack = {start}, [start]
    while stack:
        for w in adj[stack.pop()]:
            if w not in seen:
                seen.add(w)
                stack.append(w)
    return seen == s


@pytest.mark.parametrize("seed", range(150))
def test_greedy_merge_leaves_no_convex_union_of_regions(seed):
    """Section 3.1.2 merges consecutive supported operators greedily to make
    regions as large as possible.  Checked by brute force on <= 10-node DAGs:
    every supported node is in exactly one region, every region is convex and
    connected, and no union of two or more regions (every subset is tried) is
    both connected -- its operators consecutive -- and convex, i.e. no region
    could still grow by absorbing others."""
    import itertools
    g = _random_dag(seed) if seed % 2 else _dense_dag(seed)
    res = P.partition(g, [], annotators={"nn.relu": lambda n: True}, fallback_no_mac=False)
    regs = _regions(res)
    assert regs == ref.partition(g, {"nn.relu"}, fallback_no_mac=False, patterns=[])
    covered = sorted(m for r in regs for m in r)
    assert covered == sorted(nd.name for nd in g.nodes if nd.op == "nn.relu")
    for r in regs:
        assert ref.is_convex(g, r) and _weakly_connected(g, r)
    for size in range(2, len(regs) + 1):
        for sub in itertools.combinations(range(len(regs)), size):
            union = [m for i in sub for m in regs[i]]
            assert not (_weakly_connected(g, union) and ref.is_convex(g, union)), \
                f"regions {[regs[i] for i in sub]} could be merged into one convex region"
