"""CPU tests of the C ABI: the library builds and loads without a GPU,
exports every function the headers declare, and its host-side planning
(validation, epilogue fusion, batch-norm folding, weight packing) behaves as
specified.  No test here calls a CUDA function."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

from paper_2105_03215_gb300 import abi
from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import partition as P
from paper_2105_03215_gb300 import region as R

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_functions():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names.update(re.findall(r"\b(byoc_[a-z0-9_]+)\s*\(", src))
    return names


def test_library_exports_every_declared_function():
    path = abi.lib().__getattribute__("_name")
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (byoc_\w+)", out))
    declared = _declared_functions()
    assert declared, "no declarations parsed"
    assert declared <= exported, f"declared but not exported: {sorted(declared - exported)}"
    assert set(abi.declared_symbols()) == declared


def _plan(g, options=0, **kw):
    return R.whole_graph_region(g, options=options).plan(**kw)


def test_plan_fuses_composites_into_launches():
    rep = _plan(I.resnet_bottleneck(N=2, H=14, W=14, C=256, width=64)[0])
    assert rep.n_launches == 3
    assert [rep.n_ops[i] for i in range(3)] == [3, 3, 4]      # conv+bn+relu x2, conv+bn+add+relu
    assert [rep.act[i] for i in range(3)] == [1, 1, 1]
    assert rep.residual[2] == 0 and rep.residual[0] == -1     # residual = region input 0
    assert [rep.im2col[i] for i in range(3)] == [0, 2, 0]     # 1x1 as GEMM, 3x3 in slab mode
    rep = _plan(I.bert_ffn(M=64, D=128, F=256)[0])
    assert rep.n_launches == 2 and rep.act[0] == 3 and rep.act[1] == 0
    rep = _plan(I.mbv2_dw_pw(N=1, H=8, W=8)[0])
    assert [rep.kind[i] for i in range(rep.n_launches)] == [abi.LAUNCH_DEPTHWISE, abi.LAUNCH_GEMM]
    assert rep.act[0] == 2


def test_plan_fuses_depthwise_into_the_pointwise_when_asked():
    # depthwise + BN + ReLU6 -> 1x1 + BN: one fused launch (the depthwise output stays on chip)
    assert _plan(I.mbv2_dw_pw(N=1, H=8, W=8)[0]).n_launches == 2  # the default: two launches
    rep = _plan(I.mbv2_dw_pw(N=1, H=8, W=8)[0], options=abi.OPT_FUSE_DW_PW)
    assert rep.n_launches == 1 and rep.kind[0] == abi.LAUNCH_DWPW
    assert rep.n_ops[0] == 5 and rep.act[0] == 0
    assert (rep.gemm_m[0], rep.gemm_n[0], rep.gemm_k[0], rep.tile_n[0]) == (64, 24, 144, 32)
    # a depthwise whose output is also a region output stays a launch of its own
    g, _ = I.mbv2_dw_pw(N=1, H=8, W=8)
    reg = R.Region(g, [n.name for n in g.nodes], "both", outputs=[g.nodes[2].name, g.outputs[0]],
                   options=abi.OPT_FUSE_DW_PW)
    rep = reg.plan()
    assert [rep.kind[i] for i in range(rep.n_launches)] == [abi.LAUNCH_DEPTHWISE, abi.LAUNCH_GEMM]
    assert rep.act[0] == 2


def test_plan_stem_inserts_the_pixel_pair_layout():
    g, _ = I.resnet50(N=1, H=32, W=32)
    rep = R.Region(g, [n.name for n in g.nodes[:3]], "stem").plan()
    assert rep.n_launches == 2
    assert rep.kind[0] == abi.LAUNCH_S2D and rep.kind[1] == abi.LAUNCH_GEMM
    # 7x7/2 over 3 channels -> 1x4 stride-1 conv over 8 rows x 2 pixels x 4 channels (slab mode)
    assert rep.gemm_k[1] == 4 * 64 and rep.tile_k[1] == 64 and rep.im2col[1] == 2
    # 3x3/2 -> 1x2 over 4 rows x 2 pixels x 4 channels (32-element k-blocks)
    g, _ = I.stem(N=1, H=32, W=32, k=3, cout=32, C=3)
    rep = R.whole_graph_region(g).plan()
    assert rep.gemm_k[1] == 2 * 32 and rep.tile_k[1] == 32 and rep.im2col[1] == 2


def test_stem_weights_follow_the_pixel_pair_definition():
    # w'[k][b][r*8 + dx*4 + c] = w[k][c][r][2b+dx], zero where r or 2b+dx >= 7 or c >= 3
    g, _ = I.resnet50(N=1, H=32, W=32)
    reg = R.Region(g, [n.name for n in g.nodes[:3]], "stem")
    rep = reg.plan()
    w = g.nodes[0].consts["weight"].astype(np.float64)            # [64, 3, 7, 7]
    bn = g.nodes[1]
    scale = bn.consts["gamma"].astype(np.float64) / np.sqrt(
        bn.consts["moving_var"].astype(np.float64) + 1e-5)
    packed = np.frombuffer(reg.plan_constants(1, 0), dtype=np.uint16).reshape(-1, rep.gemm_k[1])
    expect = np.zeros((64, 4, 8, 2, 4), dtype=np.float64)          # [k][b][r][dx][c]
    for b in range(4):
        for r in range(7):
            for dx in range(2):
                if 2 * b + dx < 7:
                    expect[:, b, r, dx, :3] = w[:, :, r, 2 * b + dx]
    expect *= scale[:, None, None, None, None]
    want = I.bf16_bits(expect.reshape(64, -1).astype(np.float32))
    assert np.array_equal(packed[:64], want)
    # the flop count is the 7x7x3 convolution's, not the padded GEMM's
    assert rep.flops == pytest.approx(2.0 * 64 * 16 * 16 * 7 * 7 * 3, rel=1e-12)


def test_stem_layout_is_the_image_size_at_any_batch():
    # xq: 232 rows x 230 columns x 4 channels of bf16 per image (2 Ho + 8 rows,
    # 2 (Wo + 3) columns), read by one GEMM launch whatever the batch
    for N in (64, 170):
        g, _ = I.stem(N=N, H=224, W=224)
        rep = R.whole_graph_region(g).plan()
        assert rep.n_launches == 2 and rep.gemm_m[1] == N * 112 * 112
        assert [rep.kind[i] for i in range(2)] == [abi.LAUNCH_S2D, abi.LAUNCH_GEMM]
        assert rep.flops == pytest.approx(2.0 * N * 112 * 112 * 64 * 7 * 7 * 3, rel=1e-12)
        assert rep.workspace_bytes <= 256 + N * 232 * 230 * 4 * 2 + 256
        assert rep.resident_b[1] == 1 and rep.pair_units[1] == 1


def test_plan_flops_match_mac_count():
    for g, _ in [I.bert_ffn(), I.resnet_bottleneck(), I.conv_bias_relu()]:
        assert _plan(g).flops == pytest.approx(I.region_flops(g), rel=1e-12)


def test_packed_weights_are_folded_rounded_and_k_major():
    g, _ = I.conv_bias_relu(N=1, H=8, W=8, C=64, K=32, seed=3)
    g2, _ = I.mbv2_dw_pw(N=1, H=8, W=8, C=64, Cout=32)
    # conv -> bn (from the pointwise part of g2) : fold checked on the GEMM launch
    reg = R.whole_graph_region(g2, options=abi.OPT_FUSE_DW_PW)
    rep = reg.plan()
    pw = g2.nodes[3]
    bn = g2.nodes[4]
    s = bn.consts["gamma"].astype(np.float64) / np.sqrt(bn.consts["moving_var"].astype(np.float64) + 1e-5)
    shift = bn.consts["beta"] - s * bn.consts["moving_mean"]
    w = pw.consts["weight"][:, :, 0, 0].astype(np.float64) * s[:, None]
    assert rep.kind[0] == abi.LAUNCH_DWPW
    raw = np.frombuffer(reg.plan_constants(0, 2), dtype=np.uint16)   # the fused launch's 1x1 weights
    packed = raw.reshape(rep.tile_n[0], -1)
    assert packed.shape == (32, 64)
    assert np.array_equal(packed[:32, :64], I.bf16_bits(w.astype(np.float32)))
    bias = np.frombuffer(reg.plan_constants(0, 3), dtype=np.float32)
    np.testing.assert_allclose(bias[:32], shift, rtol=1e-6, atol=1e-7)
    # 3x3 conv: column index = (tap r*3+s) * Cin_pad + c
    reg = R.whole_graph_region(g)
    rep = reg.plan()
    packed = np.frombuffer(reg.plan_constants(0, 0), dtype=np.uint16).reshape(-1, rep.gemm_k[0])
    wc = g.nodes[0].consts["weight"]
    for (k, c, r, t) in [(0, 0, 0, 0), (5, 17, 2, 1), (31, 63, 1, 2)]:
        assert packed[k, (r * 3 + t) * 64 + c] == I.bf16_bits(wc[k, c, r, t:t + 1])[0]


def _bad(mutate):
    g, _ = I.conv_bias_relu(N=1, H=8, W=8, C=64, K=64)
    reg = R.whole_graph_region(g)
    desc, keep = reg.to_desc()
    mutate(desc)
    rep = abi.PlanReport()
    return abi.lib().byoc_plan(ctypes.byref(desc), 148, ctypes.byref(rep))


def test_validation_rejects_malformed_descriptors():
    assert _bad(lambda d: None) == abi.OK
    assert _bad(lambda d: setattr(d, "abi_version", 99)) == abi.ERR_INVALID_ARG
    assert _bad(lambda d: setattr(d, "n_ops", 0)) == abi.ERR_INVALID_ARG
    def bad_shape(d):
        d.tensors[1].shape[1] = 7
    assert _bad(bad_shape) == abi.ERR_INVALID_ARG
    def null_weight(d):
        d.ops[0].consts[0] = None
    assert _bad(null_weight) == abi.ERR_INVALID_ARG
    def bad_order(d):
        d.ops[1].in_[0] = 3   # reads the output of a later op
    assert _bad(bad_order) == abi.ERR_INVALID_ARG
    def fp32_act(d):
        d.tensors[0].dtype = abi.FP32
    assert _bad(fp32_act) == abi.ERR_UNSUPPORTED
    assert b"" != abi.lib().byoc_last_error()


def test_unsupported_chains_are_rejected_not_run_elsewhere():
    b = I._Builder("lone_relu")
    x = b.input("x", (1, 4, 4, 8))
    y = b.relu(x)
    g, _ = I._finish(b, [y], 0)
    with pytest.raises(abi.ByocError) as e:
        R.whole_graph_region(g).plan()
    assert e.value.status == abi.ERR_UNSUPPORTED
    g, _ = I.conv_bias_relu(N=1, H=8, W=8, C=64, K=20)   # Cout not a multiple of 8
    with pytest.raises(abi.ByocError) as e:
        R.whole_graph_region(g).plan()
    assert e.value.status == abi.ERR_UNSUPPORTED


def test_every_mobilenet_v2_region_plans_at_224():
    # The stride-2 depthwise over 112 x 112 x 96 needs 9 input rows x 113
    # columns x 96 channels = 195 KB for a full-width tile of 4 output rows:
    # the planner narrows the column tile until one buffer holds it.
    from paper_2105_03215_gb300 import partition as P
    g, _ = I.mobilenet_v2(N=64, H=224, W=224, draw=True)
    res = P.partition(g, P.PATTERN_TABLE, target=P.TARGET, max_ops=1)
    regions = res.region_objects()
    assert len(regions) == 53
    for r in regions:
        rep = r.plan()
        assert rep.n_launches >= 1
    assert sum(r.plan().flops for r in regions) == pytest.approx(I.region_flops(g), rel=1e-9)


def test_slab_pool_keeps_small_weight_matrices_resident():
    # one column tile whose packed weights fit beside two slabs: loaded once
    # per CTA; the slabs take the rest of the pool, up to 8 in flight
    g, _ = I.conv_bias_relu(N=2, H=56, W=56, C=64, K=64)
    rep = _plan(g)
    assert rep.im2col[0] == 2 and rep.tile_n[0] == 64 and rep.gemm_k[0] == 576
    assert rep.resident_b[0] == 1 and 2 <= rep.slab_slots[0] <= 8
    g, _ = I.resnet50(N=1, H=32, W=32)
    rep = R.Region(g, [n.name for n in g.nodes[:3]], "stem").plan()
    assert rep.resident_b[1] == 1 and rep.slab_slots[1] >= 4     # 1 x 115-pixel slabs of 16 KB
    # 3x3 over 128 channels to 128: 18 k-blocks x 16 KB do not fit; ringed, slabs double-buffered or more
    g, _ = I.conv_bias_relu(N=2, H=28, W=28, C=128, K=128)
    rep = _plan(g)
    assert rep.im2col[0] == 2 and rep.resident_b[0] == 0 and rep.slab_slots[0] >= 2
    # other modes carry no slab pool
    rep = _plan(I.bert_ffn(M=64, D=128, F=256)[0])
    assert rep.resident_b[0] == 0 and rep.slab_slots[0] == 0


def _report_tuple(rep):
    n = rep.n_launches
    fields = ["kind", "first_op", "n_ops", "act", "residual", "gemm_m", "gemm_n", "gemm_k", "tile_n",
              "tile_k", "im2col", "grid", "resident_b", "slab_slots"]
    return (n, tuple(tuple(getattr(rep, f)[:n]) for f in fields), rep.flops, rep.bytes,
            rep.const_bytes, rep.workspace_bytes)


@pytest.mark.parametrize("make", [
    lambda: R.whole_graph_region(I.resnet_bottleneck(N=2, H=14, W=14, C=256, width=64)[0]),
    lambda: R.whole_graph_region(I.bert_ffn(M=64, D=128, F=256)[0]),
    lambda: R.whole_graph_region(I.mbv2_dw_pw(N=1, H=8, W=8)[0]),
    lambda: R.Region(I.resnet50(N=1, H=32, W=32)[0], [n.name for n in I.resnet50(N=1, H=32, W=32)[0].nodes[:3]], "stem"),
])
def test_serialized_plan_round_trips(make):
    # Section 3.3 option 3: the serialised plan holds the same launches,
    # figures and constants as the plan it was written from
    reg = make()
    blob = reg.plan_serialized(152)
    assert blob[:8] == b"BYOCPLN1"
    assert _report_tuple(R.load_plan_report(blob)) == _report_tuple(reg.plan(152))
    # the packed constants of every launch are in the blob byte for byte
    rep = reg.plan(152)
    for i in range(rep.n_launches):
        if rep.kind[i] == abi.LAUNCH_S2D:
            continue
        w = reg.plan_constants(i, 0, 152)
        assert blob.find(w) > 0
    # deterministic: planning twice gives the same bytes
    assert reg.plan_serialized(152) == blob


def test_serialized_plan_rejects_damaged_bytes():
    reg = R.whole_graph_region(I.conv_bias_relu(N=1, H=8, W=8, C=64, K=64)[0])
    blob = bytearray(reg.plan_serialized(152))
    for bad, status in [
        (blob[:-1], abi.ERR_INVALID_ARG),                               # truncated
        (blob + b"\0", abi.ERR_INVALID_ARG),                            # trailing bytes
        (b"NOTAPLAN" + blob[8:], abi.ERR_INVALID_ARG),                  # magic
        (blob[:200] + bytes([blob[200] ^ 1]) + blob[201:], abi.ERR_INVALID_ARG),  # checksum
        (blob[:8] + (99).to_bytes(4, "little") + blob[12:], abi.ERR_UNSUPPORTED),  # format
        (b"", abi.ERR_INVALID_ARG),
    ]:
        with pytest.raises(abi.ByocError) as e:
            R.load_plan_report(bytes(bad))
        assert e.value.status == status


def test_fusion_follows_the_composites_at_every_region_size():
    # the engine fuses a region's ops greedily in descriptor order; regions
    # list their ops composite by composite, so a downsample block fuses the
    # same way (conv3 + BN + add + ReLU, residual = the downsample output)
    # whether it is one region per composite or part of a larger region
    from collections import Counter
    from paper_2105_03215_gb300 import partition as P
    g, _ = I.resnet50(N=1, H=64, W=64)

    def launches(max_ops):
        res = P.partition(g, P.PATTERN_TABLE, target=P.TARGET, max_ops=max_ops)
        c = Counter()
        for r in res.region_objects():
            rep = r.plan(152)
            for i in range(rep.n_launches):
                c[(rep.kind[i], rep.gemm_m[i], rep.gemm_n[i], rep.gemm_k[i], rep.act[i],
                   rep.residual[i] >= 0, rep.n_ops[i], rep.tile_n[i])] += 1
        return c

    base = launches(1)
    for mo in (4, 16, None):
        assert launches(mo) == base, mo


def test_split_k_for_deep_reductions_with_few_tiles():
    # BERT FFN's second dense (1024 x 3072 -> 768): 48 tiles of 128 x 128 would
    # leave most SMs idle for 48 k-blocks; three CTAs share each tile's
    # k-blocks instead (144 CTAs); the first dense (GELU epilogue) keeps one
    # CTA per tile, 192 tiles of 128 x 128 on the 152 SMs
    rep = \
        R.whole_graph_region(I.bert_ffn()[0]).plan(152)
    assert rep.splits[0] == 1 and rep.tile_n[0] == 128 and rep.grid[0] == 152
    assert rep.splits[1] == 3 and rep.tile_n[1] == 128 and rep.grid[1] == 144
    # fp32 partials [3][1024][768] + counters live in the handle's workspace
    assert rep.workspace_bytes >= 3 * 1024 * 768 * 4 + 1024 * 3072 * 2
    # a shallow reduction is not split
    rep = R.whole_graph_region(I.conv_bias_relu(N=2, H=56, W=56, C=64, K=64)[0]).plan(152)
    assert rep.splits[0] == 1


def test_pair_units_only_where_a_tile_has_few_mmas():
    # Pair units (two adjacent tiles per unit, resident weights) for slabs
    # with at most 16 MMAs per tile: the ResNet-50 stem's 1x4 GEMM at N=64.
    # The stride-1 3x3 layers (36+ MMAs per tile) stay single, and so does
    # the stem at N=1, where pairs would leave SMs idle.
    for N, want in ((64, 1), (1, 0)):
        g, _ = I.resnet50(N=N, H=224, W=224)
        part = P.partition(g, P.PATTERN_TABLE, target=P.TARGET, max_ops=1)
        slabs = 0
        for ri in range(len(part.region_objects())):
            rep = R.Region(g, part.region_nodes(ri), f"r{ri}").plan(152)
            for i in range(rep.n_launches):
                if rep.kind[i] != abi.LAUNCH_GEMM:
                    continue
                if rep.im2col[i] == 2:
                    slabs += 1
                stem = rep.n_launches == 2 and i == 1
                assert rep.pair_units[i] == (want if stem else 0), (N, ri)
        assert slabs == 12
    # a 1x4 conv over 64 channels (the stem GEMM's shape) pairs as well
    g, _ = I.conv_general(kernel=(1, 4), strides=(1, 1), padding=(0, 0, 0, 0), dilation=(1, 1),
                          N=32, H=24, W=100, C=64, K=64)
    rep = _plan(g)
    assert rep.pair_units[0] == 1 and rep.resident_b[0] == 1 and rep.slab_slots[0] >= 2


def test_source_digest_is_independent_of_the_checkout_path(tmp_path, monkeypatch):
    # bench.py reports the profiled DRAM traffic only while the sources hash
    # to the digest stored beside it: a copy of the same sources elsewhere
    # must hash the same, and any change of a source must not
    import shutil
    from paper_2105_03215_gb300 import build as B
    want = B._digest()
    root = tmp_path / "copy"
    shutil.copytree(B.CSRC, root / "pkg" / "csrc")
    shutil.copytree(B.INCLUDE, root / "include")
    csrc, inc = str(root / "pkg" / "csrc"), str(root / "include")
    monkeypatch.setattr(B, "FLAGS", [{B.INCLUDE: inc, B.CSRC: csrc}.get(f, f) for f in B.FLAGS])
    monkeypatch.setattr(B, "CSRC", csrc)
    monkeypatch.setattr(B, "INCLUDE", inc)
    assert B._digest() == want
    with open(os.path.join(csrc, "ptx.cuh"), "a") as f:
        f.write("\n")
    assert B._digest() != want


@pytest.mark.parametrize("k,C,cout", [(3, 3, 32), (5, 4, 48), (7, 1, 64)])
def test_stem_weights_for_every_filter_size(k, C, cout):
    # w'[k][b][r*8 + dx*4 + c] = w[k][c][r][2b+dx] with R = 4 row taps (k = 3)
    # or 8 (k = 5, 7) and zero where r >= k, 2b + dx >= k or c >= C
    g, _ = I.stem(N=1, H=32, W=30, k=k, cout=cout, C=C)
    reg = R.whole_graph_region(g)
    rep = reg.plan()
    k2, Rr = (k + 1) // 2, (4 if k <= 3 else 8)
    assert rep.gemm_k[1] == k2 * 8 * Rr and rep.tile_k[1] == 8 * Rr
    w = g.nodes[0].consts["weight"].astype(np.float64)            # [cout, C, k, k]
    bn = g.nodes[1]
    scale = bn.consts["gamma"].astype(np.float64) / np.sqrt(
        bn.consts["moving_var"].astype(np.float64) + bn.attrs.get("epsilon", 1e-5))
    packed = np.frombuffer(reg.plan_constants(1, 0), dtype=np.uint16).reshape(-1, rep.gemm_k[1])
    expect = np.zeros((cout, k2, Rr, 2, 4), dtype=np.float64)     # [k][b][r][dx][c]
    for b in range(k2):
        for r in range(k):
            for dx in range(2):
                if 2 * b + dx < k:
                    expect[:, b, r, dx, :C] = w[:, :, r, 2 * b + dx]
    expect *= scale[:, None, None, None, None]
    want = I.bf16_bits(expect.reshape(cout, -1).astype(np.float32))
    assert np.array_equal(packed[:cout], want)
