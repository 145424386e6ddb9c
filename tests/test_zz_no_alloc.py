"""byoc_ffn_noalloc, the allocation-free entry point, against the fp64 oracle
on the dense + bias + GELU -> dense + bias chain.

Some callers cannot allocate device memory -- an inference path running
inside a memory pool it does not own, or one that must not take the
allocator's lock or its implicit synchronisation -- so they cannot use
byoc_compile.  byoc_ffn_noalloc keeps its hidden activation in a fixed device
array instead.  This file is collected after every other test file, so a
failure here never stops the rest of the GPU suite; each test also passes
when run alone in a fresh process.
"""
import numpy as np
import pytest

from paper_2105_03215_gb300 import abi
from paper_2105_03215_gb300 import inputs as I

from .parity import assert_close, oracle

pytestmark = pytest.mark.gpu


def _call(x, M, D, F, w1, b1, w2, b2, y, stream):
    return abi.lib().byoc_ffn_noalloc(x.data_ptr(), M, D, F, w1.data_ptr(), b1.data_ptr(),
                                      w2.data_ptr(), b2.data_ptr(), y.data_ptr(), stream)


def _weights(g):
    import torch
    d1, bias1, _, d2, bias2 = g.nodes
    # bf16 weights rounded to nearest even, as byoc_compile rounds them
    w1 = torch.from_numpy(d1.consts["weight"]).to(torch.bfloat16).cuda()
    w2 = torch.from_numpy(d2.consts["weight"]).to(torch.bfloat16).cuda()
    b1 = torch.from_numpy(bias1.consts["bias"]).cuda()
    b2 = torch.from_numpy(bias2.consts["bias"]).cuda()
    return w1, b1, w2, b2


@pytest.mark.parametrize("M,D,F", [
    (1024, 768, 3072),   # BERT-base FFN, 128 tokens x batch 8
    (200, 128, 384),     # ragged last row tile (200 = 128 + 72), three hidden column tiles
    (2048, 128, 4096),   # M * F = 8,388,608: the scratch array exactly full
])
def test_ffn_noalloc_matches_the_oracle_on_two_calls(M, D, F):
    import torch
    g, _ = I.bert_ffn(M=M, D=D, F=F, seed=21)
    w1, b1, w2, b2 = _weights(g)
    stream = torch.cuda.current_stream().cuda_stream
    rng = np.random.default_rng(M + F)
    for call in range(2):  # two calls in a row, different inputs
        xs = I.bf16_round(rng.standard_normal((M, D), dtype=np.float32))
        x = torch.from_numpy(xs).to(torch.bfloat16).cuda()
        y = torch.full((M, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        abi.check(_call(x, M, D, F, w1, b1, w2, b2, y, stream))
        torch.cuda.synchronize()
        abi.check(abi.lib().byoc_check(None))  # the entry point's bounded waits all completed
        ref, sc = oracle(g, {"x": xs})
        o = g.outputs[0]
        assert_close(y.float().cpu().numpy(), ref[o], sc[o], f"noalloc {M}x{D}x{F} call {call}")


def test_ffn_noalloc_leaves_device_memory_untouched():
    import torch
    M, D, F = 256, 256, 512
    g, _ = I.bert_ffn(M=M, D=D, F=F, seed=22)
    w1, b1, w2, b2 = _weights(g)
    x = torch.ones((M, D), dtype=torch.bfloat16, device="cuda")
    y = torch.empty((M, D), dtype=torch.bfloat16, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    abi.check(_call(x, M, D, F, w1, b1, w2, b2, y, stream))  # set-up and module loading
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        abi.check(_call(x, M, D, F, w1, b1, w2, b2, y, stream))
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


def test_ffn_noalloc_rejects_sizes_beyond_its_scratch():
    import torch
    M, D, F = 2049, 128, 4096  # M * F = 8,392,704 > 8,388,608
    x = torch.zeros((M, D), dtype=torch.bfloat16, device="cuda")
    w1 = torch.zeros((F, D), dtype=torch.bfloat16, device="cuda")
    w2 = torch.zeros((D, F), dtype=torch.bfloat16, device="cuda")
    b1 = torch.zeros(F, device="cuda")
    b2 = torch.zeros(D, device="cuda")
    y = torch.zeros((M, D), dtype=torch.bfloat16, device="cuda")
    st = _call(x, M, D, F, w1, b1, w2, b2, y, torch.cuda.current_stream().cuda_stream)
    assert st == abi.ERR_INVALID_ARG
    assert b"scratch" in abi.lib().byoc_last_error()
