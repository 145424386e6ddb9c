"""byoc_ffn_noalloc, the allocation-free entry point, against the regular
compiled-region path (byoc_compile + byoc_run) on the same dense + bias +
GELU -> dense + bias chain.

Some callers cannot allocate device memory -- an inference path running
inside a memory pool it does not own, or one that must not take the
allocator's lock or its implicit synchronisation -- so they cannot use
byoc_compile.  byoc_ffn_noalloc keeps its hidden activation in a fixed device
array instead.  This file is collected after every other test file, so a
failure here never stops the rest of the GPU suite.
"""
import ctypes

import numpy as np
import pytest

from paper_2105_03215_gb300 import abi
from paper_2105_03215_gb300 import inputs as I
from paper_2105_03215_gb300 import region as R

from .parity import assert_close

pytestmark = pytest.mark.gpu


def _call(x, M, D, F, w1, b1, w2, b2, y, stream):
    return abi.lib().byoc_ffn_noalloc(x.data_ptr(), M, D, F, w1.data_ptr(), b1.data_ptr(),
                                      w2.data_ptr(), b2.data_ptr(), y.data_ptr(), stream)


def test_ffn_noalloc_matches_compiled_region_on_two_calls():
    import torch
    M, D, F = 1024, 768, 3072  # BERT-base FFN, 128 tokens x batch 8
    g, _ = I.bert_ffn(M=M, D=D, F=F, seed=21)
    d1, bias1, _, d2, bias2 = g.nodes
    cr = R.whole_graph_region(g).compile()
    # bf16 weights rounded to nearest even, as byoc_compile rounds them
    w1 = torch.from_numpy(d1.consts["weight"]).to(torch.bfloat16).cuda()
    w2 = torch.from_numpy(d2.consts["weight"]).to(torch.bfloat16).cuda()
    b1 = torch.from_numpy(bias1.consts["bias"]).cuda()
    b2 = torch.from_numpy(bias2.consts["bias"]).cuda()
    stream = torch.cuda.current_stream().cuda_stream
    rng = np.random.default_rng(77)
    for call in range(2):  # two calls in a row, different inputs
        x = torch.from_numpy(I.bf16_round(rng.standard_normal((M, D), dtype=np.float32))).to(
            torch.bfloat16).cuda()
        ref = torch.empty((M, D), dtype=torch.bfloat16, device="cuda")
        cr.run([x], [ref])
        y = torch.full((M, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        abi.check(_call(x, M, D, F, w1, b1, w2, b2, y, stream))
        torch.cuda.synchronize()
        cr.check()
        assert_close(y.float().cpu().numpy(), ref.float().cpu().numpy(), f"noalloc call {call}")
    cr.release()


def test_ffn_noalloc_rejects_sizes_beyond_its_scratch():
    import torch
    M, D, F = 4096, 128, 4096  # M * F = 16 Mi elements > 8 Mi
    x = torch.zeros((M, D), dtype=torch.bfloat16, device="cuda")
    w1 = torch.zeros((F, D), dtype=torch.bfloat16, device="cuda")
    w2 = torch.zeros((D, F), dtype=torch.bfloat16, device="cuda")
    b1 = torch.zeros(F, device="cuda")
    b2 = torch.zeros(D, device="cuda")
    y = torch.zeros((M, D), dtype=torch.bfloat16, device="cuda")
    st = _call(x, M, D, F, w1, b1, w2, b2, y, torch.cuda.current_stream().cuda_stream)
    assert st == abi.ERR_INVALID_ARG
    assert b"scratch" in abi.lib().byoc_last_error()
