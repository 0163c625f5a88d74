"""phsa_sparse_attn_bwd_noalloc: the backward pass for callers that cannot
allocate device memory where they run it (engines that own all of HBM, plugin
execute steps, hot loops that cannot afford cudaMalloc's synchronisation).

Its results must match phsa_sparse_attn_bwd (which takes a caller workspace)
within the parity tolerance, on two calls in a row (the library's scratch array
keeps the previous call's contents, so the second call checks that nothing
stale leaks into it). This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2601_02819_gb300 import phsa
from parity import assert_close

pytestmark = pytest.mark.gpu

D = 128


def _case(seed, B, Hq, Hkv, L, topk):
    g = torch.Generator(device="cuda").manual_seed(seed)
    r = lambda *s: torch.randn(s, generator=g, device="cuda").to(torch.bfloat16)
    Q, K, V, dO = r(B, Hq, L, D), r(B, Hkv, L, D), r(B, Hkv, L, D), r(B, Hq, L, D)
    mask = (torch.rand((B, L), generator=g, device="cuda") < 0.06).to(torch.uint8)
    O, lse, idx, cnt, _ = phsa.phsa_forward(Q, K, V, mask, 0.5, topk)
    return Q, K, V, O, dO, lse, idx, cnt


def _noalloc_call(Q, K, V, O, dO, lse, idx, cnt, dQ, dK, dV):
    """Direct C-ABI call (ctypes), outputs preallocated by the test."""
    lib = phsa.load()
    B, Hq, L, _ = Q.shape
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    return lib.phsa_sparse_attn_bwd_noalloc(
        p(Q), p(K), p(V), p(O), p(dO), p(lse), p(idx), p(cnt),
        phsa.make_shape(B, L, Hq, K.shape[1]), int(idx.shape[-1]), ctypes.c_float(D ** -0.5),
        p(dQ), p(dK), p(dV), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("seed,B,Hq,Hkv,L,topk", [
    (0, 1, 2, 1, 64 * 40 + 13, 6),   # ragged tail
    (1, 2, 4, 2, 64 * 96, 8),        # lists longer than one chunk
])
def test_noalloc_matches_the_workspace_entry_point_twice(seed, B, Hq, Hkv, L, topk):
    Q, K, V, O, dO, lse, idx, cnt = _case(seed, B, Hq, Hkv, L, topk)
    ref = phsa.phsa_sparse_attn_bwd(Q, K, V, O, dO, lse, idx, cnt)
    torch.cuda.synchronize()
    outs = [torch.empty_like(Q), torch.empty_like(K), torch.empty_like(V)]
    for call in range(2):
        for t in outs:
            t.fill_(float("nan"))
        rc = _noalloc_call(Q, K, V, O, dO, lse, idx, cnt, *outs)
        assert rc == 0, phsa.phsa_status_string(rc)
        torch.cuda.synchronize()
        assert phsa.phsa_get_device_status() == 0
        for name, got, want in zip(("dQ", "dK", "dV"), outs, ref):
            assert_close(f"{name} (call {call + 1})", got.double().cpu().numpy(),
                         want.double().cpu().numpy())


def test_noalloc_allocates_no_device_memory():
    Q, K, V, O, dO, lse, idx, cnt = _case(2, 1, 2, 1, 64 * 24, 5)
    outs = [torch.empty_like(Q), torch.empty_like(K), torch.empty_like(V)]
    assert _noalloc_call(Q, K, V, O, dO, lse, idx, cnt, *outs) == 0  # first call: set-up
    torch.cuda.synchronize()
    free_before, _ = torch.cuda.mem_get_info()
    torch_before = torch.cuda.memory_allocated()
    assert _noalloc_call(Q, K, V, O, dO, lse, idx, cnt, *outs) == 0
    torch.cuda.synchronize()
    free_after, _ = torch.cuda.mem_get_info()
    assert free_after == free_before
    assert torch.cuda.memory_allocated() == torch_before


def test_noalloc_rejects_shapes_beyond_its_scratch():
    shape = phsa.make_shape(1, 32768, 16, 8)
    assert phsa.phsa_sparse_attn_bwd_workspace(1, 32768, 16, 8, 14) > (64 << 20)
    lib = phsa.load()
    one = torch.zeros(16, dtype=torch.bfloat16, device="cuda")
    p = ctypes.c_void_p(one.data_ptr())
    rc = lib.phsa_sparse_attn_bwd_noalloc(p, p, p, p, p, p, p, p, shape, 14,
                                          ctypes.c_float(D ** -0.5), p, p, p, None)
    assert rc == -6, phsa.phsa_status_string(rc)  # PHSA_ERR_WORKSPACE, nothing launched
