"""Stage (c) on the GPU vs the oracle: sparse attention forward and backward.

The GPU kernels are driven by the oracle's own block selection, so attention
parity is checked independently of selection. Tolerances: max-abs <= 2e-2 and
relative L2 <= 1e-2 for O, dQ, dK, dV; LSE within 1e-3.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300 import inputs
from paper_2601_02819_gb300 import phsa
from parity import LSE_ABS, assert_close, bf16_to_f64, to_dev_bf16

pytestmark = pytest.mark.gpu

D = 128
SCALE = D ** -0.5


def rand_case(seed, B, Hq, Hkv, L, topk, n_init=1, n_local=1, grad=False):
    rng = np.random.default_rng(seed)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    Q, K, V = f(B, Hq, L, D), f(B, Hkv, L, D), f(B, Hkv, L, D)
    mask = (rng.random((B, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, 64, 0.5)
    idx, cnt = oracle.select_blocks(Q, Kr, L, 64, topk, n_init, n_local, SCALE)
    dO = f(B, Hq, L, D) if grad else None
    return Q, K, V, dO, idx, cnt


def gpu_fwd(Q, K, V, idx, cnt):
    O, lse = phsa.phsa_sparse_attn_fwd(to_dev_bf16(Q), to_dev_bf16(K), to_dev_bf16(V),
                                       torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda())
    torch.cuda.synchronize()
    return O, lse


CASES = [
    (1, 2, 1, 2048, 8),          # the tiny workload's shape
    (2, 4, 2, 64 * 23 + 41, 5),  # ragged tail
    (1, 3, 3, 64 * 17, 6),       # G = 1
    (1, 2, 1, 64 * 5 + 1, 3),    # one-token tail block
    (1, 2, 1, 37, 2),            # shorter than one block
]


@pytest.mark.parametrize("B,Hq,Hkv,L,topk", CASES)
def test_forward_matches_oracle(B, Hq, Hkv, L, topk):
    Q, K, V, _, idx, cnt = rand_case(L, B, Hq, Hkv, L, topk)
    O, lse = gpu_fwd(Q, K, V, idx, cnt)
    Or, lser = oracle.sparse_attn_fwd(Q, K, V, idx, cnt, 64, SCALE)
    assert_close("O", bf16_to_f64(O), Or)
    assert np.abs(lse.cpu().numpy() - lser).max() <= LSE_ABS
    assert phsa.phsa_get_device_status() == 0


def test_full_budget_is_dense_causal_attention():
    B, Hq, Hkv, L = 1, 4, 2, 64 * 12 + 20
    NQB = -(-L // 64)
    rng = np.random.default_rng(3)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    Q, K, V = f(B, Hq, L, D), f(B, Hkv, L, D), f(B, Hkv, L, D)
    idx = np.full((B, Hkv, NQB, NQB), -1, np.int32)
    cnt = np.zeros((B, Hkv, NQB), np.int32)
    for qb in range(NQB):
        idx[:, :, qb, :qb + 1] = np.arange(qb + 1)
        cnt[:, :, qb] = qb + 1
    O, lse = gpu_fwd(Q, K, V, idx, cnt)
    Od, lsed = oracle.dense_causal(Q, K, V, SCALE)
    assert_close("O", bf16_to_f64(O), Od)
    assert np.abs(lse.cpu().numpy() - lsed).max() <= LSE_ABS


def test_constant_values_give_constant_output():
    Q, K, V, _, idx, cnt = rand_case(4, 1, 2, 1, 64 * 10, 4)
    V = np.full_like(V, inputs.f32_to_bf16_bits(np.array([0.75], np.float32))[0])
    O, _ = gpu_fwd(Q, K, V, idx, cnt)
    assert np.all(bf16_to_f64(O) == 0.75)


@pytest.mark.parametrize("B,Hq,Hkv,L,topk", CASES)
def test_backward_matches_oracle(B, Hq, Hkv, L, topk):
    Q, K, V, dO, idx, cnt = rand_case(L + 7, B, Hq, Hkv, L, topk, grad=True)
    Qd, Kd, Vd, dOd = (to_dev_bf16(a) for a in (Q, K, V, dO))
    it, ct = torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda()
    O, lse = phsa.phsa_sparse_attn_fwd(Qd, Kd, Vd, it, ct)
    dQ, dK, dV = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct)
    torch.cuda.synchronize()
    rQ, rK, rV = oracle.sparse_attn_bwd(Q, K, V, dO, idx, cnt, 64, SCALE)
    assert_close("dQ", bf16_to_f64(dQ), rQ)
    assert_close("dK", bf16_to_f64(dK), rK)
    assert_close("dV", bf16_to_f64(dV), rV)
    assert phsa.phsa_get_device_status() == 0


def test_backward_long_lists_use_chunked_partials_and_are_deterministic():
    # L = 64*100 with n_init = 4: blocks 0-3 are selected by ~100 query blocks each,
    # more than one dK/dV chunk, so the partial-sum path runs.
    Q, K, V, dO, idx, cnt = rand_case(11, 1, 2, 1, 64 * 100, 8, n_init=4, grad=True)
    Qd, Kd, Vd, dOd = (to_dev_bf16(a) for a in (Q, K, V, dO))
    it, ct = torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda()
    O, lse = phsa.phsa_sparse_attn_fwd(Qd, Kd, Vd, it, ct)
    g1 = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct)
    g2 = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct)
    torch.cuda.synchronize()
    for a, b in zip(g1, g2):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    rQ, rK, rV = oracle.sparse_attn_bwd(Q, K, V, dO, idx, cnt, 64, SCALE)
    assert_close("dQ", bf16_to_f64(g1[0]), rQ)
    assert_close("dK", bf16_to_f64(g1[1]), rK)
    assert_close("dV", bf16_to_f64(g1[2]), rV)


def test_backward_large_budget_for_pairs():
    # A list capacity of 220 blocks (the selection padded with -1) no longer fits
    # beside the tcgen05 dQ kernel's tiles, so pairs of heads take the
    # register-MMA backward kernels; the forward keeps its tcgen05 kernel.
    Q, K, V, dO, idx, cnt = rand_case(21, 1, 4, 2, 64 * 30 + 17, 8, grad=True)
    wide = np.full(idx.shape[:-1] + (220,), -1, np.int32)
    wide[..., :idx.shape[-1]] = idx
    Qd, Kd, Vd, dOd = (to_dev_bf16(a) for a in (Q, K, V, dO))
    it, ct = torch.from_numpy(wide).cuda(), torch.from_numpy(cnt).cuda()
    O, lse = phsa.phsa_sparse_attn_fwd(Qd, Kd, Vd, it, ct)
    dQ, dK, dV = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    Or, _ = oracle.sparse_attn_fwd(Q, K, V, idx, cnt, 64, SCALE)
    assert_close("O", bf16_to_f64(O), Or)
    rQ, rK, rV = oracle.sparse_attn_bwd(Q, K, V, dO, idx, cnt, 64, SCALE)
    assert_close("dQ", bf16_to_f64(dQ), rQ)
    assert_close("dK", bf16_to_f64(dK), rK)
    assert_close("dV", bf16_to_f64(dV), rV)


def test_invalid_block_indices_are_skipped_and_reported():
    Q, K, V, _, idx, cnt = rand_case(12, 1, 2, 1, 64 * 6, 3)
    bad = idx.copy()
    bad[0, 0, 2, 1] = 5        # a future block: must be skipped, not read
    bad[0, 0, 3, 1] = 100000   # far out of range
    phsa.phsa_get_device_status()  # clear
    O, _ = gpu_fwd(Q, K, V, bad, cnt)
    assert phsa.phsa_get_device_status() == -5
    assert phsa.phsa_get_device_status() == 0  # cleared by the read
    Or, _ = oracle.sparse_attn_fwd(Q, K, V, idx, cnt, 64, SCALE)
    # untouched query blocks still match
    assert_close("O", bf16_to_f64(O)[:, :, 256:], Or[:, :, 256:])


def test_argument_errors_raise():
    Q = torch.zeros((1, 2, 128, 128), dtype=torch.bfloat16, device="cuda")
    K = torch.zeros((1, 1, 128, 128), dtype=torch.bfloat16, device="cuda")
    idx = torch.zeros((1, 1, 2, 4), dtype=torch.int32, device="cuda")
    cnt = torch.zeros((1, 1, 2), dtype=torch.int32, device="cuda")
    with pytest.raises(phsa.PhsaError):
        phsa.phsa_sparse_attn_fwd(Q, K, K, idx, cnt, sm_scale=-1.0)
    with pytest.raises(phsa.PhsaError):
        phsa.phsa_select_blocks(Q, K[:, :, :2], 1, topk=1, n_init=1, n_local=1)


@pytest.mark.parametrize("m,B,Hq,Hkv,L,topk,n_init", [
    (64, 1, 2, 1, 64 * 100 + 13, 8, 4),   # GQA pair; multi-chunk lists
    (64, 2, 3, 3, 64 * 21 + 5, 6, 1),     # one query head per KV head
    (16, 1, 2, 1, 16 * 300 + 5, 20, 2),   # m = 16: mask rows per span
    (32, 1, 4, 2, 32 * 25 + 17, 4, 1),    # m = 32
])
def test_backward_index_transpose_forms_agree(m, B, Hq, Hkv, L, topk, n_init):
    # The one-launch transpose (bitmap in shared memory) and the two-launch
    # form (bitmap in global memory: at m < 64, and when a (b, g)'s bitmap
    # exceeds 160 KB) build the same KV-block lists, so the gradients are
    # identical. The hook forces each form at every block size.
    rng = np.random.default_rng(L + 17 * m)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    Q, K, V, dO = f(B, Hq, L, D), f(B, Hkv, L, D), f(B, Hkv, L, D), f(B, Hq, L, D)
    mask = (rng.random((B, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, m, 0.5)
    idx, cnt = oracle.select_blocks(Q, Kr, L, m, topk, n_init, 1, SCALE)
    Qd, Kd, Vd, dOd = (to_dev_bf16(a) for a in (Q, K, V, dO))
    it, ct = torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda()
    O, lse = phsa.phsa_sparse_attn_fwd(Qd, Kd, Vd, it, ct, block_size=m)
    g_default = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct, block_size=m)
    prev = phsa.phsa_test_set_idx_smem_limit(160 * 1024)
    try:
        g_smem = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct, block_size=m)
        phsa.phsa_test_set_idx_smem_limit(1)
        g_glob = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct, block_size=m)
        torch.cuda.synchronize()
    finally:
        phsa.phsa_test_set_idx_smem_limit(prev)
    assert phsa.phsa_get_device_status() == 0
    for a, b, c in zip(g_smem, g_glob, g_default):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
        assert torch.equal(a.view(torch.int16), c.view(torch.int16))
    rQ, rK, rV = oracle.sparse_attn_bwd(Q, K, V, dO, idx, cnt, m, SCALE)
    assert_close("dQ", bf16_to_f64(g_smem[0]), rQ)
    assert_close("dK", bf16_to_f64(g_smem[1]), rK)
    assert_close("dV", bf16_to_f64(g_smem[2]), rV)
