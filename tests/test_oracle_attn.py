"""Pins for the oracle's sparse attention, forward and backward (Eq. 1-2, 10-11).

The independent references are PyTorch's own fp64 CPU routines
(``scaled_dot_product_attention`` with an explicit boolean mask, and autograd
through it), plus closed-form invariants. The oracle itself is plain C.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300.inputs import f32_to_bf16_bits

D = 128


def bf(x):
    return f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def rand_qkv(rng, B, Hq, Hkv, L):
    Q = bf(rng.standard_normal((B, Hq, L, D)))
    K = bf(rng.standard_normal((B, Hkv, L, D)))
    V = bf(rng.standard_normal((B, Hkv, L, D)))
    return Q, K, V


def random_selection(rng, B, Hkv, L, m, topk):
    """A valid block set per (b, g, qb): first and own block plus random earlier ones."""
    NQB = -(-L // m)
    idx = np.full((B, Hkv, NQB, topk), -1, np.int32)
    cnt = np.zeros((B, Hkv, NQB), np.int32)
    for b in range(B):
        for g in range(Hkv):
            for qb in range(NQB):
                s = {0, qb}
                extra = [t for t in range(1, qb)]
                rng.shuffle(extra)
                s |= set(extra[:max(0, topk - len(s))])
                s = sorted(s)
                idx[b, g, qb, :len(s)] = s
                cnt[b, g, qb] = len(s)
    return idx, cnt


def token_mask(idx, cnt, L, m):
    """Boolean [B, Hkv, L, L]: key j visible to query i (selected block and j <= i)."""
    B, Hkv, NQB, _ = idx.shape
    M = np.zeros((B, Hkv, L, L), bool)
    for b in range(B):
        for g in range(Hkv):
            for i in range(L):
                qb = i // m
                for t in idx[b, g, qb, :cnt[b, g, qb]]:
                    M[b, g, i, t * m:min((t + 1) * m, i + 1)] = True
    return M


def torch_ref(Q, K, V, vis, scale, dO=None):
    """fp64 PyTorch SDPA with an explicit mask; returns O, lse and optionally grads."""
    G = Q.shape[1] // K.shape[1]
    q = torch.from_numpy(oracle.bf16_to_f64(Q)).requires_grad_(dO is not None)
    k = torch.from_numpy(oracle.bf16_to_f64(K)).requires_grad_(dO is not None)
    v = torch.from_numpy(oracle.bf16_to_f64(V)).requires_grad_(dO is not None)
    ke = k.repeat_interleave(G, dim=1)
    ve = v.repeat_interleave(G, dim=1)
    mask = torch.from_numpy(np.repeat(vis, G, axis=1))
    o = torch.nn.functional.scaled_dot_product_attention(q, ke, ve, attn_mask=mask, scale=scale)
    s = (q @ ke.transpose(-1, -2)) * scale
    lse = torch.logsumexp(s.masked_fill(~mask, float("-inf")), dim=-1)
    if dO is None:
        return o.detach().numpy(), lse.detach().numpy()
    o.backward(torch.from_numpy(oracle.bf16_to_f64(dO)))
    return (o.detach().numpy(), lse.detach().numpy(), q.grad.numpy(), k.grad.numpy(),
            v.grad.numpy())


@pytest.mark.parametrize("L,m", [(256, 64), (300, 64), (300, 16), (160, 32)])
def test_full_budget_equals_dense_causal(L, m):
    rng = np.random.default_rng(10)
    Q, K, V = rand_qkv(rng, 1, 4, 2, L)
    NQB = -(-L // m)
    idx = np.tile(np.arange(NQB, dtype=np.int32), (1, 2, NQB, 1))
    cnt = np.tile(np.arange(1, NQB + 1, dtype=np.int32), (1, 2, 1))
    for qb in range(NQB):
        idx[..., qb, qb + 1:] = -1
    O, lse = oracle.sparse_attn_fwd(Q, K, V, idx, cnt, m, D ** -0.5)
    Od, lsed = oracle.dense_causal(Q, K, V, D ** -0.5)
    np.testing.assert_allclose(O, Od, rtol=0, atol=1e-13)
    np.testing.assert_allclose(lse, lsed, rtol=0, atol=1e-13)


def test_dense_causal_matches_torch_fp64():
    rng = np.random.default_rng(11)
    L = 200
    Q, K, V = rand_qkv(rng, 2, 4, 2, L)
    O, lse = oracle.dense_causal(Q, K, V, D ** -0.5)
    vis = np.broadcast_to(np.tril(np.ones((L, L), bool)), (2, 2, L, L))
    Ot, lset = torch_ref(Q, K, V, vis, D ** -0.5)
    np.testing.assert_allclose(O, Ot, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lset, rtol=0, atol=1e-12)


@pytest.mark.parametrize("L,topk,m", [(64 * 9, 4, 64), (64 * 6 + 23, 3, 64), (16 * 13 + 5, 5, 16),
                                      (32 * 7 + 9, 3, 32)])
def test_sparse_matches_torch_masked_fp64(L, topk, m):
    rng = np.random.default_rng(12)
    Q, K, V = rand_qkv(rng, 2, 4, 2, L)
    idx, cnt = random_selection(rng, 2, 2, L, m, topk)
    O, lse = oracle.sparse_attn_fwd(Q, K, V, idx, cnt, m, D ** -0.5)
    Ot, lset = torch_ref(Q, K, V, token_mask(idx, cnt, L, m), D ** -0.5)
    np.testing.assert_allclose(O, Ot, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lset, rtol=0, atol=1e-12)
    rows = np.array([[0, 0, 5], [1, 3, L - 1], [1, 2, 64], [0, 1, 130]], np.int32)
    Or, lser = oracle.sparse_attn_rows(Q, K, V, idx, cnt, m, D ** -0.5, rows)
    for n, (b, h, i) in enumerate(rows):
        np.testing.assert_array_equal(Or[n], O[b, h, i])
        assert lser[n] == lse[b, h, i]


def test_constant_values_give_constant_output():
    rng = np.random.default_rng(13)
    L, m = 64 * 5, 64
    Q, K, _ = rand_qkv(rng, 1, 2, 1, L)
    V = bf(np.full((1, 1, L, D), 1.5))
    idx, cnt = random_selection(rng, 1, 1, L, m, 3)
    O, _ = oracle.sparse_attn_fwd(Q, K, V, idx, cnt, m, D ** -0.5)
    np.testing.assert_allclose(O, 1.5, rtol=0, atol=1e-13)


def test_block_order_does_not_matter():
    rng = np.random.default_rng(14)
    L, m = 64 * 8, 64
    Q, K, V = rand_qkv(rng, 1, 2, 1, L)
    idx, cnt = random_selection(rng, 1, 1, L, m, 4)
    O, lse = oracle.sparse_attn_fwd(Q, K, V, idx, cnt, m, D ** -0.5)
    idx2 = idx.copy()
    for qb in range(idx.shape[2]):
        n = cnt[0, 0, qb]
        idx2[0, 0, qb, :n] = idx[0, 0, qb, :n][::-1]
    O2, lse2 = oracle.sparse_attn_fwd(Q, K, V, idx2, cnt, m, D ** -0.5)
    np.testing.assert_allclose(O, O2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, lse2, rtol=0, atol=1e-12)


@pytest.mark.parametrize("L,topk,m", [(64 * 5, 3, 64), (64 * 4 + 9, 2, 64), (16 * 13 + 5, 5, 16),
                                      (16 * 9, 9, 16), (32 * 7 + 3, 3, 32)])
def test_backward_matches_torch_autograd_fp64(L, topk, m):
    rng = np.random.default_rng(15 + m)
    Q, K, V = rand_qkv(rng, 1, 4, 2, L)
    dO = bf(rng.standard_normal(Q.shape))
    idx, cnt = random_selection(rng, 1, 2, L, m, topk)
    dQ, dK, dV = oracle.sparse_attn_bwd(Q, K, V, dO, idx, cnt, m, D ** -0.5)
    _, _, tq, tk, tv = torch_ref(Q, K, V, token_mask(idx, cnt, L, m), D ** -0.5, dO=dO)
    np.testing.assert_allclose(dQ, tq, rtol=0, atol=1e-11)
    np.testing.assert_allclose(dK, tk, rtol=0, atol=1e-11)
    np.testing.assert_allclose(dV, tv, rtol=0, atol=1e-11)


@pytest.mark.parametrize("L,m", [(64 * 6 + 5, 64), (16 * 20 + 7, 16)])
def test_backward_invariants(L, m):
    # Softmax rows sum to one, so sum_j dV_j = sum_i dO_i (per KV head, over its query
    # heads), and the dS of each row sums to zero, so sum_j dK_j = 0.
    rng = np.random.default_rng(16 + m)
    Q, K, V = rand_qkv(rng, 2, 4, 2, L)
    dO = bf(rng.standard_normal(Q.shape))
    idx, cnt = random_selection(rng, 2, 2, L, m, 3)
    dQ, dK, dV = oracle.sparse_attn_bwd(Q, K, V, dO, idx, cnt, m, D ** -0.5)
    go = oracle.bf16_to_f64(dO).reshape(2, 2, 2, L, D).sum(axis=(2, 3))
    np.testing.assert_allclose(dV.sum(axis=2), go, rtol=0, atol=1e-9)
    np.testing.assert_allclose(dK.sum(axis=2), 0.0, rtol=0, atol=1e-9)


def test_sampled_oracle_entry_points_agree_with_full_ones():
    # The sampled forms used at full size must give exactly the full computation's values.
    rng = np.random.default_rng(17)
    L, m = 64 * 7 + 11, 64
    Q, K, V = rand_qkv(rng, 2, 4, 2, L)
    dO = bf(rng.standard_normal(Q.shape))
    Kr = oracle.block_repr(K, (rng.random((2, L)) < 0.1).astype(np.uint8), m, 0.5)
    idx, cnt, agg = oracle.select_blocks(Q, Kr, L, m, 4, 1, 1, D ** -0.5, want_agg=True)
    units = np.array([0, 5, 7, 8 + 6, 3 * 8 + 7])
    i2, c2, a2 = oracle.select_units(Q, Kr, L, m, 4, 1, 1, D ** -0.5, units)
    fi = idx.reshape(-1, 4)[units]
    assert np.array_equal(i2, fi) and np.array_equal(c2, cnt.reshape(-1)[units])
    np.testing.assert_array_equal(a2, agg.reshape(-1, agg.shape[-1])[units])
    dQ, dK, dV = oracle.sparse_attn_bwd(Q, K, V, dO, idx, cnt, m, D ** -0.5)
    rows = np.array([[0, 0, 3], [1, 3, L - 1], [1, 2, 200]], np.int32)
    dq = oracle.sparse_attn_bwd_dq_rows(Q, K, V, dO, idx, cnt, m, D ** -0.5, rows)
    for n, (b, h, i) in enumerate(rows):
        np.testing.assert_allclose(dq[n], dQ[b, h, i], rtol=0, atol=1e-12)
    blocks = np.array([[0, 0, 0], [1, 1, 3], [1, 0, 7]], np.int32)
    dk, dv = oracle.sparse_attn_bwd_kv_blocks(Q, K, V, dO, idx, cnt, m, D ** -0.5, blocks)
    for n, (b, g, t) in enumerate(blocks):
        hi = min(L, (t + 1) * m) - t * m
        np.testing.assert_allclose(dk[n, :hi], dK[b, g, t * m:t * m + hi], rtol=0, atol=1e-12)
        np.testing.assert_allclose(dv[n, :hi], dV[b, g, t * m:t * m + hi], rtol=0, atol=1e-12)
        assert np.all(dk[n, hi:] == 0) and np.all(dv[n, hi:] == 0)
