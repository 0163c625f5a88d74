"""Block sizes 16 and 32 on the GPU vs the oracle: representative keys (Eq. 6-8),
selection (Eq. 8, Algorithm 1 step 3) and sparse attention forward (Eq. 10-11).

The paper's experiments use blocks of 16 tokens. Each stage gets the oracle's
inputs for it (the oracle's representative keys for the selection, the
oracle's block lists for the attention), so every check isolates one kernel;
the end-to-end case runs the three calls in a row.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300 import inputs, phsa
from parity import (LSE_ABS, assert_close, bf16_bits, bf16_to_f64, compare_selection,
                    to_dev_bf16, ulp_distance)

pytestmark = pytest.mark.gpu

D = 128
SCALE = D ** -0.5


def rand(rng, *s):
    return inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))


@pytest.mark.parametrize("m,L,lam", [(16, 16 * 50 + 7, 0.5), (16, 16 * 64, 0.0), (32, 32 * 33 + 31, 1.0),
                                     (32, 32 * 20, 0.3)])
def test_block_repr_matches_oracle(m, L, lam):
    rng = np.random.default_rng(m + L)
    K = rand(rng, 2, 3, L, D)
    mask = (rng.random((2, L)) < 0.08).astype(np.uint8)
    mask[0, :m] = 1      # an all-punctuation block
    mask[1, m:2 * m] = 0  # a block without punctuation
    got = phsa.phsa_build_block_repr(to_dev_bf16(K), torch.from_numpy(mask).cuda(), lam,
                                     block_size=m)
    torch.cuda.synchronize()
    ref = oracle.block_repr(K, mask, m, lam)
    assert got.shape == ref.shape == (2, 3, L // m, D)
    assert ulp_distance(bf16_bits(got), ref).max() <= 1


def gpu_select(Q, Kr, Hkv, topk, n_init, n_local, m, aggregation="softmax_sum"):
    idx, cnt = phsa.phsa_select_blocks(to_dev_bf16(Q), to_dev_bf16(Kr), Hkv, topk, n_init,
                                       n_local, SCALE, aggregation=aggregation, block_size=m)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), cnt.cpu().numpy()


@pytest.mark.parametrize("m,B,Hq,Hkv,L,topk,n_init,n_local", [
    (16, 1, 2, 1, 16 * 97 + 5, 8, 1, 1),      # G = 2, ragged tail
    (16, 2, 2, 2, 16 * 80, 6, 1, 2),          # G = 1
    (16, 1, 4, 2, 16 * 256, 56, 8, 32),       # the paper's 32k forced sets (8 + 32 blocks of 16)
    (16, 1, 2, 1, 16 * 40, 41, 1, 1),         # budget covers everything: dense rows
    (32, 1, 4, 2, 32 * 70 + 19, 10, 1, 1),    # m = 32, G = 2
    (32, 1, 3, 3, 32 * 50, 7, 2, 2),          # m = 32, G = 1
])
@pytest.mark.parametrize("aggregation", ["softmax_sum", "max_logit"])
def test_selection_matches_oracle(m, B, Hq, Hkv, L, topk, n_init, n_local, aggregation):
    rng = np.random.default_rng(L + topk)
    Q, K = rand(rng, B, Hq, L, D), rand(rng, B, Hkv, L, D)
    mask = (rng.random((B, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, m, 0.5)
    gi, gc = gpu_select(Q, Kr, Hkv, topk, n_init, n_local, m, aggregation)
    oi, oc, oa = oracle.select_blocks(Q, Kr, L, m, topk, n_init, n_local, SCALE, want_agg=True,
                                      aggregation=aggregation)
    assert gi.shape == oi.shape == (B, Hkv, -(-L // m), topk)
    bad, excl, differ, msgs = compare_selection(gi, gc, oi, oc, oa)
    assert bad == 0, msgs[:5]
    assert differ <= max(2, 0.01 * oc.size), (differ, oc.size)


def test_selection_exact_ties_go_to_the_lower_block_at_m16():
    rng = np.random.default_rng(9)
    L, T = 16 * 24, 24
    Q = rand(rng, 1, 2, L, D)
    row = rand(rng, D)
    Kr = np.broadcast_to(row, (1, 1, T, D)).copy()
    gi, gc = gpu_select(Q, Kr, 1, 6, 1, 1, 16)
    for qb in range(6, 24):
        assert list(gi[0, 0, qb]) == [0, 1, 2, 3, 4, qb], qb


def gpu_fwd(Q, K, V, idx, cnt, m):
    O, lse = phsa.phsa_sparse_attn_fwd(to_dev_bf16(Q), to_dev_bf16(K), to_dev_bf16(V),
                                       torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda(),
                                       block_size=m)
    torch.cuda.synchronize()
    return O, lse


@pytest.mark.parametrize("m,B,Hq,Hkv,L,topk", [
    (16, 1, 2, 1, 16 * 70 + 9, 7),    # G = 2, ragged tail; key tiles of four blocks, some short
    (16, 2, 4, 2, 16 * 33, 5),        # B = 2
    (16, 1, 3, 3, 16 * 41 + 1, 6),    # G = 1, a one-token tail block
    (16, 1, 2, 1, 11, 2),             # shorter than one block
    (32, 1, 4, 2, 32 * 25 + 17, 4),   # m = 32: key tiles of two blocks
    (32, 1, 2, 2, 32 * 18, 3),        # m = 32, G = 1
])
def test_forward_matches_oracle(m, B, Hq, Hkv, L, topk):
    rng = np.random.default_rng(L * 3 + m)
    Q, K, V = rand(rng, B, Hq, L, D), rand(rng, B, Hkv, L, D), rand(rng, B, Hkv, L, D)
    mask = (rng.random((B, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, m, 0.5)
    idx, cnt = oracle.select_blocks(Q, Kr, L, m, topk, 1, 1, SCALE)
    O, lse = gpu_fwd(Q, K, V, idx, cnt, m)
    Or, lser = oracle.sparse_attn_fwd(Q, K, V, idx, cnt, m, SCALE)
    assert_close("O", bf16_to_f64(O), Or)
    assert np.abs(lse.cpu().numpy() - lser).max() <= LSE_ABS
    assert phsa.phsa_get_device_status() == 0


@pytest.mark.parametrize("m", [16, 32])
def test_forward_full_budget_is_dense_causal(m):
    B, Hq, Hkv, L = 1, 4, 2, m * 21 + 5
    NQB = -(-L // m)
    rng = np.random.default_rng(m)
    Q, K, V = rand(rng, B, Hq, L, D), rand(rng, B, Hkv, L, D), rand(rng, B, Hkv, L, D)
    idx = np.full((B, Hkv, NQB, NQB), -1, np.int32)
    cnt = np.zeros((B, Hkv, NQB), np.int32)
    for qb in range(NQB):
        idx[:, :, qb, :qb + 1] = np.arange(qb + 1)
        cnt[:, :, qb] = qb + 1
    O, lse = gpu_fwd(Q, K, V, idx, cnt, m)
    Od, lsed = oracle.dense_causal(Q, K, V, SCALE)
    assert_close("O", bf16_to_f64(O), Od)
    assert np.abs(lse.cpu().numpy() - lsed).max() <= LSE_ABS


def test_forward_constant_values_give_constant_output_at_m16():
    rng = np.random.default_rng(4)
    L, m = 16 * 30, 16
    Q, K = rand(rng, 1, 2, L, D), rand(rng, 1, 1, L, D)
    V = np.full((1, 1, L, D), inputs.f32_to_bf16_bits(np.array([0.75], np.float32))[0], np.uint16)
    Kr = oracle.block_repr(K, np.zeros((1, L), np.uint8), m, 0.5)
    idx, cnt = oracle.select_blocks(Q, Kr, L, m, 5, 1, 1, SCALE)
    O, _ = gpu_fwd(Q, K, V, idx, cnt, m)
    assert np.all(bf16_to_f64(O) == 0.75)


def test_forward_path_end_to_end_at_m16():
    # (a) -> (b) -> (c) through phsa_forward with the paper's block size; the
    # selection is compared first, and the output whenever the sets agree.
    B, Hq, Hkv, L, m, topk, n_init, n_local, lam = 1, 4, 2, 16 * 150 + 3, 16, 20, 2, 8, 0.5
    rng = np.random.default_rng(77)
    pset = inputs.punct_id_set(rng)
    ids = inputs.draw_token_ids(rng, B, L, "uniform8", (9, 25), pset)
    mask = oracle.punct_mask(ids, pset)
    Q, K, V = rand(rng, B, Hq, L, D), rand(rng, B, Hkv, L, D), rand(rng, B, Hkv, L, D)
    O, lse, gi, gc, Krd = phsa.phsa_forward(to_dev_bf16(Q), to_dev_bf16(K), to_dev_bf16(V),
                                            torch.from_numpy(mask).cuda(), lam, topk, n_init,
                                            n_local, block_size=m)
    torch.cuda.synchronize()
    Kr = oracle.block_repr(K, mask, m, lam)
    assert ulp_distance(bf16_bits(Krd), Kr).max() <= 1
    oi, oc, oa = oracle.select_blocks(Q, Kr, L, m, topk, n_init, n_local, SCALE, want_agg=True)
    bad, _, differ, msgs = compare_selection(gi.cpu().numpy(), gc.cpu().numpy(), oi, oc, oa)
    assert bad == 0, msgs[:5]
    assert phsa.phsa_get_device_status() == 0
    if differ == 0:  # the same sets: the outputs must agree too
        Or, lser = oracle.sparse_attn_fwd(Q, K, V, oi, oc, m, SCALE)
        assert_close("O", bf16_to_f64(O), Or)
        assert np.abs(lse.cpu().numpy() - lser).max() <= LSE_ABS


def _sampled_selection(m, L, topk, n_init, n_local, aggregation, seed, extra_units=()):
    """GPU selection of a GQA pair vs the oracle's on sampled units (the first,
    middle and last query blocks, `extra_units` and 24 random ones)."""
    rng = np.random.default_rng(seed)
    Q, K = rand(rng, 1, 2, L, D), rand(rng, 1, 1, L, D)
    mask = (rng.random((1, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, m, 0.5)
    gi, gc = gpu_select(Q, Kr, 1, topk, n_init, n_local, m, aggregation)
    NQB = -(-L // m)
    units = np.unique(np.concatenate([[0, NQB - 1, NQB // 2], list(extra_units),
                                      rng.integers(0, NQB, 24)])).astype(np.int64)
    oi, oc, oa = oracle.select_units(Q, Kr, L, m, topk, n_init, n_local, SCALE, units,
                                     aggregation=aggregation)
    bad, _, differ, msgs = compare_selection(gi.reshape(-1, topk)[units], gc.reshape(-1)[units],
                                             oi, oc, oa)
    assert bad == 0, msgs[:5]
    assert differ <= 1
    assert phsa.phsa_get_device_status() == 0


@pytest.mark.parametrize("aggregation", ["softmax_sum", "max_logit"])
def test_selection_long_sequence_at_m16_uses_the_warp_mma_kernel(aggregation):
    # 4200 query blocks of 16: the tcgen05 kernel's per-block sums no longer fit
    # in shared memory, so the pair runs on the warp-MMA kernel; sampled units
    # against the oracle's selection.
    _sampled_selection(16, 16 * 4200 + 3, 20, 1, 2, aggregation, 4200)


@pytest.mark.parametrize("n_init,n_local", [(1, 1), (2, 8)])
@pytest.mark.parametrize("aggregation", ["softmax_sum", "max_logit"])
def test_selection_span_pair_kernel_at_m64_beyond_1024_query_blocks(n_init, n_local, aggregation):
    # Past 1024 query blocks of 64 the pair selection runs on the span-pair
    # kernel (two 64-token spans share every candidate chunk); its candidate
    # ranges reach 9 chunks, more than the ring holds for pass 2.
    NQB = 1100
    _sampled_selection(64, 64 * NQB + 17, 14, n_init, n_local, aggregation, 1100 + n_local,
                       extra_units=[NQB - 2, NQB - 3, 1025, 1024, 1023])


@pytest.mark.parametrize("m,L,topk,n_init,n_local", [
    (16, 16 * 300 + 9, 40, 1, 2),   # 37 picks per query block: beyond the two-level top-k
    (32, 32 * 200 + 5, 36, 1, 1),   # 34 picks at m = 32
])
@pytest.mark.parametrize("aggregation", ["softmax_sum", "max_logit"])
def test_selection_tcgen05_large_budget_uses_one_warp_rounds(m, L, topk, n_init, n_local,
                                                             aggregation):
    # At m < 64 the tcgen05 kernel runs each query block's top-k on its scoring
    # warps; budgets above 32 picks take the one-warp rounds instead of the
    # two-level selection. Full comparison with the oracle.
    rng = np.random.default_rng(L + topk)
    Q, K = rand(rng, 1, 2, L, D), rand(rng, 1, 1, L, D)
    mask = (rng.random((1, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, m, 0.5)
    gi, gc = gpu_select(Q, Kr, 1, topk, n_init, n_local, m, aggregation)
    oi, oc, oa = oracle.select_blocks(Q, Kr, L, m, topk, n_init, n_local, SCALE, want_agg=True,
                                      aggregation=aggregation)
    bad, _, differ, msgs = compare_selection(gi, gc, oi, oc, oa)
    assert bad == 0, msgs[:5]
    assert differ <= max(2, 0.01 * oc.size), (differ, oc.size)
    assert phsa.phsa_get_device_status() == 0


@pytest.mark.parametrize("aggregation", ["softmax_sum", "max_logit"])
def test_selection_tcgen05_more_than_2048_candidates_at_m16(aggregation):
    # 2300 query blocks of 16: the last ones have more than 2048 candidates,
    # past the two-level top-k, so the tcgen05 kernel takes the one-warp rounds.
    NQB = 2300
    _sampled_selection(16, 16 * NQB, 14, 1, 2, aggregation, 2300,
                       extra_units=[NQB - 2, NQB - 3, 2100, 2060])


@pytest.mark.parametrize("m", [16, 32])
@pytest.mark.parametrize("aggregation", ["softmax_sum", "max_logit"])
def test_selection_warp_mma_pair_kernels_on_short_inputs(m, aggregation):
    # The warp-MMA kernels for GQA pairs (select_blocks_kernel<2, m>) normally
    # run only beyond ~64k tokens at m = 16 and ~250k at m = 32; a lowered
    # switch point sends a short input to them.
    prev = phsa.phsa_test_set_select_tc_limit(1)
    try:
        L, topk = m * 150 + 7, 12
        rng = np.random.default_rng(m * 7 + len(aggregation))
        Q, K = rand(rng, 1, 4, L, D), rand(rng, 1, 2, L, D)
        mask = (rng.random((1, L)) < 0.06).astype(np.uint8)
        Kr = oracle.block_repr(K, mask, m, 0.5)
        gi, gc = gpu_select(Q, Kr, 2, topk, 1, 2, m, aggregation)
        oi, oc, oa = oracle.select_blocks(Q, Kr, L, m, topk, 1, 2, SCALE, want_agg=True,
                                          aggregation=aggregation)
        bad, _, differ, msgs = compare_selection(gi, gc, oi, oc, oa)
        assert bad == 0, msgs[:5]
        assert differ <= max(2, 0.01 * oc.size), (differ, oc.size)
        assert phsa.phsa_get_device_status() == 0
    finally:
        phsa.phsa_test_set_select_tc_limit(prev)


@pytest.mark.parametrize("m,B,Hq,Hkv,L,topk,n_init,n_local", [
    (16, 1, 2, 1, 16 * 70 + 9, 7, 1, 1),     # ragged tail; four blocks of 16 per 64-key span
    (16, 2, 4, 2, 16 * 33, 5, 1, 1),         # B = 2, two KV heads
    (16, 1, 2, 1, 16 * 300 + 5, 20, 2, 8),   # the first spans' lists exceed one work item (128)
    (16, 1, 2, 1, 16 * 24, 30, 1, 1),        # budget covers everything: dense rows
    (32, 1, 4, 2, 32 * 25 + 17, 4, 1, 1),    # m = 32: two blocks per span
    (32, 1, 2, 1, 32 * 150 + 31, 9, 2, 2),   # m = 32, lists over one work item (64)
])
def test_backward_matches_oracle(m, B, Hq, Hkv, L, topk, n_init, n_local):
    # The backward at the paper's block size on the tcgen05 kernels: dQ over the
    # union of a span's lists, dK/dV over 64-key spans with gathered query blocks.
    rng = np.random.default_rng(L * 5 + m)
    Q, K, V = rand(rng, B, Hq, L, D), rand(rng, B, Hkv, L, D), rand(rng, B, Hkv, L, D)
    dO = rand(rng, B, Hq, L, D)
    mask = (rng.random((B, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, m, 0.5)
    idx, cnt = oracle.select_blocks(Q, Kr, L, m, topk, n_init, n_local, SCALE)
    it, ct = torch.from_numpy(idx).cuda(), torch.from_numpy(cnt).cuda()
    Qd, Kd, Vd, dOd = (to_dev_bf16(x) for x in (Q, K, V, dO))
    O, lse = phsa.phsa_sparse_attn_fwd(Qd, Kd, Vd, it, ct, block_size=m)
    dQ, dK, dV = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct, block_size=m)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    rq, rk, rv = oracle.sparse_attn_bwd(Q, K, V, dO, idx, cnt, m, SCALE)
    assert_close("dQ", bf16_to_f64(dQ), rq)
    assert_close("dK", bf16_to_f64(dK), rk)
    assert_close("dV", bf16_to_f64(dV), rv)


def test_backward_at_m16_rejects_a_single_query_head_per_kv_head():
    B, Hq, Hkv, L = 1, 2, 2, 16 * 8
    assert phsa.phsa_sparse_attn_bwd_workspace(B, L, Hq, Hkv, 4, block_size=16) == 0
