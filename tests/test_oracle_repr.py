"""Pins for the oracle's representative keys (Eq. 3, 6, 7, 8; Algorithm 1 step 2).

Every expected value below is a closed form worked out by hand from the
equations for a constructed block, not a recomputation of the oracle's code.
"""
import numpy as np
import pytest

import oracle
from paper_2601_02819_gb300.inputs import f32_to_bf16_bits

M = 64


def bf(x):
    return f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def repr_vals(K, mask, lam, m=M):
    out = oracle.block_repr(K, mask, m, lam)
    return oracle.bf16_to_f64(out)


def ramp_keys(B=1, Hkv=1, L=256, D=128):
    """K[b, g, i, :] = i (the token position), exact in bf16 for i <= 256."""
    K = np.broadcast_to(np.arange(L, dtype=np.float32)[None, None, :, None], (B, Hkv, L, D))
    return bf(K)


@pytest.mark.parametrize("lam", [0.0, 0.3, 1.0])
def test_constant_block_gives_the_constant(lam):
    K = bf(np.full((1, 1, 128, 128), 0.8125))
    mask = np.zeros((1, 128), np.uint8)
    mask[0, [3, 70, 71]] = 1
    r = repr_vals(K, mask, lam)
    assert np.all(r == 0.8125)


def test_no_punctuation_is_the_mean_of_each_block():
    # Eq. 6 with K_i = i: block t averages 64t .. 64t+63 -> 64t + 31.5; bf16 rounding
    # (ties to even) turns 159.5 into 160 and 223.5 into 224. Also pins Eq. 3's blocking.
    K = ramp_keys()
    r = repr_vals(K, np.zeros((1, 256), np.uint8), 0.5)
    assert r.shape == (1, 1, 4, 128)
    assert list(r[0, 0, :, 0]) == [31.5, 95.5, 160.0, 224.0]


def test_block_size_16_means_and_one_punctuation_token():
    # Eq. 3 and 6 at m = 16 with K_i = i: block t averages 16t .. 16t+15 -> 16t + 7.5
    # (all exact in bf16 below 256). Eq. 7-8 with one punctuation token j = 37 in
    # block 2 and lambda = 0.5: 0.5 * 39.5 + 0.5 * 37 = 38.25 (exact).
    K = ramp_keys(L=128)
    r = repr_vals(K, np.zeros((1, 128), np.uint8), 0.5, m=16)
    assert r.shape == (1, 1, 8, 128)
    assert list(r[0, 0, :, 0]) == [16 * t + 7.5 for t in range(8)]
    mask = np.zeros((1, 128), np.uint8)
    mask[0, 37] = 1
    r = repr_vals(K, mask, 0.5, m=16)
    assert r[0, 0, 2, 0] == 38.25
    assert [r[0, 0, t, 0] for t in (0, 1, 3)] == [7.5, 23.5, 55.5]


@pytest.mark.parametrize("lam,j,expect", [
    (0.5, 10, 0.5 * 31.5 + 0.5 * 10),    # 20.75
    (0.25, 40, 38.0),  # 0.25*31.5 + 0.75*40 = 37.875 = 100101.111b: a bf16 tie -> even, 38
    (0.0, 17, 17.0),                     # lambda = 0: punctuation branch only
    (1.0, 17, 31.5),                     # lambda = 1: mean pooling only
])
def test_single_punctuation_token(lam, j, expect):
    # Eq. 7 with one punctuation token at j: M_p = K_j = j; Eq. 8 mixes it with M_0.
    K = ramp_keys()
    mask = np.zeros((1, 256), np.uint8)
    mask[0, j] = 1
    r = repr_vals(K, mask, lam)
    assert r[0, 0, 0, 0] == expect
    assert list(r[0, 0, 1:, 0]) == [95.5, 160.0, 224.0]  # other blocks untouched


def test_two_punctuation_tokens_average():
    # M_p = (10 + 20) / 2 = 15 in block 0; lambda = 0.5 -> 0.5 * 31.5 + 0.5 * 15 = 23.25
    K = ramp_keys()
    mask = np.zeros((1, 256), np.uint8)
    mask[0, [10, 20]] = 1
    r = repr_vals(K, mask, 0.5)
    assert r[0, 0, 0, 0] == 23.25


def test_all_punctuation_block_is_the_mean():
    K = ramp_keys()
    mask = np.zeros((1, 256), np.uint8)
    mask[0, 64:128] = 1
    r = repr_vals(K, mask, 0.3)
    assert r[0, 0, 1, 0] == 95.5


def test_columns_are_not_mixed():
    # K[i, d] = d: every block's representative key is (0, 1, ..., 127).
    K = bf(np.broadcast_to(np.arange(128, dtype=np.float32), (1, 2, 192, 128)))
    mask = np.zeros((1, 192), np.uint8)
    mask[0, 5] = 1
    r = repr_vals(K, mask, 0.5)
    assert np.all(r == np.arange(128)[None, None, None, :])


def test_batch_and_head_indexing():
    # Distinct constant per (b, g) and a per-batch mask.
    B, Hkv, L = 2, 3, 128
    vals = np.array([[1, 2, 3], [4, 5, 6]], np.float32)
    K = bf(np.broadcast_to(vals[:, :, None, None], (B, Hkv, L, 128)))
    K = K.copy()
    # make batch 1, head 2, token 7 a punctuation token with a distinct key of 14
    K[1, 2, 7, :] = bf(14.0)
    mask = np.zeros((B, L), np.uint8)
    mask[1, 7] = 1
    r = repr_vals(K, mask, 0.5)
    assert np.all(r[0, :, :, 0] == vals[0][:, None])
    # batch 1: head 0/1 have the punctuation token but a constant block -> constant
    assert r[1, 0, 0, 0] == 4 and r[1, 1, 0, 0] == 5
    # head 2 block 0: M_0 = (63*6 + 14)/64 = 6.125, M_p = 14 -> 0.5*(6.125+14) = 10.0625
    assert r[1, 2, 0, 0] == 10.0625
    assert r[1, 2, 1, 0] == 6


def test_tail_tokens_have_no_representative():
    # L = 200, m = 64 -> T = floor(200/64) = 3 (Eq. 3); tokens 192..199 belong to no block.
    K = ramp_keys(L=200)
    mask = np.zeros((1, 200), np.uint8)
    r1 = oracle.block_repr(K, mask, M, 0.5)
    K2 = K.copy()
    K2[:, :, 192:, :] = bf(99.0)
    mask2 = mask.copy()
    mask2[0, 195] = 1
    r2 = oracle.block_repr(K2, mask2, M, 0.5)
    assert r1.shape == (1, 1, 3, 128)
    assert np.array_equal(r1, r2)


def test_unrounded_values_match_closed_form():
    K = ramp_keys()
    mask = np.zeros((1, 256), np.uint8)
    mask[0, 130] = 1
    _, r64 = oracle.block_repr(K, mask, M, 0.5, want_f64=True)
    assert r64[0, 0, 2, 0] == 0.5 * 159.5 + 0.5 * 130
    assert r64[0, 0, 3, 5] == 223.5
