"""Pins for the oracle's decode functions (one new token per sequence).

Decode applies the selection rule of Section 3.3 / Algorithm 1 to a query
"block" that holds the single new row p = lens[b] - 1 of each query head of
the group, and Eq. 10-11 to that row. These tests tie it to things fixed
independently of the decode code:
  * a prefill query block whose only row is p (L = p + 1, p a multiple of m)
    is exactly the decode problem, so the prefill selection must agree bit
    for bit, aggregates included;
  * with one query head per group the softmax is monotone, so the choice is the
    per-token Top-K of raw scores q . M_t of Algorithm 1;
  * a budget that covers every block gives dense causal attention (Eq. 1-2)
    for the last row;
  * one token attends only to itself; an empty sequence has no query.
"""
import numpy as np
import pytest

import oracle
from paper_2601_02819_gb300 import inputs

D, M = 128, 64
SCALE = D ** -0.5


def _case(seed, B, Hq, Hkv, Lc):
    rng = np.random.default_rng(seed)
    f = lambda *s: inputs.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    Q, K, V = f(B, Hq, Lc, D), f(B, Hkv, Lc, D), f(B, Hkv, Lc, D)
    mask = (rng.random((B, Lc)) < 0.06).astype(np.uint8)
    return Q, K, V, mask


def _last_rows(Q, lens):
    return np.stack([Q[b, :, lens[b] - 1] for b in range(len(lens))])


@pytest.mark.parametrize("aggregation", ["softmax_sum", "max_logit"])
def test_decode_select_equals_prefill_block_with_one_row(aggregation):
    B, Hq, Hkv, Lc = 3, 4, 2, 64 * 20
    lens = np.array([64 * 7 + 1, 64 * 12 + 1, 64 * 19 + 1], np.int32)
    Q, K, _, mask = _case(1, B, Hq, Hkv, Lc)
    Kr = oracle.block_repr(K, mask, M, 0.5)
    topk = 5
    di, dc, da = oracle.decode_select(_last_rows(Q, lens), Kr, lens, Lc, M, topk, 1, 1, SCALE,
                                      want_agg=True, aggregation=aggregation)
    for b, L in enumerate(lens):
        Krb = oracle.block_repr(K[b:b + 1, :, :L], mask[b:b + 1, :L], M, 0.5)
        pi, pc, pa = oracle.select_blocks(Q[b:b + 1, :, :L], Krb, int(L), M, topk, 1, 1, SCALE,
                                          want_agg=True, aggregation=aggregation)
        qb = (L - 1) // M
        assert np.array_equal(di[b], pi[0, :, qb]), b
        assert np.array_equal(dc[b], pc[0, :, qb]), b
        T = L // M
        a_dec, a_pf = da[b, :, :T], pa[0, :, qb, :T]
        assert np.array_equal(np.isnan(a_dec), np.isnan(a_pf))
        assert np.array_equal(a_dec[~np.isnan(a_dec)], a_pf[~np.isnan(a_pf)])


def test_decode_select_with_one_head_is_per_token_topk_of_raw_scores():
    B, Hq, Hkv, Lc = 4, 2, 2, 64 * 30
    lens = np.array([64 * 30, 64 * 25 + 17, 64 * 9 + 3, 64 * 16 + 63], np.int32)
    Q, K, _, mask = _case(2, B, Hq, Hkv, Lc)
    Kr = oracle.block_repr(K, mask, M, 0.5)
    topk, n_init, n_local = 6, 1, 2
    q = _last_rows(Q, lens)
    di, dc = oracle.decode_select(q, Kr, lens, Lc, M, topk, n_init, n_local, SCALE)
    qf, Krf = oracle.bf16_to_f64(q), oracle.bf16_to_f64(Kr)
    checked = 0
    for b, L in enumerate(lens):
        qb = (L - 1) // M
        forced = set(range(n_init)) | set(range(max(0, qb - n_local + 1), qb + 1))
        cand = [t for t in range(qb) if t not in forced and t < L // M]
        for g in range(Hkv):
            s = np.array([qf[b, g] @ Krf[b, g, t] for t in cand])
            order = sorted(range(len(cand)), key=lambda c: (-s[c], cand[c]))
            k = topk - len(forced)
            gap = s[order[k - 1]] - s[order[k]]
            if gap < 1e-9:
                continue  # too close for the binary32 ranking to be decided by the score
            want = sorted(forced | {cand[c] for c in order[:k]})
            assert list(di[b, g, :dc[b, g]]) == want, (b, g)
            assert np.all(di[b, g, dc[b, g]:] == -1)
            checked += 1
    assert checked >= 6


def test_decode_full_budget_is_dense_causal_last_row():
    B, Hq, Hkv, Lc = 2, 4, 2, 64 * 9
    lens = np.array([64 * 9, 64 * 5 + 30], np.int32)
    Q, K, V, _ = _case(3, B, Hq, Hkv, Lc)
    topk = Lc // M
    idx = np.full((B, Hkv, topk), -1, np.int32)
    cnt = np.zeros((B, Hkv), np.int32)
    for b, L in enumerate(lens):
        nb = (L - 1) // M + 1
        idx[b, :, :nb] = np.arange(nb)
        cnt[b] = nb
    O, lse = oracle.decode_attn(_last_rows(Q, lens), K, V, idx, cnt, lens, M, SCALE)
    for b, L in enumerate(lens):
        Od, lsed = oracle.dense_causal(Q[b:b + 1, :, :L], K[b:b + 1, :, :L], V[b:b + 1, :, :L],
                                       SCALE)
        np.testing.assert_allclose(O[b], Od[0, :, L - 1], rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse[b], lsed[0, :, L - 1], rtol=0, atol=1e-12)


def test_decode_attn_equals_the_prefill_row_with_the_same_blocks():
    B, Hq, Hkv, Lc = 3, 4, 2, 64 * 16
    lens = np.array([64 * 16, 64 * 11 + 40, 200], np.int32)
    Q, K, V, mask = _case(4, B, Hq, Hkv, Lc)
    Kr = oracle.block_repr(K, mask, M, 0.5)
    topk = 5
    q = _last_rows(Q, lens)
    di, dc = oracle.decode_select(q, Kr, lens, Lc, M, topk, 1, 1, SCALE)
    O, lse = oracle.decode_attn(q, K, V, di, dc, lens, M, SCALE)
    for b, L in enumerate(lens):
        NQB = -(-int(L) // M)
        qb = (L - 1) // M
        pidx = np.full((1, Hkv, NQB, topk), -1, np.int32)
        pcnt = np.zeros((1, Hkv, NQB), np.int32)
        pidx[0, :, qb] = di[b]
        pcnt[0, :, qb] = dc[b]
        rows = np.array([[0, h, L - 1] for h in range(Hq)], np.int32)
        Or, lr = oracle.sparse_attn_rows(Q[b:b + 1, :, :L], K[b:b + 1, :, :L], V[b:b + 1, :, :L],
                                         pidx, pcnt, M, SCALE, rows)
        assert np.array_equal(O[b], Or) and np.array_equal(lse[b], lr)


def test_decode_degenerate_lengths():
    B, Hq, Hkv, Lc = 4, 2, 1, 64 * 4
    lens = np.array([0, 1, 64, 65], np.int32)
    Q, K, V, mask = _case(5, B, Hq, Hkv, Lc)
    Kr = oracle.block_repr(K, mask, M, 0.5)
    q = np.stack([Q[b, :, max(int(lens[b]) - 1, 0)] for b in range(B)])
    di, dc = oracle.decode_select(q, Kr, lens, Lc, M, 4, 1, 1, SCALE)
    assert dc[0, 0] == 0 and np.all(di[0, 0] == -1)      # no token, no query
    assert list(di[1, 0]) == [0, -1, -1, -1]              # p = 0: its own block
    assert list(di[2, 0]) == [0, -1, -1, -1]              # p = 63: still block 0
    assert list(di[3, 0]) == [0, 1, -1, -1]               # p = 64: forced {0, 1}, nothing to score
    O, lse = oracle.decode_attn(q, K, V, di, dc, lens, M, SCALE)
    assert np.all(O[0] == 0) and np.all(np.isneginf(lse[0]))
    # a single key: the softmax weight is 1 and the output is that key's value
    assert np.array_equal(O[1], np.broadcast_to(oracle.bf16_to_f64(V[1, 0, 0]), (Hq, D)))


def test_decode_length_beyond_capacity_is_rejected():
    B, Hq, Hkv, Lc = 1, 2, 1, 128
    Q, K, _, mask = _case(6, B, Hq, Hkv, Lc)
    Kr = oracle.block_repr(K, mask, M, 0.5)
    with pytest.raises(ValueError):
        oracle.decode_select(Q[:, :, 0], Kr, np.array([Lc + 1], np.int32), Lc, M, 3, 1, 1, SCALE)
