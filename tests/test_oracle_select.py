"""Pins for the oracle's scoring and block selection (Eq. 8; Algorithm 1 step 3).

Expected selections come from constructed inputs whose answer is fixed by
hand (one-hot representative keys give exact scores), from the per-token case
of Algorithm 1 checked with numpy's own sort, and from invariants.
"""
import numpy as np
import pytest

import oracle
from paper_2601_02819_gb300.inputs import f32_to_bf16_bits

D = 128


def bf(x):
    return f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def sel(Q, Kr, L, m, topk, n_init=1, n_local=1, scale=1.0, agg=False):
    return oracle.select_blocks(Q, Kr, L, m, topk, n_init, n_local, scale, want_agg=agg)


def onehot_repr(T, Hkv=1, B=1):
    """Krepr_t = e_t: the score of block t for a query row is q[t] exactly (scale 1)."""
    Kr = np.zeros((B, Hkv, T, D), np.float32)
    for t in range(T):
        Kr[:, :, t, t] = 1.0
    return bf(Kr)


def test_full_budget_selects_every_causal_block():
    rng = np.random.default_rng(0)
    L, m = 64 * 7, 64
    Q = bf(rng.standard_normal((1, 2, L, D)))
    Kr = bf(rng.standard_normal((1, 1, 7, D)))
    idx, cnt = sel(Q, Kr, L, m, topk=7, scale=D ** -0.5)
    for qb in range(7):
        assert cnt[0, 0, qb] == qb + 1
        assert list(idx[0, 0, qb, :qb + 1]) == list(range(qb + 1))
        assert np.all(idx[0, 0, qb, qb + 1:] == -1)


@pytest.mark.parametrize("qb,expect", [
    (0, [0]), (1, [0, 1]), (2, [0, 1, 2]), (3, [0, 1, 2, 3]),
    (5, [0, 1, 3, 4, 5]), (9, [0, 1, 7, 8, 9]),
])
def test_forced_blocks_only(qb, expect):
    # n_init = 2, n_local = 3: F_b = {0, 1} U {b-2, b-1, b}, clipped and de-duplicated.
    rng = np.random.default_rng(1)
    L, m = 64 * 10, 64
    Q = bf(rng.standard_normal((1, 1, L, D)))
    Kr = bf(rng.standard_normal((1, 1, 10, D)))
    idx, cnt = sel(Q, Kr, L, m, topk=5, n_init=2, n_local=3, scale=D ** -0.5)
    assert cnt[0, 0, qb] == len(expect)
    assert list(idx[0, 0, qb, :len(expect)]) == expect
    assert np.all(idx[0, 0, qb, len(expect):] == -1)


def test_topk_below_forced_count_is_rejected():
    Q = bf(np.zeros((1, 1, 640, D)))
    Kr = bf(np.zeros((1, 1, 10, D)))
    with pytest.raises(ValueError):
        sel(Q, Kr, 640, 64, topk=4, n_init=2, n_local=3)


def test_per_token_case_is_argsort_of_raw_scores():
    # Block size 1, one query head per KV head: each query block is one token and
    # each representative key is that token's key (M_0 = M_p = K_t), so the
    # selection must be Algorithm 1's per-token Top-K of q_i . k_t (softmax is monotone).
    rng = np.random.default_rng(2)
    L, n_init, n_local, extra = 40, 2, 3, 4
    topk = n_init + n_local + extra
    Q = bf(rng.standard_normal((1, 1, L, D)))
    K = bf(rng.standard_normal((1, 1, L, D)))
    mask = (rng.random((1, L)) < 0.3).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, 1, 0.37)
    assert np.array_equal(Kr, K)
    idx, cnt = sel(Q, Kr, L, 1, topk, n_init, n_local, scale=D ** -0.5)
    q = oracle.bf16_to_f64(Q)[0, 0]
    k = oracle.bf16_to_f64(K)[0, 0]
    S = q @ k.T
    for i in range(L):
        forced = set(range(min(n_init, i + 1))) | set(range(max(0, i - n_local + 1), i + 1))
        cands = [t for t in range(i) if t not in forced]
        order = sorted(cands, key=lambda t: (-S[i, t], t))
        expect = sorted(forced | set(order[:extra]))
        assert cnt[0, 0, i] == len(expect), i
        assert list(idx[0, 0, i, :len(expect)]) == expect, i


def test_exact_tie_goes_to_the_lower_block():
    # Blocks 2 and 5 have identical representative keys and win over the rest.
    rng = np.random.default_rng(3)
    L, m, T = 64 * 8, 64, 8
    Kr = bf(rng.standard_normal((1, 1, T, D)) * 0.05)
    u = bf(rng.standard_normal(D))
    Kr[0, 0, 2] = u
    Kr[0, 0, 5] = u
    Q = np.broadcast_to(u, (1, 1, L, D)).copy()
    idx, cnt = sel(Q, Kr, L, m, topk=3, scale=D ** -0.5)  # forced {0, 7} + one pick
    assert list(idx[0, 0, 7]) == [0, 2, 7]


def _onehot_case(row_scores_h0, row_scores_h1=None, forced_bias=0.0):
    """Query block 4 of a 5-block sequence; candidates are blocks 1, 2, 3.

    Each query row r gets q_r[t] = the score wanted for block t. Forced blocks 0
    and 4 get score ``forced_bias`` so that a reading that wrongly normalises over
    them would see them.
    """
    G = 1 if row_scores_h1 is None else 2
    L, m, T = 64 * 5, 64, 5
    Q = np.zeros((1, G, L, D), np.float32)
    for h, rs in enumerate([row_scores_h0] + ([row_scores_h1] if G == 2 else [])):
        for r, s in enumerate(rs):
            Q[0, h, 4 * m + r, [1, 2, 3]] = s
            Q[0, h, 4 * m + r, [0, 4]] = forced_bias
    return bf(Q), onehot_repr(T), L, m


def test_relevance_is_the_summed_softmax_over_candidates_only():
    # Row 0 scores (100, 0, 0); rows 1..63 score (0, 0.5, 0); forced blocks score 10.
    # Softmax over candidates summed over rows: A_1 = 1 + 63/(2+e^0.5) = 18.27,
    # A_2 = 63 e^0.5/(2+e^0.5) = 28.46 -> block 2. Raw-score sums, the max logit, or
    # a softmax that also counts the forced blocks would all pick block 1.
    rows = [(100.0, 0.0, 0.0)] + [(0.0, 0.5, 0.0)] * 63
    Q, Kr, L, m = _onehot_case(rows, forced_bias=10.0)
    idx, cnt, A = sel(Q, Kr, L, m, topk=3, agg=True)
    assert list(idx[0, 0, 4]) == [0, 2, 4]
    e = np.exp(0.5)
    np.testing.assert_allclose(A[0, 0, 4, 1:4], [1 + 63 / (2 + e), 63 * e / (2 + e),
                                                 63 / (2 + e)], rtol=1e-12, atol=1e-12)
    assert np.isnan(A[0, 0, 4, 0]) and np.isnan(A[0, 0, 4, 4])  # forced: never scored


def test_relevance_at_block_size_16():
    # The closed form above with m = 16: query block 4 has 16 rows; row 0 scores
    # (100, 0, 0), rows 1..15 score (0, 0.5, 0). A_1 = 1 + 15/(2+e^0.5) = 5.11,
    # A_2 = 15 e^0.5/(2+e^0.5) = 6.78 -> block 2 (64 rows would give the same pick
    # with other values; a block size read as 64 would see 64 rows of zeros).
    L, m, T = 16 * 5, 16, 5
    Q = np.zeros((1, 1, L, D), np.float32)
    for r in range(m):
        Q[0, 0, 4 * m + r, [1, 2, 3]] = (100.0, 0.0, 0.0) if r == 0 else (0.0, 0.5, 0.0)
        Q[0, 0, 4 * m + r, [0, 4]] = 10.0
    idx, cnt, A = sel(bf(Q), onehot_repr(T), L, m, topk=3, agg=True)
    assert list(idx[0, 0, 4]) == [0, 2, 4]
    e = np.exp(0.5)
    np.testing.assert_allclose(A[0, 0, 4, 1:4], [1 + 15 / (2 + e), 15 * e / (2 + e), 15 / (2 + e)],
                               rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("h1_score,expect", [(0.5, 1), (2.0, 2)])
def test_both_heads_of_a_group_vote(h1_score, expect):
    # Head 0 rows score (1, 0, 0), head 1 rows score (0, s, 0).
    # s = 0.5: A_1 = 64 (e/(e+2) + 1/(2+e^.5)) = 54.4 > A_2 = 64 (1/(e+2) + e^.5/(2+e^.5)) = 42.5
    # s = 2:   A_1 = 64 (e/(e+2) + 1/(e^2+2)) = 43.7 < A_2 = 64 (1/(e+2) + e^2/(e^2+2)) = 63.9
    # Using head 0 alone would give block 1 both times, head 1 alone block 2 both times.
    h0 = [(1.0, 0.0, 0.0)] * 64
    h1 = [(0.0, h1_score, 0.0)] * 64
    Q, Kr, L, m = _onehot_case(h0, h1)
    idx, cnt = sel(Q, Kr, L, m, topk=3)
    assert list(idx[0, 0, 4]) == sorted([0, 4, expect])


def test_punctuation_branch_changes_the_choice():
    # Blocks 1 and 3 hold the same keys, including one key u; in block 3 that token is
    # punctuation, in block 1 it is not. With lambda = 1 (mean pooling only) the two
    # representatives are equal and the tie goes to block 1; with lambda = 0.5 the
    # punctuation branch lifts block 3 (its representative gains 0.5 u).
    rng = np.random.default_rng(4)
    L, m = 64 * 6, 64
    K = bf(rng.standard_normal((1, 1, L, D)) * 0.1)
    u = bf(rng.standard_normal(D) * 2)
    K[0, 0, 64:128] = K[0, 0, 192:256]
    K[0, 0, 64 + 17] = u
    K[0, 0, 192 + 17] = u
    mask = np.zeros((1, L), np.uint8)
    mask[0, 192 + 17] = 1
    Q = np.broadcast_to(u, (1, 1, L, D)).copy()
    for lam, expect in [(1.0, 1), (0.5, 3)]:
        Kr = oracle.block_repr(K, mask, m, lam)
        idx, cnt = sel(Q, Kr, L, m, topk=3, scale=D ** -0.5)
        assert list(idx[0, 0, 5]) == sorted([0, 5, expect]), lam


def test_ragged_tail_query_block():
    # L = 330: NQB = 6, T = 5. The tail query block (10 rows) keeps its own partial
    # block (forced local, no representative) and picks among blocks 1-4.
    L, m = 330, 64
    Q = np.zeros((1, 1, L, D), np.float32)
    Q[0, 0, 320:, 2] = 1.0
    Q[0, 0, 320:, 4] = 0.9
    Kr = onehot_repr(5)
    idx, cnt = sel(bf(Q), Kr, L, m, topk=4)
    assert cnt[0, 0, 5] == 4
    assert list(idx[0, 0, 5]) == [0, 2, 4, 5]


def test_selection_ignores_row_order():
    rng = np.random.default_rng(5)
    L, m = 64 * 12, 64
    Q = bf(rng.standard_normal((2, 4, L, D)))
    Kr = bf(rng.standard_normal((2, 2, 12, D)))
    idx, cnt = sel(Q, Kr, L, m, topk=5, scale=D ** -0.5)
    Qp = Q.copy()
    for qb in range(12):
        perm = rng.permutation(m)
        Qp[:, :, qb * m:(qb + 1) * m] = Q[:, :, qb * m + perm]
    Qp[:, [0, 1]] = Qp[:, [1, 0]]  # swap the two heads of KV group 0
    idx2, cnt2 = sel(Qp, Kr, L, m, topk=5, scale=D ** -0.5)
    assert np.array_equal(idx, idx2) and np.array_equal(cnt, cnt2)


def test_output_is_ascending_unique_and_budgeted():
    rng = np.random.default_rng(6)
    L, m, topk = 64 * 40 + 17, 64, 9
    Q = bf(rng.standard_normal((2, 4, L, D)))
    Kr = bf(rng.standard_normal((2, 2, L // m, D)))
    idx, cnt = sel(Q, Kr, L, m, topk, n_init=2, n_local=2, scale=D ** -0.5)
    for b in range(2):
        for g in range(2):
            for qb in range(idx.shape[2]):
                n = cnt[b, g, qb]
                row = idx[b, g, qb]
                assert n == min(topk, qb + 1)
                assert np.all(np.diff(row[:n]) > 0) and np.all(row[n:] == -1)
                assert row[0] == 0 and row[n - 1] == qb
                assert {0, 1} & set(range(qb + 1)) <= set(row[:n])


# ---- the max-logit aggregation (A_t = max over the group's rows of S_{r,t}) ----

def sel_max(Q, Kr, L, m, topk, n_init=1, n_local=1, scale=1.0, agg=False):
    return oracle.select_blocks(Q, Kr, L, m, topk, n_init, n_local, scale, want_agg=agg,
                                aggregation="max_logit")


def test_max_logit_takes_the_largest_raw_score_over_rows():
    # The case above: one row scores (100, 0, 0), 63 rows (0, 0.5, 0), forced blocks 10.
    # A = (100, 0.5, 0) exactly; the forced blocks' scores play no part.
    rows = [(100.0, 0.0, 0.0)] + [(0.0, 0.5, 0.0)] * 63
    Q, Kr, L, m = _onehot_case(rows, forced_bias=10.0)
    idx, cnt, A = sel_max(Q, Kr, L, m, topk=3, agg=True)
    assert list(idx[0, 0, 4]) == [0, 1, 4]
    assert list(A[0, 0, 4, 1:4]) == [100.0, 0.5, 0.0]
    assert np.isnan(A[0, 0, 4, 0]) and np.isnan(A[0, 0, 4, 4])
    idx2, _ = sel_max(Q, Kr, L, m, topk=4)  # second pick: 0.5 beats 0
    assert list(idx2[0, 0, 4]) == [0, 1, 2, 4]


@pytest.mark.parametrize("s,expect", [(0.5, 1), (2.0, 2), (-3.0, 1)])
def test_max_logit_over_both_heads(s, expect):
    # head 0 rows score (1, 0, 0), head 1 rows (0, s, 0): A = (1, max(0, s), 0)
    Q, Kr, L, m = _onehot_case([(1.0, 0.0, 0.0)] * 64, [(0.0, s, 0.0)] * 64)
    idx, cnt, A = sel_max(Q, Kr, L, m, topk=3, agg=True)
    assert list(idx[0, 0, 4]) == [0, expect, 4]
    assert list(A[0, 0, 4, 1:4]) == [1.0, max(0.0, s), 0.0]


def test_max_logit_ranks_negative_scores():
    # every candidate's best score is negative: the least negative wins
    Q, Kr, L, m = _onehot_case([(-4.0, -1.5, -2.0)] * 64)
    idx, cnt, A = sel_max(Q, Kr, L, m, topk=4, agg=True)
    assert list(idx[0, 0, 4]) == [0, 2, 3, 4]
    assert list(A[0, 0, 4, 1:4]) == [-4.0, -1.5, -2.0]


def test_max_logit_per_token_case_is_argsort_of_raw_scores():
    # With a single row per unit both aggregations rank by q_i . k_t (Algorithm 1).
    rng = np.random.default_rng(2)
    L, n_init, n_local, extra = 40, 2, 3, 4
    topk = n_init + n_local + extra
    Q = bf(rng.standard_normal((1, 1, L, D)))
    K = bf(rng.standard_normal((1, 1, L, D)))
    idx, cnt = sel_max(Q, K, L, 1, topk, n_init, n_local, scale=D ** -0.5)
    q = oracle.bf16_to_f64(Q)[0, 0]
    k = oracle.bf16_to_f64(K)[0, 0]
    S = q @ k.T
    for i in range(L):
        forced = set(range(min(n_init, i + 1))) | set(range(max(0, i - n_local + 1), i + 1))
        order = sorted((t for t in range(i) if t not in forced), key=lambda t: (-S[i, t], t))
        expect = sorted(forced | set(order[:extra]))
        assert list(idx[0, 0, i, :len(expect)]) == expect, i
    idx_sm, cnt_sm = sel(Q, K, L, 1, topk, n_init, n_local, scale=D ** -0.5)
    assert np.array_equal(idx, idx_sm) and np.array_equal(cnt, cnt_sm)


def test_max_logit_is_scale_free_and_linear_in_the_scale():
    # A positive scale multiplies every score: the choice is unchanged and A scales
    # exactly by powers of two.
    rng = np.random.default_rng(12)
    L, m = 64 * 12 + 7, 64
    Q = bf(rng.standard_normal((1, 4, L, D)))
    Kr = bf(rng.standard_normal((1, 2, 12, D)))
    i1, c1, a1 = sel_max(Q, Kr, L, m, topk=5, scale=1.0, agg=True)
    i2, c2, a2 = sel_max(Q, Kr, L, m, topk=5, scale=4.0, agg=True)
    i3, c3 = sel_max(Q, Kr, L, m, topk=5, scale=1e-3)
    assert np.array_equal(i1, i2) and np.array_equal(i1, i3) and np.array_equal(c1, c3)
    ok = ~np.isnan(a1)
    assert np.array_equal(a2[ok], 4.0 * a1[ok])
    # A is the column maximum of the unit's score matrix: 128 rows for a full query
    # block, the 2 x 7 rows that exist for the ragged last one (L = 64 * 12 + 7)
    Qf, Kf = oracle.bf16_to_f64(Q), oracle.bf16_to_f64(Kr)
    for qb, g in ((9, 1), (12, 0)):
        rows = np.concatenate([Qf[0, 2 * g + h, qb * m:min(L, (qb + 1) * m)] for h in range(2)])
        S = rows @ Kf[0, g].T
        cands = list(range(1, qb))  # n_init = 1, n_local = 1
        assert np.array_equal(a1[0, g, qb, cands], S[:, cands].max(axis=0)), qb
