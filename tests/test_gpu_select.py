"""Stage (b) on the GPU vs the oracle: selected block indices.

Both sides get the oracle's representative keys, so this isolates the
selection. Indices must match exactly except for candidates whose oracle
aggregate lies within 1e-3 of the selection boundary (counted, must be rare).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300 import inputs
from paper_2601_02819_gb300 import phsa
from parity import compare_selection, to_dev_bf16

pytestmark = pytest.mark.gpu


def gpu_select(Q, Kr, Hkv, topk, n_init, n_local, scale):
    idx, cnt = phsa.phsa_select_blocks(to_dev_bf16(Q), to_dev_bf16(Kr), Hkv, topk, n_init,
                                       n_local, scale)
    torch.cuda.synchronize()
    return idx.cpu().numpy(), cnt.cpu().numpy()


def check(Q, Kr, L, Hkv, topk, n_init=1, n_local=1):
    scale = 128 ** -0.5
    gi, gc = gpu_select(Q, Kr, Hkv, topk, n_init, n_local, scale)
    oi, oc, oa = oracle.select_blocks(Q, Kr, L, 64, topk, n_init, n_local, scale, want_agg=True)
    bad, excl, differ, msgs = compare_selection(gi, gc, oi, oc, oa)
    assert bad == 0, msgs[:5]
    # sets may differ only inside the 1e-3 band, and only rarely
    assert differ <= max(2, 0.01 * oc.size), (differ, oc.size)
    print(f"selection: {oc.size} units, {differ} differ inside the band, "
          f"{excl} candidates in the band (not compared)")


def test_tiny_workload():
    w = inputs.WORKLOADS["tiny_2k"]
    x = inputs.make_inputs(w)
    Kr = oracle.block_repr(x["K"], x["mask"], 64, w.lam)
    check(x["Q"], Kr, w.L, w.Hkv, w.topk)


@pytest.mark.parametrize("B,Hq,Hkv,L,topk,n_init,n_local", [
    (2, 4, 2, 64 * 37 + 13, 6, 1, 1),   # ragged tail, G = 2
    (1, 3, 3, 64 * 40, 9, 2, 3),        # G = 1, wider forced set
    (1, 2, 1, 64 * 300, 12, 1, 2),      # many candidate tiles
    (1, 2, 1, 64 * 20, 25, 1, 1),       # budget covers everything: dense rows
    (1, 4, 2, 64 * 40 + 5, 20, 1, 1),   # G = 2: warp slices smaller than the budget
    (1, 2, 1, 64 * 160, 80, 1, 1),      # G = 2: budget above the two-level top-k limit
    (1, 2, 1, 64 * 601, 14, 2, 8),      # G = 2: paper forced sets, odd NQB, chunks reloaded
    (2, 4, 2, 64 * 3 + 1, 3, 1, 1),     # G = 2: first blocks (no candidates, all forced)
])
def test_shapes_and_forced_sets(B, Hq, Hkv, L, topk, n_init, n_local):
    rng = np.random.default_rng(B * 1000 + L)
    Q = inputs.f32_to_bf16_bits(rng.standard_normal((B, Hq, L, 128)).astype(np.float32))
    K = inputs.f32_to_bf16_bits(rng.standard_normal((B, Hkv, L, 128)).astype(np.float32))
    mask = (rng.random((B, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, 64, 0.5)
    check(Q, Kr, L, Hkv, topk, n_init, n_local)


def test_exact_ties_go_to_the_lower_block():
    # Every representative key identical: all aggregates tie, lowest candidates win.
    rng = np.random.default_rng(9)
    L, T = 64 * 24, 24
    Q = inputs.f32_to_bf16_bits(rng.standard_normal((1, 2, L, 128)).astype(np.float32))
    row = inputs.f32_to_bf16_bits(rng.standard_normal(128).astype(np.float32))
    Kr = np.broadcast_to(row, (1, 1, T, 128)).copy()
    gi, gc = gpu_select(Q, Kr, 1, 6, 1, 1, 128 ** -0.5)
    for qb in range(6, 24):
        assert list(gi[0, 0, qb]) == [0, 1, 2, 3, 4, qb], qb
    # duplicated pairs: blocks 3 and 11 share the strongest key; 3 must win
    Kr2 = inputs.f32_to_bf16_bits((rng.standard_normal((1, 1, T, 128)) * 0.1).astype(np.float32))
    u = inputs.f32_to_bf16_bits(rng.standard_normal(128).astype(np.float32))
    Kr2[0, 0, 3] = u
    Kr2[0, 0, 11] = u
    Q2 = np.broadcast_to(u, (1, 2, L, 128)).copy()
    gi, gc = gpu_select(Q2, Kr2, 1, 3, 1, 1, 128 ** -0.5)
    for qb in range(12, 24):
        assert list(gi[0, 0, qb]) == [0, 3, qb], qb


@pytest.mark.parametrize("name", ["train_8k_x4", "prefill_32k", "prefill_32k_paper_forced",
                                  "long_131k_p0"])
def test_full_size_sampled_units(name):
    if name == "prefill_32k_paper_forced":  # 128 initial + 512 local tokens, as the paper's 32k setting
        w = inputs.custom(name, B=1, L=32768, Hq=16, Hkv=8, topk=14, n_init=2, n_local=8,
                          punct="sentence", seed=77)
    else:
        w = inputs.WORKLOADS[name]
    x = inputs.make_inputs(w)
    Kr = oracle.block_repr(x["K"], x["mask"], 64, w.lam)
    scale = 128 ** -0.5
    gi, gc = gpu_select(x["Q"], Kr, w.Hkv, w.topk, w.n_init, w.n_local, scale)
    rng = np.random.default_rng(0)
    U = w.B * w.Hkv * w.NQB
    units = np.unique(np.concatenate([rng.choice(U, 96, replace=False),
                                      [0, U - 1, w.NQB - 1, w.NQB // 2]]))
    oi, oc, oa = oracle.select_units(x["Q"], Kr, w.L, 64, w.topk, w.n_init, w.n_local, scale,
                                     units)
    bad, excl, differ, msgs = compare_selection(gi.reshape(U, -1)[units],
                                                gc.reshape(-1)[units], oi, oc, oa)
    assert bad == 0, msgs[:5]
    assert differ <= max(2, 0.02 * len(units)), (differ, len(units))


@pytest.mark.parametrize("B,Hq,Hkv,L,topk,n_init,n_local", [
    (2, 4, 2, 64 * 37 + 13, 6, 1, 1),   # G = 2, ragged tail (rows past L excluded)
    (1, 3, 3, 64 * 40 + 9, 9, 2, 3),    # G = 1
    (1, 2, 1, 64 * 300, 14, 2, 8),      # G = 2, paper forced sets, several candidate tiles
    (1, 2, 1, 64 * 160, 80, 1, 1),      # G = 2, budget above the two-level top-k limit
])
def test_max_logit_rule_matches_oracle(B, Hq, Hkv, L, topk, n_init, n_local):
    rng = np.random.default_rng(B * 7 + L)
    Q = inputs.f32_to_bf16_bits(rng.standard_normal((B, Hq, L, 128)).astype(np.float32))
    K = inputs.f32_to_bf16_bits(rng.standard_normal((B, Hkv, L, 128)).astype(np.float32))
    mask = (rng.random((B, L)) < 0.06).astype(np.uint8)
    Kr = oracle.block_repr(K, mask, 64, 0.5)
    scale = 128 ** -0.5
    idx, cnt = phsa.phsa_select_blocks(to_dev_bf16(Q), to_dev_bf16(Kr), Hkv, topk, n_init,
                                       n_local, scale, aggregation="max_logit")
    torch.cuda.synchronize()
    oi, oc, oa = oracle.select_blocks(Q, Kr, L, 64, topk, n_init, n_local, scale, want_agg=True,
                                      aggregation="max_logit")
    bad, excl, differ, msgs = compare_selection(idx.cpu().numpy(), cnt.cpu().numpy(), oi, oc, oa)
    assert bad == 0, msgs[:5]
    assert differ <= max(2, 0.01 * oc.size), (differ, oc.size)
    # the rule changes the choice: the softmax-sum selection differs somewhere
    si, _ = phsa.phsa_select_blocks(to_dev_bf16(Q), to_dev_bf16(Kr), Hkv, topk, n_init, n_local,
                                    scale)
    assert not torch.equal(si, idx)


def test_unknown_aggregation_is_rejected():
    Q = torch.zeros((1, 2, 128, 128), dtype=torch.bfloat16, device="cuda")
    Kr = torch.zeros((1, 1, 2, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(ValueError):
        phsa.phsa_select_blocks(Q, Kr, 1, 2, aggregation="mean")
