"""End-to-end parity on the named workloads at full size (sampled where the
oracle would be too slow), run in the launch configuration bench.py times.

Nothing the GPU computes is fed to the oracle. The selection is checked on
sampled units against the oracle's own selection over its own representative
keys. The attention kernels are checked at full size on block lists drawn by
the seeded input generator, given to both sides.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2601_02819_gb300 import inputs
from paper_2601_02819_gb300 import phsa
from parity import LSE_ABS, assert_close, bf16_to_f64, compare_selection, to_dev_bf16

pytestmark = pytest.mark.gpu

SCALE = 128 ** -0.5


def gpu_forward(w, x):
    Qd, Kd, Vd = (to_dev_bf16(x[k]) for k in ("Q", "K", "V"))
    md = torch.from_numpy(x["mask"]).cuda()
    O, lse, idx, cnt, Kr = phsa.phsa_forward(Qd, Kd, Vd, md, w.lam, w.topk, w.n_init, w.n_local,
                                             block_size=w.block_size)
    torch.cuda.synchronize()
    return Qd, Kd, Vd, O, lse, idx, cnt


def check_selection_on_units(w, x, gi, gc, units):
    """The GPU's selection at flat units u = (b*Hkv + g)*NQB + qb against the
    oracle's, computed over the oracle's representative keys."""
    Kr = oracle.block_repr(x["K"], x["mask"], w.block_size, w.lam)
    oi, oc, oa = oracle.select_units(x["Q"], Kr, w.L, w.block_size, w.topk, w.n_init, w.n_local,
                                     SCALE, units)
    g_i = gi.reshape(-1, w.topk)[units]
    g_c = gc.reshape(-1)[units]
    bad, _, differ, msgs = compare_selection(g_i, g_c, oi, oc, oa)
    assert bad == 0, msgs[:5]
    assert differ <= max(1, len(units) // 50), differ


def test_tiny_workload_end_to_end():
    w = inputs.WORKLOADS["tiny_2k"]
    x = inputs.make_inputs(w)
    _, _, _, O, lse, idx, cnt = gpu_forward(w, x)
    Kr, oi, oc, Or, lser = oracle.forward(x["Q"], x["K"], x["V"], x["mask"], 64, w.lam, w.topk,
                                          w.n_init, w.n_local, SCALE)
    _, _, oa = oracle.select_blocks(x["Q"], Kr, w.L, 64, w.topk, w.n_init, w.n_local, SCALE,
                                    want_agg=True)
    gi, gc = idx.cpu().numpy(), cnt.cpu().numpy()
    bad, excl, _, msgs = compare_selection(gi, gc, oi, oc, oa)
    assert bad == 0, msgs[:5]
    same = np.all(gi == oi, axis=-1)[0, 0]  # query blocks whose selection matches exactly
    rows = np.repeat(same, 64)[:w.L]
    assert_close("O", bf16_to_f64(O)[:, :, rows], Or[:, :, rows])
    assert np.abs(lse.cpu().numpy()[:, :, rows] - lser[:, :, rows]).max() <= LSE_ABS


@pytest.mark.parametrize("name", ["prefill_32k", "prefill_32k_m16", "train_8k_x4", "long_131k_p0",
                                  "long_131k_p3", "long_131k_p15"])
def test_full_size_forward_sampled(name):
    w = inputs.WORKLOADS[name]
    m = w.block_size
    x = inputs.make_inputs(w)
    Qd, Kd, Vd, _, _, idx, cnt = gpu_forward(w, x)
    gi, gc = idx.cpu().numpy(), cnt.cpu().numpy()
    assert np.all(gc == np.minimum(w.topk, np.arange(w.NQB) + 1)[None, None, :])
    rng = np.random.default_rng(1)
    U = w.B * w.Hkv * w.NQB
    units = np.unique(np.concatenate([[U - 1, w.NQB // 2], rng.integers(0, U, 24)]))
    check_selection_on_units(w, x, gi, gc, units)
    # attention at full size on drawn block lists (the same for both sides)
    bi, bc = inputs.random_block_lists(rng, w.B, w.Hkv, w.NQB, w.topk)
    O, lse = phsa.phsa_sparse_attn_fwd(Qd, Kd, Vd, torch.from_numpy(bi).cuda(),
                                       torch.from_numpy(bc).cuda(), block_size=m)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    n = 256
    rows = np.stack([rng.integers(0, w.B, n), rng.integers(0, w.Hq, n),
                     rng.integers(0, w.L, n)], axis=1).astype(np.int32)
    rows[:4] = [[0, 0, 0], [w.B - 1, w.Hq - 1, w.L - 1], [0, 1, m - 1], [0, 0, m]]
    Or, lser = oracle.sparse_attn_rows(x["Q"], x["K"], x["V"], bi, bc, m, SCALE, rows)
    Og = bf16_to_f64(O)[rows[:, 0], rows[:, 1], rows[:, 2]]
    assert_close("O rows", Og, Or)
    lg = lse.cpu().numpy()[rows[:, 0], rows[:, 1], rows[:, 2]]
    assert np.abs(lg - lser).max() <= LSE_ABS


def backward_on_drawn_lists(w, x, seed):
    """GPU forward + backward on block lists drawn by the input generator."""
    rng = np.random.default_rng(seed)
    bi, bc = inputs.random_block_lists(rng, w.B, w.Hkv, w.NQB, w.topk)
    Qd, Kd, Vd, dOd = (to_dev_bf16(x[k]) for k in ("Q", "K", "V", "dO"))
    it, ct = torch.from_numpy(bi).cuda(), torch.from_numpy(bc).cuda()
    O, lse = phsa.phsa_sparse_attn_fwd(Qd, Kd, Vd, it, ct)
    dQ, dK, dV = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    return rng, bi, bc, dQ, dK, dV


def test_train_workload_backward_sampled():
    w = inputs.WORKLOADS["train_8k_x4"]
    x = inputs.make_inputs(w, with_grad=True)
    rng, bi, bc, dQ, dK, dV = backward_on_drawn_lists(w, x, 2)
    rows = np.stack([rng.integers(0, w.B, 64), rng.integers(0, w.Hq, 64),
                     rng.integers(0, w.L, 64)], axis=1).astype(np.int32)
    rq = oracle.sparse_attn_bwd_dq_rows(x["Q"], x["K"], x["V"], x["dO"], bi, bc, 64, SCALE, rows)
    assert_close("dQ rows", bf16_to_f64(dQ)[rows[:, 0], rows[:, 1], rows[:, 2]], rq)
    # block 0 is on every list: its lists span several dK/dV chunks
    blocks = np.array([[0, 0, 0], [1, 3, 1], [2, 5, 7], [3, 7, w.NQB - 1], [0, 2, 64],
                       [1, 1, 100]], np.int32)
    rk, rv = oracle.sparse_attn_bwd_kv_blocks(x["Q"], x["K"], x["V"], x["dO"], bi, bc, 64, SCALE,
                                              blocks)
    dKh, dVh = bf16_to_f64(dK), bf16_to_f64(dV)
    for n, (b, g, t) in enumerate(blocks):
        assert_close(f"dK block {t}", dKh[b, g, t * 64:(t + 1) * 64], rk[n])
        assert_close(f"dV block {t}", dVh[b, g, t * 64:(t + 1) * 64], rv[n])


def test_prefill_32k_backward_sampled():
    # The bench configuration: dQ on sampled rows, dK/dV on sampled KV blocks (block 0,
    # listed by every query block, is left to the smaller workloads).
    w = inputs.WORKLOADS["prefill_32k"]
    x = inputs.make_inputs(w, with_grad=True)
    rng, bi, bc, dQ, dK, dV = backward_on_drawn_lists(w, x, 3)
    rows = np.stack([np.zeros(48, np.int64), rng.integers(0, w.Hq, 48),
                     rng.integers(0, w.L, 48)], axis=1).astype(np.int32)
    rows[:2] = [[0, 0, w.L - 1], [0, w.Hq - 1, 64 * 300 + 7]]
    rq = oracle.sparse_attn_bwd_dq_rows(x["Q"], x["K"], x["V"], x["dO"], bi, bc, 64, SCALE, rows)
    assert_close("dQ rows", bf16_to_f64(dQ)[rows[:, 0], rows[:, 1], rows[:, 2]], rq)
    blocks = np.array([[0, 0, 1], [0, 3, 17], [0, 5, 200], [0, 7, w.NQB - 1], [0, 2, 450],
                       [0, 6, 64]], np.int32)
    rk, rv = oracle.sparse_attn_bwd_kv_blocks(x["Q"], x["K"], x["V"], x["dO"], bi, bc, 64, SCALE,
                                              blocks)
    dKh, dVh = bf16_to_f64(dK), bf16_to_f64(dV)
    for n, (b, g, t) in enumerate(blocks):
        assert_close(f"dK block {t}", dKh[b, g, t * 64:(t + 1) * 64], rk[n])
        assert_close(f"dV block {t}", dVh[b, g, t * 64:(t + 1) * 64], rv[n])


def test_backward_is_bitwise_deterministic_at_train_size():
    # Every sum of the backward runs in a fixed order, so repeated calls give
    # identical bits. At this size the dK/dV kernel keeps several Q/dO tiles in
    # flight; a product that read a tile before its load had landed showed up
    # here as dV differing between calls in a few KV blocks.
    w = inputs.WORKLOADS["train_8k_x4"]
    x = inputs.make_inputs(w, with_grad=True)
    rng = np.random.default_rng(2)
    bi, bc = inputs.random_block_lists(rng, w.B, w.Hkv, w.NQB, w.topk)
    Qd, Kd, Vd, dOd = (to_dev_bf16(x[k]) for k in ("Q", "K", "V", "dO"))
    it, ct = torch.from_numpy(bi).cuda(), torch.from_numpy(bc).cuda()
    O, lse = phsa.phsa_sparse_attn_fwd(Qd, Kd, Vd, it, ct)
    ref = [g.clone() for g in phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct)]
    for _ in range(6):
        got = phsa.phsa_sparse_attn_bwd(Qd, Kd, Vd, O, dOd, lse, it, ct)
        for name, a, b in zip(("dQ", "dK", "dV"), ref, got):
            assert torch.equal(a.view(torch.int16), b.view(torch.int16)), f"{name} differs between calls"
    assert phsa.phsa_get_device_status() == 0
