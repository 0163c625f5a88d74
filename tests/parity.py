"""Comparison helpers for the GPU-vs-oracle parity tests.

Tolerances (bf16 inputs, fp32 accumulation on the GPU, fp64 in the oracle):
  * representative keys: at most 1 bf16 ulp from the oracle's rounded value;
  * selected block indices: bit-exact, except candidates whose oracle
    aggregate A lies within SELECT_BAND of the selection boundary (the k-th
    chosen / first unchosen value), which are excluded and counted;
  * attention outputs and gradients: max-abs <= 2e-2 and relative L2 <= 1e-2;
  * log-sum-exp: max-abs <= 1e-3 (natural log).
"""
from __future__ import annotations

import numpy as np
import torch

MAX_ABS = 2e-2
REL_L2 = 1e-2
LSE_ABS = 1e-3
SELECT_BAND = 1e-3


def to_dev_bf16(x_bits: np.ndarray, device="cuda"):
    """uint16 bf16 bit patterns -> CUDA bf16 tensor (bit-exact)."""
    t = torch.from_numpy(np.ascontiguousarray(x_bits).view(np.int16))
    return t.to(device).view(torch.bfloat16)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def bf16_to_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def ulp_distance(a_bits: np.ndarray, b_bits: np.ndarray) -> np.ndarray:
    """Distance in bf16 ulps between two bit patterns (sign-magnitude order)."""
    def ordered(x):
        x = x.astype(np.int32)
        mag = x & 0x7FFF
        return np.where(x & 0x8000, -mag, mag)
    return np.abs(ordered(a_bits) - ordered(b_bits))


def assert_close(name, got: np.ndarray, ref: np.ndarray, max_abs=MAX_ABS, rel_l2=REL_L2):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{name}: non-finite values"
    err = np.abs(got - ref)
    mae = float(err.max()) if err.size else 0.0
    den = float(np.linalg.norm(ref))
    rl2 = float(np.linalg.norm(got - ref) / den) if den > 0 else float(np.linalg.norm(got))
    assert mae <= max_abs, f"{name}: max-abs {mae:.3e} > {max_abs}"
    assert rl2 <= rel_l2, f"{name}: rel-L2 {rl2:.3e} > {rel_l2}"
    return mae, rl2


def compare_selection(g_idx, g_cnt, o_idx, o_cnt, o_agg, band=SELECT_BAND):
    """Compare GPU and oracle selections unit by unit.

    ``*_idx`` [U, topk], ``*_cnt`` [U], ``o_agg`` [U, T] (NaN where not scored).
    Returns (n_bad_units, n_excluded_candidates, n_units_differing, messages):
    bad units differ outside the ambiguity band; excluded candidates are those
    inside the band (reported, never compared); differing units are units whose
    GPU and oracle sets differ only inside the band.
    """
    g_idx = np.asarray(g_idx).reshape(len(g_cnt.reshape(-1)), -1)
    o_idx = np.asarray(o_idx).reshape(g_idx.shape)
    g_cnt = np.asarray(g_cnt).reshape(-1)
    o_cnt = np.asarray(o_cnt).reshape(-1)
    o_agg = np.asarray(o_agg).reshape(len(o_cnt), -1)
    bad, excluded, differ, msgs = 0, 0, 0, []
    for u in range(len(o_cnt)):
        if g_cnt[u] != o_cnt[u]:
            bad += 1
            msgs.append(f"unit {u}: count {g_cnt[u]} vs {o_cnt[u]}")
            continue
        n = o_cnt[u]
        gs, os_ = set(g_idx[u, :n].tolist()), set(o_idx[u, :n].tolist())
        if not np.all(g_idx[u, n:] == -1) or not np.all(np.diff(g_idx[u, :n]) > 0):
            bad += 1
            msgs.append(f"unit {u}: malformed list {g_idx[u].tolist()}")
            continue
        A = o_agg[u]
        scored = np.nonzero(np.isfinite(A))[0]
        # A candidate is ambiguous when its aggregate is within `band` of the other
        # side of the selection boundary: a chosen t with A_t - max(unchosen) <= band,
        # or an unchosen t with min(chosen) - A_t <= band. Only those may differ.
        sel = [t for t in scored if t in os_]
        uns = [t for t in scored if t not in os_]
        hi = A[sel].min() if sel else np.inf
        lo = A[uns].max() if uns else -np.inf
        amb = {t for t in sel if A[t] - lo <= band} | {t for t in uns if hi - A[t] <= band}
        excluded += len(amb)
        diff = gs ^ os_
        if diff:
            differ += 1
        if not diff <= amb:
            bad += 1
            msgs.append(f"unit {u}: gpu {sorted(gs)} vs oracle {sorted(os_)}; "
                        f"boundary gap {hi - lo:.3e}")
    return bad, excluded, differ, msgs
