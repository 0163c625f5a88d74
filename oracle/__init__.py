"""PHSA CPU oracle -- test infrastructure only.

Python access to ``phsa_oracle.c``, a plain fp64 restatement of the paper's
Section 3 and Algorithm 1. Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package; the product library
never does. Nothing here is shared with the CUDA path.

bf16 tensors are passed as numpy ``uint16`` bit patterns.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "phsa_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "libphsa_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, IEEE semantics kept: no fast-math)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
            "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            _lib = ctypes.CDLL(build())
            _declare(_lib)
    return _lib


def _declare(L):
    P = ctypes.c_void_p
    i32, i64, f64 = ctypes.c_int, ctypes.c_int64, ctypes.c_double
    L.phsa_oracle_set_threads.argtypes = [i32]
    L.phsa_oracle_max_threads.restype = i32
    L.phsa_oracle_bf16_to_f64_array.argtypes = [P, i64, P]
    L.phsa_oracle_f64_to_bf16_array.argtypes = [P, i64, P]
    L.phsa_oracle_punct_mask.argtypes = [P, i64, P, i32, P]
    L.phsa_oracle_block_repr.argtypes = [P, P, i32, i32, i32, i32, i32, f64, P, P]
    L.phsa_oracle_select_blocks.argtypes = [P, P, i32, i32, i32, i32, i32, i32, i32, i32,
                                            i32, f64, i32, P, P, P]
    L.phsa_oracle_select_blocks.restype = i32
    L.phsa_oracle_select_units.argtypes = [P, P, i32, i32, i32, i32, i32, i32, i32, i32, i32,
                                           f64, i32, P, i64, P, P, P]
    L.phsa_oracle_select_units.restype = i32
    L.phsa_oracle_sparse_attn_bwd_dq_rows.argtypes = [P, P, P, P, P, P, i32, i32, i32, i32, i32,
                                                      i32, i32, f64, P, i64, P]
    L.phsa_oracle_sparse_attn_bwd_kv_blocks.argtypes = [P, P, P, P, P, P, i32, i32, i32, i32,
                                                        i32, i32, i32, f64, P, i64, P, P]
    L.phsa_oracle_sparse_attn_rows.argtypes = [P, P, P, P, P, i32, i32, i32, i32, i32, i32,
                                               i32, f64, P, i64, P, P]
    L.phsa_oracle_sparse_attn_fwd.argtypes = [P, P, P, P, P, i32, i32, i32, i32, i32, i32,
                                              i32, f64, P, P]
    L.phsa_oracle_sparse_attn_bwd.argtypes = [P, P, P, P, P, P, i32, i32, i32, i32, i32,
                                              i32, i32, f64, P, P, P]
    L.phsa_oracle_dense_causal.argtypes = [P, P, P, i32, i32, i32, i32, i32, f64, P, P]
    L.phsa_oracle_decode_select.argtypes = [P, P, P, i32, i32, i32, i32, i32, i32, i32, i32,
                                            i32, f64, i32, P, P, P]
    L.phsa_oracle_decode_select.restype = i32
    L.phsa_oracle_decode_attn.argtypes = [P, P, P, P, P, P, i32, i32, i32, i32, i32, i32, i32,
                                          f64, P, P]


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"], "oracle inputs must be C-contiguous"
    return a.ctypes.data_as(ctypes.c_void_p)


def _u16(a):
    return np.ascontiguousarray(a, dtype=np.uint16)


def _i32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


def set_threads(n: int) -> None:
    lib().phsa_oracle_set_threads(int(n))


def max_threads() -> int:
    return int(lib().phsa_oracle_max_threads())


def bf16_to_f64(h: np.ndarray) -> np.ndarray:
    h = _u16(h)
    out = np.empty(h.shape, dtype=np.float64)
    lib().phsa_oracle_bf16_to_f64_array(_p(h), h.size, _p(out))
    return out


def f64_to_bf16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty(x.shape, dtype=np.uint16)
    lib().phsa_oracle_f64_to_bf16_array(_p(x), x.size, _p(out))
    return out


def punct_mask(ids: np.ndarray, punct_ids) -> np.ndarray:
    """Eq. 4-5 indicator I(x in P) for every token id."""
    ids = _i32(ids)
    pset = _i32(np.asarray(punct_ids))
    out = np.empty(ids.shape, dtype=np.uint8)
    lib().phsa_oracle_punct_mask(_p(ids), ids.size, _p(pset), pset.size, _p(out))
    return out


def block_repr(K, mask, block_size: int, lam: float, want_f64: bool = False):
    """Eq. 6-8: Krepr [B,Hkv,T,D] as bf16 bits (and fp64 values if asked)."""
    K = _u16(K)
    mask = np.ascontiguousarray(mask, dtype=np.uint8)
    B, Hkv, L, D = K.shape
    T = L // block_size
    out = np.empty((B, Hkv, T, D), dtype=np.uint16)
    out64 = np.empty((B, Hkv, T, D), dtype=np.float64) if want_f64 else None
    lib().phsa_oracle_block_repr(_p(K), _p(mask), B, Hkv, L, D, block_size, float(lam),
                                 _p(out), _p(out64) if want_f64 else None)
    return (out, out64) if want_f64 else out


AGGREGATIONS = {"softmax_sum": 0, "max_logit": 1}


def _agg_mode(aggregation: str) -> int:
    if aggregation not in AGGREGATIONS:
        raise ValueError(f"aggregation must be one of {sorted(AGGREGATIONS)}")
    return AGGREGATIONS[aggregation]


def select_blocks(Q, Krepr, L: int, block_size: int, topk: int, n_init: int, n_local: int,
                  sm_scale: float, want_agg: bool = False, aggregation: str = "softmax_sum"):
    """Algorithm 1 step 3 per (query block, KV head).

    ``aggregation``: "softmax_sum" (the group's rows' softmax probabilities
    summed, Eq. 8) or "max_logit" (the largest raw score over the rows).
    Returns (block_idx [B,Hkv,NQB,topk], block_cnt [B,Hkv,NQB]) and, if
    ``want_agg``, the aggregates A [B,Hkv,NQB,T] (NaN where not scored).
    """
    Q = _u16(Q)
    Krepr = _u16(Krepr)
    B, Hq, Lq, D = Q.shape
    assert Lq == L
    Hkv = Krepr.shape[1]
    T = L // block_size
    NQB = -(-L // block_size)
    idx = np.empty((B, Hkv, NQB, topk), dtype=np.int32)
    cnt = np.empty((B, Hkv, NQB), dtype=np.int32)
    agg = np.empty((B, Hkv, NQB, max(T, 1)), dtype=np.float64) if want_agg else None
    rc = lib().phsa_oracle_select_blocks(_p(Q), _p(Krepr), B, Hq, Hkv, L, D, block_size,
                                         topk, n_init, n_local, float(sm_scale),
                                         _agg_mode(aggregation), _p(idx),
                                         _p(cnt), _p(agg) if want_agg else None)
    if rc != 0:
        raise ValueError("topk is smaller than the forced block count")
    return (idx, cnt, agg) if want_agg else (idx, cnt)


def select_units(Q, Krepr, L: int, block_size: int, topk: int, n_init: int, n_local: int,
                 sm_scale: float, units, aggregation: str = "softmax_sum"):
    """Selection for a list of flat units u = (b*Hkv + g)*NQB + qb only.

    Returns (idx [n, topk], cnt [n], agg [n, T]).
    """
    Q = _u16(Q)
    Krepr = _u16(Krepr)
    B, Hq, Lq, D = Q.shape
    assert Lq == L
    Hkv = Krepr.shape[1]
    T = L // block_size
    units = np.ascontiguousarray(np.asarray(units, dtype=np.int64).ravel())
    n = units.size
    idx = np.empty((n, topk), dtype=np.int32)
    cnt = np.empty((n,), dtype=np.int32)
    agg = np.empty((n, max(T, 1)), dtype=np.float64)
    rc = lib().phsa_oracle_select_units(_p(Q), _p(Krepr), B, Hq, Hkv, L, D, block_size, topk,
                                        n_init, n_local, float(sm_scale), _agg_mode(aggregation),
                                        _p(units), n, _p(idx),
                                        _p(cnt), _p(agg))
    if rc != 0:
        raise ValueError("topk is smaller than the forced block count")
    return idx, cnt, agg


def sparse_attn_bwd_dq_rows(Q, K, V, dO, block_idx, block_cnt, block_size: int,
                            sm_scale: float, rows):
    """dQ in fp64 for the listed rows (b, h, i) only: [n, D]."""
    Q, K, V, dO = _u16(Q), _u16(K), _u16(V), _u16(dO)
    block_idx, block_cnt = _i32(block_idx), _i32(block_cnt)
    rows = _i32(rows).reshape(-1, 3)
    B, Hq, L, D = Q.shape
    out = np.empty((rows.shape[0], D), dtype=np.float64)
    lib().phsa_oracle_sparse_attn_bwd_dq_rows(_p(Q), _p(K), _p(V), _p(dO), _p(block_idx),
                                              _p(block_cnt), B, Hq, K.shape[1], L, D, block_size,
                                              block_idx.shape[-1], float(sm_scale), _p(rows),
                                              rows.shape[0], _p(out))
    return out


def sparse_attn_bwd_kv_blocks(Q, K, V, dO, block_idx, block_cnt, block_size: int,
                              sm_scale: float, blocks):
    """dK, dV in fp64 for every key of the listed KV blocks (b, g, t): [n, m, D] each."""
    Q, K, V, dO = _u16(Q), _u16(K), _u16(V), _u16(dO)
    block_idx, block_cnt = _i32(block_idx), _i32(block_cnt)
    blocks = _i32(blocks).reshape(-1, 3)
    B, Hq, L, D = Q.shape
    n = blocks.shape[0]
    dK = np.empty((n, block_size, D), dtype=np.float64)
    dV = np.empty((n, block_size, D), dtype=np.float64)
    lib().phsa_oracle_sparse_attn_bwd_kv_blocks(_p(Q), _p(K), _p(V), _p(dO), _p(block_idx),
                                                _p(block_cnt), B, Hq, K.shape[1], L, D,
                                                block_size, block_idx.shape[-1], float(sm_scale),
                                                _p(blocks), n, _p(dK), _p(dV))
    return dK, dV


def sparse_attn_fwd(Q, K, V, block_idx, block_cnt, block_size: int, sm_scale: float):
    """Eq. 10-11 over the selected blocks: O [B,Hq,L,D] fp64, lse [B,Hq,L] fp64."""
    Q, K, V = _u16(Q), _u16(K), _u16(V)
    block_idx, block_cnt = _i32(block_idx), _i32(block_cnt)
    B, Hq, L, D = Q.shape
    Hkv = K.shape[1]
    topk = block_idx.shape[-1]
    O = np.empty((B, Hq, L, D), dtype=np.float64)
    lse = np.empty((B, Hq, L), dtype=np.float64)
    lib().phsa_oracle_sparse_attn_fwd(_p(Q), _p(K), _p(V), _p(block_idx), _p(block_cnt), B,
                                      Hq, Hkv, L, D, block_size, topk, float(sm_scale),
                                      _p(O), _p(lse))
    return O, lse


def sparse_attn_rows(Q, K, V, block_idx, block_cnt, block_size: int, sm_scale: float, rows):
    """Forward for selected rows only; rows is an int array [n, 3] of (b, h, i)."""
    Q, K, V = _u16(Q), _u16(K), _u16(V)
    block_idx, block_cnt = _i32(block_idx), _i32(block_cnt)
    rows = _i32(rows).reshape(-1, 3)
    B, Hq, L, D = Q.shape
    Hkv = K.shape[1]
    topk = block_idx.shape[-1]
    O = np.empty((rows.shape[0], D), dtype=np.float64)
    lse = np.empty((rows.shape[0],), dtype=np.float64)
    lib().phsa_oracle_sparse_attn_rows(_p(Q), _p(K), _p(V), _p(block_idx), _p(block_cnt), B,
                                       Hq, Hkv, L, D, block_size, topk, float(sm_scale),
                                       _p(rows), rows.shape[0], _p(O), _p(lse))
    return O, lse


def sparse_attn_bwd(Q, K, V, dO, block_idx, block_cnt, block_size: int, sm_scale: float):
    """Gradients (dQ, dK, dV) in fp64 of sum(O * dO) for the sparse attention."""
    Q, K, V, dO = _u16(Q), _u16(K), _u16(V), _u16(dO)
    block_idx, block_cnt = _i32(block_idx), _i32(block_cnt)
    B, Hq, L, D = Q.shape
    Hkv = K.shape[1]
    topk = block_idx.shape[-1]
    dQ = np.empty((B, Hq, L, D), dtype=np.float64)
    dK = np.empty((B, Hkv, L, D), dtype=np.float64)
    dV = np.empty((B, Hkv, L, D), dtype=np.float64)
    lib().phsa_oracle_sparse_attn_bwd(_p(Q), _p(K), _p(V), _p(dO), _p(block_idx),
                                      _p(block_cnt), B, Hq, Hkv, L, D, block_size, topk,
                                      float(sm_scale), _p(dQ), _p(dK), _p(dV))
    return dQ, dK, dV


def dense_causal(Q, K, V, sm_scale: float):
    """Eq. 1-2: dense causal attention, O and lse in fp64."""
    Q, K, V = _u16(Q), _u16(K), _u16(V)
    B, Hq, L, D = Q.shape
    Hkv = K.shape[1]
    O = np.empty((B, Hq, L, D), dtype=np.float64)
    lse = np.empty((B, Hq, L), dtype=np.float64)
    lib().phsa_oracle_dense_causal(_p(Q), _p(K), _p(V), B, Hq, Hkv, L, D, float(sm_scale),
                                   _p(O), _p(lse))
    return O, lse


def decode_select(q, Krepr, lens, Lc: int, block_size: int, topk: int, n_init: int,
                  n_local: int, sm_scale: float, want_agg: bool = False,
                  aggregation: str = "softmax_sum"):
    """Selection for one new token per sequence (the token at lens[b] - 1).

    q [B,Hq,D], Krepr [B,Hkv,Lc/m,D] (full blocks valid). Returns (block_idx
    [B,Hkv,topk], block_cnt [B,Hkv]) and, if ``want_agg``, A [B,Hkv,Lc/m].
    """
    q, Krepr, lens = _u16(q), _u16(Krepr), _i32(lens)
    B, Hq, D = q.shape
    Hkv = Krepr.shape[1]
    Tc = Lc // block_size
    assert Krepr.shape[2] == Tc and lens.shape == (B,)
    idx = np.empty((B, Hkv, topk), dtype=np.int32)
    cnt = np.empty((B, Hkv), dtype=np.int32)
    agg = np.empty((B, Hkv, max(Tc, 1)), dtype=np.float64) if want_agg else None
    rc = lib().phsa_oracle_decode_select(_p(q), _p(Krepr), _p(lens), B, Hq, Hkv, Lc, D,
                                         block_size, topk, n_init, n_local, float(sm_scale),
                                         _agg_mode(aggregation), _p(idx), _p(cnt),
                                         _p(agg) if want_agg else None)
    if rc != 0:
        raise ValueError("topk is smaller than the forced block count, or a length exceeds Lc")
    return (idx, cnt, agg) if want_agg else (idx, cnt)


def decode_attn(q, K, V, block_idx, block_cnt, lens, block_size: int, sm_scale: float):
    """Attention of each sequence's new token over its selected blocks.

    q [B,Hq,D], K/V [B,Hkv,Lc,D]; returns O [B,Hq,D] and lse [B,Hq] in fp64.
    """
    q, K, V = _u16(q), _u16(K), _u16(V)
    block_idx, block_cnt, lens = _i32(block_idx), _i32(block_cnt), _i32(lens)
    B, Hq, D = q.shape
    Hkv, Lc = K.shape[1], K.shape[2]
    topk = block_idx.shape[-1]
    O = np.empty((B, Hq, D), dtype=np.float64)
    lse = np.empty((B, Hq), dtype=np.float64)
    lib().phsa_oracle_decode_attn(_p(q), _p(K), _p(V), _p(block_idx), _p(block_cnt), _p(lens),
                                  B, Hq, Hkv, Lc, D, block_size, topk, float(sm_scale), _p(O),
                                  _p(lse))
    return O, lse


def forward(Q, K, V, mask, block_size: int, lam: float, topk: int, n_init: int,
            n_local: int, sm_scale: float):
    """Whole forward path (Algorithm 1): repr -> selection -> sparse attention."""
    Krepr = block_repr(K, mask, block_size, lam)
    L = Q.shape[2]
    idx, cnt = select_blocks(Q, Krepr, L, block_size, topk, n_init, n_local, sm_scale)
    O, lse = sparse_attn_fwd(Q, K, V, idx, cnt, block_size, sm_scale)
    return Krepr, idx, cnt, O, lse
