"""Python binding of the PHSA C ABI (``include/phsa.h``).

Argument marshalling only: each function checks tensor dtypes/devices,
allocates outputs with PyTorch when the caller passes none, and calls the
entry point of the same name in ``libphsa.so`` on the current CUDA stream.
Every step of the computation runs in the library's CUDA kernels; there is no
fallback of any kind. If the library cannot be loaded, calls raise.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

BLOCK_SIZE = 64
HEAD_DIM = 128

_lock = threading.Lock()
_lib = None


class PhsaError(RuntimeError):
    """A PHSA entry point returned a non-zero status."""

    def __init__(self, fn: str, code: int):
        self.code = code
        super().__init__(f"{fn} failed: {phsa_status_string(code)} ({code})")


class phsa_shape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("L", ctypes.c_int), ("Hq", ctypes.c_int),
                ("Hkv", ctypes.c_int), ("D", ctypes.c_int), ("block_size", ctypes.c_int)]


class phsa_select_params(ctypes.Structure):
    _fields_ = [("topk", ctypes.c_int), ("n_init", ctypes.c_int), ("n_local", ctypes.c_int),
                ("sm_scale", ctypes.c_float), ("aggregation", ctypes.c_int)]


# PHSA_AGG_* of include/phsa.h: how a unit's query rows are combined per candidate
AGGREGATIONS = {"softmax_sum": 0, "max_logit": 1}


def _params(topk, n_init, n_local, sm_scale, aggregation) -> phsa_select_params:
    if aggregation not in AGGREGATIONS:
        raise ValueError(f"aggregation must be one of {sorted(AGGREGATIONS)}")
    return phsa_select_params(int(topk), int(n_init), int(n_local), float(sm_scale),
                              AGGREGATIONS[aggregation])


def library_path() -> str:
    return _build.LIB


def load():
    """Load ``libphsa.so`` (building it first if it is missing or stale)."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build()
            lib = ctypes.CDLL(path)
            _declare(lib)
            _lib = lib
    return _lib


def _declare(L):
    P, I, F, SZ = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
    L.phsa_build_block_repr.argtypes = [P, P, phsa_shape, F, P, P]
    L.phsa_select_blocks.argtypes = [P, P, phsa_shape, phsa_select_params, P, P, P]
    L.phsa_sparse_attn_fwd.argtypes = [P, P, P, P, P, phsa_shape, I, F, P, P, P]
    L.phsa_sparse_attn_bwd_workspace.argtypes = [phsa_shape, I]
    L.phsa_sparse_attn_bwd_workspace.restype = SZ
    L.phsa_sparse_attn_bwd.argtypes = [P, P, P, P, P, P, P, P, phsa_shape, I, F, P, SZ, P, P, P, P]
    L.phsa_get_device_status.argtypes = [P]
    L.phsa_status_string.argtypes = [I]
    L.phsa_status_string.restype = ctypes.c_char_p
    L.phsa_version.restype = ctypes.c_char_p
    L.phsa_profile_enable.argtypes = [I]
    L.phsa_profile_enable.restype = I
    L.phsa_profile_read.argtypes = [I, ctypes.POINTER(ctypes.c_char_p),
                                    ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int)]
    L.phsa_profile_read.restype = I
    L.phsa_selftest_tcgen05.argtypes = [P, P, P, P, P, P]
    L.phsa_sparse_attn_bwd_noalloc.argtypes = [P, P, P, P, P, P, P, P, phsa_shape, I, F, P, P, P,
                                               P]
    L.phsa_sparse_attn_bwd_noalloc.restype = I
    L.phsa_step_host_workspace.argtypes = [phsa_shape, I]
    L.phsa_step_host_workspace.restype = SZ
    L.phsa_step_host.argtypes = [P, P, P, P, P, phsa_shape, F, phsa_select_params, P, P, P, P, P,
                                 P, P, P, SZ, P, P]
    L.phsa_step_host.restype = I
    L.phsa_step_host_release.argtypes = [P]
    L.phsa_step_host_release.restype = I
    L.phsa_decode_step.argtypes = [P, P, P, P, P, phsa_shape, F, phsa_select_params, P, P, P, P,
                                   P, P]
    L.phsa_decode_step.restype = I
    L.phsa_decode_update_repr.argtypes = [P, P, P, phsa_shape, F, P, P]
    L.phsa_decode_append.argtypes = [P, P, P, P, phsa_shape, P, P, P, P]
    L.phsa_punct_mask.argtypes = [P, ctypes.c_int64, P, I, P, P]
    L.phsa_decode_select.argtypes = [P, P, P, phsa_shape, phsa_select_params, P, P, P]
    L.phsa_decode_attn.argtypes = [P, P, P, P, P, P, phsa_shape, I, F, P, P, P]
    L.phsa_prefill_append.argtypes = [P, P, P, P, I, phsa_shape, F, P, P, P, P, P]
    L.phsa_prefill_append.restype = I
    L.phsa_test_set_select_tc_limit.argtypes = [SZ]
    L.phsa_test_set_select_tc_limit.restype = SZ
    L.phsa_test_set_idx_smem_limit.argtypes = [SZ]
    L.phsa_test_set_idx_smem_limit.restype = SZ
    for fn in ("phsa_decode_update_repr", "phsa_decode_select", "phsa_decode_attn",
               "phsa_decode_append", "phsa_punct_mask",
               "phsa_build_block_repr", "phsa_select_blocks", "phsa_sparse_attn_fwd",
               "phsa_sparse_attn_bwd", "phsa_get_device_status", "phsa_selftest_tcgen05"):
        getattr(L, fn).restype = I


def _ptr(t):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _check(t, name, dtype, ndim=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got {tuple(t.shape)}")


def _check_host(t, name, dtypes, ndim=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.is_cuda:
        raise ValueError(f"{name} must be a host (CPU) tensor")
    if t.dtype not in dtypes:
        raise TypeError(f"{name} must be one of {dtypes}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got {tuple(t.shape)}")


def make_shape(B, L, Hq, Hkv, D=HEAD_DIM, block_size=BLOCK_SIZE) -> phsa_shape:
    return phsa_shape(int(B), int(L), int(Hq), int(Hkv), int(D), int(block_size))


def _raise(fn, rc):
    if rc != 0:
        raise PhsaError(fn, rc)


def phsa_status_string(code: int) -> str:
    return load().phsa_status_string(int(code)).decode()


def phsa_version() -> str:
    return load().phsa_version().decode()


def phsa_build_block_repr(K, punct_mask, lam: float, Krepr=None, stream=None,
                          block_size: int = BLOCK_SIZE):
    """Stage (a): representative keys [B, Hkv, L // m, D] (bf16), m = block_size
    (64; 16 and 32 are accepted too)."""
    _check(K, "K", torch.bfloat16, 4)
    _check(punct_mask, "punct_mask", torch.uint8, 2)
    B, Hkv, L, D = K.shape
    if tuple(punct_mask.shape) != (B, L):
        raise ValueError("punct_mask must be [B, L]")
    T = L // int(block_size)
    if Krepr is None:
        Krepr = torch.empty((B, Hkv, T, D), dtype=torch.bfloat16, device=K.device)
    _check(Krepr, "Krepr", torch.bfloat16, 4)
    rc = load().phsa_build_block_repr(_ptr(K), _ptr(punct_mask),
                                      make_shape(B, L, Hkv, Hkv, D, block_size), float(lam),
                                      _ptr(Krepr), _stream(stream))
    _raise("phsa_build_block_repr", rc)
    return Krepr


def phsa_select_blocks(Q, Krepr, Hkv: int, topk: int, n_init: int = 1, n_local: int = 1,
                       sm_scale: float | None = None, block_idx=None, block_cnt=None,
                       stream=None, aggregation: str = "softmax_sum",
                       block_size: int = BLOCK_SIZE):
    """Stage (b): (block_idx [B, Hkv, NQB, topk] int32, block_cnt [B, Hkv, NQB] int32).
    ``aggregation``: "softmax_sum" (Eq. 8 probabilities summed over the unit's
    rows) or "max_logit" (the largest raw score over the rows)."""
    _check(Q, "Q", torch.bfloat16, 4)
    _check(Krepr, "Krepr", torch.bfloat16, 4)
    B, Hq, L, D = Q.shape
    NQB = -(-L // int(block_size))
    if sm_scale is None:
        sm_scale = D ** -0.5
    if block_idx is None:
        block_idx = torch.empty((B, Hkv, NQB, topk), dtype=torch.int32, device=Q.device)
    if block_cnt is None:
        block_cnt = torch.empty((B, Hkv, NQB), dtype=torch.int32, device=Q.device)
    _check(block_idx, "block_idx", torch.int32, 4)
    _check(block_cnt, "block_cnt", torch.int32, 3)
    p = _params(topk, n_init, n_local, sm_scale, aggregation)
    rc = load().phsa_select_blocks(_ptr(Q), _ptr(Krepr), make_shape(B, L, Hq, Hkv, D, block_size),
                                   p, _ptr(block_idx), _ptr(block_cnt), _stream(stream))
    _raise("phsa_select_blocks", rc)
    return block_idx, block_cnt


def phsa_sparse_attn_fwd(Q, K, V, block_idx, block_cnt, sm_scale: float | None = None, O=None,
                         lse=None, stream=None, block_size: int = BLOCK_SIZE):
    """Stage (c) forward: (O [B, Hq, L, D] bf16, lse [B, Hq, L] fp32)."""
    _check(Q, "Q", torch.bfloat16, 4)
    _check(K, "K", torch.bfloat16, 4)
    _check(V, "V", torch.bfloat16, 4)
    _check(block_idx, "block_idx", torch.int32, 4)
    _check(block_cnt, "block_cnt", torch.int32, 3)
    B, Hq, L, D = Q.shape
    Hkv = K.shape[1]
    topk = block_idx.shape[-1]
    if sm_scale is None:
        sm_scale = D ** -0.5
    if O is None:
        O = torch.empty_like(Q)
    if lse is None:
        lse = torch.empty((B, Hq, L), dtype=torch.float32, device=Q.device)
    _check(O, "O", torch.bfloat16, 4)
    _check(lse, "lse", torch.float32, 3)
    rc = load().phsa_sparse_attn_fwd(_ptr(Q), _ptr(K), _ptr(V), _ptr(block_idx), _ptr(block_cnt),
                                     make_shape(B, L, Hq, Hkv, D, block_size), int(topk),
                                     float(sm_scale), _ptr(O), _ptr(lse), _stream(stream))
    _raise("phsa_sparse_attn_fwd", rc)
    return O, lse


def phsa_sparse_attn_bwd_workspace(B, L, Hq, Hkv, topk, D=HEAD_DIM, block_size=BLOCK_SIZE) -> int:
    return int(load().phsa_sparse_attn_bwd_workspace(make_shape(B, L, Hq, Hkv, D, block_size),
                                                     int(topk)))


def phsa_sparse_attn_bwd(Q, K, V, O, dO, lse, block_idx, block_cnt, sm_scale=None,
                         workspace=None, dQ=None, dK=None, dV=None, stream=None,
                         block_size=BLOCK_SIZE):
    """Stage (c) backward: (dQ, dK, dV) in bf16 (block sizes 16 and 32 for two
    query heads per KV head)."""
    for name, t in (("Q", Q), ("K", K), ("V", V), ("O", O), ("dO", dO)):
        _check(t, name, torch.bfloat16, 4)
    _check(lse, "lse", torch.float32, 3)
    _check(block_idx, "block_idx", torch.int32, 4)
    _check(block_cnt, "block_cnt", torch.int32, 3)
    B, Hq, L, D = Q.shape
    Hkv = K.shape[1]
    topk = block_idx.shape[-1]
    if sm_scale is None:
        sm_scale = D ** -0.5
    ws_bytes = phsa_sparse_attn_bwd_workspace(B, L, Hq, Hkv, topk, D, block_size)
    if workspace is None:
        workspace = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=Q.device)
    _check(workspace, "workspace", torch.uint8, 1)
    dQ = torch.empty_like(Q) if dQ is None else dQ
    dK = torch.empty_like(K) if dK is None else dK
    dV = torch.empty_like(V) if dV is None else dV
    rc = load().phsa_sparse_attn_bwd(
        _ptr(Q), _ptr(K), _ptr(V), _ptr(O), _ptr(dO), _ptr(lse), _ptr(block_idx), _ptr(block_cnt),
        make_shape(B, L, Hq, Hkv, D, block_size), int(topk), float(sm_scale), _ptr(workspace),
        ctypes.c_size_t(workspace.numel()), _ptr(dQ), _ptr(dK), _ptr(dV), _stream(stream))
    _raise("phsa_sparse_attn_bwd", rc)
    return dQ, dK, dV


def phsa_sparse_attn_bwd_noalloc(Q, K, V, O, dO, lse, block_idx, block_cnt, sm_scale=None,
                                 dQ=None, dK=None, dV=None, stream=None):
    """The backward pass without any workspace: for callers that cannot allocate
    device memory where they run it. The library's fixed 64 MiB scratch array is
    used instead (shapes needing more are rejected); calls must not overlap on
    the GPU. Output tensors are allocated here only when not passed in."""
    for name, t in (("Q", Q), ("K", K), ("V", V), ("O", O), ("dO", dO)):
        _check(t, name, torch.bfloat16, 4)
    _check(lse, "lse", torch.float32, 3)
    _check(block_idx, "block_idx", torch.int32, 4)
    _check(block_cnt, "block_cnt", torch.int32, 3)
    B, Hq, L, D = Q.shape
    if sm_scale is None:
        sm_scale = D ** -0.5
    dQ = torch.empty_like(Q) if dQ is None else dQ
    dK = torch.empty_like(K) if dK is None else dK
    dV = torch.empty_like(V) if dV is None else dV
    rc = load().phsa_sparse_attn_bwd_noalloc(
        _ptr(Q), _ptr(K), _ptr(V), _ptr(O), _ptr(dO), _ptr(lse), _ptr(block_idx), _ptr(block_cnt),
        make_shape(B, L, Hq, K.shape[1], D), int(block_idx.shape[-1]), float(sm_scale), _ptr(dQ),
        _ptr(dK), _ptr(dV), _stream(stream))
    _raise("phsa_sparse_attn_bwd_noalloc", rc)
    return dQ, dK, dV


def phsa_step_host_workspace(B, L, Hq, Hkv, topk, D=HEAD_DIM) -> int:
    return int(load().phsa_step_host_workspace(make_shape(B, L, Hq, Hkv, D), int(topk)))


def phsa_step_host(Q, K, V, dO, punct_mask, lam: float, topk: int, n_init: int = 1,
                   n_local: int = 1, sm_scale: float | None = None, O=None, lse=None, dQ=None,
                   dK=None, dV=None, block_idx=None, block_cnt=None, workspace=None,
                   done_event=None, stream=None, aggregation: str = "softmax_sum"):
    """One step of the whole path for HOST tensors (preferably pinned): stage (a),
    (b), the forward and the backward for dO, with the copies overlapped with the
    kernels inside the library. Q, K, V, dO: bf16 (or int16 holding bf16 bits) CPU
    tensors [B, H, L, D]; punct_mask uint8 [B, L]. Outputs O, lse, dQ, dK, dV are
    allocated pinned when not passed; block_idx / block_cnt are copied back only
    when passed. workspace: CUDA uint8 tensor of phsa_step_host_workspace() bytes.
    done_event: a torch.cuda.Event the library records when the outputs are in
    host memory (the stream then waits only for the kernels); None makes the
    stream wait for the copies back. Returns (O, lse, dQ, dK, dV)."""
    bf = (torch.bfloat16, torch.int16)
    for name, t in (("Q", Q), ("K", K), ("V", V), ("dO", dO)):
        _check_host(t, name, bf, 4)
    _check_host(punct_mask, "punct_mask", (torch.uint8,), 2)
    B, Hq, L, D = Q.shape
    Hkv = K.shape[1]
    if sm_scale is None:
        sm_scale = D ** -0.5
    pinned = lambda shape, dt: torch.empty(shape, dtype=dt).pin_memory()
    O = pinned(Q.shape, Q.dtype) if O is None else O
    dQ = pinned(Q.shape, Q.dtype) if dQ is None else dQ
    dK = pinned(K.shape, K.dtype) if dK is None else dK
    dV = pinned(K.shape, K.dtype) if dV is None else dV
    lse = pinned((B, Hq, L), torch.float32) if lse is None else lse
    for name, t in (("O", O), ("dQ", dQ), ("dK", dK), ("dV", dV)):
        _check_host(t, name, bf, 4)
    _check_host(lse, "lse", (torch.float32,), 3)
    if block_idx is not None:
        _check_host(block_idx, "block_idx", (torch.int32,), 4)
    if block_cnt is not None:
        _check_host(block_cnt, "block_cnt", (torch.int32,), 3)
    ws_bytes = phsa_step_host_workspace(B, L, Hq, Hkv, topk, D)
    if workspace is None:
        workspace = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device="cuda")
    _check(workspace, "workspace", torch.uint8, 1)
    ev = None
    if done_event is not None:
        done_event.record(stream)  # creates the CUDA event; the library records it again
        ev = ctypes.c_void_p(done_event.cuda_event)
    p = _params(topk, n_init, n_local, sm_scale, aggregation)
    rc = load().phsa_step_host(_ptr(Q), _ptr(K), _ptr(V), _ptr(dO), _ptr(punct_mask),
                               make_shape(B, L, Hq, Hkv, D), float(lam), p, _ptr(O), _ptr(lse),
                               _ptr(dQ), _ptr(dK), _ptr(dV), _ptr(block_idx), _ptr(block_cnt),
                               _ptr(workspace), ctypes.c_size_t(workspace.numel()), ev,
                               _stream(stream))
    _raise("phsa_step_host", rc)
    return O, lse, dQ, dK, dV


def phsa_step_host_release(workspace):
    """Waits for the last phsa_step_host call on `workspace` and drops its events."""
    _raise("phsa_step_host_release", load().phsa_step_host_release(_ptr(workspace)))


def phsa_punct_mask(ids, punct_ids, mask=None, stream=None):
    """Punctuation indicator: mask[i] = 1 if ids[i] is in punct_ids, else 0.
    ids int32 (any shape, contiguous), punct_ids int32 [n_punct <= 4096];
    returns a uint8 mask of ids' shape."""
    _check(ids, "ids", torch.int32)
    _check(punct_ids, "punct_ids", torch.int32, 1)
    if mask is None:
        mask = torch.empty(ids.shape, dtype=torch.uint8, device=ids.device)
    _check(mask, "mask", torch.uint8)
    if mask.numel() != ids.numel():
        raise ValueError("mask must have as many elements as ids")
    rc = load().phsa_punct_mask(_ptr(ids), ids.numel(), _ptr(punct_ids), punct_ids.numel(),
                                _ptr(mask), _stream(stream))
    _raise("phsa_punct_mask", rc)
    return mask


def phsa_decode_append(k_new, v_new, seq_lens, K, V, flag_new=None, punct_mask=None,
                       stream=None):
    """Write the new token of every sequence at row seq_lens[b] - 1 of the
    caches: k_new/v_new [B, Hkv, D] bf16 into K/V [B, Hkv, Lc, D], and, when
    flag_new [B] uint8 is given, its flag into punct_mask [B, Lc]."""
    _check(k_new, "k_new", torch.bfloat16, 3)
    _check(v_new, "v_new", torch.bfloat16, 3)
    _check(seq_lens, "seq_lens", torch.int32, 1)
    _check(K, "K", torch.bfloat16, 4)
    _check(V, "V", torch.bfloat16, 4)
    B, Hkv, Lc, D = K.shape
    if tuple(V.shape) != tuple(K.shape) or tuple(k_new.shape) != (B, Hkv, D) or \
            tuple(v_new.shape) != (B, Hkv, D) or tuple(seq_lens.shape) != (B,):
        raise ValueError("k_new/v_new must be [B, Hkv, D], K/V [B, Hkv, Lc, D], seq_lens [B]")
    if flag_new is not None:
        _check(flag_new, "flag_new", torch.uint8, 1)
        _check(punct_mask, "punct_mask", torch.uint8, 2)
        if tuple(flag_new.shape) != (B,) or tuple(punct_mask.shape) != (B, Lc):
            raise ValueError("flag_new must be [B] and punct_mask [B, Lc]")
    rc = load().phsa_decode_append(_ptr(k_new), _ptr(v_new), _ptr(flag_new), _ptr(seq_lens),
                                   make_shape(B, Lc, Hkv, Hkv, D), _ptr(K), _ptr(V),
                                   _ptr(punct_mask), _stream(stream))
    _raise("phsa_decode_append", rc)
    return K, V


def phsa_prefill_append(k_chunk, v_chunk, seq_lens, K, V, punct_mask, Krepr, lam: float,
                        flag_chunk=None, stream=None, block_size: int = BLOCK_SIZE):
    """Append a chunk of C tokens to every sequence's caches (positions
    seq_lens[b] - C .. seq_lens[b] - 1, seq_lens counting the chunk) and write
    the representative key of every block of m = block_size the chunk
    completes, from the same loads: k_chunk/v_chunk [B, Hkv, C, D] bf16 into
    K/V [B, Hkv, Lc, D], flag_chunk [B, C] uint8 (optional) into punct_mask
    [B, Lc], keys into Krepr [B, Hkv, Lc // m, D]."""
    _check(k_chunk, "k_chunk", torch.bfloat16, 4)
    _check(v_chunk, "v_chunk", torch.bfloat16, 4)
    _check(seq_lens, "seq_lens", torch.int32, 1)
    _check(K, "K", torch.bfloat16, 4)
    _check(V, "V", torch.bfloat16, 4)
    _check(punct_mask, "punct_mask", torch.uint8, 2)
    _check(Krepr, "Krepr", torch.bfloat16, 4)
    B, Hkv, Lc, D = K.shape
    C = k_chunk.shape[2]
    if tuple(V.shape) != tuple(K.shape) or tuple(k_chunk.shape) != (B, Hkv, C, D) or \
            tuple(v_chunk.shape) != (B, Hkv, C, D) or tuple(seq_lens.shape) != (B,) or \
            tuple(punct_mask.shape) != (B, Lc) or \
            tuple(Krepr.shape) != (B, Hkv, Lc // int(block_size), D):
        raise ValueError("k_chunk/v_chunk must be [B, Hkv, C, D], K/V [B, Hkv, Lc, D], "
                         "seq_lens [B], punct_mask [B, Lc], Krepr [B, Hkv, Lc // m, D]")
    if flag_chunk is not None:
        _check(flag_chunk, "flag_chunk", torch.uint8, 2)
        if tuple(flag_chunk.shape) != (B, C):
            raise ValueError("flag_chunk must be [B, C]")
    rc = load().phsa_prefill_append(_ptr(k_chunk), _ptr(v_chunk), _ptr(flag_chunk),
                                    _ptr(seq_lens), int(C),
                                    make_shape(B, Lc, Hkv, Hkv, D, block_size), float(lam),
                                    _ptr(K), _ptr(V), _ptr(punct_mask), _ptr(Krepr),
                                    _stream(stream))
    _raise("phsa_prefill_append", rc)
    return K, V, Krepr


def phsa_decode_update_repr(K, punct_mask, seq_lens, lam: float, Krepr, stream=None,
                            block_size: int = BLOCK_SIZE):
    """Decode: refresh the representative key of every block the new token has
    just filled (a sequence whose length is a positive multiple of m = block_size).
    K [B, Hkv, Lc, D] bf16 cache, punct_mask [B, Lc] uint8, seq_lens [B] int32,
    Krepr [B, Hkv, Lc // m, D] bf16 (updated in place; returned)."""
    _check(K, "K", torch.bfloat16, 4)
    _check(punct_mask, "punct_mask", torch.uint8, 2)
    _check(seq_lens, "seq_lens", torch.int32, 1)
    _check(Krepr, "Krepr", torch.bfloat16, 4)
    B, Hkv, Lc, D = K.shape
    if tuple(punct_mask.shape) != (B, Lc) or tuple(seq_lens.shape) != (B,):
        raise ValueError("punct_mask must be [B, Lc] and seq_lens [B]")
    if tuple(Krepr.shape) != (B, Hkv, Lc // int(block_size), D):
        raise ValueError("Krepr must be [B, Hkv, Lc // m, D]")
    rc = load().phsa_decode_update_repr(_ptr(K), _ptr(punct_mask), _ptr(seq_lens),
                                        make_shape(B, Lc, Hkv, Hkv, D, block_size), float(lam),
                                        _ptr(Krepr), _stream(stream))
    _raise("phsa_decode_update_repr", rc)
    return Krepr


def phsa_decode_select(q, Krepr, seq_lens, Lc: int, topk: int, n_init: int = 1,
                       n_local: int = 1, sm_scale: float | None = None, block_idx=None,
                       block_cnt=None, stream=None, aggregation: str = "softmax_sum",
                       block_size: int = BLOCK_SIZE):
    """Decode selection for the new token of every sequence: q [B, Hq, D] bf16,
    Krepr [B, Hkv, Lc // m, D] (m = block_size); returns (block_idx [B, Hkv, topk],
    block_cnt [B, Hkv])."""
    _check(q, "q", torch.bfloat16, 3)
    _check(Krepr, "Krepr", torch.bfloat16, 4)
    _check(seq_lens, "seq_lens", torch.int32, 1)
    B, Hq, D = q.shape
    Hkv = Krepr.shape[1]
    if sm_scale is None:
        sm_scale = D ** -0.5
    if block_idx is None:
        block_idx = torch.empty((B, Hkv, topk), dtype=torch.int32, device=q.device)
    if block_cnt is None:
        block_cnt = torch.empty((B, Hkv), dtype=torch.int32, device=q.device)
    _check(block_idx, "block_idx", torch.int32, 3)
    _check(block_cnt, "block_cnt", torch.int32, 2)
    p = _params(topk, n_init, n_local, sm_scale, aggregation)
    if tuple(Krepr.shape) != (B, Hkv, Lc // int(block_size), D):
        raise ValueError("Krepr must be [B, Hkv, Lc // m, D]")
    rc = load().phsa_decode_select(_ptr(q), _ptr(Krepr), _ptr(seq_lens),
                                   make_shape(B, Lc, Hq, Hkv, D, block_size), p, _ptr(block_idx),
                                   _ptr(block_cnt), _stream(stream))
    _raise("phsa_decode_select", rc)
    return block_idx, block_cnt


def phsa_decode_attn(q, K, V, block_idx, block_cnt, seq_lens, sm_scale: float | None = None,
                     O=None, lse=None, stream=None, block_size: int = BLOCK_SIZE):
    """Decode attention of the new token over the selected blocks of m =
    block_size keys: (O [B, Hq, D] bf16, lse [B, Hq] fp32)."""
    _check(q, "q", torch.bfloat16, 3)
    _check(K, "K", torch.bfloat16, 4)
    _check(V, "V", torch.bfloat16, 4)
    _check(block_idx, "block_idx", torch.int32, 3)
    _check(block_cnt, "block_cnt", torch.int32, 2)
    _check(seq_lens, "seq_lens", torch.int32, 1)
    B, Hq, D = q.shape
    Hkv, Lc = K.shape[1], K.shape[2]
    if sm_scale is None:
        sm_scale = D ** -0.5
    O = torch.empty_like(q) if O is None else O
    lse = torch.empty((B, Hq), dtype=torch.float32, device=q.device) if lse is None else lse
    _check(O, "O", torch.bfloat16, 3)
    _check(lse, "lse", torch.float32, 2)
    rc = load().phsa_decode_attn(_ptr(q), _ptr(K), _ptr(V), _ptr(block_idx), _ptr(block_cnt),
                                 _ptr(seq_lens), make_shape(B, Lc, Hq, Hkv, D, block_size),
                                 int(block_idx.shape[-1]), float(sm_scale), _ptr(O), _ptr(lse),
                                 _stream(stream))
    _raise("phsa_decode_attn", rc)
    return O, lse


def phsa_decode_step(q, K, V, punct_mask, seq_lens, lam: float, Krepr, topk: int,
                     n_init: int = 1, n_local: int = 1, sm_scale: float | None = None,
                     block_idx=None, block_cnt=None, O=None, lse=None, stream=None,
                     aggregation: str = "softmax_sum", block_size: int = BLOCK_SIZE):
    """One decode step in two launches (selection; attention fused with the
    refresh of the blocks the new tokens have just filled). q [B, Hq, D], K/V
    [B, Hkv, Lc, D] bf16 caches, punct_mask [B, Lc] uint8, seq_lens [B] int32,
    Krepr [B, Hkv, Lc // m, D] (m = block_size; read, and updated in place).
    Returns (block_idx, block_cnt, O, lse)."""
    _check(q, "q", torch.bfloat16, 3)
    _check(K, "K", torch.bfloat16, 4)
    _check(V, "V", torch.bfloat16, 4)
    _check(punct_mask, "punct_mask", torch.uint8, 2)
    _check(seq_lens, "seq_lens", torch.int32, 1)
    _check(Krepr, "Krepr", torch.bfloat16, 4)
    B, Hq, D = q.shape
    Hkv, Lc = K.shape[1], K.shape[2]
    if sm_scale is None:
        sm_scale = D ** -0.5
    if block_idx is None:
        block_idx = torch.empty((B, Hkv, topk), dtype=torch.int32, device=q.device)
    if block_cnt is None:
        block_cnt = torch.empty((B, Hkv), dtype=torch.int32, device=q.device)
    if O is None:
        O = torch.empty_like(q)
    if lse is None:
        lse = torch.empty((B, Hq), dtype=torch.float32, device=q.device)
    if tuple(Krepr.shape) != (B, Hkv, Lc // int(block_size), D):
        raise ValueError("Krepr must be [B, Hkv, Lc // m, D]")
    p = _params(topk, n_init, n_local, sm_scale, aggregation)
    rc = load().phsa_decode_step(_ptr(q), _ptr(K), _ptr(V), _ptr(punct_mask), _ptr(seq_lens),
                                 make_shape(B, Lc, Hq, Hkv, D, block_size), float(lam), p,
                                 _ptr(Krepr), _ptr(block_idx), _ptr(block_cnt), _ptr(O),
                                 _ptr(lse),
                                 _stream(stream))
    _raise("phsa_decode_step", rc)
    return block_idx, block_cnt, O, lse


def phsa_test_set_select_tc_limit(nbytes: int) -> int:
    """Testing hook: the shared-memory switch point between the tensor-core and
    the warp-level selection of GQA pairs at block sizes 16 and 32 (0 restores
    the default of 227 KB). Returns the previous value."""
    return int(load().phsa_test_set_select_tc_limit(int(nbytes)))


def phsa_test_set_idx_smem_limit(nbytes: int) -> int:
    """Testing hook: a nonzero value makes the backward transpose the block
    lists in one launch at every block size while a (b, g)'s bitmap fits in
    min(nbytes, 160 KB) of shared memory, else in two launches; 0 restores the
    default (one launch at block size 64 while it fits in 160 KB, two launches
    otherwise). Returns the previous setting."""
    return int(load().phsa_test_set_idx_smem_limit(int(nbytes)))


def phsa_get_device_status(stream=None) -> int:
    """Synchronise the stream; return and clear the device status word."""
    return int(load().phsa_get_device_status(_stream(stream)))


def phsa_profile_enable(on: bool) -> bool:
    """Turn per-kernel event timing on or off; returns the previous setting."""
    return bool(load().phsa_profile_enable(1 if on else 0))


def phsa_profile_read() -> dict:
    """{kernel name: (total ms, launches)} since the last read; clears the records."""
    n = 32
    names = (ctypes.c_char_p * n)()
    ms = (ctypes.c_double * n)()
    cnt = (ctypes.c_int * n)()
    k = load().phsa_profile_read(n, names, ms, cnt)
    if k < 0:
        raise PhsaError("phsa_profile_read", k)
    return {names[i].decode(): (float(ms[i]), int(cnt[i])) for i in range(k)}


def phsa_selftest_tcgen05(A, B, V, stream=None):
    """Diagnostic: (S = A B^T, O = bf16(S) V) computed on the tensor cores, fp32."""
    _check(A, "A", torch.bfloat16, 2)
    _check(B, "B", torch.bfloat16, 2)
    _check(V, "V", torch.bfloat16, 2)
    if tuple(A.shape) != (128, 128) or tuple(B.shape) != (64, 128) or tuple(V.shape) != (64, 128):
        raise ValueError("A must be [128,128], B and V [64,128]")
    S = torch.empty((128, 64), dtype=torch.float32, device=A.device)
    O = torch.empty((128, 128), dtype=torch.float32, device=A.device)
    rc = load().phsa_selftest_tcgen05(_ptr(A), _ptr(B), _ptr(V), _ptr(S), _ptr(O), _stream(stream))
    _raise("phsa_selftest_tcgen05", rc)
    return S, O


def phsa_forward(Q, K, V, punct_mask, lam: float, topk: int, n_init: int = 1, n_local: int = 1,
                 sm_scale: float | None = None, stream=None, aggregation: str = "softmax_sum",
                 block_size: int = BLOCK_SIZE):
    """The whole forward hot path: (a) -> (b) -> (c). Returns (O, lse, block_idx, block_cnt, Krepr)."""
    Krepr = phsa_build_block_repr(K, punct_mask, lam, stream=stream, block_size=block_size)
    idx, cnt = phsa_select_blocks(Q, Krepr, K.shape[1], topk, n_init, n_local, sm_scale,
                                  stream=stream, aggregation=aggregation, block_size=block_size)
    O, lse = phsa_sparse_attn_fwd(Q, K, V, idx, cnt, sm_scale, stream=stream,
                                  block_size=block_size)
    return O, lse, idx, cnt, Krepr
