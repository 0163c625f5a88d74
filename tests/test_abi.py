"""The C-ABI library builds, loads and exports every entry point its header declares.

CPU only: nothing here launches a kernel.
"""
import ctypes
import os
import re

import pytest

from paper_2601_02819_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            src = open(os.path.join(ROOT, "include", fn)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(phsa_[a-z0-9_]+)\s*\(", src))
    return sorted(names)


@pytest.fixture(scope="module")
def lib():
    return ctypes.CDLL(libbuild.build())


def test_header_declares_the_hot_path():
    names = declared_functions()
    for n in ("phsa_build_block_repr", "phsa_select_blocks", "phsa_sparse_attn_fwd",
              "phsa_sparse_attn_bwd", "phsa_sparse_attn_bwd_workspace", "phsa_get_device_status",
              "phsa_decode_update_repr", "phsa_decode_select", "phsa_decode_attn"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    for n in declared_functions():
        assert hasattr(lib, n), n


def test_status_strings_and_version(lib):
    lib.phsa_status_string.restype = ctypes.c_char_p
    lib.phsa_version.restype = ctypes.c_char_p
    assert lib.phsa_status_string(0) == b"PHSA_OK"
    assert b"UNSUPPORTED" in lib.phsa_status_string(-2)
    assert lib.phsa_version().count(b".") == 2


def test_host_validation_needs_no_gpu(lib):
    # Shape and parameter checks run before any CUDA call, so they answer on a CPU machine.
    from paper_2601_02819_gb300.phsa import phsa_shape, phsa_select_params
    lib.phsa_build_block_repr.argtypes = [ctypes.c_void_p, ctypes.c_void_p, phsa_shape,
                                          ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p]
    lib.phsa_select_blocks.argtypes = [ctypes.c_void_p, ctypes.c_void_p, phsa_shape,
                                       phsa_select_params, ctypes.c_void_p, ctypes.c_void_p,
                                       ctypes.c_void_p]
    lib.phsa_sparse_attn_bwd_workspace.argtypes = [phsa_shape, ctypes.c_int]
    lib.phsa_sparse_attn_bwd_workspace.restype = ctypes.c_size_t
    ok = phsa_shape(1, 4096, 16, 8, 128, 64)
    assert lib.phsa_build_block_repr(None, None, phsa_shape(1, 4096, 16, 8, 64, 64), 0.5, None,
                                     None) == -2  # D = 64 unsupported
    for bs in (16, 32):  # the prefill forward calls take m = 16 and 32: past the block
        # size check, a null pointer is what they reject
        assert lib.phsa_build_block_repr(None, None, phsa_shape(1, 4096, 16, 8, 128, bs), 0.5,
                                         None, None) == -1
        assert lib.phsa_select_blocks(None, None, phsa_shape(1, 4096, 16, 8, 128, bs),
                                      phsa_select_params(8, 1, 1, 0.088), None, None, None) == -1
        # the backward takes m = 16 and 32 for two query heads per KV head only
        assert lib.phsa_sparse_attn_bwd_workspace(phsa_shape(1, 4096, 16, 8, 128, bs), 14) > 0
        assert lib.phsa_sparse_attn_bwd_workspace(phsa_shape(1, 4096, 8, 8, 128, bs), 14) == 0
    for bs in (8, 48, 128):
        assert lib.phsa_build_block_repr(None, None, phsa_shape(1, 4096, 16, 8, 128, bs), 0.5,
                                         None, None) == -2  # other block sizes unsupported
    assert lib.phsa_build_block_repr(None, None, phsa_shape(1, 4096, 12, 8, 128, 64), 0.5, None,
                                     None) == -1  # Hq not a multiple of Hkv
    assert lib.phsa_build_block_repr(None, None, ok, 1.5, None, None) == -1  # lambda > 1
    assert lib.phsa_build_block_repr(None, None, ok, 0.5, None, None) == -1  # null pointers
    p = phsa_select_params(2, 1, 2, 0.088)  # topk < n_init + n_local
    assert lib.phsa_select_blocks(None, None, ok, p, None, None, None) == -1
    p = phsa_select_params(8, 1, 0, 0.088)  # n_local must be >= 1
    assert lib.phsa_select_blocks(None, None, ok, p, None, None, None) == -1
    p = phsa_select_params(8, 1, 1, 0.088, 2)  # no such aggregation rule
    assert lib.phsa_select_blocks(None, None, ok, p, None, None, None) == -1
    assert lib.phsa_sparse_attn_bwd_workspace(ok, 14) > 0
    assert lib.phsa_sparse_attn_bwd_workspace(phsa_shape(1, 4096, 16, 8, 96, 64), 14) == 0


def test_host_step_validation_needs_no_gpu(lib):
    # The host-buffer step checks its arguments and workspace before any CUDA call.
    from paper_2601_02819_gb300.phsa import phsa_shape, phsa_select_params
    P = ctypes.c_void_p
    lib.phsa_step_host_workspace.argtypes = [phsa_shape, ctypes.c_int]
    lib.phsa_step_host_workspace.restype = ctypes.c_size_t
    lib.phsa_step_host.argtypes = [P, P, P, P, P, phsa_shape, ctypes.c_float, phsa_select_params,
                                   P, P, P, P, P, P, P, P, ctypes.c_size_t, P, P]
    ok = phsa_shape(1, 4096, 16, 8, 128, 64)
    ws = lib.phsa_step_host_workspace(ok, 14)
    # device copies of Q, dO, O, dQ (16 MB each) and K, V, dK, dV (8 MB each) alone
    assert ws > 4 * 16 * 2**20 + 4 * 8 * 2**20
    assert ws >= lib.phsa_sparse_attn_bwd_workspace(ok, 14)
    assert lib.phsa_step_host_workspace(phsa_shape(1, 4096, 16, 8, 96, 64), 14) == 0
    p = phsa_select_params(14, 1, 1, 0.088)
    dummy = ctypes.c_void_p(256)  # never dereferenced: every case fails validation first
    args = [dummy] * 5
    assert lib.phsa_step_host(*args, ok, 1.5, p, *([None] * 7), dummy, ws, None, None) == -1
    assert lib.phsa_step_host(*args, ok, 0.5, phsa_select_params(2, 1, 2, 0.088),
                              *([None] * 7), dummy, ws, None, None) == -1
    assert lib.phsa_step_host(*args, ok, 0.5, p, *([None] * 7), None, ws, None, None) == -6
    assert lib.phsa_step_host(*args, ok, 0.5, p, *([None] * 7), dummy, ws - 1, None, None) == -6
    assert lib.phsa_step_host(*args, phsa_shape(1, 4096, 16, 8, 64, 64), 0.5, p, *([None] * 7),
                              dummy, ws, None, None) == -2


def test_punct_mask_and_append_validation_needs_no_gpu(lib):
    # Both entry points reject bad arguments before any CUDA call.
    from paper_2601_02819_gb300.phsa import phsa_shape
    P = ctypes.c_void_p
    lib.phsa_punct_mask.argtypes = [P, ctypes.c_int64, P, ctypes.c_int, P, P]
    lib.phsa_decode_append.argtypes = [P, P, P, P, phsa_shape, P, P, P, P]
    dummy = ctypes.c_void_p(256)  # never dereferenced
    assert lib.phsa_punct_mask(dummy, 10, dummy, 4097, dummy, None) == -2  # set too large
    assert lib.phsa_punct_mask(dummy, -1, dummy, 4, dummy, None) == -1
    assert lib.phsa_punct_mask(dummy, 10, dummy, -1, dummy, None) == -1
    assert lib.phsa_punct_mask(None, 10, dummy, 4, dummy, None) == -1
    assert lib.phsa_punct_mask(dummy, 10, None, 4, dummy, None) == -1  # set without ids
    assert lib.phsa_punct_mask(None, 0, None, 4, None, None) == 0  # nothing to do
    ok = phsa_shape(2, 256, 8, 8, 128, 64)
    assert lib.phsa_decode_append(dummy, dummy, None, dummy, phsa_shape(2, 256, 8, 8, 64, 64),
                                  dummy, dummy, None, None) == -2  # D = 64
    assert lib.phsa_decode_append(None, dummy, None, dummy, ok, dummy, dummy, None, None) == -1
    assert lib.phsa_decode_append(dummy, dummy, dummy, dummy, ok, dummy, dummy, None,
                                  None) == -1  # flags without a mask
    odd = ctypes.c_void_p(264)  # not 16-byte aligned
    assert lib.phsa_decode_append(odd, dummy, None, dummy, ok, dummy, dummy, None, None) == -1
    assert lib.phsa_decode_append(None, None, None, None, phsa_shape(0, 256, 8, 8, 128, 64),
                                  None, None, None, None) == 0  # empty batch


def test_prefill_append_validation_needs_no_gpu(lib):
    from paper_2601_02819_gb300.phsa import phsa_shape
    P, I, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
    lib.phsa_prefill_append.argtypes = [P, P, P, P, I, phsa_shape, F, P, P, P, P, P]
    ok = phsa_shape(2, 512, 4, 2, 128, 64)
    f = lib.phsa_prefill_append
    assert f(None, None, None, None, 0, ok, 0.5, None, None, None, None, None) == 0   # empty chunk
    assert f(None, None, None, None, 16, ok, 1.5, None, None, None, None, None) == -1  # lambda > 1
    assert f(None, None, None, None, -1, ok, 0.5, None, None, None, None, None) == -1  # C < 0
    assert f(None, None, None, None, 513, ok, 0.5, None, None, None, None, None) == -1  # C > L
    assert f(None, None, None, None, 16, ok, 0.5, None, None, None, None, None) == -1  # null pointers
    for bs in (16, 32):  # accepted: the null pointers are what is rejected
        mb = phsa_shape(2, 512, 4, 2, 128, bs)
        assert f(None, None, None, None, 16, mb, 0.5, None, None, None, None, None) == -1
    m8 = phsa_shape(2, 512, 4, 2, 128, 8)
    assert f(None, None, None, None, 16, m8, 0.5, None, None, None, None, None) == -2  # m = 8
    d64 = phsa_shape(2, 512, 4, 2, 64, 64)
    assert f(None, None, None, None, 16, d64, 0.5, None, None, None, None, None) == -2  # D = 128 only


def test_decode_calls_take_block_sizes_16_and_32(lib):
    # past the block size check, a null pointer is what the decode calls reject
    from paper_2601_02819_gb300.phsa import phsa_shape, phsa_select_params
    P, F, I = ctypes.c_void_p, ctypes.c_float, ctypes.c_int
    lib.phsa_decode_update_repr.argtypes = [P, P, P, phsa_shape, F, P, P]
    lib.phsa_decode_select.argtypes = [P, P, P, phsa_shape, phsa_select_params, P, P, P]
    lib.phsa_decode_attn.argtypes = [P, P, P, P, P, P, phsa_shape, I, F, P, P, P]
    lib.phsa_decode_step.argtypes = [P, P, P, P, P, phsa_shape, F, phsa_select_params, P, P, P,
                                     P, P, P]
    p = phsa_select_params(12, 1, 2, 0.088)
    for bs, want in ((16, -1), (32, -1), (8, -2), (128, -2)):
        s = phsa_shape(2, 4096, 16, 8, 128, bs)
        assert lib.phsa_decode_update_repr(None, None, None, s, 0.5, None, None) == want
        assert lib.phsa_decode_select(None, None, None, s, p, None, None, None) == want
        assert lib.phsa_decode_attn(None, None, None, None, None, None, s, 12, 0.088, None, None,
                                    None) == want
        assert lib.phsa_decode_step(None, None, None, None, None, s, 0.5, p, None, None, None,
                                    None, None, None) == want
