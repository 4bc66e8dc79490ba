"""The C-ABI library loads and exports every entry point that include/namoh.h declares.

Runs without a GPU: only host-side functions are called (status strings, version,
workspace sizes, and argument checks that return before any CUDA call).
"""
import ctypes
import os
import subprocess

import pytest

from paper_2609_38832_gb300 import _abi, build


@pytest.fixture(scope="module")
def lib():
    build.build()
    return _abi.load()


def test_header_declares_the_three_calls():
    names = _abi.header_functions()
    for fn in ("namoh_route", "namoh_prefill", "namoh_decode"):
        assert fn in names


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", _abi.LIB_PATH], capture_output=True, text=True, check=True)
    exported = {line.split()[-1] for line in out.stdout.splitlines() if " T " in line}
    for fn in _abi.header_functions():
        assert fn in exported, fn
        assert fn in _abi.SIGNATURES, fn


def test_status_strings_and_version(lib):
    assert lib.namoh_status_string(0) == b"ok"
    assert b"invalid" in lib.namoh_status_string(-1)
    assert lib.namoh_status_string(-99) == b"unknown status"
    assert lib.namoh_version() >> 16 == 1


def test_workspace_sizes(lib):
    assert lib.namoh_route_workspace_size(4, 4096, 16, 4) > 0
    assert lib.namoh_route_workspace_size(0, 1, 1, 1) == 0
    assert lib.namoh_prefill_workspace_size(4, 4096, 16, 4, 128, 1) >= 4 * 4096 * 4 * 128 * 2
    assert lib.namoh_prefill_workspace_size(1, 16, 64, 32, 128, 8) > 0
    assert lib.namoh_prefill_workspace_size(1, 16, 8, 2, 96, 1) == 0  # d_head 96 not built
    assert lib.namoh_prefill_workspace_size(1, 16, 8, 3, 128, 2) == 0  # g must divide K
    assert lib.namoh_decode_workspace_size(64, 32, 4, 128, 1) > 0
    assert lib.namoh_decode_workspace_size(64, 32, 4, 80, 1) == 0


def test_argument_errors_return_before_any_launch(lib):
    P = ctypes.c_void_p
    fake = P(256)  # never dereferenced: every call below fails its host-side checks first
    st = P(512)
    # null scores
    assert lib.namoh_route(None, 1, 1, 8, 2, fake, fake, None, None, None, None, None, 0, st, None) == -1
    # K > H
    assert lib.namoh_route(fake, 1, 4, 4, 5, fake, fake, None, None, None, None, None, 0, st, None) == -1
    # H beyond the build limit
    assert lib.namoh_route(fake, 1, 4, 65, 2, fake, fake, None, None, None, None, None, 0, st, None) == -1
    # partial packed-layout outputs
    assert lib.namoh_route(fake, 1, 4, 8, 2, fake, fake, fake, None, fake, fake, None, 0, st, None) == -1
    # prefill: null q; unsupported d_head; k_cache aliasing k
    args = [fake, fake, fake, 1, 16, 8, 2, 128, 1, 10000.0, fake, fake, fake, fake, fake, fake, None, None, 0, None,
            fake, 1 << 20, st, None]
    a = list(args); a[0] = None
    assert lib.namoh_prefill(*a) == -1
    a = list(args); a[7] = 96
    assert lib.namoh_prefill(*a) == -2
    a = list(args); a[13] = a[1]
    assert lib.namoh_prefill(*a) == -1
    a = list(args); a[9] = 1.0  # rope base must exceed 1
    assert lib.namoh_prefill(*a) == -1
    # decode: null seg_base
    dargs = [fake, fake, fake, fake, fake, 2, 8, 2, 128, 1, 10000.0, fake, fake, None, fake, fake, 100, fake, fake,
             1 << 20, st, None]
    assert lib.namoh_decode(*dargs) == -1


def test_rope_flag_errors_return_before_any_launch(lib):
    P = ctypes.c_void_p
    fake = P(256)
    st = P(512)
    G, IL = _abi.NAMOH_ROPE_GLOBAL, _abi.NAMOH_ROPE_INTERLEAVED
    # prefill_ex: an unknown flag bit
    pargs = [fake, fake, fake, 1, 16, 8, 2, 128, 1, 10000.0, 0x4, fake, fake, fake, fake, fake, fake, None, None, 0,
             None, fake, 1 << 20, st, None]
    assert lib.namoh_prefill_ex(*pargs) == -1
    # rope_pack_ex: global positions need row_src
    rargs = [fake, fake, fake, 1, 16, 8, 2, 128, 1, 10000.0, G | IL, fake, None, fake, fake, fake, None, None, 0, st,
             None, 0, None]
    assert lib.namoh_rope_pack_ex(*rargs) == -1
    # decode_ex: token_pos exactly when global; unknown bits
    dargs = [fake, fake, fake, fake, fake, 2, 8, 2, 128, 1, 10000.0, G, None, fake, fake, fake, fake, fake, 100, fake,
             fake, 1 << 20, st, None]
    assert lib.namoh_decode_ex(*dargs) == -1
    a = list(dargs); a[11] = IL; a[12] = fake
    assert lib.namoh_decode_ex(*a) == -1
    a = list(dargs); a[11] = 0x8; a[12] = None
    assert lib.namoh_decode_ex(*a) == -1


def test_sa_sizes_and_argument_errors(lib):
    """SA + NAMOH: mask words and workspace for the supported block sizes, and every argument error
    (block size, alpha, null mask, too many blocks) returned before any launch."""
    assert lib.namoh_sa_mask_words(4096, 32) == 4
    assert lib.namoh_sa_mask_words(4097, 32) == 5
    assert lib.namoh_sa_mask_words(4096, 128) == 1
    assert lib.namoh_sa_mask_words(4096, 48) == 0 and lib.namoh_sa_mask_words(4096, 16) == 0
    plain = lib.namoh_prefill_workspace_size(4, 4096, 16, 4, 128, 1)
    # the dense prefill's workspace holds the rotated queries (R g d bf16) for the global-position path
    assert plain >= 65536 * 128 * 2
    # SA: the rotated queries (the selection reads them) plus the pooled keys, (R / block + B H) d bf16
    assert lib.namoh_sa_prefill_workspace_size(4, 4096, 16, 4, 128, 1, 32) >= 65536 * 128 * 2 + (65536 // 32 + 64) * 128 * 2
    assert lib.namoh_sa_prefill_workspace_size(4, 4096, 16, 4, 128, 1, 48) == 0
    P = ctypes.c_void_p
    fake = P(256)
    st = P(512)
    # q k v B T H K d g base flags seg row_src gate block num den mask y kc vc seg_base seg_cap rows seg_len ws wsb st s
    args = [fake, fake, fake, 1, 1024, 8, 2, 128, 1, 10000.0, 0, fake, fake, fake, 32, 1, 5, fake, fake, fake, fake,
            None, None, 0, None, fake, 1 << 24, st, None]
    for idx, bad in ((14, 48), (14, 16), (15, 0), (15, 6), (16, 0), (17, None), (0, None)):
        a = list(args)
        a[idx] = bad
        assert lib.namoh_sa_prefill(*a) == -1, (idx, bad)
    a = list(args)
    a[4] = 32 * 1024 + 1  # 1025 blocks of 32 keys: more than the selector holds
    assert lib.namoh_sa_prefill(*a) == -1
