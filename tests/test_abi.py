"""The C-ABI library builds for sm_103a, loads, and exports what include/spade.h declares.

CPU only: no call here launches a kernel.  Host-side validation runs before
any device query, so argument errors are checked without a GPU.
"""
import ctypes
import os
import re
import subprocess

import pytest

import paper_2608_13076_gb300 as spade
from paper_2608_13076_gb300 import _build

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "spade.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(spade_[a-z_]+)\s*\(", src)))


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return spade.load()


def test_header_declares_the_entry_points():
    names = declared_functions()
    for n in ("spade_verify_attention", "spade_verify_accept", "spade_kv_commit", "spade_verify_accept_commit",
              "spade_attn_workspace_size", "spade_accept_workspace_size", "spade_last_error",
              "spade_status_string"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", _build.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r" T (\w+)$", out, flags=re.M))
    missing = [n for n in declared_functions() if n not in exported]
    assert not missing, missing
    for n in declared_functions():
        assert hasattr(lib, n)


def test_library_is_built_for_sm103a(lib):
    # The fatbinary holds sm_103a code only (names from cuobjdump's listing, not its contents).
    r = subprocess.run(["cuobjdump", "--list-elf", _build.LIB_PATH], capture_output=True, text=True)
    assert r.returncode == 0
    assert "sm_103a" in r.stdout
    assert all("sm_103" in line for line in r.stdout.splitlines() if line.strip())


def test_status_strings(lib):
    assert lib.spade_status_string(0) == b"SPADE_OK"
    assert lib.spade_status_string(4) == b"SPADE_ERR_UNSUPPORTED_DEVICE"
    assert b"sm_103a" in lib.spade_version()


def test_null_arguments_rejected_before_any_device_work(lib):
    rc = lib.spade_verify_attention(*([None] * 8), 1, 8, 8, 128, 300, 4, 5, None, 0, None, None)
    assert rc == 1 and b"null" in lib.spade_last_error()
    rc = lib.spade_verify_accept(*([None] * 10), 1, 5, 512, 1024, None, 0, None, None)
    assert rc == 1
    rc = lib.spade_kv_commit(*([None] * 5), 1, 8, 128, 300, None, None)
    assert rc == 1
    rc = lib.spade_verify_accept_commit(*([None] * 13), 1, 5, 512, 1024, 8, 128, 300, None, 0, None, None)
    assert rc == 1
    rc = lib.spade_verify_accept_sampling(*([None] * 15), 1, 5, 512, 1024, 0, 0, 0, None, 0, None, None)
    assert rc == 1


def test_paged_accept_commit_validation_before_device_work(lib):
    p = ctypes.c_void_p(16)
    base = [p] * 10  # hidden .. next_token
    # Null table.
    assert lib.spade_verify_accept_commit_paged(*base, p, p, None, p, 1, 5, 512, 1024, 8, 128, 64, 10, 4,
                                                p, 1 << 20, p, None) == 1
    # Non-positive page size; head dim not a multiple of 8.
    assert lib.spade_verify_accept_commit_paged(*base, p, p, p, p, 1, 5, 512, 1024, 8, 128, 0, 10, 4,
                                                p, 1 << 20, p, None) == 1
    assert lib.spade_verify_accept_commit_paged(*base, p, p, p, p, 1, 5, 512, 1024, 8, 12, 64, 10, 4,
                                                p, 1 << 20, p, None) == 2


def test_sampling_entry_point_validation_before_device_work(lib):
    p = ctypes.c_void_p(16)
    base = [p] * 12  # hidden .. next_token, temperature and top_p given
    # Cache pointers: all three or none.
    assert lib.spade_verify_accept_sampling(*base, p, None, None, 1, 5, 512, 1024, 8, 128, 300,
                                            p, 1 << 20, p, None) == 1
    assert b"all of k_cache" in lib.spade_last_error()
    # Non-positive cache sizes with a commit.
    assert lib.spade_verify_accept_sampling(*base, p, p, p, 1, 5, 512, 1024, 0, 128, 300,
                                            p, 1 << 20, p, None) == 1
    # Head dim not a multiple of 8 with a commit; hidden size not a multiple of 8.
    assert lib.spade_verify_accept_sampling(*base, p, p, p, 1, 5, 512, 1024, 8, 12, 300,
                                            p, 1 << 20, p, None) == 2
    assert lib.spade_verify_accept_sampling(*base, None, None, None, 1, 5, 500, 1024, 0, 0, 0,
                                            p, 1 << 20, p, None) == 2


def test_selftest_rejects_bad_arguments_before_device_work(lib):
    assert lib.spade_selftest_wait_timeout(None, 1000, None) == 1
    p = ctypes.c_void_p(16)
    assert lib.spade_selftest_wait_timeout(p, 0, None) == 1
    assert lib.spade_selftest_wait_timeout(p, 2000000, None) == 1


def test_launch_count_rejects_invalid_sizes(lib):
    # Validation precedes the device query, so these need no GPU.
    assert lib.spade_accept_launches(0, 5, 512, 1024) == 0
    assert lib.spade_accept_launches(4, 3, 512, 1024) == 0   # R < B
    assert lib.spade_accept_launches(1, 5, 0, 1024) == 0


def test_bad_shapes_rejected(lib):
    p = ctypes.c_void_p(16)
    args = [p] * 7 + [None]
    # Hq not a multiple of Hkv
    assert lib.spade_verify_attention(*args, 1, 6, 4, 128, 300, 4, 5, p, 1 << 20, p, None) == 2
    # head dim 96 unsupported
    assert lib.spade_verify_attention(*args, 1, 8, 8, 96, 300, 4, 5, p, 1 << 20, p, None) == 2
    # hidden size not a multiple of 8
    assert lib.spade_verify_accept(*([p] * 10), 1, 5, 500, 1024, p, 1 << 20, p, None) == 2
    # head dim not a multiple of 8 for commit
    assert lib.spade_kv_commit(*([p] * 5), 1, 8, 12, 300, p, None) == 2
    assert lib.spade_verify_accept_commit(*([p] * 13), 1, 5, 512, 1024, 8, 12, 300, p, 1 << 20, p, None) == 2
    # The allocation-free attention gives the workspace entry point's codes.
    assert lib.spade_verify_attention_noalloc(*args, 1, 6, 4, 128, 300, 4, 5, p, None) == 2
    assert lib.spade_verify_attention_noalloc(*args, 1, 8, 8, 96, 300, 4, 5, p, None) == 2
    assert lib.spade_verify_attention_noalloc(*args, 0, 8, 8, 128, 300, 4, 5, p, None) == 1


def test_stats_layout_rejects_bad_arguments(lib):
    out = ctypes.c_size_t(0)
    assert lib.spade_accept_stats_layout(1, 5, 512, 1024, None, None, None) == 1
    assert lib.spade_accept_stats_layout(4, 3, 512, 1024, ctypes.byref(out), ctypes.byref(out),
                                         ctypes.byref(ctypes.c_int32(0))) == 1


def test_qkv_rope_validation_before_device_work(lib):
    p = ctypes.c_void_p(16)
    f = lib.spade_verify_qkv_rope
    assert f(*([None] * 8), 1, 5, 512, 8, 8, 128, 300, 4, ctypes.c_float(1e4), None, 0, None, None) == 1  # null
    assert f(*([p] * 8), 1, 5, 512, 8, 8, 96, 300, 4, ctypes.c_float(1e4), p, 1 << 20, p, None) == 2          # D = 96
    assert f(*([p] * 8), 1, 5, 512, 6, 4, 128, 300, 4, ctypes.c_float(1e4), p, 1 << 20, p, None) == 2         # Hq % Hkv
    assert f(*([p] * 8), 1, 5, 500, 8, 8, 128, 300, 4, ctypes.c_float(1e4), p, 1 << 20, p, None) == 2         # H % 8
    assert f(*([p] * 8), 1, 5, 512, 3, 3, 64, 300, 4, ctypes.c_float(1e4), p, 1 << 20, p, None) == 2          # (Hq+2Hkv)D % 128
    assert f(*([p] * 8), 1, 600, 512, 8, 8, 128, 900, 4, ctypes.c_float(1e4), p, 1 << 20, p, None) == 2       # R > 512
    assert f(*([p] * 8), 1, 5, 512, 8, 8, 128, 300, 4, ctypes.c_float(0.5), p, 1 << 20, p, None) == 1         # theta <= 1
