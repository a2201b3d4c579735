"""SPADE verify step on GB300: Python binding of the C-ABI library libspade.so.

This module only marshals arguments: it checks dtypes and layouts of torch
tensors and passes raw device pointers, sizes and the current CUDA stream to
the library's entry points.  Every step of the verify path runs in the
library's CUDA kernels; there is no Python or CPU fallback, and a call fails
loudly if the library is missing.

Entry points (same names as the C ABI in include/spade.h):
    spade_verify_attention  verify-position attention against the KV cache
    spade_verify_accept     LM head + softmax + accept/reject + residual sampling
    spade_kv_commit         append accepted positions, roll back rejected ones
    spade_verify_qkv_rope   QKV projection + rotary embedding of the verify block, K/V into the cache
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import _build

__all__ = [
    "SpadeError", "load", "build", "library_path",
    "spade_verify_attention", "spade_verify_accept", "spade_kv_commit", "spade_verify_attention_noalloc",
    "spade_verify_qkv_rope", "spade_qkv_workspace_size", "qkv_workspace", "spade_verify_attention_paged", "spade_kv_commit_paged",
    "spade_verify_qkv_rope_paged",
    "spade_attn_workspace_size", "spade_accept_workspace_size", "spade_accept_launches",
    "spade_accept_stats_layout", "read_accept_stats", "spade_verify_accept_commit",
    "spade_verify_accept_sampling", "spade_verify_accept_commit_paged", "spade_selftest_wait_timeout",
    "attn_workspace", "accept_workspace", "status_tensor", "check_status",
    "DEV_BAD_INDEX", "DEV_CAPACITY", "DEV_TIMEOUT", "DEV_FALLBACK",
]

DEV_BAD_INDEX = 0x1
DEV_CAPACITY = 0x2
DEV_TIMEOUT = 0x4
DEV_FALLBACK = 0x8

_lib = None


class SpadeError(RuntimeError):
    """A non-OK status returned by the library (message from spade_last_error)."""

    def __init__(self, status, message):
        super().__init__(f"{message} [status {status}]")
        self.status = status


def library_path() -> str:
    return _build.LIB_PATH


def build(force: bool = False) -> str:
    return _build.build(force=force)


_i32 = ctypes.c_int32
_vp = ctypes.c_void_p
_sz = ctypes.c_size_t


def load():
    """Load libspade.so (built in-tree); raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    path = library_path()
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build the CUDA library first "
                           "(python -c 'import __graft_entry__ as g; g.build()')")
    lib = ctypes.CDLL(path)
    lib.spade_verify_attention.restype = _i32
    lib.spade_verify_attention.argtypes = [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                           _i32, _i32, _i32, _i32, _i32, _i32, _i32,
                                           _vp, _sz, _vp, _vp]
    lib.spade_verify_attention_noalloc.restype = _i32
    lib.spade_verify_attention_noalloc.argtypes = [_vp] * 8 + [_i32] * 7 + [_vp, _vp]
    lib.spade_attn_workspace_size.restype = _sz
    lib.spade_attn_workspace_size.argtypes = [_i32] * 6
    lib.spade_verify_accept.restype = _i32
    lib.spade_verify_accept.argtypes = [_vp] * 10 + [_i32] * 4 + [_vp, _sz, _vp, _vp]
    lib.spade_verify_accept_commit.restype = _i32
    lib.spade_verify_accept_commit.argtypes = [_vp] * 13 + [_i32] * 7 + [_vp, _sz, _vp, _vp]
    lib.spade_accept_workspace_size.restype = _sz
    lib.spade_accept_workspace_size.argtypes = [_i32] * 4
    lib.spade_verify_accept_temperature.restype = _i32
    lib.spade_verify_accept_temperature.argtypes = [_vp] * 11 + [_i32] * 4 + [_vp, _sz, _vp, _vp]
    lib.spade_verify_accept_sampling.restype = _i32
    lib.spade_verify_accept_sampling.argtypes = [_vp] * 15 + [_i32] * 7 + [_vp, _sz, _vp, _vp]
    lib.spade_accept_stats_layout.restype = _i32
    lib.spade_accept_stats_layout.argtypes = [_i32] * 4 + [_vp, _vp, _vp]
    lib.spade_accept_launches.restype = _i32
    lib.spade_accept_launches.argtypes = [_i32] * 4
    lib.spade_selftest_wait_timeout.restype = _i32
    lib.spade_selftest_wait_timeout.argtypes = [_vp, _i32, _vp]
    lib.spade_verify_qkv_rope.restype = _i32
    lib.spade_verify_qkv_rope.argtypes = [_vp] * 8 + [_i32] * 8 + [ctypes.c_float, _vp, _sz, _vp, _vp]
    lib.spade_qkv_workspace_size.restype = _sz
    lib.spade_qkv_workspace_size.argtypes = [_i32] * 4
    lib.spade_verify_attention_paged.restype = _i32
    lib.spade_verify_attention_paged.argtypes = [_vp] * 9 + [_i32] * 9 + [_vp, _sz, _vp, _vp]
    lib.spade_verify_accept_commit_paged.restype = _i32
    lib.spade_verify_accept_commit_paged.argtypes = [_vp] * 14 + [_i32] * 9 + [_vp, _sz, _vp, _vp]
    lib.spade_kv_commit_paged.restype = _i32
    lib.spade_kv_commit_paged.argtypes = [_vp] * 6 + [_i32] * 6 + [_vp, _vp]
    lib.spade_verify_qkv_rope_paged.restype = _i32
    lib.spade_verify_qkv_rope_paged.argtypes = [_vp] * 9 + [_i32] * 10 + [ctypes.c_float, _vp, _sz, _vp, _vp]
    lib.spade_kv_commit.restype = _i32
    lib.spade_kv_commit.argtypes = [_vp] * 5 + [_i32] * 4 + [_vp, _vp]
    lib.spade_status_string.restype = ctypes.c_char_p
    lib.spade_status_string.argtypes = [_i32]
    lib.spade_last_error.restype = ctypes.c_char_p
    lib.spade_last_error.argtypes = []
    lib.spade_version.restype = ctypes.c_char_p
    lib.spade_version.argtypes = []
    _lib = lib
    return lib


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check_rc(rc):
    if rc != 0:
        lib = load()
        raise SpadeError(rc, f"{lib.spade_status_string(rc).decode()}: {lib.spade_last_error().decode()}")


def _need(t, name, dtype, ndim=None):
    if t is None:
        raise ValueError(f"{name} is required")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got {t.dim()}")


def status_tensor(device="cuda"):
    """A zeroed device int32 status word."""
    return torch.zeros(1, dtype=torch.int32, device=device)


def check_status(status):
    """Reads the device status word (synchronises) and returns its SPADE_DEV_* bits."""
    return int(status.item())


# ---------------------------------------------------------------------------
def spade_attn_workspace_size(B, Hq, Hkv, D, cap, max_k):
    return int(load().spade_attn_workspace_size(B, Hq, Hkv, D, cap, max_k))


def attn_workspace(B, Hq, Hkv, D, cap, max_k, device="cuda"):
    """A zeroed workspace for spade_verify_attention (zeroed once; calls keep it zeroed)."""
    n = spade_attn_workspace_size(B, Hq, Hkv, D, cap, max_k)
    if n == 0:
        raise SpadeError(-1, "spade_attn_workspace_size returned 0: " + load().spade_last_error().decode())
    return torch.zeros(n, dtype=torch.uint8, device=device)


def spade_verify_attention(q, k_cache, v_cache, ctx_lens, n_draft, cu_q, out, lse=None, *,
                           max_k, workspace, status, stream=None):
    """out[cu_q[b]+i, h] = softmax(q K^T / sqrt(D)) V over keys [0, ctx_b + i] (KV head h // G)."""
    _need(q, "q", torch.bfloat16, 3)
    _need(k_cache, "k_cache", torch.bfloat16, 4)
    _need(v_cache, "v_cache", torch.bfloat16, 4)
    for t, n in ((ctx_lens, "ctx_lens"), (n_draft, "n_draft"), (cu_q, "cu_q"), (status, "status")):
        _need(t, n, torch.int32, 1)
    _need(out, "out", torch.bfloat16, 3)
    if lse is not None:
        _need(lse, "lse", torch.float32, 2)
    _need(workspace, "workspace", torch.uint8, 1)
    if v_cache.shape != k_cache.shape:
        raise ValueError("k_cache and v_cache shapes differ")
    R, Hq, D = q.shape
    B, Hkv, cap, Dk = k_cache.shape
    if Dk != D or tuple(out.shape) != (R, Hq, D) or ctx_lens.numel() != B or n_draft.numel() != B \
            or cu_q.numel() != B + 1:
        raise ValueError("inconsistent attention shapes")
    rc = load().spade_verify_attention(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(ctx_lens), _ptr(n_draft), _ptr(cu_q), _ptr(out),
        _ptr(lse), B, Hq, Hkv, D, cap, int(max_k), R, _ptr(workspace), workspace.numel(),
        _ptr(status), _stream(stream))
    _check_rc(rc)
    return out


def spade_verify_attention_noalloc(q, k_cache, v_cache, ctx_lens, n_draft, cu_q, out, lse=None, *,
                                   max_k, status, stream=None):
    """spade_verify_attention for callers that cannot allocate: scratch in a static device array.

    Calls that overlap on the GPU share that array and race; the first call on
    a device resolves the array's address and should precede any stream capture.
    """
    R, Hq, D = q.shape
    B, Hkv, cap, _ = k_cache.shape
    for t, n in ((q, "q"), (k_cache, "k_cache"), (v_cache, "v_cache"), (out, "out")):
        _need(t, n, torch.bfloat16)
    for t, n in ((ctx_lens, "ctx_lens"), (n_draft, "n_draft"), (cu_q, "cu_q"), (status, "status")):
        _need(t, n, torch.int32, 1)
    rc = load().spade_verify_attention_noalloc(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(ctx_lens), _ptr(n_draft), _ptr(cu_q), _ptr(out),
        _ptr(lse), B, Hq, Hkv, D, cap, int(max_k), R, _ptr(status), _stream(stream))
    _check_rc(rc)
    return out


# ---------------------------------------------------------------------------
def spade_accept_workspace_size(B, R, H, V):
    return int(load().spade_accept_workspace_size(B, R, H, V))


def spade_selftest_wait_timeout(status, limit_us, stream=None):
    """One bounded wait that nothing completes: SPADE_DEV_TIMEOUT lands in `status` after limit_us."""
    _need(status, "status", torch.int32, 1)
    _check_rc(load().spade_selftest_wait_timeout(_ptr(status), int(limit_us), _stream(stream)))


def spade_accept_stats_layout(B, R, H, V):
    """Byte offsets of the merged row statistics and the draft logits in an accept workspace.

    Returns (row_stats_offset, draft_logit_offset, replica_stride); see include/spade.h.
    """
    a, b, c = ctypes.c_size_t(0), ctypes.c_size_t(0), ctypes.c_int32(0)
    _check_rc(load().spade_accept_stats_layout(B, R, H, V, ctypes.byref(a), ctypes.byref(b), ctypes.byref(c)))
    return int(a.value), int(b.value), int(c.value)


def read_accept_stats(workspace, B, R, H, V):
    """Row statistics a completed accept call left in `workspace` (reads device memory).

    Returns dict of torch CPU tensors: max [R] f32, sumexp [R] f32, argmax [R] i32,
    accept_bit [R] i32, draft_logit [R] f32 (rows with a draft only are meaningful).
    """
    off_s, off_d, _ = spade_accept_stats_layout(B, R, H, V)
    st = workspace[off_s:off_s + 16 * R].view(torch.float32).view(R, 4).cpu()
    ld = workspace[off_d:off_d + 4 * R].view(torch.float32).cpu()
    return dict(max=st[:, 0].clone(), sumexp=st[:, 1].clone(), argmax=st[:, 2].clone().view(torch.int32),
                accept_bit=st[:, 3].clone().view(torch.int32), draft_logit=ld.clone())


def spade_accept_launches(B, R, H, V):
    """Kernel launches of one accept call: 1 (logits on chip) or 2 (statistics pass, then sampling pass)."""
    return int(load().spade_accept_launches(B, R, H, V))


def accept_workspace(B, R, H, V, device="cuda"):
    """A zeroed workspace for spade_verify_accept (zeroed once; calls keep it usable)."""
    n = spade_accept_workspace_size(B, R, H, V)
    if n == 0:
        raise SpadeError(-1, "spade_accept_workspace_size returned 0: " + load().spade_last_error().decode())
    return torch.zeros(n, dtype=torch.uint8, device=device)


def spade_verify_accept(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q, n_draft,
                        accepted_len, next_token, *, workspace, status, stream=None, temperature=None):
    """Greedy / rejection-sampling verification of every sequence (see include/spade.h); with
    ``temperature`` ([B] float32) the verifier's p is softmax(logits / T)."""
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(w_lm, "w_lm", torch.bfloat16, 2)
    _need(uniforms, "uniforms", torch.float32, 1)
    for t, n in ((draft_tokens, "draft_tokens"), (mode, "mode"), (cu_q, "cu_q"), (n_draft, "n_draft"),
                 (accepted_len, "accepted_len"), (next_token, "next_token"), (status, "status")):
        _need(t, n, torch.int32, 1)
    if draft_probs is not None:
        _need(draft_probs, "draft_probs", torch.float32, 2)
    _need(workspace, "workspace", torch.uint8, 1)
    R, H = hidden.shape
    V, H2 = w_lm.shape
    B = n_draft.numel()
    if H2 != H or uniforms.numel() != R or draft_tokens.numel() != R - B or cu_q.numel() != B + 1 \
            or mode.numel() != B or accepted_len.numel() != B or next_token.numel() != B:
        raise ValueError("inconsistent accept shapes")
    if draft_probs is not None and tuple(draft_probs.shape) != (R - B, V):
        raise ValueError("draft_probs must be [R - B, V]")
    if temperature is None:
        rc = load().spade_verify_accept(
            _ptr(hidden), _ptr(w_lm), _ptr(draft_tokens), _ptr(draft_probs), _ptr(uniforms), _ptr(mode),
            _ptr(cu_q), _ptr(n_draft), _ptr(accepted_len), _ptr(next_token), B, R, H, V,
            _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream))
    else:
        _need(temperature, "temperature", torch.float32, 1)
        if temperature.numel() != B:
            raise ValueError("temperature must be [B]")
        rc = load().spade_verify_accept_temperature(
            _ptr(hidden), _ptr(w_lm), _ptr(draft_tokens), _ptr(draft_probs), _ptr(uniforms), _ptr(mode),
            _ptr(temperature), _ptr(cu_q), _ptr(n_draft), _ptr(accepted_len), _ptr(next_token), B, R, H, V,
            _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream))
    _check_rc(rc)
    return accepted_len, next_token


def spade_verify_accept_commit(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q, n_draft,
                               accepted_len, next_token, k_cache, v_cache, ctx_lens, *, workspace,
                               status, stream=None):
    """spade_verify_accept followed by spade_kv_commit in one launch (see include/spade.h)."""
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(w_lm, "w_lm", torch.bfloat16, 2)
    _need(uniforms, "uniforms", torch.float32, 1)
    for t, n in ((draft_tokens, "draft_tokens"), (mode, "mode"), (cu_q, "cu_q"), (n_draft, "n_draft"),
                 (accepted_len, "accepted_len"), (next_token, "next_token"), (status, "status"),
                 (ctx_lens, "ctx_lens")):
        _need(t, n, torch.int32, 1)
    if draft_probs is not None:
        _need(draft_probs, "draft_probs", torch.float32, 2)
    _need(workspace, "workspace", torch.uint8, 1)
    _need(k_cache, "k_cache", torch.bfloat16, 4)
    _need(v_cache, "v_cache", torch.bfloat16, 4)
    R, H = hidden.shape
    V, H2 = w_lm.shape
    B = n_draft.numel()
    Bc, Hkv, cap, D = k_cache.shape
    if H2 != H or uniforms.numel() != R or draft_tokens.numel() != R - B or cu_q.numel() != B + 1 \
            or mode.numel() != B or accepted_len.numel() != B or next_token.numel() != B \
            or Bc != B or tuple(v_cache.shape) != tuple(k_cache.shape) or ctx_lens.numel() != B:
        raise ValueError("inconsistent accept/commit shapes")
    if draft_probs is not None and tuple(draft_probs.shape) != (R - B, V):
        raise ValueError("draft_probs must be [R - B, V]")
    rc = load().spade_verify_accept_commit(
        _ptr(hidden), _ptr(w_lm), _ptr(draft_tokens), _ptr(draft_probs), _ptr(uniforms), _ptr(mode),
        _ptr(cu_q), _ptr(n_draft), _ptr(accepted_len), _ptr(next_token), _ptr(k_cache), _ptr(v_cache),
        _ptr(ctx_lens), B, R, H, V, Hkv, D, cap, _ptr(workspace), workspace.numel(), _ptr(status),
        _stream(stream))
    _check_rc(rc)
    return accepted_len, next_token


def spade_verify_accept_sampling(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q, n_draft,
                                 accepted_len, next_token, *, workspace, status, temperature=None, top_p=None,
                                 k_cache=None, v_cache=None, ctx_lens=None, stream=None):
    """spade_verify_accept with per-sequence ``temperature`` and ``top_p`` ([B] float32, either
    may be None) and, with k_cache / v_cache / ctx_lens given, the fused KV commit
    (see include/spade.h)."""
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(w_lm, "w_lm", torch.bfloat16, 2)
    _need(uniforms, "uniforms", torch.float32, 1)
    for t, n in ((draft_tokens, "draft_tokens"), (mode, "mode"), (cu_q, "cu_q"), (n_draft, "n_draft"),
                 (accepted_len, "accepted_len"), (next_token, "next_token"), (status, "status")):
        _need(t, n, torch.int32, 1)
    if draft_probs is not None:
        _need(draft_probs, "draft_probs", torch.float32, 2)
    _need(workspace, "workspace", torch.uint8, 1)
    R, H = hidden.shape
    V, H2 = w_lm.shape
    B = n_draft.numel()
    if H2 != H or uniforms.numel() != R or draft_tokens.numel() != R - B or cu_q.numel() != B + 1 \
            or mode.numel() != B or accepted_len.numel() != B or next_token.numel() != B:
        raise ValueError("inconsistent accept shapes")
    if draft_probs is not None and tuple(draft_probs.shape) != (R - B, V):
        raise ValueError("draft_probs must be [R - B, V]")
    for t, n in ((temperature, "temperature"), (top_p, "top_p")):
        if t is not None:
            _need(t, n, torch.float32, 1)
            if t.numel() != B:
                raise ValueError(f"{n} must be [B]")
    Hkv = D = cap = 0
    if (k_cache is None) != (v_cache is None) or (k_cache is None) != (ctx_lens is None):
        raise ValueError("give all of k_cache, v_cache, ctx_lens or none")
    if k_cache is not None:
        _need(k_cache, "k_cache", torch.bfloat16, 4)
        _need(v_cache, "v_cache", torch.bfloat16, 4)
        _need(ctx_lens, "ctx_lens", torch.int32, 1)
        Bc, Hkv, cap, D = k_cache.shape
        if Bc != B or tuple(v_cache.shape) != tuple(k_cache.shape) or ctx_lens.numel() != B:
            raise ValueError("inconsistent cache shapes")
    rc = load().spade_verify_accept_sampling(
        _ptr(hidden), _ptr(w_lm), _ptr(draft_tokens), _ptr(draft_probs), _ptr(uniforms), _ptr(mode),
        _ptr(temperature), _ptr(top_p), _ptr(cu_q), _ptr(n_draft), _ptr(accepted_len), _ptr(next_token),
        _ptr(k_cache), _ptr(v_cache), _ptr(ctx_lens), B, R, H, V, Hkv, D, cap, _ptr(workspace),
        workspace.numel(), _ptr(status), _stream(stream))
    _check_rc(rc)
    return accepted_len, next_token


def spade_verify_accept_commit_paged(hidden, w_lm, draft_tokens, draft_probs, uniforms, mode, cu_q, n_draft,
                                     accepted_len, next_token, k_pool, v_pool, block_table, ctx_lens, *,
                                     workspace, status, stream=None):
    """spade_verify_accept_commit on paged caches: pools [num_pages, Hkv, page_size, D] and a
    block table [B, max_pages] (see include/spade.h)."""
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(w_lm, "w_lm", torch.bfloat16, 2)
    _need(uniforms, "uniforms", torch.float32, 1)
    for t, n in ((draft_tokens, "draft_tokens"), (mode, "mode"), (cu_q, "cu_q"), (n_draft, "n_draft"),
                 (accepted_len, "accepted_len"), (next_token, "next_token"), (status, "status"),
                 (ctx_lens, "ctx_lens")):
        _need(t, n, torch.int32, 1)
    if draft_probs is not None:
        _need(draft_probs, "draft_probs", torch.float32, 2)
    _need(workspace, "workspace", torch.uint8, 1)
    _need(k_pool, "k_pool", torch.bfloat16, 4)
    _need(v_pool, "v_pool", torch.bfloat16, 4)
    _need(block_table, "block_table", torch.int32, 2)
    R, H = hidden.shape
    V, H2 = w_lm.shape
    B = n_draft.numel()
    num_pages, Hkv, page_size, D = k_pool.shape
    if H2 != H or uniforms.numel() != R or draft_tokens.numel() != R - B or cu_q.numel() != B + 1 \
            or mode.numel() != B or accepted_len.numel() != B or next_token.numel() != B \
            or tuple(v_pool.shape) != tuple(k_pool.shape) or ctx_lens.numel() != B or block_table.shape[0] != B:
        raise ValueError("inconsistent accept/commit shapes")
    if draft_probs is not None and tuple(draft_probs.shape) != (R - B, V):
        raise ValueError("draft_probs must be [R - B, V]")
    rc = load().spade_verify_accept_commit_paged(
        _ptr(hidden), _ptr(w_lm), _ptr(draft_tokens), _ptr(draft_probs), _ptr(uniforms), _ptr(mode),
        _ptr(cu_q), _ptr(n_draft), _ptr(accepted_len), _ptr(next_token), _ptr(k_pool), _ptr(v_pool),
        _ptr(block_table), _ptr(ctx_lens), B, R, H, V, Hkv, D, page_size, num_pages, block_table.shape[1],
        _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream))
    _check_rc(rc)
    return accepted_len, next_token


# ---------------------------------------------------------------------------
def spade_qkv_workspace_size(R, Hq, Hkv, D):
    return int(load().spade_qkv_workspace_size(R, Hq, Hkv, D))


def qkv_workspace(R, Hq, Hkv, D, device="cuda"):
    """A zeroed workspace for spade_verify_qkv_rope (zeroed once; calls keep its counters zeroed)."""
    n = spade_qkv_workspace_size(R, Hq, Hkv, D)
    if n == 0:
        raise SpadeError(-1, "spade_qkv_workspace_size returned 0: " + load().spade_last_error().decode())
    return torch.zeros(n, dtype=torch.uint8, device=device)


def spade_verify_qkv_rope(x, w_qkv, ctx_lens, n_draft, cu_q, q_out, k_cache, v_cache, *, Hq, Hkv,
                          rope_theta, max_k, workspace, status, stream=None):
    """q, k, v of the verify block (rotary embedding at ctx + i); K/V into cache slots ctx .. ctx + k."""
    _need(x, "x", torch.bfloat16, 2)
    _need(w_qkv, "w_qkv", torch.bfloat16, 2)
    _need(q_out, "q_out", torch.bfloat16, 3)
    _need(k_cache, "k_cache", torch.bfloat16, 4)
    _need(v_cache, "v_cache", torch.bfloat16, 4)
    for t, n in ((ctx_lens, "ctx_lens"), (n_draft, "n_draft"), (cu_q, "cu_q"), (status, "status")):
        _need(t, n, torch.int32, 1)
    R, H = x.shape
    B, Hkv2, cap, D = k_cache.shape
    if Hkv2 != Hkv or tuple(v_cache.shape) != tuple(k_cache.shape) or tuple(q_out.shape) != (R, Hq, D) \
            or tuple(w_qkv.shape) != ((Hq + 2 * Hkv) * D, H) or ctx_lens.numel() != B or n_draft.numel() != B \
            or cu_q.numel() != B + 1:
        raise ValueError("inconsistent qkv_rope shapes")
    _need(workspace, "workspace", torch.uint8, 1)
    rc = load().spade_verify_qkv_rope(
        _ptr(x), _ptr(w_qkv), _ptr(ctx_lens), _ptr(n_draft), _ptr(cu_q), _ptr(q_out), _ptr(k_cache), _ptr(v_cache),
        B, R, H, Hq, Hkv, D, cap, int(max_k), float(rope_theta), _ptr(workspace), workspace.numel(), _ptr(status),
        _stream(stream))
    _check_rc(rc)
    return q_out


# ---------------------------------------------------------------------------
# Paged KV cache: pools [num_pages, Hkv, page_size, D], block_table [B, max_pages].
def _need_paged(k_pool, v_pool, block_table):
    _need(k_pool, "k_pool", torch.bfloat16, 4)
    _need(v_pool, "v_pool", torch.bfloat16, 4)
    _need(block_table, "block_table", torch.int32, 2)
    if tuple(v_pool.shape) != tuple(k_pool.shape):
        raise ValueError("k_pool and v_pool shapes differ")
    num_pages, Hkv, page_size, D = k_pool.shape
    return num_pages, Hkv, page_size, D, block_table.shape[1]


def spade_verify_attention_paged(q, k_pool, v_pool, block_table, ctx_lens, n_draft, cu_q, out, lse=None, *,
                                 max_k, workspace, status, stream=None):
    """spade_verify_attention on a paged cache (see include/spade.h)."""
    _need(q, "q", torch.bfloat16, 3)
    _need(out, "out", torch.bfloat16, 3)
    num_pages, Hkv, page_size, D, max_pages = _need_paged(k_pool, v_pool, block_table)
    for t, n in ((ctx_lens, "ctx_lens"), (n_draft, "n_draft"), (cu_q, "cu_q"), (status, "status")):
        _need(t, n, torch.int32, 1)
    if lse is not None:
        _need(lse, "lse", torch.float32, 2)
    _need(workspace, "workspace", torch.uint8, 1)
    R, Hq, Dq = q.shape
    B = ctx_lens.numel()
    if Dq != D or tuple(out.shape) != (R, Hq, D) or block_table.shape[0] != B or n_draft.numel() != B \
            or cu_q.numel() != B + 1:
        raise ValueError("inconsistent paged attention shapes")
    rc = load().spade_verify_attention_paged(
        _ptr(q), _ptr(k_pool), _ptr(v_pool), _ptr(block_table), _ptr(ctx_lens), _ptr(n_draft), _ptr(cu_q), _ptr(out),
        _ptr(lse), B, Hq, Hkv, D, page_size, num_pages, max_pages, int(max_k), R, _ptr(workspace), workspace.numel(),
        _ptr(status), _stream(stream))
    _check_rc(rc)
    return out


def spade_kv_commit_paged(k_pool, v_pool, block_table, ctx_lens, accepted_len, n_draft, *, status, stream=None):
    """spade_kv_commit on a paged cache (see include/spade.h)."""
    num_pages, Hkv, page_size, D, max_pages = _need_paged(k_pool, v_pool, block_table)
    for t, n in ((ctx_lens, "ctx_lens"), (accepted_len, "accepted_len"), (n_draft, "n_draft"), (status, "status")):
        _need(t, n, torch.int32, 1)
    B = ctx_lens.numel()
    if block_table.shape[0] != B:
        raise ValueError("block_table must have one row per sequence")
    rc = load().spade_kv_commit_paged(_ptr(k_pool), _ptr(v_pool), _ptr(block_table), _ptr(ctx_lens),
                                      _ptr(accepted_len), _ptr(n_draft), B, Hkv, D, page_size, num_pages,
                                      max_pages, _ptr(status), _stream(stream))
    _check_rc(rc)


def spade_verify_qkv_rope_paged(x, w_qkv, block_table, ctx_lens, n_draft, cu_q, q_out, k_pool, v_pool, *, Hq,
                                rope_theta, max_k, workspace, status, stream=None):
    """spade_verify_qkv_rope writing the block's K/V into a paged cache (see include/spade.h)."""
    _need(x, "x", torch.bfloat16, 2)
    _need(w_qkv, "w_qkv", torch.bfloat16, 2)
    _need(q_out, "q_out", torch.bfloat16, 3)
    num_pages, Hkv, page_size, D, max_pages = _need_paged(k_pool, v_pool, block_table)
    for t, n in ((ctx_lens, "ctx_lens"), (n_draft, "n_draft"), (cu_q, "cu_q"), (status, "status")):
        _need(t, n, torch.int32, 1)
    R, H = x.shape
    B = ctx_lens.numel()
    if tuple(q_out.shape) != (R, Hq, D) or tuple(w_qkv.shape) != ((Hq + 2 * Hkv) * D, H) \
            or block_table.shape[0] != B or n_draft.numel() != B or cu_q.numel() != B + 1:
        raise ValueError("inconsistent paged qkv_rope shapes")
    _need(workspace, "workspace", torch.uint8, 1)
    rc = load().spade_verify_qkv_rope_paged(
        _ptr(x), _ptr(w_qkv), _ptr(block_table), _ptr(ctx_lens), _ptr(n_draft), _ptr(cu_q), _ptr(q_out),
        _ptr(k_pool), _ptr(v_pool), B, R, H, Hq, Hkv, D, page_size, num_pages, max_pages, int(max_k),
        float(rope_theta), _ptr(workspace), workspace.numel(), _ptr(status), _stream(stream))
    _check_rc(rc)
    return q_out


# ---------------------------------------------------------------------------
def spade_kv_commit(k_cache, v_cache, ctx_lens, accepted_len, n_draft, *, status, stream=None):
    """ctx_lens += accepted_len + 1; rejected draft slots of the caches are cleared."""
    _need(k_cache, "k_cache", torch.bfloat16, 4)
    _need(v_cache, "v_cache", torch.bfloat16, 4)
    for t, n in ((ctx_lens, "ctx_lens"), (accepted_len, "accepted_len"), (n_draft, "n_draft"),
                 (status, "status")):
        _need(t, n, torch.int32, 1)
    B, Hkv, cap, D = k_cache.shape
    rc = load().spade_kv_commit(_ptr(k_cache), _ptr(v_cache), _ptr(ctx_lens), _ptr(accepted_len),
                                _ptr(n_draft), B, Hkv, D, cap, _ptr(status), _stream(stream))
    _check_rc(rc)
