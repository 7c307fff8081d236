"""Python binding of the C ABI in include/specflash_verify.h (ctypes).

Argument marshalling only: tensors are checked for dtype, device, shape and
contiguity, their device pointers and the current CUDA stream are passed to
the library, and outputs/workspaces are allocated with torch when the caller
does not supply them.  Every step of the computation runs in the library's
CUDA kernels; there is no fallback.  If the compiled library is missing the
first call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build_lib

SF_OK = 0
SF_DEVICE_BAD_PAGE = 0x1
SF_DEVICE_BAD_TOKEN = 0x2
SF_DEVICE_TIMEOUT = 0x4
SF_DEVICE_BAD_SEQLEN = 0x8
SF_DEVICE_OUT_OF_PAGES = 0x10
PAGE_SIZE = 16

EXPORTED_SYMBOLS = (
    "sf_status_string", "sf_last_error", "sf_version", "sf_workspace_init",
    "sf_read_device_status", "sf_selftest_bounded_wait",
    "sf_verify_attention_workspace_size", "sf_verify_attention",
    "sf_verify_attention_noalloc", "sf_verify_attention_kernel_launches",
    "sf_accept_workspace_size", "sf_accept", "sf_accept_kernel_launches",
    "sf_kv_commit_workspace_size", "sf_kv_commit",
    "sf_draft_tail_workspace_size", "sf_lm_head", "sf_sample", "sf_draft_sample",
    "sf_visual_compress_workspace_size", "sf_visual_compress",
    "sf_verify_lm_head_accept_workspace_size", "sf_verify_lm_head_accept",
)

_lock = threading.Lock()
_lib = None


class SFError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(message)
        self.status = status


def library_path() -> str:
    return build_lib.LIB


def load_library(path: str | None = None):
    """Load (once) the compiled library; raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = path or library_path()
        if not os.path.exists(path):
            raise RuntimeError(
                f"{path} is missing: build it with paper_2505_12728_gb300.build_lib.build() "
                "(nvcc for sm_103a); the verification step has no CPU implementation")
        lib = ctypes.CDLL(path)
        P, I, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_float
        S = ctypes.c_size_t
        lib.sf_status_string.argtypes = [I]
        lib.sf_status_string.restype = ctypes.c_char_p
        lib.sf_last_error.argtypes = []
        lib.sf_last_error.restype = ctypes.c_char_p
        lib.sf_version.argtypes = []
        lib.sf_version.restype = I
        lib.sf_workspace_init.argtypes = [P, S, P]
        lib.sf_workspace_init.restype = I
        lib.sf_read_device_status.argtypes = [P, ctypes.POINTER(ctypes.c_uint32)]
        lib.sf_read_device_status.restype = I
        lib.sf_selftest_bounded_wait.argtypes = [P, S, P]
        lib.sf_selftest_bounded_wait.restype = I
        lib.sf_verify_attention_workspace_size.argtypes = [I, I, I, I, I, I, I, I]
        lib.sf_verify_attention_workspace_size.restype = S
        lib.sf_verify_attention.argtypes = [P, P, P, P, P, I, I, I, I, I, I, I, I, F, I, P, P, P,
                                            S, P]
        lib.sf_verify_attention.restype = I
        lib.sf_verify_attention_noalloc.argtypes = [P, P, P, P, P, I, I, I, I, I, I, I, I, F, I,
                                                    P, P, P]
        lib.sf_verify_attention_noalloc.restype = I
        lib.sf_verify_attention_kernel_launches.argtypes = [I] * 8
        lib.sf_verify_attention_kernel_launches.restype = I
        lib.sf_accept_workspace_size.argtypes = [I, I, I]
        lib.sf_accept_workspace_size.restype = S
        lib.sf_accept_kernel_launches.argtypes = [I, I, I]
        lib.sf_accept_kernel_launches.restype = I
        lib.sf_accept.argtypes = [P, P, P, P, P, I, I, I, P, P, P, P, S, P]
        lib.sf_accept.restype = I
        lib.sf_kv_commit_workspace_size.argtypes = []
        lib.sf_kv_commit_workspace_size.restype = S
        lib.sf_kv_commit.argtypes = [P, P, P, P, P, I, I, I, I, I, I, P, S, P]
        lib.sf_kv_commit.restype = I
        lib.sf_draft_tail_workspace_size.argtypes = [I, I]
        lib.sf_draft_tail_workspace_size.restype = S
        lib.sf_lm_head.argtypes = [P, P, I, I, I, P, P, S, P]
        lib.sf_lm_head.restype = I
        lib.sf_sample.argtypes = [P, P, P, I, I, P, P, P, S, P]
        lib.sf_sample.restype = I
        lib.sf_draft_sample.argtypes = [P, P, P, P, I, I, I, P, P, P, P, S, P]
        lib.sf_draft_sample.restype = I
        lib.sf_visual_compress_workspace_size.argtypes = [I, I, I, I]
        lib.sf_visual_compress_workspace_size.restype = S
        lib.sf_visual_compress.argtypes = [P, P, I, I, I, I, P, P, S, P]
        lib.sf_visual_compress.restype = I
        lib.sf_verify_lm_head_accept_workspace_size.argtypes = [I, I, I]
        lib.sf_verify_lm_head_accept_workspace_size.restype = S
        lib.sf_verify_lm_head_accept.argtypes = [P, P, P, P, P, P, I, I, I, I, P, P, P, P, P, S, P]
        lib.sf_verify_lm_head_accept.restype = I
        _lib = lib
        return lib


def _check(status: int):
    if status != SF_OK:
        lib = load_library()
        raise SFError(status, f"{lib.sf_status_string(status).decode()}: "
                              f"{lib.sf_last_error().decode()}")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream_handle(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need_workspace(workspace):
    """A caller-supplied workspace must be a contiguous uint8 CUDA tensor (its
    numel() is the byte count passed to the library)."""
    _need(workspace, "workspace", torch.uint8)


def _need(t, name, dtype, shape=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")


# --------------------------------------------------------------------------- #
# workspaces                                                                  #
# --------------------------------------------------------------------------- #
def verify_attention_workspace_size(B, n_q, H_q, H_kv, head_dim, max_pages_per_seq,
                                    page_size=PAGE_SIZE, num_splits=0) -> int:
    n = load_library().sf_verify_attention_workspace_size(B, n_q, H_q, H_kv, head_dim,
                                                          max_pages_per_seq, page_size,
                                                          num_splits)
    if n == 0:
        raise SFError(1, "invalid verify-attention shape: " + load_library().sf_last_error().decode())
    return int(n)


def accept_workspace_size(B, k, V) -> int:
    n = load_library().sf_accept_workspace_size(B, k, V)
    if n == 0:
        raise SFError(1, "invalid acceptance shape: " + load_library().sf_last_error().decode())
    return int(n)


def verify_attention_kernel_launches(B, n_q, H_q, H_kv, head_dim, max_pages_per_seq,
                                     num_splits=0) -> int:
    """Kernels one verify_attention call with these shapes launches (1 or 2)."""
    n = load_library().sf_verify_attention_kernel_launches(B, n_q, H_q, H_kv, head_dim,
                                                           max_pages_per_seq, PAGE_SIZE, num_splits)
    if n == 0:
        raise SFError(1, "no attention launch plan: " + load_library().sf_last_error().decode())
    return int(n)


def accept_kernel_launches(B, k, V) -> int:
    """Kernels one accept call with these shapes launches (1 or 2)."""
    n = load_library().sf_accept_kernel_launches(B, k, V)
    if n == 0:
        raise SFError(1, "no acceptance launch plan: " + load_library().sf_last_error().decode())
    return int(n)


def new_workspace(nbytes: int, device=None) -> torch.Tensor:
    """A zero-filled uint8 device buffer (the library's counters start at 0)."""
    return torch.zeros(int(nbytes), dtype=torch.uint8, device=device or "cuda")


def workspace_init(workspace: torch.Tensor, stream=None):
    _need_workspace(workspace)
    _check(load_library().sf_workspace_init(_ptr(workspace), workspace.numel(),
                                            _stream_handle(stream)))


def read_device_status(workspace: torch.Tensor) -> int:
    _need_workspace(workspace)
    v = ctypes.c_uint32(0)
    _check(load_library().sf_read_device_status(_ptr(workspace), ctypes.byref(v)))
    return int(v.value)


def selftest_bounded_wait(workspace: torch.Tensor, stream=None) -> None:
    """sf_selftest_bounded_wait: a wait that nothing completes gives up after
    about a second and sets SF_DEVICE_TIMEOUT in the workspace's status word
    (read it with read_device_status)."""
    _need_workspace(workspace)
    _check(load_library().sf_selftest_bounded_wait(_ptr(workspace), workspace.numel(),
                                                   _stream_handle(stream)))


# --------------------------------------------------------------------------- #
# verification attention                                                      #
# --------------------------------------------------------------------------- #
def verify_attention(q, k_cache, v_cache, block_table, seq_lens, *, out=None, lse=None,
                     workspace=None, softmax_scale=0.0, num_splits=0, stream=None,
                     with_lse=True):
    """sf_verify_attention: q bf16 [B][n_q][H_q][d]; k/v_cache bf16
    [pages][H_kv][16][d]; block_table int32 [B][max_pages]; seq_lens int32 [B]
    (prefix + n_q).  Returns (out bf16 [B][n_q][H_q][d], lse fp32 [B][n_q][H_q]
    or None)."""
    B, n_q, H_q, d = q.shape
    num_pages, H_kv, page, d2 = k_cache.shape
    if block_table.dim() != 2 or block_table.shape[0] != B:
        raise ValueError(f"block_table has shape {tuple(block_table.shape)}, expected ({B}, max_pages)")
    if d2 != d:
        raise ValueError("head_dim of q and caches differ")
    _need(q, "q", torch.bfloat16)
    _need(k_cache, "k_cache", torch.bfloat16)
    _need(v_cache, "v_cache", torch.bfloat16, k_cache.shape)
    _need(block_table, "block_table", torch.int32)
    _need(seq_lens, "seq_lens", torch.int32, (B,))
    max_pages = block_table.shape[1]
    if out is None:
        out = torch.empty_like(q)
    _need(out, "out", torch.bfloat16, q.shape)
    if lse is None and with_lse:
        lse = torch.empty((B, n_q, H_q), dtype=torch.float32, device=q.device)
    if lse is not None:
        _need(lse, "lse", torch.float32, (B, n_q, H_q))
    if workspace is None:
        workspace = new_workspace(verify_attention_workspace_size(
            B, n_q, H_q, H_kv, d, max_pages, page, num_splits), q.device)
    _need_workspace(workspace)
    _check(load_library().sf_verify_attention(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(seq_lens), B, n_q, H_q,
        H_kv, d, page, num_pages, max_pages, float(softmax_scale), int(num_splits), _ptr(out),
        _ptr(lse), _ptr(workspace), workspace.numel(), _stream_handle(stream)))
    return out, lse


def verify_attention_noalloc(q, k_cache, v_cache, block_table, seq_lens, *, out=None, lse=None,
                             softmax_scale=0.0, num_splits=0, stream=None, with_lse=True):
    """sf_verify_attention_noalloc: the same computation as verify_attention
    for callers that cannot allocate device memory while verifying; the
    library's own 16 MiB device scratch replaces the workspace (calls that
    overlap on the GPU race on it).  Outputs may still be allocated here when
    not supplied."""
    B, n_q, H_q, d = q.shape
    num_pages, H_kv, page, d2 = k_cache.shape
    if block_table.dim() != 2 or block_table.shape[0] != B:
        raise ValueError(f"block_table has shape {tuple(block_table.shape)}, expected ({B}, max_pages)")
    if d2 != d:
        # the library sizes the caches' tensor maps from q's head_dim: a
        # narrower cache would let the copies read past its end
        raise ValueError("head_dim of q and caches differ")
    _need(q, "q", torch.bfloat16)
    _need(k_cache, "k_cache", torch.bfloat16)
    _need(v_cache, "v_cache", torch.bfloat16, k_cache.shape)
    _need(block_table, "block_table", torch.int32)
    _need(seq_lens, "seq_lens", torch.int32, (B,))
    if out is None:
        out = torch.empty_like(q)
    _need(out, "out", torch.bfloat16, q.shape)
    if lse is None and with_lse:
        lse = torch.empty((B, n_q, H_q), dtype=torch.float32, device=q.device)
    if lse is not None:
        _need(lse, "lse", torch.float32, (B, n_q, H_q))
    _check(load_library().sf_verify_attention_noalloc(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(block_table), _ptr(seq_lens), B, n_q, H_q,
        H_kv, d, page, num_pages, block_table.shape[1], float(softmax_scale), int(num_splits),
        _ptr(out), _ptr(lse), _stream_handle(stream)))
    return out, lse


# --------------------------------------------------------------------------- #
# acceptance                                                                  #
# --------------------------------------------------------------------------- #
def accept(target_logits, draft_probs, draft_tokens, uniforms, temperature, *,
           num_accepted=None, out_tokens=None, accept_ratio=None, workspace=None, stream=None,
           with_ratio=True):
    """sf_accept: target_logits fp32 [B][k+1][V], draft_probs fp32 [B][k][V],
    draft_tokens int32 [B][k], uniforms fp32 [B][k+1], temperature fp32 [B]
    (<= 0 greedy).  Returns (num_accepted int32 [B], out_tokens int32 [B][k+1],
    accept_ratio fp32 [B][k] or None)."""
    B, k1, V = target_logits.shape
    k = k1 - 1
    _need(target_logits, "target_logits", torch.float32)
    _need(draft_probs, "draft_probs", torch.float32, (B, k, V))
    _need(draft_tokens, "draft_tokens", torch.int32, (B, k))
    _need(uniforms, "uniforms", torch.float32, (B, k + 1))
    _need(temperature, "temperature", torch.float32, (B,))
    dev = target_logits.device
    if num_accepted is None:
        num_accepted = torch.empty(B, dtype=torch.int32, device=dev)
    if out_tokens is None:
        out_tokens = torch.empty((B, k + 1), dtype=torch.int32, device=dev)
    if accept_ratio is None and with_ratio:
        accept_ratio = torch.empty((B, k), dtype=torch.float32, device=dev)
    _need(num_accepted, "num_accepted", torch.int32, (B,))
    _need(out_tokens, "out_tokens", torch.int32, (B, k + 1))
    if accept_ratio is not None:
        _need(accept_ratio, "accept_ratio", torch.float32, (B, k))
    if workspace is None:
        workspace = new_workspace(accept_workspace_size(B, k, V), dev)
    _need_workspace(workspace)
    _check(load_library().sf_accept(
        _ptr(target_logits), _ptr(draft_probs), _ptr(draft_tokens), _ptr(uniforms),
        _ptr(temperature), B, k, V, _ptr(num_accepted), _ptr(out_tokens), _ptr(accept_ratio),
        _ptr(workspace), workspace.numel(), _stream_handle(stream)))
    return num_accepted, out_tokens, accept_ratio


def verify_lm_head_accept_workspace_size(B, k, V) -> int:
    n = load_library().sf_verify_lm_head_accept_workspace_size(B, k, V)
    if n == 0:
        raise SFError(1, "invalid fused acceptance shape")
    return int(n)


def verify_lm_head_accept(hidden, weight, draft_probs, draft_tokens, uniforms, temperature, *,
                          logits=None, num_accepted=None, out_tokens=None, accept_ratio=None,
                          workspace=None, stream=None, with_ratio=True):
    """sf_verify_lm_head_accept: hidden bf16 [B][k+1][d] (the target's final
    hidden states of the verified positions), weight bf16 [V][d], then the
    acceptance rule as in accept().  Returns (logits fp32 [B][k+1][V],
    num_accepted int32 [B], out_tokens int32 [B][k+1], accept_ratio or None)."""
    B, k1, d = hidden.shape
    k = k1 - 1
    V = weight.shape[0]
    _need(hidden, "hidden", torch.bfloat16)
    _need(weight, "weight", torch.bfloat16, (V, d))
    _need(draft_probs, "draft_probs", torch.float32, (B, k, V))
    _need(draft_tokens, "draft_tokens", torch.int32, (B, k))
    _need(uniforms, "uniforms", torch.float32, (B, k + 1))
    _need(temperature, "temperature", torch.float32, (B,))
    dev = hidden.device
    if logits is None:
        logits = torch.empty((B, k + 1, V), dtype=torch.float32, device=dev)
    if num_accepted is None:
        num_accepted = torch.empty(B, dtype=torch.int32, device=dev)
    if out_tokens is None:
        out_tokens = torch.empty((B, k + 1), dtype=torch.int32, device=dev)
    if accept_ratio is None and with_ratio:
        accept_ratio = torch.empty((B, k), dtype=torch.float32, device=dev)
    _need(logits, "logits", torch.float32, (B, k + 1, V))
    _need(num_accepted, "num_accepted", torch.int32, (B,))
    _need(out_tokens, "out_tokens", torch.int32, (B, k + 1))
    if accept_ratio is not None:
        _need(accept_ratio, "accept_ratio", torch.float32, (B, k))
    if workspace is None:
        workspace = new_workspace(verify_lm_head_accept_workspace_size(B, k, V), dev)
    _need_workspace(workspace)
    _check(load_library().sf_verify_lm_head_accept(
        _ptr(hidden), _ptr(weight), _ptr(draft_probs), _ptr(draft_tokens), _ptr(uniforms),
        _ptr(temperature), B, k, V, d, _ptr(logits), _ptr(num_accepted), _ptr(out_tokens),
        _ptr(accept_ratio), _ptr(workspace), workspace.numel(), _stream_handle(stream)))
    return logits, num_accepted, out_tokens, accept_ratio


def kv_commit_workspace_size() -> int:
    return int(load_library().sf_kv_commit_workspace_size())


def kv_commit(seq_lens, block_table, free_pages, free_count, num_accepted, n_q, n_q_next, *,
              workspace=None, stream=None):
    """sf_kv_commit, in place: seq_lens int32 [B], block_table int32
    [B][max_pages], free_pages int32 [capacity] (a stack of free page ids),
    free_count int32 [1], num_accepted int32 [B] (from accept).  Keeps the
    first min(a + 1, n_q) verified rows of each sequence, prepares seq_lens
    for the next n_q_next rows and maps exactly their pages."""
    B, max_pages = block_table.shape
    _need(seq_lens, "seq_lens", torch.int32, (B,))
    _need(block_table, "block_table", torch.int32)
    _need(free_pages, "free_pages", torch.int32)
    _need(free_count, "free_count", torch.int32, (1,))
    _need(num_accepted, "num_accepted", torch.int32, (B,))
    if workspace is None:
        workspace = new_workspace(kv_commit_workspace_size(), seq_lens.device)
    _need_workspace(workspace)
    _check(load_library().sf_kv_commit(
        _ptr(seq_lens), _ptr(block_table), _ptr(free_pages), _ptr(free_count), _ptr(num_accepted),
        B, n_q, n_q_next, max_pages, PAGE_SIZE, free_pages.numel(), _ptr(workspace),
        workspace.numel(), _stream_handle(stream)))


# --------------------------------------------------------------------------- #
# draft-distribution tail                                                     #
# --------------------------------------------------------------------------- #
def draft_tail_workspace_size(R, V) -> int:
    n = load_library().sf_draft_tail_workspace_size(R, V)
    if n == 0:
        raise SFError(1, "invalid draft-tail shape: " + load_library().sf_last_error().decode())
    return int(n)


def lm_head(hidden, weight, *, logits=None, workspace=None, stream=None):
    """sf_lm_head: hidden bf16 [R][hidden_size], weight bf16 [V][hidden_size].
    Returns logits fp32 [R][V] = hidden @ weight^T."""
    R, Hd = hidden.shape
    V = weight.shape[0]
    _need(hidden, "hidden", torch.bfloat16)
    _need(weight, "weight", torch.bfloat16, (V, Hd))
    if logits is None:
        logits = torch.empty((R, V), dtype=torch.float32, device=hidden.device)
    _need(logits, "logits", torch.float32, (R, V))
    if workspace is None:
        workspace = new_workspace(draft_tail_workspace_size(R, V), hidden.device)
    _need_workspace(workspace)
    _check(load_library().sf_lm_head(_ptr(hidden), _ptr(weight), R, Hd, V, _ptr(logits),
                                     _ptr(workspace), workspace.numel(), _stream_handle(stream)))
    return logits


def sample(logits, uniforms, temperature, *, probs=None, tokens=None, workspace=None,
           stream=None):
    """sf_sample: logits fp32 [R][V], uniforms fp32 [R], temperature fp32 [R]
    (<= 0 greedy).  Returns (probs fp32 [R][V], tokens int32 [R])."""
    R, V = logits.shape
    _need(logits, "logits", torch.float32)
    _need(uniforms, "uniforms", torch.float32, (R,))
    _need(temperature, "temperature", torch.float32, (R,))
    dev = logits.device
    if probs is None:
        probs = torch.empty((R, V), dtype=torch.float32, device=dev)
    if tokens is None:
        tokens = torch.empty(R, dtype=torch.int32, device=dev)
    _need(probs, "probs", torch.float32, (R, V))
    _need(tokens, "tokens", torch.int32, (R,))
    if workspace is None:
        workspace = new_workspace(draft_tail_workspace_size(R, V), dev)
    _need_workspace(workspace)
    _check(load_library().sf_sample(_ptr(logits), _ptr(uniforms), _ptr(temperature), R, V,
                                    _ptr(probs), _ptr(tokens), _ptr(workspace), workspace.numel(),
                                    _stream_handle(stream)))
    return probs, tokens


def draft_sample(hidden, weight, uniforms, temperature, *, logits=None, probs=None, tokens=None,
                 workspace=None, stream=None):
    """sf_draft_sample: the LM-head projection and sampling of the draft
    rows in two launches.  Returns (logits fp32 [R][V], probs fp32 [R][V],
    tokens int32 [R])."""
    R, Hd = hidden.shape
    V = weight.shape[0]
    _need(hidden, "hidden", torch.bfloat16)
    _need(weight, "weight", torch.bfloat16, (V, Hd))
    _need(uniforms, "uniforms", torch.float32, (R,))
    _need(temperature, "temperature", torch.float32, (R,))
    dev = hidden.device
    if logits is None:
        logits = torch.empty((R, V), dtype=torch.float32, device=dev)
    if probs is None:
        probs = torch.empty((R, V), dtype=torch.float32, device=dev)
    if tokens is None:
        tokens = torch.empty(R, dtype=torch.int32, device=dev)
    _need(logits, "logits", torch.float32, (R, V))
    _need(probs, "probs", torch.float32, (R, V))
    _need(tokens, "tokens", torch.int32, (R,))
    if workspace is None:
        workspace = new_workspace(draft_tail_workspace_size(R, V), dev)
    _need_workspace(workspace)
    _check(load_library().sf_draft_sample(
        _ptr(hidden), _ptr(weight), _ptr(uniforms), _ptr(temperature), R, Hd, V, _ptr(logits),
        _ptr(probs), _ptr(tokens), _ptr(workspace), workspace.numel(), _stream_handle(stream)))
    return logits, probs, tokens


# --------------------------------------------------------------------------- #
# visual token compression                                                    #
# --------------------------------------------------------------------------- #
def visual_compress_workspace_size(F, N, C, d) -> int:
    n = load_library().sf_visual_compress_workspace_size(F, N, C, d)
    if n == 0:
        raise SFError(1, "invalid compressor shape")
    return int(n)


def visual_compress(queries, features, *, out=None, workspace=None, stream=None):
    """sf_visual_compress: queries bf16 [C][d], features bf16 [F][N][d].
    Returns out bf16 [F][C][d] = softmax(Q F_V^T) F_V per frame."""
    C, d = queries.shape
    F, N, d2 = features.shape
    _need(queries, "queries", torch.bfloat16)
    _need(features, "features", torch.bfloat16)
    if d2 != d:
        raise ValueError("queries and features differ in d")
    if out is None:
        out = torch.empty((F, C, d), dtype=torch.bfloat16, device=queries.device)
    _need(out, "out", torch.bfloat16, (F, C, d))
    if workspace is None:
        workspace = new_workspace(visual_compress_workspace_size(F, N, C, d), queries.device)
    _need_workspace(workspace)
    _check(load_library().sf_visual_compress(_ptr(queries), _ptr(features), F, N, C, d, _ptr(out),
                                             _ptr(workspace), workspace.numel(),
                                             _stream_handle(stream)))
    return out
