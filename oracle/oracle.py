"""ctypes front end of the fp64 CPU oracle (``specflash_oracle.c``).

TEST INFRASTRUCTURE ONLY.  The test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` are the only callers.  The product package
never imports this module, and this module imports nothing from the product
package: the oracle and the CUDA path share no code.

Each function states the passage of arXiv 2505.12728 it follows; the C file
holds the arithmetic.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "specflash_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "libspecflash_oracle.so")
# A prebuilt oracle library to load instead (used by the mutation test, which
# checks that the pins reject deliberately broken copies of the oracle).
_LIB_OVERRIDE = os.environ.get("SPECFLASH_ORACLE_LIB")

ORACLE_OK = 0
ORACLE_ERR_ARG = 1
ORACLE_ERR_BAD_PAGE = 2
ORACLE_ERR_BAD_TOKEN = 3

_lock = threading.Lock()
_lib = None


class OracleError(RuntimeError):
    pass


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP, no -ffast-math)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-fno-fast-math", "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(_LIB_OVERRIDE if _LIB_OVERRIDE else build())
        P = ctypes.c_void_p
        I = ctypes.c_int
        D = ctypes.c_double
        lib.oracle_decode_attention.argtypes = [P, P, P, I, I, D, P, P]
        lib.oracle_decode_attention.restype = I
        lib.oracle_verify_attention.argtypes = [P, P, P, P, P, I, I, I, I, I, I, I, I, D,
                                                I, I, I, P, P]
        lib.oracle_verify_attention.restype = I
        lib.oracle_target_probs.argtypes = [P, I, D, P]
        lib.oracle_target_probs.restype = I
        lib.oracle_argmax.argtypes = [P, I]
        lib.oracle_argmax.restype = I
        lib.oracle_accept.argtypes = [P, P, P, P, P, I, I, I, P, P, P, P]
        lib.oracle_accept.restype = I
        lib.oracle_kv_commit.argtypes = [P, P, P, P, P, I, I, I, I, I, I]
        lib.oracle_kv_commit.restype = I
        lib.oracle_sample.argtypes = [P, P, P, I, I, P, P, P]
        lib.oracle_sample.restype = I
        lib.oracle_visual_compress.argtypes = [P, P, I, I, I, I, P]
        lib.oracle_visual_compress.restype = I
        lib.oracle_set_threads.argtypes = [I]
        lib.oracle_set_threads.restype = None
        _lib = lib
        return lib


def set_threads(n: int) -> None:
    """Threads of the oracle's OpenMP loops (n <= 0: all host cores).  The
    results do not depend on it."""
    _load().oracle_set_threads(int(n))


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def decode_attention(q, k, v, scale):
    """One query row against T contiguous keys (Sec. 3.1; the K = 1 case of
    the draft-length ablation).  q [d], k/v [T][d] float64 -> (o [d], lse)."""
    lib = _load()
    q = _c(q, np.float64)
    k = _c(k, np.float64)
    v = _c(v, np.float64)
    T, d = k.shape
    o = np.zeros(d, np.float64)
    lse = np.zeros(1, np.float64)
    st = lib.oracle_decode_attention(_ptr(q), _ptr(k), _ptr(v), T, d, float(scale), _ptr(o),
                                     _ptr(lse))
    if st != ORACLE_OK:
        raise OracleError(f"oracle_decode_attention status {st}")
    return o, float(lse[0])


def verify_attention(q_bits, k_bits, v_bits, block_table, seq_lens, H_kv, page_size=16,
                     scale=0.0, select=(-1, -1, -1)):
    """Verification attention over the paged cache (Sec. 3.1: the K candidates
    are scored in one forward pass against the cached visual and text tokens).

    q_bits [B][n_q][H_q][d] uint16 (bf16 bits); k_bits/v_bits
    [num_pages][H_kv][page_size][d] uint16; block_table [B][max_pages] int32;
    seq_lens [B] int32 (prefix + n_q).  ``select`` = (b, i, h) restricts the
    computation to matching rows (-1 = all); other rows are returned as NaN.
    Returns (out float64 [B][n_q][H_q][d], lse float64 [B][n_q][H_q]).
    """
    lib = _load()
    q_bits = _c(q_bits, np.uint16)
    k_bits = _c(k_bits, np.uint16)
    v_bits = _c(v_bits, np.uint16)
    block_table = _c(block_table, np.int32)
    seq_lens = _c(seq_lens, np.int32)
    B, n_q, H_q, d = q_bits.shape
    num_pages = k_bits.shape[0]
    assert k_bits.shape == (num_pages, H_kv, page_size, d), k_bits.shape
    assert v_bits.shape == k_bits.shape
    max_pages = block_table.shape[1]
    out = np.full((B, n_q, H_q, d), np.nan, np.float64)
    lse = np.full((B, n_q, H_q), np.nan, np.float64)
    st = lib.oracle_verify_attention(_ptr(q_bits), _ptr(k_bits), _ptr(v_bits),
                                     _ptr(block_table), _ptr(seq_lens), B, n_q, H_q, H_kv, d,
                                     page_size, num_pages, max_pages, float(scale),
                                     int(select[0]), int(select[1]), int(select[2]),
                                     _ptr(out), _ptr(lse))
    if st != ORACLE_OK:
        raise OracleError(f"oracle_verify_attention status {st}")
    return out, lse


def target_probs(logits, tau):
    """p = softmax(logits / tau) in fp64 (Sec. 3.1: the target distribution
    P_i of a verified position; tau as in Sec. 4.2)."""
    lib = _load()
    logits = _c(logits, np.float32)
    p = np.zeros(logits.shape[0], np.float64)
    st = lib.oracle_target_probs(_ptr(logits), logits.shape[0], float(tau), _ptr(p))
    if st != ORACLE_OK:
        raise OracleError(f"oracle_target_probs status {st}")
    return p


def argmax(logits):
    """Greedy decoding's choice (tau = 0, Sec. 4.2): first maximal index."""
    lib = _load()
    logits = _c(logits, np.float32)
    return int(lib.oracle_argmax(_ptr(logits), logits.shape[0]))


def accept(target_logits, draft_probs, draft_tokens, uniforms, temperature):
    """Token-wise acceptance-rejection over a batch (Sec. 3.1 and Sec. 3.3).

    target_logits [B][k+1][V] fp32, draft_probs [B][k][V] fp32, draft_tokens
    [B][k] int32, uniforms [B][k+1] fp32, temperature [B] fp32 (<= 0 greedy).
    Returns dict(num_accepted [B] int32, out_tokens [B][k+1] int32,
    accept_ratio [B][k] float64, margin [B][k+1] float64).
    """
    lib = _load()
    target_logits = _c(target_logits, np.float32)
    draft_probs = _c(draft_probs, np.float32)
    draft_tokens = _c(draft_tokens, np.int32)
    uniforms = _c(uniforms, np.float32)
    temperature = _c(temperature, np.float32)
    B, k1, V = target_logits.shape
    k = k1 - 1
    assert draft_probs.shape == (B, k, V)
    assert draft_tokens.shape == (B, k)
    assert uniforms.shape == (B, k + 1)
    assert temperature.shape == (B,)
    num_accepted = np.zeros(B, np.int32)
    out_tokens = np.zeros((B, k + 1), np.int32)
    ratio = np.zeros((B, k), np.float64)
    margin = np.zeros((B, k + 1), np.float64)
    st = lib.oracle_accept(_ptr(target_logits), _ptr(draft_probs), _ptr(draft_tokens),
                           _ptr(uniforms), _ptr(temperature), B, k, V, _ptr(num_accepted),
                           _ptr(out_tokens), _ptr(ratio), _ptr(margin))
    if st != ORACLE_OK:
        raise OracleError(f"oracle_accept status {st}")
    return dict(num_accepted=num_accepted, out_tokens=out_tokens, accept_ratio=ratio,
                margin=margin)


ORACLE_ERR_PAGES = 5


def kv_commit(seq_lens, block_table, free_pages, free_count, num_accepted, n_q, n_q_next,
              page_size=16):
    """Cache bookkeeping after acceptance (Sec. 3.1, Sec. 3.3): keep the first
    min(a + 1, n_q) verified rows of each sequence, set seq_lens for the next
    n_q_next rows and map exactly their pages through the free-page stack.

    seq_lens [B] int32, block_table [B][max_pages] int32, free_pages
    [capacity] int32 (entries [0, free_count) are free pages), num_accepted
    [B] int32.  Inputs are not modified.  Returns (status, seq_lens,
    block_table, free_pages, free_count); status is ORACLE_OK,
    ORACLE_ERR_ARG or ORACLE_ERR_PAGES, and on an error the returned arrays
    equal the inputs.
    """
    lib = _load()
    sl = np.array(seq_lens, dtype=np.int32, copy=True, order="C")
    bt = np.array(block_table, dtype=np.int32, copy=True, order="C")
    fp = np.array(free_pages, dtype=np.int32, copy=True, order="C")
    fc = np.array([int(free_count)], dtype=np.int32)
    na = _c(num_accepted, np.int32)
    B, max_pages = bt.shape
    assert sl.shape == (B,) and na.shape == (B,)
    st = lib.oracle_kv_commit(_ptr(sl), _ptr(bt), _ptr(fp), _ptr(fc), _ptr(na), B, n_q, n_q_next,
                              max_pages, page_size, fp.shape[0])
    return int(st), sl, bt, fp, int(fc[0])


def sample(logits, uniforms, temperature):
    """Draft-tail sampling (Algorithm 1): P' = softmax(logits / tau) per row,
    T' by inverse CDF with the row's uniform (ascending token id, strict <);
    tau <= 0: first argmax, one-hot P'.  logits [R][V] fp32, uniforms [R]
    fp32, temperature [R] fp32.  Returns (probs [R][V] float64, tokens [R]
    int32, margin [R] float64: distance of each draw to the nearest CDF
    boundary)."""
    lib = _load()
    logits = _c(logits, np.float32)
    uniforms = _c(uniforms, np.float32)
    temperature = _c(temperature, np.float32)
    R, V = logits.shape
    assert uniforms.shape == (R,) and temperature.shape == (R,)
    probs = np.zeros((R, V), np.float64)
    tokens = np.zeros(R, np.int32)
    margin = np.zeros(R, np.float64)
    st = lib.oracle_sample(_ptr(logits), _ptr(uniforms), _ptr(temperature), R, V, _ptr(probs),
                           _ptr(tokens), _ptr(margin))
    if st != ORACLE_OK:
        raise OracleError(f"oracle_sample status {st}")
    return probs, tokens, margin


def lm_head_logits(hidden_bits, weight_bits):
    """LM-head projection (Algorithm 1, the step before sampling): logits =
    H W^T in float64 from bf16 hidden states H [R][hidden] and weights W
    [V][hidden] (bf16 bit patterns, uint16), decoded exactly.  A library
    matrix product is the only step."""
    h = _bf16_to_f64(np.asarray(hidden_bits, np.uint16))
    w = _bf16_to_f64(np.asarray(weight_bits, np.uint16))
    return h @ w.T


def visual_compress(query_bits, feature_bits):
    """Visual token compression (Sec. 3.2, Eq. 3; Algorithm 1):
    F^_V = softmax(Q F_V^T) F_V for each of the F frames, the softmax over the
    frame's N tokens, unscaled scores.  query_bits bf16 bits [C][d],
    feature_bits bf16 bits [F][N][d] (uint16).  Returns [F][C][d] float64."""
    lib = _load()
    q = _c(query_bits, np.uint16)
    f = _c(feature_bits, np.uint16)
    if f.ndim == 2:
        f = f[None]
    C, d = q.shape
    F, N, d2 = f.shape
    assert d2 == d
    out = np.zeros((F, C, d), np.float64)
    st = lib.oracle_visual_compress(_ptr(q), _ptr(f), F, N, C, d, _ptr(out))
    if st != ORACLE_OK:
        raise OracleError(f"oracle_visual_compress status {st}")
    return out


def _bf16_to_f64(bits):
    return (np.asarray(bits, np.uint32) << 16).view(np.float32).astype(np.float64)
