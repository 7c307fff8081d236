"""Seeded synthetic inputs for the verification step.

This module is the one place that both the CUDA path's tests/benchmark and the
CPU oracle draw their inputs from.  It holds none of the verification method's
arithmetic: it only draws random numbers (numpy PCG64, platform independent)
and lays them out.  The draft distribution q and the draft tokens belong to
the draft model, which is outside the verification step, so they are produced
here as inputs (a softmax of noisy target logits and a categorical draw, as the
draft head of Algorithm 1 samples its candidates).

The five named workloads follow the shapes of the paper's image- and
video-LMM settings: 576 visual tokens per LLaVA image (Sec. 4.2), QwenVL
images at 324 tokens, video as frames of 144 visual tokens, vocabularies of
32000 (LLaVA) and 152064 (QwenVL).  Q/K/V are N(0,1) rounded to bf16; target
logits are N(0, 3^2) in fp32; uniforms are U[0,1) in fp32; the physical page
order in the KV pool is a seeded random permutation.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

PAGE_SIZE = 16


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H_q: int
    H_kv: int
    d: int
    k: int                      # draft length K
    V: int                      # vocabulary size
    prefix: tuple               # ("fixed", L) or ("uniform", lo, hi): cached tokens before the draft block
    layers: int = 1             # independent attention layers per verification step
    mode: str = "sampling"      # "sampling" | "greedy" | "alternate" (even b greedy, odd b sampling)
    draft_sharpness: float = 1.0  # q = softmax(sharpness * logits + N(0,1))
    seed: int = 0
    n_q: int = 0                # attention rows per sequence; 0 means k
    logit_std: float = 3.0
    description: str = field(default="", compare=False)

    @property
    def rows(self) -> int:
        return self.n_q if self.n_q > 0 else self.k

    @property
    def group(self) -> int:
        return self.H_q // self.H_kv


WORKLOADS = {
    "tiny": Workload(
        "tiny", B=1, H_q=8, H_kv=8, d=64, k=4, V=32000, prefix=("fixed", 640),
        mode="sampling", seed=0,
        description="B1, 8/8 heads MHA, d64, prefix 640 (576 visual + 64 text), k4, V32000"),
    "image7b": Workload(
        "image7b", B=1, H_q=32, H_kv=32, d=128, k=5, V=32000, prefix=("fixed", 3008),
        layers=32, mode="sampling", seed=1,
        description="B1, 32 layers, 32/32 heads MHA, d128, prefix 3008 (5x576 visual + 128 text), "
                    "k5, V32000, sampling at tau=1"),
    "gqa": Workload(
        "gqa", B=8, H_q=28, H_kv=4, d=128, k=6, V=152064, prefix=("uniform", 1200, 3600),
        mode="alternate", seed=2,
        description="B8, 28/4 heads GQA, d128, prefix U[1200,3600], k6, V152064, "
                    "even sequences greedy, odd sampling"),
    "video": Workload(
        "video", B=4, H_q=28, H_kv=4, d=128, k=8, V=152064, prefix=("fixed", 4864),
        mode="sampling", draft_sharpness=1.5, seed=3,
        description="B4, 28/4 heads GQA, d128, prefix 4864 (32x144 visual + 256 text), k8, "
                    "V152064, q = softmax(1.5*logits + noise)"),
    "long": Workload(
        "long", B=16, H_q=28, H_kv=4, d=128, k=8, V=152064, prefix=("uniform", 8192, 32768),
        mode="sampling", seed=4,
        description="B16, 28/4 heads GQA, d128, prefix U[8192,32768], k in {2,4,8}, V152064"),
}


def workload(name: str, **overrides) -> Workload:
    return replace(WORKLOADS[name], **overrides)


# --------------------------------------------------------------------------- #
# bf16 helpers (layout only: round-to-nearest-even of fp32 draws to bf16 bits) #
# --------------------------------------------------------------------------- #
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32)
    rounding = ((u >> 16) & 1) + np.uint32(0x7FFF)
    return ((u + rounding) >> 16).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _normal_bf16(rng: np.random.Generator, shape) -> np.ndarray:
    n = int(np.prod(shape))
    out = np.empty(n, np.uint16)
    chunk = 1 << 24
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        out[s:e] = f32_to_bf16_bits(rng.standard_normal(e - s, dtype=np.float32))
    return out.reshape(shape)


# --------------------------------------------------------------------------- #
# attention inputs                                                            #
# --------------------------------------------------------------------------- #
def prefix_lengths(wl: Workload, rng: np.random.Generator) -> np.ndarray:
    if wl.prefix[0] == "fixed":
        return np.full(wl.B, int(wl.prefix[1]), np.int64)
    lo, hi = int(wl.prefix[1]), int(wl.prefix[2])
    return rng.integers(lo, hi + 1, size=wl.B).astype(np.int64)


@dataclass
class AttentionInputs:
    q: np.ndarray            # uint16 [layers][B][n_q][H_q][d]
    k_cache: np.ndarray      # uint16 [layers][num_pages][H_kv][page][d]
    v_cache: np.ndarray      # uint16 [layers][num_pages][H_kv][page][d]
    block_table: np.ndarray  # int32 [layers][B][max_pages]
    seq_lens: np.ndarray     # int32 [B]  (prefix + n_q)
    prefix_lens: np.ndarray  # int64 [B]
    n_q: int
    H_kv: int
    page_size: int = PAGE_SIZE

    @property
    def layers(self) -> int:
        return self.q.shape[0]

    def layer(self, l: int):
        return dict(q=self.q[l], k_cache=self.k_cache[l], v_cache=self.v_cache[l],
                    block_table=self.block_table[l], seq_lens=self.seq_lens)


def make_attention_case(B, n_q, H_q, H_kv, d, prefix_lens, seed, layers=1, page_size=PAGE_SIZE,
                        spare_pages=0, max_pages=None, kv_scale=1.0, q_scale=1.0):
    """Random paged cache for arbitrary shapes.

    Every sequence holds prefix_lens[b] + n_q tokens (the draft rows' K/V are
    already written).  Physical pages of all sequences (plus ``spare_pages``
    never referenced) are a random permutation of the pool; unused block-table
    entries hold -1.
    """
    rng = np.random.default_rng(seed)
    prefix_lens = np.asarray(prefix_lens, np.int64).reshape(B)
    seq_lens = (prefix_lens + n_q).astype(np.int32)
    pages_per_seq = (seq_lens.astype(np.int64) + page_size - 1) // page_size
    need = int(pages_per_seq.sum())
    num_pages = need + int(spare_pages)
    if max_pages is None:
        max_pages = int(pages_per_seq.max())
    q = np.empty((layers, B, n_q, H_q, d), np.uint16)
    kc = np.empty((layers, num_pages, H_kv, page_size, d), np.uint16)
    vc = np.empty_like(kc)
    bt = np.full((layers, B, max_pages), -1, np.int32)
    for l in range(layers):
        perm = rng.permutation(num_pages).astype(np.int32)
        off = 0
        for b in range(B):
            n = int(pages_per_seq[b])
            bt[l, b, :n] = perm[off:off + n]
            off += n
        if q_scale == 1.0:
            q[l] = _normal_bf16(rng, q.shape[1:])
        else:
            q[l] = f32_to_bf16_bits(q_scale * rng.standard_normal(q.shape[1:], dtype=np.float32))
        if kv_scale == 1.0:
            kc[l] = _normal_bf16(rng, kc.shape[1:])
            vc[l] = _normal_bf16(rng, vc.shape[1:])
        else:
            kc[l] = f32_to_bf16_bits(kv_scale * rng.standard_normal(kc.shape[1:], dtype=np.float32))
            vc[l] = f32_to_bf16_bits(kv_scale * rng.standard_normal(vc.shape[1:], dtype=np.float32))
    return AttentionInputs(q=q, k_cache=kc, v_cache=vc, block_table=bt, seq_lens=seq_lens,
                           prefix_lens=prefix_lens, n_q=n_q, H_kv=H_kv, page_size=page_size)


def make_attention_inputs(wl: Workload, seed=None, layers=None) -> AttentionInputs:
    seed = wl.seed if seed is None else seed
    rng = np.random.default_rng([seed, 0xA77])
    L = prefix_lengths(wl, rng)
    return make_attention_case(wl.B, wl.rows, wl.H_q, wl.H_kv, wl.d, L, seed=[seed, 0xCAC4E],
                               layers=wl.layers if layers is None else layers)


# --------------------------------------------------------------------------- #
# acceptance inputs                                                           #
# --------------------------------------------------------------------------- #
@dataclass
class AcceptInputs:
    target_logits: np.ndarray  # fp32 [B][k+1][V]
    draft_probs: np.ndarray    # fp32 [B][k][V]
    draft_tokens: np.ndarray   # int32 [B][k]
    uniforms: np.ndarray       # fp32 [B][k+1]
    temperature: np.ndarray    # fp32 [B]

    @property
    def shape(self):
        B, k1, V = self.target_logits.shape
        return B, k1 - 1, V


def temperatures(mode: str, B: int) -> np.ndarray:
    if mode == "sampling":
        return np.ones(B, np.float32)
    if mode == "greedy":
        return np.zeros(B, np.float32)
    if mode == "alternate":
        return np.where(np.arange(B) % 2 == 0, 0.0, 1.0).astype(np.float32)
    raise ValueError(mode)


def make_accept_case(B, k, V, seed, mode="sampling", draft_sharpness=1.0, logit_std=3.0,
                     noise_std=1.0):
    """Target logits ~ N(0, logit_std^2); the draft distribution is
    q = softmax(draft_sharpness * logits + N(0, noise_std^2)) over the first k
    rows; sampling sequences draw T'_i ~ q_i, greedy sequences take argmax q_i;
    uniforms ~ U[0,1)."""
    rng = np.random.default_rng(seed)
    logits = (logit_std * rng.standard_normal((B, k + 1, V), dtype=np.float32)).astype(np.float32)
    temp = temperatures(mode, B)
    z = draft_sharpness * logits[:, :k, :].astype(np.float64) + \
        noise_std * rng.standard_normal((B, k, V))
    z -= z.max(axis=-1, keepdims=True)
    np.exp(z, out=z)
    z /= z.sum(axis=-1, keepdims=True)
    q = z.astype(np.float32)
    del z
    tokens = np.empty((B, k), np.int32)
    draws = rng.random((B, k))
    for b in range(B):
        for i in range(k):
            if temp[b] > 0:
                c = np.cumsum(q[b, i].astype(np.float64))
                tokens[b, i] = min(int(np.searchsorted(c, draws[b, i] * c[-1], side="right")), V - 1)
            else:
                tokens[b, i] = int(np.argmax(q[b, i]))
    uniforms = rng.random((B, k + 1), dtype=np.float32)
    return AcceptInputs(target_logits=logits, draft_probs=q, draft_tokens=tokens,
                        uniforms=uniforms, temperature=temp)


def make_accept_inputs(wl: Workload, seed=None, mode=None) -> AcceptInputs:
    seed = wl.seed if seed is None else seed
    return make_accept_case(wl.B, wl.k, wl.V, seed=[seed, 0xACC], mode=mode or wl.mode,
                            draft_sharpness=wl.draft_sharpness, logit_std=wl.logit_std)


# --------------------------------------------------------------------------- #
# draft-tail inputs                                                           #
# --------------------------------------------------------------------------- #
# Hidden sizes of the target/draft LM heads: LLaVA-1.5-7B (Vicuna-7B) for the
# 32000-token vocabulary, Qwen2-VL-7B for the 152064-token one.
HIDDEN_SIZES = {32000: 4096, 152064: 3584}


@dataclass
class DraftTailInputs:
    hidden: np.ndarray       # uint16 bf16 bits [R][hidden_size]: draft head outputs
    weight: np.ndarray       # uint16 bf16 bits [V][hidden_size]: the LM head
    uniforms: np.ndarray     # fp32 [R]
    temperature: np.ndarray  # fp32 [R]

    @property
    def shape(self):
        return self.hidden.shape[0], self.hidden.shape[1], self.weight.shape[0]


def _scaled_normal_bf16(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    n = int(np.prod(shape))
    out = np.empty(n, np.uint16)
    chunk = 1 << 24
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        out[s:e] = f32_to_bf16_bits(np.float32(std) * rng.standard_normal(e - s, dtype=np.float32))
    return out.reshape(shape)


def _small_int_bf16(rng: np.random.Generator, shape, scale: float) -> np.ndarray:
    n = int(np.prod(shape))
    out = np.empty(n, np.uint16)
    chunk = 1 << 24
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        v = rng.integers(-3, 4, size=e - s).astype(np.float32) * np.float32(scale)
        out[s:e] = f32_to_bf16_bits(v)
    return out.reshape(shape)


def make_draft_tail_case(R, hidden_size, V, seed, temperature=None, logit_std=3.0, exact=False):
    """Hidden states ~ N(0,1) and LM-head weights ~ N(0, logit_std^2 /
    hidden_size), both rounded to bf16, so the logits are ~ N(0, logit_std^2)
    like the target logits of the acceptance inputs; uniforms ~ U[0,1);
    temperature per row (default 1).

    exact=True draws both from the integers -3..3 instead, the weights scaled
    by a power of two 2^-e (logit std within a factor 2 of logit_std): every
    product and partial sum is then a multiple of 2^-e below 2^24 * 2^-e, so
    any fp32 accumulation order gives the exact logits."""
    rng = np.random.default_rng(seed)
    if exact:
        e = int(np.floor(np.log2(4.0 * np.sqrt(hidden_size) / logit_std)))
        hidden = _small_int_bf16(rng, (R, hidden_size), 1.0)
        weight = _small_int_bf16(rng, (V, hidden_size), 2.0 ** -e)
    else:
        hidden = _normal_bf16(rng, (R, hidden_size))
        weight = _scaled_normal_bf16(rng, (V, hidden_size), logit_std / np.sqrt(hidden_size))
    uniforms = rng.random(R, dtype=np.float32)
    if temperature is None:
        temperature = np.ones(R, np.float32)
    temperature = np.asarray(temperature, np.float32).reshape(R)
    return DraftTailInputs(hidden=hidden, weight=weight, uniforms=uniforms, temperature=temperature)


def make_draft_tail_inputs(wl: Workload, seed=None, exact=False) -> DraftTailInputs:
    """The K = wl.k draft positions of each of the B sequences (row b*k + i),
    each sequence at its workload temperature."""
    seed = wl.seed if seed is None else seed
    temp = np.repeat(temperatures(wl.mode, wl.B), wl.k)
    return make_draft_tail_case(wl.B * wl.k, HIDDEN_SIZES[wl.V], wl.V, seed=[seed, 0xD4AF7],
                                temperature=temp, logit_std=wl.logit_std, exact=exact)


def make_sample_case(R, V, seed, temperature=None, logit_std=3.0):
    """fp32 logits ~ N(0, logit_std^2) [R][V] and uniforms ~ U[0,1) [R] for
    the sampler alone."""
    rng = np.random.default_rng(seed)
    logits = (logit_std * rng.standard_normal((R, V), dtype=np.float32)).astype(np.float32)
    uniforms = rng.random(R, dtype=np.float32)
    if temperature is None:
        temperature = np.ones(R, np.float32)
    return logits, uniforms, np.asarray(temperature, np.float32).reshape(R)



# --------------------------------------------------------------------------- #
# visual-compressor inputs                                                    #
# --------------------------------------------------------------------------- #
# (frames F, tokens per frame N, queries C, hidden d) per workload, at the
# paper's compression ratio C/N = 1/9: LLaVA images 576 -> 64 (d 4096), QwenVL
# images 324 -> 36 and video frames 144 -> 16 (d 3584).
COMPRESS_SHAPES = {
    "tiny": (1, 576, 64, 4096),
    "image7b": (5, 576, 64, 4096),     # the 5 images of the image7b prefix
    "gqa": (8, 324, 36, 3584),         # one QwenVL image per sequence
    "video": (128, 144, 16, 3584),     # 4 sequences x 32 frames
}


def make_compress_case(F, N, C, d, seed, q_std=2.0):
    """Features F_V ~ N(0, 1) [F][N][d] and queries ~ N(0, q_std^2 / d)
    [C][d], both bf16 bits, so the scores are ~ N(0, q_std^2)."""
    rng = np.random.default_rng(seed)
    queries = _scaled_normal_bf16(rng, (C, d), q_std / np.sqrt(d))
    features = _normal_bf16(rng, (F, N, d))
    return queries, features


def make_compress_inputs(wl: Workload, seed=None):
    seed = wl.seed if seed is None else seed
    F, N, C, d = COMPRESS_SHAPES[wl.name]
    return make_compress_case(F, N, C, d, seed=[seed, 0xC0C0])
