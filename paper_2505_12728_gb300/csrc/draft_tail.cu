// draft_tail.cu -- the draft-distribution tail of Algorithm 1 on sm_103a.
//
// The semi-autoregressive draft head ends with the frozen LM head (Sec. 3.3,
// Algorithm 1): each of the K draft positions' hidden states is projected to
// vocabulary logits, P'_i = softmax(logits_i / tau) is the draft distribution
// q that the verification rule divides by, and T'_i is drawn from it,
// independently per position.  The draw is an inverse CDF in ascending token
// order (the smallest token x with u_i * S < C(x)); tau <= 0 is greedy (the
// first argmax, a one-hot P').
//
// GB300 design.  The projection streams the whole V x hidden bf16 LM head
// (262 MB for LLaVA's 32000 x 4096, 1.09 GB for QwenVL's 152064 x 3584) for
// a few dozen rows, so it is bound by HBM and everything else hides under
// that stream:
//  * lm_head_kernel: one CTA per SM, each owning an equal contiguous range
//    of vocabulary rows (floor or ceil of V / G), cut into 128-row tiles; a
//    range's last tile is loaded with a box of exactly its remaining height
//    (two extra tensor maps), so every SM streams the same number of weight
//    bytes.  Warp 5 streams 128 x 64 weight boxes and
//    the matching 64-column box of the hidden states (rows padded to NP, a
//    multiple of 16, by the copy's zero fill) into a deep ring; warp 4 issues
//    logits^T = W H^T as tcgen05 MMAs of M = 128 (vocabulary), N = NP (draft
//    rows), K = 16, accumulating in tensor memory, double-buffered per tile;
//    warps 0-3 read a finished tile back (one vocabulary row per lane),
//    store the fp32 logits coalesced along the vocabulary and, for the fused
//    path, reduce each draft row over the tile to (max, first argmax,
//    float-float sum of exp((x - max)/tau)), merged across the CTA's tiles.
//    Weight copies run before griddepcontrol.wait (the weights are constant);
//    the hidden states are copied after it.
//  * sample_stats_kernel (sf_sample only): the same per-chunk statistics
//    from given logits, 2048 tokens per CTA.
//  * sample_finish_kernel: grid (CTAs per row, rows).  Every CTA of a row
//    combines the row's chunk statistics in the same fixed order (so all get
//    bit-identical max, sum and crossing chunk), writes probabilities for its
//    span of tokens, and the CTA whose span holds the crossing chunk's first
//    token scans that chunk in ascending order for the token.
// Arithmetic: per-token terms are fp32 (exp of a float-float argument, see
// ff_math.cuh); sums, prefixes and the crossing test are float-float in a
// fixed order, so results are deterministic.  The chunk sums are taken
// relative to each chunk's own maximum and rescaled by exp((m_c - m)/tau) when
// combined; the scan inside the crossing chunk uses terms relative to the
// row maximum, so the two differ by rounding only, and where rounding puts
// the target past the chunk's own terms the chunk's last positive token is
// taken.
#include <climits>
#include <cmath>
#include <map>
#include <mutex>
#include <tuple>

#include "ff_math.cuh"
#include "sf_device.cuh"
#include "sf_host.h"

namespace sf {

constexpr int kLmThreads = 192;
constexpr int kLmEpiThreads = 128;
constexpr int kLmMmaWarp = 4;
constexpr int kLmProducerWarp = 5;
constexpr int kLmTileV = 128;                          // vocabulary rows per tile (MMA M)
constexpr int kLmChunkK = 64;                          // hidden columns per ring slot
constexpr uint32_t kLmWBytes = kLmTileV * kLmChunkK * 2;  // 16 KB weight box
constexpr int kLmMaxStages = 12;
constexpr int kLmColGroup = 16;                        // draft rows per epilogue step
constexpr int kLmTStride = 136;                        // floats per transposed row (8 mod 32 banks)
constexpr int kLmTBufFloats = 2 * kLmColGroup * kLmTStride;
constexpr int kSampleUnit = 2048;                      // tokens per statistics chunk (sf_sample)
constexpr int kSampleSpan = 4096;                      // least tokens per finishing CTA
constexpr int kMaxStatChunks = 4096;                   // statistics chunks per row

struct LmParams {
  float *logits;     // [R][V]
  const float *tau;  // temperature of row r: tau[r / tau_div]; read only with stats
  SampStat *stats;   // [R][G], or null for the plain projection
  uint32_t *status;
  int R, V, NP;
  int G;             // CTAs; CTA c owns vocabulary rows [c*V/G, (c+1)*V/G)
  int ha, hb;        // box heights of the two last-tile weight maps
  int KC;            // hidden chunks of 64
  int stages;
  uint32_t stage_bytes;  // weight box + NP * 128 bytes of hidden states
  uint32_t tmem_cols;
  uint32_t idesc;
  int w_after_wait;  // copy the weight rows only after griddepcontrol.wait
  int w_keep;        // weight rows are re-read next: L2 evict_last instead of evict_first
  int tau_div;       // rows per temperature entry (1: one per row)
  int ks;            // hidden-dimension splits: CTA (g, s) sums chunks [s*KC/ks, (s+1)*KC/ks)
  long long part_stride;  // floats between the ks partial outputs (split s adds s * part_stride)
};

struct SampleParams {
  const float *logits;    // [R][V]
  SampStat *stats;        // [R][Cn]
  const float *u;         // [R]
  const float *tau;       // [R]
  float *probs;           // [R][V]
  int32_t *tokens;        // [R]
  int R, V;
  int Cn;                 // statistics chunks per row
  int unit, T;            // chunk c covers [e(c), e(c+1)), e(c) = min(V, unit * (c*T/Cn))
  int span;               // tokens per finishing CTA (a multiple of 4)
  int vec4;               // rows 16-byte aligned and V % 4 == 0
};

// ---------------------------------------------------------------------------
// LM-head projection (tcgen05)
// ---------------------------------------------------------------------------
struct LmSmem {
  static size_t bytes(int stages, uint32_t stage_bytes, int NP) {
    return 1024 + static_cast<size_t>(stages) * stage_bytes + 4 * kLmTBufFloats +
           static_cast<size_t>(NP) * (sizeof(SampStat) + 4) + 8 * (2 * stages + 5) + 64;
  }
};

// exp((x - m) / tau) for one token; a token at -inf (masked) has weight 0.
__device__ __forceinline__ float term_of(float x, float m, float tau) {
  return x == -INFINITY ? 0.f : exp_diff_accurate(x, m, tau);
}

// Folds one tile's (max, argmax, sum) of a row into the CTA's running
// statistics; tiles arrive in ascending order, so on equal maxima the
// earlier index stays.
__device__ __forceinline__ void stat_merge(SampStat &run, float m, int arg, ff s, float tau,
                                           bool greedy) {
  if (better(m, arg, run.m, run.arg)) {
    if (!greedy)
      run.S = run.m == -INFINITY ? s : ff_add(ff_mul(run.S, exp_diff_accurate(run.m, m, tau)), s);
    run.m = m;
    run.arg = arg;
  } else if (!greedy) {
    run.S = ff_add(run.S, ff_mul(s, term_of(m, run.m, tau)));
  }
}

__global__ void __launch_bounds__(kLmThreads, 1)
lm_head_kernel(const __grid_constant__ CUtensorMap tmap_w, const __grid_constant__ CUtensorMap tmap_wa,
               const __grid_constant__ CUtensorMap tmap_wb, const __grid_constant__ CUtensorMap tmap_h,
               const __grid_constant__ LmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = p.stages;
  const uint32_t ring = smem_addr(smem);
  float *tbuf = reinterpret_cast<float *>(smem + static_cast<size_t>(S) * p.stage_bytes);
  SampStat *run = reinterpret_cast<SampStat *>(tbuf + kLmTBufFloats);
  float *s_tau = reinterpret_cast<float *>(run + p.NP);
  uint64_t *bar_mem = reinterpret_cast<uint64_t *>(s_tau + p.NP);
  int *s_misc = reinterpret_cast<int *>(bar_mem + 2 * S + 5);
  // s_misc: [0] TMEM base, [1] abort word, [2] chunks issued, [3] chunks consumed
  volatile int *s_abort = s_misc + 1;
  const uint32_t bars = smem_addr(bar_mem);
  const int FULL = 0, EMPTY = S, DFULL = 2 * S, DEMPTY = 2 * S + 2, FIN = 2 * S + 4;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int grp = static_cast<int>(blockIdx.x) % p.G, split = static_cast<int>(blockIdx.x) / p.G;
  const int v0 = static_cast<int>(static_cast<long long>(grp) * p.V / p.G);
  const int v1 = static_cast<int>(static_cast<long long>(grp + 1) * p.V / p.G);
  const int n_tiles = (v1 - v0 + kLmTileV - 1) / kLmTileV;
  const int last_h = v1 - v0 - (n_tiles - 1) * kLmTileV;  // rows of the last tile
  const int kc0 = split * p.KC / p.ks;                      // this CTA's hidden chunks
  const int nkc = (split + 1) * p.KC / p.ks - kc0;
  float *const logits = p.logits + static_cast<long long>(split) * p.part_stride;
  const uint32_t total = static_cast<uint32_t>(n_tiles) * static_cast<uint32_t>(nkc);
  // weight map and box height of tile i
  auto tile_map = [&](int i, uint32_t &bytes) -> const CUtensorMap * {
    const int h = i == n_tiles - 1 ? last_h : kLmTileV;
    bytes = static_cast<uint32_t>(h) * (kLmChunkK * 2) + static_cast<uint32_t>(p.NP) * (kLmChunkK * 2);
    return h == kLmTileV ? &tmap_w : (h == p.ha ? &tmap_wa : &tmap_wb);
  };

  grid_launch_dependents();
  if (tid == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(bar(FULL + s), 1);
      mbar_init(bar(EMPTY + s), 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(bar(DFULL + x), 1);
      mbar_init(bar(DEMPTY + x), kLmEpiThreads);
    }
    mbar_init(bar(FIN), 1);
    fence_mbar_init();
    prefetch_tensormap(&tmap_w);
    prefetch_tensormap(&tmap_wa);
    prefetch_tensormap(&tmap_wb);
    prefetch_tensormap(&tmap_h);
    s_misc[1] = 0;
    s_misc[2] = 0;
    s_misc[3] = 0;
  }
  __syncthreads();  // barrier initialisation visible to every role
  // Tensor memory is allocated only once the previous kernel on the stream
  // has completed: a predecessor that is still waiting for its own
  // predecessor may not have allocated yet, and holding TMEM here while it
  // waits for columns could deadlock the pair.  The producer warp does not
  // need TMEM and starts its weight copies meanwhile.
  uint32_t tmem = 0;
  if (warp != kLmProducerWarp) {
    if (warp == kLmMmaWarp) {
      grid_dependency_wait();
      tmem_alloc(smem_addr(s_misc), p.tmem_cols);
      tmem_relinquish_alloc_permit();
      tc_fence_before_sync();
    }
    named_bar_sync(3, kLmEpiThreads + 32);
    tc_fence_after_sync();
    tmem = static_cast<uint32_t>(s_misc[0]);
  }

  if (warp == kLmProducerWarp) {
    if (lane == 0) {
      const uint64_t pol_w = p.w_keep ? l2_policy_evict_last() : l2_policy_evict_first();
      const uint64_t pol_h = l2_policy_evict_last();
      const uint32_t prime = total < static_cast<uint32_t>(S) ? total : static_cast<uint32_t>(S);
      // the first ring fill: weights before the dependency wait (unless
      // they may come from the previous kernel), hidden states after it
      if (p.w_after_wait) grid_dependency_wait();
      for (uint32_t q = 0; q < prime; ++q) {
        const int i = static_cast<int>(q) / nkc, kc = kc0 + static_cast<int>(q) % nkc;
        uint32_t bytes;
        const CUtensorMap *mw = tile_map(i, bytes);
        mbar_arrive_expect_tx(bar(FULL + q), bytes);
        tma_load_2d(ring + q * p.stage_bytes, mw, kc * kLmChunkK, v0 + i * kLmTileV, bar(FULL + q),
                    pol_w);
      }
      if (!p.w_after_wait) grid_dependency_wait();
      for (uint32_t q = 0; q < prime; ++q) {
        const int kc = kc0 + static_cast<int>(q) % nkc;
        tma_load_2d(ring + q * p.stage_bytes + kLmWBytes, &tmap_h, kc * kLmChunkK, 0, bar(FULL + q),
                    pol_h);
      }
      uint32_t q = prime;
      for (; q < total; ++q) {
        const uint32_t slot = q % S;
        if (!mbar_wait_or_abort(bar(EMPTY + slot), ((q / S) - 1) & 1u, s_abort)) break;
        const int i = static_cast<int>(q) / nkc, kc = kc0 + static_cast<int>(q) % nkc;
        const uint32_t dst = ring + slot * p.stage_bytes;
        uint32_t bytes;
        const CUtensorMap *mw = tile_map(i, bytes);
        mbar_arrive_expect_tx(bar(FULL + slot), bytes);
        tma_load_2d(dst, mw, kc * kLmChunkK, v0 + i * kLmTileV, bar(FULL + slot), pol_w);
        tma_load_2d(dst + kLmWBytes, &tmap_h, kc * kLmChunkK, 0, bar(FULL + slot), pol_h);
      }
      s_misc[2] = static_cast<int>(q);
    }
    __syncwarp();
  } else if (warp == kLmMmaWarp) {
    // ------------------------------------------------------------------
    // MMA issue: per 64-column chunk four MMAs (K = 16 each, +32 bytes
    // along the 128-byte swizzled rows); the slot is released by a commit.
    // Rows of a short last tile beyond its box hold stale data; their
    // accumulator rows are never stored.
    // ------------------------------------------------------------------
    uint32_t q = 0;
    bool ok = true;
    for (int i = 0; i < n_tiles && ok; ++i) {
      const uint32_t buf = static_cast<uint32_t>(i) & 1u;
      if (i >= 2) {
        int w = 1;
        if (lane == 0) w = mbar_wait_or_abort(bar(DEMPTY + buf), ((i - 2) >> 1) & 1, s_abort);
        if (!__shfl_sync(0xffffffffu, w, 0)) break;
      }
      tc_fence_after_sync();
      const uint32_t d = tmem + buf * static_cast<uint32_t>(p.NP);
      for (int kc = 0; kc < nkc; ++kc, ++q) {
        const uint32_t slot = q % S;
        int w = 1;
        if (lane == 0) w = mbar_wait_or_abort(bar(FULL + slot), (q / S) & 1u, s_abort);
        if (!__shfl_sync(0xffffffffu, w, 0)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        if (lane == 0) s_misc[3] = static_cast<int>(q + 1);
        const uint32_t wa = ring + slot * p.stage_bytes;
        const uint32_t hb = wa + kLmWBytes;
        if (elect_one()) {
#pragma unroll
          for (int kk = 0; kk < kLmChunkK / 16; ++kk) {
            const uint64_t a = smem_desc_sw128(wa + kk * 32, 16, 1024);
            const uint64_t b = smem_desc_sw128(hb + kk * 32, 16, 1024);
            tc_mma_ss(d, a, b, p.idesc, (kc > 0 || kk > 0) ? 1u : 0u);
          }
          tc_commit(bar(EMPTY + slot));
        }
        __syncwarp();
      }
      if (!ok) break;
      if (elect_one()) tc_commit(bar(DFULL + buf));
      __syncwarp();
    }
    if (elect_one()) tc_commit(bar(FIN));
    __syncwarp();
    (void)mbar_wait_bounded(bar(FIN), 0);
  } else {
    // ------------------------------------------------------------------
    // epilogue: thread = vocabulary row of the tile (TMEM lane), 16 draft
    // rows (TMEM columns) per step.  Logits go straight to global memory;
    // for the statistics the step is transposed through shared memory and
    // each draft row is reduced by 8 threads (128 values / 8, interleaved).
    // ------------------------------------------------------------------
    const bool stats = p.stats != nullptr;
    grid_dependency_wait();  // outputs and temperatures follow the previous kernel
    if (stats) {
      for (int c = tid; c < p.NP; c += kLmEpiThreads) {
        s_tau[c] = c < p.R ? p.tau[c / p.tau_div] : 1.f;
        run[c] = SampStat{-INFINITY, INT_MAX, ff_of(0.f)};
      }
    }
    named_bar_sync(1, kLmEpiThreads);
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * warp) << 16);
    const int groups = p.NP / kLmColGroup;
    uint32_t g_count = 0;
    for (int i = 0; i < n_tiles; ++i) {
      const uint32_t buf = static_cast<uint32_t>(i) & 1u;
      bool ok = mbar_wait_or_abort(bar(DFULL + buf), (i >> 1) & 1, s_abort);
      if (!named_bar_and(2, kLmEpiThreads, ok)) break;
      tc_fence_after_sync();
      const int vbase = v0 + i * kLmTileV;
      const int v = vbase + 32 * warp + lane;
      const bool vin = v < v1;
      for (int g = 0; g < groups; ++g, ++g_count) {
        const int c0 = g * kLmColGroup;
        uint32_t x[16];
        tmem_ld_32x32b_x16(lane_base + buf * static_cast<uint32_t>(p.NP) + c0, x);
        if (vin) {
#pragma unroll
          for (int j = 0; j < 16; ++j)
            if (c0 + j < p.R) logits[static_cast<size_t>(c0 + j) * p.V + v] = __uint_as_float(x[j]);
        }
        if (!stats) continue;
        float *tb = tbuf + (g_count & 1u) * (kLmColGroup * kLmTStride);
#pragma unroll
        for (int j = 0; j < 16; ++j)
          tb[j * kLmTStride + 32 * warp + lane] = vin ? __uint_as_float(x[j]) : -INFINITY;
        named_bar_sync(1, kLmEpiThreads);
        const int cl = tid >> 3, part = tid & 7, r = c0 + cl;
        const float *col = tb + cl * kLmTStride + part;
        float bv = -INFINITY;
        int bi = INT_MAX;
#pragma unroll
        for (int e = 0; e < 16; ++e) {
          const float val = col[8 * e];
          if (better(val, vbase + part + 8 * e, bv, bi)) {
            bv = val;
            bi = vbase + part + 8 * e;
          }
        }
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) {
          const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
          const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
          if (better(ov, oi, bv, bi)) {
            bv = ov;
            bi = oi;
          }
        }
        const float tau = s_tau[r];
        const bool greedy = !(tau > 0.f);
        ff s = ff_of(0.f);
        if (!greedy) {
#pragma unroll 4
          for (int e = 0; e < 16; ++e) s = ff_add(s, ff_of(term_of(col[8 * e], bv, tau)));
        }
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) s = ff_add(s, shfl_xor_ff(s, o));
        if (part == 0) stat_merge(run[r], bv, bi, s, tau, greedy);
      }
      tc_fence_before_sync();
      mbar_arrive(bar(DEMPTY + buf));
    }
    if (stats) {
      named_bar_sync(1, kLmEpiThreads);
      for (int c = tid; c < p.R; c += kLmEpiThreads)
        p.stats[static_cast<size_t>(c) * p.G + grp] = run[c];
    }
  }

  // ---- teardown ----
  __syncthreads();
  if (*s_abort) {
    if (tid == 0) set_status(p.status, SF_DEVICE_TIMEOUT);
    if (warp == kLmProducerWarp && lane == 0) {
      // copies issued but never consumed: wait (bounded) until they land
      for (uint32_t x = static_cast<uint32_t>(s_misc[3]); x < static_cast<uint32_t>(s_misc[2]); ++x)
        (void)mbar_wait_bounded(bar(FULL + x % S), (x / S) & 1u);
    }
    __syncthreads();
  }
  if (warp == kLmMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, p.tmem_cols);
  }
}

// ---------------------------------------------------------------------------
// sampling
// ---------------------------------------------------------------------------
__device__ __forceinline__ int chunk_start(const SampleParams &p, int c) {
  const long long e = static_cast<long long>(p.unit) * (static_cast<long long>(c) * p.T / p.Cn);
  return e < p.V ? static_cast<int>(e) : p.V;
}

// Statistics of one kSampleUnit chunk of one row (sf_sample): grid (Cn, R).
__global__ void __launch_bounds__(kFfThreads) sample_stats_kernel(const __grid_constant__ SampleParams p) {
  __shared__ ff s_d[32];
  __shared__ float s_v[32];
  __shared__ int s_i[32];
  grid_dependency_wait();
  grid_launch_dependents();
  const int c = blockIdx.x, r = blockIdx.y, tid = threadIdx.x;
  const float *row = p.logits + static_cast<size_t>(r) * p.V;
  const int e0 = c * kSampleUnit;
  const float tau = p.tau[r];
  const bool greedy = !(tau > 0.f);
  constexpr int kPer = kSampleUnit / kFfThreads;  // 8 tokens per thread, 4 consecutive
  float x[kPer];
#pragma unroll
  for (int h = 0; h < kPer / 4; ++h) {
    const int i0 = e0 + h * 4 * kFfThreads + 4 * tid;
    if (p.vec4 && i0 + 3 < p.V) {
      const float4 f = __ldg(reinterpret_cast<const float4 *>(row + i0));
      x[4 * h] = f.x;
      x[4 * h + 1] = f.y;
      x[4 * h + 2] = f.z;
      x[4 * h + 3] = f.w;
    } else {
#pragma unroll
      for (int j = 0; j < 4; ++j) x[4 * h + j] = i0 + j < p.V ? __ldg(row + i0 + j) : -INFINITY;
    }
  }
  float bv = -INFINITY;
  int bi = INT_MAX;
#pragma unroll
  for (int h = 0; h < kPer / 4; ++h)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int idx = e0 + h * 4 * kFfThreads + 4 * tid + j;
      if (idx < p.V && better(x[4 * h + j], idx, bv, bi)) {
        bv = x[4 * h + j];
        bi = idx;
      }
    }
  block_argmax(bv, bi, s_v, s_i);
  ff s = ff_of(0.f);
  if (!greedy) {
#pragma unroll
    for (int e = 0; e < kPer; ++e) s = ff_add(s, ff_of(term_of(x[e], bv, tau)));
    s = block_sum(s, s_d);
  }
  if (tid == 0) p.stats[static_cast<size_t>(r) * p.Cn + c] = SampStat{bv, bi, s};
}

// Combines a row's chunk statistics, writes P' for this CTA's span of
// tokens and, in the CTA holding the crossing chunk's first
// token, draws T'.  grid (ceil(V / span), R); dynamic shared memory
// holds the row's Cn statistics.
__global__ void __launch_bounds__(kFfThreads) sample_finish_kernel(const __grid_constant__ SampleParams p) {
  extern __shared__ SampStat s_st[];
  __shared__ ff s_scan[kFfWarps + 1];
  __shared__ float s_v[32];
  __shared__ int s_i[32];
  __shared__ int s_c, s_tok, s_last;
  __shared__ ff s_base;
  grid_dependency_wait();  // the statistics and logits come from the previous kernels
  grid_launch_dependents();
  const int r = blockIdx.y, tid = threadIdx.x;
  const float *row = p.logits + static_cast<size_t>(r) * p.V;
  float *prow = p.probs + static_cast<size_t>(r) * p.V;
  const SampStat *st = p.stats + static_cast<size_t>(r) * p.Cn;
  for (int c = tid; c < p.Cn; c += kFfThreads) s_st[c] = st[c];
  if (tid == 0) {
    s_c = INT_MAX;
    s_tok = INT_MAX;
    s_last = -1;
  }
  __syncthreads();

  // row maximum and its first index
  float m = -INFINITY;
  int arg = INT_MAX;
  for (int c = tid; c < p.Cn; c += kFfThreads)
    if (better(s_st[c].m, s_st[c].arg, m, arg)) {
      m = s_st[c].m;
      arg = s_st[c].arg;
    }
  block_argmax(m, arg, s_v, s_i);

  const float tau = p.tau[r];
  const int x0 = blockIdx.x * p.span;
  const int x1 = min(p.V, x0 + p.span);
  if (!(tau > 0.f)) {
    // greedy: one-hot P', T' = the first argmax
    for (int x = x0 + tid; x < x1; x += kFfThreads) prow[x] = x == arg ? 1.f : 0.f;
    if (tid == 0 && arg >= x0 && arg < x1) p.tokens[r] = arg;
    return;
  }

  // chunk masses relative to m; thread t sums chunks [c_lo, c_hi) in order
  const int c_lo = static_cast<int>(static_cast<long long>(tid) * p.Cn / kFfThreads);
  const int c_hi = static_cast<int>(static_cast<long long>(tid + 1) * p.Cn / kFfThreads);
  auto mass = [&](int c) -> ff {
    return s_st[c].m == -INFINITY ? ff_of(0.f)
                                  : ff_mul(s_st[c].S, term_of(s_st[c].m, m, tau));
  };
  ff mine = ff_of(0.f);
  for (int c = c_lo; c < c_hi; ++c) mine = ff_add(mine, mass(c));
  ff excl, Stot;
  block_inclusive_scan(mine, s_scan, &excl, &Stot);
  const ff target = ff_mul(Stot, p.u[r]);
  // the first chunk whose inclusive prefix exceeds the target
  {
    ff cum = excl;
    int cand = INT_MAX, lastpos = -1;
    ff cand_base = ff_of(0.f);
    for (int c = c_lo; c < c_hi; ++c) {
      const ff w = mass(c);
      const ff nxt = ff_add(cum, w);
      if (ff_pos(w)) lastpos = c;
      if (cand == INT_MAX && ff_lt(target, nxt)) {
        cand = c;
        cand_base = cum;
      }
      cum = nxt;
    }
    if (cand != INT_MAX) atomicMin(&s_c, cand);
    if (lastpos >= 0) atomicMax(&s_last, lastpos);
    __syncthreads();
    if (cand != INT_MAX && cand == s_c) s_base = cand_base;
    __syncthreads();
  }
  const bool crossed = s_c != INT_MAX;
  const int cs = crossed ? s_c : s_last;  // no crossing (u >= 1 or NaN): last positive chunk

  // P' for this CTA's span.  Rows are 16-byte aligned and the span a
  // multiple of 4 in the vector path, so a float4 is either wholly inside
  // the span or wholly outside; each thread issues kBatch loads before
  // the arithmetic and stores that depend on them.
  const float invS = ff_div_to_f(1.f, Stot);
  if (p.vec4) {
    constexpr int kBatch = 4;
    for (int base = x0 + 4 * tid; base < x1; base += 4 * kFfThreads * kBatch) {
      float4 f[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int x = base + j * 4 * kFfThreads;
        if (x < x1) f[j] = __ldcs(reinterpret_cast<const float4 *>(row + x));
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int x = base + j * 4 * kFfThreads;
        if (x < x1) {
          float4 o;
          o.x = __fmul_rn(term_of(f[j].x, m, tau), invS);
          o.y = __fmul_rn(term_of(f[j].y, m, tau), invS);
          o.z = __fmul_rn(term_of(f[j].z, m, tau), invS);
          o.w = __fmul_rn(term_of(f[j].w, m, tau), invS);
          *reinterpret_cast<float4 *>(prow + x) = o;
        }
      }
    }
  } else {
    for (int x = x0 + tid; x < x1; x += kFfThreads)
      prow[x] = __fmul_rn(term_of(row[x], m, tau), invS);
  }

  if (cs < 0) return;  // no positive chunk: unreachable for finite logits
  const int e0 = chunk_start(p, cs), e1 = chunk_start(p, cs + 1);
  if (e0 < x0 || e0 >= x1) return;

  // scan the chunk in ascending order, 4 consecutive tokens per thread
  __syncthreads();
  if (tid == 0) s_last = -1;
  __syncthreads();
  ff base = s_base;
  int lastpos = -1;
  for (int s0 = e0; s0 < e1; s0 += 4 * kFfThreads) {
    float t[4];
    ff tsum = ff_of(0.f);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int x = s0 + 4 * tid + j;
      t[j] = x < e1 ? term_of(row[x], m, tau) : 0.f;
      if (t[j] > 0.f) lastpos = x;
      tsum = ff_add(tsum, ff_of(t[j]));
    }
    ff ex, tot;
    block_inclusive_scan(tsum, s_scan, &ex, &tot);
    if (crossed) {
      ff cum = ff_add(base, ex);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        cum = ff_add(cum, ff_of(t[j]));
        if (ff_lt(target, cum)) {
          atomicMin(&s_tok, s0 + 4 * tid + j);
          break;
        }
      }
    }
    __syncthreads();
    if (s_tok != INT_MAX) break;
    base = ff_add(base, tot);
  }
  if (lastpos >= 0) atomicMax(&s_last, lastpos);
  __syncthreads();
  if (tid == 0) p.tokens[r] = s_tok != INT_MAX ? s_tok : s_last;
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
static int np_of(int R) { return (R + 15) / 16 * 16; }

static int lm_stages(const DeviceInfo &dev, uint32_t stage_bytes, int NP) {
  int s = kLmMaxStages;
  while (s > 2 && LmSmem::bytes(s, stage_bytes, NP) > static_cast<size_t>(dev.max_smem_optin)) --s;
  return s;
}

static int lm_setup(const DeviceInfo &dev) {
  static std::mutex mu;
  static bool done[64] = {};
  if (dev.ordinal < 0 || dev.ordinal >= 64) return fail(SF_ERR_UNSUPPORTED, "device ordinal %d", dev.ordinal);
  std::lock_guard<std::mutex> lock(mu);
  if (done[dev.ordinal]) return SF_OK;
  cudaError_t e = cudaFuncSetAttribute(lm_head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       dev.max_smem_optin);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(sample_finish_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             kMaxStatChunks * static_cast<int>(sizeof(SampStat)));
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "cudaFuncSetAttribute (draft tail): %s", cudaGetErrorString(e));
  done[dev.ordinal] = true;
  return SF_OK;
}

// Tensor maps of the weights {hidden, V} (box 64 x 128, 64 x ha, 64 x hb) and
// hidden states {hidden, R} (box 64 x NP), cached by (base, rows, hidden, box
// rows).
static int lm_tensor_map(CUtensorMap *out, const void *base, uint64_t rows, int hidden, uint32_t box_rows) {
  static std::mutex mu;
  static std::map<std::tuple<const void *, uint64_t, int, uint32_t>, CUtensorMap> maps;
  const auto key = std::make_tuple(base, rows, hidden, box_rows);
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = maps.find(key);
    if (it != maps.end()) {
      *out = it->second;
      return SF_OK;
    }
  }
  const uint64_t dims[2] = {static_cast<uint64_t>(hidden), rows};
  const uint64_t strides[1] = {static_cast<uint64_t>(hidden) * 2};
  const uint32_t box[2] = {static_cast<uint32_t>(kLmChunkK), box_rows};
  const int st = encode_tensor_map_bf16(out, base, 2, dims, strides, box);
  if (st != SF_OK) return st;
  std::lock_guard<std::mutex> lock(mu);
  if (maps.size() >= 4096) maps.clear();
  maps.emplace(key, *out);
  return SF_OK;
}

static int check_lm_args(const void *hidden, const void *weight, int R, int hidden_size, int V,
                         const float *logits) {
  if (R < 1 || R > SF_MAX_DRAFT_ROWS)
    return fail(SF_ERR_INVALID_ARG, "R=%d outside [1, %d]", R, SF_MAX_DRAFT_ROWS);
  if (hidden_size < 8 || hidden_size % 8 != 0 || hidden_size > (1 << 20))
    return fail(SF_ERR_INVALID_ARG, "hidden_size=%d must be a multiple of 8 in [8, 2^20]", hidden_size);
  if (V < 1 || V > SF_MAX_VOCAB) return fail(SF_ERR_INVALID_ARG, "V=%d outside [1, %d]", V, SF_MAX_VOCAB);
  if (!hidden || !weight || !logits) return fail(SF_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!aligned(hidden, 16) || !aligned(weight, 16))
    return fail(SF_ERR_INVALID_ARG, "hidden and weight must be 16-byte aligned");
  if (!aligned(logits, 4)) return fail(SF_ERR_INVALID_ARG, "logits must be 4-byte aligned");
  return SF_OK;
}

static int check_sample_args(int R, int V, const float *uniforms, const float *temperature,
                             const float *probs, const int32_t *tokens) {
  if (R < 1 || R > 65535) return fail(SF_ERR_INVALID_ARG, "R=%d outside [1, 65535]", R);
  if (V < 1 || V > SF_MAX_VOCAB) return fail(SF_ERR_INVALID_ARG, "V=%d outside [1, %d]", V, SF_MAX_VOCAB);
  if (!uniforms || !temperature || !probs || !tokens)
    return fail(SF_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!aligned(uniforms, 4) || !aligned(temperature, 4) || !aligned(probs, 4) || !aligned(tokens, 4))
    return fail(SF_ERR_INVALID_ARG, "buffers must be 4-byte aligned");
  return SF_OK;
}

static size_t stats_bytes(int R, int V, int sm_count) {
  const size_t cn = static_cast<size_t>((V + kSampleUnit - 1) / kSampleUnit);
  const size_t cn_max = cn > static_cast<size_t>(sm_count) ? cn : static_cast<size_t>(sm_count);
  return 256 + round_up(static_cast<size_t>(R) * cn_max * sizeof(SampStat), 256);
}

static cudaLaunchConfig_t pdl_config(dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                                     cudaLaunchAttribute *attr) {
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

// Launches the projection; with `stats` the epilogue also writes the per-CTA
// sampling statistics [R][G] and *G_out receives G.
static int launch_lm_head(const void *hidden, const void *weight, int R, int hidden_size, int V,
                          float *logits, const float *temperature, SampStat *stats, uint32_t *status,
                          int *G_out, cudaStream_t stream, bool w_after_wait = false,
                          bool w_keep = false, int ks = 1, int tau_div = 1) {
  DeviceInfo dev;
  int st = current_device(&dev);
  if (st != SF_OK) return st;
  if (dev.cc_major != 10) return fail(SF_ERR_UNSUPPORTED, "the LM-head kernel needs an sm_10x GPU");
  st = lm_setup(dev);
  if (st != SF_OK) return st;
  const int NP = np_of(R);
  LmParams prm;
  prm.logits = logits;
  prm.tau = temperature;
  prm.stats = stats;
  prm.status = status;
  prm.R = R;
  prm.V = V;
  prm.NP = NP;
  const int tiles = (V + kLmTileV - 1) / kLmTileV;
  prm.G = tiles < dev.sm_count ? tiles : dev.sm_count;
  const int q = V / prm.G;  // every CTA owns q or q + 1 rows
  prm.ha = (q - 1) % kLmTileV + 1;
  prm.hb = q % kLmTileV + 1;
  prm.KC = (hidden_size + kLmChunkK - 1) / kLmChunkK;
  prm.stage_bytes = kLmWBytes + static_cast<uint32_t>(NP) * 128u;
  prm.stages = lm_stages(dev, prm.stage_bytes, NP);
  uint32_t cols = 32;
  while (cols < 2u * static_cast<uint32_t>(NP)) cols <<= 1;
  prm.tmem_cols = cols;
  prm.idesc = idesc_bf16_f32(128, NP, 0, 0);
  prm.w_after_wait = w_after_wait ? 1 : 0;
  prm.w_keep = w_keep ? 1 : 0;
  prm.ks = ks < 1 ? 1 : (ks > prm.KC ? prm.KC : ks);
  prm.tau_div = tau_div < 1 ? 1 : tau_div;
  prm.part_stride = static_cast<long long>(R) * V;
  if (stats && prm.ks != 1) return fail(SF_ERR_INVALID_ARG, "statistics need an unsplit projection");
  const size_t smem = LmSmem::bytes(prm.stages, prm.stage_bytes, NP);
  if (smem > static_cast<size_t>(dev.max_smem_optin))
    return fail(SF_ERR_UNSUPPORTED, "LM-head ring needs %zu bytes of shared memory", smem);
  CUtensorMap tw, twa, twb, th;
  st = lm_tensor_map(&tw, weight, static_cast<uint64_t>(V), hidden_size, kLmTileV);
  if (st == SF_OK)
    st = lm_tensor_map(&twa, weight, static_cast<uint64_t>(V), hidden_size, static_cast<uint32_t>(prm.ha));
  if (st == SF_OK)
    st = lm_tensor_map(&twb, weight, static_cast<uint64_t>(V), hidden_size, static_cast<uint32_t>(prm.hb));
  if (st != SF_OK) return st;
  st = lm_tensor_map(&th, hidden, static_cast<uint64_t>(R), hidden_size, static_cast<uint32_t>(NP));
  if (st != SF_OK) return st;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = pdl_config(dim3(prm.G * prm.ks), dim3(kLmThreads), smem, stream, attr);
  cudaError_t e = cudaLaunchKernelEx(&cfg, lm_head_kernel, tw, twa, twb, th, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "LM-head launch: %s", cudaGetErrorString(e));
  if (G_out) *G_out = prm.G;
  return SF_OK;
}

// Span per finishing CTA: about one wave of CTAs (8 per SM) over all rows,
// at least kSampleSpan tokens, a multiple of kSampleSpan.
static int finish_span(int R, int V) {
  DeviceInfo dev;
  const int sms = current_device(&dev) == SF_OK ? dev.sm_count : 148;
  const long long per = ((long long)R * V + 8LL * sms - 1) / (8LL * sms);
  long long span = (per + kSampleSpan - 1) / kSampleSpan * kSampleSpan;
  if (span < kSampleSpan) span = kSampleSpan;
  if (span > V) span = (V + 3) / 4 * 4;
  return static_cast<int>(span);
}

static int launch_finish(SampleParams prm, cudaStream_t stream) {
  cudaLaunchAttribute attr[1];
  prm.span = finish_span(prm.R, prm.V);
  const int spans = (prm.V + prm.span - 1) / prm.span;
  cudaLaunchConfig_t cfg = pdl_config(dim3(spans, prm.R), dim3(kFfThreads),
                                      static_cast<size_t>(prm.Cn) * sizeof(SampStat), stream, attr);
  cudaError_t e = cudaLaunchKernelEx(&cfg, sample_finish_kernel, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "sampling launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

int launch_projection_stats(const void *hidden, const void *weight, int R, int hidden_size, int V,
                            float *logits, const float *temperature, int rows_per_temperature,
                            SampStat *stats, uint32_t *status, int *G_out, cudaStream_t stream) {
  const int st = check_lm_args(hidden, weight, R, hidden_size, V, logits);
  if (st != SF_OK) return st;
  return launch_lm_head(hidden, weight, R, hidden_size, V, logits, temperature, stats, status, G_out,
                        stream, false, false, 1, rows_per_temperature);
}

int projection_groups(int V, int sm_count) {
  const int tiles = (V + kLmTileV - 1) / kLmTileV;
  return tiles < sm_count ? tiles : sm_count;
}

int projection_splits(int V, int hidden_size, int sm_count) {
  const int tiles = (V + kLmTileV - 1) / kLmTileV;
  const int G = tiles < sm_count ? tiles : sm_count;
  const int KC = (hidden_size + kLmChunkK - 1) / kLmChunkK;
  int ks = sm_count / G;
  if (ks > KC) ks = KC;
  return ks < 1 ? 1 : ks;
}

int launch_projection(const void *rows_r, const void *rows_v, int R, int hidden_size, int V,
                      float *out, uint32_t *status, bool inputs_after_wait, bool keep_v_rows,
                      int splits, cudaStream_t stream) {
  const int st = check_lm_args(rows_r, rows_v, R, hidden_size, V, out);
  if (st != SF_OK) return st;
  return launch_lm_head(rows_r, rows_v, R, hidden_size, V, out, nullptr, nullptr, status, nullptr,
                        stream, inputs_after_wait, keep_v_rows, splits);
}

}  // namespace sf

extern "C" {

size_t sf_draft_tail_workspace_size(int R, int V) {
  using namespace sf;
  if (R < 1 || R > 65535 || V < 1 || V > SF_MAX_VOCAB) return 0;
  DeviceInfo dev;
  if (current_device(&dev) != SF_OK) return 0;
  return stats_bytes(R, V, dev.sm_count);
}

int sf_lm_head(const void *hidden, const void *weight, int R, int hidden_size, int V, float *logits,
               void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  using namespace sf;
  clear_error();
  int st = check_lm_args(hidden, weight, R, hidden_size, V, logits);
  if (st != SF_OK) return st;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < 256)
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL, 256-byte aligned and >= 256 bytes");
  return launch_lm_head(hidden, weight, R, hidden_size, V, logits, nullptr, nullptr,
                        static_cast<uint32_t *>(workspace), nullptr, stream);
}

int sf_sample(const float *logits, const float *uniforms, const float *temperature, int R, int V,
              float *probs, int32_t *tokens, void *workspace, size_t workspace_bytes,
              cudaStream_t stream) {
  using namespace sf;
  clear_error();
  int st = check_sample_args(R, V, uniforms, temperature, probs, tokens);
  if (st != SF_OK) return st;
  if (!logits || !aligned(logits, 4)) return fail(SF_ERR_INVALID_ARG, "logits NULL or misaligned");
  DeviceInfo dev;
  st = current_device(&dev);
  if (st != SF_OK) return st;
  st = lm_setup(dev);
  if (st != SF_OK) return st;
  if (!workspace || !aligned(workspace, 256))
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL and 256-byte aligned");
  const size_t need = stats_bytes(R, V, dev.sm_count);
  if (workspace_bytes < need)
    return fail(SF_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, need);
  SampleParams prm;
  prm.logits = logits;
  prm.stats = reinterpret_cast<SampStat *>(static_cast<uint8_t *>(workspace) + 256);
  prm.u = uniforms;
  prm.tau = temperature;
  prm.probs = probs;
  prm.tokens = tokens;
  prm.R = R;
  prm.V = V;
  prm.Cn = (V + kSampleUnit - 1) / kSampleUnit;
  prm.unit = kSampleUnit;
  prm.T = prm.Cn;
  prm.vec4 = (V % 4 == 0) && aligned(logits, 16) && aligned(probs, 16);
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = pdl_config(dim3(prm.Cn, R), dim3(kFfThreads), 0, stream, attr);
  cudaError_t e = cudaLaunchKernelEx(&cfg, sample_stats_kernel, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "sampling statistics launch: %s", cudaGetErrorString(e));
  return launch_finish(prm, stream);
}

int sf_draft_sample(const void *hidden, const void *weight, const float *uniforms,
                    const float *temperature, int R, int hidden_size, int V, float *logits,
                    float *probs, int32_t *tokens, void *workspace, size_t workspace_bytes,
                    cudaStream_t stream) {
  using namespace sf;
  clear_error();
  int st = check_lm_args(hidden, weight, R, hidden_size, V, logits);
  if (st != SF_OK) return st;
  st = check_sample_args(R, V, uniforms, temperature, probs, tokens);
  if (st != SF_OK) return st;
  DeviceInfo dev;
  st = current_device(&dev);
  if (st != SF_OK) return st;
  if (!workspace || !aligned(workspace, 256))
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL and 256-byte aligned");
  const size_t need = stats_bytes(R, V, dev.sm_count);
  if (workspace_bytes < need)
    return fail(SF_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, need);
  SampleParams prm;
  prm.stats = reinterpret_cast<SampStat *>(static_cast<uint8_t *>(workspace) + 256);
  int G = 0;
  st = launch_lm_head(hidden, weight, R, hidden_size, V, logits, temperature, prm.stats,
                      static_cast<uint32_t *>(workspace), &G, stream);
  if (st != SF_OK) return st;
  prm.logits = logits;
  prm.u = uniforms;
  prm.tau = temperature;
  prm.probs = probs;
  prm.tokens = tokens;
  prm.R = R;
  prm.V = V;
  prm.Cn = G;  // chunk c = CTA c's rows [c*V/G, (c+1)*V/G)
  prm.unit = 1;
  prm.T = V;
  prm.vec4 = (V % 4 == 0) && aligned(logits, 16) && aligned(probs, 16);
  return launch_finish(prm, stream);
}

}  // extern "C"
