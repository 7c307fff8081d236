// verify_attention_tc.cu -- verification attention on the 5th-generation
// tensor cores (tcgen05, accumulators in tensor memory), used for shapes
// with many query rows per KV head (GQA, R = n_q * g > 16).
//
// It computes exactly what the mma.sync kernel in verify_attention.cu
// computes (Sec. 3.1: the K draft tokens are scored in one forward pass, so
// each of the n_q new rows attends to the prefix plus the causal draft
// block).  Design points:
//  * One CTA per SM with a six-stage ring (192 KB): the prefix tiles of the
//    ring are copied before griddepcontrol.wait, so they land while the
//    previous kernel on the stream finishes.  Tensor memory (all 512
//    columns) is allocated only after that wait: a kernel that waits for
//    its predecessor never holds TMEM, so two kernels cannot each hold what
//    the other waits for.
//  * The work partition is chosen on the device from seq_lens: the
//    balanced one (all tiles cut into G equal ranges; a CTA may hold pieces
//    of several segments) or a segment-aligned one (each segment gets
//    ceil(tiles / Ta) CTAs and every CTA one piece) when its largest piece
//    is within kAlignSlackTiles of the balanced share.
//  * All R rows of a KV head are the M = 128 side of the MMAs.  The rows are
//    repeated F = 128 / RPK times (RPK = 32, 64 or 128 rows per copy): copy
//    kap occupies TMEM lanes [kap * RPK, (kap + 1) * RPK) and, in the
//    softmax, owns keys [kap * KPL, (kap + 1) * KPL) of every 64-key tile
//    (KPL = 64 / F).  A copy is a whole number of 32-lane quarters, so each
//    softmax warp reads exactly its keys' score columns.  The repeated rows
//    cost the 128-row MMAs nothing.  The F partial states of a row merge
//    through shared memory when the piece is a whole segment; a split
//    segment's pieces write one partial per copy and the merge kernel
//    combines all of them (no exchange on the split kernel's tail).
//  * Q lives in tensor memory (the A operand of S = Q K^T): each softmax
//    thread writes its lane's row.  Four S buffers: P = exp2(S') is written
//    as bf16 over the scores it came from, so Q K^T of tile n+4 (which
//    overwrites the buffer) is issued after P V of tile n, and tcgen05 MMAs
//    of one thread execute in issue order.  The softmax of four tiles can be
//    in flight behind one another.
//  * A K tile sits in shared memory as [page][8-token group][64-column
//    half][8 tokens][128 B], 128B-swizzled: one 4-D TMA box per 16-token
//    page brings both halves, and the 8-token atoms of a half are 2048 bytes
//    apart, so S = Q K^T is head_dim/16 MMAs of M=128, N=64, K=16.  A V tile
//    sits as [page][half][16 tokens][128 B] (one box per page); P =
//    exp2(S') goes back to its S buffer as bf16 and O += P V is four MMAs
//    (one per page) with A = P from TMEM and B = V as an MN-major operand.
//    Eight TMA boxes per 32 KB tile, issued by two producer warps (K and V).
//  * Warp roles: warps 0-3 softmax and epilogue (one TMEM lane quarter
//    each), warp 4 allocates TMEM and issues the MMAs (one elected lane),
//    warp 5 reads the block table and issues the K boxes, warp 6 the V
//    boxes.
//  * Hand-offs are mbarriers: full / empty per ring slot, s_full / p_full /
//    o_done per S buffer, q_full per piece.
//  * The running maximum is a reference that moves only when a row's new
//    maximum exceeds it by more than kRescaleLog2 (base-2 units), so the O
//    rescale (a TMEM read-modify-write behind the previous P V) is rare.
//  * On a sequence's first tile P V is accumulated from P = P_hi + P_lo, two
//    bf16 terms, so that P carries ~16 bits like the fp32 row sum it is
//    divided by (rows with a handful of visible keys would otherwise show
//    P's bf16 rounding).
//  * A piece that covers a whole segment writes bf16 out and the LSE; a
//    split segment's pieces write fp32 partials to the workspace, one per
//    key-split copy (O as [D/4][R] float4, so that a warp's stores are
//    contiguous), which verify_tc_merge_kernel combines across the whole
//    GPU right after this kernel.  As a separate kernel the merge also lets
//    the next call's CTAs take the SMs this grid leaves, and run their
//    prologue and first copies while it merges; one CTA merging a
//    segment's partials alone, or every CTA merging after a grid-wide
//    barrier, kept the SMs busy and exposed that prologue.
//  * K/V copies run before griddepcontrol.wait only for tiles that lie
//    wholly in the prefix; tiles holding draft positions
//    (which the previous kernel on the stream may have just written) are
//    copied after it, and so is Q.
//  * Every wait is bounded; a timeout sets SF_DEVICE_TIMEOUT, stops every
//    role, waits (bounded) for copies and MMAs in flight and frees TMEM.
#include <cmath>
#include <mutex>

#include "attn_common.cuh"
#include "sf_host.h"

namespace sf {

constexpr int kTcThreads = 224;
constexpr int kTcSoftmaxThreads = 128;
constexpr int kTcMmaWarp = 4;
constexpr int kTcKWarp = 5;
constexpr int kTcVWarp = 6;
constexpr uint32_t kTmemCols = 512;
constexpr int kNumS = 4;  // S buffers (64 columns each)
// TMEM columns: O [0, D), Q [128, 128 + D/2), S_b [192 + 64 b, 256 + 64 b);
// within S_b the bf16 P of the tile overwrites columns [0, 32) and, on a
// sequence's first tile, its low part P_lo columns [32, 64).
constexpr uint32_t kTmemO = 0, kTmemQ = 128, kTmemS = 192;
constexpr float kRescaleLog2 = 8.f;
// The segment-aligned partition is used while its largest piece is at most
// this many tiles above the balanced share (a second piece in a CTA costs
// about that much: another Q load, epilogue and pipeline start).
constexpr int kAlignSlackTiles = 3;
// Registers per thread: low enough that a merge-kernel CTA (launched early,
// waiting for this grid) fits next to a split CTA -- registers are
// partitioned per SM sub-partition (16K each), and warps w and w + 4 of
// both CTAs share one.
constexpr int kTcMaxRegs = 128;
constexpr int kTcNamedTmem = 1;     // softmax warps + MMA warp: TMEM allocated
constexpr int kTcNamedSoftmax = 2;  // softmax warps: epilogue exchange

template <int D>
struct TcConfig {
  static constexpr int kStages = D == 128 ? 6 : 12;  // 192 KB of ring either way
};

template <int D, int STAGES, int F>
struct TcSmem {
  static constexpr int kTileBytes = kTileTokens * D * 2;  // one tensor, one tile
  static constexpr int kStageBytes = 2 * kTileBytes;      // K then V
  static constexpr int kBarOffset = STAGES * kStageBytes;
  // full[S], empty[S], s_full[NS], p_full[NS], o_done[NS], q_full, fin
  static constexpr int kNumBars = 2 * STAGES + 3 * kNumS + 2;
  static constexpr int kMiscOffset = kBarOffset + 8 * kNumBars;
  static constexpr int kMiscInts = 16;
  static constexpr int kRowsPerCopy = 128 / F;
  // epilogue exchange: (max, sum) of every lane, then 32 O columns of the
  // copies kap > 0, column-major so that a warp's stores hit distinct banks
  static constexpr int kMlOffset = kMiscOffset + 4 * kMiscInts;  // float2 [128]
  static constexpr int kXOffset = kMlOffset + 8 * 128;            // float [F-1][32][RPK]
  static constexpr int kXFloats = (F - 1) * 32 * kRowsPerCopy;
  static constexpr int kPrefixOffset = kXOffset + 4 * kXFloats;
  // tiles prefix [B+1] | seq lens [B] | aligned CTA prefix [B+1]
  static int bytes(int B) { return 1024 + kPrefixOffset + 4 * (3 * B + 3); }
};

// tcgen05.ld / st of N consecutive 32-bit columns of the thread's lane.
template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t (&v)[N]) {
  if constexpr (N == 64) tmem_ld_32x32b_x64(taddr, v);
  else if constexpr (N == 32) tmem_ld_32x32b_x32(taddr, v);
  else if constexpr (N == 16) tmem_ld_32x32b_x16(taddr, v);
  else tmem_ld_32x32b_x8(taddr, v);
}
template <int N>
__device__ __forceinline__ void tmem_st_cols(uint32_t taddr, const uint32_t (&v)[N]) {
  if constexpr (N == 32) tmem_st_32x32b_x32(taddr, v);
  else if constexpr (N == 16) tmem_st_32x32b_x16(taddr, v);
  else tmem_st_32x32b_x8(taddr, v);
}

// The work partition of the split kernel, decided identically by every CTA
// (of the split kernel and of its merge kernel) from seq_lens:
//  * balanced: the batch's tiles in one ordered list cut into G equal
//    ranges (a CTA may hold pieces of several segments);
//  * segment-aligned: segment s gets ceil(tiles_s / Ta) CTAs and every CTA
//    holds one piece, with the smallest Ta whose pieces fit the grid --
//    chosen when Ta is close to the balanced share.
// s_prefix holds the exclusive prefix of per-sequence tile counts
// (tile_prefix); s_cpre receives, for the aligned partition, the first CTA
// of each sequence; s_scratch is one int per warp.  Every thread calls it.
struct TcPartition {
  TilePartition part;  // the balanced partition (also defines Tot and G)
  bool aligned;
  int Ta;
};

template <int NT>
__device__ TcPartition tc_partition(const AttnParams &p, const int *s_prefix, int *s_cpre,
                                    int *s_scratch) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t Tot = static_cast<uint32_t>(p.H_kv) * static_cast<uint32_t>(s_prefix[p.B]);
  const int G = Tot < static_cast<uint32_t>(p.G) ? static_cast<int>(Tot) : p.G;
  TcPartition tp;
  tp.part = TilePartition{Tot, static_cast<uint32_t>(G), Tot / G, Tot % G};
  tp.aligned = false;
  tp.Ta = 0;
  const int S = p.B * p.H_kv;
  if (p.G > S) {
    int Ta = static_cast<int>((Tot + static_cast<uint32_t>(p.G - S) - 1) / static_cast<uint32_t>(p.G - S));
    const int Tmin = static_cast<int>((Tot + p.G - 1) / p.G);
    tp.aligned = Ta <= Tmin + kAlignSlackTiles;
    // the smallest piece length whose pieces still fit the grid (Ta always
    // does: each segment's ceiling adds less than one CTA)
#pragma unroll 1
    for (int cand = Tmin; tp.aligned && cand < Ta; ++cand) {
      int local = 0;
#pragma unroll 1
      for (int b = tid; b < p.B; b += NT) local += (s_prefix[b + 1] - s_prefix[b] + cand - 1) / cand;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) local += __shfl_xor_sync(0xffffffffu, local, o);
      if (lane == 0) s_scratch[warp] = local;
      __syncthreads();
      int need = 0;
#pragma unroll 1
      for (int w = 0; w < NT / 32; ++w) need += s_scratch[w];
      __syncthreads();
      if (static_cast<long long>(need) * p.H_kv <= p.G) {
        Ta = cand;
        break;
      }
    }
    tp.Ta = Ta;
  }
  if (tp.aligned) {
    aligned_prefix<NT>(p, s_prefix, tp.Ta, s_cpre, s_scratch);
    __syncthreads();
  }
  return tp;
}

// First CTA and number of pieces of segment (b, h) under partition tp.
__device__ __forceinline__ void tc_segment(const TcPartition &tp, const AttnParams &p,
                                           const int *s_prefix, const int *s_cpre, int b, int h,
                                           int &c_first, int &n_pieces) {
  const int tiles_b = s_prefix[b + 1] - s_prefix[b];
  if (tp.aligned) {
    const int ns = (tiles_b + tp.Ta - 1) / tp.Ta;
    c_first = s_cpre[b] + h * ns;
    n_pieces = ns;
  } else {
    const uint32_t first = static_cast<uint32_t>(p.H_kv) * static_cast<uint32_t>(s_prefix[b]) +
                           static_cast<uint32_t>(h * tiles_b);
    c_first = static_cast<int>(tp.part.owner(first));
    n_pieces = static_cast<int>(tp.part.owner(first + tiles_b - 1)) - c_first + 1;
  }
}

template <int D, int STAGES, int F>
__global__ void __maxnreg__(kTcMaxRegs)
verify_attention_tc_kernel(const __grid_constant__ CUtensorMap tmap_k,
                           const __grid_constant__ CUtensorMap tmap_v,
                           const __grid_constant__ AttnParams p) {
  using L = TcSmem<D, STAGES, F>;
  constexpr int HALVES = D / 64;
  constexpr int kPageHalfBytes = kPageTokens * kRowBytes;  // 16 tokens x 64 columns
  constexpr int kPageBytes = HALVES * kPageHalfBytes;      // one page of one tensor
  constexpr int RPK = 128 / F;                             // M rows per key copy
  constexpr int KPL = 64 / F;                              // keys per lane and tile
  constexpr uint32_t kKSbo = HALVES == 2 ? 2048u : 1024u;  // 8-key atoms of a K tile
  constexpr float kLn2 = 0.6931471805599453f;
  constexpr uint32_t kIdescQK = idesc_bf16_f32(128, 64, 0, 0);  // Q (TMEM), K K-major
  constexpr uint32_t kIdescPV = idesc_bf16_f32(128, D, 0, 1);   // P (TMEM), V MN-major
  constexpr int kQWords = D / 2;                                 // 32-bit columns of a Q row
  // barrier indices
  constexpr int FULL = 0, EMPTY = STAGES, SFULL = 2 * STAGES, PFULL = SFULL + kNumS,
                ODONE = PFULL + kNumS, QFULL = ODONE + kNumS, FIN = QFULL + 1;
  constexpr uint32_t NS = kNumS;

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t ring = smem_addr(smem);
  const uint32_t bars = ring + L::kBarOffset;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };
  int *s_misc = reinterpret_cast<int *>(smem + L::kMiscOffset);
  // s_misc: [0] TMEM base, [1] abort word, [2] tiles with K issued, [3] tiles
  // whose full barrier the MMA warp observed, [4] tiles with V issued
  volatile int *s_abort = s_misc + 1;
  int *s_prefix = reinterpret_cast<int *>(smem + L::kPrefixOffset);
  int *s_len = s_prefix + p.B + 1;
  int *s_cpre = s_len + p.B;  // aligned partition: first CTA of each sequence

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  grid_launch_dependents();
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bar(FULL + s), 2);  // one arrival per producer warp (with its bytes)
      mbar_init(bar(EMPTY + s), 1);
    }
    for (int x = 0; x < kNumS; ++x) {
      mbar_init(bar(SFULL + x), 1);
      mbar_init(bar(PFULL + x), kTcSoftmaxThreads);
      mbar_init(bar(ODONE + x), 1);
    }
    mbar_init(bar(QFULL), kTcSoftmaxThreads);
    mbar_init(bar(FIN), 1);
    fence_mbar_init();
    prefetch_tensormap(&tmap_k);
    prefetch_tensormap(&tmap_v);
    s_misc[1] = 0;
    s_misc[2] = 0;
    s_misc[3] = 0;
    s_misc[4] = 0;
  }
  tile_prefix<kTcThreads>(p, s_prefix, s_len, s_misc + 8);
  __syncthreads();

  const TcPartition tp = tc_partition<kTcThreads>(p, s_prefix, s_cpre, s_misc + 8);
  const TilePartition &part = tp.part;
  const bool aligned = tp.aligned;
  const int Ta = tp.Ta;
  const uint32_t Tot = part.Tot;
  const int G = static_cast<int>(part.G);
  Piece apc{};  // the aligned partition's piece of this CTA
  uint32_t t_begin = Tot, t_end = Tot;
  if (aligned) {
    const int c = static_cast<int>(blockIdx.x);
    if (c < s_cpre[p.B]) {
      int lo = 0, hi = p.B - 1;  // last sequence whose first CTA is <= c
      while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (s_cpre[mid] <= c) lo = mid; else hi = mid - 1;
      }
      const int b = lo, tiles_b = s_prefix[b + 1] - s_prefix[b];
      const int ns = (tiles_b + Ta - 1) / Ta, local = c - s_cpre[b];
      const int h = local / ns, q = local % ns;
      apc.b = b;
      apc.h_kv = h;
      apc.seg = b * p.H_kv + h;
      apc.lt0 = q * tiles_b / ns;
      apc.n_tiles = (q + 1) * tiles_b / ns - apc.lt0;
      apc.c_first = s_cpre[b] + h * ns;
      apc.n_pieces = ns;
      apc.T = s_len[b];
      apc.Lb = apc.T - p.n_q;
      t_begin = static_cast<uint32_t>(p.H_kv) * static_cast<uint32_t>(s_prefix[b]) +
                static_cast<uint32_t>(h * tiles_b + apc.lt0);
      t_end = t_begin + static_cast<uint32_t>(apc.n_tiles);
    }
  } else if (static_cast<int>(blockIdx.x) < G) {
    t_begin = part.start(blockIdx.x);
    t_end = part.start(blockIdx.x + 1);
  }
  // the piece starting at tile t of this CTA's range
  auto piece_at = [&](uint32_t t) -> Piece {
    return aligned ? apc : locate_piece(t, t_end, part, s_prefix, s_len, p);
  };

  if (warp == kTcKWarp || warp == kTcVWarp) {
    // ------------------------------------------------------------------
    // producers: lanes 0-3 of the K warp issue the K boxes of a tile (one
    // per page), lanes 0-3 of the V warp its V boxes; each warp arrives on
    // the slot's full barrier with its own bytes.
    // ------------------------------------------------------------------
    const bool is_k = warp == kTcKWarp;
    const uint64_t policy = l2_policy_evict_first();
    bool waited = false;
    uint32_t n = 0;  // tiles issued by this CTA
    bool ok = true;
    for (uint32_t t = t_begin; t < t_end && ok;) {
      const Piece pc = piece_at(t);
      t += pc.n_tiles;
      // page ids of tiles base .. base+7 of the piece: lane l holds tile
      // base + l/4, page l%4
      auto window = [&](int base) -> int {
        const int lt = pc.lt0 + base + (lane >> 2);
        const int lp = lt * kPagesPerTile + (lane & 3);
        int id = kBeyondEnd;
        if (base + (lane >> 2) < pc.n_tiles && lp * kPageTokens < pc.T)
          id = p.block_table[(size_t)pc.b * p.max_pages + lp];
        return id;
      };
      int ids = kBeyondEnd;
      for (int it = 0; it < pc.n_tiles; ++it, ++n) {
        if ((it & 7) == 0) ids = window(it);
        const int pg = lane & 3;
        const int phys = __shfl_sync(0xffffffffu, ids, ((it & 7) << 2) + pg);
        const int slot = static_cast<int>(n % STAGES);
        if (n >= static_cast<uint32_t>(STAGES)) {
          int w = 1;
          if (lane == 0) w = mbar_wait_or_abort(bar(EMPTY + slot), ((n / STAGES) - 1) & 1u, s_abort);
          if (!__shfl_sync(0xffffffffu, w, 0)) {
            ok = false;
            break;
          }
        }
        // a tile that holds draft positions may have been written by the
        // previous kernel on the stream: copy it only after that kernel
        if (!waited && (pc.lt0 + it + 1) * kTileTokens > pc.Lb) {
          grid_dependency_wait();
          waited = true;
        }
        if (lane == 0) mbar_arrive_expect_tx(bar(FULL + slot), L::kTileBytes);
        __syncwarp();
        if (lane < kPagesPerTile) {
          // pages past the sequence end or outside the pool load as zeros
          int row = p.oob_row;
          if (phys != kBeyondEnd) {
            if (phys < 0 || phys >= p.num_pages) {
              if (is_k) set_status(p.status, SF_DEVICE_BAD_PAGE);
            } else {
              row = (phys * p.H_kv + pc.h_kv) * kPageTokens;
            }
          }
          const uint32_t stage = ring + slot * L::kStageBytes;
          if (is_k) {
            const uint32_t dst = stage + pg * kPageBytes;
            if constexpr (HALVES == 2) tma_load_4d(dst, &tmap_k, 0, 0, 0, row / 8, bar(FULL + slot), policy);
            else tma_load_2d(dst, &tmap_k, 0, row, bar(FULL + slot), policy);
          } else {
            const uint32_t dst = stage + L::kTileBytes + pg * kPageBytes;
            if constexpr (HALVES == 2) tma_load_3d(dst, &tmap_v, 0, row, 0, bar(FULL + slot), policy);
            else tma_load_2d(dst, &tmap_v, 0, row, bar(FULL + slot), policy);
          }
        }
        __syncwarp();
        if (lane == 0) s_misc[is_k ? 2 : 4] = static_cast<int>(n + 1);
      }
    }
  } else if (warp == kTcMmaWarp) {
    // ------------------------------------------------------------------
    // MMA warp.  TMEM is allocated after the previous kernel on the stream
    // has completed.  Then the whole warp polls, one elected lane issues and
    // commits.  Q K^T of tile m needs its K tile (full), its S buffer free
    // (P V of tile m - NS issued: the MMAs run in issue order, so that P V
    // reads its P before Q K^T overwrites it) and, for the first tile of a
    // piece, the piece's Q (q_full); P V of tile m needs its P (p_full).
    // The two streams are issued as soon as their conditions hold.
    // ------------------------------------------------------------------
    grid_dependency_wait();
    tmem_alloc(smem_addr(s_misc), kTmemCols);
    tmem_relinquish_alloc_permit();
    tc_fence_before_sync();
    named_bar_sync(kTcNamedTmem, kTcSoftmaxThreads + 32);
    tc_fence_after_sync();
    const uint32_t tmem = static_cast<uint32_t>(s_misc[0]);
    uint32_t qk = 0, pv = 0;      // next tile to multiply, CTA-wide counters
    uint32_t qk_piece_end = 0;    // end of the piece of tile qk
    uint32_t pv_piece_start = 0;  // first tile of the piece of tile pv
    uint32_t pv_piece_end = 0;
    int pv_lt0 = 0;               // first tile of pv's piece within its sequence
    uint32_t t_qk = t_begin, t_pv = t_begin;  // piece cursors (global tiles)
    int q_piece = -1, q_ready = -1;           // piece of tile qk, pieces with Q
    uint32_t total = 0;
    for (uint32_t t = t_begin; t < t_end;) {
      const Piece pc = piece_at(t);
      t += pc.n_tiles;
      total += pc.n_tiles;
    }
    unsigned long long t0 = 0;
    bool ok = true;
    while (pv < total && ok) {
      bool progress = false;
      if (qk == qk_piece_end && qk < total) {
        const Piece pc = piece_at(t_qk);
        t_qk += pc.n_tiles;
        qk_piece_end += pc.n_tiles;
        ++q_piece;
      }
      if (pv == pv_piece_end) {
        const Piece pc = piece_at(t_pv);
        t_pv += pc.n_tiles;
        pv_piece_start = pv_piece_end;
        pv_lt0 = pc.lt0;
        pv_piece_end += pc.n_tiles;
      }
      if (qk < total && qk < pv + NS) {
        bool ready = true;
        if (q_ready < q_piece) {
          ready = mbar_test_wait(bar(QFULL), static_cast<uint32_t>(q_piece) & 1u);
          if (ready) q_ready = q_piece;
        }
        const uint32_t slot = qk % STAGES;
        if (ready) ready = mbar_test_wait(bar(FULL + slot), (qk / STAGES) & 1u);
        if (__all_sync(0xffffffffu, ready)) {
          tc_fence_after_sync();
          if (lane == 0) s_misc[3] = static_cast<int>(qk + 1);
          const uint32_t kb = ring + slot * L::kStageBytes;
          const uint32_t d = tmem + kTmemS + (qk % NS) * 64u;
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              // K step kk: columns 16kk .. 16kk+15 = 32-byte column kk%4 of half kk/4
              const uint64_t b = smem_desc_sw128(kb + (kk >> 2) * 1024 + (kk & 3) * 32, 16, kKSbo);
              tc_mma_ts(d, tmem + kTmemQ + kk * 8, b, kIdescQK, kk > 0 ? 1u : 0u);
            }
            tc_commit(bar(SFULL + qk % NS));
          }
          __syncwarp();
          ++qk;
          progress = true;
        }
      }
      if (pv < qk) {
        const bool ready = mbar_test_wait(bar(PFULL + pv % NS), (pv / NS) & 1u);
        if (__all_sync(0xffffffffu, ready)) {
          tc_fence_after_sync();
          const uint32_t slot = pv % STAGES;
          const uint32_t vb = ring + slot * L::kStageBytes + L::kTileBytes;
          const bool first = pv == pv_piece_start;
          const bool seq_first = first && pv_lt0 == 0;  // the sequence's first tile: P_hi + P_lo
          if (elect_one()) {
#pragma unroll
            for (int j = 0; j < kTileTokens / 16; ++j) {
              // V page j = keys 16j..16j+15 (K): 8-key groups 1024 B apart;
              // the 64-column halves of N are kPageHalfBytes apart
              const uint64_t b = smem_desc_sw128(vb + j * kPageBytes, kPageHalfBytes, 1024);
              const uint32_t pb = tmem + kTmemS + (pv % NS) * 64u + j * 8u;
              tc_mma_ts(tmem + kTmemO, pb, b, kIdescPV, (first && j == 0) ? 0u : 1u);
              if (seq_first) tc_mma_ts(tmem + kTmemO, pb + 32u, b, kIdescPV, 1u);
            }
            tc_commit(bar(ODONE + pv % NS));
            tc_commit(bar(EMPTY + slot));
          }
          __syncwarp();
          ++pv;
          progress = true;
        }
      }
      if (progress) {
        t0 = 0;
      } else {
        // nothing ready: bounded wait (the abort word stops it early)
        if (t0 == 0) t0 = global_timer_ns();
        if (*s_abort) ok = false;
        else if (global_timer_ns() - t0 > kWaitBudgetNs) {
          *s_abort = 1;
          ok = false;
        }
        ok = __all_sync(0xffffffffu, ok);
      }
    }
    // every MMA issued has completed once this arrives
    if (elect_one()) tc_commit(bar(FIN));
    __syncwarp();
    (void)mbar_wait_bounded(bar(FIN), 0);
  } else {
    // ------------------------------------------------------------------
    // softmax + epilogue.  Thread tid owns TMEM lane tid: key copy kap =
    // tid / RPK (keys kap*KPL .. kap*KPL+KPL-1 of every tile) of query row
    // r = tid % RPK (rows >= R are padding).  Each lane keeps its own
    // reference, sum and O over its keys.
    // ------------------------------------------------------------------
    const int kap = tid / RPK, r = tid % RPK;
    const bool valid = r < p.R;
    const int qi = valid ? r / p.group : 0, qj = valid ? r % p.group : 0;
    float2 *s_ml = reinterpret_cast<float2 *>(smem + L::kMlOffset);
    float *s_x = reinterpret_cast<float *>(smem + L::kXOffset);
    // every lane waits (and acquires); the warp leaves together if any failed,
    // so the warp-collective tcgen05 instructions always see a full warp
    auto wwait = [&](uint32_t b, uint32_t parity) -> bool {
      const bool w = mbar_wait_or_abort(b, parity, s_abort);
      return __all_sync(0xffffffffu, w);
    };
    auto q_row = [&](const Piece &pc) -> const __nv_bfloat16 * {
      return p.q + (((size_t)pc.b * p.n_q + qi) * p.H_q + (size_t)pc.h_kv * p.group + qj) * D;
    };
    // this lane's Q row of piece pc (zeros for padding rows) into registers,
    // then into TMEM
    auto fetch_q = [&](const Piece &pc, uint32_t (&qw)[kQWords]) {
      const uint4 *src = reinterpret_cast<const uint4 *>(q_row(pc));
#pragma unroll
      for (int u = 0; u < D / 8; ++u) {
        const uint4 v = valid ? __ldg(src + u) : make_uint4(0u, 0u, 0u, 0u);
        qw[4 * u] = v.x; qw[4 * u + 1] = v.y; qw[4 * u + 2] = v.z; qw[4 * u + 3] = v.w;
      }
    };
    auto store_q = [&](const uint32_t (&qw)[kQWords], uint32_t tl) {
#pragma unroll
      for (int c = 0; c < kQWords; c += 32) {
        uint32_t part[32];
#pragma unroll
        for (int k = 0; k < 32; ++k) part[k] = qw[c + k];
        tmem_st_32x32b_x32(tl + kTmemQ + c, part);
      }
    };

    Piece pc0{};
    if (t_begin < t_end) {
      pc0 = piece_at(t_begin);
      if (valid) {
        const char *row = reinterpret_cast<const char *>(q_row(pc0));
        for (int x = 0; x < D * 2; x += 128) prefetch_l2(row + x);
      }
    }
    grid_dependency_wait();
    {
      // the Q loads are in flight while the MMA warp allocates TMEM
      uint32_t qw[kQWords];
      if (t_begin < t_end) fetch_q(pc0, qw);
      named_bar_sync(kTcNamedTmem, kTcSoftmaxThreads + 32);
      tc_fence_after_sync();
      const uint32_t tl0 = static_cast<uint32_t>(s_misc[0]) + (static_cast<uint32_t>(warp * 32) << 16);
      if (t_begin < t_end) store_q(qw, tl0);
    }
    const uint32_t tmem = static_cast<uint32_t>(s_misc[0]);
    const uint32_t tl = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    tmem_wait_st();
    tc_fence_before_sync();
    mbar_arrive(bar(QFULL));

    uint32_t n = 0;
    bool ok = true;
    int pi = 0;  // piece index in this CTA
    for (uint32_t t = t_begin; t < t_end; ++pi) {
      const Piece pc = pi == 0 ? pc0 : piece_at(t);
      t += pc.n_tiles;
      if (t < t_end) {
        // the next piece's Q rows into L2 (read after this piece's tiles)
        const Piece nx = piece_at(t);
        if (valid) {
          const char *row = reinterpret_cast<const char *>(q_row(nx));
          for (int x = 0; x < D * 2; x += 128) prefetch_l2(row + x);
        }
      }

      // last visible key position of this row (draft row i sees L_b + i)
      const int lim = valid ? pc.Lb + min(qi, p.n_q - 1) : -1;
      float ref = -INFINITY, l_run = 0.f;
      for (int it = 0; it < pc.n_tiles && ok; ++it, ++n) {
        const uint32_t sb = tl + kTmemS + (n % NS) * 64u;  // this tile's S buffer
        if (!wwait(bar(SFULL + n % NS), (n / NS) & 1u)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        uint32_t sv[KPL];
        tmem_ld_cols<KPL>(sb + kap * KPL, sv);
        const int tile_pos = (pc.lt0 + it) * kTileTokens;
        const bool split_p = pc.lt0 + it == 0;  // P as two bf16 terms on the sequence's first tile
        const int valid_keys = pc.T - tile_pos;
        if (valid_keys < kTileTokens) {
          // V rows past the sequence end hold whatever the page holds: zero
          // them so that 0 * v stays 0 in P V (read after p_full)
          uint8_t *vt = smem + (n % STAGES) * L::kStageBytes + L::kTileBytes;
          for (int idx = tid; idx < (kTileTokens - valid_keys) * HALVES * 8; idx += kTcSoftmaxThreads) {
            const int tok = valid_keys + idx / (HALVES * 8);
            const int rem = idx % (HALVES * 8);
            *reinterpret_cast<uint4 *>(vt + (tok >> 4) * kPageBytes + (rem >> 3) * kPageHalfBytes +
                                       (tok & 15) * kRowBytes + (rem & 7) * 16) = make_uint4(0u, 0u, 0u, 0u);
          }
          fence_proxy_async_smem();
        }
        // this lane's keys kap*KPL .. kap*KPL + KPL-1 (raw scores; the
        // scale, > 0, is applied to the maximum and folded into the exponent)
        // tile maximum as a tree (a chain of KPL dependent max operations
        // is ~5 cycles each on the softmax's critical path)
        float mx;
        {
          float t[KPL / 2];
#pragma unroll
          for (int c = 0; c < KPL / 2; ++c) t[c] = fmaxf(__uint_as_float(sv[2 * c]), __uint_as_float(sv[2 * c + 1]));
#pragma unroll
          for (int w = KPL / 4; w >= 1; w >>= 1) {
#pragma unroll
            for (int c = 0; c < w; ++c) t[c] = fmaxf(t[c], t[c + w]);
          }
          mx = t[0];
        }
        const int key0 = tile_pos + kap * KPL;
        if (key0 + KPL - 1 > lim) {
          // causal mask of the draft block, positions past the end, padding rows
          mx = -INFINITY;
#pragma unroll
          for (int c = 0; c < KPL; ++c) {
            if (key0 + c > lim) sv[c] = __float_as_uint(-INFINITY);
            mx = fmaxf(mx, __uint_as_float(sv[c]));
          }
        }
        mx *= p.scale_log2;
        // move the reference only when the maximum outgrows it
        float alpha = 1.f;
        if (mx > ref + kRescaleLog2) {
          if (ref != -INFINITY) alpha = exp2f(ref - mx);
          ref = mx;
        }
        const float mu = ref == -INFINITY ? 0.f : ref;
        uint32_t mine[KPL / 2], mine_lo[KPL / 2];
        float ps[KPL / 2];  // pair sums, added as a tree below
#pragma unroll
        for (int c2 = 0; c2 < KPL / 2; ++c2) {
          const float p0 = fast_exp2(fmaf(__uint_as_float(sv[2 * c2]), p.scale_log2, -mu));
          const float p1 = fast_exp2(fmaf(__uint_as_float(sv[2 * c2 + 1]), p.scale_log2, -mu));
          ps[c2] = p0 + p1;
          if (split_p) split_bf16x2(p0, p1, mine[c2], mine_lo[c2]);
          else mine[c2] = pack_bf16x2(p0, p1);
        }
#pragma unroll
        for (int w = KPL / 4; w >= 1; w >>= 1) {
#pragma unroll
          for (int c = 0; c < w; ++c) ps[c] += ps[c + w];
        }
        const float rs = ps[0];
        l_run = l_run * alpha + rs;
        if (__any_sync(0xffffffffu, alpha != 1.f)) {
          // O *= alpha after the P V of tile n-1 (it > 0 here: the first
          // tile of a piece starts with ref = -inf, so alpha = 1)
          if (!wwait(bar(ODONE + (n - 1) % NS), ((n - 1) / NS) & 1u)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
#pragma unroll 1
          for (int ch = 0; ch < D / 32; ++ch) {
            uint32_t ov[32];
            tmem_ld_32x32b_x32(tl + kTmemO + ch * 32, ov);
#pragma unroll
            for (int c = 0; c < 32; ++c) ov[c] = __float_as_uint(__uint_as_float(ov[c]) * alpha);
            tmem_st_32x32b_x32(tl + kTmemO + ch * 32, ov);
          }
        }
        // P over the scores: this lane's keys, zeros for the other copies'
        // keys (the A operand of P V covers the whole tile)
        {
          uint32_t pk[32];
#pragma unroll
          for (int c = 0; c < 32; ++c) pk[c] = (c / (KPL / 2) == kap) ? mine[c % (KPL / 2)] : 0u;
          tmem_st_32x32b_x32(sb, pk);
          if (split_p) {  // the sequence's first tile: P_lo too (warp-uniform)
#pragma unroll
            for (int c = 0; c < 32; ++c) pk[c] = (c / (KPL / 2) == kap) ? mine_lo[c % (KPL / 2)] : 0u;
            tmem_st_32x32b_x32(sb + 32, pk);
          }
        }
        tmem_wait_st();
        tc_fence_before_sync();
        mbar_arrive(bar(PFULL + n % NS));
      }

      // ---- the next piece's Q (every Q K^T of this piece has completed:
      // its last score tile was read above), so that the next piece's first
      // Q K^T overlaps this epilogue ----
      if (ok && t < t_end) {
        uint32_t qw[kQWords];
        fetch_q(piece_at(t), qw);
        store_q(qw, tl);
        tmem_wait_st();
        tc_fence_before_sync();
        mbar_arrive(bar(QFULL));
      }

      // ---- epilogue of the piece ----
      if (ok) {
        const uint32_t last = n - 1;
        ok = wwait(bar(ODONE + last % NS), (last / NS) & 1u);
      }
      // all four warps take the exchange barriers below, or all skip them
      if (!named_bar_and(kTcNamedSoftmax, kTcSoftmaxThreads, ok)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      if (pc.n_pieces > 1) {
        // a split segment: each key-split copy writes its own partial
        // (relative to its own reference); the merge kernel combines the
        // n_pieces x F partials, so no exchange between the copies here
        float *partk = p.partials + ((size_t)(blockIdx.x + pc.seg) * F + kap) * p.slot_stride;
#pragma unroll 1
        for (int ch = 0; ch < D / 32; ++ch) {
          uint32_t ov[32];
          tmem_ld_32x32b_x32(tl + kTmemO + ch * 32, ov);  // warp-wide: every lane loads
          if (valid) {
            float4 *dst = reinterpret_cast<float4 *>(partk) + (size_t)(ch * 8) * p.R + r;
#pragma unroll
            for (int q4 = 0; q4 < 8; ++q4)
              dst[(size_t)q4 * p.R] = make_float4(__uint_as_float(ov[4 * q4]), __uint_as_float(ov[4 * q4 + 1]),
                                                  __uint_as_float(ov[4 * q4 + 2]), __uint_as_float(ov[4 * q4 + 3]));
          }
        }
        if (valid) {
          partk[(size_t)p.R * D + r] = ref;
          partk[(size_t)p.R * D + p.R + r] = l_run;
        }
        tc_fence_before_sync();
        if (!ok) break;
        continue;
      }
      // merge the F copies of each row (M = max reference, w = 2^(ref - M));
      // copy 0 then normalises and writes a whole segment, or leaves a split
      // one's fp32 partial O [R][D] (relative to M), M [R], L [R]
      float M = ref, Ls = l_run;
      if constexpr (F > 1) {
        s_ml[tid] = make_float2(ref, l_run);
        named_bar_sync(kTcNamedSoftmax, kTcSoftmaxThreads);
#pragma unroll
        for (int k = 0; k < F; ++k) M = fmaxf(M, s_ml[k * RPK + r].x);
        Ls = 0.f;
#pragma unroll
        for (int k = 0; k < F; ++k) {
          const float2 v = s_ml[k * RPK + r];
          if (v.x != -INFINITY) Ls += v.y * exp2f(v.x - M);
        }
      }
      const float w = ref == -INFINITY ? 0.f : exp2f(ref - M);
      const bool writer = valid && kap == 0;
      const size_t row = ((size_t)pc.b * p.n_q + qi) * p.H_q + (size_t)pc.h_kv * p.group + qj;
      const bool whole = pc.n_pieces == 1;
      const float inv = whole ? 1.f / Ls : 1.f;
      float *part0 = p.partials + (size_t)(blockIdx.x + pc.seg) * p.slot_stride;
#pragma unroll 1
      for (int ch = 0; ch < D / 32; ++ch) {
        uint32_t ov[32];
        tmem_ld_32x32b_x32(tl + kTmemO + ch * 32, ov);
        float o[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) o[c] = __uint_as_float(ov[c]) * w;
        if constexpr (F > 1) {
          if (kap > 0) {
#pragma unroll
            for (int c = 0; c < 32; ++c) s_x[((kap - 1) * 32 + c) * RPK + r] = o[c];
          }
          named_bar_sync(kTcNamedSoftmax, kTcSoftmaxThreads);
          if (kap == 0) {
#pragma unroll
            for (int k = 1; k < F; ++k) {
#pragma unroll
              for (int c = 0; c < 32; ++c) o[c] += s_x[((k - 1) * 32 + c) * RPK + r];
            }
          }
        }
        if (writer && whole) {
          uint4 *dst = reinterpret_cast<uint4 *>(p.out + row * D + ch * 32);
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4) {
            uint4 wv;
            wv.x = pack_bf16x2(o[8 * q4 + 0] * inv, o[8 * q4 + 1] * inv);
            wv.y = pack_bf16x2(o[8 * q4 + 2] * inv, o[8 * q4 + 3] * inv);
            wv.z = pack_bf16x2(o[8 * q4 + 4] * inv, o[8 * q4 + 5] * inv);
            wv.w = pack_bf16x2(o[8 * q4 + 6] * inv, o[8 * q4 + 7] * inv);
            dst[q4] = wv;
          }
        } else if (writer) {
          // [D/4][R] float4: the warp's 32 rows of one quad are contiguous
          float4 *dst = reinterpret_cast<float4 *>(part0) + (size_t)(ch * 8) * p.R + r;
#pragma unroll
          for (int q4 = 0; q4 < 8; ++q4)
            dst[(size_t)q4 * p.R] = make_float4(o[4 * q4], o[4 * q4 + 1], o[4 * q4 + 2], o[4 * q4 + 3]);
        }
        if constexpr (F > 1) named_bar_sync(kTcNamedSoftmax, kTcSoftmaxThreads);
      }
      if (writer) {
        if (whole) {
          if (p.lse) p.lse[row] = (M + log2f(Ls)) * kLn2;
        } else {
          part0[(size_t)p.R * D + r] = M;
          part0[(size_t)p.R * D + p.R + r] = Ls;
        }
      }
      tc_fence_before_sync();
      if (!ok) break;
    }
    tc_fence_before_sync();
  }

  // ---- teardown: every role is done (or stopped) ----
  __syncthreads();
  if (*s_abort) {
    if (tid == 0) set_status(p.status, SF_DEVICE_TIMEOUT);
    if (warp == kTcKWarp && lane == 0) {
      // copies issued but never consumed: a tile that only one producer warp
      // reached gets the other warp's arrival here, then every issued copy
      // is waited for (bounded) before the shared memory is released
      const uint32_t kI = static_cast<uint32_t>(s_misc[2]), vI = static_cast<uint32_t>(s_misc[4]);
      const uint32_t hi = kI > vI ? kI : vI;
      for (uint32_t x = static_cast<uint32_t>(s_misc[3]); x < hi; ++x) {
        if (x >= kI) mbar_arrive(bar(FULL + x % STAGES));
        if (x >= vI) mbar_arrive(bar(FULL + x % STAGES));
        (void)mbar_wait_bounded(bar(FULL + x % STAGES), (x / STAGES) & 1u);
      }
    }
    __syncthreads();
  }
  if (warp == kTcMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(static_cast<uint32_t>(s_misc[0]), kTmemCols);
  }
}

// --------------------------------------------------------------------------
// Merge of split segments, one CTA per SM (256 threads).  Before the
// dependency wait every CTA recomputes the split kernel's partition from
// seq_lens, so that after it only the partials are read: one item per output
// quad (row r, columns 4c4 .. 4c4+3) of every split segment, consecutive
// threads on consecutive rows of one quad (the [D/4][R] slots make a warp's
// loads contiguous), with the loads of kTcMergeBatch partials in flight at
// once.  A segment's partials are its pieces' key-split copies (F per piece,
// F = 4 / 2 / 1 for R <= 32 / 64 / 128), merged in piece-then-copy order
// (deterministic):
//   M = max_q m_q,  L = sum_q l_q 2^(m_q - M),  O = sum_q 2^(m_q - M) O_q / L,
//   lse = (M + log2 L) ln 2.
// Launched right after the split kernel with programmatic stream
// serialisation: its CTAs are resident while the split grid runs.
// --------------------------------------------------------------------------
constexpr int kTcMergeThreads = 256;
constexpr int kTcMergeBatch = 12;
// 256 threads x 104 registers fit next to a split CTA (224 x 128) on one SM
constexpr int kTcMergeMaxRegs = 104;

template <int D>
__global__ void __maxnreg__(kTcMergeMaxRegs)
verify_tc_merge_kernel(const __grid_constant__ AttnParams p) {
  constexpr float kLn2 = 0.6931471805599453f;
  constexpr int C4 = D / 4;
  extern __shared__ int s_arr[];
  __shared__ int s_scratch[16];
  int *s_prefix = s_arr;             // [B+1]
  int *s_len = s_prefix + p.B + 1;   // [B]
  int *s_cpre = s_len + p.B;         // [B+1]
  grid_launch_dependents();
  tile_prefix<kTcMergeThreads>(p, s_prefix, s_len, s_scratch + 8);
  __syncthreads();
  const TcPartition tp = tc_partition<kTcMergeThreads>(p, s_prefix, s_cpre, s_scratch + 8);
  grid_dependency_wait();
  // work units of kTcMergeThreads items of one segment (32-bit indices:
  // the units of all segments number fewer than 2^31)
  const int per_seg = p.R * C4;
  const int units_per_seg = (per_seg + kTcMergeThreads - 1) / kTcMergeThreads;
  const int units = p.B * p.H_kv * units_per_seg;
  const size_t stride = (size_t)p.slot_stride;
#pragma unroll 1
  for (int unit = blockIdx.x; unit < units; unit += gridDim.x) {
    const int seg = unit / units_per_seg;
    const int rem = (unit - seg * units_per_seg) * kTcMergeThreads + threadIdx.x;
    if (rem >= per_seg) continue;
    const int c4 = rem / p.R, r = rem - c4 * p.R;
    const int b = seg / p.H_kv, h_kv = seg - b * p.H_kv;
    int c_first, n_pieces;
    tc_segment(tp, p, s_prefix, s_cpre, b, h_kv, c_first, n_pieces);
    if (n_pieces <= 1) continue;  // the split kernel wrote the output
    const int F = p.R <= 32 ? 4 : (p.R <= 64 ? 2 : 1);  // key-split copies per piece
    const float *slot0 = p.partials + (size_t)(c_first + seg) * F * stride;
    n_pieces *= F;
    float M = -INFINITY, Ls = 0.f;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int q0 = 0; q0 < n_pieces; q0 += kTcMergeBatch) {
      float mv[kTcMergeBatch], lv[kTcMergeBatch];
      float4 xv[kTcMergeBatch];
#pragma unroll
      for (int u = 0; u < kTcMergeBatch; ++u) {
        const bool in = q0 + u < n_pieces;
        const float *slot = slot0 + (size_t)(q0 + u) * stride;
        mv[u] = in ? slot[(size_t)p.R * D + r] : -INFINITY;
        lv[u] = in ? slot[(size_t)p.R * D + p.R + r] : 0.f;
        xv[u] = in ? reinterpret_cast<const float4 *>(slot)[(size_t)c4 * p.R + r]
                   : make_float4(0.f, 0.f, 0.f, 0.f);
      }
      float Mb = M;
#pragma unroll
      for (int u = 0; u < kTcMergeBatch; ++u) Mb = fmaxf(Mb, mv[u]);
      // weights 2^(m - Mb) <= 1 (fast_exp2(-inf) = 0: pieces without a
      // visible key for this row, and the empty running state of the first batch)
      const float a = fast_exp2(M - Mb);
      Ls *= a;
      acc.x *= a; acc.y *= a; acc.z *= a; acc.w *= a;
#pragma unroll
      for (int u = 0; u < kTcMergeBatch; ++u) {
        const float w = fast_exp2(mv[u] - Mb);
        Ls += lv[u] * w;
        acc.x += xv[u].x * w; acc.y += xv[u].y * w; acc.z += xv[u].z * w; acc.w += xv[u].w * w;
      }
      M = Mb;
    }
    const int i = r / p.group, j = r % p.group;
    const size_t row = ((size_t)b * p.n_q + i) * p.H_q + (size_t)h_kv * p.group + j;
    const float inv = 1.f / Ls;
    uint2 packed;
    packed.x = pack_bf16x2(acc.x * inv, acc.y * inv);
    packed.y = pack_bf16x2(acc.z * inv, acc.w * inv);
    *reinterpret_cast<uint2 *>(p.out + row * D + 4 * c4) = packed;
    if (p.lse && c4 == 0) p.lse[row] = (M + log2f(Ls)) * kLn2;
  }
}

// --------------------------------------------------------------------------
// host side
// --------------------------------------------------------------------------
using TcKernelFn = void (*)(const CUtensorMap, const CUtensorMap, const AttnParams);

// Copies of each query row (lanes per row): as many as 128 TMEM lanes allow,
// at most 4.
static int tc_key_split(int R) { return R <= 32 ? 4 : (R <= 64 ? 2 : 1); }

template <int D>
static TcKernelFn tc_kernel(int F) {
  constexpr int S = TcConfig<D>::kStages;
  if (F == 4) return verify_attention_tc_kernel<D, S, 4>;
  if (F == 2) return verify_attention_tc_kernel<D, S, 2>;
  return verify_attention_tc_kernel<D, S, 1>;
}

template <int D>
static int tc_bytes(int F, int B) {
  constexpr int S = TcConfig<D>::kStages;
  if (F == 4) return TcSmem<D, S, 4>::bytes(B);
  if (F == 2) return TcSmem<D, S, 2>::bytes(B);
  return TcSmem<D, S, 1>::bytes(B);
}

int tc_smem_bytes(int head_dim, int R, int B) {
  const int F = tc_key_split(R);
  if (head_dim == 128) return tc_bytes<128>(F, B);
  if (head_dim == 64) return tc_bytes<64>(F, B);
  return 0;
}

int tc_setup(int head_dim, int device) {
  static std::mutex mu;
  static bool done[64][2] = {};
  if (device < 0 || device >= 64) return fail(SF_ERR_UNSUPPORTED, "device ordinal %d", device);
  const int k = head_dim == 128 ? 1 : 0;
  std::lock_guard<std::mutex> lock(mu);
  if (done[device][k]) return SF_OK;
  for (int F : {1, 2, 4}) {
    TcKernelFn fn = head_dim == 128 ? tc_kernel<128>(F) : tc_kernel<64>(F);
    const int smem = head_dim == 128 ? tc_bytes<128>(F, SF_MAX_BATCH) : tc_bytes<64>(F, SF_MAX_BATCH);
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(fn, cudaFuncAttributePreferredSharedMemoryCarveout,
                               cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess)
      return fail(SF_ERR_CUDA, "cudaFuncSetAttribute (tcgen05 kernel): %s", cudaGetErrorString(e));
  }
  done[device][k] = true;
  return SF_OK;
}

int tc_launch(int head_dim, int G, int smem, const CUtensorMap &tk, const CUtensorMap &tv,
              const AttnParams &prm, cudaStream_t stream) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(G);
  cfg.blockDim = dim3(kTcThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const int F = tc_key_split(prm.R);
  TcKernelFn fn = head_dim == 128 ? tc_kernel<128>(F) : tc_kernel<64>(F);
  cudaError_t e = cudaLaunchKernelEx(&cfg, fn, tk, tv, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "verify attention (tcgen05) launch: %s", cudaGetErrorString(e));
  const long long items = (long long)prm.R * (head_dim / 4) * prm.B * prm.H_kv;
  long long ctas = (items + kTcMergeThreads - 1) / kTcMergeThreads;
  if (ctas > G) ctas = G;  // one per SM (G is the SM count unless num_splits asks for fewer)
  cfg.gridDim = dim3(static_cast<unsigned>(ctas));
  cfg.blockDim = dim3(kTcMergeThreads);
  cfg.dynamicSmemBytes = 4 * (3 * prm.B + 2);
  e = head_dim == 64 ? cudaLaunchKernelEx(&cfg, verify_tc_merge_kernel<64>, prm)
                     : cudaLaunchKernelEx(&cfg, verify_tc_merge_kernel<128>, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "verify merge launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

}  // namespace sf
