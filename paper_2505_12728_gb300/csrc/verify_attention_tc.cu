// verify_attention_tc.cu -- verification attention on the 5th-generation
// tensor cores (tcgen05, accumulators in tensor memory), used for shapes
// with many query rows per KV head (GQA, R = n_q * g > 16).
//
// It computes exactly what the mma.sync kernel in verify_attention.cu
// computes (Sec. 3.1: the K draft tokens are scored in one forward pass, so
// each of the n_q new rows attends to the prefix plus the causal draft
// block), with the same fp32 partial format, so verify_merge_kernel combines
// split segments.  What differs:
//  * The work partition is chosen on the device from seq_lens: the
//    balanced one (all tiles cut into G equal ranges; a CTA may hold pieces
//    of several segments) or a segment-aligned one (each segment gets
//    ceil(tiles / Ta) CTAs and every CTA one piece) when its largest piece
//    is within kAlignSlackTiles of the balanced share -- a CTA's second
//    piece costs another Q load, epilogue and pipeline start.
//  * All R rows of a KV head are the M = 128 side of the MMAs.  Row r sits
//    in TMEM lane 32 * (r % 4) + r / 4, so the rows spread over the four lane
//    quarters (one per softmax warp); lanes >= R hold zero rows.
//  * A K tile sits in shared memory as [64-column half][64 tokens][128 B],
//    128B-swizzled (one TMA box per page and half), so the 64 keys of a half
//    are eight 8-row swizzle atoms 1024 bytes apart and S = Q K^T is
//    head_dim/16 MMAs of M=128, N=64, K=16 straight into TMEM.  A V tile sits
//    as [page][half][16 tokens][128 B] (one box per page: a box costs the
//    TMA unit about the same whatever its size, so V takes half as many);
//    P = exp2(S') goes back to TMEM as bf16, and O += P V is four MMAs (one
//    per page of 16 keys) with A from TMEM and B = V as an MN-major operand
//    (N = head_dim, the halves 2 KB apart).
//  * Warp roles: warps 0-3 own one TMEM lane (= one query row) per thread
//    and run the online softmax with no shuffles; warp 4 allocates TMEM and
//    runs the MMA loop (one elected lane issues); warp 5 reads the block
//    table and issues the TMA copies into a STAGES-deep ring.
//  * Hand-offs are mbarriers: full / empty per ring slot (TMA bytes, MMA
//    commit), s_full / p_full / o_done per S and P buffer (two of each, so
//    Q K^T of tile n+1 runs while tile n is in the softmax), q_full per piece.
//  * The running maximum is a reference that moves only when a row's new
//    maximum exceeds it by more than kRescaleLog2 (base-2 units): the
//    weights exp2(x - ref) stay below 2^kRescaleLog2, and the O rescale (a
//    TMEM read-modify-write that must wait for the previous P V) is rare.
//    O/l and the LSE do not depend on the reference.
//  * One CTA per SM (the ring and Q fill most of shared memory), so the
//    whole 512-column TMEM is this CTA's: O of the first piece [0,128), O of
//    later pieces [128,256), S0 [256,320), S1 [320,384), P0 [384,416),
//    P1 [416,448), and the low bf16 parts of P0 and P1 [448,480), [480,512)
//    (on a sequence's first tile P V is accumulated from P = P_hi + P_lo, two
//    bf16 terms, so that it carries P to ~16 bits like the fp32 row sum it
//    is divided by: rows with a handful of visible keys, and weight
//    concentrated on the first keys, otherwise show P's bf16 rounding).
//  * A piece that covers a whole segment writes bf16 out and the LSE; a
//    split segment's pieces write fp32 partials to the workspace, which the
//    merge kernel of verify_attention.cu combines.
//  * The first copies run before griddepcontrol.wait only for tiles that lie
//    wholly in the prefix; tiles holding draft positions (which the previous
//    kernel on the stream may have just written) are copied after it.
//  * Every wait is bounded; a timeout sets SF_DEVICE_TIMEOUT, stops every
//    role, waits (bounded) for copies and MMAs in flight and frees TMEM.
#include <cmath>
#include <mutex>

#include "attn_common.cuh"
#include "sf_host.h"

namespace sf {

constexpr int kTcThreads = 192;
constexpr int kTcSoftmaxThreads = 128;
constexpr int kTcMmaWarp = 4;
constexpr int kTcProducerWarp = 5;
constexpr uint32_t kTmemCols = 512;
// O of a CTA's first piece stays in [0,128) until the end (it may be split);
// every later piece accumulates in [128,256).
constexpr uint32_t kTmemOFirst = 0, kTmemOLater = 128, kTmemS = 256, kTmemP = 384, kTmemPlo = 448;
constexpr float kRescaleLog2 = 8.f;
constexpr int kTilesBeforeQ = 5;  // K/V tiles copied before the first Q is loaded
// The segment-aligned partition is used while its largest piece is at most
// this many tiles above the balanced share (a second piece in a CTA costs
// about that much: another Q load, epilogue and pipeline start).
constexpr int kAlignSlackTiles = 3;

template <int D>
struct TcConfig {
  static constexpr int kStages = D == 128 ? 5 : 8;
};

template <int D, int STAGES>
struct TcSmem {
  static constexpr int kTileBytes = kTileTokens * D * 2;  // one tensor, one tile
  static constexpr int kStageBytes = 2 * kTileBytes;      // K then V
  static constexpr int kQOffset = STAGES * kStageBytes;
  static constexpr int kQBytes = 128 * D * 2;             // [D/64][128 rows][128 B]
  static constexpr int kBarOffset = kQOffset + kQBytes;
  // full[S], empty[S], s_full[2], p_full[2], o_done[2], q_full, fin
  static constexpr int kNumBars = 2 * STAGES + 8;
  static constexpr int kMiscOffset = kBarOffset + 8 * kNumBars;
  static constexpr int kMiscInts = 16;
  static constexpr int kPrefixOffset = kMiscOffset + 4 * kMiscInts;
  // tiles prefix [B+1] | seq lens [B] | aligned CTA prefix [B+1]
  static int bytes(int B) { return 1024 + kPrefixOffset + 4 * (3 * B + 3); }
};

template <int D, int STAGES, int F>
__global__ void __launch_bounds__(kTcThreads, 1)
verify_attention_tc_kernel(const __grid_constant__ CUtensorMap tmap_k,
                           const __grid_constant__ CUtensorMap tmap_v,
                           const __grid_constant__ AttnParams p) {
  using L = TcSmem<D, STAGES>;
  constexpr int HALVES = D / 64;
  constexpr int kPageHalfBytes = kPageTokens * kRowBytes;       // 16 tokens x 64 columns
  constexpr int kPageBytes = HALVES * kPageHalfBytes;           // one page of V
  constexpr int kTileHalfBytes = kTileTokens * kRowBytes;       // 64 tokens x 64 columns
  constexpr int kQHalfBytes = 128 * kRowBytes;                  // 128 rows x 64 columns of Q
  constexpr float kLn2 = 0.6931471805599453f;
  constexpr uint32_t kIdescQK = idesc_bf16_f32(128, 64, 0, 0);  // Q K-major, K K-major
  constexpr uint32_t kIdescPV = idesc_bf16_f32(128, D, 0, 1);   // P (TMEM), V MN-major
  // barrier indices
  constexpr int FULL = 0, EMPTY = STAGES, SFULL = 2 * STAGES, PFULL = 2 * STAGES + 2,
                ODONE = 2 * STAGES + 4, QFULL = 2 * STAGES + 6, FIN = 2 * STAGES + 7;

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t ring = smem_addr(smem);
  const uint32_t qs = ring + L::kQOffset;
  const uint32_t bars = ring + L::kBarOffset;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };
  int *s_misc = reinterpret_cast<int *>(smem + L::kMiscOffset);
  // s_misc: [0] TMEM base, [1] abort word, [2] tiles issued, [3] tiles consumed
  volatile int *s_abort = s_misc + 1;
  int *s_prefix = reinterpret_cast<int *>(smem + L::kPrefixOffset);
  int *s_len = s_prefix + p.B + 1;
  int *s_cpre = s_len + p.B;  // aligned partition: first CTA of each sequence

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  grid_launch_dependents();
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(bar(FULL + s), 1);
      mbar_init(bar(EMPTY + s), 1);
    }
    for (int x = 0; x < 2; ++x) {
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
  }
  tile_prefix<kTcThreads>(p, s_prefix, s_len, s_misc + 8);
  __syncthreads();

  // Work partition, decided identically by every CTA from seq_lens:
  //  * balanced: the batch's tiles in one ordered list cut into G equal
  //    ranges (a CTA may hold pieces of several segments);
  //  * segment-aligned: segment s gets ceil(tiles_s / Ta) CTAs, Ta =
  //    ceil(Tot / (G - S)) so that they number at most G, and every CTA holds
  //    one piece -- chosen when Ta is close to the balanced share.
  // CTAs beyond the work get an empty range.
  const uint32_t Tot = static_cast<uint32_t>(p.H_kv) * static_cast<uint32_t>(s_prefix[p.B]);
  const int G = Tot < static_cast<uint32_t>(p.G) ? static_cast<int>(Tot) : p.G;
  const TilePartition part{Tot, static_cast<uint32_t>(G), Tot / G, Tot % G};
  const int S = p.B * p.H_kv;
  bool aligned = false;
  int Ta = 0;
  if (p.G > S) {
    Ta = static_cast<int>((Tot + static_cast<uint32_t>(p.G - S) - 1) / static_cast<uint32_t>(p.G - S));
    aligned = Ta <= static_cast<int>((Tot + p.G - 1) / p.G) + kAlignSlackTiles;
  }
  Piece apc{};  // the aligned partition's piece of this CTA
  uint32_t t_begin = Tot, t_end = Tot;
  if (aligned) {
    aligned_prefix<kTcThreads>(p, s_prefix, Ta, s_cpre, s_misc + 8);
    __syncthreads();
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

  if (warp == kTcMmaWarp) {
    tmem_alloc(smem_addr(s_misc), kTmemCols);
    tmem_relinquish_alloc_permit();
    tc_fence_before_sync();
  }
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = static_cast<uint32_t>(s_misc[0]);

  if (warp == kTcProducerWarp) {
    // ------------------------------------------------------------------
    // producer: the warp reads the block table; one lane per TMA box (K:
    // page and half, V: page) issues the copies of a tile
    // ------------------------------------------------------------------
    const uint64_t policy = l2_policy_evict_first();
    bool waited = false;
    bool q_in = false;  // Q of the first piece is in shared memory
    uint32_t n = 0;     // tiles issued by this CTA
    bool ok = true;
    for (uint32_t t = t_begin; t < t_end && ok;) {
      const Piece pc = piece_at(t);
      t += pc.n_tiles;
      int ids = kBeyondEnd;
      for (int it = 0; it < pc.n_tiles; ++it, ++n) {
        if ((it & 7) == 0) {
          // page ids of tiles it .. it+7: lane l holds tile it + l/4, page l%4
          const int lt = pc.lt0 + it + (lane >> 2);
          const int lp = lt * kPagesPerTile + (lane & 3);
          ids = kBeyondEnd;
          if (it + (lane >> 2) < pc.n_tiles && lp * kPageTokens < pc.T)
            ids = p.block_table[(size_t)pc.b * p.max_pages + lp];
        }
        // lanes 0 .. 4*HALVES-1 issue the K boxes (page l / HALVES, half
        // l % HALVES), the next four lanes the V boxes (one per page)
        constexpr int kKBoxes = HALVES * kPagesPerTile;
        const bool is_v = lane >= kKBoxes;
        const int pg = is_v ? (lane - kKBoxes) & (kPagesPerTile - 1) : (lane / HALVES) & (kPagesPerTile - 1);
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
        // Q goes first: beyond kTilesBeforeQ tiles, the copies would queue
        // ahead of the Q loads that the first MMA needs
        if (!q_in && n >= static_cast<uint32_t>(kTilesBeforeQ)) {
          int w = 1;
          if (lane == 0) w = mbar_wait_or_abort(bar(QFULL), 0, s_abort);
          if (!__shfl_sync(0xffffffffu, w, 0)) {
            ok = false;
            break;
          }
          q_in = true;
        }
        if (lane == 0) mbar_arrive_expect_tx(bar(FULL + slot), L::kStageBytes);
        __syncwarp();
        if (lane < kKBoxes + kPagesPerTile) {
          // pages past the sequence end or outside the pool load as zeros
          int row = p.oob_row;
          if (phys != kBeyondEnd) {
            if (phys < 0 || phys >= p.num_pages) set_status(p.status, SF_DEVICE_BAD_PAGE);
            else row = (phys * p.H_kv + pc.h_kv) * kPageTokens;
          }
          const uint32_t stage = ring + slot * L::kStageBytes;
          if (is_v) {
            // whole page: [half][16 tokens][128 B]
            const uint32_t dst = stage + L::kTileBytes + pg * kPageBytes;
            if constexpr (HALVES == 2) tma_load_3d(dst, &tmap_v, 0, row, 0, bar(FULL + slot), policy);
            else tma_load_2d(dst, &tmap_v, 0, row, bar(FULL + slot), policy);
          } else {
            const int h = lane % HALVES;
            const uint32_t dst = stage + h * kTileHalfBytes + pg * kPageHalfBytes;
            if constexpr (HALVES == 2) tma_load_3d(dst, &tmap_k, 0, row, h, bar(FULL + slot), policy);
            else tma_load_2d(dst, &tmap_k, 0, row, bar(FULL + slot), policy);
          }
        }
        __syncwarp();
      }
    }
    if (lane == 0) s_misc[2] = static_cast<int>(n);
  } else if (warp == kTcMmaWarp) {
    // ------------------------------------------------------------------
    // MMA loop: the whole warp polls, one elected lane issues and commits.
    // Q K^T of tile m needs its K tile (full), S buffer m&1 read out
    // (p_full of tile m-2, i.e. m <= pv + 1) and, for the first tile of a
    // piece, the piece's Q (q_full); P V of tile m needs its P (p_full).
    // The two streams are issued as soon as their conditions hold, so a
    // P V never waits behind the next tile's copy.
    // ------------------------------------------------------------------
    uint32_t qk = 0, pv = 0;      // next tile to multiply, CTA-wide counters
    uint32_t qk_piece_end = 0;    // end of the piece of tile qk
    uint32_t pv_piece_start = 0;  // first tile of the piece of tile pv
    uint32_t pv_piece_end = 0;
    int pv_piece = -1;            // piece of tile pv
    int pv_lt0 = 0;               // its first tile within the sequence
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
      // advance the piece cursors
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
        ++pv_piece;
        pv_piece_end += pc.n_tiles;
      }
      if (qk < total && qk <= pv + 1) {
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
          const uint32_t d = tmem + kTmemS + (qk & 1u) * 64u;
          if (elect_one()) {
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint32_t koff = (kk >> 2) * kQHalfBytes + (kk & 3) * 32;
              const uint64_t a = smem_desc_sw128(qs + koff, 16, 1024);
              const uint64_t b = smem_desc_sw128(kb + (kk >> 2) * kTileHalfBytes + (kk & 3) * 32, 16, 1024);
              tc_mma_ss(d, a, b, kIdescQK, kk > 0 ? 1u : 0u);
            }
            tc_commit(bar(SFULL + (qk & 1u)));
          }
          __syncwarp();
          ++qk;
          progress = true;
        }
      }
      if (pv < qk) {
        const bool ready = mbar_test_wait(bar(PFULL + (pv & 1u)), (pv >> 1) & 1u);
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
              const uint32_t acc = tmem + (pv_piece == 0 ? kTmemOFirst : kTmemOLater);
              tc_mma_ts(acc, tmem + kTmemP + (pv & 1u) * 32u + j * 8u, b, kIdescPV,
                        (first && j == 0) ? 0u : 1u);
              if (seq_first) tc_mma_ts(acc, tmem + kTmemPlo + (pv & 1u) * 32u + j * 8u, b, kIdescPV, 1u);
            }
            tc_commit(bar(ODONE + (pv & 1u)));
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
    // softmax + epilogue.  Lane quarter q = warp; inside it, lane
    // rho + k * (32/F) holds query row r = 4 * rho + q for the k-th 1/F of
    // the tile's keys (the Q row is repeated F times on the M side, which
    // costs the 128-row MMAs nothing).  Each lane keeps its own reference,
    // sum and O over its keys; the F lanes of a row merge at the end of the
    // piece with shuffles, like split-KV pieces.
    // ------------------------------------------------------------------
    constexpr int RPQ = 32 / F;    // rows per lane quarter
    constexpr int KPL = 64 / F;    // keys per lane and tile
    const int rho = lane % RPQ, kap = lane / RPQ;
    const int r = rho * 4 + warp;
    const bool valid = r < p.R;
    const uint32_t tl = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    // every lane waits (and acquires); the warp leaves together if any failed,
    // so the warp-collective tcgen05 instructions always see a full warp
    auto wwait = [&](uint32_t b, uint32_t parity) -> bool {
      const bool w = mbar_wait_or_abort(b, parity, s_abort);
      return __all_sync(0xffffffffu, w);
    };
    bool waited = false;
    uint32_t n = 0;
    bool ok = true;
    int pi = 0;                          // piece index in this CTA
    for (uint32_t t = t_begin; t < t_end && ok; ++pi) {
      const Piece pc = piece_at(t);
      t += pc.n_tiles;
      const uint32_t ob = pi == 0 ? kTmemOFirst : kTmemOLater;  // this piece's O
      if (!waited) {
        // Q rows into L2 while the previous kernel drains (a prefetch has
        // no effect on the values read after the wait)
        for (int x = tid; x < p.R * (D * 2 / 128); x += kTcSoftmaxThreads) {
          const int rr = x / (D * 2 / 128), half = x % (D * 2 / 128);
          const int i = rr / p.group, j = rr % p.group;
          prefetch_l2(p.q + (((size_t)pc.b * p.n_q + i) * p.H_q + (size_t)pc.h_kv * p.group + j) * D + half * 64);
        }
        grid_dependency_wait();
        waited = true;
      }
      if (pc.lt0 == 0 && tid == 0) p.seg_desc[pc.seg] = make_int2(pc.c_first, pc.n_pieces);

      // Q rows of the piece into shared memory (every MMA of the previous
      // piece has completed): M-side row m holds query row
      // 4 * ((m % 32) % RPQ) + m / 32, 128B-swizzled like the K tiles
      // (each distinct row is loaded once and stored F times; all loads
      // first, then all stores: one memory round trip)
      {
        constexpr int kQChunks = 4 * RPQ * (D / 8) / kTcSoftmaxThreads;
        uint4 qv[kQChunks];
#pragma unroll
        for (int u = 0; u < kQChunks; ++u) {
          const int idx = tid + u * kTcSoftmaxThreads;
          const int ui = idx / (D / 8), c = idx % (D / 8);
          const int rr = (ui % RPQ) * 4 + ui / RPQ;
          qv[u] = make_uint4(0u, 0u, 0u, 0u);
          if (rr < p.R) {
            const int i = rr / p.group, j = rr % p.group;
            qv[u] = __ldg(reinterpret_cast<const uint4 *>(
                p.q + (((size_t)pc.b * p.n_q + i) * p.H_q + (size_t)pc.h_kv * p.group + j) * D + c * 8));
          }
        }
#pragma unroll
        for (int u = 0; u < kQChunks; ++u) {
          const int idx = tid + u * kTcSoftmaxThreads;
          const int ui = idx / (D / 8), c = idx % (D / 8);
#pragma unroll
          for (int k = 0; k < F; ++k) {
            const int mrow = (ui / RPQ) * 32 + ui % RPQ + k * RPQ;
            *reinterpret_cast<uint4 *>(smem + L::kQOffset + (c >> 3) * kQHalfBytes + mrow * kRowBytes +
                                       (((c & 7) ^ (mrow & 7)) << 4)) = qv[u];
          }
        }
      }
      fence_proxy_async_smem();
      tc_fence_before_sync();
      mbar_arrive(bar(QFULL));
      if (t < t_end) {
        // the next piece's Q rows into L2 (one 128-byte line per thread)
        const Piece nx = piece_at(t);
        const int lines = p.R * (D * 2 / 128);
        for (int x = tid; x < lines; x += kTcSoftmaxThreads) {
          const int rr = x / (D * 2 / 128), half = x % (D * 2 / 128);
          const int i = rr / p.group, j = rr % p.group;
          prefetch_l2(p.q + (((size_t)nx.b * p.n_q + i) * p.H_q + (size_t)nx.h_kv * p.group + j) * D + half * 64);
        }
      }

      // last visible key position of this row (draft row i sees L_b + i)
      const int lim = valid ? pc.Lb + min(r / p.group, p.n_q - 1) : -1;
      float ref = -INFINITY, l_run = 0.f;
      for (int it = 0; it < pc.n_tiles; ++it, ++n) {
        if (!wwait(bar(SFULL + (n & 1u)), (n >> 1) & 1u)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        uint32_t sv[64];
        tmem_ld_32x32b_x64(tl + kTmemS + (n & 1u) * 64u, sv);
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
        float x[KPL];
        float mx = -INFINITY;
#pragma unroll
        for (int c = 0; c < KPL; ++c) {
          uint32_t v = sv[c];
#pragma unroll
          for (int k = 1; k < F; ++k)
            if (kap == k) v = sv[k * KPL + c];
          x[c] = __uint_as_float(v);
          mx = fmaxf(mx, x[c]);
        }
        const int key0 = tile_pos + kap * KPL;
        if (key0 + KPL - 1 > lim) {
          // causal mask of the draft block, positions past the end, padding rows
          mx = -INFINITY;
#pragma unroll
          for (int c = 0; c < KPL; ++c) {
            if (key0 + c > lim) x[c] = -INFINITY;
            mx = fmaxf(mx, x[c]);
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
        float rs = 0.f;
        uint32_t mine[KPL / 2], mine_lo[KPL / 2];
#pragma unroll
        for (int c2 = 0; c2 < KPL / 2; ++c2) {
          const float p0 = fast_exp2(fmaf(x[2 * c2], p.scale_log2, -mu));
          const float p1 = fast_exp2(fmaf(x[2 * c2 + 1], p.scale_log2, -mu));
          rs += p0 + p1;
          if (split_p) split_bf16x2(p0, p1, mine[c2], mine_lo[c2]);
          else mine[c2] = pack_bf16x2(p0, p1);
        }
        l_run = l_run * alpha + rs;
        // P row of this lane: its keys' weights, zeros for the other lanes' keys
        uint32_t pk[32];
#pragma unroll
        for (int cc = 0; cc < 32; ++cc) pk[cc] = (cc / (KPL / 2) == kap) ? mine[cc % (KPL / 2)] : 0u;
        // P buffer n&1 is free once the P V of tile n-2 has completed
        if (n >= 2 && !wwait(bar(ODONE + (n & 1u)), ((n - 2) >> 1) & 1u)) {
          ok = false;
          break;
        }
        if (__any_sync(0xffffffffu, alpha != 1.f)) {
          // O *= alpha after the P V of tile n-1 (it > 0 here: the first
          // tile of a piece starts with ref = -inf, so alpha = 1)
          if (!wwait(bar(ODONE + ((n - 1) & 1u)), ((n - 1) >> 1) & 1u)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
#pragma unroll 1
          for (int ch = 0; ch < D / 32; ++ch) {
            uint32_t ov[32];
            tmem_ld_32x32b_x32(tl + ob + ch * 32, ov);
#pragma unroll
            for (int c = 0; c < 32; ++c) ov[c] = __float_as_uint(__uint_as_float(ov[c]) * alpha);
            tmem_st_32x32b_x32(tl + ob + ch * 32, ov);
          }
        }
        tmem_st_32x32b_x32(tl + kTmemP + (n & 1u) * 32u, pk);
        if (split_p) {  // the sequence's first tile: P_lo too (warp-uniform)
          uint32_t pk_lo[32];
#pragma unroll
          for (int cc = 0; cc < 32; ++cc) pk_lo[cc] = (cc / (KPL / 2) == kap) ? mine_lo[cc % (KPL / 2)] : 0u;
          tmem_st_32x32b_x32(tl + kTmemPlo + (n & 1u) * 32u, pk_lo);
        }
        tmem_wait_st();
        tc_fence_before_sync();
        mbar_arrive(bar(PFULL + (n & 1u)));
      }
      if (!ok) break;

      // ---- epilogue of the piece ----
      const uint32_t last = n - 1;
      if (!wwait(bar(ODONE + (last & 1u)), (last >> 1) & 1u)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      // merge the F lanes of each row (M = max ref, w = 2^(ref - M)); a
      // whole segment is normalised and written, a split one leaves its
      // fp32 partial O [R][D] (relative to M), M [R], L [R] in the workspace
      float M = ref;
#pragma unroll
      for (int k = RPQ; k < 32; k <<= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, k));
      const float w = ref == -INFINITY ? 0.f : exp2f(ref - M);
      float Ls = l_run * w;
#pragma unroll
      for (int k = RPQ; k < 32; k <<= 1) Ls += __shfl_xor_sync(0xffffffffu, Ls, k);
      // tcgen05.ld is warp-collective: every lane loads; lane kap == 0 of a
      // valid row stores
      const bool writer = valid && kap == 0;
      const int i = valid ? r / p.group : 0, j = valid ? r % p.group : 0;
      const size_t row = ((size_t)pc.b * p.n_q + i) * p.H_q + (size_t)pc.h_kv * p.group + j;
      const bool whole = pc.n_pieces == 1;
      const float inv = whole ? 1.f / Ls : 1.f;
      float *part0 = p.partials + (size_t)(blockIdx.x + pc.seg) * p.slot_stride;
#pragma unroll 1
      for (int ch = 0; ch < D / 32; ++ch) {
        uint32_t ov[32];
        tmem_ld_32x32b_x32(tl + ob + ch * 32, ov);
        float o[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          o[c] = __uint_as_float(ov[c]) * w;
#pragma unroll
          for (int k = RPQ; k < 32; k <<= 1) o[c] += __shfl_xor_sync(0xffffffffu, o[c], k);
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
          float4 *dst = reinterpret_cast<float4 *>(part0 + (size_t)r * D + ch * 32);
#pragma unroll
          for (int q4 = 0; q4 < 8; ++q4)
            dst[q4] = make_float4(o[4 * q4], o[4 * q4 + 1], o[4 * q4 + 2], o[4 * q4 + 3]);
        }
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
    }

    tc_fence_before_sync();
  }

  // ---- teardown: every role is done (or stopped) ----
  __syncthreads();
  if (*s_abort) {
    if (tid == 0) set_status(p.status, SF_DEVICE_TIMEOUT);
    if (warp == kTcProducerWarp && lane == 0) {
      // copies issued but never consumed: wait (bounded) until they land
      for (uint32_t x = static_cast<uint32_t>(s_misc[3]); x < static_cast<uint32_t>(s_misc[2]); ++x)
        (void)mbar_wait_bounded(bar(FULL + x % STAGES), (x / STAGES) & 1u);
    }
    __syncthreads();
  }
  if (warp == kTcMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }

}

// --------------------------------------------------------------------------
// host side
// --------------------------------------------------------------------------
using TcKernelFn = void (*)(const CUtensorMap, const CUtensorMap, const AttnParams);

// Lanes per query row: as many as 128 TMEM lanes allow, at most 4.
static int tc_key_split(int R) { return R <= 32 ? 4 : (R <= 64 ? 2 : 1); }

template <int D>
static TcKernelFn tc_kernel(int F) {
  constexpr int S = TcConfig<D>::kStages;
  if (F == 4) return verify_attention_tc_kernel<D, S, 4>;
  if (F == 2) return verify_attention_tc_kernel<D, S, 2>;
  return verify_attention_tc_kernel<D, S, 1>;
}

int tc_smem_bytes(int head_dim, int B) {
  if (head_dim == 128) return TcSmem<128, TcConfig<128>::kStages>::bytes(B);
  if (head_dim == 64) return TcSmem<64, TcConfig<64>::kStages>::bytes(B);
  return 0;
}

int tc_setup(int head_dim, int device) {
  static std::mutex mu;
  static bool done[64][2] = {};
  if (device < 0 || device >= 64) return fail(SF_ERR_UNSUPPORTED, "device ordinal %d", device);
  const int k = head_dim == 128 ? 1 : 0;
  std::lock_guard<std::mutex> lock(mu);
  if (done[device][k]) return SF_OK;
  const int smem = tc_smem_bytes(head_dim, SF_MAX_BATCH);
  for (int F : {1, 2, 4}) {
    TcKernelFn fn = head_dim == 128 ? tc_kernel<128>(F) : tc_kernel<64>(F);
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
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
  return SF_OK;
}

}  // namespace sf
