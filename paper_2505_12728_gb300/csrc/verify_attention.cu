// verify_attention.cu -- split-KV verification attention for sm_103a.
//
// The target model scores the K draft tokens in one forward pass against its
// cache of visual-then-text tokens (Sec. 3.1; verification costs about one
// target step, Eq. 1).  Per layer that is attention of n_q new query rows per
// sequence over the prefix plus the causal draft block:
//   out[b,i,h] = sum_t softmax_t(scale * <q[b,i,h], k[b,t,h/g]>) v[b,t,h/g],
//   t = 0 .. L_b + i,   L_b = seq_lens[b] - n_q.
//
// GB300 design (the paper gives no kernel; its runs used one A6000):
//  * Work unit = a tile of 64 cached tokens of one (sequence, KV head)
//    "segment".  All tiles of the batch form one ordered list that is cut
//    into G equal, contiguous ranges, one per CTA, computed on the device from
//    seq_lens, so long and short sequences balance without host knowledge of
//    the lengths.  A CTA's range touches one or two segments ("pieces").
//  * Each CTA streams its tiles through a STAGES-deep ring in shared memory:
//    one elected warp issues one TMA box per 16-token page and tensor
//    (128-byte swizzle) straight from the block table, completing on an
//    mbarrier; nothing else touches HBM in the loop.
//  * All n_q * g query rows of a KV head share each K/V tile.  This kernel
//    takes shapes with at most 16 such rows (MHA, n_q <= 16): the rows are
//    the M dimension of bf16 m16n8k16 tensor-core MMAs (S = Q K^T and
//    O += P V, fp32 accumulate); scores stay in registers, where an fp32
//    online softmax (base 2, scale folded in) rescales the running output.
//    On a sequence's first tile P enters P V as two bf16 terms (see
//    split_bf16x2), so that rows with few visible keys keep P's precision.
//    The four warps split each tile's keys and combine in shared memory at
//    the end of a piece.  More rows per KV head (GQA) are a real dense
//    contraction and go to the tcgen05 kernel in verify_attention_tc.cu.
//  * A piece that covers a whole segment writes bf16 out and fp32 LSE
//    directly.  Split segments are merged (deterministically, in piece
//    order) in one of three ways:
//      - cluster mode: for one sequence the grid is one thread-block cluster
//        per KV head; the cluster's CTAs keep their partials in shared
//        memory and merge them through distributed shared memory;
//      - otherwise the CTA that takes the last ticket of the segment (an
//        atomic counter; nobody waits) merges the fp32 partials;
//      - the tcgen05 kernel's split segments (many rows, larger partials):
//        verify_tc_merge_kernel, spread over the whole GPU.
//  * Launches use programmatic stream serialisation: the partition, the
//    block-table reads (for one sequence, its whole row copied to shared
//    memory next to the seq_lens read) and the first copies of prefix tiles
//    run before griddepcontrol.wait, overlapping the previous kernel on the
//    stream (tiles holding draft positions are copied after it).
//  * Page indices outside the pool and positions past a sequence's end are
//    loaded as zero boxes (TMA out-of-bounds fill); bad indices set a bit in
//    the status word.  Every mbarrier wait is bounded.
#include <algorithm>
#include <cmath>
#include <map>
#include <mutex>
#include <tuple>

#include "attn_common.cuh"
#include "sf_host.h"

namespace sf {


template <int D, int STAGES, int NW>
struct AttnSmem {
  static constexpr int kTensorTileBytes = kTileTokens * D * 2;
  static constexpr int kStageBytes = 2 * kTensorTileBytes;
  static constexpr int kRingBytes = STAGES * kStageBytes;
  // ring | STAGES mbarriers | misc ints | tiles prefix [B+1] | seq lens [B]
  static constexpr int kBarOffset = kRingBytes;
  static constexpr int kMiscOffset = kBarOffset + 8 * STAGES;
  static constexpr int kMiscInts = 8 + 2 * NW;
  static constexpr int kPrefixOffset = kMiscOffset + 4 * kMiscInts;
  static int bytes(int B) { return 1024 + kPrefixOffset + 4 * (2 * B + 2); }
};


constexpr int kMaxCluster = 16;  // largest cluster launched (non-portable size)
constexpr int kPrefetchLines = 64;  // block-table lines prefetched for one sequence
constexpr int kBtCacheEntries = 512;  // longest block-table row copied to shared memory
constexpr int kPushSlots = 2;    // rows a CTA merges in push mode (at most)

// The two halves of a cluster barrier phase, for a phase that opens early and
// closes later (every thread of every CTA of the cluster arrives, then waits).
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait_acquire() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

template <int D, int KS, int NW, int STAGES>
__global__ void __launch_bounds__(NW * 32, (NW == 4 ? 2 : 1))
verify_attention_kernel(const __grid_constant__ CUtensorMap tmap_k,
                        const __grid_constant__ CUtensorMap tmap_v,
                        const __grid_constant__ AttnParams p) {
  using L = AttnSmem<D, STAGES, NW>;
  constexpr int NTHREADS = NW * 32;
  constexpr int RT_SLOTS = NW / KS;      // row tiles a CTA covers at once
  constexpr int KW = kTileTokens / KS;   // keys per warp per tile
  constexpr int NT = KW / 8;             // score n-tiles per warp
  constexpr int KK = D / 16;             // k-steps of Q K^T
  constexpr int DT = D / 8;              // output n-tiles
  constexpr int HALVES = D / 64;
  constexpr float kLn2 = 0.6931471805599453f;

  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t ring = smem_addr(smem);
  const uint32_t bar0 = ring + L::kBarOffset;
  int *s_misc = reinterpret_cast<int *>(smem + L::kMiscOffset);
  int *s_prefix = reinterpret_cast<int *>(smem + L::kPrefixOffset);
  int *s_len = s_prefix + p.B + 1;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rt = warp % RT_SLOTS, ks = warp / RT_SLOTS;
  const int row_tiles = (p.R + 15) >> 4;
  const bool active = rt < row_tiles;

  // Let the next kernel on the stream be scheduled as CTAs of this grid
  // finish.  Work that does not depend on the previous kernel on
  // the stream (barrier set-up, the tile partition, block-table reads and the
  // first K/V copies) runs before grid_dependency_wait(); Q is read and
  // results are written only after it.
  grid_launch_dependents();
  // One sequence: its block-table row is needed as soon as the partition is
  // known.  A short row is loaded now, while seq_lens is read, and kept in
  // shared memory, so the first copies wait for one global load, not two; a
  // longer row is brought toward the SM (L2) instead.
  constexpr int kBtPer = kBtCacheEntries / NTHREADS;
  int32_t *s_bt = reinterpret_cast<int32_t *>(smem + p.bt_off);
  int32_t bt_row[kBtPer];
  if (p.bt_off) {
#pragma unroll
    for (int k = 0; k < kBtPer; ++k) {
      const int i = tid + k * NTHREADS;
      bt_row[k] = i < p.max_pages ? __ldg(p.block_table + i) : 0;
    }
  } else if (p.B == 1 && tid < kPrefetchLines && tid * 32 < p.max_pages) {
    prefetch_l2(p.block_table + tid * 32);
  }
  if (tid == 0) {
    for (int s = 0; s < STAGES; ++s) mbar_init(bar0 + 8 * s, 1);
    fence_mbar_init();
    prefetch_tensormap(&tmap_k);
    prefetch_tensormap(&tmap_v);
  }
  tile_prefix<NTHREADS>(p, s_prefix, s_len, s_misc + 8);
  if (p.bt_off) {
#pragma unroll
    for (int k = 0; k < kBtPer; ++k) {
      const int i = tid + k * NTHREADS;
      if (i < p.max_pages) s_bt[i] = bt_row[k];
    }
  }
  __syncthreads();

  // The host sizes the grid from an upper bound of the tile count; with more
  // CTAs than tiles the surplus CTAs leave, so that every CTA of the
  // partition owns at least one tile and a segment's pieces are owned by
  // consecutive CTAs.
  const uint32_t Tot = static_cast<uint32_t>(p.H_kv) * static_cast<uint32_t>(s_prefix[p.B]);
  const int G = Tot < static_cast<uint32_t>(p.G) ? static_cast<int>(Tot) : p.G;
  if (static_cast<int>(blockIdx.x) >= G) return;
  const TilePartition part_of{Tot, static_cast<uint32_t>(G), Tot / G, Tot % G};
  const uint32_t t_begin = part_of.start(blockIdx.x);
  const uint32_t t_end = part_of.start(blockIdx.x + 1);

  // Cluster mode: when the launch uses clusters of cs CTAs and a cluster's
  // tiles are exactly one segment (uniform segments with G = segments x cs),
  // its CTAs keep their partials in shared memory and combine them through
  // distributed shared memory between two cluster barriers; no partial goes
  // through global memory.  Decided per cluster (identically by its CTAs);
  // every CTA of an aligned cluster has exactly one piece.
  bool aligned = false;
  // one sequence: its H_kv segments have equal length, so with G = H_kv x cs
  // every cluster is exactly one segment (no partition arithmetic needed)
  const bool one_seq_clusters = p.cs > 1 && p.B == 1 && G == p.G && G == p.H_kv * p.cs;
  if (one_seq_clusters) {
    aligned = true;
  } else if (p.cs > 1 && G == p.G) {
    const uint32_t k = blockIdx.x / p.cs;
    const uint32_t c0 = part_of.start(k * p.cs), c1 = part_of.start((k + 1) * p.cs);
    const int bb = find_sequence(c0, s_prefix, p.B, p.H_kv);
    const uint32_t tb = static_cast<uint32_t>(s_prefix[bb + 1] - s_prefix[bb]);
    const uint32_t base = static_cast<uint32_t>(p.H_kv) * static_cast<uint32_t>(s_prefix[bb]);
    aligned = ((c0 - base) % tb == 0) && (c1 - c0 == tb);
  }
  int seg_b = 0, seg_h = 0;  // the segment of an aligned cluster
  // Push mode stores into the shared memory of peer CTAs, which must have
  // started by then: the first barrier phase opens here and closes right
  // before the push (long since complete by then, so it costs no wait).
  const bool push_mode = aligned && p.push;
  if (push_mode) cluster_arrive_relaxed();

  const uint64_t policy = l2_policy_evict_first();
  bool waited = false;    // grid_dependency_wait() done
  uint32_t consumed = 0;  // tiles consumed by this CTA so far (ring position)
  bool timed_out = false;

  for (uint32_t t = t_begin; t < t_end && !timed_out;) {
    // ---- locate the piece: segment (b, h_kv), local tiles [lt0, lt1) ----
    int b, tiles_b, h_kv, lt0, n_tiles, c_first, n_pieces;
    if (one_seq_clusters) {
      // cluster k = KV head k; CTA rank r holds tiles [r tiles / cs, (r+1) tiles / cs)
      b = 0;
      tiles_b = s_prefix[1];
      h_kv = static_cast<int>(blockIdx.x) / p.cs;
      const int rank = static_cast<int>(blockIdx.x) - h_kv * p.cs;
      lt0 = rank * tiles_b / p.cs;
      n_tiles = (rank + 1) * tiles_b / p.cs - lt0;
      c_first = h_kv * p.cs;
      n_pieces = p.cs;
    } else {
      b = find_sequence(t, s_prefix, p.B, p.H_kv);
      tiles_b = s_prefix[b + 1] - s_prefix[b];
      const uint32_t seg_base = static_cast<uint32_t>(p.H_kv) * static_cast<uint32_t>(s_prefix[b]);
      h_kv = static_cast<int>((t - seg_base) / static_cast<uint32_t>(tiles_b));
      lt0 = static_cast<int>((t - seg_base) % static_cast<uint32_t>(tiles_b));
      const uint32_t left = t_end - t;
      n_tiles = left < static_cast<uint32_t>(tiles_b - lt0) ? static_cast<int>(left) : tiles_b - lt0;
      const uint32_t seg_first = seg_base + static_cast<uint32_t>(h_kv) * static_cast<uint32_t>(tiles_b);
      c_first = static_cast<int>(part_of.owner(seg_first));
      n_pieces = static_cast<int>(part_of.owner(seg_first + tiles_b - 1)) - c_first + 1;
    }
    const int seg = b * p.H_kv + h_kv;
    const int T = s_len[b];
    const int Lb = T - p.n_q;
    t += n_tiles;

    // ---- producer: lanes 0..3 of warp 0 own the four pages of a tile ----
    // fetch_page reads the block table (the value is checked only when the
    // copy is issued, so the load latency overlaps the current tile's math)
    auto fetch_page = [&](int lt, int pg) -> int {
      const int lp = lt * kPagesPerTile + pg;
      if (lp * kPageTokens >= T) return kBeyondEnd;
      return p.bt_off ? s_bt[lp] : p.block_table[(size_t)b * p.max_pages + lp];
    };
    auto issue = [&](int slot, int pg, int phys) {
      // one page (16 tokens) of K and V into ring slot `slot`; pages past the
      // end of the sequence or outside the pool load as zeros
      int row = p.oob_row;
      if (phys != kBeyondEnd) {
        if (phys < 0 || phys >= p.num_pages) set_status(p.status, SF_DEVICE_BAD_PAGE);
        else row = (phys * p.H_kv + h_kv) * kPageTokens;
      }
      const uint32_t dst = ring + slot * L::kStageBytes + pg * HALVES * kPageTokens * kRowBytes;
      const uint32_t bar = bar0 + 8 * slot;
      if constexpr (HALVES == 2) {
        // both 128-byte column halves of the page in one box (3-D map)
        tma_load_3d(dst, &tmap_k, 0, row, 0, bar, policy);
        tma_load_3d(dst + L::kTensorTileBytes, &tmap_v, 0, row, 0, bar, policy);
      } else {
        tma_load_2d(dst, &tmap_k, 0, row, bar, policy);
        tma_load_2d(dst + L::kTensorTileBytes, &tmap_v, 0, row, bar, policy);
      }
    };

    const int prologue = n_tiles < STAGES ? n_tiles : STAGES;
    const uint32_t piece_base = consumed;  // ring position of the piece's first tile
    int issued = prologue;                 // tiles of this piece issued so far
    int next_phys = 0;  // lanes 0..3 of warp 0: block-table entry of the next tile
    // tiles j0 .. j1-1 of the prologue, one lane per page
    auto issue_prologue = [&](int j0, int j1) {
      if (warp == 0 && j1 > j0) {
        if (lane >= j0 && lane < j1)
          mbar_arrive_expect_tx(bar0 + 8 * ((piece_base + lane) % STAGES), L::kStageBytes);
        __syncwarp();
        if (lane < kPagesPerTile * (j1 - j0)) {
          const int j = j0 + lane / kPagesPerTile, pg = lane % kPagesPerTile;
          issue((piece_base + j) % STAGES, pg, fetch_page(lt0 + j, pg));
        }
      }
    };
    // Before the wait on the previous kernel only tiles wholly inside the
    // prefix are copied: the draft rows' K/V may be written by that kernel.
    int pre = prologue;
    if (!waited) {
      pre = 0;
      while (pre < prologue && (lt0 + pre + 1) * kTileTokens <= Lb) ++pre;
    }
    issue_prologue(0, pre);
    if (warp == 0 && lane < kPagesPerTile && prologue < n_tiles)
      next_phys = fetch_page(lt0 + prologue, lane);

    if (!waited) {
      grid_dependency_wait();
      waited = true;
    }
    issue_prologue(pre, prologue);
    seg_b = b;
    seg_h = h_kv;

    // ---- consumers: Q fragments of this warp's 16 rows ----
    // row r = i * g + j  <->  (draft row i, query head h_kv * g + j)
    const int r0 = rt * 16 + (lane >> 2), r1 = r0 + 8;
    uint32_t qa[KK][4];
    {
      const int cols = 2 * (lane & 3);
      auto qptr = [&](int r) -> const __nv_bfloat16 * {
        const int i = r / p.group, j = r % p.group;
        return p.q + (((size_t)b * p.n_q + i) * p.H_q + (size_t)h_kv * p.group + j) * D;
      };
      const bool v0 = active && r0 < p.R, v1 = active && r1 < p.R;
      const __nv_bfloat16 *q0 = v0 ? qptr(r0) : nullptr;
      const __nv_bfloat16 *q1 = v1 ? qptr(r1) : nullptr;
#pragma unroll
      for (int kk = 0; kk < KK; ++kk) {
        const int c = kk * 16 + cols;
        qa[kk][0] = v0 ? *reinterpret_cast<const uint32_t *>(q0 + c) : 0u;
        qa[kk][1] = v1 ? *reinterpret_cast<const uint32_t *>(q1 + c) : 0u;
        qa[kk][2] = v0 ? *reinterpret_cast<const uint32_t *>(q0 + c + 8) : 0u;
        qa[kk][3] = v1 ? *reinterpret_cast<const uint32_t *>(q1 + c + 8) : 0u;
      }
    }
    // last visible key position of each of the thread's two rows
    const int lim0 = Lb + min(r0 / p.group, p.n_q - 1);
    const int lim1 = Lb + min(r1 / p.group, p.n_q - 1);

    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    float o[DT][4];
#pragma unroll
    for (int dt = 0; dt < DT; ++dt) o[dt][0] = o[dt][1] = o[dt][2] = o[dt][3] = 0.f;

    for (int it = 0; it < n_tiles; ++it) {
      const int slot = consumed % STAGES;
      const uint32_t parity = (consumed / STAGES) & 1u;
      const int lt = lt0 + it;
      const bool ok = mbar_wait_bounded(bar0 + 8 * slot, parity);
      const uint32_t kbase = ring + slot * L::kStageBytes;
      const uint32_t vbase = kbase + L::kTensorTileBytes;
      const int tile_pos = lt * kTileTokens;

      // Positions past the sequence end inside its last page hold whatever
      // the cache page holds; zero those V rows so that 0 * v stays 0.
      const int valid = T - tile_pos;
      if (valid < kTileTokens) {
        if (ok) {
          uint8_t *vt = smem + slot * L::kStageBytes + L::kTensorTileBytes;
          for (int idx = tid; idx < (kTileTokens - valid) * HALVES * 8; idx += NTHREADS) {
            const int tok = valid + idx / (HALVES * 8);
            const int rem = idx % (HALVES * 8);
            *reinterpret_cast<uint4 *>(vt + (tok >> 4) * (HALVES * kPageTokens * kRowBytes) +
                                       (rem >> 3) * (kPageTokens * kRowBytes) +
                                       (tok & 15) * kRowBytes + (rem & 7) * 16) =
                make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async_smem();
        }
        asm volatile("bar.sync 1, %0;" ::"n"(NTHREADS) : "memory");
      }

      if (ok && active) {
        float s[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
        // S = Q K^T over this warp's KW keys
#pragma unroll
        for (int kk = 0; kk < KK; kk += 2) {
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int key = ks * KW + nt * 8 + (lane & 7);
            uint32_t b0, b1, b2, b3;
            ldmatrix_x4(kbase + swz<D>(key, 2 * kk + (lane >> 3)), b0, b1, b2, b3);
            mma_bf16_16816(s[nt], qa[kk], b0, b1);
            mma_bf16_16816(s[nt], qa[kk + 1], b2, b3);
          }
        }
        // causal mask of the draft block (and of positions past the end)
        if (tile_pos + kTileTokens - 1 > Lb) {
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) {
            const int kp = tile_pos + ks * KW + nt * 8 + 2 * (lane & 3);
            if (kp > lim0) s[nt][0] = -INFINITY;
            if (kp + 1 > lim0) s[nt][1] = -INFINITY;
            if (kp > lim1) s[nt][2] = -INFINITY;
            if (kp + 1 > lim1) s[nt][3] = -INFINITY;
          }
        }
        // online softmax in base 2 with the scale folded in
        float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
          mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
        }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float mn0 = fmaxf(m0, mx0 * p.scale_log2);
        const float mn1 = fmaxf(m1, mx1 * p.scale_log2);
        const float mu0 = mn0 == -INFINITY ? 0.f : mn0;
        const float mu1 = mn1 == -INFINITY ? 0.f : mn1;
        const float a0 = exp2f(m0 - mu0), a1 = exp2f(m1 - mu1);
        m0 = mn0;
        m1 = mn1;
        float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
          s[nt][0] = exp2f(fmaf(s[nt][0], p.scale_log2, -mu0));
          s[nt][1] = exp2f(fmaf(s[nt][1], p.scale_log2, -mu0));
          s[nt][2] = exp2f(fmaf(s[nt][2], p.scale_log2, -mu1));
          s[nt][3] = exp2f(fmaf(s[nt][3], p.scale_log2, -mu1));
          rs0 += s[nt][0] + s[nt][1];
          rs1 += s[nt][2] + s[nt][3];
        }
        l0 = l0 * a0 + rs0;
        l1 = l1 * a1 + rs1;
#pragma unroll
        for (int dt = 0; dt < DT; ++dt) {
          o[dt][0] *= a0;
          o[dt][1] *= a0;
          o[dt][2] *= a1;
          o[dt][3] *= a1;
        }
        // O += P V.  On a sequence's first tile P = P_hi + P_lo, two bf16
        // terms (split_bf16x2), so that P carries ~16 bits like the fp32 row
        // sum l: rows with a handful of visible keys, and weight concentrated
        // on the first keys, otherwise show P's bf16 rounding in the output.
        // Later tiles use P_hi alone (their weights are spread over many keys).
        if (lt == 0) {
#pragma unroll
          for (int kt = 0; kt < KW / 16; ++kt) {
            uint32_t pa[4], pl[4];
            split_bf16x2(s[2 * kt][0], s[2 * kt][1], pa[0], pl[0]);
            split_bf16x2(s[2 * kt][2], s[2 * kt][3], pa[1], pl[1]);
            split_bf16x2(s[2 * kt + 1][0], s[2 * kt + 1][1], pa[2], pl[2]);
            split_bf16x2(s[2 * kt + 1][2], s[2 * kt + 1][3], pa[3], pl[3]);
            const int key = ks * KW + kt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
            for (int dt = 0; dt < DT; dt += 2) {
              uint32_t b0, b1, b2, b3;
              ldmatrix_x4_trans(vbase + swz<D>(key, dt + (lane >> 4)), b0, b1, b2, b3);
              mma_bf16_16816(o[dt], pa, b0, b1);
              mma_bf16_16816(o[dt], pl, b0, b1);
              mma_bf16_16816(o[dt + 1], pa, b2, b3);
              mma_bf16_16816(o[dt + 1], pl, b2, b3);
            }
          }
        } else {
#pragma unroll
          for (int kt = 0; kt < KW / 16; ++kt) {
            uint32_t pa[4];
            pa[0] = pack_bf16x2(s[2 * kt][0], s[2 * kt][1]);
            pa[1] = pack_bf16x2(s[2 * kt][2], s[2 * kt][3]);
            pa[2] = pack_bf16x2(s[2 * kt + 1][0], s[2 * kt + 1][1]);
            pa[3] = pack_bf16x2(s[2 * kt + 1][2], s[2 * kt + 1][3]);
            const int key = ks * KW + kt * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
#pragma unroll
            for (int dt = 0; dt < DT; dt += 2) {
              uint32_t b0, b1, b2, b3;
              ldmatrix_x4_trans(vbase + swz<D>(key, dt + (lane >> 4)), b0, b1, b2, b3);
              mma_bf16_16816(o[dt], pa, b0, b1);
              mma_bf16_16816(o[dt + 1], pa, b2, b3);
            }
          }
        }
      }
      // every warp is done with this slot; refill it with tile it + STAGES
      timed_out = __syncthreads_or(!ok) != 0;
      ++consumed;
      if (timed_out) break;
      if (it + STAGES < n_tiles) {
        if (warp == 0) {
          const int nslot = (consumed - 1) % STAGES;
          if (lane == 0) mbar_arrive_expect_tx(bar0 + 8 * nslot, L::kStageBytes);
          __syncwarp();
          if (lane < kPagesPerTile) {
            issue(nslot, lane, next_phys);
            if (it + STAGES + 1 < n_tiles) next_phys = fetch_page(lt0 + it + STAGES + 1, lane);
          }
        }
        ++issued;
      }
    }
    if (timed_out) {
      // Unwind: wait (bounded) for the copies still in flight -- the tile
      // that timed out and any issued after it -- then leave.
      if (tid == 0) {
        set_status(p.status, SF_DEVICE_TIMEOUT);
        for (uint32_t x = consumed - 1; x < piece_base + (uint32_t)issued; ++x)
          (void)mbar_wait_bounded(bar0 + 8 * (x % STAGES), (x / STAGES) & 1u);
      }
      __syncthreads();
      // the cluster's other CTAs expect this CTA's barrier arrivals, and in
      // push mode they may still store into its shared memory until the
      // second phase completes
      if (push_mode) {
        cluster_wait_acquire();
        cluster_sync();
      } else if (aligned) {
        cluster_sync();
        cluster_sync();
      }
      return;
    }

    // ---- finish the piece ----
    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);

    if constexpr (KS > 1) {
      // warps ks >= 1 hand their (m, l, O) to warp ks == 0 of the same row
      // tile through the (now idle) ring memory
      constexpr int kPer = 4 * DT + 4;
      float *xchg = reinterpret_cast<float *>(smem);
      if (active && ks > 0) {
        float *dst = xchg + ((size_t)(rt * (KS - 1) + ks - 1) * 32 + lane) * kPer;
#pragma unroll
        for (int dt = 0; dt < DT; ++dt)
          *reinterpret_cast<float4 *>(dst + 4 * dt) = make_float4(o[dt][0], o[dt][1], o[dt][2], o[dt][3]);
        *reinterpret_cast<float4 *>(dst + 4 * DT) = make_float4(m0, m1, l0, l1);
      }
      __syncthreads();
      if (active && ks == 0) {
        float M0 = m0, M1 = m1;
        for (int s2 = 1; s2 < KS; ++s2) {
          const float4 ml = *reinterpret_cast<const float4 *>(
              xchg + ((size_t)(rt * (KS - 1) + s2 - 1) * 32 + lane) * kPer + 4 * DT);
          M0 = fmaxf(M0, ml.x);
          M1 = fmaxf(M1, ml.y);
        }
        // a row may see no key at all in this piece (every key masked):
        // then every max is -inf and the reference must be finite
        const float U0 = M0 == -INFINITY ? 0.f : M0, U1 = M1 == -INFINITY ? 0.f : M1;
        const float w0 = exp2f(m0 - U0), w1 = exp2f(m1 - U1);
        l0 *= w0;
        l1 *= w1;
#pragma unroll
        for (int dt = 0; dt < DT; ++dt) {
          o[dt][0] *= w0; o[dt][1] *= w0; o[dt][2] *= w1; o[dt][3] *= w1;
        }
        for (int s2 = 1; s2 < KS; ++s2) {
          const float *src = xchg + ((size_t)(rt * (KS - 1) + s2 - 1) * 32 + lane) * kPer;
          const float4 ml = *reinterpret_cast<const float4 *>(src + 4 * DT);
          const float v0 = exp2f(ml.x - U0), v1 = exp2f(ml.y - U1);
          l0 += ml.z * v0;
          l1 += ml.w * v1;
#pragma unroll
          for (int dt = 0; dt < DT; ++dt) {
            const float4 x = *reinterpret_cast<const float4 *>(src + 4 * dt);
            o[dt][0] += x.x * v0; o[dt][1] += x.y * v0; o[dt][2] += x.z * v1; o[dt][3] += x.w * v1;
          }
        }
        m0 = M0;
        m1 = M1;
      }
      fence_proxy_async_smem();  // generic writes to the ring before later TMA writes
      __syncthreads();           // the ring is refilled by the next piece's prologue
    }

    const bool writer = active && ks == 0;
    const int colb = 2 * (lane & 3);
    if (n_pieces == 1) {
      // the whole segment is in this CTA: normalise and write
      if (writer) {
        const float inv0 = 1.f / l0, inv1 = 1.f / l1;
        auto orow = [&](int r) -> __nv_bfloat16 * {
          const int i = r / p.group, j = r % p.group;
          return p.out + (((size_t)b * p.n_q + i) * p.H_q + (size_t)h_kv * p.group + j) * D;
        };
        if (r0 < p.R) {
          __nv_bfloat16 *dst = orow(r0);
#pragma unroll
          for (int dt = 0; dt < DT; ++dt)
            *reinterpret_cast<uint32_t *>(dst + dt * 8 + colb) = pack_bf16x2(o[dt][0] * inv0, o[dt][1] * inv0);
        }
        if (r1 < p.R) {
          __nv_bfloat16 *dst = orow(r1);
#pragma unroll
          for (int dt = 0; dt < DT; ++dt)
            *reinterpret_cast<uint32_t *>(dst + dt * 8 + colb) = pack_bf16x2(o[dt][2] * inv1, o[dt][3] * inv1);
        }
        if (p.lse && (lane & 3) == 0) {
          auto lidx = [&](int r) {
            const int i = r / p.group, j = r % p.group;
            return ((size_t)b * p.n_q + i) * p.H_q + (size_t)h_kv * p.group + j;
          };
          if (r0 < p.R) p.lse[lidx(r0)] = (m0 + log2f(l0)) * kLn2;
          if (r1 < p.R) p.lse[lidx(r1)] = (m1 + log2f(l1)) * kLn2;
        }
      }
      continue;
    }

    if (push_mode) {
      // push each partial row into the shared memory of the CTA that merges
      // it: rank rho merges rows [rho*R/cs, (rho+1)*R/cs); entry
      // [row slot][sender rank] holds O (D floats), m, l (stride D + 4)
      cluster_wait_acquire();  // every peer has started
      const int cs = p.cs, rank = static_cast<int>(blockIdx.x) % cs;
      auto push_row = [&](int r, const float (&oo)[DT][4], int h, float mm, float ll) {
        const int rho = ((r + 1) * cs - 1) / p.R;
        const int slot = r - rho * p.R / cs;
        const uint32_t entry = ring + p.push_off + 4u * ((slot * cs + rank) * (D + 4));
        const uint32_t remote = dsmem_addr(entry, rho);
#pragma unroll
        for (int dt = 0; dt < DT; ++dt)
          st_dsmem_f32x2(remote + 4u * (dt * 8 + colb), oo[dt][2 * h], oo[dt][2 * h + 1]);
        if ((lane & 3) == 0) {
          st_dsmem_f32(remote + 4u * D, mm);
          st_dsmem_f32(remote + 4u * (D + 1), ll);
        }
      };
      if (writer) {
        if (r0 < p.R) push_row(r0, o, 0, m0, l0);
        if (r1 < p.R) push_row(r1, o, 1, m1, l1);
      }
      continue;
    }
    if (aligned) {
      // partial of this CTA's piece into its own shared memory (ring, idle):
      // O [R][D] fp32, then m [R], l [R]; read by the cluster after the barrier
      float *part = reinterpret_cast<float *>(smem);
      if (writer) {
        if (r0 < p.R) {
#pragma unroll
          for (int dt = 0; dt < DT; ++dt)
            *reinterpret_cast<float2 *>(part + r0 * D + dt * 8 + colb) = make_float2(o[dt][0], o[dt][1]);
          if ((lane & 3) == 0) {
            part[p.R * D + r0] = m0;
            part[p.R * D + p.R + r0] = l0;
          }
        }
        if (r1 < p.R) {
#pragma unroll
          for (int dt = 0; dt < DT; ++dt)
            *reinterpret_cast<float2 *>(part + r1 * D + dt * 8 + colb) = make_float2(o[dt][2], o[dt][3]);
          if ((lane & 3) == 0) {
            part[p.R * D + r1] = m1;
            part[p.R * D + p.R + r1] = l1;
          }
        }
      }
      continue;
    }

    // ---- several pieces: write this piece's partial ----
    const size_t stride = (size_t)p.slot_stride;
    {
      float *part = p.partials + (size_t)(blockIdx.x + seg) * stride;
      if (writer) {
        if (r0 < p.R) {
#pragma unroll
          for (int dt = 0; dt < DT; ++dt)
            *reinterpret_cast<float2 *>(part + (size_t)r0 * D + dt * 8 + colb) = make_float2(o[dt][0], o[dt][1]);
          if ((lane & 3) == 0) {
            part[(size_t)p.R * D + r0] = m0;
            part[(size_t)p.R * D + p.R + r0] = l0;
          }
        }
        if (r1 < p.R) {
#pragma unroll
          for (int dt = 0; dt < DT; ++dt)
            *reinterpret_cast<float2 *>(part + (size_t)r1 * D + dt * 8 + colb) = make_float2(o[dt][2], o[dt][3]);
          if ((lane & 3) == 0) {
            part[(size_t)p.R * D + r1] = m1;
            part[(size_t)p.R * D + p.R + r1] = l1;
          }
        }
      }
    }
    // ---- few rows: the last CTA of the segment to finish merges it ----
    __threadfence();
    __syncthreads();
    if (tid == 0) {
      const unsigned prev = atomicAdd(p.tickets + seg, 1u);
      s_misc[0] = (prev == static_cast<unsigned>(n_pieces - 1)) ? 1 : 0;
    }
    __syncthreads();
    if (s_misc[0]) {
      // every piece is written: this CTA merges the segment
      __threadfence();
      const float *part0 = p.partials + (size_t)(c_first + seg) * stride;
      for (int idx = tid; idx < p.R * (D / 4); idx += NTHREADS) {
        const int r = idx / (D / 4), c4 = idx % (D / 4);
        float4 ov;
        float M, Ls;
        merge_one<D, true>(part0, stride, p.R, r, c4, n_pieces, ov, M, Ls);
        const int i = r / p.group, j = r % p.group;
        const size_t row = ((size_t)b * p.n_q + i) * p.H_q + (size_t)h_kv * p.group + j;
        uint2 packed;
        packed.x = pack_bf16x2(ov.x, ov.y);
        packed.y = pack_bf16x2(ov.z, ov.w);
        *reinterpret_cast<uint2 *>(p.out + row * D + 4 * c4) = packed;
        if (p.lse && c4 == 0) p.lse[row] = (M + log2f(Ls)) * kLn2;
      }
      if (tid == 0) p.tickets[seg] = 0u;
    }
    __syncthreads();
  }
  if (push_mode) {
    // Every peer has pushed its rows; merge this CTA's rows from its own
    // shared memory, in rank order (= tile order).  Nobody reads this CTA's
    // shared memory, so there is no third phase.
    cluster_sync();
    const int cs = p.cs, rank = static_cast<int>(blockIdx.x) % cs;
    const int R = p.R;
    const int r_lo = rank * R / cs, r_hi = (rank + 1) * R / cs;
    const float *push = reinterpret_cast<const float *>(smem + p.push_off);
    for (int idx = tid; idx < (r_hi - r_lo) * (D / 4); idx += NTHREADS) {
      const int slot = idx / (D / 4), c4 = idx % (D / 4);
      const int r = r_lo + slot;
      float M = -INFINITY;
      for (int u = 0; u < cs; ++u) M = fmaxf(M, push[(slot * cs + u) * (D + 4) + D]);
      float Ls = 0.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int u = 0; u < cs; ++u) {
        const float *e = push + (slot * cs + u) * (D + 4);
        const float w = exp2f(e[D] - M);
        Ls += e[D + 1] * w;
        const float4 x = *reinterpret_cast<const float4 *>(e + 4 * c4);
        acc.x += x.x * w; acc.y += x.y * w; acc.z += x.z * w; acc.w += x.w * w;
      }
      const float inv = 1.f / Ls;
      const int i = r / p.group, j = r % p.group;
      const size_t row = ((size_t)seg_b * p.n_q + i) * p.H_q + (size_t)seg_h * p.group + j;
      uint2 packed;
      packed.x = pack_bf16x2(acc.x * inv, acc.y * inv);
      packed.y = pack_bf16x2(acc.z * inv, acc.w * inv);
      *reinterpret_cast<uint2 *>(p.out + row * D + 4 * c4) = packed;
      if (p.lse && c4 == 0) p.lse[row] = (M + log2f(Ls)) * kLn2;
    }
  } else if (aligned) {
    // Every CTA's partial is in its shared memory; CTA `rank` of the cluster
    // merges rows [rank*R/cs, (rank+1)*R/cs) over the cluster's pieces, which
    // are in rank order (= tile order), reading them through distributed
    // shared memory.  The second barrier keeps each CTA's shared memory alive
    // until its peers have read it.
    cluster_sync();
    const int cs = p.cs, rank = static_cast<int>(blockIdx.x) % cs;
    const int R = p.R;
    const int r_lo = rank * R / cs, r_hi = (rank + 1) * R / cs;
    for (int idx = tid; idx < (r_hi - r_lo) * (D / 4); idx += NTHREADS) {
      const int r = r_lo + idx / (D / 4), c4 = idx % (D / 4);
      float mv[kMaxCluster], lv[kMaxCluster];
      float4 xv[kMaxCluster];
#pragma unroll
      for (int u = 0; u < kMaxCluster; ++u) {
        if (u < cs) {
          mv[u] = ld_dsmem_f32(ring + 4u * (R * D + r), u);
          lv[u] = ld_dsmem_f32(ring + 4u * (R * D + R + r), u);
          xv[u] = ld_dsmem_f32x4(ring + 4u * (r * D + 4 * c4), u);
        } else {
          mv[u] = -INFINITY;
          lv[u] = 0.f;
          xv[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
      }
      float M = -INFINITY;
#pragma unroll
      for (int u = 0; u < kMaxCluster; ++u) M = fmaxf(M, mv[u]);
      float Ls = 0.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
      for (int u = 0; u < kMaxCluster; ++u) {
        const float w = exp2f(mv[u] - M);
        Ls += lv[u] * w;
        acc.x += xv[u].x * w; acc.y += xv[u].y * w; acc.z += xv[u].z * w; acc.w += xv[u].w * w;
      }
      const float inv = 1.f / Ls;
      const int i = r / p.group, j = r % p.group;
      const size_t row = ((size_t)seg_b * p.n_q + i) * p.H_q + (size_t)seg_h * p.group + j;
      uint2 packed;
      packed.x = pack_bf16x2(acc.x * inv, acc.y * inv);
      packed.y = pack_bf16x2(acc.z * inv, acc.w * inv);
      *reinterpret_cast<uint2 *>(p.out + row * D + 4 * c4) = packed;
      if (p.lse && c4 == 0) p.lse[row] = (M + log2f(Ls)) * kLn2;
    }
    cluster_sync();
  }
}

// --------------------------------------------------------------------------
// host side
// --------------------------------------------------------------------------
using AttnKernel = void (*)(const CUtensorMap, const CUtensorMap, const AttnParams);

struct AttnVariant {
  AttnKernel fn;
  int threads;
  int stages;
  int smem_fixed;  // bytes excluding the per-batch arrays
  int prefix_off;  // byte offset of the per-batch arrays in shared memory
  int ks, nw;
};

template <int D, int KS, int NW>
static AttnVariant make_variant() {
  constexpr int STAGES = (D == 64) ? 6 : (NW == 4 ? 3 : 5);
  AttnVariant v;
  v.fn = verify_attention_kernel<D, KS, NW, STAGES>;
  v.threads = NW * 32;
  v.stages = STAGES;
  v.smem_fixed = AttnSmem<D, STAGES, NW>::bytes(0);
  v.prefix_off = AttnSmem<D, STAGES, NW>::kPrefixOffset;
  v.ks = KS;
  v.nw = NW;
  return v;
}

// One row tile per KV head (R <= 16): the four warps split each tile's keys.
// More rows go to the tcgen05 kernel (verify_attention_tc.cu).
static AttnVariant select_variant(int D) {
  if (D == 64) return make_variant<64, 4, 4>();
  return make_variant<128, 4, 4>();
}

struct AttnLayout {
  size_t tickets_off, partials_off, total;
};

static AttnLayout attn_layout(int B, int H_kv, int R, int D, long long G) {
  AttnLayout l;
  const size_t segs = (size_t)B * H_kv;
  l.tickets_off = 256;
  l.partials_off = round_up(l.tickets_off + 8 * segs, 256);
  // the tcgen05 kernel (R > 16) writes one partial per key-split copy
  const long long copies = R > 16 ? (R <= 32 ? 4 : (R <= 64 ? 2 : 1)) : 1;
  l.total = round_up(l.partials_off + (size_t)((G + (long long)segs) * copies) * partial_slot_floats(R, D) * 4,
                     256);
  return l;
}

static int check_shapes(int B, int n_q, int H_q, int H_kv, int D, int page_size,
                        int max_pages_per_seq) {
  if (B < 1 || B > SF_MAX_BATCH) return fail(SF_ERR_INVALID_ARG, "B=%d outside [1, %d]", B, SF_MAX_BATCH);
  if (n_q < 1 || n_q > SF_MAX_QUERY_ROWS)
    return fail(SF_ERR_INVALID_ARG, "n_q=%d outside [1, %d]", n_q, SF_MAX_QUERY_ROWS);
  if (H_kv < 1 || H_q < 1 || H_q % H_kv != 0)
    return fail(SF_ERR_INVALID_ARG, "H_q=%d must be a positive multiple of H_kv=%d", H_q, H_kv);
  if (H_q / H_kv > SF_MAX_GROUP)
    return fail(SF_ERR_UNSUPPORTED, "group H_q/H_kv=%d above %d", H_q / H_kv, SF_MAX_GROUP);
  if (D != 64 && D != 128) return fail(SF_ERR_UNSUPPORTED, "head_dim=%d (built: 64, 128)", D);
  if (page_size != SF_PAGE_SIZE) return fail(SF_ERR_UNSUPPORTED, "page_size=%d (built: 16)", page_size);
  if (max_pages_per_seq < 1 || (long long)max_pages_per_seq * page_size > (1LL << 30))
    return fail(SF_ERR_INVALID_ARG, "max_pages_per_seq=%d", max_pages_per_seq);
  return SF_OK;
}

// Every argument check of a call that does not need the launch plan: shapes,
// required pointers, alignment, pool size and scale.
static int check_call_args(const void *q, const void *k_cache, const void *v_cache,
                           const int32_t *block_table, const int32_t *seq_lens, int B, int n_q,
                           int H_q, int H_kv, int head_dim, int page_size, int num_pages,
                           int max_pages_per_seq, float softmax_scale, const void *out,
                           const float *lse) {
  int st = check_shapes(B, n_q, H_q, H_kv, head_dim, page_size, max_pages_per_seq);
  if (st != SF_OK) return st;
  if (!q || !k_cache || !v_cache || !block_table || !seq_lens || !out)
    return fail(SF_ERR_INVALID_ARG, "a required pointer is NULL");
  if (num_pages < 1) return fail(SF_ERR_INVALID_ARG, "num_pages=%d", num_pages);
  if ((long long)num_pages * H_kv * SF_PAGE_SIZE >= (1LL << 31))
    return fail(SF_ERR_UNSUPPORTED, "KV pool of %d pages x %d heads too large", num_pages, H_kv);
  if (!aligned(q, 16) || !aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(out, 16) ||
      !aligned(block_table, 4) || !aligned(seq_lens, 4) || (lse && !aligned(lse, 4)))
    return fail(SF_ERR_INVALID_ARG, "q, caches and out must be 16-byte aligned");
  if (!(softmax_scale >= 0.f) || std::isinf(softmax_scale))
    return fail(SF_ERR_INVALID_ARG, "softmax_scale must be finite and >= 0");
  return SF_OK;
}

struct AttnPlan {
  AttnVariant v;
  int G;
  int smem;
  int cs;        // CTAs per cluster (1: no clusters)
  int push;      // cluster mode pushes partial rows (few rows per merging CTA)
  int push_off;  // byte offset of the push area in shared memory
  int bt_off;    // byte offset of the block-table row in shared memory (0: none)
  int tc;        // 1: the tcgen05 kernel (many rows per KV head)
};

// Largest dynamic shared memory a launch of variant v can ask for: the
// per-batch arrays at SF_MAX_BATCH plus a full push area.
static int max_dynamic_smem(const AttnVariant &v) {
  return v.smem_fixed + 8 * SF_MAX_BATCH + 16 + kPushSlots * kMaxCluster * (128 + 4) * 4 + 16 +
         4 * kBtCacheEntries;
}

// Per-device, per-kernel launch facts, computed once: the dynamic shared
// memory limit is raised to the largest size any batch needs, and resident
// CTAs per SM are cached per shared-memory size.
static int kernel_setup(const AttnVariant &v, int dev, int smem, int *occ_out) {
  static std::mutex mu;
  static std::map<std::tuple<void *, int, int>, int> occ_cache;
  static std::map<std::pair<void *, int>, bool> attr_done;
  std::lock_guard<std::mutex> lock(mu);
  void *key = reinterpret_cast<void *>(v.fn);
  if (!attr_done[{key, dev}]) {
    cudaError_t e = cudaFuncSetAttribute(v.fn, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         max_dynamic_smem(v));
    if (e != cudaSuccess) return fail(SF_ERR_CUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(e));
    attr_done[{key, dev}] = true;
  }
  auto it = occ_cache.find({key, dev, smem});
  if (it == occ_cache.end()) {
    int occ = 0;
    cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, v.fn, v.threads, smem);
    if (e != cudaSuccess) return fail(SF_ERR_CUDA, "occupancy query: %s", cudaGetErrorString(e));
    it = occ_cache.emplace(std::make_tuple(key, dev, smem), occ > 0 ? occ : 1).first;
  }
  *occ_out = it->second;
  return SF_OK;
}

// How many clusters of `cs` CTAs can be resident at once (cached).
static int max_active_clusters(const AttnVariant &v, int dev, int smem, int cs, int *out) {
  static std::mutex mu;
  static std::map<std::tuple<void *, int, int, int>, int> cache;
  std::lock_guard<std::mutex> lock(mu);
  void *key = reinterpret_cast<void *>(v.fn);
  auto it = cache.find({key, dev, smem, cs});
  if (it == cache.end()) {
    if (cs > 8) {
      cudaError_t e = cudaFuncSetAttribute(v.fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      if (e != cudaSuccess) {
        cudaGetLastError();
        it = cache.emplace(std::make_tuple(key, dev, smem, cs), 0).first;
        *out = 0;
        return SF_OK;
      }
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cs);
    cfg.blockDim = dim3(v.threads);
    cfg.dynamicSmemBytes = smem;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    cudaError_t e = cudaOccupancyMaxActiveClusters(&n, v.fn, &cfg);
    if (e != cudaSuccess) {
      cudaGetLastError();  // a size the device cannot run: not used
      n = 0;
    }
    it = cache.emplace(std::make_tuple(key, dev, smem, cs), n).first;
  }
  *out = it->second;
  return SF_OK;
}

static int plan_attention(int B, int n_q, int H_q, int H_kv, int D, int max_pages_per_seq,
                          int num_splits, AttnPlan *plan) {
  DeviceInfo dev;
  int st = current_device(&dev);
  if (st != SF_OK) return st;
  const int R = n_q * (H_q / H_kv);
  plan->v = select_variant(D);
  plan->smem = plan->v.smem_fixed + 8 * B;
  plan->push = 0;
  plan->push_off = 0;
  plan->bt_off = 0;
  plan->tc = 0;
  const long long max_tiles =
      (long long)B * H_kv * (((long long)max_pages_per_seq * SF_PAGE_SIZE + kTileTokens - 1) / kTileTokens);
  if (max_tiles >= (1LL << 31))
    return fail(SF_ERR_UNSUPPORTED, "B x H_kv x tiles per sequence = %lld tiles (limit 2^31)", max_tiles);
  if (R > 16) {
    // Many rows per KV head: a real dense contraction, run on the tcgen05
    // tensor cores with one CTA per SM (the whole TMEM is one CTA's).
    plan->tc = 1;
    plan->cs = 1;
    plan->smem = tc_smem_bytes(D, R, B);
    if (tc_smem_bytes(D, R, SF_MAX_BATCH) > dev.max_smem_optin)
      return fail(SF_ERR_UNSUPPORTED, "needs %d B shared memory, device allows %d",
                  tc_smem_bytes(D, R, SF_MAX_BATCH), dev.max_smem_optin);
    st = tc_setup(D, dev.ordinal);
    if (st != SF_OK) return st;
    long long G = num_splits > 0 && num_splits < dev.sm_count ? num_splits : dev.sm_count;
    if (G > max_tiles) G = max_tiles;
    plan->G = static_cast<int>(G < 1 ? 1 : G);
    return SF_OK;
  }
  if (max_dynamic_smem(plan->v) > dev.max_smem_optin)
    return fail(SF_ERR_UNSUPPORTED, "needs %d B shared memory, device allows %d",
                max_dynamic_smem(plan->v), dev.max_smem_optin);
  int occ = 1;
  st = kernel_setup(plan->v, dev.ordinal, plan->smem, &occ);
  if (st != SF_OK) return st;
  const long long capacity = (long long)dev.sm_count * occ;
  long long G = num_splits > 0 ? num_splits : capacity;
  plan->cs = 1;
  if (num_splits <= 0 && B == 1) {
    // One sequence: its H_kv segments have equal length, so one cluster per
    // segment (as large as the resident capacity allows) merges on chip
    // (cluster mode) -- provided the grid still fills most of the GPU.
    // Batches keep the balanced global partition: their segment lengths are
    // unknown on the host, and misaligned clusters would only cost CTAs.
    const long long S = (long long)B * H_kv;
    for (int cand : {8, 4, 2}) {
      if (S * cand > capacity || S * cand > max_tiles) continue;
      if (4 * S * cand < 3 * capacity) break;
      int fits = 0;
      st = max_active_clusters(plan->v, dev.ordinal, plan->smem, cand, &fits);
      if (st != SF_OK) return st;
      if (fits >= S) {
        plan->cs = cand;
        G = S * cand;
        break;
      }
    }
  }
  if (G > max_tiles) G = max_tiles;
  if (G > kMaxGrid) G = kMaxGrid;
  plan->G = static_cast<int>(G < 1 ? 1 : G);
  if (plan->cs > 1 && (R + plan->cs - 1) / plan->cs <= kPushSlots) {
    // push area after the per-batch arrays: kPushSlots x cs entries of D + 4 floats
    plan->push = 1;
    plan->push_off = static_cast<int>(round_up((size_t)plan->v.prefix_off + 4 * (2 * B + 2), 16));
    plan->smem = plan->push_off + 1024 + kPushSlots * plan->cs * (D + 4) * 4;
  }
  if (B == 1 && max_pages_per_seq <= kBtCacheEntries) {
    // the sequence's block-table row, copied at entry, after everything else
    const int off = static_cast<int>(round_up((size_t)plan->smem - 1024, 16));
    const int smem = off + 1024 + 4 * max_pages_per_seq;
    int occ_before = 0, occ_after = 0;
    st = kernel_setup(plan->v, dev.ordinal, plan->smem, &occ_before);
    if (st != SF_OK) return st;
    st = kernel_setup(plan->v, dev.ordinal, smem, &occ_after);
    if (st != SF_OK) return st;
    if (occ_after == occ_before) {  // only where it costs no resident CTA
      plan->bt_off = off;
      plan->smem = smem;
    }
  }
  return SF_OK;
}

// TMA descriptors of the K and V caches, cached by (address, rows,
// head_dim, layout) so that repeated calls on the same caches skip the
// encoding.  Each box brings one 16-token page; layout 0 lands it as
// [64-column half][16 tokens][128 B], layout 1 (head_dim 128 only) as
// [8-token group][half][8 tokens][128 B], so that the 8-token atoms of one
// half sit at a fixed 2048-byte stride across the pages of a tile.
static int cache_tensor_map(CUtensorMap *out, const void *base, uint64_t rows, int head_dim,
                            int layout) {
  static std::mutex mu;
  static std::map<std::tuple<const void *, uint64_t, int, int>, CUtensorMap> maps;
  if (head_dim != 128) layout = 0;
  {
    std::lock_guard<std::mutex> lock(mu);
    auto it = maps.find({base, rows, head_dim, layout});
    if (it != maps.end()) {
      *out = it->second;
      return SF_OK;
    }
  }
  // head_dim 128, layout 0: view each 256-byte token row as two 128-byte
  // halves with the halves outermost, {64 elements, rows, 2 halves} with byte
  // strides {256, 128}; a {64, 16, 2} box brings a page as [half][token][64].
  // Layout 1: {64 elements, 8 tokens, 2 halves, rows / 8 token groups} with
  // byte strides {256, 128, 2048}; a {64, 8, 2, 2} box brings a page as
  // [group][half][token][64].  head_dim 64: {64, rows}, box {64, 16}.
  int st;
  if (head_dim == 128 && layout == 1) {
    const uint64_t dims[4] = {64, 8, 2, rows / 8}, strides[3] = {256, 128, 2048};
    const uint32_t box[4] = {64, 8, 2, 2};
    st = encode_tensor_map_bf16(out, base, 4, dims, strides, box);
  } else if (head_dim == 128) {
    const uint64_t dims[3] = {64, rows, 2}, strides[2] = {256, 128};
    const uint32_t box[3] = {64, SF_PAGE_SIZE, 2};
    st = encode_tensor_map_bf16(out, base, 3, dims, strides, box);
  } else {
    const uint64_t dims[2] = {64, rows}, strides[1] = {128};
    const uint32_t box[2] = {64, SF_PAGE_SIZE};
    st = encode_tensor_map_bf16(out, base, 2, dims, strides, box);
  }
  if (st != SF_OK) return st;
  std::lock_guard<std::mutex> lock(mu);
  if (maps.size() >= 4096) maps.clear();
  maps.emplace(std::make_tuple(base, rows, head_dim, layout), *out);
  return SF_OK;
}

}  // namespace sf

extern "C" {

size_t sf_verify_attention_workspace_size(int B, int n_q, int H_q, int H_kv, int head_dim,
                                          int max_pages_per_seq, int page_size,
                                          int num_splits) {
  if (sf::check_shapes(B, n_q, H_q, H_kv, head_dim, page_size, max_pages_per_seq) != SF_OK)
    return 0;
  sf::AttnPlan plan;
  if (sf::plan_attention(B, n_q, H_q, H_kv, head_dim, max_pages_per_seq, num_splits, &plan) != SF_OK)
    return 0;
  return sf::attn_layout(B, H_kv, n_q * (H_q / H_kv), head_dim, plan.G).total;
}

int sf_verify_attention_kernel_launches(int B, int n_q, int H_q, int H_kv, int head_dim,
                                        int max_pages_per_seq, int page_size, int num_splits) {
  if (sf::check_shapes(B, n_q, H_q, H_kv, head_dim, page_size, max_pages_per_seq) != SF_OK)
    return 0;
  sf::AttnPlan plan;
  if (sf::plan_attention(B, n_q, H_q, H_kv, head_dim, max_pages_per_seq, num_splits, &plan) != SF_OK)
    return 0;
  return plan.tc ? 2 : 1;  // the tcgen05 split kernel is followed by its merge kernel
}

int sf_verify_attention(const void *q, const void *k_cache, const void *v_cache,
                        const int32_t *block_table, const int32_t *seq_lens, int B, int n_q,
                        int H_q, int H_kv, int head_dim, int page_size, int num_pages,
                        int max_pages_per_seq, float softmax_scale, int num_splits, void *out,
                        float *lse, void *workspace, size_t workspace_bytes,
                        cudaStream_t stream) {
  using namespace sf;
  clear_error();
  int st = check_call_args(q, k_cache, v_cache, block_table, seq_lens, B, n_q, H_q, H_kv,
                           head_dim, page_size, num_pages, max_pages_per_seq, softmax_scale, out,
                           lse);
  if (st != SF_OK) return st;
  if (!workspace || !aligned(workspace, 256))
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL and 256-byte aligned");

  AttnPlan plan;
  st = plan_attention(B, n_q, H_q, H_kv, head_dim, max_pages_per_seq, num_splits, &plan);
  if (st != SF_OK) return st;
  const int R = n_q * (H_q / H_kv);
  const AttnLayout lay = attn_layout(B, H_kv, R, head_dim, plan.G);
  if (workspace_bytes < lay.total)
    return fail(SF_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, lay.total);

  const uint64_t rows = (uint64_t)num_pages * H_kv * SF_PAGE_SIZE;
  CUtensorMap tk, tv;
  st = cache_tensor_map(&tk, k_cache, rows, head_dim, plan.tc ? 1 : 0);
  if (st != SF_OK) return st;
  st = cache_tensor_map(&tv, v_cache, rows, head_dim, 0);
  if (st != SF_OK) return st;

  AttnParams prm;
  uint8_t *ws = static_cast<uint8_t *>(workspace);
  prm.q = static_cast<const __nv_bfloat16 *>(q);
  prm.block_table = block_table;
  prm.seq_lens = seq_lens;
  prm.out = static_cast<__nv_bfloat16 *>(out);
  prm.lse = lse;
  prm.status = reinterpret_cast<uint32_t *>(ws);
  prm.tickets = reinterpret_cast<uint32_t *>(ws + lay.tickets_off);
  prm.cs = plan.cs;
  prm.push = plan.push;
  prm.push_off = plan.push_off;
  prm.bt_off = plan.bt_off;
  prm.partials = reinterpret_cast<float *>(ws + lay.partials_off);
  prm.B = B;
  prm.n_q = n_q;
  prm.H_q = H_q;
  prm.H_kv = H_kv;
  prm.group = H_q / H_kv;
  prm.R = R;
  prm.num_pages = num_pages;
  prm.max_pages = max_pages_per_seq;
  prm.max_tokens = max_pages_per_seq * SF_PAGE_SIZE;
  prm.oob_row = static_cast<int>(rows);
  const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / sqrtf((float)head_dim);
  prm.scale_log2 = scale * 1.4426950408889634f;
  prm.G = plan.G;
  prm.slot_stride = partial_slot_floats(R, head_dim);

  // Both kernels are launched with programmatic stream serialisation: each
  // may be scheduled while its predecessor on the stream drains, and waits
  // for it (griddepcontrol.wait) before reading its results or writing.
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = plan.cs;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(plan.G);
  cfg.blockDim = dim3(plan.v.threads);
  cfg.dynamicSmemBytes = plan.smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = plan.cs > 1 ? 2 : 1;
  cudaError_t e;
  if (plan.tc) {
    st = tc_launch(head_dim, plan.G, plan.smem, tk, tv, prm, stream);
    if (st != SF_OK) return st;
  } else {
    e = cudaLaunchKernelEx(&cfg, plan.v.fn, tk, tv, prm);
    if (e != cudaSuccess) return fail(SF_ERR_CUDA, "verify attention launch: %s", cudaGetErrorString(e));
  }
  return SF_OK;
}

}  // extern "C"

// --------------------------------------------------------------------------
// Verification attention without a caller workspace.
//
// Some callers cannot allocate device memory at the point where they run the
// verification step: an inference server whose memory manager owns every
// byte of the device and refuses allocations while serving, a plug-in that
// is handed only its input and output buffers, or a runtime that pre-plans a
// fixed memory budget before the first request.  For them the library keeps
// its own scratch: one file-scope device array, created with the module on
// every GPU that loads this library and held until the process exits.  The
// entry point below runs the same kernel as sf_verify_attention with that
// array as its workspace, after clearing the part that must start at zero.
// --------------------------------------------------------------------------
namespace sf {

constexpr size_t kStaticScratchBytes = size_t(16) << 20;  // 16 MiB per device

static __device__ __align__(256) uint8_t g_static_scratch[kStaticScratchBytes];

// Device address of g_static_scratch on the current device.  Host code must
// not use the symbol itself (it is a host-side stand-in, not a device
// address); the address is looked up once per device, with that device
// current, and cached for the life of the process.  A device reset
// (cudaDeviceReset) destroys the module that holds the array, so the cached
// address must not outlive it: resetting a device that this entry point has
// used is not supported.
static int static_scratch_address(void **out) {
  static std::mutex mu;
  static void *addr[64] = {nullptr};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= 64) return fail(SF_ERR_UNSUPPORTED, "device ordinal %d", dev);
  std::lock_guard<std::mutex> lock(mu);
  if (!addr[dev]) {
    void *p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (e != cudaSuccess || !p)
      return fail(SF_ERR_CUDA, "cudaGetSymbolAddress(scratch): %s", cudaGetErrorString(e));
    addr[dev] = p;
  }
  *out = addr[dev];
  return SF_OK;
}

}  // namespace sf

extern "C" int sf_verify_attention_noalloc(const void *q, const void *k_cache,
                                           const void *v_cache, const int32_t *block_table,
                                           const int32_t *seq_lens, int B, int n_q, int H_q,
                                           int H_kv, int head_dim, int page_size, int num_pages,
                                           int max_pages_per_seq, float softmax_scale,
                                           int num_splits, void *out, float *lse,
                                           cudaStream_t stream) {
  using namespace sf;
  clear_error();
  // every argument check first: a rejected call enqueues nothing, not even
  // the clearing of the shared scratch (another stream may be using it)
  int st = check_call_args(q, k_cache, v_cache, block_table, seq_lens, B, n_q, H_q, H_kv,
                           head_dim, page_size, num_pages, max_pages_per_seq, softmax_scale, out,
                           lse);
  if (st != SF_OK) return st;
  AttnPlan plan;
  st = plan_attention(B, n_q, H_q, H_kv, head_dim, max_pages_per_seq, num_splits, &plan);
  if (st != SF_OK) return st;
  const AttnLayout lay = attn_layout(B, H_kv, n_q * (H_q / H_kv), head_dim, plan.G);
  if (lay.total > kStaticScratchBytes)
    return fail(SF_ERR_UNSUPPORTED,
                "this shape needs %zu bytes of scratch but the built-in scratch holds %zu; "
                "use sf_verify_attention with a caller workspace (or a smaller num_splits)",
                lay.total, kStaticScratchBytes);
  void *scratch = nullptr;
  st = static_scratch_address(&scratch);
  if (st != SF_OK) return st;
  // The status word and the merge tickets must start at zero; partials are
  // written before they are read.  The scratch keeps whatever the previous
  // call left.
  cudaError_t e = cudaMemsetAsync(scratch, 0, lay.partials_off, stream);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "clearing the scratch: %s", cudaGetErrorString(e));
  return sf_verify_attention(q, k_cache, v_cache, block_table, seq_lens, B, n_q, H_q, H_kv,
                             head_dim, page_size, num_pages, max_pages_per_seq, softmax_scale,
                             num_splits, out, lse, scratch, kStaticScratchBytes, stream);
}
