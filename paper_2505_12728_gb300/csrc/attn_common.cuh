// attn_common.cuh -- definitions shared by the verification-attention
// kernels (the mma.sync kernel and the tcgen05 kernel): kernel parameters,
// the shared-memory layout of one K/V page, the on-device tile partition.
#pragma once

#include "sf_device.cuh"

namespace sf {

constexpr int kTileTokens = 64;            // keys per ring stage
constexpr int kPageTokens = SF_PAGE_SIZE;  // 16
constexpr int kPagesPerTile = kTileTokens / kPageTokens;
constexpr int kRowBytes = 128;             // one swizzled smem row (64 bf16)
constexpr int kBeyondEnd = -2147483647 - 1;           // page past the sequence end
constexpr int kMaxGrid = 65535;  // CTAs of one launch (the partition uses 32-bit math)

struct AttnParams {
  const __nv_bfloat16 *q;
  const int32_t *block_table;
  const int32_t *seq_lens;
  __nv_bfloat16 *out;
  float *lse;
  uint32_t *status;
  uint32_t *tickets;  // [2 * B * H_kv], zero between calls (in-kernel merges)
  int cs;             // CTAs per cluster of the launch (1: no clusters)
  int push;           // cluster mode: peers push partial rows into the merging CTA
  int push_off;       // byte offset of the push area in dynamic shared memory
  int bt_off;         // one sequence: byte offset of its block-table row copied to
                      // dynamic shared memory at entry (0: read from global memory)
  float *partials;    // [G + B * H_kv][R][D + 2]
  int B, n_q, H_q, H_kv, group, R;
  int num_pages, max_pages, max_tokens;
  int oob_row;        // a tensor-map row beyond the pool: loads as zeros
  float scale_log2;   // softmax_scale * log2(e)
  int G;
  int slot_stride;    // floats per partial slot: R*D (O) + R (max) + R (sum), padded to 4
};

// The softmax weights (x, y) as two bf16 pairs: hi = their bf16 rounding,
// lo = the bf16 rounding of the remainder, so that hi + lo carries ~16
// significant bits.  P V is accumulated from both: with P rounded once to
// bf16 (8 bits) against a row sum l of the unrounded fp32 weights, rows with
// a handful of visible keys reached an output error of 1.05e-2.
__device__ __forceinline__ void split_bf16x2(float x, float y, uint32_t &hi, uint32_t &lo) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(x, y);
  const __nv_bfloat162 l = __floats2bfloat162_rn(x - __low2float(h), y - __high2float(h));
  hi = *reinterpret_cast<const uint32_t *>(&h);
  lo = *reinterpret_cast<const uint32_t *>(&l);
}

// Floats per partial slot; a multiple of 4 so every slot starts 16-byte aligned.
__host__ __device__ inline int partial_slot_floats(int R, int D) {
  return (R * (D + 2) + 3) / 4 * 4;
}

// Shared-memory layout of one K or V tile (64 tokens): one TMA box per page,
// [page][c / 8][token % 16][128 B], each 128-byte row 128B-swizzled.  Byte
// offset of 16-byte chunk `c` (head_dim / 8 index) of token `t`:
template <int D>
__device__ __forceinline__ uint32_t swz(int t, int c) {
  constexpr int kPageBytes = (D / 64) * kPageTokens * kRowBytes;
  return static_cast<uint32_t>((t >> 4) * kPageBytes + (c >> 3) * (kPageTokens * kRowBytes) +
                               (t & 15) * kRowBytes + (((c & 7) ^ (t & 7)) << 4));
}

// Exclusive prefix of per-sequence tile counts into s_prefix[0..B], clamped
// sequence lengths into s_len[0..B-1].
template <int NT>
__device__ void tile_prefix(const AttnParams &p, int *s_prefix, int *s_len, int *s_warp) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int per = (p.B + NT - 1) / NT;
  const int b0 = tid * per;
  int local = 0;
#pragma unroll 1
  for (int b = b0; b < b0 + per && b < p.B; ++b) {
    int T = p.seq_lens[b];
    if (T < p.n_q || T > p.max_tokens) {
      set_status(p.status, SF_DEVICE_BAD_SEQLEN);
      T = T < p.n_q ? p.n_q : p.max_tokens;
    }
    s_len[b] = T;
    local += (T + kTileTokens - 1) / kTileTokens;
  }
  int incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  int warp_off = 0;
#pragma unroll 1
  for (int w = 0; w < warp; ++w) warp_off += s_warp[w];
  int run = warp_off + incl - local;
#pragma unroll 1
  for (int b = b0; b < b0 + per && b < p.B; ++b) {
    s_prefix[b] = run;
    run += (s_len[b] + kTileTokens - 1) / kTileTokens;
  }
  if (tid == NT - 1) s_prefix[p.B] = warp_off + incl;
}

// The tile partition uses 32-bit arithmetic only (the host guarantees
// fewer than 2^31 tiles and G <= 65535): CTA c owns the global tiles
// [start(c), start(c+1)) with start(c) = floor(c * Tot / G), computed as
// c*q + floor(c*r / G) with q = Tot / G, r = Tot % G (c*r < G^2 < 2^32).
struct TilePartition {
  uint32_t Tot, G, q, r;
  __device__ __forceinline__ uint32_t start(uint32_t c) const { return c * q + (c * r) / G; }
  // CTA whose range contains tile t: an fp32 estimate, then exact steps
  __device__ __forceinline__ uint32_t owner(uint32_t t) const {
    int c = static_cast<int>((static_cast<float>(t) + 0.5f) * (static_cast<float>(G) / static_cast<float>(Tot)));
    c = c < 0 ? 0 : (c >= static_cast<int>(G) ? static_cast<int>(G) - 1 : c);
    while (c > 0 && start(static_cast<uint32_t>(c)) > t) --c;
    while (c + 1 < static_cast<int>(G) && start(static_cast<uint32_t>(c + 1)) <= t) ++c;
    return static_cast<uint32_t>(c);
  }
};

// Sequence b owning global tile t: H_kv * s_prefix[b] <= t < H_kv * s_prefix[b+1].
__device__ __forceinline__ int find_sequence(uint32_t t, const int *s_prefix, int B, int H_kv) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    int mid = (lo + hi + 1) >> 1;
    if (static_cast<uint32_t>(H_kv) * static_cast<uint32_t>(s_prefix[mid]) <= t) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Exclusive prefix over sequences b of H_kv * ceil(tiles_b / Ta) -- the CTAs
// a segment-aligned partition gives sequence b's H_kv segments -- into
// s_out[0..B] (s_out[B] = total).  s_warp: one int per warp.
template <int NT>
__device__ void aligned_prefix(const AttnParams &p, const int *s_prefix, int Ta, int *s_out,
                               int *s_warp) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int per = (p.B + NT - 1) / NT;
  const int b0 = tid * per;
  int local = 0;
#pragma unroll 1
  for (int b = b0; b < b0 + per && b < p.B; ++b)
    local += p.H_kv * ((s_prefix[b + 1] - s_prefix[b] + Ta - 1) / Ta);
  int incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int v = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  int warp_off = 0;
#pragma unroll 1
  for (int w = 0; w < warp; ++w) warp_off += s_warp[w];
  int run = warp_off + incl - local;
#pragma unroll 1
  for (int b = b0; b < b0 + per && b < p.B; ++b) {
    s_out[b] = run;
    run += p.H_kv * ((s_prefix[b + 1] - s_prefix[b] + Ta - 1) / Ta);
  }
  if (tid == NT - 1) s_out[p.B] = warp_off + incl;
}

// The piece of a CTA's tile range that starts at global tile t: segment
// (b, h_kv), its local tiles [lt0, lt0 + n_tiles), and how the segment is
// split over CTAs (c_first = CTA owning its first tile, n_pieces CTAs).
struct Piece {
  int b, h_kv, seg, lt0, n_tiles, c_first, n_pieces, T, Lb;
};

__device__ __forceinline__ Piece locate_piece(uint32_t t, uint32_t t_end, const TilePartition &part,
                                              const int *s_prefix, const int *s_len,
                                              const AttnParams &p) {
  Piece pc;
  pc.b = find_sequence(t, s_prefix, p.B, p.H_kv);
  const int tiles_b = s_prefix[pc.b + 1] - s_prefix[pc.b];
  const uint32_t seg_base = static_cast<uint32_t>(p.H_kv) * static_cast<uint32_t>(s_prefix[pc.b]);
  pc.h_kv = static_cast<int>((t - seg_base) / static_cast<uint32_t>(tiles_b));
  pc.lt0 = static_cast<int>((t - seg_base) % static_cast<uint32_t>(tiles_b));
  const uint32_t left = t_end - t;
  pc.n_tiles = left < static_cast<uint32_t>(tiles_b - pc.lt0) ? static_cast<int>(left) : tiles_b - pc.lt0;
  const uint32_t seg_first = seg_base + static_cast<uint32_t>(pc.h_kv) * static_cast<uint32_t>(tiles_b);
  pc.seg = pc.b * p.H_kv + pc.h_kv;
  pc.c_first = static_cast<int>(part.owner(seg_first));
  pc.n_pieces = static_cast<int>(part.owner(seg_first + tiles_b - 1)) - pc.c_first + 1;
  pc.T = s_len[pc.b];
  pc.Lb = pc.T - p.n_q;
  return pc;
}

constexpr int kMergeBatch = 16;

template <bool kBypassL1, typename T>
__device__ __forceinline__ T merge_load(const T *p) {
  if constexpr (kBypassL1) return __ldcg(p);
  else return *p;
}

// Combines the pieces of one output (row r, columns 4*c4 .. 4*c4+3) of a
// split segment, in piece order:
//   M = max_q m_q,  L = sum_q l_q 2^(m_q - M),  O = sum_q 2^(m_q - M) O_q / L.
// The pieces are read in batches of kMergeBatch with an online rescale; all
// loads of a batch are issued before any is used, so a batch costs one
// memory round trip.  Partial slot layout: O [R][D], m [R], l [R].
template <int D, bool kBypassL1, int BATCH = kMergeBatch>
__device__ __forceinline__ void merge_one(const float *part0, size_t stride, int R, int r, int c4,
                                          int n_pieces, float4 &o, float &M, float &Ls) {
  const float *mrow = part0 + (size_t)R * D + r;
  const float *lrow = mrow + R;
  const float4 *orow = reinterpret_cast<const float4 *>(part0 + (size_t)r * D) + c4;
  const size_t stride4 = stride / 4;
  M = -INFINITY;
  Ls = 0.f;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int q0 = 0; q0 < n_pieces; q0 += BATCH) {
    float mv[BATCH], lv[BATCH];
    float4 xv[BATCH];
#pragma unroll
    for (int u = 0; u < BATCH; ++u) {
      const bool in = q0 + u < n_pieces;
      mv[u] = in ? merge_load<kBypassL1>(mrow + (q0 + u) * stride) : -INFINITY;
      lv[u] = in ? merge_load<kBypassL1>(lrow + (q0 + u) * stride) : 0.f;
      xv[u] = in ? merge_load<kBypassL1>(orow + (q0 + u) * stride4) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float Mb = M;
#pragma unroll
    for (int u = 0; u < BATCH; ++u) Mb = fmaxf(Mb, mv[u]);
    const float a = exp2f(M - Mb);  // first batch: M = -inf, a = 0
    Ls *= a;
    acc.x *= a; acc.y *= a; acc.z *= a; acc.w *= a;
#pragma unroll
    for (int u = 0; u < BATCH; ++u) {
      const float w = exp2f(mv[u] - Mb);
      Ls += lv[u] * w;
      acc.x += xv[u].x * w; acc.y += xv[u].y * w; acc.z += xv[u].z * w; acc.w += xv[u].w * w;
    }
    M = Mb;
  }
  const float inv = 1.f / Ls;
  o = make_float4(acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv);
}

// Host side of the tcgen05 kernel (verify_attention_tc.cu).
// Dynamic shared memory of a launch with R rows per KV head and batch B (0
// if head_dim is not built).
int tc_smem_bytes(int head_dim, int R, int B);
// Raises the kernel's shared-memory limit once per device.
int tc_setup(int head_dim, int device);
// Launches the tcgen05 split kernel over G CTAs, then its merge kernel.
int tc_launch(int head_dim, int G, int smem, const CUtensorMap &tk, const CUtensorMap &tv,
              const AttnParams &prm, cudaStream_t stream);

}  // namespace sf
