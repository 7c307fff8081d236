// visual_compress.cu -- visual token compression of the draft model
// (Sec. 3.2, Eq. 3; Algorithm 1) on sm_103a:
//
//     F^_V = softmax(Q F_V^T) F_V
//
// per image or frame, with the learnable query set Q (C x d) shared by all
// frames, F_V (N x d) acting as both keys and values, the softmax over the
// frame's N tokens and no score scale (Eq. 3 writes none).  The sizes are
// the paper's: N = 576 -> C = 64 for LLaVA images, 324 -> 36 for QwenVL, at
// the hidden size d of the target (4096, 3584).
//
// GB300 design.  The work is 4 C N d flops per frame over 2 N d bytes of
// features: 2 C = 128 flop/byte for LLaVA, below the bf16 tensor ridge
// (~286), so the floor is reading the features once at HBM speed, and only
// tensor cores keep the arithmetic under that.  Three launches:
//  1. scores S = Q F_V^T for all frames at once ([C][F*N] fp32) with the
//     tcgen05 projection kernel of draft_tail.cu (queries as the N side, the
//     F*N feature rows streamed as the M side), the hidden dimension split
//     into ks ranges when F*N has too few 128-row tiles to fill the GPU
//     (each split writes partial sums); it copies the features after the
//     dependency wait and leaves them in L2 (evict_last) for 3.;
//  2. compress_softmax_kernel: one warp per (frame, query) sums the ks
//     partials in a fixed order, takes the row max, and writes the
//     unnormalised weights exp(s - max) rounded to bf16 into P [C][F][Np]
//     (Np = N rounded up to 64, zeros past N) and the sum of the rounded
//     weights into l [F][C];
//  3. compress_apply_kernel, one CTA per (128 output columns, frame): the
//     transposed product O^T = F_V^T P^T as a pipelined tcgen05 GEMM with
//     M = 128 feature columns (A = the frame's features, MN-major, two
//     64-column boxes per 64 tokens), N = C padded to 16 (B = P, K-major) and
//     K = 64 tokens per ring slot, the accumulator in tensor memory; warps 0-3
//     (lane = feature column) divide by l and store bf16, coalesced along d.
// N is at most 768 and C at most 128.  Every wait is bounded
// (SF_DEVICE_TIMEOUT).
#include <cmath>
#include <mutex>

#include "sf_device.cuh"
#include "sf_host.h"

namespace sf {

constexpr int kVcThreads = 192;
constexpr int kVcMmaWarp = 4;
constexpr int kVcProducerWarp = 5;
constexpr int kVcCols = 128;        // output columns per CTA (MMA M)
constexpr int kVcTokens = 64;       // tokens per ring slot (K)
constexpr int kVcMaxTokens = 768;   // N
constexpr int kVcMaxQueries = 128;  // C
constexpr int kVcMaxStages = 4;
constexpr uint32_t kVcFBytes = 2 * kVcTokens * 128;  // 64 tokens x 128 columns of features
constexpr int kVcSoftmaxWarps = 8;

struct VcSoftmaxParams {
  const float *scores;  // [ks][C][F*N]
  __nv_bfloat16 *P;     // [C][F*Np]
  float *l;             // [F][C]
  long long part_stride;  // C*F*N
  int ks, F, N, C, Np;
};

struct VcParams {
  const float *l;       // [F][C]
  __nv_bfloat16 *out;   // [F][C][d]
  uint32_t *status;
  int F, N, C, Cp, d, Np;
  int KT;               // Np / 64 ring slots per CTA
  int stages;
  uint32_t stage_bytes;
  uint32_t tmem_cols;
};

static size_t vc_smem_bytes(int stages, uint32_t stage_bytes, int C) {
  return 1024 + static_cast<size_t>(stages) * stage_bytes + 8 * (2 * stages + 1) + 64 + 4 * C;
}

// grid (F, ceil(C / 8)), 256 threads: warp w handles query 8 * blockIdx.y + w
// of frame blockIdx.x.
__global__ void __launch_bounds__(32 * kVcSoftmaxWarps)
compress_softmax_kernel(const __grid_constant__ VcSoftmaxParams p) {
  constexpr int kPer = kVcMaxTokens / 32;  // scores per lane
  grid_dependency_wait();  // the partial scores come from the projection
  grid_launch_dependents();
  const int f = blockIdx.x, c = blockIdx.y * kVcSoftmaxWarps + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (c >= p.C) return;
  const long long row = static_cast<long long>(c) * p.F * p.N + static_cast<long long>(f) * p.N;
  float x[kPer];
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    const int n = lane + 32 * i;
    x[i] = n < p.N ? __ldg(p.scores + row + n) : -INFINITY;
  }
  // the other hidden-range partials, added in split order
  for (int s = 1; s < p.ks; ++s) {
    const float *part = p.scores + s * p.part_stride + row;
#pragma unroll
    for (int i = 0; i < kPer; ++i) {
      const int n = lane + 32 * i;
      if (n < p.N) x[i] += __ldg(part + n);
    }
  }
  float m = -INFINITY;
#pragma unroll
  for (int i = 0; i < kPer; ++i) m = fmaxf(m, x[i]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  constexpr float kLog2e = 1.4426950408889634f;
  const float mb = m * kLog2e;
  __nv_bfloat16 *prow = p.P + static_cast<long long>(c) * p.F * p.Np + static_cast<long long>(f) * p.Np;
  float l = 0.f;
#pragma unroll
  for (int i = 0; i < kPer; ++i) {
    const int n = lane + 32 * i;
    if (n < p.Np) {
      const __nv_bfloat16 b = __float2bfloat16_rn(n < p.N ? fast_exp2(fmaf(x[i], kLog2e, -mb)) : 0.f);
      l += __bfloat162float(b);
      prow[n] = b;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
  if (lane == 0) p.l[f * p.C + c] = l;
}

__global__ void __launch_bounds__(kVcThreads, 1)
compress_apply_kernel(const __grid_constant__ CUtensorMap tmap_f, const __grid_constant__ CUtensorMap tmap_p,
                      const __grid_constant__ VcParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int S = p.stages;
  const uint32_t ring = smem_addr(smem);
  uint64_t *bar_mem = reinterpret_cast<uint64_t *>(smem + static_cast<size_t>(S) * p.stage_bytes);
  int *s_misc = reinterpret_cast<int *>(bar_mem + 2 * S + 1);  // [0] TMEM, [1] abort, [2] issued, [3] consumed
  float *s_inv = reinterpret_cast<float *>(s_misc + 16);       // 1 / l of the frame's queries
  volatile int *s_abort = s_misc + 1;
  const uint32_t bars = smem_addr(bar_mem);
  const int FULL = 0, EMPTY = S, DONE = 2 * S;
  auto bar = [&](int i) -> uint32_t { return bars + 8u * static_cast<uint32_t>(i); };

  const int chunk = blockIdx.x, f = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  grid_launch_dependents();
  if (tid == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(bar(FULL + i), 1);
      mbar_init(bar(EMPTY + i), 1);
    }
    mbar_init(bar(DONE), 1);
    fence_mbar_init();
    prefetch_tensormap(&tmap_f);
    prefetch_tensormap(&tmap_p);
    s_misc[1] = 0;
    s_misc[2] = 0;
    s_misc[3] = 0;
  }
  __syncthreads();  // barrier initialisation visible to every role
  // Tensor memory only once the previous kernel on the stream has completed
  // (a predecessor still waiting for its own predecessor may not have
  // allocated yet; holding TMEM here could deadlock the pair).
  uint32_t tmem = 0;
  if (warp != kVcProducerWarp) {
    if (warp == kVcMmaWarp) {
      grid_dependency_wait();
      tmem_alloc(smem_addr(s_misc), p.tmem_cols);
      tmem_relinquish_alloc_permit();
      tc_fence_before_sync();
    }
    named_bar_sync(3, 160);
    tc_fence_after_sync();
    tmem = static_cast<uint32_t>(s_misc[0]);
  }

  if (warp == kVcProducerWarp) {
    if (lane == 0) {
      grid_dependency_wait();  // P comes from the softmax kernel
      const uint64_t pol = l2_policy_evict_first();
      int k = 0;
      for (; k < p.KT; ++k) {
        const int slot = k % S;
        if (k >= S && !mbar_wait_or_abort(bar(EMPTY + slot), ((k / S) - 1) & 1, s_abort)) break;
        const uint32_t dst = ring + static_cast<uint32_t>(slot) * p.stage_bytes;
        mbar_arrive_expect_tx(bar(FULL + slot), p.stage_bytes);
        // features: tokens f*N + 64k .. +63 of columns [128 chunk, +64) and [+64, +128)
        tma_load_2d(dst, &tmap_f, chunk * kVcCols, f * p.N + k * kVcTokens, bar(FULL + slot), pol);
        tma_load_2d(dst + kVcFBytes / 2, &tmap_f, chunk * kVcCols + 64, f * p.N + k * kVcTokens,
                    bar(FULL + slot), pol);
        // weights of those tokens for every query (rows >= C are zero-filled)
        tma_load_2d(dst + kVcFBytes, &tmap_p, f * p.Np + k * kVcTokens, 0, bar(FULL + slot), pol);
      }
      s_misc[2] = k;
    }
    __syncwarp();
  } else if (warp == kVcMmaWarp) {
    const uint32_t idesc = idesc_bf16_f32(128, p.Cp, 1, 0);  // A MN-major, B K-major
    bool ok = true;
    for (int k = 0; k < p.KT; ++k) {
      const int slot = k % S;
      int w = 1;
      if (lane == 0) w = mbar_wait_or_abort(bar(FULL + slot), (k / S) & 1, s_abort);
      if (!__shfl_sync(0xffffffffu, w, 0)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      if (lane == 0) s_misc[3] = k + 1;
      const uint32_t base = ring + static_cast<uint32_t>(slot) * p.stage_bytes;
      if (elect_one()) {
#pragma unroll
        for (int kk = 0; kk < kVcTokens / 16; ++kk) {
          // A: 16 tokens = two 8-row atoms (2 KB) into each 64-column half;
          // the halves (M) are kVcFBytes / 2 apart.  B: 16 tokens = 32 bytes
          // along the 128-byte swizzled rows of P, 8-row groups 1 KB apart.
          const uint64_t a = smem_desc_sw128(base + kk * 2048u, kVcFBytes / 2, 1024);
          const uint64_t b = smem_desc_sw128(base + kVcFBytes + kk * 32u, 16, 1024);
          tc_mma_ss(tmem, a, b, idesc, (k > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(bar(EMPTY + slot));
      }
      __syncwarp();
    }
    if (ok && elect_one()) tc_commit(bar(DONE));
    __syncwarp();
    if (ok) (void)mbar_wait_bounded(bar(DONE), 0);
  } else {
    // ------------------------------------------------------------------
    // epilogue: lane = feature column 32 * warp + lane of the chunk, TMEM
    // columns = queries
    // ------------------------------------------------------------------
    grid_dependency_wait();  // l comes from the softmax kernel
    for (int c = tid; c < p.C; c += 128) {
      const float l = p.l[f * p.C + c];
      s_inv[c] = l > 0.f ? 1.f / l : 0.f;
    }
    named_bar_sync(1, 128);
    bool ok = mbar_wait_or_abort(bar(DONE), 0, s_abort);
    ok = __all_sync(0xffffffffu, ok);
    if (ok) {
      tc_fence_after_sync();
      const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * warp) << 16);
      __nv_bfloat16 *dst = p.out + static_cast<size_t>(f) * p.C * p.d + chunk * kVcCols + 32 * warp + lane;
      for (int c0 = 0; c0 < p.Cp; c0 += 16) {
        uint32_t v[16];
        tmem_ld_32x32b_x16(lane_base + static_cast<uint32_t>(c0), v);
#pragma unroll
        for (int j = 0; j < 16; ++j)
          if (c0 + j < p.C)
            dst[static_cast<size_t>(c0 + j) * p.d] = __float2bfloat16_rn(__uint_as_float(v[j]) * s_inv[c0 + j]);
      }
    }
    tc_fence_before_sync();
  }

  // ---- teardown ----
  __syncthreads();
  if (*s_abort) {
    if (tid == 0) set_status(p.status, SF_DEVICE_TIMEOUT);
    if (warp == kVcProducerWarp && lane == 0)
      for (int k = s_misc[3]; k < s_misc[2]; ++k) (void)mbar_wait_bounded(bar(FULL + k % S), (k / S) & 1);
    __syncthreads();
  }
  if (warp == kVcMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, p.tmem_cols);
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
static int vc_setup(const DeviceInfo &dev) {
  static std::mutex mu;
  static bool done[64] = {};
  if (dev.ordinal < 0 || dev.ordinal >= 64) return fail(SF_ERR_UNSUPPORTED, "device ordinal %d", dev.ordinal);
  std::lock_guard<std::mutex> lock(mu);
  if (done[dev.ordinal]) return SF_OK;
  cudaError_t e = cudaFuncSetAttribute(compress_apply_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       dev.max_smem_optin);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "cudaFuncSetAttribute (compressor): %s", cudaGetErrorString(e));
  done[dev.ordinal] = true;
  return SF_OK;
}

struct VcLayout {
  int ks;
  size_t scores, P, l, total;
};

static VcLayout vc_layout(int F, int N, int C, int d, int sm_count) {
  VcLayout L;
  L.ks = projection_splits(F * N, d, sm_count);
  const int Np = (N + kVcTokens - 1) / kVcTokens * kVcTokens;
  size_t off = 256;
  L.scores = off;
  off = round_up(off + static_cast<size_t>(L.ks) * C * F * N * sizeof(float), 256);
  L.P = off;
  off = round_up(off + static_cast<size_t>(C) * F * Np * 2, 256);
  L.l = off;
  off = round_up(off + static_cast<size_t>(F) * C * sizeof(float), 256);
  L.total = off;
  return L;
}

static int check_vc(const void *queries, const void *features, int F, int N, int C, int d, const void *out) {
  if (F < 1 || F > 65535) return fail(SF_ERR_INVALID_ARG, "F=%d outside [1, 65535]", F);
  if (N < 1 || N > kVcMaxTokens) return fail(SF_ERR_INVALID_ARG, "N=%d outside [1, %d]", N, kVcMaxTokens);
  if (C < 1 || C > kVcMaxQueries) return fail(SF_ERR_INVALID_ARG, "C=%d outside [1, %d]", C, kVcMaxQueries);
  if (d < kVcCols || d % kVcCols != 0 || d > (1 << 20))
    return fail(SF_ERR_INVALID_ARG, "d=%d must be a multiple of 128 in [128, 2^20]", d);
  if (static_cast<long long>(F) * N > SF_MAX_VOCAB)
    return fail(SF_ERR_INVALID_ARG, "F*N=%lld above %d", static_cast<long long>(F) * N, SF_MAX_VOCAB);
  if (!queries || !features || !out) return fail(SF_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!aligned(queries, 16) || !aligned(features, 16) || !aligned(out, 16))
    return fail(SF_ERR_INVALID_ARG, "queries, features and out must be 16-byte aligned");
  return SF_OK;
}

}  // namespace sf

extern "C" {

size_t sf_visual_compress_workspace_size(int F, int N, int C, int d) {
  using namespace sf;
  if (F < 1 || N < 1 || C < 1 || N > kVcMaxTokens || C > kVcMaxQueries || d < kVcCols) return 0;
  DeviceInfo dev;
  if (current_device(&dev) != SF_OK) return 0;
  return vc_layout(F, N, C, d, dev.sm_count).total;
}

int sf_visual_compress(const void *queries, const void *features, int F, int N, int C, int d,
                       void *out, void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  using namespace sf;
  clear_error();
  int st = check_vc(queries, features, F, N, C, d, out);
  if (st != SF_OK) return st;
  DeviceInfo dev;
  st = current_device(&dev);
  if (st != SF_OK) return st;
  if (dev.cc_major != 10) return fail(SF_ERR_UNSUPPORTED, "the compressor needs an sm_10x GPU");
  if (!workspace || !aligned(workspace, 256))
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL and 256-byte aligned");
  const VcLayout L = vc_layout(F, N, C, d, dev.sm_count);
  if (workspace_bytes < L.total)
    return fail(SF_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, L.total);
  st = vc_setup(dev);
  if (st != SF_OK) return st;

  uint8_t *ws = static_cast<uint8_t *>(workspace);
  uint32_t *status = reinterpret_cast<uint32_t *>(ws);
  float *scores = reinterpret_cast<float *>(ws + L.scores);
  __nv_bfloat16 *P = reinterpret_cast<__nv_bfloat16 *>(ws + L.P);
  float *lsum = reinterpret_cast<float *>(ws + L.l);
  const int Np = (N + kVcTokens - 1) / kVcTokens * kVcTokens;

  // 1. partial scores S_s = Q F_V^T over hidden range s, all frames: [ks][C][F*N]
  st = launch_projection(queries, features, C, d, F * N, scores, status, true, true, L.ks, stream);
  if (st != SF_OK) return st;

  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;

  // 2. weights P = bf16(exp(S - max)) and their sums l
  VcSoftmaxParams sp;
  sp.scores = scores;
  sp.P = P;
  sp.l = lsum;
  sp.part_stride = static_cast<long long>(C) * F * N;
  sp.ks = L.ks;
  sp.F = F;
  sp.N = N;
  sp.C = C;
  sp.Np = Np;
  cfg.gridDim = dim3(F, (C + kVcSoftmaxWarps - 1) / kVcSoftmaxWarps);
  cfg.blockDim = dim3(32 * kVcSoftmaxWarps);
  cfg.dynamicSmemBytes = 0;
  cudaError_t e = cudaLaunchKernelEx(&cfg, compress_softmax_kernel, sp);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "compressor softmax launch: %s", cudaGetErrorString(e));

  // 3. O^T = F_V^T P^T per (128 columns, frame), divided by l
  VcParams prm;
  prm.l = lsum;
  prm.out = static_cast<__nv_bfloat16 *>(out);
  prm.status = status;
  prm.F = F;
  prm.N = N;
  prm.C = C;
  prm.Cp = (C + 15) / 16 * 16;
  prm.d = d;
  prm.Np = Np;
  prm.KT = Np / kVcTokens;
  prm.stage_bytes = kVcFBytes + static_cast<uint32_t>(prm.Cp) * 128u;
  // a ring no deeper than the CTA's token chunks, and small enough for two
  // or more CTAs per SM (the CTAs are short: prologue and epilogue overlap)
  prm.stages = prm.KT < kVcMaxStages ? prm.KT : kVcMaxStages;
  while (prm.stages > 2 && vc_smem_bytes(prm.stages, prm.stage_bytes, C) > static_cast<size_t>(dev.max_smem_optin) / 2)
    --prm.stages;
  uint32_t cols = 32;
  while (cols < static_cast<uint32_t>(prm.Cp)) cols <<= 1;
  prm.tmem_cols = cols;
  CUtensorMap tmap_f, tmap_p;
  {
    const uint64_t dims[2] = {static_cast<uint64_t>(d), static_cast<uint64_t>(F) * N};
    const uint64_t strides[1] = {static_cast<uint64_t>(d) * 2};
    const uint32_t box[2] = {64, static_cast<uint32_t>(kVcTokens)};
    st = encode_tensor_map_bf16(&tmap_f, features, 2, dims, strides, box);
    if (st != SF_OK) return st;
  }
  {
    const uint64_t dims[2] = {static_cast<uint64_t>(F) * Np, static_cast<uint64_t>(C)};
    const uint64_t strides[1] = {static_cast<uint64_t>(F) * Np * 2};
    const uint32_t box[2] = {static_cast<uint32_t>(kVcTokens), static_cast<uint32_t>(prm.Cp)};
    st = encode_tensor_map_bf16(&tmap_p, P, 2, dims, strides, box);
    if (st != SF_OK) return st;
  }
  cfg.gridDim = dim3(d / kVcCols, F);
  cfg.blockDim = dim3(kVcThreads);
  cfg.dynamicSmemBytes = vc_smem_bytes(prm.stages, prm.stage_bytes, C);
  e = cudaLaunchKernelEx(&cfg, compress_apply_kernel, tmap_f, tmap_p, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "compressor launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

}  // extern "C"
