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
// tensor cores keep the arithmetic under that.  Two launches:
//  1. scores S = Q F_V^T for all frames at once ([C][F*N] fp32) with the
//     tcgen05 projection kernel of draft_tail.cu (queries as the N side,
//     the F*N feature rows streamed as the M side); it copies the features
//     after the dependency wait and leaves them in L2 (evict_last) for 2.;
//  2. compress_apply_kernel, one CTA per (128 output columns, frame): warp 5
//     copies the frame's features for those columns into shared memory
//     ([64-column half][N tokens][128 B], 128B-swizzled: the MN-major B
//     operand); warps 0-3 hold one query per TMEM lane, read its N scores,
//     and store the unnormalised weights exp(s - max) as bf16 into tensor
//     memory (the A operand); warp 4 issues O = P F_V as N/16 MMAs of M = 128
//     (queries), N = 128 (columns), K = 16 (tokens); warps 0-3 divide by the
//     sum of the bf16 weights and store bf16 rows.
// N is at most 768 (P takes N/2 TMEM columns beside the 128 of O) and C at
// most 128 (one lane per query).  Every wait is bounded (SF_DEVICE_TIMEOUT).
#include <cmath>
#include <mutex>

#include "sf_device.cuh"
#include "sf_host.h"

namespace sf {

constexpr int kVcThreads = 192;
constexpr int kVcMmaWarp = 4;
constexpr int kVcProducerWarp = 5;
constexpr int kVcCols = 128;        // output columns per CTA (MMA N)
constexpr int kVcMaxTokens = 768;   // N
constexpr int kVcMaxQueries = 128;  // C
constexpr uint32_t kVcTmemCols = 512;
constexpr uint32_t kVcTmemO = 0, kVcTmemP = 128;

struct VcParams {
  const float *scores;  // [C][F*N]
  __nv_bfloat16 *out;   // [F][C][d]
  uint32_t *status;
  long long score_stride;  // F*N
  int F, N, C, d;
  int Npad;             // N rounded up to 16 (MMA K)
  int BT;               // token rows per TMA box (divides Npad)
  int vec4;             // score rows are 16-byte aligned (N % 4 == 0)
};

static size_t vc_smem_bytes(int Npad) {
  return 1024 + 2 * static_cast<size_t>(Npad) * 128 + 64;
}

__global__ void __launch_bounds__(kVcThreads, 1)
compress_apply_kernel(const __grid_constant__ CUtensorMap tmap_f, const __grid_constant__ VcParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const uint32_t fv = smem_addr(smem);
  const uint32_t half_bytes = static_cast<uint32_t>(p.Npad) * 128u;
  uint64_t *bar_mem = reinterpret_cast<uint64_t *>(smem + 2 * static_cast<size_t>(half_bytes));
  int *s_misc = reinterpret_cast<int *>(bar_mem + 3);  // [0] TMEM base, [1] abort, [2] copies issued
  volatile int *s_abort = s_misc + 1;
  const uint32_t FVFULL = smem_addr(bar_mem), PFULL = FVFULL + 8, ODONE = FVFULL + 16;

  const int chunk = blockIdx.x, f = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  grid_launch_dependents();
  if (tid == 0) {
    mbar_init(FVFULL, 1);
    mbar_init(PFULL, 128);
    mbar_init(ODONE, 1);
    fence_mbar_init();
    prefetch_tensormap(&tmap_f);
    s_misc[1] = 0;
    s_misc[2] = 0;
  }
  if (warp == kVcMmaWarp) {
    tmem_alloc(smem_addr(s_misc), kVcTmemCols);
    tmem_relinquish_alloc_permit();
    tc_fence_before_sync();
  }
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = static_cast<uint32_t>(s_misc[0]);

  if (warp == kVcProducerWarp) {
    if (lane == 0) {
      // the features may come from the previous kernel on the stream
      grid_dependency_wait();
      const uint64_t pol = l2_policy_evict_first();
      mbar_arrive_expect_tx(FVFULL, 2 * half_bytes);
      for (int h = 0; h < 2; ++h)
        for (int t0 = 0; t0 < p.Npad; t0 += p.BT)
          tma_load_2d(fv + h * half_bytes + static_cast<uint32_t>(t0) * 128u, &tmap_f,
                      chunk * kVcCols + h * 64, f * p.N + t0, FVFULL, pol);
      s_misc[2] = 1;
    }
    __syncwarp();
  } else if (warp == kVcMmaWarp) {
    int w = 1;
    if (lane == 0)
      w = mbar_wait_or_abort(PFULL, 0, s_abort) && mbar_wait_or_abort(FVFULL, 0, s_abort);
    if (__shfl_sync(0xffffffffu, w, 0)) {
      tc_fence_after_sync();
      constexpr uint32_t kIdesc = idesc_bf16_f32(128, kVcCols, 0, 1);  // P from TMEM, F_V MN-major
      if (elect_one()) {
        for (int s = 0; s < p.Npad / 16; ++s) {
          // 16 tokens = two 8-row swizzle atoms (2 KB) per half; the two
          // 64-column halves of N are half_bytes apart
          const uint64_t b = smem_desc_sw128(fv + static_cast<uint32_t>(s) * 2048u, half_bytes, 1024);
          tc_mma_ts(tmem + kVcTmemO, tmem + kVcTmemP + static_cast<uint32_t>(s) * 8u, b, kIdesc,
                    s > 0 ? 1u : 0u);
        }
        tc_commit(ODONE);
      }
      __syncwarp();
      // every MMA has completed before the teardown frees TMEM
      (void)mbar_wait_bounded(ODONE, 0);
    }
  } else {
    // ------------------------------------------------------------------
    // weights and output: thread = query c = TMEM lane
    // ------------------------------------------------------------------
    const int c = 32 * warp + lane;
    const bool valid = c < p.C;
    const bool warp_used = 32 * warp < p.C;
    const uint32_t lane_base = tmem + (static_cast<uint32_t>(32 * warp) << 16);
    grid_dependency_wait();  // the scores come from the previous kernel
    float l = 0.f;
    if (warp_used) {
      const float *srow = p.scores + (valid ? c : 0) * p.score_stride + static_cast<long long>(f) * p.N;
      float m = -INFINITY;
      if (valid) {
        if (p.vec4) {
          for (int n = 0; n < p.N; n += 4) {
            const float4 v = __ldg(reinterpret_cast<const float4 *>(srow + n));
            m = fmaxf(m, fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w)));
          }
        } else {
          for (int n = 0; n < p.N; ++n) m = fmaxf(m, __ldg(srow + n));
        }
      }
      constexpr float kLog2e = 1.4426950408889634f;
      const float mb = m * kLog2e;
      // 64 tokens (32 TMEM columns of bf16 pairs) per store
      for (int g = 0; g < (p.Npad + 63) / 64; ++g) {
        uint32_t pk[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int n0 = g * 64 + 2 * j;
          float e0 = 0.f, e1 = 0.f;
          if (valid && n0 < p.N) e0 = fast_exp2(fmaf(__ldg(srow + n0), kLog2e, -mb));
          if (valid && n0 + 1 < p.N) e1 = fast_exp2(fmaf(__ldg(srow + n0 + 1), kLog2e, -mb));
          const __nv_bfloat16 b0 = __float2bfloat16_rn(e0), b1 = __float2bfloat16_rn(e1);
          l += __bfloat162float(b0) + __bfloat162float(b1);
          pk[j] = static_cast<uint32_t>(__bfloat16_as_ushort(b0)) |
                  (static_cast<uint32_t>(__bfloat16_as_ushort(b1)) << 16);
        }
        tmem_st_32x32b_x32(lane_base + kVcTmemP + static_cast<uint32_t>(g) * 32u, pk);
      }
      tmem_wait_st();
    }
    tc_fence_before_sync();
    mbar_arrive(PFULL);

    bool ok = mbar_wait_or_abort(ODONE, 0, s_abort);
    ok = __all_sync(0xffffffffu, ok);
    if (ok && warp_used) {
      tc_fence_after_sync();
      const float inv = valid && l > 0.f ? 1.f / l : 0.f;
#pragma unroll 1
      for (int h = 0; h < 2; ++h) {
        uint32_t v[64];
        tmem_ld_32x32b_x64(lane_base + kVcTmemO + static_cast<uint32_t>(h) * 64u, v);
        if (valid) {
          uint4 *dst = reinterpret_cast<uint4 *>(
              p.out + (static_cast<size_t>(f) * p.C + c) * p.d + chunk * kVcCols + h * 64);
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            uint4 w4;
            w4.x = pack_bf16x2(__uint_as_float(v[8 * q + 0]) * inv, __uint_as_float(v[8 * q + 1]) * inv);
            w4.y = pack_bf16x2(__uint_as_float(v[8 * q + 2]) * inv, __uint_as_float(v[8 * q + 3]) * inv);
            w4.z = pack_bf16x2(__uint_as_float(v[8 * q + 4]) * inv, __uint_as_float(v[8 * q + 5]) * inv);
            w4.w = pack_bf16x2(__uint_as_float(v[8 * q + 6]) * inv, __uint_as_float(v[8 * q + 7]) * inv);
            dst[q] = w4;
          }
        }
      }
    }
    tc_fence_before_sync();
  }

  // ---- teardown ----
  __syncthreads();
  if (*s_abort) {
    if (tid == 0) set_status(p.status, SF_DEVICE_TIMEOUT);
    // copies issued but never consumed: wait (bounded) until they land
    if (warp == kVcProducerWarp && lane == 0 && s_misc[2]) (void)mbar_wait_bounded(FVFULL, 0);
    __syncthreads();
  }
  if (warp == kVcMmaWarp) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kVcTmemCols);
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
                                       static_cast<int>(vc_smem_bytes(kVcMaxTokens)));
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "cudaFuncSetAttribute (compressor): %s", cudaGetErrorString(e));
  done[dev.ordinal] = true;
  return SF_OK;
}

// Token rows per TMA box: the largest multiple of 16 that divides Npad and
// is at most 256 (boxes tile each half exactly, 1024-byte aligned).
static int box_tokens(int Npad) {
  const int k = Npad / 16;
  int q = 16;
  while (k % q) --q;
  return 16 * q;
}

static size_t vc_workspace(int F, int N, int C) {
  return 256 + round_up(static_cast<size_t>(C) * F * N * sizeof(float), 256);
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

size_t sf_visual_compress_workspace_size(int F, int N, int C) {
  if (F < 1 || N < 1 || C < 1 || N > sf::kVcMaxTokens || C > sf::kVcMaxQueries) return 0;
  return sf::vc_workspace(F, N, C);
}

int sf_visual_compress(const void *queries, const void *features, int F, int N, int C, int d,
                       void *out, void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  using namespace sf;
  clear_error();
  int st = check_vc(queries, features, F, N, C, d, out);
  if (st != SF_OK) return st;
  if (!workspace || !aligned(workspace, 256))
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL and 256-byte aligned");
  const size_t need = vc_workspace(F, N, C);
  if (workspace_bytes < need)
    return fail(SF_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, need);
  DeviceInfo dev;
  st = current_device(&dev);
  if (st != SF_OK) return st;
  if (dev.cc_major != 10) return fail(SF_ERR_UNSUPPORTED, "the compressor needs an sm_10x GPU");
  st = vc_setup(dev);
  if (st != SF_OK) return st;

  uint8_t *ws = static_cast<uint8_t *>(workspace);
  uint32_t *status = reinterpret_cast<uint32_t *>(ws);
  float *scores = reinterpret_cast<float *>(ws + 256);
  // 1. S = Q F_V^T over all frames: [C][F*N]
  st = launch_projection(queries, features, C, d, F * N, scores, status, true, true, stream);
  if (st != SF_OK) return st;

  // 2. per (128 columns, frame): softmax over the frame's tokens and P F_V
  VcParams prm;
  prm.scores = scores;
  prm.out = static_cast<__nv_bfloat16 *>(out);
  prm.status = status;
  prm.score_stride = static_cast<long long>(F) * N;
  prm.F = F;
  prm.N = N;
  prm.C = C;
  prm.d = d;
  prm.Npad = (N + 15) / 16 * 16;
  prm.BT = box_tokens(prm.Npad);
  prm.vec4 = N % 4 == 0 ? 1 : 0;
  CUtensorMap tmap;
  const uint64_t dims[2] = {static_cast<uint64_t>(d), static_cast<uint64_t>(F) * N};
  const uint64_t strides[1] = {static_cast<uint64_t>(d) * 2};
  const uint32_t box[2] = {64, static_cast<uint32_t>(prm.BT)};
  st = encode_tensor_map_bf16(&tmap, features, 2, dims, strides, box);
  if (st != SF_OK) return st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(d / kVcCols, F);
  cfg.blockDim = dim3(kVcThreads);
  cfg.dynamicSmemBytes = vc_smem_bytes(prm.Npad);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, compress_apply_kernel, tmap, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "compressor launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

}  // extern "C"
