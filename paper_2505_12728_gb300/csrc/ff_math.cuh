// ff_math.cuh -- float-float arithmetic and fixed-order block reductions
// shared by the acceptance and draft-sampling kernels.  A float-float number
// is an unevaluated sum hi + lo of two fp32 values (~44 significant bits),
// built from exactly rounded fp32 operations (Knuth's TwoSum, FMA-based
// TwoProduct); every reduction runs in a fixed order, so results are
// deterministic.  Blocks are kFfThreads threads.
#pragma once

#include <climits>
#include <cmath>

#include "sf_device.cuh"

namespace sf {

constexpr int kFfThreads = 256;
constexpr int kFfWarps = kFfThreads / 32;

struct ff {       // float-float number hi + lo, |lo| <= ulp(hi) / 2
  float hi, lo;
};

// Softmax statistics of one chunk of one row: written by the projection
// epilogue (draft_tail.cu), read by the samplers and the fused acceptance.
struct SampStat {
  float m;  // largest logit of the chunk
  int arg;  // its first index
  ff S;     // sum of exp((x - m) / tau) over the chunk; 0 for greedy rows
};
static_assert(sizeof(SampStat) == 16, "SampStat is 16 bytes");

// (value, index) order for argmax: larger value first, then lower index.
__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

// Float-float arithmetic (Knuth's TwoSum and an FMA-based TwoProduct); the
// explicit _rn intrinsics keep the compiler from contracting or reordering.
__device__ __forceinline__ ff ff_of(float x) { return ff{x, 0.f}; }

__device__ __forceinline__ ff ff_add(ff a, ff b) {
  const float s = __fadd_rn(a.hi, b.hi);
  const float v = __fsub_rn(s, a.hi);
  float e = __fadd_rn(__fsub_rn(a.hi, __fsub_rn(s, v)), __fsub_rn(b.hi, v));
  e = __fadd_rn(e, __fadd_rn(a.lo, b.lo));
  const float hi = __fadd_rn(s, e);
  return ff{hi, __fsub_rn(e, __fsub_rn(hi, s))};
}

__device__ __forceinline__ ff ff_mul(ff a, float b) {
  const float p = __fmul_rn(a.hi, b);
  float e = __fmaf_rn(a.hi, b, -p);
  e = __fmaf_rn(a.lo, b, e);
  const float hi = __fadd_rn(p, e);
  return ff{hi, __fsub_rn(e, __fsub_rn(hi, p))};
}

__device__ __forceinline__ bool ff_lt(ff a, ff b) {
  return a.hi < b.hi || (a.hi == b.hi && a.lo < b.lo);
}

__device__ __forceinline__ bool ff_pos(ff a) { return a.hi > 0.f || (a.hi == 0.f && a.lo > 0.f); }

// a / b rounded to fp32 (one Newton correction of the fp32 quotient).
__device__ __forceinline__ float ff_div_to_f(float a, ff b) {
  const float q = __fdiv_rn(a, b.hi);
  float r = __fmaf_rn(-q, b.hi, a);  // a - q * b.hi, exact
  r = __fmaf_rn(-q, b.lo, r);
  return __fadd_rn(q, __fdiv_rn(r, b.hi));
}

// exp((x - m) / tau) with the argument carried to float-float, so that the
// result is as accurate as expf itself even for large |x - m|; 0 for a
// masked token (x = -inf), where the float-float split would give NaN.
__device__ __forceinline__ float exp_diff_accurate(float x, float m, float tau) {
  if (x == -INFINITY) return 0.f;
  float hi = __fsub_rn(x, m);
  const float v = __fsub_rn(hi, x);
  float lo = __fadd_rn(__fsub_rn(x, __fsub_rn(hi, v)), __fsub_rn(-m, v));
  if (tau != 1.0f) {
    const float qh = __fdiv_rn(hi, tau);
    const float r = __fmaf_rn(-qh, tau, hi);  // hi - qh * tau, exact
    lo = __fdiv_rn(__fadd_rn(r, lo), tau);
    hi = qh;
  }
  return __fmul_rn(expf(hi), __fadd_rn(1.0f, lo));
}

// Hardware base-2 exponential (approximate, subnormal results kept).
__device__ __forceinline__ float ex2_approx(float x) {
  float y;
  asm("ex2.approx.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// exp(a) = 2^(a log2 e) with a * log2 e carried as hi + lo (log2 e split
// into the float nearest it and the remainder, an FMA for the rounding of
// hi), 2^hi from ex2.approx and 2^lo ~ 1 + lo ln 2 (|lo| is a few ulp of
// hi).  Measured against expf on GB300 over [-103, 1]: max relative error
// 2.4e-7 (expf 1.5e-7).  For the hot loops of the acceptance, where it
// replaces expf.
__device__ __forceinline__ float exp_fast(float a) {
  constexpr float kL2eHi = 1.44269502162933349609375f;   // nearest float to log2 e
  constexpr float kL2eLo = 1.9259630335000111e-08f;       // log2 e - kL2eHi
  const float hi = __fmul_rn(a, kL2eHi);
  const float lo = __fmaf_rn(a, kL2eLo, __fmaf_rn(a, kL2eHi, -hi));
  const float r = __fmul_rn(ex2_approx(hi), __fmaf_rn(lo, 0.69314718055994531f, 1.0f));
  return a == -INFINITY ? 0.f : r;  // lo is NaN there
}

__device__ __forceinline__ ff shfl_xor_ff(ff a, int o) {
  return ff{__shfl_xor_sync(0xffffffffu, a.hi, o), __shfl_xor_sync(0xffffffffu, a.lo, o)};
}

__device__ __forceinline__ ff shfl_up_ff(ff a, int o) {
  return ff{__shfl_up_sync(0xffffffffu, a.hi, o), __shfl_up_sync(0xffffffffu, a.lo, o)};
}

__device__ __forceinline__ ff warp_sum_ff(ff v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = ff_add(v, shfl_xor_ff(v, o));
  return v;
}

__device__ __forceinline__ void warp_argmax(float &v, int &i) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (better(ov, oi, v, i)) { v = ov; i = oi; }
  }
}

// Block-wide float-float sum (fixed tree order).
__device__ inline ff block_sum(ff v, ff *s_buf) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum_ff(v);
  __syncthreads();
  if (lane == 0) s_buf[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < kFfWarps ? s_buf[lane] : ff_of(0.f);
    v = warp_sum_ff(v);
    if (lane == 0) s_buf[0] = v;
  }
  __syncthreads();
  return s_buf[0];
}

__device__ inline void block_argmax(float &v, int &i, float *s_v, int *s_i) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  warp_argmax(v, i);
  __syncthreads();
  if (lane == 0) { s_v[warp] = v; s_i[warp] = i; }
  __syncthreads();
  if (warp == 0) {
    v = lane < kFfWarps ? s_v[lane] : -INFINITY;
    i = lane < kFfWarps ? s_i[lane] : INT_MAX;
    warp_argmax(v, i);
    if (lane == 0) { s_v[0] = v; s_i[0] = i; }
  }
  __syncthreads();
  v = s_v[0];
  i = s_i[0];
}

// Inclusive float-float prefix sum over the block (fixed order).  Returns
// the thread's inclusive value; *excl receives its exclusive value (the
// previous thread's inclusive value, bit for bit) and *total the block total
// (the last thread's inclusive value).  s_buf holds kFfWarps + 1 values.
__device__ inline ff block_inclusive_scan(ff v, ff *s_buf, ff *excl, ff *total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const ff n = shfl_up_ff(v, o);
    if (lane >= o) v = ff_add(n, v);
  }
  __syncthreads();
  if (lane == 31) s_buf[warp] = v;  // warp totals
  __syncthreads();
  if (threadIdx.x == 0) {
    // warp offsets in sequence: off(w) = ff_add(off(w-1), t(w-1)) is, bit for
    // bit, the inclusive value of the last thread of warp w-1
    ff off = ff_of(0.f);
    for (int w = 0; w < kFfWarps; ++w) {
      const ff t = s_buf[w];
      s_buf[w] = off;
      off = ff_add(off, t);
    }
    s_buf[kFfWarps] = off;
  }
  __syncthreads();
  const ff off = s_buf[warp];
  const ff incl = ff_add(off, v);
  const ff prev = shfl_up_ff(incl, 1);
  *excl = lane > 0 ? prev : off;
  *total = s_buf[kFfWarps];
  __syncthreads();  // s_buf is reused by the next call
  return incl;
}

}  // namespace sf
