// sf_host.h -- host-side helpers shared by the C-ABI translation units:
// thread-local error text, per-device properties, TMA descriptor encoding.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "specflash_verify.h"

namespace sf {

// Records a formatted message as the calling thread's last error and returns
// `status` (so call sites can `return fail(SF_ERR_..., "...")`).
int fail(int status, const char *fmt, ...);
void clear_error();

// Properties of the current device, cached per device ordinal.
struct DeviceInfo {
  int ordinal = -1;
  int sm_count = 0;
  int max_smem_optin = 0;
  int cc_major = 0, cc_minor = 0;
};
int current_device(DeviceInfo *info);

// cuTensorMapEncodeTiled for a bf16 tensor of `rank` dimensions (dims[0]
// innermost; strides[i] is the byte stride of dimension i+1), fetched
// through the runtime (no link-time libcuda).  128-byte swizzle, zero fill.
int encode_tensor_map_bf16(CUtensorMap *map, const void *base, int rank, const uint64_t *dims,
                           const uint64_t *strides, const uint32_t *box);

// out[r][v] = sum_j rows_r[r][j] * rows_v[v][j] (bf16 in, fp32 out) with the
// tcgen05 projection kernel of draft_tail.cu (1 <= R <= 256).  With
// inputs_after_wait both inputs are copied only after the previous kernel on
// the stream completes; keep_v_rows leaves rows_v in L2 for a second pass.
// With splits > 1 the hidden dimension is cut into `splits` ranges and
// split s writes its partial sums to out + s * R * V (the caller adds them).
int launch_projection(const void *rows_r, const void *rows_v, int R, int hidden_size, int V,
                      float *out, uint32_t *status, bool inputs_after_wait, bool keep_v_rows,
                      int splits, cudaStream_t stream);

// Hidden-dimension splits that fill the GPU when V has few 128-row tiles.
int projection_splits(int V, int hidden_size, int sm_count);

// The projection with softmax statistics in its epilogue: logits [R][V] and,
// per row and CTA (G = projection_groups(V, SM count) CTAs, CTA g owning
// rows [g*V/G, (g+1)*V/G)), a 16-byte record {max, first argmax,
// float-float sum of exp((x - max)/tau)} at stats[r * G + g]; row r uses
// temperature[r / rows_per_temperature] (<= 0: greedy, no sum).
struct SampStat;
int launch_projection_stats(const void *hidden, const void *weight, int R, int hidden_size, int V,
                            float *logits, const float *temperature, int rows_per_temperature,
                            SampStat *stats, uint32_t *status, int *G_out, cudaStream_t stream);
int projection_groups(int V, int sm_count);

inline bool aligned(const void *p, size_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}

inline size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace sf
