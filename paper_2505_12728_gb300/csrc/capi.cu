// capi.cu -- the library-wide C entry points (status strings, last error,
// version, workspace initialisation and status read-back) and the host
// helpers declared in sf_host.h.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "sf_device.cuh"
#include "sf_host.h"

namespace sf {

static thread_local char g_last_error[512] = "";

int fail(int status, const char *fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
  va_end(ap);
  return status;
}

void clear_error() { g_last_error[0] = '\0'; }

int current_device(DeviceInfo *info) {
  static std::mutex mu;
  static DeviceInfo cache[64];
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e));
  if (dev < 0 || dev >= 64) return fail(SF_ERR_UNSUPPORTED, "device ordinal %d", dev);
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev].ordinal != dev) {
    DeviceInfo d;
    d.ordinal = dev;
    if ((e = cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&d.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&d.cc_major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&d.cc_minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess)
      return fail(SF_ERR_CUDA, "cudaDeviceGetAttribute: %s", cudaGetErrorString(e));
    cache[dev] = d;
  }
  *info = cache[dev];
  return SF_OK;
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *,
                                  const cuuint64_t *, const cuuint64_t *, const cuuint32_t *,
                                  const cuuint32_t *, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

int encode_tensor_map_bf16(CUtensorMap *map, const void *base, int rank, const uint64_t *dims,
                           const uint64_t *strides, const uint32_t *box) {
  static std::once_flag once;
  static EncodeTiledFn fn = nullptr;
  static cudaError_t fetch_err = cudaSuccess;
  std::call_once(once, [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    fetch_err = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                                 cudaEnableDefault, &q);
    if (fetch_err == cudaSuccess && q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  if (!fn)
    return fail(SF_ERR_CUDA, "cuTensorMapEncodeTiled unavailable (%s)",
                cudaGetErrorString(fetch_err));
  if (rank < 1 || rank > 5) return fail(SF_ERR_INVALID_ARG, "tensor map rank %d", rank);
  cuuint64_t d[5], st[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    d[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
    if (i + 1 < rank) st[i] = strides[i];
  }
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void *>(base), d, st, bx,
                  es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SF_ERR_CUDA, "cuTensorMapEncodeTiled failed (CUresult %d)", (int)r);
  return SF_OK;
}

// Self-test of the bounded wait every kernel uses: one thread waits for
// phase 0 of an mbarrier that nobody arrives at.  The wait gives up after
// kWaitBudgetNs and the kernel records SF_DEVICE_TIMEOUT, as the kernels do
// when a copy or a peer never completes.
__global__ void selftest_wait_kernel(uint32_t *status) {
  __shared__ alignas(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(smem_addr(&bar), 1);
    fence_mbar_init();
    if (!mbar_wait_bounded(smem_addr(&bar), 0u)) set_status(status, SF_DEVICE_TIMEOUT);
  }
}

}  // namespace sf

extern "C" {

const char *sf_status_string(int status) {
  switch (status) {
    case SF_OK: return "SF_OK";
    case SF_ERR_INVALID_ARG: return "SF_ERR_INVALID_ARG";
    case SF_ERR_UNSUPPORTED: return "SF_ERR_UNSUPPORTED";
    case SF_ERR_CUDA: return "SF_ERR_CUDA";
    case SF_ERR_WORKSPACE: return "SF_ERR_WORKSPACE";
    case SF_ERR_DEVICE_STATUS: return "SF_ERR_DEVICE_STATUS";
    default: return "SF_ERR_UNKNOWN";
  }
}

const char *sf_last_error(void) { return sf::g_last_error; }

int sf_version(void) { return 10000; }

int sf_workspace_init(void *workspace, size_t bytes, cudaStream_t stream) {
  if (!workspace || bytes == 0) return sf::fail(SF_ERR_INVALID_ARG, "workspace is NULL or empty");
  cudaError_t e = cudaMemsetAsync(workspace, 0, bytes, stream);
  if (e != cudaSuccess) return sf::fail(SF_ERR_CUDA, "cudaMemsetAsync: %s", cudaGetErrorString(e));
  return SF_OK;
}

int sf_selftest_bounded_wait(void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  sf::clear_error();
  if (!workspace || workspace_bytes < sizeof(uint32_t) || !sf::aligned(workspace, 4))
    return sf::fail(SF_ERR_WORKSPACE, "workspace must hold a 4-byte aligned status word");
  sf::selftest_wait_kernel<<<1, 32, 0, stream>>>(static_cast<uint32_t *>(workspace));
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return sf::fail(SF_ERR_CUDA, "self-test launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

int sf_read_device_status(const void *workspace, uint32_t *status_out) {
  if (!workspace || !status_out) return sf::fail(SF_ERR_INVALID_ARG, "NULL argument");
  cudaError_t e = cudaDeviceSynchronize();
  if (e == cudaSuccess) e = cudaMemcpy(status_out, workspace, sizeof(uint32_t), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return sf::fail(SF_ERR_CUDA, "status read-back: %s", cudaGetErrorString(e));
  return SF_OK;
}

}  // extern "C"
