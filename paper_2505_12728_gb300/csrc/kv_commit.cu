// kv_commit.cu -- paged-cache bookkeeping after acceptance (Sec. 3.1: the
// accepted candidates join the context and decoding continues from the first
// rejected position; Sec. 3.3: the next draft block starts from the emitted
// token).  For each sequence the first min(a + 1, n_q) verified rows stay,
// seq_lens is prepared for the next n_q_next rows, and the block table maps
// exactly the pages those need, through a stack of free pages.
//
// GB300 design: the work is a few integers per sequence, so the whole batch
// (at most 1024 sequences) is one CTA with one thread per sequence.  Block
// scans give every sequence its offsets in the stack, so the result does not
// depend on thread timing (no atomics): surplus pages are pushed in sequence
// order, a barrier, then missing pages are taken from the topmost entries.
// All or nothing: invalid sequences or a page shortage set a status bit and
// leave every array unchanged.  Latency-bound: one launch, two dependent
// global round trips.
#include <climits>

#include "sf_device.cuh"
#include "sf_host.h"

namespace sf {

constexpr int kCommitThreads = SF_MAX_BATCH;  // one thread per sequence
constexpr int kPageTokensCommit = SF_PAGE_SIZE;

struct CommitParams {
  int32_t *seq_lens;
  int32_t *block_table;
  int32_t *free_pages;
  int32_t *free_count;
  const int32_t *num_accepted;
  uint32_t *status;
  int B, n_q, n_q_next, max_pages, capacity;
};

// Block-wide exclusive scan of one int per thread (blockDim.x threads);
// returns the exclusive prefix and writes the total to *total.
__device__ __forceinline__ int block_exclusive_scan(int v, int *s_warp, int *total) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = (blockDim.x + 31) >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int x = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += x;
  }
  if (lane == 31) s_warp[warp] = incl;
  __syncthreads();
  int off = 0, sum = 0;
  for (int w = 0; w < nwarps; ++w) {
    if (w < warp) off += s_warp[w];
    sum += s_warp[w];
  }
  __syncthreads();  // s_warp may be reused by the next scan
  *total = sum;
  return off + incl - v;
}

__global__ void __launch_bounds__(kCommitThreads) kv_commit_kernel(const CommitParams p) {
  __shared__ int s_warp[kCommitThreads / 32];
  const int b = threadIdx.x;
  int push = 0, take = 0, bad = 0, had = 0, need = 0, next_len = 0;
  if (b < p.B) {
    const int T = p.seq_lens[b], a = p.num_accepted[b];
    if (T < p.n_q || a < 0) {
      bad = 1;
    } else {
      const int keep = a + 1 < p.n_q ? a + 1 : p.n_q;
      const long long nl = (long long)(T - p.n_q) + keep + p.n_q_next;
      had = (T + kPageTokensCommit - 1) / kPageTokensCommit;
      const long long nd = (nl + kPageTokensCommit - 1) / kPageTokensCommit;
      if (nd > p.max_pages || had > p.max_pages) {
        bad = 1;
      } else {
        need = static_cast<int>(nd);
        next_len = static_cast<int>(nl);
        if (need < had) push = had - need;
        else take = need - had;
      }
    }
  }
  int any_bad = 0, pushed = 0, taken = 0;
  (void)block_exclusive_scan(bad, s_warp, &any_bad);
  const int push_off = block_exclusive_scan(push, s_warp, &pushed);
  const int take_off = block_exclusive_scan(take, s_warp, &taken);
  if (any_bad) {
    if (b == 0) set_status(p.status, SF_DEVICE_BAD_SEQLEN);
    return;
  }
  const int fc0 = *p.free_count;
  const long long top = (long long)fc0 + pushed;
  if (fc0 < 0 || top > p.capacity || taken > top) {
    if (b == 0) set_status(p.status, SF_DEVICE_OUT_OF_PAGES);
    return;
  }
  int32_t *row = p.block_table + (size_t)(b < p.B ? b : 0) * p.max_pages;
  // 1. surplus pages onto the stack (sequence order, ascending logical page)
  for (int j = 0; j < push; ++j) {
    p.free_pages[fc0 + push_off + j] = row[need + j];
    row[need + j] = -1;
  }
  __syncthreads();  // every push is visible before any take
  // 2. missing pages from the topmost `taken` entries, bottom-up
  const int base = static_cast<int>(top) - taken;
  for (int j = 0; j < take; ++j) row[had + j] = p.free_pages[base + take_off + j];
  if (b < p.B) p.seq_lens[b] = next_len;
  if (b == 0) *p.free_count = base;
}

}  // namespace sf

extern "C" {

size_t sf_kv_commit_workspace_size(void) { return 256; }

int sf_kv_commit(int32_t *seq_lens, int32_t *block_table, int32_t *free_pages,
                 int32_t *free_count, const int32_t *num_accepted, int B, int n_q, int n_q_next,
                 int max_pages_per_seq, int page_size, int capacity, void *workspace,
                 size_t workspace_bytes, cudaStream_t stream) {
  using namespace sf;
  clear_error();
  if (B < 1 || B > SF_MAX_BATCH) return fail(SF_ERR_INVALID_ARG, "B=%d outside [1, %d]", B, SF_MAX_BATCH);
  if (n_q < 1 || n_q > SF_MAX_QUERY_ROWS || n_q_next < 1 || n_q_next > SF_MAX_QUERY_ROWS)
    return fail(SF_ERR_INVALID_ARG, "n_q=%d, n_q_next=%d outside [1, %d]", n_q, n_q_next,
                SF_MAX_QUERY_ROWS);
  if (page_size != SF_PAGE_SIZE) return fail(SF_ERR_UNSUPPORTED, "page_size=%d (built: 16)", page_size);
  if (max_pages_per_seq < 1 || (long long)max_pages_per_seq * page_size > (1LL << 30))
    return fail(SF_ERR_INVALID_ARG, "max_pages_per_seq=%d", max_pages_per_seq);
  if (capacity < 0) return fail(SF_ERR_INVALID_ARG, "capacity=%d", capacity);
  if (!seq_lens || !block_table || !free_pages || !free_count || !num_accepted)
    return fail(SF_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!aligned(seq_lens, 4) || !aligned(block_table, 4) || !aligned(free_pages, 4) ||
      !aligned(free_count, 4) || !aligned(num_accepted, 4))
    return fail(SF_ERR_INVALID_ARG, "int32 arrays must be 4-byte aligned");
  if (!workspace || !aligned(workspace, 256))
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL and 256-byte aligned");
  if (workspace_bytes < sf_kv_commit_workspace_size())
    return fail(SF_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes,
                sf_kv_commit_workspace_size());
  CommitParams prm;
  prm.seq_lens = seq_lens;
  prm.block_table = block_table;
  prm.free_pages = free_pages;
  prm.free_count = free_count;
  prm.num_accepted = num_accepted;
  prm.status = static_cast<uint32_t *>(workspace);
  prm.B = B;
  prm.n_q = n_q;
  prm.n_q_next = n_q_next;
  prm.max_pages = max_pages_per_seq;
  prm.capacity = capacity;
  const int threads = (B + 31) / 32 * 32;
  kv_commit_kernel<<<1, threads, 0, stream>>>(prm);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "kv commit launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

}  // extern "C"
