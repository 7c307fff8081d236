// accept.cu -- fused speculative acceptance for sm_103a.
//
// The verification rule (Sec. 3.1; Sec. 3.3 "the standard token-wise
// acceptance-rejection rule"): with p_i = softmax(target_logits_i / tau) and
// the draft distribution q_i, draft T'_{i+1} = x_i is accepted iff
// u_i * q_i(x_i) < p_i(x_i) (probability min(1, p/q)); decisions are taken in
// order up to the first rejection j; the token at position j is drawn by
// inverse CDF from norm(max(0, p_j - q_j)), or from the bonus row p_k when all
// k drafts were accepted.  tau <= 0 is greedy decoding (Sec. 4.2): accept iff
// x_i is the argmax of row i, and emit the argmax of row j.
//
// GB300 design.  The whole cost is streaming the (k+1) x V fp32 logits once
// (plus one row of q for the draw), so both kernels are coalesced 128-bit
// streaming reductions spread over many CTAs, with no tensor cores:
//  * accept_stats_kernel, grid (chunks, k+1, B): each CTA reduces a chunk of
//    one row to (max, first argmax, sum exp((x - max)/tau)) with the chunk
//    held in registers; the last CTA of a row (atomic ticket, nobody waits)
//    combines the chunks in fp64; the last row of a sequence to finish takes
//    the k accept/reject decisions in fp64 and writes the accepted tokens.
//  * accept_draw_kernel, grid (chunks, B): for sampled sequences, each CTA
//    sums the residual (or bonus) mass of a chunk of row j; the last CTA of
//    the sequence locates the chunk holding u_k * S with an fp64 scan over
//    the chunk sums, then scans that chunk element by element in ascending
//    token order.
// Per-element arithmetic is fp32 (expf, explicitly rounded products and
// differences, identical in both passes); every sum above one thread is fp64.
#include <cmath>

#include "sf_device.cuh"
#include "sf_host.h"

namespace sf {

constexpr int kAccThreads = 256;
constexpr int kMaxPerThread = 32;                       // elements held per thread
constexpr int kMaxChunk = kAccThreads * kMaxPerThread;  // 8192 elements per CTA

struct RowStat {   // one (sequence, row) or one chunk of it
  float m;         // largest raw logit
  int arg;         // its first index
  double S;        // sum of exp((x - m) / tau); 0 for greedy rows
};

struct SeqState {
  int j;           // first rejected position (k if none)
  int pad[3];
};

struct DrawPart {
  double sum_r;    // residual (or bonus) mass of the chunk
  double sum_p;    // target mass of the chunk (fallback when the residual is 0)
  int last_r;      // last index with r > 0 (-1 if none)
  int last_p;      // last index with p > 0 (-1 if none)
  int pad[2];
};

struct AccParams {
  const float *logits;   // [B][k+1][V]
  const float *q;        // [B][k][V]
  const int32_t *tokens; // [B][k]
  const float *u;        // [B][k+1]
  const float *tau;      // [B]
  int32_t *num_accepted; // [B]
  int32_t *out_tokens;   // [B][k+1]
  float *ratio;          // [B][k] or null
  uint32_t *status;
  uint32_t *row_tickets; // [B][k+1]
  uint32_t *seq_tickets; // [B]
  uint32_t *draw_tickets;// [B]
  RowStat *rows;         // [B][k+1]
  RowStat *chunks;       // [B][k+1][C1]
  SeqState *seqs;        // [B]
  DrawPart *parts;       // [B][C2]
  int B, k, V;
  int C1, CV1;           // stats chunks per row, elements per chunk
  int C2, CV2;           // draw chunks per row, elements per chunk
  int vec4;              // rows are 16-byte aligned and V % 4 == 0
};

// (value, index) order for argmax: larger value first, then lower index.
__device__ __forceinline__ bool better(float v, int i, float bv, int bi) {
  return v > bv || (v == bv && i < bi);
}

__device__ __forceinline__ float exp_scaled(float x, float m, float tau) {
  const float d = __fsub_rn(x, m);
  return expf(tau == 1.0f ? d : __fdiv_rn(d, tau));
}

// Residual (j < k) or bonus (j == k) mass of one token and its target mass.
__device__ __forceinline__ void draw_terms(float x, float qx, bool residual, float m, float tau,
                                           float invS, float &r, float &pz) {
  pz = __fmul_rn(exp_scaled(x, m, tau), invS);
  r = residual ? fmaxf(__fsub_rn(pz, qx), 0.0f) : pz;
}

template <typename T>
__device__ __forceinline__ T warp_sum(T v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Block-wide sum in fp64 (deterministic tree order).
__device__ double block_sum(double v, double *s_buf) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  v = warp_sum(v);
  __syncthreads();
  if (lane == 0) s_buf[warp] = v;
  __syncthreads();
  if (warp == 0) {
    v = lane < kAccThreads / 32 ? s_buf[lane] : 0.0;
    v = warp_sum(v);
    if (lane == 0) s_buf[0] = v;
  }
  __syncthreads();
  return s_buf[0];
}

__device__ void block_argmax(float &v, int &i, float *s_v, int *s_i) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float ov = __shfl_xor_sync(0xffffffffu, v, o);
    const int oi = __shfl_xor_sync(0xffffffffu, i, o);
    if (better(ov, oi, v, i)) { v = ov; i = oi; }
  }
  __syncthreads();
  if (lane == 0) { s_v[warp] = v; s_i[warp] = i; }
  __syncthreads();
  if (warp == 0) {
    v = lane < kAccThreads / 32 ? s_v[lane] : -INFINITY;
    i = lane < kAccThreads / 32 ? s_i[lane] : 0x7fffffff;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, v, o);
      const int oi = __shfl_xor_sync(0xffffffffu, i, o);
      if (better(ov, oi, v, i)) { v = ov; i = oi; }
    }
    if (lane == 0) { s_v[0] = v; s_i[0] = i; }
  }
  __syncthreads();
  v = s_v[0];
  i = s_i[0];
}

__global__ void __launch_bounds__(kAccThreads)
accept_stats_kernel(const __grid_constant__ AccParams p) {
  __shared__ double s_d[32];
  __shared__ float s_v[32];
  __shared__ int s_i[32];
  __shared__ int s_flag;
  __shared__ int s_acc[SF_MAX_DRAFT];

  const int c = blockIdx.x, r = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x;
  const int k = p.k, V = p.V;
  const float tau = p.tau[b];
  const bool greedy = !(tau > 0.0f);
  const float *row = p.logits + ((size_t)b * (k + 1) + r) * V;
  const int c0 = c * p.CV1;
  const int c1 = min(V, c0 + p.CV1);

  // ---- chunk reduction: max / first argmax, then sum of exp ----
  float vals[kMaxPerThread];
  int n = 0;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  if (p.vec4) {
    const float4 *row4 = reinterpret_cast<const float4 *>(row);
#pragma unroll
    for (int t = 0; t < kMaxPerThread / 4; ++t) {
      const int e = c0 + 4 * (tid + t * kAccThreads);
      if (e < c1) {
        const float4 x = row4[e / 4];
        vals[4 * t + 0] = x.x; vals[4 * t + 1] = x.y; vals[4 * t + 2] = x.z; vals[4 * t + 3] = x.w;
        if (better(x.x, e, bv, bi)) { bv = x.x; bi = e; }
        if (better(x.y, e + 1, bv, bi)) { bv = x.y; bi = e + 1; }
        if (better(x.z, e + 2, bv, bi)) { bv = x.z; bi = e + 2; }
        if (better(x.w, e + 3, bv, bi)) { bv = x.w; bi = e + 3; }
        n = 4 * t + 4;
      }
    }
  } else {
#pragma unroll
    for (int t = 0; t < kMaxPerThread; ++t) {
      const int e = c0 + tid + t * kAccThreads;
      if (e < c1) {
        const float x = row[e];
        vals[t] = x;
        if (better(x, e, bv, bi)) { bv = x; bi = e; }
        n = t + 1;
      }
    }
  }
  block_argmax(bv, bi, s_v, s_i);
  double S = 0.0;
  if (!greedy && bv != -INFINITY) {
    float acc = 0.f;
#pragma unroll
    for (int t = 0; t < kMaxPerThread; ++t)
      if (t < n) acc += exp_scaled(vals[t], bv, tau);
    S = block_sum((double)acc, s_d);
  }
  const size_t rowid = (size_t)b * (k + 1) + r;
  if (tid == 0) p.chunks[rowid * p.C1 + c] = RowStat{bv, bi, S};

  // ---- the last chunk of the row combines the row ----
  __threadfence();
  __syncthreads();
  if (tid == 0) s_flag = (atomicAdd(p.row_tickets + rowid, 1u) == (unsigned)(p.C1 - 1));
  __syncthreads();
  if (!s_flag) return;
  __threadfence();
  float mv = -INFINITY;
  int mi = 0x7fffffff;
  for (int cc = tid; cc < p.C1; cc += kAccThreads) {
    const float cm = __ldcg(&p.chunks[rowid * p.C1 + cc].m);
    const int ca = __ldcg(&p.chunks[rowid * p.C1 + cc].arg);
    if (better(cm, ca, mv, mi)) { mv = cm; mi = ca; }
  }
  block_argmax(mv, mi, s_v, s_i);
  double Srow = 0.0;
  if (!greedy && mv != -INFINITY) {
    double part = 0.0;
    for (int cc = tid; cc < p.C1; cc += kAccThreads) {
      const float cm = __ldcg(&p.chunks[rowid * p.C1 + cc].m);
      const double cS = __ldcg(&p.chunks[rowid * p.C1 + cc].S);
      if (cS > 0.0) part += cS * exp(((double)cm - (double)mv) / (double)tau);
    }
    Srow = block_sum(part, s_d);
  }
  if (tid == 0) {
    p.rows[rowid] = RowStat{mv, mi, Srow};
    p.row_tickets[rowid] = 0u;
  }

  // ---- the last row of the sequence takes the k decisions ----
  __threadfence();
  __syncthreads();
  if (tid == 0) s_flag = (atomicAdd(p.seq_tickets + b, 1u) == (unsigned)k);
  __syncthreads();
  if (!s_flag) return;
  __threadfence();
  if (tid < k) {
    const int i = tid;
    const int x = p.tokens[(size_t)b * k + i];
    const RowStat rs = {__ldcg(&p.rows[(size_t)b * (k + 1) + i].m),
                        __ldcg(&p.rows[(size_t)b * (k + 1) + i].arg),
                        __ldcg(&p.rows[(size_t)b * (k + 1) + i].S)};
    int acc = 0;
    float ratio = 0.f;
    if (x < 0 || x >= V) {
      set_status(p.status, SF_DEVICE_BAD_TOKEN);  // treated as a rejection
    } else if (greedy) {
      acc = (x == rs.arg);
      ratio = acc ? 1.f : 0.f;
    } else {
      const double lx = (double)__ldcg(p.logits + ((size_t)b * (k + 1) + i) * V + x);
      const double px = exp((lx - (double)rs.m) / (double)tau) / rs.S;
      const double qx = (double)p.q[((size_t)b * k + i) * V + x];
      const double ux = (double)p.u[(size_t)b * (k + 1) + i];
      acc = (ux * qx < px);
      ratio = qx > 0.0 ? (float)fmin(1.0, px / qx) : 1.f;
    }
    s_acc[i] = acc;
    if (p.ratio) p.ratio[(size_t)b * k + i] = ratio;
  }
  __syncthreads();
  if (tid == 0) {
    int j = k;
    for (int i = 0; i < k; ++i)
      if (!s_acc[i]) { j = i; break; }
    p.num_accepted[b] = j;
    int32_t *ob = p.out_tokens + (size_t)b * (k + 1);
    for (int i = 0; i <= k; ++i) ob[i] = i < j ? p.tokens[(size_t)b * k + i] : -1;
    if (greedy) ob[j] = __ldcg(&p.rows[(size_t)b * (k + 1) + j].arg);
    p.seqs[b].j = j;
    p.seq_tickets[b] = 0u;
  }
}

__global__ void __launch_bounds__(kAccThreads)
accept_draw_kernel(const __grid_constant__ AccParams p) {
  __shared__ double s_d[32];
  __shared__ double s_scan[kAccThreads];
  __shared__ float s_r[kMaxChunk];
  __shared__ int s_flag;
  __shared__ int s_token;
  __shared__ int s_chunk;
  __shared__ double s_base;

  const int c = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x;
  const int k = p.k, V = p.V;
  const float tau = p.tau[b];
  if (!(tau > 0.0f)) return;  // greedy sequences are complete
  const int j = p.seqs[b].j;
  const bool residual = j < k;
  const RowStat rs = p.rows[(size_t)b * (k + 1) + j];
  const float invS = (float)(1.0 / rs.S);
  const float *row = p.logits + ((size_t)b * (k + 1) + j) * V;
  const float *qrow = residual ? p.q + ((size_t)b * k + j) * V : nullptr;
  const int c0 = c * p.CV2;
  const int c1 = min(V, c0 + p.CV2);

  // ---- chunk sums of r and p (fp32 per thread, fp64 across threads) ----
  float sr = 0.f, sp = 0.f;
  int lr = -1, lp = -1;
  if (p.vec4) {
    for (int e = c0 + 4 * tid; e < c1; e += 4 * kAccThreads) {
      const float4 x = *reinterpret_cast<const float4 *>(row + e);
      const float4 qv = residual ? __ldcs(reinterpret_cast<const float4 *>(qrow + e))
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
      const float xs[4] = {x.x, x.y, x.z, x.w};
      const float qs[4] = {qv.x, qv.y, qv.z, qv.w};
#pragma unroll
      for (int t = 0; t < 4; ++t) {
        float rr, pz;
        draw_terms(xs[t], qs[t], residual, rs.m, tau, invS, rr, pz);
        sr += rr;
        sp += pz;
        if (rr > 0.f) lr = e + t;
        if (pz > 0.f) lp = e + t;
      }
    }
  } else {
    for (int e = c0 + tid; e < c1; e += kAccThreads) {
      float rr, pz;
      draw_terms(row[e], residual ? qrow[e] : 0.f, residual, rs.m, tau, invS, rr, pz);
      sr += rr;
      sp += pz;
      if (rr > 0.f) lr = e;
      if (pz > 0.f) lp = e;
    }
  }
  const double Sr = block_sum((double)sr, s_d);
  const double Sp = block_sum((double)sp, s_d);
  {
    int v = lr;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = max(v, __shfl_xor_sync(0xffffffffu, v, o));
    int w = lp;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) w = max(w, __shfl_xor_sync(0xffffffffu, w, o));
    if (tid == 0) { s_flag = -1; s_token = -1; }
    __syncthreads();
    if ((tid & 31) == 0) { atomicMax(&s_flag, v); atomicMax(&s_token, w); }
    __syncthreads();
    if (tid == 0) p.parts[(size_t)b * p.C2 + c] = DrawPart{Sr, Sp, s_flag, s_token, {0, 0}};
  }

  // ---- the last chunk of the sequence draws the token ----
  __threadfence();
  __syncthreads();
  if (tid == 0) s_flag = (atomicAdd(p.draw_tickets + b, 1u) == (unsigned)(p.C2 - 1));
  __syncthreads();
  if (!s_flag) return;
  __threadfence();

  const DrawPart *parts = p.parts + (size_t)b * p.C2;
  double total = 0.0;
  {
    double pr = 0.0;
    for (int cc = tid; cc < p.C2; cc += kAccThreads) pr += __ldcg(&parts[cc].sum_r);
    total = block_sum(pr, s_d);
  }
  const bool use_p = !(total > 0.0);  // residual with no mass (rounding only)
  if (use_p) {
    double pp = 0.0;
    for (int cc = tid; cc < p.C2; cc += kAccThreads) pp += __ldcg(&parts[cc].sum_p);
    total = block_sum(pp, s_d);
  }
  const double target = (double)p.u[(size_t)b * (k + 1) + k] * total;

  // chunk holding the target: inclusive fp64 scan over chunk sums, in order
  if (tid == 0) { s_chunk = 0x7fffffff; s_base = 0.0; }
  double carry = 0.0;
  for (int base = 0; base < p.C2; base += kAccThreads) {
    const int cc = base + tid;
    double v = 0.0;
    if (cc < p.C2) v = use_p ? __ldcg(&parts[cc].sum_p) : __ldcg(&parts[cc].sum_r);
    __syncthreads();
    s_scan[tid] = v;
    __syncthreads();
    for (int o = 1; o < kAccThreads; o <<= 1) {
      const double add = tid >= o ? s_scan[tid - o] : 0.0;
      __syncthreads();
      s_scan[tid] += add;
      __syncthreads();
    }
    // excl of chunk cc is bit-identical to incl of chunk cc-1, so the chunk
    // intervals [excl, incl) tile [0, total) without gaps or overlaps
    const double incl = carry + s_scan[tid];
    const double excl = carry + (tid > 0 ? s_scan[tid - 1] : 0.0);
    if (cc < p.C2 && v > 0.0 && target < incl && target >= excl) atomicMin(&s_chunk, cc);
    __syncthreads();
    if (s_chunk == cc && cc < p.C2) s_base = excl;
    carry += s_scan[kAccThreads - 1];
    __syncthreads();
    if (s_chunk != 0x7fffffff) break;
  }
  __syncthreads();
  int token = -1;
  if (s_chunk == 0x7fffffff) {
    // u*S at or past the total (rounding): the last token with positive mass
    int last = -1;
    for (int cc = tid; cc < p.C2; cc += kAccThreads)
      last = max(last, use_p ? __ldcg(&parts[cc].last_p) : __ldcg(&parts[cc].last_r));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, o));
    if (tid == 0) s_token = -1;
    __syncthreads();
    if ((tid & 31) == 0) atomicMax(&s_token, last);
    __syncthreads();
    token = s_token;
  } else {
    // scan the chunk in ascending token order: thread t owns a contiguous run
    const int cc = s_chunk;
    const int e0 = cc * p.CV2, e1 = min(V, e0 + p.CV2);
    const int len = e1 - e0;
    for (int e = tid; e < len; e += kAccThreads) {
      float rr, pz;
      draw_terms(row[e0 + e], residual ? qrow[e0 + e] : 0.f, residual, rs.m, tau, invS, rr, pz);
      s_r[e] = use_p ? pz : rr;
    }
    __syncthreads();
    const int per = (len + kAccThreads - 1) / kAccThreads;
    const int a0 = tid * per, a1 = min(len, a0 + per);
    double mine = 0.0;
    for (int e = a0; e < a1; ++e) mine += (double)s_r[e];
    s_scan[tid] = mine;
    __syncthreads();
    for (int o = 1; o < kAccThreads; o <<= 1) {
      const double add = tid >= o ? s_scan[tid - o] : 0.0;
      __syncthreads();
      s_scan[tid] += add;
      __syncthreads();
    }
    double cum = s_base + (tid > 0 ? s_scan[tid - 1] : 0.0);
    if (tid == 0) s_token = 0x7fffffff;
    __syncthreads();
    for (int e = a0; e < a1; ++e) {
      cum += (double)s_r[e];
      if (target < cum) { atomicMin(&s_token, e0 + e); break; }
    }
    __syncthreads();
    token = s_token;
    if (token == 0x7fffffff) {
      // rounding put the target past this chunk's own sum: its last positive token
      token = use_p ? __ldcg(&parts[cc].last_p) : __ldcg(&parts[cc].last_r);
    }
  }
  if (tid == 0) {
    p.out_tokens[(size_t)b * (k + 1) + j] = token;
    p.draw_tickets[b] = 0u;
  }
}

// --------------------------------------------------------------------------
// host side
// --------------------------------------------------------------------------
struct AccPlan {
  int C1, CV1, C2, CV2;
};

struct AccLayout {
  size_t row_tickets, seq_tickets, draw_tickets, rows, chunks, seqs, parts, total;
};

static int chunking(long long target_ctas, int V, int rows, int *C, int *CV) {
  const long long min_chunks = (V + kMaxChunk - 1) / kMaxChunk;
  const long long max_chunks = V > 1024 ? (V + 1023) / 1024 : 1;
  long long want = (target_ctas + rows - 1) / rows;
  if (want < min_chunks) want = min_chunks;
  if (want > max_chunks) want = max_chunks;
  if (want < 1) want = 1;
  long long cv = (V + want - 1) / want;
  cv = (cv + 3) / 4 * 4;
  if (cv > kMaxChunk) cv = kMaxChunk;
  *CV = static_cast<int>(cv);
  *C = static_cast<int>((V + cv - 1) / cv);
  return SF_OK;
}

static int plan_accept(int B, int k, int V, AccPlan *plan) {
  DeviceInfo dev;
  int st = current_device(&dev);
  if (st != SF_OK) return st;
  const long long target = 4LL * dev.sm_count;  // ~ 4 CTAs of 256 threads per SM
  chunking(target, V, B * (k + 1), &plan->C1, &plan->CV1);
  chunking(target, V, B, &plan->C2, &plan->CV2);
  return SF_OK;
}

static AccLayout acc_layout(int B, int k, const AccPlan &pl) {
  AccLayout l;
  const size_t R = (size_t)B * (k + 1);
  size_t off = 256;
  l.row_tickets = off; off = round_up(off + 4 * R, 256);
  l.seq_tickets = off; off = round_up(off + 4 * (size_t)B, 256);
  l.draw_tickets = off; off = round_up(off + 4 * (size_t)B, 256);
  l.rows = off; off = round_up(off + sizeof(RowStat) * R, 256);
  l.chunks = off; off = round_up(off + sizeof(RowStat) * R * pl.C1, 256);
  l.seqs = off; off = round_up(off + sizeof(SeqState) * (size_t)B, 256);
  l.parts = off; off = round_up(off + sizeof(DrawPart) * (size_t)B * pl.C2, 256);
  l.total = off;
  return l;
}

static int check_accept_shapes(int B, int k, int V) {
  if (B < 1 || B > SF_MAX_BATCH) return fail(SF_ERR_INVALID_ARG, "B=%d outside [1, %d]", B, SF_MAX_BATCH);
  if (k < 1 || k > SF_MAX_DRAFT) return fail(SF_ERR_INVALID_ARG, "k=%d outside [1, %d]", k, SF_MAX_DRAFT);
  if (V < 2 || (long long)V * (k + 1) >= (1LL << 31))
    return fail(SF_ERR_INVALID_ARG, "V=%d outside [2, 2^31/(k+1))", V);
  return SF_OK;
}

}  // namespace sf

extern "C" {

size_t sf_accept_workspace_size(int B, int k, int V) {
  if (sf::check_accept_shapes(B, k, V) != SF_OK) return 0;
  sf::AccPlan plan;
  if (sf::plan_accept(B, k, V, &plan) != SF_OK) return 0;
  return sf::acc_layout(B, k, plan).total;
}

int sf_accept(const float *target_logits, const float *draft_probs,
              const int32_t *draft_tokens, const float *uniforms, const float *temperature,
              int B, int k, int V, int32_t *num_accepted, int32_t *out_tokens,
              float *accept_ratio, void *workspace, size_t workspace_bytes,
              cudaStream_t stream) {
  using namespace sf;
  clear_error();
  int st = check_accept_shapes(B, k, V);
  if (st != SF_OK) return st;
  if (!target_logits || !draft_probs || !draft_tokens || !uniforms || !temperature ||
      !num_accepted || !out_tokens)
    return fail(SF_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!aligned(target_logits, 4) || !aligned(draft_probs, 4) || !aligned(draft_tokens, 4) ||
      !aligned(uniforms, 4) || !aligned(temperature, 4) || !aligned(num_accepted, 4) ||
      !aligned(out_tokens, 4) || (accept_ratio && !aligned(accept_ratio, 4)))
    return fail(SF_ERR_INVALID_ARG, "buffers must be 4-byte aligned");
  if (!workspace || !aligned(workspace, 256))
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL and 256-byte aligned");
  AccPlan plan;
  st = plan_accept(B, k, V, &plan);
  if (st != SF_OK) return st;
  const AccLayout lay = acc_layout(B, k, plan);
  if (workspace_bytes < lay.total)
    return fail(SF_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, lay.total);

  uint8_t *ws = static_cast<uint8_t *>(workspace);
  AccParams prm;
  prm.logits = target_logits;
  prm.q = draft_probs;
  prm.tokens = draft_tokens;
  prm.u = uniforms;
  prm.tau = temperature;
  prm.num_accepted = num_accepted;
  prm.out_tokens = out_tokens;
  prm.ratio = accept_ratio;
  prm.status = reinterpret_cast<uint32_t *>(ws);
  prm.row_tickets = reinterpret_cast<uint32_t *>(ws + lay.row_tickets);
  prm.seq_tickets = reinterpret_cast<uint32_t *>(ws + lay.seq_tickets);
  prm.draw_tickets = reinterpret_cast<uint32_t *>(ws + lay.draw_tickets);
  prm.rows = reinterpret_cast<RowStat *>(ws + lay.rows);
  prm.chunks = reinterpret_cast<RowStat *>(ws + lay.chunks);
  prm.seqs = reinterpret_cast<SeqState *>(ws + lay.seqs);
  prm.parts = reinterpret_cast<DrawPart *>(ws + lay.parts);
  prm.B = B;
  prm.k = k;
  prm.V = V;
  prm.C1 = plan.C1;
  prm.CV1 = plan.CV1;
  prm.C2 = plan.C2;
  prm.CV2 = plan.CV2;
  prm.vec4 = (V % 4 == 0) && aligned(target_logits, 16) && aligned(draft_probs, 16);

  accept_stats_kernel<<<dim3(plan.C1, k + 1, B), kAccThreads, 0, stream>>>(prm);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "accept stats launch: %s", cudaGetErrorString(e));
  accept_draw_kernel<<<dim3(plan.C2, B), kAccThreads, 0, stream>>>(prm);
  e = cudaGetLastError();
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "accept draw launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

}  // extern "C"
