// accept.cu -- fused speculative acceptance for sm_103a.
//
// The verification rule (Sec. 3.1; Sec. 3.3 names it the usual token-by-token
// accept/reject rule of speculative sampling): with
// p_i = softmax(target_logits_i / tau) and
// the draft distribution q_i, draft T'_{i+1} = x_i is accepted iff
// u_i * q_i(x_i) < p_i(x_i) (probability min(1, p/q)); decisions are taken in
// order up to the first rejection j; the token at position j is drawn by
// inverse CDF from norm(max(0, p_j - q_j)), or from the bonus row p_k when all
// k drafts were accepted.  tau <= 0 is greedy decoding (Sec. 4.2): accept iff
// x_i is the argmax of row i, and emit the argmax of row j.
//
// GB300 design.  The whole cost is streaming the (k+1) x V fp32 logits once
// (plus one row of q for the draw), so every kernel is a coalesced 128-bit
// streaming reduction spread over many CTAs, with no tensor cores, and the
// critical path is a short chain of memory round trips.  Three launch plans:
//  * V <= 16 x 2048: accept_cluster_kernel, one thread-block cluster per
//    sequence, the phases separated by cluster barriers (below);
//  * larger V: accept_chunks_kernel (every row in 1024-token chunks over
//    all SMs; the warp that completes a row combines its run records, the
//    one that completes a sequence takes the decisions) then
//    accept_draw_kernel (the residual draw in C2 CTAs per sequence over row
//    j, the last CTA of a sequence scanning for u_k * S);
//  * behind the fused LM head, whose projection already left per-CTA row
//    statistics: accept_decide_kernel then accept_draw_kernel.
// Every launch uses programmatic stream serialisation: a kernel is resident
// while the previous one drains and waits for it (griddepcontrol.wait)
// before reading its results.
// Arithmetic: per-element terms are fp32 (2^x by the hardware approximation
// of explicitly rounded differences and products; the decisions' p(x) by
// expf on a float-float difference; a term recomputed within a draw is
// recomputed identically); sums, scans and the accept tests use float-float
// numbers (an unevaluated sum hi + lo of two fp32 values, ~44 significant
// bits) built from exactly rounded fp32 operations, accumulated in a fixed
// order (results are deterministic).
// GB300's fp64 pipe is far too slow for this latency-bound path, and
// float-float gives the accuracy the decisions need.
#include <climits>
#include <cmath>
#include <mutex>

#include "ff_math.cuh"
#include "sf_device.cuh"
#include "sf_host.h"

namespace sf {

constexpr int kAccThreads = kFfThreads;
constexpr int kAccWarps = kFfWarps;
// Rows are cut into segments of 1024 tokens (a warp, eight float4 per lane):
// the unit of the chunk records and of the draw's partial sums.
constexpr int kSegTokens = 1024;


struct alignas(16) RowStat {  // a target row, or a run of its chunks (one 16-byte load)
  float m;         // largest raw logit
  int arg;         // its first index
  ff S;            // sum of exp((x - m) / tau); 0 for greedy rows
};

struct alignas(16) SeqState {  // what the draw needs, in one 16-byte load
  int j;           // first rejected position (k if none)
  float m;         // row j's largest raw logit
  ff S;            // row j's sum of exp((x - m) / tau)
};

struct alignas(16) DrawPart {  // one segment of row j
  ff sum_r;        // residual (or bonus) mass of the segment
  ff sum_p;        // target mass of the segment (fallback when the residual is 0)
  int last_r;      // last index with r > 0 (-1 if none)
  int last_p;      // last index with p > 0 (-1 if none)
  int pad[2];
};

struct AccParams {
  const float *logits;     // [B][k+1][V]
  const float *q;          // [B][k][V]
  const int32_t *tokens;   // [B][k]
  const float *u;          // [B][k+1]
  const float *tau;        // [B]
  int32_t *num_accepted;   // [B]
  int32_t *out_tokens;     // [B][k+1]
  float *ratio;            // [B][k] or null
  uint32_t *status;
  uint32_t *draw_tickets;  // [B]
  uint32_t *row_tickets;   // [B][k+1]: runs of a row whose record is written (chunk kernel)
  uint32_t *seq_tickets;   // [B]: rows of a sequence whose statistics are final
  RowStat *runs;           // [B][k+1][C1]: per row, one record per run of the chunk kernel
  RowStat *rows;           // [B][k+1]
  SeqState *seqs;          // [B]
  DrawPart *parts;         // [B][C1]
  int B, k, V;
  int C1;                  // segments per row: ceil(V / kSegTokens)
  int C2;                  // draw CTAs per row: ceil(C1 / kAccWarps)
  int NW1;                 // warps of the chunk kernel
  int vec4;                // rows are 16-byte aligned and V % 4 == 0
};


// exp((x - m) / tau) for the per-token loops (sums and draw terms); the
// decisions' p(x) use exp_diff_accurate.  Terms are summed four at a time in
// fp32 before each float-float add (a few 2^-24 of the partial).
__device__ __forceinline__ float exp_scaled(float x, float m, float tau) {
  const float d = __fsub_rn(x, m);
  return exp_fast(tau == 1.0f ? d : __fdiv_rn(d, tau));
}

__device__ __forceinline__ float sum4(float a, float b, float c, float d) {
  return __fadd_rn(__fadd_rn(a, b), __fadd_rn(c, d));
}

// Residual (j < k) or bonus (j == k) mass of one token and its target mass.
__device__ __forceinline__ void draw_terms(float x, float qx, bool residual, float m, float tau,
                                           float invS, float &r, float &pz) {
  pz = __fmul_rn(exp_scaled(x, m, tau), invS);
  r = residual ? fmaxf(__fsub_rn(pz, qx), 0.0f) : pz;
}

// The k accept/reject decisions of sequence b and its outputs, from the
// combined rows in shared memory (row rr: max s_rm, first argmax s_rarg,
// float-float sum s_rS, the draft token's logit s_rlx and draft probability
// s_rqx, s_rhx = the token lies in [0, V)).  Called by every thread of the
// block after the rows are visible; thread i < k tests draft i (my_tok,
// my_u), threads <= k write out_tokens; j goes to num_accepted and seqs.
__device__ void decide_sequence(const AccParams &p, int b, bool greedy, float tau, int my_tok,
                                float my_u, const float *s_rm, const int *s_rarg, const ff *s_rS,
                                const float *s_rlx, const float *s_rqx, const int *s_rhx,
                                int *s_acc, bool write = true, int *s_j = nullptr) {
  const int tid = threadIdx.x, k = p.k, V = p.V;
  if (tid < k) {
    const int i = tid, x = my_tok;
    int acc = 0;
    float ratio = 0.f;
    if (x < 0 || x >= V || !s_rhx[i]) {
      if (write) set_status(p.status, SF_DEVICE_BAD_TOKEN);  // treated as a rejection
    } else if (greedy) {
      acc = (x == s_rarg[i]);
      ratio = acc ? 1.f : 0.f;
    } else {
      // p(x) = exp((l_x - m) / tau) / S; accept iff u * q(x) < p(x), with the
      // product u * q kept exactly as float-float
      const float px = ff_div_to_f(exp_diff_accurate(s_rlx[i], s_rm[i], tau), s_rS[i]);
      const float qd = s_rqx[i];
      const float uq = __fmul_rn(my_u, qd);
      const ff uqf = ff{uq, __fmaf_rn(my_u, qd, -uq)};
      acc = ff_lt(uqf, ff_of(px)) ? 1 : 0;
      ratio = qd > 0.f ? fminf(1.f, __fdiv_rn(px, qd)) : 1.f;
    }
    s_acc[i] = acc;
    if (write && p.ratio) p.ratio[(size_t)b * k + i] = ratio;
  }
  __syncthreads();
  if (tid <= k) {
    // every writer finds j in shared memory; thread i writes out_tokens[i]
    int j = k;
    for (int i = 0; i < k; ++i)
      if (!s_acc[i]) { j = i; break; }
    int32_t v = -1;
    if (tid < j) v = my_tok;
    else if (tid == j && greedy) v = s_rarg[j];
    if (write && !(tid == j && !greedy)) p.out_tokens[(size_t)b * (k + 1) + tid] = v;
    if (tid == 0) {
      if (write) {
        p.num_accepted[b] = j;
        p.seqs[b] = SeqState{j, s_rm[j], s_rS[j]};
      }
      if (s_j) *s_j = j;
    }
  }
}

// Single-kernel acceptance for V <= 16 * kClusterMaxSlice: one thread-block
// cluster of cs CTAs per sequence, CTA `rank` owning tokens [rank * slice,
// (rank + 1) * slice) of every row.  Phases, separated by cluster barriers
// (the same number on every path; greedy clusters leave together after the
// decision):
//  1. each warp reduces one row of the CTA's slice to (max, first argmax,
//     float-float sum of exp((x - max)/tau));
//  2. CTA 0 combines the cs records of each row (read through distributed
//     shared memory, in rank order), takes the decisions (decide_sequence)
//     and publishes j and row j's (max, sum);
//  3. sampled sequences: each CTA writes row j's residual (or bonus) terms
//     of its slice to shared memory and their ordered sum;
//  4. every CTA adds the cs slice sums in rank order, finds the slice
//     holding u_k * S, and that CTA scans its terms in ascending order.
constexpr int kClusterMax = 16;
constexpr int kClusterMaxSlice = 2048;   // tokens per CTA: one row slice in a warp's registers
constexpr int kClusterPerThread = kClusterMaxSlice / kAccThreads;  // 8

struct alignas(16) ClusterRec {  // one row of one CTA's slice (one 16-byte remote load)
  float m;
  int arg;
  ff S;
};

struct alignas(16) ClusterDraw {  // row j's terms in one CTA's slice (two 16-byte loads)
  ff sum_r, sum_p;
  int last_r, last_p;
  int pad[2];
};
static_assert(sizeof(ClusterRec) == 16 && sizeof(ClusterDraw) == 32, "record sizes");

__global__ void __launch_bounds__(kAccThreads)
accept_cluster_kernel(const __grid_constant__ AccParams p, int cs, int slice) {
  extern __shared__ float s_terms[];  // [slice]
  __shared__ ClusterRec s_rec[SF_MAX_DRAFT + 1];
  __shared__ ClusterRec s_part[SF_MAX_DRAFT + 1][kAccWarps];  // per-warp partials of phase 1
  __shared__ ClusterDraw s_draw;
  __shared__ int s_dec_j;
  __shared__ float s_dec_m;
  __shared__ ff s_dec_S;
  __shared__ ff s_d[32];
  __shared__ ff s_scan[kAccWarps + 1];
  __shared__ int s_acc[SF_MAX_DRAFT];
  __shared__ float s_rm[SF_MAX_DRAFT + 1], s_rlx[SF_MAX_DRAFT + 1], s_rqx[SF_MAX_DRAFT + 1];
  __shared__ int s_rarg[SF_MAX_DRAFT + 1], s_rhx[SF_MAX_DRAFT + 1];
  __shared__ ff s_rS[SF_MAX_DRAFT + 1];
  __shared__ int s_i0, s_i1;
  __shared__ ff s_base, s_total;

  grid_dependency_wait();  // logits, q, tokens and the outputs follow the previous kernel
  grid_launch_dependents();
  const int rank = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = p.k, V = p.V;
  const float tau = p.tau[b];
  const bool greedy = !(tau > 0.0f);
  const int x0 = min(V, rank * slice), x1 = min(V, x0 + slice);

  // ---- 1. row statistics of the slice: warp w reduces the w-th eighth of
  // the slice of every row (rows interleaved, short dependency chains), then
  // warp r merges row r's eight partials in warp order ----
  {
    constexpr int kRG = 6;  // rows per pass
    const int sub = kClusterMaxSlice / kAccWarps;  // 256 tokens per warp
    const int w0 = x0 + warp * sub, w1 = min(x1, w0 + sub);
    for (int g = 0; g <= k; g += kRG) {
      float v[kRG][8];
#pragma unroll
      for (int i = 0; i < kRG; ++i) {
        const int r = g + i;
        const float *row = p.logits + ((size_t)b * (k + 1) + (r <= k ? r : k)) * V;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int e = w0 + 4 * (lane + 32 * h);
          float4 x = make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
          if (r <= k) {
            if (p.vec4) {
              if (e < w1) x = *reinterpret_cast<const float4 *>(row + e);
            } else {
              if (e < w1) x.x = row[e];
              if (e + 1 < w1) x.y = row[e + 1];
              if (e + 2 < w1) x.z = row[e + 2];
              if (e + 3 < w1) x.w = row[e + 3];
            }
          }
          v[i][4 * h] = x.x; v[i][4 * h + 1] = x.y; v[i][4 * h + 2] = x.z; v[i][4 * h + 3] = x.w;
        }
      }
#pragma unroll
      for (int i = 0; i < kRG; ++i) {
        float bv = -INFINITY;
        int bi = INT_MAX;
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          const int e = w0 + 4 * (lane + 32 * (t / 4)) + (t % 4);
          if (better(v[i][t], e, bv, bi)) { bv = v[i][t]; bi = e; }
        }
        warp_argmax(bv, bi);
        ff S = ff_of(0.f);
        if (!greedy && bv != -INFINITY) {
          float e[8];
#pragma unroll
          for (int t = 0; t < 8; ++t) e[t] = v[i][t] != -INFINITY ? exp_scaled(v[i][t], bv, tau) : 0.f;
          S = ff_add(ff_of(sum4(e[0], e[1], e[2], e[3])), ff_of(sum4(e[4], e[5], e[6], e[7])));
          S = warp_sum_ff(S);
        }
        if (lane == 0 && g + i <= k) s_part[g + i][warp] = ClusterRec{bv, bi, S};
      }
    }
    __syncthreads();
    for (int r = warp; r <= k; r += kAccWarps) {
      // lane w < 8 holds warp w's partial; merged in warp order
      float cm = -INFINITY;
      int ca = INT_MAX;
      ff cS = ff_of(0.f);
      if (lane < kAccWarps) {
        cm = s_part[r][lane].m;
        ca = s_part[r][lane].arg;
        cS = s_part[r][lane].S;
      }
      float mv = cm;
      int mi = ca;
      warp_argmax(mv, mi);
      ff Sr = ff_of(0.f);
      if (!greedy && mv != -INFINITY) {
        for (int w = 0; w < kAccWarps; ++w) {
          const float wm = __shfl_sync(0xffffffffu, cm, w);
          const ff wS = ff{__shfl_sync(0xffffffffu, cS.hi, w), __shfl_sync(0xffffffffu, cS.lo, w)};
          if (ff_pos(wS)) Sr = ff_add(Sr, ff_mul(wS, exp_diff_accurate(wm, mv, tau)));
        }
      }
      if (lane == 0) s_rec[r] = ClusterRec{mv, mi, Sr};
    }
  }
  cluster_sync();

  // ---- 2. CTA 0: combine the slices of every row and decide ----
  if (rank == 0) {
    int my_tok = -1;
    float my_u = 0.f;
    if (tid < k) {
      my_tok = p.tokens[(size_t)b * k + tid];
      my_u = p.u[(size_t)b * (k + 1) + tid];
    }
    for (int r = warp; r <= k; r += kAccWarps) {
      float mv = -INFINITY, cm = -INFINITY;
      int mi = INT_MAX;
      ff cS = ff_of(0.f);
      if (lane < cs) {
        const float4 rec = ld_dsmem_f32x4(smem_addr(&s_rec[r]), lane);
        cm = rec.x;
        cS = ff{rec.z, rec.w};
        mv = cm;
        mi = __float_as_int(rec.y);
      }
      warp_argmax(mv, mi);
      ff Sr = ff_of(0.f);
      if (!greedy && mv != -INFINITY) {
        if (lane < cs && ff_pos(cS)) Sr = ff_mul(cS, exp_diff_accurate(cm, mv, tau));
        Sr = warp_sum_ff(Sr);
      }
      if (lane == 0) {
        const int x = r < k ? p.tokens[(size_t)b * k + r] : -1;
        const bool ok = x >= 0 && x < V;
        s_rm[r] = mv;
        s_rarg[r] = mi;
        s_rS[r] = Sr;
        s_rlx[r] = ok ? p.logits[((size_t)b * (k + 1) + r) * V + x] : 0.f;
        s_rqx[r] = ok ? p.q[((size_t)b * k + r) * V + x] : 0.f;
        s_rhx[r] = ok ? 1 : 0;
      }
    }
    __syncthreads();
    decide_sequence(p, b, greedy, tau, my_tok, my_u, s_rm, s_rarg, s_rS, s_rlx, s_rqx, s_rhx, s_acc);
    // publish j and row j's (max, sum) into every CTA's shared memory
    if (tid < cs) {
      int j = k;
      for (int i = 0; i < k; ++i)
        if (!s_acc[i]) { j = i; break; }
      st_dsmem_f32(dsmem_addr(smem_addr(&s_dec_j), tid), __int_as_float(j));
      st_dsmem_f32(dsmem_addr(smem_addr(&s_dec_m), tid), s_rm[j]);
      st_dsmem_f32(dsmem_addr(smem_addr(&s_dec_S), tid), s_rS[j].hi);
      st_dsmem_f32(dsmem_addr(smem_addr(&s_dec_S) + 4, tid), s_rS[j].lo);
    }
  }
  cluster_sync();
  if (greedy) return;  // uniform over the cluster: the sequence is complete

  // ---- 3. row j's residual (or bonus) terms of the slice ----
  const int j = s_dec_j;
  const float mj = s_dec_m;
  const ff Sj = s_dec_S;
  const bool residual = j < k;
  const float invS = ff_div_to_f(1.0f, Sj);
  const float *row = p.logits + ((size_t)b * (k + 1) + j) * V;
  const float *qrow = residual ? p.q + ((size_t)b * k + j) * V : nullptr;
  const int len = x1 - x0;
  ff sp = ff_of(0.f);
  int lr = -1, lp = -1;
  {
    float xv[kClusterPerThread], qv[kClusterPerThread];
#pragma unroll
    for (int t = 0; t < kClusterPerThread; ++t) {
      const int e = tid + kAccThreads * t;
      xv[t] = e < len ? row[x0 + e] : 0.f;
      qv[t] = (residual && e < len) ? qrow[x0 + e] : 0.f;
    }
    float pzs[kClusterPerThread];
#pragma unroll
    for (int t = 0; t < kClusterPerThread; ++t) {
      const int e = tid + kAccThreads * t;
      pzs[t] = 0.f;
      if (e < len) {
        float rr;
        draw_terms(xv[t], qv[t], residual, mj, tau, invS, rr, pzs[t]);
        s_terms[e] = rr;
        if (rr > 0.f) lr = x0 + e;
        if (pzs[t] > 0.f) lp = x0 + e;
      }
    }
#pragma unroll
    for (int t = 0; t < kClusterPerThread; t += 4)
      sp = ff_add(sp, ff_of(sum4(pzs[t], pzs[t + 1], pzs[t + 2], pzs[t + 3])));
  }
  __syncthreads();
  // thread t owns the contiguous run [a0, a1) of the slice, summed in order
  const int per = (len + kAccThreads - 1) / kAccThreads;
  const int a0 = min(len, tid * per), a1 = min(len, a0 + per);
  {
    ff mine = ff_of(0.f);
    for (int e = a0; e < a1; ++e) mine = ff_add(mine, ff_of(s_terms[e]));
    ff ex, tot;
    block_inclusive_scan(mine, s_scan, &ex, &tot);
    const ff tp = block_sum(sp, s_d);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lr = max(lr, __shfl_xor_sync(0xffffffffu, lr, o));
      lp = max(lp, __shfl_xor_sync(0xffffffffu, lp, o));
    }
    if (tid == 0) { s_i0 = -1; s_i1 = -1; }
    __syncthreads();
    if (lane == 0) { atomicMax(&s_i0, lr); atomicMax(&s_i1, lp); }
    __syncthreads();
    if (tid == 0) s_draw = ClusterDraw{tot, tp, s_i0, s_i1, {0, 0}};
  }
  cluster_sync();

  // ---- 4. the slice holding u_k * S draws the token ----
  if (warp == 0) {
    // lane l reads slice l's record (all in flight together); the sums run
    // in rank order through shuffles, identically in every CTA
    ff r_l = ff_of(0.f), p_l = ff_of(0.f);
    int lr_l = -1, lp_l = -1;
    if (lane < cs) {
      const uint32_t a = smem_addr(&s_draw);
      const float4 s0 = ld_dsmem_f32x4(a, lane), s1 = ld_dsmem_f32x4(a + 16, lane);
      r_l = ff{s0.x, s0.y};
      p_l = ff{s0.z, s0.w};
      lr_l = __float_as_int(s1.x);
      lp_l = __float_as_int(s1.y);
    }
    ff tr = ff_of(0.f), tp = ff_of(0.f);
    for (int l = 0; l < cs; ++l) {
      tr = ff_add(tr, ff{__shfl_sync(0xffffffffu, r_l.hi, l), __shfl_sync(0xffffffffu, r_l.lo, l)});
      tp = ff_add(tp, ff{__shfl_sync(0xffffffffu, p_l.hi, l), __shfl_sync(0xffffffffu, p_l.lo, l)});
    }
    const bool use_p = !ff_pos(tr);  // residual with no mass (rounding only)
    const ff total = use_p ? tp : tr;
    const ff target = ff_mul(total, p.u[(size_t)b * (k + 1) + k]);
    // slice l covers [cum_l, cum_l + sum_l); cum_{l+1} = ff_add(cum_l, sum_l) exactly
    int cross = -1, last = -1;
    ff cum = ff_of(0.f), base = ff_of(0.f);
    for (int l = 0; l < cs; ++l) {
      const ff mine = use_p ? p_l : r_l;
      const ff sl = ff{__shfl_sync(0xffffffffu, mine.hi, l), __shfl_sync(0xffffffffu, mine.lo, l)};
      const ff nxt = ff_add(cum, sl);
      last = max(last, __shfl_sync(0xffffffffu, use_p ? lp_l : lr_l, l));
      if (cross < 0 && ff_pos(sl) && ff_lt(target, nxt) && !ff_lt(target, cum)) {
        cross = l;
        base = cum;
      }
      cum = nxt;
    }
    if (lane == 0) {
      s_i0 = cross;
      s_i1 = use_p ? 1 : 0;
      s_total = target;
      s_base = base;
      // no slice holds the target (rounding): the last token with positive mass
      if (cross < 0 && rank == 0) p.out_tokens[(size_t)b * (k + 1) + j] = last;
    }
  }
  __syncthreads();
  if (s_i0 == rank) {
    const bool use_p = s_i1 != 0;
    if (use_p) {
      for (int e = tid; e < len; e += kAccThreads) {
        float rr, pz;
        draw_terms(row[x0 + e], 0.f, false, mj, tau, invS, rr, pz);
        s_terms[e] = pz;
      }
      __syncthreads();
    }
    const ff target = s_total;
    ff mine = ff_of(0.f);
    for (int e = a0; e < a1; ++e) mine = ff_add(mine, ff_of(s_terms[e]));
    ff ex, tot;
    block_inclusive_scan(mine, s_scan, &ex, &tot);
    ff c = ff_add(s_base, ex);
    if (tid == 0) s_i0 = INT_MAX;
    __syncthreads();
    for (int e = a0; e < a1; ++e) {
      c = ff_add(c, ff_of(s_terms[e]));
      if (ff_lt(target, c)) { atomicMin(&s_i0, x0 + e); break; }
    }
    __syncthreads();
    if (tid == 0)
      p.out_tokens[(size_t)b * (k + 1) + j] =
          s_i0 != INT_MAX ? s_i0 : (use_p ? s_draw.last_p : s_draw.last_r);
  }
  cluster_sync();  // peers may still read this CTA's s_draw
}

// Fused path: the decisions from the projection's per-CTA row statistics
// (launch_projection_stats, G records per row) instead of a pass over the
// logits.  grid (B), kAccThreads threads: warp w combines rows w, w + 8, ...
__global__ void __launch_bounds__(kAccThreads)
accept_decide_kernel(const __grid_constant__ AccParams p, const SampStat *__restrict__ stats, int G) {
  __shared__ int s_acc[SF_MAX_DRAFT];
  __shared__ float s_rm[SF_MAX_DRAFT + 1], s_rlx[SF_MAX_DRAFT + 1], s_rqx[SF_MAX_DRAFT + 1];
  __shared__ int s_rarg[SF_MAX_DRAFT + 1], s_rhx[SF_MAX_DRAFT + 1];
  __shared__ ff s_rS[SF_MAX_DRAFT + 1];
  grid_dependency_wait();  // statistics and logits come from the projection
  grid_launch_dependents();
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = p.k, V = p.V;
  const float tau = p.tau[b];
  const bool greedy = !(tau > 0.0f);
  int my_tok = -1;
  float my_u = 0.f;
  if (tid < k) {
    my_tok = p.tokens[(size_t)b * k + tid];
    my_u = p.u[(size_t)b * (k + 1) + tid];
  }
  for (int rr = warp; rr <= k; rr += kAccWarps) {
    const size_t row = (size_t)b * (k + 1) + rr;
    const SampStat *cr = stats + row * G;
    float mv = -INFINITY;
    int mi = INT_MAX;
    for (int c = lane; c < G; c += 32)
      if (better(cr[c].m, cr[c].arg, mv, mi)) { mv = cr[c].m; mi = cr[c].arg; }
    warp_argmax(mv, mi);
    ff Sr = ff_of(0.f);
    if (!greedy && mv != -INFINITY) {
      for (int c = lane; c < G; c += 32)
        if (ff_pos(cr[c].S)) Sr = ff_add(Sr, ff_mul(cr[c].S, exp_diff_accurate(cr[c].m, mv, tau)));
      Sr = warp_sum_ff(Sr);
    }
    if (lane == 0) {
      const int x = rr < k ? p.tokens[(size_t)b * k + rr] : -1;
      const bool ok = x >= 0 && x < V;
      s_rm[rr] = mv;
      s_rarg[rr] = mi;
      s_rS[rr] = Sr;
      s_rlx[rr] = ok ? p.logits[row * V + x] : 0.f;
      s_rqx[rr] = ok ? p.q[((size_t)b * k + rr) * V + x] : 0.f;
      s_rhx[rr] = ok ? 1 : 0;
      p.rows[row] = RowStat{mv, mi, Sr};
    }
  }
  __syncthreads();
  decide_sequence(p, b, greedy, tau, my_tok, my_u, s_rm, s_rarg, s_rS, s_rlx, s_rqx, s_rhx, s_acc);
}

// The residual (j < k) or bonus (j == k) draw of sequence b (grid (C2, B)
// of kAccThreads threads; rs holds row j's max, argmax and sum).  Warp w of
// CTA c sums the residual and target masses of segment c * kAccWarps + w of
// row j (float-float) into its part; the last CTA of the sequence to finish
// (one atomic ticket; nobody waits) locates the segment holding u_k * S with
// a float-float scan over the segment sums in order, and scans that segment
// in ascending token order, four tokens per thread.
__device__ void draw_residual(const AccParams &p, int b, int c, int j, RowStat rs, float tau,
                              float u_k) {
  __shared__ ff s_d[32];
  __shared__ ff s_scan[kAccWarps + 1];
  __shared__ int s_flag, s_seg, s_token;
  __shared__ ff s_base;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int k = p.k, V = p.V, NS = p.C1;
  const bool residual = j < k;
  const float invS = ff_div_to_f(1.0f, rs.S);
  const float *row = p.logits + ((size_t)b * (k + 1) + j) * V;
  const float *qrow = residual ? p.q + ((size_t)b * k + j) * V : nullptr;
  DrawPart *parts = p.parts + (size_t)b * NS;
  // four consecutive tokens from e (past V: logit -inf and q 0, terms 0)
  auto load4 = [&](int e, float4 &x, float4 &qq) {
    if (p.vec4) {
      x = e < V ? *reinterpret_cast<const float4 *>(row + e)
                : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
      qq = (e < V && residual) ? __ldcs(reinterpret_cast<const float4 *>(qrow + e))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
    } else {
      x.x = e < V ? row[e] : -INFINITY;
      x.y = e + 1 < V ? row[e + 1] : -INFINITY;
      x.z = e + 2 < V ? row[e + 2] : -INFINITY;
      x.w = e + 3 < V ? row[e + 3] : -INFINITY;
      qq.x = (e < V && residual) ? qrow[e] : 0.f;
      qq.y = (e + 1 < V && residual) ? qrow[e + 1] : 0.f;
      qq.z = (e + 2 < V && residual) ? qrow[e + 2] : 0.f;
      qq.w = (e + 3 < V && residual) ? qrow[e + 3] : 0.f;
    }
  };

  // ---- segment sums of r and p: lane sums of 32 terms added pairwise in
  // fp32, then a float-float warp sum ----
  const int sg = c * kAccWarps + warp;
  if (sg < NS) {
    float4 xv[8], qv[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) load4(sg * kSegTokens + 128 * i + 4 * lane, xv[i], qv[i]);
    float gr[8], gp[8];
    int lr = -1, lp = -1;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int e = sg * kSegTokens + 128 * i + 4 * lane;
      const float xs[4] = {xv[i].x, xv[i].y, xv[i].z, xv[i].w};
      const float qs[4] = {qv[i].x, qv[i].y, qv[i].z, qv[i].w};
      float rr[4], pz[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        draw_terms(xs[u], qs[u], residual, rs.m, tau, invS, rr[u], pz[u]);
        lr = rr[u] > 0.f ? e + u : lr;
        lp = pz[u] > 0.f ? e + u : lp;
      }
      gr[i] = sum4(rr[0], rr[1], rr[2], rr[3]);
      gp[i] = sum4(pz[0], pz[1], pz[2], pz[3]);
    }
    const ff Sr = warp_sum_ff(ff_of(__fadd_rn(__fadd_rn(__fadd_rn(gr[0], gr[1]), __fadd_rn(gr[2], gr[3])),
                                              __fadd_rn(__fadd_rn(gr[4], gr[5]), __fadd_rn(gr[6], gr[7])))));
    const ff Sp = warp_sum_ff(ff_of(__fadd_rn(__fadd_rn(__fadd_rn(gp[0], gp[1]), __fadd_rn(gp[2], gp[3])),
                                              __fadd_rn(__fadd_rn(gp[4], gp[5]), __fadd_rn(gp[6], gp[7])))));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      lr = max(lr, __shfl_xor_sync(0xffffffffu, lr, o));
      lp = max(lp, __shfl_xor_sync(0xffffffffu, lp, o));
    }
    if (lane == 0) parts[sg] = DrawPart{Sr, Sp, lr, lp, {0, 0}};
  }

  // ---- the last CTA of the sequence draws the token ----
  __syncthreads();  // every part of this CTA is written
  if (tid == 0)     // release this CTA's parts, acquire the others'
    s_flag = atom_add_acq_rel_gpu(p.draw_tickets + b, 1u) == static_cast<unsigned>(p.C2 - 1);
  __syncthreads();
  if (!s_flag) return;

  auto part_sum = [&](int cc, bool pmass) -> ff {
    const float4 v = __ldcg(reinterpret_cast<const float4 *>(parts + cc));
    return pmass ? ff{v.z, v.w} : ff{v.x, v.y};
  };
  ff target;
  bool use_p;
  int my_last_r = -1, my_last_p = -1;  // one segment per thread: its last indices
  if (tid == 0) { s_seg = INT_MAX; s_base = ff_of(0.f); }
  if (NS <= kAccThreads) {
    // one segment per thread: every part is loaded once, and one scan gives
    // both the segment intervals and the total (its last inclusive value, so
    // that the intervals tile [0, total) exactly)
    float4 v0 = make_float4(0.f, 0.f, 0.f, 0.f);
    if (tid < NS) {
      v0 = __ldcg(reinterpret_cast<const float4 *>(parts + tid));
      my_last_r = __ldcg(&parts[tid].last_r);
      my_last_p = __ldcg(&parts[tid].last_p);
    }
    ff v = ff{v0.x, v0.y};
    ff excl, total;
    ff incl = block_inclusive_scan(v, s_scan, &excl, &total);
    use_p = !ff_pos(total);  // residual with no mass (rounding only)
    if (use_p) {
      v = ff{v0.z, v0.w};
      incl = block_inclusive_scan(v, s_scan, &excl, &total);
    }
    target = ff_mul(total, u_k);
    if (tid < NS && ff_pos(v) && ff_lt(target, incl) && !ff_lt(target, excl)) atomicMin(&s_seg, tid);
    __syncthreads();
    if (s_seg == tid) s_base = excl;
  } else {
    ff total;
    {
      ff pr = ff_of(0.f);
      for (int cc = tid; cc < NS; cc += kAccThreads) pr = ff_add(pr, part_sum(cc, false));
      total = block_sum(pr, s_d);
    }
    use_p = !ff_pos(total);  // residual with no mass (rounding only)
    if (use_p) {
      ff pp = ff_of(0.f);
      for (int cc = tid; cc < NS; cc += kAccThreads) pp = ff_add(pp, part_sum(cc, true));
      total = block_sum(pp, s_d);
    }
    target = ff_mul(total, u_k);
    // segment holding the target: inclusive float-float scan over the
    // segment sums in order; segment cc covers [excl, incl), and excl of cc
    // is bit-identical to incl of cc - 1, so the intervals tile [0, total)
    ff carry = ff_of(0.f);
    for (int base = 0; base < NS; base += kAccThreads) {
      const int cc = base + tid;
      const ff v = cc < NS ? part_sum(cc, use_p) : ff_of(0.f);
      ff excl_local, blk_total;
      const ff incl_local = block_inclusive_scan(v, s_scan, &excl_local, &blk_total);
      const ff excl = ff_add(carry, excl_local), incl = ff_add(carry, incl_local);
      if (cc < NS && ff_pos(v) && ff_lt(target, incl) && !ff_lt(target, excl)) atomicMin(&s_seg, cc);
      __syncthreads();
      if (s_seg == cc) s_base = excl;
      carry = ff_add(carry, blk_total);
      __syncthreads();
      if (s_seg != INT_MAX) break;
    }
  }
  __syncthreads();
  int token = -1;
  if (s_seg == INT_MAX) {
    // u*S at or past the total (rounding): the last token with positive mass
    int last = -1;
    if (NS <= kAccThreads) {
      last = use_p ? my_last_p : my_last_r;
    } else {
      for (int cc = tid; cc < NS; cc += kAccThreads)
        last = max(last, use_p ? __ldcg(&parts[cc].last_p) : __ldcg(&parts[cc].last_r));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) last = max(last, __shfl_xor_sync(0xffffffffu, last, o));
    if (tid == 0) s_token = -1;
    __syncthreads();
    if (lane == 0) atomicMax(&s_token, last);
    __syncthreads();
    token = s_token;
  } else {
    // the segment in ascending token order: thread t owns tokens 4t .. 4t+3
    // (terms recomputed exactly as in the segment sums)
    const int cc = s_seg;
    const int e = cc * kSegTokens + 4 * tid;
    float4 xv, qv;
    load4(e, xv, qv);
    const float xs[4] = {xv.x, xv.y, xv.z, xv.w};
    const float qs[4] = {qv.x, qv.y, qv.z, qv.w};
    float t[4];
    ff mine = ff_of(0.f);
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      float rr, pz;
      draw_terms(xs[u], qs[u], residual, rs.m, tau, invS, rr, pz);
      t[u] = use_p ? pz : rr;
      mine = ff_add(mine, ff_of(t[u]));
    }
    ff excl, unused;
    block_inclusive_scan(mine, s_scan, &excl, &unused);
    ff cum = ff_add(s_base, excl);
    if (tid == 0) s_token = INT_MAX;
    __syncthreads();
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      cum = ff_add(cum, ff_of(t[u]));
      if (t[u] > 0.f && ff_lt(target, cum)) {
        atomicMin(&s_token, e + u);
        break;
      }
    }
    __syncthreads();
    token = s_token;
    if (token == INT_MAX) {
      // rounding put the target past the segment's own running sum: its last
      // positive token
      token = use_p ? __ldcg(&parts[cc].last_p) : __ldcg(&parts[cc].last_r);
    }
  }
  if (tid == 0) {
    p.out_tokens[(size_t)b * (k + 1) + j] = token;
    p.draw_tickets[b] = 0u;
  }
}


__global__ void __launch_bounds__(kAccThreads, 3)
accept_draw_kernel(const __grid_constant__ AccParams p) {
  // The previous kernel (the decision kernel of this call) lets this grid
  // start only after it has itself waited for the kernel before the call, so
  // the call's inputs (temperature, uniforms) are in place already; j and
  // the row statistics are waited for.
  grid_launch_dependents();
  const int c = blockIdx.x, b = blockIdx.y;
  const int k = p.k;
  const float tau = p.tau[b];
  if (!(tau > 0.0f)) return;  // greedy sequences are complete
  const float u_k = p.u[(size_t)b * (k + 1) + k];
  grid_dependency_wait();     // j and row j's statistics come from the previous kernel
  const int4 sq = __ldcg(reinterpret_cast<const int4 *>(p.seqs + b));
  const int j = sq.x;
  if (j < 0 || j > k) {       // no decision was written (a timed-out statistics pass)
    if (c == 0 && threadIdx.x == 0) set_status(p.status, SF_DEVICE_TIMEOUT);
    return;
  }
  const RowStat rs = {__int_as_float(sq.y), 0, ff{__int_as_float(sq.z), __int_as_float(sq.w)}};
  draw_residual(p, b, c, j, rs, tau, u_k);
}

// --------------------------------------------------------------------------
// Two-kernel acceptance for vocabularies beyond one cluster (V > 16 x 2048).
//
// accept_chunks_kernel streams the (k+1) x V logits of every sequence once.
// The B (k+1) rows are cut into 1024-token segments ("chunks"), numbered row
// by row, and warp g of NW1 owns chunks [g U / NW1, (g+1) U / NW1) of the U
// in all: a few consecutive chunks, at most two or three rows.  Lane l reads
// tokens 128 i + 4 l .. +3 of a chunk (eight 16-byte loads), and the next
// chunk's loads are in flight while the current one is folded into per-lane
// running state (max, first index, float-float sum of exp((x - max)/tau)).
// At the end of each run of chunks of one row the warp combines its lanes
// and writes one run record; the runs of row R are stored in warp order, so
// that run t of the row is the one of warp warp_of(R C1) + t.
//
// The warp that writes a row's last run record (a ticket per row) combines
// the row's runs in run order into its final statistics; the warp that
// finalises a sequence's k + 1 rows (a ticket per sequence) takes the k
// decisions.  accept_draw_kernel, grid (C2, B), then draws the token of row
// j for the sampled sequences.
// --------------------------------------------------------------------------

// The warp of the chunk kernel owning chunk u: the largest g with
// floor(g U / NW) <= u (warps with empty ranges are never returned).
__device__ __forceinline__ int warp_of(int u, int U, int NW) {
  return static_cast<int>(((long long)(u + 1) * NW - 1) / U);
}

// The 32 tokens of lane `lane` in chunk c of a row: c*1024 + 128 i + 4 lane + t
// (tokens at or past V read as -inf).
__device__ __forceinline__ void load_chunk(const AccParams &p, int row, int c, int lane,
                                           float4 (&x)[8]) {
  const float *rp = p.logits + (size_t)row * p.V;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int e = c * kSegTokens + 128 * i + 4 * lane;
    if (p.vec4) {
      x[i] = e < p.V ? __ldcg(reinterpret_cast<const float4 *>(rp + e))
                     : make_float4(-INFINITY, -INFINITY, -INFINITY, -INFINITY);
    } else {
      x[i].x = e < p.V ? __ldcg(rp + e) : -INFINITY;
      x[i].y = e + 1 < p.V ? __ldcg(rp + e + 1) : -INFINITY;
      x[i].z = e + 2 < p.V ? __ldcg(rp + e + 2) : -INFINITY;
      x[i].w = e + 3 < p.V ? __ldcg(rp + e + 3) : -INFINITY;
    }
  }
}

// State of one warp over its current run (consecutive chunks of one row).
// Each lane keeps the max of its own tokens so far, the first index holding
// it and the float-float sum of exp((x - max)/tau) over them; the warp
// combines the lanes once, at the end of the run.
struct RunState {
  int row, c, start_chunk, len;
  float tau, scale;  // scale = log2(e) / tau, rounded once
  bool greedy;
  float lm;          // lane max
  int li;            // its first index
  ff lS;             // lane sum, relative to lm
};

__device__ __forceinline__ void run_begin(const AccParams &p, RunState &st, int row, int c) {
  st.row = row;
  st.c = c;
  st.start_chunk = c;
  st.len = 0;
  st.tau = __ldg(p.tau + row / (p.k + 1));
  st.greedy = !(st.tau > 0.0f);
  st.scale = st.greedy ? 0.f : __fdiv_rn(1.44269504088896341f, st.tau);
  st.lm = -INFINITY;
  st.li = INT_MAX;
  st.lS = ff_of(0.f);
}

// Folds chunk st.c (its tokens in x) into the lane state.
__device__ __forceinline__ void run_chunk(RunState &st, int lane, const float4 (&x)[8]) {
  float cm = -INFINITY;
#pragma unroll
  for (int i = 0; i < 8; ++i) cm = fmaxf(cm, fmaxf(fmaxf(x[i].x, x[i].y), fmaxf(x[i].z, x[i].w)));
  if (st.len == 0 || cm > st.lm) {
    // new lane max (or the run's first chunk): its first index in this chunk,
    // and the sum so far moved to the new reference
    int fi = INT_MAX;
#pragma unroll
    for (int i = 7; i >= 0; --i) {  // descending, so the first match wins
      const int e = st.c * kSegTokens + 128 * i + 4 * lane;
      fi = x[i].w == cm ? e + 3 : fi;
      fi = x[i].z == cm ? e + 2 : fi;
      fi = x[i].y == cm ? e + 1 : fi;
      fi = x[i].x == cm ? e : fi;
    }
    if (ff_pos(st.lS)) st.lS = ff_mul(st.lS, exp_diff_accurate(st.lm, cm, st.tau));
    st.lm = cm;
    st.li = fi;
  }
  if (!st.greedy && st.lm != -INFINITY) {
    // 2^((x - lm) log2(e)/tau): the difference and the product each rounded
    // once per token (a term's relative error grows with |x - lm| x 1e-7
    // with no common bias), 2^ by the hardware approximation; the 32 terms
    // are added pairwise in fp32 before one float-float add
    float t[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
      t[i] = sum4(ex2_approx(__fmul_rn(__fsub_rn(x[i].x, st.lm), st.scale)),
                  ex2_approx(__fmul_rn(__fsub_rn(x[i].y, st.lm), st.scale)),
                  ex2_approx(__fmul_rn(__fsub_rn(x[i].z, st.lm), st.scale)),
                  ex2_approx(__fmul_rn(__fsub_rn(x[i].w, st.lm), st.scale)));
    st.lS = ff_add(st.lS, ff_of(__fadd_rn(__fadd_rn(__fadd_rn(t[0], t[1]), __fadd_rn(t[2], t[3])),
                                          __fadd_rn(__fadd_rn(t[4], t[5]), __fadd_rn(t[6], t[7])))));
  }
  ++st.len;
}

__device__ __forceinline__ RowStat combine_runs(const AccParams &p, int row, float tau,
                                                bool greedy);

// The k accept/reject decisions of sequence b by one warp, from the final
// row statistics (lane i < k tests draft i, exactly as decide_sequence
// does); writes every output except, for a sampled sequence, out_tokens[j],
// which the draw kernel writes.
__device__ void decide_warp(const AccParams &p, int b) {
  const int lane = threadIdx.x & 31, k = p.k, V = p.V;
  const float tau = p.tau[b];
  const bool greedy = !(tau > 0.0f);
  const RowStat *rows = p.rows + (size_t)b * (k + 1);
  float rm = 0.f;
  int rarg = -1;
  ff rS = ff_of(0.f);
  if (lane <= k) {
    const float4 v = __ldcg(reinterpret_cast<const float4 *>(rows + lane));
    rm = v.x;
    rarg = __float_as_int(v.y);
    rS = ff{v.z, v.w};
  }
  int tok = -1;
  float u = 0.f, lx = 0.f, qx = 0.f;
  bool in_range = false;
  if (lane < k) {
    tok = p.tokens[(size_t)b * k + lane];
    u = p.u[(size_t)b * (k + 1) + lane];
    in_range = tok >= 0 && tok < V;
    if (in_range) {
      lx = p.logits[((size_t)b * (k + 1) + lane) * V + tok];
      qx = p.q[((size_t)b * k + lane) * V + tok];
    }
  }
  int acc = 0;
  if (lane < k) {
    float ratio = 0.f;
    if (!in_range) {
      set_status(p.status, SF_DEVICE_BAD_TOKEN);  // treated as a rejection
    } else if (greedy) {
      acc = tok == rarg;
      ratio = acc ? 1.f : 0.f;
    } else {
      // p(x) = exp((l_x - m) / tau) / S; accept iff u * q(x) < p(x), with the
      // product u * q kept exactly as float-float
      const float px = ff_div_to_f(exp_diff_accurate(lx, rm, tau), rS);
      const float uq = __fmul_rn(u, qx);
      const ff uqf = ff{uq, __fmaf_rn(u, qx, -uq)};
      acc = ff_lt(uqf, ff_of(px)) ? 1 : 0;
      ratio = qx > 0.f ? fminf(1.f, __fdiv_rn(px, qx)) : 1.f;
    }
    if (p.ratio) p.ratio[(size_t)b * k + lane] = ratio;
  }
  const unsigned rejected = __ballot_sync(0xffffffffu, lane < k && !acc);
  const int j = rejected ? __ffs(rejected) - 1 : k;
  const int arg_j = __shfl_sync(0xffffffffu, rarg, j);
  const float m_j = __shfl_sync(0xffffffffu, rm, j);
  const ff S_j = ff{__shfl_sync(0xffffffffu, rS.hi, j), __shfl_sync(0xffffffffu, rS.lo, j)};
  if (lane <= k) {
    int v = -1;
    if (lane < j) v = tok;
    else if (lane == j && greedy) v = arg_j;
    if (!(lane == j && !greedy)) p.out_tokens[(size_t)b * (k + 1) + lane] = v;
  }
  if (lane == 0) {
    p.num_accepted[b] = j;
    p.seqs[b] = SeqState{j, m_j, S_j};
  }
}

// A run record whose row ticket is taken: the row, its number of runs and
// (lane 0) the ticket's value before this warp's add.
struct PendingTicket {
  int row;          // -1: none
  int n_runs;       // runs of the row
  uint32_t ticket;  // lane 0: the row ticket before this warp's add
};

// Ends the warp's run: combines the lanes, writes the run's record and
// takes the row's ticket (lane 0; one atomic per run; nobody waits).
__device__ __forceinline__ PendingTicket run_end(const AccParams &p, const RunState &st, int lane,
                                                 int gw, int U) {
  float wm = st.lm;
  int wi = st.li;
  warp_argmax(wm, wi);
  ff S = ff_of(0.f);
  if (!st.greedy && wm != -INFINITY) {
    ff mine = ff_of(0.f);
    if (ff_pos(st.lS)) mine = ff_mul(st.lS, exp_diff_accurate(st.lm, wm, st.tau));
    S = warp_sum_ff(mine);
  }
  const int CPR = p.C1;
  const int g0 = warp_of(st.row * CPR, U, p.NW1);
  PendingTicket pt{st.row, warp_of(st.row * CPR + CPR - 1, U, p.NW1) - g0 + 1, 0u};
  if (lane == 0) {
    p.runs[(size_t)st.row * CPR + (gw - g0)] = RowStat{wm, wi, S};  // run gw - g0 of its row
    // the release covers the record; the acquire, the other runs' records
    pt.ticket = atom_add_acq_rel_gpu(p.row_tickets + pt.row, 1u);
  }
  return pt;
}

// Looks at a taken row ticket: the warp that wrote the row's last record
// combines the row's runs in run order into its final statistics, and the
// warp that finalises a sequence's k + 1 rows takes its decisions.
__device__ __forceinline__ void resolve_ticket(const AccParams &p, const PendingTicket &pt, int lane) {
  const bool last = __shfl_sync(0xffffffffu, pt.ticket == static_cast<uint32_t>(pt.n_runs - 1), 0);
  if (!last) return;
  __syncwarp();
  const float tau = __ldg(p.tau + pt.row / (p.k + 1));
  const RowStat rs = combine_runs(p, pt.row, tau, !(tau > 0.0f));
  const int b = pt.row / (p.k + 1);
  uint32_t last_row = 0;
  if (lane == 0) {
    p.rows[pt.row] = rs;
    p.row_tickets[pt.row] = 0u;  // zero again for the next call
    last_row = atom_add_acq_rel_gpu(p.seq_tickets + b, 1u) == static_cast<uint32_t>(p.k);
  }
  if (!__shfl_sync(0xffffffffu, last_row, 0)) return;
  __syncwarp();
  decide_warp(p, b);
  if (lane == 0) p.seq_tickets[b] = 0u;
}

// Chunk ring of the bulk-copy path: kChunkStages 4 KB stages per warp (the
// chunks a warp has requested ahead of the one it reduces) and one mbarrier
// per stage.  Two CTAs per SM keep 192 KB of logits in flight per SM.
constexpr int kChunkStages = 3;
constexpr int kChunkRingBytes = kAccWarps * kChunkStages * kSegTokens * 4;
constexpr int kChunkSmemBytes = kChunkRingBytes + kAccWarps * kChunkStages * 8;

// kBulk (rows 16-byte aligned, V % 4 == 0): each warp's lane 0 requests its
// chunks into the warp's ring with 1-D bulk copies, kChunkStages ahead, and
// the warp reduces them from shared memory; otherwise two register buffers
// (chunk u + 1 loads while chunk u is reduced).
template <bool kBulk>
__global__ void __launch_bounds__(kAccThreads, 2)
accept_chunks_kernel(const __grid_constant__ AccParams p) {
  extern __shared__ __align__(128) uint8_t s_ring[];
  // Every input may come from the previous kernel on the stream: wait for
  // it before reading anything, and only then let the finishing kernel be
  // scheduled (so that it too starts after that kernel completed).
  grid_dependency_wait();
  grid_launch_dependents();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gw = blockIdx.x * kAccWarps + warp;
  const int CPR = p.C1;
  const int U = p.B * (p.k + 1) * CPR;  // < 2^31: the host checks V * (k + 1) and B
  const int u0 = static_cast<int>((long long)gw * U / p.NW1);
  const int u1 = static_cast<int>((long long)(gw + 1) * U / p.NW1);
  if (u0 >= u1) return;
  RunState st;
  run_begin(p, st, u0 / CPR, u0 % CPR);
  // the next chunk: the row boundary ends the run and looks at its ticket
  auto advance = [&](int u) {
    int nrow = st.row, nc = st.c + 1;
    if (nc == CPR) { nc = 0; ++nrow; }
    if (nc == 0 || u + 1 == u1) {
      const PendingTicket now = run_end(p, st, lane, gw, U);
      resolve_ticket(p, now, lane);
      if (u + 1 < u1) run_begin(p, st, nrow, 0);
    } else {
      st.c = nc;
    }
  };
  if constexpr (kBulk) {
    const float4 *ring = reinterpret_cast<const float4 *>(s_ring + warp * kChunkStages * kSegTokens * 4);
    const uint32_t ring_s = smem_addr(ring);
    const uint32_t bar0 = smem_addr(s_ring + kChunkRingBytes) + static_cast<uint32_t>(warp * kChunkStages * 8);
    if (lane == 0) {
#pragma unroll 1
      for (int s = 0; s < kChunkStages; ++s) mbar_init(bar0 + 8u * s, 1);
      fence_mbar_init();
    }
    __syncwarp();
    // lane 0: chunk u (row u / CPR, tokens from (u % CPR) * 1024) into stage s
    auto request = [&](int u, int s) {
      const int row = u / CPR, c = u - row * CPR;
      const int n = min(kSegTokens, p.V - c * kSegTokens);
      const uint32_t bytes = static_cast<uint32_t>(n) * 4u;
      mbar_arrive_expect_tx(bar0 + 8u * s, bytes);
      bulk_copy_g2s(ring_s + static_cast<uint32_t>(s * kSegTokens * 4),
                    p.logits + (size_t)row * p.V + (size_t)c * kSegTokens, bytes, bar0 + 8u * s);
    };
    if (lane == 0) {
#pragma unroll 1
      for (int s = 0; s < kChunkStages && u0 + s < u1; ++s) request(u0 + s, s);
    }
    int issued = min(kChunkStages, u1 - u0);
#pragma unroll 1
    for (int u = u0; u < u1; ++u) {
      const int i = u - u0, s = i % kChunkStages;
      const bool ok = mbar_wait_bounded(bar0 + 8u * s, static_cast<uint32_t>(i / kChunkStages) & 1u);
      if (!__all_sync(0xffffffffu, ok)) {
        // a copy never completed (not expected): flag it, wait (bounded)
        // for the other requested stages, and stop this warp
        if (lane == 0) {
          set_status(p.status, SF_DEVICE_TIMEOUT);
#pragma unroll 1
          for (int x = i + 1; x < issued; ++x)
            (void)mbar_wait_bounded(bar0 + 8u * (x % kChunkStages), static_cast<uint32_t>(x / kChunkStages) & 1u);
        }
        return;
      }
      float4 x[8];
#pragma unroll
      for (int t = 0; t < 8; ++t) x[t] = ring[s * (kSegTokens / 4) + 32 * t + lane];
      if ((st.c + 1) * kSegTokens > p.V) {
        // the row's last chunk: tokens at or past V were not copied
#pragma unroll
        for (int t = 0; t < 8; ++t) {
          const int e = st.c * kSegTokens + 128 * t + 4 * lane;
          if (e >= p.V) x[t].x = -INFINITY;
          if (e + 1 >= p.V) x[t].y = -INFINITY;
          if (e + 2 >= p.V) x[t].z = -INFINITY;
          if (e + 3 >= p.V) x[t].w = -INFINITY;
        }
      }
      run_chunk(st, lane, x);
      // the stage's reads are complete (their values are consumed): the
      // next request may overwrite it
      __syncwarp();
      if (issued < u1 - u0 && i + kChunkStages == issued) {
        if (lane == 0) {
          fence_proxy_async_smem();
          request(u0 + issued, s);
        }
        ++issued;
      }
      advance(u);
    }
  } else {
    // two register buffers: chunk u + 1 is loading while chunk u is reduced
    float4 xa[8], xb[8];
    load_chunk(p, st.row, st.c, lane, xa);
    auto step = [&](int u, const float4 (&cur)[8], float4 (&nxt)[8]) {
      int nrow = st.row, nc = st.c + 1;
      if (nc == CPR) { nc = 0; ++nrow; }
      if (u + 1 < u1) load_chunk(p, nrow, nc, lane, nxt);
      run_chunk(st, lane, cur);
      advance(u);
    };
    for (int u = u0; u < u1; u += 2) {
      step(u, xa, xb);
      if (u + 1 < u1) step(u + 1, xb, xa);
    }
  }
}

// Combines the run records of target row `row` (in run order, which is
// chunk order) into the row's max, first argmax and float-float sum rescaled
// to the max.  Executed by one whole warp; all loads are issued before any
// is used.
__device__ __forceinline__ RowStat combine_runs(const AccParams &p, int row, float tau,
                                                bool greedy) {
  constexpr int kPer = 4;  // records per lane and pass
  const int lane = threadIdx.x & 31, CPR = p.C1;
  const int U = p.B * (p.k + 1) * CPR;
  const int g0 = warp_of(row * CPR, U, p.NW1);
  const int n = warp_of(row * CPR + CPR - 1, U, p.NW1) - g0 + 1;
  const float4 *rr = reinterpret_cast<const float4 *>(p.runs + (size_t)row * CPR);
  float mv = -INFINITY;
  int mi = INT_MAX;
  ff Sr = ff_of(0.f);
  for (int base = 0; base < n; base += 32 * kPer) {  // one pass unless n > 128
    float4 a[kPer];
#pragma unroll
    for (int t = 0; t < kPer; ++t) {
      const int i = base + lane + 32 * t;
      a[t] = i < n ? __ldcg(rr + i) : make_float4(-INFINITY, __int_as_float(INT_MAX), 0.f, 0.f);
    }
    float bm = -INFINITY;
    int bi = INT_MAX;
#pragma unroll
    for (int t = 0; t < kPer; ++t)
      if (better(a[t].x, __float_as_int(a[t].y), bm, bi)) { bm = a[t].x; bi = __float_as_int(a[t].y); }
    warp_argmax(bm, bi);
    if (!greedy) {
      // the pass's sums relative to its max, then the running sum moved to
      // the larger of the two maxima
      ff ps = ff_of(0.f);
#pragma unroll
      for (int t = 0; t < kPer; ++t) {
        const ff cS = ff{a[t].z, a[t].w};
        if (ff_pos(cS)) ps = ff_add(ps, ff_mul(cS, exp_diff_accurate(a[t].x, bm, tau)));
      }
      ps = warp_sum_ff(ps);
      if (bm > mv) {
        if (ff_pos(Sr)) Sr = ff_mul(Sr, exp_diff_accurate(mv, bm, tau));
        Sr = ff_add(Sr, ps);
      } else if (ff_pos(ps)) {
        Sr = ff_add(Sr, ff_mul(ps, exp_diff_accurate(bm, mv, tau)));
      }
    }
    if (better(bm, bi, mv, mi)) { mv = bm; mi = bi; }
  }
  return RowStat{mv, mi, Sr};
}

// --------------------------------------------------------------------------
// host side
// --------------------------------------------------------------------------
struct AccPlan {
  int C1, C2;  // segments per row, draw CTAs per row
};

struct AccLayout {
  size_t draw_tickets, row_tickets, seq_tickets, runs, rows, seqs, parts, total;
};

static int plan_accept(int V, AccPlan *plan) {
  plan->C1 = (V + kSegTokens - 1) / kSegTokens;
  plan->C2 = (plan->C1 + kAccWarps - 1) / kAccWarps;
  return SF_OK;
}

static AccLayout acc_layout(int B, int k, const AccPlan &pl) {
  AccLayout l;
  const size_t R = (size_t)B * (k + 1);
  size_t off = 256;
  l.draw_tickets = off; off = round_up(off + 4 * (size_t)B, 256);
  l.row_tickets = off; off = round_up(off + 4 * R, 256);
  l.seq_tickets = off; off = round_up(off + 4 * (size_t)B, 256);
  l.runs = off; off = round_up(off + sizeof(RowStat) * R * pl.C1, 256);
  l.rows = off; off = round_up(off + sizeof(RowStat) * R, 256);
  l.seqs = off; off = round_up(off + sizeof(SeqState) * (size_t)B, 256);
  l.parts = off; off = round_up(off + sizeof(DrawPart) * (size_t)B * pl.C1, 256);
  l.total = off;
  return l;
}

// Cluster size and slice of the single-kernel path: up to 16 CTAs per
// sequence, slices of at most kClusterMaxSlice tokens (a multiple of 4);
// false when V needs more (the two-kernel path spreads those rows over
// many more CTAs).
static bool cluster_plan(int V, int *cs, int *slice) {
  int c = (V + kClusterMaxSlice - 1) / kClusterMaxSlice;
  if (c > kClusterMax) c = kClusterMax;
  if (c < 1) c = 1;
  int sl = (V + c - 1) / c;
  sl = (sl + 3) / 4 * 4;
  if (sl > kClusterMaxSlice) return false;
  *cs = c;
  *slice = sl;
  return true;
}

// Sets the kernel attributes once per device and reports whether a cluster
// of cs CTAs can be resident (*ok false: use the two-kernel path).
static int cluster_setup(int cs, bool *ok) {
  static std::mutex mu;
  static int state[64][kClusterMax + 1] = {};  // 0 unknown, 1 usable, 2 not usable
  DeviceInfo dev;
  int st = current_device(&dev);
  if (st != SF_OK) return st;
  if (dev.ordinal < 0 || dev.ordinal >= 64) return fail(SF_ERR_UNSUPPORTED, "device ordinal %d", dev.ordinal);
  std::lock_guard<std::mutex> lock(mu);
  if (state[dev.ordinal][cs] == 0) {
    cudaError_t e = cudaFuncSetAttribute(accept_cluster_kernel,
                                         cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(accept_cluster_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(sizeof(float) * kClusterMaxSlice));
    if (e != cudaSuccess)
      return fail(SF_ERR_CUDA, "cudaFuncSetAttribute (accept cluster): %s", cudaGetErrorString(e));
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cs, 1);
    cfg.blockDim = dim3(kAccThreads);
    cfg.dynamicSmemBytes = sizeof(float) * kClusterMaxSlice;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, accept_cluster_kernel, &cfg);
    if (e != cudaSuccess) (void)cudaGetLastError();  // not usable: clear the error
    state[dev.ordinal][cs] = (e == cudaSuccess && n > 0) ? 1 : 2;
  }
  *ok = state[dev.ordinal][cs] == 1;
  return SF_OK;
}

// Raises the bulk-copy chunk kernel's dynamic shared memory limit once per
// device.
static int chunks_setup(int device) {
  static std::mutex mu;
  static bool done[64] = {};
  if (device < 0 || device >= 64) return fail(SF_ERR_UNSUPPORTED, "device ordinal %d", device);
  std::lock_guard<std::mutex> lock(mu);
  if (!done[device]) {
    const cudaError_t e = cudaFuncSetAttribute(accept_chunks_kernel<true>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, kChunkSmemBytes);
    if (e != cudaSuccess)
      return fail(SF_ERR_CUDA, "cudaFuncSetAttribute (accept chunks): %s", cudaGetErrorString(e));
    done[device] = true;
  }
  return SF_OK;
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
  if (sf::plan_accept(V, &plan) != SF_OK) return 0;
  return sf::acc_layout(B, k, plan).total;
}

int sf_accept_kernel_launches(int B, int k, int V) {
  using namespace sf;
  if (check_accept_shapes(B, k, V) != SF_OK) return 0;
  int cs = 0, slice = 0;
  bool cluster_ok = false;
  if (cluster_plan(V, &cs, &slice) && cluster_setup(cs, &cluster_ok) != SF_OK) return 0;
  return cluster_ok ? 1 : 2;
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
  st = plan_accept(V, &plan);
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
  prm.draw_tickets = reinterpret_cast<uint32_t *>(ws + lay.draw_tickets);
  prm.row_tickets = reinterpret_cast<uint32_t *>(ws + lay.row_tickets);
  prm.seq_tickets = reinterpret_cast<uint32_t *>(ws + lay.seq_tickets);
  prm.runs = reinterpret_cast<RowStat *>(ws + lay.runs);
  prm.rows = reinterpret_cast<RowStat *>(ws + lay.rows);
  prm.seqs = reinterpret_cast<SeqState *>(ws + lay.seqs);
  prm.parts = reinterpret_cast<DrawPart *>(ws + lay.parts);
  prm.B = B;
  prm.k = k;
  prm.V = V;
  prm.C1 = plan.C1;
  prm.C2 = plan.C2;
  prm.NW1 = 0;
  prm.vec4 = (V % 4 == 0) && aligned(target_logits, 16) && aligned(draft_probs, 16);

  // One cluster per sequence when a row fits 16 slices: a single launch
  int cs = 0, slice = 0;
  bool cluster_ok = false;
  if (cluster_plan(V, &cs, &slice)) {
    st = cluster_setup(cs, &cluster_ok);
    if (st != SF_OK) return st;
  }
  if (cluster_ok) {
    cudaLaunchAttribute cattr[2];
    cattr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    cattr[0].val.programmaticStreamSerializationAllowed = 1;
    cattr[1].id = cudaLaunchAttributeClusterDimension;
    cattr[1].val.clusterDim.x = cs;
    cattr[1].val.clusterDim.y = 1;
    cattr[1].val.clusterDim.z = 1;
    cudaLaunchConfig_t ccfg = {};
    ccfg.gridDim = dim3(cs, B);
    ccfg.blockDim = dim3(kAccThreads);
    ccfg.dynamicSmemBytes = sizeof(float) * slice;
    ccfg.stream = stream;
    ccfg.attrs = cattr;
    ccfg.numAttrs = 2;
    cudaError_t ce = cudaLaunchKernelEx(&ccfg, accept_cluster_kernel, prm, cs, slice);
    if (ce != cudaSuccess) return fail(SF_ERR_CUDA, "accept cluster launch: %s", cudaGetErrorString(ce));
    return SF_OK;
  }

  // Both kernels are launched with programmatic stream serialisation: each
  // may be scheduled while the previous kernel on the stream drains and
  // waits for it (griddepcontrol.wait) before writing or reading its results.
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  DeviceInfo dev;
  st = current_device(&dev);
  if (st != SF_OK) return st;
  // at most one warp per chunk, so that every warp owns at least one chunk
  // (a row's runs are then exactly the warps between its first and last
  // chunk's owners), and at most two CTAs per SM
  const long long units = (long long)B * (k + 1) * plan.C1;
  long long nw = units < 2LL * dev.sm_count * kAccWarps ? units : 2LL * dev.sm_count * kAccWarps;
  const long long ctas = (nw + kAccWarps - 1) / kAccWarps;
  prm.NW1 = static_cast<int>(nw);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(ctas));
  cfg.blockDim = dim3(kAccThreads);
  cfg.dynamicSmemBytes = prm.vec4 ? kChunkSmemBytes : 0;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (prm.vec4) {
    st = chunks_setup(dev.ordinal);
    if (st != SF_OK) return st;
  }
  cudaError_t e = prm.vec4 ? cudaLaunchKernelEx(&cfg, accept_chunks_kernel<true>, prm)
                           : cudaLaunchKernelEx(&cfg, accept_chunks_kernel<false>, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "accept chunks launch: %s", cudaGetErrorString(e));
  cfg.gridDim = dim3(plan.C2, B);
  cfg.dynamicSmemBytes = 0;
  e = cudaLaunchKernelEx(&cfg, accept_draw_kernel, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "accept draw launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

size_t sf_verify_lm_head_accept_workspace_size(int B, int k, int V) {
  using namespace sf;
  if (check_accept_shapes(B, k, V) != SF_OK || B * (k + 1) > SF_MAX_DRAFT_ROWS) return 0;
  AccPlan plan;
  if (plan_accept(V, &plan) != SF_OK) return 0;
  DeviceInfo dev;
  if (current_device(&dev) != SF_OK) return 0;
  const size_t G = static_cast<size_t>(projection_groups(V, dev.sm_count));
  return acc_layout(B, k, plan).total + round_up(sizeof(SampStat) * B * (k + 1) * G, 256);
}

int sf_verify_lm_head_accept(const void *hidden, const void *weight, const float *draft_probs,
                             const int32_t *draft_tokens, const float *uniforms,
                             const float *temperature, int B, int k, int V, int d, float *logits,
                             int32_t *num_accepted, int32_t *out_tokens, float *accept_ratio,
                             void *workspace, size_t workspace_bytes, cudaStream_t stream) {
  using namespace sf;
  clear_error();
  int st = check_accept_shapes(B, k, V);
  if (st != SF_OK) return st;
  if (B * (k + 1) > SF_MAX_DRAFT_ROWS)
    return fail(SF_ERR_INVALID_ARG, "B*(k+1)=%d above %d rows", B * (k + 1), SF_MAX_DRAFT_ROWS);
  if (!draft_probs || !draft_tokens || !uniforms || !temperature || !num_accepted || !out_tokens)
    return fail(SF_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!aligned(draft_probs, 4) || !aligned(draft_tokens, 4) || !aligned(uniforms, 4) ||
      !aligned(temperature, 4) || !aligned(num_accepted, 4) || !aligned(out_tokens, 4) ||
      (accept_ratio && !aligned(accept_ratio, 4)))
    return fail(SF_ERR_INVALID_ARG, "buffers must be 4-byte aligned");
  if (!workspace || !aligned(workspace, 256))
    return fail(SF_ERR_WORKSPACE, "workspace must be non-NULL and 256-byte aligned");
  AccPlan plan;
  st = plan_accept(V, &plan);
  if (st != SF_OK) return st;
  DeviceInfo dev;
  st = current_device(&dev);
  if (st != SF_OK) return st;
  const AccLayout lay = acc_layout(B, k, plan);
  const int R = B * (k + 1);
  const size_t G = static_cast<size_t>(projection_groups(V, dev.sm_count));
  const size_t need = lay.total + round_up(sizeof(SampStat) * R * G, 256);
  if (workspace_bytes < need)
    return fail(SF_ERR_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, need);

  uint8_t *ws = static_cast<uint8_t *>(workspace);
  SampStat *stats = reinterpret_cast<SampStat *>(ws + lay.total);
  int Gl = 0;
  // target logits and their per-CTA row statistics; row b*(k+1)+i uses tau_b
  st = launch_projection_stats(hidden, weight, R, d, V, logits, temperature, k + 1, stats,
                               reinterpret_cast<uint32_t *>(ws), &Gl, stream);
  if (st != SF_OK) return st;

  AccParams prm;
  prm.logits = logits;
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
  prm.runs = reinterpret_cast<RowStat *>(ws + lay.runs);
  prm.rows = reinterpret_cast<RowStat *>(ws + lay.rows);
  prm.seqs = reinterpret_cast<SeqState *>(ws + lay.seqs);
  prm.parts = reinterpret_cast<DrawPart *>(ws + lay.parts);
  prm.B = B;
  prm.k = k;
  prm.V = V;
  prm.C1 = plan.C1;
  prm.C2 = plan.C2;
  prm.NW1 = 0;
  prm.vec4 = (V % 4 == 0) && aligned(logits, 16) && aligned(draft_probs, 16);

  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(B);
  cfg.blockDim = dim3(kAccThreads);
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, accept_decide_kernel, prm,
                                     static_cast<const SampStat *>(stats), Gl);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "accept decide launch: %s", cudaGetErrorString(e));
  cfg.gridDim = dim3(plan.C2, B);
  e = cudaLaunchKernelEx(&cfg, accept_draw_kernel, prm);
  if (e != cudaSuccess) return fail(SF_ERR_CUDA, "accept draw launch: %s", cudaGetErrorString(e));
  return SF_OK;
}

}  // extern "C"
