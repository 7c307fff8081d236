/*
 * specflash_verify.h -- C ABI of the GB300 (sm_103a) verification step of
 * SpecFLASH speculative decoding (arXiv 2505.12728).
 *
 * The verification step has two parts (Sec. 3.1, "Preliminaries"; Sec. 3.3):
 *   1. the target model scores all K draft tokens together, in one forward
 *      pass: per layer, attention of the K new query rows over the cached
 *      (mostly visual) prefix plus the causal draft block
 *      (sf_verify_attention);
 *   2. the token-wise acceptance-rejection rule: candidate T'_i is kept with
 *      probability min(1, p_i/q_i), candidates after the first rejection are
 *      discarded, and the token at the rejected position is drawn from the
 *      residual distribution norm(max(0, p - q)); at temperature 0 (greedy
 *      decoding, Sec. 4.2) a candidate is kept iff it is the target argmax
 *      (sf_accept).
 *
 * Conventions for every entry point:
 *   - Pointers are DEVICE pointers unless stated otherwise.  The caller owns
 *     every buffer; the library never allocates, frees or synchronises, and
 *     enqueues its kernels on `stream` (0 = the legacy default stream).
 *   - Return value: SF_OK (0) or an sf_status code.  Argument errors are
 *     detected on the host before any launch; nothing is enqueued then.
 *     sf_last_error() gives a thread-local description of the last failure.
 *   - Data errors that only the device can see (a page index outside the
 *     pool, a draft token outside [0, V)) never fault: the offending access
 *     is replaced by a zero page / a rejection, and a bit is set in the
 *     status word at the start of the workspace (SF_DEVICE_* below), which
 *     sf_read_device_status() returns.
 *   - Workspaces must be zero-filled once before their first use
 *     (sf_workspace_init, or cudaMemset to 0).  The kernels leave their
 *     counters at zero on exit, so a workspace can be reused by later calls
 *     on the same stream; calls that overlap on the GPU must use distinct
 *     workspaces.  Re-initialise after a nonzero device status.
 *   - Results are deterministic: for fixed shapes, inputs and num_splits they
 *     are bit-identical from run to run (no floating-point atomics).
 *   - Stream order: kernels are launched with programmatic dependent launch,
 *     so each may start while the previous kernel on `stream` drains.  Before
 *     waiting for that kernel, sf_verify_attention reads the block table, the
 *     sequence lengths and the prefix part of the KV cache (positions below
 *     seq_lens[b] - n_q), and the LM-head projections read the weights;
 *     these, and the workspace, must already be in place when the previous
 *     kernel on the stream starts (so neither it nor a kernel it may overlap
 *     writes them).  Everything else (q, hidden states, the draft rows' K/V,
 *     logits, probabilities, tokens, uniforms, temperatures) may come from
 *     the previous kernel: every kernel waits for it before reading them.
 */
#ifndef SPECFLASH_VERIFY_H
#define SPECFLASH_VERIFY_H

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SF_OK = 0,
  SF_ERR_INVALID_ARG = 1,   /* bad shape, NULL pointer, misaligned buffer      */
  SF_ERR_UNSUPPORTED = 2,   /* valid but not built: head_dim, page size, ...   */
  SF_ERR_CUDA = 3,          /* a CUDA runtime/driver call failed               */
  SF_ERR_WORKSPACE = 4,     /* workspace NULL or smaller than required         */
  SF_ERR_DEVICE_STATUS = 5  /* the device status word is nonzero               */
} sf_status;

/* Bits of the device status word (first 4 bytes of every workspace). */
#define SF_DEVICE_BAD_PAGE 0x1u  /* block_table entry outside [0, num_pages)  */
#define SF_DEVICE_BAD_TOKEN 0x2u /* draft token outside [0, V)                */
#define SF_DEVICE_TIMEOUT 0x4u   /* a bounded wait on a copy gave up (~1 s)   */
#define SF_DEVICE_BAD_SEQLEN 0x8u /* seq_lens[b] outside [n_q, max_pages*16]   */
#define SF_DEVICE_OUT_OF_PAGES 0x10u /* sf_kv_commit: free-page stack too small */

/* Compile-time limits of the library (calls beyond them return an error). */
#define SF_PAGE_SIZE 16      /* tokens per KV page                            */
#define SF_MAX_BATCH 1024    /* sequences per call                            */
#define SF_MAX_QUERY_ROWS 16 /* n_q: draft rows scored per sequence           */
#define SF_MAX_GROUP 8       /* H_q / H_kv                                    */
#define SF_MAX_DRAFT 16      /* k: draft length                               */
#define SF_MAX_DRAFT_ROWS 256 /* R: rows of one LM-head projection            */
#define SF_MAX_VOCAB 8388608  /* V for sf_lm_head / sf_sample / sf_draft_sample */

/* Static string naming a status code. */
const char *sf_status_string(int status);

/* Thread-local, human-readable detail of the last failing call ("" if none). */
const char *sf_last_error(void);

/* Library version: major * 10000 + minor * 100 + patch. */
int sf_version(void);

/* Zero-fill `bytes` of `workspace` on `stream` (asynchronous). */
int sf_workspace_init(void *workspace, size_t bytes, cudaStream_t stream);

/* Synchronously read the device status word of a workspace (tests and
 * diagnostics only: it waits for all work on the device).  On success
 * *status_out holds the SF_DEVICE_* bits; returns SF_OK or SF_ERR_CUDA. */
int sf_read_device_status(const void *workspace, uint32_t *status_out);

/* Self-test of the bounded waits (diagnostics): launches one CTA whose      */
/* thread waits on an mbarrier that nothing completes.  The wait gives up    */
/* after about one second (the budget of every wait in these kernels) and    */
/* sets SF_DEVICE_TIMEOUT in the status word at the start of `workspace`     */
/* (>= 4 bytes, 4-byte aligned); the context stays usable.  Returns SF_OK or */
/* SF_ERR_WORKSPACE / SF_ERR_CUDA; asynchronous on `stream`.                 */
int sf_selftest_bounded_wait(void *workspace, size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* Verification attention (Sec. 3.1: the K candidates' probabilities come  */
/* from one parallel forward pass of the target model; the verify costs     */
/* about one target step, Eq. 1).                                            */
/*                                                                           */
/* For each sequence b, draft row i < n_q and query head h (KV head          */
/* h / (H_q / H_kv)): the visible keys are the L_b = seq_lens[b] - n_q       */
/* cached prefix tokens (visual first, then text) plus draft rows 0..i,      */
/* s_t = softmax_scale * <q, k_t>, lse = ln sum_t exp(s_t),                  */
/* out = sum_t exp(s_t - lse) * v_t.                                         */
/*                                                                           */
/* q            bf16 [B][n_q][H_q][head_dim], already position-encoded.      */
/* k_cache      bf16 [num_pages][H_kv][page_size][head_dim]; 16-byte aligned */
/* v_cache      bf16, same layout as k_cache.                                */
/* block_table  int32 [B][max_pages_per_seq]: logical page -> physical page. */
/*              Entries past a sequence's last page are never read.          */
/* seq_lens     int32 [B]: L_b + n_q, the draft rows' K/V already written at */
/*              positions L_b..L_b+n_q-1.  Must satisfy                      */
/*              n_q <= seq_lens[b] <= max_pages_per_seq * page_size; values  */
/*              outside are clamped and flagged with SF_DEVICE_BAD_SEQLEN.   */
/* head_dim     64 or 128; page_size 16; 1 <= n_q <= 16; H_q % H_kv == 0,    */
/*              H_q / H_kv <= 8; 1 <= B <= 1024.                             */
/* softmax_scale  0 selects 1/sqrt(head_dim).                                */
/* num_splits   number of cooperating CTAs the batch's KV tiles are divided */
/*              among (at most 65535); 0 picks the grid from the SM count    */
/*              (and, for one sequence, one thread-block cluster per KV      */
/*              head).  With more than 16 rows per KV head                   */
/*              (n_q * H_q / H_kv > 16) the tcgen05 kernel runs one CTA per  */
/*              SM and uses min(num_splits, SM count) CTAs.  The result      */
/*              depends on it only through rounding.                         */
/* out          bf16 [B][n_q][H_q][head_dim].                                */
/* lse          fp32 [B][n_q][H_q] (natural log, scaled scores); may be NULL.*/
/* workspace    >= sf_verify_attention_workspace_size(...) bytes, 256-byte   */
/*              aligned, zero-filled before first use.                       */
/* Accuracy: scores and softmax statistics in fp32; P V on bf16 tensor cores */
/* with P carried as two bf16 terms on each sequence's first 64-token tile   */
/* and as one on later tiles.  Against the exact result, out is within 1e-2  */
/* (bf16 rounding of out included, for |out| < 4) and lse within 1e-3 on the */
/* tested inputs (N(0,1) q, k, v in bf16, 1 to 32K keys).                    */
/* ------------------------------------------------------------------------ */
size_t sf_verify_attention_workspace_size(int B, int n_q, int H_q, int H_kv, int head_dim,
                                          int max_pages_per_seq, int page_size,
                                          int num_splits);

int sf_verify_attention(const void *q, const void *k_cache, const void *v_cache,
                        const int32_t *block_table, const int32_t *seq_lens, int B, int n_q,
                        int H_q, int H_kv, int head_dim, int page_size, int num_pages,
                        int max_pages_per_seq, float softmax_scale, int num_splits, void *out,
                        float *lse, void *workspace, size_t workspace_bytes,
                        cudaStream_t stream);

/* Kernels one sf_verify_attention call with these shapes launches on the    */
/* current device: 1 (at most 16 rows per KV head: the split kernel merges  */
/* in place) or 2 (the tcgen05 split kernel, then the merge kernel); 0 for   */
/* shapes sf_verify_attention rejects or without a usable CUDA device       */
/* (sf_last_error says which).  For graph and launch planning.              */
int sf_verify_attention_kernel_launches(int B, int n_q, int H_q, int H_kv, int head_dim,
                                        int max_pages_per_seq, int page_size, int num_splits);

/* ------------------------------------------------------------------------ */
/* Verification attention without a caller workspace.  The paper has no      */
/* counterpart: this is a deployment convenience of this library.            */
/*                                                                           */
/* For callers that cannot allocate device memory when they verify: a        */
/* serving runtime whose memory manager owns the whole device and refuses    */
/* allocations mid-request, a plug-in that receives only its input and       */
/* output buffers, or a runtime with a memory budget fixed before serving.   */
/* Same arguments and results as sf_verify_attention, minus the workspace:   */
/* the library uses its own scratch, a 16 MiB device array that exists on    */
/* every GPU that loads the library until the process exits.  Shapes whose   */
/* workspace (sf_verify_attention_workspace_size) exceeds 16 MiB are         */
/* rejected with SF_ERR_UNSUPPORTED before anything is enqueued.             */
/* The call allocates nothing: it clears the scratch's counters with         */
/* cudaMemsetAsync on `stream`, then launches the kernel.                    */
/* Its first call on a device looks up the scratch's device address (once    */
/* per device, cached); make that first call before any stream capture.      */
/* The cached address lives as long as the process: resetting a device       */
/* (cudaDeviceReset) after this entry point has used it is not supported.    */
/* Every argument check runs before the scratch is touched: a rejected call  */
/* enqueues nothing.                                                          */
/* All calls share the one scratch array, which keeps the previous call's    */
/* contents: calls that may overlap on the GPU (different streams, or        */
/* threads without ordering) race and give wrong results; serialise them.    */
/* Device data errors never fault here either, but their status bits stay   */
/* in the library's scratch; use sf_verify_attention to read them.           */
/* ------------------------------------------------------------------------ */
int sf_verify_attention_noalloc(const void *q, const void *k_cache, const void *v_cache,
                                const int32_t *block_table, const int32_t *seq_lens, int B,
                                int n_q, int H_q, int H_kv, int head_dim, int page_size,
                                int num_pages, int max_pages_per_seq, float softmax_scale,
                                int num_splits, void *out, float *lse, cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* Acceptance (Sec. 3.1: acceptance probability as the ratio of target to    */
/* draft probability, discard from the first rejection on, resample from the */
/* residual distribution; Sec. 3.3: "the standard token-wise acceptance-     */
/* rejection rule"; Sec. 4.2: tau = 0 is greedy decoding).                   */
/*                                                                           */
/* target_logits fp32 [B][k+1][V]: row i < k scores draft T'_{i+1}; row k is */
/*               the bonus row used when all k drafts are accepted.          */
/* draft_probs   fp32 [B][k][V]: draft distributions q_i, used as given.     */
/* draft_tokens  int32 [B][k].                                               */
/* uniforms      fp32 [B][k+1] in [0,1): u_i for test i, u_k for the draw.   */
/* temperature   fp32 [B]: p = softmax(logits / tau); tau <= 0 selects       */
/*               greedy matching for that sequence (mixed batches allowed).  */
/* num_accepted  int32 [B] in [0, k].                                        */
/* out_tokens    int32 [B][k+1]: the accepted drafts, then the corrected     */
/*               (or bonus) token; entries past num_accepted are -1.         */
/* accept_ratio  fp32 [B][k] = min(1, p_i(T'_i)/q_i(T'_i)) for every i      */
/*               (greedy: 1 on a match, else 0); may be NULL.                */
/* Rule details: accept iff u_i * q < p (strict); greedy ties go to the      */
/* lowest token id; a residual with zero mass falls back to p_j; the draw is */
/* the smallest token x with u_k * S < C(x) in ascending token order.        */
/* Limits: 1 <= B <= 1024, 1 <= k <= 16, 2 <= V < 2^31 / (k + 1).            */
/* ------------------------------------------------------------------------ */
size_t sf_accept_workspace_size(int B, int k, int V);

/* Kernels one sf_accept call with these shapes launches on the current      */
/* device: 1 (a row fits one 16-CTA thread-block cluster, V <= 32768, and    */
/* such a cluster can be resident) or 2 (statistics and decisions, then the  */
/* draw); 0 for shapes sf_accept rejects or without a usable CUDA device     */
/* (sf_last_error says which).  For graph and launch planning.              */
int sf_accept_kernel_launches(int B, int k, int V);

int sf_accept(const float *target_logits, const float *draft_probs,
              const int32_t *draft_tokens, const float *uniforms, const float *temperature,
              int B, int k, int V, int32_t *num_accepted, int32_t *out_tokens,
              float *accept_ratio, void *workspace, size_t workspace_bytes,
              cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* Fused target LM head + acceptance (Sec. 3.1: the target scores the K     */
/* candidates in one forward pass; its LM head turns the k+1 verified       */
/* positions' final hidden states into the logits the rule above reads).   */
/* target_logits[b][i][v] = sum_j hidden[b][i][j] * weight[v][j] (bf16 in,  */
/* fp32 accumulate), then exactly the rule of sf_accept, with the rows'     */
/* max, argmax and softmax sums reduced in the projection's epilogue        */
/* instead of a second pass over the logits.                                */
/*                                                                           */
/* hidden        bf16 [B][k+1][d], 16-byte aligned.                          */
/* weight        bf16 [V][d] (the target's LM head), 16-byte aligned.        */
/* logits        fp32 [B][k+1][V], output (also read by the draw).           */
/* other arguments and outputs as for sf_accept.                             */
/* Limits: those of sf_accept, B * (k + 1) <= 256, d a multiple of 8 in    */
/* [8, 2^20].  workspace >= sf_verify_lm_head_accept_workspace_size(B, k, V)*/
/* bytes, 256-byte aligned, zero-filled before first use.                   */
/* The weight copies start before the previous kernel on the stream        */
/* completes (the weights must be in place when that kernel starts).        */
/* ------------------------------------------------------------------------ */
size_t sf_verify_lm_head_accept_workspace_size(int B, int k, int V);

int sf_verify_lm_head_accept(const void *hidden, const void *weight, const float *draft_probs,
                             const int32_t *draft_tokens, const float *uniforms,
                             const float *temperature, int B, int k, int V, int d, float *logits,
                             int32_t *num_accepted, int32_t *out_tokens, float *accept_ratio,
                             void *workspace, size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* KV commit after acceptance (Sec. 3.1: the accepted candidates join the    */
/* context and decoding continues from the first rejected position; Sec.    */
/* 3.3: the next draft block starts from the emitted token).  The paper      */
/* gives no cache mechanics; this call keeps a paged cache consistent on the */
/* device, with no host round trip, between two verification steps.         */
/*                                                                           */
/* For each sequence b, with a = num_accepted[b] (from sf_accept): of the    */
/* n_q rows verified at cache positions L_b .. L_b + n_q - 1                 */
/* (L_b = seq_lens[b] - n_q), the first keep = min(a + 1, n_q) stay -- row i */
/* holds the i-th token of the verified block, whose first token is the one  */
/* emitted by the previous step -- and the rest are dropped.  The next step  */
/* verifies n_q_next rows written at L_b + keep ..:                           */
/*   seq_lens[b] <- L_b + keep + n_q_next,                                   */
/* and the block table maps exactly need_b = ceil(seq_lens[b] / 16) logical  */
/* pages (it mapped ceil(old seq_lens[b] / 16) before):                      */
/*   1. pages no longer needed are pushed onto the free-page stack, in       */
/*      sequence order and ascending logical page, and their entries set to  */
/*      -1;                                                                  */
/*   2. missing pages are then taken from the topmost stack entries, assigned */
/*      bottom-up in sequence order and ascending logical page.              */
/* Deterministic; all or nothing: if any seq_lens[b] < n_q, num_accepted[b]  */
/* < 0 or need_b > max_pages_per_seq, SF_DEVICE_BAD_SEQLEN is set, and if the */
/* stack would run out of pages or overflow `capacity`,                      */
/* SF_DEVICE_OUT_OF_PAGES is set; in both cases nothing is modified.         */
/*                                                                           */
/* seq_lens      int32 [B], in/out.                                          */
/* block_table   int32 [B][max_pages_per_seq], in/out.                       */
/* free_pages    int32 [capacity], in/out: entries [0, *free_count) are free  */
/*               physical page ids (a stack, top at the end).                */
/* free_count    int32 [1], in/out (device memory).                          */
/* num_accepted  int32 [B] in [0, k].                                        */
/* B <= 1024; 1 <= n_q, n_q_next <= 16; page_size 16.                        */
/* workspace     >= sf_kv_commit_workspace_size() bytes, 256-byte aligned,   */
/*               zero-filled before first use (status word).                 */
/* The next sf_verify_attention reads seq_lens and the block table before    */
/* waiting for the kernel that precedes it on the stream, so that kernel must */
/* not be this one (in a decoding loop the K/V append of the next draft rows */
/* comes in between).                                                        */
/* ------------------------------------------------------------------------ */
size_t sf_kv_commit_workspace_size(void);

int sf_kv_commit(int32_t *seq_lens, int32_t *block_table, int32_t *free_pages,
                 int32_t *free_count, const int32_t *num_accepted, int B, int n_q, int n_q_next,
                 int max_pages_per_seq, int page_size, int capacity, void *workspace,
                 size_t workspace_bytes, cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* Draft-distribution tail (Sec. 3.3, Algorithm 1: the semi-autoregressive   */
/* head's outputs for the K draft positions pass through the frozen LM head; */
/* the K candidates are then sampled from the resulting distributions       */
/* independently).  These calls produce the draft_probs / draft_tokens that  */
/* sf_accept consumes (rows R = B * k, row b * k + i for draft position i). */
/*                                                                           */
/* sf_lm_head:  logits[r][v] = sum_j hidden[r][j] * weight[v][j], bf16       */
/*              inputs, fp32 accumulation (tensor cores), fp32 output.       */
/* sf_sample:   for each row r, with tau = temperature[r]:                   */
/*              probs[r] = softmax(logits[r] / tau), and tokens[r] = the     */
/*              smallest token x with uniforms[r] * S < C(x), where C is the */
/*              cumulative sum of exp(logits/tau - max) in ascending token   */
/*              order and S its total; tau <= 0 (or NaN) selects greedy      */
/*              decoding: tokens[r] = the first argmax, probs[r] one-hot.    */
/*              Tokens at -inf get probability 0.  Where rounding leaves no  */
/*              token past the target (uniforms[r] >= 1 or NaN), the last    */
/*              token of positive probability is taken.                      */
/* sf_draft_sample: sf_lm_head then sf_sample, with the per-row max and sum  */
/*              reduced in the projection's epilogue, so the logits are read */
/*              once more (for probs) instead of three times.                */
/*                                                                           */
/* hidden       bf16 [R][hidden_size], 16-byte aligned.                      */
/* weight       bf16 [V][hidden_size] (the LM head), 16-byte aligned.        */
/*              hidden_size a multiple of 8 in [8, 2^20]; 1 <= R <= 256      */
/*              (sf_sample alone: R <= 65535); 1 <= V <= SF_MAX_VOCAB.       */
/* logits       fp32 [R][V]: output of sf_lm_head / sf_draft_sample, input   */
/*              of sf_sample.                                                */
/* uniforms     fp32 [R] in [0, 1).   temperature  fp32 [R].                 */
/* probs        fp32 [R][V].          tokens       int32 [R].                */
/* workspace    >= sf_draft_tail_workspace_size(R, V) bytes, 256-byte        */
/*              aligned, zero-filled before first use (status word).        */
/* Stream order: the projection copies weight tiles before waiting for the   */
/* previous kernel on the stream (the weights must be in place when that     */
/* kernel starts); hidden, temperature, uniforms and the outputs follow it.  */
/* Results are deterministic; SF_DEVICE_TIMEOUT is the only device status.   */
/* ------------------------------------------------------------------------ */
size_t sf_draft_tail_workspace_size(int R, int V);

int sf_lm_head(const void *hidden, const void *weight, int R, int hidden_size, int V,
               float *logits, void *workspace, size_t workspace_bytes, cudaStream_t stream);

int sf_sample(const float *logits, const float *uniforms, const float *temperature, int R, int V,
              float *probs, int32_t *tokens, void *workspace, size_t workspace_bytes,
              cudaStream_t stream);

int sf_draft_sample(const void *hidden, const void *weight, const float *uniforms,
                    const float *temperature, int R, int hidden_size, int V, float *logits,
                    float *probs, int32_t *tokens, void *workspace, size_t workspace_bytes,
                    cudaStream_t stream);

/* ------------------------------------------------------------------------ */
/* Visual token compression of the draft model (Sec. 3.2, Eq. 3; Algorithm */
/* 1): each image or video frame's N visual features F_V (the target's      */
/* second-to-top layer) are compressed to C features with the learnable     */
/* query set Q, F_V serving as keys and values:                             */
/*     out[f] = softmax(Q F_V[f]^T) F_V[f],                                 */
/* the softmax over the frame's N tokens for each query, scores unscaled.  */
/*                                                                           */
/* queries   bf16 [C][d], 16-byte aligned.                                  */
/* features  bf16 [F][N][d], 16-byte aligned.                               */
/* out       bf16 [F][C][d], 16-byte aligned.                               */
/* Limits: 1 <= F <= 65535, 1 <= N <= 768, 1 <= C <= 128, d a multiple of   */
/* 128 in [128, 2^20], F * N <= SF_MAX_VOCAB.                               */
/* workspace >= sf_visual_compress_workspace_size(F, N, C, d) bytes (fp32  */
/*           partial scores, bf16 weights, their sums), 256-byte aligned,   */
/*           zero-filled before first use (status word).                    */
/* Three launches; each copies its inputs only after the previous kernel on */
/* the stream completes.  Deterministic; SF_DEVICE_TIMEOUT is the only      */
/* device status.                                                            */
/* ------------------------------------------------------------------------ */
size_t sf_visual_compress_workspace_size(int F, int N, int C, int d);

int sf_visual_compress(const void *queries, const void *features, int F, int N, int C, int d,
                       void *out, void *workspace, size_t workspace_bytes, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SPECFLASH_VERIFY_H */
