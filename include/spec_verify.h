/*
 * spec_verify.h -- C ABI of the GB300 (sm_103a) verify step of lossless
 * diffusion-drafted decoding ("Unlocking Lossless Speedups in LLMs via Discrete
 * Diffusion": Psi-Spec, Sec. 4 and Appendix B.3).
 *
 * In one decode step, the drafter proposes a block of gamma tokens
 * [x^{L+1}, x~^1 .. x~^{gamma-1}] (gamma is the paper's block size B), and the
 * autoregressive verifier scores the whole block in one forward pass. This library
 * implements the two data-parallel parts of that verify step:
 *   (a) block-causal attention of the gamma block queries against a paged bf16 KV
 *       cache with grouped-query heads (spec_verify_attention);
 *   (b) the vocabulary-wide softmax of target and drafter logits and the lossless
 *       acceptance rule: accept draft i with probability min(1, p_i/q_i), on the
 *       first rejection n draw from Norm([p_n - q_n]_+), otherwise draw the bonus
 *       token from p_B; at temperature 0, greedy argmax matching
 *       (spec_accept_block).
 * spec_verify_step runs both on one stream.
 *
 * Conventions shared by every entry point
 *   - Every tensor argument is a DEVICE pointer owned by the caller, row-major and
 *     densely packed in the layout stated beside it. The library allocates no device
 *     memory and never synchronizes the stream (except spec_read_device_status).
 *     Calls are asynchronous on `stream`.
 *   - Each call makes the device of `stream` current while it runs and restores the
 *     calling thread's current device before it returns.
 *   - State kept between calls: cached SM counts, the driver's tensor-map encoder,
 *     and, for the fused steps only, one side stream with two events per (host
 *     thread, device, caller stream), at most 16 per thread (the least recently
 *     used one that is not under capture is released to make room). Calls on
 *     different streams never wait for each other's work.
 *   - `ws` is a caller-owned device workspace of at least spec_workspace_size()
 *     bytes, 256-byte aligned. A new workspace must be zero-filled once (e.g.
 *     spec_workspace_init); every call leaves its internal counters at zero again.
 *     Concurrent calls need distinct workspaces. A workspace holds the counters of
 *     one call configuration (the entry point, which of its parts are given, and
 *     their sizes): calls of another configuration lay their scratch data out
 *     differently and may leave non-zero words where this one keeps counters, so
 *     give each configuration its own workspace, or zero-fill it again when
 *     switching (CUDA graphs captured for different configurations included).
 *   - Host-side argument checks happen before any launch and return
 *     SPEC_ERR_INVALID_ARGUMENT / SPEC_ERR_UNSUPPORTED / SPEC_ERR_WORKSPACE_TOO_SMALL
 *     without touching the device. Launch failures return SPEC_ERR_CUDA.
 *   - Bad device-resident data (a token id outside [0, vocab), a page id outside
 *     [0, num_pages), kv_len outside [gamma, max_pages_per_seq * page_size], NaN or
 *     +inf logits) never traps: the kernels set a bit in the workspace status word
 *     (SPEC_FLAG_*), write the documented sentinel outputs for the affected
 *     sequence, and carry on. spec_read_device_status reads and clears the word.
 *   - Kernels never wait on other thread blocks; every internal wait on an
 *     asynchronous copy or tensor-core operation is bounded, and a timeout sets
 *     SPEC_FLAG_TIMEOUT instead of hanging.
 */
#ifndef SPEC_VERIFY_H
#define SPEC_VERIFY_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A cudaStream_t (the runtime's stream handle); NULL is the legacy default stream. */
typedef struct CUstream_st* spec_stream_t;

typedef enum {
  SPEC_OK = 0,
  SPEC_ERR_INVALID_ARGUMENT = 1,  /* null pointer, non-positive size, inconsistent shape   */
  SPEC_ERR_UNSUPPORTED = 2,       /* a shape outside the supported limits below            */
  SPEC_ERR_WORKSPACE_TOO_SMALL = 3,
  SPEC_ERR_CUDA = 4,              /* a CUDA runtime/driver call or a launch failed          */
  SPEC_ERR_DEVICE_INPUT = 5,      /* spec_read_device_status found SPEC_FLAG_BAD_* bits    */
  SPEC_ERR_TIMEOUT = 6            /* spec_read_device_status found SPEC_FLAG_TIMEOUT       */
} spec_status_t;

typedef enum { SPEC_F32 = 0, SPEC_BF16 = 1 } spec_dtype_t;

/* Attention kernel selection (spec_attn_args_t.path). */
typedef enum {
  SPEC_ATTN_AUTO = 0,          /* tensor cores when (Hq/Hkv)*gamma >= the crossover, else CUDA cores */
  SPEC_ATTN_CUDA_CORES = 1,    /* fp32 CUDA-core kernel                                  */
  SPEC_ATTN_TENSOR_CORES = 2,  /* tcgen05 (TMEM accumulators, TMA-staged KV pages), the
                                  row-tile kernel (M = 128 query rows per tile); with 33
                                  to 64 query rows per KV head and an even Hkv (batch <=
                                  407 for head_dim 128) one block serves two adjacent KV
                                  heads, reading 8 KB page boxes                          */
  SPEC_ATTN_TENSOR_CORES_KEYS_ON_LANES = 3  /* tcgen05 with the keys of a tile on the MMA's
                                  M dimension (S^T = K Q^T, O^T = V^T P^T), where it applies
                                  (head_dim 128, at most 64 query rows per KV head, 64 %
                                  group == 0, batch <= 2048, no tree mask), else as 2; same
                                  results within the tolerance. Measured slower than 2 on
                                  GB300 at the named workloads, so AUTO does not pick it */
} spec_attn_path_t;

/* Device status word bits. */
#define SPEC_FLAG_BAD_TOKEN 0x1u   /* a block token outside [0, vocab)                      */
#define SPEC_FLAG_BAD_LOGITS 0x2u  /* a used logits row with NaN, +inf, or no finite entry */
#define SPEC_FLAG_BAD_PAGE 0x4u    /* a page id of a visible key outside [0, num_pages)      */
#define SPEC_FLAG_BAD_KV_LEN 0x8u  /* kv_len outside [gamma, max_pages_per_seq * page_size] */
#define SPEC_FLAG_TIMEOUT 0x10u    /* a bounded internal wait ran out                        */
#define SPEC_FLAG_BAD_FILTER 0x20u /* a tempered sequence's top_k or top_p out of range       */
#define SPEC_FLAG_BAD_TREE 0x40u   /* a candidate tree whose parents are not a tree          */

/*
 * Part (a): block-causal verify attention (Sec. 4.1: the block [x^{L+1}, z] is
 * processed while the prefix stays in the KV cache; Alg. "Lossless Psi-Spec":
 * p <- x_theta([x^{L+1}, x~]; x) is one causal pass over the block).
 *
 * For sequence b, kv_len[b] = ctx_b + gamma keys are in the cache: the prefix at
 * positions 0 .. ctx_b-1 and the block's own keys at ctx_b .. ctx_b+gamma-1 (already
 * written). Block query j of head h attends to keys k <= ctx_b + j of KV head
 * h / (num_q_heads / num_kv_heads):
 *   out[b][j][h] = sum_k softmax_k(scale * q.k_k) v_k,
 *   lse[b][j][h] = log sum_k exp(scale * q.k_k)       (natural log).
 * Logical key k lives in physical page page_table[b][k / page_size], slot
 * k % page_size. Accumulation is fp32; out is rounded to bf16.
 * A sequence flagged BAD_PAGE or BAD_KV_LEN gets out = 0 and lse = -inf.
 *
 * Tree attention (Sec. 4.2: several candidates are verified in one pass, arranged as a
 * prefix tree under tree attention): with tree_mask set, the gamma block positions are
 * the nodes of a candidate tree, and block query j sees the prefix keys k < ctx_b and
 * the block keys ctx_b + i for every bit i set in tree_mask[b][j] (itself and its
 * ancestors) instead of every k <= ctx_b + j. A mask with bits 0..j set is the causal
 * block. Device memory, caller-owned; gamma <= 64.
 */
typedef struct {
  int32_t batch;              /* >= 1                                                       */
  int32_t gamma;              /* block size, 1 .. 64                                        */
  int32_t num_q_heads;        /* Hq, a multiple of num_kv_heads                             */
  int32_t num_kv_heads;       /* Hkv                                                        */
  int32_t head_dim;           /* D: 64 or 128                                               */
  int32_t page_size;          /* 16, 32 or 64 tokens                                        */
  int32_t max_pages_per_seq;  /* page_table row length                                      */
  int32_t num_pages;          /* physical pages in k_cache / v_cache                        */
  float softmax_scale;        /* 0 => 1/sqrt(head_dim)                                      */
  int32_t path;               /* spec_attn_path_t                                           */
  const void* q;              /* bf16 [batch][gamma][Hq][D]                                 */
  const void* k_cache;        /* bf16 [num_pages][Hkv][page_size][D], 16-byte aligned       */
  const void* v_cache;        /* bf16 [num_pages][Hkv][page_size][D], 16-byte aligned       */
  const int32_t* page_table;  /* [batch][max_pages_per_seq]; entries past the sequence unread */
  const int32_t* kv_len;      /* [batch]                                                    */
  void* out;                  /* bf16 [batch][gamma][Hq][D]                                 */
  float* lse;                 /* fp32 [batch][gamma][Hq], or NULL                           */
  const uint64_t* tree_mask;  /* [batch][gamma], or NULL: tree attention (below)           */
} spec_attn_args_t;

/*
 * Part (b): lossless acceptance (Alg. "Lossless Psi-Spec decoding (Linear
 * Sampler)", the steps after the verifier pass; Sec. 4.2).
 *
 * Row conventions (gamma = B): target row j is the verifier's distribution of block
 * token j+1, so the algorithm's p_i is target row i-1 and the bonus row p_B is row
 * gamma-1; drafter row j is the distribution block token j was drawn from, so q_i is
 * drafter row i (drafter row 0 is never read). With T = temperature[b] > 0,
 * p = softmax(target / T), q = softmax(drafter / T), and
 *   n = min({i in 1..gamma-1 : uniforms[b][i-1] > min(1, p_i(t_i) / q_i(t_i))} U {gamma});
 * the final token is the smallest x with C(x) >= uniforms[b][gamma-1] * C(vocab-1),
 * C the ascending-token cumulative sum of p_B (n = gamma) or of [p_n - q_n]_+.
 * With T = 0 (greedy): n = the first i whose token is not the lowest-index argmax of
 * target row i-1, and the final token is that argmax of target row n-1.
 *
 * The classic speculative-decoding convention (k drafts d_1..d_k drawn from q_1..q_k,
 * k + 1 target rows p_1..p_{k+1}, the last one the bonus) is this call with
 * gamma = k + 1: block tokens [the last emitted token, d_1, .., d_k], target rows
 * p_1..p_{k+1}, drafter rows [any row, q_1, .., q_k] (row 0 is never read, so it may
 * hold anything, even NaN), uniforms [u_1, .., u_k, u_draw]; out_tokens[0] echoes the
 * last emitted token and num_accepted counts accepted drafts.
 * Outputs: out_tokens[b] = [t_0, t_1 .. t_{n-1}, final, -1 ...] (gamma+1 entries),
 * num_accepted[b] = n - 1 in [0, gamma-1], num_emitted[b] = n + 1 in [2, gamma+1].
 * A sequence flagged BAD_TOKEN or BAD_LOGITS gets num_accepted = -1,
 * num_emitted = 0 and out_tokens = -1.
 */
typedef struct {
  int32_t batch;               /* >= 1                                                      */
  int32_t gamma;               /* 1 .. 64                                                   */
  int32_t vocab;               /* >= 1                                                      */
  int32_t logits_dtype;        /* spec_dtype_t                                              */
  const void* target_logits;   /* [batch][gamma][vocab]                                     */
  const void* drafter_logits;  /* [batch][gamma][vocab]; row 0 of each sequence unread      */
  const int32_t* block_tokens; /* [batch][gamma]: t_0 = x^{L+1}, t_1.. = drafts            */
  const float* temperature;    /* [batch]; 0 => greedy                                      */
  const float* uniforms;       /* [batch][gamma] in (0, 1]; [i-1] tests draft i, [gamma-1] draws the final token */
  int32_t* num_accepted;       /* [batch]                                                   */
  int32_t* out_tokens;         /* [batch][gamma+1]                                          */
  int32_t* num_emitted;        /* [batch]                                                   */
  float* diag;                 /* [batch][gamma][2] = (p_i(t_i), q_i(t_i)) for the decisions
                                  taken (entry 0 = (0, 0); untaken = NaN; greedy: (match, 1);
                                  a sequence with bad input: all NaN), or NULL              */
} spec_accept_args_t;

/* Bytes of workspace the calls below need for these arguments (either may be NULL). */
size_t spec_workspace_size(const spec_attn_args_t* attn, const spec_accept_args_t* accept);

/* Zero-fills a workspace (cudaMemsetAsync on `stream`). */
spec_status_t spec_workspace_init(void* ws, size_t ws_bytes, spec_stream_t stream);

/* Part (a) alone. */
spec_status_t spec_verify_attention(const spec_attn_args_t* attn, void* ws, size_t ws_bytes,
                                    spec_stream_t stream);

/* Part (b) alone. */
spec_status_t spec_accept_block(const spec_accept_args_t* accept, void* ws, size_t ws_bytes,
                                spec_stream_t stream);

/* The whole verify step: parts (a) and (b), ordered on `stream` (they share no data:
 * the logits are inputs). Either argument may be NULL to run only the other part. With
 * both, part (b) runs on a second stream that belongs to the calling host thread and
 * to `stream` (created on the first such call) between a fork event recorded on
 * `stream` and a join event that `stream` waits for, so the two parts overlap; this
 * also holds under stream capture. Steps issued on different streams therefore never
 * wait for each other. The filtered step (spec_verify_step_filtered) does the same. */
spec_status_t spec_verify_step(const spec_attn_args_t* attn, const spec_accept_args_t* accept,
                               void* ws, size_t ws_bytes, spec_stream_t stream);

/*
 * Seeded uniforms for the acceptance rule (Alg. "Lossless Psi-Spec": r ~ U[0,1]).
 * out_dev[i] = ((x >> 8) + 1) * 2^-24 in (0, 1], x = word (offset+i) & 3 of
 * Philox4x32-10 (Salmon et al., SC'11) with key (seed low, seed high) and counter
 * ((offset+i) >> 2 low, high, 0, 0). n >= 0; out_dev is fp32 device memory.
 */
spec_status_t spec_philox_uniforms(uint64_t seed, uint64_t offset, int64_t n, float* out_dev,
                                   spec_stream_t stream);

/* Synchronizes `stream`, reads the workspace status word into *flags_out and clears
 * it. Returns SPEC_ERR_TIMEOUT if SPEC_FLAG_TIMEOUT is set, SPEC_ERR_DEVICE_INPUT if
 * another flag is set, else SPEC_OK. */
spec_status_t spec_read_device_status(void* ws, spec_stream_t stream, uint32_t* flags_out);

/* A static, human-readable name of a status code. */
const char* spec_status_string(spec_status_t status);

/* The (Hq/Hkv)*gamma at and above which SPEC_ATTN_AUTO picks the tensor-core kernel. */
int32_t spec_attn_tensor_core_min_rows(void);

/*
 * Filtered acceptance: spec_accept_block with top-k / top-p filtering of both
 * distributions, the sampling of the paper's evaluations (top-k 50 and top-p 0.95 for
 * drafting and verification: Sec. 5.1, Sec. 5.2, Appendix C.1).
 *
 * For a tempered sequence b (temperature[b] > 0), every target row and every used
 * drafter row is replaced by its filtered form before the rule: rank the tokens by
 * logit, equal logits by lower token id; keep the first k = min(top_k[b], vocab);
 * of those, keep the shortest rank-order prefix whose mass under their renormalised
 * distribution reaches top_p[b] (top_p = 1 keeps all k); renormalise over the kept
 * tokens; every other token has probability 0. The rule of spec_accept_block then runs
 * on the filtered p' and q', with one addition: a draft with q'_i(t_i) = 0 (outside
 * the filtered proposal) is accepted iff p'_i(t_i) > 0. The final draw is over the
 * kept tokens of p'_n in ascending token order. Drafts should be drawn from q' for
 * the output to follow the filtered target exactly. Greedy sequences (T = 0) are
 * verified as by spec_accept_block; their top_k / top_p are not read.
 *   - accept: as spec_accept_block (same layouts, outputs and sentinels); diag holds
 *     (p'_i(t_i), q'_i(t_i)).
 *   - filter->top_k: int32 [batch], device; 1 <= top_k[b] <= filter->max_top_k.
 *   - filter->top_p: fp32 [batch], device; 0 < top_p[b] <= 1.
 *   - filter->max_top_k: host bound on top_k, 1 .. SPEC_FILTER_MAX_TOP_K; it sizes
 *     the workspace (spec_filtered_workspace_size).
 *   - A tempered sequence whose top_k or top_p is out of range sets
 *     SPEC_FLAG_BAD_FILTER and gets the sentinel outputs; other sequences are unaffected.
 *   - Precision: the filter and the decisions are evaluated in fp64 on the logits
 *     (z = l / T); ranking uses the logits themselves, so it is exact.
 *   - Workspace: as for every call, zero-filled once when new; each call leaves its
 *     per-sequence counters at zero again.
 */
#define SPEC_FILTER_MAX_TOP_K 1024
typedef struct {
  const int32_t* top_k;  /* [batch]                                                   */
  const float* top_p;    /* [batch]                                                   */
  int32_t max_top_k;     /* 1 .. SPEC_FILTER_MAX_TOP_K                                */
} spec_filter_args_t;

/* Bytes of workspace the filtered calls below need (attn may be NULL; 0 if an
 * argument is invalid). */
size_t spec_filtered_workspace_size(const spec_attn_args_t* attn, const spec_accept_args_t* accept,
                                    const spec_filter_args_t* filter);

/* Part (b) with filtering. */
spec_status_t spec_accept_block_filtered(const spec_accept_args_t* accept,
                                         const spec_filter_args_t* filter, void* ws,
                                         size_t ws_bytes, spec_stream_t stream);

/* The whole verify step with filtering: part (a) (attn may be NULL) and the filtered
 * part (b) on one stream, as spec_verify_step. */
spec_status_t spec_verify_step_filtered(const spec_attn_args_t* attn,
                                        const spec_accept_args_t* accept,
                                        const spec_filter_args_t* filter, void* ws,
                                        size_t ws_bytes, spec_stream_t stream);

/*
 * Draft-side sampling (Alg. "Lossless Psi-Spec decoding (Linear Sampler)": sample the
 * free clean token x^{L+1} ~ q_0 and the B-1 drafts x~ ~ q, in parallel). Block token j
 * of sequence b is drawn from drafter row j (row 0 = q_0, the AR pathway's
 * distribution; rows 1.. = q, the diffusion drafter's) at temperature[b]: the smallest
 * x with C(x) >= uniforms[b][j] * C(vocab-1), C the ascending-token cumulative sum of
 * softmax(row / T), top-k / top-p filtered first when filter is not NULL (as in
 * spec_accept_block_filtered); at T = 0 the row's lowest-index argmax. The result is the
 * block_tokens input of the verify step.
 *   - A sequence with a row that has NaN, +inf (T > 0) or no finite logit (T > 0) sets
 *     SPEC_FLAG_BAD_LOGITS and gets block_tokens = -1 (and q_tok = NaN) in every row; a
 *     tempered sequence with an out-of-range filter sets SPEC_FLAG_BAD_FILTER likewise.
 *   - Unfiltered draws keep one 8-byte (max, sum) pair per 64 logits (32 without 16-byte
 *     alignment) in shared memory: vocab up to 1,600,000 (800,000); larger is
 *     SPEC_ERR_UNSUPPORTED.
 */
typedef struct {
  int32_t batch;               /* >= 1                                                      */
  int32_t gamma;               /* 1 .. 64                                                   */
  int32_t vocab;               /* >= 1                                                      */
  int32_t logits_dtype;        /* spec_dtype_t                                              */
  const void* drafter_logits;  /* [batch][gamma][vocab]                                     */
  const float* temperature;    /* [batch]; 0 => argmax                                      */
  const float* uniforms;       /* [batch][gamma] in (0, 1]; [j] draws block token j         */
  int32_t* block_tokens;       /* [batch][gamma], written                                   */
  float* q_tok;                /* [batch][gamma]: the drawn token's (filtered) probability,
                                  1 at T = 0; or NULL                                       */
} spec_draft_args_t;

size_t spec_draft_workspace_size(const spec_draft_args_t* draft, const spec_filter_args_t* filter);
spec_status_t spec_sample_block(const spec_draft_args_t* draft, const spec_filter_args_t* filter,
                                void* ws, size_t ws_bytes, spec_stream_t stream);

/*
 * The noise tokens that start a draft pass (Alg. line 1: z ~ U[V], i.i.d.):
 * out_dev[i] = floor(x * vocab / 2^32), x = the Philox4x32-10 word of
 * spec_philox_uniforms' definition at index offset + i. n >= 0, vocab >= 1.
 */
spec_status_t spec_noise_tokens(uint64_t seed, uint64_t offset, int64_t n, int32_t vocab,
                                int32_t* out_dev, spec_stream_t stream);

/*
 * KV commit: roll a paged KV cache back to the accepted prefix of a verify step (the
 * Algorithm returns [x, x^{L+1}, x~^{1:n-1}, z~]: the block keys past x~^{n-1} are not
 * part of the sequence). On entry kv_len[b] = ctx_b + gamma (the verify layout); on exit
 * kv_len[b] = ctx_b + n_b, n_b = num_accepted[b] + 1 (ctx_b if num_accepted[b] = -1,
 * a failed step). The final token z~ has no key yet: the next pass computes it.
 *   - reserve = 1: each sequence keeps its pages and takes, from the top of the free
 *     list, the pages it lacks to hold gamma more keys (the next block). Requests are
 *     served in batch order while their running total fits the list; a refused request
 *     still counts against the later ones (flag 2, its length still committed), as does a
 *     sequence whose table cannot hold the pages.
 *   - reserve = 0 (the sequence stops): pages wholly past the new length are pushed onto
 *     the free list in batch order (entries set to -1), under the same prefix rule
 *     against free_capacity; a sequence whose pages do not fit keeps them (flag 2).
 *   - kv_len outside [gamma, max_pages_per_seq * page_size] or num_accepted outside
 *     [-1, gamma-1]: the sequence is left unchanged (flag 1).
 * All pointers are device memory; one launch of one block, no workspace. The paper
 * keeps its cache inside its serving framework; this call is that framework's step.
 */
typedef struct {
  int32_t batch, gamma, page_size, max_pages_per_seq;
  int32_t* kv_len;              /* [batch], read and written                                 */
  const int32_t* num_accepted;  /* [batch], from the verify step                            */
  int32_t* page_table;          /* [batch][max_pages_per_seq], read and written             */
  int32_t* free_pages;          /* [free_capacity]: the free list, its top at free_count     */
  int32_t* free_count;          /* [1], read and written                                     */
  int32_t free_capacity;
  int32_t reserve;              /* 1: reserve for the next block; 0: release                 */
  int32_t* flags;               /* [batch]: 0, 1 or 2 as above; or NULL                      */
} spec_commit_args_t;

spec_status_t spec_commit_kv(const spec_commit_args_t* commit, spec_stream_t stream);

/*
 * Tree verification (Sec. 4.2: several candidates verified at once as a prefix tree,
 * with the standard speculative-decoding rejection correction; Sec. 3.3, "Tree
 * Sampler"), greedy (T = 0) or sampled (T > 0).
 *
 * A candidate tree of num_nodes <= 64 nodes per sequence: node 0 is the root (the free
 * token x^{L+1}); parents[b][c] < c is node c's parent (-1 for the root); tokens[b][c]
 * is its token. The verify pass runs on the nodes as the block (spec_verify_attention
 * with tree_mask = each node's ancestor bits); target row c (target_logits
 * [batch][num_nodes][vocab]) is the verifier's distribution of the token after node c.
 *
 * spec_accept_tree, greedy sequences (temperature NULL, or temperature[b] <= 0): from
 * the root, move to the child (lowest node index first) whose token is the lowest-index
 * argmax of the current node's target row; stop where there is none; the final token is
 * that argmax.
 * Sampled sequences (temperature[b] > 0): at the current node, with p = softmax(target
 * row / T), its children are tried in node order as point-mass proposals: child c is
 * accepted iff uniforms[b][c] <= p'(tokens[b][c]), where p' is p with the tokens of the
 * children rejected so far at this node removed and renormalised (min(1, p'/q) with q
 * the point mass; its residual Norm([p' - q]_+) removes the token). On acceptance the
 * walk moves to c. If none is accepted, or the node has no child, the final token is
 * drawn from p' by inverse CDF in ascending token order with uniforms[b][0]. The
 * emitted tokens then follow the target's own distribution exactly (lossless).
 * Outputs: path[b] = the visited nodes (-1 padded), out_tokens[b] = their tokens then
 * the final token (-1 padded, num_nodes + 1 entries), num_accepted = path length - 1,
 * num_emitted = path length + 1. A sequence with a token outside [0, vocab), parents
 * that are not a tree (SPEC_FLAG_BAD_TREE), a NaN in a target row, or (sampled) a
 * target row with +inf or no finite logit (SPEC_FLAG_BAD_LOGITS) gets
 * num_accepted = -1, num_emitted = 0 and -1 outputs.
 */
typedef struct {
  int32_t batch, num_nodes, vocab, logits_dtype;
  const void* target_logits;   /* [batch][num_nodes][vocab]                                */
  const int32_t* tokens;       /* [batch][num_nodes]                                       */
  const int32_t* parents;      /* [batch][num_nodes]                                       */
  int32_t* path;               /* [batch][num_nodes], written                              */
  int32_t* num_accepted;       /* [batch], written                                         */
  int32_t* out_tokens;         /* [batch][num_nodes + 1], written                          */
  int32_t* num_emitted;        /* [batch], written                                         */
  const float* temperature;    /* [batch], or NULL: every sequence greedy                  */
  const float* uniforms;       /* [batch][num_nodes] in (0, 1] (needed with temperature):
                                  [c] tests node c, [0] draws the final token              */
} spec_tree_accept_args_t;

size_t spec_tree_workspace_size(const spec_tree_accept_args_t* tree);
spec_status_t spec_accept_tree(const spec_tree_accept_args_t* tree, void* ws, size_t ws_bytes,
                               spec_stream_t stream);

/*
 * After spec_accept_tree: keep the accepted path in the paged KV cache. The nodes' keys
 * sit at positions ctx_b .. ctx_b + num_nodes - 1 (kv_len[b] = ctx_b + num_nodes); the
 * key and value rows (every KV head) of path node path[b][d] move to position ctx_b + d
 * for d = 1 .. num_accepted[b], and kv_len[b] becomes ctx_b + num_accepted[b] + 1
 * (ctx_b when num_accepted[b] = -1). The result is that of moving the rows one by one
 * in increasing d. A sequence with kv_len[b] outside [num_nodes, max_pages_per_seq *
 * page_size] (SPEC_FLAG_BAD_KV_LEN), num_accepted outside [-1, num_nodes) or a path that
 * does not start at node 0 and rise strictly below num_nodes (SPEC_FLAG_BAD_TREE), or a
 * moved row's page id outside [0, num_pages) (SPEC_FLAG_BAD_PAGE) is left unchanged,
 * kv_len included, and the flag is set in *status (if given). Two launches, no workspace.
 */
typedef struct {
  int32_t batch, num_nodes, num_kv_heads, head_dim, page_size, max_pages_per_seq, num_pages;
  void* k_cache;                /* bf16 [num_pages][Hkv][page_size][D], updated              */
  void* v_cache;                /* bf16, same layout, updated                                */
  const int32_t* page_table;    /* [batch][max_pages_per_seq]                               */
  int32_t* kv_len;              /* [batch], updated                                          */
  const int32_t* path;          /* [batch][num_nodes] from spec_accept_tree                 */
  const int32_t* num_accepted;  /* [batch] from spec_accept_tree                            */
  uint32_t* status;             /* a status word (e.g. a workspace's first word), or NULL   */
} spec_tree_commit_args_t;

spec_status_t spec_commit_tree_kv(const spec_tree_commit_args_t* commit, spec_stream_t stream);

/*
 * The tree sampler (Sec. 3.3, "Tree Sampler", with (B, K, V) = (gamma, top_k,
 * num_nodes - 1)): the candidate tree that spec_accept_tree verifies, built from the
 * drafter's rows. Block position d = 1 .. gamma-1 draws from drafter row d
 * (drafter_logits[b][d]; row 0 is not read). Its candidates are the top_k tokens of
 * log q_d = log softmax(row / T), T = temperature[b] (T <= 0 or NaN ranks at T = 1),
 * ranked by probability, equal ones by lower token id. Node 0 is the root, token
 * root_tokens[b] (the free token x^{L+1}). Each of the num_nodes - 1 steps adds the
 * best child on offer, where every node at depth d < gamma - 1 offers its next unused
 * candidate of position d + 1, scored by the sum of log q along its path; equal scores
 * go to the lower parent index. The nodes are then the most probable num_nodes - 1
 * prefixes, each after its parent, in the order they were taken. log q is computed in
 * fp32 and path scores are summed in double-float (two fp32 words, about 48 bits).
 *
 * Outputs: tokens, parents (-1 for the root), depth (optional; the root is 0) and
 * tree_mask (optional; bit i of node j set iff node i is j or one of its ancestors, the
 * input of tree attention), each [batch][num_nodes]. A sequence whose used drafter rows
 * hold a NaN or +inf or no finite logit (SPEC_FLAG_BAD_LOGITS) or whose root token is
 * outside [0, vocab) (SPEC_FLAG_BAD_TOKEN) gets -1 tokens, parents and depths and a
 * zero mask. SPEC_ERR_INVALID_ARGUMENT when the positions cannot hold num_nodes - 1
 * nodes: sum over d = 1 .. gamma-1 of min(top_k, vocab)^d < num_nodes - 1.
 */
typedef struct {
  int32_t batch, gamma, vocab, logits_dtype;
  int32_t top_k;                /* K >= 1                                                  */
  int32_t num_nodes;            /* 1 .. 64                                                 */
  const void* drafter_logits;   /* [batch][gamma][vocab]                                   */
  const float* temperature;     /* [batch]                                                 */
  const int32_t* root_tokens;   /* [batch]                                                 */
  int32_t* tokens;              /* [batch][num_nodes], written                             */
  int32_t* parents;             /* [batch][num_nodes], written                             */
  int32_t* depth;               /* [batch][num_nodes], written, or NULL                    */
  uint64_t* tree_mask;          /* [batch][num_nodes], written, or NULL                    */
} spec_tree_build_args_t;

size_t spec_tree_build_workspace_size(const spec_tree_build_args_t* build);
spec_status_t spec_build_tree(const spec_tree_build_args_t* build, void* ws, size_t ws_bytes,
                              spec_stream_t stream);

/*
 * The target's LM head with the row statistics of the acceptance fused into it (the
 * verifier pass of Sec. 4.2 scores the block rows with the target's output layer;
 * Appendix B.3's rule reads p = softmax(logits / T) through its normaliser, its
 * maximum and the logit of a drafted token): logits = hidden_states . weight^T on the
 * tensor cores (bf16 operands, fp32 accumulation), reduced per row as they leave the
 * accumulator, so the [rows][vocab] logits need not be written.
 *
 * Row r belongs to sequence r / rows_per_seq, whose temperature is T. Outputs per row:
 * row_max = max_v l_v; row_sum = sum_v exp((l_v - row_max) / T) (T <= 0 or NaN sums at
 * T = 1); row_argmax = the lowest index of the maximum; token_logit (if given) = l at
 * tokens[r] (NaN where tokens is NULL or tokens[r] is outside [0, vocab)). logits (if
 * given) receives every logit as bf16 [rows][vocab] (the rounding of the fp32 value).
 * A row with a NaN or an infinite logit sets SPEC_FLAG_BAD_LOGITS and gets
 * row_argmax = -1. Device memory, caller-owned; hidden_states and weight 16-byte
 * aligned, hidden a multiple of 8.
 */
typedef struct {
  int32_t rows, hidden, vocab, rows_per_seq;
  const void* hidden_states;   /* bf16 [rows][hidden]                                    */
  const void* weight;          /* bf16 [vocab][hidden]: output row v of the LM head       */
  const float* temperature;    /* [ceil(rows / rows_per_seq)]                             */
  const int32_t* tokens;       /* [rows], or NULL                                         */
  float* row_max;              /* [rows], written                                         */
  float* row_sum;              /* [rows], written                                         */
  int32_t* row_argmax;         /* [rows], written                                         */
  float* token_logit;          /* [rows], written, or NULL                                */
  void* logits;                /* bf16 [rows][vocab], written, or NULL                    */
} spec_lm_head_args_t;

size_t spec_lm_head_workspace_size(const spec_lm_head_args_t* lm);
spec_status_t spec_lm_head_stats(const spec_lm_head_args_t* lm, void* ws, size_t ws_bytes,
                                 spec_stream_t stream);

/*
 * spec_accept_block without a workspace, for callers that cannot allocate device
 * memory when they verify (for example, code confined to a fixed, pre-planned memory
 * arena, or code that must not call an allocator). It computes exactly what
 * spec_accept_block computes; the paper has no counterpart to this call. Its scratch
 * lives in one device array of SPEC_NOALLOC_SCRATCH_BYTES owned by the library, which
 * every GPU that loads the library keeps until the process exits.
 *   - Arguments: as spec_accept_block (device pointers, same layouts); no workspace.
 *   - Limit: the scratch this batch needs (16 bytes per (sequence, row, 4096-entry
 *     vocab chunk), 32 bytes per sequence, and 16 bytes per (sequence, 4096-entry
 *     slice), rounded up) must fit
 *     in SPEC_NOALLOC_SCRATCH_BYTES; otherwise SPEC_ERR_WORKSPACE_TOO_SMALL, with
 *     nothing launched. Other argument errors as spec_accept_block.
 *   - Allocates nothing: no cudaMalloc, cudaFree or allocating library routine. The
 *     first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current; make that first call before
 *     any stream capture.
 *   - Every call shares the one array per device, and each call clears the part of it
 *     that must start at zero, so calls that overlap on the GPU (concurrent streams)
 *     race and give wrong results: serialize them.
 *   - Bad device data is still reported through the sentinel outputs; there is no
 *     status word to read back.
 */
#define SPEC_NOALLOC_SCRATCH_BYTES (4u << 20)
spec_status_t spec_accept_block_noalloc(const spec_accept_args_t* accept, spec_stream_t stream);

/* ---------------------------------------------------------------------------------------
 * Test hooks for the timeout path (not part of the verify step)
 *
 * The kernels' internal waits on asynchronous copies and tensor-core operations are
 * bounded (about 1 s of SM clock); one that runs out sets SPEC_FLAG_TIMEOUT, the block
 * releases its resources and returns, and the context stays usable. These two calls make
 * that happen on purpose, so that it can be tested: each is the launch of its product
 * call (spec_verify_attention on the tensor-core row-tile path, spec_lm_head_stats), with
 * the same arguments, workspace rules and errors, except that the kernel's copy producer
 * issues nothing, so every consumer's wait runs out (about 1 s). Afterwards the workspace
 * status word holds SPEC_FLAG_TIMEOUT (spec_read_device_status returns
 * SPEC_ERR_TIMEOUT and clears it), the outputs are undefined, and the workspace's
 * counters are still zero, so the same workspace serves the next product call.
 * spec_test_attention_wait_timeout returns SPEC_ERR_UNSUPPORTED for shapes the
 * tensor-core row-tile kernel does not take. Nothing traps, faults or waits without bound.
 * ------------------------------------------------------------------------------------- */
spec_status_t spec_test_attention_wait_timeout(const spec_attn_args_t* attn, void* ws,
                                               size_t ws_bytes, spec_stream_t stream);
spec_status_t spec_test_lm_head_wait_timeout(const spec_lm_head_args_t* lm, void* ws,
                                             size_t ws_bytes, spec_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SPEC_VERIFY_H */
