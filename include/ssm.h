/*
 * ssm.h -- C ABI of libssm: one structured-suffix (SSM) denoising step of a
 * block-wise diffusion language model on an NVIDIA GB300 (sm_103a).
 *
 * The step (paper: "Accelerating Diffusion Language Models via Structured
 * Suffix Modeling") has four stages, each one entry point here:
 *   1. ssm_select_suffix      -- retained suffix positions R_t (Sec. 3.2, Eqs. 1-5)
 *   2. ssm_build_step_input   -- sparse input X~_t = [P; B_t; R_t] with original
 *                                positions and soft suffix embeddings (Eqs. 6-8)
 *   3. ssm_attention          -- bidirectional MHA/GQA attention with rotary
 *                                encodings at the original positions
 *   4. ssm_unmask             -- vocabulary softmax, confidence, argmax and the
 *                                threshold / top-k / margin commit (Sec. 4.2, 4.6)
 * and, around the step, ssm_suffix_topk (the retained suffix positions' top-k
 * candidates for the next step's Eq. 6), ssm_cache_append (the prefix-cache
 * update at a block boundary, Sec. 4.8 "+PC.") and ssm_early_stop (early
 * termination after a block, Sec. 3.2).
 *
 * Conventions (all entry points):
 *   - Every function returns ssm_status; nothing throws across the ABI.
 *   - Pointers are DEVICE pointers unless the name starts with h_ (host).
 *     The caller allocates and owns every buffer; the library allocates no
 *     device memory.  Scratch memory, where a stage needs it, is a caller
 *     buffer of at least the size the matching *_workspace_size() returns.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t; NULL is the
 *     legacy default stream).  Argument checks are synchronous, on the host:
 *     a call that returns an error has enqueued nothing.
 *   - Errors found on the device (an out-of-range token id, a wait that timed
 *     out) do not stop the stream: the kernel writes zeros or skips the item
 *     and records a code in a device error word; ssm_get_device_error()
 *     synchronises the stream and returns (and clears) that code.
 *   - Tensors are dense, row-major, with the innermost dimension last, in the
 *     layouts given per argument.  bf16 data are IEEE bfloat16 bit patterns.
 *   - The library looks up the device addresses of its own device variables
 *     (the error word, ssm_unmask_noalloc's scratch) once per device and keeps
 *     them.  Destroying a device's primary context (cudaDeviceReset) makes those
 *     addresses stale: after a reset, reload the library (a new process) before
 *     calling it again on that device.
 */
#ifndef SSM_H_
#define SSM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* ssm_stream_t; /* identical to cudaStream_t */

typedef enum {
  SSM_OK = 0,
  SSM_ERR_INVALID_ARG = 1,  /* null pointer, negative size, budget, alpha outside [0,1] ... */
  SSM_ERR_SHAPE = 2,        /* inconsistent shapes (G % B != 0, H_q % H_kv != 0 ...) */
  SSM_ERR_CAPACITY = 3,     /* output or workspace smaller than required */
  SSM_ERR_CUDA = 4,         /* a CUDA runtime/driver call failed */
  SSM_ERR_TIMEOUT = 5,      /* (device) a bounded wait inside a kernel expired */
  SSM_ERR_UNSUPPORTED = 6,  /* valid but not implemented (head_dim not 64/128 ...) */
  SSM_ERR_DEVICE_INPUT = 7  /* (device) an input value was out of range (token id >= vocab ...) */
} ssm_status;

typedef enum { SSM_DTYPE_BF16 = 0, SSM_DTYPE_F32 = 1 } ssm_dtype;

typedef enum {
  SSM_COMMIT_THRESHOLD = 0, /* "Par.": commit masked positions with confidence > threshold */
  SSM_COMMIT_TOPK = 1,      /* "Vanilla" is topk = 1: the k most confident masked positions */
  SSM_COMMIT_MARGIN = 2     /* commit masked positions with p1 - p2 > threshold */
} ssm_commit_mode;

const char* ssm_status_str(ssm_status s);
const char* ssm_version(void);

/* Synchronises `stream`, returns the first device-side error recorded by any
 * libssm kernel since the last call (SSM_OK if none) and clears it. */
ssm_status ssm_get_device_error(ssm_stream_t stream);

/* Device-side wait limit, in nanoseconds, for every bounded spin inside the
 * libssm kernels (default 2e9).  A wait that exceeds it records
 * SSM_ERR_TIMEOUT and the kernel leaves the work item.  0 restores the default. */
ssm_status ssm_set_wait_limit_ns(uint64_t ns);

/* ------------------------------------------------------------------------- */
/* 1. Structured suffix selection (Sec. 3.2 "Suffix Region Partition" Eq. 1,  */
/*    "Suffix Token Retention" Eqs. 2-5).                                     */
/* ------------------------------------------------------------------------- */

/* Sequence layout: the prompt occupies positions [0, prompt_len); the
 * generation [prompt_len, prompt_len + gen_len) is cut into gen_len/block_len
 * blocks; block_idx is the block being decoded and the suffix is every later
 * block.  Budgets are token counts:
 *   local_budget  L: the first L suffix tokens are kept (Eq. 2; the paper's w
 *                    blocks are L = w * block_len); if the whole suffix fits in
 *                    L, every suffix token is kept;
 *   middle_budget M: the start token of each middle block (Eq. 3), at most M
 *                    of them (evenly strided, block q*nm/M, if there are more);
 *   tail_budget   T: T evenly spaced tokens of the last block, start and end
 *                    included (Eq. 4 is T = 2). */
typedef struct {
  int32_t prompt_len, gen_len, block_len, block_idx;
  int32_t local_budget, middle_budget, tail_budget;
} ssm_suffix_cfg;

/* Host only, pure: region sizes of R_t for `cfg` (the three add up to |R_t|;
 * h_n_tail counts tail tokens not already local).  Any output may be NULL. */
ssm_status ssm_suffix_count(const ssm_suffix_cfg* cfg, int32_t* h_n_local, int32_t* h_n_mid,
                            int32_t* h_n_tail);

/* Writes R_t for `cfg` to positions[0 .. |R_t|) as ascending absolute int32
 * positions, and |R_t| to *h_count (host).  capacity = length of `positions`;
 * if capacity < |R_t| returns SSM_ERR_CAPACITY with *h_count set and enqueues
 * nothing. */
ssm_status ssm_select_suffix(const ssm_suffix_cfg* cfg, int32_t* positions, int32_t capacity,
                             int32_t* h_count, ssm_stream_t stream);

/* Several selections in one launch (e.g. sequences of a serving batch, each at
 * its own block index).  h_cfgs: host array of n configs.  The sets are
 * written back to back into `positions`; h_offsets (host, n + 1 entries) gets
 * the start of each set and the total in h_offsets[n]. */
ssm_status ssm_select_suffix_batch(const ssm_suffix_cfg* h_cfgs, int32_t n, int32_t* positions,
                                   int64_t capacity, int64_t* h_offsets, ssm_stream_t stream);

/* ------------------------------------------------------------------------- */
/* 2. Sparse step input with soft suffix embeddings (Sec. 3.2 "Soft Suffix    */
/*    Embedding Mixing" Eqs. 6-8, "Sparse Input Construction").               */
/* ------------------------------------------------------------------------- */

/* For every batch row b the output rows are
 *   [0, n_prefix)                 x = E[prefix_tokens[b, j]]          (prompt, when recomputed)
 *   [n_prefix, n_prefix+B)        x = E[block_tokens[b, j]]           (current block; a masked
 *                                                                     position carries mask_id)
 *   [n_prefix+B, n_prefix+B+R)    x = (1-alpha) E[mask_id] + alpha * sum_j p~_j E[ids_j]
 * with p~_j = p_j / sum_j p_j over the previous step's top-k candidates of
 * that suffix position (Eq. 6-8).  Candidates with id -1 are absent; a row with
 * no candidate (or zero mass) is E[mask_id].  Sums are in fp32, the stored
 * value is rounded to bf16 (nearest even).  pos_out gets the original absolute
 * positions: 0..n_prefix-1, block_start..block_start+B-1, suffix_pos[0..R).
 *
 *   block_tokens   int32 [batch, block_len]
 *   prefix_tokens  int32 [batch, n_prefix]             (NULL iff n_prefix == 0)
 *   suffix_pos     int32 [n_suffix]                    (from ssm_select_suffix)
 *   embed          bf16  [vocab, hidden]; hidden % 8 == 0, 16-byte aligned
 *   prev_topk_ids  int32 [batch, n_suffix, k]          (NULL: no prediction anywhere)
 *   prev_topk_prob fp32  [batch, n_suffix, k]          (previous-step probabilities)
 *   x_out          bf16  [batch, n_prefix + block_len + n_suffix, hidden]
 *   pos_out        int32 [n_prefix + block_len + n_suffix]   (may be NULL)
 * 0 <= k <= 32, alpha in [0, 1].  A token id outside [0, vocab) (other than a
 * -1 candidate) records SSM_ERR_DEVICE_INPUT and zeroes that row. */
ssm_status ssm_build_step_input(const int32_t* block_tokens, const int32_t* prefix_tokens,
                                int32_t batch, int32_t n_prefix, int32_t block_len,
                                int32_t block_start, const int32_t* suffix_pos, int32_t n_suffix,
                                const void* embed, int64_t vocab, int32_t hidden, int32_t mask_id,
                                const int32_t* prev_topk_ids, const float* prev_topk_prob,
                                int32_t k, float alpha, void* x_out, int32_t* pos_out,
                                ssm_stream_t stream);

/* Ragged form: n_problems independent steps (one sequence each, e.g. every
 * block index of a sweep, or a serving batch at mixed block indices) in one
 * launch.  problems is a DEVICE array; problem p reads
 *   block_tokens[block_tok_off .. + block_len), prefix_tokens[prefix_tok_off .. + n_prefix),
 *   suffix_pos[suffix_off .. + n_suffix), prev_topk_*[(suffix_off)*k .. + n_suffix*k)
 * and writes rows out_row .. out_row + n_prefix + block_len + n_suffix of
 * x_out [*, hidden] and the same entries of pos_out.  max_rows bounds
 * n_prefix + block_len + n_suffix over all problems (grid size). */
typedef struct {
  int64_t block_tok_off;
  int64_t prefix_tok_off;
  int64_t suffix_off;
  int64_t out_row;
  int32_t n_prefix;
  int32_t n_suffix;
  int32_t block_start;
  int32_t reserved;
} ssm_step_problem;

ssm_status ssm_build_step_input_varlen(const ssm_step_problem* problems, int32_t n_problems,
                                       int32_t max_rows, int32_t block_len,
                                       const int32_t* block_tokens, const int32_t* prefix_tokens,
                                       const int32_t* suffix_pos, const void* embed,
                                       int64_t vocab, int32_t hidden, int32_t mask_id,
                                       const int32_t* prev_topk_ids, const float* prev_topk_prob,
                                       int32_t k, float alpha, void* x_out, int32_t* pos_out,
                                       ssm_stream_t stream);

/* Selection and sparse input in one launch: ssm_select_suffix_batch followed by
 * ssm_build_step_input_varlen, with every retained suffix row placing itself at
 * the position of its rank in R_t (the closed form of Eqs. 2-5) instead of
 * reading a selection written by an earlier launch.
 *   cfgs            DEVICE array of n_problems ssm_suffix_cfg: problem p's
 *                   selection; its |R_t| must equal problems[p].n_suffix
 *                   (ssm_suffix_count), else SSM_ERR_DEVICE_INPUT is recorded
 *                   and that problem's suffix rows are zeroed
 *   suffix_pos_out  int32, R_t of problem p written at problems[p].suffix_off
 *                   (the positions ssm_select_suffix_batch gives; may be NULL)
 * Other arguments, outputs and errors as ssm_build_step_input_varlen, whose
 * results this equals. */
ssm_status ssm_select_build_step_input_varlen(const ssm_step_problem* problems, const ssm_suffix_cfg* cfgs,
                                              int32_t n_problems, int32_t max_rows, int32_t block_len,
                                              const int32_t* block_tokens, const int32_t* prefix_tokens,
                                              int32_t* suffix_pos_out, const void* embed, int64_t vocab,
                                              int32_t hidden, int32_t mask_id, const int32_t* prev_topk_ids,
                                              const float* prev_topk_prob, int32_t k, float alpha, void* x_out,
                                              int32_t* pos_out, ssm_stream_t stream);

/* ------------------------------------------------------------------------- */
/* 3. Bidirectional attention over prefix cache + block + retained suffix     */
/*    (Sec. 1 and Sec. 2: DLM attention is bidirectional; Sec. 3.2 "Sparse    */
/*    Input Construction": retained tokens keep their original rotary         */
/*    encodings; Table 4: prefix cache "PC.").                                 */
/* ------------------------------------------------------------------------- */

/* O = softmax(scale * Q^ K^T) V with no mask, per (batch, query head h), over
 * keys [cache rows; new rows].  Q^ = RoPE(q, pos), new keys are RoPE(k_new,
 * pos); cached keys are used as given (already rotated at their own positions).
 * RoPE: rotate-half pairs (i, i + d/2), angle pos * theta^(-2i/d); theta == 0
 * disables it.  The angle pos * f (f the fp64 frequency) is taken modulo one
 * turn in 0.64 fixed point (exact to below 2^-33 turns for any int32 position),
 * its sine and cosine in fp32, the rotation in fp32 and rounded to bf16 before
 * the tensor-core products.
 * GQA: query head h reads key/value head h / (h_q / h_kv).
 * bf16 inputs, fp32 accumulation (tcgen05 tensor cores), bf16 output.
 *
 *   q            bf16 [batch, n_new, h_q, d]
 *   k_new, v_new bf16 [batch, n_new, h_kv, d]    (the same rows as q)
 *   pos          int32 [n_new]                   (shared by the batch)
 *   k_cache, v_cache bf16 [batch, n_cache, h_kv, d]  (NULL iff n_cache == 0)
 *   out          bf16 [batch, n_new, h_q, d]
 *   lse          fp32 [batch, n_new, h_q]  natural-log sum-exp of the scaled
 *                scores (may be NULL)
 *   workspace    >= ssm_attention_workspace_size(batch * n_new, h_q, h_kv, d)
 *                bytes, 256-byte aligned; holds the rotated queries and keys
 *                (and, for the ragged form, the work plan and a row map).
 * d in {64, 128}; h_q % h_kv == 0; every pointer 16-byte aligned. */
size_t ssm_attention_workspace_size(int64_t total_new_rows, int32_t h_q, int32_t h_kv,
                                    int32_t head_dim);

ssm_status ssm_attention(const void* q, const void* k_new, const void* v_new, const int32_t* pos,
                         const void* k_cache, const void* v_cache, int32_t batch, int32_t n_new,
                         int32_t n_cache, int32_t h_q, int32_t h_kv, int32_t head_dim,
                         float rope_theta, float scale, void* out, float* lse, void* workspace,
                         size_t ws_bytes, ssm_stream_t stream);

/* Ragged form: independent problems packed along the row dimension.
 * problems is a DEVICE array; problem p owns rows new_row .. new_row + n_new
 * of q / k_new / v_new / out / lse / pos (packed [total_new_rows, h, d]) and
 * rows cache_row .. cache_row + n_cache of k_cache / v_cache (packed
 * [total_cache_rows, h_kv, d]; several problems may share cache rows).
 * max_n_new / max_n_cache bound the per-problem sizes (grid size).  A tile at
 * the ragged end of a problem may read rows of the same buffers beyond it
 * (multiplied by an exact zero): keep every row of the packed buffers finite.
 * When every problem reads one shared cache (equal cache_row; prefixes of
 * different lengths, e.g. the block indices of one sequence) and the problems'
 * new rows follow one another from row 0, the rows of consecutive problems may
 * share query tiles (each row still sees only its own prefix and its own new
 * rows); the result is the same either way. */
typedef struct {
  int64_t new_row;
  int64_t cache_row;
  int32_t n_new;
  int32_t n_cache;
} ssm_attn_problem;

ssm_status ssm_attention_varlen(const void* q, const void* k_new, const void* v_new,
                                const int32_t* pos, const void* k_cache, const void* v_cache,
                                int64_t total_new_rows, int64_t total_cache_rows,
                                const ssm_attn_problem* problems, int32_t n_problems,
                                int32_t max_n_new, int32_t max_n_cache, int32_t h_q,
                                int32_t h_kv, int32_t head_dim, float rope_theta, float scale,
                                void* out, float* lse, void* workspace, size_t ws_bytes,
                                ssm_stream_t stream);

/* The two launches ssm_attention_varlen makes, as separate calls with the same
 * arguments, for a caller that schedules or times them apart:
 *   ..._rotate writes the rotated queries (packed by GQA group), the rotated
 *              new keys and the work plan into `workspace` (the RoPE pre-pass;
 *              q, k_new, pos and the problem table are read, v/cache/out/lse
 *              are not touched);
 *   ..._core   runs the attention forward from that workspace (q, k_new and pos
 *              are not read again).
 * ..._core must follow a ..._rotate with the same arguments and workspace, in
 * stream order; ssm_attention_varlen(args) equals ..._rotate(args) followed by
 * ..._core(args).  Errors as ssm_attention_varlen. */
ssm_status ssm_attention_varlen_rotate(const void* q, const void* k_new, const void* v_new,
                                       const int32_t* pos, const void* k_cache, const void* v_cache,
                                       int64_t total_new_rows, int64_t total_cache_rows,
                                       const ssm_attn_problem* problems, int32_t n_problems,
                                       int32_t max_n_new, int32_t max_n_cache, int32_t h_q,
                                       int32_t h_kv, int32_t head_dim, float rope_theta, float scale,
                                       void* out, float* lse, void* workspace, size_t ws_bytes,
                                       ssm_stream_t stream);
ssm_status ssm_attention_varlen_core(const void* q, const void* k_new, const void* v_new,
                                     const int32_t* pos, const void* k_cache, const void* v_cache,
                                     int64_t total_new_rows, int64_t total_cache_rows,
                                     const ssm_attn_problem* problems, int32_t n_problems,
                                     int32_t max_n_new, int32_t max_n_cache, int32_t h_q,
                                     int32_t h_kv, int32_t head_dim, float rope_theta, float scale,
                                     void* out, float* lse, void* workspace, size_t ws_bytes,
                                     ssm_stream_t stream);

/* ------------------------------------------------------------------------- */
/* 4. Confidence-based unmasking (Sec. 4.2 "Baselines": Vanilla top-1 and     */
/*    parallel threshold decoding; Sec. 4.6: margin decoding).                */
/* ------------------------------------------------------------------------- */

/* For every masked block position (masked[b, j] != 0): the softmax over the
 * vocabulary in fp32, conf = largest probability, argmax = lowest id among the
 * largest logits, p2 = second-largest probability (a tied maximum counts
 * twice).  Unmasked positions get conf = 0, argmax = -1, p2 = 0, commit = 0
 * and their logits are never read.  Then, per batch row:
 *   THRESHOLD: commit masked positions with conf > threshold;
 *   MARGIN:    commit masked positions with conf - p2 > threshold;
 *   TOPK:      commit the `topk` masked positions of highest confidence;
 * and (THRESHOLD, MARGIN) if fewer than min_commit passed, the most confident
 * remaining masked positions are added up to min_commit.  Ties between
 * positions go to the lower position.
 *
 *   logits   [batch, block_len, vocab] of `dtype` (bf16 or fp32), 16-byte aligned
 *   masked   uint8 [batch, block_len]
 *   conf, p2 fp32 [batch, block_len]; argmax int32 [batch, block_len]
 *            (p2 may be NULL unless mode == MARGIN)
 *   commit   uint8 [batch, block_len]
 *   workspace >= ssm_unmask_workspace_size(batch, block_len, vocab, dtype) bytes,
 *            256-byte aligned (the partial reductions of each row: one per
 *            streaming range of the vocabulary that meets the row).
 * block_len <= 1024. */
size_t ssm_unmask_workspace_size(int32_t batch, int32_t block_len, int64_t vocab, ssm_dtype dtype);

ssm_status ssm_unmask(const void* logits, ssm_dtype dtype, int32_t batch, int32_t block_len,
                      int64_t vocab, const uint8_t* masked, ssm_commit_mode mode, float threshold,
                      int32_t topk, int32_t min_commit, float* conf, int32_t* argmax, float* p2,
                      uint8_t* commit, void* workspace, size_t ws_bytes, ssm_stream_t stream);

/* Everything a denoising step takes from its logits, in one call: ssm_unmask
 * of the block rows (Sec. 4.2 / 4.6 commit rules) and ssm_suffix_topk of the
 * retained suffix rows (Sec. 3.2 "Soft Suffix Embedding Mixing": the top-k
 * candidates and full-vocabulary probabilities that the next step's Eq. 6
 * renormalizes -- ssm_build_step_input's prev_topk_ids / prev_topk_prob).  The
 * two streaming passes are enqueued back to back on `stream`.
 * Block-row arguments, outputs and workspace as ssm_unmask; suffix rows as
 * ssm_suffix_topk:
 *   suffix_logits  same dtype and vocab as logits, [n_suffix_rows, vocab]
 *   ids, probs     int32 / fp32 [n_suffix_rows, k], 1 <= k <= 8
 * Every condition of both calls is checked before anything is enqueued
 * (n_suffix_rows == 0 is ssm_unmask).  The results equal the two separate
 * calls'. */
ssm_status ssm_unmask_topk(const void* logits, ssm_dtype dtype, int32_t batch, int32_t block_len, int64_t vocab,
                           const uint8_t* masked, ssm_commit_mode mode, float threshold, int32_t topk,
                           int32_t min_commit, float* conf, int32_t* argmax, float* p2, uint8_t* commit,
                           const void* suffix_logits, int64_t n_suffix_rows, int32_t k, int32_t* ids,
                           float* probs, void* workspace, size_t ws_bytes, ssm_stream_t stream);

/* ssm_unmask_noalloc -- ssm_unmask for callers that cannot allocate device
 * memory.  The paper has no counterpart: this is a deployment convenience.
 *
 * Some callers cannot call cudaMalloc or hand out a scratch buffer: a host
 * program whose device memory is owned by another framework's allocator, or a
 * code path where allocation is not permitted.  This entry point takes the
 * same arguments as ssm_unmask minus the workspace and allocates nothing: its
 * scratch is a fixed 2 MiB array in device global memory that the library
 * holds on every GPU that loads it, until the process exits.
 *   - Limit: ssm_unmask_workspace_size(batch, block_len, vocab, dtype) must be
 *     at most 2 MiB (with a 126464-entry bf16 or fp32 vocabulary that holds
 *     every call of up to 65535 positions, the most ssm_unmask takes); larger
 *     calls return SSM_ERR_CAPACITY and enqueue nothing.
 *   - The first call on a device looks up the array's device address (with
 *     that device current); make that first call before any stream capture.
 *     The address is kept for the life of the process: a cudaDeviceReset makes
 *     it stale, so after a reset reload the library before calling this again.
 *   - Every call shares the one array: two calls that overlap on the GPU (on
 *     different streams, or from different threads) race and corrupt each
 *     other's results.  Serialise them.  The array keeps the last call's
 *     contents; nothing in it needs to start at zero.
 *   - No cudaMalloc, cudaFree or allocating library routine is called. */
ssm_status ssm_unmask_noalloc(const void* logits, ssm_dtype dtype, int32_t batch, int32_t block_len,
                              int64_t vocab, const uint8_t* masked, ssm_commit_mode mode, float threshold,
                              int32_t topk, int32_t min_commit, float* conf, int32_t* argmax, float* p2,
                              uint8_t* commit, ssm_stream_t stream);

/* ------------------------------------------------------------------------- */
/* 4b. The next step's soft-embedding candidates of the retained suffix       */
/*     positions (Sec. 3.2 "Soft Suffix Embedding Mixing", the set T^i_{t+1}  */
/*     and p^i_{t+1}(v) of Eq. 6).                                            */
/* ------------------------------------------------------------------------- */

/* For every row r of logits (one retained suffix position): ids[r, j] = the
 * j-th most probable token (j < k; equal logits: lower id first) and
 * probs[r, j] its probability under the softmax over the whole vocabulary
 * (fp32; Eq. 6 renormalizes them within the set at the next step, which is
 * what ssm_build_step_input's prev_topk_ids / prev_topk_prob take).
 *   logits     bf16 or fp32 [n_rows, vocab], rows 16-byte aligned (vocab *
 *              element size a multiple of 16 and logits 16-byte aligned;
 *              otherwise SSM_ERR_UNSUPPORTED)
 *   ids        int32 [n_rows, k];  probs  fp32 [n_rows, k]
 * 1 <= k <= 8 (SSM_ERR_UNSUPPORTED otherwise), k <= vocab; vocab up to
 * 2,744,320 (bf16) or 684,032 (fp32) entries (a row's per-slice maxima are kept
 * in shared memory; SSM_ERR_UNSUPPORTED beyond).  No workspace. */
ssm_status ssm_suffix_topk(const void* logits, ssm_dtype dtype, int64_t n_rows, int64_t vocab, int32_t k,
                           int32_t* ids, float* probs, ssm_stream_t stream);

/* ------------------------------------------------------------------------- */
/* 5. Prefix-cache append at a block boundary (prefix caching, "+PC." of      */
/*    Sec. 4.8, Table 4).                                                      */
/* ------------------------------------------------------------------------- */

/* Once a block is decoded, the keys and values of its rows join the prefix
 * cache that ssm_attention reads as already rotated: for every sequence b and
 * row i < n_rows,
 *   k_cache[b, start_row + i, h, :] = RoPE(k_new[b, i, h, :], pos[i], rope_theta)
 *   v_cache[b, start_row + i, h, :] = v_new[b, i, h, :]
 * with ssm_attention's rotation (the same bf16 bits as its pre-pass produces for
 * the same key and position).  Other cache rows are not touched.
 *   k_new, v_new      bf16 [batch, n_rows, h_kv, d]
 *   pos               int32 [n_rows] (shared by the batch)
 *   k_cache, v_cache  bf16 [batch, cache_rows, h_kv, d], caller-owned, written
 *                     in place; they must not overlap k_new / v_new.
 * d in {64, 128}; every bf16 pointer 16-byte aligned.  start_row + n_rows >
 * cache_rows returns SSM_ERR_CAPACITY and writes nothing. */
ssm_status ssm_cache_append(const void* k_new, const void* v_new, const int32_t* pos, int32_t batch,
                            int32_t n_rows, int32_t h_kv, int32_t head_dim, float rope_theta, void* k_cache,
                            void* v_cache, int64_t cache_rows, int64_t start_row, ssm_stream_t stream);

/* ------------------------------------------------------------------------- */
/* 6. Early termination after a decoded block (Sec. 3.2 "Early Termination"). */
/* ------------------------------------------------------------------------- */

/* For every sequence s with finished[s] == 0: if the generated tokens of block
 * block_idx (positions block_idx*block_len .. +block_len-1 of tokens[s]) hold
 * eos_id, set finished[s] = 1 and write eos_id at every generated position
 * after the first EOS (the rest of that block and every later block).
 * Sequences already finished are not touched.  n_active (optional, device
 * int32) receives the number of sequences still running after the call.
 *   tokens    int32 [batch, gen_len] (the generated region only), in place
 *   finished  uint8 [batch], in place
 * gen_len % block_len != 0 returns SSM_ERR_SHAPE; a block past the end returns
 * SSM_ERR_INVALID_ARG. */
ssm_status ssm_early_stop(int32_t* tokens, int32_t batch, int32_t gen_len, int32_t block_len, int32_t block_idx,
                          int32_t eos_id, uint8_t* finished, int32_t* n_active, ssm_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* SSM_H_ */
