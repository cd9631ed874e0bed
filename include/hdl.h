/*
 * libhdl -- GB300 (sm_103a) kernels for the hot path of Hindsight-Divergence
 * Localization (HDL, arXiv 2609.36864): teacher-forced re-scoring of every
 * root token under the original and the hindsight context, the per-token
 * hindsight-divergence score, top-k branch-point selection per root, the
 * allocation of continuations to branch points, and suffix-only loss masks.
 *
 * Conventions shared by every entry point
 *   - Array arguments are DEVICE pointers unless stated otherwise.  The caller
 *     owns every buffer; the library allocates no device memory and keeps no
 *     per-call state between calls.  (The one exception is the module's own
 *     static scratch array, which only hdl_rescore_noalloc uses; it is loaded
 *     with the library on each device, see there.)
 *   - Calls are asynchronous on `cuda_stream` (a cudaStream_t; NULL = the
 *     legacy default stream).  Argument errors are detected on the host and
 *     returned before anything is launched.  A failed launch returns
 *     HDL_ERR_CUDA.  Errors that only the device can see (a wait that ran out,
 *     a target id outside [0, vocab)) are recorded in the status word of the
 *     re-scoring workspace and read back with hdl_device_status().
 *   - Packed ragged layout: root r occupies tokens [root_offsets[r],
 *     root_offsets[r+1]) of the packed token arrays; positions reported per
 *     root (branch points) are relative to the root's first token.
 */
#ifndef HDL_H
#define HDL_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define HDL_ABI_VERSION 2

/* Exported symbols keep default visibility when the library is built with
 * -fvisibility=hidden. */
#if defined(__GNUC__)
#define HDL_API __attribute__((visibility("default")))
#else
#define HDL_API
#endif

typedef enum {
  HDL_OK = 0,
  HDL_ERR_INVALID_ARG = 1,  /* null pointer, negative size, misaligned buffer */
  HDL_ERR_UNSUPPORTED = 2,  /* valid but not supported (d % 64 != 0, k > 16, ...) */
  HDL_ERR_WORKSPACE = 3,    /* workspace missing or smaller than required */
  HDL_ERR_CUDA = 4,         /* a CUDA runtime/driver call or a launch failed */
  HDL_ERR_TIMEOUT = 5,      /* device: a pipeline wait ran out; outputs invalid */
  HDL_ERR_BAD_TARGET = 6    /* device: a target id outside [0, vocab) */
} hdl_status;

typedef enum { HDL_BF16 = 0, HDL_F32 = 1 } hdl_dtype;

/* Returns HDL_ABI_VERSION of the loaded library. */
HDL_API int32_t hdl_abi_version(void);

/* Static, human-readable name of a status code. */
HDL_API const char* hdl_status_string(hdl_status s);

/* ------------------------------------------------------------------------
 * Re-scoring: log p(y_t) under both contexts, and the divergence.
 *
 * Section 3.1, Eq. (hindsight-contexts): the same policy, the same root
 * prefix y_<t, two contexts; p^0_t = softmax(h^0_t W^T) and
 * p^H_t = softmax(h^H_t W^T) at temperature 1 (the rollout temperature,
 * Section 4.1).  Section 3.2, Eq. (div): delta_t = |log p^H_t(y_t) - log p^0_t(y_t)|.
 *
 *   h_orig, h_hind  [n_tokens, d] row-major hidden states (final layer,
 *                   after the final norm) of the original and the hindsight
 *                   context.  Row t is the state whose LM-head output
 *                   predicts targets[t] (the caller applies the usual causal
 *                   shift).  Element type `dt`; 16-byte aligned.
 *   w_lmhead        [vocab, d] row-major LM head (nn.Linear layout), type `dt`,
 *                   16-byte aligned; shared by both contexts.
 *   dt              HDL_BF16: bf16 inputs, bf16 x bf16 products with fp32
 *                   accumulation on the tensor cores.  HDL_F32: fp32 inputs
 *                   rounded to tf32 (to nearest), tf32 x tf32 products with
 *                   fp32 accumulation.
 *   targets         [n_tokens] int32 token ids y_t in [0, vocab).
 *   n_tokens        N >= 0 tokens per context (N == 0: returns HDL_OK, no launch).
 *   d               hidden size; a positive multiple of 64, at most 65536.
 *   vocab           V >= 1.
 *   logp_orig, logp_hind  [n_tokens] float outputs.
 *   delta           [n_tokens] float output, or NULL to skip it.
 *   workspace       device scratch of at least
 *                   hdl_rescore_workspace_bytes(n_tokens, d, vocab, dt) bytes,
 *                   256-byte aligned, owned by the caller.  Its first word is
 *                   the device status word; it and the merge counters after
 *                   it are cleared (one memset) at the start of each call.
 *                   Two calls in flight at once must not share a workspace.
 * The [2N, V] logits are never written to memory: one persistent tensor-core
 * kernel walks the vocabulary tiles, keeps a running max and sum of
 * exponentials per row and picks out the target logit; the same kernel
 * merges the per-vocabulary-chunk partial sums of each 32 tokens as soon as
 * the last of them is written (one memset + one kernel launch per call).
 */
HDL_API size_t hdl_rescore_workspace_bytes(int64_t n_tokens, int32_t d, int32_t vocab,
                                   hdl_dtype dt);

HDL_API hdl_status hdl_rescore(const void* h_orig, const void* h_hind,
                       const void* w_lmhead, hdl_dtype dt,
                       const int32_t* targets, int64_t n_tokens, int32_t d,
                       int32_t vocab, float* logp_orig, float* logp_hind,
                       float* delta, void* workspace, size_t workspace_bytes,
                       void* cuda_stream);

/* Options of hdl_rescore_ex.  A zero-initialised struct (or NULL) gives
 * exactly hdl_rescore. */
typedef struct {
  /* [n_tokens] float outputs or NULL: the entropy (nats) of the next-token
   * distribution, H_t = -sum_v p_t(v) log p_t(v), under the original / the
   * hindsight context -- the ranking signal of the paper's Entropy selector
   * (Section 4.1, "Rollout protocols"; the paper uses the original context).
   * Computed in the same vocabulary walk (one more multiply-add per logit),
   * as log Z - E_p[z]. */
  float* entropy_orig;
  float* entropy_hind;
  /* Limit of each pipeline wait inside the kernel, ns; 0 = 4 s. */
  uint64_t wait_timeout_ns;
  /* Test hook, 0 in normal use.  Bit 0: the kernel's copy producer issues no
   * loads, so the first pipeline wait runs out after wait_timeout_ns and the
   * call reports HDL_ERR_TIMEOUT through hdl_device_status (nothing faults or
   * hangs).  Other bits: HDL_ERR_INVALID_ARG. */
  uint32_t fault_inject;
  uint32_t reserved;
} hdl_rescore_opts;

/* Workspace of hdl_rescore_ex with these options (entropy outputs need
 * 4 more bytes per row and vocabulary chunk); 0 for unsupported shapes. */
HDL_API size_t hdl_rescore_ex_workspace_bytes(int64_t n_tokens, int32_t d, int32_t vocab,
                                      hdl_dtype dt, const hdl_rescore_opts* opts);

/* hdl_rescore with options (opts may be NULL).  Same arguments, layout,
 * ownership and errors as hdl_rescore; the workspace must hold
 * hdl_rescore_ex_workspace_bytes(..., opts) bytes. */
HDL_API hdl_status hdl_rescore_ex(const void* h_orig, const void* h_hind,
                          const void* w_lmhead, hdl_dtype dt,
                          const int32_t* targets, int64_t n_tokens, int32_t d,
                          int32_t vocab, float* logp_orig, float* logp_hind,
                          float* delta, const hdl_rescore_opts* opts,
                          void* workspace, size_t workspace_bytes,
                          void* cuda_stream);

/* ------------------------------------------------------------------------
 * Vocabulary-parallel re-scoring (a tensor-parallel LM head: each GPU holds
 * rows [vocab_offset, vocab_offset + vocab_shard) of W).  The softmax
 * normaliser of Section 3.1 splits over shards exactly: with per-shard
 * m_p = max z (log2 units) and s_p = sum 2^(z log2e - m_p),
 *   log Z = ln2 * (M + log2 sum_p s_p 2^(m_p - M)),  M = max_p m_p,
 * so one exchange of 16 bytes per row and context (e.g. an all-gather)
 * followed by hdl_merge_vocab_shards gives the same log-probs as one GPU.
 *
 * hdl_rescore_shard writes stats, [2][n_tokens] float4 (context 0 = original,
 * 16-byte aligned): x = m_p, y = s_p, z = the target logit z_{y_t} if this
 * shard holds y_t else NaN, w = sum 2^(z log2e - m_p) * z (for the entropy).
 * Arguments otherwise as hdl_rescore (w_shard is [vocab_shard, d]; targets
 * are global ids); the workspace holds
 * hdl_rescore_shard_workspace_bytes(n_tokens, d, vocab_shard, dt) bytes. */
HDL_API size_t hdl_rescore_shard_workspace_bytes(int64_t n_tokens, int32_t d,
                                         int32_t vocab_shard, hdl_dtype dt);

HDL_API hdl_status hdl_rescore_shard(const void* h_orig, const void* h_hind,
                             const void* w_shard, hdl_dtype dt,
                             const int32_t* targets, int64_t n_tokens, int32_t d,
                             int32_t vocab_shard, int32_t vocab_offset,
                             float* stats, void* workspace,
                             size_t workspace_bytes, void* cuda_stream);

/* Merge n_shards shards' stats, laid out back to back (shard p at
 * stats + p * 2 * n_tokens * 4 floats), into log-probs, |Delta| and
 * (optional, NULL to skip) entropies.  A token whose target no shard holds
 * gets NaN log-probs.  delta, entropy_orig, entropy_hind may be NULL. */
HDL_API hdl_status hdl_merge_vocab_shards(const float* stats, int32_t n_shards,
                                  int64_t n_tokens, float* logp_orig,
                                  float* logp_hind, float* delta,
                                  float* entropy_orig, float* entropy_hind,
                                  void* cuda_stream);

/* ------------------------------------------------------------------------
 * The update after branch selection: group-relative advantages and the
 * clipped, token-aggregated policy loss on the suffix-only masks.
 *
 * Section 3: A_j = R_j - (1/G) sum_{k in group} R_k (no standard-deviation
 * normalisation, Section 4.1); the group's roots and continuations form one
 * group (Section 3.3).  Section 4.1 "Training": asymmetric clipping with
 * thresholds 0.2 / 0.28, no KL penalty, losses aggregated at the token level:
 *   r_t = exp(logp_new_t - logp_old_t),
 *   obj_t = min(r_t A_j, clip(r_t, 1 - eps_low, 1 + eps_high) A_j),
 *   loss = - sum_t mask_t obj_t / sum_t mask_t,
 *   grad_t = d loss / d logp_new_t (= -mask_t r_t A_j / sum mask when the
 *            unclipped term is the minimum, else 0).
 *
 *   logp_new, logp_old  [n_tokens] float, packed trajectories.
 *   mask            [n_tokens] uint8: the loss mask (hdl_suffix_mask for
 *                   continuations, the valid mask for roots).
 *   traj_offsets    [n_traj + 1] int64, non-decreasing: trajectory j = tokens
 *                   [traj_offsets[j], traj_offsets[j+1]); they should cover
 *                   [0, n_tokens) (tokens outside every trajectory carry no loss).
 *   rewards         [n_traj] float verifier rewards.
 *   group_offsets   [n_groups + 1] int32: group g = trajectories
 *                   [group_offsets[g], group_offsets[g+1]).
 *   eps_low, eps_high  clip thresholds, 0 <= eps_low < 1, eps_high >= 0.
 *   advantages      [n_traj] float out, NULL only when n_traj == 0
 *                   (trajectories outside every group are not written).
 *   grad            [n_tokens] float out or NULL.
 *   stats           [4] float out: loss, masked tokens, fraction of masked
 *                   tokens whose clipped term is strictly smaller, mean ratio.
 *   workspace       hdl_grpo_loss_workspace_bytes() bytes, 256-byte aligned.
 * The loss is reduced in double precision in a fixed order.  Every array is
 * aligned to its element type; the token streams are read 16 bytes at a time
 * when the addresses of logp_new, logp_old and grad (/ 4) and of mask agree
 * mod 4, else one token at a time (same results). */
HDL_API size_t hdl_grpo_loss_workspace_bytes(void);

HDL_API hdl_status hdl_grpo_loss(const float* logp_new, const float* logp_old,
                         const uint8_t* mask, int64_t n_tokens,
                         const int64_t* traj_offsets, int32_t n_traj,
                         const float* rewards, const int32_t* group_offsets,
                         int32_t n_groups, float eps_low, float eps_high,
                         float* advantages, float* grad, float* stats,
                         void* workspace, size_t workspace_bytes,
                         void* cuda_stream);

/* Allocation-free variant of hdl_rescore (the paper has no counterpart: this
 * is an interface convenience).  It is for callers that must not allocate
 * device memory while they run: plugin "enqueue" callbacks of inference
 * runtimes, which forbid allocation during enqueue; processes whose device
 * memory is owned by a pooling allocator, where a cudaMalloc can fail or
 * fragment the pool; and latency-critical loops, where cudaMalloc/cudaFree
 * can synchronise the device.  Instead of a caller-provided workspace it uses
 * one file-scope device array of HDL_STATIC_SCRATCH_BYTES (64 MiB) that every
 * GPU which loads the library holds until the process exits.  It calls no
 * cudaMalloc, cudaFree or allocating library routine.
 *
 * Arguments and results are those of hdl_rescore, without the workspace.
 *   - Returns HDL_ERR_UNSUPPORTED, before launching anything, when the
 *     problem needs more than HDL_STATIC_SCRATCH_BYTES of scratch, i.e. when
 *     hdl_rescore_workspace_bytes(n_tokens, d, vocab, dt) exceeds it
 *     (e.g. at d = 3584, vocab = 152064 about 28,000 tokens fit; at d = 2048,
 *     vocab = 32000 about 250,000).
 *   - The first call on a device looks up the array's device address (with
 *     that device current) and caches it, keyed on the context's
 *     process-unique id; make that first call before any stream capture.  A
 *     call from a new context of the device (for instance after
 *     cudaDeviceReset re-created the primary context) looks the address up
 *     again, so that call, too, should come before any capture.
 *   - Every call on a device shares the one array and leaves its contents
 *     behind; each call clears the status word it needs.  Calls that overlap
 *     on the GPU (e.g. on two streams at once) race on the array: serialise
 *     them.
 *   - scratch_out (host pointer, may be NULL) receives the array's device
 *     address, which hdl_device_status() accepts (with
 *     HDL_STATIC_SCRATCH_BYTES) to read the device status of the last call. */
#define HDL_STATIC_SCRATCH_BYTES ((size_t)64 << 20)

HDL_API hdl_status hdl_rescore_noalloc(const void* h_orig, const void* h_hind,
                               const void* w_lmhead, hdl_dtype dt,
                               const int32_t* targets, int64_t n_tokens,
                               int32_t d, int32_t vocab, float* logp_orig,
                               float* logp_hind, float* delta,
                               const void** scratch_out, void* cuda_stream);

/* Synchronises `cuda_stream`, then reads the status word of a re-scoring
 * workspace.  Returns HDL_OK, HDL_ERR_TIMEOUT or HDL_ERR_BAD_TARGET (the
 * device condition), or HDL_ERR_CUDA / HDL_ERR_INVALID_ARG for the call
 * itself.  `raw_word` (host pointer, may be NULL) receives the raw status
 * bits: bit 0 timeout, bit 1 bad target, bits 8..15 the pipeline role that
 * timed out first (1 producer, 2 MMA issuer, 3 epilogue). */
HDL_API hdl_status hdl_device_status(const void* workspace, size_t workspace_bytes,
                             void* cuda_stream, uint32_t* raw_word);

/* ------------------------------------------------------------------------
 * Branch-point selection (Section 3.2: rank each root's candidate positions
 * by delta and take the highest; Section 3.1: only policy-generated tokens
 * are candidates; Section 4.4: of points that sit too near each other only
 * one is kept).
 *
 * For root r the candidates are positions t (relative to the root start) in
 * the window [lo, hi) -- hi <= 0 means the root's end -- with valid != 0 and
 * a delta that is not NaN.  They are ranked by delta, descending, ties to the
 * lower t (the paper does not fix a tie rule).
 *   min_gap == 0: the first k ranked candidates.
 *   min_gap > 0, gap_mode 0 (greedy): walk the ranked list, skip every point
 *       with |t - a| < min_gap for an accepted a, stop at k points.
 *   min_gap > 0, gap_mode 1 (drop-lower): take the first k ranked candidates,
 *       then drop, in rank order, every point with |t - a| < min_gap for a
 *       kept higher-ranked a.
 */
typedef struct {
  int32_t min_gap;   /* 0 = no spacing rule (default) */
  int32_t gap_mode;  /* 0 = greedy, 1 = drop-lower */
  int32_t lo, hi;    /* candidate window relative to the root start */
} hdl_select_opts;

/*   delta          [n_tokens] float scores (e.g. the output of hdl_rescore).
 *   valid          [n_tokens] uint8, nonzero = policy-generated, or NULL (all).
 *   n_tokens       length of delta/valid; tokens outside [0, n_tokens) are
 *                  never read (a root reaching past it loses those positions).
 *   root_offsets   [n_roots + 1] int64, non-decreasing (a root whose end is
 *                  before its start is treated as empty).
 *   k              0 <= k <= 16.
 *   opts           NULL = {0, 0, 0, 0}.  min_gap >= 0, gap_mode in {0, 1}.
 *   branch_pos     [n_roots * k] int32 out: root-relative positions in rank
 *                  order, -1 after the last selected one.
 *   n_selected     [n_roots] int32 out: number of points selected (<= k).
 *   branch_delta   [n_roots * k] float out or NULL: delta at each point, NaN
 *                  padding.
 * Every array is aligned to its element type.  The scores are read 16 bytes
 * at a time when delta's address / 4 and valid's address agree mod 4 (both
 * from the same token offset of aligned buffers, for instance), else one
 * element at a time (same results). */
HDL_API hdl_status hdl_select_branches(const float* delta, const uint8_t* valid,
                               int64_t n_tokens, const int64_t* root_offsets,
                               int32_t n_roots, int32_t k,
                               const hdl_select_opts* opts, int32_t* branch_pos,
                               int32_t* n_selected, float* branch_delta,
                               void* cuda_stream);

/* ------------------------------------------------------------------------
 * Continuation allocation (Section 4.1: two points per root with three and
 * four continuations, G = 2 x (1 + 3 + 4) = 16; Table fork-ablation: 2x1 -> 7,
 * 4x2 -> 1 + 2; Section 4.4: a root left with one point samples all of its
 * continuations from it).
 *
 * Root r's conts_per_root[r] continuations are laid out after those of
 * roots < r.  Over its n = n_selected[r] points (rank order) point j gets
 * floor(C / n) + [j < C mod n] continuations (extra_to_higher != 0) or
 * floor(C / n) + [j >= n - C mod n] (extra_to_higher == 0), consecutively.
 *   n_selected, branch_pos  as written by hdl_select_branches (same k).
 *   conts_per_root  [n_roots] int32 (negative counts as 0).
 *   cont_branch     [n_cont_capacity] int32 out: each continuation's
 *                   root-relative branch position; -1 if its root has no
 *                   point.  Entries past n_cont_capacity are not written. */
HDL_API hdl_status hdl_assign_continuations(const int32_t* n_selected,
                                    const int32_t* branch_pos, int32_t n_roots,
                                    int32_t k, const int32_t* conts_per_root,
                                    int32_t extra_to_higher,
                                    int32_t* cont_branch,
                                    int64_t n_cont_capacity, void* cuda_stream);

/* ------------------------------------------------------------------------
 * Suffix-only loss mask (Section 3.3: a root is trained on all its generated
 * tokens; a continuation y~ = y_<i || y~_>=i of Eq. (branch-sampling) only on
 * the newly sampled tokens, positions >= i, including i itself).
 *
 * Continuation c occupies mask bytes [cont_offsets[c], cont_offsets[c+1]);
 * its token t (relative to its start) gets
 *     mask = (b >= 0) && (t >= b) && (cont_valid == NULL || cont_valid[.] != 0)
 * with b = cont_branch[c].  Pass b = 0 for a root (mask = its valid tokens).
 *   cont_offsets  [n_cont + 1] int64, non-decreasing.
 *   cont_valid    [mask_len] uint8, same packing as mask, or NULL.
 *   mask          [mask_len] uint8 out; bytes outside
 *                 [cont_offsets[0], cont_offsets[n_cont]) are left untouched.
 * 16-byte vectors are used when mask and cont_valid have the same address
 * mod 16, else single bytes (same results).
 */
HDL_API hdl_status hdl_suffix_mask(const int32_t* cont_branch,
                           const int64_t* cont_offsets, int32_t n_cont,
                           const uint8_t* cont_valid, uint8_t* mask,
                           int64_t mask_len, void* cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* HDL_H */
