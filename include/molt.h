/*
 * molt.h — C ABI of the GB300 (sm_103a) policy-update hot path of MOLT
 * (arxiv 2607.21653): GRPO group advantages, the LM-head log-probability /
 * entropy forward, and the fused clipped-surrogate forward + backward with the
 * token-mean normalisation of Eq. 2.
 *
 * Conventions shared by every call
 *   - All array pointers are DEVICE pointers owned by the caller; the library
 *     never frees them.  bf16 tensors are passed as their 16-bit patterns
 *     (uint16_t), row-major, 16-byte aligned.
 *   - Calls are asynchronous on `stream`.  Arguments are validated on the host
 *     before anything is launched; a non-OK return means nothing was launched
 *     and no output was written.  The thread-local molt_last_error() explains
 *     the last non-OK return.
 *   - Conditions that only the device can see (a token id out of range on an
 *     active row, a zero token count when the denominator is taken from the
 *     mask, unsorted group ids, a pipeline wait that timed out) set bits of a
 *     per-device status word that molt_device_status() reads and clears.
 *   - Workspace: calls that need scratch memory take (workspace, bytes).  The
 *     size comes from the matching *_workspace_bytes() query.  Passing NULL
 *     makes the call allocate and free it stream-ordered (cudaMallocAsync).
 *   - The library keeps no state between calls except cached device
 *     properties, the per-device status word, the kernel-launch counter, the
 *     no-allocation forward's fixed scratch array, and, for the loss call's
 *     vocabulary split and the zeroing of its backward targets, one side stream
 *     with fork, join and zeroed events per (device, caller stream), created on
 *     first use (at most 64, never while the
 *     caller's stream is being captured) and kept for the life of the process.
 *     It is safe to call from several threads on different streams with
 *     different workspaces; calls sharing a stream must come from one thread at
 *     a time (their launches would interleave on it).
 */
#ifndef MOLT_H_
#define MOLT_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MOLT_OK = 0,
  MOLT_ERR_INVALID_ARG = 1,       /* null / misaligned pointer, negative size, bad clip range */
  MOLT_ERR_UNSUPPORTED_SHAPE = 2, /* H not a positive multiple of 64, or a size beyond int32 */
  MOLT_ERR_UNSORTED_GROUPS = 3,   /* (device status) group ids decrease somewhere */
  MOLT_ERR_ZERO_DENOM = 4,        /* (device status) Eq. 2 denominator is zero */
  MOLT_ERR_CUDA = 5,              /* a CUDA runtime/driver call failed */
  MOLT_ERR_DEVICE_TIMEOUT = 6,    /* (device status) a pipeline wait gave up */
  MOLT_ERR_NO_MEMORY = 7,         /* workspace allocation failed */
  MOLT_ERR_TOKEN_RANGE = 8,       /* (device status) tokens[t] outside [0, V) on an active row */
  MOLT_ERR_WORKSPACE = 9          /* caller workspace smaller than *_workspace_bytes() */
} molt_status;

/* bits of the device status word */
#define MOLT_DEV_TIMEOUT 1u
#define MOLT_DEV_TOKEN_RANGE 2u
#define MOLT_DEV_ZERO_DENOM 4u
#define MOLT_DEV_UNSORTED_GROUPS 8u

/* Window statistics written (device memory) by molt_policy_loss_fwd_bwd.
 * Counts and sums run over active (mask = 1) tokens of this call. */
typedef struct {
  double denom;             /* D actually used in Eq. 2 */
  double loss;              /* sum_i m_i l_i / D */
  double sum_ratio;         /* sum of rho_i */
  double sum_entropy;       /* sum of per-token entropies (nats) */
  double max_abs_log_ratio; /* max |logp_i - b_i| */
  int64_t n_active;         /* sum_i m_i */
  int64_t n_clip_low;       /* tokens on the clipped branch with A_i < 0 (rho < 1 - eps_lo) */
  int64_t n_clip_high;      /* tokens on the clipped branch with A_i > 0 (rho > 1 + eps_hi) */
  int64_t n_grad_rows;      /* active tokens whose gradient coefficient is not 0: the rows
                               the backward processes (masked, clipped, A = 0 and rejected
                               rows carry no gradient and are left out) */
} molt_stats;

const char* molt_status_string(molt_status s);
/* Text of the last non-OK status returned on the calling thread. */
const char* molt_last_error(void);
int molt_version(void);
/* Process-wide number of CUDA kernels the library has enqueued so far (every
 * entry point and device; a call that fails part-way counts what it did
 * enqueue).  For launch accounting in benchmarks and tests. */
uint64_t molt_kernel_launches(void);

/* Self-test of the device-side wait bound (no paper counterpart).  One warp
 * waits, exactly as the deterministic backward's turn waits do, on a counter
 * that nothing raises: the wait gives up after its time limit (about 4 s),
 * sets MOLT_DEV_TIMEOUT in the status word and the kernel returns, leaving the
 * context usable.  Asynchronous on `stream` (scratch from cudaMallocAsync);
 * read the outcome with molt_device_status. */
molt_status molt_selftest_wait_timeout(cudaStream_t stream);

/* Synchronises `stream`, returns the current device's status word in *flags
 * (MOLT_DEV_* bits) and clears it.  Returns the molt_status of the highest
 * priority set bit (MOLT_OK if none). */
molt_status molt_device_status(cudaStream_t stream, uint32_t* flags);

/*
 * GRPO group-normalised advantages (Sec. 4.5 lists GRPO among the advantage
 * estimators; Sec. 4.2: segments of one rollout share its reward, which group
 * estimators count once).
 *   rewards   [n_resp] fp32, one reward per rollout (not per segment)
 *   group_ids [n_resp] int32, non-decreasing; a prompt group is a maximal
 *             run of equal consecutive ids.  An id smaller than its
 *             predecessor sets MOLT_DEV_UNSORTED_GROUPS (each run is still
 *             normalised on its own).
 *   eps       added to the unbiased (n-1) standard deviation
 *   adv_out   [n_resp] fp32: A_j = (r_j - mean_g) / (std_g + eps); groups of one
 *             response and zero-variance groups give exactly 0.
 * Arithmetic is fp64 in index order with correctly rounded operations, so the
 * result is bit-identical to a sequential fp64 evaluation rounded to fp32.
 */
molt_status molt_group_advantages(const float* rewards, const int32_t* group_ids, int64_t n_resp, double eps,
                                  float* adv_out, cudaStream_t stream);

/* The advantage estimators Sec. 4.5 lists, per rollout (one reward each):
 *   MOLT_ADV_GRPO          (r - mean_g) / (std_g + eps), unbiased std
 *                          (identical to molt_group_advantages)
 *   MOLT_ADV_GROUP_MEAN    r - mean_g (group-mean baseline)
 *   MOLT_ADV_DR_GRPO       r - mean_g: Dr. GRPO drops the std division; its
 *                          length normalisation is the token mean of Eq. 2
 *   MOLT_ADV_RLOO          r_j - (sum_g r - r_j) / (n_g - 1) (leave-one-out)
 *   MOLT_ADV_REINFORCE_PP  (r - mean_B) / (std_B + eps) over the whole batch;
 *                          group_ids is ignored and may be NULL
 * A group (or batch) of one response gives 0.  Same arithmetic contract as
 * molt_group_advantages: fp64 in index order, bit-identical to a sequential
 * fp64 evaluation rounded once to fp32. */
typedef enum {
  MOLT_ADV_GRPO = 0,
  MOLT_ADV_GROUP_MEAN = 1,
  MOLT_ADV_DR_GRPO = 2,
  MOLT_ADV_RLOO = 3,
  MOLT_ADV_REINFORCE_PP = 4
} molt_adv_estimator;
molt_status molt_advantages(const float* rewards, const int32_t* group_ids, int64_t n_resp, int estimator,
                            double eps, float* adv_out, cudaStream_t stream);

/* Per-token advantages: adv_tok[t] = adv_resp[resp_of_token[t]] (Sec. 4.2: the
 * rollout-level result is mapped back to its segments' tokens).
 * resp_of_token [T] int32 in [0, n_resp); out-of-range ids give 0. */
molt_status molt_broadcast_advantages(const float* adv_resp, const int32_t* resp_of_token, int64_t n_resp,
                                      int64_t T, float* adv_tok, cudaStream_t stream);

/* Number of active tokens sum_i m_i (the Eq. 2 denominator of one call),
 * written as an int64 to device memory `count_out`.  mask [T] uint8 (0/1). */
molt_status molt_mask_count(const uint8_t* mask, int64_t T, int64_t* count_out, cudaStream_t stream);

/*
 * Recomputed log-probabilities and entropies of the generated tokens
 * (Sec. 4.5: the actor's recomputed probabilities), without materialising the
 * [T, V] logits:
 *   z_tv = sum_k hidden[t,k] W[v,k];  lse_t = log sum_v exp z_tv
 *   logp_out[t] = z_{t,tokens[t]} - lse_t
 *   entropy_out[t] = lse_t - sum_v softmax(z_t)_v z_tv        (nats)
 *   hidden [T,H] bf16, W [V,H] bf16 (nn.Linear layout), tokens [T] int32,
 *   mask [T] uint8 or NULL (= all active).  Rows with mask 0 are skipped and
 *   their outputs are 0.  entropy_out may be NULL.
 * Shapes: T >= 0, V >= 1, H a positive multiple of 64, T, V < 2^31.
 * bf16 products accumulate in fp32 on the tensor cores; outputs are fp32.
 */
size_t molt_token_logprobs_workspace_bytes(int64_t T, int64_t H, int64_t V);
molt_status molt_token_logprobs_fwd(const uint16_t* hidden, const uint16_t* W, const int32_t* tokens,
                                    const uint8_t* mask, int64_t T, int64_t H, int64_t V, float* logp_out,
                                    float* entropy_out, void* workspace, size_t workspace_bytes,
                                    cudaStream_t stream);

/*
 * Fused clipped-surrogate policy loss with Eq. 2 normalisation, forward and
 * backward (Sec. 4.5):
 *   rho_t = exp(logp_t - behavior_logp[t])                 importance ratio
 *   l_t   = -min(rho_t A_t, clip(rho_t, 1 - clip_lo, 1 + clip_hi) A_t)
 *   loss  = sum_t m_t l_t / D,  D = denom if denom > 0, else sum_t m_t
 *   dL/dz_tv = (m_t / D) c_t (softmax(z_t)_v - [v == tokens[t]]),
 *              c_t = rho_t A_t on the unclipped branch, 0 on the clipped one
 *   dhidden = dL/dz W   [T,H] bf16 (rows with mask 0 are exactly 0)
 *   dW     (+)= dL/dz^T hidden   [V,H] fp32; accumulate_dW = 0 overwrites,
 *              1 adds to the caller's buffer (microbatches of one window).
 * Inputs: hidden [T,H] bf16, W [V,H] bf16, tokens [T] int32, behavior_logp [T]
 * fp32, adv [T] fp32 per-token advantages, mask [T] uint8 or NULL.
 * Use one window-wide `denom` for every microbatch of an optimizer window
 * (Eq. 2); with denom <= 0 and no active token the loss and gradients are 0
 * and MOLT_DEV_ZERO_DENOM is set.
 * Outputs: loss_out (device fp32 scalar), dhidden_out, dW_out; optional
 * (may be NULL): logp_out [T], entropy_out [T], token_loss_out [T] (= m_t l_t),
 * stats_out (device molt_stats).
 * The [T,V] logits and gradients never reach global memory: each vocab tile is
 * recomputed on chip in the backward pass and fed to the dhidden / dW tensor-
 * core products from shared memory.
 * Streams: all work is ordered on `stream`.  Part of the backward, and the
 * zeroing of dW and of the fp32 dhidden accumulator (during the forward), may
 * run on an internal lowest-priority stream of the library (one per device and
 * caller stream, created on the first such call), forked from `stream` and
 * joined back to it with events before the call's later work, so nothing needs
 * to be synchronised by the caller.  The call can be captured into a CUDA graph;
 * the side stream is only used under capture if an earlier uncaptured call on
 * the same stream created it.
 */
size_t molt_policy_loss_workspace_bytes(int64_t T, int64_t H, int64_t V);
molt_status molt_policy_loss_fwd_bwd(const uint16_t* hidden, const uint16_t* W, const int32_t* tokens,
                                     const float* behavior_logp, const float* adv, const uint8_t* mask,
                                     int64_t T, int64_t H, int64_t V, float clip_lo, float clip_hi,
                                     double denom, float* loss_out, uint16_t* dhidden_out, float* dW_out,
                                     int accumulate_dW, float* logp_out, float* entropy_out,
                                     float* token_loss_out, molt_stats* stats_out, void* workspace,
                                     size_t workspace_bytes, cudaStream_t stream);

/*
 * Extended objective (Sec. 4.5 lists KL control and rejection / weighting rules
 * among the configurable parts of the policy update).  Per active token t:
 *   l_t = w_t (l_pg,t + kl_coef KL_t - entropy_coef H_t)
 *   KL_t = exp(r_t) - r_t - 1,  r_t = ref_logp[t] - logp_t   (non-negative
 *          per-token estimator of KL(pi || pi_ref))
 *   H_t  = entropy of softmax(z_t); the bonus carries a gradient
 *   w_t  = sequence-gate weight in {0, 1}: a sequence is rejected (w = 0 on all
 *          its tokens) when the geometric mean of its active tokens' ratios,
 *          exp(mean_t (logp_t - behavior_logp[t])), lies outside
 *          [gate_lo, gate_hi].  D is not renormalised by the rejections (Eq. 2).
 *   dL/dz_tv = (m_t w_t / D) [ (c_t + kl_coef (exp(r_t) - 1)) (p_tv - [v == x_t])
 *                             + entropy_coef p_tv (z_tv - sum_u p_tu z_tu) ]
 * Fields:
 *   kl_coef       >= 0; 0 disables the KL term (ref_logp may then be NULL)
 *   entropy_coef  finite; 0 disables the bonus and its gradient
 *   ref_logp      [T] device fp32, reference-policy log-prob of tokens[t]
 *   seq_of_token  [T] device int32 sequence ids, non-decreasing (a sequence is
 *                 the run of tokens sharing an id); NULL disables the gate.
 *                 Decreasing ids set MOLT_DEV_UNSORTED_GROUPS.
 *   gate_lo, gate_hi   acceptance band of the geometric-mean ratio,
 *                 0 <= gate_lo <= gate_hi (gate_hi may be +inf)
 *   deterministic 1: dW and dhidden are bitwise reproducible for the same inputs
 *                 (no paper counterpart).  The backward then fixes the order of
 *                 every partial-sum reduction: the partial products of a
 *                 512-token quad x 512-column vocabulary block are reduce-added
 *                 into dW in token-quad order and into dhidden in vocabulary
 *                 block order, each [32 x 128] slab waiting its turn on a
 *                 counter in the workspace.  The order does not depend on the
 *                 number C of clusters of four CTAs the backward runs (see
 *                 det_clusters).  The C clusters wait on one another, so they
 *                 must be resident together: if other work keeps SMs busy for
 *                 seconds, a wait gives up after about 4 s, the call's backward
 *                 returns early with dW and dhidden incomplete, and
 *                 molt_device_status reports MOLT_ERR_DEVICE_TIMEOUT
 *                 (MOLT_DEV_TIMEOUT bit); nothing hangs.  Needs H % 128 == 0
 *                 (MOLT_ERR_UNSUPPORTED_SHAPE otherwise) and the workspace of
 *                 molt_policy_loss_workspace_bytes_ex (the raster's plus the
 *                 counters).  0: reduce-adds in arrival order (results agree
 *                 to fp32 rounding).
 *   det_clusters  deterministic mode only: the number C of clusters to run, a
 *                 multiple of 4 from 4 up to the number that fit on the device
 *                 at once (36 on a GB300); 0 takes that maximum.  A caller that
 *                 shares the GPU with other work can leave SMs to it with a
 *                 smaller C.  The results are the same bits for every C.  Other
 *                 values return MOLT_ERR_INVALID_ARG.
 */
typedef struct {
  float kl_coef;
  float entropy_coef;
  const float* ref_logp;
  const int32_t* seq_of_token;
  double gate_lo;
  double gate_hi;
  int deterministic;
  int det_clusters;
} molt_loss_options;

/* molt_stats plus the extended objective's counters (device memory). */
typedef struct {
  molt_stats base;           /* as above; n_clip_* count accepted tokens only */
  double sum_kl;             /* sum of KL_t over accepted active tokens */
  int64_t n_tokens_rejected; /* active tokens of rejected sequences */
  int64_t n_seq_rejected;    /* sequences (with at least one active token) rejected */
} molt_stats_ex;

/* Workspace of molt_policy_loss_fwd_bwd_ex with these options (opts may be
 * NULL); 0 for unsupported shapes.  Queries the current device. */
size_t molt_policy_loss_workspace_bytes_ex(int64_t T, int64_t H, int64_t V, const molt_loss_options* opts);

/*
 * molt_policy_loss_fwd_bwd with the extended objective above.  Arguments as in
 * molt_policy_loss_fwd_bwd; opts NULL (or all terms disabled) gives the same
 * results.  token_loss_out[t] = m_t l_t with the extended l_t.  The workspace
 * size is molt_policy_loss_workspace_bytes_ex(T, H, V, opts).
 */
molt_status molt_policy_loss_fwd_bwd_ex(const uint16_t* hidden, const uint16_t* W, const int32_t* tokens,
                                        const float* behavior_logp, const float* adv, const uint8_t* mask,
                                        int64_t T, int64_t H, int64_t V, float clip_lo, float clip_hi,
                                        double denom, const molt_loss_options* opts, float* loss_out,
                                        uint16_t* dhidden_out, float* dW_out, int accumulate_dW,
                                        float* logp_out, float* entropy_out, float* token_loss_out,
                                        molt_stats_ex* stats_out, void* workspace, size_t workspace_bytes,
                                        cudaStream_t stream);

/*
 * Vocabulary-parallel LM head (Sec. 4.1: the actor composes tensor parallelism
 * with FSDP2, Table 2 --fsdp.tp_size).  With W split by vocabulary rows over
 * n_shards ranks, rank r holding W_shard = W[v_begin_r, v_begin_r + V_r) with
 * the shards covering [0, V) in order, one policy-loss step is:
 *   1. every rank: molt_vp_partials on its shard -> partials_r [T, 4];
 *   2. the caller gathers them in shard order into partials [n_shards, T, 4]
 *      (an all-gather of 16 bytes per token);
 *   3. every rank: molt_vp_loss on the gathered statistics -> the loss of
 *      Eq. 2, lse and m c / D per token (identical on every rank);
 *   4. every rank: molt_vp_backward on its shard -> its dW shard and its
 *      contribution to dhidden; the caller sums the contributions over the
 *      ranks (an all-reduce of T x H fp32).
 * The library performs no collective; the exchange of steps 2 and 4 is the
 * caller's (NCCL, or any other transport).  Results agree with
 * molt_policy_loss_fwd_bwd on the whole W to fp32 rounding.
 */

/* Per-token statistics of one vocabulary shard:
 *   partials_out[t] = (M, S, Q, z_x) fp32, 16-byte aligned [T, 4], with z the
 *   logits of the shard's columns, M = max z, S = sum exp(z - M),
 *   Q = sum exp(z - M) (z - M), and z_x the logit of tokens[t] if it lies in
 *   [v_begin, v_begin + V_shard), else -inf.  Rows with mask 0 (mask may be
 *   NULL) get (-inf, 0, 0, -inf).
 * hidden [T,H] bf16, W_shard [V_shard,H] bf16, tokens [T] int32 (global ids).
 * Workspace as molt_token_logprobs_fwd (NULL allocates stream-ordered). */
size_t molt_vp_partials_workspace_bytes(int64_t T, int64_t H, int64_t V_shard);
molt_status molt_vp_partials(const uint16_t* hidden, const uint16_t* W_shard, const int32_t* tokens,
                             const uint8_t* mask, int64_t T, int64_t H, int64_t V_shard, int64_t v_begin,
                             float* partials_out, void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* Merge of the shards' statistics (partials [n_shards, T, 4], shard order,
 * 16-byte aligned) into each active row's lse = M + log S (M the largest
 * shard max, S = sum_s S_s exp(M_s - M)), logp = z_x - lse and entropy, then
 * the clipped surrogate and Eq. 2 exactly as molt_policy_loss_fwd_bwd's
 * forward half: loss_out (device fp32 scalar), lse_out [T] and coef_out [T]
 * (= m c / D, the inputs of molt_vp_backward; 0 on masked and clipped rows),
 * optional logp_out, entropy_out, token_loss_out [T] and stats_out (its
 * n_grad_rows counts the rows with coef != 0).  The reductions run in a fixed
 * order, so every rank that merges the same statistics gets the same bits.  A
 * row whose token lies in no shard sets MOLT_DEV_TOKEN_RANGE. */
size_t molt_vp_loss_workspace_bytes(int64_t T);
molt_status molt_vp_loss(const float* partials, int n_shards, const float* behavior_logp, const float* adv,
                         const uint8_t* mask, int64_t T, float clip_lo, float clip_hi, double denom, float* loss_out,
                         float* lse_out, float* coef_out, float* logp_out, float* entropy_out, float* token_loss_out,
                         molt_stats* stats_out, void* workspace, size_t workspace_bytes, cudaStream_t stream);

/* Backward of one shard: with g_tv = coef[t] (softmax(z_t)_v - [v == tokens[t]])
 * over the shard's columns (lse and coef from molt_vp_loss),
 *   dhidden_partial_out [T,H] fp32 = g W_shard (this shard's term of dhidden;
 *                                    rows with coef 0 are exactly 0)
 *   dW_shard_out [V_shard,H] fp32 (+)= g^T hidden (accumulate_dW as in
 *                                    molt_policy_loss_fwd_bwd).
 * Only rows with coef != 0 are computed.  16-byte-aligned outputs.  The
 * workspace holds the packed rows and an fp32 [T,H] accumulator. */
size_t molt_vp_backward_workspace_bytes(int64_t T, int64_t H, int64_t V_shard);
molt_status molt_vp_backward(const uint16_t* hidden, const uint16_t* W_shard, const int32_t* tokens,
                             const float* lse, const float* coef, int64_t T, int64_t H, int64_t V_shard,
                             int64_t v_begin, float* dhidden_partial_out, float* dW_shard_out, int accumulate_dW,
                             void* workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * Allocation-free variant of molt_token_logprobs_fwd (the paper has no
 * counterpart; it exists for callers, not for the method).
 *
 * Some callers cannot let a library allocate device memory: a training or
 * serving runtime that reserves the GPU's memory up front and hands it out only
 * through its own pool, or a process whose memory budget leaves nothing outside
 * that pool.  This call allocates nothing (no cudaMalloc, cudaMallocAsync or
 * cudaFree).  Its scratch is one fixed device array of about 4 MB, sized for
 * MOLT_NOALLOC_MAX_TOKENS tokens, that every GPU which loads the library keeps
 * until the process exits.  The caller still owns and passes all inputs and
 * outputs, with the same meaning as in molt_token_logprobs_fwd.
 *   - T > MOLT_NOALLOC_MAX_TOKENS returns MOLT_ERR_UNSUPPORTED_SHAPE and
 *     launches nothing; split larger batches into several calls.
 *   - All calls on a device share the one scratch array and each call leaves
 *     its contents behind (the call clears what it needs before use).  Calls
 *     whose kernels may overlap on the GPU (different streams, or different
 *     host threads, without ordering between them) race on that array: order
 *     them, e.g. by issuing them on one stream.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress, with that device current); later calls reuse it.
 *     A lookup that fails is not remembered: the next call tries again.
 *     Make the first call on a device before any stream capture on it.
 *   - The timing hook (molt_set_timing_events) records kernel groups 1 (the
 *     forward kernel) and 2 (the merge) of this call.
 * Masked rows are computed and then written as 0 (there is no compaction),
 * so prefer molt_token_logprobs_fwd when allocation is allowed.
 */
#define MOLT_NOALLOC_MAX_TOKENS 32768
molt_status molt_token_logprobs_fwd_noalloc(const uint16_t* hidden, const uint16_t* W, const int32_t* tokens,
                                            const uint8_t* mask, int64_t T, int64_t H, int64_t V,
                                            float* logp_out, float* entropy_out, cudaStream_t stream);

/*
 * Per-kernel timing hook for benchmarks.  While set, every LM-head call made
 * from the calling thread records starts[k] / stops[k] (caller-created CUDA
 * events) on its stream around kernel group k:
 *   k = 0  active-row compaction and packed gather
 *   k = 1  LM-head forward kernel (online log-softmax)
 *   k = 2  split merge, surrogate loss, the fixed-order reductions and the
 *          packing of the rows with a gradient for the backward
 *   k = 3  LM-head backward kernel (dhidden / dW products)
 *   k = 4  dhidden cast
 * Slots beyond n are ignored.  n = 0 (or NULL arrays) turns the hook off.
 * The arrays are read at each call, not copied: keep them alive while set.
 */
#define MOLT_TIMING_SLOTS 5
void molt_set_timing_events(cudaEvent_t* starts, cudaEvent_t* stops, int n);

#ifdef __cplusplus
}
#endif
#endif /* MOLT_H_ */
