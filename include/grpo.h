/*
 * grpo.h -- C ABI of the fused GRPO token-scoring + loss + backward library (GB300, sm_103a).
 *
 * One GRPO update (arxiv 2510.17158, Alg. 1) scores K sampled completions per prompt, normalises
 * their rewards within the group, and takes a gradient step on
 *     L = E_{x~pi}[ -w(x) log pi(x|c) ] + beta KL(pi || pi_ref)                  (Eq. 1)
 * using the clipped-ratio surrogate of standard GRPO, which Sec. 6.1 keeps. This library
 * computes the data-parallel core of that step for the LM head: logits z = W h per token over
 * the whole vocabulary (never written to memory), log-softmax at the sampled token, entropy and
 * argmax, group advantages, the per-token surrogate + KL loss, and dL/dH, dL/dW.
 *
 * Conventions (every entry point):
 *  - All array arguments are DEVICE pointers unless stated; the caller owns every buffer, the
 *    workspace and the stream. The library allocates and frees nothing and never synchronises,
 *    except grpo_last_device_error() and grpo_timing_read(), which say so.
 *  - Work is enqueued asynchronously on `stream` (a cudaStream_t; 0 = legacy default stream).
 *    Outputs are overwritten, never accumulated into.
 *  - Layouts are row-major and contiguous:
 *      H       [S, T, d]   hidden states of every position (bf16 or f32; padding must be finite)
 *      W       [V, d]      LM-head weight (same dtype as H)
 *      tokens  [S, T]      int32 sampled token ids, in [0, V) where mask != 0
 *      mask    [S, T]      uint8, nonzero = scored completion token (prompt padding, tool-result
 *                          text and tail padding are 0; holes inside a completion are allowed)
 *      per-token f32 arrays [S, T]; per-sequence arrays [S].
 *    Sequences of one group are contiguous: group g owns sequences
 *    group_offsets[g] .. group_offsets[g+1]-1.
 *  - Host-side argument checks run before any launch and return a negative status with nothing
 *    enqueued. Faults only the device can see (a token id outside [0, V) at a scored position,
 *    invalid group offsets, a bounded wait that ran out) write a status word in the workspace;
 *    read it with grpo_last_device_error().
 *  - Unscored positions get logp = lse = entropy = 0, argmax = -1, g = 0 and dH rows = 0.
 */
#ifndef GRPO_GB300_H
#define GRPO_GB300_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* grpo_stream_t; /* same object as cudaStream_t */

typedef enum {
  GRPO_OK = 0,
  GRPO_ERR_INVALID_ARG = -1,  /* null pointer, non-positive size, bad enum, ...            */
  GRPO_ERR_UNSUPPORTED = -2,  /* shape/dtype combination this build does not implement     */
  GRPO_ERR_CUDA = -3,         /* a CUDA runtime call or a launch failed                      */
  GRPO_ERR_WORKSPACE = -4,    /* workspace too small or misaligned                           */
  GRPO_ERR_TOKEN_RANGE = -5,  /* device: a scored token id outside [0, V)                    */
  GRPO_ERR_TIMEOUT = -6,      /* device: a bounded wait inside a kernel ran out              */
  GRPO_ERR_GROUPS = -7        /* device: group offsets not non-decreasing from 0 to S        */
} grpo_status;

typedef enum { GRPO_F32 = 0, GRPO_BF16 = 1 } grpo_dtype;
typedef enum { GRPO_STD_UNBIASED = 0, GRPO_STD_POPULATION = 1 } grpo_std_mode;
typedef enum { GRPO_AGG_SEQ_MEAN = 0, GRPO_AGG_TOKEN_MEAN = 1 } grpo_agg;

/* Bytes of workspace needed for a problem of this shape. `vocab_chunk` is how many vocabulary
 * columns of dL/dz the backward keeps at once (rounded up to a multiple of 256); 0 = the whole
 * vocabulary in one chunk (fastest; S*ceil(T/128)*128*V*2 bytes of scratch). Returns 0 for
 * invalid shapes. The workspace must be 256-byte aligned. With less than this, the backward
 * takes the widest vocabulary chunk that fits next to an f32 dH accumulator, and returns
 * GRPO_ERR_WORKSPACE only if not even the fixed regions and one 256-column chunk fit. The
 * exact-KL entry points (grpo_score_fwd_kl, grpo_loss_bwd_kl) also hold the reference model's
 * packed hidden states and forward statistics: grpo_workspace_bytes_kl gives their size for the
 * same chunking (bf16 only; 0 for f32), and a workspace of that size serves every entry point. */
size_t grpo_workspace_bytes(int32_t S, int32_t T, int32_t d, int32_t V, int32_t dtype,
                            int32_t vocab_chunk);
size_t grpo_workspace_bytes_kl(int32_t S, int32_t T, int32_t d, int32_t V, int32_t dtype,
                               int32_t vocab_chunk);

/* Clears the workspace's status word. Call once after allocating a workspace. */
int grpo_workspace_init(void* workspace, size_t workspace_bytes, grpo_stream_t stream);

/* Group-relative advantages (Eq. 1's w(x): rewards normalised within each group, Sec. 2.1 and
 * Alg. 1).
 *   rewards        [num_seqs] f32
 *   group_offsets  [num_groups+1] int32, device; must rise from 0 to num_seqs (else the status
 *                  word gets GRPO_ERR_GROUPS and the affected advantages are NaN)
 *   adv_out        [num_seqs] f32: (r - mean_g) / (std_g + std_eps); std unbiased (default) or
 *                  population; exactly 0 for a group of one or a group whose rewards are all equal
 * Needs >= 256 bytes of workspace (status word only). */
int group_advantages(const float* rewards, const int32_t* group_offsets, int32_t num_groups,
                     int32_t num_seqs, int32_t std_mode, float std_eps, float* adv_out,
                     void* workspace, size_t workspace_bytes, grpo_stream_t stream);

/* Forward scoring of Eq. 1's log pi(x|c) per token: z_t = W h_t over all V columns, reduced on
 * chip (the [tokens x V] logits never reach memory) to
 *   lse_t = log sum_v exp(z_tv), logp_t = z_t[y_t] - lse_t, entropy_t = lse_t - sum_v p_tv z_tv
 *   (nats), argmax_t = lowest v with the largest z_tv; valid_count_i = #scored tokens of seq i.
 * dtype GRPO_BF16: bf16 H, W, tensor-core products with f32 accumulation (d % 64 == 0).
 * dtype GRPO_F32 : f32 H, W, f32 CUDA-core arithmetic (small problems, d <= 4096).
 * Outputs: logp, lse, entropy f32 [S,T]; argmax int32 [S,T]; valid_count int32 [S]. */
int grpo_score_fwd(const void* H, const void* W, int32_t dtype, const int32_t* tokens,
                   const uint8_t* mask, int32_t S, int32_t T, int32_t d, int32_t V, float* logp,
                   float* lse, float* entropy, int32_t* argmax, int32_t* valid_count,
                   void* workspace, size_t workspace_bytes, grpo_stream_t stream);

/* Bytes of the library-owned device scratch array used by grpo_score_fwd_static. */
#define GRPO_STATIC_SCRATCH_BYTES (64u * 1024u * 1024u)

/* grpo_score_fwd without a workspace, for callers that cannot allocate device memory -- e.g. a
 * plugin whose host framework owns every device allocation and forbids extensions from making
 * their own, or a latency-critical section where an allocation (which can synchronise the
 * device) is not allowed. The paper has no counterpart; this is a deployment convenience.
 * Arguments, outputs and results are those of grpo_score_fwd, except:
 *  - the scratch is a GRPO_STATIC_SCRATCH_BYTES (64 MiB) __device__ array inside the library,
 *    held on every GPU that loads the library until the process exits. A batch whose scratch
 *    (for bf16 about R * (16 * ceil(V/256) + 2 * d + 4) + 8 * S*T bytes, R = S*T rounded up to
 *    a multiple of 128) does not fit returns GRPO_ERR_WORKSPACE before anything is enqueued;
 *  - it allocates nothing and calls no allocating routine;
 *  - the first call made with a given device current looks up the array's device address
 *    (cudaGetSymbolAddress) and caches it: make that first call before any stream capture (a
 *    first call inside a capture returns GRPO_ERR_CUDA). Later calls whose stream is not being
 *    captured look the address up again, so a context re-created by cudaDeviceReset is handled;
 *    calls inside a capture use the cached address;
 *  - its launches are counted by the kernel accounting below like those of grpo_score_fwd, and
 *    grpo_debug_inject_stall applies to its tensor-core GEMM;
 *  - all calls share the one array and each overwrites it: calls that overlap on the GPU
 *    (different streams, or different host threads on one device) race and corrupt each
 *    other's results;
 *  - the device status word (e.g. GRPO_ERR_TOKEN_RANGE) is cleared at the start of each call and
 *    copied at its end into *status_out (one device int32; may be NULL). */
int grpo_score_fwd_static(const void* H, const void* W, int32_t dtype, const int32_t* tokens,
                          const uint8_t* mask, int32_t S, int32_t T, int32_t d, int32_t V,
                          float* logp, float* lse, float* entropy, int32_t* argmax,
                          int32_t* valid_count, int32_t* status_out, grpo_stream_t stream);

/* GRPO loss and its gradient (Eq. 1 with the clipped-ratio surrogate of Sec. 6.1; Alg. 1's
 * gradient step), per scored token t of sequence i:
 *   rho = exp(logp - old_logp);  surr = min(rho A_i, clip(rho, 1-eps_low, 1+eps_high) A_i)
 *   delta = ref_logp - logp;     kl = e^delta - delta - 1;      l_t = -surr + beta kl
 *   L = (1/S') sum_i (1/n_i) sum_t l_t   (GRPO_AGG_SEQ_MEAN)   or   sum l_t / N' (TOKEN_MEAN)
 * where S' = S and N' = sum_i n_i unless `norm` > 0 overrides them (data-parallel shards pass
 * the global count). g_t = dL/dlogp_t takes the unclipped branch when it is active, boundaries
 * inclusive. Then dz_t = g_t (onehot(y_t) - softmax(z_t)) is recomputed from H, W and lse,
 * rounded to bf16, and contracted: dH_t = dz_t W (written in H's dtype), dW = sum_t dz_t h_t
 * (f32). logp/lse/valid_count are grpo_score_fwd's outputs for the same H, W, tokens, mask.
 * ref_logp may be NULL only when beta == 0. loss_out is one device f32. */
int grpo_loss_bwd(const void* H, const void* W, int32_t dtype, const int32_t* tokens,
                  const uint8_t* mask, int32_t S, int32_t T, int32_t d, int32_t V,
                  const float* logp, const float* lse, const float* old_logp,
                  const float* ref_logp, const float* adv, const int32_t* valid_count,
                  float eps_low, float eps_high, float beta, int32_t agg, double norm,
                  float* loss_out, void* dH, float* dW, void* workspace, size_t workspace_bytes,
                  grpo_stream_t stream);

/* Distillation loss and gradient (Sec. 6.2: the small model is fine-tuned by supervised
 * learning on the large model's filtered traces, tool-call tokens kept in the targets): token
 * cross-entropy l_t = -logp_t over the scored tokens, aggregated like grpo_loss_bwd
 * (GRPO_AGG_TOKEN_MEAN is the usual choice), so g_t = -w_t; then the same recompute + dz + dH +
 * dW contractions as grpo_loss_bwd. Arguments as in grpo_loss_bwd. */
int grpo_sft_loss_bwd(const void* H, const void* W, int32_t dtype, const int32_t* tokens,
                      const uint8_t* mask, int32_t S, int32_t T, int32_t d, int32_t V,
                      const float* logp, const float* lse, const int32_t* valid_count,
                      int32_t agg, double norm, float* loss_out, void* dH, float* dW,
                      void* workspace, size_t workspace_bytes, grpo_stream_t stream);

/* Rewards of n completions (Eq. 2: r = r_perf + r_tools), the input of group_advantages:
 *   r_perf (Eq. 3) = -2 if correct[i] == 0; -1 if t_new[i] > t_base[i] (correct but slower);
 *                    else min(10, t_base[i] / t_new[i] - 1)
 *   r_tools (Eq. 4) = lambda_tools * tools_used[i] / tools_avail[i] (the paper: 0.5; unique
 *                    tools used out of the 4-6 made available); NaN unless
 *                    0 <= tools_used <= tools_avail and tools_avail >= 1.
 * correct uint8 [n], t_base / t_new f32 [n] (seconds), tools_used / tools_avail int32 [n],
 * r_out f32 [n]. */
int grpo_rewards(const uint8_t* correct, const float* t_base, const float* t_new,
                 const int32_t* tools_used, const int32_t* tools_avail, int32_t n,
                 float lambda_tools, float* r_out, grpo_stream_t stream);

/* Exact KL variant. Eq. 1 writes the full-distribution KL(pi_theta(.|c) || pi_ref(.|c)); with
 * the frozen reference model of Alg. 1 (same d and V) its per-position term is
 *   KL_t = sum_v p_tv (log p_tv - log q_tv),  p = softmax(W h_t),  q = softmax(W_ref h_ref_t).
 * grpo_score_fwd_kl computes grpo_score_fwd's outputs plus lse_ref [S,T] and kl [S,T] (0 at
 * unscored positions); both products stream through one tensor-core tile per 128 x 256 block,
 * the logits of neither model reach memory. H_ref [S,T,d], W_ref [V,d] bf16. Workspace:
 * grpo_workspace_bytes_kl. */
int grpo_score_fwd_kl(const void* H, const void* W, const void* H_ref, const void* W_ref,
                      int32_t dtype, const int32_t* tokens, const uint8_t* mask, int32_t S,
                      int32_t T, int32_t d, int32_t V, float* logp, float* lse, float* entropy,
                      int32_t* argmax, int32_t* valid_count, float* lse_ref, float* kl,
                      void* workspace, size_t workspace_bytes, grpo_stream_t stream);

/* grpo_loss_bwd with the exact KL: l_t = -surr_t + beta KL_t (the clipped surrogate as in
 * grpo_loss_bwd), and dz_t = g_t (onehot(y_t) - p_t) + beta w_t p_t (log p_t - log q_t - KL_t)
 * from both recomputed products; dH, dW as in grpo_loss_bwd (nothing flows to the frozen
 * reference). logp, lse, lse_ref, kl are grpo_score_fwd_kl's outputs. bf16 only. Workspace:
 * grpo_workspace_bytes_kl. */
int grpo_loss_bwd_kl(const void* H, const void* W, const void* H_ref, const void* W_ref,
                     int32_t dtype, const int32_t* tokens, const uint8_t* mask, int32_t S,
                     int32_t T, int32_t d, int32_t V, const float* logp, const float* lse,
                     const float* lse_ref, const float* kl, const float* old_logp,
                     const float* adv, const int32_t* valid_count, float eps_low, float eps_high,
                     float beta, int32_t agg, double norm, float* loss_out, void* dH, float* dW,
                     void* workspace, size_t workspace_bytes, grpo_stream_t stream);

/* Vocabulary-parallel (tensor-parallel) variant. The paper shards the policy over GPUs with
 * tensor parallelism (Sec. 6.3); sharding the LM head by vocabulary rows needs one exchange of
 * per-token statistics after the forward and one sum of dH after the backward.
 *
 * grpo_score_fwd_shard: this rank holds rows [v_offset, v_offset + V_shard) of W (W_shard
 * [V_shard, d], bf16); tokens are global ids in [0, V_total). Writes, per position,
 *   stats [S,T,4] f32: (m = max z, sum e^{z-m}, sum e^{z-m} z, argmax) over the shard, the
 *                      argmax as the bit pattern of an int32 global index (16-byte aligned);
 *   zy    [S,T] f32:   z at the sampled token if this shard owns it, else -inf.
 * Unscored positions get (-inf, 0, 0, -1) and -inf. Workspace: grpo_workspace_bytes with
 * V = V_shard. */
int grpo_score_fwd_shard(const void* H, const void* W_shard, int32_t dtype,
                         const int32_t* tokens, const uint8_t* mask, int32_t S, int32_t T,
                         int32_t d, int32_t V_shard, int32_t v_offset, int32_t V_total,
                         float* stats, float* zy, void* workspace, size_t workspace_bytes,
                         grpo_stream_t stream);

/* Merges the statistics of all shards after they were exchanged (e.g. all-gathered so that
 * stats is [num_shards, S, T, 4] and zy [num_shards, S, T]) into grpo_score_fwd's outputs:
 * lse = M + log sum_p s_p e^{m_p - M}, logp = z_y - lse, entropy = lse - U/S, argmax = lowest
 * global index attaining M; valid_count as in grpo_score_fwd. Needs 256 bytes of
 * workspace. */
int grpo_merge_shard_stats(const float* stats, const float* zy, int32_t num_shards,
                           const int32_t* tokens, const uint8_t* mask, int32_t S, int32_t T,
                           int32_t V_total, float* logp, float* lse, float* entropy,
                           int32_t* argmax, int32_t* valid_count, void* workspace,
                           size_t workspace_bytes, grpo_stream_t stream);

/* The shard's part of grpo_loss_bwd: logp/lse are the merged (global) values; the loss is the
 * full loss (every rank computes it); dz is formed for this shard's columns only, so
 * dH_partial [S,T,d] f32 is this shard's contribution (sum it over the ranks) and dW_shard
 * [V_shard, d] f32 is this shard's rows of dW. bf16 only. */
int grpo_loss_bwd_shard(const void* H, const void* W_shard, int32_t dtype,
                        const int32_t* tokens, const uint8_t* mask, int32_t S, int32_t T,
                        int32_t d, int32_t V_shard, int32_t v_offset, int32_t V_total,
                        const float* logp, const float* lse, const float* old_logp,
                        const float* ref_logp, const float* adv, const int32_t* valid_count,
                        float eps_low, float eps_high, float beta, int32_t agg, double norm,
                        float* loss_out, float* dH_partial, float* dW_shard, void* workspace,
                        size_t workspace_bytes, grpo_stream_t stream);

/* Synchronises `stream`, returns the first device-side status recorded in the workspace since
 * the last call (GRPO_OK if none) and clears it. *where_out (may be NULL) gets a code naming the
 * kernel and wait that recorded it. */
int grpo_last_device_error(void* workspace, int32_t* where_out, grpo_stream_t stream);

const char* grpo_status_string(int status);

/* Kernel accounting, for measurement. Every launch made by this library bumps a per-kernel
 * counter. With timing enabled, each launch is bracketed by a pair of CUDA events recorded on
 * its stream (host-side objects; no device memory). */
enum {
  GRPO_K_MASK_SCAN = 0, GRPO_K_PACK, GRPO_K_GROUP_ADV, GRPO_K_FWD_GEMM, GRPO_K_FWD_MERGE,
  GRPO_K_LOSS_TOKENS, GRPO_K_LOSS_FINAL, GRPO_K_BWD_DZ_GEMM, GRPO_K_BWD_DH_GEMM,
  GRPO_K_BWD_DW_GEMM, GRPO_K_DH_ZERO, GRPO_K_F32_FWD, GRPO_K_F32_DH, GRPO_K_F32_DW,
  GRPO_K_REWARDS, GRPO_K_SHARD_STATS, GRPO_K_MERGE_SHARDS, GRPO_K_GATHER, GRPO_K_COUNT
};
const char* grpo_kernel_name(int32_t kernel_id);
int grpo_timing_enable(int32_t enable);   /* 1 = record events from now on, 0 = stop */
int grpo_timing_reset(void);              /* forget recorded events and counters */
/* Synchronises on the recorded events; returns launches and summed device time of one kernel. */
int grpo_timing_read(int32_t kernel_id, int64_t* launches, double* total_ms);

/* Fault-injection hook for tests of the bounded waits (failure detection without a GPU fault):
 * while `on` is nonzero, CTA 0 of every tensor-core GEMM launched afterwards leaves its first
 * pipeline stage unfilled; its MMA warp's wait then runs out after about 2 s, the kernel records
 * GRPO_ERR_TIMEOUT in the workspace status word, releases its tensor memory and exits. Outputs of
 * such a call are undefined. Process-wide; not for production use. */
int grpo_debug_inject_stall(int32_t on);

/* Tensor-core tile mode of the four LM-head GEMM roles, process-wide, for launches made
 * afterwards (the exact-KL GEMMs always use single-CTA tiles). Every mode sums each output
 * element over K in the same k-block order; modes 1 and 2 issue the same M = 256 MMAs and give
 * bitwise identical results in every role, and agree with mode 0 (M = 128 MMAs) within rounding. Every TMA
 * copy lands in the issuing CTA's own shared memory (no multicast).
 *   GRPO_TILE_SINGLE        (0): one CTA per 128 x 256 tile (tcgen05 cta_group::1), two TMEM
 *                           accumulators (a tile's epilogue overlaps the next tile's MMAs).
 *   GRPO_TILE_CTA_PAIR      (1): clusters of two CTAs on one TPC compute 256 x 256 tiles with
 *                           cta_group::2, each CTA staging its 128 rows of A and half of B.
 *   GRPO_TILE_CTA_PAIR_WIDE (2): the CTA pair computes 256 x 512 tiles: two N = 256 MMAs per
 *                           k-step into one 512-column accumulator, each CTA staging 128 rows
 *                           of A and 256 rows of B per k-block, i.e. half of mode 0's operand
 *                           bytes per flop; eight epilogue warps each read one half. Made for
 *                           the long-K roles dH and dW; a forward or dz work unit is then two
 *                           vocabulary tiles.
 *   GRPO_TILE_DEFAULT      (-1): the library's per-role choice, in force at load: the forward
 *                           product and the dz recompute in mode 0, dH and dW in mode 2.
 * Roles: GRPO_ROLE_FWD (forward scoring product), GRPO_ROLE_DZ (its recompute into dz),
 * GRPO_ROLE_DH, GRPO_ROLE_DW.
 * grpo_set_tile_mode(m) puts every role in mode m (m = -1: each role's default);
 * grpo_set_role_tile_mode(r, m) sets one role (m = -1: that role's default).
 * grpo_get_tile_mode returns the mode all four roles share, or -1 when they differ (as they do
 * by default); grpo_get_role_tile_mode returns the mode role r runs in.
 * grpo_set_cta_pair(on) is grpo_set_tile_mode(on ? 1 : 0).
 * Setters return GRPO_ERR_INVALID_ARG, changing nothing, for a mode or role outside these
 * ranges; grpo_get_role_tile_mode returns GRPO_ERR_INVALID_ARG for a role outside 0..3. */
enum {
  GRPO_TILE_DEFAULT = -1,
  GRPO_TILE_SINGLE = 0,
  GRPO_TILE_CTA_PAIR = 1,
  GRPO_TILE_CTA_PAIR_WIDE = 2
};
enum { GRPO_ROLE_FWD = 0, GRPO_ROLE_DZ = 1, GRPO_ROLE_DH = 2, GRPO_ROLE_DW = 3 };
int grpo_set_tile_mode(int32_t mode);
int grpo_get_tile_mode(void);
int grpo_set_cta_pair(int32_t on);
int grpo_set_role_tile_mode(int32_t role, int32_t mode);
int grpo_get_role_tile_mode(int32_t role);

/* Progress window of the long-K tensor-core GEMMs (dH and dW; the forward and dz GEMMs never
 * wait), process-wide, for launches made afterwards. At every checkpoint the TMA producer of each
 * CTA waits (at most 0.5 ms) until the CTAs of the launch are on average within `lag`
 * checkpoints of it, so that CTAs reading the same operand tiles read them close enough in time
 * to hit L2 (CTAs that share a tile otherwise drift apart over successive long-K units and
 * re-read their operands from HBM). Checkpoints fall every `check_kblocks` k-blocks of 64
 * (check_kblocks > 0) or, for check_kblocks < 0, at the start of every (-check_kblocks)-th work
 * unit (an output tile): with lag 1 a barrier between the waves of units. Default
 * (GRPO_GEMM_WINDOW_DEFAULT_CHECK, GRPO_GEMM_WINDOW_DEFAULT_LAG) = (256, 1): a barrier every 256
 * k-blocks. Results do not depend on it. check_kblocks == 0 turns it off. Returns
 * GRPO_ERR_INVALID_ARG for a negative lag or for check_kblocks != 0 with lag == 0. */
enum { GRPO_GEMM_WINDOW_DEFAULT_CHECK = 256, GRPO_GEMM_WINDOW_DEFAULT_LAG = 1 };
int grpo_set_gemm_window(int32_t check_kblocks, int32_t lag);

#ifdef __cplusplus
}
#endif
#endif /* GRPO_GB300_H */
