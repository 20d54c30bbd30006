/*
 * mc.h — C ABI of libmc: the fused LM-head log-prob / entropy forward, the
 * MirrorPop sequence filter, and the fused backward, for one NVIDIA GB300
 * (sm_103a).
 *
 * Every entry point takes plain pointers and sizes. Unless a parameter says
 * "host", every pointer is DEVICE memory on the current CUDA device, owned by
 * the caller, and must stay valid until the work queued on `stream` has
 * finished. The library allocates no device memory: scratch comes in through
 * `workspace` arguments sized by the matching *_workspace_size() query.
 *
 * Calls are stream-ordered and asynchronous. The tensor-core kernels of the
 * forward and backward are persistent cooperative launches, one CTA per SM
 * with every CTA resident (the CTAs keep their waves in step through a
 * bounded wait on a counter in the caller's workspace): such a kernel starts
 * only when every SM has room for one of its CTAs at once.
 * Errors that can be found on the
 * host (null or misaligned pointers, bad sizes, a workspace that is too small,
 * no sm_103 device) return a non-zero mc_status synchronously and queue no
 * work. Errors found on the device (a target outside [0, V), a bounded wait
 * that gave up) set bits of the caller's `dev_status` word (MC_DEV_* flags,
 * never cleared by the library) and mark the affected outputs NaN.
 *
 * Layouts: matrices are row-major. hidden is [N, d] bf16, w_vocab is [V, d]
 * bf16 (the LM head, one row per vocabulary entry), so the logits are
 * z[t, v] = (hidden[t, :] . w_vocab[v, :]) * inv_temperature and are never
 * written to memory. Row t's hidden state is the one that predicts targets[t]
 * (the caller applies the usual one-token shift). Token arrays are packed
 * over all sequences; cu_seqlens[B+1] gives the sequence boundaries.
 *
 * The paper: MusaCoder (arXiv 2606.04847). §4.4.1 Eq. 4 defines the token
 * importance ratio, Eq. 5 the GRPO objective; §4.5.2 Eq. 17 the masked
 * objective and Eq. 18-21 the sequence statistics and MirrorPop mask.
 */
#ifndef MC_H_
#define MC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A cudaStream_t (NULL = the legacy default stream). */
typedef struct CUstream_st* mc_stream_t;

typedef enum {
  MC_OK = 0,
  MC_ERR_INVALID_ARG = 1,   /* null/misaligned pointer, size out of range */
  MC_ERR_UNSUPPORTED = 2,   /* a valid request the library does not run (e.g. no sm_103 GPU) */
  MC_ERR_CUDA = 3,          /* a CUDA runtime or driver call failed; see mc_last_cuda_error() */
  MC_ERR_TIMEOUT = 4,       /* reported through dev_status: see MC_DEV_TIMEOUT */
  MC_ERR_WORKSPACE = 5,     /* workspace pointer null/misaligned or smaller than the query */
  MC_ERR_TARGET_RANGE = 6,  /* reported through dev_status: see MC_DEV_TARGET_RANGE */
  MC_ERR_SCRATCH_LIMIT = 7  /* mc_token_logprobs_noalloc: the request needs more scratch than
                               the library's fixed MC_NOALLOC_SCRATCH_BYTES */
} mc_status;

/* Bits the kernels OR into *dev_status (an int32 in device memory). */
#define MC_DEV_TIMEOUT      0x1  /* a bounded device-side wait gave up; outputs of that call are invalid */
#define MC_DEV_TARGET_RANGE 0x2  /* some targets[t] was outside [0, V); those rows are NaN */

/* Static text for a status code. */
const char* mc_status_string(mc_status s);
/* Text of the last CUDA error seen by this thread inside the library ("" if none). */
const char* mc_last_cuda_error(void);
/* ABI version: (major << 16) | minor. */
int32_t mc_version(void);
/* Kernels this library has enqueued in this process since it was loaded, over
 * every entry point and thread (a relaxed atomic counter). For launch
 * accounting: the difference across a region of calls is the number of
 * kernels those calls launched. Calls captured into a CUDA graph count once,
 * at capture, not at each replay. */
uint64_t mc_kernel_launches(void);

/* ------------------------------------------------------------------------
 * Forward: per-token target log-prob, entropy and log-sum-exp.
 *
 * Computes, for every row t < N (pi_theta of Eq. 4 / Eq. 5, §4.4.1, taken as
 * the softmax of the LM-head logits; the entropy is the Shannon entropy in
 * nats of the same softmax, the diagnostic tracked in §5.4.6):
 *   lse[t]     = log sum_v exp(z[t, v])
 *   logp[t]    = z[t, targets[t]] - lse[t]
 *   entropy[t] = -sum_v p log p,  p = exp(z[t, :] - lse[t])
 * in one pass over the vocabulary (online max / sum / entropy update), fp32
 * accumulation of bf16 products on the tensor cores.
 *
 *   hidden        bf16 [N, d], 16-byte aligned rows
 *   w_vocab       bf16 [V, d], 16-byte aligned rows
 *   targets       int32 [N]; a value outside [0, V) sets MC_DEV_TARGET_RANGE and
 *                 makes that row's logp, entropy and lse NaN
 *   N             rows, 0 <= N < 2^31 (N == 0 queues nothing and returns MC_OK)
 *   d             hidden size, a positive multiple of 64, <= 16384
 *   V             vocabulary size, 1 <= V < 2^31
 *   inv_temperature  1/tau > 0 (tau = sampling temperature; 1 for none)
 *   logp          fp32 [N] out
 *   entropy, lse  fp32 [N] out, each may be NULL
 *   workspace     device scratch of >= mc_token_logprobs_workspace_size(N, d, V)
 *                 bytes, 256-byte aligned; contents on entry are ignored
 *   dev_status    int32 [1] (may be NULL): MC_DEV_* bits are ORed in
 * ------------------------------------------------------------------------ */
size_t mc_token_logprobs_workspace_size(int64_t N, int32_t d, int32_t V);

mc_status mc_token_logprobs(const void* hidden, const void* w_vocab, const int32_t* targets,
                            int64_t N, int32_t d, int32_t V, float inv_temperature,
                            float* logp, float* entropy, float* lse,
                            void* workspace, size_t workspace_bytes,
                            int32_t* dev_status, mc_stream_t stream);

/* ------------------------------------------------------------------------
 * Vocabulary-sharded forward: the building block of a tensor-parallel LM
 * head (the paper trains its 27B model with tensor parallelism, §5.1).
 *
 * mc_token_logprob_state computes, for one slice of the vocabulary — the rows
 * w_shard [V_shard, d] holding global ids [v_begin, v_begin + V_shard) — the
 * softmax state of every row t, in natural units:
 *   state[t] = (m, s, u, z_y):  m = max_v z[t, v],  s = sum_v exp(z - m),
 *              u = sum_v exp(z - m) (z - m),
 *              z_y = z[t, targets[t]] if the slice holds targets[t], else -inf
 * (fp32 [N, 4], 16-byte aligned). targets are global ids. The workspace is
 * mc_token_logprobs_workspace_size(N, d, V_shard) bytes.
 *
 * mc_merge_logprob_states combines P slice states (fp32 [P, N, 4], slice-major:
 * the concatenation of the P state arrays, e.g. after an all-gather) into the
 * full-vocabulary outputs of mc_token_logprobs:
 *   M = max_p m_p, S = sum_p s_p e^(m_p - M), U = sum_p e^(m_p - M)(u_p + (m_p - M) s_p),
 *   lse = M + log S, entropy = log S - U / S, logp = z_y - lse.
 * The slices must partition the vocabulary; a row whose target no slice holds
 * gets NaN outputs and sets MC_DEV_TARGET_RANGE.
 * ------------------------------------------------------------------------ */
mc_status mc_token_logprob_state(const void* hidden, const void* w_shard, const int32_t* targets,
                                 int64_t N, int32_t d, int32_t V_shard, int32_t v_begin,
                                 float inv_temperature, float* state,
                                 void* workspace, size_t workspace_bytes,
                                 int32_t* dev_status, mc_stream_t stream);

mc_status mc_merge_logprob_states(const float* states, int32_t P, int64_t N,
                                  float* logp, float* entropy, float* lse,
                                  int32_t* dev_status, mc_stream_t stream);

/* ------------------------------------------------------------------------
 * Forward for callers that cannot allocate device memory. (The paper has no
 * counterpart: this is a deployment variant of mc_token_logprobs.)
 *
 * Some callers may not call cudaMalloc and have no spare buffer to pass as a
 * workspace: a host process whose memory manager owns every device
 * allocation, a plugin running inside such a host, or a latency-critical loop
 * that cannot take the device-wide synchronisation an allocation may cause.
 * This entry point computes exactly what mc_token_logprobs computes, with the
 * same arguments minus the workspace; its scratch is a fixed array of
 * MC_NOALLOC_SCRATCH_BYTES compiled into libmc, which every GPU that loads
 * the library holds until the process exits. It allocates nothing itself.
 *
 *   Limit: requests with mc_token_logprobs_workspace_size(N, d, V) greater than
 *   MC_NOALLOC_SCRATCH_BYTES are rejected with MC_ERR_SCRATCH_LIMIT before any
 *   work is queued (about 171,000 rows for V >= 4096; more for smaller V).
 *   Set-up: the first call on each device looks up the array's device address
 *   with that device current and caches it; make that first call before any
 *   stream capture begins. The cached address belongs to the device's context
 *   as it was at that first call: cudaDeviceReset() on the device invalidates
 *   it, and this entry point must not be called again on that device in the
 *   same process afterwards.
 *   Sharing: all calls on a device use the same array and it keeps the last
 *   call's contents (the call clears, on its stream, what must start at zero).
 *   Calls whose work overlaps on the GPU (different streams without ordering
 *   between them) race on the array; order them.
 * ------------------------------------------------------------------------ */
#define MC_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)

mc_status mc_token_logprobs_noalloc(const void* hidden, const void* w_vocab, const int32_t* targets,
                                    int64_t N, int32_t d, int32_t V, float inv_temperature,
                                    float* logp, float* entropy, float* lse,
                                    int32_t* dev_status, mc_stream_t stream);

/* ------------------------------------------------------------------------
 * Backward of the forward above.
 *
 * For upstream gradients g[t] = dL/dlogp[t] and gH[t] = dL/dentropy[t]
 * (gH may be NULL = 0), with p = exp(z - lse):
 *   dZ[t, v]        = inv_temperature * ( g[t] (1[v = targets[t]] - p[t, v])
 *                                         - gH[t] p[t, v] (log p[t, v] + entropy[t]) )
 *   grad_hidden     = dZ . w_vocab           bf16 [N, d] (overwritten)
 *   grad_w          = dZ^T . hidden          fp32 [V, d] (overwritten, or added to
 *                                            when accumulate != 0)
 * This is the gradient of the log-prob and entropy with respect to the LM-head
 * inputs, which the masked GRPO objective (Eq. 17, §4.5.2) reaches through
 * rho (Eq. 4). Eq. 17 multiplies every token of response i by its mask M_i:
 * `row_keep` (uint8 [N], nullable = all kept) applies that gate, so
 * g[t] and gH[t] count only where row_keep[t] != 0 (pass the filter's
 * token_keep). Rows with a zero effective upstream gradient contribute
 * nothing: their grad_hidden rows are written as zero. The logits are
 * recomputed per tile on the tensor cores and never stored; dZ (a gradient)
 * is staged in bf16 in the workspace.
 *
 *   lse, entropy  fp32 [N] from the forward (entropy may be NULL when gH is NULL)
 *   grad_logp     fp32 [N]; grad_entropy fp32 [N] or NULL
 *   workspace     >= mc_token_logprobs_bwd_workspace_size(N, d, V, 256) bytes
 *                 (chunks of 256 rows; rows_per_chunk rounds up to a multiple
 *                 of 256); more workspace lets the rows run in fewer, larger
 *                 chunks (mc_token_logprobs_bwd_workspace_size(N, d, V, N) =
 *                 one chunk). The call uses as many rows per chunk as
 *                 workspace_bytes holds.
 *   Other arguments as for the forward. A target outside [0, V) sets
 *   MC_DEV_TARGET_RANGE; that row's gradient terms are dropped.
 * ------------------------------------------------------------------------ */
size_t mc_token_logprobs_bwd_workspace_size(int64_t N, int32_t d, int32_t V, int64_t rows_per_chunk);

mc_status mc_token_logprobs_bwd(const void* hidden, const void* w_vocab, const int32_t* targets,
                                const float* lse, const float* entropy,
                                const float* grad_logp, const float* grad_entropy,
                                const uint8_t* row_keep, int64_t N, int32_t d, int32_t V, float inv_temperature,
                                void* grad_hidden, float* grad_w, int32_t accumulate,
                                void* workspace, size_t workspace_bytes,
                                int32_t* dev_status, mc_stream_t stream);

/* ------------------------------------------------------------------------
 * Sequence importance-ratio statistics and the MirrorPop keep-mask.
 *
 * With log rho[t] = logp_policy[t] - logp_behaviour[t] (Eq. 4: policy over
 * rollout/behaviour) and T_i = { t in [cu_seqlens[i], cu_seqlens[i+1]) :
 * loss_mask[t] != 0 }, L_i = |T_i|:
 *   n_tokens[i]    = L_i
 *   signed_mean[i] = (1/L_i) sum_{T_i} log rho      (exponent of Eq. 18)
 *   abs_mean[i]    = (1/L_i) sum_{T_i} |log rho|    (exponent of Eq. 20)
 *   keep[i]        = abs_mean[i] <= delta           (Eq. 21)
 *   keep_vanilla[i]= |signed_mean[i]| <= delta_vanilla (the conventional
 *                    sequence mask, read as a symmetric log-space interval;
 *                    0 when delta_vanilla < 0)
 *   token_ratio[t] = exp(log rho[t])                (Eq. 4)
 *   token_keep[t]  = keep[seq(t)] && loss_mask[t]
 * A sequence with L_i = 0 gets signed_mean = abs_mean = 0 and keep = 0.
 *
 *   logp_policy, logp_behaviour  fp32 [N]
 *   loss_mask     uint8 [N] or NULL (= all tokens count)
 *   cu_seqlens    int64 [B+1], cu[0] = 0, non-decreasing, cu[B] = N
 *                 (checked on the device only as far as needed to stay in bounds:
 *                 a segment is clamped to [0, N))
 *   B             sequences, 1 <= B < 2^31;  N tokens, 0 <= N < 2^40
 *   delta         MirrorPop threshold in log-ratio space, >= 0
 *   signed_mean, abs_mean  fp32 [B] out; n_tokens int32 [B] out; keep uint8 [B] out
 *   keep_vanilla  uint8 [B] out or NULL;  token_ratio fp32 [N] out or NULL;
 *   token_keep    uint8 [N] out or NULL
 * ------------------------------------------------------------------------ */
mc_status mc_seq_ratio_filter(const float* logp_policy, const float* logp_behaviour,
                              const uint8_t* loss_mask, const int64_t* cu_seqlens,
                              int32_t B, int64_t N, float delta, float delta_vanilla,
                              float* signed_mean, float* abs_mean, int32_t* n_tokens,
                              uint8_t* keep, uint8_t* keep_vanilla,
                              float* token_ratio, uint8_t* token_keep, mc_stream_t stream);

/* ------------------------------------------------------------------------
 * Masked GRPO objective and the upstream gradient of the backward.
 *
 * With rho_t = exp(logp_policy[t] - logp_behaviour[t]) (Eq. 4), response i's
 * advantage A_i = advantages[i] (Eq. 3), mask M_i = keep[i] (Eq. 21) and
 * L_i = n_tokens[i] (its loss-masked token count, as mc_seq_ratio_filter
 * returns it), over the tokens T_i of response i with loss_mask != 0:
 *   s_t          = min(rho_t A_i, clip(rho_t, 1 - eps_low, 1 + eps_high) A_i)   (Eq. 5)
 *   k_t          = e^r - r - 1,  r = logp_ref[t] - logp_policy[t]  (per-token
 *                  estimate of KL(pi_theta || pi_ref); the paper does not fix
 *                  the estimator, this is the non-negative one used with GRPO)
 *   *kl          = (1 / Z) sum_i M_i sum_{t in T_i} k_t
 *   *loss        = -(1 / Z) sum_i M_i sum_{t in T_i} s_t + beta * kl,
 *                  Z = sum_i M_i L_i                                             (Eq. 17)
 *   grad_logp[t] = dL / dlogp_policy[t] = (M_i / Z) (-rho_t A_i [where the
 *                  unclipped term attains the minimum, ties included]
 *                  + beta (1 - e^r)); 0 for tokens with loss_mask == 0;
 *                  everything 0 when Z == 0.
 * With logp_ref == NULL the KL term is absent (k_t = 0). grad_logp is the
 * grad_logp argument of mc_token_logprobs_bwd (dropped responses already
 * carry zero gradient).
 *
 *   advantages    fp32 [B]; keep uint8 [B]; n_tokens int32 [B]
 *   eps_low       in [0, 1); eps_high >= 0
 *   logp_ref      fp32 [N] or NULL (reference-policy log-probs of the same tokens)
 *   beta          KL weight >= 0 (ignored without logp_ref)
 *   loss          fp32 [1] out
 *   grad_logp     fp32 [N] out
 *   seq_loss      fp32 [B] out or NULL: response i's share of *loss
 *   n_clipped     int32 [1] out or NULL: tokens of kept responses whose clipped
 *                 term was strictly smaller
 *   kl            fp32 [1] out or NULL
 *   workspace     >= mc_grpo_masked_loss_workspace_size(B) bytes, 256-byte aligned
 * Other arguments, layouts and error behaviour as for mc_seq_ratio_filter.
 * ------------------------------------------------------------------------ */
size_t mc_grpo_masked_loss_workspace_size(int32_t B);

mc_status mc_grpo_masked_loss(const float* logp_policy, const float* logp_behaviour,
                              const uint8_t* loss_mask, const int64_t* cu_seqlens,
                              const float* advantages, const uint8_t* keep, const int32_t* n_tokens,
                              int32_t B, int64_t N, float eps_low, float eps_high,
                              const float* logp_ref, float beta,
                              float* loss, float* grad_logp, float* seq_loss, int32_t* n_clipped, float* kl,
                              void* workspace, size_t workspace_bytes, mc_stream_t stream);

/* ------------------------------------------------------------------------
 * PrimeEcho trajectory reward and group-normalised advantage (§4.4.3).
 *
 * For trajectory i with per-turn scores s_{i,k} = scores[i*K + k - 1] and
 * verification outcomes success[i*K + k - 1], over its n_turns[i] turns
 * (clamped to [1, K]; turns beyond it did not run):
 *   reward[i]    = alpha s_{i,1} + (1 - alpha) max_k s_{i,k}
 *                  + beta1 1[success_{i,1}] + beta2 1[!success_{i,1} && success_{i,2}]   (Eq. 9-10)
 *   advantage[i] = (reward[i] - mean_G) / (std_G + eps)                                  (Eq. 12)
 * over groups of group_size consecutive trajectories (the G samples of one
 * prompt); std_G is the sample standard deviation (divisor G - 1) and a group
 * of one gets advantage 0. K = 1 with beta1 = beta2 = 0 is the single-turn
 * GRPO advantage of Eq. 3 with reward[i] = s_{i,1}.
 *
 *   scores fp32 [T, K]; success uint8 [T, K]; n_turns int32 [T]
 *   T a positive multiple of group_size; K >= 1; alpha in [0, 1];
 *   beta1, beta2 >= 0 (the paper sets beta1 > beta2 >= 0 so that earlier
 *   success earns more; the library does not require the order); eps >= 0
 *   reward fp32 [T] out or NULL; advantage fp32 [T] out (feed it to
 *   mc_grpo_masked_loss as `advantages`)
 * ------------------------------------------------------------------------ */
mc_status mc_prime_echo_advantages(const float* scores, const uint8_t* success, const int32_t* n_turns,
                                   int32_t T, int32_t K, int32_t group_size, float alpha, float beta1,
                                   float beta2, float eps, float* reward, float* advantage,
                                   mc_stream_t stream);

/* ------------------------------------------------------------------------
 * Self-test of the bounded device waits used by every pipelined kernel: one
 * CTA waits on a shared-memory barrier that nothing ever signals and, in a
 * second warp, on a global counter that nothing ever raises (the wait of the
 * GEMMs' wave gate); each gives up after `timeout_ns` nanoseconds
 * (1e6 <= timeout_ns <= 1e10), sets MC_DEV_TIMEOUT in *dev_status and
 * returns. Exercises the failure path without faulting or hanging the GPU.
 * (No counterpart in the paper.)
 * ------------------------------------------------------------------------ */
mc_status mc_selftest_bounded_wait(int32_t* dev_status, int64_t timeout_ns, mc_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* MC_H_ */
