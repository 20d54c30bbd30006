// mc_internal.h — launch entry points shared between the kernel translation
// units and the C-ABI layer (mc_api.cu). Not part of the public ABI.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace mc {

// Launch accounting: every kernel the library enqueues is counted (a
// process-wide relaxed atomic, read through mc_kernel_launches()).
void note_launches(unsigned n = 1);
// After a kernel launch: its error status, counting the launch if it was enqueued.
inline cudaError_t launched() {
  const cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) note_launches();
  return e;
}

// Forward: persistent tcgen05 kernel (online log-softmax epilogue) followed by
// the per-row merge of the split partials.
struct FwdArgs {
  CUtensorMap tm_hidden;  // K-major {d, N}, box {64, 128}
  CUtensorMap tm_w;       // K-major {d, V}, box {64, 256}
  const int32_t* targets;
  long long N;
  int d, V;
  float inv_temperature;
  int splits;
  long long n_pad;
  float* part;            // workspace: [3][splits * halves][n_pad]
  float* zy;              // workspace: [n_pad]
  int32_t* ws_status;     // workspace: internal status word (zeroed by the caller)
  unsigned int* wave_ctr; // workspace: the projection's wave gate counter (zeroed by the caller)
  float* logp;
  float* entropy;
  float* lse;
  int32_t* dev_status;
  int grid;
  uint64_t timeout_ns;
  int wide;               // 1 = 256-row tiles (TileCfg<2>), 0 = 128-row
  int halves;             // 256-row tiles: 2 = two epilogue warp groups per sub-block, one per
                          // column half, each with its own partial slot (needs 2 * splits <= 16)
  int v_offset;           // global vocabulary id of W's row 0 (shards); 0 otherwise
  float* state;           // non-null: write the slice state [N, 4] instead of logp/entropy/lse
};
cudaError_t launch_forward(const FwdArgs& a, cudaStream_t stream);
cudaError_t launch_merge_states(const float* states, int P, long long N, float* logp, float* entropy, float* lse,
                                int32_t* dev_status, cudaStream_t stream);

// Backward building blocks. Rows are first compacted on the device (idx[],
// *count); every later stage takes its extent from *count.
struct SelectArgs {
  const void* hidden;     // bf16 [N, d]
  const uint8_t* row_keep;
  const float* grad_logp;
  const float* grad_entropy;
  const int32_t* targets;
  long long N;
  int d, V;
  int32_t* idx;           // workspace: [N] selected original rows, ascending
  int32_t* count;         // workspace: number selected
  int32_t* slab;          // workspace: [ceil(N / 1024)] per-slab offsets (any region the gather writes later)
  void* hc;               // workspace: bf16 [n_pad, d] gathered hidden rows
  int32_t* ws_status;
  int grid;
};
cudaError_t launch_select_gather(const SelectArgs& a, cudaStream_t stream);

struct DzArgs {
  CUtensorMap tm_hidden;  // K-major {d, rows} over Hc + row_offset, box {64, 128}
  CUtensorMap tm_w;       // K-major {d, V}, box {64, 256}
  const int32_t* targets; // original-row arrays (indexed through idx)
  const float* lse;
  const float* entropy;
  const float* grad_logp;
  const float* grad_entropy;
  const int32_t* idx;     // idx + row_offset
  const int32_t* count;
  long long row_offset;   // first compacted row of this chunk
  long long rows;         // chunk capacity (rows of the dZ buffer used)
  int d, V;
  float inv_temperature;
  int splits;
  void* dz;               // bf16 [rows, ld]
  long long ld;
  CUtensorMap tm_dz_st;   // dz {V, rows}, box {32, 32}, 64-byte swizzle (the epilogue's TMA stores)
  int32_t* ws_status;
  int grid;
  unsigned int* wave_ctr;   // workspace: the wave gate counter (zeroed before each launch)
  uint64_t timeout_ns;
  int wide;               // 1 = 256-row tiles (TileCfg<2>), 0 = 128-row
};
cudaError_t launch_dz(const DzArgs& a, cudaStream_t stream);

struct DhArgs {           // grad_hidden[idx[j], :] = (dZ . W)[j, :]
  CUtensorMap tm_dz;      // K-major {V, rows}, box {64, 128}
  CUtensorMap tm_w_mn;    // N-major {d, V}, box {64, 64}
  const int32_t* idx;     // idx + row_offset
  const int32_t* count;
  long long row_offset;
  long long rows;
  int d, V;
  void* grad_hidden;      // bf16 [N, d]
  int32_t* ws_status;
  int grid;
  unsigned int* wave_ctr;   // workspace: the wave gate counter (zeroed before each launch)
  uint64_t timeout_ns;
};
cudaError_t launch_dh(const DhArgs& a, cudaStream_t stream);

struct DwArgs {           // grad_w[V, d] (+)= dZ[rows, V]^T . Hc[rows, d]
  CUtensorMap tm_dz_mn;   // M-major {V, rows}, box {64, 64}
  CUtensorMap tm_h_mn;    // N-major {d, rows} over Hc + row_offset, box {64, 64}
  const int32_t* count;
  long long row_offset;
  long long rows;
  int d, V;
  float* grad_w;
  int accumulate;
  int32_t* ws_status;
  int grid;
  unsigned int* wave_ctr;   // workspace: the wave gate counter (zeroed before each launch)
  uint64_t timeout_ns;
};
cudaError_t launch_dw(const DwArgs& a, cudaStream_t stream);

// Propagates the internal status word to the caller's (if any).
cudaError_t launch_status_merge(const int32_t* ws_status, int32_t* dev_status, cudaStream_t stream);

struct FilterArgs {
  const float* logp_policy;
  const float* logp_behaviour;
  const uint8_t* loss_mask;
  const int64_t* cu_seqlens;
  int B;
  long long N;
  float delta, delta_vanilla;
  float* signed_mean;
  float* abs_mean;
  int32_t* n_tokens;
  uint8_t* keep;
  uint8_t* keep_vanilla;
  float* token_ratio;
  uint8_t* token_keep;
  int vec_ok;             // all float arrays 16-byte and loss_mask 4-byte aligned
  int keep_vec_ok;        // token_keep and loss_mask 16-byte aligned: 16-token keep stores
  int grid;               // persistent CTAs (sequences are strided over them)
};
cudaError_t launch_filter(const FilterArgs& a, cudaStream_t stream);
// CTAs of the filter kernel one SM keeps resident (from its register and
// thread counts, queried once): a grid of SMs x this runs in a single wave.
int filter_ctas_per_sm();

struct LossArgs {
  const float* logp_policy;
  const float* logp_behaviour;
  const uint8_t* loss_mask;
  const int64_t* cu_seqlens;
  const float* advantages;
  const uint8_t* keep;
  const int32_t* n_tokens;
  int B;
  long long N;
  float eps_low, eps_high;
  const float* logp_ref;  // null: no KL term
  float beta;
  float* loss;
  float* grad_logp;
  float* seq_loss;
  int32_t* n_clipped;
  float* kl;
  long long* Z;           // workspace (zeroed by the launch, with the ticket after it)
  unsigned int* ticket;   // workspace: CTAs done, for the last-CTA sum
  float* seq_share;       // workspace [B]
  float* seq_kl;          // workspace [B]
  int vec_ok;
  int grid;               // persistent CTAs (sequences are strided over them)
};
cudaError_t launch_grpo_loss(const LossArgs& a, cudaStream_t stream);

struct AdvArgs {
  const float* scores;     // [T, K]
  const uint8_t* success;  // [T, K]
  const int32_t* n_turns;  // [T]
  long long n_groups;
  int G, K;
  float alpha, beta1, beta2, eps;
  float* reward;           // [T] or null
  float* advantage;        // [T]
  int vec4;                // K == 4, scores 16-byte and success 4-byte aligned: vector row loads
};
cudaError_t launch_group_advantage(const AdvArgs& a, cudaStream_t stream);

cudaError_t launch_selftest_wait(int32_t* dev_status, uint64_t timeout_ns, cudaStream_t stream);


}  // namespace mc
