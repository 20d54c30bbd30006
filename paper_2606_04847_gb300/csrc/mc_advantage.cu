// mc_advantage.cu — PrimeEcho trajectory reward (§4.4.3, Eq. 9-10) and the
// group-normalised advantage A_i (Eq. 12; Eq. 3 for single-turn rewards) that
// the masked GRPO loss takes per response.
//
//   R_i = alpha s_{i,1} + (1 - alpha) max_{k <= K_i} s_{i,k}
//         + beta1 1[success_{i,1}] + beta2 1[!success_{i,1} && success_{i,2}]
//   A_i = (R_i - mean_G R) / (std_G R + eps),  std with divisor G - 1
//
// One thread per group of G consecutive trajectories (a few hundred groups per
// batch): it forms the G rewards, then the mean and the standard deviation in
// two passes. Latency-bound by design.
#include "mc_internal.h"

namespace mc {

namespace {

constexpr int kAdvThreads = 128;

__device__ __forceinline__ float trajectory_reward(const AdvArgs& p, long long i) {
  int k = p.n_turns[i];
  k = k < 1 ? 1 : (k > p.K ? p.K : k);
  const float* s = p.scores + i * p.K;
  const uint8_t* ok = p.success + i * p.K;
  float best = s[0];
  for (int j = 1; j < k; ++j) best = fmaxf(best, s[j]);
  const bool first_ok = ok[0] != 0;
  const bool second_ok = k >= 2 && ok[1] != 0;
  const float bonus = (first_ok ? p.beta1 : 0.f) + ((!first_ok && second_ok) ? p.beta2 : 0.f);
  return p.alpha * s[0] + (1.f - p.alpha) * best + bonus;
}

__global__ void __launch_bounds__(kAdvThreads) group_advantage_kernel(AdvArgs p) {
  const long long g = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (g >= p.n_groups) return;
  const long long i0 = g * p.G;
  float sum = 0.f;
  for (int j = 0; j < p.G; ++j) {
    const float r = trajectory_reward(p, i0 + j);
    if (p.reward) p.reward[i0 + j] = r;
    sum += r;
  }
  const float mean = sum / static_cast<float>(p.G);
  float ss = 0.f;
  for (int j = 0; j < p.G; ++j) {
    const float dv = trajectory_reward(p, i0 + j) - mean;
    ss = fmaf(dv, dv, ss);
  }
  const float sd = p.G > 1 ? sqrtf(ss / static_cast<float>(p.G - 1)) : 0.f;
  const float inv = 1.f / (sd + p.eps);
  for (int j = 0; j < p.G; ++j) {
    const float dv = trajectory_reward(p, i0 + j) - mean;
    p.advantage[i0 + j] = (p.G > 1 && sd + p.eps > 0.f) ? dv * inv : 0.f;
  }
}

}  // namespace

cudaError_t launch_group_advantage(const AdvArgs& a, cudaStream_t stream) {
  if (a.n_groups <= 0) return cudaSuccess;
  const long long blocks = (a.n_groups + kAdvThreads - 1) / kAdvThreads;
  group_advantage_kernel<<<static_cast<unsigned>(blocks), kAdvThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace mc
