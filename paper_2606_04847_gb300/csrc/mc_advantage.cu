// mc_advantage.cu — PrimeEcho trajectory reward (§4.4.3, Eq. 9-10) and the
// group-normalised advantage A_i (Eq. 12; Eq. 3 for single-turn rewards) that
// the masked GRPO loss takes per response.
//
//   R_i = alpha s_{i,1} + (1 - alpha) max_{k <= K_i} s_{i,k}
//         + beta1 1[success_{i,1}] + beta2 1[!success_{i,1} && success_{i,2}]
//   A_i = (R_i - mean_G R) / (std_G R + eps),  std with divisor G - 1
//
// Group sizes dividing 32 (the paper's G = 8 among them): a group's G
// trajectories on G consecutive lanes of a warp (a group never straddles two
// warps), its mean and standard deviation formed by xor-shuffle butterflies
// inside those lanes; a warp reads 32 consecutive trajectory rows, and each
// thread handles four rows one block apart. Other group sizes: one thread per group forms the G
// rewards, then the mean and the standard deviation in two passes.
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

// K = 4 turns with aligned arrays: one 16-byte load of the row's scores and
// one 4-byte load of its success flags.
__device__ __forceinline__ float trajectory_reward4(const AdvArgs& p, long long i) {
  int k = p.n_turns[i];
  k = k < 1 ? 1 : (k > 4 ? 4 : k);
  const float4 s = reinterpret_cast<const float4*>(p.scores)[i];
  const uchar4 ok = reinterpret_cast<const uchar4*>(p.success)[i];
  float best = s.x;
  if (k >= 2) best = fmaxf(best, s.y);
  if (k >= 3) best = fmaxf(best, s.z);
  if (k >= 4) best = fmaxf(best, s.w);
  const bool first_ok = ok.x != 0;
  const bool second_ok = k >= 2 && ok.y != 0;
  const float bonus = (first_ok ? p.beta1 : 0.f) + ((!first_ok && second_ok) ? p.beta2 : 0.f);
  return p.alpha * s.x + (1.f - p.alpha) * best + bonus;
}

// Trajectories per thread in the lanes kernel: thread t of a block handles
// trajectories base + t + u * blockDim.x, u < kAdvUnroll (whole warps, so
// whole groups, per u). All of a thread's row loads issue before any reward
// is formed: four rows' 24 bytes each in flight per thread instead of one.
constexpr int kAdvUnroll = 4;

template <int G>
__global__ void __launch_bounds__(kAdvThreads) group_advantage_lanes_kernel(AdvArgs p) {
  static_assert(32 % G == 0, "a group must fit the lanes of one warp");
  const long long T = p.n_groups * G;
  const long long base = static_cast<long long>(blockIdx.x) * (blockDim.x * kAdvUnroll) + threadIdx.x;
  float r[kAdvUnroll];
#pragma unroll
  for (int u = 0; u < kAdvUnroll; ++u) {
    const long long i = base + static_cast<long long>(u) * blockDim.x;
    // Whole groups: the tail's dead lanes form dead groups.
    r[u] = i >= T ? 0.f : (p.vec4 ? trajectory_reward4(p, i) : trajectory_reward(p, i));
  }
#pragma unroll
  for (int u = 0; u < kAdvUnroll; ++u) {
    const long long i = base + static_cast<long long>(u) * blockDim.x;
    float sum = r[u];
#pragma unroll
    for (int off = G / 2; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
    const float mean = sum / static_cast<float>(G);
    const float dv = r[u] - mean;
    float ss = dv * dv;
#pragma unroll
    for (int off = G / 2; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    if (i >= T) continue;
    const float sd = G > 1 ? sqrtf(ss / static_cast<float>(G - 1)) : 0.f;
    if (p.reward) __stcs(p.reward + i, r[u]);
    __stcs(p.advantage + i, (G > 1 && sd + p.eps > 0.f) ? dv * (1.f / (sd + p.eps)) : 0.f);
  }
}

template <int G>
cudaError_t launch_lanes(const AdvArgs& a, cudaStream_t stream) {
  const long long T = a.n_groups * G;
  const long long per_block = static_cast<long long>(kAdvThreads) * kAdvUnroll;
  const long long blocks = (T + per_block - 1) / per_block;
  group_advantage_lanes_kernel<G><<<static_cast<unsigned>(blocks), kAdvThreads, 0, stream>>>(a);
  return launched();
}

}  // namespace

cudaError_t launch_group_advantage(const AdvArgs& a, cudaStream_t stream) {
  if (a.n_groups <= 0) return cudaSuccess;
  switch (a.G) {
    case 1: return launch_lanes<1>(a, stream);
    case 2: return launch_lanes<2>(a, stream);
    case 4: return launch_lanes<4>(a, stream);
    case 8: return launch_lanes<8>(a, stream);
    case 16: return launch_lanes<16>(a, stream);
    case 32: return launch_lanes<32>(a, stream);
    default: break;
  }
  const long long blocks = (a.n_groups + kAdvThreads - 1) / kAdvThreads;
  group_advantage_kernel<<<static_cast<unsigned>(blocks), kAdvThreads, 0, stream>>>(a);
  return launched();
}

}  // namespace mc
