// mc_loss.cu — the masked GRPO objective (Eq. 17 without the KL term) and its
// gradient with respect to the policy log-probs, which is the upstream
// gradient g_t the fused backward consumes.
//
//   rho_t  = exp(logp_policy_t - logp_behaviour_t)                  (Eq. 4)
//   s_t    = min(rho_t A_i, clip(rho_t, 1 - eps_low, 1 + eps_high) A_i)
//   L      = -(1 / Z) sum_i M_i sum_{t in T_i} s_t,  Z = sum_i M_i L_i   (Eq. 17)
//   dL/dlogp_t = -M_i rho_t A_i / Z if rho_t A_i <= the clipped term, else 0
//
// Three launches: (1) one CTA forms Z from the filter's keep / n_tokens;
// (2) persistent CTAs stride over the sequences, write g_t for every token
// (16-byte loads and stores, two vectors in flight per thread) and each
// response's share of L; (3) one CTA sums the shares in a fixed order.
// All reductions are fixed-order, so results are bitwise reproducible.
#include "mc_internal.h"
#include "mc_ptx.cuh"

namespace mc {

namespace {

constexpr int kLossThreads = 256;
constexpr int kReduceThreads = 1024;

__global__ void __launch_bounds__(kReduceThreads) grpo_norm_kernel(const uint8_t* __restrict__ keep,
                                                                   const int32_t* __restrict__ n_tokens, int B,
                                                                   long long* Z, int32_t* n_clipped) {
  __shared__ long long part[kReduceThreads / 32];
  long long acc = 0;
  for (int i = threadIdx.x; i < B; i += blockDim.x)
    if (keep[i]) acc += n_tokens[i] > 0 ? n_tokens[i] : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    long long z = 0;
    for (int w = 0; w < kReduceThreads / 32; ++w) z += part[w];
    *Z = z;
    if (n_clipped) *n_clipped = 0;
  }
}

struct TokAcc {
  float s;
  int clipped;
};

__device__ __forceinline__ float token_grad(float lp, float lb, bool counted, float A, float lo, float hi, float kz,
                                            TokAcc& acc) {
  if (!counted) return 0.f;
  const float rho = __expf(lp - lb);                 // Eq. 4
  const float u = rho * A;                           // unclipped surrogate
  const float c = fminf(fmaxf(rho, lo), hi) * A;     // clipped surrogate
  const bool clipped = c < u;                        // ties take the unclipped branch
  acc.s += clipped ? c : u;
  acc.clipped += clipped ? 1 : 0;
  return clipped ? 0.f : -kz * u;                    // -M_i rho A / Z
}

__device__ __forceinline__ float4 vec_grad(const float4& lp, const float4& lb, uchar4 mk, float A, float lo, float hi,
                                           float kz, TokAcc& acc) {
  float4 g;
  g.x = token_grad(lp.x, lb.x, mk.x != 0, A, lo, hi, kz, acc);
  g.y = token_grad(lp.y, lb.y, mk.y != 0, A, lo, hi, kz, acc);
  g.z = token_grad(lp.z, lb.z, mk.z != 0, A, lo, hi, kz, acc);
  g.w = token_grad(lp.w, lb.w, mk.w != 0, A, lo, hi, kz, acc);
  return g;
}

__global__ void __launch_bounds__(kLossThreads) grpo_loss_kernel(LossArgs p) {
  __shared__ TokAcc warp_acc[kLossThreads / 32];
  const long long Z = *p.Z;
  const float lo = 1.f - p.eps_low, hi = 1.f + p.eps_high;
  const float4* lp4 = reinterpret_cast<const float4*>(p.logp_policy);
  const float4* lb4 = reinterpret_cast<const float4*>(p.logp_behaviour);
  const uchar4* m4 = reinterpret_cast<const uchar4*>(p.loss_mask);
  float4* g4 = reinterpret_cast<float4*>(p.grad_logp);
  for (int i = blockIdx.x; i < p.B; i += gridDim.x) {
    long long b = p.cu_seqlens[i];
    long long e = p.cu_seqlens[i + 1];
    b = b < 0 ? 0 : (b > p.N ? p.N : b);
    e = e < b ? b : (e > p.N ? p.N : e);
    const float M = (p.keep[i] != 0 && Z > 0) ? 1.f : 0.f;
    const float A = p.advantages[i];
    const float kz = Z > 0 ? M / static_cast<float>(Z) : 0.f;

    TokAcc acc{0.f, 0};
    long long hb = p.vec_ok ? ((b + 3) & ~3LL) : e;
    if (hb > e) hb = e;
    const long long vend = hb + ((e - hb) & ~3LL);
    for (long long t = b + threadIdx.x; t < hb; t += blockDim.x)
      p.grad_logp[t] = token_grad(p.logp_policy[t], p.logp_behaviour[t],
                                  p.loss_mask ? p.loss_mask[t] != 0 : true, A, lo, hi, kz, acc);
    const long long q1 = vend >> 2;
    for (long long q = (hb >> 2) + threadIdx.x; q < q1; q += 2LL * blockDim.x) {
      const long long r = q + blockDim.x;
      const bool two = r < q1;
      const float4 lpa = __ldcs(lp4 + q), lba = __ldcs(lb4 + q);
      const uchar4 ma = p.loss_mask ? m4[q] : make_uchar4(1, 1, 1, 1);
      float4 lpb = make_float4(0.f, 0.f, 0.f, 0.f), lbb = lpb;
      uchar4 mb = make_uchar4(0, 0, 0, 0);
      if (two) {
        lpb = __ldcs(lp4 + r);
        lbb = __ldcs(lb4 + r);
        mb = p.loss_mask ? m4[r] : make_uchar4(1, 1, 1, 1);
      }
      __stcs(g4 + q, vec_grad(lpa, lba, ma, A, lo, hi, kz, acc));
      if (two) __stcs(g4 + r, vec_grad(lpb, lbb, mb, A, lo, hi, kz, acc));
    }
    for (long long t = vend + threadIdx.x; t < e; t += blockDim.x)
      p.grad_logp[t] = token_grad(p.logp_policy[t], p.logp_behaviour[t],
                                  p.loss_mask ? p.loss_mask[t] != 0 : true, A, lo, hi, kz, acc);

#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      acc.s += __shfl_xor_sync(0xffffffffu, acc.s, o);
      acc.clipped += __shfl_xor_sync(0xffffffffu, acc.clipped, o);
    }
    if ((threadIdx.x & 31) == 0) warp_acc[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
      TokAcc tot{0.f, 0};
      for (int w = 0; w < kLossThreads / 32; ++w) {
        tot.s += warp_acc[w].s;
        tot.clipped += warp_acc[w].clipped;
      }
      const float share = -tot.s * kz;  // this response's share of L
      p.seq_share[i] = share;
      if (p.seq_loss) p.seq_loss[i] = share;
      if (p.n_clipped && M != 0.f && tot.clipped) atomicAdd(p.n_clipped, tot.clipped);
    }
    __syncthreads();  // warp_acc is reused by the next sequence
  }
}

__global__ void __launch_bounds__(kReduceThreads) grpo_final_kernel(const float* __restrict__ seq_share, int B,
                                                                    float* loss) {
  __shared__ float part[kReduceThreads / 32];
  float acc = 0.f;
  for (int i = threadIdx.x; i < B; i += blockDim.x) acc += seq_share[i];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float l = 0.f;
    for (int w = 0; w < kReduceThreads / 32; ++w) l += part[w];
    *loss = l;
  }
}

}  // namespace

cudaError_t launch_grpo_loss(const LossArgs& a, cudaStream_t stream) {
  grpo_norm_kernel<<<1, kReduceThreads, 0, stream>>>(a.keep, a.n_tokens, a.B, a.Z, a.n_clipped);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int grid = a.B < a.grid ? a.B : a.grid;
  grpo_loss_kernel<<<grid, kLossThreads, 0, stream>>>(a);
  if ((e = cudaGetLastError()) != cudaSuccess) return e;
  grpo_final_kernel<<<1, kReduceThreads, 0, stream>>>(a.seq_share, a.B, a.loss);
  return cudaGetLastError();
}

}  // namespace mc
