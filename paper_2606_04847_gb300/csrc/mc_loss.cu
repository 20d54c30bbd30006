// mc_loss.cu — the masked GRPO objective (Eq. 5 / Eq. 17) and its gradient
// with respect to the policy log-probs, which is the upstream gradient g_t the
// fused backward consumes.
//
//   rho_t  = exp(logp_policy_t - logp_behaviour_t)                  (Eq. 4)
//   s_t    = min(rho_t A_i, clip(rho_t, 1 - eps_low, 1 + eps_high) A_i)
//   k_t    = e^r - r - 1,  r = logp_ref_t - logp_policy_t   (KL estimate, optional)
//   L      = -(1 / Z) sum_i M_i sum_{t in T_i} s_t + beta (1 / Z) sum_i M_i sum_t k_t,
//            Z = sum_i M_i L_i                                      (Eq. 17)
//   dL/dlogp_t = M_i / Z (-rho_t A_i [unclipped branch] + beta (1 - e^r))
//
// Two launches: (1) Z from the filter's keep / n_tokens, an exact integer
// sum over many CTAs; (2) persistent CTAs stride over the sequences, write g_t
// for every token (16-byte loads and stores, two vectors in flight per
// thread) and each response's shares of L and of the KL estimate; the last
// CTA to finish sums the shares in a fixed order. Every floating-point
// reduction has a fixed order, so results are bitwise reproducible.
#include "mc_internal.h"
#include "mc_ptx.cuh"

namespace mc {

namespace {

constexpr int kLossThreads = 256;
constexpr int kReduceThreads = 1024;

// Z = sum_i M_i L_i over every sequence: an integer sum, so CTAs may add
// their warps' parts with 64-bit atomics in any order and Z stays exact.
// (*Z is zeroed on the stream before.) Block 0 also zeroes the clip count.
__global__ void __launch_bounds__(kReduceThreads) grpo_norm_kernel(const uint8_t* __restrict__ keep,
                                                                   const int32_t* __restrict__ n_tokens, int B,
                                                                   long long* Z, int32_t* n_clipped) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  long long v = 0;
  if (i < B && keep[i]) v = n_tokens[i] > 0 ? n_tokens[i] : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if ((threadIdx.x & 31) == 0 && v != 0)
    atomicAdd(reinterpret_cast<unsigned long long*>(Z), static_cast<unsigned long long>(v));
  if (blockIdx.x == 0 && threadIdx.x == 0 && n_clipped) *n_clipped = 0;
}

struct TokAcc {
  float s;    // sum of surrogates
  float kl;   // sum of KL estimates
  int clipped;
};

struct SeqConst {
  float A, lo, hi;
  float kz;     // M_i / Z
  float kbeta;  // beta M_i / Z
};

template <bool kRef>
__device__ __forceinline__ float token_grad(float lp, float lb, float lr, bool counted, const SeqConst& c,
                                            TokAcc& acc) {
  if (!counted) return 0.f;
  const float rho = __expf(lp - lb);                 // Eq. 4
  const float u = rho * c.A;                         // unclipped surrogate
  const float cl = fminf(fmaxf(rho, c.lo), c.hi) * c.A;
  const bool clipped = cl < u;                       // ties take the unclipped branch
  acc.s += clipped ? cl : u;
  acc.clipped += clipped ? 1 : 0;
  float g = clipped ? 0.f : -c.kz * u;               // -M_i rho A / Z
  if (kRef) {
    const float r = lr - lp;
    const float er = __expf(r);
    acc.kl += er - r - 1.f;
    g = fmaf(c.kbeta, 1.f - er, g);                  // + beta M_i (1 - e^r) / Z
  }
  return g;
}

template <bool kRef>
__device__ __forceinline__ float4 vec_grad(const float4& lp, const float4& lb, const float4& lr, uchar4 mk,
                                           const SeqConst& c, TokAcc& acc) {
  float4 g;
  g.x = token_grad<kRef>(lp.x, lb.x, lr.x, mk.x != 0, c, acc);
  g.y = token_grad<kRef>(lp.y, lb.y, lr.y, mk.y != 0, c, acc);
  g.z = token_grad<kRef>(lp.z, lb.z, lr.z, mk.z != 0, c, acc);
  g.w = token_grad<kRef>(lp.w, lb.w, lr.w, mk.w != 0, c, acc);
  return g;
}

template <bool kRef>
__global__ void __launch_bounds__(kLossThreads) grpo_loss_kernel(LossArgs p) {
  __shared__ TokAcc warp_acc[kLossThreads / 32];
  const long long Z = *p.Z;
  const float4* lp4 = reinterpret_cast<const float4*>(p.logp_policy);
  const float4* lb4 = reinterpret_cast<const float4*>(p.logp_behaviour);
  const float4* lr4 = reinterpret_cast<const float4*>(p.logp_ref);
  const uchar4* m4 = reinterpret_cast<const uchar4*>(p.loss_mask);
  float4* g4 = reinterpret_cast<float4*>(p.grad_logp);
  const float4 zero4 = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int i = blockIdx.x; i < p.B; i += gridDim.x) {
    long long b = p.cu_seqlens[i];
    long long e = p.cu_seqlens[i + 1];
    b = b < 0 ? 0 : (b > p.N ? p.N : b);
    e = e < b ? b : (e > p.N ? p.N : e);
    const float M = (p.keep[i] != 0 && Z > 0) ? 1.f : 0.f;
    SeqConst c;
    c.A = p.advantages[i];
    c.lo = 1.f - p.eps_low;
    c.hi = 1.f + p.eps_high;
    c.kz = Z > 0 ? M / static_cast<float>(Z) : 0.f;
    c.kbeta = p.beta * c.kz;

    TokAcc acc{0.f, 0.f, 0};
    long long hb = p.vec_ok ? ((b + 3) & ~3LL) : e;
    if (hb > e) hb = e;
    const long long vend = hb + ((e - hb) & ~3LL);
    for (long long t = b + threadIdx.x; t < hb; t += blockDim.x)
      p.grad_logp[t] = token_grad<kRef>(p.logp_policy[t], p.logp_behaviour[t], kRef ? p.logp_ref[t] : 0.f,
                                        p.loss_mask ? p.loss_mask[t] != 0 : true, c, acc);
    const long long q1 = vend >> 2;
    for (long long q = (hb >> 2) + threadIdx.x; q < q1; q += 2LL * blockDim.x) {
      const long long r = q + blockDim.x;
      const bool two = r < q1;
      const float4 lpa = __ldcs(lp4 + q), lba = __ldcs(lb4 + q);
      const float4 lra = kRef ? __ldcs(lr4 + q) : zero4;
      const uchar4 ma = p.loss_mask ? m4[q] : make_uchar4(1, 1, 1, 1);
      float4 lpb = zero4, lbb = zero4, lrb = zero4;
      uchar4 mb = make_uchar4(0, 0, 0, 0);
      if (two) {
        lpb = __ldcs(lp4 + r);
        lbb = __ldcs(lb4 + r);
        if (kRef) lrb = __ldcs(lr4 + r);
        mb = p.loss_mask ? m4[r] : make_uchar4(1, 1, 1, 1);
      }
      __stcs(g4 + q, vec_grad<kRef>(lpa, lba, lra, ma, c, acc));
      if (two) __stcs(g4 + r, vec_grad<kRef>(lpb, lbb, lrb, mb, c, acc));
    }
    for (long long t = vend + threadIdx.x; t < e; t += blockDim.x)
      p.grad_logp[t] = token_grad<kRef>(p.logp_policy[t], p.logp_behaviour[t], kRef ? p.logp_ref[t] : 0.f,
                                        p.loss_mask ? p.loss_mask[t] != 0 : true, c, acc);

#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      acc.s += __shfl_xor_sync(0xffffffffu, acc.s, o);
      acc.kl += __shfl_xor_sync(0xffffffffu, acc.kl, o);
      acc.clipped += __shfl_xor_sync(0xffffffffu, acc.clipped, o);
    }
    if ((threadIdx.x & 31) == 0) warp_acc[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
      TokAcc tot{0.f, 0.f, 0};
      for (int w = 0; w < kLossThreads / 32; ++w) {
        tot.s += warp_acc[w].s;
        tot.kl += warp_acc[w].kl;
        tot.clipped += warp_acc[w].clipped;
      }
      const float kl_share = tot.kl * c.kz;                 // this response's share of KL
      const float share = -tot.s * c.kz + p.beta * kl_share;  // and of L
      p.seq_share[i] = share;
      p.seq_kl[i] = kl_share;
      if (p.seq_loss) p.seq_loss[i] = share;
      if (p.n_clipped && M != 0.f && tot.clipped) atomicAdd(p.n_clipped, tot.clipped);
    }
    __syncthreads();  // warp_acc is reused by the next sequence
  }

  // The last CTA to finish sums the per-sequence shares in a fixed order
  // (deterministic): every CTA publishes its shares, then takes a ticket.
  __shared__ bool last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(p.ticket, 1u) == gridDim.x - 1;
  __syncthreads();
  if (!last) return;
  __threadfence();
  // Four consecutive shares per thread and step (one 16-byte load from each
  // 256-byte-aligned workspace array), four partial sums combined in order.
  float la[4] = {0.f, 0.f, 0.f, 0.f}, ka[4] = {0.f, 0.f, 0.f, 0.f};
  const int B4 = p.B & ~3;
#pragma unroll 4
  for (int i = 4 * threadIdx.x; i < B4; i += 4 * blockDim.x) {
    const float4 sv = __ldcg(reinterpret_cast<const float4*>(p.seq_share + i));
    const float4 kv = __ldcg(reinterpret_cast<const float4*>(p.seq_kl + i));
    la[0] += sv.x;
    la[1] += sv.y;
    la[2] += sv.z;
    la[3] += sv.w;
    ka[0] += kv.x;
    ka[1] += kv.y;
    ka[2] += kv.z;
    ka[3] += kv.w;
  }
  if (threadIdx.x < p.B - B4) {
    la[0] += __ldcg(p.seq_share + B4 + threadIdx.x);
    ka[0] += __ldcg(p.seq_kl + B4 + threadIdx.x);
  }
  float l = (la[0] + la[1]) + (la[2] + la[3]);
  float k = (ka[0] + ka[1]) + (ka[2] + ka[3]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    l += __shfl_xor_sync(0xffffffffu, l, o);
    k += __shfl_xor_sync(0xffffffffu, k, o);
  }
  if ((threadIdx.x & 31) == 0) {
    warp_acc[threadIdx.x >> 5].s = l;
    warp_acc[threadIdx.x >> 5].kl = k;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float lt = 0.f, kt = 0.f;
    for (int w = 0; w < kLossThreads / 32; ++w) {
      lt += warp_acc[w].s;
      kt += warp_acc[w].kl;
    }
    *p.loss = lt;
    if (p.kl) *p.kl = kt;
  }
}

}  // namespace

cudaError_t launch_grpo_loss(const LossArgs& a, cudaStream_t stream) {
  // Z and the ticket counter start at zero.
  cudaError_t e = cudaMemsetAsync(a.Z, 0, sizeof(long long) + sizeof(unsigned int), stream);
  if (e != cudaSuccess) return e;
  grpo_norm_kernel<<<(a.B + kReduceThreads - 1) / kReduceThreads, kReduceThreads, 0, stream>>>(
      a.keep, a.n_tokens, a.B, a.Z, a.n_clipped);
  e = launched();
  if (e != cudaSuccess) return e;
  const int grid = a.B < a.grid ? a.B : a.grid;
  if (a.logp_ref != nullptr)
    grpo_loss_kernel<true><<<grid, kLossThreads, 0, stream>>>(a);
  else
    grpo_loss_kernel<false><<<grid, kLossThreads, 0, stream>>>(a);
  return launched();
}

}  // namespace mc
