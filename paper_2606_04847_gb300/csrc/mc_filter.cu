// mc_filter.cu — per-sequence importance-ratio statistics and the MirrorPop
// keep-mask (§4.5.2, Eq. 18-21), plus per-token ratios (Eq. 4).
//
// Persistent CTAs of 128 threads, as many as the SMs keep resident at once (12
// per SM at the kernel's 37 registers: one wave, no late second wave at low
// occupancy), stride over the sequences, one sequence at a time per CTA. Each
// thread walks its share of the sequence's packed tokens with 16-byte loads
// (4 tokens of logp_policy / logp_behaviour, 4 mask bytes; two vectors in
// flight), accumulates sum(log rho), sum(|log rho|) and the count over
// loss-masked tokens, and writes rho = exp(log rho) on the way (streaming
// stores). Warp shuffles then a shared-memory step reduce the three sums in a
// fixed order (deterministic for a given launch shape). Thread 0 forms the
// statistics and the masks; a second sweep writes token_keep once keep_i is
// known, 16 tokens per 16-byte load of the mask and store. The kernel is
// HBM-bound: 4 + 4 + 1 bytes read and up to 4 + 1 bytes written per token.
#include "mc_internal.h"
#include "mc_ptx.cuh"

namespace mc {

namespace {

constexpr int kFilterThreads = 128;

struct Acc {
  float s, a;
  int n;
};

__device__ __forceinline__ void add_token(Acc& acc, float lp, float lb, bool m, float* ratio_out) {
  const float d = lp - lb;  // log rho
  if (ratio_out) *ratio_out = __expf(d);
  if (m) {
    acc.s += d;
    acc.a += fabsf(d);
    acc.n += 1;
  }
}

__device__ __forceinline__ void add_vec(Acc& acc, const float4& lp, const float4& lb, uchar4 mk, float* ratio_out) {
  const float d0 = lp.x - lb.x, d1 = lp.y - lb.y, d2 = lp.z - lb.z, d3 = lp.w - lb.w;
  if (ratio_out) __stcs(reinterpret_cast<float4*>(ratio_out), make_float4(__expf(d0), __expf(d1), __expf(d2), __expf(d3)));
  if (mk.x) { acc.s += d0; acc.a += fabsf(d0); acc.n += 1; }
  if (mk.y) { acc.s += d1; acc.a += fabsf(d1); acc.n += 1; }
  if (mk.z) { acc.s += d2; acc.a += fabsf(d2); acc.n += 1; }
  if (mk.w) { acc.s += d3; acc.a += fabsf(d3); acc.n += 1; }
}

// 0x01 in every byte of w that is nonzero, 0x00 elsewhere: the low seven bits
// of a byte plus 0x7F reach bit 7 exactly when they are not all zero (no carry
// leaves the byte), and OR-ing the byte itself covers its own bit 7.
__device__ __forceinline__ uint32_t nonzero_bytes(uint32_t w) {
  return ((((w & 0x7F7F7F7Fu) + 0x7F7F7F7Fu) | w) & 0x80808080u) >> 7;
}
__device__ __forceinline__ uint4 nonzero_bytes(uint4 v) {
  return make_uint4(nonzero_bytes(v.x), nonzero_bytes(v.y), nonzero_bytes(v.z), nonzero_bytes(v.w));
}

// Persistent over sequences (CTA c handles sequences c, c + gridDim.x, ...).
__global__ void __launch_bounds__(kFilterThreads) seq_filter_kernel(FilterArgs p) {
  __shared__ Acc warp_acc[kFilterThreads / 32];
  __shared__ int keep_s;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = blockIdx.x; i < p.B; i += gridDim.x) {
    long long b = p.cu_seqlens[i];
    long long e = p.cu_seqlens[i + 1];
    // Clamp the segment to [0, N) so malformed cu_seqlens cannot index out of bounds.
    b = b < 0 ? 0 : (b > p.N ? p.N : b);
    e = e < b ? b : (e > p.N ? p.N : e);

    Acc acc{0.f, 0.f, 0};
    // Scalar head up to a multiple of 4 tokens, then 4-token vectors (two in
    // flight per thread: both loads issue before either is used), then the tail.
    // (p.vec_ok = 0 when some pointer is not aligned for vector access: all scalar.)
    long long hb = p.vec_ok ? ((b + 3) & ~3LL) : e;
    if (hb > e) hb = e;
    const long long vend = hb + ((e - hb) & ~3LL);
    for (long long t = b + threadIdx.x; t < hb; t += blockDim.x)
      add_token(acc, p.logp_policy[t], p.logp_behaviour[t], p.loss_mask ? p.loss_mask[t] != 0 : true,
                p.token_ratio ? p.token_ratio + t : nullptr);
    const long long q1 = vend >> 2;
    const float4* lp4 = reinterpret_cast<const float4*>(p.logp_policy);
    const float4* lb4 = reinterpret_cast<const float4*>(p.logp_behaviour);
    const uchar4* m4 = reinterpret_cast<const uchar4*>(p.loss_mask);
    for (long long q = (hb >> 2) + threadIdx.x; q < q1; q += 2LL * blockDim.x) {
      const long long r = q + blockDim.x;
      const bool two = r < q1;
      const float4 lp0 = __ldcs(lp4 + q);
      const float4 lb0 = __ldcs(lb4 + q);
      const uchar4 m0 = p.loss_mask ? m4[q] : make_uchar4(1, 1, 1, 1);
      float4 lp1 = make_float4(0.f, 0.f, 0.f, 0.f), lb1 = lp1;
      uchar4 m1 = make_uchar4(0, 0, 0, 0);
      if (two) {
        lp1 = __ldcs(lp4 + r);
        lb1 = __ldcs(lb4 + r);
        m1 = p.loss_mask ? m4[r] : make_uchar4(1, 1, 1, 1);
      }
      add_vec(acc, lp0, lb0, m0, p.token_ratio ? p.token_ratio + 4 * q : nullptr);
      if (two) add_vec(acc, lp1, lb1, m1, p.token_ratio ? p.token_ratio + 4 * r : nullptr);
    }
    for (long long t = vend + threadIdx.x; t < e; t += blockDim.x)
      add_token(acc, p.logp_policy[t], p.logp_behaviour[t], p.loss_mask ? p.loss_mask[t] != 0 : true,
                p.token_ratio ? p.token_ratio + t : nullptr);

#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      acc.s += __shfl_xor_sync(0xffffffffu, acc.s, off);
      acc.a += __shfl_xor_sync(0xffffffffu, acc.a, off);
      acc.n += __shfl_xor_sync(0xffffffffu, acc.n, off);
    }
    if (lane == 0) warp_acc[warp] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
      Acc tot{0.f, 0.f, 0};
      for (int w = 0; w < kFilterThreads / 32; ++w) {
        tot.s += warp_acc[w].s;
        tot.a += warp_acc[w].a;
        tot.n += warp_acc[w].n;
      }
      float S = 0.f, A = 0.f;
      int keep = 0, keep_v = 0;
      if (tot.n > 0) {
        S = tot.s / static_cast<float>(tot.n);
        A = tot.a / static_cast<float>(tot.n);
        keep = A <= p.delta ? 1 : 0;                                   // Eq. 21
        keep_v = (p.delta_vanilla >= 0.f && fabsf(S) <= p.delta_vanilla) ? 1 : 0;
      }
      p.signed_mean[i] = S;
      p.abs_mean[i] = A;
      p.n_tokens[i] = tot.n;
      p.keep[i] = static_cast<uint8_t>(keep);
      if (p.keep_vanilla) p.keep_vanilla[i] = static_cast<uint8_t>(keep_v);
      keep_s = keep;
    }
    __syncthreads();
    if (p.token_keep != nullptr) {
      const uint8_t k = static_cast<uint8_t>(keep_s);
      // token_keep = keep_i & (mask != 0): scalar up to a 16-token boundary,
      // then 16 tokens per 16-byte load / store, then the tail (all scalar
      // when the bases are not 16-byte aligned).
      long long hb = p.keep_vec_ok ? ((b + 15) & ~15LL) : e;
      if (hb > e) hb = e;
      const long long vend = hb + ((e - hb) & ~15LL);
      for (long long t = b + threadIdx.x; t < hb; t += blockDim.x)
        p.token_keep[t] = static_cast<uint8_t>(k & (p.loss_mask ? (p.loss_mask[t] != 0) : 1));
      const uint4* m16 = reinterpret_cast<const uint4*>(p.loss_mask);
      uint4* k16 = reinterpret_cast<uint4*>(p.token_keep);
      for (long long q = (hb >> 4) + threadIdx.x; q < (vend >> 4); q += blockDim.x) {
        uint4 o = make_uint4(0u, 0u, 0u, 0u);
        if (k) o = p.loss_mask ? nonzero_bytes(m16[q]) : make_uint4(0x01010101u, 0x01010101u, 0x01010101u,
                                                                    0x01010101u);
        k16[q] = o;
      }
      for (long long t = vend + threadIdx.x; t < e; t += blockDim.x)
        p.token_keep[t] = static_cast<uint8_t>(k & (p.loss_mask ? (p.loss_mask[t] != 0) : 1));
    }
    __syncthreads();  // warp_acc / keep_s are reused by the next sequence
  }
}

// A global counter nothing ever raises (zero for the life of the module).
__device__ unsigned int g_selftest_counter;

// Waits, through the two bounded waits the pipelined kernels use, on a
// barrier nothing arrives at (warp 0) and on a global counter nothing raises
// (warp 1, the wave gate's wait); each must give up and set MC_DEV_TIMEOUT.
__global__ void selftest_wait_kernel(int32_t* dev_status, uint64_t timeout_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_flag, timeout_ns, dev_status);
  if (threadIdx.x == 32) counter_wait_geq(&g_selftest_counter, 1u, nullptr, timeout_ns, dev_status);
}

}  // namespace

int filter_ctas_per_sm() {
  static const int n = [] {
    int b = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, seq_filter_kernel, kFilterThreads, 0) != cudaSuccess ||
        b < 1) {
      cudaGetLastError();  // clear the failed query, so the launch check after it does not report it
      b = 1;
    }
    return b;
  }();
  return n;
}

cudaError_t launch_filter(const FilterArgs& a, cudaStream_t stream) {
  if (a.B <= 0) return cudaSuccess;
  const int grid = a.B < a.grid ? a.B : a.grid;
  seq_filter_kernel<<<grid, kFilterThreads, 0, stream>>>(a);
  return launched();
}

cudaError_t launch_selftest_wait(int32_t* dev_status, uint64_t timeout_ns, cudaStream_t stream) {
  selftest_wait_kernel<<<1, 64, 0, stream>>>(dev_status, timeout_ns);
  return launched();
}

}  // namespace mc
