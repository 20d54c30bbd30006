// mc_fwd.cu — fused LM-head projection + online log-softmax / entropy.
//
// The projection z = (h . w) * inv_temperature runs on the tensor cores
// (mc_gemm.cuh); the accumulator tiles are consumed in TMEM by the epilogue
// below and never reach memory. Each epilogue thread owns one token row and
// keeps, in base 2 (a = z * log2 e),
//     m = max a,   s = sum 2^(a - m),   t = sum 2^(a - m) (a - m)
// over the vocabulary columns of its unit. When a new chunk raises the
// maximum from m to m', s <- s 2^(m - m') and t <- 2^(m - m') (t + (m - m') s).
// At the end of the unit (m, s, t) goes to the split's partial slot; the
// target logit z_y is written by whichever unit holds column y. A second
// kernel merges the splits of each row with the same rule and finishes
//     lse = ln2 (m + log2 s),  entropy = ln2 (log2 s - t / s),  logp = z_y - lse.
// This single-pass form equals the two-pass definition of the log-softmax
// and of the Shannon entropy (-sum p log p) exactly in real arithmetic.
#include <cuda_bf16.h>

#include "mc_gemm.cuh"
#include "mc_internal.h"

namespace mc {

namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

struct FwdParams {
  const int32_t* targets;
  long long N;
  int V;
  float scale2;  // inv_temperature * log2(e)
  float inv_temp;
  float* part;   // [3][slots][n_pad]
  float* zy;     // [n_pad]
  long long n_pad;
  int slots;     // partial states per row: vocabulary splits x column halves
  int v_offset;  // global id of column 0 (a vocabulary shard), 0 for the full vocabulary
};

// H = 2 (256-row tiles only): two warp groups per 128-row sub-block, each
// keeping its own online state over one half of every tile's 256 columns;
// the two halves' states go to slots 2 split and 2 split + 1 and are merged
// by the finalize kernel like any other split.
template <int H>
struct FwdEpiT {
  using Params = FwdParams;
  static constexpr int kColumnHalves = H;
  static constexpr int kChunks = BN / 32 / H;  // 32-column chunks this warp reads per tile

  float m, s0, s1, t0, t1;
  int y;
  int half = 0;

  __device__ __forceinline__ void setup(const Params&, long long, bool) {}
  __device__ __forceinline__ void set_half(int h) { half = h; }

  __device__ __forceinline__ void begin(const Params& p, long long row, int, int) {
    m = -INFINITY;
    s0 = s1 = t0 = t1 = 0.f;
    y = row < p.N ? __ldg(p.targets + row) - p.v_offset : -1;  // column of the target in this W
  }

  // Online update with 32 values of which the first `nvalid` are real columns.
  template <bool kFull>
  __device__ __forceinline__ void update(const float (&x)[32], int nvalid, float scale2) {
    float cm = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (kFull || i < nvalid) cm = fmaxf(cm, x[i]);
    cm *= scale2;
    if (cm > m) {
      if (s0 + s1 > 0.f) {
        const float dm = m - cm;
        const float r = ex2_approx(dm);
        t0 = r * fmaf(dm, s0, t0);
        t1 = r * fmaf(dm, s1, t1);
        s0 *= r;
        s1 *= r;
      }
      m = cm;
    }
    const float nm = -m;
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
      if (kFull || i < nvalid) {
        const float a = fmaf(x[i], scale2, nm);
        const float e = ex2_approx(a);
        s0 += e;
        t0 = fmaf(e, a, t0);
      }
      if (kFull || i + 1 < nvalid) {
        const float a = fmaf(x[i + 1], scale2, nm);
        const float e = ex2_approx(a);
        s1 += e;
        t1 = fmaf(e, a, t1);
      }
    }
  }

  __device__ __forceinline__ void tile(const Params& p, long long row, int n_tile, uint32_t taddr) {
    const int v0 = n_tile * BN;
#pragma unroll 1
    for (int c = half * kChunks; c < (half + 1) * kChunks; ++c) {
      float x[32];
      tmem_ld32(taddr + c * 32, x);
      const int vc = v0 + c * 32;
      const int rel = y - vc;
      if (rel >= 0 && rel < 32) {  // this row's target lies in this chunk
        float zv = x[0];
#pragma unroll
        for (int i = 1; i < 32; ++i) zv = (i == rel) ? x[i] : zv;
        p.zy[row] = zv * p.inv_temp;
      }
      const int nvalid = p.V - vc;
      if (nvalid >= 32)
        update<true>(x, 32, p.scale2);
      else if (nvalid > 0)
        update<false>(x, nvalid, p.scale2);
    }
  }

  __device__ __forceinline__ void end(const Params& p, long long row, int, int split, bool ok) {
    const long long plane = static_cast<long long>(p.slots) * p.n_pad;
    const long long o = static_cast<long long>(split * H + half) * p.n_pad + row;
    p.part[o] = ok ? m : NAN;
    p.part[plane + o] = s0 + s1;
    p.part[2 * plane + o] = t0 + t1;
  }
};

__global__ void fwd_finalize(const int32_t* __restrict__ targets, long long N, int V, int splits,
                             long long n_pad, const float* __restrict__ part, const float* __restrict__ zy,
                             float* __restrict__ logp, float* __restrict__ entropy, float* __restrict__ lse,
                             const int32_t* __restrict__ ws_status, int32_t* dev_status) {
  const long long row = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (blockIdx.x == 0 && threadIdx.x == 0 && dev_status != nullptr && *ws_status != 0)
    atomicOr(dev_status, *ws_status);
  if (row >= N) return;
  bool bad = (*ws_status & MC_DEV_TIMEOUT) != 0;
  const int y = targets[row];
  const bool y_bad = y < 0 || y >= V;
  if (__any_sync(__activemask(), y_bad) && dev_status != nullptr && (threadIdx.x & 31) == 0)
    atomicOr(dev_status, MC_DEV_TARGET_RANGE);
  bad |= y_bad;

  const long long plane = static_cast<long long>(splits) * n_pad;
  float M = -INFINITY;
  for (int k = 0; k < splits; ++k) {
    const float mk = part[static_cast<long long>(k) * n_pad + row];
    bad |= isnan(mk);
    M = fmaxf(M, mk);
  }
  float S = 0.f, T = 0.f;
  for (int k = 0; k < splits; ++k) {
    const long long o = static_cast<long long>(k) * n_pad + row;
    const float mk = part[o];
    const float sk = part[plane + o];
    const float tk = part[2 * plane + o];
    if (!(sk > 0.f)) continue;
    const float dm = mk - M;
    const float r = exp2f(dm);
    S = fmaf(sk, r, S);
    T = fmaf(r, fmaf(dm, sk, tk), T);
  }
  const float l2s = log2f(S);
  const float lse_v = kLn2 * (M + l2s);
  const float ent_v = kLn2 * (l2s - T / S);
  const float logp_v = bad ? NAN : zy[row] - lse_v;
  logp[row] = logp_v;
  if (entropy) entropy[row] = bad ? NAN : ent_v;
  if (lse) lse[row] = bad ? NAN : lse_v;
}

// Shard mode: the merged split partials of each row as a natural-unit state
// (m, s, t, z_y) of this vocabulary slice; z_y = -inf when the slice does not
// hold the row's target.
__global__ void fwd_state_finalize(const int32_t* __restrict__ targets, long long N, int V, int v_offset,
                                   int splits, long long n_pad, const float* __restrict__ part,
                                   const float* __restrict__ zy, float4* __restrict__ state,
                                   const int32_t* __restrict__ ws_status, int32_t* dev_status) {
  const long long row = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (blockIdx.x == 0 && threadIdx.x == 0 && dev_status != nullptr && *ws_status != 0)
    atomicOr(dev_status, *ws_status);
  if (row >= N) return;
  bool bad = (*ws_status & MC_DEV_TIMEOUT) != 0;
  const long long plane = static_cast<long long>(splits) * n_pad;
  float M = -INFINITY;
  for (int k = 0; k < splits; ++k) {
    const float mk = part[static_cast<long long>(k) * n_pad + row];
    bad |= isnan(mk);
    M = fmaxf(M, mk);
  }
  float S = 0.f, T = 0.f;
  for (int k = 0; k < splits; ++k) {
    const long long o = static_cast<long long>(k) * n_pad + row;
    const float sk = part[plane + o];
    if (!(sk > 0.f)) continue;
    const float dm = part[o] - M;
    const float r = exp2f(dm);
    S = fmaf(sk, r, S);
    T = fmaf(r, fmaf(dm, sk, part[2 * plane + o]), T);
  }
  const int local = targets[row] - v_offset;
  const float zv = (local >= 0 && local < V) ? zy[row] : -INFINITY;
  state[row] = bad ? make_float4(NAN, NAN, NAN, NAN) : make_float4(kLn2 * M, S, kLn2 * T, zv);
}

// Per row: combine the P slice states into the full-vocabulary log-sum-exp,
// entropy and target log-prob (the same rescale-to-a-common-max rule as the
// online update). A row whose target no slice holds gets NaN and sets
// MC_DEV_TARGET_RANGE.
__global__ void merge_states_kernel(const float4* __restrict__ states, int P, long long N, float* __restrict__ logp,
                                    float* __restrict__ entropy, float* __restrict__ lse, int32_t* dev_status) {
  const long long row = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (row >= N) return;
  float M = -INFINITY, zv = -INFINITY;
  bool bad = false;
  for (int p = 0; p < P; ++p) {
    const float4 s = states[static_cast<long long>(p) * N + row];
    bad |= isnan(s.x);
    M = fmaxf(M, s.x);
    zv = fmaxf(zv, s.w);
  }
  float S = 0.f, T = 0.f;
  for (int p = 0; p < P; ++p) {
    const float4 s = states[static_cast<long long>(p) * N + row];
    if (!(s.y > 0.f)) continue;
    const float dm = s.x - M;
    const float r = __expf(dm);
    S = fmaf(s.y, r, S);
    T = fmaf(r, fmaf(dm, s.y, s.z), T);
  }
  const bool no_target = !(zv > -INFINITY);
  if (__any_sync(__activemask(), no_target) && dev_status != nullptr && (threadIdx.x & 31) == 0)
    atomicOr(dev_status, MC_DEV_TARGET_RANGE);
  bad |= no_target;
  const float ls = logf(S);
  const float lse_v = M + ls;
  logp[row] = bad ? NAN : zv - lse_v;
  if (entropy) entropy[row] = bad ? NAN : ls - T / S;
  if (lse) lse[row] = bad ? NAN : lse_v;
}

}  // namespace

template <int MS, int H>
cudaError_t run_forward_gemm(const FwdArgs& a, const Schedule& sch, const FwdParams& ep, cudaStream_t stream) {
  using Epi = FwdEpiT<H>;
  auto kern = gemm_persistent<Epi, false, false, MS>;
  constexpr size_t smem = TileFor<Epi, MS>::template smem_bytes<Epi>();
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int units = sch.m_blocks * sch.splits;
  const int grid = units < a.grid ? units : a.grid;
  // Cooperative launch: the wave gate needs every CTA resident (one per SM).
  Schedule gated = sch;
  gated.wave_ctr = a.wave_ctr;
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(TileFor<Epi, MS>::THREADS);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, kern, a.tm_hidden, a.tm_w, gated, ep, a.timeout_ns, a.ws_status);
  if (e != cudaSuccess) return e;
  return launched();
}

cudaError_t launch_merge_states(const float* states, int P, long long N, float* logp, float* entropy, float* lse,
                                int32_t* dev_status, cudaStream_t stream) {
  if (N <= 0) return cudaSuccess;
  const int threads = 256;
  const long long blocks = (N + threads - 1) / threads;
  merge_states_kernel<<<static_cast<unsigned>(blocks), threads, 0, stream>>>(
      reinterpret_cast<const float4*>(states), P, N, logp, entropy, lse, dev_status);
  return launched();
}

cudaError_t launch_forward(const FwdArgs& a, cudaStream_t stream) {
  cudaError_t e;
  Schedule sch;
  const int row_block = a.wide ? 2 * BM : BM;
  sch.m_blocks = static_cast<int>((a.N + row_block - 1) / row_block);
  sch.n_tiles = (a.V + BN - 1) / BN;
  sch.splits = a.splits;
  sch.k_blocks = a.d / BK;
  const int halves = (a.wide && a.halves == 2) ? 2 : 1;
  const int slots = a.splits * halves;
  FwdParams ep;
  ep.targets = a.targets;
  ep.N = a.N;
  ep.V = a.V;
  ep.scale2 = a.inv_temperature * kLog2e;
  ep.inv_temp = a.inv_temperature;
  ep.part = a.part;
  ep.zy = a.zy;
  ep.n_pad = a.n_pad;
  ep.slots = slots;
  ep.v_offset = a.v_offset;
  if (a.wide && halves == 2) {
    e = run_forward_gemm<2, 2>(a, sch, ep, stream);
  } else if (a.wide) {
    e = run_forward_gemm<2, 1>(a, sch, ep, stream);
  } else {
    e = run_forward_gemm<1, 1>(a, sch, ep, stream);
  }
  if (e != cudaSuccess) return e;
  const int threads = 256;
  const long long blocks = (a.N + threads - 1) / threads;
  if (a.state != nullptr)
    fwd_state_finalize<<<static_cast<unsigned>(blocks), threads, 0, stream>>>(
        a.targets, a.N, a.V, a.v_offset, slots, a.n_pad, a.part, a.zy, reinterpret_cast<float4*>(a.state),
        a.ws_status, a.dev_status);
  else
    fwd_finalize<<<static_cast<unsigned>(blocks), threads, 0, stream>>>(
        a.targets, a.N, a.V, slots, a.n_pad, a.part, a.zy, a.logp, a.entropy, a.lse, a.ws_status,
        a.dev_status);
  return launched();
}

}  // namespace mc
