// mc_bwd.cu — backward of the fused log-prob / entropy forward.
//
// Stage 1 (dZ producer): the forward's tensor-core mainloop recomputes each
// 128 x 256 logit tile in TMEM; the epilogue turns it into
//     p        = 2^(z log2e - lse log2e)
//     dZ[t, v] = inv_temp ( g_t (1[v = y_t] - p) - gH_t p (log p + H_t) )
// and stores dZ as bf16 (a gradient, not the logits) to the workspace.
// Stage 2: grad_hidden = dZ . W     (A = dZ K-major, B = W read N-major)
// Stage 3: grad_w (+)= dZ^T . H     (A = dZ read M-major, B = H read N-major)
// Both are plain tcgen05 GEMMs of the same engine with store epilogues.
#include <cuda_bf16.h>

#include "mc_gemm.cuh"
#include "mc_internal.h"

namespace mc {

namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

struct DzEpi {
  struct Params {
    const int32_t* targets;
    const float* lse;
    const float* entropy;
    const float* grad_logp;
    const float* grad_entropy;
    long long rows;
    int V;
    float scale2;
    float inv_temp;
    __nv_bfloat16* dz;
    long long ld;
    int32_t* status;
  };

  float lse2, cg, cgh, hrow;
  int y;
  bool valid;

  __device__ __forceinline__ void begin(const Params& p, long long row, int, int) {
    valid = row < p.rows;
    y = -1;
    lse2 = cg = cgh = hrow = 0.f;
    if (!valid) return;
    y = __ldg(p.targets + row);
    cg = __ldg(p.grad_logp + row) * p.inv_temp;
    cgh = p.grad_entropy ? __ldg(p.grad_entropy + row) * p.inv_temp : 0.f;
    hrow = (p.grad_entropy && p.entropy) ? __ldg(p.entropy + row) : 0.f;
    lse2 = __ldg(p.lse + row) * kLog2e;
    if (y < 0 || y >= p.V) {  // invalid target: drop the row's gradient terms
      atomicOr(p.status, MC_DEV_TARGET_RANGE);
      cg = cgh = 0.f;
      lse2 = 0.f;
    }
  }

  __device__ __forceinline__ void tile(const Params& p, long long row, int n_tile, uint32_t taddr) {
    const int v0 = n_tile * BN;
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      float x[32];
      tmem_ld32(taddr + c * 32, x);
      const int vc = v0 + c * 32;
      if (!valid || vc >= p.V) continue;
      const float nl = -lse2;
      uint32_t w[16];
#pragma unroll
      for (int i = 0; i < 32; i += 2) {
        float d2[2];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const float a = fmaf(x[i + j], p.scale2, nl);  // log2 p
          const float pr = ex2_approx(a);
          const float oh = (vc + i + j == y) ? 1.f : 0.f;
          d2[j] = fmaf(cg, oh - pr, -cgh * pr * fmaf(a, kLn2, hrow));
        }
        w[i / 2] = pack_bf16x2(d2[0], d2[1]);
      }
      __nv_bfloat16* dst = p.dz + row * p.ld + vc;
      if (vc + 32 <= p.V) {
        uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
        for (int q = 0; q < 4; ++q) d4[q] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
      } else {
        const int n = p.V - vc;
        for (int i = 0; i < n; ++i) {
          const uint32_t pair = w[i / 2];
          const uint16_t bits = (i & 1) ? static_cast<uint16_t>(pair >> 16) : static_cast<uint16_t>(pair & 0xFFFFu);
          reinterpret_cast<uint16_t*>(dst)[i] = bits;
        }
      }
    }
  }

  __device__ __forceinline__ void end(const Params&, long long, int, int, bool) {}
};

// out[row, col] = acc (bf16), rows < p.rows, cols < p.cols (cols % 32 == 0).
struct StoreBf16Epi {
  struct Params {
    __nv_bfloat16* out;
    long long ld;
    long long rows;
    int cols;
  };
  __device__ __forceinline__ void begin(const Params&, long long, int, int) {}
  __device__ __forceinline__ void tile(const Params& p, long long row, int n_tile, uint32_t taddr) {
    const int n0 = n_tile * BN;
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      float x[32];
      tmem_ld32(taddr + c * 32, x);
      const int col = n0 + c * 32;
      if (row >= p.rows || col >= p.cols) continue;
      uint4* d4 = reinterpret_cast<uint4*>(p.out + row * p.ld + col);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        d4[q] = make_uint4(pack_bf16x2(x[8 * q + 0], x[8 * q + 1]), pack_bf16x2(x[8 * q + 2], x[8 * q + 3]),
                           pack_bf16x2(x[8 * q + 4], x[8 * q + 5]), pack_bf16x2(x[8 * q + 6], x[8 * q + 7]));
    }
  }
  __device__ __forceinline__ void end(const Params&, long long, int, int, bool) {}
};

// out[row, col] (+)= acc (fp32), rows < p.rows, cols < p.cols (cols % 32 == 0).
struct StoreF32Epi {
  struct Params {
    float* out;
    long long ld;
    long long rows;
    int cols;
    int accumulate;
  };
  __device__ __forceinline__ void begin(const Params&, long long, int, int) {}
  __device__ __forceinline__ void tile(const Params& p, long long row, int n_tile, uint32_t taddr) {
    const int n0 = n_tile * BN;
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      float x[32];
      tmem_ld32(taddr + c * 32, x);
      const int col = n0 + c * 32;
      if (row >= p.rows || col >= p.cols) continue;
      float4* d4 = reinterpret_cast<float4*>(p.out + row * p.ld + col);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 v = make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3]);
        if (p.accumulate) {
          const float4 o = d4[q];
          v.x += o.x;
          v.y += o.y;
          v.z += o.z;
          v.w += o.w;
        }
        d4[q] = v;
      }
    }
  }
  __device__ __forceinline__ void end(const Params&, long long, int, int, bool) {}
};

template <class Epi, bool A_MN, bool B_MN>
cudaError_t run_gemm(const CUtensorMap& ta, const CUtensorMap& tb, const Schedule& sch,
                     const typename Epi::Params& ep, int grid_cap, uint64_t timeout_ns, int32_t* status,
                     cudaStream_t stream) {
  auto kern = gemm_persistent<Epi, A_MN, B_MN>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(GEMM_SMEM_BYTES));
  if (e != cudaSuccess) return e;
  const int units = sch.m_blocks * sch.splits;
  const int grid = units < grid_cap ? units : grid_cap;
  if (grid <= 0) return cudaSuccess;
  kern<<<grid, GEMM_THREADS, GEMM_SMEM_BYTES, stream>>>(ta, tb, sch, ep, timeout_ns, status);
  return cudaGetLastError();
}

__global__ void status_merge(const int32_t* ws_status, int32_t* dev_status) {
  if (*ws_status != 0) atomicOr(dev_status, *ws_status);
}

}  // namespace

cudaError_t launch_dz(const DzArgs& a, cudaStream_t stream) {
  Schedule sch;
  sch.m_blocks = static_cast<int>((a.rows + BM - 1) / BM);
  sch.n_tiles = (a.V + BN - 1) / BN;
  sch.splits = a.splits;
  sch.k_blocks = a.d / BK;
  DzEpi::Params ep;
  ep.targets = a.targets;
  ep.lse = a.lse;
  ep.entropy = a.entropy;
  ep.grad_logp = a.grad_logp;
  ep.grad_entropy = a.grad_entropy;
  ep.rows = a.rows;
  ep.V = a.V;
  ep.scale2 = a.inv_temperature * kLog2e;
  ep.inv_temp = a.inv_temperature;
  ep.dz = static_cast<__nv_bfloat16*>(a.dz);
  ep.ld = a.ld;
  ep.status = a.ws_status;
  return run_gemm<DzEpi, false, false>(a.tm_hidden, a.tm_w, sch, ep, a.grid, a.timeout_ns, a.ws_status,
                                       stream);
}

cudaError_t launch_dh(const DhArgs& a, cudaStream_t stream) {
  Schedule sch;
  sch.m_blocks = static_cast<int>((a.rows + BM - 1) / BM);
  sch.n_tiles = (a.d + BN - 1) / BN;
  sch.splits = sch.n_tiles;  // one output tile per unit
  sch.k_blocks = (a.V + BK - 1) / BK;
  StoreBf16Epi::Params ep;
  ep.out = static_cast<__nv_bfloat16*>(a.grad_hidden);
  ep.ld = a.d;
  ep.rows = a.rows;
  ep.cols = a.d;
  return run_gemm<StoreBf16Epi, false, true>(a.tm_dz, a.tm_w_mn, sch, ep, a.grid, a.timeout_ns, a.ws_status,
                                             stream);
}

cudaError_t launch_dw(const DwArgs& a, cudaStream_t stream) {
  Schedule sch;
  sch.m_blocks = (a.V + BM - 1) / BM;
  sch.n_tiles = (a.d + BN - 1) / BN;
  sch.splits = sch.n_tiles;
  sch.k_blocks = static_cast<int>((a.rows + BK - 1) / BK);
  StoreF32Epi::Params ep;
  ep.out = a.grad_w;
  ep.ld = a.d;
  ep.rows = a.V;
  ep.cols = a.d;
  ep.accumulate = a.accumulate;
  return run_gemm<StoreF32Epi, true, true>(a.tm_dz_mn, a.tm_h_mn, sch, ep, a.grid, a.timeout_ns, a.ws_status,
                                           stream);
}

cudaError_t launch_status_merge(const int32_t* ws_status, int32_t* dev_status, cudaStream_t stream) {
  if (dev_status == nullptr) return cudaSuccess;
  status_merge<<<1, 1, 0, stream>>>(ws_status, dev_status);
  return cudaGetLastError();
}

}  // namespace mc
