// mc_bwd.cu — backward of the fused log-prob / entropy forward.
//
// Stage 0 (row selection): rows whose effective upstream gradient is zero
// (row_keep[t] == 0, i.e. M_i = 0 in Eq. 17, or g_t = gH_t = 0, or an invalid
// target) contribute nothing; one CTA scans the rows in order and writes the
// indices of the others (idx[], count). Their hidden rows are gathered into a
// dense block Hc, zero-padded to a multiple of 256 rows. All later extents come
// from the device-side count, so nothing waits on the host.
// Stage 1 (dZ producer): the forward's tensor-core mainloop recomputes each
// 128 x 256 logit tile of the selected rows in TMEM; the epilogue turns it into
//     p        = 2^(z log2e - lse log2e)
//     dZ[j, v] = inv_temp ( g (1[v = y] - p) - gH p (log p + H) )
// and stores dZ as bf16 (a gradient, not the logits) to the workspace.
// Stage 2: grad_hidden[idx[j]] = (dZ . W)[j]   (A = dZ K-major, B = W N-major)
// Stage 3: grad_w (+)= dZ^T . Hc                (A = dZ M-major, B = Hc N-major)
// Stages 2-3 are plain tcgen05 GEMMs of the same engine with store epilogues,
// one output tile per unit, 256-row tiles once K is long (TileCfg<2>) and
// tiles grouped so that a wave reads few operand bytes (Schedule::n_group).
// Every epilogue store is evict-first (st.cs): no output is read again
// before it has left L2, and the operand tiles that the concurrent CTAs
// share stay resident.
#include <cuda_bf16.h>

#include "mc_gemm.cuh"
#include "mc_internal.h"

namespace mc {

namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr int kSelectThreads = 1024;
constexpr int kHcRowPad = 2 * BM;  // gathered rows are zero-padded to whole 256-row blocks

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}

// ---------------------------------------------------------------- stage 0

// Ordered compaction of the rows with a nonzero effective upstream gradient,
// in three launches over slabs of kSelectThreads rows: (1) each slab's count
// of selected rows (and the target range check), (2) one CTA turns the counts
// into exclusive offsets and writes the total, (3) each slab writes its rows'
// indices from its offset, in row order (a block scan of warp ballots). No CTA
// waits on another.
__device__ __forceinline__ int select_flag(const uint8_t* __restrict__ row_keep, const float* __restrict__ g,
                                           const float* __restrict__ gh, const int32_t* __restrict__ targets,
                                           int V, long long t, bool& bad_target) {
  const int y = targets[t];
  const bool yok = y >= 0 && y < V;
  bad_target |= !yok;
  const bool live = g[t] != 0.f || (gh != nullptr && gh[t] != 0.f);
  return (yok && live && (row_keep == nullptr || row_keep[t] != 0)) ? 1 : 0;
}

__global__ void __launch_bounds__(kSelectThreads) select_count_kernel(
    const uint8_t* __restrict__ row_keep, const float* __restrict__ g, const float* __restrict__ gh,
    const int32_t* __restrict__ targets, int V, long long N, int32_t* __restrict__ slab, int32_t* status) {
  const long long t = static_cast<long long>(blockIdx.x) * kSelectThreads + threadIdx.x;
  bool bad = false;
  const int f = t < N ? select_flag(row_keep, g, gh, targets, V, t, bad) : 0;
  const int n = __syncthreads_count(f);
  const int any_bad = __syncthreads_or(bad);
  if (threadIdx.x == 0) {
    slab[blockIdx.x] = n;
    if (any_bad) atomicOr(status, MC_DEV_TARGET_RANGE);
  }
}

// Exclusive prefix sum of the slab counts, in place, in chunks of
// kSelectThreads; *count = the total.
__global__ void __launch_bounds__(kSelectThreads) select_scan_kernel(int32_t* __restrict__ slab, long long nslabs,
                                                                     int32_t* count) {
  __shared__ int warp_off[kSelectThreads / 32];
  __shared__ int chunk_total;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  int base = 0;
  for (long long s0 = 0; s0 < nslabs; s0 += kSelectThreads) {
    const long long s = s0 + tid;
    const int c = s < nslabs ? slab[s] : 0;
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    if (lane == 31) warp_off[warp] = incl;
    __syncthreads();
    if (warp == 0) {
      const int w = warp_off[lane];
      int wi = w;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, wi, o);
        if (lane >= o) wi += n;
      }
      warp_off[lane] = wi - w;
      if (lane == 31) chunk_total = wi;
    }
    __syncthreads();
    if (s < nslabs) slab[s] = base + warp_off[warp] + incl - c;
    base += chunk_total;
    __syncthreads();
  }
  if (tid == 0) *count = base;
}

__global__ void __launch_bounds__(kSelectThreads) select_write_kernel(
    const uint8_t* __restrict__ row_keep, const float* __restrict__ g, const float* __restrict__ gh,
    const int32_t* __restrict__ targets, int V, long long N, const int32_t* __restrict__ slab,
    int32_t* __restrict__ idx) {
  __shared__ int warp_off[kSelectThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const long long t = static_cast<long long>(blockIdx.x) * kSelectThreads + tid;
  bool bad = false;
  const int f = t < N ? select_flag(row_keep, g, gh, targets, V, t, bad) : 0;
  const unsigned bal = __ballot_sync(0xffffffffu, f);
  const int in_warp = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) warp_off[warp] = __popc(bal);
  __syncthreads();
  if (warp == 0) {
    const int c = warp_off[lane];
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    warp_off[lane] = incl - c;
  }
  __syncthreads();
  if (f) idx[slab[blockIdx.x] + warp_off[warp] + in_warp] = static_cast<int32_t>(t);
}

// Hc[j] = H[idx[j]] for j < count, zero rows up to the next multiple of 256
// (a whole row block of either tile height).
__global__ void gather_rows_kernel(const uint4* __restrict__ H, int row_vec, const int32_t* __restrict__ idx,
                                   const int32_t* __restrict__ count, uint4* __restrict__ Hc) {
  const long long cnt = *count;
  const long long lim = (cnt + kHcRowPad - 1) / kHcRowPad * kHcRowPad;
  for (long long j = blockIdx.x; j < lim; j += gridDim.x) {
    uint4* dst = Hc + j * row_vec;
    if (j < cnt) {
      const uint4* src = H + static_cast<long long>(idx[j]) * row_vec;
      for (int k = threadIdx.x; k < row_vec; k += blockDim.x) dst[k] = src[k];
    } else {
      for (int k = threadIdx.x; k < row_vec; k += blockDim.x) dst[k] = make_uint4(0, 0, 0, 0);
    }
  }
}

// ---------------------------------------------------------------- stage 1

struct DzParams {
  CUtensorMap tm_st;  // dz as {V, rows}, box {32 columns, 32 rows}, 64-byte swizzle: the staged stores
  const int32_t* targets;
  const float* lse;
  const float* entropy;
  const float* grad_logp;
  const float* grad_entropy;
  const int32_t* idx;  // compacted row -> original row (this chunk's slice)
  long long rows;      // rows of this chunk (host bound; the device count may be lower)
  int V;
  float scale2;
  float inv_temp;
};

// kEntropy = false when there is no entropy gradient (gH == 0 for every row):
// then dZ = -g p everywhere except the target column, which gets g (1 - p).
// H = 2 (256-row tiles only): two warp groups per 128-row sub-block, each
// draining one half of every tile's 256 columns (16 epilogue warps, more of
// them to hide TMEM-load and store latency behind each other's arithmetic;
// the 9B-class backward call ran 0.6 % faster than with 8, three interleaved
// runs with the wave gates).
template <bool kEntropy, int H = 1>
struct DzEpi {
  using Params = DzParams;
  static constexpr int kColumnHalves = H;
  static constexpr int kChunks = BN / 32 / H;  // 32-column chunks this warp drains per tile
  static constexpr int kBuffers = H == 2 ? 1 : 2;  // staging buffers per warp (see below)

  // Staged stores: each epilogue warp writes its 32 rows x 32 columns of
  // bf16 into a 2 KB shared-memory buffer in the 64-byte swizzle (row r's
  // 16-byte piece q at position q ^ ((r >> 1) & 3), conflict-free), and one
  // lane stores the box with TMA: whole lines reach L2 instead of 32
  // scattered 16-byte pieces per warp store instruction. The tensor map's
  // extent clips rows past the chunk and columns past V. Eight warps take two
  // buffers each (one fills while a store still reads the other); sixteen
  // take one each, which is what shared memory holds beside the operand ring.
  static constexpr int kStageBytes = 2048 * kBuffers;

  long long rows_lim;
  float lse2, cg, cgh, hrow;
  int y;
  int half = 0;
  bool valid;
  uint8_t* sbuf;
  uint32_t nstore;

  __device__ __forceinline__ void setup(const Params& p, long long rows_eff, bool) {
    rows_lim = rows_eff >= 0 ? rows_eff : p.rows;
    nstore = 0;
  }
  __device__ __forceinline__ void stage(uint8_t* buf) { sbuf = buf; }
  __device__ __forceinline__ void set_half(int h) { half = h; }
  // The last stores must have completed before the CTA exits.
  __device__ __forceinline__ void finish() {
    if ((threadIdx.x & 31) == 0) bulk_wait_group_all();
    __syncwarp();
  }

  __device__ __forceinline__ void begin(const Params& p, long long row, int, int) {
    valid = row < rows_lim;
    y = -1;
    lse2 = cg = cgh = hrow = 0.f;
    if (!valid) return;
    const long long o = p.idx ? p.idx[row] : row;
    y = __ldg(p.targets + o);
    cg = __ldg(p.grad_logp + o) * p.inv_temp;
    cgh = p.grad_entropy ? __ldg(p.grad_entropy + o) * p.inv_temp : 0.f;
    hrow = (p.grad_entropy && p.entropy) ? __ldg(p.entropy + o) : 0.f;
    lse2 = __ldg(p.lse + o) * kLog2e;
  }

  // Rows past the device count inside the last row block get dZ = 0, so the
  // K tail of the grad_w GEMM reads zeros.
  __device__ __forceinline__ void tile(const Params& p, long long row, int n_tile, uint32_t taddr) {
    const int v0 = n_tile * BN;
#pragma unroll 1
    for (int c = half * kChunks; c < (half + 1) * kChunks; ++c) {
      float x[32];
      tmem_ld32(taddr + c * 32, x);
      const int vc = v0 + c * 32;
      if (vc >= p.V) continue;  // the same for the whole warp
      uint32_t w[16];
      if (valid) {
        const float nl = -lse2;
        if (kEntropy) {
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
        } else {
          const float ncg = -cg;
          float dv[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) dv[i] = ncg * ex2_approx(fmaf(x[i], p.scale2, nl));
          const int rel = y - vc;
          if (rel >= 0 && rel < 32) {  // the target column of this row lies in this chunk
#pragma unroll
            for (int i = 0; i < 32; ++i) dv[i] = (i == rel) ? dv[i] + cg : dv[i];
          }
#pragma unroll
          for (int i = 0; i < 32; i += 2) w[i / 2] = pack_bf16x2(dv[i], dv[i + 1]);
        }
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) w[i] = 0u;
      }
      const int lane = threadIdx.x & 31;
      if (row - lane >= p.rows) continue;  // the warp's rows all lie past the chunk: nothing to store
      uint8_t* buf = sbuf + (nstore % kBuffers) * 2048u;
      if (lane == 0) bulk_wait_group_read<kBuffers - 1>();  // the store that last used this buffer has read it
      __syncwarp();
      uint4* r4 = reinterpret_cast<uint4*>(buf + lane * 64);
      const int sw = (lane >> 1) & 3;
#pragma unroll
      for (int q = 0; q < 4; ++q) r4[q ^ sw] = make_uint4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
      fence_proxy_async_shared();
      __syncwarp();
      if (lane == 0) {
        tma_store_2d(&p.tm_st, buf, vc, static_cast<int32_t>(row - lane));
        bulk_commit_group();
      }
      ++nstore;
    }
  }

  __device__ __forceinline__ void end(const Params&, long long, int, int, bool) {}
};

// ---------------------------------------------------------------- stages 2-3

// out[idx[row], col] = acc (bf16) for row < rows (device count), col < cols (cols % 32 == 0).
struct StoreBf16Epi {
  struct Params {
    __nv_bfloat16* out;
    const int32_t* idx;  // nullable: identity
    long long ld;
    long long rows;
    int cols;
  };
  long long rows_lim;
  __device__ __forceinline__ void setup(const Params& p, long long rows_eff, bool) {
    rows_lim = rows_eff >= 0 ? rows_eff : p.rows;
  }
  __device__ __forceinline__ void begin(const Params&, long long, int, int) {}
  __device__ __forceinline__ void tile(const Params& p, long long row, int n_tile, uint32_t taddr) {
    const int n0 = n_tile * BN;
    const long long orow = (row < rows_lim) ? (p.idx ? p.idx[row] : row) : -1;
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      float x[32];
      tmem_ld32(taddr + c * 32, x);
      const int col = n0 + c * 32;
      if (orow < 0 || col >= p.cols) continue;
      uint4* d4 = reinterpret_cast<uint4*>(p.out + orow * p.ld + col);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        __stcs(d4 + q, make_uint4(pack_bf16x2(x[8 * q + 0], x[8 * q + 1]), pack_bf16x2(x[8 * q + 2], x[8 * q + 3]),
                                  pack_bf16x2(x[8 * q + 4], x[8 * q + 5]), pack_bf16x2(x[8 * q + 6], x[8 * q + 7])));
    }
  }
  __device__ __forceinline__ void end(const Params&, long long, int, int, bool) {}
};

// out[row, col] (+)= acc (fp32), rows < p.rows, cols < p.cols (cols % 32 == 0).
// With an empty K extent the product is zero: overwrite writes zeros,
// accumulate leaves `out` as it is.
struct StoreF32Epi {
  struct Params {
    float* out;
    long long ld;
    long long rows;
    int cols;
    int accumulate;
  };
  bool kvalid;
  __device__ __forceinline__ void setup(const Params&, long long, bool k_nonempty) { kvalid = k_nonempty; }
  __device__ __forceinline__ void begin(const Params&, long long, int, int) {}
  __device__ __forceinline__ void tile(const Params& p, long long row, int n_tile, uint32_t taddr) {
    const int n0 = n_tile * BN;
#pragma unroll 1
    for (int c = 0; c < BN / 32; ++c) {
      float x[32];
      tmem_ld32(taddr + c * 32, x);
      const int col = n0 + c * 32;
      if (row >= p.rows || col >= p.cols) continue;
      if (!kvalid && p.accumulate) continue;
      float4* d4 = reinterpret_cast<float4*>(p.out + row * p.ld + col);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        float4 v = kvalid ? make_float4(x[4 * q], x[4 * q + 1], x[4 * q + 2], x[4 * q + 3])
                          : make_float4(0.f, 0.f, 0.f, 0.f);
        if (p.accumulate) {
          const float4 o = __ldcs(d4 + q);
          v.x += o.x;
          v.y += o.y;
          v.z += o.z;
          v.w += o.w;
        }
        __stcs(d4 + q, v);
      }
    }
  }
  __device__ __forceinline__ void end(const Params&, long long, int, int, bool) {}
};

template <class Epi, bool A_MN, bool B_MN, int MS = 1>
cudaError_t run_gemm(const CUtensorMap& ta, const CUtensorMap& tb, const Schedule& sch,
                     const typename Epi::Params& ep, int grid_cap, uint64_t timeout_ns, int32_t* status,
                     cudaStream_t stream) {
  auto kern = gemm_persistent<Epi, A_MN, B_MN, MS>;
  constexpr size_t smem = TileFor<Epi, MS>::template smem_bytes<Epi>();
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int units = sch.m_blocks * sch.splits;  // host upper bound; the kernel may find fewer
  const int grid = units < grid_cap ? units : grid_cap;
  if (grid <= 0) return cudaSuccess;
  // Cooperative launch with the wave gate (its counter zeroed on the stream
  // first): every CTA resident, and no CTA starts a wave before the previous
  // one has been issued in full. Measured on the 9B-class backward: 1.1 %
  // faster (283.5 against 286.8 ms, three interleaved runs).
  if (sch.wave_ctr != nullptr) {
    e = cudaMemsetAsync(sch.wave_ctr, 0, sizeof(unsigned int), stream);
    if (e != cudaSuccess) return e;
  }
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
  e = cudaLaunchKernelEx(&cfg, kern, ta, tb, sch, ep, timeout_ns, status);
  if (e != cudaSuccess) return e;
  return launched();
}

__global__ void status_merge(const int32_t* ws_status, int32_t* dev_status) {
  if (*ws_status != 0) atomicOr(dev_status, *ws_status);
}

}  // namespace

cudaError_t launch_select_gather(const SelectArgs& a, cudaStream_t stream) {
  const long long nslabs = (a.N + kSelectThreads - 1) / kSelectThreads;
  if (nslabs > 0) {
    select_count_kernel<<<static_cast<unsigned>(nslabs), kSelectThreads, 0, stream>>>(
        a.row_keep, a.grad_logp, a.grad_entropy, a.targets, a.V, a.N, a.slab, a.ws_status);
    cudaError_t e = launched();
    if (e != cudaSuccess) return e;
  }
  select_scan_kernel<<<1, kSelectThreads, 0, stream>>>(a.slab, nslabs, a.count);
  cudaError_t e = launched();
  if (e != cudaSuccess) return e;
  if (nslabs > 0) {
    select_write_kernel<<<static_cast<unsigned>(nslabs), kSelectThreads, 0, stream>>>(
        a.row_keep, a.grad_logp, a.grad_entropy, a.targets, a.V, a.N, a.slab, a.idx);
    e = launched();
    if (e != cudaSuccess) return e;
  }
  const int row_vec = a.d * 2 / 16;
  gather_rows_kernel<<<a.grid, 256, 0, stream>>>(static_cast<const uint4*>(a.hidden), row_vec, a.idx, a.count,
                                                 static_cast<uint4*>(a.hc));
  return launched();
}

cudaError_t launch_dz(const DzArgs& a, cudaStream_t stream) {
  Schedule sch;
  const int rb = a.wide ? 2 * BM : BM;
  sch.m_blocks = static_cast<int>((a.rows + rb - 1) / rb);
  sch.n_tiles = (a.V + BN - 1) / BN;
  sch.splits = a.splits;
  sch.k_blocks = a.d / BK;
  sch.dyn_count = a.count;
  sch.dyn_offset = a.row_offset;
  sch.dyn_cap = a.rows;
  sch.dyn_mode = DYN_ROWS;
  sch.wave_ctr = a.wave_ctr;
  DzParams ep;
  ep.targets = a.targets;
  ep.lse = a.lse;
  ep.entropy = a.entropy;
  ep.grad_logp = a.grad_logp;
  ep.grad_entropy = a.grad_entropy;
  ep.idx = a.idx;
  ep.rows = a.rows;
  ep.V = a.V;
  ep.scale2 = a.inv_temperature * kLog2e;
  ep.inv_temp = a.inv_temperature;
  ep.tm_st = a.tm_dz_st;
  if (a.wide) {
    if (a.grad_entropy != nullptr)
      return run_gemm<DzEpi<true, 2>, false, false, 2>(a.tm_hidden, a.tm_w, sch, ep, a.grid, a.timeout_ns,
                                                    a.ws_status, stream);
    return run_gemm<DzEpi<false, 2>, false, false, 2>(a.tm_hidden, a.tm_w, sch, ep, a.grid, a.timeout_ns,
                                                   a.ws_status, stream);
  }
  if (a.grad_entropy != nullptr)
    return run_gemm<DzEpi<true>, false, false>(a.tm_hidden, a.tm_w, sch, ep, a.grid, a.timeout_ns, a.ws_status,
                                               stream);
  return run_gemm<DzEpi<false>, false, false>(a.tm_hidden, a.tm_w, sch, ep, a.grid, a.timeout_ns, a.ws_status,
                                              stream);
}

// Tiles per group for a one-tile-per-unit long-K GEMM whose waves hold `conc`
// units: the divisor b of n_tiles that minimises the operand extent one wave
// streams, rb * conc / b (A rows) + BN * b (B columns), among those whose wave
// still spans conc / b <= m_blocks row blocks. 0 = ungrouped.
static int tile_group(int n_tiles, long long m_blocks, int conc, int rb) {
  int best = 0;
  double best_cost = double(rb) * conc / n_tiles + double(BN) * n_tiles;
  for (int b = 1; b < n_tiles; ++b) {
    if (n_tiles % b != 0 || static_cast<long long>(conc / b) > m_blocks) continue;
    const double cost = double(rb) * conc / b + double(BN) * b;
    if (cost < best_cost) {
      best_cost = cost;
      best = b;
    }
  }
  return best;
}

// K extent (in BK blocks) from which grad_hidden / grad_w use the wide
// 256-row tile: measured on the 9B-class shapes, grad_w (K = kept rows) runs
// ~2 % faster on it at K = 4,096 and 4-9 % faster at 6,144-12,288; its
// un-overlapped epilogue stays small next to a K loop of 64+ blocks.
constexpr int kWideMinKBlocks = 64;

cudaError_t launch_dh(const DhArgs& a, cudaStream_t stream) {
  Schedule sch;
  sch.k_blocks = (a.V + BK - 1) / BK;
  const bool wide = sch.k_blocks >= kWideMinKBlocks;
  const int rb = wide ? 2 * BM : BM;
  sch.m_blocks = static_cast<int>((a.rows + rb - 1) / rb);
  sch.n_tiles = (a.d + BN - 1) / BN;
  sch.splits = sch.n_tiles;  // one output tile per unit
  sch.n_group = tile_group(sch.n_tiles, sch.m_blocks, a.grid, rb);
  sch.dyn_count = a.count;
  sch.dyn_offset = a.row_offset;
  sch.dyn_cap = a.rows;
  sch.dyn_mode = DYN_ROWS;
  sch.wave_ctr = a.wave_ctr;
  StoreBf16Epi::Params ep;
  ep.out = static_cast<__nv_bfloat16*>(a.grad_hidden);
  ep.idx = a.idx;
  ep.ld = a.d;
  ep.rows = a.rows;
  ep.cols = a.d;
  if (wide)
    return run_gemm<StoreBf16Epi, false, true, 2>(a.tm_dz, a.tm_w_mn, sch, ep, a.grid, a.timeout_ns,
                                                  a.ws_status, stream);
  return run_gemm<StoreBf16Epi, false, true>(a.tm_dz, a.tm_w_mn, sch, ep, a.grid, a.timeout_ns, a.ws_status,
                                             stream);
}

cudaError_t launch_dw(const DwArgs& a, cudaStream_t stream) {
  Schedule sch;
  sch.k_blocks = static_cast<int>((a.rows + BK - 1) / BK);  // host bound; the kernel reads the count
  const bool wide = sch.k_blocks >= kWideMinKBlocks;
  const int rb = wide ? 2 * BM : BM;
  sch.m_blocks = (a.V + rb - 1) / rb;
  sch.n_tiles = (a.d + BN - 1) / BN;
  sch.splits = sch.n_tiles;
  sch.n_group = tile_group(sch.n_tiles, sch.m_blocks, a.grid, rb);
  sch.dyn_count = a.count;
  sch.dyn_offset = a.row_offset;
  sch.dyn_cap = a.rows;
  sch.dyn_mode = DYN_K;
  sch.wave_ctr = a.wave_ctr;
  StoreF32Epi::Params ep;
  ep.out = a.grad_w;
  ep.ld = a.d;
  ep.rows = a.V;
  ep.cols = a.d;
  ep.accumulate = a.accumulate;
  if (wide)
    return run_gemm<StoreF32Epi, true, true, 2>(a.tm_dz_mn, a.tm_h_mn, sch, ep, a.grid, a.timeout_ns,
                                                a.ws_status, stream);
  return run_gemm<StoreF32Epi, true, true>(a.tm_dz_mn, a.tm_h_mn, sch, ep, a.grid, a.timeout_ns, a.ws_status,
                                           stream);
}

cudaError_t launch_status_merge(const int32_t* ws_status, int32_t* dev_status, cudaStream_t stream) {
  if (dev_status == nullptr) return cudaSuccess;
  status_merge<<<1, 1, 0, stream>>>(ws_status, dev_status);
  return launched();
}

}  // namespace mc
