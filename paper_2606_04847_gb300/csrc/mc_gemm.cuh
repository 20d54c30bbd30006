// mc_gemm.cuh — persistent warp-specialised tcgen05 GEMM engine for sm_103a.
//
// C[m, n] = sum_k A[m, k] B[n, k], bf16 operands, fp32 accumulation in TMEM.
// The accumulator tile (128 x 256, or 256 x 256 with MS = 2) is handed to an
// epilogue functor and never written to memory by the engine itself: the
// forward turns it into an online log-sum-exp / entropy update, the backward
// into dZ, the backward GEMMs into plain stores.
//
// CTA = 2 + 4 * MS * H warps, one CTA per SM (the SMEM ring takes 192 KB, plus
// the epilogue's own staging buffers when it asks for them):
//   warp 0        TMA producer: loads A/B k-blocks (BK = 64) into the ring
//                 (4 x 48 KB stages; 3 x 64 KB with MS = 2)
//   warp 1        TMEM allocator + MMA issuer (one thread): 4 x MS
//                 tcgen05.mma (M=128, N=256, K=16) per k-block into TMEM
//                 (2 x 256 fp32 columns = all 512 columns)
//   warps 2..     epilogue (4 warps per 128-row sub-block, or per sub-block
//                 and column half when the epilogue asks for H = 2 halves):
//                 warp w reads TMEM lanes 32*(w%4)..+31 of its sub-block, one
//                 output row per thread, 32 columns per tcgen05.ld
// With MS = 1 the two 256-column accumulators let the epilogue of tile j
// overlap the MMAs of tile j+1; with MS = 2 they hold the two 128-row halves
// of one 256 x 256 tile (see TileCfg). Barriers: full[s]/empty[s] per ring
// stage, tfull[a]/tempty[a] per accumulator slot. Every wait is bounded
// (mbar_wait), and on the way out each role drains what it has in flight (TMA
// loads, MMAs, the epilogue's TMA stores) before TMEM is freed.
//
// Work decomposition: the M dimension is cut into row blocks, the N
// dimension into BN-column tiles, and the tiles of one row block into
// `splits` contiguous ranges. A unit = (row block, range). Units are dealt
// round-robin to the persistent CTAs (unit u -> CTA u % gridDim.x), so the
// CTAs running at the same time share a few row blocks (A stays in L2) and
// sweep the same B tiles together (B is read from HBM about once per wave).
// The library launches every GEMM cooperatively with a wave gate
// (Schedule::wave_ctr) that keeps the waves in step.
// Within a unit the tiles run in order, so an epilogue can carry per-row
// state across them (the forward's online softmax).
//
// Operand layouts: A is [M, K] K-major (A_MN = false) or [K, M] M-major
// (A_MN = true); B is [N, K] K-major or [K, N] N-major. All tiles use the
// 128-byte swizzle; TMA boxes are 64 elements (128 B) wide in the contiguous
// dimension. K-major A: one box {64 k, 128 m} per sub-block; M-major A: two
// boxes {64 m, 64 k} per sub-block; K-major B: one box {64 k, 256 n}; N-major
// B: four boxes {64 n, 64 k}. Out-of-range rows/columns are zero-filled by
// TMA.
#pragma once

#include <type_traits>

#include "mc_ptx.cuh"

namespace mc {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;
constexpr int UMMA_K = 16;
constexpr int NUM_STAGES = 4;
constexpr int NUM_ACC = 2;
constexpr int TMEM_COLS = NUM_ACC * BN;  // 512
constexpr int A_STAGE_BYTES = BM * BK * 2;  // 16 KB
constexpr int B_STAGE_BYTES = BN * BK * 2;  // 32 KB
constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
constexpr int GEMM_THREADS = 192;
constexpr int EPI_WARP_BEGIN = 2;
constexpr int NUM_EPI_WARPS = 4;
constexpr int MN_BOX_BYTES = 64 * 64 * 2;  // one {64, 64} bf16 box = 8 KB

struct GemmShared {
  uint64_t full[NUM_STAGES];
  uint64_t empty[NUM_STAGES];
  uint64_t tfull[NUM_ACC];
  uint64_t tempty[NUM_ACC];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

constexpr size_t GEMM_SMEM_BYTES = size_t(NUM_STAGES) * STAGE_BYTES + sizeof(GemmShared) + 1024;

// Epilogues may ask for shared memory of their own: `static constexpr int
// kStageBytes` per epilogue warp (1024-byte aligned). The engine then calls
// `epi.stage(buffer)` after setup and `epi.finish()` after the last unit.
template <class E, class = void>
struct EpiStage {
  static constexpr int bytes = 0;
};
template <class E>
struct EpiStage<E, std::void_t<decltype(E::kStageBytes)>> {
  static constexpr int bytes = E::kStageBytes;
};
constexpr size_t kEpiStageOffset = (size_t(NUM_STAGES) * STAGE_BYTES + sizeof(GemmShared) + 1023) / 1024 * 1024;

// Epilogues may also ask, through `static constexpr int kColumnHalves = 2`,
// for two warp groups per 128-row sub-block of a 256-row tile, each draining
// half of the tile's 256 columns (16 epilogue warps: twice the warps hiding
// TMEM-load and arithmetic latency while the MMAs wait for the drain). The
// engine then calls `epi.set_half(h)` once, h = the warp's column half. Their
// staging buffers (kStageBytes each) must fit beside the operand ring.
template <class E, class = void>
struct EpiColumnHalves {
  static constexpr int value = 1;
};
template <class E>
struct EpiColumnHalves<E, std::void_t<decltype(E::kColumnHalves)>> {
  static constexpr int value = E::kColumnHalves;
};

enum DynMode : int { DYN_NONE = 0, DYN_ROWS = 1, DYN_K = 2 };

struct Schedule {
  int m_blocks;  // ceil(M / BM)
  int n_tiles;   // ceil(N / BN)
  int splits;    // tile ranges per row block, 1 <= splits <= n_tiles
  int k_blocks;  // ceil(K / BK)
  // Optional extent known only on the device (a count written by an earlier
  // kernel on the stream): c = clamp(*dyn_count - dyn_offset, 0, dyn_cap)
  // replaces M (DYN_ROWS: m_blocks = ceil(c / BM)) or K (DYN_K).
  const int32_t* dyn_count = nullptr;
  long long dyn_offset = 0;
  long long dyn_cap = 0;
  int dyn_mode = DYN_NONE;
  // One-tile units only (splits == n_tiles): when 0 < n_group < n_tiles and
  // n_group divides n_tiles, units are ordered (tile group, row block, tile in
  // group), so the CTAs running at once cover ~grid/n_group row blocks x
  // n_group tiles instead of ~grid/n_tiles x all tiles. A long-K GEMM re-reads
  // both operands once per wave; this shape reads fewer bytes per wave.
  int n_group = 0;
  // Optional wave gate (a counter that is zero at launch; the launch must be
  // cooperative, so that every CTA is resident). Each CTA's producer raises
  // it after issuing a unit's loads and, before its k-th unit (k >= 1), waits
  // until min(k * gridDim.x, units) units have been issued: no CTA starts a
  // wave before every CTA has finished the one before. The CTAs that share a
  // unit's B tiles then read each tile within a few tiles of one another, and
  // the tile is still in L2 for all of them; without the gate they drift
  // apart over many waves and re-read B from HBM.
  unsigned int* wave_ctr = nullptr;

  __device__ __forceinline__ int units() const { return m_blocks * splits; }
  __device__ __forceinline__ void unit(int u, int& mb, int& split, int& t0, int& t1) const {
    if (n_group > 0) {
      const int per = m_blocks * n_group;
      const int g = u / per;
      const int r = u - g * per;
      mb = r / n_group;
      split = g * n_group + (r - mb * n_group);
      t0 = split;
      t1 = split + 1;
      return;
    }
    mb = u / splits;
    split = u - mb * splits;
    t0 = static_cast<int>((static_cast<long long>(split) * n_tiles) / splits);
    t1 = static_cast<int>((static_cast<long long>(split + 1) * n_tiles) / splits);
  }
};

// Epilogue functor contract (one instance per epilogue thread):
//   struct Epi {
//     struct Params;
//     __device__ void setup(const Params&, long long rows_eff, bool k_nonempty);
//     __device__ void begin(const Params&, long long row, int mb, int split);
//     __device__ void tile(const Params&, long long row, int n_tile, uint32_t taddr);
//     __device__ void end(const Params&, long long row, int mb, int split, bool ok);
//   };
// `row` = global M index of the thread's row (may be >= M: padding rows),
// `taddr` = TMEM address of the thread's warp's lane quadrant, column 0 of the
// accumulator holding tile `n_tile`. `ok` is false when the pipeline gave up.
// `rows_eff` is the device-side row count under DYN_ROWS (else -1);
// `k_nonempty` is false when a DYN_K extent is 0 (the accumulator is then
// never written and must be read as zero).

// MS = row sub-blocks per tile. MS = 1: 128 x 256 tiles, 4 x 48 KB stages,
// two tiles in flight in TMEM (the epilogue of one overlaps the MMAs of the
// next). MS = 2 ("wide"): 256 x 256 tiles computed as two M = 128 MMAs that
// share each B stage, 3 x 64 KB stages, both TMEM accumulators on the one
// tile in flight, and 8 epilogue warps that drain the two halves at once (16
// when the epilogue asks for H = 2 column halves). A
// wide tile streams ~29 % fewer operand bytes per output from HBM and a third
// fewer from L2, and its ring covers longer operand latency; the epilogue no
// longer overlaps the MMAs, which costs a GEMM little when its K loop is long
// or its epilogue short. Unit row blocks are then 256 rows.
template <int MS, int H = 1>
struct TileCfg {
  static_assert(MS == 1 || MS == 2, "one or two 128-row sub-blocks");
  static_assert(H == 1 || (H == 2 && MS == 2), "column halves only with 256-row tiles");
  static constexpr int TBM = BM * MS;
  static constexpr int STAGES = MS == 1 ? NUM_STAGES : 3;
  static constexpr int SBYTES = MS * A_STAGE_BYTES + B_STAGE_BYTES;
  static constexpr int SLOTS = NUM_ACC / MS;  // tiles in flight in TMEM
  static constexpr int HALVES = H;            // warp groups per sub-block (column halves)
  static constexpr int EPI_WARPS = NUM_EPI_WARPS * MS * H;  // 4 per 128-row sub-block and column half
  static constexpr int THREADS = 32 * (EPI_WARP_BEGIN + EPI_WARPS);
  // Dynamic shared memory of the kernel running epilogue E.
  template <class E>
  static constexpr size_t smem_bytes() {
    return EpiStage<E>::bytes > 0 ? kEpiStageOffset + size_t(EPI_WARPS) * EpiStage<E>::bytes + 1024
                                  : GEMM_SMEM_BYTES;
  }
  static_assert(STAGES * SBYTES <= NUM_STAGES * STAGE_BYTES, "ring exceeds the SMEM budget");
  static_assert(STAGES <= NUM_STAGES && SLOTS >= 1, "barrier arrays are sized for the narrow tile");
};

// The tile configuration a kernel with epilogue E and MS sub-blocks runs:
// E's column halves apply to 256-row tiles only.
template <class E, int MS>
using TileFor = TileCfg<MS, (MS == 2 ? EpiColumnHalves<E>::value : 1)>;

template <class Epi, bool A_MN, bool B_MN, int MS = 1>
__global__ void __launch_bounds__(TileFor<Epi, MS>::THREADS, 1)
    gemm_persistent(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const Schedule sch_in, const __grid_constant__ typename Epi::Params ep,
                    const uint64_t timeout_ns, int32_t* dev_status) {
  using C = TileFor<Epi, MS>;
  static_assert(C::template smem_bytes<Epi>() <= 227 * 1024, "shared memory of one CTA exceeded");
  Schedule sch = sch_in;
  long long rows_eff = -1;
  bool k_nonempty = true;
  if (sch.dyn_count != nullptr) {
    long long c = static_cast<long long>(*sch.dyn_count) - sch.dyn_offset;
    c = c < 0 ? 0 : (c > sch.dyn_cap ? sch.dyn_cap : c);
    if (sch.dyn_mode == DYN_ROWS) {
      sch.m_blocks = static_cast<int>((c + C::TBM - 1) / C::TBM);
      rows_eff = c;
    } else if (sch.dyn_mode == DYN_K) {
      sch.k_blocks = static_cast<int>((c + BK - 1) / BK);
      k_nonempty = sch.k_blocks > 0;
    }
  }
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  GemmShared* sh = reinterpret_cast<GemmShared*>(smem + NUM_STAGES * STAGE_BYTES);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
#pragma unroll
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&sh->full[s], 1);
      mbar_init(&sh->empty[s], 1);
    }
#pragma unroll
    for (int a = 0; a < C::SLOTS; ++a) {
      mbar_init(&sh->tfull[a], 1);
      mbar_init(&sh->tempty[a], C::EPI_WARPS);
    }
    mbar_init(&sh->drain, 1);
    sh->abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(&sh->tmem_base, TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sh->tmem_base;
  volatile int* abort = &sh->abort;
  const int n_units = sch.units();

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      uint32_t it = 0;
      bool ok = true;
      for (int u = blockIdx.x, wave = 0; u < n_units && ok; u += gridDim.x, ++wave) {
        if (sch.wave_ctr != nullptr && wave > 0) {
          const unsigned need = min(static_cast<unsigned>(wave) * gridDim.x, static_cast<unsigned>(n_units));
          if (!counter_wait_geq(sch.wave_ctr, need, abort, timeout_ns, dev_status)) {
            ok = false;
            break;
          }
        }
        int mb, split, t0, t1;
        sch.unit(u, mb, split, t0, t1);
        const int row0 = mb * C::TBM;
        for (int t = t0; t < t1 && ok; ++t) {
          for (int kb = 0; kb < sch.k_blocks; ++kb) {
            const int s = static_cast<int>(it % C::STAGES);
            const uint32_t ph = (it / C::STAGES) & 1u;
            if (!mbar_wait(&sh->empty[s], ph ^ 1u, abort, timeout_ns, dev_status)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&sh->full[s], C::SBYTES);
            uint8_t* a = smem + s * C::SBYTES;
            uint8_t* b = a + MS * A_STAGE_BYTES;
            // Sub-block j of A lands at a + j * A_STAGE_BYTES in both layouts.
            if (!A_MN) {
#pragma unroll
              for (int j = 0; j < MS; ++j)
                tma_load_2d(a + j * A_STAGE_BYTES, &tmA, &sh->full[s], kb * BK, row0 + j * BM);
            } else {
#pragma unroll
              for (int j = 0; j < C::TBM / 64; ++j)
                tma_load_2d(a + j * MN_BOX_BYTES, &tmA, &sh->full[s], row0 + j * 64, kb * BK);
            }
            if (!B_MN) {
              tma_load_2d(b, &tmB, &sh->full[s], kb * BK, t * BN);
            } else {
#pragma unroll
              for (int j = 0; j < BN / 64; ++j)
                tma_load_2d(b + j * MN_BOX_BYTES, &tmB, &sh->full[s], t * BN + j * 64, kb * BK);
            }
            ++it;
          }
        }
        if (sch.wave_ctr != nullptr && ok) atomicAdd(sch.wave_ctr, 1u);
      }
      // Let every load this thread issued land before the CTA can exit.
      const uint32_t last = it < C::STAGES ? it : C::STAGES;
      for (uint32_t j = it - last; j < it; ++j)
        mbar_wait(&sh->full[j % C::STAGES], (j / C::STAGES) & 1u, nullptr, timeout_ns, dev_status);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN, A_MN, B_MN);
      uint32_t it = 0, tc = 0;
      bool ok = true;
      for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
        int mb, split, t0, t1;
        sch.unit(u, mb, split, t0, t1);
        for (int t = t0; t < t1 && ok; ++t) {
          const uint32_t acc = tc % C::SLOTS;
          const uint32_t aph = (tc / C::SLOTS) & 1u;
          if (!mbar_wait(&sh->tempty[acc], aph ^ 1u, abort, timeout_ns, dev_status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem + acc * (MS * BN);
          for (int kb = 0; kb < sch.k_blocks; ++kb) {
            const int s = static_cast<int>(it % C::STAGES);
            const uint32_t ph = (it / C::STAGES) & 1u;
            if (!mbar_wait(&sh->full[s], ph, abort, timeout_ns, dev_status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a_addr = smem_u32(smem + s * C::SBYTES);
            const uint32_t b_addr = a_addr + MS * A_STAGE_BYTES;
#pragma unroll
            for (int k = 0; k < BK / UMMA_K; ++k) {
              const uint64_t bdesc = B_MN ? smem_desc_sw128(b_addr + k * (UMMA_K * 128), MN_BOX_BYTES, 1024)
                                          : smem_desc_sw128(b_addr + k * (UMMA_K * 2), 16, 1024);
#pragma unroll
              for (int j = 0; j < MS; ++j) {
                const uint32_t aj = a_addr + j * A_STAGE_BYTES;
                const uint64_t adesc = A_MN ? smem_desc_sw128(aj + k * (UMMA_K * 128), MN_BOX_BYTES, 1024)
                                            : smem_desc_sw128(aj + k * (UMMA_K * 2), 16, 1024);
                umma_bf16(d_tmem + j * BN, adesc, bdesc, IDESC, (kb | k) != 0 ? 1u : 0u);
              }
            }
            umma_commit(&sh->empty[s]);  // frees the stage once these MMAs have read it
            ++it;
          }
          if (!ok) break;
          umma_commit(&sh->tfull[acc]);  // accumulator(s) ready for the epilogue
          ++tc;
        }
      }
      // No MMA may still be writing TMEM when it is freed.
      umma_commit(&sh->drain);
      mbar_wait(&sh->drain, 0, nullptr, timeout_ns, dev_status);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    // Warps 2.. in groups of four, group g draining row sub-block g % MS
    // (and, with two column halves, columns [128 h, 128 h + 128) of it,
    // h = g / MS); within a group, warp w may access TMEM lane quadrant w % 4
    // only.
    const int group = (warp - EPI_WARP_BEGIN) / NUM_EPI_WARPS;
    const int sub = group % MS;
    const int quad = warp & 3;
    const int row_in_tile = sub * BM + quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t tc = 0;
    Epi epi;
    epi.setup(ep, rows_eff, k_nonempty);
    if constexpr (EpiStage<Epi>::bytes > 0)
      epi.stage(smem + kEpiStageOffset + (warp - EPI_WARP_BEGIN) * EpiStage<Epi>::bytes);
    if constexpr (C::HALVES > 1) epi.set_half(group / MS);
    bool ok = true;
    for (int u = blockIdx.x; u < n_units && ok; u += gridDim.x) {
      int mb, split, t0, t1;
      sch.unit(u, mb, split, t0, t1);
      const long long row = static_cast<long long>(mb) * C::TBM + row_in_tile;
      epi.begin(ep, row, mb, split);
      for (int t = t0; t < t1; ++t) {
        const uint32_t acc = tc % C::SLOTS;
        const uint32_t aph = (tc / C::SLOTS) & 1u;
        // Every lane polls; the warp proceeds only if all lanes saw the phase
        // complete, so the warp-collective tcgen05.ld below stays converged.
        const bool got = mbar_wait(&sh->tfull[acc], aph, abort, timeout_ns, dev_status);
        if (!__all_sync(0xffffffffu, got)) {
          ok = false;
          break;
        }
        tc_fence_after();
        epi.tile(ep, row, t, tmem + (acc * MS + sub) * BN + lane_off);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&sh->tempty[acc]);
        ++tc;
      }
      epi.end(ep, row, mb, split, ok);
    }
    if constexpr (EpiStage<Epi>::bytes > 0) epi.finish();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
}

}  // namespace mc
