// mc_gemm2.cuh — the persistent tcgen05 GEMM engine on CTA pairs (cta_group::2).
//
// Same contract as mc_gemm.cuh (Schedule, epilogue functors, bounded waits),
// but two CTAs of a cluster compute one 256 x 256 output tile together:
//   * CTA rank r (r = 0, 1) loads rows [128 r, 128 r + 128) of the tile's A
//     operand and columns [128 r, 128 r + 128) of its B operand into its own
//     shared memory: 16 + 16 KB per 64-deep k-block instead of 16 + 32 KB, so
//     each SM pulls a third less data from L2 per FLOP and the ring holds six
//     stages instead of four (more latency hidden);
//   * the leader (rank 0) issues tcgen05.mma.cta_group::2 (M = 256, N = 256,
//     K = 16), which reads A and B from both CTAs and accumulates rows
//     [128 r, 128 r + 128) into CTA r's TMEM;
//   * each CTA's epilogue warps read their own TMEM, exactly as in the
//     one-CTA engine, so the epilogue functors are shared.
// Barriers: full[s] lives in the leader and counts both CTAs' TMA bytes (the
// peer's loads signal it across the pair); empty[s] and tfull[a] live in both
// CTAs and receive the leader's multicast commits; tempty[a] lives in the
// leader and collects the four epilogue warps of each CTA (the peer's arrive
// remotely). A wait that gives up raises the abort word of both CTAs.
// Every pipeline wait is bounded; the only unbounded waits are the two
// cluster barriers at kernel start and end, which every thread reaches
// unconditionally.
#pragma once

#include "mc_gemm.cuh"
#include "mc_internal.h"

namespace mc {

constexpr int PAIR_BM = 256;  // rows per pair tile (128 per CTA)
constexpr int PAIR_STAGES = 6;
constexpr int PAIR_A_BYTES = 128 * BK * 2;  // 16 KB
constexpr int PAIR_B_BYTES = 128 * BK * 2;  // 16 KB: this CTA's half of BN
constexpr int PAIR_STAGE_BYTES = PAIR_A_BYTES + PAIR_B_BYTES;

struct PairShared {
  uint64_t full[PAIR_STAGES];
  uint64_t empty[PAIR_STAGES];
  uint64_t tfull[NUM_ACC];
  uint64_t tempty[NUM_ACC];
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
};

// A 16 KB guard after the ring: even a descriptor read of a full 256-row
// operand tile from the last stage stays inside this CTA's shared memory.
constexpr int PAIR_GUARD_BYTES = 16 * 1024;
constexpr size_t GEMM2_SMEM_BYTES =
    size_t(PAIR_STAGES) * PAIR_STAGE_BYTES + PAIR_GUARD_BYTES + sizeof(PairShared) + 1024;

// Schedule.m_blocks counts 256-row pair blocks here; DYN_ROWS divides the
// device-side row count by 256.
template <class Epi, bool A_MN, bool B_MN>
__global__ void __launch_bounds__(GEMM_THREADS, 1)
    gemm_pair(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
              const Schedule sch_in, const typename Epi::Params ep, const uint64_t timeout_ns,
              int32_t* dev_status) {
  Schedule sch = sch_in;
  long long rows_eff = -1;
  bool k_nonempty = true;
  if (sch.dyn_count != nullptr) {
    long long c = static_cast<long long>(*sch.dyn_count) - sch.dyn_offset;
    c = c < 0 ? 0 : (c > sch.dyn_cap ? sch.dyn_cap : c);
    if (sch.dyn_mode == DYN_ROWS) {
      sch.m_blocks = static_cast<int>((c + PAIR_BM - 1) / PAIR_BM);
      rows_eff = c;
    } else if (sch.dyn_mode == DYN_K) {
      sch.k_blocks = static_cast<int>((c + BK - 1) / BK);
      k_nonempty = sch.k_blocks > 0;
    }
  }
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  PairShared* sh = reinterpret_cast<PairShared*>(smem + PAIR_STAGES * PAIR_STAGE_BYTES + PAIR_GUARD_BYTES);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int cluster = static_cast<int>(blockIdx.x >> 1);
  const int n_clusters = static_cast<int>(gridDim.x >> 1);

  if (threadIdx.x == 0) {
#pragma unroll
    for (int s = 0; s < PAIR_STAGES; ++s) {
      mbar_init(&sh->full[s], 1);
      mbar_init(&sh->empty[s], 1);
    }
#pragma unroll
    for (int a = 0; a < NUM_ACC; ++a) {
      mbar_init(&sh->tfull[a], 1);
      mbar_init(&sh->tempty[a], 2 * NUM_EPI_WARPS);
    }
    mbar_init(&sh->drain, 1);
    sh->abort = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc_pair(&sh->tmem_base, TMEM_COLS);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers exist before either signals the other
  tc_fence_after();
  const uint32_t tmem = sh->tmem_base;
  volatile int* abort = &sh->abort;
  const uint32_t peer_abort = mapa_shared(smem_u32(&sh->abort), rank ^ 1u);
  const int n_units = sch.units();

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer (both CTAs)
    if (lane == 0) {
      tma_prefetch_desc(&tmA);
      tma_prefetch_desc(&tmB);
      uint32_t it = 0;
      bool ok = true;
      for (int u = cluster; u < n_units && ok; u += n_clusters) {
        int mb, split, t0, t1;
        sch.unit(u, mb, split, t0, t1);
        const int row0 = mb * PAIR_BM + static_cast<int>(rank) * 128;
        for (int t = t0; t < t1 && ok; ++t) {
          const int n0 = t * BN + static_cast<int>(rank) * 128;
          for (int kb = 0; kb < sch.k_blocks; ++kb) {
            const int s = static_cast<int>(it % PAIR_STAGES);
            const uint32_t ph = (it / PAIR_STAGES) & 1u;
            if (!mbar_wait_pair(&sh->empty[s], ph ^ 1u, abort, peer_abort, timeout_ns, dev_status)) {
              ok = false;
              break;
            }
            if (leader) mbar_arrive_expect_tx(&sh->full[s], 2 * PAIR_STAGE_BYTES);
            const uint32_t full_leader = mapa_shared(smem_u32(&sh->full[s]), 0u);
            uint8_t* a = smem + s * PAIR_STAGE_BYTES;
            uint8_t* b = a + PAIR_A_BYTES;
            if (!A_MN) {
              tma_load_2d_pair(a, &tmA, full_leader, kb * BK, row0);
            } else {
#pragma unroll
              for (int j = 0; j < 2; ++j)
                tma_load_2d_pair(a + j * MN_BOX_BYTES, &tmA, full_leader, row0 + j * 64, kb * BK);
            }
            if (!B_MN) {
              tma_load_2d_pair(b, &tmB, full_leader, kb * BK, n0);
            } else {
#pragma unroll
              for (int j = 0; j < 2; ++j)
                tma_load_2d_pair(b + j * MN_BOX_BYTES, &tmB, full_leader, n0 + j * 64, kb * BK);
            }
            ++it;
          }
        }
      }
      // The leader's full barriers count both CTAs' bytes: it waits for every
      // load of the pair to land (the peer then leaves only after the final
      // cluster barrier, i.e. after this drain).
      if (leader) {
        const uint32_t last = it < PAIR_STAGES ? it : PAIR_STAGES;
        for (uint32_t j = it - last; j < it; ++j)
          mbar_wait(&sh->full[j % PAIR_STAGES], (j / PAIR_STAGES) & 1u, nullptr, timeout_ns, dev_status);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (leader only)
    if (lane == 0 && leader) {
      constexpr uint32_t IDESC = idesc_bf16_f32(PAIR_BM, BN, A_MN, B_MN);
      uint32_t it = 0, tc = 0;
      bool ok = true;
      for (int u = cluster; u < n_units && ok; u += n_clusters) {
        int mb, split, t0, t1;
        sch.unit(u, mb, split, t0, t1);
        for (int t = t0; t < t1 && ok; ++t) {
          const uint32_t acc = tc & 1u;
          const uint32_t aph = (tc >> 1) & 1u;
          if (!mbar_wait_pair(&sh->tempty[acc], aph ^ 1u, abort, peer_abort, timeout_ns, dev_status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem + acc * BN;
          for (int kb = 0; kb < sch.k_blocks; ++kb) {
            const int s = static_cast<int>(it % PAIR_STAGES);
            const uint32_t ph = (it / PAIR_STAGES) & 1u;
            if (!mbar_wait_pair(&sh->full[s], ph, abort, peer_abort, timeout_ns, dev_status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a_addr = smem_u32(smem + s * PAIR_STAGE_BYTES);
            const uint32_t b_addr = a_addr + PAIR_A_BYTES;
#pragma unroll
            for (int k = 0; k < BK / UMMA_K; ++k) {
              const uint64_t adesc = A_MN ? smem_desc_sw128(a_addr + k * (UMMA_K * 128), MN_BOX_BYTES, 1024)
                                          : smem_desc_sw128(a_addr + k * (UMMA_K * 2), 16, 1024);
              const uint64_t bdesc = B_MN ? smem_desc_sw128(b_addr + k * (UMMA_K * 128), MN_BOX_BYTES, 1024)
                                          : smem_desc_sw128(b_addr + k * (UMMA_K * 2), 16, 1024);
              umma_bf16_pair(d_tmem, adesc, bdesc, IDESC, (kb | k) != 0 ? 1u : 0u);
            }
            umma_commit_pair(&sh->empty[s], 0x3);  // frees stage s in both CTAs
            ++it;
          }
          if (!ok) break;
          umma_commit_pair(&sh->tfull[acc], 0x3);  // both halves of the tile are ready
          ++tc;
        }
      }
      umma_commit_pair(&sh->drain, 0x1);
      mbar_wait(&sh->drain, 0, nullptr, timeout_ns, dev_status);
    }
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs)
    const int quad = warp & 3;
    const int row_in_pair = static_cast<int>(rank) * 128 + quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    uint32_t tc = 0;
    Epi epi;
    epi.setup(ep, rows_eff, k_nonempty);
    bool ok = true;
    for (int u = cluster; u < n_units && ok; u += n_clusters) {
      int mb, split, t0, t1;
      sch.unit(u, mb, split, t0, t1);
      const long long row = static_cast<long long>(mb) * PAIR_BM + row_in_pair;
      epi.begin(ep, row, mb, split);
      for (int t = t0; t < t1; ++t) {
        const uint32_t acc = tc & 1u;
        const uint32_t aph = (tc >> 1) & 1u;
        const bool got = mbar_wait_pair(&sh->tfull[acc], aph, abort, peer_abort, timeout_ns, dev_status);
        if (!__all_sync(0xffffffffu, got)) {
          ok = false;
          break;
        }
        tc_fence_after();
        epi.tile(ep, row, t, tmem + acc * BN + lane_off);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (leader)
            mbar_arrive(&sh->tempty[acc]);
          else
            mbar_arrive_cluster(mapa_shared(smem_u32(&sh->tempty[acc]), 0u));
        }
        ++tc;
      }
      epi.end(ep, row, mb, split, ok);
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // no CTA leaves while its peer may still touch its shared memory
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc_pair(tmem, TMEM_COLS);
  }
}

}  // namespace mc

namespace mc {

// Launches the pair engine as 2-CTA clusters: as many clusters as can be
// resident at once (persistent), never more than there are units.
template <class Epi, bool A_MN, bool B_MN>
cudaError_t run_gemm_pair(const CUtensorMap& ta, const CUtensorMap& tb, const Schedule& sch,
                          const typename Epi::Params& ep, uint64_t timeout_ns, int32_t* status,
                          cudaStream_t stream) {
  auto kern = gemm_pair<Epi, A_MN, B_MN>;
  static int max_clusters = 0;  // per instantiation; all GPUs of a process are the same part
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(GEMM2_SMEM_BYTES));
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 2;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.blockDim = dim3(GEMM_THREADS, 1, 1);
  cfg.dynamicSmemBytes = GEMM2_SMEM_BYTES;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (max_clusters == 0) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    cfg.gridDim = dim3(static_cast<unsigned>(sms & ~1), 1, 1);
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, kern, &cfg);
    if (e != cudaSuccess) return e;
    max_clusters = n > 0 ? n : 1;
  }
  const long long units = static_cast<long long>(sch.m_blocks) * sch.splits;
  const int clusters = static_cast<int>(units < max_clusters ? units : max_clusters);
  if (clusters <= 0) return cudaSuccess;
  cfg.gridDim = dim3(static_cast<unsigned>(2 * clusters), 1, 1);
  e = cudaLaunchKernelEx(&cfg, kern, ta, tb, sch, ep, timeout_ns, status);
  if (e == cudaSuccess) note_launches();
  return e;
}

}  // namespace mc
