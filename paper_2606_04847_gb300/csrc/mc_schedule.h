// mc_schedule.h — the launch-shaping policy of the C-ABI layer (host code,
// included by mc_api.cu only): the row-block height of a projection launch, and how many vocabulary splits its row blocks get.
// These choices decide how often W is streamed from HBM and how busy the SMs
// are; the kernels themselves live in mc_gemm.cuh / mc_fwd.cu / mc_bwd.cu.
#pragma once

#include <cmath>

namespace mc {
namespace sched {

constexpr int kBM = 128;       // rows one CTA owns in a tile (TMA box height for A)
constexpr int kBN = 256;       // vocabulary / output columns per tile
constexpr int kRowPad = 256;   // row padding of workspaces: one row block of either tile height
constexpr int kMaxSplits = 16;

inline long long ceil_div(long long a, long long b) { return (a + b - 1) / b; }

// Projection launches (forward, dZ) with at least this
// many rows use 256-row tiles (TileCfg<2>: a third less operand traffic per
// FLOP, 8 epilogue warps); fewer rows keep 128-row tiles so that small
// launches still spread over the SMs. Measured on the 9B-class shapes: the
// 256-row forward is 7-10 % faster from 2,304 rows up and 1 % slower at 2,048.
constexpr long long kWideMinRows = 2304;
inline bool wide_rows(long long rows) { return rows >= kWideMinRows; }

// Rows per scheduled row block of a projection launch over `rows` rows; one
// unit runs per SM at a time.
inline int row_block(long long rows) { return wide_rows(rows) ? 256 : kBM; }
inline int concurrent_units(int sms) { return sms; }

// Vocabulary tile ranges per row block. A wave of `conc` concurrent units
// streams W once and keeps its conc / s row blocks of hidden rows in L2, so
// s is at least the count that holds those rows under kWaveRowBytes. Among
// the counts allowed, the one with the shortest critical path in tiles,
// waves(s) x ceil(n_tiles / s); counts within kPathSlack of the best resolve
// to the fewest splits. W is read from HBM once per wave, so fewer splits
// (fewer, larger waves) stream it fewer times: under the GPU's power cap the
// DRAM energy saved buys more SM clock than a slightly longer tail costs.
// Past ~100 MB of rows per wave the hidden rows no longer stay in L2.
constexpr double kWaveRowBytes = 80.0 * (1 << 20);
constexpr double kPathSlack = 1.015;

inline int choose_splits(long long m_blocks, int n_tiles, int conc, int rb, int d) {
  long long lo = static_cast<long long>(std::ceil(double(conc) * rb * d * 2.0 / kWaveRowBytes));
  if (lo < 1) lo = 1;
  long long hi = kMaxSplits;
  if (hi > n_tiles) hi = n_tiles;
  if (lo > hi) lo = hi;
  double best_path = 0.0;
  for (long long s = lo; s <= hi; ++s) {
    const double path = double(ceil_div(m_blocks * s, conc)) * double(ceil_div(n_tiles, s));
    if (s == lo || path < best_path) best_path = path;
  }
  for (long long s = lo; s <= hi; ++s) {
    const double path = double(ceil_div(m_blocks * s, conc)) * double(ceil_div(n_tiles, s));
    if (path <= best_path * kPathSlack) return static_cast<int>(s);
  }
  return static_cast<int>(hi);
}

inline int max_splits(int V) {
  const int n_tiles = static_cast<int>(ceil_div(V, kBN));
  return n_tiles < kMaxSplits ? n_tiles : kMaxSplits;
}

}  // namespace sched
}  // namespace mc
