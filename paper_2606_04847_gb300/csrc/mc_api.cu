// mc_api.cu — the C ABI declared in include/mc.h.
//
// Host side only: checks arguments (before touching CUDA, so a bad call never
// launches anything), checks the device is an sm_103 part, lays out the
// caller's workspace, encodes the TMA descriptors and queues the kernels on
// the caller's stream. No device memory is allocated here.
#include <atomic>
#include <cmath>
#include <cstdio>
#include <string>

#include <cuda.h>
#include <cuda_runtime.h>

#include "mc.h"
#include "mc_internal.h"
#include "mc_schedule.h"

namespace {

using namespace mc::sched;

constexpr size_t kStatusBytes = 256;
constexpr int kMaxDevices = 64;

thread_local std::string g_last_cuda_error;

mc_status cuda_fail(cudaError_t e, const char* what) {
  g_last_cuda_error = std::string(what) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
  return MC_ERR_CUDA;
}

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// ---- cached device attributes (the only state the library keeps)
std::atomic<int> g_dev_sms[kMaxDevices];
std::atomic<int> g_dev_cc[kMaxDevices];

mc_status device_info(int* sms) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return MC_ERR_UNSUPPORTED;
  int cc = g_dev_cc[dev].load(std::memory_order_relaxed);
  int n = g_dev_sms[dev].load(std::memory_order_relaxed);
  if (cc == 0) {
    int major = 0, minor = 0;
    if ((e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) != cudaSuccess)
      return cuda_fail(e, "cudaDeviceGetAttribute");
    if ((e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess)
      return cuda_fail(e, "cudaDeviceGetAttribute");
    if ((e = cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return cuda_fail(e, "cudaDeviceGetAttribute");
    cc = major * 10 + minor;
    g_dev_sms[dev].store(n, std::memory_order_relaxed);
    g_dev_cc[dev].store(cc, std::memory_order_relaxed);
  }
  if (cc != 103) return MC_ERR_UNSUPPORTED;  // kernels are built for sm_103a only
  *sms = n;
  return MC_OK;
}

// Limit of every bounded pipeline wait: far above any healthy wait (the
// longest, an MMA issuer waiting for one operand stage, takes microseconds).
constexpr uint64_t kWaitTimeoutNs = 4000000000ull;  // 4 s

// ---- TMA descriptors
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                              CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
  static EncodeFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) !=
            cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      return static_cast<EncodeFn>(nullptr);
    return reinterpret_cast<EncodeFn>(p);
  }();
  return fn;
}

// 2-D bf16 tensor [outer, inner] with row stride `stride_elems`, 128-byte
// swizzled boxes of {64, box_outer}; out-of-range elements read as zero.
mc_status make_tmap_box(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t stride_elems,
                        uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle swizzle) {
  EncodeFn fn = encode_fn();
  if (fn == nullptr) {
    g_last_cuda_error = "cuTensorMapEncodeTiled not available from the driver";
    return MC_ERR_CUDA;
  }
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {stride_elems * 2};
  const cuuint32_t box[2] = {box_inner, box_outer};
  const cuuint32_t estr[2] = {1, 1};
  const CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    char buf[128];
    std::snprintf(buf, sizeof buf, "cuTensorMapEncodeTiled failed (CUresult %d)", static_cast<int>(r));
    g_last_cuda_error = buf;
    return MC_ERR_CUDA;
  }
  return MC_OK;
}

// Operand tiles of the GEMM engines: boxes 64 elements (128 bytes) wide,
// 128-byte swizzle.
mc_status make_tmap(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer, uint64_t stride_elems,
                    uint32_t box_outer) {
  return make_tmap_box(m, base, inner, outer, stride_elems, 64, box_outer, CU_TENSOR_MAP_SWIZZLE_128B);
}

bool valid_common(int64_t N, int32_t d, int32_t V, float inv_temperature) {
  if (N < 0 || N >= (1LL << 31)) return false;
  if (V < 1) return false;
  if (d <= 0 || d % 64 != 0 || d > 16384) return false;
  if (!(inv_temperature > 0.f) || !std::isfinite(inv_temperature)) return false;
  return true;
}

struct FwdLayout {
  size_t status_off, part_off, zy_off, total;
  long long n_pad;
};

FwdLayout fwd_layout(int64_t N, int32_t V) {
  FwdLayout L;
  L.n_pad = ceil_div(N, kRowPad) * kRowPad;
  const size_t part_bytes = size_t(3) * max_splits(V) * size_t(L.n_pad) * 4;
  L.status_off = 0;
  L.part_off = kStatusBytes;
  L.zy_off = align_up(L.part_off + part_bytes, 256);
  L.total = align_up(L.zy_off + size_t(L.n_pad) * 4, 256);
  return L;
}

long long v_pad(int32_t V) { return ceil_div(V, 64) * 64; }

// Backward workspace: [status | wave gate counter (offset 64) | count (offset
// 128)] header, selected-row indices, the
// gathered hidden rows (zero-padded to a 256-row multiple), then the dZ chunk
// buffer.
struct BwdLayout {
  size_t status_off, count_off, idx_off, hc_off, fixed;
  long long n_pad;
};

BwdLayout bwd_layout(int64_t N, int32_t d) {
  BwdLayout L;
  L.n_pad = ceil_div(N, kRowPad) * kRowPad;
  L.status_off = 0;
  L.count_off = 128;
  L.idx_off = kStatusBytes;
  L.hc_off = align_up(L.idx_off + size_t(L.n_pad) * 4, 256);
  L.fixed = align_up(L.hc_off + size_t(L.n_pad) * size_t(d) * 2, 256);
  return L;
}

}  // namespace

namespace mc {
namespace {
std::atomic<unsigned long long> g_kernel_launches{0};
}  // namespace
void note_launches(unsigned n) { g_kernel_launches.fetch_add(n, std::memory_order_relaxed); }
}  // namespace mc

extern "C" {

const char* mc_status_string(mc_status s) {
  switch (s) {
    case MC_OK: return "MC_OK";
    case MC_ERR_INVALID_ARG: return "MC_ERR_INVALID_ARG: invalid argument (null/misaligned pointer or size out of range)";
    case MC_ERR_UNSUPPORTED: return "MC_ERR_UNSUPPORTED: unsupported shape or device (needs sm_103, d % 64 == 0)";
    case MC_ERR_CUDA: return "MC_ERR_CUDA: a CUDA call failed (see mc_last_cuda_error)";
    case MC_ERR_TIMEOUT: return "MC_ERR_TIMEOUT: a bounded device wait gave up";
    case MC_ERR_WORKSPACE: return "MC_ERR_WORKSPACE: workspace missing, misaligned or too small";
    case MC_ERR_TARGET_RANGE: return "MC_ERR_TARGET_RANGE: a target index outside [0, V)";
    case MC_ERR_SCRATCH_LIMIT:
      return "MC_ERR_SCRATCH_LIMIT: request needs more than the fixed MC_NOALLOC_SCRATCH_BYTES scratch";
  }
  return "unknown mc_status";
}

const char* mc_last_cuda_error(void) { return g_last_cuda_error.c_str(); }

int32_t mc_version(void) { return (1 << 16) | 1; }

uint64_t mc_kernel_launches(void) { return mc::g_kernel_launches.load(std::memory_order_relaxed); }

size_t mc_token_logprobs_workspace_size(int64_t N, int32_t d, int32_t V) {
  if (!valid_common(N, d, V, 1.f)) return 0;
  return fwd_layout(N, V).total;
}

}  // extern "C"

namespace {

// Queues the forward over the rows of W (a whole vocabulary, or a slice whose
// row 0 is global id v_offset). Writes logp/entropy/lse, or with `state` the
// slice state. Arguments are already validated.
mc_status queue_forward(const void* hidden, const void* w_vocab, const int32_t* targets, int64_t N, int32_t d,
                        int32_t V, int32_t v_offset, float inv_temperature, float* logp, float* entropy, float* lse,
                        float* state, void* workspace, size_t workspace_bytes, int32_t* dev_status,
                        mc_stream_t stream) {
  const FwdLayout L = fwd_layout(N, V);
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < L.total) return MC_ERR_WORKSPACE;
  int sms = 0;
  mc_status st = device_info(&sms);
  if (st != MC_OK) return st;

  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  mc::FwdArgs a;
  if ((st = make_tmap(&a.tm_hidden, hidden, d, N, d, kBM)) != MC_OK) return st;
  if ((st = make_tmap(&a.tm_w, w_vocab, d, V, d, kBN)) != MC_OK) return st;
  const long long m_blocks = ceil_div(N, row_block(N));
  const int n_tiles = static_cast<int>(ceil_div(V, kBN));
  a.targets = targets;
  a.N = N;
  a.d = d;
  a.V = V;
  a.inv_temperature = inv_temperature;
  a.splits = choose_splits(m_blocks, n_tiles, concurrent_units(sms), row_block(N), d);
  a.n_pad = L.n_pad;
  a.part = reinterpret_cast<float*>(ws + L.part_off);
  a.zy = reinterpret_cast<float*>(ws + L.zy_off);
  a.ws_status = reinterpret_cast<int32_t*>(ws + L.status_off);
  a.wave_ctr = reinterpret_cast<unsigned int*>(ws + L.status_off + 64);
  a.logp = logp;
  a.entropy = entropy;
  a.lse = lse;
  a.dev_status = dev_status;
  a.grid = sms;
  a.timeout_ns = kWaitTimeoutNs;
  a.wide = wide_rows(N) ? 1 : 0;
  // Two column halves per sub-block when twice the split partials still fit
  // the max_splits(V) slots per row that the workspace holds.
  a.halves = (a.wide && 2 * a.splits <= max_splits(V)) ? 2 : 1;
  a.v_offset = v_offset;
  a.state = state;
  cudaError_t e = cudaMemsetAsync(ws + L.status_off, 0, 128, s);  // status word and wave gate counter
  if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
  e = mc::launch_forward(a, s);
  if (e != cudaSuccess) return cuda_fail(e, "forward launch");
  return MC_OK;
}

}  // namespace

extern "C" {

mc_status mc_token_logprobs(const void* hidden, const void* w_vocab, const int32_t* targets, int64_t N,
                            int32_t d, int32_t V, float inv_temperature, float* logp, float* entropy,
                            float* lse, void* workspace, size_t workspace_bytes, int32_t* dev_status,
                            mc_stream_t stream) {
  if (!valid_common(N, d, V, inv_temperature)) return MC_ERR_INVALID_ARG;
  if (N == 0) return MC_OK;
  if (!hidden || !w_vocab || !targets || !logp) return MC_ERR_INVALID_ARG;
  if (!aligned(hidden, 16) || !aligned(w_vocab, 16) || !aligned(targets, 4) || !aligned(logp, 4) ||
      (entropy && !aligned(entropy, 4)) || (lse && !aligned(lse, 4)) || (dev_status && !aligned(dev_status, 4)))
    return MC_ERR_INVALID_ARG;
  return queue_forward(hidden, w_vocab, targets, N, d, V, 0, inv_temperature, logp, entropy, lse, nullptr,
                       workspace, workspace_bytes, dev_status, stream);
}

mc_status mc_token_logprob_state(const void* hidden, const void* w_shard, const int32_t* targets, int64_t N,
                                 int32_t d, int32_t V_shard, int32_t v_begin, float inv_temperature, float* state,
                                 void* workspace, size_t workspace_bytes, int32_t* dev_status, mc_stream_t stream) {
  if (!valid_common(N, d, V_shard, inv_temperature) || v_begin < 0) return MC_ERR_INVALID_ARG;
  if (N == 0) return MC_OK;
  if (!hidden || !w_shard || !targets || !state) return MC_ERR_INVALID_ARG;
  if (!aligned(hidden, 16) || !aligned(w_shard, 16) || !aligned(targets, 4) || !aligned(state, 16) ||
      (dev_status && !aligned(dev_status, 4)))
    return MC_ERR_INVALID_ARG;
  return queue_forward(hidden, w_shard, targets, N, d, V_shard, v_begin, inv_temperature, nullptr, nullptr, nullptr,
                       state, workspace, workspace_bytes, dev_status, stream);
}

mc_status mc_merge_logprob_states(const float* states, int32_t P, int64_t N, float* logp, float* entropy, float* lse,
                                  int32_t* dev_status, mc_stream_t stream) {
  if (P < 1 || N < 0 || N >= (1LL << 31)) return MC_ERR_INVALID_ARG;
  if (N == 0) return MC_OK;
  if (!states || !logp || !aligned(states, 16) || !aligned(logp, 4) || (entropy && !aligned(entropy, 4)) ||
      (lse && !aligned(lse, 4)) || (dev_status && !aligned(dev_status, 4)))
    return MC_ERR_INVALID_ARG;
  int sms = 0;
  mc_status st = device_info(&sms);
  if (st != MC_OK) return st;
  cudaError_t e = mc::launch_merge_states(states, P, N, logp, entropy, lse, dev_status,
                                          reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "state merge launch");
  return MC_OK;
}

size_t mc_token_logprobs_bwd_workspace_size(int64_t N, int32_t d, int32_t V, int64_t rows_per_chunk) {
  if (!valid_common(N, d, V, 1.f) || rows_per_chunk < 1) return 0;
  long long r = rows_per_chunk < N ? rows_per_chunk : N;
  r = ceil_div(r < 1 ? 1 : r, kRowPad) * kRowPad;
  return bwd_layout(N, d).fixed + align_up(size_t(r) * size_t(v_pad(V)) * 2, 256);
}

mc_status mc_token_logprobs_bwd(const void* hidden, const void* w_vocab, const int32_t* targets, const float* lse,
                                const float* entropy, const float* grad_logp, const float* grad_entropy,
                                const uint8_t* row_keep, int64_t N, int32_t d, int32_t V, float inv_temperature,
                                void* grad_hidden, float* grad_w, int32_t accumulate, void* workspace,
                                size_t workspace_bytes, int32_t* dev_status, mc_stream_t stream) {
  if (!valid_common(N, d, V, inv_temperature)) return MC_ERR_INVALID_ARG;
  if (!grad_w || !aligned(grad_w, 16)) return MC_ERR_INVALID_ARG;
  if (N > 0) {
    if (!hidden || !w_vocab || !targets || !lse || !grad_logp || !grad_hidden) return MC_ERR_INVALID_ARG;
    if (grad_entropy && !entropy) return MC_ERR_INVALID_ARG;
    if (!aligned(hidden, 16) || !aligned(w_vocab, 16) || !aligned(grad_hidden, 16) || !aligned(targets, 4) ||
        !aligned(lse, 4) || !aligned(grad_logp, 4) || (entropy && !aligned(entropy, 4)) ||
        (grad_entropy && !aligned(grad_entropy, 4)) || (dev_status && !aligned(dev_status, 4)))
      return MC_ERR_INVALID_ARG;
  }
  const long long vp = v_pad(V);
  const BwdLayout L = bwd_layout(N, d);
  long long R = 0;
  if (N > 0) {
    if (!workspace || !aligned(workspace, 256) || workspace_bytes < mc_token_logprobs_bwd_workspace_size(N, d, V, kRowPad))
      return MC_ERR_WORKSPACE;
    R = static_cast<long long>((workspace_bytes - L.fixed) / (size_t(vp) * 2));
    R = R / kRowPad * kRowPad;
    if (R > L.n_pad) R = L.n_pad;
    if (R < kRowPad) return MC_ERR_WORKSPACE;
  }
  int sms = 0;
  mc_status st = device_info(&sms);
  if (st != MC_OK) return st;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (N == 0) {
    if (!accumulate) {
      e = cudaMemsetAsync(grad_w, 0, size_t(V) * size_t(d) * sizeof(float), s);
      if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
    }
    return MC_OK;
  }
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  int32_t* ws_status = reinterpret_cast<int32_t*>(ws + L.status_off);
  int32_t* count = reinterpret_cast<int32_t*>(ws + L.count_off);
  int32_t* idx = reinterpret_cast<int32_t*>(ws + L.idx_off);
  uint16_t* hc = reinterpret_cast<uint16_t*>(ws + L.hc_off);
  void* dz = ws + L.fixed;
  if ((e = cudaMemsetAsync(ws, 0, kStatusBytes, s)) != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync");
  // Rows outside the selection keep a zero gradient.
  if ((e = cudaMemsetAsync(grad_hidden, 0, size_t(N) * size_t(d) * 2, s)) != cudaSuccess)
    return cuda_fail(e, "cudaMemsetAsync");

  const uint64_t tmo = kWaitTimeoutNs;
  mc::SelectArgs sa;
  sa.hidden = hidden;
  sa.row_keep = row_keep;
  sa.grad_logp = grad_logp;
  sa.grad_entropy = grad_entropy;
  sa.targets = targets;
  sa.N = N;
  sa.d = d;
  sa.V = V;
  sa.idx = idx;
  sa.count = count;
  sa.hc = hc;
  // The slab offsets of the row selection live at the start of the gathered-
  // rows region: selection finishes with them before the gather writes it
  // (n_pad * d * 2 bytes, far more than the ceil(N / 1024) * 4 they take).
  sa.slab = reinterpret_cast<int32_t*>(hc);
  sa.ws_status = ws_status;
  sa.grid = sms * 8;
  if ((e = mc::launch_select_gather(sa, s)) != cudaSuccess) return cuda_fail(e, "row selection launch");

  CUtensorMap tm_w_k, tm_w_mn;
  if ((st = make_tmap(&tm_w_k, w_vocab, d, V, d, kBN)) != MC_OK) return st;
  if ((st = make_tmap(&tm_w_mn, w_vocab, d, V, d, 64)) != MC_OK) return st;
  const int n_tiles = static_cast<int>(ceil_div(V, kBN));

  // Chunks of R compacted rows; chunks past the device-side count do no work.
  for (long long r0 = 0; r0 < N; r0 += R) {
    const long long rows = (N - r0) < R ? (N - r0) : R;
    const void* hc_chunk = hc + r0 * d;
    mc::DzArgs za;
    if ((st = make_tmap(&za.tm_hidden, hc_chunk, d, rows, d, kBM)) != MC_OK) return st;
    za.tm_w = tm_w_k;
    za.targets = targets;
    za.lse = lse;
    za.entropy = entropy;
    za.grad_logp = grad_logp;
    za.grad_entropy = grad_entropy;
    za.idx = idx + r0;
    za.count = count;
    za.row_offset = r0;
    za.rows = rows;
    za.d = d;
    za.V = V;
    za.inv_temperature = inv_temperature;
    const int rb = row_block(rows);
    za.splits = choose_splits(ceil_div(rows, rb), n_tiles, concurrent_units(sms), rb, d);
    za.dz = dz;
    za.ld = vp;
    if ((st = make_tmap_box(&za.tm_dz_st, dz, V, rows, vp, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B)) != MC_OK) return st;
    za.ws_status = ws_status;
    za.grid = sms;
    za.timeout_ns = tmo;
    za.wave_ctr = reinterpret_cast<unsigned int*>(ws + 64);
    za.wide = wide_rows(rows) ? 1 : 0;
    if ((e = mc::launch_dz(za, s)) != cudaSuccess) return cuda_fail(e, "dZ launch");

    mc::DhArgs ha;
    if ((st = make_tmap(&ha.tm_dz, dz, V, rows, vp, kBM)) != MC_OK) return st;
    ha.tm_w_mn = tm_w_mn;
    ha.idx = idx + r0;
    ha.count = count;
    ha.row_offset = r0;
    ha.rows = rows;
    ha.d = d;
    ha.V = V;
    ha.grad_hidden = grad_hidden;
    ha.ws_status = ws_status;
    ha.grid = sms;
    ha.timeout_ns = tmo;
    ha.wave_ctr = reinterpret_cast<unsigned int*>(ws + 64);
    if ((e = mc::launch_dh(ha, s)) != cudaSuccess) return cuda_fail(e, "dH launch");

    mc::DwArgs wa;
    if ((st = make_tmap(&wa.tm_dz_mn, dz, V, rows, vp, 64)) != MC_OK) return st;
    if ((st = make_tmap(&wa.tm_h_mn, hc_chunk, d, rows, d, 64)) != MC_OK) return st;
    wa.count = count;
    wa.row_offset = r0;
    wa.rows = rows;
    wa.d = d;
    wa.V = V;
    wa.grad_w = grad_w;
    wa.accumulate = (accumulate || r0 > 0) ? 1 : 0;
    wa.ws_status = ws_status;
    wa.grid = sms;
    wa.timeout_ns = tmo;
    wa.wave_ctr = reinterpret_cast<unsigned int*>(ws + 64);
    if ((e = mc::launch_dw(wa, s)) != cudaSuccess) return cuda_fail(e, "dW launch");
  }
  if ((e = mc::launch_status_merge(ws_status, dev_status, s)) != cudaSuccess) return cuda_fail(e, "status launch");
  return MC_OK;
}

mc_status mc_seq_ratio_filter(const float* logp_policy, const float* logp_behaviour, const uint8_t* loss_mask,
                              const int64_t* cu_seqlens, int32_t B, int64_t N, float delta, float delta_vanilla,
                              float* signed_mean, float* abs_mean, int32_t* n_tokens, uint8_t* keep,
                              uint8_t* keep_vanilla, float* token_ratio, uint8_t* token_keep, mc_stream_t stream) {
  if (B < 1 || N < 0 || N >= (1LL << 40)) return MC_ERR_INVALID_ARG;
  if (!(delta >= 0.f) || !std::isfinite(delta) || std::isnan(delta_vanilla)) return MC_ERR_INVALID_ARG;
  if (!cu_seqlens || !signed_mean || !abs_mean || !n_tokens || !keep) return MC_ERR_INVALID_ARG;
  if (N > 0 && (!logp_policy || !logp_behaviour)) return MC_ERR_INVALID_ARG;
  if (!aligned(cu_seqlens, 8) || !aligned(signed_mean, 4) || !aligned(abs_mean, 4) || !aligned(n_tokens, 4) ||
      (logp_policy && !aligned(logp_policy, 4)) || (logp_behaviour && !aligned(logp_behaviour, 4)) ||
      (token_ratio && !aligned(token_ratio, 4)))
    return MC_ERR_INVALID_ARG;
  int sms = 0;
  mc_status st = device_info(&sms);
  if (st != MC_OK) return st;
  mc::FilterArgs a;
  a.logp_policy = logp_policy;
  a.logp_behaviour = logp_behaviour;
  a.loss_mask = loss_mask;
  a.cu_seqlens = cu_seqlens;
  a.B = B;
  a.N = N;
  a.delta = delta;
  a.delta_vanilla = delta_vanilla;
  a.signed_mean = signed_mean;
  a.abs_mean = abs_mean;
  a.n_tokens = n_tokens;
  a.keep = keep;
  a.keep_vanilla = keep_vanilla;
  a.token_ratio = token_ratio;
  a.token_keep = token_keep;
  a.vec_ok = aligned(logp_policy, 16) && aligned(logp_behaviour, 16) && (!token_ratio || aligned(token_ratio, 16)) &&
             (!loss_mask || aligned(loss_mask, 4));
  a.keep_vec_ok = aligned(token_keep, 16) && (!loss_mask || aligned(loss_mask, 16));
  a.grid = mc::filter_ctas_per_sm() * sms;
  cudaError_t e = mc::launch_filter(a, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "filter launch");
  return MC_OK;
}

size_t mc_grpo_masked_loss_workspace_size(int32_t B) {
  if (B < 1) return 0;
  return kStatusBytes + 2 * align_up(size_t(B) * sizeof(float), 256);
}

mc_status mc_grpo_masked_loss(const float* logp_policy, const float* logp_behaviour, const uint8_t* loss_mask,
                              const int64_t* cu_seqlens, const float* advantages, const uint8_t* keep,
                              const int32_t* n_tokens, int32_t B, int64_t N, float eps_low, float eps_high,
                              const float* logp_ref, float beta, float* loss, float* grad_logp, float* seq_loss,
                              int32_t* n_clipped, float* kl, void* workspace, size_t workspace_bytes,
                              mc_stream_t stream) {
  if (B < 1 || N < 0 || N >= (1LL << 40)) return MC_ERR_INVALID_ARG;
  if (!(eps_low >= 0.f && eps_low < 1.f) || !(eps_high >= 0.f) || !std::isfinite(eps_high))
    return MC_ERR_INVALID_ARG;
  if (!(beta >= 0.f) || !std::isfinite(beta)) return MC_ERR_INVALID_ARG;
  if ((logp_ref && !aligned(logp_ref, 4)) || (kl && !aligned(kl, 4))) return MC_ERR_INVALID_ARG;
  if (!cu_seqlens || !advantages || !keep || !n_tokens || !loss) return MC_ERR_INVALID_ARG;
  if (N > 0 && (!logp_policy || !logp_behaviour || !grad_logp)) return MC_ERR_INVALID_ARG;
  if (!aligned(cu_seqlens, 8) || !aligned(advantages, 4) || !aligned(n_tokens, 4) || !aligned(loss, 4) ||
      (logp_policy && !aligned(logp_policy, 4)) || (logp_behaviour && !aligned(logp_behaviour, 4)) ||
      (grad_logp && !aligned(grad_logp, 4)) || (seq_loss && !aligned(seq_loss, 4)) ||
      (n_clipped && !aligned(n_clipped, 4)))
    return MC_ERR_INVALID_ARG;
  if (!workspace || !aligned(workspace, 256) || workspace_bytes < mc_grpo_masked_loss_workspace_size(B))
    return MC_ERR_WORKSPACE;
  int sms = 0;
  mc_status st = device_info(&sms);
  if (st != MC_OK) return st;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  mc::LossArgs a;
  a.logp_policy = logp_policy;
  a.logp_behaviour = logp_behaviour;
  a.loss_mask = loss_mask;
  a.cu_seqlens = cu_seqlens;
  a.advantages = advantages;
  a.keep = keep;
  a.n_tokens = n_tokens;
  a.B = B;
  a.N = N;
  a.eps_low = eps_low;
  a.eps_high = eps_high;
  a.logp_ref = N > 0 ? logp_ref : nullptr;
  a.beta = logp_ref ? beta : 0.f;
  a.loss = loss;
  a.grad_logp = grad_logp;
  a.seq_loss = seq_loss;
  a.n_clipped = n_clipped;
  a.kl = kl;
  a.Z = reinterpret_cast<long long*>(ws);
  a.ticket = reinterpret_cast<unsigned int*>(ws + sizeof(long long));
  a.seq_share = reinterpret_cast<float*>(ws + kStatusBytes);
  a.seq_kl = reinterpret_cast<float*>(ws + kStatusBytes + align_up(size_t(B) * sizeof(float), 256));
  a.vec_ok = aligned(logp_policy, 16) && aligned(logp_behaviour, 16) && aligned(grad_logp, 16) &&
             (!logp_ref || aligned(logp_ref, 16)) && (!loss_mask || aligned(loss_mask, 4));
  a.grid = 16 * sms;
  cudaError_t e = mc::launch_grpo_loss(a, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "GRPO loss launch");
  return MC_OK;
}

mc_status mc_prime_echo_advantages(const float* scores, const uint8_t* success, const int32_t* n_turns, int32_t T,
                                   int32_t K, int32_t group_size, float alpha, float beta1, float beta2, float eps,
                                   float* reward, float* advantage, mc_stream_t stream) {
  if (T < 1 || K < 1 || group_size < 1 || T % group_size != 0) return MC_ERR_INVALID_ARG;
  if (!(alpha >= 0.f && alpha <= 1.f) || !(beta1 >= 0.f) || !(beta2 >= 0.f) || !(eps >= 0.f) ||
      !std::isfinite(beta1) || !std::isfinite(beta2) || !std::isfinite(eps))
    return MC_ERR_INVALID_ARG;
  if (!scores || !success || !n_turns || !advantage) return MC_ERR_INVALID_ARG;
  if (!aligned(scores, 4) || !aligned(n_turns, 4) || !aligned(advantage, 4) || (reward && !aligned(reward, 4)))
    return MC_ERR_INVALID_ARG;
  int sms = 0;
  mc_status st = device_info(&sms);
  if (st != MC_OK) return st;
  mc::AdvArgs a;
  a.scores = scores;
  a.success = success;
  a.n_turns = n_turns;
  a.n_groups = T / group_size;
  a.G = group_size;
  a.K = K;
  a.alpha = alpha;
  a.beta1 = beta1;
  a.beta2 = beta2;
  a.eps = eps;
  a.reward = reward;
  a.advantage = advantage;
  a.vec4 = (K == 4 && aligned(scores, 16) && aligned(success, 4)) ? 1 : 0;
  cudaError_t e = mc::launch_group_advantage(a, reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "advantage launch");
  return MC_OK;
}

mc_status mc_selftest_bounded_wait(int32_t* dev_status, int64_t timeout_ns, mc_stream_t stream) {
  if (!dev_status || !aligned(dev_status, 4)) return MC_ERR_INVALID_ARG;
  if (timeout_ns < 1000000LL || timeout_ns > 10000000000LL) return MC_ERR_INVALID_ARG;
  int sms = 0;
  mc_status st = device_info(&sms);
  if (st != MC_OK) return st;
  cudaError_t e = mc::launch_selftest_wait(dev_status, static_cast<uint64_t>(timeout_ns),
                                           reinterpret_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "self-test launch");
  return MC_OK;
}

}  // extern "C"
