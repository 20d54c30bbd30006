// mc_noalloc.cu — the forward (mc_token_logprobs) for callers that cannot
// allocate device memory.
//
// Some callers may not call cudaMalloc: a host process whose memory manager
// owns every device allocation and forbids libraries from making their own, a
// plugin that runs inside such a host, or a latency-critical loop that cannot
// afford the device-wide synchronisation an allocation may cause. They also
// may have no spare buffer to hand over as a workspace. For them the scratch
// the forward needs (the per-split softmax partials, the target logits and a
// status word) lives in a fixed array compiled into this library. Every GPU
// that loads the library holds that array (MC_NOALLOC_SCRATCH_BYTES) until
// the process exits.
#include <mutex>

#include <cuda_runtime.h>

#include "mc.h"

namespace {

constexpr size_t kScratchBytes = MC_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

// The scratch itself. In host code this name is only a host-side stand-in for
// the device array, never a device address: the address comes from
// cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

std::mutex g_mu;
void* g_scratch_dev_ptr[kMaxDevices] = {};

// Device address of the scratch on the current device, looked up once per
// device (with that device current) and cached for the life of the process:
// a cudaDeviceReset() unloads the module and leaves the cached address stale.
mc_status scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return MC_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_scratch_dev_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return MC_ERR_CUDA;
    g_scratch_dev_ptr[dev] = p;
  }
  *out = g_scratch_dev_ptr[dev];
  return MC_OK;
}

}  // namespace

extern "C" mc_status mc_token_logprobs_noalloc(const void* hidden, const void* w_vocab, const int32_t* targets,
                                               int64_t N, int32_t d, int32_t V, float inv_temperature,
                                               float* logp, float* entropy, float* lse, int32_t* dev_status,
                                               mc_stream_t stream) {
  const size_t need = mc_token_logprobs_workspace_size(N, d, V);
  if (need > kScratchBytes) return MC_ERR_SCRATCH_LIMIT;
  void* scratch = nullptr;
  if (need > 0) {
    const mc_status st = scratch_address(&scratch);
    if (st != MC_OK) return st;
  }
  // Same checks, kernels and launch sequence as the workspace entry point; the
  // status word at the start of the scratch is cleared on the stream there.
  return mc_token_logprobs(hidden, w_vocab, targets, N, d, V, inv_temperature, logp, entropy, lse, scratch,
                           kScratchBytes, dev_status, stream);
}
