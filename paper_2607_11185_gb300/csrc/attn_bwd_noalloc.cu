// attn_bwd_noalloc.cu - the attention backward for callers that cannot
// allocate device memory.
//
// vcs_attn_bwd needs a caller-provided workspace (an fp32 dQ accumulator and
// the per-row terms D).  Some callers cannot provide one: a plugin whose host
// framework owns all device memory and hands it only the input and output
// tensors, or a latency-critical loop that must not call cudaMalloc (which
// can synchronise the device and can fail when memory is nearly full).  This
// entry point takes its workspace from a fixed array compiled into the
// library instead, so neither the caller nor the library allocates anything.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds kNoallocScratchBytes of it until the process exits.  Host code
// must not hand the array's name to a kernel (on the host it names a
// host-side stand-in, not device memory); the device address is looked up once
// per device with cudaGetSymbolAddress and cached.
#include <cstdint>
#include <mutex>

#include "internal.h"

namespace vcs {
namespace {

constexpr size_t kNoallocScratchBytes = size_t(32) << 20;
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_bwd_scratch[kNoallocScratchBytes];

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (set-up on first use).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_bwd_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

}  // namespace
}  // namespace vcs

extern "C" vcs_status vcs_attn_bwd_noalloc(const void* q, const void* k, const void* v, const void* o,
                                           const float* lse, const void* dout, const int32_t* cu_seqlens,
                                           int32_t num_segments, int64_t num_tokens, int32_t max_seqlen,
                                           int32_t hq, int32_t hkv, int32_t d, float softmax_scale, void* dq,
                                           void* dk, void* dv, int32_t* dev_status, void* stream) {
  vcs::ApiRange nvtx_range("vcs_attn_bwd_noalloc");
  const size_t need = vcs_attn_bwd_workspace_size(num_segments, num_tokens, max_seqlen, hq, hkv, d);
  if (need > vcs::kNoallocScratchBytes) return VCS_ERR_WORKSPACE;
  void* scratch = nullptr;
  if (vcs::scratch_address(&scratch) != cudaSuccess) return VCS_ERR_CUDA;
  // vcs_attn_bwd clears the status header and zeroes the dQ accumulator it
  // finds in the workspace before use, so the previous call's contents do
  // not leak into this one.
  const vcs_status s = vcs_attn_bwd(q, k, v, o, lse, dout, cu_seqlens, num_segments, num_tokens, max_seqlen, hq,
                                    hkv, d, softmax_scale, dq, dk, dv, scratch, vcs::kNoallocScratchBytes, stream);
  if (s != VCS_OK) return s;
  if (dev_status != nullptr &&
      cudaMemcpyAsync(dev_status, scratch, sizeof(int32_t), cudaMemcpyDeviceToDevice,
                      static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return VCS_ERR_CUDA;
  return VCS_OK;
}
