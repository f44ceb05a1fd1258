// reuse.cu - the common prefix of consecutive segments of a trajectory (prefix reuse).
//
// A fresh stream re-tokenises the text of the steps before its window (Algorithm 1,
// Sec. 3.4 / App. C.1), and the steps that leave the window join that text, so segment
// s of a trajectory starts with the tokens segment s-1 starts with.  Causal attention row
// r depends only on tokens 0..r of its segment, so over the common prefix the rows of the
// two segments are equal (the forward with prefix reuse computes them once).
//
//   seg_shared[s] = max n with tok_gather[cu[s] + i] == tok_gather[cu[s-1] + i] for i < n,
//                   n <= min(L_s, L_{s-1}); 0 when s is its trajectory's first segment
//
// One block per segment: each thread scans a strided subset of the positions up to its
// first mismatch and the block takes the minimum.
#include <cstdint>

#include "internal.h"

namespace vcs {
namespace {

constexpr int kThreads = 256;

__global__ void __launch_bounds__(kThreads) shared_prefix_kernel(const int32_t* __restrict__ cu_seqlens,
                                                                 const int32_t* __restrict__ seg_traj,
                                                                 const int32_t* __restrict__ tok_gather,
                                                                 int32_t num_segments, int32_t num_tokens,
                                                                 int32_t* __restrict__ seg_shared, int32_t* status) {
  const int s = blockIdx.x;
  __shared__ int smin[kThreads / 32];
  if (s == 0 || seg_traj[s] != seg_traj[s - 1]) {
    if (threadIdx.x == 0) seg_shared[s] = 0;
    return;
  }
  const int pb = cu_seqlens[s - 1], b = cu_seqlens[s], e = cu_seqlens[s + 1];
  if (pb < 0 || b < pb || e < b || e > num_tokens) {
    if (threadIdx.x == 0) {
      seg_shared[s] = 0;
      if (status != nullptr) atomicCAS(status, 0, VCS_ERR_DEVICE_CHECK);
    }
    return;
  }
  const int n = min(e - b, b - pb);
  int first = n;
  for (int i = threadIdx.x; i < n; i += kThreads) {
    if (__ldg(&tok_gather[b + i]) != __ldg(&tok_gather[pb + i])) {
      first = i;
      break;
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) first = min(first, __shfl_xor_sync(0xffffffffu, first, off));
  if ((threadIdx.x & 31) == 0) smin[threadIdx.x >> 5] = first;
  __syncthreads();
  if (threadIdx.x == 0) {
    int m = smin[0];
    for (int w = 1; w < kThreads / 32; ++w) m = min(m, smin[w]);
    seg_shared[s] = m;
  }
}

}  // namespace

cudaError_t launch_shared_prefix(const int32_t* cu_seqlens, const int32_t* seg_traj, const int32_t* tok_gather,
                                 int32_t num_segments, int32_t num_tokens, int32_t* seg_shared, int32_t* status,
                                 cudaStream_t st) {
  if (num_segments == 0) return cudaSuccess;
  shared_prefix_kernel<<<(unsigned)num_segments, kThreads, 0, st>>>(cu_seqlens, seg_traj, tok_gather, num_segments,
                                                                     num_tokens, seg_shared, status);
  return cudaGetLastError();
}

}  // namespace vcs
