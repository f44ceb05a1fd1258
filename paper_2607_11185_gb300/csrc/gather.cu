// gather.cu - packed segment rows from trajectory rows.
//
// After a prune, Algorithm 1 (Sec. 3.4) re-tokenises the retained history into
// a fresh stream: every segment token is a token of its trajectory, so the
// packed Q/K/V of a segment are rows of the trajectory-layout tensors at the
// builder's gather map.  The copy is HBM-bound: every 16-byte chunk of every
// destination row is read once and written once, with consecutive threads on
// consecutive chunks (coalesced on both sides whenever consecutive segment
// tokens map to consecutive trajectory tokens, which is the common case).
#include <cstdint>

#include "internal.h"
#include "sm100.cuh"

namespace vcs {
namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;

__device__ __forceinline__ int4 ld_stream(const int4* p) {
  int4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.s32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}
__device__ __forceinline__ void st_stream(int4* p, int4 v) {
  asm volatile("st.global.cs.v4.s32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

// One thread moves kUnroll chunks (stride = grid size) per iteration so that
// several independent loads are in flight before the stores.
__global__ void __launch_bounds__(kThreads) gather_rows(const int4* __restrict__ src, int64_t traj_tokens,
                                                        const int32_t* __restrict__ tok_gather, int64_t num_tokens,
                                                        int64_t row_chunks, int4* __restrict__ dst,
                                                        int32_t* status) {
  const int64_t total = num_tokens * row_chunks;
  const int64_t stride = (int64_t)gridDim.x * kThreads;
  for (int64_t c0 = blockIdx.x * (int64_t)kThreads + threadIdx.x; c0 < total; c0 += stride * kUnroll) {
    int4 v[kUnroll];
    int64_t dsti[kUnroll];
    bool ok[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t c = c0 + u * stride;
      ok[u] = false;
      if (c < total) {
        const int64_t n = c / row_chunks;
        const int64_t off = c - n * row_chunks;
        const int64_t s = __ldg(&tok_gather[n]);
        if (s >= 0 && s < traj_tokens) {
          v[u] = ld_stream(src + s * row_chunks + off);
          dsti[u] = c;
          ok[u] = true;
        } else if (off == 0) {
          dev::set_status(status, VCS_ERR_DEVICE_CHECK);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (ok[u]) st_stream(dst + dsti[u], v[u]);
  }
}

}  // namespace

cudaError_t launch_gather(const void* src, int64_t traj_tokens, const int32_t* tok_gather, int64_t num_tokens,
                          int64_t row_bytes, void* dst, int32_t* dev_status, cudaStream_t st) {
  if (num_tokens == 0) return cudaSuccess;
  const int64_t row_chunks = row_bytes / 16;
  const int64_t total = num_tokens * row_chunks;
  int64_t blocks = (total + (int64_t)kThreads * kUnroll - 1) / ((int64_t)kThreads * kUnroll);
  const int64_t cap = 152 * 16;
  if (blocks > cap) blocks = cap;
  gather_rows<<<(unsigned)blocks, kThreads, 0, st>>>(static_cast<const int4*>(src), traj_tokens, tok_gather,
                                                     num_tokens, row_chunks, static_cast<int4*>(dst), dev_status);
  return cudaGetLastError();
}

}  // namespace vcs
