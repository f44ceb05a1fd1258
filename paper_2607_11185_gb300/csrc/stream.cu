// stream.cu - Algorithm 1's token-ID stream fields over the segment layout
// (App. C.1) and the ordered list of trainable tokens, sm_103a.
//
//   ids[n]  = traj_ids[tok_gather[n]]
//   logp[n] = tok_loss_mask[n] ? traj_logp[tok_gather[n]] : 0
// (trainable response tokens keep their rollout log-probability; observation
// tokens and the re-tokenised history of a fresh stream carry 0), and
//   idx = the n with tok_loss_mask[n] = 1, in increasing order.
//
// Both are HBM-bound.  The compaction is three launches: per-chunk counts, one
// block scanning the chunk counts, and a per-chunk ordered write (warp ballots
// and a block-wide prefix over the warps).
#include <cstdint>

#include "internal.h"

namespace vcs {
namespace {

constexpr int kThreads = 256;
constexpr int kChunk = kThreads * 16;  // tokens per compaction block

__device__ __forceinline__ void set_status(int32_t* status, int32_t code) {
  if (status != nullptr) atomicCAS(status, 0, code);
}

__global__ void __launch_bounds__(kThreads) stream_fields_kernel(const int32_t* __restrict__ traj_ids,
                                                                 const float* __restrict__ traj_logp,
                                                                 int64_t traj_tokens,
                                                                 const int32_t* __restrict__ tok_gather,
                                                                 const uint8_t* __restrict__ mask, int64_t num_tokens,
                                                                 int32_t* __restrict__ ids, float* __restrict__ logp,
                                                                 int32_t* status) {
  for (int64_t n = blockIdx.x * (int64_t)kThreads + threadIdx.x; n < num_tokens; n += (int64_t)gridDim.x * kThreads) {
    const int32_t g = __ldg(&tok_gather[n]);
    if (g < 0 || g >= traj_tokens) {
      set_status(status, VCS_ERR_DEVICE_CHECK);
      ids[n] = 0;
      logp[n] = 0.f;
      continue;
    }
    ids[n] = __ldg(&traj_ids[g]);
    logp[n] = __ldg(&mask[n]) != 0 ? __ldg(&traj_logp[g]) : 0.f;
  }
}

__global__ void __launch_bounds__(kThreads) compact_count(const uint8_t* __restrict__ mask, int64_t num_tokens,
                                                          int64_t* __restrict__ counts) {
  const int64_t base = blockIdx.x * (int64_t)kChunk;
  int c = 0;
  for (int i = threadIdx.x; i < kChunk; i += kThreads) {
    const int64_t n = base + i;
    if (n < num_tokens && __ldg(&mask[n]) != 0) ++c;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) c += __shfl_down_sync(0xffffffffu, c, off);
  __shared__ int red[kThreads / 32];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    int s = 0;
    for (int w = 0; w < kThreads / 32; ++w) s += red[w];
    counts[blockIdx.x] = s;
  }
}

// exclusive scan of the chunk counts in place (one block); total -> *count
__global__ void __launch_bounds__(kThreads) compact_scan(int64_t* __restrict__ counts, int nchunks,
                                                         int64_t* __restrict__ count) {
  __shared__ int64_t carry;
  __shared__ int64_t warp_sum[kThreads / 32];
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < nchunks; base += kThreads) {
    const int i = base + threadIdx.x;
    const int64_t v = i < nchunks ? counts[i] : 0;
    int64_t x = v;  // inclusive scan within the warp
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int64_t y = __shfl_up_sync(0xffffffffu, x, off);
      if ((threadIdx.x & 31) >= off) x += y;
    }
    if ((threadIdx.x & 31) == 31) warp_sum[threadIdx.x >> 5] = x;
    __syncthreads();
    int64_t before = carry;
    for (int w = 0; w < (int)(threadIdx.x >> 5); ++w) before += warp_sum[w];
    if (i < nchunks) counts[i] = before + x - v;
    __syncthreads();
    if (threadIdx.x == kThreads - 1) carry = before + x;
    __syncthreads();
  }
  if (threadIdx.x == 0) *count = carry;
}

__global__ void __launch_bounds__(kThreads) compact_write(const uint8_t* __restrict__ mask, int64_t num_tokens,
                                                          const int64_t* __restrict__ offsets,
                                                          int32_t* __restrict__ idx, int64_t capacity,
                                                          int32_t* status) {
  __shared__ int warp_cnt[kThreads / 32];
  const int64_t base = blockIdx.x * (int64_t)kChunk;
  int64_t out = offsets[blockIdx.x];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int it = 0; it < kChunk / kThreads; ++it) {
    const int64_t n = base + it * kThreads + threadIdx.x;
    const bool take = n < num_tokens && __ldg(&mask[n]) != 0;
    const unsigned bal = __ballot_sync(0xffffffffu, take);
    if (lane == 0) warp_cnt[warp] = __popc(bal);
    __syncthreads();
    int64_t pos = out + __popc(bal & ((1u << lane) - 1u));
    int total = 0;
    for (int w = 0; w < kThreads / 32; ++w) {
      if (w < warp) pos += warp_cnt[w];
      total += warp_cnt[w];
    }
    if (take) {
      if (pos < capacity) idx[pos] = (int32_t)n;
      else set_status(status, VCS_ERR_CAPACITY);
    }
    out += total;
    __syncthreads();
  }
}

}  // namespace

cudaError_t launch_stream_fields(const int32_t* traj_ids, const float* traj_logp, int64_t traj_tokens,
                                 const int32_t* tok_gather, const uint8_t* mask, int64_t num_tokens, int32_t* ids,
                                 float* logp, int32_t* status, cudaStream_t st) {
  if (num_tokens == 0) return cudaSuccess;
  int64_t blocks = (num_tokens + kThreads - 1) / kThreads;
  if (blocks > 152 * 16) blocks = 152 * 16;
  stream_fields_kernel<<<(unsigned)blocks, kThreads, 0, st>>>(traj_ids, traj_logp, traj_tokens, tok_gather, mask,
                                                              num_tokens, ids, logp, status);
  return cudaGetLastError();
}

size_t compact_ws_bytes(int64_t num_tokens) {
  const int64_t nchunks = (num_tokens + kChunk - 1) / kChunk;
  return kWsHeader + (size_t)(nchunks > 0 ? nchunks : 1) * sizeof(int64_t);
}

cudaError_t launch_compact(const uint8_t* mask, int64_t num_tokens, int32_t* idx, int64_t capacity, int64_t* count,
                           void* ws, cudaStream_t st) {
  int32_t* status = static_cast<int32_t*>(ws);
  int64_t* counts = reinterpret_cast<int64_t*>(static_cast<char*>(ws) + kWsHeader);
  const int64_t nchunks = (num_tokens + kChunk - 1) / kChunk;
  if (cudaMemsetAsync(status, 0, sizeof(int32_t), st) != cudaSuccess) return cudaErrorUnknown;
  if (nchunks == 0) return cudaMemsetAsync(count, 0, sizeof(int64_t), st);
  compact_count<<<(unsigned)nchunks, kThreads, 0, st>>>(mask, num_tokens, counts);
  compact_scan<<<1, kThreads, 0, st>>>(counts, (int)nchunks, count);
  compact_write<<<(unsigned)nchunks, kThreads, 0, st>>>(mask, num_tokens, counts, idx, capacity, status);
  return cudaGetLastError();
}

}  // namespace vcs
