// loss.cu - the token-level RL objective over packed segments (App. C.2), sm_103a.
//
// For every segment token t (trajectory b(t), advantage A = adv[b(t)], loss
// mask m_t from the segment builder):
//   rho = exp(logp - old_logp)
//   o   = min(rho A, clip(rho, 1 - eps_l, 1 + eps_h) A), and for A < 0 also
//         o = max(o, c A)   (the clip-ratio cap c)
//   k   = exp(r) - r - 1 with r = ref_logp - logp   (per-token KL estimate)
//   loss   = (1/N_traj) sum_t m_t (-o + lambda k)
//   dlogp  = (m_t/N_traj) (-do/dlogp + lambda (1 - exp(r))),  do/dlogp = rho A
//            on the rho-dependent branch, 0 where o is clipped to a constant.
// The branch is taken in float32; the per-token terms are float32 and the sum
// is accumulated in double, per block and then over the blocks in a fixed
// order (the result does not depend on scheduling).
//
// HBM-bound: 17 bytes per token (three fp32 inputs, the mask byte, the fp32
// gradient), plus a log2(num_segments) lookup of the token's segment in
// cu_seqlens (L1-resident).
#include <cstdint>

#include "internal.h"

namespace vcs {
namespace {

constexpr int kThreads = 256;
constexpr int kPerThread = 8;
constexpr int kChunk = kThreads * kPerThread;  // tokens per block
constexpr int kMaxBlocks = 152 * 8;

__device__ __forceinline__ void set_status(int32_t* status, int32_t code) { atomicCAS(status, 0, code); }

// last s in [0, num_segments) with cu[s] <= t (t < cu[num_segments])
__device__ __forceinline__ int segment_of(const int32_t* __restrict__ cu, int num_segments, int t) {
  int lo = 0, hi = num_segments;  // invariant: cu[lo] <= t < cu[hi]
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(&cu[mid]) <= t) lo = mid;
    else hi = mid;
  }
  return lo;
}

__global__ void __launch_bounds__(kThreads) grpo_loss_tokens(
    const float* __restrict__ logp, const float* __restrict__ old_logp, const float* __restrict__ ref_logp,
    const uint8_t* __restrict__ mask, const int32_t* __restrict__ cu_seqlens, const int32_t* __restrict__ seg_traj,
    int32_t num_segments, int32_t num_tokens, const float* __restrict__ adv, int32_t num_traj, float lo, float hi,
    float cap, float kl_coef, float inv_ntraj, float* __restrict__ dlogp, double* __restrict__ partial,
    int32_t* status) {
  double acc = 0.0;
  for (int base = blockIdx.x * kChunk; base < num_tokens; base += gridDim.x * kChunk) {
#pragma unroll
    for (int i = 0; i < kPerThread; ++i) {
      const int t = base + i * kThreads + threadIdx.x;
      if (t >= num_tokens) break;
      float g = 0.f;
      if (__ldg(&mask[t]) != 0) {
        const int s = segment_of(cu_seqlens, num_segments, t);
        const int b = __ldg(&seg_traj[s]);
        if (b < 0 || b >= num_traj) {
          set_status(status, VCS_ERR_DEVICE_CHECK);
        } else {
          const float A = __ldg(&adv[b]);
          const float lp = __ldg(&logp[t]);
          const float rho = expf(lp - __ldg(&old_logp[t]));
          float o, dobj;
          if (A >= 0.f) {
            if (rho <= hi) { o = rho * A; dobj = o; }
            else { o = hi * A; dobj = 0.f; }
          } else {
            if (rho < lo) { o = lo * A; dobj = 0.f; }
            else if (rho > cap) { o = cap * A; dobj = 0.f; }
            else { o = rho * A; dobj = o; }
          }
          const float r = __ldg(&ref_logp[t]) - lp;
          const float em1 = expm1f(r);
          acc += (double)(-o + kl_coef * (em1 - r));
          g = (-dobj - kl_coef * em1) * inv_ntraj;
        }
      }
      if (dlogp != nullptr) dlogp[t] = g;
    }
  }
  // block sum (double) in a fixed order
  __shared__ double red[kThreads / 32];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, off);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double sum = 0.0;
    for (int w = 0; w < kThreads / 32; ++w) sum += red[w];
    partial[blockIdx.x] = sum;
  }
}

__global__ void grpo_loss_finish(const double* __restrict__ partial, int nblocks, double inv_ntraj,
                                 double* __restrict__ loss) {
  __shared__ double red[32];
  double acc = 0.0;
  for (int i = threadIdx.x; i < nblocks; i += blockDim.x) acc += partial[i];
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_down_sync(0xffffffffu, acc, off);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double sum = 0.0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) sum += red[w];
    *loss = sum * inv_ntraj;
  }
}

// one thread per group: mean and population standard deviation in double
__global__ void group_advantage_kernel(const float* __restrict__ rewards, int64_t num_groups, int32_t group_size,
                                       float eps, float* __restrict__ adv) {
  for (int64_t gi = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; gi < num_groups;
       gi += (int64_t)gridDim.x * blockDim.x) {
    const float* r = rewards + gi * group_size;
    double mean = 0.0;
    for (int j = 0; j < group_size; ++j) mean += r[j];
    mean /= group_size;
    double var = 0.0;
    for (int j = 0; j < group_size; ++j) {
      const double d = r[j] - mean;
      var += d * d;
    }
    const double den = sqrt(var / group_size) + (double)eps;
    for (int j = 0; j < group_size; ++j) adv[gi * group_size + j] = (float)((r[j] - mean) / den);
  }
}

int loss_blocks(int64_t num_tokens) {
  int64_t b = (num_tokens + kChunk - 1) / kChunk;
  if (b < 1) b = 1;
  return (int)(b < kMaxBlocks ? b : kMaxBlocks);
}

}  // namespace

size_t grpo_loss_ws_bytes(int64_t num_tokens) { return kWsHeader + (size_t)loss_blocks(num_tokens) * sizeof(double); }

cudaError_t launch_grpo_loss(const float* logp, const float* old_logp, const float* ref_logp, const uint8_t* mask,
                             const int32_t* cu_seqlens, const int32_t* seg_traj, int32_t num_segments,
                             int32_t num_tokens, const float* adv, int32_t num_traj, float lo, float hi,
                             float clip_cap, float kl_coef, double* loss, float* dlogp, void* ws, cudaStream_t st) {
  int32_t* status = static_cast<int32_t*>(ws);
  double* partial = reinterpret_cast<double*>(static_cast<char*>(ws) + kWsHeader);
  const int nb = loss_blocks(num_tokens);
  cudaMemsetAsync(status, 0, sizeof(int32_t), st);
  grpo_loss_tokens<<<nb, kThreads, 0, st>>>(logp, old_logp, ref_logp, mask, cu_seqlens, seg_traj, num_segments,
                                            num_tokens, adv, num_traj, lo, hi, clip_cap,
                                            kl_coef, 1.f / (float)num_traj, dlogp, partial, status);
  grpo_loss_finish<<<1, 256, 0, st>>>(partial, nb, 1.0 / (double)num_traj, loss);
  return cudaGetLastError();
}

cudaError_t launch_group_advantage(const float* rewards, int64_t num_groups, int32_t group_size, float eps,
                                   float* adv, cudaStream_t st) {
  if (num_groups == 0) return cudaSuccess;
  int64_t blocks = (num_groups + 255) / 256;
  if (blocks > 152 * 8) blocks = 152 * 8;
  group_advantage_kernel<<<(unsigned)blocks, 256, 0, st>>>(rewards, num_groups, group_size, eps, adv);
  return cudaGetLastError();
}

}  // namespace vcs
