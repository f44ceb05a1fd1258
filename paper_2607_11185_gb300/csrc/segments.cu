// segments.cu - the Visual Context Segmentation layout builder (Sec. 3.4,
// Algorithm 1; App. C.1), as integer scans and a per-token expansion.
//
// Algorithm 1 keeps a running token stream per rollout and prunes it when the
// screenshot count exceeds K + delta.  Because a prune depends only on the
// number of steps seen, the segment boundaries have a closed form per
// trajectory (K = keep, delta = window, steps 1-based):
//   first segment: new steps 1..min(K+delta, T), screenshots for all of them;
//   segment j >= 1: new steps s_j = K+delta+(j-1)*delta+1 .. e_j =
//   min(s_j+delta-1, T); screenshots for a_j = max(1, s_j-K) .. e_j; steps
//   before a_j appear as their response tokens only (the fresh, re-tokenised
//   stream after a prune).
// Segment j's length is therefore
//   L_j = sum_{t<a_j} txt_t + sum_{t=a_j..e_j} (img_t + txt_t),
// which two global exclusive scans over the steps give in O(1).
//
// Kernels (all on the caller's stream, no host synchronisation):
//   seg_scan_steps  one CTA: exclusive scans of img+txt and txt over all steps
//   seg_traj_plan   one thread per trajectory: segment count, tokens, max length
//   seg_scan_traj   one CTA: scans over trajectories, totals, overflow and
//                   capacity checks, the vcs_sizes record
//   seg_write       one thread per trajectory: cu_seqlens, seg_traj and the
//                   per-segment step bounds used by the expansion
//   seg_expand      one warp per 4,096 segment tokens: gather index, source
//                   step, position, loss mask, streamed run by run (one run per
//                   step of the segment), 32 consecutive tokens per store
#include <climits>
#include <cstdint>

#include "internal.h"
#include "sm100.cuh"

namespace vcs {
namespace {

constexpr int kScanThreads = 1024;
constexpr int kScanItems = 4;

// Inclusive block-wide scan of two int64 values per thread; *tot receives the block totals.
__device__ void block_scan2(long long& a, long long& b, long long& tot_a, long long& tot_b) {
  __shared__ long long sa[32], sb[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nwarps = blockDim.x >> 5;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    long long ta = __shfl_up_sync(0xffffffffu, a, o);
    long long tb = __shfl_up_sync(0xffffffffu, b, o);
    if (lane >= o) {
      a += ta;
      b += tb;
    }
  }
  if (lane == 31) {
    sa[warp] = a;
    sb[warp] = b;
  }
  __syncthreads();
  if (warp == 0) {
    long long xa = lane < nwarps ? sa[lane] : 0, xb = lane < nwarps ? sb[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      long long ta = __shfl_up_sync(0xffffffffu, xa, o);
      long long tb = __shfl_up_sync(0xffffffffu, xb, o);
      if (lane >= o) {
        xa += ta;
        xb += tb;
      }
    }
    sa[lane] = xa;
    sb[lane] = xb;
  }
  __syncthreads();
  if (warp > 0) {
    a += sa[warp - 1];
    b += sb[warp - 1];
  }
  tot_a = sa[nwarps - 1];
  tot_b = sb[nwarps - 1];
  __syncthreads();
}

__device__ __forceinline__ void fail(int64_t* totals, int code) {
  atomicCAS(reinterpret_cast<unsigned long long*>(&totals[3]), 0ull, (unsigned long long)code);
}

__global__ void __launch_bounds__(kScanThreads) seg_scan_steps(const int32_t* __restrict__ step_img,
                                                                const int32_t* __restrict__ step_txt,
                                                                int64_t num_steps, SegWorkspace w) {
  long long carry_a = 0, carry_b = 0;
  for (int64_t base = 0; base < num_steps; base += (int64_t)kScanThreads * kScanItems) {
    const int64_t i0 = base + (int64_t)threadIdx.x * kScanItems;
    long long fa[kScanItems], fb[kScanItems];
    long long sa = 0, sb = 0;
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
      long long im = 0, tx = 0;
      if (i0 + i < num_steps) {
        im = step_img[i0 + i];
        tx = step_txt[i0 + i];
        if (im < 0 || tx < 0) {
          fail(w.totals, VCS_ERR_DEVICE_CHECK);
          im = im < 0 ? 0 : im;
          tx = tx < 0 ? 0 : tx;
        }
      }
      fa[i] = im + tx;
      fb[i] = tx;
      sa += fa[i];
      sb += fb[i];
    }
    long long ia = sa, ib = sb, ta, tb;
    block_scan2(ia, ib, ta, tb);
    long long ea = carry_a + ia - sa, eb = carry_b + ib - sb;
#pragma unroll
    for (int i = 0; i < kScanItems; ++i) {
      if (i0 + i < num_steps) {
        w.step_off[i0 + i] = ea;
        w.txt_pre[i0 + i] = eb;
      }
      ea += fa[i];
      eb += fb[i];
    }
    carry_a += ta;
    carry_b += tb;
  }
  if (threadIdx.x == 0) {
    w.step_off[num_steps] = carry_a;
    w.txt_pre[num_steps] = carry_b;
  }
}

// Segment j of a T-step trajectory: 1-based (a, s, e).
__device__ __forceinline__ void seg_bounds(int j, int T, int keep, int window, int& a, int& s, int& e) {
  if (j == 0) {
    s = 1;
    e = min(keep + window, T);
  } else {
    s = keep + window + (j - 1) * window + 1;
    e = min(s + window - 1, T);
  }
  a = max(1, s - keep);
}

__device__ __forceinline__ int seg_count(int T, int keep, int window) {
  if (T <= 0) return 0;
  if (T <= keep + window) return 1;
  return 1 + (T - keep - window + window - 1) / window;
}

__global__ void seg_traj_plan(const int32_t* __restrict__ cu_steps, int32_t num_traj, int64_t num_steps,
                              int32_t window, int32_t keep, SegWorkspace w) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= num_traj) return;
  const int64_t g0 = cu_steps[b], g1 = cu_steps[b + 1];
  bool ok = g0 >= 0 && g1 >= g0 && g1 <= num_steps && (b > 0 || g0 == 0) && (b < num_traj - 1 || g1 == num_steps);
  if (!ok) {
    fail(w.totals, VCS_ERR_DEVICE_CHECK);
    w.traj_nseg[b] = 0;
    w.traj_ntok[b] = 0;
    w.traj_maxlen[b] = 0;
    return;
  }
  const int T = (int)(g1 - g0);
  const int nseg = seg_count(T, keep, window);
  long long ntok = 0, maxlen = 0;
  for (int j = 0; j < nseg; ++j) {
    int a, s, e;
    seg_bounds(j, T, keep, window, a, s, e);
    const long long L =
        (w.txt_pre[g0 + a - 1] - w.txt_pre[g0]) + (w.step_off[g0 + e] - w.step_off[g0 + a - 1]);
    ntok += L;
    maxlen = L > maxlen ? L : maxlen;
  }
  if (maxlen > INT_MAX) fail(w.totals, VCS_ERR_OVERFLOW);
  w.traj_nseg[b] = nseg;
  w.traj_ntok[b] = ntok;
  w.traj_maxlen[b] = (int32_t)(maxlen > INT_MAX ? INT_MAX : maxlen);
}

__global__ void __launch_bounds__(kScanThreads) seg_scan_traj(int32_t num_traj, int64_t num_steps,
                                                               int64_t seg_capacity, int64_t tok_capacity,
                                                               vcs_sizes* sizes, SegWorkspace w) {
  __shared__ int smax[32];
  long long carry_a = 0, carry_b = 0;
  int mx = 0;
  for (int64_t i = threadIdx.x; i < num_traj; i += kScanThreads) mx = max(mx, w.traj_maxlen[i]);
  for (int o = 16; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if ((threadIdx.x & 31) == 0) smax[threadIdx.x >> 5] = mx;
  __syncthreads();
  if (threadIdx.x < 32) {
    mx = smax[threadIdx.x];
    for (int o = 16; o > 0; o >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  for (int64_t base = 0; base < num_traj; base += kScanThreads) {
    const int64_t i = base + threadIdx.x;
    long long a = i < num_traj ? w.traj_nseg[i] : 0;
    long long b = i < num_traj ? w.traj_ntok[i] : 0;
    long long ia = a, ib = b, ta, tb;
    block_scan2(ia, ib, ta, tb);
    if (i < num_traj) {
      w.seg_base[i] = carry_a + ia - a;
      w.tok_base[i] = carry_b + ib - b;
    }
    carry_a += ta;
    carry_b += tb;
  }
  if (threadIdx.x == 0) {
    w.seg_base[num_traj] = carry_a;
    w.tok_base[num_traj] = carry_b;
    if (carry_b > INT_MAX || w.step_off[num_steps] > INT_MAX) fail(w.totals, VCS_ERR_OVERFLOW);
    if (seg_capacity >= 0 && (carry_a > seg_capacity || carry_b > tok_capacity)) fail(w.totals, VCS_ERR_CAPACITY);
    w.totals[0] = carry_a;
    w.totals[1] = carry_b;
    w.totals[2] = mx;
    __threadfence();
    const int64_t status = atomicAdd(reinterpret_cast<unsigned long long*>(&w.totals[3]), 0ull);
    sizes->num_segments = carry_a;
    sizes->num_tokens = carry_b;
    sizes->max_seqlen = mx;
    sizes->status = (int32_t)status;
  }
}

__global__ void seg_write(const int32_t* __restrict__ cu_steps, int32_t num_traj, int32_t window, int32_t keep,
                          int32_t* __restrict__ cu_seqlens, int32_t* __restrict__ seg_traj, SegWorkspace w) {
  if (w.totals[3] != 0) return;
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b == 0) {
    cu_seqlens[w.totals[0]] = (int32_t)w.totals[1];
    w.seg_start[w.totals[0]] = w.totals[1];
  }
  if (b >= num_traj) return;
  const int g0 = cu_steps[b];
  const int T = cu_steps[b + 1] - g0;
  const int nseg = w.traj_nseg[b];
  int64_t start = w.tok_base[b];
  for (int j = 0; j < nseg; ++j) {
    int a, s, e;
    seg_bounds(j, T, keep, window, a, s, e);
    const int64_t seg = w.seg_base[b] + j;
    cu_seqlens[seg] = (int32_t)start;
    if (seg_traj != nullptr) seg_traj[seg] = b;
    w.seg_start[seg] = start;
    w.seg_first[seg] = g0;
    w.seg_full[seg] = g0 + a - 1;
    w.seg_new[seg] = g0 + s - 1;
    w.seg_last[seg] = g0 + e - 1;
    start += (w.txt_pre[g0 + a - 1] - w.txt_pre[g0]) + (w.step_off[g0 + e] - w.step_off[g0 + a - 1]);
  }
}

// Largest index u in [lo, hi] with arr[u] <= x (arr non-decreasing, arr[lo] <= x).
__device__ __forceinline__ int64_t last_le(const int64_t* __restrict__ arr, int64_t lo, int64_t hi, int64_t x) {
  while (lo < hi) {
    const int64_t mid = (lo + hi + 1) >> 1;
    if (__ldg(&arr[mid]) <= x)
      lo = mid;
    else
      hi = mid - 1;
  }
  return lo;
}

// One warp per chunk of kExpandChunk consecutive segment tokens.  A segment is a sequence of
// runs, one per step: the response tokens of each step before a_j (text-only history), then
// the screenshot-and-response tokens of each step a_j..e_j; inside a run the gather index,
// the position and the mask follow from the run's start, so the warp finds the run of its
// first token once (two binary searches, uniform across the lanes) and then streams the runs
// in order, the lanes writing 32 consecutive tokens per store.
constexpr int kExpandChunk = 4096;

__global__ void __launch_bounds__(256) seg_expand(const int32_t* __restrict__ step_img,
                                                  int32_t* __restrict__ tok_gather, int32_t* __restrict__ tok_src_step,
                                                  int32_t* __restrict__ tok_pos, uint8_t* __restrict__ tok_loss_mask,
                                                  SegWorkspace w) {
  if (w.totals[3] != 0) return;
  const int64_t nseg = w.totals[0], ntok = w.totals[1];
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t c = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); c * kExpandChunk < ntok;
       c += warps) {
    int64_t n = c * kExpandChunk;
    const int64_t nend = min(n + (int64_t)kExpandChunk, ntok);
    int64_t seg = last_le(w.seg_start, 0, nseg - 1, n);
    while (n < nend) {
      while (w.seg_start[seg + 1] <= n) ++seg;  // skip segments without tokens
      const int64_t start = w.seg_start[seg], next = w.seg_start[seg + 1];
      const int64_t g0 = w.seg_first[seg], A = w.seg_full[seg], S = w.seg_new[seg], E = w.seg_last[seg];
      const int64_t t0 = w.txt_pre[g0], H = w.txt_pre[A] - t0, f0 = w.step_off[A];
      // the run (step u) of position p = n - start, and its bounds [lo, hi) in the segment
      const int64_t p = n - start;
      int64_t u = p < H ? last_le(w.txt_pre, g0, A - 1, t0 + p) : last_le(w.step_off, A, E, f0 + (p - H));
      const int64_t send = min(next, nend);
      while (n < send) {
        const bool hist = u < A;
        const int64_t lo = hist ? w.txt_pre[u] - t0 : H + (w.step_off[u] - f0);
        const int64_t hi = hist ? w.txt_pre[u + 1] - t0 : H + (w.step_off[u + 1] - f0);
        const int64_t img = step_img[u];
        // token at position q of the run's step: history tokens are the step's response
        // tokens (after its screenshot); a full step's tokens start with the screenshot
        const int64_t g_base = hist ? w.step_off[u] + img - lo : w.step_off[u] - lo;
        const bool trainable_step = !hist && u >= S;
        const int64_t rend = min(start + hi, send);
        for (int64_t m = n + lane; m < rend; m += 32) {
          const int64_t q = m - start;
          tok_gather[m] = (int32_t)(g_base + q);
          tok_src_step[m] = (int32_t)u;
          tok_pos[m] = (int32_t)q;
          if (tok_loss_mask != nullptr) tok_loss_mask[m] = (trainable_step && q - lo >= img) ? 1 : 0;
        }
        n = max(n, rend);
        ++u;
      }
      ++seg;
    }
  }
}

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

}  // namespace

size_t seg_workspace_bytes(int32_t num_traj, int64_t num_steps) {
  const size_t S = (size_t)num_steps, B = (size_t)num_traj;
  size_t n = 0;
  n += align256((S + 1) * 8) * 2;       // step_off, txt_pre
  n += align256(B * 4) * 2;             // traj_nseg, traj_maxlen
  n += align256(B * 8);                 // traj_ntok
  n += align256((B + 1) * 8) * 2;       // seg_base, tok_base
  n += align256((S + 1) * 8);           // seg_start
  n += align256(S * 4) * 4;             // seg_full/new/last/first
  n += align256(4 * 8);                 // totals
  return n;
}

SegWorkspace seg_workspace_carve(void* ws, int32_t num_traj, int64_t num_steps) {
  const size_t S = (size_t)num_steps, B = (size_t)num_traj;
  char* p = static_cast<char*>(ws);
  auto take = [&](size_t bytes) {
    char* r = p;
    p += align256(bytes);
    return r;
  };
  SegWorkspace w;
  w.totals = reinterpret_cast<int64_t*>(take(4 * 8));
  w.step_off = reinterpret_cast<int64_t*>(take((S + 1) * 8));
  w.txt_pre = reinterpret_cast<int64_t*>(take((S + 1) * 8));
  w.traj_nseg = reinterpret_cast<int32_t*>(take(B * 4));
  w.traj_maxlen = reinterpret_cast<int32_t*>(take(B * 4));
  w.traj_ntok = reinterpret_cast<int64_t*>(take(B * 8));
  w.seg_base = reinterpret_cast<int64_t*>(take((B + 1) * 8));
  w.tok_base = reinterpret_cast<int64_t*>(take((B + 1) * 8));
  w.seg_start = reinterpret_cast<int64_t*>(take((S + 1) * 8));
  w.seg_full = reinterpret_cast<int32_t*>(take(S * 4));
  w.seg_new = reinterpret_cast<int32_t*>(take(S * 4));
  w.seg_last = reinterpret_cast<int32_t*>(take(S * 4));
  w.seg_first = reinterpret_cast<int32_t*>(take(S * 4));
  return w;
}

cudaError_t launch_seg_plan(const int32_t* cu_steps, int32_t num_traj, int64_t num_steps, const int32_t* step_img,
                            const int32_t* step_txt, int32_t window, int32_t keep, int64_t seg_capacity,
                            int64_t tok_capacity, vcs_sizes* sizes, const SegWorkspace& w, cudaStream_t st) {
  cudaError_t e = cudaMemsetAsync(w.totals, 0, 4 * sizeof(int64_t), st);
  if (e != cudaSuccess) return e;
  seg_scan_steps<<<1, kScanThreads, 0, st>>>(step_img, step_txt, num_steps, w);
  const int tb = 128;
  const int nb = num_traj > 0 ? (num_traj + tb - 1) / tb : 1;
  seg_traj_plan<<<nb, tb, 0, st>>>(cu_steps, num_traj, num_steps, window, keep, w);
  seg_scan_traj<<<1, kScanThreads, 0, st>>>(num_traj, num_steps, seg_capacity, tok_capacity, sizes, w);
  return cudaGetLastError();
}

cudaError_t launch_seg_build(const int32_t* cu_steps, int32_t num_traj, int32_t window, int32_t keep,
                             const int32_t* step_img, int32_t* cu_seqlens, int32_t* seg_traj, int32_t* tok_gather,
                             int32_t* tok_src_step, int32_t* tok_pos, uint8_t* tok_loss_mask,
                             const SegWorkspace& w, cudaStream_t st) {
  const int tb = 128;
  const int nb = num_traj > 0 ? (num_traj + tb - 1) / tb : 1;
  seg_write<<<nb, tb, 0, st>>>(cu_steps, num_traj, window, keep, cu_seqlens, seg_traj, w);
  seg_expand<<<152 * 16, 256, 0, st>>>(step_img, tok_gather, tok_src_step, tok_pos, tok_loss_mask, w);
  return cudaGetLastError();
}

}  // namespace vcs
