// attn_fwd.cu - causal grouped-query softmax attention forward over packed
// variable-length segments, for sm_103a (tcgen05 + TMEM + TMA).
//
// Every training segment that Algorithm 1 (Sec. 3.4) emits is an independent
// causal sequence; the packed buffer holds them back to back (cu_seqlens).
//   s_ij = scale <q_i, k_j> for j <= i in the same segment
//   o_i  = sum_j softmax_j(s_ij) v_j,   lse_i = ln sum_j exp(s_ij)
//
// Work unit (one CTA): a segment, a query head h, and a PAIR of consecutive
// 128-row query tiles (m0 = 2p, m1 = 2p+1).  Both tiles stream the same K/V
// tiles of kv-head h / (hq/hkv), so each K/V tile brought into shared memory
// feeds 256 query rows.  Tiles above the diagonal are never visited; only the
// diagonal tile is masked element-wise.
//
// Grid: two small kernels first list the launch's work units in device memory
// (fwd_item_scan counts each segment's pairs and checks the segment bounds,
// fwd_item_fill writes {start, end, pair, head} per unit), in the order
// (segment, kv-head, pair index from the last, query head in the group); CTA
// b takes unit b.  The CTAs sharing a K/V stream run together, so those tiles
// are read from HBM about once and then served from L2, and the longest pairs
// of each stream start first.  Pairs beyond a segment's end are not listed
// (a grid sized by the longest segment would launch them only to exit), and
// neither are pairs that prefix reuse copies from the previous segment; the
// grid is an upper bound of the count, and the few CTAs past it exit at once.
//
// Warp roles (384 threads):
//   warp 0      TMA producer: Q0/Q1 once, then K and V tiles into a 5-slot ring
//               (K runs one tile ahead of V: K0, K1, V0, K2, V1, ...)
//   warp 1      TMEM allocator and single-thread tcgen05.mma issuer
//   warps 2-3   idle (they keep the softmax warps on TMEM lane quadrants 0-3)
//   warps 4-7   softmax + epilogue for tile 0 (thread = query row)
//   warps 8-11  softmax + epilogue for tile 1
// TMEM (512 columns x 128 lanes, fp32): S0 [0,128), S1 [128,256),
// O0 [256,256+D), O1 [384,384+D).  P_k (bf16, two per column) overwrites the
// first 64 columns of S_k and is the A operand of O_k += P_k V read straight
// from TMEM, so P never touches shared memory.
//
// Per K/V tile j the MMA thread issues, for each tile k once its P_k(j) is in
// TMEM: O_k += P_k(j) V_j, then S_k(j+1) = Q_k K_{j+1}^T.  The tensor pipe
// executes in order, so the completion of S_k(j+1) also means that P_k(j) has
// been consumed and O_k is up to date, which is all the softmax warps wait
// for.  The two tiles alternate, so one tile's MMAs run while the other
// tile's softmax warps work.  The MMA thread commits only what the softmax
// warps wait for (a commit holds it, and the pipe, about as long as an MMA);
// the K/V ring slots are handed back to the producer by one softmax thread of
// the last tile, whose S(j+1) completing means their reads are done.  (The
// gathered variant, whose producer issues its loads more slowly, has them
// handed back by commits as soon as the MMAs are done.)  The ring order puts
// the two tiles step j reads, K_{j+1} and V_j, next to each other, so the
// tiled loads complete one barrier per step and the MMA thread waits once a
// step for its K/V, at the top of the step.
//
// Online softmax with a lazy running maximum: the row maximum used for P is
// only raised (and O, l rescaled) when a new tile's maximum exceeds it by more
// than 2^8 in the exp2 domain; otherwise P may reach 2^8, which bf16 and the
// fp32 accumulators hold without loss of relative precision.
#include <cfloat>
#include <cstdint>

#include "internal.h"
#include "sm100.cuh"

namespace vcs {
namespace {

using namespace dev;

constexpr int kThreads = 384;
// registers per thread after rebalancing: the producer/MMA warpgroup gives up
// what the two softmax warpgroups take (the block launches with 168)
constexpr int kRegLaunch = 168, kRegCtrl = 80, kRegSoftmax = 208;
static_assert(kRegCtrl + 2 * kRegSoftmax <= 3 * kRegLaunch, "setmaxnreg targets exceed the launch registers");
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct Fwd {
  static constexpr int BM = 128;
  static constexpr int BN = 128;
  static constexpr int KB = D / 64;                 // 128-byte column blocks per row
  static constexpr int TILE = BM * D * 2;           // bytes of a 128 x D bf16 tile
  static constexpr int BLOCK = BM * 128;            // bytes of one 128 x 64 column block
  static constexpr int NSLOT = 5;
  static constexpr int NGRP = 4;                    // ring-item group barriers (tiled loads)
  static constexpr int OFF_Q0 = 0;
  static constexpr int OFF_Q1 = TILE;
  static constexpr int OFF_KV = 2 * TILE;
  static constexpr int OFF_BAR = OFF_KV + NSLOT * TILE;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr int TM_S0 = 0, TM_S1 = 128, TM_O0 = 256, TM_O1 = 384;
  static constexpr uint32_t IDESC_S = idesc_bf16(128, 128, 0, 0);   // Q (K-major) x K^T (K-major)
  static constexpr uint32_t IDESC_PV = idesc_bf16(128, D, 0, 1);    // P (TMEM) x V (MN-major)
};
static_assert(Fwd<128>::SMEM <= 232448, "shared memory budget");

struct Bars {
  uint64_t q_full;
  uint64_t kv_full[5];   // per ring slot (gathered loads)
  uint64_t kv_empty[5];
  uint64_t grp_full[4];  // per pair of ring items consumed in one step (tiled loads)
  uint64_t s_full[2];
  uint64_t p_full[2];
  uint64_t o_done[2];
  uint32_t tmem_base;
  int32_t abort;
};

// workspace header: the number of listed work units sits after the status word
constexpr size_t kWsItemTotal = 128;

__device__ __forceinline__ void on_timeout(Bars* b, int32_t* status) {
  set_status(status, VCS_ERR_DEVICE_TIMEOUT);
  *reinterpret_cast<volatile int32_t*>(&b->abort) = 1;
}
__device__ __forceinline__ bool aborted(Bars* b) { return *reinterpret_cast<volatile int32_t*>(&b->abort) != 0; }

// S = Q K^T; qd, kd are K-major descriptors of the Q tile and the K tile.
template <int D>
__device__ __forceinline__ void issue_s(uint32_t tmem_d, uint64_t qd, uint64_t kd) {
  using C = Fwd<D>;
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    const uint32_t off = (kk >> 2) * C::BLOCK + (kk & 3) * 32;
    tc_mma_ss(tmem_d, desc_at(qd, off), desc_at(kd, off), C::IDESC_S, kk > 0);
  }
}

// O (+)= P V with P (128 x 128 keys, bf16) in TMEM columns p_tmem .. p_tmem+63;
// vd is the MN-major descriptor of the V tile.
template <int D>
__device__ __forceinline__ void issue_pv(uint32_t tmem_d, uint32_t p_tmem, uint64_t vd, bool accumulate) {
  using C = Fwd<D>;
  const uint32_t acc0 = accumulate ? 1u : 0u;
#pragma unroll
  for (int kk = 0; kk < C::BN / 16; ++kk)
    tc_mma_ts(tmem_d, p_tmem + kk * 8, desc_at(vd, kk * 16 * 128), C::IDESC_PV, kk > 0 ? 1u : acc0);
}

// Prefix reuse: rows [0, skip) of segment s, skip the shared prefix with segment s-1
// rounded down to whole pairs of query tiles, equal rows [0, skip) of segment s-1 and are
// copied from there instead of computed.  A shared length that segment s-1 cannot have
// (negative, longer than either segment, or given for segment 0) is recorded as a device
// check and read as 0.
__device__ __forceinline__ int reuse_skip_rows(const int32_t* __restrict__ seg_shared,
                                               const int32_t* __restrict__ cu_seqlens, int s, int32_t* status) {
  if (seg_shared == nullptr) return 0;
  const int sh = seg_shared[s];
  if (sh == 0) return 0;
  const int L = cu_seqlens[s + 1] - cu_seqlens[s];
  if (s == 0 || sh < 0 || sh > L || sh > cu_seqlens[s] - cu_seqlens[s - 1]) {
    set_status(status, VCS_ERR_DEVICE_CHECK);
    return 0;
  }
  return sh / 256 * 256;
}

// Pairs of query tiles of segment s the forward computes: none for a segment whose bounds are
// invalid (recorded as a device check), and none of those that prefix reuse copies from the
// previous segment.  Pairs [np - count, np) remain, np = ceil(L / 256).
__device__ __forceinline__ int seg_item_pairs(const int32_t* __restrict__ cu_seqlens, int32_t num_segments,
                                              int32_t num_tokens, int32_t max_seqlen,
                                              const int32_t* __restrict__ seg_shared, int s, int32_t* status) {
  const int start = cu_seqlens[s], end = cu_seqlens[s + 1];
  if (start < 0 || end < start || end > num_tokens || end - start > max_seqlen || (s == 0 && start != 0) ||
      (s == num_segments - 1 && end != num_tokens)) {
    set_status(status, VCS_ERR_DEVICE_CHECK);
    return 0;
  }
  const int np = (end - start + 255) / 256;
  return np - reuse_skip_rows(seg_shared, cu_seqlens, s, status) / 256;
}

// off[s] = hq * (pairs of segments 0 .. s-1), off[S] = *total: one block, in chunks of 1024
// segments (warp scans, then a scan of the warp sums), in 64-bit.  Consistent segments list at
// most `capacity` units (the workspace's room); segments that overlap, which only inconsistent
// bounds allow, can list more: the offsets are then clipped to the capacity, the count is 0 (no
// unit runs, so no CTA reads a unit the fill did not write) and the call records
// VCS_ERR_DEVICE_CHECK (already recorded for the inconsistent segment).
__global__ void __launch_bounds__(1024) fwd_item_scan(const int32_t* __restrict__ cu_seqlens, int32_t num_segments,
                                                      int32_t num_tokens, int32_t max_seqlen, int32_t hq,
                                                      const int32_t* __restrict__ seg_shared, int32_t capacity,
                                                      int32_t* __restrict__ off, int32_t* __restrict__ total,
                                                      int32_t* status) {
  __shared__ long long wsum[32];
  __shared__ long long carry;
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  if (threadIdx.x == 0) carry = 0;
  __syncthreads();
  for (int base = 0; base < num_segments; base += 1024) {
    const int s = base + (int)threadIdx.x;
    const long long cnt =
        s < num_segments
            ? (long long)hq * seg_item_pairs(cu_seqlens, num_segments, num_tokens, max_seqlen, seg_shared, s, status)
            : 0;
    long long x = cnt;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const long long y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane == 31) wsum[wid] = x;
    __syncthreads();
    if (wid == 0) {
      long long w = wsum[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, w, o);
        if (lane >= o) w += y;
      }
      wsum[lane] = w;
    }
    __syncthreads();
    const long long incl = carry + (wid > 0 ? wsum[wid - 1] : 0) + x;
    if (s < num_segments) off[s] = (int32_t)(incl - cnt < capacity ? incl - cnt : capacity);
    __syncthreads();
    if (threadIdx.x == 1023) carry = incl;
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const int32_t t = carry <= capacity ? (int32_t)carry : 0;
    if (carry > capacity) set_status(status, VCS_ERR_DEVICE_CHECK);
    off[num_segments] = t;
    *total = t;
  }
}

// The units of segment s at off[s] .. off[s+1]-1, in the order (kv head, pair from the last,
// query head in the group): {segment start, segment end, pair index, query head}.  A segment
// whose units would not all fit in the capacity (clipped by fwd_item_scan) writes none.
__global__ void __launch_bounds__(256) fwd_item_fill(const int32_t* __restrict__ cu_seqlens, int32_t num_segments,
                                                     int32_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv,
                                                     const int32_t* __restrict__ seg_shared, int32_t capacity,
                                                     const int32_t* __restrict__ off, int4* __restrict__ items,
                                                     int32_t* status) {
  const int G = hq / hkv;
  for (int s = blockIdx.x; s < num_segments; s += gridDim.x) {
    const int cnt = seg_item_pairs(cu_seqlens, num_segments, num_tokens, max_seqlen, seg_shared, s, status);
    const long long base = off[s], n = (long long)hq * cnt;
    if (cnt == 0 || base + n > capacity) continue;
    const int start = cu_seqlens[s], end = cu_seqlens[s + 1];
    const int np = (end - start + 255) / 256;  // pairs np - cnt .. np - 1
    for (int r = threadIdx.x; r < (int)n; r += blockDim.x) {
      const int hh = r % G, r2 = r / G;
      const int pr = r2 % cnt, g = r2 / cnt;
      items[base + r] = make_int4(start, end, np - 1 - pr, g * G + hh);
    }
  }
}

template <int D, bool GATHER>
__global__ void __launch_bounds__(kThreads, 1)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ CUtensorMap tm_v, const int4* __restrict__ items,
                    const int32_t* __restrict__ item_total, int32_t num_tokens, int32_t hq, int32_t hkv,
                    float scale_log2, __nv_bfloat16* __restrict__ out, float* __restrict__ lse,
                    int32_t* status, const int32_t* __restrict__ tok_gather, int32_t traj_tokens,
                    const __grid_constant__ CUtensorMap tm_qr, const __grid_constant__ CUtensorMap tm_kr,
                    const __grid_constant__ CUtensorMap tm_vr,
                    const __grid_constant__ CUtensorMap tm_qs, const __grid_constant__ CUtensorMap tm_ks,
                    const __grid_constant__ CUtensorMap tm_vs) {
  using C = Fwd<D>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + C::OFF_BAR);

  // CTA b takes listed unit b; the unit, the count and the status word are loaded together
  const int G = hq / hkv;
  const int4 e = items[blockIdx.x];
  const int total = *item_total;
  const int st = *reinterpret_cast<volatile int32_t*>(status);
  if ((int)blockIdx.x >= total) return;  // the grid is an upper bound of the listed units
  // once any CTA of this launch has given up on a wait, the rest stand down
  if (st == VCS_ERR_DEVICE_TIMEOUT) return;
  const int start = e.x, end = e.y, p = e.z, h = e.w, g = h / G;
  const int L = end - start;
  const int m0 = 2 * p, m1 = 2 * p + 1;
  const bool has1 = m1 * C::BM < L;
  const int nkv = has1 ? m1 + 1 : m0 + 1;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t sbase = smem_u32(smem);

  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    for (int i = 0; i < C::NSLOT; ++i) {
      mbar_init(&bars->kv_full[i], 1);
      mbar_init(&bars->kv_empty[i], 1);
    }
    for (int i = 0; i < C::NGRP; ++i) mbar_init(&bars->grp_full[i], 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->p_full[i], 128);
      mbar_init(&bars->o_done[i], 1);
    }
    bars->abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;

  if (warp < 4) {
    setmaxnreg_dec<kRegCtrl>();
    if (warp == 0 && (GATHER || lane == 0)) {
    // ------------------------------------------------------------ producer
      if constexpr (GATHER) {
        // the whole warp: lane 0 posts each tile's bytes and waits for free slots
        if (lane == 0) {
          tma_prefetch_desc(&tm_q);
          tma_prefetch_desc(&tm_k);
          tma_prefetch_desc(&tm_v);
          mbar_arrive_expect_tx(&bars->q_full, (has1 ? 2 : 1) * C::TILE);
        }
        __syncwarp();
        load_traj_tile<C::KB, C::BLOCK>(smem + C::OFF_Q0, &tm_q, &tm_qr, &tm_qs, &bars->q_full, h, D, start + m0 * C::BM, end - 1,
                                     tok_gather, traj_tokens, status, lane);
        if (has1)
          load_traj_tile<C::KB, C::BLOCK>(smem + C::OFF_Q1, &tm_q, &tm_qr, &tm_qs, &bars->q_full, h, D, start + m1 * C::BM, end - 1,
                                       tok_gather, traj_tokens, status, lane);
        for (int c = 0; c < 2 * nkv; ++c) {
          const bool is_v = c == 2 * nkv - 1 || (c > 0 && (c & 1) == 0);
          const int j = c == 2 * nkv - 1 ? nkv - 1 : (is_v ? (c - 2) >> 1 : (c + 1) >> 1);
          const int slot = c % C::NSLOT, round = c / C::NSLOT;
          int go = 1;
          if (lane == 0) {
            if (c >= C::NSLOT && !mbar_wait(&bars->kv_empty[slot], (round - 1) & 1)) {
              on_timeout(bars, status);
              go = 0;
            } else if (aborted(bars)) {
              go = 0;
            } else {
              mbar_arrive_expect_tx(&bars->kv_full[slot], C::TILE);
            }
          }
          if (!__shfl_sync(0xffffffffu, go, 0)) break;
          load_traj_tile<C::KB, C::BLOCK>(smem + C::OFF_KV + slot * C::TILE, is_v ? &tm_v : &tm_k,
                                          is_v ? &tm_vr : &tm_kr, is_v ? &tm_vs : &tm_ks, &bars->kv_full[slot], g, D, start + j * C::BN,
                                          end - 1, tok_gather, traj_tokens, status, lane);
        }
      } else {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_k);
        tma_prefetch_desc(&tm_v);
        mbar_arrive_expect_tx(&bars->q_full, (has1 ? 2 : 1) * C::TILE);
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb) {
          tma_load_3d(smem + C::OFF_Q0 + kb * C::BLOCK, &tm_q, &bars->q_full, kb * 64, h, start + m0 * C::BM);
          if (has1)
            tma_load_3d(smem + C::OFF_Q1 + kb * C::BLOCK, &tm_q, &bars->q_full, kb * 64, h, start + m1 * C::BM);
        }
        const uint64_t keep_l2 = l2_policy_evict_last();
        // ring order K0, K1, V0, K2, V1, ..., K_{n-1}, V_{n-2}, V_{n-1}
        for (int c = 0; c < 2 * nkv; ++c) {
          const bool is_v = c == 2 * nkv - 1 || (c > 0 && (c & 1) == 0);
          const int j = c == 2 * nkv - 1 ? nkv - 1 : (is_v ? (c - 2) >> 1 : (c + 1) >> 1);
          const int slot = c % C::NSLOT, round = c / C::NSLOT;
          if (c >= C::NSLOT && !mbar_wait(&bars->kv_empty[slot], (round - 1) & 1)) {
            on_timeout(bars, status);
            break;
          }
          if (aborted(bars)) break;
          // items 2m-1, 2m (K_m, V_{m-1}) are the ones step m-1 consumes: they complete one
          // barrier, armed for both by the first; group 0 (K_0) and group nkv (V_{nkv-1})
          // hold one item
          const int m = (c + 1) >> 1;
          uint64_t* gb = &bars->grp_full[m % C::NGRP];
          if (c == 0 || (c & 1)) mbar_arrive_expect_tx(gb, (m == 0 || m == nkv ? 1 : 2) * C::TILE);
          const CUtensorMap* tm = is_v ? &tm_v : &tm_k;
#pragma unroll
          for (int kb = 0; kb < C::KB; ++kb)
            tma_load_3d_hint(smem + C::OFF_KV + slot * C::TILE + kb * C::BLOCK, tm, gb, kb * 64, g, start + j * C::BN,
                             keep_l2);
        }
      }
    } else if (warp == 1 && lane == 0) {
    // ------------------------------------------------------------ MMA issuer
      bool ok = mbar_wait(&bars->q_full, 0);
      // descriptors built once; the issue loops only add compile-time offsets
      const uint64_t q0d = smem_desc(sbase + C::OFF_Q0, 16, 1024), q1d = desc_at(q0d, C::TILE);
      const uint64_t kv_kmaj = smem_desc(sbase + C::OFF_KV, 16, 1024);
      const uint64_t kv_mnmaj = smem_desc(sbase + C::OFF_KV, C::BLOCK, 1024);
      // positions of K_j and V_j in the producer's ring order, and their slots' byte offsets
      auto k_item = [&](int j) { return j == 0 ? 0 : 2 * j - 1; };
      auto v_item = [&](int j) { return j == nkv - 1 ? 2 * nkv - 1 : 2 * j + 2; };
      auto k_off = [&](int j) { return (uint32_t)((k_item(j) % C::NSLOT) * C::TILE); };
      auto v_off = [&](int j) { return (uint32_t)((v_item(j) % C::NSLOT) * C::TILE); };
      // tiled loads: group m holds K_m and V_{m-1} (group 0 only K_0, group nkv only
      // V_{nkv-1}); gathered loads: one barrier per ring item
      auto acquire_group = [&](int m) -> bool {
        if constexpr (GATHER) {
          if (m < nkv && !mbar_wait(&bars->kv_full[k_item(m) % C::NSLOT], (k_item(m) / C::NSLOT) & 1)) return false;
          if (m > 0 && !mbar_wait(&bars->kv_full[v_item(m - 1) % C::NSLOT], (v_item(m - 1) / C::NSLOT) & 1))
            return false;
        } else {
          if (!mbar_wait(&bars->grp_full[m % C::NGRP], (m / C::NGRP) & 1)) return false;
        }
        tc_fence_after();
        return true;
      };
      uint32_t kaddr = k_off(0), vaddr = 0;  // slot byte offsets of K_{j+1} and V_j
      if (ok) ok = acquire_group(0);
      if (ok) {
        issue_s<D>(tmem + C::TM_S0, q0d, desc_at(kv_kmaj, kaddr));
        tc_commit(&bars->s_full[0]);
        if (has1) {
          issue_s<D>(tmem + C::TM_S1, q1d, desc_at(kv_kmaj, kaddr));
          tc_commit(&bars->s_full[1]);
        }
        if constexpr (GATHER) tc_commit(&bars->kv_empty[0]);
      }
      // step j reads V_j and K_{j+1}, one group: acquired at the top of the step, one wait a
      // step (a barrier wait stalls the issuing thread for hundreds of cycles while the pipe
      // streams from shared memory, so the fewer the better), a step after the producer asked
      // for it
      for (int j = 0; ok && j < nkv; ++j) {
        const bool next = j + 1 < nkv;
        if (!acquire_group(j + 1)) { ok = false; break; }
        vaddr = v_off(j);
        if (next) kaddr = k_off(j + 1);
        // tile 0: O0 += P0(j) V_j, then S0(j+1)
        if (j <= m0) {
          if (!mbar_wait(&bars->p_full[0], j & 1)) { ok = false; break; }
          tc_fence_after();
          issue_pv<D>(tmem + C::TM_O0, tmem + C::TM_S0, desc_at(kv_mnmaj, vaddr), j > 0);
          if (next && j + 1 <= m0) {
            issue_s<D>(tmem + C::TM_S0, q0d, desc_at(kv_kmaj, kaddr));
            tc_commit(&bars->s_full[0]);
          } else {
            tc_commit(&bars->o_done[0]);
          }
        }
        // tile 1
        if (has1) {
          if (!mbar_wait(&bars->p_full[1], j & 1)) { ok = false; break; }
          tc_fence_after();
          issue_pv<D>(tmem + C::TM_O1, tmem + C::TM_S1, desc_at(kv_mnmaj, vaddr), j > 0);
          if (next) {
            issue_s<D>(tmem + C::TM_S1, q1d, desc_at(kv_kmaj, kaddr));
            tc_commit(&bars->s_full[1]);
          } else {
            tc_commit(&bars->o_done[1]);
          }
        }
        if constexpr (GATHER) {
          // the gathering producer needs its slots back as soon as the MMAs are done with them
          if (next) tc_commit(&bars->kv_empty[k_item(j + 1) % C::NSLOT]);
          tc_commit(&bars->kv_empty[v_item(j) % C::NSLOT]);
        }
      }
      if (!ok) on_timeout(bars, status);
    }
  } else {
    // ------------------------------------------------------------ softmax
    setmaxnreg_inc<kRegSoftmax>();
    const int wg = (warp - 4) >> 2;
    const int quad = warp & 3;
    const int r = quad * 32 + lane;  // query row within the tile
    if (wg == 0 || has1) {
      const int mt = wg == 0 ? m0 : m1;
      const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
      const uint32_t s_col = wg == 0 ? C::TM_S0 : C::TM_S1;
      const uint32_t o_col = wg == 0 ? C::TM_O0 : C::TM_O1;
      const uint64_t sc2 = f2pack(scale_log2, scale_log2);
      float m_run = -FLT_MAX, l = 0.f;
      bool ok = true;
      // The K/V ring slots are handed back from here rather than by commits of the MMA thread
      // (a tcgen05.commit holds that thread, and the tensor pipe, for about as long as an MMA):
      // once S_k(j) of the last tile is complete, in-order execution has also completed every
      // MMA that reads K_j (the S(j) of both tiles) and V_{j-1} (the P V of both tiles at
      // step j-1), so one thread of that tile's warpgroup frees their slots.  The last V_{n-1}
      // is not handed back: the producer has issued every load by then.
      const bool releaser = !GATHER && (has1 ? wg == 1 : wg == 0) && quad == 0 && lane == 0;
      for (int j = 0; j <= mt; ++j) {
        // S(j) complete also means P(j-1) was consumed and O holds P(j-1) V.  The wait's
        // outcome is the warp's: the TMEM loads and votes below are warp-collective.
        if (!mbar_wait_warp(&bars->s_full[wg], j & 1)) { ok = false; break; }
        if (releaser) {
          // ring items: K_j is 0 for j = 0, else 2j-1; V_{j-1} is 2(j-1)+2 = 2j (j-1 < nkv-1 here)
          mbar_arrive(&bars->kv_empty[(j == 0 ? 0 : 2 * j - 1) % C::NSLOT]);
          if (j > 0) mbar_arrive(&bars->kv_empty[(2 * j) % C::NSLOT]);
        }
        tc_fence_after();
        uint32_t s[128];
#pragma unroll
        for (int c = 0; c < 4; ++c)
          tmem_ld_32x32b_x32(trow + s_col + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&s[c * 32]));
        tmem_ld_wait();
        reg_fence<128>(s);
        if (j == mt) {  // diagonal tile: key c is visible to row r iff c <= r
#pragma unroll
          for (int c = 0; c < 128; ++c)
            if (c > r) s[c] = __float_as_uint(-FLT_MAX);
        }
        // row maximum: 8 independent three-input chains
        float pm[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) pm[u] = fmaxf(__uint_as_float(s[2 * u]), __uint_as_float(s[2 * u + 1]));
#pragma unroll
        for (int c = 16; c < 128; c += 16)
#pragma unroll
          for (int u = 0; u < 8; ++u)
            pm[u] = fmax3(pm[u], __uint_as_float(s[c + 2 * u]), __uint_as_float(s[c + 2 * u + 1]));
        const float mx = fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7]));
        const float mx2 = mx * scale_log2;
        float alpha = 1.f;
        bool rescale = false;
        if (j == 0) {
          m_run = mx2;
        } else if (mx2 > m_run + kRescaleThreshold) {
          alpha = ex2(m_run - mx2);
          m_run = mx2;
          rescale = true;
        }
        // P = exp2(s*scale*log2e - m) as bf16 pairs, packed over S; the
        // scale-and-shift and the row sums run on packed fp32 pairs
        const uint64_t nm2 = f2pack(-m_run, -m_run);
        uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
        for (int c2 = 0; c2 < 64; ++c2) {
          float x0, x1;
          f2unpack(ffma2(f2pack(__uint_as_float(s[2 * c2]), __uint_as_float(s[2 * c2 + 1])), sc2, nm2), x0, x1);
          const float p0 = ex2(x0), p1 = ex2(x1);
          acc[c2 & 3] = fadd2(acc[c2 & 3], f2pack(p0, p1));
          s[c2] = pack_bf16(p0, p1);
        }
        float a0, a1, b0, b1;
        f2unpack(fadd2(acc[0], acc[1]), a0, a1);
        f2unpack(fadd2(acc[2], acc[3]), b0, b1);
        l = l * alpha + ((a0 + a1) + (b0 + b1));
        // P over the first 64 columns of S (the MMA reads it from there)
        tmem_st_32x32b_x32(trow + s_col, *reinterpret_cast<uint32_t(*)[32]>(&s[0]));
        tmem_st_32x32b_x32(trow + s_col + 32, *reinterpret_cast<uint32_t(*)[32]>(&s[32]));
        if (j > 0 && __any_sync(0xffffffffu, rescale)) {
          const uint64_t al2 = f2pack(alpha, alpha);
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            uint32_t o[32];
            tmem_ld_32x32b_x32(trow + o_col + c * 32, o);
            tmem_ld_wait();
            reg_fence<32>(o);
#pragma unroll
            for (int e = 0; e < 32; e += 2) {
              float x0, x1;
              f2unpack(fmul2(f2pack(__uint_as_float(o[e]), __uint_as_float(o[e + 1])), al2), x0, x1);
              o[e] = __float_as_uint(x0);
              o[e + 1] = __float_as_uint(x1);
            }
            tmem_st_32x32b_x32(trow + o_col + c * 32, o);
          }
        }
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(&bars->p_full[wg]);
        if (__any_sync(0xffffffffu, aborted(bars))) { ok = false; break; }
      }
      if (ok) ok = mbar_wait_warp(&bars->o_done[wg], 0);
      if (!ok) {
        on_timeout(bars, status);
      } else {
        tc_fence_after();
        const int row = mt * C::BM + r;
        const bool valid = row < L;
        const float inv_l = 1.f / l;
        const uint64_t il2 = f2pack(inv_l, inv_l);
        __nv_bfloat16* orow = out + ((size_t)(start + row) * hq + h) * D;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld_32x32b_x32(trow + o_col + c * 32, o);
          tmem_ld_wait();
          reg_fence<32>(o);
          uint32_t pk[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) {
            float x0, x1;
            f2unpack(fmul2(f2pack(__uint_as_float(o[2 * e]), __uint_as_float(o[2 * e + 1])), il2), x0, x1);
            pk[e] = pack_bf16(x0, x1);
          }
          if (valid) {
            uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
            for (int v4 = 0; v4 < 4; ++v4) dst[v4] = make_uint4(pk[4 * v4], pk[4 * v4 + 1], pk[4 * v4 + 2], pk[4 * v4 + 3]);
          }
        }
        if (valid) lse[(size_t)h * num_tokens + start + row] = (m_run + lg2(l)) * 0.69314718055994531f;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Prefix reuse: O and lse of the rows the forward skipped, from the segment that computed
// them (walk back through the previous segments while the row lies in their skipped
// prefix).  One warp per segment token; 16-byte pieces of the O row, then the lse values.
__global__ void __launch_bounds__(256) fwd_reuse_copy(const int32_t* __restrict__ cu_seqlens, int32_t num_segments,
                                                      int32_t num_tokens, const int32_t* __restrict__ seg_shared,
                                                      int32_t hq, int32_t d, __nv_bfloat16* __restrict__ out,
                                                      float* __restrict__ lse, int32_t* status) {
  const int warps = gridDim.x * 8;
  const int lane = threadIdx.x & 31;
  for (int n = blockIdx.x * 8 + (threadIdx.x >> 5); n < num_tokens; n += warps) {
    int lo = 0, hi = num_segments - 1;  // the segment s with cu[s] <= n < cu[s+1]
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (cu_seqlens[mid] <= n) lo = mid;
      else hi = mid - 1;
    }
    const int r = n - cu_seqlens[lo];
    int src = lo;
    while (r < reuse_skip_rows(seg_shared, cu_seqlens, src, status)) --src;
    if (src == lo) continue;
    const int m = cu_seqlens[src] + r;  // the same row of the segment that computed it
    const int chunks = hq * d / 8;
    const uint4* from = reinterpret_cast<const uint4*>(out + (size_t)m * hq * d);
    uint4* to = reinterpret_cast<uint4*>(out + (size_t)n * hq * d);
    for (int c = lane; c < chunks; c += 32) to[c] = from[c];
    for (int h = lane; h < hq; h += 32) lse[(size_t)h * num_tokens + n] = lse[(size_t)h * num_tokens + m];
  }
}

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Upper bound of a launch's work units: hq * sum_s ceil(L_s / 256) <= hq * (T / 256 + S + 1).
inline int64_t fwd_max_items(const AttnArgs& a) {
  return (int64_t)a.hq * (a.num_tokens / 256 + (int64_t)a.num_segments + 1);
}

template <int D, bool GATHER>
cudaError_t launch_fwd_d(const AttnArgs& a, void* o, float* lse, void* ws, cudaStream_t st) {
  using C = Fwd<D>;
  alignas(64) CUtensorMap tq, tk, tv, tqr, tkr, tvr, tqs, tks, tvs;
  if (GATHER) {
    if (!encode_tma_rows_bf16(&tq, a.q, (uint64_t)a.hq * D, a.traj_tokens) ||
        !encode_tma_rows_bf16(&tk, a.k, (uint64_t)a.hkv * D, a.traj_tokens) ||
        !encode_tma_rows_bf16(&tv, a.v, (uint64_t)a.hkv * D, a.traj_tokens) ||
        !encode_tma_3d_bf16(&tqr, a.q, D, a.hq, a.traj_tokens, 64, 128) ||
        !encode_tma_3d_bf16(&tkr, a.k, D, a.hkv, a.traj_tokens, 64, 128) ||
        !encode_tma_3d_bf16(&tvr, a.v, D, a.hkv, a.traj_tokens, 64, 128) ||
        !encode_tma_3d_bf16(&tqs, a.q, D, a.hq, a.traj_tokens, 64, 32) ||
        !encode_tma_3d_bf16(&tks, a.k, D, a.hkv, a.traj_tokens, 64, 32) ||
        !encode_tma_3d_bf16(&tvs, a.v, D, a.hkv, a.traj_tokens, 64, 32))
      return cudaErrorInvalidValue;
  } else if (!encode_tma_3d_bf16(&tq, a.q, D, a.hq, a.num_tokens, 64, 128) ||
             !encode_tma_3d_bf16(&tk, a.k, D, a.hkv, a.num_tokens, 64, 128) ||
             !encode_tma_3d_bf16(&tv, a.v, D, a.hkv, a.num_tokens, 64, 128)) {
    return cudaErrorInvalidValue;
  }
  static std::atomic<int> regs_cache{-1};
  bool regs_ok = false;
  if (cudaError_t e = launch_regs_match(reinterpret_cast<const void*>(attn_fwd_kernel<D, GATHER>), kRegLaunch,
                                        &regs_cache, &regs_ok);
      e != cudaSuccess)
    return e;
  if (!regs_ok) return cudaErrorInvalidConfiguration;
  cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel<D, GATHER>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const int64_t max_items = fwd_max_items(a);
  if (max_items > INT32_MAX) return cudaErrorInvalidConfiguration;
  // workspace: header (status word, unit count), off[S+1], the units
  char* w = static_cast<char*>(ws);
  int32_t* total = reinterpret_cast<int32_t*>(w + kWsItemTotal);
  int32_t* off = reinterpret_cast<int32_t*>(w + kWsHeader);
  int4* items = reinterpret_cast<int4*>(w + kWsHeader + align256(((size_t)a.num_segments + 1) * 4));
  fwd_item_scan<<<1, 1024, 0, st>>>(a.cu_seqlens, a.num_segments, (int32_t)a.num_tokens, a.max_seqlen, a.hq,
                                    a.seg_shared, (int32_t)max_items, off, total, a.status);
  const int fill_blocks = a.num_segments < 152 * 8 ? a.num_segments : 152 * 8;
  fwd_item_fill<<<fill_blocks, 256, 0, st>>>(a.cu_seqlens, a.num_segments, (int32_t)a.num_tokens, a.max_seqlen,
                                             a.hq, a.hkv, a.seg_shared, (int32_t)max_items, off, items, a.status);
  const float scale_log2 = a.scale * 1.4426950408889634f;
  attn_fwd_kernel<D, GATHER><<<(unsigned)max_items, kThreads, C::SMEM, st>>>(
      tq, tk, tv, items, total, (int32_t)a.num_tokens, a.hq, a.hkv, scale_log2, static_cast<__nv_bfloat16*>(o),
      lse, a.status, a.tok_gather, (int32_t)a.traj_tokens, GATHER ? tqr : tq, GATHER ? tkr : tk,
      GATHER ? tvr : tv, GATHER ? tqs : tq, GATHER ? tks : tk, GATHER ? tvs : tv);
  if (a.seg_shared != nullptr) {
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    int64_t blocks = (a.num_tokens + 7) / 8;
    if (blocks > 152 * 16) blocks = 152 * 16;
    fwd_reuse_copy<<<(unsigned)blocks, 256, 0, st>>>(a.cu_seqlens, a.num_segments, (int32_t)a.num_tokens,
                                                     a.seg_shared, a.hq, D, static_cast<__nv_bfloat16*>(o), lse,
                                                     a.status);
  }
  return cudaGetLastError();
}

}  // namespace

// Header (status word, unit count), the per-segment unit offsets and the list of work units
// (16 bytes each).
size_t attn_fwd_ws_bytes(const AttnArgs& a) {
  const int64_t items = fwd_max_items(a);
  return kWsHeader + align256(((size_t)(a.num_segments > 0 ? a.num_segments : 0) + 1) * 4) +
         align256((size_t)(items > 0 ? items : 0) * 16);
}

cudaError_t launch_attn_fwd(const AttnArgs& a, void* o, float* lse, void* ws, cudaStream_t st) {
  if (a.tok_gather != nullptr) {
    if (a.d == 64) return launch_fwd_d<64, true>(a, o, lse, ws, st);
    return launch_fwd_d<128, true>(a, o, lse, ws, st);
  }
  if (a.d == 64) return launch_fwd_d<64, false>(a, o, lse, ws, st);
  return launch_fwd_d<128, false>(a, o, lse, ws, st);
}

}  // namespace vcs
