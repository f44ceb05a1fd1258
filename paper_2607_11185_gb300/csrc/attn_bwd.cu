// attn_bwd.cu - backward of the packed-segment causal GQA attention, sm_103a.
//
// For an upstream gradient dO of o_i = sum_j P_ij v_j (P the causal softmax of
// s_ij = scale <q_i, k_j> within one segment):
//   D_i   = <dO_i, o_i>
//   dP_ij = <dO_i, v_j>,   dS_ij = P_ij (dP_ij - D_i)
//   dq_i  = scale sum_j dS_ij k_j
//   dk_j  = scale sum_{h in group} sum_i dS_ij q_i
//   dv_j  = sum_{h in group} sum_i P_ij dO_i
// P is recomputed from the forward's log-sum-exp: P_ij = exp(s_ij - lse_i).
//
// Three kernels on the caller's stream:
//   bwd_pre     D = rowsum(dO * O) (fp32, [hq, N]) and zeroes the fp32 dQ accumulator
//   bwd_main    one CTA per (segment, 128-key tile n, kv-head g); loops over the
//               G query heads of the group and the query tiles m >= n.  dK and
//               dV of the tile accumulate in TMEM across the whole loop (GQA head
//               sharing: the K/V tile is loaded once for all G heads); the dQ
//               contribution of every (m, h) is added to the fp32 accumulator
//               with vector reductions.
//   bwd_dq_cvt  fp32 dQ accumulator -> bf16 dq
//
// bwd_main per (m, h), with the key rows of the tile on TMEM lanes:
//   St  = K_n Q_m^T                 (TMEM cols [0,128))
//   dPt = V_n dO_m^T                (TMEM cols [128,256))
//   compute warps: Pt = exp2(St*scale*log2e - lse*log2e) (causal + validity mask),
//                  dSt = scale * Pt * (dPt - D); both to shared memory as bf16
//   dV += Pt dO_m, dK += dSt Q_m    (TMEM cols [256,256+D), [384,384+D))
//   dQ  = dSt^T K_n                 (TMEM cols [0,D), reusing St)
//   compute warps: dQ rows (query rows on TMEM lanes) -> red.global.add.v4.f32
// Warp roles as in the forward: warp 0 TMA, warp 1 MMA, warps 4-11 compute
// (two warpgroups, each owning half of the 128 query columns / D columns).
// For head_dim 128, bwd_main_d128 replaces bwd_main: P^T kept in TMEM, dQ
// computed with query rows on TMEM lanes, and a fourth warpgroup that drains it
// with TMA bulk reduce-adds (described at the kernel).
#include <cfloat>
#include <cstdint>

#include "internal.h"
#include "sm100.cuh"

namespace vcs {
namespace {

using namespace dev;

constexpr int kThreads = 384;
constexpr int kPreThreads = 256;

template <int D>
struct Bwd {
  static constexpr int BM = 128;                 // key rows of the tile
  static constexpr int BN = 128;                 // query rows per iteration
  static constexpr int KB = D / 64;
  static constexpr int TILE = BM * D * 2;
  static constexpr int BLOCK = BM * 128;
  static constexpr int PTILE = BM * BN * 2;
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = TILE;
  static constexpr int OFF_Q = 2 * TILE;
  static constexpr int OFF_DO = 3 * TILE;
  static constexpr int OFF_PT = 4 * TILE;
  static constexpr int OFF_DST = OFF_PT + PTILE;
  static constexpr int OFF_ROW = OFF_DST + PTILE;        // lse2[2][128], dvec[2][128] fp32
  static constexpr int OFF_BAR = OFF_ROW + 4 * 128 * 4;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr int TM_ST = 0, TM_DPT = 128, TM_DV = 256, TM_DK = 384, TM_DQ = 0;
  static constexpr uint32_t IDESC_S = idesc_bf16(128, 128, 0, 0);   // K (K-major) x Q^T (K-major)
  static constexpr uint32_t IDESC_KV = idesc_bf16(128, D, 0, 1);    // Pt/dSt (K-major) x dO/Q (MN-major)
  static constexpr uint32_t IDESC_DQ = idesc_bf16(128, D, 1, 1);    // dS (MN-major) x K (MN-major)
};

struct BwdBars {
  uint64_t kv_full;
  uint64_t qdo_full;
  uint64_t qdo_empty;
  uint64_t s_full;
  uint64_t p_full;
  uint64_t dq_full;
  uint64_t dq_free;
  uint32_t tmem_base;
  int32_t abort;
};

__device__ __forceinline__ void on_timeout(BwdBars* b, int32_t* status) {
  set_status(status, VCS_ERR_DEVICE_TIMEOUT);
  *reinterpret_cast<volatile int32_t*>(&b->abort) = 1;
}
__device__ __forceinline__ bool aborted(BwdBars* b) {
  return *reinterpret_cast<volatile int32_t*>(&b->abort) != 0;
}

__device__ __forceinline__ void red_add_v4(float* p, float a, float b, float c, float d) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(a), "f"(b), "f"(c), "f"(d) : "memory");
}

// ------------------------------------------------------------------ bwd_pre
// One 16-byte chunk (8 elements) per thread; D/8 consecutive threads share a row.
template <int D>
__global__ void __launch_bounds__(kPreThreads) bwd_pre(const __nv_bfloat16* __restrict__ o,
                                                       const __nv_bfloat16* __restrict__ dout, int64_t rows,
                                                       int32_t hq, int64_t num_tokens, float* __restrict__ dvec,
                                                       float* __restrict__ dq_acc) {
  constexpr int CPR = D / 8;  // chunks per row
  const int64_t total = rows * CPR;
  for (int64_t c = blockIdx.x * (int64_t)kPreThreads + threadIdx.x; c - threadIdx.x < total;
       c += (int64_t)gridDim.x * kPreThreads) {
    float acc = 0.f;
    if (c < total) {
      const uint4 a = __ldg(reinterpret_cast<const uint4*>(o) + c);
      const uint4 b = __ldg(reinterpret_cast<const uint4*>(dout) + c);
      const __nv_bfloat162* pa = reinterpret_cast<const __nv_bfloat162*>(&a);
      const __nv_bfloat162* pb = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const float2 fa = __bfloat1622float2(pa[e]);
        const float2 fb = __bfloat1622float2(pb[e]);
        acc = fmaf(fa.x, fb.x, acc);
        acc = fmaf(fa.y, fb.y, acc);
      }
      float4* z = reinterpret_cast<float4*>(dq_acc) + 2 * c;
      z[0] = make_float4(0.f, 0.f, 0.f, 0.f);
      z[1] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int off = CPR / 2; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
    if (c < total && (c % CPR) == 0) {
      const int64_t row = c / CPR;           // row = token * hq + head
      const int64_t tok = row / hq;
      const int64_t h = row - tok * hq;
      dvec[h * num_tokens + tok] = acc;
    }
  }
}

// ------------------------------------------------------------------ bwd_dq_cvt
__global__ void __launch_bounds__(256) bwd_dq_cvt(const float* __restrict__ acc, __nv_bfloat16* __restrict__ dq,
                                                  int64_t n8) {
  for (int64_t c = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; c < n8; c += (int64_t)gridDim.x * blockDim.x) {
    const float4 a = __ldg(reinterpret_cast<const float4*>(acc) + 2 * c);
    const float4 b = __ldg(reinterpret_cast<const float4*>(acc) + 2 * c + 1);
    uint4 r;
    r.x = pack_bf16(a.x, a.y);
    r.y = pack_bf16(a.z, a.w);
    r.z = pack_bf16(b.x, b.y);
    r.w = pack_bf16(b.z, b.w);
    reinterpret_cast<uint4*>(dq)[c] = r;
  }
}

// ------------------------------------------------------------------ bwd_dq_scatter
// Gathered backward: dq_traj[tok_gather[n]] += dq_acc[n] (fp32, all heads of the row), one
// 16-byte chunk per thread; a segment token's rows are contiguous, so consecutive threads
// add to one trajectory row.
__global__ void __launch_bounds__(256) bwd_dq_scatter(const float* __restrict__ dq_acc,
                                                      const int32_t* __restrict__ tok_gather, int64_t num_tokens,
                                                      int32_t row_chunks, int32_t traj_tokens,
                                                      float* __restrict__ dq_traj) {
  const int64_t total = num_tokens * row_chunks;
  for (int64_t i = blockIdx.x * 256ll + threadIdx.x; i < total; i += (int64_t)gridDim.x * 256) {
    const int64_t n = i / row_chunks;
    const int c = (int)(i - n * row_chunks);
    const int t = __ldg(&tok_gather[n]);
    if (t < 0 || t >= traj_tokens) continue;  // recorded by the attention kernels' gathers
    const float4 x = reinterpret_cast<const float4*>(dq_acc)[i];
    red_add_v4(dq_traj + ((int64_t)t * row_chunks + c) * 4, x.x, x.y, x.z, x.w);
  }
}

// ------------------------------------------------------------------ bwd_main
template <int D>
__device__ __forceinline__ void issue_st(uint32_t tmem_d, uint32_t a_addr, uint32_t b_addr) {
  using C = Bwd<D>;
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    const uint32_t off = (kk >> 2) * C::BLOCK + (kk & 3) * 32;
    tc_mma_ss(tmem_d, smem_desc(a_addr + off, 16, 1024), smem_desc(b_addr + off, 16, 1024), C::IDESC_S, kk > 0);
  }
}
// D(tmem) (+)= A(128 x 128, K-major, K = query) x B(128 queries x D, MN-major)
template <int D>
__device__ __forceinline__ void issue_kv(uint32_t tmem_d, uint32_t a_addr, uint32_t b_addr, bool accumulate) {
  using C = Bwd<D>;
#pragma unroll
  for (int kk = 0; kk < C::BN / 16; ++kk) {
    const uint32_t aoff = (kk >> 2) * C::BLOCK + (kk & 3) * 32;
    tc_mma_ss(tmem_d, smem_desc(a_addr + aoff, 16, 1024), smem_desc(b_addr + kk * 2048, C::BLOCK, 1024),
              C::IDESC_KV, (accumulate || kk > 0) ? 1u : 0u);
  }
}
// dQ(tmem) = dS (128 queries x 128 keys, MN-major view of dSt) x K (128 keys x D, MN-major)
template <int D>
__device__ __forceinline__ void issue_dq(uint32_t tmem_d, uint32_t dst_addr, uint32_t k_addr) {
  using C = Bwd<D>;
#pragma unroll
  for (int kk = 0; kk < C::BM / 16; ++kk) {
    tc_mma_ss(tmem_d, smem_desc(dst_addr + kk * 2048, C::BLOCK, 1024), smem_desc(k_addr + kk * 2048, C::BLOCK, 1024),
              C::IDESC_DQ, kk > 0);
  }
}

// GATHER: Q, K and V are trajectory-layout tensors read through tok_gather, one warp per
// tile (TMA gather4 with the 2-D maps tm_q/k/v, or tiled loads with the 3-D maps
// tm_qr/kr/vr and tm_qs/ks/vs, 128- and 32-row boxes, where a tile or a 32-row group is one
// run of consecutive trajectory rows), and dK, dV are added
// in fp32 to trajectory-layout accumulators (dk_acc, dv_acc) at row tok_gather[key];
// otherwise segment-layout tiled loads, bf16 dK, dV, and tm_qr/kr/vr unused.
template <int D, bool GATHER>
__global__ void __launch_bounds__(kThreads, 1)
    bwd_main(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
             const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_do,
             const int32_t* __restrict__ cu_seqlens, int32_t num_segments, int32_t num_tokens, int32_t max_seqlen,
             int32_t hq, int32_t hkv, int32_t ntiles, float scale, float scale_log2,
             const float* __restrict__ lse, const float* __restrict__ dvec, float* __restrict__ dq_acc,
             __nv_bfloat16* __restrict__ dk, __nv_bfloat16* __restrict__ dv, int32_t* status,
             const int32_t* __restrict__ tok_gather, int32_t traj_tokens, float* __restrict__ dk_acc,
             float* __restrict__ dv_acc, const __grid_constant__ CUtensorMap tm_qr,
             const __grid_constant__ CUtensorMap tm_kr, const __grid_constant__ CUtensorMap tm_vr,
                    const __grid_constant__ CUtensorMap tm_qs, const __grid_constant__ CUtensorMap tm_ks,
                    const __grid_constant__ CUtensorMap tm_vs) {
  using C = Bwd<D>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  BwdBars* bars = reinterpret_cast<BwdBars*>(smem + C::OFF_BAR);
  float* lse2_s = reinterpret_cast<float*>(smem + C::OFF_ROW);         // [2][128]
  float* dvec_s = lse2_s + 2 * 128;                                    // [2][128]

  if (*reinterpret_cast<volatile int32_t*>(status) == VCS_ERR_DEVICE_TIMEOUT) return;
  // x = key tile (fastest), so the CTAs resident at one time mostly belong to
  // one (segment, kv-head) and their dQ reductions hit the same rows in L2
  const int sg = (int)(blockIdx.z * 65535u + blockIdx.y);
  if (sg >= num_segments * hkv) return;
  const int seg = sg / hkv;
  const int g = sg - seg * hkv;
  const int n = blockIdx.x;  // key tile
  const int start = cu_seqlens[seg];
  const int end = cu_seqlens[seg + 1];
  if (start < 0 || end < start || end > num_tokens || end - start > max_seqlen ||
      (seg == 0 && start != 0) || (seg == num_segments - 1 && end != num_tokens)) {
    if (threadIdx.x == 0 && n == 0 && g == 0) set_status(status, VCS_ERR_DEVICE_CHECK);
    return;
  }
  const int L = end - start;
  const int nq = (L + C::BN - 1) / C::BN;
  if (n >= nq) return;
  const int G = hq / hkv;
  const int per_head = nq - n;            // query tiles m = n .. nq-1
  const int iters = G * per_head;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t sbase = smem_u32(smem);

  if (threadIdx.x == 0) {
    mbar_init(&bars->kv_full, 1);
    mbar_init(&bars->qdo_full, 1);
    mbar_init(&bars->qdo_empty, 1);
    mbar_init(&bars->s_full, 1);
    mbar_init(&bars->p_full, 256);
    mbar_init(&bars->dq_full, 1);
    mbar_init(&bars->dq_free, 256);
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

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if constexpr (GATHER) {
      // the whole warp gathers Q, K, V; lane 0 posts the bytes, waits for free stages, loads dO
      if (lane == 0) {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_k);
        tma_prefetch_desc(&tm_v);
        tma_prefetch_desc(&tm_do);
        mbar_arrive_expect_tx(&bars->kv_full, 2 * C::TILE);
      }
      __syncwarp();
      load_traj_tile<C::KB, C::BLOCK>(smem + C::OFF_K, &tm_k, &tm_kr, &tm_ks, &bars->kv_full, g, D, start + n * C::BM, end - 1,
                                   tok_gather, traj_tokens, status, lane);
      load_traj_tile<C::KB, C::BLOCK>(smem + C::OFF_V, &tm_v, &tm_vr, &tm_vs, &bars->kv_full, g, D, start + n * C::BM, end - 1,
                                   tok_gather, traj_tokens, status, lane);
      for (int it = 0; it < iters; ++it) {
        const int h = g * G + it / per_head;
        const int m = n + it % per_head;
        int go = 1;
        if (lane == 0) {
          if (it > 0 && !mbar_wait(&bars->qdo_empty, (it - 1) & 1)) {
            on_timeout(bars, status);
            go = 0;
          } else if (aborted(bars)) {
            go = 0;
          } else {
            mbar_arrive_expect_tx(&bars->qdo_full, 2 * C::TILE);
#pragma unroll
            for (int kb = 0; kb < C::KB; ++kb)
              tma_load_3d(smem + C::OFF_DO + kb * C::BLOCK, &tm_do, &bars->qdo_full, kb * 64, h, start + m * C::BN);
          }
        }
        if (!__shfl_sync(0xffffffffu, go, 0)) break;
        load_traj_tile<C::KB, C::BLOCK>(smem + C::OFF_Q, &tm_q, &tm_qr, &tm_qs, &bars->qdo_full, h, D, start + m * C::BN, end - 1,
                                     tok_gather, traj_tokens, status, lane);
      }
    } else if (lane == 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      tma_prefetch_desc(&tm_do);
      mbar_arrive_expect_tx(&bars->kv_full, 2 * C::TILE);
#pragma unroll
      for (int kb = 0; kb < C::KB; ++kb) {
        tma_load_3d(smem + C::OFF_K + kb * C::BLOCK, &tm_k, &bars->kv_full, kb * 64, g, start + n * C::BM);
        tma_load_3d(smem + C::OFF_V + kb * C::BLOCK, &tm_v, &bars->kv_full, kb * 64, g, start + n * C::BM);
      }
      for (int it = 0; it < iters; ++it) {
        const int h = g * G + it / per_head;
        const int m = n + it % per_head;
        if (it > 0 && !mbar_wait(&bars->qdo_empty, (it - 1) & 1)) {
          on_timeout(bars, status);
          break;
        }
        if (aborted(bars)) break;
        mbar_arrive_expect_tx(&bars->qdo_full, 2 * C::TILE);
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb) {
          tma_load_3d(smem + C::OFF_Q + kb * C::BLOCK, &tm_q, &bars->qdo_full, kb * 64, h, start + m * C::BN);
          tma_load_3d(smem + C::OFF_DO + kb * C::BLOCK, &tm_do, &bars->qdo_full, kb * 64, h, start + m * C::BN);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      bool ok = mbar_wait(&bars->kv_full, 0);
      tc_fence_after();
      for (int it = 0; ok && it < iters; ++it) {
        if (!mbar_wait(&bars->qdo_full, it & 1)) { ok = false; break; }
        if (it > 0 && !mbar_wait(&bars->dq_free, (it - 1) & 1)) { ok = false; break; }
        tc_fence_after();
        issue_st<D>(tmem + C::TM_ST, sbase + C::OFF_K, sbase + C::OFF_Q);
        issue_st<D>(tmem + C::TM_DPT, sbase + C::OFF_V, sbase + C::OFF_DO);
        tc_commit(&bars->s_full);
        if (!mbar_wait(&bars->p_full, it & 1)) { ok = false; break; }
        tc_fence_after();
        issue_kv<D>(tmem + C::TM_DV, sbase + C::OFF_PT, sbase + C::OFF_DO, it > 0);
        issue_kv<D>(tmem + C::TM_DK, sbase + C::OFF_DST, sbase + C::OFF_Q, it > 0);
        issue_dq<D>(tmem + C::TM_DQ, sbase + C::OFF_DST, sbase + C::OFF_K);
        tc_commit(&bars->dq_full);
        tc_commit(&bars->qdo_empty);
        if (aborted(bars)) { ok = false; break; }
      }
      if (!ok) on_timeout(bars, status);
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------ compute
    const int wg = (warp - 4) >> 2;          // query-column half / D-column half
    const int quad = warp & 3;
    const int r = quad * 32 + lane;          // TMEM lane: key row (P phase) / query row (dQ phase)
    const int tw = threadIdx.x - 128 - wg * 128;  // 0..127 within the warpgroup
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    const int kpos = n * C::BM + r;
    bool ok = true;
    // per-query lse (log2 domain) and D of this warpgroup's 64 query columns,
    // loaded one iteration ahead so the global-load latency is off the critical path
    auto load_row_terms = [&](int it, float& l2, float& dd) {
      const int h = g * G + it / per_head;
      const int m = n + it % per_head;
      const int qpos = m * C::BN + wg * 64 + tw;
      l2 = __int_as_float(0x7f800000);  // +inf: query outside the segment -> P = 0
      dd = 0.f;
      if (tw < 64 && qpos < L) {
        l2 = __ldg(&lse[(size_t)h * num_tokens + start + qpos]) * 1.4426950408889634f;
        dd = __ldg(&dvec[(size_t)h * num_tokens + start + qpos]);
      }
    };
    float next_l2, next_dd;
    load_row_terms(0, next_l2, next_dd);
    for (int it = 0; it < iters; ++it) {
      const int h = g * G + it / per_head;
      const int m = n + it % per_head;
      const int buf = it & 1;
      if (tw < 64) {
        lse2_s[buf * 128 + wg * 64 + tw] = next_l2;
        dvec_s[buf * 128 + wg * 64 + tw] = next_dd;
      }
      if (it + 1 < iters) load_row_terms(it + 1, next_l2, next_dd);
      // the warpgroup goes on only if every thread finished the previous tile and no role has
      // given up (a decision all 128 threads take together, so none waits here alone)
      if (!named_bar_and(1 + wg, 128, ok && !aborted(bars))) { ok = false; break; }
      // each wait's outcome is the warp's: the TMEM loads that follow are warp-collective
      if (!mbar_wait_warp(&bars->s_full, it & 1)) { ok = false; continue; }
      tc_fence_after();
      uint32_t sv[64], pv[64];
      tmem_ld_32x32b_x32(trow + C::TM_ST + wg * 64, *reinterpret_cast<uint32_t(*)[32]>(&sv[0]));
      tmem_ld_32x32b_x32(trow + C::TM_ST + wg * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(&sv[32]));
      tmem_ld_32x32b_x32(trow + C::TM_DPT + wg * 64, *reinterpret_cast<uint32_t(*)[32]>(&pv[0]));
      tmem_ld_32x32b_x32(trow + C::TM_DPT + wg * 64 + 32, *reinterpret_cast<uint32_t(*)[32]>(&pv[32]));
      tmem_ld_wait();
      reg_fence<64>(sv);
      reg_fence<64>(pv);
      const bool diag = (m == n);
      const uint32_t pt_addr = sbase + C::OFF_PT + wg * C::BLOCK + r * 128;
      const uint32_t ds_addr = sbase + C::OFF_DST + wg * C::BLOCK + r * 128;
#pragma unroll
      for (int ch = 0; ch < 8; ++ch) {
        uint32_t wp[4], wd[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          float pe[2], de[2];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const int c = ch * 8 + e * 2 + u;          // column within this half
            const int qi = wg * 64 + c;
            const float l2 = lse2_s[buf * 128 + qi];
            float p = ex2(fmaf(__uint_as_float(sv[c]), scale_log2, -l2));
            if (diag && r > qi) p = 0.f;               // key after query
            pe[u] = p;
            de[u] = p * (__uint_as_float(pv[c]) - dvec_s[buf * 128 + qi]) * scale;
          }
          wp[e] = pack_bf16(pe[0], pe[1]);
          wd[e] = pack_bf16(de[0], de[1]);
        }
        const uint32_t sw = (uint32_t)((ch ^ (r & 7)) << 4);
        st_shared_v4(pt_addr + sw, wp[0], wp[1], wp[2], wp[3]);
        st_shared_v4(ds_addr + sw, wd[0], wd[1], wd[2], wd[3]);
      }
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(&bars->p_full);
      // dQ of this (m, h): query rows on TMEM lanes, this warpgroup's D/2 columns
      if (!mbar_wait_warp(&bars->dq_full, it & 1)) { ok = false; continue; }
      tc_fence_after();
      const int qrow = m * C::BN + r;
      float* dst = dq_acc + ((size_t)(start + qrow) * hq + h) * D + wg * (D / 2);
      // drain this warpgroup's dQ columns into registers, release TMEM, then reduce
      uint32_t q32[D / 2];
#pragma unroll
      for (int c = 0; c < D / 64; ++c)
        tmem_ld_32x32b_x32(trow + C::TM_DQ + wg * (D / 2) + c * 32,
                           *reinterpret_cast<uint32_t(*)[32]>(&q32[c * 32]));
      tmem_ld_wait();
      reg_fence<D / 2>(q32);
      tc_fence_before();
      mbar_arrive(&bars->dq_free);
      if (qrow < L) {
#pragma unroll
        for (int e = 0; e < D / 8; ++e)
          red_add_v4(dst + e * 4, __uint_as_float(q32[e * 4]), __uint_as_float(q32[e * 4 + 1]),
                     __uint_as_float(q32[e * 4 + 2]), __uint_as_float(q32[e * 4 + 3]));
      }
    }
    if (!ok) {
      on_timeout(bars, status);
    } else {
      // dK, dV rows of the tile (key rows on TMEM lanes), this warpgroup's D/2 columns
      bool valid = kpos < L;
      size_t base = ((size_t)(start + kpos) * hkv + g) * D + wg * (D / 2);
      if (GATHER && valid) {  // fp32 add at the key's trajectory row
        const int t = tok_gather[start + kpos];
        valid = t >= 0 && t < traj_tokens;
        base = ((size_t)(valid ? t : 0) * hkv + g) * D + wg * (D / 2);
      }
#pragma unroll
      for (int which = 0; which < 2; ++which) {
        const uint32_t col = (which == 0 ? C::TM_DK : C::TM_DV) + wg * (D / 2);
        __nv_bfloat16* outp = (which == 0 ? dk : dv) + base;
#pragma unroll
        for (int c = 0; c < D / 64; ++c) {
          uint32_t v32[32];
          tmem_ld_32x32b_x32(trow + col + c * 32, v32);
          tmem_ld_wait();
          reg_fence<32>(v32);
          if (GATHER) {
            if (valid) {
              float* acc = (which == 0 ? dk_acc : dv_acc) + base + c * 32;
#pragma unroll
              for (int e = 0; e < 8; ++e)
                red_add_v4(acc + e * 4, __uint_as_float(v32[e * 4]), __uint_as_float(v32[e * 4 + 1]),
                           __uint_as_float(v32[e * 4 + 2]), __uint_as_float(v32[e * 4 + 3]));
            }
          } else if (valid) {
            uint4* d4 = reinterpret_cast<uint4*>(outp + c * 32);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              uint4 pk;
              pk.x = pack_bf16(__uint_as_float(v32[q * 8 + 0]), __uint_as_float(v32[q * 8 + 1]));
              pk.y = pack_bf16(__uint_as_float(v32[q * 8 + 2]), __uint_as_float(v32[q * 8 + 3]));
              pk.z = pack_bf16(__uint_as_float(v32[q * 8 + 4]), __uint_as_float(v32[q * 8 + 5]));
              pk.w = pack_bf16(__uint_as_float(v32[q * 8 + 6]), __uint_as_float(v32[q * 8 + 7]));
              d4[q] = pk;
            }
          }
        }
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

// ------------------------------------------------------------------ bwd_main_d128 (head_dim 128)
// Same work unit and result as bwd_main, with every MMA at N = 128 (the
// tensor pipe's full rate; N = 64 runs at 2/3).  The query rows of each
// (query tile, head) are processed as 128-row tiles in one stream; the two
// compute warpgroups split a tile's query columns.
//   WG0   warp 0: TMA producer (K and V once, Q/dO 128-row tiles through a 2-stage ring)
//         warp 1: TMEM allocation and the single MMA-issuing thread
//   WG1/2 compute in four phases of 32 query columns, warpgroup k taking 16
//         columns of each: S^T, dP^T -> P^T and dS^T (bf16, written back to TMEM
//         over the warpgroup's own 16 dP^T columns, 8 each: the A operands of
//         dV += P^T dO and dK += dS^T Q, which then read only their B operand
//         from shared memory) and dS^T once more in shared memory (for
//         dQ = dS K); dV and dK over a phase's columns run while the next phase
//         is computed
//   WG3   dQ drain: once a tile's MMAs are complete, dQ (query rows on TMEM
//         lanes) is read two 32-column parts at a time and copied into the tile's
//         freed Q/dO stage, the columns are handed back, and TMA bulk reduce-adds
//         add it to the fp32 accumulator
// Registers are rebalanced per warpgroup with setmaxnreg (96 / 168 / 168 / 80
// per thread; the block launches with 128).
// With a 64-query sub-tile and two streams (compute of one stream overlapping
// the other's MMAs) the N = 64 MMAs held the backward 5% lower on the
// long-horizon workload than this single stream of 128-query tiles.
//   TMEM: dV [0,128), dK [128,256); S^T then dQ, and dP^T then P^T/dS^T, in [256,384) and
//         [384,512), swapping roles every tile so that S^T(u+1) can be computed while
//         dQ(u) is drained
//   smem: K, V (64 KB), 2-stage Q/dO ring (128 KB; a freed stage also stages dQ),
//         dS^T (32 KB), row terms (1 KB)

// dst (global, tensor map) += src (shared) for one box, asynchronously (bulk group).
__device__ __forceinline__ void tma_reduce_add_3d(const void* map, const void* src, int x, int y, int z) {
  asm volatile(
      "cp.reduce.async.bulk.tensor.3d.global.shared::cta.add.tile.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(map),
      "r"(smem_u32(src)), "r"(x), "r"(y), "r"(z)
      : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// all but the most recent bulk group have finished reading their shared-memory sources
__device__ __forceinline__ void bulk_wait_read1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// TMEM loads / stores of N consecutive 32-bit columns of the warp's 32 lanes.
template <int N>
__device__ __forceinline__ void tmem_ld_cols(uint32_t taddr, uint32_t (&r)[N]) {
  static_assert(N == 16 || N == 32, "16 or 32 columns");
  if constexpr (N == 32) tmem_ld_32x32b_x32(taddr, r);
  else tmem_ld_32x32b_x16(taddr, r);
}
template <int N>
__device__ __forceinline__ void tmem_st_cols(uint32_t taddr, const uint32_t (&r)[N]) {
  static_assert(N == 8 || N == 16, "8 or 16 columns");
  if constexpr (N == 16) tmem_st_32x32b_x16(taddr, r);
  else tmem_st_32x32b_x8(taddr, r);
}

// One compute thread's share of one phase: key row r against NC query columns.
//   P^T  = 2^(S^T * scale*log2e - lse*log2e)     (zero where the key follows the query)
//   dS^T = P^T * (dP^T - D) * scale
// The row terms come as {-lse*log2e, -D*scale} of each column pair, one 16-byte load
// {nl(c), nl(c+1), nd(c), nd(c+1)} per pair.  P^T goes to pt and dS^T to dt as bf16 pairs
// (for TMEM), and dS^T also to 16-byte chunks CH0 .. CH0+NC/8-1 of the thread's 128-byte row
// of the swizzled K-major shared block.  The causal test is compiled
// only into the diagonal instantiation (column c is masked when c < dlim), so the
// off-diagonal tiles run a branch-free body the compiler can interleave.
template <int NC, bool DIAG>
__device__ __forceinline__ void d128_phase_math(const uint32_t (&sv)[NC], const uint32_t (&pv)[NC],
                                                uint32_t (&pt)[NC / 2], uint32_t (&dt)[NC / 2],
                                                const uint4 (&rq)[NC / 2], uint64_t sl2,
                                                uint64_t sc2, int dlim, uint32_t ds_row, int ch0, int r) {
#pragma unroll
  for (int ch = 0; ch < NC / 8; ++ch) {
    uint32_t wd[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int c = ch * 8 + e * 2;
      const float4 q = make_float4(__uint_as_float(rq[c / 2].x), __uint_as_float(rq[c / 2].y),
                                   __uint_as_float(rq[c / 2].z), __uint_as_float(rq[c / 2].w));
      float x0, x1;
      f2unpack(ffma2(f2pack(__uint_as_float(sv[c]), __uint_as_float(sv[c + 1])), sl2, f2pack(q.x, q.y)), x0, x1);
      float p0 = ex2(x0), p1 = ex2(x1);
      if (DIAG) {
        if (c < dlim) p0 = 0.f;
        if (c + 1 < dlim) p1 = 0.f;
      }
      const uint64_t pp = f2pack(p0, p1);
      const uint64_t t = ffma2(f2pack(__uint_as_float(pv[c]), __uint_as_float(pv[c + 1])), sc2, f2pack(q.z, q.w));
      float d0, d1;
      f2unpack(fmul2(pp, t), d0, d1);
      pt[ch * 4 + e] = pack_bf16(p0, p1);
      wd[e] = pack_bf16(d0, d1);
      dt[ch * 4 + e] = wd[e];
    }
    st_shared_v4(ds_row + (uint32_t)(((ch0 + ch) ^ (r & 7)) << 4), wd[0], wd[1], wd[2], wd[3]);
  }
}

struct D128 {
  static constexpr int D = 128;
  static constexpr int BM = 128;                 // key rows of the tile
  static constexpr int BQ = 128;                 // query rows per tile
  static constexpr int NST = 2;                  // Q/dO ring stages
  // The compute runs in NPH phases of PW query columns; warpgroup k takes columns
  // [PW*ph + HW*k, PW*ph + HW*k + HW) of phase ph, and dV, dK over a phase's columns are
  // issued as soon as both warpgroups have written them.
  static constexpr int NPH = 4;
  static constexpr int PW = 128 / NPH;
  static constexpr int HW = PW / 2;
  static constexpr int KPP = PW / 16;            // K = 16 MMA steps (16 queries each) per phase
  static constexpr int THREADS = 512;
  static constexpr int TILE = 128 * D * 2;       // 32 KB: K, V, a Q or a dO tile
  static constexpr int BLOCK = 128 * 128;        // one 64-column block of a 128-row tile
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = TILE;
  static constexpr int OFF_Q = 2 * TILE;                       // stage s: Q at +s*2*TILE, dO at +TILE
  static constexpr int OFF_DS = OFF_Q + NST * 2 * TILE;        // dS^T [128 keys][128 queries], two 64-query blocks
  static constexpr int OFF_ROW = OFF_DS + TILE;                // WG k: -lse*log2e, -D*scale of 64 queries
  static constexpr int OFF_BAR = OFF_ROW + 2 * 2 * 64 * 4;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr int TM_DV = 0, TM_DK = 128, TM_A = 256, TM_B = 384;
  // tile u: S^T (later dQ) in TM_A for even u, TM_B for odd u; dP^T (later P^T) in the other
  __device__ static uint32_t col_s(int u) { return (u & 1) ? TM_B : TM_A; }
  __device__ static uint32_t col_p(int u) { return (u & 1) ? TM_A : TM_B; }
  // P^T of queries [16kk, 16kk+16) (8 columns of bf16 pairs) is written by the warpgroup that
  // computes them, into the first columns of the dP^T columns it has itself just read
  __host__ __device__ static constexpr uint32_t pt_col(int kk) {
    return PW * (kk / KPP) + HW * ((kk % KPP) / (KPP / 2)) + 8 * (kk % (KPP / 2));
  }
  // ... and its dS^T (the A operand of dK += dS^T Q) in the 8 columns after them: each
  // warpgroup's 16 dP^T columns of a phase hold exactly one K = 16 step of each
  static constexpr int REG_CTRL = 96, REG_COMPUTE = 168, REG_DRAIN = 80;
  static constexpr int REG_LAUNCH = 65536 / THREADS;
  static constexpr uint32_t IDESC_S = idesc_bf16(128, 128, 0, 0);   // K or V (K-major) x Q or dO (K-major)
  static constexpr uint32_t IDESC_KV = idesc_bf16(128, 128, 0, 1);  // P^T / dS^T (TMEM) x dO / Q (MN-major)
  static constexpr uint32_t IDESC_DQ = idesc_bf16(128, 128, 1, 1);  // dS (MN-major) x K (MN-major)
};
static_assert(D128::SMEM <= 232448, "shared memory budget");
static_assert(D128::HW == 16, "a warpgroup's phase columns hold one K step of P^T and one of dS^T");
static_assert(D128::REG_CTRL + 2 * D128::REG_COMPUTE + D128::REG_DRAIN <= 4 * D128::REG_LAUNCH,
              "setmaxnreg targets exceed the registers the block is launched with");

struct D128Bars {
  uint64_t kv_full;
  uint64_t q_full[D128::NST];      // Q of the stage's tile has landed
  uint64_t do_full[D128::NST];     // dO of the stage's tile has landed and the drain has read the
                                   // previous tile's dQ out of TMEM (its columns take dP^T next)
  uint64_t kv_done[D128::NST];     // the tile's MMAs are complete: its Q/dO stage may be overwritten
  uint64_t q_free[D128::NST];      // the drain's reduce-adds have read the stage's Q half
  uint64_t do_free[D128::NST];     // ... and its dO half
  uint64_t s_full;
  uint64_t p_full[D128::NPH];  // the query columns of phase ph of the tile: P^T and dS^T written
  uint64_t acc_done;
  uint32_t tmem_base;
  int32_t abort;
};


// GATHER: as for bwd_main (Q, K, V gathered from trajectory-layout tensors, dK and dV
// added in fp32 at the keys' trajectory rows).
template <bool GATHER>
__global__ void __launch_bounds__(D128::THREADS, 1)
    bwd_main_d128(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                  const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_do,
                  const __grid_constant__ CUtensorMap tm_dq, const int32_t* __restrict__ cu_seqlens,
                  int32_t num_segments, int32_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv, float scale,
                  float scale_log2, const float* __restrict__ lse, const float* __restrict__ dvec,
                  __nv_bfloat16* __restrict__ dk, __nv_bfloat16* __restrict__ dv, int32_t* status,
                  const int32_t* __restrict__ tok_gather, int32_t traj_tokens, float* __restrict__ dk_acc,
                  float* __restrict__ dv_acc, const __grid_constant__ CUtensorMap tm_qr,
                  const __grid_constant__ CUtensorMap tm_kr, const __grid_constant__ CUtensorMap tm_vr,
                    const __grid_constant__ CUtensorMap tm_qs, const __grid_constant__ CUtensorMap tm_ks,
                    const __grid_constant__ CUtensorMap tm_vs) {
  using C = D128;
  constexpr int D = C::D;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  D128Bars* bars = reinterpret_cast<D128Bars*>(smem + C::OFF_BAR);

  const int sg = (int)(blockIdx.z * 65535u + blockIdx.y);
  if (sg >= num_segments * hkv) return;
  const int seg = sg / hkv;
  const int g = sg - seg * hkv;
  const int n = blockIdx.x;  // key tile
  const int start = cu_seqlens[seg];
  const int end = cu_seqlens[seg + 1];
  if (start < 0 || end < start || end > num_tokens || end - start > max_seqlen ||
      (seg == 0 && start != 0) || (seg == num_segments - 1 && end != num_tokens)) {
    if (threadIdx.x == 0 && n == 0 && g == 0) set_status(status, VCS_ERR_DEVICE_CHECK);
    return;
  }
  const int L = end - start;
  if (n * C::BM >= L) return;
  // once any CTA of this launch has given up on a wait, the rest stand down (read only by the
  // CTAs that have a key tile)
  if (*reinterpret_cast<volatile int32_t*>(status) == VCS_ERR_DEVICE_TIMEOUT) return;
  const int G = hq / hkv;
  const int nsub = (L - n * C::BM + C::BQ - 1) / C::BQ;  // 128-row query tiles at or after this key tile
  const int U = G * nsub;
  // Tile u covers query rows n*BM + sub_of(u)*BQ ... +BQ-1 of head head_of(u), swept from the
  // segment end toward the key tile with the G heads of one row block in turn, so that the key
  // tiles of one (segment, kv head) running together meet the same Q/dO/dQ lines in L2.
  auto sub_of = [&](int u) { return nsub - 1 - u / G; };
  auto head_of = [&](int u) { return g * G + u % G; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t sbase = smem_u32(smem);

  if (threadIdx.x == 0) {
    mbar_init(&bars->kv_full, 1);
    for (int i = 0; i < C::NST; ++i) {
      mbar_init(&bars->q_full[i], 1);
      mbar_init(&bars->do_full[i], 1 + 128);  // the producer's bytes + the drain's 128 threads
      mbar_init(&bars->kv_done[i], 1);
      mbar_init(&bars->q_free[i], 1);
      mbar_init(&bars->do_free[i], 1);
    }
    mbar_init(&bars->s_full, 1);
    for (int i = 0; i < C::NPH; ++i) mbar_init(&bars->p_full[i], 256);
    mbar_init(&bars->acc_done, 1);
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
  auto abort_now = [&]() {
    set_status(status, VCS_ERR_DEVICE_TIMEOUT);
    *reinterpret_cast<volatile int32_t*>(&bars->abort) = 1;
  };
  auto aborted_now = [&]() { return *reinterpret_cast<volatile int32_t*>(&bars->abort) != 0; };

  if (warp < 4) {
    setmaxnreg_dec<C::REG_CTRL>();
    if (GATHER && warp == 0) {
      // ---------------------------------------------------------- producer (gathered)
      // the whole warp gathers K, V and each tile's Q; lane 0 posts the bytes, waits for
      // free stages and loads dO
      if (lane == 0) {
        tma_prefetch_desc(&tm_q);
        tma_prefetch_desc(&tm_k);
        tma_prefetch_desc(&tm_v);
        tma_prefetch_desc(&tm_do);
        mbar_arrive_expect_tx(&bars->kv_full, 2 * C::TILE);
      }
      __syncwarp();
      load_traj_tile<2, C::BLOCK>(smem + C::OFF_K, &tm_k, &tm_kr, &tm_ks, &bars->kv_full, g, D, start + n * C::BM, end - 1, tok_gather,
                               traj_tokens, status, lane);
      load_traj_tile<2, C::BLOCK>(smem + C::OFF_V, &tm_v, &tm_vr, &tm_vs, &bars->kv_full, g, D, start + n * C::BM, end - 1, tok_gather,
                               traj_tokens, status, lane);
      for (int u = 0; u < U; ++u) {
        const int h = head_of(u);
        const int q0 = n * C::BM + sub_of(u) * C::BQ;
        const int stage = u % C::NST;
        uint8_t* qs = smem + C::OFF_Q + stage * 2 * C::TILE;
        int go = 1;
        if (lane == 0) {
          if (u >= C::NST && !mbar_wait(&bars->q_free[stage], ((u / C::NST) - 1) & 1)) {
            abort_now();
            go = 0;
          } else if (aborted_now()) {
            go = 0;
          } else {
            mbar_arrive_expect_tx(&bars->q_full[stage], C::TILE);
          }
        }
        if (!__shfl_sync(0xffffffffu, go, 0)) break;
        load_traj_tile<2, C::BLOCK>(qs, &tm_q, &tm_qr, &tm_qs, &bars->q_full[stage], h, D, start + q0, end - 1, tok_gather, traj_tokens,
                                 status, lane);
        if (lane == 0) {
          if (u >= C::NST && !mbar_wait(&bars->do_free[stage], ((u / C::NST) - 1) & 1)) {
            abort_now();
            go = 0;
          } else {
            mbar_arrive_expect_tx(&bars->do_full[stage], C::TILE);
#pragma unroll
            for (int kb = 0; kb < 2; ++kb)
              tma_load_3d(qs + C::TILE + kb * C::BLOCK, &tm_do, &bars->do_full[stage], kb * 64, h, start + q0);
          }
        }
        if (!__shfl_sync(0xffffffffu, go, 0)) break;
      }
    } else if (warp == 0 && lane == 0) {
      // ---------------------------------------------------------- producer
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_k);
      tma_prefetch_desc(&tm_v);
      tma_prefetch_desc(&tm_do);
      mbar_arrive_expect_tx(&bars->kv_full, 2 * C::TILE);
#pragma unroll
      for (int kb = 0; kb < 2; ++kb) {
        tma_load_3d(smem + C::OFF_K + kb * C::BLOCK, &tm_k, &bars->kv_full, kb * 64, g, start + n * C::BM);
        tma_load_3d(smem + C::OFF_V + kb * C::BLOCK, &tm_v, &bars->kv_full, kb * 64, g, start + n * C::BM);
      }
      for (int u = 0; u < U; ++u) {
        const int h = head_of(u);
        const int q0 = n * C::BM + sub_of(u) * C::BQ;
        const int stage = u % C::NST;
        uint8_t* qs = smem + C::OFF_Q + stage * 2 * C::TILE;
        // Q and dO are refilled separately: the drain's reduce-adds read the Q half first
        if (u >= C::NST && !mbar_wait(&bars->q_free[stage], ((u / C::NST) - 1) & 1)) {
          abort_now();
          break;
        }
        if (aborted_now()) break;
        mbar_arrive_expect_tx(&bars->q_full[stage], C::TILE);
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
          tma_load_3d(qs + kb * C::BLOCK, &tm_q, &bars->q_full[stage], kb * 64, h, start + q0);
        if (u >= C::NST && !mbar_wait(&bars->do_free[stage], ((u / C::NST) - 1) & 1)) {
          abort_now();
          break;
        }
        mbar_arrive_expect_tx(&bars->do_full[stage], C::TILE);
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
          tma_load_3d(qs + C::TILE + kb * C::BLOCK, &tm_do, &bars->do_full[stage], kb * 64, h, start + q0);
      }
    } else if (warp == 1 && lane == 0) {
      // ---------------------------------------------------------- MMA issuer
      bool ok = mbar_wait(&bars->kv_full, 0);
      // descriptors built once; the issue loops only add compile-time offsets
      const uint64_t k_kmaj = smem_desc(sbase + C::OFF_K, 16, 1024);
      const uint64_t v_kmaj = smem_desc(sbase + C::OFF_V, 16, 1024);
      const uint64_t k_mnmaj = smem_desc(sbase + C::OFF_K, C::BLOCK, 1024);
      const uint64_t q_kmaj = smem_desc(sbase + C::OFF_Q, 16, 1024);
      const uint64_t q_mnmaj = smem_desc(sbase + C::OFF_Q, C::BLOCK, 1024);
      const uint64_t ds_mnmaj = smem_desc(sbase + C::OFF_DS, C::BLOCK, 1024);
      for (int u = 0; ok && u < U; ++u) {
        const int stage = u % C::NST;
        const uint32_t cs = tmem + C::col_s(u), cp = tmem + C::col_p(u);
        // S^T = K Q^T needs Q/dO of u; its columns held P^T of u-1, which dV(u-1), issued
        // before, reads first (in-order execution), so it overlaps the drain of dQ(u-1).
        if (!mbar_wait(&bars->q_full[stage], (u / C::NST) & 1) || aborted_now()) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint64_t qd = desc_at(q_kmaj, stage * 2 * C::TILE), dd = desc_at(qd, C::TILE);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t o = (kk >> 2) * C::BLOCK + (kk & 3) * 32;
          tc_mma_ss(cs, desc_at(k_kmaj, o), desc_at(qd, o), C::IDESC_S, kk > 0);
        }
        // dP^T = V dO^T goes where dQ(u-1) was: one wait for dO and for the drain to have read
        // dQ(u-1)
        if (!mbar_wait(&bars->do_full[stage], (u / C::NST) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint32_t o = (kk >> 2) * C::BLOCK + (kk & 3) * 32;
          tc_mma_ss(cp, desc_at(v_kmaj, o), desc_at(dd, o), C::IDESC_S, kk > 0);
        }
        tc_commit(&bars->s_full);
        // dV += P^T dO and dK += dS^T Q over each phase's queries as soon as they are written
        // (overlapping the compute of the next phase), then, after the last phase, dQ = dS K
        // and the last phase's dV, dK.  In-order execution keeps S(u+1) from overwriting P^T or
        // dS^T first.  P^T of queries [16kk, 16kk+16) sits at C::pt_col(kk) of its columns, their
        // dS^T 8 columns further.
        const uint64_t qmn = desc_at(q_mnmaj, stage * 2 * C::TILE), dmn = desc_at(qmn, C::TILE);
        const uint32_t acc0 = u > 0 ? 1u : 0u;
        auto issue_dvdk = [&](int kk0) {
#pragma unroll
          for (int kk = kk0; kk < kk0 + C::KPP; ++kk)
            tc_mma_ts(tmem + C::TM_DV, cp + C::pt_col(kk), desc_at(dmn, kk * 2048), C::IDESC_KV,
                      kk > 0 ? 1u : acc0);
#pragma unroll
          for (int kk = kk0; kk < kk0 + C::KPP; ++kk)
            tc_mma_ts(tmem + C::TM_DK, cp + C::pt_col(kk) + 8, desc_at(qmn, kk * 2048), C::IDESC_KV,
                      kk > 0 ? 1u : acc0);
        };
#pragma unroll
        for (int ph = 0; ph < C::NPH - 1; ++ph) {
          if (!mbar_wait(&bars->p_full[ph], u & 1)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_dvdk(ph * C::KPP);
        }
        if (!ok || !mbar_wait(&bars->p_full[C::NPH - 1], u & 1)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < C::BM / 16; ++kk)
          tc_mma_ss(cs, desc_at(ds_mnmaj, kk * 2048), desc_at(k_mnmaj, kk * 2048), C::IDESC_DQ,
                    kk > 0 ? 1u : 0u);
        issue_dvdk((C::NPH - 1) * C::KPP);
        tc_commit(&bars->kv_done[stage]);
      }
      tc_commit(&bars->acc_done);
      if (!ok) abort_now();
    }
  } else if (warp < 12) {
    // ------------------------------------------------------------ compute
    setmaxnreg_inc<C::REG_COMPUTE>();
    const int k = (warp - 4) >> 2;   // query columns [32k, 32k+32) and [64+32k, 96+32k) of the tile
    const int quad = warp & 3;
    const int r = quad * 32 + lane;  // TMEM lane: key row
    const int tw = threadIdx.x - 128 - k * 128;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    // row terms of the warpgroup's 64 query columns, per phase (16 columns):
    // {nl(c), nl(c+1), nd(c), nd(c+1)}
    // for each column pair, nl = -lse*log2e and nd = -D*scale
    float* rt_s = reinterpret_cast<float*>(smem + C::OFF_ROW) + k * 128;
    const uint32_t rt_u32 = smem_u32(rt_s);
    // thread tw < 64 stages the terms of column HW*k + PW*(tw / HW) + tw % HW; phase ph's terms
    // start at rt_s + PW*ph
    const int rt_slot = (tw / C::HW) * C::PW + ((tw % C::HW) >> 1) * 4 + (tw & 1);
    const uint64_t sl2 = f2pack(scale_log2, scale_log2), sc2 = f2pack(scale, scale);
    auto row_terms = [&](int u, float& nl2, float& nds) {
      nl2 = __int_as_float(0xff800000);  // -inf: query outside the segment -> P = 0
      nds = 0.f;
      if (u < U && tw < 64) {
        const int h = head_of(u);
        const int q = n * C::BM + sub_of(u) * C::BQ + C::PW * (tw / C::HW) + C::HW * k + tw % C::HW;
        if (q < L) {
          nl2 = -__ldg(&lse[(size_t)h * num_tokens + start + q]) * 1.4426950408889634f;
          nds = -__ldg(&dvec[(size_t)h * num_tokens + start + q]) * scale;
        }
      }
    };
    float next_nl2, next_nds;
    row_terms(0, next_nl2, next_nds);
    bool ok = true;
    for (int u = 0; u < U; ++u) {
      const bool diag = sub_of(u) == 0;  // the query rows are the key tile's own: mask keys after queries
      if (tw < 64) {
        rt_s[rt_slot] = next_nl2;
        rt_s[rt_slot + 2] = next_nds;
      }
      named_bar_sync(1 + k, 128);
      row_terms(u + 1, next_nl2, next_nds);
      // the wait's outcome is the warp's (the TMEM loads below are warp-collective); the
      // warpgroup decides together at the barrier that closes the tile
      const bool got = mbar_wait_warp(&bars->s_full, u & 1);
      if (got) {
        tc_fence_after();
        // phase ph: query columns [PW*ph + HW*k, PW*ph + HW*k + HW); its P^T and dS^T (HW/2
        // words each) go over its own dP^T columns, and its dS^T also into HW/8 16-byte chunks
        // of the shared block of its 64 queries
        // the next phase's S^T and dP^T columns are loaded while this phase is computed
        uint32_t sv[2][C::HW], pv[2][C::HW];
        tmem_ld_cols<C::HW>(trow + C::col_s(u) + C::HW * k, sv[0]);
        tmem_ld_cols<C::HW>(trow + C::col_p(u) + C::HW * k, pv[0]);
        tmem_ld_wait();
        reg_fence<C::HW>(sv[0]);
        reg_fence<C::HW>(pv[0]);
#pragma unroll
        for (int ph = 0; ph < C::NPH; ++ph) {
          const int cur = ph & 1;
          const uint32_t col = C::PW * ph + C::HW * k;
          if (ph + 1 < C::NPH) {
            tmem_ld_cols<C::HW>(trow + C::col_s(u) + col + C::PW, sv[cur ^ 1]);
            tmem_ld_cols<C::HW>(trow + C::col_p(u) + col + C::PW, pv[cur ^ 1]);
          }
          // the phase's row terms, all loads issued back to back so that their latencies overlap
          uint4 rq[C::HW / 2];
#pragma unroll
          for (int e = 0; e < C::HW / 2; ++e) rq[e] = ld_shared_v4(rt_u32 + (uint32_t)(C::PW * ph + 4 * e) * 4);
          uint32_t pt[C::HW / 2], dt[C::HW / 2];
          const uint32_t ds_row = sbase + C::OFF_DS + (col / 64) * C::BLOCK + r * 128;
          const int ch0 = (int)(col % 64) / 8;
          if (diag)
            d128_phase_math<C::HW, true>(sv[cur], pv[cur], pt, dt, rq, sl2, sc2, r - (int)col, ds_row, ch0, r);
          else
            d128_phase_math<C::HW, false>(sv[cur], pv[cur], pt, dt, rq, sl2, sc2, 0, ds_row, ch0, r);
          // dS^T (shared memory) is published to the tensor pipe while the TMEM stores of P^T and
          // dS^T complete
          fence_proxy_async_smem();
          tmem_st_cols<C::HW / 2>(trow + C::col_p(u) + col, pt);
          tmem_st_cols<C::HW / 2>(trow + C::col_p(u) + col + C::HW / 2, dt);
          tmem_st_wait();
          tc_fence_before();
          mbar_arrive(&bars->p_full[ph]);
          if (ph + 1 < C::NPH) {
            tmem_ld_wait();
            reg_fence<C::HW>(sv[cur ^ 1]);
            reg_fence<C::HW>(pv[cur ^ 1]);
          }
        }
      }
      // everyone is done with this tile's row terms; go on only if every thread got its tile and
      // no other role has given up
      if (!named_bar_and(1 + k, 128, got && !aborted_now())) { ok = false; break; }
    }
    if (ok) ok = mbar_wait_warp(&bars->acc_done, 0);
    if (!ok) {
      abort_now();
    } else {
      tc_fence_after();
      // warpgroup 1 writes dK, warpgroup 2 writes dV (key row r on the TMEM lane)
      const int kpos = n * C::BM + r;
      const uint32_t col = k == 0 ? C::TM_DK : C::TM_DV;
      __nv_bfloat16* outp = (k == 0 ? dk : dv) + ((size_t)(start + kpos) * hkv + g) * D;
      float* accp = nullptr;  // gathered: fp32 add at the key's trajectory row
      if (GATHER && kpos < L) {
        const int t = tok_gather[start + kpos];
        if (t >= 0 && t < traj_tokens) accp = (k == 0 ? dk_acc : dv_acc) + ((size_t)t * hkv + g) * D;
      }
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t v32[32];
        tmem_ld_32x32b_x32(trow + col + c * 32, v32);
        tmem_ld_wait();
        reg_fence<32>(v32);
        if (GATHER) {
          if (accp != nullptr) {
#pragma unroll
            for (int e = 0; e < 8; ++e)
              red_add_v4(accp + c * 32 + e * 4, __uint_as_float(v32[e * 4]), __uint_as_float(v32[e * 4 + 1]),
                         __uint_as_float(v32[e * 4 + 2]), __uint_as_float(v32[e * 4 + 3]));
          }
        } else if (kpos < L) {
          uint4* d4 = reinterpret_cast<uint4*>(outp + c * 32);
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            uint4 pk;
            pk.x = pack_bf16(__uint_as_float(v32[q * 8 + 0]), __uint_as_float(v32[q * 8 + 1]));
            pk.y = pack_bf16(__uint_as_float(v32[q * 8 + 2]), __uint_as_float(v32[q * 8 + 3]));
            pk.z = pack_bf16(__uint_as_float(v32[q * 8 + 4]), __uint_as_float(v32[q * 8 + 5]));
            pk.w = pack_bf16(__uint_as_float(v32[q * 8 + 6]), __uint_as_float(v32[q * 8 + 7]));
            d4[q] = pk;
          }
        }
      }
    }
  } else {
    // ------------------------------------------------------------ dQ drain
    // Once a tile's MMAs are complete its Q/dO stage is free: dQ (query rows on TMEM lanes) is
    // copied there as four [128 rows][32 dims] fp32 blocks in the 128-byte swizzled layout of
    // the accumulator's tensor map, added to the accumulator with four TMA bulk reduce-adds
    // (rows past the segment end are exact zeros), and the stage is handed back to the producer
    // once the reduce-adds have read it.
    setmaxnreg_dec<C::REG_DRAIN>();
    const int quad = warp & 3;
    const int l = quad * 32 + lane;  // TMEM lane: query row of the tile
    const int dw = threadIdx.x - 12 * 32;
    const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
    bool ok = true;
    // each tile's dP^T waits, with its dO, for the drain to have read the previous tile's dQ;
    // tile 0 has none
    mbar_arrive(&bars->do_full[0]);
    for (int u = 0; u < U; ++u) {
      const int stage = u % C::NST;
      const bool got = mbar_wait_warp(&bars->kv_done[stage], (u / C::NST) & 1);
      uint8_t* stg = smem + C::OFF_Q + stage * 2 * C::TILE;
      if (got) {
        tc_fence_after();
        const uint32_t srow = smem_u32(stg) + l * 128;
        // two 32-column parts per TMEM round trip, so that the columns are handed back after two
        // rounds of loads
#pragma unroll
        for (int pp = 0; pp < D / 64; ++pp) {
          uint32_t a[2][32];
          tmem_ld_32x32b_x32(trow + C::col_s(u) + pp * 64, a[0]);
          tmem_ld_32x32b_x32(trow + C::col_s(u) + pp * 64 + 32, a[1]);
          tmem_ld_wait();
          reg_fence<32>(a[0]);
          reg_fence<32>(a[1]);
          if (pp == D / 64 - 1 && u + 1 < U) {
            tc_fence_before();
            mbar_arrive(&bars->do_full[(u + 1) % C::NST]);
          }
#pragma unroll
          for (int i = 0; i < 2; ++i)
#pragma unroll
            for (int j = 0; j < 8; ++j)
              st_shared_v4(srow + (2 * pp + i) * (128 * 128) + (uint32_t)((j ^ (l & 7)) << 4), a[i][4 * j],
                           a[i][4 * j + 1], a[i][4 * j + 2], a[i][4 * j + 3]);
        }
        fence_proxy_async_smem();
      }
      // the staged tile is complete, and the warpgroup goes on (or gives up) together
      if (!named_bar_and(3, 128, got && !aborted_now())) { ok = false; break; }
      if (dw == 0) {
        const int h = head_of(u);
        const int q0 = n * C::BM + sub_of(u) * C::BQ;
        // blocks 0, 1 sit in the Q half, 2, 3 in the dO half: release each half once read
#pragma unroll
        for (int part = 0; part < D / 32; ++part) {
          tma_reduce_add_3d(&tm_dq, stg + part * (128 * 128), part * 32, h, start + q0);
          if (part == 1 || part == 3) bulk_commit();
        }
        bulk_wait_read1();
        mbar_arrive(&bars->q_free[stage]);
        bulk_wait_read();
        mbar_arrive(&bars->do_free[stage]);
      }
    }
    if (dw == 0) bulk_wait_all();
    if (!ok) abort_now();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

template <int D, bool GATHER>
cudaError_t launch_bwd_d(const AttnArgs& a, const void* o, const float* lse, const void* dout, void* dq, void* dk,
                         void* dv, void* ws, cudaStream_t st) {
  using C = Bwd<D>;
  char* w = static_cast<char*>(ws) + kWsHeader;
  float* dvec = reinterpret_cast<float*>(w);
  float* dq_acc = reinterpret_cast<float*>(w + align256((size_t)a.hq * a.num_tokens * 4));
  // gathered: fp32 trajectory-layout accumulators of dQ, dK, dV after the segment-layout dQ
  float *dq_t = nullptr, *dk_t = nullptr, *dv_t = nullptr;
  const int64_t rows = a.num_tokens * a.hq;
  if (GATHER) {
    char* t0 = reinterpret_cast<char*>(dq_acc) + align256((size_t)a.num_tokens * a.hq * D * 4);
    const size_t qb = align256((size_t)a.traj_tokens * a.hq * D * 4), kb = align256((size_t)a.traj_tokens * a.hkv * D * 4);
    dq_t = reinterpret_cast<float*>(t0);
    dk_t = reinterpret_cast<float*>(t0 + qb);
    dv_t = reinterpret_cast<float*>(t0 + qb + kb);
    if (cudaMemsetAsync(t0, 0, qb + 2 * kb, st) != cudaSuccess) return cudaErrorUnknown;
  }
  {
    const int64_t total = rows * (D / 8);
    int64_t blocks = (total + kPreThreads - 1) / kPreThreads;
    if (blocks > 152 * 32) blocks = 152 * 32;
    bwd_pre<D><<<(unsigned)blocks, kPreThreads, 0, st>>>(static_cast<const __nv_bfloat16*>(o),
                                                         static_cast<const __nv_bfloat16*>(dout), rows, a.hq,
                                                         a.num_tokens, dvec, dq_acc);
  }
  alignas(64) CUtensorMap tq, tk, tv, tdo, tqr, tkr, tvr, tqs, tks, tvs;
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
  if (!encode_tma_3d_bf16(&tdo, dout, D, a.hq, a.num_tokens, 64, 128)) return cudaErrorInvalidValue;
  const int ntiles = (a.max_seqlen + C::BM - 1) / C::BM;
  const int64_t gx = (int64_t)a.num_segments * a.hkv;
  if (gx > (int64_t)65535 * 65535) return cudaErrorInvalidConfiguration;
  dim3 grid((unsigned)ntiles, (unsigned)(gx < 65535 ? gx : 65535), (unsigned)((gx + 65534) / 65535));
  if (ntiles > 0) {
    if (D == 128) {
      static std::atomic<int> regs_cache{-1};
      bool regs_ok = false;
      if (cudaError_t e = launch_regs_match(reinterpret_cast<const void*>(bwd_main_d128<GATHER>), D128::REG_LAUNCH,
                                            &regs_cache, &regs_ok);
          e != cudaSuccess)
        return e;
      if (!regs_ok) return cudaErrorInvalidConfiguration;
      alignas(64) CUtensorMap tdq32;  // fp32 accumulator, [128 rows][32 dims] boxes, 128-byte swizzle
      if (!encode_tma_3d_f32(&tdq32, dq_acc, D, a.hq, a.num_tokens, 32, 128, true)) return cudaErrorInvalidValue;
      cudaError_t e =
          cudaFuncSetAttribute(bwd_main_d128<GATHER>, cudaFuncAttributeMaxDynamicSharedMemorySize, D128::SMEM);
      if (e != cudaSuccess) return e;
      bwd_main_d128<GATHER><<<grid, D128::THREADS, D128::SMEM, st>>>(
          tq, tk, tv, tdo, tdq32, a.cu_seqlens, a.num_segments, (int32_t)a.num_tokens, a.max_seqlen, a.hq, a.hkv,
          a.scale, a.scale * 1.4426950408889634f, lse, dvec, static_cast<__nv_bfloat16*>(dk),
          static_cast<__nv_bfloat16*>(dv), a.status, a.tok_gather, (int32_t)a.traj_tokens, dk_t, dv_t,
          GATHER ? tqr : tq, GATHER ? tkr : tk, GATHER ? tvr : tv, GATHER ? tqs : tq, GATHER ? tks : tk,
          GATHER ? tvs : tv);
    } else {
      cudaError_t e =
          cudaFuncSetAttribute(bwd_main<D, GATHER>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
      if (e != cudaSuccess) return e;
      bwd_main<D, GATHER><<<grid, kThreads, C::SMEM, st>>>(
          tq, tk, tv, tdo, a.cu_seqlens, a.num_segments, (int32_t)a.num_tokens, a.max_seqlen, a.hq, a.hkv, ntiles,
          a.scale, a.scale * 1.4426950408889634f, lse, dvec, dq_acc, static_cast<__nv_bfloat16*>(dk),
          static_cast<__nv_bfloat16*>(dv), a.status, a.tok_gather, (int32_t)a.traj_tokens, dk_t, dv_t,
          GATHER ? tqr : tq, GATHER ? tkr : tk, GATHER ? tvr : tv, GATHER ? tqs : tq, GATHER ? tks : tk,
          GATHER ? tvs : tv);
    }
  }
  auto convert = [&](const float* acc, void* out, int64_t elems) {
    const int64_t n8 = elems / 8;
    int64_t blocks = (n8 + 255) / 256;
    if (blocks > 152 * 32) blocks = 152 * 32;
    if (n8 > 0) bwd_dq_cvt<<<(unsigned)blocks, 256, 0, st>>>(acc, static_cast<__nv_bfloat16*>(out), n8);
  };
  if (GATHER) {
    const int32_t row_chunks = a.hq * D / 4;
    const int64_t total = a.num_tokens * row_chunks;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 152 * 32) blocks = 152 * 32;
    if (total > 0)
      bwd_dq_scatter<<<(unsigned)blocks, 256, 0, st>>>(dq_acc, a.tok_gather, a.num_tokens, row_chunks,
                                                       (int32_t)a.traj_tokens, dq_t);
    convert(dq_t, dq, a.traj_tokens * a.hq * D);
    convert(dk_t, dk, a.traj_tokens * a.hkv * D);
    convert(dv_t, dv, a.traj_tokens * a.hkv * D);
  } else {
    convert(dq_acc, dq, rows * D);
  }
  return cudaGetLastError();
}

}  // namespace

size_t attn_bwd_ws_bytes(const AttnArgs& a) {
  if (a.num_tokens < 0 || a.hq <= 0 || a.hkv <= 0 || a.d <= 0 || a.traj_tokens < 0) return kWsHeader;
  size_t b = kWsHeader + align256((size_t)a.hq * a.num_tokens * 4) + align256((size_t)a.num_tokens * a.hq * a.d * 4);
  if (a.traj_tokens > 0)  // gathered: fp32 trajectory-layout dQ, dK, dV accumulators
    b += align256((size_t)a.traj_tokens * a.hq * a.d * 4) + 2 * align256((size_t)a.traj_tokens * a.hkv * a.d * 4);
  return b;
}

cudaError_t launch_attn_bwd(const AttnArgs& a, const void* o, const float* lse, const void* dout, void* dq, void* dk,
                            void* dv, void* ws, cudaStream_t st) {
  if (a.tok_gather != nullptr) {
    if (a.d == 64) return launch_bwd_d<64, true>(a, o, lse, dout, dq, dk, dv, ws, st);
    return launch_bwd_d<128, true>(a, o, lse, dout, dq, dk, dv, ws, st);
  }
  if (a.d == 64) return launch_bwd_d<64, false>(a, o, lse, dout, dq, dk, dv, ws, st);
  return launch_bwd_d<128, false>(a, o, lse, dout, dq, dk, dv, ws, st);
}

}  // namespace vcs
