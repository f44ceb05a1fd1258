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
// diagonal tile is masked element-wise.  Grid: x = (segment, head), y = pair
// index in decreasing order, so the longest rows of work start first.
//
// Warp roles (384 threads):
//   warp 0      TMA producer: Q0/Q1 once, then K0,V0,K1,V1,... into a 3-slot ring
//   warp 1      TMEM allocator and single-thread tcgen05.mma issuer
//   warps 2-3   idle (they keep the softmax warps on TMEM lane quadrants 0-3)
//   warps 4-7   softmax + epilogue for tile 0 (thread = query row)
//   warps 8-11  softmax + epilogue for tile 1
// TMEM (512 columns x 128 lanes, fp32): S0 [0,128), S1 [128,256),
// O0 [256,256+D), O1 [384,384+D).
//
// Per K/V tile j the MMA thread issues, in order,
//   S0(j+1) = Q0 K_{j+1}^T  once softmax 0 has copied S0(j) to registers,
//   S1(j+1) = Q1 K_{j+1}^T  likewise for tile 1,
//   PV0(j):  O0 += P0(j) V_j once P0(j) is in shared memory,
//   PV1(j):  O1 += P1(j) V_j,
// so the next scores are computed while the softmax warps still work on the
// current ones, and the two tiles keep the tensor pipe busy in turn.  P goes
// through shared memory in the 128-byte-swizzled K-major layout the MMA
// reads; a softmax warp computes its P in registers and only waits for the
// previous P.V of its tile before storing it.
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
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct Fwd {
  static constexpr int BM = 128;
  static constexpr int BN = 128;
  static constexpr int KB = D / 64;                 // 128-byte column blocks per row
  static constexpr int TILE = BM * D * 2;           // bytes of a 128 x D bf16 tile
  static constexpr int BLOCK = BM * 128;            // bytes of one 128 x 64 column block
  static constexpr int PTILE = BM * BN * 2;         // bytes of a 128 x 128 bf16 P tile
  static constexpr int NSLOT = 3;
  static constexpr int OFF_Q0 = 0;
  static constexpr int OFF_Q1 = TILE;
  static constexpr int OFF_KV = 2 * TILE;
  static constexpr int OFF_P0 = OFF_KV + NSLOT * TILE;
  static constexpr int OFF_P1 = OFF_P0 + PTILE;
  static constexpr int OFF_BAR = OFF_P1 + PTILE;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr int TM_S0 = 0, TM_S1 = 128, TM_O0 = 256, TM_O1 = 384;
  static constexpr uint32_t IDESC_S = idesc_bf16(128, 128, 0, 0);   // Q (K-major) x K^T (K-major)
  static constexpr uint32_t IDESC_PV = idesc_bf16(128, D, 0, 1);    // P (K-major) x V (MN-major)
};

struct Bars {
  uint64_t q_full;
  uint64_t kv_full[3];
  uint64_t kv_empty[3];
  uint64_t s_full[2];
  uint64_t s_consumed[2];
  uint64_t p_full[2];
  uint64_t pv_done[2];
  uint32_t tmem_base;
  int32_t abort;
};

__device__ __forceinline__ void on_timeout(Bars* b, int32_t* status) {
  set_status(status, VCS_ERR_DEVICE_TIMEOUT);
  *reinterpret_cast<volatile int32_t*>(&b->abort) = 1;
}
__device__ __forceinline__ bool aborted(Bars* b) { return *reinterpret_cast<volatile int32_t*>(&b->abort) != 0; }

template <int D>
__device__ __forceinline__ void issue_s(uint32_t tmem_d, uint32_t q_addr, uint32_t k_addr) {
  using C = Fwd<D>;
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    const uint32_t off = (kk >> 2) * C::BLOCK + (kk & 3) * 32;
    tc_mma_ss(tmem_d, smem_desc(q_addr + off, 16, 1024), smem_desc(k_addr + off, 16, 1024), C::IDESC_S, kk > 0);
  }
}

template <int D>
__device__ __forceinline__ void issue_pv(uint32_t tmem_d, uint32_t p_addr, uint32_t v_addr, bool accumulate) {
  using C = Fwd<D>;
#pragma unroll
  for (int kk = 0; kk < C::BN / 16; ++kk) {
    const uint32_t aoff = (kk >> 2) * C::BLOCK + (kk & 3) * 32;
    const uint32_t boff = kk * 16 * 128;  // 16 key rows of 128 bytes
    tc_mma_ss(tmem_d, smem_desc(p_addr + aoff, 16, 1024), smem_desc(v_addr + boff, C::BLOCK, 1024), C::IDESC_PV,
              (accumulate || kk > 0) ? 1u : 0u);
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ CUtensorMap tm_v, const int32_t* __restrict__ cu_seqlens,
                    int32_t num_segments, int32_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv,
                    int32_t npairs, float scale_log2, __nv_bfloat16* __restrict__ out, float* __restrict__ lse,
                    int32_t* status) {
  using C = Fwd<D>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + C::OFF_BAR);

  // once any CTA of this launch has given up on a wait, the rest stand down
  if (*reinterpret_cast<volatile int32_t*>(status) == VCS_ERR_DEVICE_TIMEOUT) return;
  const int seg = blockIdx.x / hq;
  const int h = blockIdx.x - seg * hq;
  const int p = npairs - 1 - (int)blockIdx.y;
  const int start = cu_seqlens[seg];
  const int end = cu_seqlens[seg + 1];
  if (start < 0 || end < start || end > num_tokens || end - start > max_seqlen ||
      (seg == 0 && start != 0) || (seg == num_segments - 1 && end != num_tokens)) {
    if (threadIdx.x == 0 && p == 0 && h == 0) set_status(status, VCS_ERR_DEVICE_CHECK);
    return;
  }
  const int L = end - start;
  if (p * 2 * C::BM >= L) return;  // this pair of query tiles lies beyond the segment
  const int m0 = 2 * p, m1 = 2 * p + 1;
  const bool has1 = m1 * C::BM < L;
  const int nkv = has1 ? m1 + 1 : m0 + 1;
  const int g = h / (hq / hkv);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t sbase = smem_u32(smem);

  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    for (int i = 0; i < 3; ++i) {
      mbar_init(&bars->kv_full[i], 1);
      mbar_init(&bars->kv_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->s_consumed[i], 128);
      mbar_init(&bars->p_full[i], 128);
      mbar_init(&bars->pv_done[i], 1);
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

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
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
      // ring order K0, K1, V0, K2, V1, ..., K_{n-1}, V_{n-2}, V_{n-1}: keys run one
      // tile ahead of values, since S(j+1) is issued before P(j).V_j
      for (int c = 0; c < 2 * nkv; ++c) {
        const bool is_v = c == 2 * nkv - 1 || (c > 0 && (c & 1) == 0);
        const int j = c == 2 * nkv - 1 ? nkv - 1 : (is_v ? (c - 2) >> 1 : (c + 1) >> 1);
        const int slot = c % 3, round = c / 3;
        if (c >= 3 && !mbar_wait(&bars->kv_empty[slot], (round - 1) & 1)) {
          on_timeout(bars, status);
          break;
        }
        if (aborted(bars)) break;
        mbar_arrive_expect_tx(&bars->kv_full[slot], C::TILE);
        const CUtensorMap* tm = is_v ? &tm_v : &tm_k;
#pragma unroll
        for (int kb = 0; kb < C::KB; ++kb)
          tma_load_3d_hint(smem + C::OFF_KV + slot * C::TILE + kb * C::BLOCK, tm, &bars->kv_full[slot], kb * 64, g,
                           start + j * C::BN, keep_l2);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      bool ok = mbar_wait(&bars->q_full, 0);
      auto acquire = [&](int c, uint32_t& addr) -> bool {
        const int slot = c % 3;
        if (!mbar_wait(&bars->kv_full[slot], (c / 3) & 1)) return false;
        tc_fence_after();
        addr = sbase + C::OFF_KV + slot * C::TILE;
        return true;
      };
      // positions of K_j and V_j in the producer's ring order
      auto k_item = [&](int j) { return j == 0 ? 0 : 2 * j - 1; };
      auto v_item = [&](int j) { return j == nkv - 1 ? 2 * nkv - 1 : 2 * j + 2; };
      uint32_t kaddr = 0, vaddr = 0;
      if (ok) ok = acquire(0, kaddr);
      if (ok) {
        issue_s<D>(tmem + C::TM_S0, sbase + C::OFF_Q0, kaddr);
        tc_commit(&bars->s_full[0]);
        if (has1) {
          issue_s<D>(tmem + C::TM_S1, sbase + C::OFF_Q1, kaddr);
          tc_commit(&bars->s_full[1]);
        }
        tc_commit(&bars->kv_empty[0]);
      }
      for (int j = 0; ok && j < nkv; ++j) {
        const bool next = j + 1 < nkv;
        // S(j+1) of each tile as soon as its softmax has pulled S(j) out of TMEM
        if (next) {
          if (!acquire(k_item(j + 1), kaddr)) { ok = false; break; }
          if (j + 1 <= m0) {
            if (!mbar_wait(&bars->s_consumed[0], j & 1)) { ok = false; break; }
            tc_fence_after();
            issue_s<D>(tmem + C::TM_S0, sbase + C::OFF_Q0, kaddr);
            tc_commit(&bars->s_full[0]);
          }
          if (has1) {
            if (!mbar_wait(&bars->s_consumed[1], j & 1)) { ok = false; break; }
            tc_fence_after();
            issue_s<D>(tmem + C::TM_S1, sbase + C::OFF_Q1, kaddr);
            tc_commit(&bars->s_full[1]);
          }
          tc_commit(&bars->kv_empty[k_item(j + 1) % 3]);
        }
        // then O += P(j) V_j as each tile's P arrives
        if (!acquire(v_item(j), vaddr)) { ok = false; break; }
        if (j <= m0) {
          if (!mbar_wait(&bars->p_full[0], j & 1)) { ok = false; break; }
          tc_fence_after();
          issue_pv<D>(tmem + C::TM_O0, sbase + C::OFF_P0, vaddr, j > 0);
          tc_commit(&bars->pv_done[0]);
        }
        if (has1) {
          if (!mbar_wait(&bars->p_full[1], j & 1)) { ok = false; break; }
          tc_fence_after();
          issue_pv<D>(tmem + C::TM_O1, sbase + C::OFF_P1, vaddr, j > 0);
          tc_commit(&bars->pv_done[1]);
        }
        tc_commit(&bars->kv_empty[v_item(j) % 3]);
        if (aborted(bars)) { ok = false; break; }
      }
      if (!ok) on_timeout(bars, status);
    }
  } else if (warp >= 4) {
    // ------------------------------------------------------------ softmax
    const int wg = (warp - 4) >> 2;
    const int quad = warp & 3;
    const int r = quad * 32 + lane;  // query row within the tile
    if (wg == 0 || has1) {
      const int mt = wg == 0 ? m0 : m1;
      const uint32_t trow = tmem + ((uint32_t)(quad * 32) << 16);
      const uint32_t s_col = wg == 0 ? C::TM_S0 : C::TM_S1;
      const uint32_t o_col = wg == 0 ? C::TM_O0 : C::TM_O1;
      const uint32_t p_addr = sbase + (wg == 0 ? C::OFF_P0 : C::OFF_P1);
      float m_run = -FLT_MAX, l = 0.f;
      bool ok = true;
      for (int j = 0; j <= mt; ++j) {
        if (!mbar_wait(&bars->s_full[wg], j & 1)) { ok = false; break; }
        tc_fence_after();
        uint32_t s[128];
#pragma unroll
        for (int c = 0; c < 4; ++c)
          tmem_ld_32x32b_x32(trow + s_col + c * 32, *reinterpret_cast<uint32_t(*)[32]>(&s[c * 32]));
        tmem_ld_wait();
        reg_fence<128>(s);
        // S of this tile is in registers: the MMA may overwrite it with S(j+1)
        tc_fence_before();
        mbar_arrive(&bars->s_consumed[wg]);
        if (j == mt) {  // diagonal tile: key c is visible to row r iff c <= r
#pragma unroll
          for (int c = 0; c < 128; ++c)
            if (c > r) s[c] = __float_as_uint(-FLT_MAX);
        }
        // row maximum: 8 independent three-input chains (short dependency chains,
        // two elements per instruction)
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
        // P in registers (bf16 pairs, packed over S) before waiting for the previous P.V;
        // the scale-and-shift and the row sums run on packed fp32 pairs
        const uint64_t sc2 = f2pack(scale_log2, scale_log2);
        const uint64_t nm2 = f2pack(-m_run, -m_run);
        uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};  // independent partial row sums
#pragma unroll
        for (int c2 = 0; c2 < 64; ++c2) {
          float x0, x1;
          f2unpack(ffma2(f2pack(__uint_as_float(s[2 * c2]), __uint_as_float(s[2 * c2 + 1])), sc2, nm2), x0, x1);
          const float p0 = ex2(x0), p1 = ex2(x1);
          acc[c2 & 3] = fadd2(acc[c2 & 3], f2pack(p0, p1));
          s[c2] = pack_bf16(p0, p1);
        }
        float rsp[4];
        {
          float a0, a1, b0, b1;
          f2unpack(fadd2(acc[0], acc[1]), a0, a1);
          f2unpack(fadd2(acc[2], acc[3]), b0, b1);
          rsp[0] = a0;
          rsp[1] = a1;
          rsp[2] = b0;
          rsp[3] = b1;
        }
        // the previous P.V of this tile must be done before P and O change
        if (j > 0) {
          if (!mbar_wait(&bars->pv_done[wg], (j - 1) & 1)) { ok = false; break; }
          tc_fence_after();
        }
#pragma unroll
        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
          for (int ch = 0; ch < 8; ++ch) {
            const int w0 = kb * 32 + ch * 4;
            st_shared_v4(p_addr + kb * C::BLOCK + r * 128 + ((ch ^ (r & 7)) << 4), s[w0], s[w0 + 1], s[w0 + 2],
                         s[w0 + 3]);
          }
        l = l * alpha + ((rsp[0] + rsp[1]) + (rsp[2] + rsp[3]));
        if (j > 0 && __any_sync(0xffffffffu, rescale)) {
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            uint32_t o[32];
            tmem_ld_32x32b_x32(trow + o_col + c * 32, o);
            tmem_ld_wait();
            reg_fence<32>(o);
#pragma unroll
            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
            tmem_st_32x32b_x32(trow + o_col + c * 32, o);
          }
          tmem_st_wait();
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(&bars->p_full[wg]);
        if (aborted(bars)) { ok = false; break; }
      }
      if (ok && !mbar_wait(&bars->pv_done[wg], mt & 1)) ok = false;
      if (!ok) {
        on_timeout(bars, status);
      } else {
        tc_fence_after();
        const int row = mt * C::BM + r;
        const bool valid = row < L;
        const float inv_l = 1.f / l;
        __nv_bfloat16* orow = out + ((size_t)(start + row) * hq + h) * D;
#pragma unroll
        for (int c = 0; c < D / 32; ++c) {
          uint32_t o[32];
          tmem_ld_32x32b_x32(trow + o_col + c * 32, o);
          tmem_ld_wait();
          reg_fence<32>(o);
          if (valid) {
            uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
            for (int v4 = 0; v4 < 4; ++v4) {
              uint4 pk;
              pk.x = pack_bf16(__uint_as_float(o[v4 * 8 + 0]) * inv_l, __uint_as_float(o[v4 * 8 + 1]) * inv_l);
              pk.y = pack_bf16(__uint_as_float(o[v4 * 8 + 2]) * inv_l, __uint_as_float(o[v4 * 8 + 3]) * inv_l);
              pk.z = pack_bf16(__uint_as_float(o[v4 * 8 + 4]) * inv_l, __uint_as_float(o[v4 * 8 + 5]) * inv_l);
              pk.w = pack_bf16(__uint_as_float(o[v4 * 8 + 6]) * inv_l, __uint_as_float(o[v4 * 8 + 7]) * inv_l);
              dst[v4] = pk;
            }
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

template <int D>
cudaError_t launch_fwd_d(const AttnArgs& a, void* o, float* lse, cudaStream_t st) {
  using C = Fwd<D>;
  alignas(64) CUtensorMap tq, tk, tv;
  if (!encode_tma_3d_bf16(&tq, a.q, D, a.hq, a.num_tokens, 64, 128) ||
      !encode_tma_3d_bf16(&tk, a.k, D, a.hkv, a.num_tokens, 64, 128) ||
      !encode_tma_3d_bf16(&tv, a.v, D, a.hkv, a.num_tokens, 64, 128))
    return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  const int npairs = (a.max_seqlen + 2 * C::BM - 1) / (2 * C::BM);
  if (npairs == 0) return cudaSuccess;
  const int64_t gx = (int64_t)a.num_segments * a.hq;
  if (gx > INT32_MAX || npairs > 65535) return cudaErrorInvalidConfiguration;
  const float scale_log2 = a.scale * 1.4426950408889634f;
  dim3 grid((unsigned)gx, (unsigned)npairs, 1);
  attn_fwd_kernel<D><<<grid, kThreads, C::SMEM, st>>>(tq, tk, tv, a.cu_seqlens, a.num_segments, (int32_t)a.num_tokens,
                                                     a.max_seqlen, a.hq, a.hkv, npairs, scale_log2,
                                                     static_cast<__nv_bfloat16*>(o), lse, a.status);
  return cudaGetLastError();
}

}  // namespace

size_t attn_fwd_ws_bytes(const AttnArgs& a) {
  (void)a;
  return kWsHeader;
}

cudaError_t launch_attn_fwd(const AttnArgs& a, void* o, float* lse, void* ws, cudaStream_t st) {
  (void)ws;
  if (a.d == 64) return launch_fwd_d<64>(a, o, lse, st);
  return launch_fwd_d<128>(a, o, lse, st);
}

}  // namespace vcs
