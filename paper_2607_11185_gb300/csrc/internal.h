// internal.h - launchers shared between the C-ABI layer (api.cu) and the
// kernel translation units.  Not part of the public interface.
#pragma once

#include <atomic>
#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>

#include "vcs.h"

namespace vcs {

// A named NVTX range around one C-ABI call, so that a profiler's timeline (Nsight Systems,
// Nsight Compute's range filters) shows each entry point and the launches it made.  NVTX is
// header-only here: with no tool attached a push or pop costs a few nanoseconds.
struct ApiRange {
  explicit ApiRange(const char* name) { nvtxRangePushA(name); }
  ~ApiRange() { nvtxRangePop(); }
  ApiRange(const ApiRange&) = delete;
  ApiRange& operator=(const ApiRange&) = delete;
};

// ---- segment builder (segments.cu) ----
struct SegWorkspace {
  int64_t* step_off;    // [num_steps+1] exclusive prefix of img+txt over all steps
  int64_t* txt_pre;     // [num_steps+1] exclusive prefix of txt over all steps
  int32_t* traj_nseg;   // [num_traj]
  int64_t* traj_ntok;   // [num_traj]
  int32_t* traj_maxlen; // [num_traj]
  int64_t* seg_base;    // [num_traj+1]
  int64_t* tok_base;    // [num_traj+1]
  int64_t* seg_start;   // [num_steps+1] start of every segment in the packed buffer
  int32_t* seg_full;    // [num_steps] global step of the first full (screenshot) step a_j
  int32_t* seg_new;     // [num_steps] global step of the first new step s_j
  int32_t* seg_last;    // [num_steps] global step of the last step e_j
  int32_t* seg_first;   // [num_steps] global step of the trajectory's first step
  int64_t* totals;      // [4]: num_segments, num_tokens, max_seqlen, status
};
size_t seg_workspace_bytes(int32_t num_traj, int64_t num_steps);
SegWorkspace seg_workspace_carve(void* ws, int32_t num_traj, int64_t num_steps);

cudaError_t launch_seg_plan(const int32_t* cu_steps, int32_t num_traj, int64_t num_steps, const int32_t* step_img,
                            const int32_t* step_txt, int32_t window, int32_t keep, int64_t seg_capacity,
                            int64_t tok_capacity, vcs_sizes* sizes, const SegWorkspace& w, cudaStream_t st);
cudaError_t launch_seg_build(const int32_t* cu_steps, int32_t num_traj, int32_t window, int32_t keep,
                             const int32_t* step_img, int32_t* cu_seqlens, int32_t* seg_traj, int32_t* tok_gather,
                             int32_t* tok_src_step, int32_t* tok_pos, uint8_t* tok_loss_mask,
                             const SegWorkspace& w, cudaStream_t st);

// ---- gather (gather.cu) ----
cudaError_t launch_gather(const void* src, int64_t traj_tokens, const int32_t* tok_gather, int64_t num_tokens,
                          int64_t row_bytes, void* dst, int32_t* dev_status, cudaStream_t st);

// ---- attention (attn_fwd.cu, attn_bwd.cu) ----
struct AttnArgs {
  const void* q;
  const void* k;
  const void* v;
  const int32_t* cu_seqlens;
  int32_t num_segments;
  int64_t num_tokens;
  int32_t max_seqlen;
  int32_t hq, hkv, d;
  float scale;
  int32_t* status;  // device status word (workspace header)
  // gathered variants: q, k, v are trajectory-layout [traj_tokens, heads, d] tensors and
  // segment token n reads trajectory row tok_gather[n]; nullptr for segment-layout inputs
  const int32_t* tok_gather = nullptr;
  int64_t traj_tokens = 0;
  // prefix reuse (forward): per segment, the length of its common prefix with the previous
  // segment of its trajectory (vcs_shared_prefix); nullptr computes every row
  const int32_t* seg_shared = nullptr;
};
size_t attn_fwd_ws_bytes(const AttnArgs& a);
cudaError_t launch_attn_fwd(const AttnArgs& a, void* o, float* lse, void* ws, cudaStream_t st);
size_t attn_bwd_ws_bytes(const AttnArgs& a);
cudaError_t launch_attn_bwd(const AttnArgs& a, const void* o, const float* lse, const void* dout, void* dq, void* dk,
                            void* dv, void* ws, cudaStream_t st);

// ---- RL objective over segments (loss.cu) ----
size_t grpo_loss_ws_bytes(int64_t num_tokens);
cudaError_t launch_grpo_loss(const float* logp, const float* old_logp, const float* ref_logp, const uint8_t* mask,
                             const int32_t* cu_seqlens, const int32_t* seg_traj, int32_t num_segments,
                             int32_t num_tokens, const float* adv, int32_t num_traj, float lo, float hi,
                             float clip_cap, float kl_coef, double* loss, float* dlogp, void* ws, cudaStream_t st);
cudaError_t launch_group_advantage(const float* rewards, int64_t num_groups, int32_t group_size, float eps,
                                   float* adv, cudaStream_t st);

// ---- token-ID stream fields and trainable-token compaction (stream.cu) ----
cudaError_t launch_stream_fields(const int32_t* traj_ids, const float* traj_logp, int64_t traj_tokens,
                                 const int32_t* tok_gather, const uint8_t* mask, int64_t num_tokens, int32_t* ids,
                                 float* logp, int32_t* status, cudaStream_t st);
size_t compact_ws_bytes(int64_t num_tokens);
cudaError_t launch_compact(const uint8_t* mask, int64_t num_tokens, int32_t* idx, int64_t capacity, int64_t* count,
                           void* ws, cudaStream_t st);

cudaError_t launch_shared_prefix(const int32_t* cu_seqlens, const int32_t* seg_traj, const int32_t* tok_gather,
                                 int32_t num_segments, int32_t num_tokens, int32_t* seg_shared, int32_t* status,
                                 cudaStream_t st);

// TMA descriptor encoding through the driver entry point (no libcuda link).
bool encode_tma_3d_bf16(void* map /*CUtensorMap*/, const void* base, uint64_t d, uint64_t heads, uint64_t tokens,
                        uint32_t box_d, uint32_t box_rows);

// 2-D map over a row-major [rows, row_elems] bf16 tensor with a 64-column x 1-row box and the
// 128-byte swizzle: the map of the TMA gather4 loads (one row per gathered token)
bool encode_tma_rows_bf16(void* map, const void* base, uint64_t row_elems, uint64_t rows);
// fp32 variant of encode_tma_3d_bf16 (bulk reduce-add targets): no swizzle, or the 128-byte
// swizzle (box_d * 4 must then be 128).
bool encode_tma_3d_f32(void* map, const void* base, uint64_t d, uint64_t heads, uint64_t tokens, uint32_t box_d,
                       uint32_t box_rows, bool swizzle128 = false);

constexpr size_t kWsHeader = 256;  // attention workspace header (status word first)

// Whether kernel fn was built with exactly `want` registers per thread: a kernel whose
// warpgroups move registers with setmaxnreg is served from the registers its block is launched
// with, so a build that got another count must not run.  The answer is cached in *cache
// (-1 until first asked); concurrent first calls from several host threads are safe.
inline cudaError_t launch_regs_match(const void* fn, int want, std::atomic<int>* cache, bool* ok) {
  int c = cache->load(std::memory_order_relaxed);
  if (c < 0) {
    cudaFuncAttributes fa;
    const cudaError_t e = cudaFuncGetAttributes(&fa, fn);
    if (e != cudaSuccess) return e;
    c = fa.numRegs == want ? 1 : 0;
    cache->store(c, std::memory_order_relaxed);
  }
  *ok = c == 1;
  return cudaSuccess;
}

}  // namespace vcs
