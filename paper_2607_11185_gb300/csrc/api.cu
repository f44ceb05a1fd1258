// api.cu - the extern "C" boundary of libvcs.so (declared in include/vcs.h).
//
// Host-side validation happens here, before any launch: pointers, counts,
// alignment, supported shapes, workspace size.  Everything that depends on
// device data (cu_steps, cu_seqlens, gather indices) is validated by the
// kernels themselves, which record a status word instead of trapping.
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "internal.h"

namespace vcs {

namespace {

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline cudaStream_t as_stream(void* s) { return static_cast<cudaStream_t>(s); }

PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::once_flag g_encode_once;

void load_encode_fn() {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
      q == cudaDriverEntryPointSuccess)
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
}

vcs_status check_attn(const AttnArgs& a) {
  if (a.q == nullptr || a.k == nullptr || a.v == nullptr || a.cu_seqlens == nullptr) return VCS_ERR_INVALID_ARG;
  if (a.num_segments < 0 || a.num_tokens < 0 || a.max_seqlen < 0 || a.hq <= 0 || a.hkv <= 0)
    return VCS_ERR_INVALID_ARG;
  if (a.num_tokens > INT32_MAX - 256) return VCS_ERR_OVERFLOW;
  if (a.d != 64 && a.d != 128) return VCS_ERR_UNSUPPORTED;
  if (a.hq % a.hkv != 0) return VCS_ERR_UNSUPPORTED;
  if (a.hq > 65535 || a.hkv > 65535) return VCS_ERR_UNSUPPORTED;
  if (!aligned16(a.q) || !aligned16(a.k) || !aligned16(a.v)) return VCS_ERR_INVALID_ARG;
  return VCS_OK;
}

}  // namespace

bool encode_tma_3d_bf16(void* map, const void* base, uint64_t d, uint64_t heads, uint64_t tokens, uint32_t box_d,
                        uint32_t box_rows) {
  std::call_once(g_encode_once, load_encode_fn);
  if (g_encode == nullptr) return false;
  // dims innermost first: (d, heads, tokens); a box is box_d x 1 head x box_rows tokens
  cuuint64_t dims[3] = {d, heads, tokens > 0 ? tokens : 1};
  cuuint64_t strides[2] = {d * 2, heads * d * 2};
  cuuint32_t box[3] = {box_d, 1, box_rows};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(static_cast<CUtensorMap*>(map), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base),
                        dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_tma_rows_bf16(void* map, const void* base, uint64_t row_elems, uint64_t rows) {
  std::call_once(g_encode_once, load_encode_fn);
  if (g_encode == nullptr) return false;
  cuuint64_t dims[2] = {row_elems, rows > 0 ? rows : 1};
  cuuint64_t strides[1] = {row_elems * 2};
  cuuint32_t box[2] = {64, 1};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(static_cast<CUtensorMap*>(map), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base),
                        dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_tma_3d_f32(void* map, const void* base, uint64_t d, uint64_t heads, uint64_t tokens, uint32_t box_d,
                       uint32_t box_rows, bool swizzle128) {
  std::call_once(g_encode_once, load_encode_fn);
  if (g_encode == nullptr) return false;
  cuuint64_t dims[3] = {d, heads, tokens > 0 ? tokens : 1};
  cuuint64_t strides[2] = {d * 4, heads * d * 4};
  cuuint32_t box[3] = {box_d, 1, box_rows};
  cuuint32_t estr[3] = {1, 1, 1};
  if (swizzle128 && box_d * 4 != 128) return false;
  CUresult r = g_encode(static_cast<CUtensorMap*>(map), CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(base),
                        dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace vcs

using namespace vcs;

extern "C" {

const char* vcs_status_string(int32_t status) {
  switch (status) {
    case VCS_OK: return "VCS_OK";
    case VCS_ERR_INVALID_ARG: return "VCS_ERR_INVALID_ARG: null pointer, negative count, misaligned pointer or bad window";
    case VCS_ERR_UNSUPPORTED: return "VCS_ERR_UNSUPPORTED: head_dim must be 64 or 128 and hq a multiple of hkv";
    case VCS_ERR_CAPACITY: return "VCS_ERR_CAPACITY: an output buffer is smaller than the layout";
    case VCS_ERR_OVERFLOW: return "VCS_ERR_OVERFLOW: a token count exceeds INT32_MAX";
    case VCS_ERR_CUDA: return "VCS_ERR_CUDA: a CUDA call failed";
    case VCS_ERR_DEVICE_CHECK: return "VCS_ERR_DEVICE_CHECK: a kernel found inconsistent input data";
    case VCS_ERR_DEVICE_TIMEOUT: return "VCS_ERR_DEVICE_TIMEOUT: a bounded device wait gave up";
    case VCS_ERR_WORKSPACE: return "VCS_ERR_WORKSPACE: workspace missing or too small";
    default: return "VCS_ERR_UNKNOWN";
  }
}

const char* vcs_version(void) { return "libvcs 0.1 sm_103a"; }

size_t vcs_segments_workspace_size(int32_t num_traj, int64_t num_steps) {
  if (num_traj < 0 || num_steps < 0) return 0;
  return seg_workspace_bytes(num_traj, num_steps);
}

static vcs_status check_seg_args(const int32_t* cu_steps, int32_t num_traj, int64_t num_steps, const int32_t* step_img,
                                 const int32_t* step_txt, int32_t window, int32_t keep, const void* sizes,
                                 const void* ws, size_t ws_bytes) {
  if (cu_steps == nullptr || sizes == nullptr) return VCS_ERR_INVALID_ARG;
  if (num_traj < 0 || num_steps < 0 || window < 1 || keep < 0) return VCS_ERR_INVALID_ARG;
  if (num_steps > 0 && (step_img == nullptr || step_txt == nullptr)) return VCS_ERR_INVALID_ARG;
  if (num_steps > INT32_MAX - 1) return VCS_ERR_OVERFLOW;
  if ((int64_t)keep + window > INT32_MAX / 2) return VCS_ERR_INVALID_ARG;
  if (ws == nullptr || ws_bytes < seg_workspace_bytes(num_traj, num_steps)) return VCS_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) & 255u) != 0) return VCS_ERR_INVALID_ARG;
  return VCS_OK;
}

vcs_status vcs_plan_segments(const int32_t* cu_steps, int32_t num_traj, int64_t num_steps, const int32_t* step_img,
                             const int32_t* step_txt, int32_t window, int32_t keep, vcs_sizes* sizes, void* ws,
                             size_t ws_bytes, void* stream) {
  vcs::ApiRange nvtx_range("vcs_plan_segments");
  vcs_status s = check_seg_args(cu_steps, num_traj, num_steps, step_img, step_txt, window, keep, sizes, ws, ws_bytes);
  if (s != VCS_OK) return s;
  SegWorkspace w = seg_workspace_carve(ws, num_traj, num_steps);
  if (launch_seg_plan(cu_steps, num_traj, num_steps, step_img, step_txt, window, keep, -1, -1, sizes, w,
                      as_stream(stream)) != cudaSuccess)
    return VCS_ERR_CUDA;
  return VCS_OK;
}

vcs_status vcs_build_segments(const int32_t* cu_steps, int32_t num_traj, int64_t num_steps, const int32_t* step_img,
                              const int32_t* step_txt, int32_t window, int32_t keep, int64_t seg_capacity,
                              int64_t tok_capacity, int32_t* cu_seqlens, int32_t* seg_traj, int32_t* tok_gather,
                              int32_t* tok_src_step, int32_t* tok_pos, uint8_t* tok_loss_mask, vcs_sizes* sizes,
                              void* ws, size_t ws_bytes, void* stream) {
  vcs::ApiRange nvtx_range("vcs_build_segments");
  vcs_status s = check_seg_args(cu_steps, num_traj, num_steps, step_img, step_txt, window, keep, sizes, ws, ws_bytes);
  if (s != VCS_OK) return s;
  if (seg_capacity < 0 || tok_capacity < 0 || cu_seqlens == nullptr) return VCS_ERR_INVALID_ARG;
  if (tok_capacity > 0 && (tok_gather == nullptr || tok_src_step == nullptr || tok_pos == nullptr))
    return VCS_ERR_INVALID_ARG;
  SegWorkspace w = seg_workspace_carve(ws, num_traj, num_steps);
  cudaStream_t st = as_stream(stream);
  if (launch_seg_plan(cu_steps, num_traj, num_steps, step_img, step_txt, window, keep, seg_capacity, tok_capacity,
                      sizes, w, st) != cudaSuccess)
    return VCS_ERR_CUDA;
  if (launch_seg_build(cu_steps, num_traj, window, keep, step_img, cu_seqlens, seg_traj, tok_gather, tok_src_step,
                       tok_pos, tok_loss_mask, w, st) != cudaSuccess)
    return VCS_ERR_CUDA;
  return VCS_OK;
}

vcs_status vcs_gather(const void* q_traj, const void* k_traj, const void* v_traj, int64_t traj_tokens,
                      const int32_t* tok_gather, int64_t num_tokens, int32_t hq, int32_t hkv, int32_t d, void* q,
                      void* k, void* v, int32_t* dev_status, void* stream) {
  vcs::ApiRange nvtx_range("vcs_gather");
  if (traj_tokens < 0 || num_tokens < 0 || hq <= 0 || d <= 0) return VCS_ERR_INVALID_ARG;
  if (num_tokens > 0 && (tok_gather == nullptr || q_traj == nullptr || q == nullptr)) return VCS_ERR_INVALID_ARG;
  const bool with_kv = k_traj != nullptr || v_traj != nullptr || k != nullptr || v != nullptr;
  if (with_kv && (k_traj == nullptr || v_traj == nullptr || k == nullptr || v == nullptr || hkv <= 0))
    return VCS_ERR_INVALID_ARG;
  if ((d * 2) % 16 != 0) return VCS_ERR_UNSUPPORTED;
  const void* ptrs[6] = {q_traj, k_traj, v_traj, q, k, v};
  for (const void* p : ptrs)
    if (p != nullptr && !aligned16(p)) return VCS_ERR_INVALID_ARG;
  cudaStream_t st = as_stream(stream);
  if (launch_gather(q_traj, traj_tokens, tok_gather, num_tokens, (int64_t)hq * d * 2, q, dev_status, st) !=
      cudaSuccess)
    return VCS_ERR_CUDA;
  if (with_kv) {
    if (launch_gather(k_traj, traj_tokens, tok_gather, num_tokens, (int64_t)hkv * d * 2, k, dev_status, st) !=
        cudaSuccess)
      return VCS_ERR_CUDA;
    if (launch_gather(v_traj, traj_tokens, tok_gather, num_tokens, (int64_t)hkv * d * 2, v, dev_status, st) !=
        cudaSuccess)
      return VCS_ERR_CUDA;
  }
  return VCS_OK;
}

static AttnArgs make_args(const void* q, const void* k, const void* v, const int32_t* cu_seqlens,
                          int32_t num_segments, int64_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv,
                          int32_t d, float scale) {
  AttnArgs a;
  a.q = q;
  a.k = k;
  a.v = v;
  a.cu_seqlens = cu_seqlens;
  a.num_segments = num_segments;
  a.num_tokens = num_tokens;
  a.max_seqlen = max_seqlen;
  a.hq = hq;
  a.hkv = hkv;
  a.d = d;
  a.scale = (scale > 0.f && std::isfinite(scale)) ? scale : 1.0f / std::sqrt((float)(d > 0 ? d : 1));
  a.status = nullptr;
  return a;
}

size_t vcs_attn_fwd_workspace_size(int32_t num_segments, int64_t num_tokens, int32_t max_seqlen, int32_t hq,
                                   int32_t hkv, int32_t d) {
  AttnArgs a = make_args(nullptr, nullptr, nullptr, nullptr, num_segments, num_tokens, max_seqlen, hq, hkv, d, 0.f);
  return attn_fwd_ws_bytes(a);
}

vcs_status vcs_attn_fwd(const void* q, const void* k, const void* v, const int32_t* cu_seqlens, int32_t num_segments,
                        int64_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv, int32_t d,
                        float softmax_scale, void* o, float* lse, void* ws, size_t ws_bytes, void* stream) {
  vcs::ApiRange nvtx_range("vcs_attn_fwd");
  AttnArgs a = make_args(q, k, v, cu_seqlens, num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale);
  vcs_status s = check_attn(a);
  if (s != VCS_OK) return s;
  if (o == nullptr || lse == nullptr || !aligned16(o) || !aligned16(lse)) return VCS_ERR_INVALID_ARG;
  if (ws == nullptr || ws_bytes < attn_fwd_ws_bytes(a) || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return VCS_ERR_WORKSPACE;
  a.status = static_cast<int32_t*>(ws);
  cudaStream_t st = as_stream(stream);
  if (cudaMemsetAsync(ws, 0, kWsHeader, st) != cudaSuccess) return VCS_ERR_CUDA;
  if (num_tokens == 0 || num_segments == 0) return VCS_OK;
  if (launch_attn_fwd(a, o, lse, ws, st) != cudaSuccess) return VCS_ERR_CUDA;
  return VCS_OK;
}

size_t vcs_attn_bwd_workspace_size(int32_t num_segments, int64_t num_tokens, int32_t max_seqlen, int32_t hq,
                                   int32_t hkv, int32_t d) {
  AttnArgs a = make_args(nullptr, nullptr, nullptr, nullptr, num_segments, num_tokens, max_seqlen, hq, hkv, d, 0.f);
  return attn_bwd_ws_bytes(a);
}

vcs_status vcs_stream_fields(const int32_t* traj_ids, const float* traj_logp, int64_t traj_tokens,
                             const int32_t* tok_gather, const uint8_t* tok_loss_mask, int64_t num_tokens,
                             int32_t* ids, float* logp, int32_t* dev_status, void* stream) {
  vcs::ApiRange nvtx_range("vcs_stream_fields");
  if (traj_tokens < 0 || num_tokens < 0) return VCS_ERR_INVALID_ARG;
  if (traj_tokens > INT32_MAX || num_tokens > INT32_MAX) return VCS_ERR_OVERFLOW;
  if (num_tokens > 0 && (traj_ids == nullptr || traj_logp == nullptr || tok_gather == nullptr ||
                         tok_loss_mask == nullptr || ids == nullptr || logp == nullptr))
    return VCS_ERR_INVALID_ARG;
  if (launch_stream_fields(traj_ids, traj_logp, traj_tokens, tok_gather, tok_loss_mask, num_tokens, ids, logp,
                           dev_status, as_stream(stream)) != cudaSuccess)
    return VCS_ERR_CUDA;
  return VCS_OK;
}

size_t vcs_compact_workspace_size(int64_t num_tokens) { return compact_ws_bytes(num_tokens < 0 ? 0 : num_tokens); }

vcs_status vcs_compact_trainable(const uint8_t* tok_loss_mask, int64_t num_tokens, int32_t* idx, int64_t idx_capacity,
                                 int64_t* count, void* ws, size_t ws_bytes, void* stream) {
  vcs::ApiRange nvtx_range("vcs_compact_trainable");
  if (num_tokens < 0 || idx_capacity < 0 || count == nullptr) return VCS_ERR_INVALID_ARG;
  if (num_tokens > INT32_MAX) return VCS_ERR_OVERFLOW;
  if (num_tokens > 0 && tok_loss_mask == nullptr) return VCS_ERR_INVALID_ARG;
  if (idx_capacity > 0 && idx == nullptr) return VCS_ERR_INVALID_ARG;
  if (ws == nullptr || ws_bytes < compact_ws_bytes(num_tokens) || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return VCS_ERR_WORKSPACE;
  if (launch_compact(tok_loss_mask, num_tokens, idx, idx_capacity, count, ws, as_stream(stream)) != cudaSuccess)
    return VCS_ERR_CUDA;
  return VCS_OK;
}

size_t vcs_grpo_loss_workspace_size(int64_t num_tokens) {
  return grpo_loss_ws_bytes(num_tokens < 0 ? 0 : num_tokens);
}

vcs_status vcs_grpo_loss(const float* logp, const float* old_logp, const float* ref_logp,
                         const uint8_t* tok_loss_mask, const int32_t* cu_seqlens, const int32_t* seg_traj,
                         int64_t num_segments, int64_t num_tokens, const float* adv, int64_t num_traj, float eps_low,
                         float eps_high, float clip_cap, float kl_coef, double* loss, float* dlogp, void* ws,
                         size_t ws_bytes, void* stream) {
  vcs::ApiRange nvtx_range("vcs_grpo_loss");
  if (num_segments < 0 || num_tokens < 0 || num_traj <= 0 || loss == nullptr) return VCS_ERR_INVALID_ARG;
  if (num_tokens > INT32_MAX || num_segments > INT32_MAX || num_traj > INT32_MAX) return VCS_ERR_OVERFLOW;
  if (!(eps_low >= 0.f && eps_low < 1.f) || !(eps_high >= 0.f) || !(clip_cap > 1.f + eps_high) ||
      !(kl_coef >= 0.f))
    return VCS_ERR_INVALID_ARG;
  if (num_tokens > 0 && (logp == nullptr || old_logp == nullptr || ref_logp == nullptr || tok_loss_mask == nullptr ||
                         cu_seqlens == nullptr || seg_traj == nullptr || adv == nullptr || num_segments == 0))
    return VCS_ERR_INVALID_ARG;
  if (ws == nullptr || ws_bytes < grpo_loss_ws_bytes(num_tokens) || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return VCS_ERR_WORKSPACE;
  // branch thresholds rounded once from double, as a float32 reading of 1 - eps_l, 1 + eps_h
  const float lo = (float)(1.0 - (double)eps_low), hi = (float)(1.0 + (double)eps_high);
  if (launch_grpo_loss(logp, old_logp, ref_logp, tok_loss_mask, cu_seqlens, seg_traj, (int32_t)num_segments,
                       (int32_t)num_tokens, adv, (int32_t)num_traj, lo, hi, clip_cap, kl_coef, loss, dlogp, ws,
                       as_stream(stream)) != cudaSuccess)
    return VCS_ERR_CUDA;
  return VCS_OK;
}

vcs_status vcs_group_advantage(const float* rewards, int64_t num_groups, int32_t group_size, float eps, float* adv,
                               void* stream) {
  vcs::ApiRange nvtx_range("vcs_group_advantage");
  if (num_groups < 0 || group_size <= 0 || !(eps >= 0.f)) return VCS_ERR_INVALID_ARG;
  if (num_groups > 0 && (rewards == nullptr || adv == nullptr)) return VCS_ERR_INVALID_ARG;
  if (launch_group_advantage(rewards, num_groups, group_size, eps, adv, as_stream(stream)) != cudaSuccess)
    return VCS_ERR_CUDA;
  return VCS_OK;
}

vcs_status vcs_attn_bwd(const void* q, const void* k, const void* v, const void* o, const float* lse,
                        const void* dout, const int32_t* cu_seqlens, int32_t num_segments, int64_t num_tokens,
                        int32_t max_seqlen, int32_t hq, int32_t hkv, int32_t d, float softmax_scale, void* dq,
                        void* dk, void* dv, void* ws, size_t ws_bytes, void* stream) {
  vcs::ApiRange nvtx_range("vcs_attn_bwd");
  AttnArgs a = make_args(q, k, v, cu_seqlens, num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale);
  vcs_status s = check_attn(a);
  if (s != VCS_OK) return s;
  const void* outs[6] = {o, lse, dout, dq, dk, dv};
  for (const void* p : outs)
    if (p == nullptr || !aligned16(p)) return VCS_ERR_INVALID_ARG;
  if (ws == nullptr || ws_bytes < attn_bwd_ws_bytes(a) || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return VCS_ERR_WORKSPACE;
  a.status = static_cast<int32_t*>(ws);
  cudaStream_t st = as_stream(stream);
  if (cudaMemsetAsync(ws, 0, kWsHeader, st) != cudaSuccess) return VCS_ERR_CUDA;
  if (num_tokens == 0 || num_segments == 0) return VCS_OK;
  if (launch_attn_bwd(a, o, lse, dout, dq, dk, dv, ws, st) != cudaSuccess) return VCS_ERR_CUDA;
  return VCS_OK;
}

// ---------------------------------------------------------------- prefix reuse
vcs_status vcs_shared_prefix(const int32_t* cu_seqlens, const int32_t* seg_traj, const int32_t* tok_gather,
                             int32_t num_segments, int64_t num_tokens, int32_t* seg_shared, int32_t* dev_status,
                             void* stream) {
  vcs::ApiRange nvtx_range("vcs_shared_prefix");
  if (num_segments < 0 || num_tokens < 0) return VCS_ERR_INVALID_ARG;
  if (num_tokens > INT32_MAX) return VCS_ERR_OVERFLOW;
  if (num_segments > 0 && (cu_seqlens == nullptr || seg_traj == nullptr || seg_shared == nullptr ||
                           (num_tokens > 0 && tok_gather == nullptr)))
    return VCS_ERR_INVALID_ARG;
  if (launch_shared_prefix(cu_seqlens, seg_traj, tok_gather, num_segments, (int32_t)num_tokens, seg_shared,
                           dev_status, as_stream(stream)) != cudaSuccess)
    return VCS_ERR_CUDA;
  return VCS_OK;
}

vcs_status vcs_attn_fwd_reuse(const void* q, const void* k, const void* v, const int32_t* cu_seqlens,
                              const int32_t* seg_shared, int32_t num_segments, int64_t num_tokens, int32_t max_seqlen,
                              int32_t hq, int32_t hkv, int32_t d, float softmax_scale, void* o, float* lse, void* ws,
                              size_t ws_bytes, void* stream) {
  vcs::ApiRange nvtx_range("vcs_attn_fwd_reuse");
  AttnArgs a = make_args(q, k, v, cu_seqlens, num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale);
  vcs_status s = check_attn(a);
  if (s != VCS_OK) return s;
  if (num_segments > 0 && seg_shared == nullptr) return VCS_ERR_INVALID_ARG;
  a.seg_shared = seg_shared;
  if ((num_tokens > 0 && (o == nullptr || lse == nullptr)) || !aligned16(o) || !aligned16(lse))
    return VCS_ERR_INVALID_ARG;
  if (ws == nullptr || ws_bytes < attn_fwd_ws_bytes(a) || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return VCS_ERR_WORKSPACE;
  a.status = static_cast<int32_t*>(ws);
  cudaStream_t st = as_stream(stream);
  if (cudaMemsetAsync(ws, 0, kWsHeader, st) != cudaSuccess) return VCS_ERR_CUDA;
  if (num_tokens == 0 || num_segments == 0) return VCS_OK;
  if (launch_attn_fwd(a, o, lse, ws, st) != cudaSuccess) return VCS_ERR_CUDA;
  return VCS_OK;
}

// ---------------------------------------------------------------- gathered attention
// The attention forward/backward reading Q, K, V straight from trajectory-layout tensors
// through the builder's gather map (no materialised segment-layout copies); the backward
// returns dQ, dK, dV in trajectory layout, the contributions of a token's copies summed.
static vcs_status check_gathered(const AttnArgs& a, int64_t traj_tokens, const int32_t* tok_gather) {
  vcs_status s = check_attn(a);
  if (s != VCS_OK) return s;
  if (traj_tokens < 0) return VCS_ERR_INVALID_ARG;
  if (traj_tokens > INT32_MAX) return VCS_ERR_OVERFLOW;
  if (a.num_tokens > 0 && (traj_tokens == 0 || tok_gather == nullptr)) return VCS_ERR_INVALID_ARG;
  return VCS_OK;
}

vcs_status vcs_attn_fwd_gathered(const void* q_traj, const void* k_traj, const void* v_traj, int64_t traj_tokens,
                                 const int32_t* tok_gather, const int32_t* cu_seqlens, int32_t num_segments,
                                 int64_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv, int32_t d,
                                 float softmax_scale, void* o, float* lse, void* ws, size_t ws_bytes, void* stream) {
  vcs::ApiRange nvtx_range("vcs_attn_fwd_gathered");
  AttnArgs a =
      make_args(q_traj, k_traj, v_traj, cu_seqlens, num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale);
  vcs_status s = check_gathered(a, traj_tokens, tok_gather);
  if (s != VCS_OK) return s;
  a.tok_gather = tok_gather;
  a.traj_tokens = traj_tokens;
  if ((num_tokens > 0 && (o == nullptr || lse == nullptr)) || !aligned16(o) || !aligned16(lse))
    return VCS_ERR_INVALID_ARG;  // o, lse may be NULL when there are no segment tokens
  if (ws == nullptr || ws_bytes < attn_fwd_ws_bytes(a) || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return VCS_ERR_WORKSPACE;
  a.status = static_cast<int32_t*>(ws);
  cudaStream_t st = as_stream(stream);
  if (cudaMemsetAsync(ws, 0, kWsHeader, st) != cudaSuccess) return VCS_ERR_CUDA;
  if (num_tokens == 0 || num_segments == 0) return VCS_OK;
  if (launch_attn_fwd(a, o, lse, ws, st) != cudaSuccess) return VCS_ERR_CUDA;
  return VCS_OK;
}

size_t vcs_attn_bwd_gathered_workspace_size(int32_t num_segments, int64_t num_tokens, int32_t max_seqlen,
                                            int64_t traj_tokens, int32_t hq, int32_t hkv, int32_t d) {
  AttnArgs a = make_args(nullptr, nullptr, nullptr, nullptr, num_segments, num_tokens, max_seqlen, hq, hkv, d, 0.f);
  a.traj_tokens = traj_tokens;
  return attn_bwd_ws_bytes(a);
}

vcs_status vcs_attn_bwd_gathered(const void* q_traj, const void* k_traj, const void* v_traj, int64_t traj_tokens,
                                 const int32_t* tok_gather, const void* o, const float* lse, const void* dout,
                                 const int32_t* cu_seqlens, int32_t num_segments, int64_t num_tokens,
                                 int32_t max_seqlen, int32_t hq, int32_t hkv, int32_t d, float softmax_scale,
                                 void* dq_traj, void* dk_traj, void* dv_traj, void* ws, size_t ws_bytes,
                                 void* stream) {
  vcs::ApiRange nvtx_range("vcs_attn_bwd_gathered");
  AttnArgs a =
      make_args(q_traj, k_traj, v_traj, cu_seqlens, num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale);
  vcs_status s = check_gathered(a, traj_tokens, tok_gather);
  if (s != VCS_OK) return s;
  a.tok_gather = tok_gather;
  a.traj_tokens = traj_tokens;
  const void* seg_ptrs[3] = {o, lse, dout};            // may be NULL when there are no segment tokens
  const void* traj_ptrs[3] = {dq_traj, dk_traj, dv_traj};
  for (const void* p : seg_ptrs)
    if ((num_tokens > 0 && p == nullptr) || !aligned16(p)) return VCS_ERR_INVALID_ARG;
  for (const void* p : traj_ptrs)
    if ((traj_tokens > 0 && p == nullptr) || !aligned16(p)) return VCS_ERR_INVALID_ARG;
  if (ws == nullptr || ws_bytes < attn_bwd_ws_bytes(a) || (reinterpret_cast<uintptr_t>(ws) & 255u) != 0)
    return VCS_ERR_WORKSPACE;
  a.status = static_cast<int32_t*>(ws);
  cudaStream_t st = as_stream(stream);
  if (cudaMemsetAsync(ws, 0, kWsHeader, st) != cudaSuccess) return VCS_ERR_CUDA;
  if (num_tokens == 0 || num_segments == 0) {  // no segment token reads the trajectory: zero gradients
    const size_t qb = (size_t)traj_tokens * hq * d * 2, kb = (size_t)traj_tokens * hkv * d * 2;
    if (traj_tokens > 0 && (cudaMemsetAsync(dq_traj, 0, qb, st) != cudaSuccess ||
                            cudaMemsetAsync(dk_traj, 0, kb, st) != cudaSuccess ||
                            cudaMemsetAsync(dv_traj, 0, kb, st) != cudaSuccess))
      return VCS_ERR_CUDA;
    return VCS_OK;
  }
  if (launch_attn_bwd(a, o, lse, dout, dq_traj, dk_traj, dv_traj, ws, st) != cudaSuccess) return VCS_ERR_CUDA;
  return VCS_OK;
}

}  // extern "C"
