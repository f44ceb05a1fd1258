/*
 * vcs.h - C ABI of libvcs.so, the GB300 (sm_103a) hot path of Visual Context
 * Segmentation (arXiv 2607.11185, Sec. 3.4, Algorithm 1, App. C.1).
 *
 * A GUI trajectory of T steps (screenshot tokens followed by response tokens
 * per step) is cut into training segments that keep a sliding window of the
 * most recent screenshots as image tokens and carry the earlier steps as text
 * (Algorithm 1).  The library builds the packed segment layout, gathers the
 * bf16 Q/K/V rows of every segment token from trajectory-layout tensors, and
 * runs causal (per-segment) grouped-query softmax attention forward and
 * backward over the packed segments.
 *
 * Conventions shared by every call:
 *   - Plain C, no allocation, no global state: every buffer is owned by the
 *     caller.  Device pointers must point to memory of the current CUDA
 *     device.  Tensors are contiguous, row-major, 16-byte aligned.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default).
 *     Every call is asynchronous on that stream.
 *   - The return value is a vcs_status.  Argument errors that the host can
 *     see are returned before anything is launched.  Errors that only the
 *     device can see (inconsistent offsets, out-of-range indices, too-small
 *     capacities, a bounded wait that gave up) are written as a non-zero
 *     vcs_status into a device-visible int32 status word named by each call;
 *     the offending work is skipped, never trapped.  The caller reads that
 *     word after synchronising.
 *   - Counts of tokens, steps and segments are limited to INT32_MAX.
 *
 * Step model (the readings of the paper that the layout follows):
 *   step t of a trajectory contributes step_img[t] screenshot tokens followed
 *   by step_txt[t] response tokens; the trajectory token buffer is the
 *   concatenation of the steps, trajectories are concatenated in order.  A
 *   segment holds at most keep + window screenshots (Algorithm 1's prune
 *   trigger n_img > K + delta, with K = keep and delta = window).  The first
 *   segment takes steps 1..min(keep+window, T); each later one takes the next
 *   `window` steps as new steps and retains the `keep` steps before them with
 *   their screenshots.  Earlier steps appear as their response tokens only.
 *   Only the response tokens of a segment's new steps are trainable (each
 *   response is optimised exactly once, App. C.1).  keep = 0 gives a window
 *   of the `window` most recent screenshots; keep = 0, window = 1 gives
 *   step-wise decomposition (Sec. 1); keep + window >= T gives one segment
 *   per trajectory.
 */
#ifndef VCS_H_
#define VCS_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum vcs_status {
  VCS_OK = 0,
  VCS_ERR_INVALID_ARG = 1,     /* null pointer, negative count, misaligned pointer, bad window */
  VCS_ERR_UNSUPPORTED = 2,     /* head_dim not 64/128, hq not a multiple of hkv, ... */
  VCS_ERR_CAPACITY = 3,        /* an output buffer is smaller than the layout needs */
  VCS_ERR_OVERFLOW = 4,        /* a token count does not fit int32 */
  VCS_ERR_CUDA = 5,            /* a CUDA runtime or driver call failed */
  VCS_ERR_DEVICE_CHECK = 6,    /* a kernel found inconsistent input data */
  VCS_ERR_DEVICE_TIMEOUT = 7,  /* a bounded device-side wait gave up */
  VCS_ERR_WORKSPACE = 8        /* workspace pointer NULL or smaller than the size query */
} vcs_status;

/* Sizes of a segment layout, written by the device.  Must live in device
 * memory or in pinned (mapped) host memory. */
typedef struct vcs_sizes {
  int64_t num_segments;
  int64_t num_tokens;
  int32_t max_seqlen;
  int32_t status;              /* vcs_status of device-side checks, 0 = OK */
} vcs_sizes;

/* Human-readable name of a status code (static storage, never NULL). */
const char* vcs_status_string(int32_t status);

/* Library version / build string (static storage). */
const char* vcs_version(void);

/* ------------------------------------------------------------------------ *
 * Segment builder (Sec. 3.4, Algorithm 1; App. C.1)
 * ------------------------------------------------------------------------ */

/* Workspace bytes for vcs_plan_segments / vcs_build_segments. */
size_t vcs_segments_workspace_size(int32_t num_traj, int64_t num_steps);

/* Phase 1: sizes of the segment layout.
 *   cu_steps  [num_traj+1] int32 device: step range of each trajectory
 *             (cu_steps[0] = 0, non-decreasing, cu_steps[num_traj] = num_steps)
 *   step_img  [num_steps] int32 device: screenshot tokens of each step (>= 0)
 *   step_txt  [num_steps] int32 device: response tokens of each step (>= 0)
 *   window    delta of Algorithm 1 (>= 1): new screenshots per segment
 *   keep      K of Algorithm 1 (>= 0): screenshots retained across a prune
 *   sizes     device-visible output: segment count, segment-token count,
 *             longest segment, device status (VCS_ERR_DEVICE_CHECK for
 *             inconsistent cu_steps or negative counts, VCS_ERR_OVERFLOW when
 *             a token count exceeds INT32_MAX)
 *   ws        device workspace of vcs_segments_workspace_size() bytes
 * Asynchronous: synchronise `stream` before reading *sizes. */
vcs_status vcs_plan_segments(const int32_t* cu_steps, int32_t num_traj, int64_t num_steps,
                             const int32_t* step_img, const int32_t* step_txt,
                             int32_t window, int32_t keep, vcs_sizes* sizes,
                             void* ws, size_t ws_bytes, void* stream);

/* Phase 2: the token-level layout (same inputs as phase 1).
 *   cu_seqlens    [num_segments+1] int32: segment boundaries in the packed buffer
 *   seg_traj      [num_segments] int32 or NULL: trajectory of each segment
 *   tok_gather    [num_tokens] int32: index into the trajectory token buffer
 *   tok_src_step  [num_tokens] int32: global step index (into step_img/step_txt)
 *   tok_pos       [num_tokens] int32: position in the segment, 0..L-1
 *   tok_loss_mask [num_tokens] uint8 or NULL: 1 on trainable response tokens
 *   seg_capacity / tok_capacity: element capacities of the segment / token
 *   arrays.  If the layout needs more, nothing is written past the capacity
 *   and sizes->status becomes VCS_ERR_CAPACITY.  sizes receives the same
 *   values as in phase 1. */
vcs_status vcs_build_segments(const int32_t* cu_steps, int32_t num_traj, int64_t num_steps,
                              const int32_t* step_img, const int32_t* step_txt,
                              int32_t window, int32_t keep,
                              int64_t seg_capacity, int64_t tok_capacity,
                              int32_t* cu_seqlens, int32_t* seg_traj, int32_t* tok_gather,
                              int32_t* tok_src_step, int32_t* tok_pos, uint8_t* tok_loss_mask,
                              vcs_sizes* sizes, void* ws, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------ *
 * Gather: packed segment rows from trajectory rows (the re-tokenised fresh
 * stream of Algorithm 1 re-uses trajectory tokens).
 *   q_traj [traj_tokens, hq, d], k_traj / v_traj [traj_tokens, hkv, d] bf16 device
 *   tok_gather [num_tokens] int32 device (from vcs_build_segments)
 *   q [num_tokens, hq, d], k / v [num_tokens, hkv, d] bf16 device outputs
 *   dev_status  int32 device word or NULL: set to VCS_ERR_DEVICE_CHECK if a
 *               gather index is outside [0, traj_tokens) (that row is skipped)
 * k_traj/v_traj/k/v may all be NULL to gather Q only.  Bit-exact copy.
 * ------------------------------------------------------------------------ */
vcs_status vcs_gather(const void* q_traj, const void* k_traj, const void* v_traj, int64_t traj_tokens,
                      const int32_t* tok_gather, int64_t num_tokens, int32_t hq, int32_t hkv, int32_t d,
                      void* q, void* k, void* v, int32_t* dev_status, void* stream);

/* ------------------------------------------------------------------------ *
 * Attention over packed segments.  Token i of segment s attends to the
 * tokens j of the same segment with j <= i (causal), query head h uses
 * key/value head h / (hq / hkv).  softmax_scale <= 0 selects 1/sqrt(d).
 * Layouts: q, o, dout, dq [num_tokens, hq, d]; k, v, dk, dv
 * [num_tokens, hkv, d]; all bf16.  lse [hq, num_tokens] fp32, natural log.
 * cu_seqlens [num_segments+1] int32 device, non-decreasing from 0 to
 * num_tokens, every segment at most max_seqlen long.  Supported: d in
 * {64, 128}, hq % hkv == 0, num_tokens < 2^31.  The workspace starts with a
 * 256-byte header whose first int32 is the device status word
 * (VCS_ERR_DEVICE_CHECK for inconsistent cu_seqlens, VCS_ERR_DEVICE_TIMEOUT
 * for a wait that gave up); every call clears it first.
 * ------------------------------------------------------------------------ */

/* Forward workspace: the header, then the list of the launch's work units (one
 * per segment, query head and pair of 128-row query tiles, 16 bytes each, at
 * most hq * (num_tokens / 256 + num_segments + 1) of them) and their
 * per-segment offsets, built on the device by the call itself; about
 * hq * num_tokens / 16 bytes.  Also the size for vcs_attn_fwd_reuse and
 * vcs_attn_fwd_gathered.  Inconsistent cu_seqlens can describe overlapping
 * segments with more units than that: then no unit runs (nothing is written
 * past the list) and the status word reports VCS_ERR_DEVICE_CHECK. */
size_t vcs_attn_fwd_workspace_size(int32_t num_segments, int64_t num_tokens, int32_t max_seqlen,
                                   int32_t hq, int32_t hkv, int32_t d);

/* Forward: o = softmax(scale q k^T, causal within the segment) v, and lse. */
vcs_status vcs_attn_fwd(const void* q, const void* k, const void* v, const int32_t* cu_seqlens,
                        int32_t num_segments, int64_t num_tokens, int32_t max_seqlen,
                        int32_t hq, int32_t hkv, int32_t d, float softmax_scale,
                        void* o, float* lse, void* ws, size_t ws_bytes, void* stream);

size_t vcs_attn_bwd_workspace_size(int32_t num_segments, int64_t num_tokens, int32_t max_seqlen,
                                   int32_t hq, int32_t hkv, int32_t d);

/* Backward: dq, dk, dv of sum(o * dout), given q, k, v, the forward's o and lse.
 * dk / dv sum over the hq / hkv query heads that share a key/value head.
 * The workspace also holds an fp32 dq accumulator and the row terms
 * D = rowsum(dout * o). */
vcs_status vcs_attn_bwd(const void* q, const void* k, const void* v, const void* o, const float* lse,
                        const void* dout, const int32_t* cu_seqlens, int32_t num_segments,
                        int64_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv, int32_t d,
                        float softmax_scale, void* dq, void* dk, void* dv,
                        void* ws, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------ *
 * Backward for callers that cannot allocate device memory.
 *
 * The paper has no counterpart to this call; it exists for users of this
 * library.  vcs_attn_bwd needs a workspace from the caller.  Some callers
 * cannot allocate one: a plugin whose host framework owns all device memory
 * and passes it only the input and output tensors, or a latency-critical
 * loop that must not call cudaMalloc (it can synchronise the device, and it
 * can fail when memory is nearly full).  This variant computes exactly what
 * vcs_attn_bwd computes (same arguments, layouts and errors, minus the
 * workspace) but takes its workspace from a fixed array of
 * VCS_NOALLOC_SCRATCH_BYTES compiled into the library, which every GPU that
 * loads the library holds until the process exits.  Neither the caller nor
 * the library allocates anything; the caller still passes all inputs and
 * outputs.
 *
 *   dev_status  int32 device word or NULL: receives the device status word
 *               (as the first int32 of vcs_attn_bwd's workspace would)
 * Returns VCS_ERR_WORKSPACE, before any launch, when the problem needs more
 * than VCS_NOALLOC_SCRATCH_BYTES (vcs_attn_bwd_workspace_size() tells the
 * need: 256 + 4*hq*num_tokens + 4*num_tokens*hq*d bytes, each term rounded up
 * to 256; e.g. hq = 28, d = 128 allows about 2,300 tokens).
 * The first call on each device performs a one-time set-up (it looks up the
 * array's device address); make that first call before any stream capture.
 * Every call on a device shares the one array, which keeps the last call's
 * contents (each call clears what must start at zero): calls that can overlap
 * on the GPU (different streams without ordering between them) race on it and
 * must not be issued.
 * ------------------------------------------------------------------------ */
#define VCS_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)

vcs_status vcs_attn_bwd_noalloc(const void* q, const void* k, const void* v, const void* o, const float* lse,
                                const void* dout, const int32_t* cu_seqlens, int32_t num_segments,
                                int64_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv, int32_t d,
                                float softmax_scale, void* dq, void* dk, void* dv, int32_t* dev_status,
                                void* stream);

/* ------------------------------------------------------------------------
 * Gathered attention: the forward and backward above, with Q, K and V read
 * straight from the trajectory-layout tensors through the builder's gather
 * map instead of from vcs_gather's segment-layout copies.  A segment holds
 * copies of trajectory tokens (the text history re-tokenised into each fresh
 * stream, Alg. 1, App. C.1; the screenshots kept across segments), so segment
 * token n is trajectory token tok_gather[n]; the paper names no kernel for
 * this, and these calls only fuse the copy into the attention's tile loads.
 *
 *   q_traj      bf16 [traj_tokens, hq, d] device, row-major
 *   k_traj, v_traj  bf16 [traj_tokens, hkv, d] device
 *   traj_tokens number of trajectory tokens (rows of the three tensors)
 *   tok_gather  int32 [num_tokens] device, from vcs_build_segments; every
 *               entry in [0, traj_tokens) (an entry outside is recorded as
 *               VCS_ERR_DEVICE_CHECK in the workspace status word and read as
 *               row 0)
 *   cu_seqlens .. lse / dout   as for vcs_attn_fwd / vcs_attn_bwd (segment
 *               layout: o, lse and dout have num_tokens rows; NULL allowed
 *               when num_tokens is 0)
 *   dq_traj     bf16 [traj_tokens, hq, d] device (written): the sum over the
 *               segment copies n of trajectory token t (tok_gather[n] = t) of
 *               dQ of copy n; dk_traj, dv_traj bf16 [traj_tokens, hkv, d]
 *               likewise (tokens no segment reads get 0)
 * The forward's o and lse equal vcs_attn_fwd's on vcs_gather's copies bit
 * for bit.  The backward accumulates in fp32 (atomic adds, so the order of
 * the additions and the last bits of dq, dk, dv vary from run to run) and
 * needs the workspace vcs_attn_bwd_gathered_workspace_size() gives:
 * vcs_attn_bwd's plus 4*traj_tokens*(hq + 2*hkv)*d bytes, each term rounded
 * up to 256.  Errors as for vcs_attn_fwd / vcs_attn_bwd, plus
 * VCS_ERR_INVALID_ARG for num_tokens > 0 with traj_tokens = 0 or a NULL
 * tok_gather and VCS_ERR_OVERFLOW for traj_tokens above INT32_MAX.
 * ------------------------------------------------------------------------ */
vcs_status vcs_attn_fwd_gathered(const void* q_traj, const void* k_traj, const void* v_traj, int64_t traj_tokens,
                                 const int32_t* tok_gather, const int32_t* cu_seqlens, int32_t num_segments,
                                 int64_t num_tokens, int32_t max_seqlen, int32_t hq, int32_t hkv, int32_t d,
                                 float softmax_scale, void* o, float* lse, void* ws, size_t ws_bytes,
                                 void* stream);

size_t vcs_attn_bwd_gathered_workspace_size(int32_t num_segments, int64_t num_tokens, int32_t max_seqlen,
                                            int64_t traj_tokens, int32_t hq, int32_t hkv, int32_t d);

vcs_status vcs_attn_bwd_gathered(const void* q_traj, const void* k_traj, const void* v_traj, int64_t traj_tokens,
                                 const int32_t* tok_gather, const void* o, const float* lse, const void* dout,
                                 const int32_t* cu_seqlens, int32_t num_segments, int64_t num_tokens,
                                 int32_t max_seqlen, int32_t hq, int32_t hkv, int32_t d, float softmax_scale,
                                 void* dq_traj, void* dk_traj, void* dv_traj, void* ws, size_t ws_bytes,
                                 void* stream);

/* ------------------------------------------------------------------------
 * Prefix reuse (forward).  A fresh stream re-tokenises the text of the steps
 * before its window (Alg. 1, Sec. 3.4 / App. C.1) and the steps that leave the
 * window join that text, so a trajectory's segment s starts with the tokens
 * its segment s-1 starts with.  Causal attention row r depends only on tokens
 * 0..r of its segment (positions restart at 0 in every stream), so over the
 * common prefix the two segments' rows are equal.  The paper does not use
 * this; it only removes repeated forward work.
 *
 * vcs_shared_prefix: seg_shared[s] = the largest n <= min(L_s, L_{s-1}) with
 * tok_gather[cu[s] + i] == tok_gather[cu[s-1] + i] for all i < n, and 0 when
 * seg_traj[s] != seg_traj[s-1] or s = 0.
 *   cu_seqlens, seg_traj, tok_gather  from vcs_build_segments (device)
 *   seg_shared  int32 [num_segments] device (written)
 *   dev_status  int32 device word or NULL: VCS_ERR_DEVICE_CHECK for
 *               inconsistent cu_seqlens (that segment gets 0)
 *
 * vcs_attn_fwd_reuse: vcs_attn_fwd's result (bit for bit) with seg_shared
 * from vcs_shared_prefix: the query-tile pairs (256 rows) of segment s that
 * lie wholly below seg_shared[s] are not computed; their o and lse rows are
 * copied from the segment that computed them (going back through the
 * trajectory's segments).  Arguments and errors as vcs_attn_fwd, plus
 * VCS_ERR_INVALID_ARG for a NULL seg_shared with segments present; a
 * seg_shared[s] larger than either segment, negative, or non-zero for s = 0
 * is recorded as VCS_ERR_DEVICE_CHECK in the workspace status word and read
 * as 0.  (A seg_shared larger than the true common prefix gives wrong rows,
 * not a fault: pass vcs_shared_prefix's.)
 * ------------------------------------------------------------------------ */
vcs_status vcs_shared_prefix(const int32_t* cu_seqlens, const int32_t* seg_traj, const int32_t* tok_gather,
                             int32_t num_segments, int64_t num_tokens, int32_t* seg_shared, int32_t* dev_status,
                             void* stream);

vcs_status vcs_attn_fwd_reuse(const void* q, const void* k, const void* v, const int32_t* cu_seqlens,
                              const int32_t* seg_shared, int32_t num_segments, int64_t num_tokens, int32_t max_seqlen,
                              int32_t hq, int32_t hkv, int32_t d, float softmax_scale, void* o, float* lse, void* ws,
                              size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Token-ID stream fields (App. C.1, Algorithm 1's (ids, mask, logp) stream).
 * Response tokens enter a segment's stream as trainable tokens with their
 * rollout log-probabilities; observation tokens and the re-tokenised history
 * of a fresh stream enter with mask 0 and log-probability 0.  Over the
 * segment layout, for segment token n:
 *   ids[n]  = traj_ids[tok_gather[n]]
 *   logp[n] = tok_loss_mask[n] ? traj_logp[tok_gather[n]] : 0
 *   traj_ids   int32 [traj_tokens] device: the trajectories' token IDs
 *   traj_logp  fp32 [traj_tokens] device: rollout log-probabilities of the
 *              trajectories' tokens (read only for response tokens)
 *   tok_gather, tok_loss_mask  from vcs_build_segments
 *   ids, logp  int32 / fp32 [num_tokens] device (written)
 *   dev_status int32 device word or NULL: VCS_ERR_DEVICE_CHECK when a gather
 *              index is outside [0, traj_tokens) (that token gets 0, 0)
 * Returns VCS_ERR_INVALID_ARG for a negative count or a null pointer,
 * VCS_ERR_OVERFLOW for counts above INT32_MAX.
 * ------------------------------------------------------------------------ */
vcs_status vcs_stream_fields(const int32_t* traj_ids, const float* traj_logp, int64_t traj_tokens,
                             const int32_t* tok_gather, const uint8_t* tok_loss_mask, int64_t num_tokens,
                             int32_t* ids, float* logp, int32_t* dev_status, void* stream);

/* vcs_compact_trainable: the indices n with tok_loss_mask[n] != 0, in
 * increasing order (each response token of the batch appears exactly once,
 * App. C.1).
 *   idx        int32 [idx_capacity] device (written: the first min(count,
 *              idx_capacity) entries)
 *   count      int64 device, 1 value (written): the number of trainable tokens
 *   ws         device workspace of vcs_compact_workspace_size(num_tokens) bytes,
 *              256-byte aligned; its first int32 is the device status word
 *              (VCS_ERR_CAPACITY when count > idx_capacity)
 * Returns VCS_ERR_INVALID_ARG for negative counts or null pointers,
 * VCS_ERR_WORKSPACE for a small or misaligned workspace. */
size_t vcs_compact_workspace_size(int64_t num_tokens);

vcs_status vcs_compact_trainable(const uint8_t* tok_loss_mask, int64_t num_tokens, int32_t* idx, int64_t idx_capacity,
                                 int64_t* count, void* ws, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * RL objective over the segments (App. C.2, Eq. "RL objective" and the
 * hyperparameter table: DAPO asymmetric clipping eps_l = 0.2, eps_h = 0.28,
 * clip-ratio cap c = 3.0, KL weight lambda = 1e-4, group-relative advantage
 * shared by every segment of a rollout, loss masks so that each response is
 * optimised exactly once).  Readings where the paper gives no formula:
 *   - the cap is dual clipping: a token with A < 0 contributes
 *     max(min(rho A, clip(rho, 1-eps_l, 1+eps_h) A), c A);
 *   - the KL term is the per-token estimate exp(r) - r - 1, r = ref_logp - logp,
 *     over the same trainable tokens;
 *   - the expectations over tasks and rollouts are a mean over trajectories:
 *       loss = (1/num_traj) sum_t mask_t (-o_t + kl_coef k_t).
 *
 * vcs_grpo_loss: forward and backward in one pass.
 *   logp, old_logp, ref_logp  fp32 [num_tokens] device, segment layout: the
 *               token log-probabilities under the policy being trained, the
 *               rollout policy and the reference policy
 *   tok_loss_mask u8 [num_tokens] device (vcs_build_segments' loss mask)
 *   cu_seqlens, seg_traj  the layout from vcs_build_segments
 *   adv         fp32 [num_traj] device: advantage of each trajectory
 *   loss        fp64 device, 1 value (written)
 *   dlogp       fp32 [num_tokens] device or NULL: d loss / d logp (written;
 *               zero for masked tokens)
 *   ws          device workspace of vcs_grpo_loss_workspace_size(num_tokens)
 *               bytes, 256-byte aligned; its first int32 is the device status
 *               word (VCS_ERR_DEVICE_CHECK when a segment names a trajectory
 *               outside [0, num_traj); that token is skipped)
 * Per token the ratio rho = exp(logp - old_logp) and the branch are float32;
 * the sum is accumulated in double in a fixed order (deterministic).
 * Returns VCS_ERR_INVALID_ARG for negative counts, num_traj <= 0, a null
 * pointer, eps_low outside [0,1), eps_high < 0, clip_cap <= 1 + eps_high or
 * kl_coef < 0; VCS_ERR_WORKSPACE for a small or misaligned workspace.
 * ------------------------------------------------------------------------ */
size_t vcs_grpo_loss_workspace_size(int64_t num_tokens);

vcs_status vcs_grpo_loss(const float* logp, const float* old_logp, const float* ref_logp,
                         const uint8_t* tok_loss_mask, const int32_t* cu_seqlens, const int32_t* seg_traj,
                         int64_t num_segments, int64_t num_tokens, const float* adv, int64_t num_traj, float eps_low,
                         float eps_high, float clip_cap, float kl_coef, double* loss, float* dlogp, void* ws,
                         size_t ws_bytes, void* stream);

/* vcs_group_advantage: GRPO's group-relative advantage (App. C.2: computed
 * over the n rollouts of each task).  rewards fp32 [num_groups * group_size]
 * device, each group's rollouts consecutive; adv (same shape, written) =
 * (r - mean) / (std + eps) per group, population standard deviation, computed
 * in double.  Returns VCS_ERR_INVALID_ARG for num_groups < 0, group_size <= 0,
 * eps < 0 or a null pointer. */
vcs_status vcs_group_advantage(const float* rewards, int64_t num_groups, int32_t group_size, float eps, float* adv,
                               void* stream);

/* ------------------------------------------------------------------------ *
 * Self-test of the bounded device waits.
 *
 * The paper has no counterpart to this call.  Every pipeline wait inside the
 * attention kernels is bounded: a wait that runs out records
 * VCS_ERR_DEVICE_TIMEOUT in the call's status word and the kernel's roles
 * leave their loops.  This call checks the bounded-wait primitive itself, and
 * only that: one single-thread kernel waits on a barrier that nothing ever
 * arrives on for limit_cycles SM clock cycles and then writes
 * VCS_ERR_DEVICE_TIMEOUT into *dev_status.  How the attention kernels' roles
 * give up together (warpgroup barriers, TMEM release) is not exercised by it.
 *
 *   dev_status    int32 device word, 4-byte aligned, zeroed by the caller (a
 *                 nonzero word is left as it is)
 *   limit_cycles  1 .. 4,000,000,000 (the attention kernels' own limit, about
 *                 2 s at 2 GHz)
 * Returns VCS_ERR_INVALID_ARG for a null or misaligned dev_status or a limit
 * outside that range, before any launch.
 * ------------------------------------------------------------------------ */
vcs_status vcs_selftest_bounded_wait(int32_t* dev_status, int64_t limit_cycles, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* VCS_H_ */
