"""ctypes binding over libvcs.so (the C ABI in include/vcs.h).

The raw functions carry the C names and argument order and do argument
marshalling only (torch tensors -> device pointers, the current CUDA stream).
Every step of the path runs in the library's CUDA kernels; there is no CPU
or PyTorch fallback: importing this module raises if libvcs.so is missing.

Convenience wrappers (``build_segments``, ``gather``, ``attn_fwd``,
``attn_bwd``) allocate outputs with torch and raise ``VcsError`` on a
non-zero status.
"""
from __future__ import annotations

import ctypes
import math
import os
from typing import Optional

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libvcs.so")
if not os.path.exists(_LIB_PATH):
    raise ImportError(f"{_LIB_PATH} is not built; run `python -m paper_2607_11185_gb300.build` "
                      "(the CUDA path has no fallback)")
_lib = ctypes.CDLL(_LIB_PATH)

_p = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_sz = ctypes.c_size_t
_f32 = ctypes.c_float


class VcsSizes(ctypes.Structure):
    _fields_ = [("num_segments", ctypes.c_int64), ("num_tokens", ctypes.c_int64),
                ("max_seqlen", ctypes.c_int32), ("status", ctypes.c_int32)]


def _sig(name, res, args):
    f = getattr(_lib, name)
    f.restype = res
    f.argtypes = args
    return f


_lib_status_string = _sig("vcs_status_string", ctypes.c_char_p, [_i32])
_lib_version = _sig("vcs_version", ctypes.c_char_p, [])
_lib_seg_ws = _sig("vcs_segments_workspace_size", _sz, [_i32, _i64])
_lib_plan = _sig("vcs_plan_segments", _i32, [_p, _i32, _i64, _p, _p, _i32, _i32, _p, _p, _sz, _p])
_lib_build = _sig("vcs_build_segments", _i32,
                  [_p, _i32, _i64, _p, _p, _i32, _i32, _i64, _i64, _p, _p, _p, _p, _p, _p, _p, _p, _sz, _p])
_lib_gather = _sig("vcs_gather", _i32, [_p, _p, _p, _i64, _p, _i64, _i32, _i32, _i32, _p, _p, _p, _p, _p])
_lib_fwd_ws = _sig("vcs_attn_fwd_workspace_size", _sz, [_i32, _i64, _i32, _i32, _i32, _i32])
_lib_fwd = _sig("vcs_attn_fwd", _i32,
                [_p, _p, _p, _p, _i32, _i64, _i32, _i32, _i32, _i32, _f32, _p, _p, _p, _sz, _p])
_lib_bwd_ws = _sig("vcs_attn_bwd_workspace_size", _sz, [_i32, _i64, _i32, _i32, _i32, _i32])
_lib_bwd = _sig("vcs_attn_bwd", _i32,
                [_p, _p, _p, _p, _p, _p, _p, _i32, _i64, _i32, _i32, _i32, _i32, _f32, _p, _p, _p, _p, _sz, _p])

_lib_bwd_noalloc = _sig("vcs_attn_bwd_noalloc", _i32,
                        [_p, _p, _p, _p, _p, _p, _p, _i32, _i64, _i32, _i32, _i32, _i32, _f32, _p, _p, _p, _p, _p])
_lib_fwd_g = _sig("vcs_attn_fwd_gathered", _i32,
                  [_p, _p, _p, _i64, _p, _p, _i32, _i64, _i32, _i32, _i32, _i32, _f32, _p, _p, _p, _sz, _p])
_lib_shared = _sig("vcs_shared_prefix", _i32, [_p, _p, _p, _i32, _i64, _p, _p, _p])
_lib_fwd_reuse = _sig("vcs_attn_fwd_reuse", _i32,
                      [_p, _p, _p, _p, _p, _i32, _i64, _i32, _i32, _i32, _i32, _f32, _p, _p, _p, _sz, _p])
_lib_bwd_g_ws = _sig("vcs_attn_bwd_gathered_workspace_size", _sz, [_i32, _i64, _i32, _i64, _i32, _i32, _i32])
_lib_bwd_g = _sig("vcs_attn_bwd_gathered", _i32,
                  [_p, _p, _p, _i64, _p, _p, _p, _p, _p, _i32, _i64, _i32, _i32, _i32, _i32, _f32, _p, _p, _p, _p,
                   _sz, _p])

_f64 = ctypes.c_double
_lib_loss_ws = _sig("vcs_grpo_loss_workspace_size", _sz, [_i64])
_lib_loss = _sig("vcs_grpo_loss", _i32,
                 [_p, _p, _p, _p, _p, _p, _i64, _i64, _p, _i64, _f32, _f32, _f32, _f32, _p, _p, _p, _sz, _p])
_lib_adv = _sig("vcs_group_advantage", _i32, [_p, _i64, _i32, _f32, _p, _p])
_lib_fields = _sig("vcs_stream_fields", _i32, [_p, _p, _i64, _p, _p, _i64, _p, _p, _p, _p])
_lib_compact_ws = _sig("vcs_compact_workspace_size", _sz, [_i64])
_lib_compact = _sig("vcs_compact_trainable", _i32, [_p, _i64, _p, _i64, _p, _p, _sz, _p])
_lib_selftest_wait = _sig("vcs_selftest_bounded_wait", _i32, [_p, _i64, _p])

EXPORTED = ["vcs_status_string", "vcs_version", "vcs_segments_workspace_size", "vcs_plan_segments",
            "vcs_build_segments", "vcs_gather", "vcs_attn_fwd_workspace_size", "vcs_attn_fwd",
            "vcs_attn_bwd_workspace_size", "vcs_attn_bwd", "vcs_attn_bwd_noalloc", "vcs_grpo_loss_workspace_size",
            "vcs_grpo_loss", "vcs_group_advantage", "vcs_stream_fields", "vcs_compact_workspace_size",
            "vcs_compact_trainable", "vcs_attn_fwd_gathered", "vcs_attn_bwd_gathered_workspace_size",
            "vcs_attn_bwd_gathered", "vcs_shared_prefix", "vcs_attn_fwd_reuse", "vcs_selftest_bounded_wait"]

LIB_PATH = _LIB_PATH


class VcsError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {vcs_status_string(status)}")
        self.status = status


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, ctypes.Structure):
        return ctypes.addressof(t)
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


# ---------------------------------------------------------------- raw C calls

def vcs_status_string(status: int) -> str:
    return _lib_status_string(int(status)).decode()


def vcs_version() -> str:
    return _lib_version().decode()


def vcs_segments_workspace_size(num_traj: int, num_steps: int) -> int:
    return int(_lib_seg_ws(num_traj, num_steps))


def vcs_plan_segments(cu_steps, num_traj, num_steps, step_img, step_txt, window, keep, sizes, ws, ws_bytes,
                      stream=None) -> int:
    return _lib_plan(_ptr(cu_steps), num_traj, num_steps, _ptr(step_img), _ptr(step_txt), window, keep,
                     _ptr(sizes), _ptr(ws), ws_bytes, _stream(stream))


def vcs_build_segments(cu_steps, num_traj, num_steps, step_img, step_txt, window, keep, seg_capacity,
                       tok_capacity, cu_seqlens, seg_traj, tok_gather, tok_src_step, tok_pos, tok_loss_mask,
                       sizes, ws, ws_bytes, stream=None) -> int:
    return _lib_build(_ptr(cu_steps), num_traj, num_steps, _ptr(step_img), _ptr(step_txt), window, keep,
                      seg_capacity, tok_capacity, _ptr(cu_seqlens), _ptr(seg_traj), _ptr(tok_gather),
                      _ptr(tok_src_step), _ptr(tok_pos), _ptr(tok_loss_mask), _ptr(sizes), _ptr(ws), ws_bytes,
                      _stream(stream))


def vcs_gather(q_traj, k_traj, v_traj, traj_tokens, tok_gather, num_tokens, hq, hkv, d, q, k, v, dev_status,
               stream=None) -> int:
    return _lib_gather(_ptr(q_traj), _ptr(k_traj), _ptr(v_traj), traj_tokens, _ptr(tok_gather), num_tokens, hq,
                       hkv, d, _ptr(q), _ptr(k), _ptr(v), _ptr(dev_status), _stream(stream))


def vcs_attn_fwd_workspace_size(num_segments, num_tokens, max_seqlen, hq, hkv, d) -> int:
    return int(_lib_fwd_ws(num_segments, num_tokens, max_seqlen, hq, hkv, d))


def vcs_attn_fwd(q, k, v, cu_seqlens, num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale, o, lse,
                 ws, ws_bytes, stream=None) -> int:
    return _lib_fwd(_ptr(q), _ptr(k), _ptr(v), _ptr(cu_seqlens), num_segments, num_tokens, max_seqlen, hq, hkv, d,
                    softmax_scale, _ptr(o), _ptr(lse), _ptr(ws), ws_bytes, _stream(stream))


def vcs_attn_bwd_workspace_size(num_segments, num_tokens, max_seqlen, hq, hkv, d) -> int:
    return int(_lib_bwd_ws(num_segments, num_tokens, max_seqlen, hq, hkv, d))


def vcs_attn_bwd(q, k, v, o, lse, dout, cu_seqlens, num_segments, num_tokens, max_seqlen, hq, hkv, d,
                 softmax_scale, dq, dk, dv, ws, ws_bytes, stream=None) -> int:
    return _lib_bwd(_ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), _ptr(dout), _ptr(cu_seqlens), num_segments,
                    num_tokens, max_seqlen, hq, hkv, d, softmax_scale, _ptr(dq), _ptr(dk), _ptr(dv), _ptr(ws),
                    ws_bytes, _stream(stream))


def vcs_attn_fwd_gathered(q_traj, k_traj, v_traj, traj_tokens, tok_gather, cu_seqlens, num_segments, num_tokens,
                          max_seqlen, hq, hkv, d, softmax_scale, o, lse, ws, ws_bytes, stream=None) -> int:
    return _lib_fwd_g(_ptr(q_traj), _ptr(k_traj), _ptr(v_traj), traj_tokens, _ptr(tok_gather), _ptr(cu_seqlens),
                      num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale, _ptr(o), _ptr(lse), _ptr(ws),
                      ws_bytes, _stream(stream))


def vcs_shared_prefix(cu_seqlens, seg_traj, tok_gather, num_segments, num_tokens, seg_shared, dev_status=None,
                      stream=None) -> int:
    return _lib_shared(_ptr(cu_seqlens), _ptr(seg_traj), _ptr(tok_gather), num_segments, num_tokens,
                       _ptr(seg_shared), _ptr(dev_status), _stream(stream))


def vcs_attn_fwd_reuse(q, k, v, cu_seqlens, seg_shared, num_segments, num_tokens, max_seqlen, hq, hkv, d,
                       softmax_scale, o, lse, ws, ws_bytes, stream=None) -> int:
    return _lib_fwd_reuse(_ptr(q), _ptr(k), _ptr(v), _ptr(cu_seqlens), _ptr(seg_shared), num_segments, num_tokens,
                          max_seqlen, hq, hkv, d, softmax_scale, _ptr(o), _ptr(lse), _ptr(ws), ws_bytes,
                          _stream(stream))


def vcs_attn_bwd_gathered_workspace_size(num_segments, num_tokens, max_seqlen, traj_tokens, hq, hkv, d) -> int:
    return int(_lib_bwd_g_ws(num_segments, num_tokens, max_seqlen, traj_tokens, hq, hkv, d))


def vcs_attn_bwd_gathered(q_traj, k_traj, v_traj, traj_tokens, tok_gather, o, lse, dout, cu_seqlens, num_segments,
                          num_tokens, max_seqlen, hq, hkv, d, softmax_scale, dq_traj, dk_traj, dv_traj, ws, ws_bytes,
                          stream=None) -> int:
    return _lib_bwd_g(_ptr(q_traj), _ptr(k_traj), _ptr(v_traj), traj_tokens, _ptr(tok_gather), _ptr(o), _ptr(lse),
                      _ptr(dout), _ptr(cu_seqlens), num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale,
                      _ptr(dq_traj), _ptr(dk_traj), _ptr(dv_traj), _ptr(ws), ws_bytes, _stream(stream))


def vcs_attn_bwd_noalloc(q, k, v, o, lse, dout, cu_seqlens, num_segments, num_tokens, max_seqlen, hq, hkv, d,
                         softmax_scale, dq, dk, dv, dev_status, stream=None) -> int:
    """vcs_attn_bwd with the library's fixed scratch instead of a caller workspace.

    For callers that cannot allocate device memory (see include/vcs.h): all
    inputs and outputs are still the caller's; the problem must fit the fixed
    scratch, else VCS_ERR_WORKSPACE is returned before any launch.
    """
    return _lib_bwd_noalloc(_ptr(q), _ptr(k), _ptr(v), _ptr(o), _ptr(lse), _ptr(dout), _ptr(cu_seqlens),
                            num_segments, num_tokens, max_seqlen, hq, hkv, d, softmax_scale, _ptr(dq), _ptr(dk),
                            _ptr(dv), _ptr(dev_status), _stream(stream))


NOALLOC_SCRATCH_BYTES = 32 << 20


def vcs_grpo_loss_workspace_size(num_tokens: int) -> int:
    return int(_lib_loss_ws(num_tokens))


def vcs_grpo_loss(logp, old_logp, ref_logp, tok_loss_mask, cu_seqlens, seg_traj, num_segments, num_tokens, adv,
                  num_traj, eps_low, eps_high, clip_cap, kl_coef, loss, dlogp, ws, ws_bytes, stream=None) -> int:
    return _lib_loss(_ptr(logp), _ptr(old_logp), _ptr(ref_logp), _ptr(tok_loss_mask), _ptr(cu_seqlens),
                     _ptr(seg_traj), num_segments, num_tokens, _ptr(adv), num_traj, eps_low, eps_high, clip_cap,
                     kl_coef, _ptr(loss), _ptr(dlogp), _ptr(ws), ws_bytes, _stream(stream))


def vcs_group_advantage(rewards, num_groups, group_size, eps, adv, stream=None) -> int:
    return _lib_adv(_ptr(rewards), num_groups, group_size, eps, _ptr(adv), _stream(stream))


def vcs_stream_fields(traj_ids, traj_logp, traj_tokens, tok_gather, tok_loss_mask, num_tokens, ids, logp,
                      dev_status, stream=None) -> int:
    return _lib_fields(_ptr(traj_ids), _ptr(traj_logp), traj_tokens, _ptr(tok_gather), _ptr(tok_loss_mask),
                       num_tokens, _ptr(ids), _ptr(logp), _ptr(dev_status), _stream(stream))


def vcs_compact_workspace_size(num_tokens: int) -> int:
    return int(_lib_compact_ws(num_tokens))


def vcs_compact_trainable(tok_loss_mask, num_tokens, idx, idx_capacity, count, ws, ws_bytes, stream=None) -> int:
    return _lib_compact(_ptr(tok_loss_mask), num_tokens, _ptr(idx), idx_capacity, _ptr(count), _ptr(ws), ws_bytes,
                        _stream(stream))


def vcs_selftest_bounded_wait(dev_status, limit_cycles, stream=None) -> int:
    return _lib_selftest_wait(_ptr(dev_status), int(limit_cycles), _stream(stream))


# ---------------------------------------------------------------- conveniences

def _check(status: int, where: str):
    if status != 0:
        raise VcsError(status, where)


def _ws(nbytes: int, device) -> torch.Tensor:
    return torch.empty(max(nbytes, 256), dtype=torch.uint8, device=device)


def plan_segments(cu_steps, step_img, step_txt, window: int, keep: int = 0, stream=None):
    """Segment count, token count and longest segment (synchronises once)."""
    dev = cu_steps.device
    num_traj, num_steps = cu_steps.numel() - 1, step_img.numel()
    nb = vcs_segments_workspace_size(num_traj, num_steps)
    ws = _ws(nb, dev)
    sizes = torch.zeros(3, dtype=torch.int64, device=dev)   # 24 bytes = vcs_sizes
    _check(vcs_plan_segments(cu_steps, num_traj, num_steps, step_img, step_txt, window, keep, sizes, ws, nb,
                             stream), "vcs_plan_segments")
    host = sizes.cpu()
    ns, nt = int(host[0]), int(host[1])
    mx = int(host[2] & 0xFFFFFFFF)
    st = int((host[2] >> 32) & 0xFFFFFFFF)
    _check(st, "vcs_plan_segments (device)")
    return ns, nt, mx


def build_segments(cu_steps, step_img, step_txt, window: int, keep: int = 0, with_mask: bool = True,
                   stream=None):
    """Plan + build: returns a dict of device tensors and the sizes."""
    dev = cu_steps.device
    num_traj, num_steps = cu_steps.numel() - 1, step_img.numel()
    ns, nt, mx = plan_segments(cu_steps, step_img, step_txt, window, keep, stream)
    nb = vcs_segments_workspace_size(num_traj, num_steps)
    ws = _ws(nb, dev)
    sizes = torch.zeros(3, dtype=torch.int64, device=dev)
    out = dict(cu_seqlens=torch.empty(ns + 1, dtype=torch.int32, device=dev),
               seg_traj=torch.empty(ns, dtype=torch.int32, device=dev),
               tok_gather=torch.empty(nt, dtype=torch.int32, device=dev),
               tok_src_step=torch.empty(nt, dtype=torch.int32, device=dev),
               tok_pos=torch.empty(nt, dtype=torch.int32, device=dev),
               tok_loss_mask=torch.empty(nt, dtype=torch.uint8, device=dev) if with_mask else None)
    _check(vcs_build_segments(cu_steps, num_traj, num_steps, step_img, step_txt, window, keep, ns, nt,
                              out["cu_seqlens"], out["seg_traj"], out["tok_gather"], out["tok_src_step"],
                              out["tok_pos"], out["tok_loss_mask"], sizes, ws, nb, stream), "vcs_build_segments")
    st = int((sizes[2].item() >> 32) & 0xFFFFFFFF)
    _check(st, "vcs_build_segments (device)")
    out.update(num_segments=ns, num_tokens=nt, max_seqlen=mx)
    return out


def gather(q_traj, k_traj, v_traj, tok_gather, stream=None):
    nt = tok_gather.numel()
    _, hq, d = q_traj.shape
    hkv = k_traj.shape[1]
    dev = q_traj.device
    q = torch.empty((nt, hq, d), dtype=q_traj.dtype, device=dev)
    k = torch.empty((nt, hkv, d), dtype=k_traj.dtype, device=dev)
    v = torch.empty((nt, hkv, d), dtype=v_traj.dtype, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    _check(vcs_gather(q_traj, k_traj, v_traj, q_traj.shape[0], tok_gather, nt, hq, hkv, d, q, k, v, status,
                      stream), "vcs_gather")
    _check(int(status.item()), "vcs_gather (device)")
    return q, k, v


def attn_fwd(q, k, v, cu_seqlens, max_seqlen: int, softmax_scale: float = 0.0, stream=None, check=True):
    nt, hq, d = q.shape
    hkv = k.shape[1]
    ns = cu_seqlens.numel() - 1
    o = torch.empty_like(q)
    lse = torch.empty((hq, nt), dtype=torch.float32, device=q.device)
    nb = vcs_attn_fwd_workspace_size(ns, nt, max_seqlen, hq, hkv, d)
    ws = _ws(nb, q.device)
    _check(vcs_attn_fwd(q, k, v, cu_seqlens, ns, nt, max_seqlen, hq, hkv, d, softmax_scale, o, lse, ws, nb,
                        stream), "vcs_attn_fwd")
    if check:
        _check(int(ws[:4].view(torch.int32).item()), "vcs_attn_fwd (device)")
    return o, lse


def attn_bwd(q, k, v, o, lse, dout, cu_seqlens, max_seqlen: int, softmax_scale: float = 0.0, stream=None,
             check=True):
    nt, hq, d = q.shape
    hkv = k.shape[1]
    ns = cu_seqlens.numel() - 1
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    nb = vcs_attn_bwd_workspace_size(ns, nt, max_seqlen, hq, hkv, d)
    ws = _ws(nb, q.device)
    _check(vcs_attn_bwd(q, k, v, o, lse, dout, cu_seqlens, ns, nt, max_seqlen, hq, hkv, d, softmax_scale, dq, dk,
                        dv, ws, nb, stream), "vcs_attn_bwd")
    if check:
        _check(int(ws[:4].view(torch.int32).item()), "vcs_attn_bwd (device)")
    return dq, dk, dv


def shared_prefix(cu_seqlens, seg_traj, tok_gather, stream=None):
    """Per segment, its common prefix length with the previous segment of its trajectory."""
    ns = cu_seqlens.numel() - 1
    out = torch.empty(max(ns, 0), dtype=torch.int32, device=cu_seqlens.device)
    status = torch.zeros(1, dtype=torch.int32, device=cu_seqlens.device)
    _check(vcs_shared_prefix(cu_seqlens, seg_traj, tok_gather, ns, tok_gather.numel(), out, status, stream),
           "vcs_shared_prefix")
    _check(int(status.item()), "vcs_shared_prefix (device)")
    return out


def attn_fwd_reuse(q, k, v, cu_seqlens, seg_shared, max_seqlen: int, softmax_scale: float = 0.0, stream=None,
                   check=True):
    """vcs_attn_fwd's o and lse, computing each shared prefix row once per trajectory."""
    nt, hq, d = q.shape
    hkv = k.shape[1]
    ns = cu_seqlens.numel() - 1
    o = torch.empty_like(q)
    lse = torch.empty((hq, nt), dtype=torch.float32, device=q.device)
    nb = vcs_attn_fwd_workspace_size(ns, nt, max_seqlen, hq, hkv, d)
    ws = _ws(nb, q.device)
    _check(vcs_attn_fwd_reuse(q, k, v, cu_seqlens, seg_shared, ns, nt, max_seqlen, hq, hkv, d, softmax_scale, o, lse,
                              ws, nb, stream), "vcs_attn_fwd_reuse")
    if check:
        _check(int(ws[:4].view(torch.int32).item()), "vcs_attn_fwd_reuse (device)")
    return o, lse


def attn_fwd_gathered(q_traj, k_traj, v_traj, tok_gather, cu_seqlens, max_seqlen: int, softmax_scale: float = 0.0,
                      stream=None, check=True):
    """Attention forward over the segments, reading trajectory-layout q/k/v through tok_gather;
    o [num_tokens, hq, d] and lse [hq, num_tokens] in segment layout."""
    tt, hq, d = q_traj.shape
    hkv = k_traj.shape[1]
    nt = tok_gather.numel()
    ns = cu_seqlens.numel() - 1
    o = torch.empty((nt, hq, d), dtype=q_traj.dtype, device=q_traj.device)
    lse = torch.empty((hq, nt), dtype=torch.float32, device=q_traj.device)
    nb = vcs_attn_fwd_workspace_size(ns, nt, max_seqlen, hq, hkv, d)
    ws = _ws(nb, q_traj.device)
    _check(vcs_attn_fwd_gathered(q_traj, k_traj, v_traj, tt, tok_gather, cu_seqlens, ns, nt, max_seqlen, hq, hkv, d,
                                 softmax_scale, o, lse, ws, nb, stream), "vcs_attn_fwd_gathered")
    if check:
        _check(int(ws[:4].view(torch.int32).item()), "vcs_attn_fwd_gathered (device)")
    return o, lse


def attn_bwd_gathered(q_traj, k_traj, v_traj, tok_gather, o, lse, dout, cu_seqlens, max_seqlen: int,
                      softmax_scale: float = 0.0, stream=None, check=True):
    """Attention backward over the segments with trajectory-layout q/k/v read through tok_gather;
    returns dq, dk, dv in trajectory layout (each token's segment copies summed)."""
    tt, hq, d = q_traj.shape
    hkv = k_traj.shape[1]
    nt = tok_gather.numel()
    ns = cu_seqlens.numel() - 1
    dq, dk, dv = torch.empty_like(q_traj), torch.empty_like(k_traj), torch.empty_like(v_traj)
    nb = vcs_attn_bwd_gathered_workspace_size(ns, nt, max_seqlen, tt, hq, hkv, d)
    ws = _ws(nb, q_traj.device)
    _check(vcs_attn_bwd_gathered(q_traj, k_traj, v_traj, tt, tok_gather, o, lse, dout, cu_seqlens, ns, nt,
                                 max_seqlen, hq, hkv, d, softmax_scale, dq, dk, dv, ws, nb, stream),
           "vcs_attn_bwd_gathered")
    if check:
        _check(int(ws[:4].view(torch.int32).item()), "vcs_attn_bwd_gathered (device)")
    return dq, dk, dv


def grpo_loss(logp, old_logp, ref_logp, tok_loss_mask, cu_seqlens, seg_traj, adv, eps_low: float = 0.2,
              eps_high: float = 0.28, clip_cap: float = 3.0, kl_coef: float = 1e-4, with_grad: bool = True,
              stream=None, check=True):
    """Loss (fp64 device scalar) and d loss / d logp (fp32, or None)."""
    nt = logp.numel()
    dev = logp.device
    loss = torch.empty(1, dtype=torch.float64, device=dev)
    dlogp = torch.empty(nt, dtype=torch.float32, device=dev) if with_grad else None
    nb = vcs_grpo_loss_workspace_size(nt)
    ws = _ws(nb, dev)
    _check(vcs_grpo_loss(logp, old_logp, ref_logp, tok_loss_mask, cu_seqlens, seg_traj, seg_traj.numel(), nt, adv,
                         adv.numel(), eps_low, eps_high, clip_cap, kl_coef, loss, dlogp, ws, nb, stream),
           "vcs_grpo_loss")
    if check:
        _check(int(ws[:4].view(torch.int32).item()), "vcs_grpo_loss (device)")
    return loss, dlogp


def stream_fields(traj_ids, traj_logp, tok_gather, tok_loss_mask, stream=None):
    """(ids int32, logp fp32) of every segment token (Algorithm 1's stream fields)."""
    nt = tok_gather.numel()
    dev = tok_gather.device
    ids = torch.empty(nt, dtype=torch.int32, device=dev)
    logp = torch.empty(nt, dtype=torch.float32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    _check(vcs_stream_fields(traj_ids, traj_logp, traj_ids.numel(), tok_gather, tok_loss_mask, nt, ids, logp, status,
                             stream), "vcs_stream_fields")
    _check(int(status.item()), "vcs_stream_fields (device)")
    return ids, logp


def compact_trainable(tok_loss_mask, capacity=None, stream=None):
    """Indices of the trainable tokens in order (int32 device tensor)."""
    nt = tok_loss_mask.numel()
    dev = tok_loss_mask.device
    cap = nt if capacity is None else capacity
    idx = torch.empty(max(cap, 1), dtype=torch.int32, device=dev)
    count = torch.zeros(1, dtype=torch.int64, device=dev)
    nb = vcs_compact_workspace_size(nt)
    ws = _ws(nb, dev)
    _check(vcs_compact_trainable(tok_loss_mask, nt, idx, cap, count, ws, nb, stream), "vcs_compact_trainable")
    _check(int(ws[:4].view(torch.int32).item()), "vcs_compact_trainable (device)")
    return idx[: int(count.item())]


def group_advantage(rewards, group_size: int, eps: float = 1e-6, stream=None):
    adv = torch.empty_like(rewards)
    _check(vcs_group_advantage(rewards, rewards.numel() // group_size, group_size, eps, adv, stream),
           "vcs_group_advantage")
    return adv


def selftest_bounded_wait(limit_cycles: int = 200_000_000, device="cuda", stream=None) -> int:
    """Runs the bounded-wait self-test (a wait on a barrier nothing arrives on, given up after
    limit_cycles SM cycles) and returns the device status it left: VCS_ERR_DEVICE_TIMEOUT (7)
    when the mechanism works.  Synchronises the device."""
    status = torch.zeros(1, dtype=torch.int32, device=device)
    _check(vcs_selftest_bounded_wait(status, limit_cycles, stream), "vcs_selftest_bounded_wait")
    torch.cuda.synchronize(status.device)
    return int(status.item())


def default_scale(d: int) -> float:
    return 1.0 / math.sqrt(d)
