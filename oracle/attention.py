"""Attention oracle over packed segments, fp64 (test infrastructure).

The paper trains its policy with the segments that Algorithm 1 emits
(Sec. 3.4; the actor-update and reference-policy phases of App. C.2); it does
not spell the attention out.  What is computed here is the plain definition
of causal softmax self-attention restricted to one segment, with grouped
query heads, read as follows:

  token i of segment sigma(i) at in-segment position p(i), query head h,
  key/value head g(h) = floor(h * Hkv / Hq):
    s_ij   = scale * <q_{i,h}, k_{j,g}>   for sigma(j) = sigma(i), p(j) <= p(i)
    lse_ih = ln sum_j exp(s_ij)
    o_ih   = sum_j exp(s_ij - lse_ih) v_{j,g}
  backward, for an upstream gradient dO:
    D_ih   = <dO_ih, o_ih>
    dS_ij  = P_ij (<dO_ih, v_{j,g}> - D_ih)
    dq_ih  = scale sum_j dS_ij k_{j,g}
    dk_jg  = scale sum_{h in g} sum_i dS_ij q_{i,h}
    dv_jg  = sum_{h in g} sum_i P_ij dO_ih

scale defaults to 1/sqrt(d).  Each query row is evaluated on its own; rows
are handled a block at a time only to bound memory (a row's keys are exactly
the keys at or before it, so no sum is reordered within a row).
"""
from __future__ import annotations

import math

import numpy as np


def _f64(x):
    if hasattr(x, "detach"):                       # torch tensor (any dtype)
        return x.detach().to("cpu").double().numpy()
    return np.asarray(x, dtype=np.float64)


def kv_head(h: int, hq: int, hkv: int) -> int:
    return (h * hkv) // hq


def _segments(cu_seqlens):
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    return [(int(cu[i]), int(cu[i + 1])) for i in range(len(cu) - 1)]


def _scores(qh, kh, rows, scale):
    """Masked score block: rows (in-segment positions) x keys 0..rows[-1]."""
    r0, r1 = rows
    s = scale * (qh[r0:r1] @ kh[:r1].T)
    pos_q = np.arange(r0, r1)[:, None]
    pos_k = np.arange(r1)[None, :]
    s[pos_k > pos_q] = -np.inf
    return s


def attn_fwd(q, k, v, cu_seqlens, scale=None, row_block=1024):
    """O [N,Hq,d] and lse [Hq,N] (natural log), fp64."""
    q, k, v = _f64(q), _f64(k), _f64(v)
    n, hq, d = q.shape
    hkv = k.shape[1]
    scale = 1.0 / math.sqrt(d) if scale is None or scale <= 0 else float(scale)
    o = np.zeros((n, hq, d))
    lse = np.zeros((hq, n))
    for b, e in _segments(cu_seqlens):
        for h in range(hq):
            g = kv_head(h, hq, hkv)
            qh, kh, vh = q[b:e, h], k[b:e, g], v[b:e, g]
            for r0 in range(0, e - b, row_block):
                r1 = min(e - b, r0 + row_block)
                s = _scores(qh, kh, (r0, r1), scale)
                m = s.max(axis=1)
                l = m + np.log(np.exp(s - m[:, None]).sum(axis=1))
                p = np.exp(s - l[:, None])
                lse[h, b + r0:b + r1] = l
                o[b + r0:b + r1, h] = p @ vh[:r1]
    return o, lse


def attn_bwd(q, k, v, do, cu_seqlens, scale=None, row_block=1024, o=None, lse=None):
    """dQ, dK, dV (fp64) from the definition; O and lse from ``attn_fwd`` unless given."""
    q, k, v, do = _f64(q), _f64(k), _f64(v), _f64(do)
    n, hq, d = q.shape
    hkv = k.shape[1]
    scale = 1.0 / math.sqrt(d) if scale is None or scale <= 0 else float(scale)
    if o is None or lse is None:
        o, lse = attn_fwd(q, k, v, cu_seqlens, scale, row_block)
    o, lse = _f64(o), _f64(lse)
    dmat = (do * o).sum(axis=-1)                  # D [N, Hq]
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    for b, e in _segments(cu_seqlens):
        for h in range(hq):
            g = kv_head(h, hq, hkv)
            qh, kh, vh, doh = q[b:e, h], k[b:e, g], v[b:e, g], do[b:e, h]
            for r0 in range(0, e - b, row_block):
                r1 = min(e - b, r0 + row_block)
                s = _scores(qh, kh, (r0, r1), scale)
                p = np.exp(s - lse[h, b + r0:b + r1][:, None])
                dp = doh[r0:r1] @ vh[:r1].T
                ds = p * (dp - dmat[b + r0:b + r1, h][:, None])
                dq[b + r0:b + r1, h] = scale * (ds @ kh[:r1])
                dk[b:b + r1, g] += scale * (ds.T @ qh[r0:r1])
                dv[b:b + r1, g] += p.T @ doh[r0:r1]
    return dq, dk, dv


# ---------------------------------------------------------------------------
# Sampled evaluation for segments too long for the full oracle.  Every value
# is the same definition evaluated for selected rows only.
# ---------------------------------------------------------------------------

def rows_fwd(q, k, v, seg, heads, rows, scale=None):
    """O and lse for query rows ``rows`` (in-segment positions) of segment ``seg=(b,e)``.

    Returns o [len(rows), len(heads), d], lse [len(heads), len(rows)].
    """
    b, e = seg
    d = q.shape[-1]
    hq, hkv = q.shape[1], k.shape[1]
    scale = 1.0 / math.sqrt(d) if scale is None or scale <= 0 else float(scale)
    o = np.zeros((len(rows), len(heads), d))
    lse = np.zeros((len(heads), len(rows)))
    for a, h in enumerate(heads):
        g = kv_head(h, hq, hkv)
        for c, i in enumerate(rows):
            qi = _f64(q[b + i, h])
            kk = _f64(k[b:b + i + 1, g])
            vv = _f64(v[b:b + i + 1, g])
            s = scale * (kk @ qi)
            m = s.max()
            l = m + np.log(np.exp(s - m).sum())
            o[c, a] = np.exp(s - l) @ vv
            lse[a, c] = l
    return o, lse


def rows_dq(q, k, v, do, seg, heads, rows, scale=None):
    """dQ for query rows ``rows`` of segment ``seg`` (each row needs only its own keys)."""
    b, e = seg
    d = q.shape[-1]
    hq, hkv = q.shape[1], k.shape[1]
    scale = 1.0 / math.sqrt(d) if scale is None or scale <= 0 else float(scale)
    dq = np.zeros((len(rows), len(heads), d))
    for a, h in enumerate(heads):
        g = kv_head(h, hq, hkv)
        for c, i in enumerate(rows):
            qi = _f64(q[b + i, h])
            doi = _f64(do[b + i, h])
            kk = _f64(k[b:b + i + 1, g])
            vv = _f64(v[b:b + i + 1, g])
            s = scale * (kk @ qi)
            m = s.max()
            p = np.exp(s - m)
            p /= p.sum()
            oi = p @ vv
            dp = vv @ doi
            ds = p * (dp - doi @ oi)
            dq[c, a] = scale * (ds @ kk)
    return dq


def keys_dkdv(q, k, v, do, seg, g, keys, scale=None):
    """dK, dV of kv-head ``g`` for key rows ``keys`` of segment ``seg``.

    Key j receives from every query row i >= j of every q-head of its group,
    so the cost grows with (L - min(keys)) * L; callers pick keys near the end
    of long segments.
    """
    b, e = seg
    L = e - b
    d = q.shape[-1]
    hq, hkv = q.shape[1], k.shape[1]
    scale = 1.0 / math.sqrt(d) if scale is None or scale <= 0 else float(scale)
    j0 = int(min(keys))
    kk = _f64(k[b:e, g])
    vv = _f64(v[b:e, g])
    keys = np.asarray(keys)
    dk = np.zeros((len(keys), d))
    dv = np.zeros((len(keys), d))
    for h in range(hq):
        if kv_head(h, hq, hkv) != g:
            continue
        for i in range(j0, L):
            qi = _f64(q[b + i, h])
            doi = _f64(do[b + i, h])
            s = scale * (kk[: i + 1] @ qi)
            m = s.max()
            p = np.exp(s - m)
            p /= p.sum()
            oi = p @ vv[: i + 1]
            dd = doi @ oi
            sel = keys <= i
            if not sel.any():
                continue
            kj = keys[sel]
            dsj = p[kj] * (vv[kj] @ doi - dd)
            dk[sel] += scale * dsj[:, None] * qi[None, :]
            dv[sel] += p[kj][:, None] * doi[None, :]
    return dk, dv


def keys_dkdv_blocked(q, k, v, do, seg, g, keys, scale=None, row_block=512):
    """dK, dV of kv-head ``g`` for key rows ``keys`` of segment ``seg`` (the same
    definition as ``keys_dkdv``), with the query rows taken a block at a time.

    A key receives from every later query row of every q-head of its group, and each
    such row needs its own lse and D = <dO, o>, which depend on all of that row's
    keys: so every row from min(keys) on is evaluated in full (as in ``attn_fwd``),
    then its P and dS restricted to the chosen keys are accumulated.  The cost is
    that of the forward over those rows, which makes keys near the start of long
    segments reachable.
    """
    b, e = seg
    L = e - b
    d = q.shape[-1]
    hq, hkv = q.shape[1], k.shape[1]
    scale = 1.0 / math.sqrt(d) if scale is None or scale <= 0 else float(scale)
    keys = np.asarray(keys, dtype=np.int64)
    kk = _f64(k[b:e, g])
    vv = _f64(v[b:e, g])
    dk = np.zeros((len(keys), d))
    dv = np.zeros((len(keys), d))
    for h in range(hq):
        if kv_head(h, hq, hkv) != g:
            continue
        qh = _f64(q[b:e, h])
        doh = _f64(do[b:e, h])
        for r0 in range(int(keys.min()), L, row_block):
            r1 = min(L, r0 + row_block)
            s = _scores(qh, kk, (r0, r1), scale)
            m = s.max(axis=1)
            lse = m + np.log(np.exp(s - m[:, None]).sum(axis=1))
            p = np.exp(s - lse[:, None])
            dd = (doh[r0:r1] * (p @ vv[:r1])).sum(axis=1)
            inside = keys < r1                 # later keys are masked for every row of the block
            kj = keys[inside]
            pk = p[:, kj]
            ds = pk * (doh[r0:r1] @ vv[kj].T - dd[:, None])
            dk[inside] += scale * (ds.T @ qh[r0:r1])
            dv[inside] += pk.T @ doh[r0:r1]
    return dk, dv
