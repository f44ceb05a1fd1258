"""Token-level RL objective over segments, fp64 (test infrastructure).

The segments Algorithm 1 emits are consumed by the RL objective of App. C.2
(Eq. "RL objective" and the hyperparameter table): for task i and rollout j
with group-relative advantage A_ij shared by every segment of that rollout,

  L = - E_i E_j  sum_{s in S_ij} sum_{t in s, mask_t = 1}
          min( rho_t A_ij, clip(rho_t, 1 - eps_l, 1 + eps_h) A_ij )
      + lambda * KL(pi_theta || pi_ref),

rho_t = pi_theta(a_t | x_<t) / pi_rollout(a_t | x_<t), asymmetric clipping
eps_l = 0.2, eps_h = 0.28 (DAPO), a clip-ratio cap c = 3.0 and a KL weight
lambda = 1e-4.  The paper gives no formula for the cap or the KL estimator and
no normaliser beyond the expectations; this oracle reads them as follows:

  * cap: dual clipping for negative advantages, the objective of a token with
    A < 0 is max(min(rho A, clip(rho) A), c A);
  * KL: the per-token estimator exp(r) - r - 1 with r = log pi_ref - log pi_theta,
    taken over the same trainable tokens as the policy term;
  * the expectations are means over the batch's trajectories (tasks x
    rollouts): L = (1/N_traj) sum_t mask_t ( -o_t + lambda k_t );
  * group-relative advantage: (r - mean_g r) / (std_g r + eps) over the n
    rollouts of each task, population standard deviation.

Inputs are log-probabilities.  Everything, including the branch of the
clipped objective a token takes (a comparison of rho_t with 1 - eps_l,
1 + eps_h and c), is evaluated in fp64 from the given values.  The objective
is continuous in rho_t, so only the gradient of a token whose ratio lies on a
branch point depends on the side it is assigned to; there both sides are
valid sub-gradients.
"""
from __future__ import annotations

import numpy as np


def group_advantage(rewards, group_size: int, eps: float = 1e-6):
    """GRPO group-relative advantage (App. C.2): rewards are [num_groups * group_size],
    grouped consecutively; returns (r - mean) / (std + eps) per element, fp64."""
    r = np.asarray(rewards, dtype=np.float64).reshape(-1, group_size)
    mean = r.mean(axis=1, keepdims=True)
    std = np.sqrt(((r - mean) ** 2).mean(axis=1, keepdims=True))
    return ((r - mean) / (std + eps)).reshape(-1)


def token_traj(cu_seqlens, seg_traj):
    """Trajectory index of every segment token (segments in order)."""
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    st = np.asarray(seg_traj, dtype=np.int64)
    return np.repeat(st, np.diff(cu))


def grpo_loss(logp, old_logp, ref_logp, mask, cu_seqlens, seg_traj, adv, num_traj: int,
              eps_low: float = 0.2, eps_high: float = 0.28, clip_cap: float = 3.0, kl_coef: float = 1e-4):
    """Loss value and its gradient with respect to logp (both fp64).

    logp, old_logp, ref_logp: [num_tokens] per segment token; mask: [num_tokens]
    (1 = trainable); cu_seqlens / seg_traj: the builder's layout; adv: [num_traj].
    Returns (loss, dlogp)."""
    lp = np.asarray(logp, dtype=np.float64)
    old = np.asarray(old_logp, dtype=np.float64)
    ref = np.asarray(ref_logp, dtype=np.float64)
    m = np.asarray(mask).astype(np.float64)
    a = np.asarray(adv, dtype=np.float64)[token_traj(cu_seqlens, seg_traj)]
    n = lp.shape[0]
    loss_terms = np.zeros(n)
    grad = np.zeros(n)
    lo, hi = 1.0 - eps_low, 1.0 + eps_high
    for t in range(n):
        if m[t] == 0.0:
            continue
        rho = np.exp(lp[t] - old[t])
        A = a[t]
        # policy objective o and do/dlogp (rho-dependent branch -> rho*A, constant branch -> 0)
        if A >= 0.0:
            if rho <= hi:
                o, g = rho * A, rho * A
            else:
                o, g = hi * A, 0.0
        else:
            if rho < lo:
                o, g = lo * A, 0.0
            elif rho > clip_cap:
                o, g = clip_cap * A, 0.0
            else:
                o, g = rho * A, rho * A
        r = ref[t] - lp[t]
        k = np.exp(r) - r - 1.0
        dk = 1.0 - np.exp(r)          # d k / d logp
        loss_terms[t] = -o + kl_coef * k
        grad[t] = (-g + kl_coef * dk) / num_traj
    return float(loss_terms.sum() / num_traj), grad


def grpo_loss_vec(logp, old_logp, ref_logp, mask, cu_seqlens, seg_traj, adv, num_traj: int,
                  eps_low: float = 0.2, eps_high: float = 0.28, clip_cap: float = 3.0, kl_coef: float = 1e-4):
    """grpo_loss written with whole-array operations (same branches and values), for
    batches too large for the per-token loop.  Returns (loss, dlogp)."""
    lp = np.asarray(logp, dtype=np.float64)
    old = np.asarray(old_logp, dtype=np.float64)
    ref = np.asarray(ref_logp, dtype=np.float64)
    m = np.asarray(mask) != 0
    a = np.asarray(adv, dtype=np.float64)[token_traj(cu_seqlens, seg_traj)]
    rho = np.exp(lp - old)
    lo, hi = 1.0 - eps_low, 1.0 + eps_high
    pos = a >= 0.0
    const_pos = rho > hi
    const_lo = rho < lo
    const_cap = rho > clip_cap
    o = np.where(pos, np.where(const_pos, hi * a, rho * a),
                 np.where(const_lo, lo * a, np.where(const_cap, clip_cap * a, rho * a)))
    dobj = np.where(pos, np.where(const_pos, 0.0, rho * a), np.where(const_lo | const_cap, 0.0, rho * a))
    r = ref - lp
    k = np.exp(r) - r - 1.0
    terms = np.where(m, -o + kl_coef * k, 0.0)
    grad = np.where(m, (-dobj + kl_coef * (1.0 - np.exp(r))) / num_traj, 0.0)
    return float(terms.sum() / num_traj), grad
