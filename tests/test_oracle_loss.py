"""Pins for oracle/loss.py (App. C.2 RL objective): hand-worked values, closed
forms, finite differences and invariants.  CPU only."""
import math

import numpy as np
import pytest

from oracle import loss as oloss
from oracle import segments as oseg


def _two_traj_example():
    # trajectory 0: A = +2, segment 0 (4 tokens); trajectory 1: A = -1, segment 1 (4 tokens)
    rho = np.array([1.0, 1.0, 1.5, 0.5, 0.5, 1.1, 4.0, 2.0])
    mask = np.array([0, 1, 1, 1, 1, 1, 1, 1], np.uint8)
    old = np.full(8, -1.0)
    logp = old + np.log(rho)
    return dict(logp=logp, old=old, ref=logp.copy(), mask=mask, cu=np.array([0, 4, 8]), seg_traj=np.array([0, 1]),
                adv=np.array([2.0, -1.0]))


def test_hand_worked_clipping_branches():
    e = _two_traj_example()
    loss, g = oloss.grpo_loss(e["logp"], e["old"], e["ref"], e["mask"], e["cu"], e["seg_traj"], e["adv"], 2)
    # objectives by hand: traj 0 (A=2): rho=1 -> 2, rho=1.5 -> 1.28*2 (clipped), rho=0.5 -> 1.0
    #                     traj 1 (A=-1): rho=0.5 -> 0.8*-1 (clipped low), rho=1.1 -> -1.1,
    #                                    rho=4 -> 3*-1 (dual-clip cap), rho=2 -> -2
    objs = [2.0, 2.56, 1.0, -0.8, -1.1, -3.0, -2.0]
    assert loss == pytest.approx(-sum(objs) / 2, abs=1e-12)
    # gradients: rho*A on the rho-dependent branch, 0 on a constant branch, divided by N_traj = 2
    want = np.array([0.0, -1.0, 0.0, -0.5, 0.0, 0.55, 0.0, 1.0])
    np.testing.assert_allclose(g, want, atol=1e-12)


def test_kl_closed_form():
    # rho = 1, A = 0: only the KL estimator exp(r) - r - 1, r = ref - logp, remains
    r = 0.3
    logp = np.array([-2.0])
    loss, g = oloss.grpo_loss(logp, logp, logp + r, np.array([1]), [0, 1], [0], [0.0], 1, kl_coef=0.5)
    assert loss == pytest.approx(0.5 * (math.exp(r) - r - 1.0), abs=1e-14)
    assert g[0] == pytest.approx(0.5 * (1.0 - math.exp(r)), abs=1e-14)


def test_on_policy_reduces_to_advantage_sum():
    # rho = 1 and pi_ref = pi_theta: L = -(1/N) sum_t mask_t A_traj(t), dL/dlogp = -mask A / N
    rng = np.random.default_rng(0)
    cu = np.array([0, 5, 9, 20])
    seg_traj = np.array([0, 0, 2])
    adv = rng.normal(size=3)
    mask = rng.integers(0, 2, size=20).astype(np.uint8)
    logp = rng.normal(size=20) - 3.0
    loss, g = oloss.grpo_loss(logp, logp, logp, mask, cu, seg_traj, adv, 3)
    a_tok = adv[np.repeat(seg_traj, np.diff(cu))]
    mf = mask.astype(np.float64)
    assert loss == pytest.approx(-(mf * a_tok).sum() / 3, abs=1e-12)
    np.testing.assert_allclose(g, -mf * a_tok / 3, atol=1e-14)


def _random_case(seed, n=64, ntraj=4):
    rng = np.random.default_rng(seed)
    lens = rng.integers(1, 12, size=9)
    cu = np.concatenate([[0], np.cumsum(lens)])
    n = int(cu[-1])
    seg_traj = np.sort(rng.integers(0, ntraj, size=9))
    adv = rng.normal(size=ntraj) * 2
    old = rng.normal(size=n) - 2.0
    # keep rho away from the branch points 0.8, 1.28 and 3 so that finite differences stay on one branch
    rho = np.exp(rng.normal(size=n) * 0.6)
    for b in (0.8, 1.28, 3.0):
        close = np.abs(rho - b) < 0.02
        rho[close] = b + 0.05
    logp = old + np.log(rho)
    ref = logp + rng.normal(size=n) * 0.2
    mask = rng.integers(0, 2, size=n).astype(np.uint8)
    return logp, old, ref, mask, cu, seg_traj, adv, ntraj


@pytest.mark.parametrize("seed", range(3))
def test_finite_differences(seed):
    logp, old, ref, mask, cu, st, adv, nt = _random_case(seed)
    _, g = oloss.grpo_loss(logp, old, ref, mask, cu, st, adv, nt, kl_coef=0.3)
    h = 1e-6
    for t in range(len(logp)):
        lp_p, lp_m = logp.copy(), logp.copy()
        lp_p[t] += h
        lp_m[t] -= h
        fp, _ = oloss.grpo_loss(lp_p, old, ref, mask, cu, st, adv, nt, kl_coef=0.3)
        fm, _ = oloss.grpo_loss(lp_m, old, ref, mask, cu, st, adv, nt, kl_coef=0.3)
        assert (fp - fm) / (2 * h) == pytest.approx(g[t], rel=1e-5, abs=1e-8), t


def test_masked_tokens_do_not_contribute():
    logp, old, ref, mask, cu, st, adv, nt = _random_case(7)
    loss, g = oloss.grpo_loss(logp, old, ref, mask, cu, st, adv, nt)
    assert np.all(g[mask == 0] == 0.0)
    lp2 = logp.copy()
    lp2[mask == 0] += 5.0
    loss2, _ = oloss.grpo_loss(lp2, old, ref, mask, cu, st, adv, nt)
    assert loss2 == loss


def test_advantage_scaling_is_linear_without_kl():
    logp, old, ref, mask, cu, st, adv, nt = _random_case(11)
    l1, g1 = oloss.grpo_loss(logp, old, ref, mask, cu, st, adv, nt, kl_coef=0.0)
    l2, g2 = oloss.grpo_loss(logp, old, ref, mask, cu, st, 2.5 * adv, nt, kl_coef=0.0)
    assert l2 == pytest.approx(2.5 * l1, rel=1e-12, abs=1e-14)
    np.testing.assert_allclose(g2, 2.5 * g1, rtol=1e-12, atol=1e-15)


def test_group_advantage():
    rng = np.random.default_rng(3)
    r = rng.normal(size=(5, 8))
    a = oloss.group_advantage(r.reshape(-1), 8, eps=0.0).reshape(5, 8)
    np.testing.assert_allclose(a.mean(axis=1), 0.0, atol=1e-12)
    np.testing.assert_allclose(a.std(axis=1), 1.0, atol=1e-12)
    # a group whose rollouts all score the same has zero advantage
    assert np.all(oloss.group_advantage(np.full(8, 0.7), 8) == 0.0)
    # hand-worked: rewards 0, 1 -> mean 0.5, population std 0.5 -> -1, +1
    np.testing.assert_allclose(oloss.group_advantage([0.0, 1.0], 2, eps=0.0), [-1.0, 1.0])


def test_token_trajectory_map_follows_the_builder():
    cu_steps = np.array([0, 3, 3, 8])
    img = np.full(8, 5)
    txt = np.arange(1, 9)
    lay = oseg.build(cu_steps, img, txt, 2, 0)
    tt = oloss.token_traj(lay["cu_seqlens"], lay["seg_traj"])
    # every segment token's source step lies inside the trajectory the map names
    step_traj = np.repeat(np.arange(3), np.diff(cu_steps))
    assert np.array_equal(step_traj[lay["tok_src_step"]], tt)


@pytest.mark.parametrize("seed", range(4))
def test_vectorised_form_equals_the_token_loop(seed):
    logp, old, ref, mask, cu, st, adv, nt = _random_case(seed + 20)
    # include tokens exactly on the branch points
    old[:3] = logp[:3] - np.log(np.array([0.8, 1.28, 3.0]))
    l1, g1 = oloss.grpo_loss(logp, old, ref, mask, cu, st, adv, nt, kl_coef=0.2)
    l2, g2 = oloss.grpo_loss_vec(logp, old, ref, mask, cu, st, adv, nt, kl_coef=0.2)
    assert l2 == pytest.approx(l1, rel=1e-12, abs=1e-14)
    np.testing.assert_allclose(g2, g1, rtol=1e-12, atol=1e-15)
