"""GPU parity of vcs_grpo_loss / vcs_group_advantage (App. C.2 objective) against
the fp64 oracle: hand-worked branches, random batches over builder layouts,
edge cases and the device-side check."""
import numpy as np
import pytest
import torch

from oracle import loss as oloss

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _vcs():
    from paper_2607_11185_gb300 import vcs
    return vcs


def _layout(seed, num_traj=6, steps=(3, 12)):
    """A builder layout (GPU builder, window 3) for random step counts."""
    vcs = _vcs()
    rng = np.random.default_rng(seed)
    T = rng.integers(steps[0], steps[1] + 1, size=num_traj)
    cu = np.concatenate([[0], np.cumsum(T)]).astype(np.int32)
    img = rng.integers(0, 300, size=int(T.sum())).astype(np.int32)
    txt = rng.integers(0, 60, size=int(T.sum())).astype(np.int32)
    lay = vcs.build_segments(torch.from_numpy(cu).to(DEV), torch.from_numpy(img).to(DEV),
                             torch.from_numpy(txt).to(DEV), 3, 0)
    return lay, num_traj


def _inputs(n, seed):
    g = torch.Generator().manual_seed(seed)
    logp = -torch.rand(n, generator=g, dtype=torch.float64) * 8.0
    old = logp + torch.randn(n, generator=g, dtype=torch.float64) * 0.4
    ref = logp + torch.randn(n, generator=g, dtype=torch.float64) * 0.1
    return logp.float(), old.float(), ref.float()


def _tol_check(loss_g, dlogp_g, logp, old, ref, mask, cu, st, adv, ntraj, **kw):
    loss_o, g_o = oloss.grpo_loss_vec(logp.numpy(), old.numpy(), ref.numpy(), mask, cu, st, adv, ntraj, **kw)
    # per-token terms are fp32: compare the sum against the sum of magnitudes
    lp = logp.double().numpy()
    rho = np.exp(lp - old.double().numpy())
    a_tok = np.asarray(adv, np.float64)[oloss.token_traj(cu, st)]
    r = ref.double().numpy() - lp
    kl = kw.get("kl_coef", 1e-4) * np.abs(np.exp(r) - r - 1.0)
    scale = ((np.abs(rho * a_tok) + kl) * (np.asarray(mask) != 0)).sum() / ntraj + 1e-30
    assert abs(loss_g - loss_o) <= 2e-6 * scale + 1e-12, (loss_g, loss_o, scale)
    # gradient element by element; a token whose fp32 ratio sits on a branch point may take
    # either branch (both are valid sub-gradients)
    diff = np.abs(dlogp_g - g_o)
    tol = 1e-5 * np.abs(g_o) + 1e-7 * np.abs(g_o).max() + 1e-12
    bad = diff > tol
    if bad.any():
        rb = rho[bad]
        near = np.zeros(bad.sum(), bool)
        for b in (1.0 - kw.get("eps_low", 0.2), 1.0 + kw.get("eps_high", 0.28), kw.get("clip_cap", 3.0)):
            near |= np.abs(rb / b - 1.0) < 1e-5
        assert near.all(), (np.flatnonzero(bad)[:10], diff[bad][:10], tol[bad][:10])


def _run(vcs, logp, old, ref, lay, adv, **kw):
    loss, dlogp = vcs.grpo_loss(logp.to(DEV), old.to(DEV), ref.to(DEV), lay["tok_loss_mask"], lay["cu_seqlens"],
                                lay["seg_traj"], adv.to(DEV), **kw)
    return float(loss.item()), dlogp.cpu().double().numpy()


def test_hand_worked_branches():
    vcs = _vcs()
    rho = torch.tensor([1.0, 1.0, 1.5, 0.5, 0.5, 1.1, 4.0, 2.0], dtype=torch.float64)
    old = torch.full((8,), -1.0, dtype=torch.float64)
    logp = (old + rho.log()).float()
    mask = torch.tensor([0, 1, 1, 1, 1, 1, 1, 1], dtype=torch.uint8)
    lay = dict(tok_loss_mask=mask.to(DEV), cu_seqlens=torch.tensor([0, 4, 8], dtype=torch.int32, device=DEV),
               seg_traj=torch.tensor([0, 1], dtype=torch.int32, device=DEV))
    adv = torch.tensor([2.0, -1.0])
    loss, g = _run(vcs, logp, old.float(), logp, lay, adv)
    objs = [2.0, 2.56, 1.0, -0.8, -1.1, -3.0, -2.0]
    assert loss == pytest.approx(-sum(objs) / 2, abs=1e-5)
    np.testing.assert_allclose(g, [0.0, -1.0, 0.0, -0.5, 0.0, 0.55, 0.0, 1.0], atol=1e-5)


@pytest.mark.parametrize("seed", range(4))
def test_random_layouts(seed):
    vcs = _vcs()
    lay, ntraj = _layout(seed)
    n = lay["num_tokens"]
    logp, old, ref = _inputs(n, seed)
    rewards = torch.from_numpy((np.random.default_rng(seed).random(ntraj) < 0.5).astype(np.float32))
    adv = oloss.group_advantage(rewards.numpy(), 2).astype(np.float32)
    kw = dict(eps_low=0.2, eps_high=0.28, clip_cap=3.0, kl_coef=0.05)
    loss, g = _run(vcs, logp, old, ref, lay, torch.from_numpy(adv), **kw)
    _tol_check(loss, g, logp, old, ref, lay["tok_loss_mask"].cpu().numpy(), lay["cu_seqlens"].cpu().numpy(),
               lay["seg_traj"].cpu().numpy(), adv, ntraj, **kw)


def test_workload_scale():
    # the 32-trajectory workload's layout (4.2 M segment tokens), paper hyperparameters
    from paper_2607_11185_gb300 import workloads
    vcs = _vcs()
    w = workloads.WORKLOADS["traj32_w3"]
    cu, img, txt = workloads.draw_steps(w)
    lay = vcs.build_segments(torch.from_numpy(cu).to(DEV), torch.from_numpy(img).to(DEV),
                             torch.from_numpy(txt).to(DEV), w.window, w.keep)
    n = lay["num_tokens"]
    logp, old, ref = _inputs(n, 99)
    rewards = (np.random.default_rng(5).random(w.num_traj) < 0.4).astype(np.float32)
    adv = oloss.group_advantage(rewards, 8).astype(np.float32)
    loss, g = _run(vcs, logp, old, ref, lay, torch.from_numpy(adv))
    _tol_check(loss, g, logp, old, ref, lay["tok_loss_mask"].cpu().numpy(), lay["cu_seqlens"].cpu().numpy(),
               lay["seg_traj"].cpu().numpy(), adv, w.num_traj)


def test_deterministic():
    vcs = _vcs()
    lay, ntraj = _layout(3, num_traj=12, steps=(20, 40))
    logp, old, ref = _inputs(lay["num_tokens"], 3)
    adv = torch.randn(ntraj, generator=torch.Generator().manual_seed(1))
    a = _run(vcs, logp, old, ref, lay, adv)
    b = _run(vcs, logp, old, ref, lay, adv)
    assert a[0] == b[0]
    assert np.array_equal(a[1], b[1])


def test_edge_cases():
    vcs = _vcs()
    # no tokens: loss 0
    z = torch.zeros(0, device=DEV)
    loss, g = vcs.grpo_loss(z, z, z, torch.zeros(0, dtype=torch.uint8, device=DEV),
                            torch.zeros(1, dtype=torch.int32, device=DEV), torch.zeros(0, dtype=torch.int32, device=DEV),
                            torch.ones(1, device=DEV))
    assert float(loss.item()) == 0.0
    # everything masked: loss 0 and zero gradient
    lay, ntraj = _layout(8)
    logp, old, ref = _inputs(lay["num_tokens"], 8)
    lay["tok_loss_mask"].zero_()
    loss, g = _run(vcs, logp, old, ref, lay, torch.ones(ntraj))
    assert loss == 0.0 and not g.any()
    # empty segments inside cu_seqlens (zero-token steps) keep the token -> trajectory map right
    cu = torch.tensor([0, 3, 3, 3, 7], dtype=torch.int32, device=DEV)
    st = torch.tensor([0, 1, 1, 2], dtype=torch.int32, device=DEV)
    m = torch.ones(7, dtype=torch.uint8, device=DEV)
    lp = torch.full((7,), -1.0)
    loss, g = _run(vcs, lp, lp, lp, dict(tok_loss_mask=m, cu_seqlens=cu, seg_traj=st), torch.tensor([1.0, 5.0, -2.0]))
    want = -(3 * 1.0 + 4 * -2.0) / 3
    assert loss == pytest.approx(want, abs=1e-6)
    np.testing.assert_allclose(g, [-1 / 3] * 3 + [2 / 3] * 4, atol=1e-6)


def test_device_check_bad_trajectory():
    vcs = _vcs()
    cu = torch.tensor([0, 2, 4], dtype=torch.int32, device=DEV)
    st = torch.tensor([0, 5], dtype=torch.int32, device=DEV)        # 5 is outside [0, 2)
    m = torch.ones(4, dtype=torch.uint8, device=DEV)
    lp = torch.full((4,), -1.0, device=DEV)
    with pytest.raises(vcs.VcsError) as e:
        vcs.grpo_loss(lp, lp, lp, m, cu, st, torch.ones(2, device=DEV))
    assert e.value.status == 6


def test_host_argument_errors():
    vcs = _vcs()
    lp = torch.zeros(4, device=DEV)
    m = torch.ones(4, dtype=torch.uint8, device=DEV)
    cu = torch.tensor([0, 4], dtype=torch.int32, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    adv = torch.ones(1, device=DEV)
    loss = torch.empty(1, dtype=torch.float64, device=DEV)
    nb = vcs.vcs_grpo_loss_workspace_size(4)
    ws = torch.empty(nb, dtype=torch.uint8, device=DEV)
    ok = vcs.vcs_grpo_loss(lp, lp, lp, m, cu, st, 1, 4, adv, 1, 0.2, 0.28, 3.0, 1e-4, loss, None, ws, nb)
    assert ok == 0
    assert vcs.vcs_grpo_loss(lp, lp, lp, m, cu, st, 1, 4, adv, 0, 0.2, 0.28, 3.0, 1e-4, loss, None, ws, nb) == 1
    assert vcs.vcs_grpo_loss(lp, lp, lp, m, cu, st, 1, 4, adv, 1, 0.2, 0.28, 1.1, 1e-4, loss, None, ws, nb) == 1
    assert vcs.vcs_grpo_loss(lp, lp, lp, m, cu, st, 1, 4, adv, 1, 0.2, 0.28, 3.0, 1e-4, loss, None, ws, 8) == 8
    assert vcs.vcs_grpo_loss(None, lp, lp, m, cu, st, 1, 4, adv, 1, 0.2, 0.28, 3.0, 1e-4, loss, None, ws, nb) == 1


@pytest.mark.parametrize("group_size", [1, 2, 8, 16])
def test_group_advantage(group_size):
    vcs = _vcs()
    r = torch.rand(37 * group_size, generator=torch.Generator().manual_seed(group_size))
    r[: group_size] = 0.5                                  # one group with equal rewards
    a = vcs.group_advantage(r.to(DEV), group_size).cpu().double().numpy()
    want = oloss.group_advantage(r.double().numpy(), group_size)
    np.testing.assert_allclose(a, want, rtol=1e-6, atol=1e-6)
