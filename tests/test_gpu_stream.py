"""GPU parity of vcs_stream_fields / vcs_compact_trainable (Algorithm 1's token-ID
stream, App. C.1) against the oracle: bit-exact on builder layouts of every
workload and comparison layout, hand-worked fixture, edge cases."""
import numpy as np
import pytest
import torch

from oracle import segments as oseg
from oracle import stream as ostream
from paper_2607_11185_gb300 import workloads

pytestmark = pytest.mark.gpu

DEV = "cuda"


def _vcs():
    from paper_2607_11185_gb300 import vcs
    return vcs


def _check_layout(cu, img, txt, window, keep, seed):
    vcs = _vcs()
    lay = vcs.build_segments(torch.from_numpy(np.asarray(cu, np.int32)).to(DEV),
                             torch.from_numpy(np.asarray(img, np.int32)).to(DEV),
                             torch.from_numpy(np.asarray(txt, np.int32)).to(DEV), window, keep)
    ntraj_tok = int(np.sum(img, dtype=np.int64) + np.sum(txt, dtype=np.int64))
    rng = np.random.default_rng(seed)
    ids = rng.integers(0, 200000, size=ntraj_tok).astype(np.int32)
    lp = (-rng.random(ntraj_tok) * 6).astype(np.float32)
    g_ids, g_lp = vcs.stream_fields(torch.from_numpy(ids).to(DEV), torch.from_numpy(lp).to(DEV), lay["tok_gather"],
                                    lay["tok_loss_mask"])
    gather = lay["tok_gather"].cpu().numpy()
    mask = lay["tok_loss_mask"].cpu().numpy()
    o_ids, o_lp = ostream.stream_fields(ids, lp, gather, mask)
    assert np.array_equal(g_ids.cpu().numpy(), o_ids)
    assert np.array_equal(g_lp.cpu().numpy().view(np.uint32), o_lp.view(np.uint32))
    idx = vcs.compact_trainable(lay["tok_loss_mask"]).cpu().numpy()
    assert np.array_equal(idx, ostream.compact_trainable(mask))


def test_hand_worked():
    vcs = _vcs()
    ids = torch.tensor([10, 11, 12, 20, 21, 22, 30, 31, 32], dtype=torch.int32, device=DEV)
    lp = torch.tensor([0, 0, -1.5, 0, 0, -2.5, 0, 0, -3.5], dtype=torch.float32, device=DEV)
    lay = vcs.build_segments(torch.tensor([0, 3], dtype=torch.int32, device=DEV),
                             torch.tensor([2, 2, 2], dtype=torch.int32, device=DEV),
                             torch.tensor([1, 1, 1], dtype=torch.int32, device=DEV), 2, 0)
    g_ids, g_lp = vcs.stream_fields(ids, lp, lay["tok_gather"], lay["tok_loss_mask"])
    assert g_ids.tolist() == [10, 11, 12, 20, 21, 22, 12, 22, 30, 31, 32]
    assert g_lp.tolist() == [0, 0, -1.5, 0, 0, -2.5, 0, 0, 0, 0, -3.5]
    assert vcs.compact_trainable(lay["tok_loss_mask"]).tolist() == [2, 5, 10]


@pytest.mark.parametrize("name", ["tiny", "traj8_w3", "traj32_w3"])
def test_workloads(name):
    w = workloads.WORKLOADS[name]
    cu, img, txt = workloads.draw_steps(w)
    _check_layout(cu, img, txt, w.window, w.keep, w.seed)


@pytest.mark.parametrize("layout", list(workloads.COMPARISON_LAYOUTS))
def test_comparison_layouts(layout):
    window, keep = workloads.COMPARISON_LAYOUTS[layout]
    cu, img, txt = workloads.draw_steps(workloads.WORKLOADS["traj8_w3"])
    _check_layout(cu, img, txt, window, keep, 4)


@pytest.mark.parametrize("seed", range(4))
def test_random_with_empty_and_zero_counts(seed):
    rng = np.random.default_rng(seed + 50)
    T = rng.integers(0, 30, size=40)
    cu = np.concatenate([[0], np.cumsum(T)])
    img = rng.integers(0, 40, size=int(T.sum()))
    txt = rng.integers(0, 9, size=int(T.sum()))
    _check_layout(cu, img, txt, int(rng.integers(1, 5)), int(rng.integers(0, 4)), seed)


def test_compaction_many_chunks_and_capacity():
    vcs = _vcs()
    rng = np.random.default_rng(9)
    mask = (rng.random(1_000_003) < 0.3).astype(np.uint8)          # ~245 compaction chunks, ragged tail
    m = torch.from_numpy(mask).to(DEV)
    idx = vcs.compact_trainable(m).cpu().numpy()
    assert np.array_equal(idx, np.flatnonzero(mask))
    # too small an output: the first entries are written, the device reports the capacity
    with pytest.raises(vcs.VcsError) as e:
        vcs.compact_trainable(m, capacity=100)
    assert e.value.status == 3
    # no tokens / no trainable token
    assert vcs.compact_trainable(torch.zeros(0, dtype=torch.uint8, device=DEV)).numel() == 0
    assert vcs.compact_trainable(torch.zeros(5000, dtype=torch.uint8, device=DEV)).numel() == 0


def test_device_check_bad_gather_index():
    vcs = _vcs()
    ids = torch.arange(10, dtype=torch.int32, device=DEV)
    lp = torch.zeros(10, device=DEV)
    g = torch.tensor([0, 3, 10], dtype=torch.int32, device=DEV)       # 10 is out of range
    m = torch.ones(3, dtype=torch.uint8, device=DEV)
    with pytest.raises(vcs.VcsError) as e:
        vcs.stream_fields(ids, lp, g, m)
    assert e.value.status == 6


def test_loss_over_the_stream_fields():
    # the stream's logp (rollout log-probabilities) feeds the objective as old_logp
    from oracle import loss as oloss
    vcs = _vcs()
    w = workloads.WORKLOADS["traj8_w3"]
    cu, img, txt = workloads.draw_steps(w)
    lay = vcs.build_segments(torch.from_numpy(cu).to(DEV), torch.from_numpy(img).to(DEV),
                             torch.from_numpy(txt).to(DEV), w.window, w.keep)
    ntok = int(img.sum() + txt.sum())
    rng = np.random.default_rng(1)
    traj_lp = (-rng.random(ntok) * 4).astype(np.float32)
    ids = rng.integers(0, 1000, size=ntok).astype(np.int32)
    _, old = vcs.stream_fields(torch.from_numpy(ids).to(DEV), torch.from_numpy(traj_lp).to(DEV), lay["tok_gather"],
                               lay["tok_loss_mask"])
    logp = old + torch.randn(old.shape, generator=torch.Generator(DEV).manual_seed(0), device=DEV) * 0.3
    adv = torch.from_numpy(oloss.group_advantage(rng.random(w.num_traj), 4).astype(np.float32)).to(DEV)
    loss, g = vcs.grpo_loss(logp, old, logp, lay["tok_loss_mask"], lay["cu_seqlens"], lay["seg_traj"], adv)
    lo, go = oloss.grpo_loss_vec(logp.cpu().numpy(), old.cpu().numpy(), logp.cpu().numpy(),
                                 lay["tok_loss_mask"].cpu().numpy(), lay["cu_seqlens"].cpu().numpy(),
                                 lay["seg_traj"].cpu().numpy(), adv.cpu().numpy(), w.num_traj)
    assert float(loss.item()) == pytest.approx(lo, rel=1e-5, abs=1e-6)
    np.testing.assert_allclose(g.cpu().numpy(), go, rtol=1e-4, atol=1e-7)
