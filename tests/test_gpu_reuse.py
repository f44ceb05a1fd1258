"""GPU parity of prefix reuse: vcs_shared_prefix against the oracle's common-prefix
definition (bit-exact), and vcs_attn_fwd_reuse against vcs_attn_fwd (bit for bit: a
reused row is the same computation on the same tokens) and against the fp64 oracle on
sampled rows; edge cases and the device check on an impossible shared length."""
import numpy as np
import pytest
import torch

from oracle import attention as oatt
from oracle import reuse as oreuse
from paper_2607_11185_gb300 import workloads
from tests.gpu_cases import random_steps

pytestmark = pytest.mark.gpu


def _vcs():
    from paper_2607_11185_gb300 import vcs
    return vcs


def _layout(cu, img, txt, window, keep):
    vcs = _vcs()
    return vcs.build_segments(*(torch.from_numpy(np.asarray(x, np.int32)).cuda() for x in (cu, img, txt)), window,
                              keep)


def _check_prefix(lay):
    vcs = _vcs()
    sp = vcs.shared_prefix(lay["cu_seqlens"], lay["seg_traj"], lay["tok_gather"])
    want = oreuse.shared_prefix(lay["cu_seqlens"].cpu().numpy(), lay["seg_traj"].cpu().numpy(),
                                lay["tok_gather"].cpu().numpy())
    assert np.array_equal(sp.cpu().numpy(), want)
    return sp


@pytest.mark.parametrize("name", ["tiny", "traj8_w3", "traj32_w3", "traj16x50_w8"])
def test_shared_prefix_workloads(name):
    w = workloads.WORKLOADS[name]
    _check_prefix(_layout(*workloads.draw_steps(w), w.window, w.keep))


@pytest.mark.parametrize("layout", list(workloads.COMPARISON_LAYOUTS))
def test_shared_prefix_layouts(layout):
    window, keep = workloads.COMPARISON_LAYOUTS[layout]
    _check_prefix(_layout(*workloads.draw_steps(workloads.WORKLOADS["traj8_w3"]), window, keep))


@pytest.mark.parametrize("seed", range(4))
def test_shared_prefix_random_with_zero_counts(seed):
    cu, img, txt = random_steps(seed + 70)
    _check_prefix(_layout(cu, img, txt, int(seed % 3 + 1), int(seed % 2)))


def _fwd_pair(name, window=None, keep=None, hq=None, hkv=None, d=None):
    vcs = _vcs()
    w = workloads.WORKLOADS[name]
    cu, img, txt = workloads.draw_steps(w)
    lay = _layout(cu, img, txt, w.window if window is None else window, w.keep if keep is None else keep)
    ntraj = workloads.trajectory_tokens(img, txt)
    qt, kt, vt, _ = workloads.draw_dense(w.seed, ntraj, hq or w.hq, hkv or w.hkv, d or w.d, device="cuda")
    q, k, v = vcs.gather(qt, kt, vt, lay["tok_gather"])
    sp = _check_prefix(lay)
    o, lse = vcs.attn_fwd(q, k, v, lay["cu_seqlens"], lay["max_seqlen"])
    o_r, lse_r = vcs.attn_fwd_reuse(q, k, v, lay["cu_seqlens"], sp, lay["max_seqlen"])
    return lay, sp, (q, k, v), (o, lse), (o_r, lse_r)


@pytest.mark.parametrize("name,window,keep", [("tiny", None, None), ("traj8_w3", None, None), ("traj8_w3", 1, 0),
                                               ("traj8_w3", 2, 1), ("traj32_w3", None, None)])
def test_fwd_reuse_equals_full_forward(name, window, keep):
    lay, sp, _, (o, lse), (o_r, lse_r) = _fwd_pair(name, window, keep)
    if name != "tiny":                      # the tiny workload's segments share no prefix
        assert (sp.cpu().numpy() >= 256).any()  # some pairs are reused
    assert torch.equal(o_r, o)
    assert torch.equal(lse_r, lse)


def test_fwd_reuse_small_heads_vs_oracle():
    # d = 64 with 4:2 heads on a step-wise layout; rows of reused and computed pairs vs fp64
    lay, sp, (q, k, v), _, (o_r, lse_r) = _fwd_pair("traj8_w3", 1, 0, hq=4, hkv=2, d=64)
    cus = lay["cu_seqlens"].cpu().numpy()
    spn = sp.cpu().numpy()
    s = int(np.argmax(spn))
    b, e = int(cus[s]), int(cus[s + 1])
    rows = sorted({0, 255, int(spn[s]) - 1, int(spn[s]), e - b - 1})
    rows = [r for r in rows if 0 <= r < e - b]
    ro, rl = oatt.rows_fwd(q.cpu(), k.cpu(), v.cpu(), (b, e), list(range(4)), rows)
    got = o_r[[b + r for r in rows]].float().cpu().numpy()
    assert np.abs(got - ro).max() <= 2e-2
    assert np.abs(lse_r[:, [b + r for r in rows]].cpu().numpy() - rl).max() <= 2e-3


def test_device_check_and_errors():
    vcs = _vcs()
    q, k, v, _ = workloads.draw_dense(3, 600, 2, 1, 64, device="cuda")
    cu = torch.tensor([0, 300, 600], dtype=torch.int32, device="cuda")
    bad = torch.tensor([0, 400], dtype=torch.int32, device="cuda")        # longer than either segment
    with pytest.raises(vcs.VcsError) as e:
        vcs.attn_fwd_reuse(q, k, v, cu, bad, 300)
    assert e.value.status == 6
    bad0 = torch.tensor([256, 0], dtype=torch.int32, device="cuda")       # segment 0 has no predecessor
    with pytest.raises(vcs.VcsError) as e:
        vcs.attn_fwd_reuse(q, k, v, cu, bad0, 300)
    assert e.value.status == 6
    o = torch.empty_like(q)
    lse = torch.empty((2, 600), dtype=torch.float32, device="cuda")
    nb = vcs.vcs_attn_fwd_workspace_size(2, 600, 300, 2, 1, 64)
    ws = torch.zeros(nb, dtype=torch.uint8, device="cuda")
    assert vcs.vcs_attn_fwd_reuse(q, k, v, cu, None, 2, 600, 300, 2, 1, 64, 0.0, o, lse, ws, nb) == 1
    # no shared prefix: same as the plain forward
    zero = torch.zeros(2, dtype=torch.int32, device="cuda")
    o1, l1 = vcs.attn_fwd_reuse(q, k, v, cu, zero, 300)
    o2, l2 = vcs.attn_fwd(q, k, v, cu, 300)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    # shared_prefix on an empty layout
    empty = vcs.shared_prefix(torch.zeros(1, dtype=torch.int32, device="cuda"),
                              torch.zeros(0, dtype=torch.int32, device="cuda"),
                              torch.zeros(0, dtype=torch.int32, device="cuda"))
    assert empty.numel() == 0
