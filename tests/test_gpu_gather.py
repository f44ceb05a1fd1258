"""GPU gather vs the oracle: bit-exact packed rows."""
import numpy as np
import pytest
import torch

from oracle import gather as ogather
from oracle import segments as oseg
from paper_2607_11185_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["tiny", "traj8_w3"])
def test_gather_matches_oracle(name):
    from paper_2607_11185_gb300 import vcs
    w = workloads.WORKLOADS[name]
    cu, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu, img, txt, w.window, w.keep)
    ntraj = workloads.trajectory_tokens(img, txt)
    q, k, v = workloads.draw_traj_qkv(w, ntraj, device="cuda")
    g = torch.from_numpy(lay["tok_gather"]).cuda()
    qs, ks, vs = vcs.gather(q, k, v, g)
    for src, got in ((q, qs), (k, ks), (v, vs)):
        ref = ogather.gather_rows(src.cpu(), lay["tok_gather"])
        assert torch.equal(got.cpu(), ref)


def test_gather_full_size_sampled_rows():
    from paper_2607_11185_gb300 import vcs
    w = workloads.WORKLOADS["traj32_w3"]
    cu, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu, img, txt, w.window, w.keep)
    ntraj = workloads.trajectory_tokens(img, txt)
    q, k, v = workloads.draw_traj_qkv(w, ntraj, device="cuda")
    g = torch.from_numpy(lay["tok_gather"]).cuda()
    qs, ks, vs = vcs.gather(q, k, v, g)
    rows = np.random.default_rng(0).integers(0, len(lay["tok_gather"]), size=2000)
    rows_t = torch.from_numpy(rows).cuda()
    src = torch.from_numpy(lay["tok_gather"][rows].astype(np.int64)).cuda()
    assert torch.equal(qs[rows_t], q[src]) and torch.equal(ks[rows_t], k[src]) and torch.equal(vs[rows_t], v[src])


def test_gather_q_only_and_odd_row_sizes():
    from paper_2607_11185_gb300 import vcs
    q = torch.randn(50, 3, 8, device="cuda").to(torch.bfloat16)   # 48-byte rows
    g = torch.tensor([5, 6, 7, 0, 49, 49, 13], dtype=torch.int32, device="cuda")
    out = torch.empty(7, 3, 8, dtype=torch.bfloat16, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert vcs.vcs_gather(q, None, None, 50, g, 7, 3, 0, 8, out, None, None, st) == 0
    torch.cuda.synchronize()
    assert st.item() == 0 and torch.equal(out, q[g.long()])


def test_gather_out_of_range_index_reported():
    from paper_2607_11185_gb300 import vcs
    q = torch.randn(10, 2, 64, device="cuda").to(torch.bfloat16)
    g = torch.tensor([1, 10, 3, -1], dtype=torch.int32, device="cuda")
    out = torch.zeros(4, 2, 64, dtype=torch.bfloat16, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert vcs.vcs_gather(q, None, None, 10, g, 4, 2, 0, 64, out, None, None, st) == 0
    torch.cuda.synchronize()
    assert st.item() == 6
    assert torch.equal(out[0], q[1]) and torch.equal(out[2], q[3])
    assert torch.all(out[1] == 0) and torch.all(out[3] == 0)


def test_gather_long_horizon_chunk_sampled_rows():
    """The long-horizon workload's first benchmark chunk (40 query / 8 kv heads: 10 KB Q rows,
    2 KB K and V rows), built and gathered on the GPU from the chunk's own trajectory rows as
    the benchmark runs it: the chunk's gather map bit-exact against the oracle's, and 4,096
    sampled rows of Q, K and V (plus the first and last) bit-exact against the oracle's
    gather."""
    import dataclasses
    from paper_2607_11185_gb300 import vcs
    from tests.gpu_cases import bench_chunks
    w = workloads.WORKLOADS["traj16x50_w8"]
    cu, img, txt = workloads.draw_steps(w)
    lay = oseg.build(cu, img, txt, w.window, w.keep)
    s0, s1 = bench_chunks(w, lay, len(cu) - 1)[0]
    b1 = int(lay["seg_traj"][s1 - 1]) + 1                     # the chunk's trajectories: 0 .. b1-1
    g1 = int(cu[b1])
    ttok = workloads.trajectory_tokens(img[:g1], txt[:g1])    # its trajectory rows: 0 .. ttok-1
    t1 = int(lay["cu_seqlens"][s1])
    glay = vcs.build_segments(*(torch.from_numpy(np.ascontiguousarray(x, np.int32)).cuda()
                                for x in (cu[:b1 + 1], img[:g1], txt[:g1])), w.window, w.keep)
    want_map = lay["tok_gather"][:t1]
    assert np.array_equal(glay["tok_gather"].cpu().numpy(), want_map)
    q, k, v = workloads.draw_traj_qkv(dataclasses.replace(w, num_traj=b1), ttok, device="cuda")
    qs, ks, vs = vcs.gather(q, k, v, glay["tok_gather"])
    rng = np.random.default_rng(55)
    rows = np.concatenate([[0, t1 - 1], rng.integers(0, t1, size=4096)])
    rows_t = torch.from_numpy(rows).cuda()
    for src, got in ((q, qs), (k, ks), (v, vs)):
        ref = ogather.gather_rows(src.cpu(), want_map[rows])
        assert torch.equal(got[rows_t].cpu(), ref)
