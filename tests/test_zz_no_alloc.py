"""The allocation-free selection entry point (rs3_select_queries_noalloc),
for callers that cannot obtain a device workspace, must give exactly what the
regular entry point gives.  Checked through the C ABI on two consecutive
frames, so the second call runs on scratch that still holds the first call's
contents.  This file is collected last on purpose."""
import numpy as np
import pytest
import torch

from paper_2608_22526_gb300 import rs3, synth

pytestmark = pytest.mark.gpu


def _dev(x):
    if x.dtype == np.uint16:
        return torch.from_numpy(x.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


@pytest.mark.parametrize("name,union_mode", [("sam2_8obj", 0), ("multistream", 1)])
def test_noalloc_selection_matches_workspace_selection(name, union_mode):
    w = synth.WORKLOADS[name]
    seq = synth.Sequence(w)
    p = rs3.default_params(rho=w.rho, r_s=w.r_s, c=w.c, union_mode=union_mode)
    k = rs3.rs3_kmax(p.rho, w.mn)
    ug = torch.tensor(w.unit_group(), dtype=torch.int32, device="cuda")
    ws = torch.empty(rs3.rs3_select_workspace_bytes(w.G, w.U, w.m, w.n), dtype=torch.uint8,
                     device="cuda")
    track_a = torch.zeros((w.U, 6), dtype=torch.int32, device="cuda")
    track_b = torch.zeros_like(track_a)
    st_a = torch.zeros(1, dtype=torch.int32, device="cuda")
    st_b = torch.zeros_like(st_a)
    for t in (1, 2):                       # two calls in a row
        z = _dev(seq.z(t))
        prev = _dev(seq.masks(t - 1))
        idx_a = torch.full((w.U, k), -7, dtype=torch.int32, device="cuda")
        idx_b = torch.full_like(idx_a, -7)
        cnt_a = torch.full((w.U,), -7, dtype=torch.int32, device="cuda")
        cnt_b = torch.full_like(cnt_a, -7)
        rs3.rs3_select_queries(z, w.dtype, w.G, w.m, w.n, w.C, prev, ug, w.U, track_a, p, idx_a,
                               cnt_a, ws, st_a)
        rs3.rs3_select_queries_noalloc(z, w.dtype, w.G, w.m, w.n, w.C, prev, ug, w.U, track_b, p,
                                       idx_b, cnt_b, st_b)
        torch.cuda.synchronize()
        ca, cb = cnt_a.cpu().numpy(), cnt_b.cpu().numpy()
        assert np.array_equal(ca, cb)
        assert ca.min() >= 0 and ca.max() <= k and ca.sum() > 0
        ia, ib = idx_a.cpu().numpy(), idx_b.cpu().numpy()
        for u in range(w.U):
            assert np.array_equal(ia[u, : ca[u]], ib[u, : cb[u]])
        assert torch.equal(track_a, track_b)
        assert int(st_a.item()) == 0 and int(st_b.item()) == 0


def test_noalloc_rejects_sizes_beyond_its_scratch():
    w = synth.WORKLOADS["multistream"]
    p = rs3.default_params()
    G, U, m, n = 512, 512, 128, 128          # far more than 8 MiB of scratch
    assert rs3.rs3_select_workspace_bytes(G, U, m, n) > (8 << 20)
    one = torch.zeros(16, dtype=torch.int32, device="cuda")
    with pytest.raises(rs3.RS3Error) as e:
        rs3.rs3_select_queries_noalloc(one, "bf16", G, m, n, 256, one, one, U, one, p, one, one, one)
    assert e.value.code == rs3.RS3_ECAPACITY
