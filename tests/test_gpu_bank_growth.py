"""Paper-mode write keep-set on the device (Sec. 3.2, Eq. 8): K_w is computed
once from the object's seed mask (its first frame), dilated by D_w grid cells
and held fixed, so every commit adds the same |K_w| rows to the bank -- the
constant per-frame stride that bounds bank growth at O(T |K_w|) instead of
O(T mn)."""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2608_22526_gb300 import rs3, synth
from paper_2608_22526_gb300.pipeline import Pipeline
from tests._harness import to_dev, to_host

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("D_w", [12, 24])
def test_paper_kw_constant_stride_on_device(D_w):
    w = synth.scaled(synth.WORKLOADS["long_video"], frames=24)
    seq = synth.Sequence(w)
    ug = w.unit_group()
    p = rs3.default_params(rho=w.rho, r_s=w.r_s, c=w.c, union_mode=w.union_mode, D_w=D_w)
    seed = seq.masks(0)
    kw = torch.empty((w.U, w.mn), dtype=torch.uint8, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    rs3.rs3_write_keepset(to_dev(seed), to_dev(ug), w.U, w.m, w.n, p, kw, st)
    kw_np = to_host(kw)
    assert int(st.item()) == 0
    assert np.array_equal(kw_np, orc.write_keepset(seed, ug, w.m, w.n, D_w, union_mode=w.union_mode))
    n_kw = kw_np.reshape(w.U, -1).astype(np.int64).sum(axis=1)
    assert (n_kw > 0).all() and (n_kw < w.mn).all()      # a real prune, no fall-through here

    pipe = Pipeline(w, ring_cap=w.frames * w.mn, params=p)
    ob = orc.OracleBank(w.U, w.D, w.dtype, w.mn, w.n_cond, w.window, pipe.bank.ring_cap,
                        pipe.bank.max_frames, w.n_ptr)
    for t in range(w.frames):
        kn, vn = seq.kv_new(t)
        is_cond = int(t == 0 and w.n_cond > 0)
        pipe.commit(to_dev(kn), to_dev(vn), kw, is_cond)
        assert ob.commit(kn, vn, kw_np, is_cond) == [0] * w.U
        meta, fr = rs3.rs3_bank_read_meta(pipe.bank)
        ring = t if w.n_cond > 0 else t + 1                 # ring frames held after frame t
        for u in range(w.U):
            assert meta[u, 7] == (t + 1) * n_kw[u]          # constant stride: |K_w| rows per frame
            assert meta[u, 3] == ring
            assert [tuple(x) for x in fr[u, :ring]] == [(i * n_kw[u], n_kw[u]) for i in range(ring)]
    assert pipe.status_code() == 0
    ks, vs = to_host(pipe.bank.k_store), to_host(pipe.bank.v_store)
    for u in range(w.U):
        rows = ob.logical_rows(u)
        assert len(rows) == w.frames * n_kw[u]
        assert np.array_equal(ks[u][rows], ob.K[u][rows]) and np.array_equal(vs[u][rows], ob.V[u][rows])
