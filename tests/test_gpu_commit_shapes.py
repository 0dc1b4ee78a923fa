"""Bank commit (Sec. 3.2, Eq. 8; Algorithm 1's sparse write) on shapes the
benchmark workloads do not reach.  The grids are odd, so a unit's mask row is
not 16-byte aligned and its last chunk is ragged.  The rows are 1 KB (2 heads
of 256 bf16), so each lane copies more than one 16-byte piece per row.
Launches both small (64-cell chunks) and large (128-cell chunks), through
ring wrap and eviction, with keys stored plain and rotated.  Every bank row
and counter is checked against the oracle's bank."""
import numpy as np
import pytest

from oracle import oracle as orc
from paper_2608_22526_gb300 import rs3, synth
from paper_2608_22526_gb300.pipeline import Pipeline
from tests._harness import to_dev, to_host, widen

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("m,n,U,frames,rope", [(37, 45, 2, 16, False), (37, 45, 2, 16, True),
                                                (69, 71, 8, 12, False)])
def test_commit_odd_grid_wide_rows_wrap(m, n, U, frames, rope):
    # 37 x 45 x 2 units: 64-cell chunks; 69 x 71 x 8 units: 128-cell chunks
    # on a 152-SM part.  1 conditioning frame, a window of 3 ring frames,
    # masks covering 20-50%.
    w = synth.Workload("commit_shape", 11, m, n, 2, 256, "bf16", 1, U, frames, 0.2, 0.5, 1, 3, 0)
    seq = synth.Sequence(w)
    pipe = Pipeline(w)
    ob = orc.OracleBank(w.U, w.D, w.dtype, w.mn, w.n_cond, w.window, pipe.bank.ring_cap,
                        pipe.bank.max_frames, w.n_ptr)
    tab = seq.rope_table() if rope else None
    tab_dev = to_dev(tab) if rope else None
    for t in range(w.frames):
        kn, vn = seq.kv_new(t)
        mask = seq.masks(t)
        is_cond = int(t == 0)
        pipe.commit(to_dev(kn), to_dev(vn), to_dev(mask), is_cond, rope=tab_dev)
        assert ob.commit(kn, vn, mask, is_cond, rope=tab) == [0] * w.U
    assert pipe.status_code() == 0

    meta, fr = rs3.rs3_bank_read_meta(pipe.bank)
    for u in range(w.U):
        assert meta[u, 0] == ob.state[u, 0] and meta[u, 1] == ob.state[u, 1]
        assert meta[u, 2] == ob.state[u, 2] and meta[u, 3] == ob.state[u, 3]
        assert meta[u, 5] == ob.state[u, 5] and meta[u, 7] == ob.length(u)
        assert [tuple(x) for x in fr[u, : meta[u, 3]]] == ob.frames(u)
    # the ring wrapped: some unit's tail (a logical position) passed its capacity
    assert (meta[:, 1] > pipe.bank.ring_cap).any()

    ks, vs = to_host(pipe.bank.k_store), to_host(pipe.bank.v_store)
    for u in range(w.U):
        rows = ob.logical_rows(u)
        assert np.array_equal(vs[u][rows], ob.V[u][rows]), f"V rows of unit {u}"
        if not rope:
            assert np.array_equal(ks[u][rows], ob.K[u][rows]), f"K rows of unit {u}"
        else:
            # fp32 rotation on the device, fp64 in the oracle, one rounding to
            # bf16 on each side: one unit in the last place apart at most, plus
            # the fp32 error of k0 cos - k1 sin where it cancels
            g = widen(ks[u][rows], "bf16")
            r = widen(ob.K[u][rows], "bf16")
            tol = 2.0 ** -7 * np.abs(r) + 2.0 ** -20 * max(float(np.abs(r).max()), 1e-30)
            assert (np.abs(g - r) <= tol).all(), f"K rows of unit {u}"
            assert (ks[u][rows] == ob.K[u][rows]).mean() > 0.99, f"K rows of unit {u}"
