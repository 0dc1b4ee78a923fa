"""GPU edge cases through the C ABI: degenerate sizes, the write keep-set,
status-word errors, resets, the largest grid."""
import dataclasses

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2608_22526_gb300 import rs3, synth
from paper_2608_22526_gb300.pipeline import Pipeline
from tests._harness import check_readout, Report, to_dev, to_host, widen

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS


def _bf16(rng, shape):
    return synth.f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32))


def test_empty_bank_reads_zero_and_keeps_residual():
    w = synth.scaled(W["sam2_1obj"], frames=2)
    pipe = Pipeline(w)
    seq = synth.Sequence(w)
    z = seq.z(1)
    pipe.select(to_dev(z), to_dev(seq.masks(0)))
    res = to_dev(z[w.unit_group()])
    before = to_host(res).copy()
    pipe.readout(to_dev(z), res, res)
    torch.cuda.synchronize()
    # nothing was committed: A = 0, so out == residual + 0 exactly
    assert np.array_equal(to_host(res), before)
    out = torch.empty_like(res)
    pipe.readout(to_dev(z), None, out)
    assert np.all(widen(to_host(out), "bf16") == 0.0)
    assert pipe.status_code() == 0


def test_rho_zero_selects_nothing():
    w = dataclasses.replace(synth.scaled(W["sam2_8obj"], frames=3), rho=0.0)
    pipe = Pipeline(w)
    assert pipe.k_max == 0
    seq = synth.Sequence(w)
    kn, vn = seq.kv_new(0)
    pipe.commit(to_dev(kn), to_dev(vn), to_dev(seq.masks(0)), 1)
    z = seq.z(1)
    pipe.select(to_dev(z), to_dev(seq.masks(0)))
    assert np.all(to_host(pipe.count) == 0)
    res = to_dev(z[w.unit_group()])
    before = to_host(res).copy()
    pipe.readout(to_dev(z), res, res)
    assert np.array_equal(to_host(res), before)
    assert pipe.status_code() == 0


def test_largest_grid_selection_bitexact():
    """mn = 16384 (the largest supported grid), 2 groups in union mode."""
    w = synth.Workload("big", 9, 128, 128, 1, 64, "bf16", 2, 2, 2, 0.05, 0.3, 1, 6, 0,
                       union_mode=1)
    seq = synth.Sequence(w)
    pipe = Pipeline(w)
    z = seq.z(1)
    prev = seq.masks(0)
    pipe.select(to_dev(z), to_dev(prev))
    track = np.zeros((w.U, 6), np.int32)
    sel = orc.select(z, "bf16", prev, w.unit_group(), track, w.m, w.n, w.rho, w.r_s, w.c, 1)
    cnt = to_host(pipe.count)
    assert np.array_equal(cnt, sel.count)
    idx = to_host(pipe.idx)
    for u in range(w.U):
        assert np.array_equal(idx[u, : cnt[u]], sel.keep(u))


def test_bbox_mode_seed_prior():
    """Eq. 1: the seed prior is the dilated tight box of the seed mask."""
    w = synth.scaled(W["sam2_8obj"], frames=2)
    p = rs3.default_params(rho=w.rho, r_s=w.r_s, c=w.c, union_mode=0, bbox_mode=1)
    pipe = Pipeline(w, params=p)
    seq = synth.Sequence(w)
    z, prev = seq.z(1), seq.masks(0)
    pipe.select(to_dev(z), to_dev(prev))
    track = np.zeros((w.U, 6), np.int32)
    sel = orc.select(z, "bf16", prev, w.unit_group(), track, w.m, w.n, w.rho, w.r_s, w.c, 0,
                     bbox_mode=1)
    cnt = to_host(pipe.count)
    assert np.array_equal(cnt, sel.count)
    for u in range(w.U):
        assert np.array_equal(to_host(pipe.idx)[u, : cnt[u]], sel.keep(u))


@pytest.mark.parametrize("union_mode", [0, 1])
@pytest.mark.parametrize("D_w", [0, 3, 24])
def test_write_keepset_matches_oracle(union_mode, D_w):
    rng = np.random.default_rng(5 + D_w)
    m = n = 40
    U = 6
    ug = np.array([0, 0, 1, 1, 1, 2], np.int32)
    seeds = np.zeros((U, m * n), np.uint8)
    for u in range(U):
        y, x = rng.integers(0, 34, size=2)
        h, wd = rng.integers(1, 7, size=2)
        seeds[u].reshape(m, n)[y:y + h, x:x + wd] = 1
    seeds[5] = 0
    seeds[5, : int(0.96 * m * n)] = 1          # > 95%: falls through to the full grid
    p = rs3.default_params(D_w=D_w, union_mode=union_mode)
    kw = torch.empty((U, m * n), dtype=torch.uint8, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    rs3.rs3_write_keepset(to_dev(seeds), to_dev(ug), U, m, n, p, kw, st)
    ref = orc.write_keepset(seeds, ug, m, n, D_w, union_mode=union_mode)
    assert np.array_equal(to_host(kw), ref)
    assert int(st.item()) == 0


def test_bank_overflow_latches_capacity_and_drops_whole_frame():
    w = synth.Workload("ovf", 8, 16, 16, 1, 64, "bf16", 1, 2, 4, 0.1, 0.2, 0, -1, 0)
    pipe = Pipeline(w, ring_cap=300)
    ones = torch.ones((w.U, w.mn), dtype=torch.uint8, device="cuda")
    rng = np.random.default_rng(1)
    kn = to_dev(_bf16(rng, (w.U, w.mn, w.D)))
    pipe.commit(kn, kn, ones, 0)                    # 256 of 300 rows
    meta0, _ = rs3.rs3_bank_read_meta(pipe.bank)
    assert pipe.status_code() == 0 and list(meta0[:, 7]) == [256, 256]
    pipe.commit(kn, kn, ones, 0)                    # 512 > 300: dropped
    meta1, _ = rs3.rs3_bank_read_meta(pipe.bank)
    assert pipe.status_code() == rs3.RS3_ECAPACITY
    assert np.array_equal(meta0, meta1)
    # a cond commit into a bank without pinned frames is refused on the host
    with pytest.raises(rs3.RS3Error):
        pipe.commit(kn, kn, ones, 1)


def test_bad_group_id_latches_einval():
    w = synth.scaled(W["sam2_8obj"], frames=2, units_per_group=2)
    pipe = Pipeline(w)
    pipe.unit_group[1] = 7                          # out of [0, G)
    seq = synth.Sequence(w)
    pipe.select(to_dev(seq.z(1)), to_dev(seq.masks(0)))
    assert pipe.status_code() == rs3.RS3_EINVAL
    assert int(to_host(pipe.count)[1]) == 0


def test_count_above_kmax_latches_einval():
    w = synth.scaled(W["sam2_1obj"], frames=2)
    pipe = Pipeline(w)
    seq = synth.Sequence(w)
    kn, vn = seq.kv_new(0)
    pipe.commit(to_dev(kn), to_dev(vn), to_dev(seq.masks(0)), 1)
    z = seq.z(1)
    pipe.select(to_dev(z), to_dev(seq.masks(0)))
    pipe.count.fill_(pipe.k_max + 5)
    res = to_dev(z[w.unit_group()])
    pipe.readout(to_dev(z), res, res)
    torch.cuda.synchronize()
    assert pipe.status_code() == rs3.RS3_EINVAL


def test_reset_empties_banks_and_restarts():
    w = synth.scaled(W["sam2_8obj"], frames=3, units_per_group=3)
    pipe = Pipeline(w)
    seq = synth.Sequence(w)
    for t in range(3):
        kn, vn = seq.kv_new(t)
        pipe.commit(to_dev(kn), to_dev(vn), to_dev(seq.masks(t)), int(t == 0))
    meta, _ = rs3.rs3_bank_read_meta(pipe.bank)
    assert np.all(meta[:, 7] > 0)
    rs3.rs3_bank_reset(pipe.bank, 1)
    meta, _ = rs3.rs3_bank_read_meta(pipe.bank)
    assert meta[1, 7] == 0 and meta[0, 7] > 0 and meta[2, 7] > 0
    rs3.rs3_bank_reset(pipe.bank, -1)
    meta, _ = rs3.rs3_bank_read_meta(pipe.bank)
    assert np.all(meta == 0)


def test_ragged_counts_across_units_and_tiles():
    """Units with very different keep-set sizes (1 .. k_max), banks crossing
    the ring end: every row of every unit against the oracle."""
    rng = np.random.default_rng(9)
    w = synth.Workload("ragged", 10, 48, 48, 1, 128, "bf16", 1, 5, 12, 0.01, 0.5, 1, 3, 5)
    from tests._harness import run_lockstep
    run_lockstep(w, check_frames={1, 5, 11}, residual_mode="inplace")


def test_readout_wait_limit_runs_out_and_the_context_stays_usable():
    """Every wait of the tensor-core readout has a time limit.  With the limit
    at 0 ns the waits give up at once: the launch returns, latches
    RS3_ETIMEOUT, and frees its tensor memory (the following launches on
    every SM allocate it again); later calls with the default limit are
    correct against the oracle."""
    from tests._harness import check_fused
    w = synth.scaled(W["sam2_1obj"], frames=3)
    pipe = Pipeline(w)
    seq = synth.Sequence(w)
    kn, vn = seq.kv_new(0)
    pipe.commit(to_dev(kn), to_dev(vn), to_dev(seq.masks(0)), 1)
    kp, vp = seq.pointers()
    pipe.set_pointers(to_dev(kp), to_dev(vp))
    z = seq.z(1)
    pipe.select(to_dev(z), to_dev(seq.masks(0)))
    torch.cuda.synchronize()
    assert rs3.rs3_get_wait_limit_ns() == 10 ** 9
    x = z[w.unit_group()]
    rs3.rs3_set_wait_limit_ns(0)
    try:
        for _ in range(2):
            res = to_dev(x)
            pipe.readout(to_dev(z), res, res)
        torch.cuda.synchronize()
    finally:
        rs3.rs3_set_wait_limit_ns(10 ** 9)
    assert pipe.status_code() == rs3.RS3_ETIMEOUT
    pipe.status.zero_()
    # the oracle's view of the bank and keep-set
    ob = orc.OracleBank(w.U, w.D, w.dtype, w.mn, w.n_cond, w.window, pipe.bank.ring_cap,
                        pipe.bank.max_frames, w.n_ptr)
    ob.commit(kn, vn, seq.masks(0), 1)
    ob.set_pointers(kp, vp)
    track = np.zeros((w.U, 6), np.int32)
    sel = orc.select(z, w.dtype, seq.masks(0), w.unit_group(), track, w.m, w.n, w.rho, w.r_s, w.c,
                     w.union_mode)
    keep = sel.keep(0)
    K, V = ob.kv(0)
    A = orc.readout(z[0], w.dtype, w.H, w.d, keep, K, V, w.dtype, threads=8)
    rep = Report()
    for _ in range(3):
        res = to_dev(x)
        pipe.readout(to_dev(z), res, res)
        out = to_host(res)
        check_fused(w.dtype, out[0][keep], x[0][keep], A, rep, "after the timeout")
        others = np.setdiff1d(np.arange(w.mn), keep)
        assert np.array_equal(out[0][others], x[0][others])
    assert pipe.status_code() == 0
