"""GPU parity: the CUDA path through the C ABI against the CPU oracle on the
same seeded inputs.  Keep-sets, counts, tracker state, bank counters and bank
rows bit for bit; readouts within max-abs 2e-2 / mean-abs 2e-3 (bf16) or 1e-4
relative (fp32); unselected cells bit-identical to the residual."""
import numpy as np
import pytest
import torch

from paper_2608_22526_gb300 import synth
from tests._harness import run_lockstep

pytestmark = pytest.mark.gpu

W = synth.WORKLOADS


@pytest.mark.parametrize("residual_mode", ["inplace", "none", "outofplace"])
@pytest.mark.parametrize("rope", [False, True])
def test_tiny_fp32_single_step(residual_mode, rope):
    rep = run_lockstep(W["tiny_fp32"], check_frames={0}, rope=rope, residual_mode=residual_mode)
    assert rep.frames_checked == 1 and rep.rows_checked > 0


@pytest.mark.parametrize("residual_mode", ["inplace", "none"])
def test_sam2_single_object_small(residual_mode):
    w = synth.scaled(W["sam2_1obj"], frames=12)
    rep = run_lockstep(w, check_frames={1, 2, 7, 8, 11}, residual_mode=residual_mode)
    assert rep.frames_checked == 5


def test_sam2_single_object_rope_out_of_place():
    w = synth.scaled(W["sam2_1obj"], frames=9)
    run_lockstep(w, check_frames={1, 8}, rope=True, residual_mode="outofplace")


def test_sam2_single_object_full_sequence():
    """The benchmark workload: all 60 frames, every kept row at six frames."""
    rep = run_lockstep(W["sam2_1obj"], check_frames={1, 2, 7, 8, 30, 59}, threads=16)
    assert rep.select_frames == 59


def test_multi_object_full():
    """8 objects on one grid, per-object selections and banks, 100 frames."""
    run_lockstep(W["sam2_8obj"], check_frames={1, 50, 99}, rows_per_unit=96, threads=16)


def test_multi_object_union_mode():
    """The paper's Eq. 2 reading: one prior per stream, the union of objects."""
    import dataclasses
    w = dataclasses.replace(synth.scaled(W["sam2_8obj"], frames=10, units_per_group=4),
                            union_mode=1)
    run_lockstep(w, check_frames={1, 9}, rows_per_unit=64)


def test_multistream_full_size():
    """16 streams x 3 objects, 96x96 grid, 4 heads x 64: full per-frame size,
    enough frames for the banks to reach their steady window."""
    run_lockstep(W["multistream"], frames=24, check_frames={1, 12, 23}, rows_per_unit=24,
                 threads=16)


@pytest.mark.parametrize("name", ["sam2_1obj", "multistream"])
def test_rope_on_queries_and_keys(name):
    """Eq. 7 on both sides: queries rotated by their cell in the readout, keys
    stored rotated by their cell at commit (pointer rows unrotated); the bank
    holds the oracle's rotated keys to one bf16 unit and the readout matches
    the oracle's attention over them."""
    w = synth.scaled(W[name], frames=10)
    run_lockstep(w, check_frames={1, 9}, rope=True, rope_keys=True, rows_per_unit=64)


def test_multistream_rope_small():
    w = synth.scaled(W["multistream"], frames=8, G=2)
    run_lockstep(w, check_frames={1, 7}, rope=True, rows_per_unit=64)


@pytest.mark.slow
def test_long_video_full():
    """1000 frames, unbounded write-pruned bank (~600k keys at the end)."""
    run_lockstep(W["long_video"], check_frames={1, 500, 999}, rows_per_unit=24, threads=16)


def test_long_video_split_kv_small():
    w = synth.scaled(W["long_video"], frames=80)
    run_lockstep(w, check_frames={1, 40, 79}, rows_per_unit=64)


def test_long_bank_single_query_tile_split_across_many_ctas():
    """Few kept queries (one 128-row tile) over a long bank: the one group is
    cut into more than 32 pieces whose partials the combine merges."""
    import dataclasses
    w = dataclasses.replace(synth.scaled(W["long_video"], frames=80), rho=0.03)
    run_lockstep(w, check_frames={1, 79}, rows_per_unit=64)


def test_dense_rho1_identity():
    """rho = 1, full prior, unpruned bank: every cell is selected in order and
    the readout is dense memory attention (Sec. 3.1, after Eq. 7)."""
    w = synth.scaled(W["sam2_1obj"], frames=4)
    rep = run_lockstep(w, check_frames={1, 3}, dense=True, rows_per_unit=256)
    assert rep.frames_checked == 2


def test_disappearing_objects_fallback():
    """Objects vanish for 20 frames: the streak-counted box prior (Eq. 4)."""
    w = synth.scaled(W["sam2_8obj"], frames=40)
    vanish = {0: [range(5, 25)], 3: [range(2, 39)], 5: [range(10, 12), range(20, 30)]}
    run_lockstep(w, check_frames={6, 26, 39}, rows_per_unit=32, vanish=vanish)
