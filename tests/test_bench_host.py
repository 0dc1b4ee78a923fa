"""Host-side pieces of bench.py that need no GPU: the algorithmic work a
frame is credited with, the key that ties a stored ncu traffic figure to the
readout sources, and the config string of every workload."""
import os
import shutil
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_22526_gb300 import synth  # noqa: E402


def test_frame_work_closed_form():
    w = synth.WORKLOADS["sam2_8obj"]
    counts = [1228, 600, 0, 5, 1228, 1000, 1, 300]
    banks = [5000, 4000, 7000, 0, 100, 6000, 28672, 16]
    kw = [800, 0, 1600, 4096, 10, 20, 30, 40]
    flops, cbytes, sbytes = bench.frame_work(w, counts, banks, kw)
    # Eq. 6 per unit: q~ K^T and P V, each 2 |K_r| N d flops per head
    assert flops == sum(4.0 * c * n * w.H * w.d for c, n in zip(counts, banks))
    # commit: every unit's mask, K and V rows read and written (bf16)
    assert cbytes == w.U * w.mn + sum(4 * L * w.D * 2 for L in kw)
    # selection: the group's grid z, each unit's previous mask, the keep-set
    # indices and counts written, the tracker state (6 int32) read and written
    assert sbytes == w.G * w.mn * w.D * 2 + w.U * w.mn + 4 * sum(counts) + 4 * w.U + 2 * 6 * 4 * w.U


def test_traffic_key_ignores_comments_not_code(tmp_path, monkeypatch):
    src = os.path.join(ROOT, "paper_2608_22526_gb300", "csrc")
    dst = tmp_path / "paper_2608_22526_gb300" / "csrc"
    dst.mkdir(parents=True)
    for f in ("rs3_readout.cu", "rs3_readout_tc.cu", "rs3_readout_common.cuh", "rs3_tc_ptx.cuh"):
        shutil.copy(os.path.join(src, f), dst / f)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.readout_source_hash()
    p = dst / "rs3_readout.cu"
    text = p.read_text()
    p.write_text("// a new comment line\n/* and a block\n   comment */\n" + text.replace("\n", "\n\n", 3))
    assert bench.readout_source_hash() == h0
    p.write_text(text.replace("a->plan_ov = p.kind == 1 ? 12 : 1;", "a->plan_ov = p.kind == 1 ? 13 : 1;"))
    assert bench.readout_source_hash() != h0


def test_traffic_record_is_used_only_with_its_sources(tmp_path, monkeypatch):
    """A stored DRAM-traffic figure is reported only while the readout
    sources hash to the key it was stored with; otherwise the bench reports
    null."""
    import json
    w = synth.WORKLOADS["sam2_8obj"]
    src = os.path.join(ROOT, "paper_2608_22526_gb300", "csrc")
    dst = tmp_path / "paper_2608_22526_gb300" / "csrc"
    dst.mkdir(parents=True)
    for f in ("rs3_readout.cu", "rs3_readout_tc.cu", "rs3_readout_common.cuh", "rs3_tc_ptx.cuh"):
        shutil.copy(os.path.join(src, f), dst / f)
    (tmp_path / "profiles").mkdir()
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    rec = {"source_hash": bench.readout_source_hash(), "per_launch_bytes": {w.name: 12345}}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    assert bench._traffic_record(w) == 12345
    rec["source_hash"] = "0" * 16
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    assert bench._traffic_record(w) is None


@pytest.mark.parametrize("name", sorted(synth.WORKLOADS))
def test_workload_config_names_the_workload(name):
    w = synth.WORKLOADS[name]
    cfg = bench.workload_config(w, 1)
    assert cfg["workload"].startswith(name + ":")
    assert f"{w.m}x{w.n}" in cfg["workload"] and f"{w.frames} frames" in cfg["workload"]
    assert cfg["parallelism"] == "replicas x1"


def test_close_argmax_work_closed_form():
    w = synth.WORKLOADS["sam2_8obj"]
    # 8 objects x 256^2 fp32 logits read, one 256^2 palette and 8 grid masks written
    assert bench.close_argmax_work(w) == 8 * 256 * 256 * 4 + 256 * 256 + 8 * 64 * 64
    w = synth.WORKLOADS["multistream"]
    assert bench.close_argmax_work(w) == 48 * 384 * 384 * 4 + 16 * 384 * 384 + 48 * 96 * 96


class _Rec:
    """Stands in for the pipeline and the device inputs: records the calls."""

    def __init__(self, w):
        self.w = w
        self.calls = []
        self.track = self
        self.bank = None

    def zero_(self):
        self.calls.append(("track_zero",))

    def use_buffer(self, i):
        self.calls.append(("buffer", i))

    def select(self, z, prev, stream=None):
        self.calls.append(("select", z[1], prev[1]))

    def commit(self, k, v, mask, is_cond, rope=None):
        self.calls.append(("commit", k[1], None if mask is None else mask[1], is_cond))


class _Data:
    def __init__(self, w):
        self.T = w.frames + w.prefill_frames
        self.P = w.prefill_frames
        self.rope = None

    @staticmethod
    def frame(key, t):
        return (key, t)


@pytest.mark.parametrize("name", sorted(synth.WORKLOADS))
def test_per_call_graphs_issue_the_pass_calls(name, monkeypatch):
    """The per-call times divide graphs of one kind of call by the readout
    frames: "select" holds one selection per readout frame (on its keep-set
    buffer), "commit" every commit of the pass in order, "setup" the commits
    before the first readout frame, so commit minus setup is one commit per
    readout frame."""
    from paper_2608_22526_gb300 import rs3
    monkeypatch.setattr(rs3, "rs3_bank_reset", lambda *a, **k: None)
    w = synth.WORKLOADS[name]
    data = _Data(w)
    first = data.P + (1 if w.n_cond > 0 else 0)
    readout = list(range(first, data.T))
    out = {}
    for what in ("select", "commit", "setup"):
        pipe = _Rec(w)
        bench.calls_only(pipe, data, what)
        out[what] = [c for c in pipe.calls if c[0] != "track_zero"]
    sel = out["select"]
    assert sel == [c for t in readout for c in (("buffer", t % 2), ("select", t, t))]
    setup = [("commit", t, None, 0) for t in range(data.P)]
    if w.n_cond > 0:
        setup.append(("commit", data.P, data.P, 1))
    assert out["setup"] == setup
    assert out["commit"] == setup + [("commit", t, t, 0) for t in readout]
