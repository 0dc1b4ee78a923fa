"""The readout in two phases (rs3_memory_readout_attend, then
rs3_memory_readout_merge on another stream, with the frame's bank commit
running beside the merge) gives the same bytes as rs3_memory_readout, frame
after frame, and leaves the same bank behind."""
import numpy as np
import pytest

from paper_2608_22526_gb300 import synth

from _harness import to_dev, to_host

W = synth.WORKLOADS


def _sequence(w, split: bool):
    import torch
    from paper_2608_22526_gb300.pipeline import Pipeline
    seq = synth.Sequence(w)
    pipe = Pipeline(w)
    torch.cuda.synchronize()                    # the bank's set-up ran on the default stream
    ug = w.unit_group()
    main = torch.cuda.Stream()
    merge = torch.cuda.Stream()
    outs = []
    with torch.cuda.stream(main):
        for t in range(w.frames):
            kn, vn = (to_dev(a) for a in seq.kv_new(t))
            mk = to_dev(seq.masks(t))
            if t == 0 and w.n_cond > 0:
                pipe.commit(kn, vn, mk, 1)
                if w.n_ptr > 0:
                    pipe.set_pointers(*(to_dev(a) for a in seq.pointers()))
                continue
            z_np = seq.z(t)
            z = to_dev(z_np)
            prev = to_dev(seq.masks(t - 1) if t > 0 else np.zeros_like(seq.masks(t)))
            pipe.select(z, prev)
            x = to_dev(np.ascontiguousarray(z_np[ug]))
            if split:
                pipe.readout_attend(z, x, x)
                attended = torch.cuda.Event()
                attended.record(main)
                merge.wait_event(attended)
                pipe.readout_merge(z, x, x, stream=merge)
                pipe.commit(kn, vn, mk, 0)          # beside the merge: it reads no bank
                merged = torch.cuda.Event()
                merged.record(merge)
                main.wait_event(merged)
            else:
                pipe.readout(z, x, x)
                pipe.commit(kn, vn, mk, 0)
            outs.append(to_host(x))
    torch.cuda.synchronize()
    return outs, pipe


@pytest.mark.gpu
@pytest.mark.parametrize("name,frames", [("sam2_8obj", 8), ("sam2_1obj", 8)])
def test_two_phase_readout_matches_single_call(name, frames):
    w = synth.scaled(W[name], frames=frames)
    ref, pa = _sequence(w, split=False)
    got, pb = _sequence(w, split=True)
    assert pa.status_code() == 0 and pb.status_code() == 0
    for t, (a, b) in enumerate(zip(ref, got)):
        assert np.array_equal(a, b), f"frame {t + 1}"
    assert np.array_equal(to_host(pa.bank.meta), to_host(pb.bank.meta))
    assert np.array_equal(to_host(pa.bank.k_store), to_host(pb.bank.k_store))
    assert np.array_equal(to_host(pa.bank.v_store), to_host(pb.bank.v_store))
