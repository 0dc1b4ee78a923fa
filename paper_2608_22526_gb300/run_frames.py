"""Runs the first frames of a synthetic workload through the library, one
frame at a time (select, readout, commit), and prints the status word and
the kept-query counts of the last frame.  A short, self-contained invocation
of the hot path for profilers:

    python -m paper_2608_22526_gb300.run_frames --workload sam2_8obj --frames 12 [--dense]

With --dense every cell is selected and nothing is write-pruned (rho = 1,
all-ones masks): the unpruned comparison of the same kernels.

    python -m paper_2608_22526_gb300.run_frames --workload sam2_8obj --close-argmax 3

runs only the decoder-side call instead: rs3_close_argmax (the 9 x 9 closure
per object, the palette argmax and down_s) on the workload's streams and
objects, with 256 x 256 logits per 64 x 64 grid, the given number of times.
"""
from __future__ import annotations

import argparse

import numpy as np
import torch

from . import synth
from .pipeline import Pipeline


def _dev(x: np.ndarray) -> torch.Tensor:
    if x.dtype == np.uint16:
        return torch.from_numpy(x.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def run(workload: str, frames: int, dense: bool) -> Pipeline:
    w = synth.WORKLOADS[workload]
    seq = synth.Sequence(w)
    pipe = Pipeline(w, dense=dense)
    ug = w.unit_group()
    first = 1 if w.n_cond > 0 else 0
    for t in range(min(frames, w.frames)):
        kn, vn = seq.kv_new(t)
        mk = seq.masks(t)
        if t < first:
            pipe.commit(_dev(kn), _dev(vn), _dev(mk), 1)
            if w.n_ptr > 0:
                kp, vp = seq.pointers()
                pipe.set_pointers(_dev(kp), _dev(vp))
            continue
        z = _dev(seq.z(t))
        prev = np.ones_like(mk) if dense else (seq.masks(t - 1) if t > 0 else np.zeros_like(mk))
        pipe.select(z, _dev(prev))
        x = _dev(seq.z(t)[ug])
        pipe.readout(z, x, x)
        pipe.commit(_dev(kn), _dev(vn), _dev(mk), 0)
    torch.cuda.synchronize()
    return pipe


def close_argmax(workload: str, launches: int) -> int:
    from . import rs3
    w = synth.WORKLOADS[workload]
    h, wd = 4 * w.m, 4 * w.n
    logits = _dev(synth.decoder_logits(np.random.default_rng(w.seed + 101), w.U, h, wd))
    gs = torch.arange(0, w.U + 1, w.units_per_group, dtype=torch.int32, device="cuda")
    pal = torch.empty((w.G, h, wd), dtype=torch.uint8, device="cuda")
    grid = torch.empty((w.U, w.m, w.n), dtype=torch.uint8, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for _ in range(launches):
        rs3.rs3_close_argmax(logits, gs, w.G, w.U, h, wd, 4, 4, pal, None, grid, status)
    torch.cuda.synchronize()
    return int(status.item())


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="sam2_1obj", choices=sorted(synth.WORKLOADS))
    ap.add_argument("--frames", type=int, default=12)
    ap.add_argument("--dense", action="store_true")
    ap.add_argument("--close-argmax", type=int, default=0, metavar="N",
                    help="run rs3_close_argmax N times instead of the frames")
    args = ap.parse_args()
    if args.close_argmax > 0:
        st = close_argmax(args.workload, args.close_argmax)
        print("status", st)
        raise SystemExit(0 if st == 0 else 1)
    pipe = run(args.workload, args.frames, args.dense)
    print("status", pipe.status_code(), "count", pipe.count.tolist())


if __name__ == "__main__":
    main()
