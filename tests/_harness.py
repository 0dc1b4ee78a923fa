"""Lockstep runner: the CUDA path (through the C ABI) and the CPU oracle
consume the same seeded inputs frame by frame; every integer result is
compared bit for bit and the readout within the stated tolerances."""
from __future__ import annotations

import dataclasses
from typing import Iterable, Optional

import numpy as np
import torch

from oracle import oracle as orc
from paper_2608_22526_gb300 import synth

# bf16 I/O: max-abs 2e-2 and mean-abs 2e-3 against fp64; fp32: 1e-4 relative
BF16_MAX_ABS = 2e-2
BF16_MEAN_ABS = 2e-3
F32_REL = 1e-4


def to_dev(x: np.ndarray, dtype: str = None, device="cuda") -> torch.Tensor:
    """numpy -> device tensor; uint16 arrays are bf16 bit patterns."""
    if x.dtype == np.uint16:
        return torch.from_numpy(x.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x)).to(device)


def to_host(t: torch.Tensor) -> np.ndarray:
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def widen(x: np.ndarray, dtype: str) -> np.ndarray:
    return orc.widen(x, dtype).astype(np.float64)


@dataclasses.dataclass
class Report:
    frames_checked: int = 0
    rows_checked: int = 0
    max_abs: float = 0.0
    mean_abs_worst: float = 0.0
    max_rel: float = 0.0
    select_frames: int = 0
    commit_frames: int = 0


def check_readout(dtype: str, got: np.ndarray, ref: np.ndarray, rep: Report, what: str):
    """got: GPU output rows (stored dtype), ref: oracle rows (fp64 or stored)."""
    g = widen(got, dtype)
    r = widen(ref, dtype) if ref.dtype != np.float64 else ref
    if g.size == 0:
        return
    err = np.abs(g - r)
    if dtype == "bf16":
        mx, mean = float(err.max()), float(err.mean())
        rep.max_abs = max(rep.max_abs, mx)
        rep.mean_abs_worst = max(rep.mean_abs_worst, mean)
        assert mx <= BF16_MAX_ABS, f"{what}: max-abs {mx}"
        assert mean <= BF16_MEAN_ABS, f"{what}: mean-abs {mean}"
    else:
        rel = float(err.max() / max(np.abs(r).max(), 1e-30))
        rep.max_rel = max(rep.max_rel, rel)
        assert rel <= F32_REL, f"{what}: rel {rel}"


def bf16_ulp(x: np.ndarray) -> np.ndarray:
    """Spacing of bf16 values at |x| (8 significant bits)."""
    ax = np.maximum(np.abs(x), 2.0 ** -126)
    return 2.0 ** (np.floor(np.log2(ax)) - 7)


def check_fused(dtype: str, got: np.ndarray, res: np.ndarray, A: np.ndarray, rep: Report, what: str):
    """The fused residual output out = x + A is rounded once to the output
    dtype.  Its error is the attention error plus that one rounding, so bf16
    allows max-abs 2e-2 plus half a bf16 step of x + A per element (a step is
    2^-5 at |x| in [4, 8), more than 2e-2 on its own), and the mean-abs bound.
    fp32: the relative bound on x + A."""
    g = widen(got, dtype)
    exact = widen(res, dtype) + A
    err = np.abs(g - exact)
    if g.size == 0:
        return
    if dtype == "bf16":
        excess = float(np.max(err - 0.5 * bf16_ulp(exact)))
        rep.max_abs = max(rep.max_abs, float(err.max()))
        assert excess <= BF16_MAX_ABS, f"{what}: error beyond one rounding {excess}"
        assert float(err.mean()) <= BF16_MEAN_ABS, f"{what}: mean-abs {err.mean()}"
    else:
        rel = float(err.max() / max(np.abs(exact).max(), 1e-30))
        rep.max_rel = max(rep.max_rel, rel)
        assert rel <= F32_REL, f"{what}: rel {rel}"


def sample_rows(count: int, limit: Optional[int], rng: np.random.Generator) -> np.ndarray:
    if limit is None or count <= limit:
        return np.arange(count)
    pick = rng.choice(np.arange(1, count - 1), size=limit - 2, replace=False)
    return np.sort(np.concatenate([[0, count - 1], pick]))


def run_lockstep(w: synth.Workload, frames: Optional[int] = None,
                 check_frames: Iterable[int] = (), rows_per_unit: Optional[int] = None,
                 rope: bool = False, residual_mode: str = "inplace", dense: bool = False,
                 vanish: Optional[dict] = None, threads: int = 8, seed: int = 0,
                 rope_keys: bool = False) -> Report:
    """rope: queries rotated by their own cell in the readout (Eq. 7);
    rope_keys: keys also stored rotated by their own cell at commit (Eq. 7 on
    the key side, rs3_bank_commit_rope), pointer rows unrotated."""
    from paper_2608_22526_gb300.pipeline import Pipeline
    from paper_2608_22526_gb300 import rs3

    frames = w.frames if frames is None else frames
    check_frames = set(check_frames)
    seq = synth.Sequence(w, vanish=vanish)
    pipe = Pipeline(w, dense=dense)
    ug = w.unit_group()
    ob = orc.OracleBank(w.U, w.D, w.dtype, w.mn, w.n_cond, w.window, pipe.bank.ring_cap,
                        pipe.bank.max_frames, w.n_ptr)
    track = np.zeros((w.U, 6), np.int32)
    rho = 1.0 if dense else w.rho
    rope_tab = seq.rope_table() if (rope or rope_keys) else None
    rope_dev = to_dev(rope_tab) if (rope or rope_keys) else None
    key_tab = rope_tab if rope_keys else None
    key_dev = rope_dev if rope_keys else None
    rng = np.random.default_rng(seed)
    rep = Report()
    row_bytes_dt = np.uint16 if w.dtype == "bf16" else np.float32

    def commit_both(s: int, is_cond: int, mask: Optional[np.ndarray]):
        kn, vn = seq.kv_new(s)
        pipe.commit(to_dev(kn), to_dev(vn), None if mask is None else to_dev(mask), is_cond, rope=key_dev)
        st = ob.commit(kn, vn, None if (mask is None or dense) else mask, is_cond, rope=key_tab)
        assert st == [0] * w.U, st
        rep.commit_frames += 1

    def check_bank(full: bool):
        meta, fr = rs3.rs3_bank_read_meta(pipe.bank)
        for u in range(w.U):
            assert meta[u, 0] == ob.state[u, 0] and meta[u, 1] == ob.state[u, 1], (u, meta[u], ob.state[u])
            assert meta[u, 2] == ob.state[u, 2] and meta[u, 3] == ob.state[u, 3]
            assert meta[u, 5] == ob.state[u, 5] and meta[u, 6] == ob.ptr_len[u]
            assert meta[u, 7] == ob.length(u)
            assert [tuple(x) for x in fr[u, : meta[u, 3]]] == ob.frames(u)
        if full:
            ks = to_host(pipe.bank.k_store)
            vs = to_host(pipe.bank.v_store)
            for u in range(w.U):
                rows = ob.logical_rows(u)
                if key_tab is None or w.dtype != "bf16":
                    assert np.array_equal(ks[u][rows], ob.K[u][rows]), f"K rows of unit {u}"
                else:
                    # the device rotates in fp32, the oracle in fp64: after the one
                    # rounding to bf16 they differ by one unit in the last place
                    # plus the fp32 error of k0 cos - k1 sin where it cancels
                    # (absolute, a few 2^-24 of the keys' size), and almost never
                    g = widen(ks[u][rows], "bf16").astype(np.float64)
                    r = widen(ob.K[u][rows], "bf16").astype(np.float64)
                    tol = 2.0 ** -7 * np.abs(r) + 2.0 ** -20 * max(float(np.abs(r).max()), 1e-30)
                    assert (np.abs(g - r) <= tol).all(), f"K rows of unit {u}"
                    assert (ks[u][rows] == ob.K[u][rows]).mean() > 0.99, f"K rows of unit {u}"
                assert np.array_equal(vs[u][rows], ob.V[u][rows]), f"V rows of unit {u}"

    for s in range(w.prefill_frames):
        commit_both(s, 0, None)
    for t in range(frames):
        s = w.prefill_frames + t
        mask_t = seq.masks(s)
        if dense:
            mask_t_commit = None
        else:
            mask_t_commit = mask_t
        if t == 0 and w.n_cond > 0:
            commit_both(s, 1, mask_t_commit)
            if w.n_ptr > 0:
                kp, vp = seq.pointers()
                pipe.set_pointers(to_dev(kp), to_dev(vp))
                ob.set_pointers(kp, vp)
            check_bank(True)
            continue
        prev = seq.masks(s - 1) if s >= 1 else np.zeros((w.U, w.mn), np.uint8)
        if dense:
            prev = np.ones_like(prev)
        z = seq.z(s)
        z_dev = to_dev(z)
        pipe.select(z_dev, to_dev(prev))
        sel = orc.select(z, w.dtype, prev, ug, track, w.m, w.n, rho, w.r_s, w.c, w.union_mode)
        cnt = to_host(pipe.count)
        idx = to_host(pipe.idx)
        assert np.array_equal(cnt, sel.count), (t, cnt, sel.count)
        for u in range(w.U):
            assert np.array_equal(idx[u, : cnt[u]], sel.keep(u)), (t, u)
        assert np.array_equal(to_host(pipe.track), track), t
        rep.select_frames += 1

        # readout on the bank as it stands before this frame's commit
        if residual_mode == "none":
            res_np = None
            out_dev = torch.empty((w.U, w.mn, w.D), dtype=synth_torch_dtype(w), device="cuda")
            res_dev = None
        else:
            res_np = np.ascontiguousarray(np.repeat(z[ug], 1, axis=0))   # residual = z of the unit's group
            res_dev = to_dev(res_np)
            if residual_mode == "inplace":
                out_dev = res_dev
            else:
                out_dev = torch.empty_like(res_dev)
        attn = None
        if t in check_frames and res_np is not None:
            # the attention output itself (Eq. 6 with zeros elsewhere)
            attn_dev = torch.empty((w.U, w.mn, w.D), dtype=synth_torch_dtype(w), device="cuda")
            pipe.readout(z_dev, None, attn_dev, rope=rope_dev)
            attn = to_host(attn_dev)
        pipe.readout(z_dev, res_dev, out_dev, rope=rope_dev)
        if t in check_frames:
            out = to_host(out_dev)
            if attn is None:
                attn = out
            for u in range(w.U):
                keep = sel.keep(u)
                rows = sample_rows(keep.size, rows_per_unit, rng)
                K, V = ob.kv(u)
                A = orc.readout(z[ug[u]], w.dtype, w.H, w.d, keep[rows], K, V, w.dtype,
                                rope=rope_tab, threads=threads)
                cells = keep[rows]
                others = np.setdiff1d(np.arange(w.mn), keep)
                check_readout(w.dtype, attn[u][cells], A, rep, f"frame {t} unit {u}")
                assert np.all(widen(attn[u][others], w.dtype) == 0.0), f"zeros off K_r {t} {u}"
                if res_np is not None:
                    check_fused(w.dtype, out[u][cells], res_np[u][cells], A, rep, f"frame {t} unit {u}")
                    assert np.array_equal(out[u][others], res_np[u][others]), f"pass-through {t} {u}"
                rep.rows_checked += rows.size
            rep.frames_checked += 1
        commit_both(s, 0, mask_t_commit)
        check_bank(t == frames - 1 or t in check_frames)
    assert int(pipe.status.item()) == 0
    return rep


def synth_torch_dtype(w: synth.Workload):
    return torch.bfloat16 if w.dtype == "bf16" else torch.float32
