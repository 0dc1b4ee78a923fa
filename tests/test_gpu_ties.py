"""Top-k keep-sets with equal energies at the k-th place (Eq. 5 and the keep
ratio of Table 4), on the GPU through the C ABI, bit for bit against the
oracle.

The ranking key is (energy desc, cell index asc): among cells of equal energy
the lower indices are kept.  Gaussian grids almost never produce two equal
fp32 energies, so these inputs are built to: channels in {-1, 0, +1} make every
energy an integer (a few dozen distinct values over thousands of cells), all
channels +-1 make every energy equal, and rows that are permutations of one
vector give energies that are equal in exact arithmetic but may differ in the
last bits of the canonical fp32 sum.  Prior sizes sit just below, at and just
above k_max, and well above it."""
import dataclasses
import zlib

import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2608_22526_gb300 import rs3, synth
from paper_2608_22526_gb300.pipeline import Pipeline
from tests._harness import to_dev, to_host


def _workload(m, n, H, d, dtype, G, upg, union_mode, r_s):
    w = synth.Workload("ties", 40, m, n, H, d, dtype, G, upg, 2, 0.05, 0.3, 1, 6, 0,
                       union_mode=union_mode)
    return dataclasses.replace(w, r_s=r_s)


def _z(kind, rng, w):
    if kind == "ternary":
        return synth.ternary_grid(rng, w.G, w.mn, w.C, 0.5, w.dtype)
    if kind == "ternary_sparse":
        return synth.ternary_grid(rng, w.G, w.mn, w.C, 0.3, w.dtype)
    if kind == "all_equal":
        return synth.ternary_grid(rng, w.G, w.mn, w.C, 1.0, w.dtype)
    return synth.permuted_rows(rng, w.G, w.mn, w.C, w.dtype)


def _sizes(k, mn, U, rng):
    base = [k - 1, k, k + 1, k + 2, k + 97, min(mn, 2 * k + 5), mn, 0]
    return [max(0, min(mn, s)) for s in (base * ((U + 7) // 8))[:U]]


def _select_both(w, z, prev, sp):
    rho, r_s, c, union_mode = sp
    params = rs3.default_params(rho=rho, r_s=r_s, c=c, union_mode=union_mode)
    pipe = Pipeline(w, params=params)
    pipe.select(to_dev(z), to_dev(prev))
    track = np.zeros((w.U, 6), np.int32)
    sel = orc.select(z, w.dtype, prev, w.unit_group(), track, w.m, w.n, rho, r_s, c, union_mode)
    return pipe, sel, track


def _boundary_ties(sel, w):
    """Units whose k-th and (k+1)-th ranked prior cells have the same energy."""
    ties = 0
    for u in range(w.U):
        g = int(w.unit_group()[u])
        P = np.flatnonzero(sel.prior[u]) if not w.union_mode else None
        if P is None:
            members = np.flatnonzero(w.unit_group() == g)
            P = np.flatnonzero(np.any(sel.prior[members] != 0, axis=0))
        if P.size <= sel.k:
            continue
        e = np.sort(sel.energy[g][P])[::-1]
        ties += int(e[sel.k - 1] == e[sel.k])
    return ties


CASES = [
    # name,          m,  n, H,   d, dtype,  G, upg, union, r_s, z kind
    ("64x64_unit",   64, 64, 1, 256, "bf16", 1, 8, 0, 0, "ternary"),
    ("64x64_equal",  64, 64, 1, 256, "bf16", 1, 8, 0, 0, "all_equal"),
    ("64x64_perm",   64, 64, 1, 256, "bf16", 1, 8, 0, 0, "permuted"),
    ("64x64_union",  64, 64, 1, 256, "bf16", 2, 4, 1, 4, "ternary"),
    ("96x96_unit",   96, 96, 4, 64, "bf16", 2, 8, 0, 0, "ternary_sparse"),
    ("96x96_union",  96, 96, 4, 64, "bf16", 3, 3, 1, 2, "ternary"),
    ("32x32_fp32",   32, 32, 1, 64, "f32", 1, 8, 0, 0, "ternary"),
]


def _inputs(case):
    name, m, n, H, d, dtype, G, upg, union_mode, r_s, kind = case
    w = _workload(m, n, H, d, dtype, G, upg, union_mode, r_s)
    rng = np.random.default_rng(zlib.crc32(name.encode()))
    z = _z(kind, rng, w)
    k = orc.kmax(w.rho, w.mn)
    if union_mode:
        # random priors of mixed sizes; the union decides |P|
        prev = synth.cell_subset_masks(rng, w.U, w.mn, rng.integers(20, w.mn // 6, size=w.U))
    else:
        prev = synth.cell_subset_masks(rng, w.U, w.mn, _sizes(k, w.mn, w.U, rng))
    return w, z, prev, (w.rho, r_s, w.c, union_mode)


@pytest.mark.parametrize("case", [c for c in CASES if c[-1] != "permuted"], ids=lambda c: c[0])
def test_tie_inputs_put_equal_keys_at_the_kth_place(case):
    """CPU check of the inputs above (oracle only): every tie case has at
    least one unit whose k-th and (k+1)-th ranked cells share an energy, and
    the oracle's keep-set is the first k cells of P ordered by (energy desc,
    index asc) with numpy's lexicographic sort."""
    w, z, prev, sp = _inputs(case)
    rho, r_s, c, union_mode = sp
    track = np.zeros((w.U, 6), np.int32)
    sel = orc.select(z, w.dtype, prev, w.unit_group(), track, w.m, w.n, rho, r_s, c, union_mode)
    assert _boundary_ties(sel, w) >= 1
    for u in range(w.U):
        g = int(w.unit_group()[u])
        if w.union_mode:
            members = np.flatnonzero(w.unit_group() == g)
            P = np.flatnonzero(np.any(sel.prior[members] != 0, axis=0))
        else:
            P = np.flatnonzero(sel.prior[u])
        e = sel.energy[g][P].astype(np.float64)
        order = np.lexsort((P, -e))                # energy desc, then cell asc
        want = np.sort(P[order[: sel.k]])
        assert np.array_equal(sel.keep(u), want), u


@pytest.mark.gpu
@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_topk_ties_bitexact(case):
    kind = case[-1]
    w, z, prev, sp = _inputs(case)
    pipe, sel, track = _select_both(w, z, prev, sp)
    cnt = to_host(pipe.count)
    idx = to_host(pipe.idx)
    assert np.array_equal(cnt, sel.count), (cnt, sel.count)
    for u in range(w.U):
        assert np.array_equal(idx[u, : cnt[u]], sel.keep(u)), f"unit {u} (|K_r| = {cnt[u]})"
    assert np.array_equal(to_host(pipe.track), track)
    assert pipe.status_code() == 0
    if kind in ("ternary", "all_equal", "ternary_sparse"):
        # the case really puts equal keys across the k-th place
        assert _boundary_ties(sel, w) >= 1


@pytest.mark.gpu
def test_topk_ties_repeated_calls_same_grid():
    """The same tied grid selected twice from different priors: nothing of
    the first call's ranking leaks into the second."""
    w = _workload(64, 64, 1, 256, "bf16", 1, 8, 0, 0)
    rng = np.random.default_rng(77)
    z = synth.ternary_grid(rng, w.G, w.mn, w.C, 0.5, w.dtype)
    k = rs3.rs3_kmax(w.rho, w.mn)
    params = rs3.default_params(rho=w.rho, r_s=0, c=w.c, union_mode=0)
    pipe = Pipeline(w, params=params)
    for rep in range(2):
        prev = synth.cell_subset_masks(rng, w.U, w.mn, _sizes(k, w.mn, w.U, rng)[::-1])
        pipe.track.zero_()
        pipe.select(to_dev(z), to_dev(prev))
        track = np.zeros((w.U, 6), np.int32)
        sel = orc.select(z, w.dtype, prev, w.unit_group(), track, w.m, w.n, w.rho, 0, w.c, 0)
        cnt = to_host(pipe.count)
        assert np.array_equal(cnt, sel.count)
        idx = to_host(pipe.idx)
        for u in range(w.U):
            assert np.array_equal(idx[u, : cnt[u]], sel.keep(u)), (rep, u)
    torch.cuda.synchronize()
    assert pipe.status_code() == 0
