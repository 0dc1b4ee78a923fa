"""Pins for the CPU oracle: each test checks the oracle against something other
than itself -- values the paper prints, closed forms, invariants, a library
routine, brute force on tiny inputs -- so that a dropped term, a wrong sign or
index, or a transposed operand fails somewhere.  CPU only."""
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bf16_bits(x):
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    return ((u + ((u >> 16) & 1) + 0x7FFF) >> 16).astype(np.uint16)


# ---------------------------------------------------------------------------
# k = floor(rho * mn): Table 4 (keep-ratio sweep) and Sec. 4.2
# ---------------------------------------------------------------------------

def _table4():
    rows = []
    with open(os.path.join(GOLDEN, "table4_kr_max.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                r, mn, k = line.split()
                rows.append((float(r), int(mn), int(k)))
    return rows


@pytest.mark.parametrize("rho,mn,k", _table4())
def test_kmax_matches_table4(rho, mn, k):
    assert orc.kmax(rho, mn) == k


def test_selection_count_is_exactly_k_when_prior_is_larger():
    rng = np.random.default_rng(1)
    m = n = 64
    z = _bf16_bits(rng.standard_normal((1, m * n, 64), dtype=np.float32))
    masks = np.ones((1, m * n), np.uint8)              # prior = whole grid
    track = np.zeros((1, 6), np.int32)
    for rho, _, k in _table4():
        tr = track.copy()
        r = orc.select(z, "bf16", masks, np.zeros(1, np.int32), tr, m, n, rho, 4, 14, 1)
        assert r.count[0] == k
        assert np.all(np.diff(r.keep(0)) > 0)          # ascending, distinct


# ---------------------------------------------------------------------------
# geometry: bbox and Chebyshev dilation against brute force
# ---------------------------------------------------------------------------

def _brute_dilate(M, m, n, r):
    out = np.zeros((m, n), np.uint8)
    pts = [(y, x) for y in range(m) for x in range(n) if M[y * n + x]]
    for y in range(m):
        for x in range(n):
            out[y, x] = any(abs(y - a) <= r and abs(x - b) <= r for a, b in pts)
    return out.reshape(-1)


@pytest.mark.parametrize("m,n,r,p", [(7, 9, 0, 0.2), (7, 9, 1, 0.1), (8, 8, 2, 0.05),
                                     (5, 11, 4, 0.08), (9, 6, 3, 0.0), (6, 6, 7, 0.03)])
def test_dilate_matches_bruteforce(m, n, r, p):
    rng = np.random.default_rng(m * 100 + n * 10 + r)
    for _ in range(4):
        M = (rng.random(m * n) < p).astype(np.uint8)
        assert np.array_equal(orc.dilate(M, m, n, r), _brute_dilate(M, m, n, r))


def test_bbox_matches_scan():
    rng = np.random.default_rng(2)
    for _ in range(20):
        m, n = rng.integers(1, 12, size=2)
        M = (rng.random(m * n) < 0.15).astype(np.uint8)
        ys, xs = np.nonzero(M.reshape(m, n))
        got = orc.bbox(M, m, n)
        if ys.size == 0:
            assert got is None
        else:
            assert got == (ys.min(), xs.min(), ys.max(), xs.max())


# ---------------------------------------------------------------------------
# priors: Eq. 1 (seed box), Eq. 2 (mask), Eq. 4 (streak-counted fallback)
# ---------------------------------------------------------------------------

def _rect_area(y0, x0, y1, x1, r, m, n):
    ya, yb = max(0, y0 - r), min(m - 1, y1 + r)
    xa, xb = max(0, x0 - r), min(n - 1, x1 + r)
    return (yb - ya + 1) * (xb - xa + 1)


def test_fallback_radius_grows_then_saturates():
    """Eq. 4: an object missing for t frames is searched at radius
    r_s + min(t, c); the cap is r_s + c; the cached box persists."""
    m = n = 96
    r_s, c = 4, 14
    M = np.zeros((m, n), np.uint8)
    M[40:46, 50:60] = 1                                # box (40,50)-(45,59)
    track = np.zeros(6, np.int32)
    P = orc.prior_unit(M.reshape(-1), m, n, track, r_s, c)
    assert tuple(track) == (40, 50, 45, 59, 1, 0)
    assert P.sum() == orc.dilate(M.reshape(-1), m, n, r_s).sum()
    empty = np.zeros(m * n, np.uint8)
    for t in range(1, 21):
        P = orc.prior_unit(empty, m, n, track, r_s, c)
        r = r_s + min(t, c)
        assert track[5] == t and track[4] == 1
        assert P.sum() == _rect_area(40, 50, 45, 59, r, m, n), t
        ys, xs = np.nonzero(P.reshape(m, n))
        assert (ys.min(), xs.min(), ys.max(), xs.max()) == (max(0, 40 - r), max(0, 50 - r),
                                                            min(m - 1, 45 + r), min(n - 1, 59 + r))
    # reappearance resets the streak and the box follows the new mask
    M2 = np.zeros((m, n), np.uint8)
    M2[10:12, 10:13] = 1
    orc.prior_unit(M2.reshape(-1), m, n, track, r_s, c)
    assert tuple(track) == (10, 10, 11, 12, 1, 0)


def test_never_seen_object_has_empty_prior():
    m = n = 16
    track = np.zeros(6, np.int32)
    P = orc.prior_unit(np.zeros(m * n, np.uint8), m, n, track, 4, 14)
    assert P.sum() == 0 and track[4] == 0 and track[5] == 1


def test_seed_bbox_mode_is_dilated_rectangle():
    """Eq. 1: the seed prior dilates the tight box, not the mask."""
    m = n = 32
    M = np.zeros((m, n), np.uint8)
    M[5, 5] = M[12, 20] = 1                             # box (5,5)-(12,20)
    track = np.zeros(6, np.int32)
    P = orc.prior_unit(M.reshape(-1), m, n, track, 4, 14, bbox_mode=1)
    assert P.sum() == _rect_area(5, 5, 12, 20, 4, m, n)
    P2 = orc.prior_unit(M.reshape(-1), m, n, np.zeros(6, np.int32), 4, 14, bbox_mode=0)
    assert P2.sum() == 2 * 81                            # two disjoint 9x9 squares


def test_union_mode_unions_group_priors():
    """Eq. 2: P(t) is the union over the objects of one stream."""
    rng = np.random.default_rng(3)
    m = n = 24
    masks = np.zeros((4, m * n), np.uint8)
    for u in range(4):
        y, x = rng.integers(2, 20, size=2)
        masks[u].reshape(m, n)[y:y + 3, x:x + 2] = 1
    ug = np.array([0, 0, 1, 1], np.int32)
    z = _bf16_bits(rng.standard_normal((2, m * n, 32), dtype=np.float32))
    per = orc.select(z, "bf16", masks, ug, np.zeros((4, 6), np.int32), m, n, 1.0, 2, 14, 0)
    uni = orc.select(z, "bf16", masks, ug, np.zeros((4, 6), np.int32), m, n, 1.0, 2, 14, 1)
    for u in range(4):
        mates = [v for v in range(4) if ug[v] == ug[u]]
        assert np.array_equal(uni.prior[u], np.bitwise_or.reduce(per.prior[mates], axis=0))
        # rho = 1 keeps the whole prior
        assert np.array_equal(np.flatnonzero(uni.prior[u]), uni.keep(u))


# ---------------------------------------------------------------------------
# energy ||z||^2 in the canonical fp32 order
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("C", [8, 32, 64, 256, 264, 512])
def test_energy_small_integers_exact(C):
    """With small integer channels every partial sum is exact, so the canonical
    order must give the exact integer sum: a dropped or doubled channel fails."""
    rng = np.random.default_rng(C)
    z = rng.integers(-3, 4, size=(50, C)).astype(np.float32)
    e = orc.energy_canonical(z)
    assert np.array_equal(e.astype(np.int64), (z.astype(np.int64) ** 2).sum(axis=1))
    # one-hot rows: every channel contributes exactly once
    oh = np.zeros((C, C), np.float32)
    oh[np.arange(C), np.arange(C)] = 2.0
    assert np.all(orc.energy_canonical(oh) == 4.0)


def test_energy_within_fp32_bound_of_exact():
    rng = np.random.default_rng(5)
    for C in (64, 256):
        z = (rng.standard_normal((400, C)) * rng.uniform(0.1, 3.0, size=(400, 1))).astype(np.float32)
        zb = (_bf16_bits(z).astype(np.uint32) << 16).view(np.float32)
        e = orc.energy_canonical(zb).astype(np.float64)
        ex = orc.energy_exact(zb)
        # exact sum of fractions as the reference
        for i in range(0, 400, 37):
            ref = sum(Fraction(float(v)) ** 2 for v in zb[i])
            assert ex[i] == float(ref) or abs(ex[i] - float(ref)) <= 1e-15 * float(ref)
        # recursive summation bound: |err| <= (depth) * u * sum, depth <= C/32 + 5
        bound = (C / 32 + 6) * 2.0 ** -24 * ex
        assert np.all(np.abs(e - ex) <= bound)


# ---------------------------------------------------------------------------
# top-k keep-set (Eq. 5) against brute-force rank counting
# ---------------------------------------------------------------------------

def _brute_topk(P, e, k):
    cells = [i for i in range(P.size) if P[i]]
    keep = []
    for i in cells:
        better = sum(1 for j in cells if (e[j] > e[i]) or (e[j] == e[i] and j < i))
        if better < k:
            keep.append(i)
    return np.array(sorted(keep), dtype=np.int32)


def test_topk_matches_bruteforce():
    rng = np.random.default_rng(7)
    for trial in range(40):
        mn = int(rng.integers(1, 120))
        P = (rng.random(mn) < rng.uniform(0.0, 1.0)).astype(np.uint8)
        e = rng.choice(np.array([0.0, 0.5, 1.0, 1.5, 2.0], np.float32), size=mn) \
            if trial % 2 else rng.random(mn).astype(np.float32)
        k = int(rng.integers(0, mn + 2))
        assert np.array_equal(orc.topk(P, e, k), _brute_topk(P, e, k)), trial


def test_topk_ties_take_lower_index():
    e = np.ones(20, np.float32)
    P = np.ones(20, np.uint8)
    assert np.array_equal(orc.topk(P, e, 5), np.arange(5))
    e[17] = 2.0
    assert np.array_equal(orc.topk(P, e, 3), np.array([0, 1, 17]))


def test_small_prior_keeps_everything():
    P = np.zeros(100, np.uint8)
    P[[3, 50, 99]] = 1
    e = np.arange(100, dtype=np.float32)
    assert np.array_equal(orc.topk(P, e, 10), np.array([3, 50, 99]))
    assert orc.topk(P, e, 0).size == 0


def test_canonical_ranking_agrees_with_exact_up_to_near_ties():
    """The fp32 ranking key selects the same cells as exact energies, except
    where exact energies at the boundary agree to within 2^-20 relative."""
    rng = np.random.default_rng(11)
    m = n = 32
    for C in (64, 256):
        z = (rng.standard_normal((m * n, C))).astype(np.float32)
        zb = (_bf16_bits(z).astype(np.uint32) << 16).view(np.float32)
        e32 = orc.energy_canonical(zb)
        ex = orc.energy_exact(zb)
        P = np.ones(m * n, np.uint8)
        k = orc.kmax(0.3, m * n)
        a = set(orc.topk(P, e32, k).tolist())
        order = sorted(range(m * n), key=lambda i: (-ex[i], i))
        b = set(order[:k])
        diff = a ^ b
        if diff:
            kth = ex[order[k - 1]]
            for i in diff:
                assert abs(ex[i] - kth) <= 2.0 ** -20 * kth


# ---------------------------------------------------------------------------
# readout (Eq. 6): high precision, library attention, closed forms, invariants
# ---------------------------------------------------------------------------

def _mp_attention(q, K, V, scale):
    import mpmath
    mpmath.mp.dps = 50
    out = []
    for qi in q:
        s = [mpmath.mpf(scale) * mpmath.fsum(mpmath.mpf(float(a)) * mpmath.mpf(float(b))
                                             for a, b in zip(qi, kt)) for kt in K]
        mx = max(s)
        w = [mpmath.exp(x - mx) for x in s]
        tot = mpmath.fsum(w)
        out.append([float(mpmath.fsum(wt * mpmath.mpf(float(v[c])) for wt, v in zip(w, V)) / tot)
                    for c in range(V.shape[1])])
    return np.array(out)


def test_readout_matches_high_precision():
    rng = np.random.default_rng(13)
    for (mn, d, N) in [(12, 8, 16), (9, 4, 1), (16, 16, 7)]:
        q = rng.standard_normal((mn, d)).astype(np.float32)
        K = rng.standard_normal((N, d)).astype(np.float32) * 2
        V = rng.standard_normal((N, d)).astype(np.float32)
        idx = np.array(sorted(rng.choice(mn, size=min(mn, 8), replace=False)), np.int32)
        A = orc.readout(q, "f32", 1, d, idx, K, V, "f32")
        ref = _mp_attention(q[idx].astype(np.float64), K.astype(np.float64),
                            V.astype(np.float64), 1 / math.sqrt(d))
        assert np.max(np.abs(A - ref)) < 1e-12


def test_rho1_equals_dense_library_attention():
    """At rho = 1 the gather and scatter are identities (Sec. 3.1, after Eq. 7):
    the readout is dense attention, here torch's fp64 SDPA, per head."""
    rng = np.random.default_rng(17)
    m, n, H, d, N = 6, 5, 4, 16, 40
    mn = m * n
    z = rng.standard_normal((1, mn, H * d)).astype(np.float32)
    K = rng.standard_normal((N, H * d)).astype(np.float32)
    V = rng.standard_normal((N, H * d)).astype(np.float32)
    sel = orc.select(z, "f32", np.ones((1, mn), np.uint8), np.zeros(1, np.int32),
                     np.zeros((1, 6), np.int32), m, n, 1.0, 1, 14, 1)
    assert np.array_equal(sel.keep(0), np.arange(mn))
    A = orc.readout(z[0], "f32", H, d, sel.keep(0), K, V, "f32")
    qt = torch.from_numpy(z[0].astype(np.float64)).view(mn, H, d).transpose(0, 1)
    kt = torch.from_numpy(K.astype(np.float64)).view(N, H, d).transpose(0, 1)
    vt = torch.from_numpy(V.astype(np.float64)).view(N, H, d).transpose(0, 1)
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt)
    ref = ref.transpose(0, 1).reshape(mn, H * d).numpy()
    assert np.max(np.abs(A - ref)) < 1e-12
    # and the scatter of the full keep-set with no residual is exactly A
    out = orc.scatter_output(None, "f32", mn, H * d, sel.keep(0), A)
    assert np.array_equal(out, A.astype(np.float32))


def test_pruned_rows_equal_dense_rows():
    """Pruning only drops query rows: each kept row equals the dense row."""
    rng = np.random.default_rng(19)
    mn, d, N = 40, 32, 50
    q = rng.standard_normal((mn, d)).astype(np.float32)
    K = rng.standard_normal((N, d)).astype(np.float32)
    V = rng.standard_normal((N, d)).astype(np.float32)
    full = orc.readout(q, "f32", 1, d, np.arange(mn, dtype=np.int32), K, V, "f32")
    idx = np.array([1, 7, 8, 30, 39], np.int32)
    part = orc.readout(q, "f32", 1, d, idx, K, V, "f32")
    assert np.array_equal(part, full[idx])


def test_single_key_reads_its_value():
    rng = np.random.default_rng(23)
    q = rng.standard_normal((5, 8)).astype(np.float32)
    K = rng.standard_normal((1, 8)).astype(np.float32)
    V = rng.standard_normal((1, 8)).astype(np.float32)
    A = orc.readout(q, "f32", 1, 8, np.arange(5, dtype=np.int32), K, V, "f32")
    assert np.array_equal(A, np.repeat(V.astype(np.float64), 5, axis=0))


def test_identical_keys_average_values():
    rng = np.random.default_rng(29)
    q = rng.standard_normal((3, 16)).astype(np.float32)
    K = np.repeat(rng.standard_normal((1, 16)).astype(np.float32), 9, axis=0)
    V = rng.standard_normal((9, 16)).astype(np.float32)
    A = orc.readout(q, "f32", 1, 16, np.arange(3, dtype=np.int32), K, V, "f32")
    assert np.max(np.abs(A - V.astype(np.float64).mean(axis=0))) < 1e-14


def test_key_shift_invariance_and_scale():
    """Adding one vector c to every key shifts all logits of a query by q.c, so
    the softmax (hence A) is unchanged; doubling the scale equals doubling K."""
    rng = np.random.default_rng(31)
    q = rng.standard_normal((4, 8)).astype(np.float32)
    K = rng.standard_normal((12, 8)).astype(np.float32)
    V = rng.standard_normal((12, 8)).astype(np.float32)
    idx = np.arange(4, dtype=np.int32)
    A = orc.readout(q, "f32", 1, 8, idx, K, V, "f32")
    c = np.float32(0.5) * rng.standard_normal((1, 8)).astype(np.float32)
    Ks = (K + c).astype(np.float32)
    # exact fp32 adds differ from K + c in fp64 only by rounding of Ks itself
    A2 = orc.readout(q, "f32", 1, 8, idx, Ks, V, "f32")
    assert np.max(np.abs(A - A2)) < 1e-5
    s = 1 / math.sqrt(8)
    A3 = orc.readout(q, "f32", 1, 8, idx, (2 * K).astype(np.float32), V, "f32", scale=s)
    A4 = orc.readout(q, "f32", 1, 8, idx, K, V, "f32", scale=2 * s)
    assert np.max(np.abs(A3 - A4)) < 1e-13


def test_empty_bank_reads_zero():
    q = np.ones((4, 8), np.float32)
    A = orc.readout(q, "f32", 2, 4, np.array([0, 3], np.int32), np.zeros((0, 8), np.float32),
                    np.zeros((0, 8), np.float32), "f32")
    assert A.shape == (2, 8) and np.all(A == 0)


# ---------------------------------------------------------------------------
# RoPE by index (Eq. 7)
# ---------------------------------------------------------------------------

def _rope_table(mn, d, rng):
    ang = rng.uniform(-np.pi, np.pi, size=(mn, d // 2))
    return np.stack([np.cos(ang), np.sin(ang)], -1).astype(np.float32), ang


def test_rope_gather_equals_rotate_then_gather():
    rng = np.random.default_rng(37)
    mn, H, d, N = 20, 2, 8, 11
    q = rng.standard_normal((mn, H * d)).astype(np.float32)
    K = rng.standard_normal((N, H * d)).astype(np.float32)
    V = rng.standard_normal((N, H * d)).astype(np.float32)
    tab, _ = _rope_table(mn, d, rng)
    idx = np.array([2, 5, 6, 13, 19], np.int32)
    A = orc.readout(q, "f32", H, d, idx, K, V, "f32", rope=tab)
    # rotate the full grid with numpy complex arithmetic, then gather without RoPE
    f = tab[..., 0].astype(np.float64) + 1j * tab[..., 1].astype(np.float64)
    qc = q.astype(np.float64).reshape(mn, H, d // 2, 2)
    qz = (qc[..., 0] + 1j * qc[..., 1]) * f[:, None, :]
    qrot = np.stack([qz.real, qz.imag], -1).reshape(mn, H * d)
    Kd = K.astype(np.float64)
    Vd = V.astype(np.float64)
    ref = []
    for j in idx:
        row = []
        for h in range(H):
            s = Kd[:, h * d:(h + 1) * d] @ qrot[j, h * d:(h + 1) * d] / math.sqrt(d)
            w = np.exp(s - s.max())
            row.append(w @ Vd[:, h * d:(h + 1) * d] / w.sum())
        ref.append(np.concatenate(row))
    assert np.max(np.abs(A - np.array(ref))) < 1e-12
    # the prefix slice f[:|K_r|] (what an untouched implementation would use)
    # gives a different answer, which is what Eq. 7 corrects
    prefix = np.zeros_like(tab)
    prefix[idx] = tab[: idx.size]
    Abad = orc.readout(q, "f32", H, d, idx, K, V, "f32", rope=prefix)
    assert np.max(np.abs(Abad - A)) > 1e-3


def test_key_rotation_is_the_complex_product():
    """Eq. 7 on the key side: each pair (2p, 2p+1) of every head of row i,
    read as a complex number, times cos + i sin of the table's entry (i, p)."""
    rng = np.random.default_rng(43)
    mn, H, d = 12, 2, 8
    x = rng.standard_normal((mn, H * d)).astype(np.float32)
    tab, _ = _rope_table(mn, d, rng)
    y = orc.rotate_rows(x, "f32", tab).astype(np.float64).reshape(mn, H, d // 2, 2)
    f = tab[..., 0].astype(np.float64) + 1j * tab[..., 1].astype(np.float64)
    xc = x.astype(np.float64).reshape(mn, H, d // 2, 2)
    z = (xc[..., 0] + 1j * xc[..., 1]) * f[:, None, :]
    assert np.max(np.abs(y[..., 0] - z.real)) < 1e-6 and np.max(np.abs(y[..., 1] - z.imag)) < 1e-6
    # bf16 storage: the fp64 rotation rounded once to nearest-even
    xb = orc.round_to(x.astype(np.float64), "bf16")
    yb = orc.rotate_rows(xb, "bf16", tab)
    xbc = orc.widen(xb, "bf16").astype(np.float64).reshape(mn, H, d // 2, 2)
    zb = (xbc[..., 0] + 1j * xbc[..., 1]) * f[:, None, :]
    ref = np.stack([zb.real, zb.imag], -1).reshape(mn, H * d)
    assert np.array_equal(yb, orc.round_to(ref, "bf16"))


def test_key_rotation_zero_angle_keeps_keys_bit_for_bit():
    rng = np.random.default_rng(47)
    mn, d = 9, 16
    tab = np.zeros((mn, d // 2, 2), np.float32)
    tab[..., 0] = 1.0
    xb = orc.round_to(rng.standard_normal((mn, 2 * d)), "bf16")
    assert np.array_equal(orc.rotate_rows(xb, "bf16", tab), xb)


def test_rotated_bank_equals_rotating_keys_at_read_time():
    """Storing keys rotated by their own cell and reading them with rotated
    queries is the attention of Eq. 6/7 with both sides rotated at read time."""
    rng = np.random.default_rng(53)
    mn, H, d = 16, 2, 8
    q = rng.standard_normal((mn, H * d)).astype(np.float32)
    kx = rng.standard_normal((mn, H * d)).astype(np.float32)
    V = rng.standard_normal((mn, H * d)).astype(np.float32)
    tab, _ = _rope_table(mn, d, rng)
    key_cells = np.array([1, 4, 5, 9, 12, 15])
    krot = orc.rotate_rows(kx, "f32", tab)[key_cells]
    idx = np.array([0, 3, 8, 14], np.int32)
    A = orc.readout(q, "f32", H, d, idx, krot, V[key_cells], "f32", rope=tab)
    f = tab[..., 0].astype(np.float64) + 1j * tab[..., 1].astype(np.float64)

    def rot(x, cells):
        xc = x.astype(np.float64).reshape(-1, H, d // 2, 2)
        z = (xc[..., 0] + 1j * xc[..., 1]) * f[cells][:, None, :]
        return np.stack([z.real, z.imag], -1).reshape(-1, H * d)
    qr, kr = rot(q[idx], idx), rot(kx[key_cells], key_cells)
    Vd = V[key_cells].astype(np.float64)
    ref = np.zeros((idx.size, H * d))
    for h in range(H):
        sl = slice(h * d, (h + 1) * d)
        s = qr[:, sl] @ kr[:, sl].T / math.sqrt(d)
        w = np.exp(s - s.max(axis=1, keepdims=True))
        ref[:, sl] = (w / w.sum(axis=1, keepdims=True)) @ Vd[:, sl]
    assert np.max(np.abs(A - ref)) < 1e-5               # keys held in fp32 after their rotation


def test_rotated_queries_and_keys_see_only_relative_positions():
    """With a 1-D rotary table (angle = position x frequency), rotating the
    query by its cell and the keys by theirs makes every score depend on the
    cells' difference only: shifting all cells together leaves the attention
    unchanged.  A sign mismatch between the two rotations would break this."""
    rng = np.random.default_rng(59)
    mn, d = 64, 8
    freq = np.array([1.0, 0.31, 0.097, 0.029])
    ang = np.arange(mn)[:, None] * freq[None, :]
    tab = np.stack([np.cos(ang), np.sin(ang)], -1).astype(np.float64)
    tab32 = tab.astype(np.float32)
    qv = rng.standard_normal(d).astype(np.float32)
    kv = rng.standard_normal((5, d)).astype(np.float32)
    V = rng.standard_normal((5, d)).astype(np.float32)
    outs = []
    for shift in (0, 17, 40):
        qcell = 3 + shift
        kcells = np.array([0, 2, 5, 9, 20]) + shift
        q = np.zeros((mn, d), np.float32)
        q[qcell] = qv
        kx = np.zeros((mn, d), np.float32)
        kx[kcells] = kv
        krot = orc.rotate_rows(kx, "f32", tab32)[kcells]
        outs.append(orc.readout(q, "f32", 1, d, np.array([qcell], np.int32), krot, V, "f32", rope=tab32))
    assert np.max(np.abs(outs[1] - outs[0])) < 1e-5 and np.max(np.abs(outs[2] - outs[0])) < 1e-5
    # keys rotated the opposite way do not have the property
    bad = np.stack([tab32[..., 0], -tab32[..., 1]], -1)
    outs_bad = []
    for shift in (0, 17):
        qcell, kcells = 3 + shift, np.array([0, 2, 5, 9, 20]) + shift
        q = np.zeros((mn, d), np.float32)
        q[qcell] = qv
        kx = np.zeros((mn, d), np.float32)
        kx[kcells] = kv
        outs_bad.append(orc.readout(q, "f32", 1, d, np.array([qcell], np.int32),
                                    orc.rotate_rows(kx, "f32", bad)[kcells], V, "f32", rope=tab32))
    assert np.max(np.abs(outs_bad[1] - outs_bad[0])) > 1e-3


def test_rope_zero_angle_is_identity():
    rng = np.random.default_rng(41)
    mn, d = 10, 8
    q = rng.standard_normal((mn, d)).astype(np.float32)
    K = rng.standard_normal((6, d)).astype(np.float32)
    V = rng.standard_normal((6, d)).astype(np.float32)
    tab = np.zeros((mn, d // 2, 2), np.float32)
    tab[..., 0] = 1.0
    idx = np.arange(0, mn, 3, dtype=np.int32)
    assert np.array_equal(orc.readout(q, "f32", 1, d, idx, K, V, "f32", rope=tab),
                          orc.readout(q, "f32", 1, d, idx, K, V, "f32"))


# ---------------------------------------------------------------------------
# scatter (Eq. 6) and output rounding
# ---------------------------------------------------------------------------

def test_scatter_leaves_unselected_rows_bit_identical():
    rng = np.random.default_rng(43)
    mn, D = 30, 16
    res = _bf16_bits(rng.standard_normal((mn, D)).astype(np.float32))
    idx = np.array([0, 4, 29], np.int32)
    A = rng.standard_normal((3, D))
    out = orc.scatter_output(res, "bf16", mn, D, idx, A)
    keep = np.setdiff1d(np.arange(mn), idx)
    assert np.array_equal(out[keep], res[keep])
    zero = orc.scatter_output(None, "bf16", mn, D, idx, A)
    assert np.all(zero[keep] == 0)


def test_round_bf16_matches_library_on_fp32_values():
    rng = np.random.default_rng(47)
    x = np.concatenate([rng.standard_normal(20000).astype(np.float32) * 7,
                        # exact ties: bf16 value + half a bf16 step
                        (((np.arange(0, 400, dtype=np.uint32) + 0x3C00) << 16) | 0x8000)
                        .view(np.float32),
                        np.array([1.0, -2.5, 3.0e-3, 65504.0], np.float32)])
    ours = orc.round_to(x.astype(np.float64), "bf16")
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


# ---------------------------------------------------------------------------
# write side: commit (Algorithm 1 sparse write), keep-set (Eq. 8)
# ---------------------------------------------------------------------------

def _bank(U=2, D=8, mn=30, n_cond=1, window=3, n_ptr=2, ring_cap=None, max_frames=None,
          dtype="bf16"):
    ring_cap = ring_cap if ring_cap is not None else max(window, 1) * mn
    max_frames = max_frames if max_frames is not None else (window if window > 0 else 64)
    return orc.OracleBank(U, D, dtype, mn, n_cond, window, ring_cap, max_frames, n_ptr)


def test_commit_holds_exactly_the_masked_rows_in_order():
    rng = np.random.default_rng(53)
    U, D, mn, W = 2, 8, 30, 3
    b = _bank(U, D, mn, 1, W, 2)
    frames = []
    for t in range(7):
        kn = rng.integers(0, 65535, size=(U, mn, D), dtype=np.uint16)
        vn = rng.integers(0, 65535, size=(U, mn, D), dtype=np.uint16)
        mk = (rng.random((U, mn)) < 0.4).astype(np.uint8)
        st = b.commit(kn, vn, mk, is_cond=int(t == 0))
        assert st == [0, 0]
        frames.append((kn, vn, mk, t == 0))
    kp = rng.integers(0, 65535, size=(U, 2, D), dtype=np.uint16)
    b.set_pointers(kp, kp)
    for u in range(U):
        cond = [f for f in frames if f[3]]
        recent = [f for f in frames if not f[3]][-W:]
        expK = np.concatenate([f[0][u][f[2][u].astype(bool)] for f in cond + recent] + [kp[u]])
        expV = np.concatenate([f[1][u][f[2][u].astype(bool)] for f in cond + recent] + [kp[u]])
        K, V = b.kv(u)
        assert np.array_equal(K, expK) and np.array_equal(V, expV)
        assert [ln for _, ln in b.frames(u)] == [int(f[2][u].sum()) for f in recent]
        assert b.length(u) == expK.shape[0]


def test_fixed_write_keepset_gives_constant_stride():
    """Sec. 3.2: K_w fixed at the seed frame -> every stored frame has |K_w| rows."""
    rng = np.random.default_rng(59)
    m = n = 16
    seed = np.zeros((1, m * n), np.uint8)
    seed[0].reshape(m, n)[5:9, 6:10] = 1
    kw = orc.write_keepset(seed, np.zeros(1, np.int32), m, n, D_w=2)
    b = _bank(1, 4, m * n, 0, -1, 0, ring_cap=20 * m * n, max_frames=32, dtype="f32")
    for t in range(12):
        kn = rng.standard_normal((1, m * n, 4)).astype(np.float32)
        assert b.commit(kn, kn, kw, 0) == [0]
    lens = [ln for _, ln in b.frames(0)]
    assert lens == [int(kw.sum())] * 12
    offs = [o for o, _ in b.frames(0)]
    assert offs == [int(kw.sum()) * t for t in range(12)]
    # bank growth O(T |K_w|), not O(T mn)
    assert b.length(0) == 12 * int(kw.sum()) < 12 * m * n


def test_commit_overflow_changes_nothing():
    rng = np.random.default_rng(61)
    mn, D = 10, 4
    b = _bank(1, D, mn, 1, -1, 0, ring_cap=15, max_frames=8, dtype="f32")
    kn = rng.standard_normal((1, mn, D)).astype(np.float32)
    assert b.commit(kn, kn, None, 1) == [0]           # pinned
    assert b.commit(kn, kn, None, 1) == [2]           # only one pinned slot
    assert b.commit(kn, kn, None, 0) == [0]           # 10 of 15 ring rows
    before = (b.state.copy(), b.K.copy())
    assert b.commit(kn, kn, None, 0) == [2]           # 20 > 15: dropped whole
    assert np.array_equal(b.state, before[0]) and np.array_equal(b.K, before[1])
    half = np.zeros((1, mn), np.uint8)
    half[0, :5] = 1
    assert b.commit(kn, kn, half, 0) == [0]           # exactly fills the ring
    assert b.length(0) == 10 + 15


def test_ring_wraps_and_keeps_order():
    rng = np.random.default_rng(67)
    mn, D, W = 8, 2, 2
    b = _bank(1, D, mn, 0, W, 0, ring_cap=2 * mn, max_frames=W, dtype="f32")
    hist = []
    for t in range(9):
        kn = rng.standard_normal((1, mn, D)).astype(np.float32)
        mk = (rng.random((1, mn)) < 0.7).astype(np.uint8)
        assert b.commit(kn, kn, mk, 0) == [0]
        hist.append(kn[0][mk[0].astype(bool)])
        K, _ = b.kv(0)
        assert np.array_equal(K, np.concatenate(hist[-W:]))


@pytest.mark.parametrize("cells,expect_full", [(19, True), (20, False), (21, False),
                                               (379, False), (380, False), (381, True)])
def test_write_fall_through_boundaries(cells, expect_full):
    """Sec. 3.2: seeds covering > 95% or < 5% of mn write the full grid.
    On a 20x20 grid 5% is 20 cells and 95% is 380 cells (strict bounds)."""
    m = n = 20
    seed = np.zeros((1, m * n), np.uint8)
    seed[0, :cells] = 1
    kw = orc.write_keepset(seed, np.zeros(1, np.int32), m, n, D_w=0)
    assert bool(kw.all()) == expect_full
    if not expect_full:
        assert np.array_equal(kw[0], seed[0])          # D_w = 0: the seed itself


def test_write_keepset_is_union_of_dilations():
    rng = np.random.default_rng(71)
    m = n = 24
    seeds = np.zeros((3, m * n), np.uint8)
    for u in range(3):
        y, x = rng.integers(0, 20, size=2)
        seeds[u].reshape(m, n)[y:y + 4, x:x + 3] = 1
    ug = np.zeros(3, np.int32)
    kw = orc.write_keepset(seeds, ug, m, n, D_w=3)
    ref = np.zeros(m * n, np.uint8)
    for u in range(3):
        ref |= _brute_dilate(seeds[u], m, n, 3)
    for u in range(3):
        assert np.array_equal(kw[u], ref)


def test_read_prior_inside_write_keepset_when_dw_covers_fallback():
    """Sec. 3.2 / appendix: P(t) within K_w whenever D_w >= r_s + c, for
    predicted masks that stay inside the seed footprint (including the
    fallback after the object vanishes)."""
    rng = np.random.default_rng(73)
    m = n = 64
    r_s, c = 4, 14
    seed = np.zeros((1, m * n), np.uint8)
    seed[0].reshape(m, n)[20:34, 25:41] = 1
    kw = orc.write_keepset(seed, np.zeros(1, np.int32), m, n, D_w=r_s + c)
    track = np.zeros(6, np.int32)
    for t in range(40):
        M = np.zeros((m, n), np.uint8)
        if not (10 <= t < 30):                           # vanishes for 20 frames
            y, x = rng.integers(20, 30), rng.integers(25, 37)
            M[y:y + 4, x:x + 4] = 1
            M &= seed[0].reshape(m, n)
        P = orc.prior_unit(M.reshape(-1), m, n, track, r_s, c)
        assert np.all(kw[0][P.astype(bool)] == 1), t
