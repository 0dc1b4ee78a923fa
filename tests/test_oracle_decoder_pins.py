"""Pins for the oracle's decoder-side and front-end functions: the per-object
9 x 9 closure and palette argmax of Sec. 3.3, and the down_s / seed-box
projection of Sec. 3.1.  Each test checks the oracle against a library
routine, brute force on tiny images, a closed form or an invariant.  CPU only."""
import numpy as np
import pytest

from oracle import oracle as orc


def _rng(seed):
    return np.random.default_rng(seed)


def _plane_closing_scipy(M, r):
    """Closing in the unbounded plane through scipy: a zero frame 2r wide,
    scipy's binary closing with the (2r+1)^2 square, then the frame removed."""
    nd = pytest.importorskip("scipy.ndimage")
    if r == 0:
        return M.astype(np.uint8)
    h, w = M.shape
    P = np.zeros((h + 4 * r, w + 4 * r), dtype=bool)
    P[2 * r:2 * r + h, 2 * r:2 * r + w] = M.astype(bool)
    C = nd.binary_closing(P, structure=np.ones((2 * r + 1, 2 * r + 1), dtype=bool))
    return C[2 * r:2 * r + h, 2 * r:2 * r + w].astype(np.uint8)


def _plane_closing_brute(M, r):
    """p is in the closing iff every (2r+1)^2 window of the plane that holds p
    also holds a set pixel (pixels outside the image are unset)."""
    h, w = M.shape
    out = np.zeros((h, w), dtype=np.uint8)
    for py in range(h):
        for px in range(w):
            keep = 1
            for ty in range(py - 2 * r, py + 1):
                for tx in range(px - 2 * r, px + 1):
                    hit = False
                    for y in range(max(ty, 0), min(ty + 2 * r, h - 1) + 1):
                        for x in range(max(tx, 0), min(tx + 2 * r, w - 1) + 1):
                            if M[y, x]:
                                hit = True
                                break
                        if hit:
                            break
                    if not hit:
                        keep = 0
                        break
                if not keep:
                    break
            out[py, px] = keep
    return out


# ---------------------------------------------------------------------------
# closure (Sec. 3.3)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("r", [0, 1, 2, 4, 8])
@pytest.mark.parametrize("density", [0.1, 0.5, 0.9])
def test_close_matches_scipy_plane_closing(r, density):
    rng = _rng(100 + r)
    for h, w in [(37, 45), (9, 64), (70, 13)]:
        M = (rng.random((h, w)) < density).astype(np.uint8)
        assert np.array_equal(orc.close(M, h, w, r), _plane_closing_scipy(M, r))


@pytest.mark.parametrize("r", [1, 2])
def test_close_matches_brute_force_windows(r):
    rng = _rng(7 + r)
    for h, w in [(9, 11), (6, 7)]:
        for density in (0.2, 0.6):
            M = (rng.random((h, w)) < density).astype(np.uint8)
            assert np.array_equal(orc.close(M, h, w, r), _plane_closing_brute(M, r))


def test_close_invariants():
    rng = _rng(3)
    h, w = 48, 40
    for density in (0.05, 0.3, 0.7):
        M = (rng.random((h, w)) < density).astype(np.uint8)
        C = orc.close(M, h, w, 4)
        assert np.all(C >= M)                                    # extensive
        assert np.array_equal(orc.close(C, h, w, 4), C)          # idempotent
        M2 = np.maximum(M, (rng.random((h, w)) < 0.1).astype(np.uint8))
        assert np.all(orc.close(M2, h, w, 4) >= C)               # monotone
        assert np.array_equal(orc.close(M, h, w, 0), M)          # r = 0: identity


@pytest.mark.parametrize("box", [(5, 6, 20, 30), (0, 0, 10, 12), (30, 25, 47, 39), (0, 3, 47, 3), (17, 0, 17, 39)])
def test_close_keeps_rectangles(box):
    """A rectangle (also one touching the border, or one pixel thin) is its
    own closing: the outer boundary does not grow."""
    h, w = 48, 40
    M = np.zeros((h, w), dtype=np.uint8)
    y0, x0, y1, x1 = box
    M[y0:y1 + 1, x0:x1 + 1] = 1
    assert np.array_equal(orc.close(M, h, w, 4), M)


@pytest.mark.parametrize("side,filled", [(1, True), (8, True), (9, False), (12, False)])
def test_close_fills_holes_smaller_than_the_element(side, filled):
    h, w = 64, 64
    M = np.ones((h, w), dtype=np.uint8)
    M[20:20 + side, 25:25 + side] = 0
    C = orc.close(M, h, w, 4)
    assert np.array_equal(C, np.ones_like(M) if filled else M)


@pytest.mark.parametrize("gap,bridged", [(1, True), (8, True), (9, False)])
def test_close_reknits_gaps(gap, bridged):
    h, w = 40, 60
    M = np.zeros((h, w), dtype=np.uint8)
    M[10:30, 5:20] = 1
    M[10:30, 20 + gap:45] = 1
    hull = np.zeros_like(M)
    hull[10:30, 5:45] = 1
    assert np.array_equal(orc.close(M, h, w, 4), hull if bridged else M)


# ---------------------------------------------------------------------------
# palette argmax after the closure (Sec. 3.3)
# ---------------------------------------------------------------------------

def _palette_brute(L, r):
    nobj, h, w = L.shape
    closed = np.stack([_plane_closing_scipy(L[o] > 0, r) for o in range(nobj)])
    pal = np.zeros((h, w), dtype=np.uint8)
    for y in range(h):
        for x in range(w):
            best = -1
            for o in range(nobj):
                if closed[o, y, x] and (best < 0 or L[o, y, x] > L[best, y, x]):
                    best = o
            pal[y, x] = best + 1
    return closed, pal


@pytest.mark.parametrize("r", [1, 4])
def test_palette_matches_per_pixel_loop(r):
    rng = _rng(11 + r)
    nobj, h, w = 3, 24, 32
    L = rng.normal(-0.3, 1.0, size=(nobj, h, w)).astype(np.float32)
    L[1, 5:15, 5:20] = np.abs(L[1, 5:15, 5:20]) + 0.1
    L[2, 10:20, 12:28] = np.abs(L[2, 10:20, 12:28]) + 0.1
    L[2, 12, 14] = L[1, 12, 14] = 1.5                         # an exact tie
    closed, pal = orc.close_argmax(L, r)
    c_ref, p_ref = _palette_brute(L, r)
    assert np.array_equal(closed, c_ref)
    assert np.array_equal(pal, p_ref)
    assert pal[12, 14] == 2                                     # tie -> lower object


def test_palette_single_and_disjoint_objects():
    h, w = 50, 60
    L = np.full((2, h, w), -1.0, dtype=np.float32)
    L[0, 5:20, 5:20] = 2.0
    L[0, 10, 10] = -1.0                                          # a hole the closure fills
    L[1, 30:45, 35:55] = 0.5
    closed, pal = orc.close_argmax(L[:1], 4)
    assert np.array_equal(pal, closed[0])
    assert pal[10, 10] == 1
    closed, pal = orc.close_argmax(L, 4)
    assert np.array_equal(pal, closed[0] * 1 + closed[1] * 2)


def test_palette_threshold_is_strict_and_background_is_zero():
    L = np.zeros((2, 16, 16), dtype=np.float32)                 # logit 0 is not set
    closed, pal = orc.close_argmax(L, 4)
    assert closed.sum() == 0 and pal.sum() == 0
    L[1, 4:8, 4:8] = 1e-30
    closed, pal = orc.close_argmax(L, 4)
    assert set(np.unique(pal)) == {0, 2} and (pal == 2).sum() == 16


def test_palette_overlap_goes_to_the_larger_logit():
    h, w = 32, 32
    L = np.full((3, h, w), -2.0, dtype=np.float32)
    L[0, 4:20, 4:20] = 1.0
    L[2, 10:28, 10:28] = 3.0
    _, pal = orc.close_argmax(L, 4)
    assert np.all(pal[10:20, 10:20] == 3)
    assert np.all(pal[4:10, 4:20] == 1) and np.all(pal[20:28, 20:28] == 3)
    assert not np.any(pal == 2)


# ---------------------------------------------------------------------------
# down_s and the seed box (Sec. 3.1, Eq. 1)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("s", [1, 4, 16])
def test_downsample_takes_the_top_left_pixel(s):
    rng = _rng(s)
    m, n = 6, 5
    pattern = (rng.random((m, n)) < 0.5).astype(np.uint8)
    M = (rng.random((m * s, n * s)) < 0.5).astype(np.uint8)
    for i in range(m):
        for j in range(n):
            M[i * s, j * s] = pattern[i, j] * (1 + (i + j) % 3)      # any non-zero value is set
    assert np.array_equal(orc.downsample(M, s), pattern)


@pytest.mark.parametrize("s", [1, 4, 16])
def test_seed_track_projects_the_pixel_box(s):
    rng = _rng(40 + s)
    h, w = 4 * 16, 3 * 16
    for _ in range(5):
        M = np.zeros((h, w), dtype=np.uint8)
        ys = rng.integers(0, h, size=4)
        xs = rng.integers(0, w, size=4)
        M[ys, xs] = 7
        t = orc.seed_track(M, s)
        assert list(t) == [ys.min() // s, xs.min() // s, ys.max() // s, xs.max() // s, 1, 0]
    M = np.zeros((h, w), dtype=np.uint8)
    assert list(orc.seed_track(M, s)) == [0, 0, 0, 0, 0, 0]
    M[h - 1, w - 1] = 1
    assert list(orc.seed_track(M, s)) == [(h - 1) // s, (w - 1) // s, (h - 1) // s, (w - 1) // s, 1, 0]


# ---------------------------------------------------------------------------
# the seeded pixel-resolution inputs the GPU tests and the benchmark share
# ---------------------------------------------------------------------------

def test_decoder_logits_are_seeded_and_shaped_like_the_recipe():
    from paper_2608_22526_gb300 import synth
    a = synth.decoder_logits(np.random.default_rng(5), 3, 64, 96)
    b = synth.decoder_logits(np.random.default_rng(5), 3, 64, 96)
    assert a.shape == (3, 64, 96) and a.dtype == np.float32 and np.array_equal(a, b)
    assert np.all(np.abs(a) >= 0.5)                      # no logit on the threshold
    cov = (a > 0).mean(axis=(1, 2))
    assert np.all(cov > 0.005) and np.all(cov < 0.35)
    # the salt-and-pepper holes are there for the closure to fill
    closed = np.stack([orc.close(a[o] > 0, 64, 96, 4) for o in range(3)])
    assert (closed.astype(int) - (a > 0)).sum() > 0


def test_pixel_masks_are_seeded():
    from paper_2608_22526_gb300 import synth
    a = synth.pixel_masks(np.random.default_rng(8), 4, 128, 64)
    b = synth.pixel_masks(np.random.default_rng(8), 4, 128, 64)
    assert a.shape == (4, 128, 64) and a.dtype == np.uint8 and np.array_equal(a, b)
    assert set(np.unique(a)) <= {0, 255} and np.all(a.reshape(4, -1).max(axis=1) == 255)
