"""rs3_close_argmax (Sec. 3.3: per-object closure, palette argmax, down_s of
the closed masks) and rs3_seed_from_masks (Sec. 3.1, Eq. 1: seed box and
down_s from pixel masks) against the oracle, bit for bit, through the C ABI."""
import numpy as np
import pytest

from oracle import oracle as orc
from paper_2608_22526_gb300 import synth

from _harness import to_dev, to_host

SENTINEL = 77


def _close_gpu(L, objs, R, s, want=("palette", "closed", "grid")):
    import torch
    from paper_2608_22526_gb300 import rs3
    U, h, w = L.shape
    G = len(objs)
    gs = np.concatenate([[0], np.cumsum(objs)]).astype(np.int32)
    dev = lambda shape: torch.full(shape, SENTINEL, dtype=torch.uint8, device="cuda")
    pal = dev((G, h, w)) if "palette" in want else None
    clo = dev((U, h, w)) if "closed" in want else None
    grd = dev((U, h // s, w // s)) if "grid" in want else None
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    rs3.rs3_close_argmax(to_dev(L), to_dev(gs), G, U, h, w, R, s, pal, clo, grd, status)
    torch.cuda.synchronize()
    get = lambda t: None if t is None else to_host(t)
    return get(pal), get(clo), get(grd), int(to_host(status)[0])


@pytest.mark.gpu
@pytest.mark.parametrize("objs,h,w,R,s,seed", [
    ([8], 256, 256, 4, 4, 1),             # one SAM2 stream, 8 objects, 256^2 low-res masks, 64^2 grid
    ([1, 3, 2], 100, 96, 4, 4, 2),        # ragged tiles in both directions
    ([2, 0], 37, 32, 8, 1, 3),            # largest radius, odd height, an empty stream
    ([3], 64, 288, 0, 8, 4),              # radius 0: the closure is the identity
    ([2], 40, 64, 1, 2, 5),
    ([3] * 16, 384, 384, 4, 4, 6),        # 16 streams x 3 objects, 96^2 grid
    ([4, 4], 512, 512, 3, 8, 7),          # tall tiles with a radius other than the paper's
])
def test_close_argmax_matches_oracle(objs, h, w, R, s, seed):
    rng = np.random.default_rng(1000 + seed)
    L = synth.decoder_logits(rng, sum(objs), h, w)
    pal, clo, grd, st = _close_gpu(L, objs, R, s)
    assert st == 0
    gs = np.concatenate([[0], np.cumsum(objs)])
    for g in range(len(objs)):
        c_ref, p_ref = orc.close_argmax(L[gs[g]:gs[g + 1]], R)
        assert np.array_equal(pal[g], p_ref), f"palette of stream {g}"
        assert np.array_equal(clo[gs[g]:gs[g + 1]], c_ref), f"closed masks of stream {g}"
        for o in range(objs[g]):
            assert np.array_equal(grd[gs[g] + o], orc.downsample(c_ref[o], s)), f"grid mask of unit {gs[g] + o}"


@pytest.mark.gpu
def test_close_argmax_full_resolution():
    """1024^2 decoder output (SAM2's upsampled masks), 8 objects, the 9 x 9
    closure, down_s by the encoder stride 16."""
    rng = np.random.default_rng(2024)
    L = synth.decoder_logits(rng, 8, 1024, 1024)
    pal, clo, grd, st = _close_gpu(L, [8], 4, 16)
    assert st == 0
    c_ref, p_ref = orc.close_argmax(L, 4)
    assert np.array_equal(pal[0], p_ref)
    assert np.array_equal(clo, c_ref)
    for o in range(8):
        assert np.array_equal(grd[o], orc.downsample(c_ref[o], 16))


@pytest.mark.gpu
def test_close_argmax_ties_and_optional_outputs():
    h, w = 64, 64
    L = np.full((3, h, w), -1.0, dtype=np.float32)
    L[0, 10:40, 10:40] = 2.0
    L[1, 20:50, 20:50] = 2.0              # equal logits on the overlap: object 0 keeps it
    L[2, 5:9, 50:60] = 1.0
    L[0, 15, 15] = -3.0                   # a hole the closure fills
    pal, clo, grd, st = _close_gpu(L, [3], 4, 4, want=("palette",))
    assert st == 0 and clo is None and grd is None
    _, p_ref = orc.close_argmax(L, 4)
    assert np.array_equal(pal[0], p_ref)
    assert np.all(pal[0, 20:40, 20:40] == 1) and pal[0, 15, 15] == 1
    _, clo, grd, st = _close_gpu(L, [3], 4, 4, want=("grid",))
    assert st == 0 and clo is None
    c_ref, _ = orc.close_argmax(L, 4)
    assert np.array_equal(grd[1], orc.downsample(c_ref[1], 4))


@pytest.mark.gpu
def test_close_argmax_rejects_bad_streams_on_the_device():
    """A stream whose unit range leaves [0, U] or holds more than 255 objects
    latches RS3_EINVAL and is skipped; the other streams are processed."""
    import torch
    from paper_2608_22526_gb300 import rs3
    h, w = 32, 32
    rng = np.random.default_rng(9)
    U = 300
    L = synth.decoder_logits(rng, U, h, w)
    for gs in ([0, 2, 300], [0, 2, 301]):
        gs = np.array(gs, dtype=np.int32)
        pal = torch.full((2, h, w), SENTINEL, dtype=torch.uint8, device="cuda")
        status = torch.zeros(1, dtype=torch.int32, device="cuda")
        rs3.rs3_close_argmax(to_dev(L), to_dev(gs), 2, U, h, w, 4, 1, pal, None, None, status)
        torch.cuda.synchronize()
        assert int(to_host(status)[0]) == rs3.RS3_EINVAL
        p = to_host(pal)
        assert np.array_equal(p[0], orc.close_argmax(L[0:2], 4)[1])
        assert np.all(p[1] == SENTINEL)


def _seed_gpu(M, s):
    import torch
    from paper_2608_22526_gb300 import rs3
    U, h, w = M.shape
    track = torch.full((U, 6), -5, dtype=torch.int32, device="cuda")
    grd = torch.full((U, h // s, w // s), SENTINEL, dtype=torch.uint8, device="cuda")
    box = torch.full((U, h // s, w // s), SENTINEL, dtype=torch.uint8, device="cuda")
    rs3.rs3_seed_from_masks(to_dev(M), U, h, w, s, track, grd, box)
    torch.cuda.synchronize()
    return to_host(track), to_host(grd), to_host(box)


@pytest.mark.gpu
@pytest.mark.parametrize("U,h,w,s", [(8, 1024, 1024, 16), (3, 48, 32, 16), (2, 64, 80, 1), (5, 256, 256, 4)])
def test_seed_from_masks_matches_oracle(U, h, w, s):
    rng = np.random.default_rng(U * 7 + s)
    M = synth.pixel_masks(rng, U, h, w)
    M[U - 1] = 0                                    # an object with no pixels
    if U > 1:
        M[0, h - 1, w - 1] = 9                      # an isolated pixel at the far corner
    track, grd, box = _seed_gpu(M, s)
    m, n = h // s, w // s
    for u in range(U):
        t_ref = orc.seed_track(M[u], s)
        assert list(track[u]) == list(t_ref), f"unit {u}"
        assert np.array_equal(grd[u], orc.downsample(M[u], s))
        b_ref = np.zeros((m, n), dtype=np.uint8)
        if t_ref[4]:
            b_ref[t_ref[0]:t_ref[2] + 1, t_ref[1]:t_ref[3] + 1] = 1
        assert np.array_equal(box[u], b_ref)
