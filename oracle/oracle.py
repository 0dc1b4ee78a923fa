"""CPU oracle for the RS3-Prune hot path (Python side).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg are the only callers.  Nothing here is imported by
the CUDA library or its binding, and nothing here imports them.

The arithmetic lives in ``rs3_oracle.c`` (fp64 explicit loops); this module
builds that file with gcc, marshals numpy arrays, and models the per-unit
memory bank.  Each function cites the part of the paper it follows:

  select()         Sec. 3.1: Eq. 1 / Eq. 2 / Eq. 4 priors, Eq. 5 top-k
  readout()        Sec. 3.1: Eq. 6 sparse memory attention, Eq. 7 RoPE gather
  scatter_output() Sec. 3.1: Eq. 6 scatter S_K back onto the m x n grid
  OracleBank       Sec. 3.2: Eq. 8 write-pruned commit, Algorithm 1 sparse write
  rotate_rows()    Sec. 3.1: Eq. 7 on the key side (keys rotated by their own cell)
  write_keepset()  Sec. 3.2: Eq. 8 with the 5% / 95% fall-through
  close_argmax()   Sec. 3.3: 9 x 9 closure per object, then the palette argmax
  downsample(), seed_track()
                   Sec. 3.1: down_s of pixel masks, the seed box of Eq. 1
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import List, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "rs3_oracle.c")
_SO = os.path.join(_HERE, "librs3_oracle.so")
_lock = threading.Lock()
_handle = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no FP contraction, so fp64 expressions mean
    exactly what they say on every host)."""
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
               "-shared", "-pthread", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _SO)
    return _SO


def _lib():
    global _handle
    with _lock:
        if _handle is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32, i64, f64 = ctypes.c_int, ctypes.c_long, ctypes.c_double
            lib.or_bbox.argtypes = [P, i32, i32, P]
            lib.or_bbox.restype = i32
            lib.or_dilate.argtypes = [P, i32, i32, i32, P]
            lib.or_prior_unit.argtypes = [P, i32, i32, P, i32, i32, i32, P]
            lib.or_energy_canonical.argtypes = [P, i64, i32, P]
            lib.or_energy_exact.argtypes = [P, i64, i32, P]
            lib.or_kmax.argtypes = [f64, i64]
            lib.or_kmax.restype = i64
            lib.or_topk.argtypes = [P, P, i64, i64, P]
            lib.or_topk.restype = i64
            lib.or_select.argtypes = [P, i32, i32, i32, i32, P, P, i32, P, f64, i32, i32,
                                      i32, i32, P, P, P, P]
            lib.or_readout.argtypes = [P, i64, i32, i32, P, i64, P, P, i64, P, f64, P, i32]
            lib.or_round_bf16_array.argtypes = [P, i64, P]
            lib.or_write_keepset.argtypes = [P, P, i32, i32, i32, i32, f64, f64, i32, i32, P]
            lib.or_commit_unit.argtypes = [P, P, i64, P, P, P, i64, i32, i32, i64, i64, i32,
                                           P, P, P]
            lib.or_commit_unit.restype = i32
            lib.or_erode.argtypes = [P, i32, i32, i32, P]
            lib.or_close.argtypes = [P, i32, i32, i32, P]
            lib.or_close_argmax.argtypes = [P, i32, i32, i32, i32, P, P]
            lib.or_downsample.argtypes = [P, i32, i32, i32, P]
            lib.or_seed_track.argtypes = [P, i32, i32, i32, P]
            lib.or_seed_track.restype = i32
            _handle = lib
    return _handle


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


# ---------------------------------------------------------------------------
# value conversion (the oracle's own)
# ---------------------------------------------------------------------------

def widen(x: np.ndarray, dtype: str) -> np.ndarray:
    """Stored values -> fp32 numbers: bf16 bit patterns widen exactly."""
    if dtype == "bf16":
        b = np.ascontiguousarray(x, dtype=np.uint16)
        return (b.astype(np.uint32) << np.uint32(16)).view(np.float32)
    return np.ascontiguousarray(x, dtype=np.float32)


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """fp64 -> output dtype with one rounding (nearest-even)."""
    x = _c(x, np.float64)
    if dtype == "bf16":
        out = np.empty(x.shape, dtype=np.uint16)
        _lib().or_round_bf16_array(_p(x), x.size, _p(out))
        return out
    return x.astype(np.float32)   # IEEE fp64 -> fp32 conversion rounds to nearest-even


# ---------------------------------------------------------------------------
# read side (Sec. 3.1)
# ---------------------------------------------------------------------------

def kmax(rho: float, mn: int) -> int:
    """k = floor(rho * mn): Table 4's |K_r|max column (819, 1228, 2048, 2867,
    4096 at mn = 4096)."""
    return int(_lib().or_kmax(float(rho), int(mn)))


def bbox(M: np.ndarray, m: int, n: int):
    box = np.zeros(4, dtype=np.int32)
    ok = _lib().or_bbox(_p(_c(M, np.uint8)), m, n, _p(box))
    return tuple(int(v) for v in box) if ok else None


def dilate(M: np.ndarray, m: int, n: int, r: int) -> np.ndarray:
    Mc = _c(M, np.uint8).reshape(-1)
    out = np.empty(m * n, dtype=np.uint8)
    _lib().or_dilate(_p(Mc), m, n, int(r), _p(out))
    return out


def prior_unit(M: np.ndarray, m: int, n: int, track: np.ndarray, r_s: int, c: int,
               bbox_mode: int = 0) -> np.ndarray:
    """Eq. 2 (or Eq. 1 in bbox mode) when M is non-empty, Eq. 4 otherwise;
    `track` (int32[6]: y0, x0, y1, x1, valid, streak) is updated in place."""
    assert track.dtype == np.int32 and track.flags.c_contiguous
    out = np.empty(m * n, dtype=np.uint8)
    _lib().or_prior_unit(_p(_c(M, np.uint8)), m, n, _p(track), int(r_s), int(c),
                         int(bbox_mode), _p(out))
    return out


def energy_canonical(z32: np.ndarray) -> np.ndarray:
    z = _c(z32, np.float32)
    rows, C = z.reshape(-1, z.shape[-1]).shape
    e = np.empty(rows, dtype=np.float32)
    _lib().or_energy_canonical(_p(z), rows, C, _p(e))
    return e


def energy_exact(z32: np.ndarray) -> np.ndarray:
    z = _c(z32, np.float32)
    rows, C = z.reshape(-1, z.shape[-1]).shape
    e = np.empty(rows, dtype=np.float64)
    _lib().or_energy_exact(_p(z), rows, C, _p(e))
    return e


def topk(P: np.ndarray, e: np.ndarray, k: int) -> np.ndarray:
    P = _c(P, np.uint8)
    e = _c(e, np.float32)
    idx = np.empty(max(k, 1), dtype=np.int32)
    cnt = _lib().or_topk(_p(P), _p(e), P.size, int(k), _p(idx))
    return idx[:cnt].copy()


class SelectResult:
    def __init__(self, idx, count, prior, energy, k):
        self.idx = idx          # int32 [U, k]
        self.count = count      # int32 [U]
        self.prior = prior      # uint8 [U, mn]
        self.energy = energy    # float32 [G, mn]
        self.k = k

    def keep(self, u: int) -> np.ndarray:
        return self.idx[u, : self.count[u]]


def select(z: np.ndarray, dtype: str, masks: np.ndarray, unit_group: np.ndarray,
           track: np.ndarray, m: int, n: int, rho: float, r_s: int, c: int,
           union_mode: int, bbox_mode: int = 0) -> SelectResult:
    """Read-side selection of one frame (Algorithm 1 up to the arg-top):
    z [G, mn, C] (stored dtype), masks [U, mn] of the previous frame,
    track [U, 6] int32 updated in place."""
    zf = widen(z, dtype)
    G, mn, C = zf.shape
    U = masks.shape[0]
    k = kmax(rho, mn)
    idx = np.zeros((U, max(k, 1)), dtype=np.int32)
    count = np.zeros(U, dtype=np.int32)
    prior = np.zeros((U, mn), dtype=np.uint8)
    energy = np.zeros((G, mn), dtype=np.float32)
    assert track.dtype == np.int32 and track.shape == (U, 6) and track.flags.c_contiguous
    _lib().or_select(_p(zf), G, m, n, C, _p(_c(masks, np.uint8)),
                     _p(_c(unit_group, np.int32)), U, _p(track), float(rho), int(r_s),
                     int(c), int(union_mode), int(bbox_mode), _p(idx), _p(count), _p(prior),
                     _p(energy))
    return SelectResult(idx[:, :k] if k > 0 else idx[:, :0], count, prior, energy, k)


def readout(q: np.ndarray, dtype: str, H: int, d: int, idx: np.ndarray, K: np.ndarray,
            V: np.ndarray, bank_dtype: str, rope: Optional[np.ndarray] = None,
            scale: Optional[float] = None, threads: int = 1) -> np.ndarray:
    """Eq. 6 with Eq. 7: A[j] = softmax(q~_j K^T * scale) V per head, in fp64.
    q [mn, H*d] (stored dtype); idx [cnt]; K, V [N, H*d] logical bank rows."""
    qd = widen(q, dtype).astype(np.float64)
    Kd = widen(K, bank_dtype).astype(np.float64).reshape(-1, H * d)
    Vd = widen(V, bank_dtype).astype(np.float64).reshape(-1, H * d)
    idx = _c(idx, np.int32)
    cnt = idx.size
    if scale is None or scale == 0.0:
        scale = 1.0 / np.sqrt(float(d))
    A = np.zeros((cnt, H * d), dtype=np.float64)
    rp = None if rope is None else _c(rope, np.float32)
    _lib().or_readout(_p(qd), qd.shape[0], H, d, _p(idx), cnt, _p(Kd), _p(Vd), Kd.shape[0],
                      _p(rp), float(scale), _p(A), int(threads))
    return A


def scatter_output(residual: Optional[np.ndarray], dtype: str, mn: int, D: int,
                   idx: np.ndarray, A: np.ndarray) -> np.ndarray:
    """Eq. 6's scatter S_K: the grid output is the residual (zeros when there is
    none) with A added at the kept cells, rounded once to the output dtype."""
    if residual is None:
        base = np.zeros((mn, D), dtype=np.float64)
        out = round_to(base, dtype)
    else:
        out = np.array(residual, copy=True).reshape(mn, D)
        base = widen(out, dtype).astype(np.float64)
    if idx.size:
        out[idx] = round_to(base[idx] + A, dtype)
    return out


# ---------------------------------------------------------------------------
# write side (Sec. 3.2)
# ---------------------------------------------------------------------------

def rotate_rows(x: np.ndarray, dtype: str, rope: np.ndarray) -> np.ndarray:
    """Eq. 7 applied to the keys: row i of x [mn, H*d] (stored dtype) rotated
    by the table entries of its own cell i -- in every head, elements
    (2p, 2p+1) turn by the angle whose (cos, sin) is rope[i, p] -- in fp64,
    then rounded once to the stored dtype.  rope: [mn, d/2, 2]."""
    rope = np.asarray(rope, dtype=np.float64)
    mn, half = rope.shape[0], rope.shape[1]
    xd = widen(x, dtype).astype(np.float64).reshape(mn, -1, half, 2)      # [mn, H, d/2, (even, odd)]
    cs = rope[:, None, :, 0]
    sn = rope[:, None, :, 1]
    ev, od = xd[..., 0], xd[..., 1]
    y = np.stack([ev * cs - od * sn, ev * sn + od * cs], axis=-1)
    return round_to(y.reshape(mn, -1), dtype)


def write_keepset(seeds: np.ndarray, unit_group: np.ndarray, m: int, n: int, D_w: int,
                  fall_lo: float = 0.05, fall_hi: float = 0.95, fall_through: int = 1,
                  union_mode: int = 1) -> np.ndarray:
    S = _c(seeds, np.uint8)
    U = S.shape[0]
    kw = np.empty((U, m * n), dtype=np.uint8)
    _lib().or_write_keepset(_p(S), _p(_c(unit_group, np.int32)), U, m, n, int(D_w),
                            float(fall_lo), float(fall_hi), int(fall_through),
                            int(union_mode), _p(kw))
    return kw


class OracleBank:
    """Per-unit memory bank (K, V): pinned conditioning frames, a ring of recent
    frames (window eviction keeps the newest `window`), and pointer rows.
    Storage per unit: pinned_cap = n_cond * mn rows, then ring_cap rows, then
    n_ptr pointer rows."""

    def __init__(self, U: int, D: int, dtype: str, mn: int, n_cond: int, window: int,
                 ring_cap: int, max_frames: int, n_ptr: int):
        self.U, self.D, self.dtype, self.mn = U, D, dtype, mn
        self.n_cond, self.window, self.n_ptr = n_cond, window, n_ptr
        self.pinned_cap = n_cond * mn
        self.ring_cap = ring_cap
        self.max_frames = max_frames
        self.rows = self.pinned_cap + ring_cap + n_ptr
        self.npdt = np.uint16 if dtype == "bf16" else np.float32
        self.K = np.zeros((U, self.rows, D), dtype=self.npdt)
        self.V = np.zeros((U, self.rows, D), dtype=self.npdt)
        self.state = np.zeros((U, 8), dtype=np.int64)
        self.state[:, 7] = n_cond
        self.foff = np.zeros((U, max(max_frames, 1)), dtype=np.int64)
        self.flen = np.zeros((U, max(max_frames, 1)), dtype=np.int32)
        self.ptr_len = np.zeros(U, dtype=np.int64)

    def reset(self, unit: int = -1):
        us = range(self.U) if unit < 0 else [unit]
        for u in us:
            self.state[u, :7] = 0
            self.ptr_len[u] = 0

    def commit(self, knew: np.ndarray, vnew: np.ndarray, mask: Optional[np.ndarray],
               is_cond: int, rope: Optional[np.ndarray] = None) -> List[int]:
        """Algorithm 1's sparse write for every unit: rows with mask = 1, in
        ascending grid order.  With a RoPE table every key row is first rotated
        by its own cell (rotate_rows), so the bank holds rotated keys.  Returns
        the per-unit status (0 or 2 = capacity)."""
        if rope is not None:
            knew = np.stack([rotate_rows(knew[u], self.dtype, rope) for u in range(self.U)])
        st = []
        row_bytes = self.D * np.dtype(self.npdt).itemsize
        for u in range(self.U):
            kn = _c(knew[u], self.npdt)
            vn = _c(vnew[u], self.npdt)
            mk = None if mask is None else _c(mask[u], np.uint8)
            Ku = self.K[u]
            Vu = self.V[u]
            s = _c(self.state[u], np.int64)
            fo = _c(self.foff[u], np.int64)
            fl = _c(self.flen[u], np.int32)
            rc = _lib().or_commit_unit(_p(Ku), _p(Vu), row_bytes, _p(kn), _p(vn), _p(mk),
                                       self.mn, int(is_cond), int(self.window),
                                       self.pinned_cap, self.ring_cap, self.max_frames,
                                       _p(s), _p(fo), _p(fl))
            self.state[u] = s
            self.foff[u] = fo
            self.flen[u] = fl
            st.append(int(rc))
        return st

    def set_pointers(self, kp: np.ndarray, vp: np.ndarray):
        base = self.pinned_cap + self.ring_cap
        for u in range(self.U):
            self.K[u, base: base + self.n_ptr] = kp[u]
            self.V[u, base: base + self.n_ptr] = vp[u]
            self.ptr_len[u] = self.n_ptr

    # -- views ---------------------------------------------------------------
    def ring_rows(self, u: int) -> np.ndarray:
        """Physical row numbers of the ring frames, oldest first."""
        head, tail = int(self.state[u, 0]), int(self.state[u, 1])
        return self.pinned_cap + (np.arange(head, tail, dtype=np.int64) % max(self.ring_cap, 1))

    def logical_rows(self, u: int) -> np.ndarray:
        """Physical row numbers of the unit's bank in logical order: pinned
        frames, ring frames oldest first, pointer rows."""
        cond = np.arange(int(self.state[u, 2]), dtype=np.int64)
        ptr = self.pinned_cap + self.ring_cap + np.arange(int(self.ptr_len[u]), dtype=np.int64)
        return np.concatenate([cond, self.ring_rows(u), ptr])

    def kv(self, u: int):
        r = self.logical_rows(u)
        return self.K[u][r], self.V[u][r]

    def length(self, u: int) -> int:
        return int(self.state[u, 2] + (self.state[u, 1] - self.state[u, 0]) + self.ptr_len[u])

    def frames(self, u: int):
        """[(logical offset, length)] of the ring frames, oldest first."""
        n, o = int(self.state[u, 3]), int(self.state[u, 4])
        return [(int(self.foff[u, (o + i) % self.max_frames]),
                 int(self.flen[u, (o + i) % self.max_frames])) for i in range(n)]


# ---------------------------------------------------------------------------
# decoder side (Sec. 3.3) and the pixel-space front end (Sec. 3.1)
# ---------------------------------------------------------------------------

def erode(M: np.ndarray, h: int, w: int, r: int) -> np.ndarray:
    """Square erosion by r with the window clipped to the image."""
    out = np.empty(h * w, dtype=np.uint8)
    _lib().or_erode(_p(_c(M, np.uint8)), h, w, int(r), _p(out))
    return out.reshape(h, w)


def close(M: np.ndarray, h: int, w: int, r: int) -> np.ndarray:
    """close_r(M) = erode_r(dilate_r(M)) (Sec. 3.3: r = 4, the 9 x 9 square)."""
    out = np.empty(h * w, dtype=np.uint8)
    _lib().or_close(_p(_c(M, np.uint8)), h, w, int(r), _p(out))
    return out.reshape(h, w)


def close_argmax(logits: np.ndarray, r: int):
    """One group: logits [nobj, h, w] fp32 -> (closed [nobj, h, w] uint8,
    palette [h, w] uint8 with 0 = background and 1 + o = object o)."""
    L = _c(logits, np.float32)
    nobj, h, w = L.shape
    closed = np.empty((nobj, h, w), dtype=np.uint8)
    palette = np.empty((h, w), dtype=np.uint8)
    _lib().or_close_argmax(_p(L), nobj, h, w, int(r), _p(closed), _p(palette))
    return closed, palette


def downsample(M: np.ndarray, s: int) -> np.ndarray:
    """down_s: grid cell (i, j) takes pixel (i*s, j*s); [h, w] -> [h/s, w/s]."""
    M = _c(M, np.uint8)
    h, w = M.shape
    out = np.empty((h // s, w // s), dtype=np.uint8)
    _lib().or_downsample(_p(M), h, w, int(s), _p(out))
    return out


def seed_track(M: np.ndarray, s: int) -> np.ndarray:
    """The seed box of Eq. 1 on the grid: int32 [6] = (y0, x0, y1, x1, valid,
    streak) from the tight pixel box of M, corners divided by s (floor)."""
    M = _c(M, np.uint8)
    h, w = M.shape
    t = np.zeros(6, dtype=np.int32)
    _lib().or_seed_track(_p(M), h, w, int(s), _p(t))
    return t
