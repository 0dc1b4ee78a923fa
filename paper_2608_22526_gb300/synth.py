"""Seeded synthetic workloads shaped like the paper's SAM2-style VOS inputs.

This module only draws random inputs; it holds none of the method's
arithmetic (no dilation, no energy, no selection, no attention).  Both the CUDA
path and the CPU oracle consume exactly the arrays produced here.

Stand-ins (the paper's datasets and checkpoints are not available):
  * encoder token grid Z_t [mn, C] (Sec. 3, the output of the image encoder,
    stride s=16, so a 1024x1024 frame gives a 64x64 grid): N(0,1), scaled by
    1.25 on cells inside any of the group's current object masks so that object
    tokens carry more energy, as Sec. 3.1 argues they do on real encoders;
  * queries q_t = Z_t (identity projection);
  * memory-encoder output K_t, V_t [mn, D] per unit: N(0,1);
  * per-object masks at grid resolution: filled ellipses whose centre drifts
    with a bounded velocity (reflecting at the borders) and whose area sweeps
    the configured coverage range along the sequence;
  * RoPE table f [mn, d/2] as (cos, sin), 2-D axial frequencies (Sec. 3.1, Eq. 7
    uses a table indexed by grid position).

bf16 tensors are produced as uint16 bit patterns, rounded to nearest-even from
fp32, so that every consumer starts from the same bits.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional

import numpy as np


# ----------------------------------------------------------------------------
# bf16 helpers (bit-pattern conversion only)
# ----------------------------------------------------------------------------

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (nearest-even) and return the uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    rounding = ((u >> np.uint64(16)) & np.uint64(1)) + np.uint64(0x7FFF)
    return ((u + rounding) >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp32."""
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# ----------------------------------------------------------------------------
# Workload configurations
# ----------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic workload.  A *unit* is one (stream, object) pair; a *group*
    is the set of units that share one query grid (the objects of one stream).
    """
    name: str
    cid: int              # config id, also the seed offset
    m: int
    n: int
    H: int                # heads
    d: int                # head dim
    dtype: str            # "f32" or "bf16"
    G: int                # groups (streams)
    units_per_group: int  # objects per stream
    frames: int
    cov_lo: float         # mask coverage range (fraction of mn)
    cov_hi: float
    n_cond: int           # pinned conditioning frames per unit bank
    window: int           # non-pinned frames held (-1 = unbounded)
    n_ptr: int            # pointer rows per unit
    prefill_frames: int = 0   # unpruned frames committed before the sequence
    union_mode: int = 0       # 1: one prior per group (union over its objects)
    rho: float = 0.3
    r_s: int = 4
    c: int = 14
    seed_base: int = 20260

    @property
    def mn(self) -> int:
        return self.m * self.n

    @property
    def D(self) -> int:
        return self.H * self.d

    @property
    def C(self) -> int:
        return self.H * self.d

    @property
    def U(self) -> int:
        return self.G * self.units_per_group

    @property
    def seed(self) -> int:
        return self.seed_base + self.cid

    def unit_group(self) -> np.ndarray:
        return np.repeat(np.arange(self.G, dtype=np.int32), self.units_per_group)

    def ring_cap_rows(self) -> int:
        """Ring rows per unit that always hold the configured window."""
        if self.window > 0:
            return self.window * self.mn
        # unbounded: every frame of the sequence plus the prefill, at full size
        return (self.frames + self.prefill_frames) * self.mn

    def ring_cap_rows_tight(self) -> int:
        """Unbounded banks sized from the coverage bound instead of mn."""
        if self.window > 0:
            return self.ring_cap_rows()
        per = int(math.ceil(self.cov_hi * 1.10 * self.mn)) + 8
        return self.prefill_frames * self.mn + self.frames * min(per, self.mn)

    def max_frames(self) -> int:
        if self.window > 0:
            return self.window
        return self.frames + self.prefill_frames


WORKLOADS = {
    # tiny single step, fp32: 32x32 grid, 1 head x 64; bank = 2 unpruned frames
    "tiny_fp32": Workload("tiny_fp32", 1, 32, 32, 1, 64, "f32", 1, 1, 1,
                          0.08, 0.12, 0, -1, 0, prefill_frames=2),
    # SAM2-shaped single object, bf16: 64x64, 1 head x 256, cond + 6 recent
    # frames write-pruned to their masks + 16 pointer rows, 60 frames
    "sam2_1obj": Workload("sam2_1obj", 2, 64, 64, 1, 256, "bf16", 1, 1, 60,
                          0.05, 0.30, 1, 6, 16),
    # 8 objects on one 64x64 grid, per-object banks of 7 frames, 100 frames
    "sam2_8obj": Workload("sam2_8obj", 3, 64, 64, 1, 256, "bf16", 1, 8, 100,
                          0.02, 0.40, 1, 6, 0),
    # long video: 1 object, 1000 frames, unbounded write-pruned bank (~15%)
    "long_video": Workload("long_video", 4, 64, 64, 1, 256, "bf16", 1, 1, 1000,
                           0.14, 0.16, 1, -1, 0),
    # 16 streams x 3 objects, 96x96 grid, 4 heads x 64, 7 frames + 16 pointers
    "multistream": Workload("multistream", 5, 96, 96, 4, 64, "bf16", 16, 3, 200,
                            0.03, 0.25, 1, 6, 16),
}

CONFIG_ORDER = ["tiny_fp32", "sam2_1obj", "sam2_8obj", "long_video", "multistream"]


def scaled(w: Workload, frames: Optional[int] = None, G: Optional[int] = None,
           units_per_group: Optional[int] = None, m: Optional[int] = None,
           n: Optional[int] = None, name_suffix: str = "_small") -> Workload:
    """A reduced copy of a workload (fewer frames / streams) with the same
    per-frame structure, for the oracle-sized parity cases."""
    kw = {}
    if frames is not None:
        kw["frames"] = frames
    if G is not None:
        kw["G"] = G
    if units_per_group is not None:
        kw["units_per_group"] = units_per_group
    if m is not None:
        kw["m"] = m
    if n is not None:
        kw["n"] = n
    return dataclasses.replace(w, name=w.name + name_suffix, **kw)


# ----------------------------------------------------------------------------
# Mask trajectories
# ----------------------------------------------------------------------------

def ellipse_mask(m: int, n: int, cy: float, cx: float, a: float, b: float,
                 theta: float) -> np.ndarray:
    """Filled ellipse on the m x n grid.  Cell (y, x) is inside iff its centre
    (y+0.5, x+0.5) satisfies the rotated-ellipse inequality (fp64)."""
    yy, xx = np.mgrid[0:m, 0:n].astype(np.float64)
    u = xx + 0.5 - cx
    v = yy + 0.5 - cy
    ct, st = math.cos(theta), math.sin(theta)
    xr = (u * ct + v * st) / a
    yr = (-u * st + v * ct) / b
    return ((xr * xr + yr * yr) <= 1.0).astype(np.uint8)


@dataclasses.dataclass
class Trajectory:
    cy: np.ndarray
    cx: np.ndarray
    a: np.ndarray
    b: np.ndarray
    theta: np.ndarray
    visible: np.ndarray   # bool per frame (False = empty mask)


def make_trajectory(rng: np.random.Generator, m: int, n: int, frames: int,
                    cov_lo: float, cov_hi: float,
                    vanish: Optional[List[range]] = None) -> Trajectory:
    """Drifting ellipse: |velocity| <= 1.5 cells/frame, reflecting so that the
    ellipse stays on the grid; its coverage sweeps [cov_lo, cov_hi] along the
    sequence (a sinusoid of random phase and a period near the length)."""
    mn = m * n
    # coverage sweeps the configured range along the sequence (random phase)
    phase = rng.uniform(0.0, 2 * math.pi)
    period = rng.uniform(0.8, 1.2) * max(30, frames)
    aspect = rng.uniform(0.6, 1.6)
    theta = rng.uniform(0.0, math.pi)
    speed = rng.uniform(0.3, 1.5)
    ang = rng.uniform(0.0, 2 * math.pi)
    vy, vx = speed * math.sin(ang), speed * math.cos(ang)
    cy = rng.uniform(0.4 * m, 0.6 * m)
    cx = rng.uniform(0.4 * n, 0.6 * n)
    out = {k: np.zeros(frames) for k in ("cy", "cx", "a", "b", "theta")}
    for t in range(frames):
        cov = cov_lo + (cov_hi - cov_lo) * 0.5 * (1.0 + math.sin(phase + 2 * math.pi * t / period))
        area = cov * mn
        a = math.sqrt(area * aspect / math.pi)
        b = math.sqrt(area / (aspect * math.pi))
        out["cy"][t], out["cx"][t] = cy, cx
        out["a"][t], out["b"][t], out["theta"][t] = a, b, theta
        # advance
        theta += rng.normal(0.0, 0.05)
        vy += rng.normal(0.0, 0.15)
        vx += rng.normal(0.0, 0.15)
        sp = math.hypot(vy, vx)
        if sp > 1.5:
            vy, vx = vy * 1.5 / sp, vx * 1.5 / sp
        cy += vy
        cx += vx
        # keep the whole ellipse on the grid (half-extents of the rotated
        # ellipse's bounding box), reflecting the velocity at the borders
        ct, st = math.cos(theta), math.sin(theta)
        hx = math.sqrt((a * ct) ** 2 + (b * st) ** 2)
        hy = math.sqrt((a * st) ** 2 + (b * ct) ** 2)
        lo_y, hi_y = min(hy, m / 2.0), max(m - hy, m / 2.0)
        lo_x, hi_x = min(hx, n / 2.0), max(n - hx, n / 2.0)
        if cy < lo_y or cy > hi_y:
            vy = -vy
            cy = min(hi_y, max(lo_y, cy))
        if cx < lo_x or cx > hi_x:
            vx = -vx
            cx = min(hi_x, max(lo_x, cx))
    visible = np.ones(frames, dtype=bool)
    for r in vanish or []:
        for t in r:
            if 0 <= t < frames:
                visible[t] = False
    return Trajectory(out["cy"], out["cx"], out["a"], out["b"], out["theta"], visible)


# ----------------------------------------------------------------------------
# The sequence generator
# ----------------------------------------------------------------------------

class Sequence:
    """Deterministic per-frame inputs for one workload.

    Every array is a function of (workload seed, frame, stream/unit), so any
    frame can be regenerated on its own without materialising the sequence.
    """

    def __init__(self, w: Workload, vanish: Optional[dict] = None):
        self.w = w
        rng = np.random.default_rng([w.seed, 0xA5])
        self.traj: List[Trajectory] = []
        for u in range(w.U):
            van = (vanish or {}).get(u)
            self.traj.append(make_trajectory(rng, w.m, w.n, w.frames + w.prefill_frames,
                                             w.cov_lo, w.cov_hi, van))
        self.ptr_seed = [w.seed, 0x9E]

    # -- masks ---------------------------------------------------------------
    def mask(self, t: int, u: int) -> np.ndarray:
        """uint8 [mn] mask of unit u at sequence frame t (prefill frames first)."""
        tr = self.traj[u]
        if not tr.visible[t]:
            return np.zeros(self.w.mn, dtype=np.uint8)
        return ellipse_mask(self.w.m, self.w.n, tr.cy[t], tr.cx[t], tr.a[t], tr.b[t],
                            tr.theta[t]).reshape(-1)

    def masks(self, t: int) -> np.ndarray:
        """uint8 [U, mn] masks of all units at frame t."""
        return np.stack([self.mask(t, u) for u in range(self.w.U)])

    # -- token grids ---------------------------------------------------------
    def _dtype_out(self, x: np.ndarray) -> np.ndarray:
        if self.w.dtype == "bf16":
            return f32_to_bf16_bits(x)
        return np.ascontiguousarray(x, dtype=np.float32)

    def z(self, t: int) -> np.ndarray:
        """Query grid per group, [G, mn, C] (uint16 bf16 bits or fp32)."""
        w = self.w
        out = np.empty((w.G, w.mn, w.C), dtype=np.float32)
        masks = self.masks(t)
        for g in range(w.G):
            rng = np.random.default_rng([w.seed, 1, t, g])
            zg = rng.standard_normal((w.mn, w.C), dtype=np.float32)
            inside = np.zeros(w.mn, dtype=bool)
            for u in range(g * w.units_per_group, (g + 1) * w.units_per_group):
                inside |= masks[u].astype(bool)
            zg[inside] *= np.float32(1.25)
            out[g] = zg
        return self._dtype_out(out)

    def kv_new(self, t: int) -> tuple:
        """Memory-encoder output per unit, (K_new, V_new) each [U, mn, D]."""
        w = self.w
        rng = np.random.default_rng([w.seed, 2, t])
        k = rng.standard_normal((w.U, w.mn, w.D), dtype=np.float32)
        v = rng.standard_normal((w.U, w.mn, w.D), dtype=np.float32)
        return self._dtype_out(k), self._dtype_out(v)

    def pointers(self) -> tuple:
        """Pointer rows per unit, (K_ptr, V_ptr) each [U, n_ptr, D]."""
        w = self.w
        rng = np.random.default_rng(self.ptr_seed)
        k = rng.standard_normal((w.U, w.n_ptr, w.D), dtype=np.float32)
        v = rng.standard_normal((w.U, w.n_ptr, w.D), dtype=np.float32)
        return self._dtype_out(k), self._dtype_out(v)

    def rope_table(self, theta_base: float = 10000.0) -> np.ndarray:
        """fp32 [mn, d/2, 2] (cos, sin) of a 2-D axial frequency table: the first
        d/4 pairs rotate with the column index, the rest with the row index."""
        w = self.w
        d2 = w.d // 2
        half = d2 // 2
        ys, xs = np.divmod(np.arange(w.mn), w.n)
        freqs = theta_base ** (-np.arange(half, dtype=np.float64) / max(half, 1))
        ang = np.zeros((w.mn, d2), dtype=np.float64)
        ang[:, :half] = xs[:, None] * freqs[None, :]
        ang[:, half:2 * half] = ys[:, None] * freqs[None, :]
        out = np.stack([np.cos(ang), np.sin(ang)], axis=-1).astype(np.float32)
        return np.ascontiguousarray(out)


def random_bf16(rng: np.random.Generator, shape, scale: float = 1.0) -> np.ndarray:
    return f32_to_bf16_bits(rng.standard_normal(shape, dtype=np.float32) * np.float32(scale))


def ternary_grid(rng: np.random.Generator, G: int, mn: int, C: int, p_nonzero: float,
                 dtype: str = "bf16") -> np.ndarray:
    """Token grids whose channels are -1, 0 or +1 (nonzero with probability
    p_nonzero, either sign equally likely).  Every squared norm is an integer
    in [0, C], so many cells share one, which puts equal keys at the k-th
    place of a top-k.  Returns bf16 bits or fp32 [G, mn, C]."""
    mag = (rng.random((G, mn, C)) < p_nonzero).astype(np.float32)
    sign = np.where(rng.random((G, mn, C)) < 0.5, -1.0, 1.0).astype(np.float32)
    z = mag * sign
    return f32_to_bf16_bits(z) if dtype == "bf16" else z


def permuted_rows(rng: np.random.Generator, G: int, mn: int, C: int,
                  dtype: str = "bf16") -> np.ndarray:
    """Token grids whose rows are permutations of one N(0,1) vector per grid:
    every cell of a grid has the same multiset of channel values."""
    base = rng.standard_normal((G, C), dtype=np.float32)
    z = np.empty((G, mn, C), dtype=np.float32)
    for g in range(G):
        z[g] = base[g][rng.permuted(np.tile(np.arange(C), (mn, 1)), axis=1)]
    return f32_to_bf16_bits(z) if dtype == "bf16" else z


def cell_subset_masks(rng: np.random.Generator, U: int, mn: int, sizes) -> np.ndarray:
    """Masks [U, mn] with exactly sizes[u] set cells each, at random positions."""
    M = np.zeros((U, mn), np.uint8)
    for u in range(U):
        M[u, rng.choice(mn, size=int(sizes[u]), replace=False)] = 1
    return M


# ----------------------------------------------------------------------------
# Pixel-resolution inputs: decoder logits and seed masks
# ----------------------------------------------------------------------------

def decoder_logits(rng: np.random.Generator, n_obj: int, h: int, w: int,
                   cov_lo: float = 0.02, cov_hi: float = 0.25,
                   hole_rate: float = 0.01, speck_rate: float = 0.002) -> np.ndarray:
    """Stand-in for a mask decoder's per-object logits [n_obj, h, w] fp32 at
    its output resolution: a rotated ellipse per object (coverage drawn from
    [cov_lo, cov_hi], objects may overlap and touch the border) with logits
    |N(0,1)| + 0.5 inside and -(|N(0,1)| + 0.5) outside, then salt-and-pepper
    noise -- isolated negative pixels inside ("holes", the artefact the paper's
    closure removes) and isolated positive specks outside."""
    out = np.empty((n_obj, h, w), dtype=np.float32)
    for o in range(n_obj):
        cov = rng.uniform(cov_lo, cov_hi)
        aspect = rng.uniform(0.6, 1.6)
        area = cov * h * w
        a = math.sqrt(area * aspect / math.pi)
        b = area / (math.pi * a)
        cy, cx = rng.uniform(0.0, h), rng.uniform(0.0, w)
        inside = ellipse_mask(h, w, cy, cx, a, b, rng.uniform(0.0, math.pi)).astype(bool)
        mag = np.abs(rng.standard_normal((h, w), dtype=np.float32)) + np.float32(0.5)
        lg = np.where(inside, mag, -mag)
        holes = inside & (rng.random((h, w)) < hole_rate)
        specks = ~inside & (rng.random((h, w)) < speck_rate)
        lg[holes] = -lg[holes]
        lg[specks] = -lg[specks]
        out[o] = lg
    return out


def pixel_masks(rng: np.random.Generator, n_obj: int, h: int, w: int,
                cov_lo: float = 0.02, cov_hi: float = 0.25) -> np.ndarray:
    """First-frame object masks at pixel resolution [n_obj, h, w] uint8
    (rotated ellipses, value 255 where set)."""
    out = np.empty((n_obj, h, w), dtype=np.uint8)
    for o in range(n_obj):
        cov = rng.uniform(cov_lo, cov_hi)
        aspect = rng.uniform(0.6, 1.6)
        area = cov * h * w
        a = math.sqrt(area * aspect / math.pi)
        b = area / (math.pi * a)
        cy, cx = rng.uniform(0.1 * h, 0.9 * h), rng.uniform(0.1 * w, 0.9 * w)
        out[o] = ellipse_mask(h, w, cy, cx, a, b, rng.uniform(0.0, math.pi)) * np.uint8(255)
    return out
