"""Python binding of librs3 (include/rs3.h): argument marshalling only.

Every step of the hot path runs in the CUDA library; this module turns torch
tensors into pointers and checks return codes.  There is no fallback: if the
library is missing the import of this module fails.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "librs3.so")

RS3_OK, RS3_EINVAL, RS3_ECAPACITY, RS3_EUNSUPPORTED, RS3_ECUDA, RS3_EINTERNAL, RS3_ETIMEOUT = range(7)
RS3_F32, RS3_BF16 = 0, 1
DTYPES = {"f32": RS3_F32, "bf16": RS3_BF16}
TORCH_DTYPES = {"f32": torch.float32, "bf16": torch.bfloat16}


class RS3Error(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"{what}: rs3 status {code} ({status_string(code)})")
        self.code = code


class Params(ctypes.Structure):
    _fields_ = [("rho", ctypes.c_double), ("r_s", ctypes.c_int32), ("c", ctypes.c_int32),
                ("D_w", ctypes.c_int32), ("union_mode", ctypes.c_int32),
                ("fall_lo", ctypes.c_double), ("fall_hi", ctypes.c_double),
                ("fall_through", ctypes.c_int32), ("bbox_mode", ctypes.c_int32)]


class BankDesc(ctypes.Structure):
    _fields_ = [("U", ctypes.c_int32), ("H", ctypes.c_int32), ("d", ctypes.c_int32),
                ("D", ctypes.c_int32), ("dtype", ctypes.c_int32), ("mn", ctypes.c_int32),
                ("n_cond", ctypes.c_int32), ("window", ctypes.c_int32),
                ("max_frames", ctypes.c_int32), ("n_ptr", ctypes.c_int32),
                ("pinned_cap", ctypes.c_int64), ("ring_cap", ctypes.c_int64),
                ("rows_per_unit", ctypes.c_int64), ("meta_stride", ctypes.c_int64),
                ("k_store", ctypes.c_void_p), ("v_store", ctypes.c_void_p),
                ("meta", ctypes.c_void_p), ("magic", ctypes.c_uint32),
                ("reserved", ctypes.c_uint32)]


# Exported symbols and their signatures (checked against include/rs3.h by the tests)
_P = ctypes.c_void_p
_I = ctypes.c_int
_I64 = ctypes.c_int64
_SZ = ctypes.c_size_t
SIGNATURES = {
    "rs3_default_params": (None, [_P]),
    "rs3_kmax": (_I64, [ctypes.c_double, _I64]),
    "rs3_status_string": (ctypes.c_char_p, [_I]),
    "rs3_version": (_I, []),
    "rs3_select_workspace_bytes": (_SZ, [_I, _I, _I, _I]),
    "rs3_select_queries": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _I, _P, _P, _P, _P, _P, _SZ, _P, _P]),
    "rs3_select_queries_noalloc": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _I, _P, _P, _P, _P, _P, _P]),
    "rs3_bank_layout": (_I, [_I, _I, _I, _I, _I, _I, _I, _I64, _I, _I, _P, _P]),
    "rs3_bank_init": (_I, [_P, _I, _I, _I, _I, _I, _I, _I, _I64, _I, _I, _P, _P, _P, _P]),
    "rs3_bank_commit": (_I, [_P, _P, _P, _P, _I, _P, _P]),
    "rs3_bank_commit_rope": (_I, [_P, _P, _P, _P, _I, _P, _P, _P]),
    "rs3_bank_set_pointers": (_I, [_P, _P, _P, _P, _P]),
    "rs3_bank_reset": (_I, [_P, _I, _P]),
    "rs3_bank_read_meta": (_I, [_P, _P, _P, _P]),
    "rs3_readout_workspace_bytes": (_SZ, [_I, _I, _I, _I, _I]),
    "rs3_memory_readout": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _P, _I, _P, _P, _P, _P,
                                ctypes.c_float, _P, _SZ, _P, _P]),
    "rs3_memory_readout_attend": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _P, _I, _P, _P, _P, _P,
                                ctypes.c_float, _P, _SZ, _P, _P]),
    "rs3_memory_readout_merge": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _P, _I, _P, _P, _P, _P,
                                ctypes.c_float, _P, _SZ, _P, _P]),
    "rs3_memory_readout_plan": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _P, _I, _P, _P, _P, _P,
                                ctypes.c_float, _P, _SZ, _P, _P]),
    "rs3_memory_readout_run": (_I, [_P, _I, _I, _I, _I, _I, _P, _P, _P, _I, _P, _P, _P, _P,
                                ctypes.c_float, _P, _SZ, _P, _P]),
    "rs3_set_wait_limit_ns": (None, [ctypes.c_uint64]),
    "rs3_get_wait_limit_ns": (ctypes.c_uint64, []),
    "rs3_write_keepset": (_I, [_P, _P, _I, _I, _I, _P, _P, _P, _P]),
    "rs3_close_argmax": (_I, [_P, _P, _I, _I, _I, _I, _I, _I, _P, _P, _P, _P, _P]),
    "rs3_seed_from_masks": (_I, [_P, _I, _I, _I, _I, _P, _P, _P, _P]),
}


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"librs3.so is not built ({LIB_PATH}); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


lib = _load()


def status_string(code: int) -> str:
    return lib.rs3_status_string(int(code)).decode()


def _check(code: int, what: str):
    if code != RS3_OK:
        raise RS3Error(code, what)


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors passed to librs3 must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


# ---------------------------------------------------------------------------
# small helpers
# ---------------------------------------------------------------------------

def default_params(**over) -> Params:
    p = Params()
    lib.rs3_default_params(ctypes.byref(p))
    for k, v in over.items():
        setattr(p, k, v)
    return p


def rs3_kmax(rho: float, mn: int) -> int:
    return int(lib.rs3_kmax(float(rho), int(mn)))


def rs3_select_workspace_bytes(G: int, U: int, m: int, n: int) -> int:
    return int(lib.rs3_select_workspace_bytes(G, U, m, n))


def rs3_readout_workspace_bytes(U: int, H: int, d: int, k_max: int, dtype: str) -> int:
    return int(lib.rs3_readout_workspace_bytes(U, H, d, k_max, DTYPES[dtype]))


# ---------------------------------------------------------------------------
# read side
# ---------------------------------------------------------------------------

def rs3_select_queries(z, dtype: str, G: int, m: int, n: int, C: int, prev_masks, unit_group,
                       U: int, track, params: Params, idx, count, workspace, status, stream=None):
    rc = lib.rs3_select_queries(_ptr(z), DTYPES[dtype], G, m, n, C, _ptr(prev_masks),
                                _ptr(unit_group), U, _ptr(track), ctypes.byref(params), _ptr(idx),
                                _ptr(count), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                _ptr(status), _stream(stream))
    _check(rc, "rs3_select_queries")


def rs3_select_queries_noalloc(z, dtype: str, G: int, m: int, n: int, C: int, prev_masks,
                               unit_group, U: int, track, params: Params, idx, count, status,
                               stream=None):
    """rs3_select_queries with the library's built-in scratch (no workspace)."""
    rc = lib.rs3_select_queries_noalloc(_ptr(z), DTYPES[dtype], G, m, n, C, _ptr(prev_masks),
                                        _ptr(unit_group), U, _ptr(track), ctypes.byref(params),
                                        _ptr(idx), _ptr(count), _ptr(status), _stream(stream))
    _check(rc, "rs3_select_queries_noalloc")


def rs3_memory_readout(q, dtype: str, G: int, mn: int, H: int, d: int, unit_group, idx, count,
                       k_max: int, bank: "Bank", rope, residual, out, scale: float, workspace,
                       status, stream=None):
    rc = lib.rs3_memory_readout(_ptr(q), DTYPES[dtype], G, mn, H, d, _ptr(unit_group), _ptr(idx),
                                _ptr(count), k_max, ctypes.byref(bank.desc), _ptr(rope),
                                _ptr(residual), _ptr(out), float(scale), _ptr(workspace),
                                workspace.numel() * workspace.element_size(), _ptr(status),
                                _stream(stream))
    _check(rc, "rs3_memory_readout")


def _readout_phase(fn, name, q, dtype, G, mn, H, d, unit_group, idx, count, k_max, bank, rope, residual,
                   out, scale, workspace, status, stream):
    rc = fn(_ptr(q), DTYPES[dtype], G, mn, H, d, _ptr(unit_group), _ptr(idx), _ptr(count), k_max,
            ctypes.byref(bank.desc), _ptr(rope), _ptr(residual), _ptr(out), float(scale), _ptr(workspace),
            workspace.numel() * workspace.element_size(), _ptr(status), _stream(stream))
    _check(rc, name)


def rs3_memory_readout_attend(q, dtype: str, G: int, mn: int, H: int, d: int, unit_group, idx, count,
                              k_max: int, bank: "Bank", rope, residual, out, scale: float, workspace,
                              status, stream=None):
    _readout_phase(lib.rs3_memory_readout_attend, "rs3_memory_readout_attend", q, dtype, G, mn, H, d,
                   unit_group, idx, count, k_max, bank, rope, residual, out, scale, workspace, status, stream)


def rs3_memory_readout_plan(q, dtype: str, G: int, mn: int, H: int, d: int, unit_group, idx, count,
                            k_max: int, bank: "Bank", rope, residual, out, scale: float, workspace,
                            status, stream=None):
    _readout_phase(lib.rs3_memory_readout_plan, "rs3_memory_readout_plan", q, dtype, G, mn, H, d,
                   unit_group, idx, count, k_max, bank, rope, residual, out, scale, workspace, status, stream)


def rs3_memory_readout_run(q, dtype: str, G: int, mn: int, H: int, d: int, unit_group, idx, count,
                           k_max: int, bank: "Bank", rope, residual, out, scale: float, workspace,
                           status, stream=None):
    _readout_phase(lib.rs3_memory_readout_run, "rs3_memory_readout_run", q, dtype, G, mn, H, d,
                   unit_group, idx, count, k_max, bank, rope, residual, out, scale, workspace, status, stream)


def rs3_memory_readout_merge(q, dtype: str, G: int, mn: int, H: int, d: int, unit_group, idx, count,
                             k_max: int, bank: "Bank", rope, residual, out, scale: float, workspace,
                             status, stream=None):
    _readout_phase(lib.rs3_memory_readout_merge, "rs3_memory_readout_merge", q, dtype, G, mn, H, d,
                   unit_group, idx, count, k_max, bank, rope, residual, out, scale, workspace, status, stream)


def rs3_write_keepset(seed_masks, unit_group, U: int, m: int, n: int, params: Params, kw_out,
                      status, stream=None):
    rc = lib.rs3_write_keepset(_ptr(seed_masks), _ptr(unit_group), U, m, n, ctypes.byref(params),
                               _ptr(kw_out), _ptr(status), _stream(stream))
    _check(rc, "rs3_write_keepset")


# ---------------------------------------------------------------------------
# memory bank
# ---------------------------------------------------------------------------

def rs3_bank_layout(U, H, d, dtype, mn, n_cond, window, ring_cap, max_frames, n_ptr):
    rows = ctypes.c_int64()
    mb = ctypes.c_size_t()
    rc = lib.rs3_bank_layout(U, H, d, DTYPES[dtype], mn, n_cond, window, ring_cap, max_frames,
                             n_ptr, ctypes.byref(rows), ctypes.byref(mb))
    _check(rc, "rs3_bank_layout")
    return rows.value, mb.value


class Bank:
    """A set of U per-unit banks whose storage is owned by torch tensors."""

    def __init__(self, U: int, H: int, d: int, dtype: str, mn: int, n_cond: int, window: int,
                 ring_cap: int, max_frames: int, n_ptr: int, device="cuda", stream=None):
        rows, mb = rs3_bank_layout(U, H, d, dtype, mn, n_cond, window, ring_cap, max_frames, n_ptr)
        self.U, self.H, self.d, self.D, self.dtype, self.mn = U, H, d, H * d, dtype, mn
        self.rows_per_unit = rows
        tdt = TORCH_DTYPES[dtype]
        self.k_store = torch.empty((U, rows, H * d), dtype=tdt, device=device)
        self.v_store = torch.empty((U, rows, H * d), dtype=tdt, device=device)
        self.meta = torch.empty(max(mb // 8, 1), dtype=torch.int64, device=device)
        self.desc = BankDesc()
        rc = lib.rs3_bank_init(ctypes.byref(self.desc), U, H, d, DTYPES[dtype], mn, n_cond, window,
                               ring_cap, max_frames, n_ptr, _ptr(self.k_store), _ptr(self.v_store),
                               _ptr(self.meta), _stream(stream))
        _check(rc, "rs3_bank_init")

    @property
    def pinned_cap(self):
        return self.desc.pinned_cap

    @property
    def ring_cap(self):
        return self.desc.ring_cap

    @property
    def max_frames(self):
        return self.desc.max_frames


def rs3_bank_commit(bank: Bank, k_new, v_new, keep_mask, is_cond: int, status, stream=None):
    rc = lib.rs3_bank_commit(ctypes.byref(bank.desc), _ptr(k_new), _ptr(v_new), _ptr(keep_mask),
                             int(is_cond), _ptr(status), _stream(stream))
    _check(rc, "rs3_bank_commit")


def rs3_bank_commit_rope(bank: Bank, k_new, v_new, keep_mask, is_cond: int, rope, status, stream=None):
    rc = lib.rs3_bank_commit_rope(ctypes.byref(bank.desc), _ptr(k_new), _ptr(v_new), _ptr(keep_mask),
                                  int(is_cond), _ptr(rope), _ptr(status), _stream(stream))
    _check(rc, "rs3_bank_commit_rope")


def rs3_bank_set_pointers(bank: Bank, k_ptr, v_ptr, status, stream=None):
    rc = lib.rs3_bank_set_pointers(ctypes.byref(bank.desc), _ptr(k_ptr), _ptr(v_ptr), _ptr(status),
                                   _stream(stream))
    _check(rc, "rs3_bank_set_pointers")


def rs3_bank_reset(bank: Bank, unit: int = -1, stream=None):
    rc = lib.rs3_bank_reset(ctypes.byref(bank.desc), int(unit), _stream(stream))
    _check(rc, "rs3_bank_reset")


def rs3_bank_read_meta(bank: Bank, stream=None):
    """(counters int64 [U, 8], frames int64 [U, max_frames, 2]); synchronises."""
    import numpy as np
    out = np.zeros((bank.U, 8), dtype=np.int64)
    fr = np.zeros((bank.U, bank.max_frames, 2), dtype=np.int64)
    rc = lib.rs3_bank_read_meta(ctypes.byref(bank.desc), out.ctypes.data_as(ctypes.c_void_p),
                                fr.ctypes.data_as(ctypes.c_void_p), _stream(stream))
    _check(rc, "rs3_bank_read_meta")
    return out, fr


# ---------------------------------------------------------------------------
# decoder side and pixel-space front end
# ---------------------------------------------------------------------------

def rs3_close_argmax(logits, group_start, G: int, U: int, h: int, w: int, radius: int, s: int,
                     palette, closed, grid_masks, status, stream=None):
    rc = lib.rs3_close_argmax(_ptr(logits), _ptr(group_start), G, U, h, w, radius, s, _ptr(palette),
                              _ptr(closed), _ptr(grid_masks), _ptr(status), _stream(stream))
    _check(rc, "rs3_close_argmax")


def rs3_seed_from_masks(masks, U: int, h: int, w: int, s: int, track, grid_masks, box_masks,
                        stream=None):
    rc = lib.rs3_seed_from_masks(_ptr(masks), U, h, w, s, _ptr(track), _ptr(grid_masks),
                                 _ptr(box_masks), _stream(stream))
    _check(rc, "rs3_seed_from_masks")


def rs3_set_wait_limit_ns(ns: int):
    lib.rs3_set_wait_limit_ns(int(ns))


def rs3_get_wait_limit_ns() -> int:
    return int(lib.rs3_get_wait_limit_ns())
