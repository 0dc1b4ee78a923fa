"""The C ABI library builds, loads without a GPU, exports every function that
include/rs3.h declares, and rejects bad arguments on the host before touching
the device.  CPU only: no call here reaches a kernel."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "rs3.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    return sorted(set(re.findall(r"\b(rs3_[a-z_0-9]+)\s*\(", src)))


@pytest.fixture(scope="module")
def binding():
    from paper_2608_22526_gb300 import _build
    _build.build()
    from paper_2608_22526_gb300 import rs3
    return rs3


def test_header_declares_the_boundary():
    names = _declared()
    for required in ("rs3_select_queries", "rs3_memory_readout", "rs3_bank_commit",
                     "rs3_bank_reset", "rs3_bank_init", "rs3_write_keepset",
                     "rs3_bank_set_pointers"):
        assert required in names


def test_library_exports_every_declared_symbol(binding):
    lib = ctypes.CDLL(binding.LIB_PATH)
    missing = [n for n in _declared() if not hasattr(lib, n)]
    assert not missing, missing
    # the binding covers exactly the declared functions
    assert sorted(binding.SIGNATURES) == _declared()


def test_struct_sizes_match_header(binding):
    assert ctypes.sizeof(binding.Params) == 48
    assert ctypes.sizeof(binding.BankDesc) == 104


def test_kmax_and_defaults(binding):
    assert binding.rs3_kmax(0.3, 4096) == 1228
    assert binding.rs3_kmax(0.2, 4096) == 819
    assert binding.rs3_kmax(1.0, 9216) == 9216
    assert binding.rs3_kmax(1.5, 10) == -1
    p = binding.default_params()
    assert (p.rho, p.r_s, p.c, p.D_w, p.union_mode) == (0.3, 4, 14, 24, 1)
    assert (p.fall_lo, p.fall_hi, p.fall_through, p.bbox_mode) == (0.05, 0.95, 1, 0)
    assert binding.status_string(2) == "capacity exceeded"


def test_bank_layout_rules(binding):
    rows, mb = binding.rs3_bank_layout(8, 1, 256, "bf16", 4096, 1, 6, 6 * 4096, 6, 16)
    assert rows == 4096 + 6 * 4096 + 16
    assert mb > 0
    bad = [
        (8, 1, 256, "bf16", 4096, 1, 6, 6 * 4096 - 1, 6, 16),   # ring cannot hold the window
        (8, 1, 256, "bf16", 4096, 1, 6, 6 * 4096, 5, 16),       # frame table != window
        (8, 1, 256, "bf16", 4096, 1, 0, 4096, 1, 0),            # window 0
        (8, 1, 3, "bf16", 4096, 1, -1, 4096, 4, 0),             # rows not 16-byte multiples
        (0, 1, 256, "bf16", 4096, 1, -1, 4096, 4, 0),           # no units
    ]
    for args in bad:
        with pytest.raises(binding.RS3Error) as e:
            binding.rs3_bank_layout(*args)
        assert e.value.code == binding.RS3_EINVAL
    for args in [(1, 1, 64, "bf16", 20000, 0, -1, 10, 4, 0),     # mn above 16384
                 (65536, 1, 64, "bf16", 16, 0, -1, 16, 1, 0)]:    # more units than a grid column
        with pytest.raises(binding.RS3Error) as e:
            binding.rs3_bank_layout(*args)
        assert e.value.code == binding.RS3_EUNSUPPORTED
    assert binding.rs3_bank_layout(65535, 1, 64, "bf16", 16, 0, -1, 16, 1, 0)[0] == 16


def test_workspace_sizes(binding):
    a = binding.rs3_select_workspace_bytes(1, 8, 64, 64)
    assert a >= 8 * 4096 + 4096 * 4
    assert binding.rs3_select_workspace_bytes(0, 1, 1, 1) == 0
    b = binding.rs3_readout_workspace_bytes(8, 1, 256, 1228, "bf16")
    c = binding.rs3_readout_workspace_bytes(8, 1, 256, 2456, "bf16")
    assert 0 < b <= c


def test_null_arguments_are_rejected_on_host(binding):
    lib = binding.lib
    p = binding.default_params()
    one = ctypes.c_void_p(16)     # a non-null, aligned dummy that is never dereferenced
    rc = lib.rs3_select_queries(None, 1, 1, 64, 64, 256, one, one, 1, one, ctypes.byref(p), one,
                                one, one, 1 << 20, one, None)
    assert rc == binding.RS3_EINVAL
    rc = lib.rs3_select_queries(one, 1, 1, 64, 64, 250, one, one, 1, one, ctypes.byref(p), one,
                                one, one, 1 << 20, one, None)           # C % 8 != 0
    assert rc == binding.RS3_EINVAL
    rc = lib.rs3_select_queries(one, 1, 1, 200, 200, 256, one, one, 1, one, ctypes.byref(p), one,
                                one, one, 1 << 30, one, None)           # mn > 16384
    assert rc == binding.RS3_EUNSUPPORTED
    rc = lib.rs3_select_queries(one, 1, 1, 64, 64, 256, one, one, 1, one, ctypes.byref(p), one,
                                one, one, 16, one, None)                # workspace too small
    assert rc == binding.RS3_ECAPACITY
    bad = binding.default_params(rho=1.5)
    rc = lib.rs3_select_queries(one, 1, 1, 64, 64, 256, one, one, 1, one, ctypes.byref(bad), one,
                                one, one, 1 << 20, one, None)
    assert rc == binding.RS3_EINVAL
    # an uninitialised bank descriptor is refused by every bank call
    desc = binding.BankDesc()
    assert lib.rs3_bank_commit(ctypes.byref(desc), one, one, None, 0, one, None) == binding.RS3_EINVAL
    assert lib.rs3_bank_commit_rope(ctypes.byref(desc), one, one, None, 0, one, one, None) == binding.RS3_EINVAL
    assert lib.rs3_bank_commit_rope(ctypes.byref(desc), one, one, None, 0, None, one, None) == binding.RS3_EINVAL
    assert lib.rs3_bank_reset(ctypes.byref(desc), -1, None) == binding.RS3_EINVAL
    assert lib.rs3_memory_readout(one, 1, 1, 4096, 1, 256, one, one, one, 1228, ctypes.byref(desc),
                                  None, None, one, 0.0, one, 1 << 30, one, None) == binding.RS3_EINVAL
    assert lib.rs3_write_keepset(None, one, 1, 8, 8, ctypes.byref(p), one, one, None) == binding.RS3_EINVAL


def test_mask_calls_reject_bad_arguments_on_host(binding):
    lib = binding.lib
    one = ctypes.c_void_p(16)
    E, U = binding.RS3_EINVAL, binding.RS3_EUNSUPPORTED
    # logits, group_start, G, U, h, w, radius, s, palette, closed, grid, status, stream
    assert lib.rs3_close_argmax(None, one, 1, 1, 64, 64, 4, 4, one, None, None, one, None) == E
    assert lib.rs3_close_argmax(one, one, 1, 1, 64, 64, 4, 4, one, None, None, None, None) == E
    assert lib.rs3_close_argmax(one, one, 1, 1, 64, 48, 4, 4, one, None, None, one, None) == U   # w % 32
    assert lib.rs3_close_argmax(one, one, 1, 1, 64, 64, 9, 4, one, None, None, one, None) == U   # radius > 8
    assert lib.rs3_close_argmax(one, one, 1, 1, 64, 64, -1, 4, one, None, None, one, None) == E
    assert lib.rs3_close_argmax(one, one, 0, 1, 64, 64, 4, 4, one, None, None, one, None) == E
    assert lib.rs3_close_argmax(one, one, 1, 1, 66, 64, 4, 4, None, None, one, one, None) == E   # h % s with grid
    # masks, U, h, w, s, track, grid, box, stream
    assert lib.rs3_seed_from_masks(None, 1, 64, 64, 16, one, None, None, None) == E
    assert lib.rs3_seed_from_masks(one, 1, 64, 64, 16, None, None, None, None) == E
    assert lib.rs3_seed_from_masks(one, 1, 64, 40, 8, one, None, None, None) == E      # w % 16
    assert lib.rs3_seed_from_masks(one, 1, 64, 64, 24, one, None, None, None) == E     # w % s
    assert lib.rs3_seed_from_masks(ctypes.c_void_p(17), 1, 64, 64, 16, one, None, None, None) == E
    assert lib.rs3_seed_from_masks(one, 0, 64, 64, 16, one, None, None, None) == E


def test_oversized_readout_plan_is_refused(binding):
    """The readout's work-item indices are 32-bit: a request whose list could
    reach 2^30 entries (4096 units x 512 heads x 512 query tiles of the fp32
    path, k_max 16384) is refused on the host with RS3_EUNSUPPORTED; a small
    request with the same descriptor shape gets as far as the workspace-size
    check."""
    lib = binding.lib
    one = ctypes.c_void_p(16)

    def bank(U):
        b = binding.BankDesc()
        b.U, b.H, b.d, b.D, b.dtype, b.mn = U, 512, 16, 512 * 16, 0, 16384
        b.n_cond, b.window, b.max_frames, b.n_ptr = 0, -1, 4, 0
        b.pinned_cap, b.ring_cap, b.rows_per_unit, b.meta_stride = 0, 64, 64, 8 * 24
        b.k_store = b.v_store = b.meta = one
        b.magic = 0x52533342           # what rs3_bank_init stores
        return b

    big, small = bank(4096), bank(8)
    args = lambda b, ws: (one, 0, 1, 16384, 512, 16, one, one, one, 16384, ctypes.byref(b), None, None,
                          one, 0.0, one, ws, one, None)
    assert lib.rs3_memory_readout(*args(big, 1 << 62)) == binding.RS3_EUNSUPPORTED
    assert lib.rs3_memory_readout_attend(*args(big, 1 << 62)) == binding.RS3_EUNSUPPORTED
    assert lib.rs3_memory_readout(*args(small, 16)) == binding.RS3_ECAPACITY
