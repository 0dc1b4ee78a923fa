"""Per-frame driver of the hot path (Algorithm 1's per-frame loop, restricted
to what the library implements): device buffers for one workload and the three
library calls of a frame -- select (Eq. 1/2/4/5), readout (Eq. 6/7) and
commit (Eq. 8).  Buffers come from torch; all arithmetic runs in librs3.
"""
from __future__ import annotations

from typing import Optional

import torch

from . import rs3
from .synth import Workload


class Pipeline:
    def __init__(self, w: Workload, device="cuda", dense: bool = False,
                 ring_cap: Optional[int] = None, params: Optional[rs3.Params] = None,
                 stream=None):
        self.w = w
        self.device = torch.device(device)
        self.dense = dense
        rho = 1.0 if dense else w.rho
        self.params = params if params is not None else rs3.default_params(
            rho=rho, r_s=w.r_s, c=w.c, union_mode=w.union_mode)
        self.k_max = rs3.rs3_kmax(self.params.rho, w.mn)
        dev = self.device
        self.unit_group = torch.tensor(w.unit_group(), dtype=torch.int32, device=dev)
        self.track = torch.zeros((w.U, 6), dtype=torch.int32, device=dev)
        # two keep-set buffers, so the selection of frame t+1 can be issued
        # while the readout of frame t still reads its own keep-set
        self.idx_buf = [torch.zeros((w.U, max(self.k_max, 1)), dtype=torch.int32, device=dev)
                        for _ in range(2)]
        self.count_buf = [torch.zeros(w.U, dtype=torch.int32, device=dev) for _ in range(2)]
        self.idx, self.count = self.idx_buf[0], self.count_buf[0]
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.ws_select = torch.empty(rs3.rs3_select_workspace_bytes(w.G, w.U, w.m, w.n),
                                     dtype=torch.uint8, device=dev)
        # two readout workspaces, paired with the keep-set buffers: the merge of
        # frame t reads its workspace while frame t+1 plans and attends in the other
        nws = rs3.rs3_readout_workspace_bytes(w.U, w.H, w.d, self.k_max, w.dtype)
        self.ws_buf = [torch.empty(nws, dtype=torch.uint8, device=dev) for _ in range(2)]
        self.ws_readout = self.ws_buf[0]
        if ring_cap is None:
            ring_cap = w.ring_cap_rows() if (dense or w.window > 0) else w.ring_cap_rows_tight()
        self.bank = rs3.Bank(w.U, w.H, w.d, w.dtype, w.mn, w.n_cond, w.window, ring_cap,
                             w.max_frames(), w.n_ptr, device=dev, stream=stream)
        self.stream = stream

    # -- library calls -------------------------------------------------------
    def use_buffer(self, i: int):
        """Selects which keep-set buffer (and readout workspace) the next
        select / readout use."""
        self.idx, self.count = self.idx_buf[i], self.count_buf[i]
        self.ws_readout = self.ws_buf[i]

    def select(self, z: torch.Tensor, prev_masks: torch.Tensor, stream=None):
        w = self.w
        rs3.rs3_select_queries(z, w.dtype, w.G, w.m, w.n, w.C, prev_masks, self.unit_group, w.U,
                               self.track, self.params, self.idx, self.count, self.ws_select,
                               self.status, stream if stream is not None else self.stream)

    def readout(self, q: torch.Tensor, residual: Optional[torch.Tensor], out: torch.Tensor,
                rope: Optional[torch.Tensor] = None, scale: float = 0.0):
        w = self.w
        rs3.rs3_memory_readout(q, w.dtype, w.G, w.mn, w.H, w.d, self.unit_group, self.idx,
                               self.count, self.k_max, self.bank, rope, residual, out, scale,
                               self.ws_readout, self.status, self.stream)

    def readout_attend(self, q: torch.Tensor, residual: Optional[torch.Tensor], out: torch.Tensor,
                       rope: Optional[torch.Tensor] = None, scale: float = 0.0, stream=None):
        """First phase of readout(): the attention over the bank."""
        w = self.w
        rs3.rs3_memory_readout_attend(q, w.dtype, w.G, w.mn, w.H, w.d, self.unit_group, self.idx,
                                      self.count, self.k_max, self.bank, rope, residual, out, scale,
                                      self.ws_readout, self.status,
                                      stream if stream is not None else self.stream)

    def readout_plan(self, q: torch.Tensor, residual: Optional[torch.Tensor], out: torch.Tensor,
                     rope: Optional[torch.Tensor] = None, scale: float = 0.0, stream=None):
        """First launch of readout_attend(): the pass-through and the work list."""
        w = self.w
        rs3.rs3_memory_readout_plan(q, w.dtype, w.G, w.mn, w.H, w.d, self.unit_group, self.idx,
                                    self.count, self.k_max, self.bank, rope, residual, out, scale,
                                    self.ws_readout, self.status,
                                    stream if stream is not None else self.stream)

    def readout_run(self, q: torch.Tensor, residual: Optional[torch.Tensor], out: torch.Tensor,
                    rope: Optional[torch.Tensor] = None, scale: float = 0.0, stream=None):
        """Second launch of readout_attend(): the attention kernel alone."""
        w = self.w
        rs3.rs3_memory_readout_run(q, w.dtype, w.G, w.mn, w.H, w.d, self.unit_group, self.idx,
                                   self.count, self.k_max, self.bank, rope, residual, out, scale,
                                   self.ws_readout, self.status,
                                   stream if stream is not None else self.stream)

    def readout_merge(self, q: torch.Tensor, residual: Optional[torch.Tensor], out: torch.Tensor,
                      rope: Optional[torch.Tensor] = None, scale: float = 0.0, stream=None):
        """Second phase of readout(): the split-KV merge; reads no bank."""
        w = self.w
        rs3.rs3_memory_readout_merge(q, w.dtype, w.G, w.mn, w.H, w.d, self.unit_group, self.idx,
                                     self.count, self.k_max, self.bank, rope, residual, out, scale,
                                     self.ws_readout, self.status,
                                     stream if stream is not None else self.stream)

    def commit(self, k_new: torch.Tensor, v_new: torch.Tensor, mask: Optional[torch.Tensor],
               is_cond: int, rope: Optional[torch.Tensor] = None):
        """Eq. 8's sparse write; with a RoPE table the keys are stored rotated
        by their own cell (Eq. 7 on the key side)."""
        m = None if self.dense else mask
        if rope is None:
            rs3.rs3_bank_commit(self.bank, k_new, v_new, m, is_cond, self.status, self.stream)
        else:
            rs3.rs3_bank_commit_rope(self.bank, k_new, v_new, m, is_cond, rope, self.status, self.stream)

    def set_pointers(self, kp: torch.Tensor, vp: torch.Tensor):
        rs3.rs3_bank_set_pointers(self.bank, kp, vp, self.status, self.stream)

    def reset(self):
        rs3.rs3_bank_reset(self.bank, -1, self.stream)
        self.track.zero_()
        self.status.zero_()

    def status_code(self) -> int:
        return int(self.status.item())
