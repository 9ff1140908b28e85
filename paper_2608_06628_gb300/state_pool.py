"""Device memory for per-request states: one slab, one slot per request.

The slab is a torch allocation; a batch names its requests through a device
array of slot pointers (int64), which is what the C ABI's d_state_ptrs takes.
Any subset of slots, in any order, forms a valid ragged batch.
"""
from __future__ import annotations

import torch

from . import hybrid as H


class StatePool:
    def __init__(self, cfg: H.hybrid_cfg, n_slots: int, device="cuda"):
        self.cfg = cfg
        self.n_slots = n_slots
        self.slot_bytes = H.hybrid_state_bytes(cfg)
        if self.slot_bytes == 0:
            raise ValueError(f"unsupported cfg {cfg}")
        assert self.slot_bytes % 16 == 0
        self.slab = torch.empty(n_slots * self.slot_bytes // 4, dtype=torch.float32, device=device)
        self.base = self.slab.data_ptr()

    def slot_ptr(self, slot: int) -> int:
        return self.base + slot * self.slot_bytes

    def ptr_array(self, slots) -> torch.Tensor:
        """Device int64 array of slot pointers for the given slots (in order)."""
        slots = torch.as_tensor(list(slots), dtype=torch.int64)
        return (slots * self.slot_bytes + self.base).to(self.slab.device)

    def all_ptrs(self) -> torch.Tensor:
        return self.ptr_array(range(self.n_slots))

    def slot_view(self, slot: int) -> torch.Tensor:
        n = self.slot_bytes // 4
        return self.slab[slot * n:(slot + 1) * n]
