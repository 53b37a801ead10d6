"""Host arrays of one batch -> device tensors in the layout the C ABI takes."""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


@dataclass
class DeviceBatch:
    n: int
    tags: object      # torch int64 (bit pattern of u64), shape (D, n), contiguous
    off: object       # torch int32 (bit pattern of u32), shape (n+1,)
    payload: object   # torch int32
    score: object     # torch float32 or None

    def nbytes(self) -> int:
        t = self.tags.numel() * 8 + self.off.numel() * 4 + self.payload.numel() * 4
        return t + (self.score.numel() * 4 if self.score is not None else 0)


def to_device(batch: dict, device="cuda", pin=False, non_blocking=False) -> DeviceBatch:
    """Copy a batch dict (tags (D,n) u64, off u32, payload int32, score f32)
    to the device."""
    import torch

    def t(a, dt):
        x = torch.from_numpy(np.ascontiguousarray(a).view(dt))
        if pin:
            x = x.pin_memory()
        return x.to(device, non_blocking=non_blocking)

    score = batch.get("score")
    return DeviceBatch(
        n=int(batch["n"]),
        tags=t(batch["tags"], np.int64),
        off=t(batch["off"], np.int32),
        payload=t(batch["payload"], np.int32),
        score=None if score is None else t(score, np.float32),
    )
