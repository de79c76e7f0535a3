"""Helpers for the GPU tests: guarded device buffers (canary bands around the
view a kernel writes, checked afterwards in place of a memory sanitizer) and
host copies of bf16 tensors as bit patterns."""
import numpy as np
import torch

SENTINEL = {torch.bfloat16: 0x7FA5, torch.float16: 0x7FA5, torch.float32: 0x7FA5A5A5}


class Guarded:
    """A rows x cols view with row stride ld inside a larger allocation whose
    bytes outside the view hold a sentinel pattern."""

    def __init__(self, rows, cols, dtype, ld=None, pad_elems=64):
        self.rows, self.cols, self.dtype = rows, cols, dtype
        self.ld = cols if ld is None else ld
        self.pad = pad_elems
        n = self.pad * 2 + max(rows * self.ld, 1)
        itype = torch.int16 if dtype in (torch.bfloat16, torch.float16) else torch.int32
        self._sent = SENTINEL[dtype]            # positive, fits the signed type
        self.base = torch.full((n,), self._sent, dtype=itype, device="cuda").view(dtype)
        flat = self.base[self.pad:self.pad + rows * self.ld]
        self.view = flat.view(rows, self.ld)[:, :cols]

    def canaries_intact(self) -> bool:
        itype = torch.int16 if self.dtype in (torch.bfloat16, torch.float16) else torch.int32
        raw = self.base.view(itype).cpu().numpy()
        mask = np.ones(raw.size, dtype=bool)
        for r in range(self.rows):
            s = self.pad + r * self.ld
            mask[s:s + self.cols] = False
        return bool(np.all(raw[mask] == self._sent))


def bits16(t: torch.Tensor) -> np.ndarray:
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def to_bf16_tensor(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def to_f16_tensor(bits: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.float16).cuda()
