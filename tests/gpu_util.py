"""Helpers shared by the GPU tests: seeded inputs on the host and device,
and the oracle's expected result for the same bits."""
from __future__ import annotations

import numpy as np
import torch

from paper_2109_12626_gb300 import inputs as I

NP_DT = {"int32": np.int32, "float32": np.float32, "mat2x2u32": np.uint32,
         "mat2x2f32": np.float32}
TORCH_DT = {"int32": torch.int32, "float32": torch.float32, "mat2x2u32": torch.int32,
            "mat2x2f32": torch.float32}


def host_inputs(kind, seed, p, m, **kw):
    """[p][m] numpy array (matrices as [p][m][4] uint32) of the seeded input."""
    rows = [I.rank_values(kind, seed, i, m, **kw) for i in range(p)]
    if kind == "mat2x2u32":
        a = torch.stack(rows).numpy().view(np.uint32)
        return a.reshape(p, m, 4)
    return torch.stack(rows).numpy() if p else np.zeros((0, m), NP_DT[kind])


def to_device(arr, kind, dev, pad_front=0):
    """One device tensor per rank.  pad_front > 0 offsets each buffer by that
    many 4-byte words from a 16-byte-aligned allocation (misaligned case)."""
    out, keep = [], []
    for row in arr:
        flat = torch.from_numpy(np.ascontiguousarray(row).view(np.int32).reshape(-1))
        if kind == "float32":
            flat = flat.view(torch.float32)
        if pad_front:
            base = torch.empty(flat.numel() + pad_front, dtype=flat.dtype, device=dev)
            t = base[pad_front:]
            t.copy_(flat)
            keep.append(base)
        else:
            t = flat.to(dev)
        out.append(t)
    return out, keep


def empty_like_ranks(xs, fill=-3, pad_front=0):
    ys, keep = [], []
    for x in xs:
        if pad_front:
            base = torch.full((x.numel() + pad_front,), fill, dtype=x.dtype, device=x.device)
            ys.append(base[pad_front:])
            keep.append(base)
        else:
            ys.append(torch.full_like(x, fill))
    return ys, keep


def bits(t) -> np.ndarray:
    """Raw 32-bit words of a tensor (float32 compared bit for bit)."""
    return t.detach().cpu().contiguous().view(torch.int32).numpy().reshape(-1)


def expect_bits(want: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(want).view(np.int32).reshape(-1)
