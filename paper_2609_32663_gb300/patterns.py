"""Saved retention patterns. A pattern M in {0,1}^{L x H x D} is exported once
(Eq. 3, App. A.3) and reused for every input (Sec. 3.4); this module stores it
with the geometry it was exported for (sink S, recent R, bin width W), so that a
loaded pattern is mapped with the same position-to-bin rule (Eqs. 4 and 5).

Format: a NumPy .npz with `M` (uint8 [L][H][D]), `sink`, `recent`, `bin_width`
(int64 scalars) and `meta` (a JSON string: the generator, seed, budget, ...)."""
from __future__ import annotations

import json

import numpy as np


def save_pattern(path, M, sink: int, recent: int, bin_width: int, meta: dict | None = None) -> None:
    M = np.asarray(M)
    if M.ndim != 3:
        raise ValueError(f"M must be [L][H][D], got shape {M.shape}")
    if M.size and not np.isin(M, (0, 1)).all():
        raise ValueError("M entries must be 0 or 1")
    if min(sink, recent) < 0 or bin_width < 1:
        raise ValueError("sink and recent must be >= 0, bin_width >= 1")
    with open(path, "wb") as f:
        np.savez_compressed(f, M=M.astype(np.uint8), sink=np.int64(sink), recent=np.int64(recent),
                            bin_width=np.int64(bin_width), meta=np.array(json.dumps(meta or {})))


def load_pattern(path):
    """Returns (M uint8 [L][H][D], {"sink", "recent", "bin_width"}, meta dict)."""
    with np.load(path, allow_pickle=False) as z:
        M = np.ascontiguousarray(z["M"], np.uint8)
        geo = {k: int(z[k]) for k in ("sink", "recent", "bin_width")}
        meta = json.loads(str(z["meta"]))
    if M.ndim != 3 or (M.size and not np.isin(M, (0, 1)).all()):
        raise ValueError(f"{path}: not a 0/1 pattern of shape [L][H][D]")
    return M, geo, meta


def check_geometry(geo: dict, shape) -> None:
    """Raise if a loaded pattern's geometry differs from the shape it is mapped with
    (any object with L, H, D, sink, recent, bin_width attributes)."""
    for k in ("sink", "recent", "bin_width"):
        if int(getattr(shape, k)) != geo[k]:
            raise ValueError(f"pattern was exported with {k}={geo[k]}, shape has {getattr(shape, k)}")
