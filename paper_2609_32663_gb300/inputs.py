"""Seeded synthetic inputs for the Distance-KV decode path.

This module only draws inputs: retention patterns M, context lengths, and the
bf16 K/V/q tensors. It holds none of the path's arithmetic (no distance bins, no
retention mask, no union of positions, no packing, no attention), so both the
CUDA path and the CPU oracle can be fed from it without sharing any of the
computation. To hit exact budgets the pattern generators pick the top-scoring
entries and count group columns; those helpers (the `_gen_` functions) are
private to the generators, and no test, smoke check or benchmark takes an
expected value from them: expected masks, maps, bytes and outputs all come from
the oracle.

The workloads stand in for the paper's efficiency setting (Sec. 4.3, App. C:
Llama-3.1-8B and Qwen2.5-7B caches up to 128K context on one GPU). No model
weights or datasets are used: K, V, q are N(0, 1) bf16 draws, and patterns come
from seeded generators shaped like the learned ones (Sec. 4.5: near-heavy, a
far rise for some heads, partial heads).
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

SINK = 128      # Sec. 3.4: first 128 context positions always kept
RECENT = 1024   # Sec. 3.4: most recent 1,024 context positions always kept


@dataclass(frozen=True)
class Workload:
    """One benchmark/test workload: model head geometry, context mix, pattern recipe."""
    name: str
    L: int
    H: int
    Hkv: int
    T: int                      # maximum (and, unless ragged, every) context length
    B: int
    D: int                      # distance bins of the pattern
    W: int                      # bin width in tokens (a property of the pattern)
    pattern: str                # "bernoulli" | "profile"
    rate: float                 # bernoulli: P(M=1); profile: fraction of union bins kept
    physical_target: float | None = None  # profile: choose K_U for this overall physical retention
    ragged: tuple | None = None  # (lo, hi): per-sequence lengths uniform in [lo, hi]
    outlier_frac: float = 0.0   # fraction of key rows scaled by 8 (exact in bf16)
    seed: int = 0
    steps: int = 256
    head_dim: int = 128
    sink: int = SINK
    recent: int = RECENT
    extra: dict = field(default_factory=dict)

    @property
    def G(self) -> int:
        return self.H // self.Hkv

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


def _w(T, D):
    return (T - SINK - RECENT) // D


# The five benchmark workloads (Llama-3.1-8B: 32 layers, 32 q-heads, 8 KV heads;
# Qwen2.5-7B: 28 layers, 28 q-heads, 4 KV heads; head_dim 128 for both).
WORKLOADS = {
    "llama8b-1layer-4k": Workload("llama8b-1layer-4k", L=1, H=32, Hkv=8, T=4096, B=1, D=32,
                                  W=_w(4096, 32), pattern="bernoulli", rate=0.35, seed=1),
    "llama8b-32k": Workload("llama8b-32k", L=32, H=32, Hkv=8, T=32768, B=1, D=64,
                            W=_w(32768, 64), pattern="profile", rate=0.35, seed=2),
    # All 256 slabs of the model at a 16K context: about 5 GB on the device with
    # the page-backed copies of the in-place path, a small case for profiles of
    # the kernels whose parallelism is one CTA per slab.
    "llama8b-16k": Workload("llama8b-16k", L=32, H=32, Hkv=8, T=16384, B=1, D=32,
                            W=_w(16384, 32), pattern="profile", rate=0.35, seed=6),
    "llama8b-128k": Workload("llama8b-128k", L=32, H=32, Hkv=8, T=131072, B=1, D=128,
                             W=_w(131072, 128), pattern="profile", rate=0.346,
                             physical_target=0.346, outlier_frac=0.01, seed=3),
    # Same head shape, pattern recipe and per-layer sizes as llama8b-128k, 4 layers only:
    # a small case (about 3 GB on the device) for detailed profiles of the same kernels.
    "llama8b-128k-l4": Workload("llama8b-128k-l4", L=4, H=32, Hkv=8, T=131072, B=1, D=128,
                                W=_w(131072, 128), pattern="profile", rate=0.346,
                                physical_target=0.346, outlier_frac=0.01, seed=3),
    # Structural ablations of llama8b-128k at matched physical retention (Sec. 4.5,
    # App. B): the same caches, patterns with parts of the structure removed.
    # Head-only makes the most ragged slabs (whole heads or sink + recent only).
    **{f"llama8b-128k-{k.replace('_', '-')}": Workload(f"llama8b-128k-{k.replace('_', '-')}", L=32, H=32, Hkv=8,
                                                       T=131072, B=1, D=128, W=_w(131072, 128),
                                                       pattern=f"ablation:{k}", rate=0.346, physical_target=0.346,
                                                       outlier_frac=0.01, seed=3)
       for k in ("distance_shuffled", "fully_shuffled", "head_only", "distance_only")},
    "llama8b-b16-ragged": Workload("llama8b-b16-ragged", L=32, H=32, Hkv=8, T=65536, B=16, D=64,
                                   W=_w(65536, 64), pattern="profile", rate=0.25,
                                   ragged=(8192, 65536), seed=4),
    "qwen7b-64k-b4-r20": Workload("qwen7b-64k-b4-r20", L=28, H=28, Hkv=4, T=65536, B=4, D=64,
                                  W=_w(65536, 64), pattern="profile", rate=0.20, seed=5),
    "qwen7b-64k-b4-r35": Workload("qwen7b-64k-b4-r35", L=28, H=28, Hkv=4, T=65536, B=4, D=64,
                                  W=_w(65536, 64), pattern="profile", rate=0.35, seed=5),
    "qwen7b-64k-b4-r50": Workload("qwen7b-64k-b4-r50", L=28, H=28, Hkv=4, T=65536, B=4, D=64,
                                  W=_w(65536, 64), pattern="profile", rate=0.50, seed=5),
}


def context_lengths(wl: Workload) -> np.ndarray:
    """Per-sequence context lengths T_c[b] (int32)."""
    if wl.ragged is None:
        return np.full(wl.B, wl.T, np.int32)
    rng = np.random.default_rng([wl.seed, 11])
    lo, hi = wl.ragged
    return rng.integers(lo, hi + 1, size=wl.B, dtype=np.int64).astype(np.int32)


def _gen_top_entries(scores: np.ndarray, k: int) -> np.ndarray:
    """Generator-only: the k highest-scoring entries of a score tensor become 1
    (ties to the lower flat index), which gives the profile generator an exact
    budget of union bins. No test takes an expected mask from it: the export's
    expected masks come from the oracle."""
    flat = scores.reshape(-1)
    k = int(max(0, min(k, flat.size)))
    order = np.argsort(-flat, kind="stable")
    out = np.zeros(flat.size, np.uint8)
    out[order[:k]] = 1
    return out.reshape(scores.shape)


def _gen_round(x: float) -> int:
    """Generator-only: floor(x + 0.5), the rounding of the generators' budgets."""
    return int(np.floor(x + 0.5))


def bernoulli_pattern(wl: Workload, rng: np.random.Generator) -> np.ndarray:
    """Per (layer, q-head, bin) Bernoulli(rate), with the nearest bin (d=0) always on."""
    M = (rng.random((wl.L, wl.H, wl.D)) < wl.rate).astype(np.uint8)
    if wl.D > 0:
        M[:, :, 0] = 1
    return M


def union_bins_target(wl: Workload) -> int:
    """Number K_U of (layer, KV head, bin) entries the profile generator keeps."""
    if wl.physical_target is not None:
        # Overall physical retention r of a T-token context: kept rows per head
        # = S + R + K_U * W / (L * Hkv) = r * T.
        per_head_bins = (wl.physical_target * wl.T - wl.sink - wl.recent) / wl.W
        return _gen_round(per_head_bins * wl.L * wl.Hkv)
    return _gen_round(wl.rate * wl.L * wl.Hkv * wl.D)


def profile_pattern(wl: Workload, rng: np.random.Generator) -> np.ndarray:
    """Near/far retention profile per (layer, KV head), exact union budget,
    then a random non-empty subset of the group's q-heads per kept bin.

    score_d = w (1 - x_d) + (1 - w) x_d + 0.25 U(0,1), x_d = d / (D - 1),
    w ~ Beta(2, 2) per (layer, KV head). A global Top-K keeps K_U union entries.
    Each kept union bin is given to each q-head of the group with probability
    1/2, redrawn until at least one q-head has it, so the GQA union of M is
    exactly the selected set.
    """
    L, Hkv, D, G = wl.L, wl.Hkv, wl.D, wl.G
    w = rng.beta(2.0, 2.0, size=(L, Hkv, 1))
    x = (np.arange(D) / max(D - 1, 1))[None, None, :]
    score = w * (1.0 - x) + (1.0 - w) * x + 0.25 * rng.random((L, Hkv, D))
    U = _gen_top_entries(score, union_bins_target(wl))
    M = np.zeros((L, Hkv, G, D), np.uint8)
    sel = np.argwhere(U == 1)
    for (l, g, d) in sel:
        while True:
            pick = rng.random(G) < 0.5
            if pick.any():
                break
        M[l, g, :, d] = pick
    return M.reshape(L, Hkv * G, D)


def retention_probs(wl: Workload, levels: int | None = None, seed_offset: int = 0) -> np.ndarray:
    """Synthetic learned retention probabilities P in (0, 1)^{L x H x D} (float32),
    the input of the exact-budget export (Eq. 3): per (layer, q-head) a Beta(2, 2)
    near/far mix w (1 - x_d) + (1 - w) x_d plus noise, squashed by a logistic.
    With `levels`, P is rounded to that many values, which makes many ties."""
    rng = np.random.default_rng([wl.seed, 13, seed_offset])
    w = rng.beta(2.0, 2.0, size=(wl.L, wl.H, 1))
    x = (np.arange(wl.D) / max(wl.D - 1, 1))[None, None, :]
    z = 6.0 * (w * (1.0 - x) + (1.0 - w) * x - 0.5) + rng.normal(0.0, 1.0, (wl.L, wl.H, wl.D))
    P = 1.0 / (1.0 + np.exp(-z))
    if levels:
        P = np.round(P * (levels - 1)) / (levels - 1)
    return P.astype(np.float32)


# ---------------------------------------------------------------- structural ablations
# The paper's ablations (Sec. 4.5 ablation study, App. B) compare Distance-KV
# with patterns of matched physical KV retention that break parts of its
# structure. These recipes derive them from a reference pattern M. The GQA union
# count below only sizes these inputs: it counts (layer, KV head, bin) columns
# with any query head on, i.e. physical bins at full context coverage.

def _gen_group_columns(M: np.ndarray, G: int) -> int:
    """Generator-only: (layer, KV head, bin) columns with any query head on,
    which sizes the ablation patterns."""
    L, H, D = M.shape
    return int(M.reshape(L, H // G, G, D).max(axis=2).sum())


def ablate_distance_shuffled(M: np.ndarray, G: int, rng: np.random.Generator) -> np.ndarray:
    """Per (layer, KV head) one random permutation of the D bins, applied to all
    of its query heads: per-head counts and each group's union count are kept,
    the distance assignment is lost."""
    L, H, D = M.shape
    out = np.empty_like(M)
    for l in range(L):
        for g in range(H // G):
            perm = rng.permutation(D)
            out[l, g * G:(g + 1) * G] = M[l, g * G:(g + 1) * G][:, perm]
    return out


def ablate_fully_shuffled(M: np.ndarray, G: int, rng: np.random.Generator) -> np.ndarray:
    """The G-head columns M[l, gG:(g+1)G, d] permuted over all (layer, KV head,
    bin) positions, and the heads permuted within each column: the logical count
    and the union (physical) count are kept, every layer / head / distance
    correspondence is lost."""
    L, H, D = M.shape
    cols = M.reshape(L, H // G, G, D).transpose(0, 1, 3, 2).reshape(-1, G)  # [(l, g, d)][j]
    cols = cols[rng.permutation(cols.shape[0])]
    cols = np.take_along_axis(cols, np.argsort(rng.random(cols.shape), axis=1), axis=1)
    return np.ascontiguousarray(cols.reshape(L, H // G, D, G).transpose(0, 1, 3, 2).reshape(L, H, D))


def ablate_head_only(M: np.ndarray, G: int) -> np.ndarray:
    """One decision per query head for all its bins. Whole KV groups are kept,
    which is what a kept head costs physically, in descending order of the
    group's union count in M (ties to the lower index), as many as round(U / D)
    for the union count U of M."""
    L, H, D = M.shape
    score = M.reshape(L, H // G, G, D).max(axis=2).sum(axis=2).reshape(-1)  # union bins per (l, g)
    n_groups = int(np.floor(_gen_group_columns(M, G) / D + 0.5))
    order = np.argsort(-score, kind="stable")[:n_groups]
    keep = np.zeros(L * (H // G), np.uint8)
    keep[order] = 1
    return np.ascontiguousarray(np.repeat(keep.reshape(L, H // G, 1, 1), G, axis=2)
                                .repeat(D, axis=3).reshape(L, H, D))


def ablate_distance_only(M: np.ndarray, G: int) -> np.ndarray:
    """One decision per (layer, bin) shared by all query heads of the layer. A
    kept (layer, bin) costs H/G physical bins; the round(U / (H/G)) with the most
    query heads on in M are kept (ties to the lower index)."""
    L, H, D = M.shape
    Hkv = H // G
    score = M.sum(axis=1).reshape(-1)  # query heads on per (l, d)
    n_keep = int(np.floor(_gen_group_columns(M, G) / Hkv + 0.5))
    order = np.argsort(-score, kind="stable")[:n_keep]
    keep = np.zeros(L * D, np.uint8)
    keep[order] = 1
    return np.ascontiguousarray(np.repeat(keep.reshape(L, 1, D), H, axis=1))


ABLATIONS = ("distance_shuffled", "fully_shuffled", "head_only", "distance_only")


def make_pattern(wl: Workload) -> np.ndarray:
    """The workload's retention pattern M in {0,1}^{L x H x D} (uint8)."""
    rng = np.random.default_rng([wl.seed, 7])
    if wl.pattern.startswith("ablation:"):
        kind = wl.pattern.split(":", 1)[1]
        base = make_pattern(wl.with_(pattern="profile"))
        arng = np.random.default_rng([wl.seed, 23])
        if kind == "distance_shuffled":
            return ablate_distance_shuffled(base, wl.G, arng)
        if kind == "fully_shuffled":
            return ablate_fully_shuffled(base, wl.G, arng)
        if kind == "head_only":
            return ablate_head_only(base, wl.G)
        if kind == "distance_only":
            return ablate_distance_only(base, wl.G)
        raise ValueError(f"unknown ablation {kind!r}")
    if wl.pattern == "bernoulli":
        return bernoulli_pattern(wl, rng)
    if wl.pattern == "profile":
        return profile_pattern(wl, rng)
    if wl.pattern == "ones":
        return np.ones((wl.L, wl.H, wl.D), np.uint8)
    if wl.pattern == "zeros":
        return np.zeros((wl.L, wl.H, wl.D), np.uint8)
    raise ValueError(f"unknown pattern recipe {wl.pattern!r}")


def dense_kv(wl: Workload, T_stride: int | None = None, device="cpu", layer_chunk: int = 1):
    """Dense post-RoPE caches K, V, bf16 [L][B][Hkv][T_stride][head_dim] ~ N(0,1).

    Drawn with a torch generator seeded from the workload, K then V, one layer at
    a time (so the device never holds an fp32 copy of a whole cache). A fraction
    `outlier_frac` of key rows (Bernoulli per (layer, b, KV head, position)) is
    multiplied by 8, which is exact in bf16. Rows past a sequence's length are
    drawn as well; the path never reads them.
    """
    import torch
    T_stride = T_stride or wl.T
    shape = (wl.L, wl.B, wl.Hkv, T_stride, wl.head_dim)
    gen = torch.Generator(device=device)
    gen.manual_seed(wl.seed * 1000 + 17)
    K = torch.empty(shape, dtype=torch.bfloat16, device=device)
    V = torch.empty(shape, dtype=torch.bfloat16, device=device)
    for t in (K, V):
        for l0 in range(0, wl.L, layer_chunk):
            l1 = min(wl.L, l0 + layer_chunk)
            t[l0:l1].copy_(torch.randn((l1 - l0,) + shape[1:], generator=gen, device=device,
                                       dtype=torch.float32).to(torch.bfloat16))
    if wl.outlier_frac > 0:
        for l in range(wl.L):
            hit = torch.rand(shape[1:4], generator=gen, device=device) < wl.outlier_frac
            K[l][hit] = K[l][hit] * 8
    return K, V


def decode_inputs(wl: Workload, steps: int, device="cpu", seed_offset: int = 0):
    """Per-step decode inputs, bf16 ~ N(0,1):
    q [steps][L][B][H][hd], k_new and v_new [steps][L][B][Hkv][hd]."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(wl.seed * 1000 + 29 + seed_offset)
    hd = wl.head_dim

    def draw(*shape):
        return torch.randn(shape, generator=gen, device=device,
                           dtype=torch.float32).to(torch.bfloat16)
    q = draw(steps, wl.L, wl.B, wl.H, hd)
    k_new = draw(steps, wl.L, wl.B, wl.Hkv, hd)
    v_new = draw(steps, wl.L, wl.B, wl.Hkv, hd)
    return q, k_new, v_new


def bf16_bits(t) -> np.ndarray:
    """Raw bf16 bit patterns of a (CPU or CUDA) torch bf16 tensor as uint16."""
    import torch
    return t.detach().to("cpu").contiguous().view(torch.int16).numpy().view(np.uint16)


__all__ = ["Workload", "WORKLOADS", "SINK", "RECENT", "context_lengths", "make_pattern", "retention_probs",
           "ABLATIONS", "ablate_distance_shuffled", "ablate_fully_shuffled", "ablate_head_only",
           "ablate_distance_only",
           "union_bins_target", "dense_kv", "decode_inputs",
           "bf16_bits"]
