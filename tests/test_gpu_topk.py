"""Exact-budget pattern export on the GPU (dkv_topk_mask, Eq. 3 / App. A.3)
against the oracle's global Top-K: the masks must be identical bit for bit,
including ties (lower flat index first), NaN (last), +0 == -0 and the budget
edge cases K = 0, 1, n - 1, n."""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2609_32663_gb300.dkv as dkv
from paper_2609_32663_gb300 import inputs as I

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built(cuda):
    from paper_2609_32663_gb300 import build
    build.build_library()
    torch.cuda.set_device(cuda)


def gpu_mask(P, K, cuda):
    Pd = torch.from_numpy(np.ascontiguousarray(P, np.float32)).to(cuda)
    Md = torch.full(Pd.shape, 7, dtype=torch.uint8, device=cuda)  # every byte must be written
    ws = torch.empty(dkv.dkv_topk_workspace_bytes() // 4 + 1, dtype=torch.int32, device=cuda)
    ws[0] = 0
    dkv.dkv_topk_mask(Pd, K, Md, ws)
    torch.cuda.synchronize()
    if 0 < K < P.size:
        assert int(ws[0].item()) == 0  # no grid barrier wait ran out
    return Md.cpu().numpy()


@pytest.mark.parametrize("name", ["llama8b-128k", "qwen7b-64k-b4-r35", "llama8b-1layer-4k", "llama8b-32k"])
@pytest.mark.parametrize("rho", [0.05, 0.2, 0.346, 0.5, 0.9])
def test_workload_shaped_probabilities(name, rho, cuda):
    wl = I.WORKLOADS[name]
    P = I.retention_probs(wl)
    K = dkv.dkv_budget(rho, wl.L, wl.H, wl.D)
    assert K == O.budget(rho, wl.L, wl.H, wl.D)
    M = gpu_mask(P, K, cuda)
    assert np.array_equal(M, O.topk_mask(P, K))
    assert int(M.sum()) == K


@pytest.mark.parametrize("levels", [2, 3, 17, 256])
def test_heavy_ties_go_to_lower_index(levels, cuda):
    wl = I.WORKLOADS["llama8b-128k"]
    P = I.retention_probs(wl, levels=levels)
    n = P.size
    for K in (1, 777, n // 3, n // 2 + 1, n - 1):
        assert np.array_equal(gpu_mask(P, K, cuda), O.topk_mask(P, K)), (levels, K)


def test_special_values(cuda):
    rng = np.random.default_rng(5)
    vals = np.array([0.0, -0.0, np.nan, np.inf, -np.inf, 1.0, -1.0, 0.5, 1e-38, -1e-38, 3e38], np.float32)
    P = rng.choice(vals, 50000).astype(np.float32)
    n = P.size
    for K in (0, 1, 2, 100, 20000, n - 5000, n - 1, n):
        assert np.array_equal(gpu_mask(P, K, cuda), O.topk_mask(P, K)), K


def test_all_equal_takes_first_k(cuda):
    P = np.full(100003, 0.25, np.float32)
    for K in (0, 1, 50000, 100002, 100003):
        want = np.zeros(P.size, np.uint8)
        want[:K] = 1
        assert np.array_equal(gpu_mask(P, K, cuda), want)


def test_tiny_and_ragged_sizes(cuda):
    rng = np.random.default_rng(9)
    for n in (1, 2, 31, 32, 33, 255, 256, 257, 4095, 4096, 4097, 70001):
        P = rng.random(n).astype(np.float32)
        for K in sorted({0, 1, n // 2, max(n - 1, 0), n}):
            assert np.array_equal(gpu_mask(P, K, cuda), O.topk_mask(P, K)), (n, K)


@pytest.mark.parametrize("n", [393_215, 400_000, 1_000_003])
def test_special_values_on_many_ctas(n, cuda):
    """Ties, NaN, +-0 and +-inf spread over many CTAs of the grid (the tie
    prefix crosses CTA and warp ranges)."""
    rng = np.random.default_rng(n)
    vals = np.array([0.0, -0.0, np.nan, np.inf, -np.inf, 1.0, -1.0, 0.5, 0.25, 1e-30], np.float32)
    P = rng.choice(vals, n).astype(np.float32)
    for K in (1, n // 3, n - 2):
        assert np.array_equal(gpu_mask(P, K, cuda), O.topk_mask(P, K)), (n, K)


def test_large_input_many_ctas(cuda):
    rng = np.random.default_rng(11)
    n = 8 * 1024 * 1024 + 12345
    P = (rng.integers(0, 1 << 20, n) / float(1 << 20)).astype(np.float32)  # many ties
    for K in (1, n // 7, n - 3):
        assert np.array_equal(gpu_mask(P, K, cuda), O.topk_mask(P, K)), K


def test_repeated_calls_reuse_workspace(cuda):
    wl = I.WORKLOADS["qwen7b-64k-b4-r35"]
    P = I.retention_probs(wl, seed_offset=1)
    K = dkv.dkv_budget(0.35, wl.L, wl.H, wl.D)
    a, b = gpu_mask(P, K, cuda), gpu_mask(P, K, cuda)
    assert np.array_equal(a, b)


def test_exported_pattern_feeds_the_map(cuda):
    """The exported pattern is a valid dkv_map_pattern input, and the map of it
    equals the oracle's map of the oracle's mask."""
    wl = I.WORKLOADS["llama8b-1layer-4k"]
    P = I.retention_probs(wl)
    K = dkv.dkv_budget(0.35, wl.L, wl.H, wl.D)
    M = gpu_mask(P, K, cuda)
    Tc = I.context_lengths(wl)
    sh = dkv.Shape(L=wl.L, H=wl.H, H_kv=wl.Hkv, D=wl.D, sink=wl.sink, recent=wl.recent, bin_width=wl.W)
    geo = O.Geometry(L=wl.L, H=wl.H, Hkv=wl.Hkv, D=wl.D, sink=wl.sink, recent=wl.recent, bin_width=wl.W)
    plan = dkv.dkv_map_pattern(M, Tc, sh)
    ln, off, ioff, idx = dkv.dkv_plan_read(plan)
    om = O.map_pattern(O.topk_mask(P, K), Tc, geo)
    assert np.array_equal(ln, om.len) and np.array_equal(idx, om.idx)
    plan.close()


def test_grid_barrier_wait_runs_out_and_reports(monkeypatch, cuda):
    """DKV_FAULT=barrier: the export's grid barriers wait for one CTA more than
    the grid has. The first wait runs out at its bound (2 s), the status word
    in the workspace is set and the kernel returns; the next call is exact."""
    import time
    rng = np.random.default_rng(3)
    P = rng.random(300_000).astype(np.float32)
    K = 1000
    Pd = torch.from_numpy(P).to(cuda)
    Md = torch.zeros(P.shape, dtype=torch.uint8, device=cuda)
    ws = torch.zeros(dkv.dkv_topk_workspace_bytes() // 4 + 1, dtype=torch.int32, device=cuda)
    monkeypatch.setenv("DKV_FAULT", "barrier")
    t0 = time.time()
    dkv.dkv_topk_mask(Pd, K, Md, ws)
    torch.cuda.synchronize()
    elapsed = time.time() - t0
    monkeypatch.delenv("DKV_FAULT")
    assert int(ws[0].item()) != 0 and elapsed < 60
    assert np.array_equal(gpu_mask(P, K, cuda), O.topk_mask(P, K))
