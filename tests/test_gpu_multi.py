"""Multi-query decode over one compressed cache (dkv_decode_multi): every query
of a sequence attends over the same packed + appended rows, against the fp64
oracle run once per query, every output row within the parity tolerances.
Covers the mma.sync kernels (one and two column tiles: Q x G <= 8 and <= 16)
and the tcgen05 kernel with its combine launch (17 to 64 columns), G = 1 to 8,
appended rows, ragged and empty slabs, slabs shorter than a tile, slabs over
many CTAs, outlier keys (running-max rescales), and full-size workloads."""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2609_32663_gb300.dkv as dkv
from paper_2609_32663_gb300 import inputs as I
from parity import Case, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built(cuda):
    from paper_2609_32663_gb300 import build
    build.build_library()
    torch.cuda.set_device(cuda)


def wl(name="m", **kw):
    base = dict(L=2, H=8, Hkv=2, T=5000, B=3, D=12, W=-(-(5000 - 1152) // 12), pattern="profile", rate=0.4,
                ragged=(0, 5000), seed=21)
    base.update(kw)
    return I.Workload(name, **base)


def multi_q(w, Q, seed=0):
    g = torch.Generator().manual_seed(1234 + seed)
    return torch.randn((w.L, w.B, Q, w.H, w.head_dim), generator=g).to(torch.bfloat16)


def run_case(w, Q, steps_before=2):
    case = Case(w, reserve=8)
    # a few decode steps with appends, so the multi-query calls also see appended rows
    if steps_before:
        case.decode_steps(steps_before, append=True)
    na = np.full(w.B, steps_before, np.int32)
    n_app = torch.from_numpy(na).to(case.dev)
    q = multi_q(w, Q)
    out = torch.full((w.B, Q, w.H, w.head_dim), float("nan"), dtype=torch.float32, device=case.dev)
    for layer in range(w.L):
        dkv.dkv_decode_multi(case.plan, layer, q[layer].to(case.dev), Q, n_app, case.Kc, case.Vc, out)
        torch.cuda.synchronize()
        got = out.double().cpu().numpy()
        for qi in range(Q):
            want = O.decode(case.om, layer, w.B, w.H, w.Hkv, I.bf16_bits(q[layer][:, qi]), case.oKc, case.oVc,
                            n_rows_app=na)
            assert_close(got[:, qi], want, f"layer {layer} query {qi}")
    assert dkv.dkv_plan_status(case.plan) == 0
    case.close()


@pytest.mark.parametrize("G,Q", [(4, 1), (4, 2), (4, 3), (4, 4), (7, 1), (7, 2), (8, 2), (1, 8), (1, 16), (2, 5),
                                 (3, 5), (5, 3), (6, 2), (2, 8)])
def test_multi_query_matches_oracle(G, Q):
    run_case(wl(H=2 * G, Hkv=2, seed=G * 10 + Q), Q)


# (G, Q) with Q x G in 17..64: the tcgen05 kernel.
TC_CASES = [(1, 17), (1, 64), (2, 9), (3, 6), (4, 5), (4, 8), (4, 16), (5, 4), (6, 3), (7, 4), (7, 9), (8, 3),
            (8, 8)]


@pytest.mark.parametrize("G,Q", TC_CASES, ids=[f"G{g}-Q{q}" for g, q in TC_CASES])
def test_multi_query_tcgen05_matches_oracle(G, Q):
    run_case(wl(H=2 * G, Hkv=2, seed=300 + G * 10 + Q), Q)


@pytest.mark.parametrize("G,Q", [(4, 8), (7, 9), (1, 64)])
def test_multi_query_tcgen05_long_slabs_with_outliers(G, Q):
    """Slabs of ~14-30 K rows over many CTAs (several 64-row tiles each, partials
    merged by the combine launch) with 1 % of key rows x 8 (scores that move the
    running max late in a segment)."""
    w = wl(L=2, H=2 * G, Hkv=2, T=40000, B=2, D=24, W=-(-(40000 - 1152) // 24), ragged=(20000, 40000),
           outlier_frac=0.01, seed=400 + G)
    run_case(w, Q, steps_before=1)


@pytest.mark.parametrize("Tc", [[0, 1, 63, 64, 65], [1152, 1153, 1300, 2000, 5]])
def test_multi_query_tcgen05_short_and_empty_slabs(Tc):
    """Contexts of 0 to a few tiles: empty slabs (zeros), slabs shorter than a
    tile, tiles straddling slabs, several segments per CTA."""
    w = wl(L=2, H=16, Hkv=2, T=max(Tc), B=len(Tc), D=8, W=200, pattern="bernoulli", rate=0.5, ragged=None,
           seed=77)
    case = Case(w, reserve=4, Tc=np.array(Tc, np.int32))
    Q = 5  # G = 8: 40 columns
    na = np.zeros(w.B, np.int32)
    n_app = torch.from_numpy(na).to(case.dev)
    q = multi_q(w, Q, seed=5)
    out = torch.full((w.B, Q, w.H, w.head_dim), float("nan"), dtype=torch.float32, device=case.dev)
    for layer in range(w.L):
        dkv.dkv_decode_multi(case.plan, layer, q[layer].to(case.dev), Q, n_app, case.Kc, case.Vc, out)
        torch.cuda.synchronize()
        got = out.double().cpu().numpy()
        for qi in range(Q):
            want = O.decode(case.om, layer, w.B, w.H, w.Hkv, I.bf16_bits(q[layer][:, qi]), case.oKc, case.oVc,
                            n_rows_app=na)
            assert_close(got[:, qi], want, f"layer {layer} query {qi}")
    assert dkv.dkv_plan_status(case.plan) == 0
    case.close()


def test_multi_query_tcgen05_slab_aligned_partition(cuda):
    """Few slabs of uneven lengths, two of them empty: the tcgen05 kernel gives
    each slab a whole number of CTAs (no CTA range holds a slab boundary) and an
    empty slab lies inside the CTA that starts the next one. Two layers, with
    rows appended in an earlier step (the appended rows move every boundary)."""
    Tc = [30000, 0, 12000, 25000]
    w = wl(L=2, H=16, Hkv=2, T=max(Tc), B=len(Tc), D=24, W=-(-(30000 - 1152) // 24), ragged=None,
           outlier_frac=0.01, seed=123)
    case = Case(w, reserve=4, Tc=np.array(Tc, np.int32))
    Q = 5  # G = 8: 40 columns
    gen = torch.Generator().manual_seed(4321)
    kn = torch.randn((w.L, w.B, w.Hkv, w.head_dim), generator=gen).to(torch.bfloat16)
    vn = torch.randn((w.L, w.B, w.Hkv, w.head_dim), generator=gen).to(torch.bfloat16)
    n_app = torch.zeros(w.B, dtype=torch.int32, device=case.dev)
    na = np.zeros(w.B, np.int32)
    step_out = torch.empty((w.B, w.H, w.head_dim), dtype=torch.float32, device=case.dev)
    qs = torch.randn((w.L, w.B, w.H, w.head_dim), generator=gen).to(torch.bfloat16)
    for layer in range(w.L):
        dkv.dkv_decode_attn(case.plan, layer, qs[layer].to(case.dev), kn[layer].to(case.dev), vn[layer].to(case.dev),
                            n_app, case.Kc, case.Vc, step_out)
        O.append(case.om, layer, w.B, w.Hkv, case.reserve, na, I.bf16_bits(kn[layer]), I.bf16_bits(vn[layer]),
                 case.oKc, case.oVc)
    dkv.dkv_advance(case.plan, n_app)
    na += 1
    q = multi_q(w, Q, seed=13)
    out = torch.full((w.B, Q, w.H, w.head_dim), float("nan"), dtype=torch.float32, device=case.dev)
    for layer in range(w.L):
        dkv.dkv_decode_multi(case.plan, layer, q[layer].to(case.dev), Q, n_app, case.Kc, case.Vc, out)
        torch.cuda.synchronize()
        got = out.double().cpu().numpy()
        for qi in range(Q):
            want = O.decode(case.om, layer, w.B, w.H, w.Hkv, I.bf16_bits(q[layer][:, qi]), case.oKc, case.oVc,
                            n_rows_app=na)
            assert_close(got[:, qi], want, f"layer {layer} query {qi}")
    assert dkv.dkv_plan_status(case.plan) == 0
    case.close()


def test_multi_query_tcgen05_twice_in_a_row_and_after_the_decode_step(cuda):
    """The tcgen05 kernel's workspace and slab bounds are reused: two calls in a
    row on different layers, then a decode step, then the multi-query again."""
    w = wl(seed=91, H=8, Hkv=2)
    case = Case(w, reserve=4)
    Q = 6  # G = 4: 24 columns
    n_app = torch.zeros(w.B, dtype=torch.int32, device=cuda)
    q = multi_q(w, Q, seed=9)
    outs = [torch.full((w.B, Q, w.H, w.head_dim), float("nan"), dtype=torch.float32, device=cuda) for _ in range(3)]
    dkv.dkv_decode_multi(case.plan, 0, q[0].to(cuda), Q, n_app, case.Kc, case.Vc, outs[0])
    dkv.dkv_decode_multi(case.plan, 1, q[1].to(cuda), Q, n_app, case.Kc, case.Vc, outs[1])
    step = torch.empty((w.B, w.H, w.head_dim), dtype=torch.float32, device=cuda)
    dkv.dkv_decode_attn(case.plan, 0, q[0][:, 0].contiguous().to(cuda), None, None, n_app, case.Kc, case.Vc, step)
    dkv.dkv_decode_multi(case.plan, 0, q[0].to(cuda), Q, n_app, case.Kc, case.Vc, outs[2])
    torch.cuda.synchronize()
    na = np.zeros(w.B, np.int32)
    for k, layer in ((0, 0), (1, 1), (2, 0)):
        got = outs[k].double().cpu().numpy()
        for qi in range(Q):
            want = O.decode(case.om, layer, w.B, w.H, w.Hkv, I.bf16_bits(q[layer][:, qi]), case.oKc, case.oVc,
                            n_rows_app=na)
            assert_close(got[:, qi], want, f"call {k} query {qi}")
    assert dkv.dkv_plan_status(case.plan) == 0
    case.close()


def test_multi_query_without_appended_rows():
    run_case(wl(seed=5), 4, steps_before=0)


def test_single_query_equals_decode_step_without_append(cuda):
    w = wl(seed=8)
    case = Case(w, reserve=4)
    q = multi_q(w, 1)
    n_app = torch.zeros(w.B, dtype=torch.int32, device=cuda)
    a = torch.empty((w.B, 1, w.H, w.head_dim), dtype=torch.float32, device=cuda)
    b = torch.empty((w.B, w.H, w.head_dim), dtype=torch.float32, device=cuda)
    for layer in range(w.L):
        dkv.dkv_decode_multi(case.plan, layer, q[layer].to(cuda), 1, n_app, case.Kc, case.Vc, a)
        dkv.dkv_decode_attn(case.plan, layer, q[layer][:, 0].contiguous().to(cuda), None, None, n_app, case.Kc,
                            case.Vc, b)
        torch.cuda.synchronize()
        assert torch.allclose(a[:, 0], b, rtol=1e-5, atol=1e-5)
    case.close()


def test_multi_query_rejects_bad_counts(cuda):
    w = wl(seed=9)
    case = Case(w, reserve=2)
    n_app = torch.zeros(w.B, dtype=torch.int32, device=cuda)
    for Q in (0, 17):  # G = 4: Q x G must be <= 64
        q = torch.zeros((w.B, max(Q, 1), w.H, w.head_dim), dtype=torch.bfloat16, device=cuda)
        out = torch.zeros((w.B, max(Q, 1), w.H, w.head_dim), dtype=torch.float32, device=cuda)
        with pytest.raises(dkv.DkvError):
            dkv.dkv_decode_multi(case.plan, 0, q, Q, n_app, case.Kc, case.Vc, out)
    case.close()


@pytest.mark.slow
@pytest.mark.parametrize("name,Q", [("llama8b-128k", 4), ("llama8b-128k", 16), ("qwen7b-64k-b4-r35", 4)])
def test_multi_query_full_size_sampled(cuda, name, Q):
    """Full-size workloads with bench.py's plan and reserve, sampled slabs
    against the oracle: llama8b-128k with 4 queries (16 columns: the two-tile
    mma.sync kernel) and 16 queries (64 columns: tcgen05), qwen7b-64k-b4-r35
    with 4 queries (28 columns: tcgen05)."""
    import bench
    w = I.WORKLOADS[name]
    reserve = bench.reserve_rows(bench.DEFAULT_STEPS, bench.DEFAULT_WARMUP)
    env = bench.setup(w, cuda, reserve)
    dkv.dkv_compact(env["plan"], env["K"], env["V"], env["Kc"], env["Vc"], T_stride=env["T_stride"])
    q = multi_q(w.with_(L=1), Q, seed=3)[0]
    n_app = torch.zeros(w.B, dtype=torch.int32, device=cuda)
    out = torch.empty((w.B, Q, w.H, w.head_dim), dtype=torch.float32, device=cuda)
    layer = 7
    dkv.dkv_decode_multi(env["plan"], layer, q.to(cuda), Q, n_app, env["Kc"], env["Vc"], out)
    torch.cuda.synchronize()
    got = out.double().cpu().numpy()
    _, geo = __import__("parity").shapes(w)
    om = O.map_pattern(env["M"], env["Tc"], geo, reserve=reserve)
    NHl = w.B * w.Hkv
    for b, g in ((0, 0), (w.B - 1, w.Hkv - 1), (w.B // 2, w.Hkv // 2)):
        h = layer * NHl + b * w.Hkv + g
        kept = torch.from_numpy(om.idx[om.ioff[h]:om.ioff[h + 1]].astype(np.int64)).to(cuda)
        Krows = I.bf16_bits(env["K"][layer, b, g].index_select(0, kept))
        Vrows = I.bf16_bits(env["V"][layer, b, g].index_select(0, kept))
        for qi in range(Q):
            want = O.attend(I.bf16_bits(q[b, qi, g * w.G:(g + 1) * w.G]), Krows, Vrows)
            assert_close(got[b, qi, g * w.G:(g + 1) * w.G], want, f"{name} Q={Q} seq {b} KV head {g} query {qi}")
    assert dkv.dkv_plan_status(env["plan"]) == 0
    env["plan"].close()
    del env
    torch.cuda.empty_cache()
