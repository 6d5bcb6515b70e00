"""Multi-query decode over one compressed cache (dkv_decode_multi): every query
of a sequence attends over the same packed + appended rows, against the fp64
oracle run once per query. Covers one and two column tiles (Q x G <= 8 and
<= 16), G = 1, 4, 7, 8, appended rows, ragged and empty slabs."""
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
    for Q in (0, 5):  # G = 4: Q x G must be <= 16
        q = torch.zeros((w.B, max(Q, 1), w.H, w.head_dim), dtype=torch.bfloat16, device=cuda)
        out = torch.zeros((w.B, max(Q, 1), w.H, w.head_dim), dtype=torch.float32, device=cuda)
        with pytest.raises(dkv.DkvError):
            dkv.dkv_decode_multi(case.plan, 0, q, Q, n_app, case.Kc, case.Vc, out)
    case.close()


@pytest.mark.slow
def test_multi_query_full_size_sampled(cuda):
    """llama8b-128k, 4 queries per sequence (16 columns: the two-tile kernel),
    bench.py's plan and reserve, sampled slabs against the oracle."""
    import bench
    w = I.WORKLOADS["llama8b-128k"]
    reserve = bench.reserve_rows(bench.DEFAULT_STEPS, bench.DEFAULT_WARMUP)
    env = bench.setup(w, cuda, reserve)
    dkv.dkv_compact(env["plan"], env["K"], env["V"], env["Kc"], env["Vc"], T_stride=env["T_stride"])
    Q = 4
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
    for g in (0, 3, 7):
        h = layer * NHl + g
        kept = torch.from_numpy(om.idx[om.ioff[h]:om.ioff[h + 1]].astype(np.int64)).to(cuda)
        Krows = I.bf16_bits(env["K"][layer, 0, g].index_select(0, kept))
        Vrows = I.bf16_bits(env["V"][layer, 0, g].index_select(0, kept))
        for qi in range(Q):
            want = O.attend(I.bf16_bits(q[0, qi, g * w.G:(g + 1) * w.G]), Krows, Vrows)
            assert_close(got[0, qi, g * w.G:(g + 1) * w.G], want, f"KV head {g} query {qi}")
    env["plan"].close()
