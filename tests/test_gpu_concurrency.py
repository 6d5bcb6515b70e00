"""Use patterns a host framework relies on: two plans decoding at once on two
streams, the entry points captured in CUDA graphs, and plans created and freed
repeatedly without growing device memory."""
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


def wl(seed, **kw):
    base = dict(L=2, H=8, Hkv=2, T=7000, B=2, D=8, W=(7000 - 1152) // 8, pattern="profile", rate=0.4,
                ragged=(500, 7000), seed=seed)
    base.update(kw)
    return I.Workload(f"c{seed}", **base)


def test_two_plans_on_two_streams():
    a, b = Case(wl(61)), Case(wl(62, H=14, Hkv=2))
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    qa, _, _ = I.decode_inputs(a.wl, 1)
    qb, _, _ = I.decode_inputs(b.wl, 1)
    outs = {}
    torch.cuda.synchronize()
    for layer in range(2):
        for c, q, s, tag in ((a, qa, sa, "a"), (b, qb, sb, "b")):
            with torch.cuda.stream(s):
                o = torch.empty((c.wl.B, c.wl.H, 128), dtype=torch.float32, device=c.dev)
                dkv.dkv_decode_attn(c.plan, layer, q[0, layer].to(c.dev), None, None, None, c.Kc, c.Vc, o,
                                    stream=s)
                outs[(tag, layer)] = o
    torch.cuda.synchronize()
    for c, q, tag in ((a, qa, "a"), (b, qb, "b")):
        for layer in range(2):
            want = O.decode(c.om, layer, c.wl.B, c.wl.H, c.wl.Hkv, I.bf16_bits(q[0, layer]), c.oKc, c.oVc)
            assert_close(outs[(tag, layer)].double().cpu().numpy(), want, f"{tag} layer {layer}")
    a.close()
    b.close()


def test_multi_query_and_export_in_graphs(cuda):
    c = Case(wl(63))
    w = c.wl
    Q = 2
    q = torch.randn((w.B, Q, w.H, 128), device=c.dev).to(torch.bfloat16)
    out = torch.empty((w.B, Q, w.H, 128), dtype=torch.float32, device=c.dev)
    P = torch.from_numpy(I.retention_probs(I.WORKLOADS["llama8b-32k"])).to(c.dev)
    K = P.numel() // 3
    M = torch.empty(P.shape, dtype=torch.uint8, device=c.dev)
    ws = torch.empty(dkv.dkv_topk_workspace_bytes() // 4 + 1, dtype=torch.int32, device=c.dev)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        dkv.dkv_decode_multi(c.plan, 0, q, Q, None, c.Kc, c.Vc, out)
        dkv.dkv_topk_mask(P, K, M, ws)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        dkv.dkv_decode_multi(c.plan, 0, q, Q, None, c.Kc, c.Vc, out)
        dkv.dkv_topk_mask(P, K, M, ws)
    out.fill_(float("nan"))
    M.fill_(7)
    g.replay()
    torch.cuda.synchronize()
    qh = I.bf16_bits(q)
    for j in range(Q):
        want = O.decode(c.om, 0, w.B, w.H, w.Hkv, qh[:, j], c.oKc, c.oVc)
        assert_close(out[:, j].double().cpu().numpy(), want, f"query {j}")
    assert np.array_equal(M.cpu().numpy(), O.topk_mask(P.cpu().numpy(), K))
    c.close()


def test_plans_do_not_leak_device_memory():
    w = wl(64)
    sh = dkv.Shape(L=w.L, H=w.H, H_kv=w.Hkv, D=w.D, sink=w.sink, recent=w.recent, bin_width=w.W)
    M, Tc = I.make_pattern(w), I.context_lengths(w)
    dkv.dkv_map_pattern(M, Tc, sh, reserve_rows=2).close()
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(20):
        dkv.dkv_map_pattern(M, Tc, sh, reserve_rows=2).close()
        dkv.dkv_map_pattern_inplace(M, Tc, sh, int(Tc.max()) + 2, reserve_rows=2).close()
    torch.cuda.synchronize()
    assert free0 - torch.cuda.mem_get_info()[0] < (4 << 20)
