"""dkv_decode_attn_noalloc: the decode entry point for callers that may not
allocate device memory (a host framework that owns the device pool and forbids
cudaMalloc). It must give the same output as dkv_decode_attn on the same inputs,
on consecutive calls that reuse its fixed scratch array, and must not allocate.

This file is named to be collected last, so a run stopped at its first failure
has already run every other test.
"""
import numpy as np
import pytest
import torch

import paper_2609_32663_gb300.dkv as dkv
from paper_2609_32663_gb300 import inputs as I
from parity import MAX_ABS, REL_L2, Case

pytestmark = pytest.mark.gpu


def close(a, b):
    a = a.double().cpu().numpy()
    b = b.double().cpu().numpy()
    assert np.isfinite(a).all()
    err = np.abs(a - b).max()
    rel = np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30)
    assert err <= MAX_ABS and rel <= REL_L2, (err, rel)


@pytest.fixture(scope="module")
def case(cuda):
    from paper_2609_32663_gb300 import build
    build.build_library()
    torch.cuda.set_device(cuda)
    wl = I.Workload("noalloc", L=2, H=16, Hkv=4, T=20000, B=3, D=16, W=(20000 - 1152) // 16 + 1,
                    pattern="profile", rate=0.35, ragged=(3000, 20000), seed=91)
    c = Case(wl, reserve=4)
    yield c
    c.close()


def metadata(c):
    info = dkv.dkv_plan_query(c.plan)
    return info.d_len, info.d_off, info.d_ioff


def test_noalloc_matches_decode_attn_on_two_calls(case):
    c, wl = case, case.wl
    d_len, d_off, d_ioff = metadata(c)
    q, _, _ = I.decode_inputs(wl, 2, seed_offset=5)
    ref = torch.empty((wl.B, wl.H, 128), dtype=torch.float32, device=c.dev)
    got = torch.empty_like(ref)
    for call in range(2):
        for layer in range(wl.L):
            qd = q[call, layer].to(c.dev)
            dkv.dkv_decode_attn(c.plan, layer, qd, None, None, None, c.Kc, c.Vc, ref)
            got.fill_(float("nan"))
            dkv.dkv_decode_attn_noalloc(c.sh, wl.B, layer, c.reserve, d_len, d_off, d_ioff, qd, None, None, None,
                                        c.Kc, c.Vc, got)
            torch.cuda.synchronize()
            close(got, ref)


def test_noalloc_appends_like_decode_attn(case):
    """Two steps with this step's token appended: outputs and cache bytes agree."""
    c, wl = case, case.wl
    d_len, d_off, d_ioff = metadata(c)
    Kc2, Vc2 = c.Kc.clone(), c.Vc.clone()
    q, kn, vn = I.decode_inputs(wl, 2, seed_offset=9)
    n1 = torch.zeros(wl.B, dtype=torch.int32, device=c.dev)
    n2 = torch.zeros_like(n1)
    st = torch.zeros(1, dtype=torch.int32, device=c.dev)
    ref = torch.empty((wl.B, wl.H, 128), dtype=torch.float32, device=c.dev)
    got = torch.empty_like(ref)
    for step in range(2):
        for layer in range(wl.L):
            args = (q[step, layer].to(c.dev), kn[step, layer].to(c.dev), vn[step, layer].to(c.dev))
            dkv.dkv_decode_attn(c.plan, layer, *args, n1, c.Kc, c.Vc, ref)
            dkv.dkv_decode_attn_noalloc(c.sh, wl.B, layer, c.reserve, d_len, d_off, d_ioff, *args, n2, Kc2, Vc2,
                                        got, status=st)
            torch.cuda.synchronize()
            close(got, ref)
        dkv.dkv_advance(c.plan, n1)
        dkv.dkv_advance(c.plan, n2)
    assert torch.equal(c.Kc.view(torch.int16), Kc2.view(torch.int16))
    assert torch.equal(c.Vc.view(torch.int16), Vc2.view(torch.int16))
    assert int(st.item()) == 0


def test_noalloc_allocates_nothing(case):
    c, wl = case, case.wl
    d_len, d_off, d_ioff = metadata(c)
    q = torch.randn((wl.B, wl.H, 128), device=c.dev).to(torch.bfloat16)
    out = torch.empty((wl.B, wl.H, 128), dtype=torch.float32, device=c.dev)
    dkv.dkv_decode_attn_noalloc(c.sh, wl.B, 0, c.reserve, d_len, d_off, d_ioff, q, None, None, None, c.Kc, c.Vc, out)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    torch_bytes = torch.cuda.memory_allocated()
    calls = 64
    for i in range(calls):
        dkv.dkv_decode_attn_noalloc(c.sh, wl.B, i % wl.L, c.reserve, d_len, d_off, d_ioff, q, None, None, None,
                                    c.Kc, c.Vc, out)
    torch.cuda.synchronize()
    # Device-wide free memory also moves with the driver's own bookkeeping, so the
    # check is for growth: an allocation per call would lose >= 64 x its size.
    assert free0 - torch.cuda.mem_get_info()[0] < (2 << 20)
    assert torch.cuda.memory_allocated() == torch_bytes


def test_noalloc_rejects_workspace_beyond_the_static_array(case):
    c = case
    big = dkv.Shape(L=1, H=64, H_kv=8, D=1)  # 512 sequences x 8 KV heads x G=8 partials > 8 MiB
    d_len, d_off, d_ioff = metadata(c)
    out = torch.empty((512, 64, 128), dtype=torch.float32, device=c.dev)
    q = torch.zeros((512, 64, 128), dtype=torch.bfloat16, device=c.dev)
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_decode_attn_noalloc(big, 512, 0, 0, d_len, d_off, d_ioff, q, None, None, None, c.Kc, c.Vc, out)
    assert e.value.status == dkv.DKV_ERR_INVALID_ARG
    assert b"static scratch" in dkv.lib().dkv_last_error()
