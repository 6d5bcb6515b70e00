"""dkv_decode_attn_noalloc: the decode entry point for callers that may not
allocate device memory (a host framework that owns the device pool and forbids
cudaMalloc). On consecutive calls that reuse its fixed scratch array it must
match the fp64 oracle (per output row, the tolerances of every parity test) and
give the same output as dkv_decode_attn on the same inputs, and it must not
allocate.

Group sizes 1, 3, 4, 5, 7 and 8 cover both shapes of the fp32 kernel it runs
(8 lanes a row for G <= 4, 16 lanes a row for G >= 5); odd G with an odd number
of (sequence, KV head) slabs per layer gives an odd count of partial records,
the case where an unpadded workspace carve-up would misalign the warp records.

This file is named to be collected last, so a run stopped at its first failure
has already run every other test.
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2609_32663_gb300.dkv as dkv
from paper_2609_32663_gb300 import inputs as I
from parity import MAX_ABS, REL_L2, Case, assert_close

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


# (G, H_kv, B): odd G with B * H_kv odd, MQA (H_kv = 1) among them.
GROUPS = [(1, 3, 1), (3, 1, 3), (4, 2, 2), (5, 1, 1), (7, 1, 3), (8, 1, 2)]


@pytest.mark.parametrize("G,Hkv,B", GROUPS, ids=[f"G{g}-Hkv{k}-B{b}" for g, k, b in GROUPS])
def test_noalloc_matches_oracle_and_decode_attn_on_two_calls(G, Hkv, B, cuda):
    """Two decode steps in a row, each appending the step's key/value: every
    output row against the oracle, the whole output against dkv_decode_attn on a
    copy of the cache, and the cache bytes after the appends."""
    from paper_2609_32663_gb300 import build
    build.build_library()
    torch.cuda.set_device(cuda)
    wl = I.Workload(f"noalloc-G{G}", L=2, H=G * Hkv, Hkv=Hkv, T=9000, B=B, D=12, W=(9000 - 1152) // 12 + 1,
                    pattern="profile", rate=0.35, ragged=(1500, 9000), seed=100 + G)
    c = Case(wl, reserve=3)
    try:
        d_len, d_off, d_ioff = metadata(c)
        Kc2, Vc2 = c.Kc.clone(), c.Vc.clone()
        q, kn, vn = I.decode_inputs(wl, 2, seed_offset=11)
        n1 = torch.zeros(wl.B, dtype=torch.int32, device=c.dev)
        n2 = torch.zeros_like(n1)
        na = np.zeros(wl.B, np.int32)
        st = torch.zeros(1, dtype=torch.int32, device=c.dev)
        ref = torch.empty((wl.B, wl.H, 128), dtype=torch.float32, device=c.dev)
        got = torch.empty_like(ref)
        for step in range(2):
            for layer in range(wl.L):
                args = (q[step, layer].to(c.dev), kn[step, layer].to(c.dev), vn[step, layer].to(c.dev))
                got.fill_(float("nan"))
                dkv.dkv_decode_attn_noalloc(c.sh, wl.B, layer, c.reserve, d_len, d_off, d_ioff, *args, n2, Kc2,
                                            Vc2, got, status=st)
                dkv.dkv_decode_attn(c.plan, layer, *args, n1, c.Kc, c.Vc, ref)
                O.append(c.om, layer, wl.B, wl.Hkv, c.reserve, na, I.bf16_bits(kn[step, layer]),
                         I.bf16_bits(vn[step, layer]), c.oKc, c.oVc)
                want = O.decode(c.om, layer, wl.B, wl.H, wl.Hkv, I.bf16_bits(q[step, layer]), c.oKc, c.oVc,
                                n_rows_app=na + 1)
                torch.cuda.synchronize()
                assert_close(got.double().cpu().numpy(), want, f"G={G} step {step} layer {layer} (oracle)")
                close(got, ref)
            dkv.dkv_advance(c.plan, n1)
            dkv.dkv_advance(c.plan, n2)
            na += 1
        assert int(st.item()) == 0
        assert torch.equal(c.Kc.view(torch.int16), Kc2.view(torch.int16))
        assert torch.equal(c.Vc.view(torch.int16), Vc2.view(torch.int16))
        c.check_packed_with_appends(na)
    finally:
        c.close()


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
            want = O.decode(c.om, layer, wl.B, wl.H, wl.Hkv, I.bf16_bits(q[call, layer]), c.oKc, c.oVc)
            assert_close(got.double().cpu().numpy(), want, f"call {call} layer {layer} (oracle)")
            close(got, ref)


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
