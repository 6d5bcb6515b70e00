"""CUDA path (through the C ABI) against the CPU oracle on seeded inputs.

Bit-exact: lengths, slab offsets, index offsets, kept index lists, packed K/V
bytes (also after appends). Attention output: rel-L2 <= 1e-3 and max-abs <= 5e-3
against fp64. Sizes span several map chunks (8192 positions), many decode tiles
and ragged tails, and the edge cases of the method.
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2609_32663_gb300.dkv as dkv
from golden_io import map_cases
from paper_2609_32663_gb300 import inputs as I
from parity import Case, assert_close, check_map, shapes

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built(cuda):
    from paper_2609_32663_gb300 import build
    build.build_library()
    torch.cuda.set_device(cuda)


def wl(name="t", **kw):
    base = dict(L=2, H=8, Hkv=2, T=3000, B=1, D=10, W=200, pattern="profile", rate=0.4, seed=3)
    base.update(kw)
    return I.Workload(name, **base)


# ---------------------------------------------------------------- map (bit-exact)

@pytest.mark.parametrize("case", map_cases(), ids=lambda c: c["name"])
def test_map_hand_worked_cases_on_gpu(case):
    g = case["geometry"]
    sh = dkv.Shape(L=g["L"], H=g["H"], H_kv=g["Hkv"], D=g["D"], sink=g["sink"], recent=g["recent"],
                   bin_width=g["bin_width"])
    plan = dkv.dkv_map_pattern(case["M"], case["ctx"], sh)
    ln, off, ioff, idx = dkv.dkv_plan_read(plan)
    got = [list(idx[ioff[h]:ioff[h + 1]]) for h in range(len(ln))]
    assert got == case["kept"]
    plan.close()


@pytest.mark.parametrize("G", [1, 2, 4, 7, 8])
@pytest.mark.parametrize("reserve", [0, 5])
def test_map_matches_oracle(G, reserve):
    w = wl(H=2 * G, Hkv=2, T=40000, B=3, D=24, W=-(-(40000 - 1152) // 24), ragged=(0, 40000), seed=G)
    M = I.make_pattern(w)
    Tc = I.context_lengths(w)
    Tc[0] = 40000  # full pattern span, several 8192-position map chunks
    sh, geo = shapes(w)
    plan = dkv.dkv_map_pattern(M, Tc, sh, reserve_rows=reserve)
    check_map(plan, O.map_pattern(M, Tc, geo, reserve=reserve))
    plan.close()


@pytest.mark.parametrize("Tc", [[0], [1], [1151], [1152], [1153], [8191, 8192, 8193], [16385, 3, 0, 9000]])
def test_map_edge_lengths(Tc):
    w = wl(B=len(Tc), T=max(Tc + [1]), D=16, W=1000, pattern="bernoulli", rate=0.5)
    M = I.make_pattern(w)
    sh, geo = shapes(w)
    plan = dkv.dkv_map_pattern(M, Tc, sh, reserve_rows=2)
    check_map(plan, O.map_pattern(M, Tc, geo, reserve=2))
    plan.close()


def test_map_random_geometries():
    """Sink or recent window of 0, bins of 1 to 100 positions (runs shorter than
    a warp's stride), contexts from 0 to the pattern's full span, random
    patterns and reserves: bit-exact against the oracle's position walk."""
    rng = np.random.default_rng(17)
    for trial in range(40):
        L, Hkv, G, B = int(rng.integers(1, 3)), int(rng.integers(1, 3)), int(rng.integers(1, 5)), int(rng.integers(1, 4))
        S, R = int(rng.choice([0, 1, 3, 16])), int(rng.choice([0, 1, 5, 33]))
        W, D = int(rng.choice([1, 2, 7, 31, 32, 33, 100])), int(rng.integers(1, 80))
        Tc = rng.integers(0, S + R + D * W + 1, size=B).astype(np.int32)
        if trial % 5 == 0:
            Tc[:] = S + R + D * W
        M = (rng.random((L, G * Hkv, D)) < rng.random()).astype(np.uint8)
        reserve = int(rng.integers(0, 3))
        sh = dkv.Shape(L=L, H=G * Hkv, H_kv=Hkv, D=D, sink=S, recent=R, bin_width=W)
        geo = O.Geometry(L=L, H=G * Hkv, Hkv=Hkv, D=D, sink=S, recent=R, bin_width=W)
        plan = dkv.dkv_map_pattern(M, Tc, sh, reserve_rows=reserve)
        check_map(plan, O.map_pattern(M, Tc, geo, reserve=reserve))
        plan.close()


@pytest.mark.parametrize("fill", [0, 1])
def test_map_all_drop_and_all_keep(fill):
    w = wl(T=20000, D=20, W=1000)
    M = np.full((w.L, w.H, w.D), fill, np.uint8)
    sh, geo = shapes(w)
    plan = dkv.dkv_map_pattern(M, [20000], sh)
    ln, *_ = dkv.dkv_plan_read(plan)
    assert (ln == (20000 if fill else 1152)).all()
    check_map(plan, O.map_pattern(M, [20000], geo))
    plan.close()


# ---------------------------------------------------------------- packing (bit-exact)

@pytest.mark.parametrize("G,B,reserve", [(4, 1, 0), (7, 2, 3), (1, 3, 1)])
def test_compact_bytes_match_oracle(G, B, reserve):
    c = Case(wl(H=2 * G, Hkv=2, T=12000, B=B, D=12, W=904, ragged=(2000, 12000), seed=10 + G),
             reserve=reserve)
    check_map(c.plan, c.om)
    c.check_packed()
    c.close()


# ---------------------------------------------------------------- decode (tolerance)

@pytest.mark.parametrize("G", [1, 2, 3, 4, 5, 6, 7, 8])
def test_decode_matches_oracle_without_append(G):
    c = Case(wl(H=2 * G, Hkv=2, T=6000, B=2, D=8, W=606, ragged=(1000, 6000), seed=20 + G))
    c.decode_steps(1, append=False)
    c.close()


@pytest.mark.parametrize("G", [1, 3, 4, 5, 6, 7])
def test_decode_with_appends_over_steps(G):
    c = Case(wl(H=2 * G, Hkv=2, T=5000, B=3, D=8, W=500, ragged=(100, 5000), seed=30 + G), reserve=6)
    c.decode_steps(4, append=True)
    c.close()


@pytest.mark.parametrize("T", [1, 2, 7, 8, 9, 15, 16, 17, 31, 32, 33, 100, 1151, 1153])
def test_decode_short_and_ragged_lengths(T):
    """Lengths around the 8-row tile, the warp's 2-row step and the sink+recent span."""
    c = Case(wl(H=4, Hkv=1, T=T, B=1, D=2, W=600, pattern="bernoulli", rate=0.5, seed=T), reserve=2)
    c.decode_steps(2, append=True)
    c.close()


def test_decode_empty_context_with_and_without_append():
    w = wl(H=8, Hkv=2, T=10, B=3, D=2, W=8)
    c = Case(w, reserve=3, Tc=[0, 5, 0])
    c.decode_steps(1, append=False)   # slabs with no rows give zeros
    c.decode_steps(2, append=True)
    c.close()


def test_decode_many_sequences_uneven():
    """Many slabs of very different lengths: CTA ranges cross slab boundaries."""
    w = wl(L=1, H=16, Hkv=4, T=30000, B=9, D=16, W=(30000 - 1152) // 16, ragged=(0, 30000), seed=77)
    c = Case(w, reserve=2)
    c.decode_steps(2, append=True)
    c.close()


@pytest.mark.parametrize("G", [4, 7])
def test_decode_more_slabs_than_the_shared_table(G):
    """B * H_kv >= 1024 slabs in a layer: the kernels read slab starts and cache
    offsets from global memory instead of their shared-memory copy."""
    w = wl(L=1, H=8 * G, Hkv=8, T=1300, B=130, D=2, W=(1300 - 1152) // 2, ragged=(0, 1300), seed=80 + G)
    assert w.B * w.Hkv >= 1024
    c = Case(w, reserve=2)
    c.decode_steps(1, append=True)
    c.close()


def test_decode_outlier_keys_and_custom_scale():
    w = wl(H=8, Hkv=2, T=9000, D=8, W=(9000 - 1152) // 8, outlier_frac=0.05, seed=5)
    c = Case(w)
    c.decode_steps(1, append=False, scale=0.2)
    c.decode_steps(1, append=False, scale=0.0)
    c.close()


@pytest.mark.parametrize("G", [4, 7])
def test_separate_partial_and_combine_entry_points(G):
    """dkv_decode_partial + dkv_decode_combine (two launches) give the oracle's answer,
    with this step's token appended, like dkv_decode_attn does in one launch."""
    w = wl(H=2 * G, Hkv=2, T=7000, B=3, D=8, W=800, ragged=(500, 7000), seed=40 + G)
    c = Case(w, reserve=3)
    q, kn, vn = I.decode_inputs(w, 2)
    n_app = torch.zeros(w.B, dtype=torch.int32, device=c.dev)
    na = np.zeros(w.B, np.int32)
    out = torch.full((w.B, w.H, 128), float("nan"), dtype=torch.float32, device=c.dev)
    for s in range(2):
        for layer in range(w.L):
            dkv.dkv_decode_partial(c.plan, layer, q[s, layer].to(c.dev), kn[s, layer].to(c.dev),
                                   vn[s, layer].to(c.dev), n_app, c.Kc, c.Vc)
            dkv.dkv_decode_combine(c.plan, layer, n_app, True, out)
            O.append(c.om, layer, w.B, w.Hkv, c.reserve, na, I.bf16_bits(kn[s, layer]), I.bf16_bits(vn[s, layer]),
                     c.oKc, c.oVc)
            want = O.decode(c.om, layer, w.B, w.H, w.Hkv, I.bf16_bits(q[s, layer]), c.oKc, c.oVc, n_rows_app=na + 1)
            assert_close(out.cpu().numpy(), want, f"two-launch step {s} layer {layer}")
        dkv.dkv_advance(c.plan, n_app)
        na += 1
    c.check_packed_with_appends(na)
    c.close()


def test_decode_repeated_calls_reuse_counters():
    """Many consecutive single-launch calls on one plan (the fused combine's slab
    counters reset themselves) stay equal to the oracle."""
    w = wl(H=8, Hkv=2, T=9000, B=2, D=8, W=(9000 - 1152) // 8 + 1, ragged=(2000, 9000), seed=51)
    c = Case(w)
    q, _, _ = I.decode_inputs(w, 1)
    out = torch.empty((w.B, w.H, 128), dtype=torch.float32, device=c.dev)
    want = [O.decode(c.om, l, w.B, w.H, w.Hkv, I.bf16_bits(q[0, l]), c.oKc, c.oVc) for l in range(w.L)]
    for rep in range(6):
        for layer in range(w.L):
            dkv.dkv_decode_attn(c.plan, layer, q[0, layer].to(c.dev), None, None, None, c.Kc, c.Vc, out)
            assert_close(out.cpu().numpy(), want[layer], f"rep {rep} layer {layer}")
    c.close()


def test_all_keep_equals_dense_plan():
    """M = 1 gives the same output as the dense-cache plan over the uncompressed K/V."""
    w = wl(H=8, Hkv=2, T=7000, B=2, D=8, W=800, ragged=(3000, 7000), seed=9)
    M = np.ones((w.L, w.H, w.D), np.uint8)
    c = Case(w, M=M)
    sh, _ = shapes(w)
    dense = dkv.dkv_plan_dense(c.Tc, sh, T_stride=c.T_stride)
    q, _, _ = I.decode_inputs(w, 1)
    o1 = torch.empty((w.B, w.H, 128), dtype=torch.float32, device=c.dev)
    o2 = torch.empty_like(o1)
    for layer in range(w.L):
        qd = q[0, layer].to(c.dev)
        dkv.dkv_decode_attn(c.plan, layer, qd, None, None, None, c.Kc, c.Vc, o1)
        dkv.dkv_decode_attn(dense, layer, qd, None, None, None, c.Kd, c.Vd, o2)
        want = O.decode(c.om, layer, w.B, w.H, w.Hkv, I.bf16_bits(q[0, layer]), c.oKc, c.oVc)
        assert_close(o1.cpu().numpy(), want, "packed")
        assert_close(o2.cpu().numpy(), want, "dense")
    dense.close()
    c.close()


def test_dense_plan_with_appends_matches_oracle():
    w = wl(H=8, Hkv=2, T=3000, B=2, D=4, W=600, ragged=(1500, 3000), seed=12)
    Tc = I.context_lengths(w)
    sh, geo = shapes(w)
    T_stride = int(Tc.max()) + 4
    K, V = I.dense_kv(w.with_(T=T_stride))
    Kd, Vd = K.cuda(), V.cuda()
    plan = dkv.dkv_plan_dense(Tc, sh, T_stride=T_stride)
    # The oracle's view of the dense layout: every position kept, slab h at h*T_stride.
    om = O.map_pattern(np.ones((w.L, w.H, w.D), np.uint8), Tc, geo, reserve=0)
    NH = w.L * w.B * w.Hkv
    om.off = np.arange(NH + 1, dtype=np.int64) * T_stride
    oK = I.bf16_bits(K).reshape(-1, 128).copy()
    oV = I.bf16_bits(V).reshape(-1, 128).copy()
    q, kn, vn = I.decode_inputs(w, 3)
    n_app = torch.zeros(w.B, dtype=torch.int32, device="cuda")
    out = torch.empty((w.B, w.H, 128), dtype=torch.float32, device="cuda")
    na = np.zeros(w.B, np.int32)
    reserve = T_stride - int(Tc.max())
    for s in range(3):
        for layer in range(w.L):
            dkv.dkv_decode_attn(plan, layer, q[s, layer].cuda(), kn[s, layer].cuda(), vn[s, layer].cuda(),
                                n_app, Kd, Vd, out)
            O.append(om, layer, w.B, w.Hkv, T_stride, na, I.bf16_bits(kn[s, layer]), I.bf16_bits(vn[s, layer]),
                     oK, oV)
            want = O.decode(om, layer, w.B, w.H, w.Hkv, I.bf16_bits(q[s, layer]), oK, oV, n_rows_app=na + 1)
            assert_close(out.cpu().numpy(), want, f"dense step {s} layer {layer}")
        dkv.dkv_advance(plan, n_app)
        na += 1
    assert reserve >= 3 and dkv.dkv_plan_status(plan) == 0
    plan.close()


# ---------------------------------------------------------------- device status word

def test_append_past_reserve_sets_status_and_is_skipped():
    w = wl(H=4, Hkv=1, T=2000, D=2, W=600)
    c = Case(w, reserve=1)
    q, kn, vn = I.decode_inputs(w, 1)
    n_app = torch.ones(1, dtype=torch.int32, device="cuda")  # reserve already used
    out = torch.empty((1, 4, 128), dtype=torch.float32, device="cuda")
    before = c.Kc.clone()
    dkv.dkv_decode_attn(c.plan, 0, q[0, 0].cuda(), kn[0, 0].cuda(), vn[0, 0].cuda(), n_app, c.Kc, c.Vc, out)
    word = dkv.dkv_plan_status(c.plan, clear=True)
    assert word & dkv.DKV_DEV_APPEND_OVERFLOW
    assert torch.equal(before.view(torch.int16), c.Kc.view(torch.int16))  # nothing written
    # The output covers the rows that exist: len + 1 already-appended (never written: NaN-free
    # only because n_app is clamped to the reserve, so compare against that view).
    dkv.dkv_advance(c.plan, n_app)
    assert dkv.dkv_plan_status(c.plan, clear=True) & dkv.DKV_DEV_APPEND_OVERFLOW
    assert dkv.dkv_plan_status(c.plan) == 0
    c.close()


def test_injected_launch_failure(monkeypatch):
    w = wl(H=4, Hkv=1, T=2000, D=2, W=600)
    c = Case(w)
    monkeypatch.setenv("DKV_FAULT", "launch")
    out = torch.empty((1, 4, 128), dtype=torch.float32, device="cuda")
    q = torch.zeros((1, 4, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_decode_attn(c.plan, 0, q, None, None, None, c.Kc, c.Vc, out)
    assert e.value.status == dkv.DKV_ERR_CUDA
    monkeypatch.delenv("DKV_FAULT")
    torch.cuda.synchronize()
    c.close()


def test_copy_wait_runs_out_and_reports(monkeypatch):
    """DKV_FAULT=copy gives the decode kernel tensor maps whose boxes bring half
    the bytes each stage's mbarrier expects: every copy wait runs out at its
    bound (2 s or 2^22 polls), the kernel sets DKV_DEV_TMA_TIMEOUT, drains and
    returns. Nothing faults; the context stays usable and the next call is
    exact again."""
    import time
    w = wl(H=8, Hkv=2, T=6000, D=8, W=606, seed=23)
    c = Case(w)
    q = torch.zeros((w.B, w.H, 128), dtype=torch.bfloat16, device=c.dev)
    out = torch.empty((w.B, w.H, 128), dtype=torch.float32, device=c.dev)
    monkeypatch.setenv("DKV_FAULT", "copy")
    t0 = time.time()
    dkv.dkv_decode_attn(c.plan, 0, q, None, None, None, c.Kc, c.Vc, out)
    torch.cuda.synchronize()
    elapsed = time.time() - t0
    monkeypatch.delenv("DKV_FAULT")
    assert dkv.dkv_plan_status(c.plan, clear=True) & dkv.DKV_DEV_TMA_TIMEOUT
    assert elapsed < 60
    c.decode_steps(1, append=False)  # exact again; checks the status word is clear
    c.close()



def test_merge_wait_runs_out_and_reports(monkeypatch):
    """DKV_FAULT=merge makes the last CTA of each fused (slab, head) merge wait
    for one CTA partial more than the slab has: the wait runs out at its bound
    (2 s or 2^22 polls), the kernel sets DKV_DEV_MERGE_TIMEOUT, makes the slab
    counters ready for the next call and skips that merge. Nothing faults; the
    next call is exact again."""
    import time
    w = wl(H=8, Hkv=2, T=6000, D=8, W=606, seed=29)
    c = Case(w)
    q = torch.zeros((w.B, w.H, 128), dtype=torch.bfloat16, device=c.dev)
    out = torch.empty((w.B, w.H, 128), dtype=torch.float32, device=c.dev)
    monkeypatch.setenv("DKV_FAULT", "merge")
    t0 = time.time()
    dkv.dkv_decode_attn(c.plan, 0, q, None, None, None, c.Kc, c.Vc, out)
    torch.cuda.synchronize()
    elapsed = time.time() - t0
    monkeypatch.delenv("DKV_FAULT")
    assert dkv.dkv_plan_status(c.plan, clear=True) & dkv.DKV_DEV_MERGE_TIMEOUT
    assert elapsed < 60
    c.decode_steps(2, append=False)  # exact again; checks the status word is clear
    c.close()


def test_unaligned_pointer_rejected():
    w = wl(H=4, Hkv=1, T=2000, D=2, W=600)
    c = Case(w)
    out = torch.empty((1, 4, 128 + 1), dtype=torch.float32, device="cuda")
    q = torch.zeros((1, 4, 128), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(dkv.DkvError) as e:
        dkv.dkv_decode_attn(c.plan, 0, q, None, None, None, c.Kc, c.Vc, out[:, :, 1:])
    assert e.value.status == dkv.DKV_ERR_INVALID_ARG
    with pytest.raises(dkv.DkvError):
        dkv.dkv_decode_attn(c.plan, 2, q, None, None, None, c.Kc, c.Vc, out)  # layer out of range
    c.close()


def test_binding_refuses_host_and_mistyped_buffers(cuda):
    """The Python binding checks device-buffer arguments before the call: a host
    tensor, a wrong element type or a short cache is refused with
    DKV_ERR_INVALID_ARG (a host address reaching a kernel would fault)."""
    c = Case(wl(seed=9))
    w = c.wl
    q = torch.zeros((w.B, w.H, 128), dtype=torch.bfloat16, device=c.dev)
    out = torch.empty((w.B, w.H, 128), dtype=torch.float32, device=c.dev)
    bad = [
        dict(q=q.cpu()),
        dict(q=q.float()),
        dict(out=out.to(torch.bfloat16)),
        dict(out=torch.empty((w.B, w.H + 1, 128), dtype=torch.float32, device=c.dev)),
        dict(Kc=c.Kc[:-1]),
    ]
    for b in bad:
        args = dict(q=q, Kc=c.Kc, Vc=c.Vc, out=out)
        args.update(b)
        with pytest.raises(dkv.DkvError) as e:
            dkv.dkv_decode_attn(c.plan, 0, args["q"], None, None, None, args["Kc"], args["Vc"], args["out"])
        assert e.value.status == dkv.DKV_ERR_INVALID_ARG
    dkv.dkv_decode_attn(c.plan, 0, q, None, None, None, c.Kc, c.Vc, out)  # the valid call still runs
    torch.cuda.synchronize()
    c.close()


def test_decode_at_the_batch_limit():
    """B = 512 sequences (the kernels' per-call table limit), one KV head each."""
    w = wl(L=1, H=4, Hkv=1, T=1300, B=512, D=2, W=(1300 - 1152) // 2, ragged=(0, 1300), seed=88)
    c = Case(w, reserve=1)
    c.decode_steps(1, append=True)
    c.close()


def test_batch_above_the_limit_is_refused():
    w = wl(L=1, H=4, Hkv=1, T=64, B=513, D=2, W=64, seed=89)
    sh, _ = shapes(w)
    with pytest.raises(dkv.DkvError):
        dkv.dkv_map_pattern(I.make_pattern(w), I.context_lengths(w), sh, reserve_rows=0)
