"""In-place prune-and-pack (dkv_map_pattern_inplace + dkv_compact_inplace): the
packed cache lives in the dense buffer, slab h at rows h * T_stride. Against the
oracle's ordered pack with the same slab offsets: bit-exact rows [0, len) of
every slab, then decode steps with appended tokens over the in-place cache."""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2609_32663_gb300.dkv as dkv
from paper_2609_32663_gb300 import inputs as I
from parity import assert_close, shapes

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built(cuda):
    from paper_2609_32663_gb300 import build
    build.build_library()
    torch.cuda.set_device(cuda)


def wl(name="ip", **kw):
    base = dict(L=2, H=8, Hkv=2, T=9000, B=3, D=20, W=-(-(9000 - 1152) // 20), pattern="profile", rate=0.35,
                ragged=(0, 9000), seed=41)
    base.update(kw)
    return I.Workload(name, **base)


def inplace_mapping(om, T_stride):
    NH = len(om.len)
    return O.Mapping(om.len, np.arange(NH + 1, dtype=np.int64) * T_stride, om.ioff, om.idx)


def run(w, reserve, M=None, Tc=None, extra_stride=0, steps=3, cuda="cuda:0"):
    M = I.make_pattern(w) if M is None else M
    Tc = I.context_lengths(w) if Tc is None else np.asarray(Tc, np.int32)
    sh, geo = shapes(w)
    T_stride = int(Tc.max()) + reserve + extra_stride
    K, V = I.dense_kv(w.with_(T=T_stride))  # CPU bf16 [L][B][Hkv][T_stride][128]
    om = O.map_pattern(M, Tc, geo, reserve=reserve)
    im = inplace_mapping(om, T_stride)
    oKc, oVc = O.compact(im, w.L, w.B, w.Hkv, I.bf16_bits(K), I.bf16_bits(V), T_stride)

    plan = dkv.dkv_map_pattern_inplace(M, Tc, sh, T_stride, reserve_rows=reserve)
    ln, off, ioff, idx = dkv.dkv_plan_read(plan)
    assert np.array_equal(ln, om.len) and np.array_equal(ioff, om.ioff) and np.array_equal(idx, om.idx)
    assert np.array_equal(off, im.off)
    Kd, Vd = K.to(cuda), V.to(cuda)
    dkv.dkv_compact_inplace(plan, Kd, Vd)
    torch.cuda.synchronize()
    gK = I.bf16_bits(Kd.reshape(-1, 128))
    gV = I.bf16_bits(Vd.reshape(-1, 128))
    for h in range(len(om.len)):
        r = slice(int(im.off[h]), int(im.off[h] + om.len[h]))
        assert np.array_equal(gK[r], oKc[r]) and np.array_equal(gV[r], oVc[r]), f"slab {h}"

    # decode steps with appends over the in-place cache
    q, kn, vn = I.decode_inputs(w, steps)
    n_app = torch.zeros(w.B, dtype=torch.int32, device=cuda)
    na = np.zeros(w.B, np.int32)
    out = torch.empty((w.B, w.H, 128), dtype=torch.float32, device=cuda)
    Kc, Vc = Kd.reshape(-1, 128), Vd.reshape(-1, 128)
    for s in range(steps):
        for layer in range(w.L):
            dkv.dkv_decode_attn(plan, layer, q[s, layer].to(cuda), kn[s, layer].to(cuda), vn[s, layer].to(cuda),
                                n_app, Kc, Vc, out)
            O.append(im, layer, w.B, w.Hkv, reserve, na, I.bf16_bits(kn[s, layer]), I.bf16_bits(vn[s, layer]),
                     oKc, oVc)
            want = O.decode(im, layer, w.B, w.H, w.Hkv, I.bf16_bits(q[s, layer]), oKc, oVc, n_rows_app=na + 1)
            assert_close(out.double().cpu().numpy(), want, f"step {s} layer {layer}")
        dkv.dkv_advance(plan, n_app)
        na += 1
    assert dkv.dkv_plan_status(plan) == 0
    plan.close()


@pytest.mark.parametrize("G", [1, 4, 7])
def test_inplace_matches_oracle(G, cuda):
    run(wl(H=2 * G, Hkv=2, seed=40 + G), reserve=4, cuda=cuda)


def test_inplace_wider_stride(cuda):
    run(wl(seed=50), reserve=2, extra_stride=777, steps=2, cuda=cuda)


def test_inplace_all_keep_moves_nothing(cuda):
    w = wl(seed=51, ragged=None)
    M = np.ones((w.L, w.H, w.D), np.uint8)
    run(w, reserve=3, M=M, cuda=cuda)


def test_inplace_all_drop_and_short_contexts(cuda):
    w = wl(seed=52)
    M = np.zeros((w.L, w.H, w.D), np.uint8)
    Tc = np.array([0, 700, 9000], np.int32)  # empty, shorter than sink + recent, long
    run(w, reserve=2, M=M, Tc=Tc, steps=2, cuda=cuda)


def test_inplace_many_short_slabs(cuda):
    """More slabs than SMs, most of them short: the kernel's CTAs claim slabs
    one after another, and slabs where no row moves are skipped."""
    w = wl(L=4, H=8, Hkv=4, B=16, T=3000, D=20, W=-(-(3000 - 1152) // 20), ragged=(0, 3000), seed=54)
    run(w, reserve=2, steps=1, cuda=cuda)


def test_inplace_rejects_short_stride_and_wrong_plan(cuda):
    w = wl(seed=53)
    sh, _ = shapes(w)
    M = I.make_pattern(w)
    Tc = I.context_lengths(w)
    with pytest.raises(dkv.DkvError):
        dkv.dkv_map_pattern_inplace(M, Tc, sh, int(Tc.max()) + 1, reserve_rows=4)  # stride < Tmax + reserve
    packed = dkv.dkv_map_pattern(M, Tc, sh, reserve_rows=4)
    x = torch.zeros((8, 128), dtype=torch.bfloat16, device=cuda)
    with pytest.raises(dkv.DkvError):
        dkv.dkv_compact_inplace(packed, x, x.clone())  # a packed plan is not an in-place plan
    packed.close()


@pytest.mark.slow
def test_inplace_full_size_llama_128k(cuda):
    """llama8b-128k: every packed byte after the in-place move (the expected rows
    are gathered at the oracle's indices before the move), then one decode step."""
    import bench
    w = I.WORKLOADS["llama8b-128k"]
    reserve = bench.reserve_rows(bench.DEFAULT_STEPS, bench.DEFAULT_WARMUP)
    M, Tc = I.make_pattern(w), I.context_lengths(w)
    sh, geo = shapes(w)
    T_stride = int(Tc.max()) + reserve
    K, V = I.dense_kv(w.with_(T=T_stride), device=cuda)
    om = O.map_pattern(M, Tc, geo, reserve=reserve)
    NHl = w.B * w.Hkv
    want_K, want_V = [], []
    for layer in range(w.L):
        src = np.concatenate([(h % NHl) * T_stride + om.idx[om.ioff[h]:om.ioff[h + 1]].astype(np.int64)
                              for h in range(layer * NHl, (layer + 1) * NHl)])
        src = torch.from_numpy(src).to(cuda)
        want_K.append(K[layer].reshape(-1, 128).index_select(0, src).view(torch.int16))
        want_V.append(V[layer].reshape(-1, 128).index_select(0, src).view(torch.int16))
    plan = dkv.dkv_map_pattern_inplace(M, Tc, sh, T_stride, reserve_rows=reserve)
    dkv.dkv_compact_inplace(plan, K, V)
    torch.cuda.synchronize()
    Kf, Vf = K.reshape(-1, 128), V.reshape(-1, 128)
    for layer in range(w.L):
        dst = np.concatenate([h * T_stride + np.arange(om.len[h], dtype=np.int64)
                              for h in range(layer * NHl, (layer + 1) * NHl)])
        dst = torch.from_numpy(dst).to(cuda)
        assert torch.equal(Kf.index_select(0, dst).view(torch.int16), want_K[layer]), f"K layer {layer}"
        assert torch.equal(Vf.index_select(0, dst).view(torch.int16), want_V[layer]), f"V layer {layer}"
    plan.close()
