"""Page-backed caches (dkv_vmm_*) on the in-place path: dense K/V in page-backed
buffers, in-place compaction, then the pages with no kept, reserve or guard row
are released, and decode steps with appends still match the oracle. The page
rule itself is checked on the CPU (tests/test_abi_cpu.py)."""
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


def test_trim_releases_pages_and_decode_still_matches(cuda):
    # Slabs of 65,536 rows (16 MiB each), a sparse pattern: most of each slab is released.
    w = I.Workload("vmm", L=2, H=8, Hkv=2, T=65536 - 8, B=2, D=16, W=-(-(65536 - 8 - 1152) // 16),
                   pattern="profile", rate=0.2, seed=61)
    reserve = 8
    M, Tc = I.make_pattern(w), I.context_lengths(w)
    sh, geo = shapes(w)
    T_stride = int(Tc.max()) + reserve  # 65,536
    NH = w.L * w.B * w.Hkv
    nbytes = NH * T_stride * 256
    bufK, bufV = dkv.VmmBuffer(nbytes), dkv.VmmBuffer(nbytes)
    try:
        assert bufK.mapped_bytes() >= nbytes
        K = bufK.tensor((w.L, w.B, w.Hkv, T_stride, 128), torch.bfloat16)
        V = bufV.tensor((w.L, w.B, w.Hkv, T_stride, 128), torch.bfloat16)
        Kh, Vh = I.dense_kv(w.with_(T=T_stride))
        K.copy_(Kh.to(cuda))
        V.copy_(Vh.to(cuda))
        om = O.map_pattern(M, Tc, geo, reserve=reserve)
        im = O.Mapping(om.len, np.arange(NH + 1, dtype=np.int64) * T_stride, om.ioff, om.idx)
        oKc, oVc = O.compact(im, w.L, w.B, w.Hkv, I.bf16_bits(Kh), I.bf16_bits(Vh), T_stride)

        plan = dkv.dkv_map_pattern_inplace(M, Tc, sh, T_stride, reserve_rows=reserve)
        dkv.dkv_compact_inplace(plan, K, V)
        torch.cuda.synchronize()
        before = bufK.mapped_bytes()
        with pytest.raises(dkv.DkvError):
            bufK.trim(plan, guard_rows=15)  # guard below a decode tile
        freed_k, freed_v = bufK.trim(plan, guard_rows=16), bufV.trim(plan, guard_rows=16)
        assert freed_k > 0 and freed_k == freed_v
        assert bufK.mapped_bytes() == before - freed_k
        # what is left mapped: each slab's len + reserve + guard rows, rounded up to pages
        page = bufK.page_bytes()
        keep = dkv.dkv_vmm_pages_to_keep(om.len, T_stride, reserve, 16, page, -(-nbytes // page))
        assert bufK.mapped_bytes() == int(keep.sum()) * page
        assert bufK.trim(plan, guard_rows=16) == 0  # idempotent

        # kept rows survived, and decode with appends works over the trimmed buffers
        Kc, Vc = K.reshape(-1, 128), V.reshape(-1, 128)
        q, kn, vn = I.decode_inputs(w, 3)
        n_app = torch.zeros(w.B, dtype=torch.int32, device=cuda)
        na = np.zeros(w.B, np.int32)
        out = torch.empty((w.B, w.H, 128), dtype=torch.float32, device=cuda)
        for s in range(3):
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
        del K, V, Kc, Vc
    finally:
        bufK.close()
        bufV.close()
