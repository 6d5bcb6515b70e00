"""Runs only against the bounds-checked build (DKV_LIBRARY=.../libdkv_debug.so;
tests/test_gpu_bounds_build.py starts it that way): a mistake the host cannot
see is planted in the call, and the kernels' own range checks must catch it.

The planted mistake is a dense stride shorter than some kept positions passed
to dkv_compact. The host cannot check it: it does not know the dense buffers'
stride. Every address the kernel could form with the shorter stride still lies
inside the real dense buffers (slab h's rows start at h x stride, before the
real h x T), so even an unchecked build reads nothing out of bounds; the check
must flag the rows whose position is past the stride and skip them."""
import numpy as np
import pytest
import torch

import paper_2609_32663_gb300.dkv as dkv
from paper_2609_32663_gb300 import inputs as I
from parity import BOUNDS_CHECKED, Case

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not BOUNDS_CHECKED, reason="needs the bounds-checked build (DKV_LIBRARY)")]


def test_short_dense_stride_is_flagged_and_its_rows_skipped(cuda):
    wl = I.Workload("planted", L=2, H=8, Hkv=2, T=6000, B=2, D=12, W=(6000 - 1152) // 12 + 1,
                    pattern="profile", rate=0.4, ragged=(2500, 6000), seed=7)
    c = Case(wl)
    try:
        assert dkv.dkv_plan_status(c.plan) == 0  # the map and the real compaction are clean
        T = c.T_stride
        short = T // 2
        Kc = torch.full_like(c.Kc, float("nan"))
        Vc = torch.full_like(c.Vc, float("nan"))
        dkv.dkv_compact(c.plan, c.Kd, c.Vd, Kc, Vc, T_stride=short)
        torch.cuda.synchronize()
        word = dkv.dkv_plan_status(c.plan, clear=True)
        assert word & dkv.DKV_DEV_BOUNDS
        # Rows whose position fits the short stride are copied from h x short + position;
        # the others are skipped (left as the NaN fill).
        K = I.bf16_bits(c.K).reshape(-1, 128)
        got = I.bf16_bits(Kc)
        nan = I.bf16_bits(torch.full((1, 128), float("nan"), dtype=torch.bfloat16))[0]
        om = c.om
        skipped = 0
        for h in range(len(om.len)):
            for r in range(int(om.len[h])):
                pos = int(om.idx[om.ioff[h] + r])
                row = got[int(om.off[h]) + r]
                if pos < short:
                    assert np.array_equal(row, K[h * short + pos]), (h, r)
                else:
                    assert np.array_equal(row, nan), (h, r)
                    skipped += 1
        assert skipped > 0
        assert dkv.dkv_plan_status(c.plan) == 0
    finally:
        c.close()
