"""Shared helpers of the GPU parity tests: run the CUDA path through the C ABI and
the CPU oracle on the same seeded inputs, and compare."""
import json
import os

import numpy as np
import torch

import oracle as O
import paper_2609_32663_gb300.dkv as dkv
from paper_2609_32663_gb300 import inputs as I

# True when the tests run against the bounds-checked build (DKV_LIBRARY=.../libdkv_debug.so).
BOUNDS_CHECKED = os.environ.get("DKV_LIBRARY", "").endswith("libdkv_debug.so")

# Tolerances of the fp32 attention output against the fp64 oracle.
REL_L2 = 1e-3
MAX_ABS = 5e-3


def shapes(wl):
    sh = dkv.Shape(L=wl.L, H=wl.H, H_kv=wl.Hkv, D=wl.D, sink=wl.sink, recent=wl.recent, bin_width=wl.W)
    geo = O.Geometry(L=wl.L, H=wl.H, Hkv=wl.Hkv, D=wl.D, sink=wl.sink, recent=wl.recent, bin_width=wl.W)
    return sh, geo


def row_errors(got, want):
    """Per output row (the last axis: one head's 128 dims for one query): max-abs
    error and rel-L2 error (relative to the oracle row's norm; absolute for a zero
    row, the output of an empty slab)."""
    got = np.asarray(got, np.float64).reshape(-1, np.shape(want)[-1] if np.ndim(want) else 1)
    want = np.asarray(want, np.float64).reshape(got.shape)
    diff = got - want
    err = np.abs(diff).max(axis=1) if got.size else np.zeros(0)
    nrm = np.linalg.norm(want, axis=1)
    dn = np.linalg.norm(diff, axis=1)
    rel = np.where(nrm > 0, dn / np.where(nrm > 0, nrm, 1.0), dn)
    return err, rel


def assert_close(got, want, what=""):
    """Every output row (each (sequence, query, head) of 128 dims) within rel-L2
    <= REL_L2 and max-abs <= MAX_ABS of the fp64 oracle. Returns the worst row's
    (rel-L2, max-abs); with DKV_PARITY_LOG set, also appends them to that file."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, f"{what}: shape {got.shape} != {want.shape}"
    assert np.isfinite(got).all(), f"{what}: non-finite output"
    if got.size == 0:
        return 0.0, 0.0
    err, rel = row_errors(got, want)
    bad = np.flatnonzero((err > MAX_ABS) | (rel > REL_L2))
    assert bad.size == 0, (f"{what}: {bad.size} of {err.size} rows out of tolerance; row {bad[0]}: "
                           f"max-abs {err[bad[0]]:.3e}, rel-L2 {rel[bad[0]]:.3e}")
    worst = (float(rel.max()), float(err.max()))
    log = os.environ.get("DKV_PARITY_LOG")
    if log:
        with open(log, "a") as f:
            f.write(json.dumps({"what": what, "rows": int(err.size), "worst_rel_l2": worst[0],
                                "worst_max_abs": worst[1]}) + "\n")
    return worst


def check_map(plan, om):
    ln, off, ioff, idx = dkv.dkv_plan_read(plan)
    assert np.array_equal(ln, om.len), "lengths differ"
    assert np.array_equal(off, om.off), "slab offsets differ"
    assert np.array_equal(ioff, om.ioff), "index offsets differ"
    assert np.array_equal(idx, om.idx), "kept index lists differ"


class Case:
    """A small end-to-end case: pattern, caches, plan, packed caches, on both sides."""

    def __init__(self, wl, reserve=0, M=None, Tc=None, device="cuda:0", T_stride=None):
        self.wl = wl
        self.reserve = reserve
        self.M = I.make_pattern(wl) if M is None else np.ascontiguousarray(M, np.uint8)
        self.Tc = I.context_lengths(wl) if Tc is None else np.ascontiguousarray(Tc, np.int32)
        self.sh, self.geo = shapes(wl)
        self.dev = torch.device(device)
        self.T_stride = T_stride or max(int(self.Tc.max()), 1)
        self.K, self.V = I.dense_kv(wl.with_(T=self.T_stride))  # CPU bf16
        self.om = O.map_pattern(self.M, self.Tc, self.geo, reserve=reserve)
        self.plan = dkv.dkv_map_pattern(self.M, self.Tc, self.sh, reserve_rows=reserve)
        self.info = dkv.dkv_plan_query(self.plan)
        self.Kd, self.Vd = self.K.to(self.dev), self.V.to(self.dev)
        n = max(self.info.total_rows, 1)
        self.Kc = torch.full((n, 128), float("nan"), dtype=torch.bfloat16, device=self.dev)
        self.Vc = torch.full((n, 128), float("nan"), dtype=torch.bfloat16, device=self.dev)
        dkv.dkv_compact(self.plan, self.Kd, self.Vd, self.Kc, self.Vc, T_stride=self.T_stride)
        self.oKc, self.oVc = O.compact(self.om, wl.L, wl.B, wl.Hkv, I.bf16_bits(self.K),
                                       I.bf16_bits(self.V), self.T_stride)

    def check_packed(self):
        gK, gV = I.bf16_bits(self.Kc), I.bf16_bits(self.Vc)
        for h in range(len(self.om.len)):
            r = slice(int(self.om.off[h]), int(self.om.off[h] + self.om.len[h]))
            assert np.array_equal(gK[r], self.oKc[r]), f"K bytes of slab {h} differ"
            assert np.array_equal(gV[r], self.oVc[r]), f"V bytes of slab {h} differ"

    def decode_steps(self, steps, append=True, scale=0.0, layers=None):
        """Run `steps` decode steps (every layer, then dkv_advance) on both sides and
        compare every layer's output."""
        wl = self.wl
        q, kn, vn = I.decode_inputs(wl, steps)
        n_app = torch.zeros(wl.B, dtype=torch.int32, device=self.dev)
        na = np.zeros(wl.B, np.int32)
        out = torch.full((wl.B, wl.H, 128), float("nan"), dtype=torch.float32, device=self.dev)
        layers = range(wl.L) if layers is None else layers
        for s in range(steps):
            for layer in layers:
                qd = q[s, layer].to(self.dev)
                if append:
                    dkv.dkv_decode_attn(self.plan, layer, qd, kn[s, layer].to(self.dev),
                                        vn[s, layer].to(self.dev), n_app, self.Kc, self.Vc, out, scale=scale)
                    O.append(self.om, layer, wl.B, wl.Hkv, self.reserve, na, I.bf16_bits(kn[s, layer]),
                             I.bf16_bits(vn[s, layer]), self.oKc, self.oVc)
                    rows = na + 1
                else:
                    dkv.dkv_decode_attn(self.plan, layer, qd, None, None, n_app, self.Kc, self.Vc, out,
                                        scale=scale)
                    rows = na
                want = O.decode(self.om, layer, wl.B, wl.H, wl.Hkv, I.bf16_bits(q[s, layer]), self.oKc,
                                self.oVc, n_rows_app=rows, scale=scale)
                assert_close(out.double().cpu().numpy(), want, f"step {s} layer {layer}")
            if append:
                dkv.dkv_advance(self.plan, n_app)
                na += 1
        assert dkv.dkv_plan_status(self.plan) == 0
        if append:
            assert np.array_equal(n_app.cpu().numpy(), na)
            self.check_packed_with_appends(na)

    def check_packed_with_appends(self, na):
        gK, gV = I.bf16_bits(self.Kc), I.bf16_bits(self.Vc)
        for h in range(len(self.om.len)):
            b = (h // self.wl.Hkv) % self.wl.B
            r = slice(int(self.om.off[h]), int(self.om.off[h] + self.om.len[h] + na[b]))
            assert np.array_equal(gK[r], self.oKc[r]) and np.array_equal(gV[r], self.oVc[r]), \
                f"slab {h} bytes differ after appends"

    def close(self):
        # Under the bounds-checked build every case also asserts that no kernel
        # flagged an out-of-range index or offset.
        word = dkv.dkv_plan_status(self.plan) if BOUNDS_CHECKED else 0
        self.plan.close()
        assert not word & dkv.DKV_DEV_BOUNDS, f"bounds-checked build flagged an access (status {word:#x})"
