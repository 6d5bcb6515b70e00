"""Parity at the benchmark workloads' full sizes, in the launch configuration
bench.py times.

Every workload runs the following, as the benchmark does:

- the map, with bench.py's reserve;
- the prune-and-pack of the whole model's dense caches;
- a few replays of the decode-step CUDA graph. A replay is one
  dkv_decode_attn per layer, appending the step's key/value, then
  dkv_advance.

What is checked:

- the map, bit-exact and in full, against the oracle's map over every position;
- every packed K/V byte. The expected bytes are a gather of the dense caches at
  the oracle's kept indices;
- the attention output of sampled slabs (first, last, longest, shortest, random
  ones), every query head of their group, against the fp64 oracle. The oracle
  computes it from the dense inputs, with the step's appended rows;
- that every output is finite, the device status word is clear and the
  per-sequence counters advanced once per replay.
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2609_32663_gb300.dkv as dkv
from paper_2609_32663_gb300 import inputs as I
from parity import assert_close, check_map, shapes

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

REPLAYS = 3  # decode steps replayed before the outputs are compared


@pytest.fixture(scope="module", autouse=True)
def _built(cuda):
    from paper_2609_32663_gb300 import build
    build.build_library()
    torch.cuda.set_device(cuda)


def _sample_slabs(wl, ln, rng, n_random=2):
    NHl = wl.B * wl.Hkv
    picks = {0, wl.L * NHl - 1, int(np.argmax(ln)), int(np.argmin(ln))}
    picks.update(int(x) for x in rng.integers(0, wl.L * NHl, size=n_random))
    return sorted(picks)


def _packed_rows(om, slabs):
    """Rows of the packed cache holding the kept rows of `slabs` (int64)."""
    return np.concatenate([np.arange(om.off[h], om.off[h] + om.len[h], dtype=np.int64) for h in slabs])


def _dense_rows(wl, om, slabs, T_stride):
    """Rows of the dense cache, flattened per layer as [B][Hkv][T_stride], that the
    oracle keeps for `slabs` (int64), in packing order."""
    NHl = wl.B * wl.Hkv
    out = []
    for h in slabs:
        base = (h % NHl) * T_stride
        out.append(base + om.idx[om.ioff[h]:om.ioff[h + 1]].astype(np.int64))
    return np.concatenate(out)


@pytest.mark.parametrize("name", ["llama8b-1layer-4k", "llama8b-16k", "llama8b-32k", "llama8b-128k", "llama8b-b16-ragged",
                                  "qwen7b-64k-b4-r20", "qwen7b-64k-b4-r35", "qwen7b-64k-b4-r50",
                                  "llama8b-128k-head-only", "llama8b-128k-distance-only",
                                  "llama8b-128k-distance-shuffled", "llama8b-128k-fully-shuffled"])
def test_full_size_workload(name, cuda):
    import bench
    wl = I.WORKLOADS[name]
    reserve = bench.reserve_rows(bench.DEFAULT_STEPS, bench.DEFAULT_WARMUP)
    env = bench.setup(wl, cuda, reserve)
    plan, Kc, Vc, T_stride = env["plan"], env["Kc"], env["Vc"], env["T_stride"]
    _, geo = shapes(wl)
    NHl = wl.B * wl.Hkv
    try:
        # Map: bit-exact, every slab.
        om = O.map_pattern(env["M"], env["Tc"], geo, reserve=reserve)
        check_map(plan, om)

        # Pack: every byte, layer by layer, against a gather at the oracle's indices.
        dkv.dkv_compact(plan, env["K"], env["V"], Kc, Vc, T_stride=T_stride)
        torch.cuda.synchronize()
        for layer in range(wl.L):
            slabs = range(layer * NHl, (layer + 1) * NHl)
            src = torch.from_numpy(_dense_rows(wl, om, slabs, T_stride)).to(cuda)
            dst = torch.from_numpy(_packed_rows(om, slabs)).to(cuda)
            for dense, packed, what in ((env["K"], Kc, "K"), (env["V"], Vc, "V")):
                want = dense[layer].reshape(-1, wl.head_dim).index_select(0, src).view(torch.int16)
                got = packed.index_select(0, dst).view(torch.int16)
                assert torch.equal(got, want), f"{name}: packed {what} bytes of layer {layer} differ"
            del src, dst

        # Decode: the benchmark's graph, replayed.
        runner = bench.DecodeRunner(wl, plan, Kc, Vc, cuda)
        runner.capture()
        for _ in range(REPLAYS):
            runner.replay()
        torch.cuda.synchronize()
        assert dkv.dkv_plan_status(plan) == 0
        assert (runner.n_app.cpu().numpy() == REPLAYS).all()
        out = runner.out.double().cpu().numpy()  # [L][B][H][hd]
        assert np.isfinite(out).all(), f"{name}: non-finite decode output"

        # Oracle inputs straight from the seeded generators (never from the CUDA path).
        q, kn, vn = I.decode_inputs(wl, 1, device=cuda)
        qb, knb, vnb = I.bf16_bits(q[0]), I.bf16_bits(kn[0]), I.bf16_bits(vn[0])
        rng = np.random.default_rng([wl.seed, 99])
        for h in _sample_slabs(wl, om.len, rng):
            layer, b, g = h // NHl, (h % NHl) // wl.Hkv, h % wl.Hkv
            kept = torch.from_numpy(om.idx[om.ioff[h]:om.ioff[h + 1]].astype(np.int64)).to(cuda)
            Krows = I.bf16_bits(env["K"][layer, b, g].index_select(0, kept))
            Vrows = I.bf16_bits(env["V"][layer, b, g].index_select(0, kept))
            # The step's own key/value was appended once per replay.
            Krows = np.concatenate([Krows, np.repeat(knb[layer, b, g][None], REPLAYS, 0)])
            Vrows = np.concatenate([Vrows, np.repeat(vnb[layer, b, g][None], REPLAYS, 0)])
            heads = slice(g * wl.G, (g + 1) * wl.G)
            want = O.attend(qb[layer, b, heads], Krows, Vrows)
            assert_close(out[layer, b, heads], want, f"{name}: layer {layer} seq {b} KV head {g}")
        del runner
    finally:
        plan.close()
        del env
        torch.cuda.empty_cache()
