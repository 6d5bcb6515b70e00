"""Benchmark of the Distance-KV decode hot path on one GB300 (per process).

A step is one decode step of the whole model: for every layer, dkv_decode_attn
(one launch: the split-K pass, which also appends the step's key/value to the
packed cache, with the combine fused in), then dkv_advance -- replayed as one
CUDA graph. Before the
timed steps the path runs its one-shot part once per context: the pattern map
and the prune-and-pack (timed separately and reported as compaction GB/s).

Default workload: Llama-3.1-8B-shaped cache (32 layers, 32 q-heads, 8 KV heads,
head_dim 128), batch 1, 131,072-token context, 34.6 % physical retention,
1 % outlier keys, synthetic N(0,1) bf16 K/V/q.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl dkv|reference]

--impl reference times the CPU oracle on the same workload (bounded sample of
the heads of each step, scaled to a full step). Under torchrun every rank runs
its own replica (the path does not exchange data between GPUs); the timing is
the max over ranks and rank 0 prints one JSON line.
"""
import argparse
import contextlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_32663_gb300 import inputs as I  # noqa: E402

# DRAM traffic of the decode kernel from one ncu capture: dram__bytes_read.sum +
# dram__bytes_write.sum of layer 0 of llama8b-128k-l4 (the per-layer sizes of
# llama8b-128k, 4 layers), against that launch's algorithmic bytes. Traffic grows
# with the rows a launch streams, so a launch of the full workload is credited
# ratio x its own algorithmic bytes -- only while the kernel sources still hash to
# the value the capture was taken on (else the traffic is unknown: null).
DECODE_TRAFFIC = {
    "sources": ("paper_2609_32663_gb300/csrc/dkv_decode_mma.cu", "paper_2609_32663_gb300/csrc/dkv_decode_common.cuh",
                "paper_2609_32663_gb300/csrc/dkv_ptx.cuh", "paper_2609_32663_gb300/csrc/dkv_internal.cuh"),
    "sha256": "d649ba7e47f67652d62273e1110a9e0bfd4e9e5fe7e5dbf1a8032ce3e8b55ffb",
    # ncu of decode_mma_kernel<4, 1, 1, 0>, llama8b-128k-l4, the 13th launch (layer 0
    # with 2 rows appended before it and one by it: 376,646 + 8 x 3 rows)
    "dram_bytes": 194_389_504 + 3_045_376,
    "algorithmic_bytes": 376_670 * 512 + 32 * (256 + 512) + 4 * 8 * 256,
}


def decode_traffic_per_launch(bytes_per_launch):
    """ncu-measured DRAM bytes of one decode launch scaled to `bytes_per_launch`, or None."""
    import hashlib
    h = hashlib.sha256()
    for f in DECODE_TRAFFIC["sources"]:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    if DECODE_TRAFFIC["sha256"] is None or h.hexdigest() != DECODE_TRAFFIC["sha256"]:
        return None
    return int(round(bytes_per_launch * DECODE_TRAFFIC["dram_bytes"] / DECODE_TRAFFIC["algorithmic_bytes"]))


METRIC = "compacted decode-attention us/step (Llama-3.1-8B KV shape, 131072 ctx, 34.6% retention)"
UNIT = "us/step"


DEFAULT_STEPS = 256
DEFAULT_WARMUP = 8


@contextlib.contextmanager
def nvtx(name):
    """An NVTX range around a bench phase (visible to a timeline profiler)."""
    import torch
    torch.cuda.nvtx.range_push(name)
    try:
        yield
    finally:
        torch.cuda.nvtx.range_pop()


def reserve_rows(steps, warmup):
    """Rows each slab keeps free for appended tokens: every step the run makes
    (the timed and warm-up graph replays, the instrumented eager steps, the e2e
    run) appends one, with room to spare."""
    return steps + warmup + 64


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=DEFAULT_STEPS)
    ap.add_argument("--warmup", type=int, default=DEFAULT_WARMUP)
    ap.add_argument("--impl", default="dkv", choices=["dkv", "reference"])
    ap.add_argument("--workload", default="llama8b-128k", choices=sorted(I.WORKLOADS))
    ap.add_argument("--no-dense", action="store_true", help="skip the dense-cache baseline")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--no-workloads", action="store_true", help="skip the other workloads' lines")
    ap.add_argument("--cpu-layers", type=int, default=2, help="layers of one step the CPU oracle times")
    ap.add_argument("--profile", action="store_true", help="few steps, no baselines (for ncu)")
    return ap.parse_args()


# ---------------------------------------------------------------- distributed plumbing
class Dist:
    def __init__(self, n):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        self.cuda = False
        if self.world > 1:
            import torch
            import torch.distributed as dist
            self.cuda = torch.cuda.is_available()
            if self.cuda:
                # One GPU per rank: the rank's device is current before NCCL binds to it.
                torch.cuda.set_device(self.local)
                dist.init_process_group("nccl", device_id=torch.device("cuda", self.local))
            else:
                dist.init_process_group("gloo")
            self.pg = dist

    def barrier(self):
        if self.pg:
            if self.cuda:
                self.pg.barrier(device_ids=[self.local])
            else:
                self.pg.barrier()

    def max(self, x):
        if not self.pg:
            return x
        import torch
        dev = torch.device("cuda", self.local) if self.cuda else "cpu"
        t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


# ---------------------------------------------------------------- clocks
class Clocks:
    """nvidia-smi sampler over the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.idx = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
            t0 = time.time()
            while not self.lines and time.time() - t0 < 3.0 and self.proc.poll() is None:
                time.sleep(0.01)  # the sampler is running before the timed region starts
            self.lines.clear()
        except (OSError, FileNotFoundError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons, power = [], None, set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax = float(f[2])
                power.append(float(f[3]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_max": max(power) if power else None}


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


# ---------------------------------------------------------------- workload set-up
def setup(wl, dev, reserve):
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    M = I.make_pattern(wl)
    Tc = I.context_lengths(wl)
    shape = dkv.Shape(L=wl.L, H=wl.H, H_kv=wl.Hkv, D=wl.D, sink=wl.sink, recent=wl.recent, bin_width=wl.W)
    T_stride = int(Tc.max()) + reserve  # room for the dense baseline's appended tokens
    K, V = I.dense_kv(wl.with_(T=T_stride), device=dev)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    plan = dkv.dkv_map_pattern(M, Tc, shape, reserve_rows=reserve)
    torch.cuda.synchronize()  # the call returns before its last kernel (the index list) ends
    map_first_ms = (time.perf_counter() - t0) * 1e3
    # The first call also pays the library's one-time set-up in this process
    # (kernel loading, launch configurations); a plan built again costs this:
    again = []
    for _ in range(3):
        t0 = time.perf_counter()
        p2 = dkv.dkv_map_pattern(M, Tc, shape, reserve_rows=reserve)
        torch.cuda.synchronize()
        again.append((time.perf_counter() - t0) * 1e3)
        p2.close()
    map_ms = statistics.median(again)
    info = dkv.dkv_plan_query(plan)
    Kc = torch.empty((info.total_rows, wl.head_dim), dtype=torch.bfloat16, device=dev)
    Vc = torch.empty_like(Kc)
    return dict(M=M, Tc=Tc, shape=shape, T_stride=T_stride, K=K, V=V, plan=plan, info=info, Kc=Kc, Vc=Vc,
                map_ms=map_ms, map_first_ms=map_first_ms, reserve=reserve)


def time_compaction(env, reps=10):
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    st = torch.cuda.current_stream()
    times = []
    for i in range(reps + 2):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        dkv.dkv_compact(env["plan"], env["K"], env["V"], env["Kc"], env["Vc"], T_stride=env["T_stride"])
        e1.record(st)
        e1.synchronize()
        if i >= 2:
            times.append(e0.elapsed_time(e1) * 1e-3)
    t = statistics.median(times)
    kept = env["info"].kept_rows
    algo = kept * (2 * 256 * 2 + 4)  # read K,V rows + write K,V rows + read the 4-byte index
    return {"gbs": algo / t / 1e9, "ms": t * 1e3, "algorithmic_bytes": algo, "reps": reps}


def time_topk(wl, dev, reps=10):
    """The exact-budget pattern export (dkv_topk_mask) on the workload's
    L x H x D probabilities and on a large synthetic one. `us`: CUDA events
    around `reps` back-to-back calls, per call; `us_single`: the median of single
    calls, each bracketed by its own events (host launch cost included).
    Algorithmic bytes: P read once + M written (5 bytes an entry); the radix
    select (one cooperative launch after a workspace memset) streams P four
    times, from L2 after the first at these sizes, and writes M."""
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    ws = torch.empty(dkv.dkv_topk_workspace_bytes() // 4 + 1, dtype=torch.int32, device=dev)
    out = {}
    big = wl.with_(L=80, H=64, D=2048)
    for tag, w in (("pattern", wl), ("large", big)):
        P = torch.from_numpy(I.retention_probs(w)).to(dev)
        M = torch.empty(P.shape, dtype=torch.uint8, device=dev)
        K = dkv.dkv_budget(0.35, w.L, w.H, w.D)
        times = []
        for i in range(reps + 2):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            dkv.dkv_topk_mask(P, K, M, ws)
            e1.record()
            e1.synchronize()
            if i >= 2:
                times.append(e0.elapsed_time(e1) * 1e-3)
        single = statistics.median(times)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            dkv.dkv_topk_mask(P, K, M, ws)
        e1.record()
        e1.synchronize()
        t = e0.elapsed_time(e1) * 1e-3 / reps
        n = P.numel()
        out[tag] = {"shape": [w.L, w.H, w.D], "n": n, "K": K, "us": round(t * 1e6, 2),
                    "us_single": round(single * 1e6, 2), "algorithmic_gbs": round(5 * n / t / 1e9, 1),
                    "streamed_gbs": round(17 * n / t / 1e9, 1), "launches": 1}
    return out


def time_compaction_inplace(wl, env, reps=5):
    """The in-place path on page-backed caches: the dense K and V are copied into
    dkv_vmm buffers, dkv_compact_inplace is timed there (median of reps; later
    reps move already-moved bytes, the same volume), then dkv_vmm_trim releases
    the pages no slab needs. Bytes: the rows that move (from the first dropped
    position of each slab on), read and written, plus their indices."""
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    T_stride, reserve = env["T_stride"], env["reserve"]
    plan = dkv.dkv_map_pattern_inplace(env["M"], env["Tc"], env["shape"], T_stride, reserve_rows=reserve)
    ln, _, ioff, idx = dkv.dkv_plan_read(plan)
    moved = 0
    for h in range(len(ln)):
        ids = idx[ioff[h]:ioff[h + 1]]
        stay = np.flatnonzero(ids != np.arange(ids.size))
        moved += ids.size - (int(stay[0]) if stay.size else ids.size)
    shape = tuple(env["K"].shape)
    nbytes = env["K"].numel() * 2
    bufK, bufV = dkv.VmmBuffer(nbytes), dkv.VmmBuffer(nbytes)
    try:
        K, V = bufK.tensor(shape, torch.bfloat16), bufV.tensor(shape, torch.bfloat16)
        K.copy_(env["K"])
        V.copy_(env["V"])
        times = []
        st = torch.cuda.current_stream()
        for i in range(reps + 1):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(st)
            dkv.dkv_compact_inplace(plan, K, V)
            e1.record(st)
            e1.synchronize()
            if i >= 1:
                times.append(e0.elapsed_time(e1) * 1e-3)
        mapped0 = bufK.mapped_bytes() + bufV.mapped_bytes()
        freed = bufK.trim(plan, guard_rows=16) + bufV.trim(plan, guard_rows=16)
        mapped1 = bufK.mapped_bytes() + bufV.mapped_bytes()
        del K, V
    finally:
        plan.close()
        bufK.close()
        bufV.close()
    t = statistics.median(times)
    algo = moved * (2 * 256 * 2 + 4)
    return {"ms": round(t * 1e3, 3), "gbs": round(algo / t / 1e9, 1), "moved_rows": int(moved),
            "kept_rows": int(ln.sum()), "dense_bytes": int(mapped0), "mapped_after_trim": int(mapped1),
            "freed_bytes": int(freed), "mapped_fraction": round(mapped1 / mapped0, 4),
            "packed_bytes": int(ln.sum()) * 512, "how": "median of %d on dkv_vmm buffers, then dkv_vmm_trim" % reps}


def time_multi_query(wl, env, dev, Q, steps, warmup):
    """Q queries per sequence over the compressed cache (dkv_decode_multi), one
    CUDA graph of L launches per step; the K/V rows are read once for all Q."""
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    g = torch.Generator(device=dev)
    g.manual_seed(wl.seed * 1000 + 31)
    q = torch.randn((wl.L, wl.B, Q, wl.H, wl.head_dim), generator=g, device=dev).to(torch.bfloat16)
    out = torch.empty((wl.L, wl.B, Q, wl.H, wl.head_dim), dtype=torch.float32, device=dev)
    n_app = torch.zeros(wl.B, dtype=torch.int32, device=dev)

    def step():
        for layer in range(wl.L):
            dkv.dkv_decode_multi(env["plan"], layer, q[layer], Q, n_app, env["Kc"], env["Vc"], out[layer])

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for _ in range(warmup):
        graph.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        graph.replay()
    e1.record()
    e1.synchronize()
    return e0.elapsed_time(e1) * 1e-3 / steps


def profile_multi_query(wl, env, dev, Qs=(2, 4, 8, 16)):
    """Eager dkv_decode_multi launches, one per layer for each Q, untimed: the
    timed multi-query runs are graph replays, and these are the launches a
    profiler selects."""
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    n_app = torch.zeros(wl.B, dtype=torch.int32, device=dev)
    for Q in (q for q in Qs if q * wl.G <= 64):
        q = torch.randn((wl.B, Q, wl.H, wl.head_dim), device=dev).to(torch.bfloat16)
        out = torch.empty((wl.B, Q, wl.H, wl.head_dim), dtype=torch.float32, device=dev)
        for layer in range(wl.L):
            dkv.dkv_decode_multi(env["plan"], layer, q, Q, n_app, env["Kc"], env["Vc"], out)
    torch.cuda.synchronize()


def l2_label(kv_bytes, l2_bytes):
    """How the timed steps meet the rule against L2-resident inputs: a step's
    K/V bytes well above L2, or else an honest note (the `workloads` block times
    such a workload over rotated copies instead)."""
    if kv_bytes >= 4 * l2_bytes:
        return "inputs larger than L2 (%.2f GB of K/V per step)" % (kv_bytes / 1e9)
    return ("L2-resident: %.3f GB of K/V per step against a %.0f MB L2, not flushed between steps; "
            "the workloads block of the default run times this configuration over rotated copies"
            % (kv_bytes / 1e9, l2_bytes / 1e6))


def step_bytes(wl, Tc_rows_per_layer, with_new=True):
    """Algorithmic bytes of one decode step: retained K/V rows (with appended
    tokens) + q read + o written + the new K/V row written."""
    kv = Tc_rows_per_layer * 2 * 256
    q = wl.B * wl.H * wl.head_dim * 2
    o = wl.B * wl.H * wl.head_dim * 4
    new = 2 * wl.B * wl.Hkv * 256 if with_new else 0
    return kv + q + o + new


class DecodeRunner:
    """One decode step over all layers as a CUDA graph (dkv_decode_attn per layer,
    then dkv_advance), or the same launches eagerly with per-launch events."""

    def __init__(self, wl, plan, Kc, Vc, dev, seed_offset=0):
        import torch

        import paper_2609_32663_gb300.dkv as dkv
        self.dkv, self.torch = dkv, torch
        self.wl, self.plan, self.Kc, self.Vc = wl, plan, Kc, Vc
        q, kn, vn = I.decode_inputs(wl, 1, device=dev, seed_offset=seed_offset)
        self.q, self.kn, self.vn = q[0].contiguous(), kn[0].contiguous(), vn[0].contiguous()
        self.n_app = torch.zeros(wl.B, dtype=torch.int32, device=dev)
        self.out = torch.empty((wl.L, wl.B, wl.H, wl.head_dim), dtype=torch.float32, device=dev)
        self.graph = None

    def launch_step(self):
        d = self.dkv
        for layer in range(self.wl.L):
            d.dkv_decode_attn(self.plan, layer, self.q[layer], self.kn[layer], self.vn[layer], self.n_app,
                              self.Kc, self.Vc, self.out[layer])
        d.dkv_advance(self.plan, self.n_app)

    def capture(self):
        torch = self.torch
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.launch_step()  # warm the launch path outside capture
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        self.n_app.zero_()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            self.launch_step()
        torch.cuda.synchronize()
        self.n_app.zero_()

    def replay(self):
        self.graph.replay()

    def timed_launches(self, steps):
        """Eager steps with CUDA events around every decode launch: mean duration."""
        torch, d = self.torch, self.dkv
        st = torch.cuda.current_stream()
        durs = []
        for _ in range(steps):
            evs = []
            for layer in range(self.wl.L):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(st)
                d.dkv_decode_attn(self.plan, layer, self.q[layer], self.kn[layer], self.vn[layer], self.n_app,
                                  self.Kc, self.Vc, self.out[layer])
                e1.record(st)
                evs.append((e0, e1))
            d.dkv_advance(self.plan, self.n_app)
            torch.cuda.synchronize()
            durs.extend(e0.elapsed_time(e1) * 1e-3 for e0, e1 in evs)
        return statistics.mean(durs), len(durs)


def workload_line(name, dev, steps, warmup, dist, peak):
    """One more workload at full size, timed like the headline one: map, pack,
    the decode-step graph replayed `steps` times after `warmup`, and the dense
    baseline (same kernels, uncompressed cache). Inputs larger than L2."""
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    wl = I.WORKLOADS[name]
    reserve = reserve_rows(steps, warmup)
    env = setup(wl, dev, reserve)
    try:
        dkv.dkv_compact(env["plan"], env["K"], env["V"], env["Kc"], env["Vc"], T_stride=env["T_stride"])
        NHl = wl.B * wl.Hkv
        kept = env["info"].kept_rows
        runner = DecodeRunner(wl, env["plan"], env["Kc"], env["Vc"], dev)
        runner.capture()
        t, _ = time_graph(runner, steps, warmup, dist)
        t = dist.max(t)
        del runner
        rows = kept + wl.L * NHl * (warmup + (steps - 1) / 2.0 + 1)
        algo = step_bytes(wl, rows)
        out = {"us_per_step": round(t * 1e6, 2), "gb_per_step": round(algo / 1e9, 4),
               "gbs": round(algo / t / 1e9, 1), "frac_of_hbm": round(algo / t / 1e9 / peak, 4),
               "physical_retention": round(kept / (wl.L * wl.Hkv * float(env["Tc"].sum())), 4),
               "steps": steps, "l2": "inputs larger than L2 (%.2f GB of K/V per step)" % (rows * 512 / 1e9)}
        dense = dkv.dkv_plan_dense(env["Tc"], env["shape"], T_stride=env["T_stride"])
        dr = DecodeRunner(wl, dense, env["K"], env["V"], dev)
        dr.capture()
        td, _ = time_graph(dr, steps, warmup, dist)
        td = dist.max(td)
        del dr
        dense.close()
        drows = wl.L * wl.Hkv * float(env["Tc"].sum()) + wl.L * NHl * (warmup + (steps - 1) / 2.0 + 1)
        out.update({"dense_us_per_step": round(td * 1e6, 2), "dense_gbs": round(step_bytes(wl, drows) / td / 1e9, 1),
                    "speedup_of_compacted": round(td / t, 3), "ideal_speedup": round(drows / rows, 3)})
        return out
    finally:
        env["plan"].close()
        del env
        torch.cuda.empty_cache()


def rotated_small_workload(name, dev, steps, warmup, dist, peak, l2_multiple=4):
    """A workload whose caches fit in L2 (the 1-layer 4K one: 14.7 MB a step),
    measured from HBM: N copies of the packed caches (and of the dense ones for
    the baseline), N chosen so that they span at least `l2_multiple` x L2, and a
    graph of N decode steps, step i on copy i (each copy with its own appended-
    row counter). Consecutive steps read different bytes, and a copy is read
    again only after the other N - 1, far more than L2 holds, were streamed."""
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    wl = I.WORKLOADS[name]
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    reserve = reserve_rows(steps, warmup)
    env = setup(wl, dev, reserve)
    try:
        dkv.dkv_compact(env["plan"], env["K"], env["V"], env["Kc"], env["Vc"], T_stride=env["T_stride"])
        kept = env["info"].kept_rows
        NHl = wl.B * wl.Hkv
        q, kn, vn = I.decode_inputs(wl, 1, device=dev)
        q, kn, vn = q[0].contiguous(), kn[0].contiguous(), vn[0].contiguous()
        out = torch.empty((wl.L, wl.B, wl.H, wl.head_dim), dtype=torch.float32, device=dev)

        def timed(plan, K, V, rows_bytes):
            n = max(2, -(-l2_multiple * l2 // rows_bytes))
            caches = [(K.clone(), V.clone(), torch.zeros(wl.B, dtype=torch.int32, device=dev)) for _ in range(n)]

            def launch():
                for Kx, Vx, na in caches:
                    for layer in range(wl.L):
                        dkv.dkv_decode_attn(plan, layer, q[layer], kn[layer], vn[layer], na, Kx, Vx, out[layer])
                    dkv.dkv_advance(plan, na)

            st = torch.cuda.Stream()
            st.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(st):
                launch()
            torch.cuda.current_stream().wait_stream(st)
            torch.cuda.synchronize()
            for _, _, na in caches:
                na.zero_()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                launch()
            reps = max(1, -(-steps // n))
            for _ in range(max(1, -(-warmup // n))):
                g.replay()
            torch.cuda.synchronize()
            dist.barrier()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(reps):
                g.replay()
            e1.record()
            e1.synchronize()
            t = dist.max(e0.elapsed_time(e1) * 1e-3 / (reps * n))
            napp_mid = max(1, -(-warmup // n)) + (reps - 1) / 2.0
            return t, n, reps, napp_mid, n * rows_bytes

        packed_bytes = env["info"].total_rows * 512
        t, n, reps, napp_mid, span = timed(env["plan"], env["Kc"], env["Vc"], packed_bytes)
        rows = kept + wl.L * NHl * (napp_mid + 1)
        algo = step_bytes(wl, rows)
        res = {"us_per_step": round(t * 1e6, 2), "gb_per_step": round(algo / 1e9, 5),
               "gbs": round(algo / t / 1e9, 1), "frac_of_hbm": round(algo / t / 1e9 / peak, 4),
               "steps": reps * n,
               "l2": "rotating %d copies of the packed caches, %.0f MB in all (%.1f x the %.0f MB L2)"
                     % (n, span / 1e6, span / l2, l2 / 1e6)}
        dense = dkv.dkv_plan_dense(env["Tc"], env["shape"], T_stride=env["T_stride"])
        td, dn, _, dmid, dspan = timed(dense, env["K"], env["V"], env["K"].numel() * 4)
        dense.close()
        drows = wl.L * wl.Hkv * float(env["Tc"].sum()) + wl.L * NHl * (dmid + 1)
        res.update({"dense_us_per_step": round(td * 1e6, 2), "dense_gbs": round(step_bytes(wl, drows) / td / 1e9, 1),
                    "dense_l2": "rotating %d copies of the dense caches, %.0f MB" % (dn, dspan / 1e6),
                    "speedup_of_compacted": round(td / t, 3), "ideal_speedup": round(drows / rows, 3)})
        return res
    finally:
        env["plan"].close()
        del env
        torch.cuda.empty_cache()


def time_graph(runner, steps, warmup, dist, clocks=None):
    import torch
    for _ in range(warmup):
        runner.replay()
    torch.cuda.synchronize()
    dist.barrier()
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
    st = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(steps):
        runner.replay()
    e1.record(st)
    e1.synchronize()
    torch.cuda.synchronize()
    clk = clocks.stop() if clocks else None
    dist.barrier()
    return e0.elapsed_time(e1) * 1e-3 / steps, clk


def run_e2e(wl, plan, Kc, Vc, dev, steps, warmup):
    """Same step through the public API with host buffers: every step copies its
    q, k_new, v_new from pinned host memory and reads all layers' outputs back."""
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    q, kn, vn = I.decode_inputs(wl, 1, seed_offset=7)
    hq, hk, hv = q[0].pin_memory(), kn[0].pin_memory(), vn[0].pin_memory()
    hout = torch.empty((wl.L, wl.B, wl.H, wl.head_dim), dtype=torch.float32).pin_memory()
    dq, dk, dv = torch.empty_like(hq, device=dev), torch.empty_like(hk, device=dev), torch.empty_like(hv, device=dev)
    out = torch.empty((wl.L, wl.B, wl.H, wl.head_dim), dtype=torch.float32, device=dev)
    n_app = torch.zeros(wl.B, dtype=torch.int32, device=dev)

    def step():
        dq.copy_(hq, non_blocking=True)
        dk.copy_(hk, non_blocking=True)
        dv.copy_(hv, non_blocking=True)
        for layer in range(wl.L):
            dkv.dkv_decode_attn(plan, layer, dq[layer], dk[layer], dv[layer], n_app, Kc, Vc, out[layer])
        dkv.dkv_advance(plan, n_app)
        hout.copy_(out, non_blocking=True)

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        step()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step()
    for _ in range(warmup):
        g.replay()
    torch.cuda.synchronize()
    st = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(st)
    for _ in range(steps):
        g.replay()
    e1.record(st)
    e1.synchronize()
    t = e0.elapsed_time(e1) * 1e-3 / steps
    bi = hq.numel() * 2 + hk.numel() * 2 + hv.numel() * 2
    bo = hout.numel() * 4
    return t, bi, bo


def cpu_oracle_step(wl, env, layers, dev):
    """CPU oracle (single thread, fp64) on `layers` layers of one decode step over
    the packed cache built on the GPU; returns seconds per full step (scaled by L)."""
    import torch

    import oracle as O
    import paper_2609_32663_gb300.dkv as dkv
    ln, off, ioff, idx = dkv.dkv_plan_read(env["plan"])
    NHl = wl.B * wl.Hkv
    q, _, _ = I.decode_inputs(wl, 1, seed_offset=3)
    total = 0.0
    rows = 0
    for layer in range(layers):
        lo, hi = int(off[layer * NHl]), int(off[(layer + 1) * NHl])
        Kh = I.bf16_bits(env["Kc"][lo:hi])
        Vh = I.bf16_bits(env["Vc"][lo:hi])
        m = O.Mapping(ln, off - lo, ioff, idx)
        qb = I.bf16_bits(q[0, layer])
        t0 = time.perf_counter()
        O.decode(m, layer, wl.B, wl.H, wl.Hkv, qb, Kh, Vh)
        total += time.perf_counter() - t0
        rows += int(ln[layer * NHl:(layer + 1) * NHl].sum())
    return total / layers * wl.L, rows


def cpu_oracle_step_threads(wl, env, threads):
    """The CPU oracle on `threads` layers of one decode step at once, one layer a
    thread (the oracle's C call releases the interpreter lock); returns seconds
    per full step (wall time scaled by L / threads) and the threads used."""
    import concurrent.futures as cf

    import oracle as O
    import paper_2609_32663_gb300.dkv as dkv
    ln, off, ioff, idx = dkv.dkv_plan_read(env["plan"])
    NHl = wl.B * wl.Hkv
    q, _, _ = I.decode_inputs(wl, 1, seed_offset=3)
    n = max(1, min(threads, wl.L))
    jobs = []
    for layer in range(n):
        lo, hi = int(off[layer * NHl]), int(off[(layer + 1) * NHl])
        jobs.append((layer, O.Mapping(ln, off - lo, ioff, idx), I.bf16_bits(q[0, layer]),
                     I.bf16_bits(env["Kc"][lo:hi]), I.bf16_bits(env["Vc"][lo:hi])))
    with cf.ThreadPoolExecutor(max_workers=n) as ex:
        t0 = time.perf_counter()
        list(ex.map(lambda j: O.decode(j[1], j[0], wl.B, wl.H, wl.Hkv, j[2], j[3], j[4]), jobs))
        t = time.perf_counter() - t0
    return t * wl.L / n, n


def cpu_oracle_compaction(wl, env, layer=0):
    """CPU oracle (single thread) prune-and-pack of one layer of the dense caches,
    the same bytes the GPU pack moves; returns seconds per full pass (scaled by L)
    and the layer's kept rows."""
    import oracle as O
    import paper_2609_32663_gb300.dkv as dkv
    ln, off, ioff, idx = dkv.dkv_plan_read(env["plan"])
    NHl = wl.B * wl.Hkv
    a, b = layer * NHl, (layer + 1) * NHl
    m = O.Mapping(ln[a:b].copy(), (off[a:b + 1] - off[a]).copy(), (ioff[a:b + 1] - ioff[a]).copy(),
                  idx[int(ioff[a]):int(ioff[b])].copy())
    Kh = I.bf16_bits(env["K"][layer])
    Vh = I.bf16_bits(env["V"][layer])
    t0 = time.perf_counter()
    O.compact(m, 1, wl.B, wl.Hkv, Kh, Vh, env["T_stride"])
    t = time.perf_counter() - t0
    return t * wl.L, int(ln[a:b].sum())


def cpu_model():
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                if ln.lower().startswith(("model name", "cpu part")):
                    return ln.split(":", 1)[1].strip()
    except OSError:
        pass
    return "unknown"


# ---------------------------------------------------------------- arms
def run_dkv(args, dist):
    import torch

    import paper_2609_32663_gb300.dkv as dkv
    from paper_2609_32663_gb300 import build
    build.build_library()
    dev = torch.device("cuda", dist.local)
    torch.cuda.set_device(dev)
    wl = I.WORKLOADS[args.workload]
    steps, warmup = args.steps, max(args.warmup, 3)
    if args.profile:
        steps, warmup = min(steps, 2), min(warmup, 3)
    reserve = reserve_rows(steps, warmup)
    with nvtx("setup: map, dense caches"):
        env = setup(wl, dev, reserve)
    with nvtx("compaction"):
        comp = time_compaction(env, reps=3 if args.profile else 10)
    info = env["info"]
    NHl = wl.B * wl.Hkv
    ln, *_ = dkv.dkv_plan_read(env["plan"])
    rows_layer = [int(ln[l * NHl:(l + 1) * NHl].sum()) for l in range(wl.L)]

    runner = DecodeRunner(wl, env["plan"], env["Kc"], env["Vc"], dev)
    runner.capture()
    clocks = Clocks(dist.local)
    with nvtx("decode step graph (timed)"):
        t_step, clk = time_graph(runner, steps, warmup, dist, clocks)
    t_step = dist.max(t_step)
    # Rows attended per step (the cache grows by one row per slab per step).
    napp_mid = warmup + (steps - 1) / 2.0
    rows_step = sum(rows_layer) + wl.L * NHl * (napp_mid + 1)
    algo_step = step_bytes(wl, rows_step)

    # Dominant kernel: the decode kernel (split-K pass with the combine fused), per
    # launch (one layer): retained K/V rows + q read + o written + new K/V row in and out.
    n_inst = 4 if args.profile else 16
    before = runner.n_app.clone()
    with nvtx("decode launches (eager, timed)"):
        t_part, n_launch = runner.timed_launches(n_inst)
    if args.profile:
        with nvtx("multi-query launches (eager)"):
            profile_multi_query(wl, env, dev)
    napp_inst = float(before[0].item()) + (n_inst - 1) / 2.0
    rows_launch = (sum(rows_layer) + wl.L * NHl * (napp_inst + 1)) / wl.L
    part_bytes = rows_launch * 512 + wl.B * wl.H * (256 + 512) + 4 * wl.B * wl.Hkv * 256
    peaks, src = measured_peaks()
    peak = float(peaks["hbm_gbs"])
    # In the timed graph consecutive decode launches overlap (programmatic dependent
    # launch), so a launch's duration there is the timed region / launches; the
    # advance kernel's share is left in (an upper bound on the decode launch).
    t_launch = t_step / wl.L
    achieved = part_bytes / t_launch / 1e9

    res = {
        "metric": METRIC, "value": round(t_step * 1e6, 2), "unit": UNIT, "n_gpus": dist.world,
        "steps": steps, "warmup": warmup, "ms_per_step": round(t_step * 1e3, 4),
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16 in, fp32 accumulate; P.V with P as a bf16 hi+lo pair (~16 significant bits)",
        "io_dtype": "bf16 q/K/V, fp32 out", "data": "synthetic",
        "config": {"workload": wl.name, "layers": wl.L, "q_heads": wl.H, "kv_heads": wl.Hkv, "head_dim": wl.head_dim,
                   "batch": wl.B, "ctx_len": [int(x) for x in env["Tc"]][:16], "bins": wl.D, "bin_width": wl.W,
                   "sink": wl.sink, "recent": wl.recent,
                   "physical_retention": round(info.kept_rows / (wl.L * wl.Hkv * float(env["Tc"].sum())), 4),
                   "logical_retention": round(float(env["M"].mean()), 4),
                   "parallelism": f"replicas x{dist.world}",
                   "l2": l2_label(rows_step * 512, torch.cuda.get_device_properties(dev).L2_cache_size),
                   "graph": "one CUDA graph per step: %d x dkv_decode_attn + dkv_advance" % wl.L},
        "tokens_per_s": round(wl.B * dist.world / t_step, 1),
        "algorithmic_gb_per_step": round(algo_step / 1e9, 4),
        "step_gbs": round(algo_step / t_step / 1e9, 1),
        "step_frac_of_hbm": round(algo_step / t_step / 1e9 / peak, 4),
        "roofline": {"bound": "hbm", "kernel": "decode_mma_kernel<G, fused>", "achieved": round(achieved, 1),
                     "peak": peak, "unit": "GB/s", "frac": round(achieved / peak, 4), "peak_source": src,
                     "frac_of_nominal_8000": round(achieved / 8000.0, 4),
                     "bytes_per_launch": int(part_bytes), "avg_launch_us": round(t_launch * 1e6, 2),
                     "launches_timed": steps * wl.L,
                     "how": "CUDA events around the timed graph replays; avg launch = region / (steps x layers)",
                     "isolated_launch_us": round(t_part * 1e6, 2), "isolated_launches": n_launch,
                     "traffic": decode_traffic_per_launch(part_bytes),
                     "traffic_how": "ncu dram__bytes_read.sum + dram__bytes_write.sum of one launch of the "
                                    "4-layer case with the same per-layer sizes, scaled by algorithmic bytes; "
                                    "null if the kernel sources changed since"},
        "compaction": {"gbs": round(comp["gbs"], 1), "ms": round(comp["ms"], 3),
                       "frac_of_hbm": round(comp["gbs"] / peak, 4), "kept_rows": info.kept_rows},
        "map_ms": round(env["map_ms"], 3),
        "map_first_call_ms": round(env["map_first_ms"], 3),
        "map_how": "wall time of dkv_map_pattern + a device sync: median of 3 plans built after the first; "
                   "the first call of the process also loads the library's kernels",
        "gpu_launches": steps * (wl.L + 1),
        "clocks": clk,
    }
    del runner

    if not args.no_dense and not args.profile:
        dense = dkv.dkv_plan_dense(env["Tc"], env["shape"], T_stride=env["T_stride"])
        dr = DecodeRunner(wl, dense, env["K"], env["V"], dev)
        dr.capture()
        with nvtx("dense baseline graph (timed)"):
            t_dense, _ = time_graph(dr, steps, warmup, dist)
        t_dense = dist.max(t_dense)
        dense_rows = wl.L * float(env["Tc"].sum()) * wl.Hkv + wl.L * NHl * (napp_mid + 1)
        res["dense_baseline"] = {"us_per_step": round(t_dense * 1e6, 2),
                                 "gbs": round(step_bytes(wl, dense_rows) / t_dense / 1e9, 1),
                                 "speedup_of_compacted": round(t_dense / t_step, 3),
                                 "ideal_speedup": round(dense_rows / rows_step, 3)}
        del dr
        dense.close()

    # End to end through the public API with host buffers (fresh plan state).
    env2_plan = env["plan"]
    with nvtx("e2e graph with host copies (timed)"):
        t_e2e, bi, bo = run_e2e(wl, env2_plan, env["Kc"], env["Vc"], dev, max(8, min(steps, 32)), warmup)
    t_e2e = dist.max(t_e2e)
    res["e2e"] = {"value": round(t_e2e * 1e6, 2), "unit": UNIT, "h2d_bytes_per_step": int(bi),
                  "d2h_bytes_per_step": int(bo), "steps": max(8, min(steps, 32)),
                  "how": "CUDA graph of: H2D q/k_new/v_new from pinned host, L x dkv_decode_attn, dkv_advance, "
                         "D2H of all layers' outputs"}

    if dist.rank == 0 and dist.world == 1 and not args.no_cpu and not args.profile:
        layers = max(1, min(args.cpu_layers, wl.L))
        with nvtx("CPU oracle"):
            t_cpu, rows = cpu_oracle_step(wl, env, layers, dev)
        res["cpu_baseline"] = {"value": round(t_cpu * 1e6, 1), "unit": UNIT, "cores": 1, "kind": "oracle",
                               "sample": f"fp64 scalar oracle, {layers} of {wl.L} layers of one decode step "
                                         f"({rows} rows x G={wl.G} heads), scaled x{wl.L / layers:g} to a step",
                               "cpu": cpu_model(), "nproc": os.cpu_count()}
        with nvtx("CPU oracle, all cores"):
            t_all, n_thr = cpu_oracle_step_threads(wl, env, os.cpu_count() or 1)
        res["cpu_baseline_all_cores"] = {"value": round(t_all * 1e6, 1), "unit": UNIT, "cores": n_thr,
                                         "kind": "oracle",
                                         "sample": f"{n_thr} layers of one decode step, one a thread, "
                                                   f"scaled x{wl.L / n_thr:g} to a step"}
        with nvtx("CPU oracle compaction"):
            t_cc, kept_cc = cpu_oracle_compaction(wl, env)
        res["cpu_compaction"] = {"ms_per_pass": round(t_cc * 1e3, 1), "cores": 1, "kind": "oracle",
                                 "gbs": round(2 * 512 * kept_cc * wl.L / t_cc / 1e9, 2),
                                 "sample": f"row-by-row pack of layer 0 of {wl.L} ({kept_cc} kept rows), "
                                           f"scaled x{wl.L} to a pass"}
    if not args.profile:
        with nvtx("pattern export"):
            res["pattern_export"] = time_topk(wl, dev)
        mq = {}
        for Q in sorted({1, max(1, 8 // wl.G), max(1, 16 // wl.G), max(1, 32 // wl.G), max(1, 64 // wl.G)}):
            with nvtx(f"multi-query Q={Q} graph (timed)"):
                t_q = dist.max(time_multi_query(wl, env, dev, Q, min(steps, 64), warmup))
            rows_q = sum(rows_layer)  # no appends in these calls
            # K/V rows once for all Q queries, plus every query's q read and out written.
            bytes_q = step_bytes(wl, rows_q, with_new=False) + (Q - 1) * wl.B * wl.H * wl.head_dim * (2 + 4)
            gbs_q = bytes_q / t_q / 1e9
            mq[f"Q{Q}"] = {"us_per_step": round(t_q * 1e6, 2), "queries_per_s": round(wl.B * Q * dist.world / t_q, 1),
                           "columns": Q * wl.G, "kernel": "tcgen05" if Q * wl.G > 16 else "mma.sync",
                           "gbs": round(gbs_q, 1), "frac_of_hbm": round(gbs_q / peak, 4)}
        res["multi_query"] = mq
    if not args.profile:
        with nvtx("in-place compaction"):
            res["compaction_inplace"] = time_compaction_inplace(wl, env)  # last: overwrites the dense caches
    st = dkv.dkv_plan_status(env["plan"])
    res["device_status_word"] = st
    env["plan"].close()
    del env
    torch.cuda.empty_cache()
    if not args.profile and not args.no_workloads:
        # The other workloads of the benchmark set that fit a few seconds: the
        # 32K Llama cache and the 64K Qwen cache (35 % budget), and the 1-layer
        # 4K case measured from HBM over rotated copies.
        wls = {}
        for name in ("llama8b-32k", "qwen7b-64k-b4-r35"):
            if name != wl.name:
                with nvtx(f"workload {name} (timed)"):
                    wls[name] = workload_line(name, dev, steps, warmup, dist, peak)
        with nvtx("workload llama8b-1layer-4k, rotated caches (timed)"):
            wls["llama8b-1layer-4k"] = rotated_small_workload("llama8b-1layer-4k", dev, steps, warmup, dist, peak)
        res["workloads"] = wls
    return res


def run_reference(args, dist):
    """The oracle as it stands, timed on the host cores, per decode step of the
    same workload (bounded sample of layers per step, scaled to a full step)."""
    import oracle as O
    wl = I.WORKLOADS[args.workload]
    M = I.make_pattern(wl)
    Tc = I.context_lengths(wl)
    layers = 1
    # The sample: layer 0 of the workload (its pattern, contexts, and K/V and q
    # drawn by the workload's own generators for a model of one layer), mapped
    # and packed by the oracle; each timed step decodes that layer and is
    # scaled to the model's L layers.
    one = wl.with_(L=layers)
    sub = O.Geometry(L=layers, H=wl.H, Hkv=wl.Hkv, D=wl.D, sink=wl.sink, recent=wl.recent, bin_width=wl.W)
    m = O.map_pattern(M[:layers], Tc, sub, reserve=0)
    K, V = I.dense_kv(one)
    Kc, Vc = O.compact(m, layers, wl.B, wl.Hkv, I.bf16_bits(K), I.bf16_bits(V), wl.T)
    del K, V
    steps, warmup = max(1, min(args.steps, 3)), min(args.warmup, 1)
    qs, _, _ = I.decode_inputs(one, warmup + steps)
    times = []
    for i in range(warmup + steps):
        q = I.bf16_bits(qs[i, 0])
        t0 = time.perf_counter()
        O.decode(m, 0, wl.B, wl.H, wl.Hkv, q, Kc, Vc)
        if i >= warmup:
            times.append((time.perf_counter() - t0) * wl.L / layers)
    t = statistics.mean(times)
    return {"impl": "reference", "metric": METRIC, "value": round(t * 1e6, 1), "unit": UNIT, "n_gpus": dist.world,
            "steps": steps, "warmup": warmup, "ms_per_step": round(t * 1e3, 3), "higher_is_better": False,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": wl.name, "layers": wl.L, "q_heads": wl.H, "kv_heads": wl.Hkv, "batch": wl.B,
                       "ctx_len": [int(x) for x in Tc][:16]},
            "cpu_baseline": {"value": round(t * 1e6, 1), "unit": UNIT, "kind": "oracle", "cores": 1,
                             "sample": f"layer 0 of {wl.L} per step (all its KV heads; the workload's pattern, K/V and q recipe), scaled to a step",
                             "cpu": cpu_model(), "nproc": os.cpu_count()},
            "e2e": {"value": round(t * 1e6, 1), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    args = parse()
    dist = Dist(args.gpus)
    try:
        if args.impl == "reference":
            if dist.rank != 0:
                return
            res = run_reference(args, dist)
        else:
            res = run_dkv(args, dist)
        if dist.rank == 0:
            print(json.dumps(res), flush=True)
    finally:
        dist.close()


if __name__ == "__main__":
    main()
