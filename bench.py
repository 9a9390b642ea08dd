"""Benchmark of one LTD draft-and-verify cycle on GB300.

A step is one whole cycle of the hot path on one batch of synthetic input:
tree reset, L draft-tree expansions, top-N selection, tree attention in every
layer, acceptance and KV compaction in every layer.  Default workload: the
8B-class shape (batch 1, 32 query / 8 KV heads, head_dim 128, context 4096,
vocab 128256, depth 6, k 10, N 60, 32 layers, bf16, greedy).

Prints one JSON line.  `value` is device time per cycle in microseconds
(lower is better) with every input resident in HBM; `e2e` repeats the
measurement through the Python binding with the step's inputs copied from
pinned host memory and the result read back.  `--impl reference` times the
fp64 CPU oracle on the same workload instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "draft-verify cycle µs at 8B shape; tree-attn HBM GB/s vs ~8 TB/s peak"
N_LAYERS = {"tiny": 1, "8b": 32, "13b": 40, "32b": 64, "70b": 80}


def _args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="8b", choices=list(N_LAYERS))
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-policy", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-sample-s", type=float, default=15.0)
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the other workloads' summaries (configs) after the headline")
    ap.add_argument("--min-timed-ms", type=float, default=250.0,
                    help="each step replays the cycle graph enough times that the K timed steps "
                         "last at least this long (so the clock sampler sees the load)")
    ap.add_argument("--next-hint", action="store_true",
                    help="give every layer's attention call the next layer's caches as an L2 "
                         "prefetch hint (measured slower on GB300 at these shapes: off by default)")
    ap.add_argument("--no-next-hint", action="store_true",
                    help="the default (kept so older command lines still run)")
    ap.add_argument("--profile-case", default=None, choices=["draft", "select", "accept"],
                    help="no timing: run one phase of the --config workload three times, eagerly, "
                         "for a profiler to capture (draft: reset + levels 1..3; select: the whole "
                         "draft + selection; accept: the acceptance row pass and walk)")
    return ap.parse_args()


def run_profile_case(args):
    """Eager calls of one phase for an external profiler; prints "ok"."""
    import torch
    from paper_2603_01639_gb300 import build, ltd
    from paper_2603_01639_gb300 import workload as wl
    build.build()
    cfg = wl.config(args.config)
    device = torch.device("cuda")
    cyc = Cycle(cfg, 1, args.seed, device)
    for _ in range(3):
        if args.profile_case == "accept":
            ltd.ltd_accept(cyc.tree, cyc.target, cyc.draft, cyc.sel[0], cyc.n_verify, cyc.mode, cyc.ctx,
                           seed=1234, cycle=0, workspace=cyc.acc_ws, out=cyc.acc)
            continue
        ltd.ltd_tree_reset(cyc.tree, cyc.root)
        last = 3 if args.profile_case == "draft" else cyc.max_depth
        for level in range(1, last + 1):
            ltd.ltd_expand_tree(cyc.tree, level, cyc.draft, active=cyc.actives[level])
        if args.profile_case == "select":
            ltd.ltd_select_verify(cyc.tree, cyc.n_verify, cfg.max_n, cyc.ctx, out=cyc.sel)
    torch.cuda.synchronize()
    if ltd.ltd_check() != 0:
        raise RuntimeError("device error flagged")
    print("ok", args.profile_case, args.config)
    return 0


def _dist():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def config_obj(cfg, layers):
    """The `config` object of the JSON line, the same in both arms."""
    kv = 2 * layers * cfg.batch * cfg.hkv * cfg.s_cap * cfg.head_dim * (2 if cfg.dtype == "bf16" else 4)
    return {"workload": workload_desc(cfg, layers), "batch_per_gpu": cfg.batch, "layers": layers,
            "l2": f"inputs larger than L2: {kv / 1e6:.0f} MB of KV cache streamed per cycle between "
                  f"reuses of any buffer"}


def load_peaks():
    """(HBM GB/s, dense bf16 TFLOP/s sustained, source): the measured copy and
    GEMM peaks of this machine, else the recipe's fallback figures."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d.get("bf16_tflops_sustained") or d["bf16_tflops"]), \
            "measured"
    except (OSError, ValueError, KeyError):
        return 6800.0, 1700.0, "fallback"


# the resource that binds tree attention at each workload's shape (flops per
# algorithmic byte against the measured ridge of ~280): HBM at 8B (227) and
# 13B (16-92), the tensor pipe at 32B (375) and 70B (461)
BINDING = {"tiny": "hbm", "8b": "hbm", "13b": "hbm", "32b": "tensor", "70b": "tensor"}


def workload_desc(cfg, layers):
    return (f"{cfg.name}-class: batch {cfg.batch}, {cfg.hq} query / {cfg.hkv} KV heads, "
            f"head_dim {cfg.head_dim}, ctx {cfg.ctx_range[0]}..{cfg.ctx_range[1]}, "
            f"vocab {cfg.vocab}, depth {cfg.depth_range[0]}..{cfg.depth_range[1]}, k {cfg.W}, "
            f"N {cfg.n_range or cfg.n_choices}, {layers} layers, {cfg.dtype}, {cfg.mode}")


# ---------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-i", str(index), "-lms", "200"], stdout=subprocess.PIPE,
                stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = [r.split(", ") for r in out.strip().splitlines() if r.count(",") >= 7]
        if not rows:
            return None
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(rows)}


class NvmlClockSampler:
    """SM clock, power and clock-event reasons polled every millisecond by a
    thread through the driver's NVML library (read-only queries), so that a
    timed region of a few milliseconds still gets samples."""

    REASONS = {0x8: "hw_slowdown", 0x40: "hw_thermal_slowdown", 0x20: "sw_thermal_slowdown",
               0x4: "sw_power_cap", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, index: int):
        import ctypes
        import threading
        self.ok = False
        try:
            self.lib = ctypes.CDLL("libnvidia-ml.so.1")
        except OSError:
            return
        L = self.lib
        if L.nvmlInit_v2() != 0:
            return
        count = ctypes.c_uint(0)
        if L.nvmlDeviceGetCount_v2(ctypes.byref(count)) != 0 or count.value == 0:
            return
        self.h = ctypes.c_void_p()
        idx = index if index < count.value else 0
        if L.nvmlDeviceGetHandleByIndex_v2(idx, ctypes.byref(self.h)) != 0:
            return
        self.reasons_fn = getattr(L, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            getattr(L, "nvmlDeviceGetCurrentClocksThrottleReasons", None)
        mx = ctypes.c_uint(0)
        self.max_mhz = float(mx.value) if L.nvmlDeviceGetMaxClockInfo(self.h, 1, ctypes.byref(mx)) == 0 \
            else None
        if self.max_mhz is not None:
            self.max_mhz = float(mx.value)
        self.samples = []
        self.stop_flag = threading.Event()
        self.ctypes = ctypes
        self.thread = threading.Thread(target=self._run, daemon=True)
        self.ok = True
        self.thread.start()

    def _run(self):
        c = self.ctypes
        mhz, bits, mw = c.c_uint(0), c.c_ulonglong(0), c.c_uint(0)
        while not self.stop_flag.is_set():
            if self.lib.nvmlDeviceGetClockInfo(self.h, 1, c.byref(mhz)) == 0:
                r = self.reasons_fn(self.h, c.byref(bits)) if self.reasons_fn else 1
                p = self.lib.nvmlDeviceGetPowerUsage(self.h, c.byref(mw))
                self.samples.append((mhz.value, bits.value if r == 0 else 0, mw.value if p == 0 else 0))
            time.sleep(0.001)

    def stop(self):
        if not self.ok:
            return None
        self.stop_flag.set()
        self.thread.join(timeout=2)
        try:
            self.lib.nvmlShutdown()
        except Exception:
            pass
        if not self.samples:
            return None
        reasons = sorted({name for _, b, _ in self.samples for bit, name in self.REASONS.items()
                          if b & bit})
        return {"sm_mhz": statistics.median(s[0] for s in self.samples), "sm_max_mhz": self.max_mhz,
                "reasons": reasons, "samples": len(self.samples),
                "power_w_max": round(max(s[2] for s in self.samples) / 1000.0, 1),
                "source": "nvml, 1 ms"}


def clock_sampler(index: int):
    s = NvmlClockSampler(index)
    return s if s.ok else ClockSampler(index)


# ---------------------------------------------------------- the GPU cycle
class Cycle:
    """All device buffers of one synthetic cycle and the calls that run it."""

    def __init__(self, cfg, layers, seed, device):
        import torch
        from paper_2603_01639_gb300 import ltd
        from paper_2603_01639_gb300 import workload as wl
        self.torch, self.ltd, self.wl = torch, ltd, wl
        self.cfg, self.layers, self.device = cfg, layers, device
        tdt = torch.bfloat16 if cfg.dtype == wl.BF16 else torch.float32
        self.tdt = tdt
        B, d = cfg.batch, cfg.head_dim
        g = torch.Generator(device=device).manual_seed(seed)
        self.q = [torch.randn(B, cfg.max_n, cfg.hq, d, generator=g, device=device).to(tdt)
                  for _ in range(layers)]
        self.k = [torch.randn(B, cfg.hkv, cfg.s_cap, d, generator=g, device=device).to(tdt)
                  for _ in range(layers)]
        self.v = [torch.randn(B, cfg.hkv, cfg.s_cap, d, generator=g, device=device).to(tdt)
                  for _ in range(layers)]
        self.out = torch.zeros(B, cfg.max_n, cfg.hq, d, dtype=tdt, device=device)
        self.kv = ltd.KVCache(self.k, self.v)
        self.tree = ltd.Tree(B, cfg.max_depth, cfg.W, cfg.vocab)
        self.att_ws = ltd.attention_workspace(B, cfg.hq, cfg.hkv, d, cfg.max_n, cfg.max_ctx, tdt,
                                              device)
        self.acc_ws = ltd.accept_workspace(B, cfg.max_n, cfg.vocab, device)
        self.sel = (torch.empty(B, cfg.max_n, dtype=torch.int32, device=device),
                    torch.empty(B, cfg.max_n, dtype=torch.int32, device=device),
                    torch.empty(B, cfg.max_n, (cfg.max_n + 31) // 32, dtype=torch.int32,
                                device=device))
        self.acc = {"path": torch.empty(B, cfg.max_depth + 1, dtype=torch.int32, device=device),
                    "accept_len": torch.empty(B, dtype=torch.int32, device=device),
                    "bonus": torch.empty(B, dtype=torch.int32, device=device),
                    "new_ctx": torch.empty(B, dtype=torch.int32, device=device)}
        self.load(wl.draw_cycle(cfg, seed), seed)

    def load(self, ci, seed):
        """The per-cycle inputs of one drawn cycle (depths, verify sizes, contexts,
        modes, draft rows) and its target logits, planted on the tree this
        draft produces (the draft runs once to learn it)."""
        torch, wl, cfg, device = self.torch, self.wl, self.cfg, self.device
        self.ci = ci
        i32 = lambda x: torch.as_tensor(np.asarray(x, np.int32), device=device)  # noqa: E731
        self.root, self.depth = i32(ci.root), ci.depth
        self.n_verify, self.ctx, self.mode = i32(ci.n_verify), i32(ci.ctx), i32(ci.mode)
        self.draft = torch.from_numpy(ci.draft_rows).to(device).to(self.tdt)
        self.max_depth = int(ci.depth.max())
        self.actives = {}
        for level in range(1, self.max_depth + 1):
            m = (ci.depth >= level)
            self.actives[level] = None if m.all() else i32(m.astype(np.int32))
        self.draft_phase()
        torch.cuda.synchronize(device)
        view = {k: v.cpu().numpy() for k, v in self.tree.view().items()}
        ids = self.sel[0].cpu().numpy()
        target = wl.draw_target_rows(cfg, ci)
        rng = np.random.default_rng(seed + 99)
        for b in range(cfg.batch):
            N = int(ci.n_verify[b])
            wl.plant_agreement(cfg, target[b], ids[b, :N], view["parent"][b], view["token"][b],
                               view["depth"][b], rng, greedy=(ci.mode[b] == 0))
        self.target = torch.from_numpy(target).to(device).to(self.tdt)

    # phases ---------------------------------------------------------------
    def draft_phase(self):
        ltd = self.ltd
        ltd.ltd_tree_reset(self.tree, self.root)
        for level in range(1, self.max_depth + 1):
            ltd.ltd_expand_tree(self.tree, level, self.draft, active=self.actives[level])
        ltd.ltd_select_verify(self.tree, self.n_verify, self.cfg.max_n, self.ctx, out=self.sel)

    def verify_phase(self, hint=False):
        # with hint, each layer asks L2 for the next layer's keys and values
        # (a hint the library skips when one layer's K/V would crowd L2); the
        # launches are latency-bound, so the prefetch only competes with the
        # current layer's reads and the cycle runs without it
        for l in range(self.layers):
            nxt = l + 1 < self.layers and hint
            self.ltd.ltd_tree_attention(self.q[l], self.k[l], self.v[l], self.ctx, self.cfg.max_ctx,
                                        self.n_verify, self.sel[2], out=self.out,
                                        workspace=self.att_ws,
                                        next_k=self.k[l + 1] if nxt else None,
                                        next_v=self.v[l + 1] if nxt else None)

    def verify_phase_plain(self):
        self.verify_phase(hint=False)

    def verify_phase_hinted(self):
        self.verify_phase(hint=True)

    def accept_phase(self, cycle_no=0):
        self.ltd.ltd_accept(self.tree, self.target, self.draft, self.sel[0], self.n_verify,
                            self.mode, self.ctx, seed=1234, cycle=cycle_no, kv=self.kv,
                            workspace=self.acc_ws, out=self.acc)

    def attention_kernel(self):
        cfg = self.cfg
        return self.ltd.ltd_attention_kernel(self.tdt, cfg.batch, cfg.hq, cfg.hkv, cfg.head_dim,
                                             cfg.max_n, cfg.max_ctx)

    def launches_per_step(self):
        # reset, one expansion per level, selection, attention per layer,
        # acceptance (row statistics, walk) and the compaction of every layer
        return 1 + self.max_depth + 1 + self.layers * self.attention_kernel()[1] + 3

    # algorithmic bytes / flops of one attention launch
    def attention_algorithmic(self):
        cfg, ci = self.cfg, self.ci
        es = 2 if self.cfg.dtype == self.wl.BF16 else 4
        d = cfg.head_dim
        byts = flops = 0
        for b in range(cfg.batch):
            N, c = int(ci.n_verify[b]), int(ci.ctx[b])
            byts += N * cfg.hq * d * es * 2                    # q in, out
            byts += 2 * (c + N) * cfg.hkv * d * es             # K and V rows read
            byts += N * ((cfg.max_n + 31) // 32) * 4           # mask
            flops += 4 * N * cfg.hq * (c + N) * d
        return byts, flops


def _graph(torch, fn):
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        fn()
    torch.cuda.current_stream().wait_stream(s)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g


def _traffic_from_profiles(kernel_tag: str, sha: str):
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(kernel_tag)
    except (OSError, ValueError):
        return None
    if not rec or rec.get("source_sha") != sha:
        return None
    return rec.get("bytes_per_launch")


def _source_sha(files):
    h = hashlib.sha256()
    for fn in files:
        with open(os.path.join(ROOT, "paper_2603_01639_gb300", "csrc", fn), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def replica_seed(seed: int, rank: int) -> int:
    """Each rank drafts and verifies its own independent sequences."""
    return seed + 1000 * rank


def aggregate(total_ms: float, steps: int, batch: int, world: int, device=None):
    """Job time = the slowest rank's time (max over ranks); value = job time
    per cycle over the cycles all ranks completed.  Returns (ms per step,
    µs per cycle)."""
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([total_ms], dtype=torch.float64,
                         device=device if dist.get_backend() == "nccl" else "cpu")
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    ms_per_step = total_ms / steps
    return ms_per_step, ms_per_step * 1e3 / (batch * world)


# ----------------------------------------------------------- CPU baseline
def time_oracle_cycle(cfg, layers, seed, budget_s):
    """The fp64 oracle on the same workload: draft, selection, acceptance and
    attention; attention runs on one layer's KV (values do not change its
    cost) once per layer.  Returns (seconds per cycle, cycles timed, detail)."""
    import oracle
    from paper_2603_01639_gb300 import workload as wl
    ci = wl.draw_cycle(cfg, seed)
    q, k, v = wl.draw_attention(cfg, seed, ci.ctx, ci.n_verify)
    target = wl.draw_target_rows(cfg, ci)
    scale = 1.0 / math.sqrt(cfg.head_dim)
    draft64 = ci.draft_rows.astype(np.float64)
    q64, k64, v64 = q.astype(np.float64), k.astype(np.float64), v.astype(np.float64)

    def one():
        for b in range(cfg.batch):
            t = oracle.grow_tree(int(ci.root[b]), draft64[b], cfg.W, int(ci.depth[b]))
            N, c = int(ci.n_verify[b]), int(ci.ctx[b])
            ids, pos, mask, _ = oracle.select_verify(t, N, c)
            for _ in range(layers):
                oracle.tree_attention(q64[b, :N], k64[b], v64[b], c, mask, scale)
            rows = target[b, :N].astype(np.float64)
            if ci.mode[b] == 0:
                path, a, bonus = oracle.accept_greedy(t, ids, rows)
            else:
                path, a, bonus, _ = oracle.accept_stochastic(t, ids, rows, draft64[b], 1234, b, 0)
            for l in range(layers):
                oracle.compact_kv(k64[b, :, c:c + N + 1], 0, path)

    times = []
    t_start = time.perf_counter()
    while True:
        t0 = time.perf_counter()
        one()
        times.append(time.perf_counter() - t0)
        if time.perf_counter() - t_start > budget_s or len(times) >= 50:
            break
    return statistics.median(times), len(times)


def blas_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads", 1) for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return max(n)
    except Exception:
        pass
    return os.cpu_count() or 1


def cpu_baseline(cfg, layers, seed, budget_s):
    sec, n = time_oracle_cycle(cfg, layers, seed, budget_s)
    return {"value": round(sec * 1e6, 1), "unit": "us", "cores": blas_threads(), "kind": "oracle",
            "sample": f"{n} full oracle cycle(s) of the {cfg.name} workload (fp64 numpy; "
                      f"attention over {layers} layers reusing one layer's KV); median"}


def time_replays(torch, g, reps, device):
    """Mean device time of one replay of graph `g` over `reps` replays (CUDA
    events on the launching stream), in milliseconds."""
    stream = torch.cuda.current_stream(device)
    g.replay()
    torch.cuda.synchronize(device)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(reps):
        g.replay()
    e1.record(stream)
    torch.cuda.synchronize(device)
    return e0.elapsed_time(e1) / reps


def phases_in_cycle(torch, cyc, verify, reps, device):
    """Per-phase device time inside one CUDA graph of the whole cycle: event
    record nodes between the phases (each one makes the next phase's first
    kernel wait for the previous phase to finish, so the three add up to a
    little more than the clean cycle).  The per-phase graphs of phases_us
    also pay a graph launch each."""
    names = ("draft_select", "attention_all_layers", "accept_compact")
    try:
        evs = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(4)]

        def full_ev():
            evs[0].record()
            cyc.draft_phase()
            evs[1].record()
            verify()
            evs[2].record()
            cyc.accept_phase()
            evs[3].record()

        g = _graph(torch, full_ev)
        acc = [0.0, 0.0, 0.0]
        for _ in range(reps):
            g.replay()
            torch.cuda.synchronize(device)
            for i in range(3):
                acc[i] += evs[i].elapsed_time(evs[i + 1])
        del g
        return {k: round(v / reps * 1e3, 2) for k, v in zip(names, acc)}
    except (TypeError, RuntimeError) as e:
        return {"unavailable": str(e).splitlines()[0][:160] if str(e) else type(e).__name__}


def attention_roofline(cyc, launch_ms, bound):
    """Roofline of one tree-attention launch against its binding resource."""
    hbm, tc, src = load_peaks()
    byts, flops = cyc.attention_algorithmic()
    gbs = byts / (launch_ms * 1e-3) / 1e9
    tfs = flops / (launch_ms * 1e-3) / 1e12
    if bound == "tensor":
        achieved, peak, unit = tfs, tc, "TFLOP/s"
    else:
        achieved, peak, unit = gbs, hbm, "GB/s"
    return {"bound": bound, "achieved": round(achieved, 1), "peak": peak, "unit": unit,
            "frac": round(achieved / peak, 4), "peak_source": src + " (hbm_gbs; bf16_tflops_sustained)",
            "launch_us": round(launch_ms * 1e3, 3), "algorithmic_bytes_per_launch": byts,
            "flops_per_launch": flops, "gbs": round(gbs, 1), "tflops": round(tfs, 1),
            "hbm_frac": round(gbs / hbm, 4)}


# the target models' hidden sizes (public model configs of the paper's
# targets: Llama-3.1-8B, Vicuna-13B, Qwen3-32B, a 70B-class model), for the LM
# head over the verified tokens
HIDDEN = {"8b": 4096, "13b": 5120, "32b": 5120, "70b": 8192}


def time_lm_head(cfg, name, device, reps):
    """ltd_lm_head_row_stats over the verified tokens of one cycle (batch x
    n_max rows, up to the 256 one call takes) at the target's hidden size,
    statistics only, seeded random bf16 hidden states and weights; the
    weight (more than L2) streams from HBM at every replay."""
    import torch
    from paper_2603_01639_gb300 import ltd
    rows = cfg.batch * cfg.max_n
    if name not in HIDDEN or cfg.dtype != "bf16" or rows > 256:
        return None
    H = HIDDEN[name]
    g = torch.Generator(device=device).manual_seed(7)
    hid = torch.randn(rows, H, generator=g, device=device).to(torch.bfloat16)
    w = (torch.randn(cfg.vocab, H, generator=g, device=device) / math.sqrt(H)).to(torch.bfloat16)
    ws = torch.empty(ltd.lib().ltd_lm_head_workspace_bytes(rows, cfg.vocab, H), dtype=torch.uint8,
                     device=device)
    call = lambda: ltd.ltd_lm_head_row_stats(hid, w, workspace=ws)  # noqa: E731
    call()
    torch.cuda.synchronize(device)
    g_lm = _graph(torch, call)
    ms = time_replays(torch, g_lm, reps, device)
    ltd.ltd_check()
    hbm, tc, src = load_peaks()
    byts = cfg.vocab * H * 2 + rows * H * 2 + rows * 12
    gbs = byts / (ms * 1e-3) / 1e9
    res = {"rows": rows, "vocab": cfg.vocab, "hidden": H, "us": round(ms * 1e3, 2),
           "roofline": {"bound": "hbm", "achieved": round(gbs, 1), "peak": hbm, "unit": "GB/s",
                        "frac": round(gbs / hbm, 4), "peak_source": src,
                        "algorithmic_bytes_per_launch": byts,
                        "tflops": round(2 * rows * cfg.vocab * H / (ms * 1e-3) / 1e12, 1)},
           "launches": 2,
           "how": "the LM-head GEMM with row max / log-sum-exp / argmax in its epilogue and the "
                  "one-CTA merge, one CUDA graph, CUDA events over the replays"}
    del hid, w, ws, g_lm
    torch.cuda.empty_cache()
    return res


def summarize_config(name, args, device, seed, reps):
    """Full-cycle latency, phases, the attention roofline against the shape's
    binding resource and e2e for one workload (the 8B-class one is the
    headline line itself)."""
    import torch
    from paper_2603_01639_gb300 import workload as wl
    cfg = wl.config(name)
    layers = N_LAYERS[name]
    cyc = Cycle(cfg, layers, seed, device)

    def full():
        cyc.draft_phase()
        cyc.verify_phase()
        cyc.accept_phase()

    for _ in range(3):
        full()
    torch.cuda.synchronize(device)
    cyc.ltd.ltd_check()
    g_cycle, g_draft = _graph(torch, full), _graph(torch, cyc.draft_phase)
    g_verify, g_plain = _graph(torch, cyc.verify_phase), _graph(torch, cyc.verify_phase_plain)
    g_accept = _graph(torch, cyc.accept_phase)
    cycle_ms = time_replays(torch, g_cycle, reps, device)
    phases = {"draft_select": time_replays(torch, g_draft, reps, device),
              "attention_all_layers": time_replays(torch, g_verify, reps, device),
              "accept_compact": time_replays(torch, g_accept, reps, device)}
    plain_ms = time_replays(torch, g_plain, reps, device)
    cyc.ltd.ltd_check()
    g_accept.replay()
    torch.cuda.synchronize(device)
    acc_len = cyc.acc["accept_len"].cpu().numpy()
    res = {"workload": workload_desc(cfg, layers), "cycle_us": round(cycle_ms * 1e3, 2),
           "cycle_us_per_sequence": round(cycle_ms * 1e3 / cfg.batch, 2),
           "phases_us": {k: round(v * 1e3, 2) for k, v in phases.items()},
           "phases_in_cycle_us": phases_in_cycle(torch, cyc, cyc.verify_phase, reps, device),
           "attention": attention_roofline(cyc, plain_ms / layers, BINDING[name]),
           "attention_launch_us_in_cycle": round(phases["attention_all_layers"] * 1e3 / layers, 3),
           "tokens_per_cycle": int((acc_len + 1).sum()),
           "gpu_launches_per_cycle": cyc.launches_per_step(), "reps": reps}
    if name == "32b":
        # the compaction of the accepted path in every layer, timed alone
        path, alen = cyc.acc["path"], cyc.acc["accept_len"]
        g_comp = _graph(torch, lambda: cyc.ltd.ltd_kv_compact(cyc.kv, path, alen, cyc.ctx))
        comp_ms = time_replays(torch, g_comp, reps, device)
        a = int(acc_len.max())
        moved = 2 * (a + 1) * cfg.hkv * cfg.head_dim * 2 * layers * cfg.batch
        res["compaction"] = {"us": round(comp_ms * 1e3, 2), "accepted": a,
                             "bytes_read_and_written_each": moved,
                             "how": "ltd_kv_compact of the cycle's accepted path in all layers, one "
                                    "launch, CUDA graph replays"}
    lm = time_lm_head(cfg, name, device, reps)
    if lm is not None:
        res["lm_head"] = lm
    if not args.no_e2e:
        res["e2e"] = run_e2e(cyc, args, device)
    del cyc, g_cycle, g_draft, g_verify, g_plain, g_accept
    torch.cuda.empty_cache()
    return res


def sweep_13b(args, device, seed, cycles, reps):
    """The 13B-class workload over `cycles` seeded cycles, each with its own
    draft depth in 3..8 and verify size in {16, 32, 48, 64, 96} (the size and
    depth choices a policy would make), on one set of caches."""
    import torch
    from paper_2603_01639_gb300 import workload as wl
    cfg = wl.config("13b")
    layers = N_LAYERS["13b"]
    cyc = Cycle(cfg, layers, seed, device)
    per = []
    for c in range(cycles):
        s = seed + 1 + c
        cyc.load(wl.draw_cycle(cfg, s), s)

        def full():
            cyc.draft_phase()
            cyc.verify_phase()
            cyc.accept_phase(cycle_no=s)

        full()
        torch.cuda.synchronize(device)
        g = _graph(torch, full)
        gv = _graph(torch, cyc.verify_phase_plain)
        ms = time_replays(torch, g, reps, device)
        vms = time_replays(torch, gv, reps, device)
        g.replay()
        torch.cuda.synchronize(device)
        per.append({"depth": int(cyc.ci.depth[0]), "n_verify": int(cyc.ci.n_verify[0]),
                    "cycle_us": round(ms * 1e3, 2),
                    "attention_launch_us": round(vms * 1e3 / layers, 3),
                    "accepted": int(cyc.acc["accept_len"][0].item()),
                    "attention_hbm_frac": attention_roofline(cyc, vms / layers, "hbm")["frac"]})
        del g, gv
    cyc.ltd.ltd_check()
    del cyc
    torch.cuda.empty_cache()
    cyc_us = [p["cycle_us"] for p in per]
    return {"cycles": cycles, "cycle_us_mean": round(statistics.mean(cyc_us), 2),
            "cycle_us_min": min(cyc_us), "cycle_us_max": max(cyc_us),
            "attention_hbm_frac_mean": round(statistics.mean(p["attention_hbm_frac"] for p in per), 4),
            "tokens_per_cycle_mean": round(statistics.mean(p["accepted"] + 1 for p in per), 3),
            "per_cycle": per}


# ------------------------------------------------------------------ main
def run_reference(args):
    rank, world, _ = _dist()
    from paper_2603_01639_gb300 import workload as wl
    cfg = wl.config(args.config)
    layers = N_LAYERS[args.config]
    if rank != 0:
        return 0
    for _ in range(args.warmup):
        time_oracle_cycle(cfg, layers, args.seed, 0.0)
    times = []
    for _ in range(args.steps):
        t, _ = time_oracle_cycle(cfg, layers, args.seed, 0.0)
        times.append(t)
    v = statistics.mean(times) * 1e6
    line = {"impl": "reference", "metric": METRIC, "value": round(v, 1), "unit": "us",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(v / 1e3, 3), "higher_is_better": False, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_obj(cfg, layers),
            "cpu_baseline": {"value": round(v, 1), "unit": "us", "cores": blas_threads(),
                             "kind": "oracle",
                             "sample": f"each step one full oracle cycle (fp64 numpy); "
                                       f"attention over {layers} layers reusing one layer's KV"},
            "e2e": {"value": round(v, 1), "unit": "us", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args):
    import torch
    rank, world, local = _dist()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    from paper_2603_01639_gb300 import ltd
    from paper_2603_01639_gb300 import workload as wl
    from paper_2603_01639_gb300.build import build
    build()
    cfg = wl.config(args.config)
    layers = N_LAYERS[args.config]
    cyc = Cycle(cfg, layers, replica_seed(args.seed, rank), device)

    verify = cyc.verify_phase_hinted if args.next_hint else cyc.verify_phase_plain

    def full():
        cyc.draft_phase()
        verify()
        cyc.accept_phase()

    for _ in range(max(args.warmup, 3)):
        full()
    torch.cuda.synchronize(device)
    ltd.ltd_check()
    g_draft = _graph(torch, cyc.draft_phase)
    g_verify = _graph(torch, verify)
    g_plain = _graph(torch, cyc.verify_phase_plain)
    g_accept = _graph(torch, cyc.accept_phase)
    # the whole cycle as one graph (the timed value); the per-phase graphs
    # give the breakdown
    g_cycle = _graph(torch, full)
    for _ in range(2):
        g_draft.replay(); g_verify.replay(); g_accept.replay(); g_cycle.replay()
    torch.cuda.synchronize(device)

    K = args.steps
    # a step is R replays of the cycle graph, R chosen so that the K timed
    # steps last at least --min-timed-ms (the same R on every rank)
    one_ms = time_replays(torch, g_cycle, 5, device)
    R = max(1, int(math.ceil(args.min_timed_ms / max(K * one_ms, 1e-3))))
    if world > 1:
        t = torch.tensor([R], dtype=torch.int64, device=device)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        R = int(t.item())
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(K)]
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize(device)
    clocks = clock_sampler(local)
    stream = torch.cuda.current_stream()
    c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    c0.record(stream)
    for i in range(K):
        for _ in range(R):
            g_cycle.replay()
    c1.record(stream)
    torch.cuda.synchronize(device)
    clk = clocks.stop()
    if world > 1:
        torch.distributed.barrier()
    for i in range(K):
        ev[i][0].record(stream)
        g_draft.replay()
        ev[i][1].record(stream)
        g_verify.replay()
        ev[i][2].record(stream)
        g_accept.replay()
        ev[i][3].record(stream)
    torch.cuda.synchronize(device)
    ltd.ltd_check()
    total_ms = c0.elapsed_time(c1) / R  # per cycle-graph replay, summed over the K steps
    draft_ms = statistics.mean(ev[i][0].elapsed_time(ev[i][1]) for i in range(K))
    verify_ms = statistics.mean(ev[i][1].elapsed_time(ev[i][2]) for i in range(K))
    accept_ms = statistics.mean(ev[i][2].elapsed_time(ev[i][3]) for i in range(K))
    in_cycle = phases_in_cycle(torch, cyc, verify, max(K, 10), device)
    ms_per_step, value_us = aggregate(total_ms, K, cfg.batch, world, device)

    # roofline of the dominant kernel (tree attention), on launches without
    # the next-layer hint, so that no byte is fetched outside the launch it
    # is counted for (the KV of all layers exceeds L2, so nothing is reused)
    torch.cuda.synchronize(device)
    pa, pb = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    pa.record(stream)
    for _ in range(K):
        g_plain.replay()
    pb.record(stream)
    torch.cuda.synchronize(device)
    plain_ms = pa.elapsed_time(pb) / K
    att_bytes, att_flops = cyc.attention_algorithmic()
    att_launch_ms = plain_ms / layers
    peaks_path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    peak_note = "measured"
    try:
        with open(peaks_path) as f:
            hbm_peak = float(json.load(f)["hbm_gbs"])
    except (OSError, ValueError, KeyError):
        hbm_peak, peak_note = 6800.0, "fallback"
    achieved = att_bytes / (att_launch_ms * 1e-3) / 1e9
    code, _ = cyc.attention_kernel()
    tag = "attn_tc" if code == 1 else "attn_simt"
    sha = _source_sha(ltd.attention_kernel_sources(code))
    traffic = _traffic_from_profiles(f"{tag}:{cfg.name}", sha)
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm_peak,
                "unit": "GB/s", "frac": round(achieved / hbm_peak, 4), "traffic": traffic,
                "peak_source": peak_note, "kernel": tag,
                "algorithmic_bytes_per_launch": att_bytes, "launch_us": round(att_launch_ms * 1e3, 3),
                "launch_us_in_cycle": round(verify_ms / layers * 1e3, 3),
                "note": "launch_us and achieved from launches without the next-layer L2 hint; "
                        "launch_us_in_cycle is the cycle's own per-layer time",
                "tflops": round(att_flops / (att_launch_ms * 1e-3) / 1e12, 1),
                "frac_of_8tbs": round(achieved / 8000.0, 4)}

    # the acceptance phase under each verification rule on this cycle (all
    # sequences on one rule; the timed cycle above keeps the workload's)
    rules = {}
    saved_mode = cyc.mode.clone()
    for rname, rmode in (("greedy", ltd.LTD_GREEDY), ("stochastic", ltd.LTD_STOCHASTIC),
                         ("point_mass", ltd.LTD_STOCHASTIC_POINT_MASS),
                         ("no_replacement", ltd.LTD_STOCHASTIC_NO_REPLACEMENT)):
        cyc.mode.fill_(rmode)
        g_rule = _graph(torch, cyc.accept_phase)
        g_rule.replay()
        torch.cuda.synchronize(device)
        r0, r1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        r0.record(stream)
        for _ in range(K):
            g_rule.replay()
        r1.record(stream)
        torch.cuda.synchronize(device)
        rules[rname] = round(r0.elapsed_time(r1) / K * 1e3, 2)
    cyc.mode.copy_(saved_mode)
    ltd.ltd_check()
    # re-run the workload's own acceptance so the outputs below are its own
    g_accept.replay()
    torch.cuda.synchronize(device)

    # the cycle's throughput, the reward of section 3.1: tokens emitted
    # (accepted + bonus) over the device time of the cycle
    acc_len = cyc.acc["accept_len"].cpu().numpy()
    reward = {"accept_len": acc_len.tolist(),
              "tokens_per_cycle": int((acc_len + 1).sum()),
              "tokens_per_s": round(float((acc_len + 1).sum()) / (ms_per_step * 1e-3), 1),
              "how": "(accepted + 1) summed over the batch / device time of one cycle"}

    pol = None
    if not args.no_policy:
        pol = time_policies(cyc, verify, K, device)

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(cyc, args, device)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(cfg, layers, args.seed, args.cpu_sample_s)

    lm_head = time_lm_head(cfg, args.config, device, max(10, min(K, 50))) if world == 1 else None

    # the other workloads: full-cycle latency, phases and the attention
    # roofline against each shape's binding resource (one GPU only)
    configs = None
    if world == 1 and not args.no_configs:
        reps = max(10, min(K, 50))
        configs = {}
        for name in N_LAYERS:
            if name == args.config:
                continue
            configs[name] = summarize_config(name, args, device, args.seed, reps)
            if name == "13b":
                configs[name]["sweep"] = sweep_13b(args, device, args.seed + 500, 32, reps)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value_us, 2), "unit": "us", "n_gpus": world,
            "steps": K, "warmup": args.warmup, "ms_per_step": round(ms_per_step * R, 4),
            "cycles_per_step": R,
            "higher_is_better": False, "scaling": "weak", "vs_baseline": None,
            "dtype": cfg.dtype, "data": "synthetic",
            "config": config_obj(cfg, layers),
            "timing": "CUDA events around K steps of R replays each of one CUDA graph of the "
                      "whole cycle; value = job time / cycles of all ranks; phases_us from "
                      "per-phase graphs timed after it (a graph launch each), phases_in_cycle_us "
                      "from event nodes inside one graph of the cycle; attention layers " +
                      ("with" if args.next_hint else "without") + " the next-layer L2 hint",
            "phases_us": {"draft_select": round(draft_ms * 1e3, 2),
                          "attention_all_layers": round(verify_ms * 1e3, 2),
                          "accept_compact": round(accept_ms * 1e3, 2)},
            "phases_in_cycle_us": in_cycle,
            "accept_rules_us": rules,
            "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "policy": pol, "reward": reward,
            "gpu_launches": cyc.launches_per_step() * K * R, "clocks": clk,
            "lm_head": lm_head, "configs": configs,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def time_policies(cyc, verify, steps, device):
    """The cycle with both learned policies in the loop (section 3.1): after
    every level the depth observation is gathered on the device, read back
    and fed to the depth policy; after the draft the size observation goes
    to the size policy.  Each decision needs the host, so this cycle runs as
    eager calls with one stream sync per decision.  The policies' weights are
    seeded random and their decisions are computed but not applied (depth
    and N stay the workload's), so the device work equals the timed cycle's;
    the same eager cycle without the policies is timed beside it.  Then the
    same networks run on the device (ltd_depth_policy / ltd_size_policy), the
    cycle captured as one CUDA graph with and without them."""
    import torch
    from paper_2603_01639_gb300 import policy
    ltd, cfg, tree = cyc.ltd, cyc.cfg, cyc.tree
    B, kk, v_pad = cfg.batch, cfg.W * cfg.W, tree.max_nodes
    pi_d, pi_v = policy.DepthPolicy(cfg.W, seed=0), policy.SizePolicy(v_pad, seed=1)
    d_obs = torch.empty(B, kk + 2, dtype=torch.float32, device=device)
    s_obs = torch.empty(B, v_pad + 2, dtype=torch.float32, device=device)
    h_d = torch.empty(B, kk + 2, dtype=torch.float32).pin_memory()
    h_s = torch.empty(B, v_pad + 2, dtype=torch.float32).pin_memory()
    stream = torch.cuda.current_stream(device)
    mlp_s = {"depth": [], "size": []}

    def decide(net, d_src, h_dst, key):
        h_dst.copy_(d_src, non_blocking=True)
        stream.synchronize()
        t0 = time.perf_counter()
        net.decide(h_dst.numpy())
        mlp_s[key].append(time.perf_counter() - t0)

    def adaptive():
        ltd.ltd_tree_reset(tree, cyc.root)
        for level in range(1, cyc.max_depth + 1):
            ltd.ltd_expand_tree(tree, level, cyc.draft, active=cyc.actives[level])
            ltd.ltd_depth_observation(tree, cyc.ctx, out=d_obs)
            decide(pi_d, d_obs, h_d, "depth")
        ltd.ltd_size_observation(tree, cyc.ctx, v_pad, out=s_obs)
        decide(pi_v, s_obs, h_s, "size")
        ltd.ltd_select_verify(tree, cyc.n_verify, cfg.max_n, cyc.ctx, out=cyc.sel)
        verify()
        cyc.accept_phase()

    def fixed():
        cyc.draft_phase()
        verify()
        cyc.accept_phase()

    # the same policies on the device: each decision is written where the
    # next launch reads it, and the whole cycle stays one CUDA graph
    dnet, snet = pi_d.net.device(device), pi_v.net.device(device)
    act_scr = torch.empty(B, dtype=torch.int32, device=device)
    n_scr = torch.empty(B, dtype=torch.int32, device=device)

    def device_adaptive():
        ltd.ltd_tree_reset(tree, cyc.root)
        for level in range(1, cyc.max_depth + 1):
            ltd.ltd_expand_tree(tree, level, cyc.draft, active=cyc.actives[level])
            ltd.ltd_depth_policy(tree, cyc.ctx, dnet, active_in=cyc.actives[level],
                                 active_out=act_scr)
        ltd.ltd_size_policy(tree, cyc.ctx, snet, cfg.max_n, v_pad=v_pad, n_verify=n_scr)
        ltd.ltd_select_verify(tree, cyc.n_verify, cfg.max_n, cyc.ctx, out=cyc.sel)
        verify()
        cyc.accept_phase()

    def depth_only():
        ltd.ltd_depth_policy(tree, cyc.ctx, dnet, active_in=None, active_out=act_scr)

    def size_only():
        ltd.ltd_size_policy(tree, cyc.ctx, snet, cfg.max_n, v_pad=v_pad, n_verify=n_scr)

    dev = {}
    for name, fn in (("graph_fixed", fixed), ("graph_with_device_policies", device_adaptive),
                     ("depth_policy_launch", depth_only), ("size_policy_launch", size_only)):
        fn()
        torch.cuda.synchronize(device)
        g = _graph(torch, fn)
        for _ in range(3):
            g.replay()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            g.replay()
        e1.record(stream)
        torch.cuda.synchronize(device)
        dev[name] = e0.elapsed_time(e1) / steps * 1e3
    cyc.ltd.ltd_check()

    res = {}
    for name, fn in (("eager_fixed", fixed), ("eager_with_policies", adaptive)):
        for _ in range(3):
            fn()
        torch.cuda.synchronize(device)
        for v in mlp_s.values():
            v.clear()
        t0 = time.perf_counter()
        for _ in range(steps):
            fn()
        torch.cuda.synchronize(device)
        res[name] = (time.perf_counter() - t0) / steps * 1e6
    over = res["eager_with_policies"] - res["eager_fixed"]
    return {"cycle_us_eager_with_policies": round(res["eager_with_policies"], 1),
            "cycle_us_eager_fixed": round(res["eager_fixed"], 1),
            "overhead_us": round(over, 1),
            "overhead_frac": round(over / res["eager_with_policies"], 4),
            "depth_decisions_per_cycle": cyc.max_depth,
            "depth_mlp_us": round(statistics.median(mlp_s["depth"]) * 1e6, 1),
            "size_mlp_us": round(statistics.median(mlp_s["size"]) * 1e6, 1),
            "mlp": "numpy fp32 on the host, seeded random weights, batch " + str(B),
            "how": "host wall clock over K eager cycles; decisions computed, not applied",
            "device": {
                "cycle_us_graph_with_device_policies": round(dev["graph_with_device_policies"], 2),
                "cycle_us_graph_fixed": round(dev["graph_fixed"], 2),
                "overhead_us": round(dev["graph_with_device_policies"] - dev["graph_fixed"], 2),
                "overhead_frac": round(1 - dev["graph_fixed"] / dev["graph_with_device_policies"], 4),
                "depth_policy_us": round(dev["depth_policy_launch"], 2),
                "size_policy_us": round(dev["size_policy_launch"], 2),
                "how": "the same networks in mlp_policy_kernel, decisions written to device "
                       "buffers (not applied), each cycle one CUDA graph; CUDA events over K "
                       "replays; the policy launches timed alone as graphs of one launch"}}


def run_e2e(cyc, args, device):
    """The same cycle through the public binding: per step, copy the draft
    logits, every layer's q and new K/V rows and the target logits from pinned
    host memory, run the cycle, read back path / accept length / bonus / ctx.
    The step's inputs sit in one pinned buffer and go over in one copy into
    one device buffer that holds the draft and target logits and every q in
    place; every layer's new K/V rows are then placed into its cache on the
    device by one ltd_kv_append launch (a host copy straight into the
    cache's strided rows ran at a few GB/s, one device copy per layer and
    tensor cost a launch each)."""
    import torch
    ltd, cfg = cyc.ltd, cyc.cfg
    c0 = int(cyc.ci.ctx.min())
    N = cfg.max_n
    # buffer order: draft logits | every q, every layer's new K, new V |
    # target logits | root
    knew = torch.stack([k[:, :, c0:c0 + N] for k in cyc.k])
    vnew = torch.stack([v[:, :, c0:c0 + N] for v in cyc.v])
    parts = [cyc.draft] + list(cyc.q) + [knew, vnew, cyc.target, cyc.root]
    offs, total = [], 0
    for t in parts:
        offs.append(total)
        total += (t.numel() * t.element_size() + 255) // 256 * 256
    h_buf = torch.empty(total, dtype=torch.uint8).pin_memory()
    d_buf = torch.empty(total, dtype=torch.uint8, device=device)
    views = []
    for t, o in zip(parts, offs):
        nbytes = t.numel() * t.element_size()
        h_buf[o:o + nbytes].view(t.dtype).view(t.shape).copy_(t.cpu().contiguous())
        views.append(d_buf[o:o + nbytes].view(t.dtype).view(t.shape))
    L = cyc.layers
    cyc.draft = views[0]
    cyc.q = views[1:1 + L]
    d_knew, d_vnew = views[1 + L], views[2 + L]
    cyc.target, cyc.root = views[-2], views[-1]
    # three spans of the buffer: what the draft phase needs, what attention
    # needs, what acceptance needs (then the root)
    a0, a1, a2 = offs[1], offs[-2], offs[-1]
    outs = {k: torch.empty(v.shape, dtype=v.dtype).pin_memory() for k, v in cyc.acc.items()}
    h2d = sum(t.numel() * t.element_size() for t in parts)
    d2h = sum(v.numel() * v.element_size() for v in outs.values())
    side = torch.cuda.Stream(device)
    ev_kv, ev_tgt = torch.cuda.Event(), torch.cuda.Event()

    def step():
        # side stream: attention's inputs (and their placement into the
        # caches), then acceptance's, while the main stream copies the draft
        # logits and drafts.  (Finer steps -- the draft rows level by level,
        # each layer's inputs behind its own event -- measured slower: the
        # cross-stream waits break the chain of programmatic launches.)
        main = torch.cuda.current_stream(device)
        side.wait_stream(main)
        d_buf[a2:].copy_(h_buf[a2:], non_blocking=True)  # root
        d_buf[:a0].copy_(h_buf[:a0], non_blocking=True)
        with torch.cuda.stream(side):
            d_buf[a0:a1].copy_(h_buf[a0:a1], non_blocking=True)
            # every layer's new rows into its cache, one launch
            ltd.ltd_kv_append(cyc.kv, d_knew, d_vnew, cyc.ctx, cyc.n_verify)
            ev_kv.record(side)
            d_buf[a1:a2].copy_(h_buf[a1:a2], non_blocking=True)
            ev_tgt.record(side)
        cyc.draft_phase()
        main.wait_event(ev_kv)
        cyc.verify_phase()
        main.wait_event(ev_tgt)
        cyc.accept_phase()
        for k in outs:
            outs[k].copy_(cyc.acc[k], non_blocking=True)

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(device)
    # the whole step (copies in, the three phases, copies out) as one CUDA
    # graph, as a serving loop would replay it
    try:
        g = _graph(torch, step)
        run, how = g.replay, "one CUDA graph per step: h2d copies from pinned memory (attention and acceptance inputs on a second stream, overlapping the draft phase), phases, d2h copies"
    except RuntimeError as exc:  # capture refused: time the eager calls
        torch.cuda.synchronize(device)
        run, how = step, f"eager calls (graph capture failed: {str(exc)[:80]})"
    for _ in range(max(3, args.warmup)):
        run()
    torch.cuda.synchronize(device)
    s, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s.record()
    for _ in range(args.steps):
        run()
    e.record()
    torch.cuda.synchronize(device)
    us = s.elapsed_time(e) * 1e3 / args.steps / cfg.batch
    return {"value": round(us, 2), "unit": "us", "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "how": how}


def main():
    args = _args()
    if args.profile_case:
        return run_profile_case(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
