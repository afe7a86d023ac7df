#!/usr/bin/env python3
"""Benchmark of the TaskPress compression path on GB300.

One step = the fused compression (V scales, guide scores, per-head
top-budget selection, compaction) of every layer of the workload in one
tp_compress_layers call, with K/V already resident in HBM.  The metric is context tokens
compressed per second per layer (all heads): value = n_tokens * layers / t_step.

Default workload: the Llama-3-8B-shaped 32-layer stack at 128K context with a
128-token guide (32 q / 8 KV heads, d = 128, keep 10%).  `--config 2` runs the
32K single layer.  Each layer's K+V (512 MiB at 128K) exceeds the 129 MB L2,
and consecutive layers use different buffers, so no L2 flush is needed.

Also reported on the same JSON line:
  roofline      the dominant kernel, timed per launch with CUDA events over a
                staged pass of the same workload (the fused call's kernels
                launched one entry point at a time), against the burst tensor
                peak (a kernel timed alone);
  hbm_fused     algorithmic bytes of the fused layer / its time / HBM peak;
  kernels       every kernel of the layer against its own bound (CUDA events,
                staged pass);
  workload_legs the other workloads of the metric, each through the same
                call: the 32K Llama layer, the 64K wide-GQA layer at its four
                keep ratios and the ragged 8-document batch (value, hbm_fused,
                staged kernel times), and the guide sweep of the paper's
                prefill table (64K layer, 64-, 256- and 1024-token guides);
  e2e           the same metric through the public API with the inputs in
                pinned host memory, H2D and D2H copies inside the timed region;
  cpu_baseline  the CPU oracle on every host core (a bounded sample of layer 0);
  clocks        nvidia-smi samples taken during the timed region;
  per_layer_calls  the same stack as one tp_compress_layer call per layer;
  graph_replay  the step's call captured as a CUDA graph and replayed;
  lse_given     the same stack through tp_compress_layers_lse, the row
                normalisers supplied by the caller (one scoring pass over K);
  literal_normaliser  the same stack through tp_compress_layer_guide (the
                guide's causal prefix folded into the normalisers).

`--impl reference` times the CPU oracle (the only other implementation of
this path) on the same workload and metric.
"""
from __future__ import annotations

import argparse
import datetime
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "context tokens compressed/s per layer (all heads) at 32K/128K; % of HBM roofline"
UNIT = "tokens/s/layer"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", type=int, default=3, choices=[1, 2, 3, 4, 5])
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--layers", type=int, default=0, help="override the workload's layer count")
    ap.add_argument("--e2e-layers", type=int, default=4)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-legs", action="store_true", help="skip the 32K / 64K / ragged workload legs")
    return ap.parse_args()


def dist_env():
    from paper_2608_03276_gb300 import replicas
    return replicas.dist_env()


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    """nvidia-smi clock and throttle-reason samples every 20 ms, time-stamped;
    summary() keeps the samples that fall inside the marked timed window."""
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None
        self.t_start = self.t_end = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def mark_start(self):
        self.t_start = datetime.datetime.now()

    def mark_end(self):
        self.t_end = datetime.datetime.now()

    def __exit__(self, *a):
        time.sleep(0.05)
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 10:
                    continue
                try:
                    ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f")
                    rows.append((ts, float(parts[2]), float(parts[3]),
                                 {nm for nm, val in zip(names, parts[6:10]) if val.lower().startswith("active")}))
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        margin = datetime.timedelta(milliseconds=25)
        inside = rows
        if self.t_start is not None and self.t_end is not None:
            inside = [r for r in rows if self.t_start - margin <= r[0] <= self.t_end + margin]
        window = len(inside)
        if not inside:  # timed region shorter than the sampling period: nearest sample after its start
            later = [r for r in rows if self.t_start is None or r[0] >= self.t_start]
            inside = later[:1] or rows[-1:]
        reasons = set()
        for r in inside:
            reasons |= r[3]
        return {"sm_mhz": statistics.median(r[1] for r in inside), "sm_max_mhz": max(r[2] for r in inside),
                "samples": len(inside), "samples_in_window": window,
                "window_ms": round((self.t_end - self.t_start).total_seconds() * 1e3, 1)
                if self.t_start and self.t_end else None,
                "reasons": sorted(reasons)}


# ---------------------------------------------------------------------------
# Algorithmic bytes / flops (per layer)
# ---------------------------------------------------------------------------
def layer_algorithmic(w, kept_total_tokens):
    """K + V read once, the compressed cache written once (Kc, Vc, int8 Vc, scale,
    index per kept token and head), the guide queries read once."""
    d = w.head_dim
    n = w.n_total
    read = 4 * d * n * w.n_heads_kv + 2 * d * w.batch * w.n_heads_q * w.guide_len
    write = (2 * d + 2 * d + d + 4 + 4) * kept_total_tokens
    flops_one_pass = 2 * w.rows * d * n * w.n_heads_kv
    return read, write, flops_one_pass


def traffic_record(kernel: str, workload: str):
    """Per-launch DRAM bytes of a kernel from the committed ncu summary, if the
    kernel source has not changed since the capture (else None)."""
    src = os.path.join(ROOT, "paper_2608_03276_gb300", "csrc", "score_tc.cu")
    try:
        sha = hashlib.sha256(open(src, "rb").read()).hexdigest()[:12]
        with open(os.path.join(ROOT, "profiles", "ncu_traffic.txt")) as f:
            for line in f:
                parts = line.split()
                if len(parts) >= 4 and not line.startswith("#") and parts[0] == kernel \
                        and parts[1] == workload and parts[2] == sha:
                    return float(parts[3])
    except Exception:
        pass
    return None


# ---------------------------------------------------------------------------
# CPU oracle sample (the cpu_baseline leg and the reference arm)
# ---------------------------------------------------------------------------
def cpu_model() -> str:
    """The host CPU's model name (x86 'model name', Arm 'CPU part' or lscpu)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu part")):
                    return line.split(":", 1)[1].strip()
    except Exception:
        pass
    import platform
    return platform.processor() or platform.machine()


def _oracle_worker_init():
    os.environ["OPENBLAS_NUM_THREADS"] = "1"
    os.environ["OMP_NUM_THREADS"] = "1"
    import numpy  # noqa: F401  (import cost outside the timed map)
    from oracle import taskpress_oracle  # noqa: F401


def _oracle_unit(args):
    """One (document 0, KV head) unit of the oracle: the whole per-head path
    (Eq. 2 scales, both scoring passes in fp64, pooling, full sort, gather)."""
    qf, kf, vf, g, keep_ratio, budget = args
    import numpy as np
    from oracle import taskpress_oracle as O
    q, k, v = np.load(qf), np.load(kf, mmap_mode="r"), np.load(vf, mmap_mode="r")
    t0 = time.perf_counter()
    out = O.compress_layer(q, k, v, [0, k.shape[1]], n_heads_q=g, n_heads_kv=1,
                           keep_ratio=keep_ratio, fixed_budget=budget)
    O.gather_rows(k, v, out["gamma"], out["vq"], 0, 0, out["idx"][(0, 0)])
    return time.perf_counter() - t0


class OracleSample:
    """The CPU oracle on every host core: document 0 of layer 0 of the workload
    is split into its KV heads, and each of the nproc worker processes (spawned
    before any timing, BLAS single-threaded) compresses one head; with more
    cores than heads, heads are repeated.  value = tokens x (units / H_kv) /
    wall, i.e. context tokens compressed per second per layer."""

    def __init__(self, w, cores=None):
        import multiprocessing as mp
        import numpy as np
        from paper_2608_03276_gb300 import synth
        self.w = w
        self.cores = cores or os.cpu_count() or 1
        one_doc = w.with_(doc_lens=(w.doc_lens[0],))
        x = synth.make_layer(one_doc)
        self.n = one_doc.n_total
        self.tmp = tempfile.mkdtemp(prefix="tp_oracle_")
        g = w.group
        files = []
        for h in range(w.n_heads_kv):
            fq, fk, fv = (os.path.join(self.tmp, f"{t}{h}.npy") for t in "qkv")
            np.save(fq, np.ascontiguousarray(x.q[:, h * g:(h + 1) * g]))
            np.save(fk, np.ascontiguousarray(x.k[h:h + 1]))
            np.save(fv, np.ascontiguousarray(x.v[h:h + 1]))
            files.append((fq, fk, fv))
        self.units = [files[i % w.n_heads_kv] + (g, w.keep_ratio, w.budget)
                      for i in range(self.cores)]
        self.pool = mp.get_context("spawn").Pool(processes=self.cores, initializer=_oracle_worker_init)
        self.pool.map(_oracle_worker_init_probe, range(self.cores))  # every worker is up

    def run(self):
        t0 = time.perf_counter()
        per_unit = self.pool.map(_oracle_unit, self.units, chunksize=1)
        wall = time.perf_counter() - t0
        layers = len(self.units) / self.w.n_heads_kv
        value = self.n * layers / wall
        detail = (f"{self.w.name}: document 0 of layer 0 (n={self.n}), {len(self.units)} (KV head) "
                  f"units = {layers:g} layer(s) of {self.w.n_heads_kv} heads on {self.cores} "
                  f"processes (one unit each, heads repeated when cores > heads), fp64 numpy; "
                  f"wall {wall:.1f}s, CPU {sum(per_unit):.1f}s")
        return value, detail

    def close(self):
        self.pool.close()
        self.pool.join()
        import shutil
        shutil.rmtree(self.tmp, ignore_errors=True)


def _oracle_worker_init_probe(_):
    return os.getpid()


def run_reference(args, w):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    sample = OracleSample(w)
    times = []
    detail = ""
    try:
        for i in range(args.warmup + args.steps):
            v, detail = sample.run()
            if i >= args.warmup:
                times.append(v)
    finally:
        sample.close()
    value = statistics.median(times)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "layers_sampled": 1, "heads_sampled": w.n_heads_kv},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": sample.cores, "kind": "oracle",
                         "cpu_model": cpu_model(), "sample": detail},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
def kept_tokens_of(w, binding, keep_ratio=None):
    r = w.keep_ratio if keep_ratio is None else keep_ratio
    return sum(int(min(w.budget, n)) if w.budget >= 0 else binding.tp_budget(int(n), r)
               for n in w.doc_lens) * w.n_heads_kv


def hbm_fused_of(w, kept_tokens, t_layer_s, hbm_peak, peak_src):
    """Algorithmic bytes of one layer (K + V read once, the compressed cache
    written once, the guide read once) over the layer's time, against HBM."""
    read_b, write_b, _ = layer_algorithmic(w, kept_tokens)
    ach = (read_b + write_b) / t_layer_s / 1e9
    return {"algorithmic_bytes": read_b + write_b, "achieved_gbs": ach, "peak_gbs": hbm_peak,
            "frac": ach / hbm_peak, "frac_of_nominal_8tbs": ach * 1e9 / 8e12,
            "peak_source": f"{peak_src} copy bandwidth"}


def staged_times(binding, torch, p, w, layers, outs, ws, stream, reps, keep_ratio=None):
    """Per-kernel CUDA-event times, one entry point at a time on the launching
    stream: pass 1 with the Eq. 2 scales (tp_guide_lse), pass 2 (tp_guide_key_scores),
    pass 2 forming the Eq. 2 scales as well (tp_guide_key_scores with V: the scoring
    kernel of the caller-normaliser path), the selection (tp_select) and the
    compaction (tp_compact) as standalone kernels."""
    dev = outs[0].idx.device
    r = w.keep_ratio if keep_ratio is None else keep_ratio
    lse = torch.empty((w.batch, w.n_heads_kv, w.rows), dtype=torch.float32, device=dev)
    skey = torch.empty((w.n_heads_kv, w.n_total), dtype=torch.float32, device=dev)
    gamma = torch.empty((w.n_heads_kv, w.n_total), dtype=torch.float32, device=dev)
    scores = torch.empty((w.n_heads_kv, w.n_total), dtype=torch.float32, device=dev)
    names = ["lse+vscale", "keyscore", "keyscore+vscale", "select", "gather"]
    acc = {s: 0.0 for s in names}
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)]
    nl = min(len(layers), 8)
    for _ in range(max(1, reps)):
        for li in range(nl):
            (q, k, v), o = layers[li], outs[li]
            binding.tp_guide_scores(p, q, k, gamma, scores, ws, stream)  # scores for select; not timed
            evs[0].record(stream)
            binding.tp_guide_lse(p, q, k, lse, ws, stream, v=v, gamma=gamma)
            evs[1].record(stream)
            binding.tp_guide_key_scores(p, q, k, lse, skey, stream)
            evs[2].record(stream)
            binding.tp_guide_key_scores(p, q, k, lse, skey, stream, v=v, gamma=gamma)
            evs[3].record(stream)
            binding.tp_select(p, scores, r, w.budget, o.idx, ws, stream)
            evs[4].record(stream)
            binding.tp_compact(p, k, v, gamma, o.idx, r, w.budget, o.kc, o.vc, o.vqc, o.gammac, stream)
            evs[5].record(stream)
            torch.cuda.synchronize()
            for i, name in enumerate(names):
                acc[name] += evs[i].elapsed_time(evs[i + 1])
    n = max(1, reps) * nl
    return {s: v / n for s, v in acc.items()}


def time_calls(torch, fn, steps, warmup, stream):
    for _ in range(warmup):
        fn()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(steps):
        fn()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def workload_leg(binding, torch, synth, w, n_layers, args, dev, stream, hbm_peak, peak_src,
                 keep_ratios=None):
    """Another workload of the metric (32K layer, 64K wide-GQA layer, ragged
    batch): tp_compress_layers over n_layers distinct layers per step (their
    K + V exceed L2 together), plus the staged per-kernel times."""
    L = n_layers
    p = binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, w.doc_offsets())
    layers = [synth.make_layer_torch(w, l, dev) for l in range(L)]
    out = {"workload": w.name, "n_ctx": w.n_total, "layers_per_step": L, "docs": w.batch,
           "guide_len": w.guide_len, "heads_q": w.n_heads_q, "heads_kv": w.n_heads_kv}
    legs = {}
    for r in (keep_ratios or (w.keep_ratio,)):
        outs = [binding.CompressOutputs(p, r, w.budget, dev, with_scores=False) for _ in range(L)]
        # the stack's workspace: short layers are selected several per launch
        ws = torch.empty(binding.tp_workspace_bytes_stack(p, r, w.budget, L), dtype=torch.uint8,
                         device=dev)
        for o in outs:
            o.ws = ws

        def step():
            binding.tp_compress_layers(p, layers, r, w.budget, outs, ws, stream)

        steps = max(args.steps, 20)
        with ClockSampler(dev.index or 0) as clocks:
            for _ in range(max(args.warmup, 3)):
                step()
            torch.cuda.synchronize()
            clocks.mark_start()
            ms = time_calls(torch, step, steps, 0, stream)
            clocks.mark_end()
        st = binding.tp_check_status(ws)
        if st != 0:
            raise RuntimeError(f"{w.name}: device status {binding.tp_status_string(st)}")
        kept = kept_tokens_of(w, binding, r)
        t_layer = ms / L / 1e3
        legs[f"keep_{r:g}" if w.budget < 0 else f"budget_{w.budget}"] = {
            "value": w.n_total / t_layer, "unit": UNIT, "ms_per_layer": ms / L,
            "hbm_fused": hbm_fused_of(w, kept, t_layer, hbm_peak, peak_src),
            "stages_ms": staged_times(binding, torch, p, w, layers, outs, ws, stream, 3, r),
            "kernels_per_layer": binding.tp_compress_kernel_count(p, r, w.budget, binding.MODE_TWO_PASS),
            "layers_per_selection": binding.tp_stack_layers_per_selection(p, r, w.budget, L, ws.numel()),
            "clocks": clocks.summary()}
        del outs, ws
    out["results"] = legs
    del layers
    torch.cuda.empty_cache()
    return out


def guide_sweep_leg(binding, torch, synth, args, dev, stream, tf_burst):
    """The setting of the paper's prefill table (Sec. 4.2.3): a Llama-3-8B-shaped
    layer (32 q / 8 KV heads, d = 128) at 64K context with 64-, 256- and
    1024-token guides at 75% eviction (keep 25%), through tp_compress_layers
    over two layers per step.  Guides above 512 stacked rows run in blocks of
    512 rows; the two exact passes then cost 4 * M * n * d flops per head."""
    base = synth.WORKLOADS[2].with_(name="llama8b-64k-guides", doc_lens=(65536,), keep_ratio=0.25)
    out = {"workload": base.name, "n_ctx": base.n_total, "layers_per_step": 2, "keep_ratio": 0.25,
           "heads_q": base.n_heads_q, "heads_kv": base.n_heads_kv}
    res = {}
    for lt in (64, 256, 1024):
        w = base.with_(guide_len=lt)
        L = 2
        p = binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, w.doc_offsets())
        layers = [synth.make_layer_torch(w, l, dev) for l in range(L)]
        outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, dev, with_scores=False)
                for _ in range(L)]
        ws = outs[0].ws
        for o in outs[1:]:
            o.ws = ws

        def step():
            binding.tp_compress_layers(p, layers, w.keep_ratio, w.budget, outs, ws, stream)

        with ClockSampler(dev.index or 0) as clocks:
            for _ in range(max(args.warmup, 3)):
                step()
            torch.cuda.synchronize()
            clocks.mark_start()
            ms = time_calls(torch, step, max(args.steps, 10), 0, stream)
            clocks.mark_end()
        st = binding.tp_check_status(ws)
        if st != 0:
            raise RuntimeError(f"guide {lt}: device status {binding.tp_status_string(st)}")
        t_layer = ms / L / 1e3
        flops = 4.0 * w.rows * w.n_total * w.head_dim * w.n_heads_kv
        res[f"guide_{lt}"] = {
            "rows": w.rows, "row_blocks": -(-w.rows // binding.TP_MAX_ROWS),
            "value": w.n_total / t_layer, "unit": UNIT, "ms_per_layer": ms / L,
            "tensor_frac_of_burst": flops / t_layer / 1e12 / tf_burst,
            "kernels_per_layer": binding.tp_compress_kernel_count(p, w.keep_ratio, w.budget,
                                                                  binding.MODE_TWO_PASS),
            "clocks": clocks.summary()}
        del outs, ws, layers
    out["results"] = res
    torch.cuda.empty_cache()
    return out


def run_ours(args, w):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2608_03276_gb300 import replicas

    rank, world, local = dist_env()
    if world > 1:
        replicas.init("nccl" if torch.cuda.is_available() else "gloo")
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_03276_gb300 import binding, synth

    hbm_peak, tf_burst, tf_sust, peak_src = measured_peaks()
    stream = torch.cuda.current_stream()

    # the metric's other workloads first, each with its own clock samples
    # (before the long 128K stack, so that none of them runs on a GPU that has
    # just spent seconds at its power limit)
    legs = {}
    if rank == 0 and not args.no_legs and args.config == 3:
        for cfg, nl, ratios in ((2, 4, None), (4, 4, (0.05, 0.10, 0.25, 0.50)), (5, 2, None)):
            wl = synth.WORKLOADS[cfg]
            legs[wl.name] = workload_leg(binding, torch, synth, wl.with_(seed=replicas.rank_seed(wl.seed, rank)),
                                         nl, args, dev, stream, hbm_peak, peak_src, ratios)
        legs["guide_sweep"] = guide_sweep_leg(binding, torch, synth, args, dev, stream, tf_burst)
    L = w.layers
    p = binding.Problem(w.n_heads_q, w.n_heads_kv, w.head_dim, w.guide_len, w.doc_offsets())
    # each rank compresses its own stack (weak scaling; no data-path collective)
    wr = w.with_(seed=replicas.rank_seed(w.seed, rank))
    layers = [synth.make_layer_torch(wr, l, dev) for l in range(L)]
    outs = [binding.CompressOutputs(p, w.keep_ratio, w.budget, dev, with_scores=False)
            for _ in range(L)]
    ws = outs[0].ws
    for o in outs[1:]:
        o.ws = ws
    cap = outs[0].cap
    kept_tokens = sum(int(min(w.budget, n)) if w.budget >= 0 else binding.tp_budget(int(n), w.keep_ratio)
                      for n in w.doc_lens) * w.n_heads_kv

    def step():
        # the whole stack in one call: one workspace reset, each layer's first
        # kernel a programmatic dependent of the previous layer's last
        binding.tp_compress_layers(p, layers, w.keep_ratio, w.budget, outs, ws, stream)

    def step_layers():
        for (q, k, v), o in zip(layers, outs):
            binding.compress(p, q, k, v, w.keep_ratio, w.budget, o, stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    st = binding.tp_check_status(ws)
    if st != 0:
        raise RuntimeError(f"device status after warm-up: {binding.tp_status_string(st)}")

    # ---- timed region (fused path)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        # the sampler's start-up pause lets the GPU idle: warm it up again, at
        # least W steps and 50 ms of work, so a short timed region does not
        # start on lowered clocks
        t_warm = time.perf_counter() + 0.05
        n_warm = 0
        while n_warm < args.warmup or time.perf_counter() < t_warm:
            step()
            torch.cuda.synchronize()
            n_warm += 1
        replicas.barrier()
        torch.cuda.synchronize()
        clocks.mark_start()
        ev0.record(stream)
        for _ in range(args.steps):
            step()
        ev1.record(stream)
        torch.cuda.synchronize()
        clocks.mark_end()
    replicas.barrier()
    ms = replicas.max_over_ranks(ev0.elapsed_time(ev1) / args.steps, dev)
    value = replicas.whole_job_value(w.n_total, L, world, ms)
    kernels_per_call = binding.tp_compress_kernel_count(p, w.keep_ratio, w.budget, binding.MODE_TWO_PASS)
    gpu_launches = kernels_per_call * L * args.steps

    # ---- staged pass: per-kernel CUDA-event times of the same launches
    rows = w.rows
    stage_ms = staged_times(binding, torch, p, w, layers, outs, ws, stream, args.steps)

    # ---- the same stack as one tp_compress_layer call per layer, and the
    # one-call stack captured into a CUDA graph and replayed
    for _ in range(args.warmup):
        step_layers()
    ev0.record(stream)
    for _ in range(args.steps):
        step_layers()
    ev1.record(stream)
    torch.cuda.synchronize()
    ms_layers = ev0.elapsed_time(ev1) / args.steps
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        binding.tp_compress_layers(p, layers, w.keep_ratio, w.budget, outs, ws)
    for _ in range(args.warmup):
        graph.replay()
    ev0.record(stream)
    for _ in range(args.steps):
        graph.replay()
    ev1.record(stream)
    torch.cuda.synchronize()
    ms_graph = ev0.elapsed_time(ev1) / args.steps
    del graph
    per_layer_calls = {"value": w.n_total * L * world / (ms_layers / 1e3), "unit": UNIT,
                       "ms_per_step": ms_layers, "path": "one tp_compress_layer call per layer"}
    graph_replay = {"value": w.n_total * L * world / (ms_graph / 1e3), "unit": UNIT,
                    "ms_per_step": ms_graph, "path": "the tp_compress_layers call captured as a CUDA graph"}

    # ---- the single-pass variant: row normalisers supplied by the caller
    # (tp_compress_layer_lse), computed once per layer outside the timed region
    lses = []
    for (q, k, v) in layers:
        t = torch.empty((w.batch, w.n_heads_kv, rows), dtype=torch.float32, device=dev)
        binding.tp_guide_lse(p, q, k, t, ws, stream)
        lses.append(t)

    def step_lse():
        # the whole stack in one call: per layer one kernel for the key scores
        # and the V scales (K and V read once), the selection, the compaction
        binding.tp_compress_layers_lse(p, layers, lses, w.keep_ratio, w.budget, outs, ws, stream)

    for _ in range(args.warmup):
        step_lse()
    ev0.record(stream)
    for _ in range(args.steps):
        step_lse()
    ev1.record(stream)
    torch.cuda.synchronize()
    ms_lse = ev0.elapsed_time(ev1) / args.steps
    lse_given = {"value": w.n_total * L * world / (ms_lse / 1e3), "unit": UNIT,
                 "ms_per_step": ms_lse,
                 "hbm_fused": hbm_fused_of(w, kept_tokens, ms_lse / L / 1e3, hbm_peak, peak_src),
                 "kernels_per_layer": binding.tp_compress_kernel_count(p, w.keep_ratio, w.budget,
                                                                       binding.MODE_CALLER_LSE),
                 "path": "tp_compress_layers_lse: caller row normalisers; per layer one kernel reads K "
                         "and V once for the key scores and the Eq. 2 scales (CTA pairs above 256 "
                         "guide rows), then the selection and the compaction"}
    del lses

    # ---- the literal normaliser: guide keys given (tp_compress_layer_guide)
    kgs = [synth.make_guide_keys_torch(wr, l, dev) for l in range(L)]

    def step_literal():
        for (q, k, v), o, kg in zip(layers, outs, kgs):
            binding.compress(p, q, k, v, w.keep_ratio, w.budget, o, stream, k_guide=kg)

    for _ in range(args.warmup):
        step_literal()
    ev0.record(stream)
    for _ in range(args.steps):
        step_literal()
    ev1.record(stream)
    torch.cuda.synchronize()
    ms_lit = ev0.elapsed_time(ev1) / args.steps
    literal = {"value": w.n_total * L * world / (ms_lit / 1e3), "unit": UNIT, "ms_per_step": ms_lit,
               "hbm_fused": hbm_fused_of(w, kept_tokens, ms_lit / L / 1e3, hbm_peak, peak_src),
               "path": "tp_compress_layer_guide: guide prefix folded into the normalisers"}
    del kgs

    read_b, write_b, flops1 = layer_algorithmic(w, kept_tokens)
    dom = max(("lse+vscale", "keyscore"), key=lambda s: stage_ms[s])
    dom_ms = stage_ms[dom]
    achieved = flops1 / (dom_ms / 1e3) / 1e12
    kname = {"lse+vscale": "tp_lse_kernel", "keyscore": "tp_keyscore_kernel"}[dom]
    # the staged times are single launches timed alone: the burst tensor peak applies
    roofline = {"bound": "tensor", "kernel": kname, "achieved": achieved,
                "peak": tf_burst, "unit": "TFLOP/s", "frac": achieved / tf_burst,
                "peak_source": f"{peak_src} bf16 burst (the kernel is timed alone, per launch)",
                "frac_of_sustained": achieved / tf_sust,
                "traffic": traffic_record(kname, w.name),
                "per_launch_ms": dom_ms,
                "flops_per_launch": flops1}
    t_layer_s = ms / L / 1e3
    # every kernel of the layer against its own bound: the scoring passes
    # against the burst tensor peak (one QK^T each; pass 1 also streams V),
    # the compaction against HBM (kept rows of K and V read, the cache written)
    d = w.head_dim
    gather_bytes = kept_tokens * (2 * 2 * d + 2 * 2 * d + d + 4 + 4)
    kernels = {
        "tp_lse_kernel": {"ms": stage_ms["lse+vscale"], "bound": "tensor",
                          "frac": flops1 / (stage_ms["lse+vscale"] / 1e3) / 1e12 / tf_burst,
                          "hbm_frac": 4 * d * w.n_total * w.n_heads_kv / (stage_ms["lse+vscale"] / 1e3) / 1e9 / hbm_peak},
        "tp_keyscore_kernel": {"ms": stage_ms["keyscore"], "bound": "tensor",
                               "frac": flops1 / (stage_ms["keyscore"] / 1e3) / 1e12 / tf_burst},
        "keyscore_with_scales": {
            "ms": stage_ms["keyscore+vscale"], "bound": "tensor",
            "kernel": "tp_keyscore_pair_kernel" if w.rows > 256 else "tp_keyscore_kernel with V",
            "frac": flops1 / (stage_ms["keyscore+vscale"] / 1e3) / 1e12 / tf_burst,
            "hbm_frac": 4 * d * w.n_total * w.n_heads_kv / (stage_ms["keyscore+vscale"] / 1e3) / 1e9 / hbm_peak,
            "note": "the scoring kernel of the caller-normaliser path: one QK^T, the Eq. 2 scales, "
                    "K and V read once"},
        "tp_select_kernel": {"ms": stage_ms["select"], "bound": "latency"},
        "tp_gather_kernel": {"ms": stage_ms["gather"], "bound": "hbm", "bytes_touched": gather_bytes,
                             "touched_frac": gather_bytes / (stage_ms["gather"] / 1e3) / 1e9 / hbm_peak,
                             "note": "bytes the kernel reads and writes (kept K and V rows, the cache); "
                                     "part of the writes is absorbed by L2 and reaches DRAM after the "
                                     "kernel, so this is a throughput of bytes touched, not DRAM bandwidth"},
    }
    lse_given["scoring_kernel"] = kernels["keyscore_with_scales"]
    fused_tail_ms = ms / L - stage_ms["lse+vscale"] - stage_ms["keyscore"]
    hbm_fused = hbm_fused_of(w, kept_tokens, t_layer_s, hbm_peak, peak_src)

    # ---- e2e: host buffers through the public API, copies inside the timed region
    Le = max(1, min(args.e2e_layers, L))
    hq = [tuple(t.cpu().pin_memory() for t in layers[l]) for l in range(Le)]
    dq = [tuple(torch.empty_like(t) for t in layers[l]) for l in range(Le)]
    host_out = [(torch.empty(o.idx.shape, dtype=o.idx.dtype, pin_memory=True),
                 torch.empty(o.kc.shape, dtype=o.kc.dtype, pin_memory=True),
                 torch.empty(o.vc.shape, dtype=o.vc.dtype, pin_memory=True),
                 torch.empty(o.vqc.shape, dtype=o.vqc.dtype, pin_memory=True),
                 torch.empty(o.gammac.shape, dtype=o.gammac.dtype, pin_memory=True))
                for o in outs[:Le]]
    h2d = sum(t.numel() * t.element_size() for l in range(Le) for t in hq[l])
    d2h = sum(t.numel() * t.element_size() for l in range(Le) for t in host_out[l])

    # Three streams: uploads, compression, downloads.  Layer l's upload waits
    # for the previous compression that read its device buffers, layer l's
    # compression waits for its upload and for the previous download of its
    # outputs, and its download waits for its compression.
    s_up, s_down = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    ev_up = [torch.cuda.Event() for _ in range(Le)]
    ev_done = [torch.cuda.Event() for _ in range(Le)]
    ev_down = [torch.cuda.Event() for _ in range(Le)]
    for l in range(Le):  # every event starts recorded
        ev_done[l].record(stream)
        ev_down[l].record(stream)

    def e2e_step():
        for l in range(Le):
            s_up.wait_event(ev_done[l])
            with torch.cuda.stream(s_up):
                for dst, src in zip(dq[l], hq[l]):
                    dst.copy_(src, non_blocking=True)
            ev_up[l].record(s_up)
            stream.wait_event(ev_up[l])
            stream.wait_event(ev_down[l])
            o = outs[l]
            binding.compress(p, *dq[l], w.keep_ratio, w.budget, o, stream)
            ev_done[l].record(stream)
            s_down.wait_event(ev_done[l])
            with torch.cuda.stream(s_down):
                for dst, src in zip(host_out[l], (o.idx, o.kc, o.vc, o.vqc, o.gammac)):
                    dst.copy_(src, non_blocking=True)
            ev_down[l].record(s_down)

    for _ in range(2):
        e2e_step()
    torch.cuda.synchronize()
    replicas.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    s_up.wait_event(e0)
    s_down.wait_event(e0)
    esteps = max(1, args.steps)
    for _ in range(esteps):
        e2e_step()
    for l in range(Le):  # the timed region ends when every download has landed
        stream.wait_event(ev_down[l])
    e1.record(stream)
    torch.cuda.synchronize()
    ems = replicas.max_over_ranks(e0.elapsed_time(e1) / esteps, dev)
    e2e = {"value": replicas.whole_job_value(w.n_total, Le, world, ems), "unit": UNIT,
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "layers_per_step": Le,
           "ms_per_step": ems}

    clk = clocks.summary()
    st = binding.tp_check_status(ws)
    if st != 0:
        raise RuntimeError(f"device status after timing: {binding.tp_status_string(st)}")

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        sample = OracleSample(w)
        try:
            cv, detail = sample.run()
        finally:
            sample.close()
        cpu = {"value": cv, "unit": UNIT, "cores": sample.cores, "cpu_model": cpu_model(),
               "kind": "oracle", "sample": detail}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name, "layers": L, "n_ctx": w.n_total, "guide_len": w.guide_len,
                       "heads_q": w.n_heads_q, "heads_kv": w.n_heads_kv, "head_dim": w.head_dim,
                       "keep_ratio": w.keep_ratio if w.budget < 0 else None,
                       "budget": w.budget if w.budget >= 0 else None,
                       "l2": "inputs larger than L2 (each layer's K+V exceeds 129 MB; layers use distinct buffers)",
                       "parallelism": f"replicas{world}"},
            "roofline": roofline, "hbm_fused": hbm_fused, "stages_ms": stage_ms, "kernels": kernels,
            "fused_layer_ms": ms / L, "kernels_per_layer": kernels_per_call,
            "layer_minus_scoring_passes_ms": fused_tail_ms,
            "workload_legs": legs,
            "e2e": e2e, "gpu_launches": gpu_launches, "clocks": clk, "per_layer_calls": per_layer_calls,
            "graph_replay": graph_replay, "lse_given": lse_given,
            "literal_normaliser": literal,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    from paper_2608_03276_gb300 import synth
    w = synth.WORKLOADS[args.config]
    if args.layers > 0:
        w = w.with_(layers=args.layers)
    if args.impl == "reference":
        run_reference(args, w)
    else:
        run_ours(args, w)


if __name__ == "__main__":
    main()
