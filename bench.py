#!/usr/bin/env python
"""Throughput of the SparseCoder hot path on GB300: kept tokens per second of the
12-layer pruned sparse-attention stack at L = 4096 (and its roofline fraction).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]
                    [--workload cfg4|cfg2|cfg3|cfg5_L512|...|cfg5_L4096[_theta0]
                                |abs_theta|top_ratio|window_w16|...|window_w512
                                |encoder_cfg2]

Besides the default, the workloads cover the other keep rules (abs_theta: the
absolute per-layer thresholds 0.01 l / 12 of RQ4; top_ratio: a kept ratio per
layer, 0.95 -> 0.8) and the window-size ablation of RQ3 (window_wNN: sparse
attention alone, nothing pruned, L = 1024, B = 8); encoder_cfg2 times 12 whole
encoder layers around the path (projections, attention with pruning, layer
norms, feed-forward on the kept tokens; random-init weights) on the config-2
shape.  Each prints its own line.

One step = one call of sc_stack_forward over the whole workload: padding removal,
then per layer the rows kernel (band + global attention, O, row LSE) and the
cols kernel (column scores, threshold, compaction), 12 layers, inputs resident in
HBM.  The default workload is the 12-layer stack B=2, L=4096, H=12, d=64, window
+-256, token 0 plus 8 seeded global positions, 5% salient keys x4, alpha 0.4->1.0.
The inputs of one step (453 MB of Q/K/V) are larger than the 129 MB L2, so no
flush is needed between steps.

e2e: the same metric through sc_stack_forward_host, the call that takes the
inputs and results in page-locked host memory: each step the kernels read the
rows each layer uses over the host link and write the defined result slots back
(replayed as a CUDA graph, like the device-resident steps).

Metric: kept tokens/s = sum over layers and sequences of the tokens entering the
layer (token-layers processed) / stack time.  Under torchrun each rank runs an
independent replica (weak scaling, no collective on the data path); value is the
sum over ranks divided by the slowest rank's time.

--impl reference times the fp64 CPU oracle (the only reference this method has)
on the host cores, each step a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads as wk  # noqa: E402

METRIC = "kept-tokens/sec per 12-layer pruned stack at L=4096; fraction of roofline"


def metric_name(wl: wk.Workload) -> str:
    """The metric's name for a workload (the default's is METRIC)."""
    return "kept-tokens/sec per %d-layer pruned stack at L=%d; fraction of roofline" % (
        wl.n_layers, wl.L)
UNIT = "kept-tokens/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
BYTES_PER_TOKEN = 6152      # Q,K,V read (3*12*64*2) + O write (12*64*2) + score (4) + position (4)
FLOPS_PER_PAIR = 4 * 64 * 12  # QK^T and PV, multiply-add = 2 flops, 12 heads


def pick_workload(name: str) -> wk.Workload:
    if name in wk.CONFIGS:
        return wk.CONFIGS[name]
    if name.startswith("cfg5_L"):
        rest = name[len("cfg5_L"):]
        control = rest.endswith("_theta0")
        return wk.cfg5(int(rest.replace("_theta0", "")), control=control)
    if name == "encoder_cfg2":
        return wk.ENCODER_CFG2
    if name == "abs_theta":
        return wk.ABS_THETA
    if name == "top_ratio":
        return wk.TOP_RATIO
    if name.startswith("window_w"):
        return wk.window_sweep(int(name[len("window_w"):]))
    raise SystemExit("unknown workload %s" % name)


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"


# ---------------------------------------------------------------------------
# algorithmic work of one (sequence, layer)
# ---------------------------------------------------------------------------
def nnz_allowed(n: int, w: int, gcur) -> int:
    """Number of (query, key) pairs in the allowed sets of n current tokens."""
    if n == 0:
        return 0
    i = np.arange(n)
    band = np.minimum(n - 1, i + w) - np.maximum(0, i - w) + 1
    isg = np.zeros(n, bool)
    isg[list(gcur)] = True
    total = int(band[~isg].sum())
    for g in gcur:  # global keys outside the band of non-global rows
        far = (~isg) & (np.abs(i - g) > w)
        total += int(far.sum())
    total += int(isg.sum()) * n  # global rows see every key
    return total


def layer_work(wl, inp, pos, lens):
    """[n_layers] lists of (bytes, flops) summed over the batch, from the kept sets."""
    gset = set(int(g) for g in inp["global_pos"])
    out = []
    for l in range(wl.n_layers):
        B_, F_ = 0, 0
        for b in range(wl.B):
            n = int(lens[l, b])
            gcur = [c for c in range(n) if int(pos[l, b, c]) in gset]
            B_ += BYTES_PER_TOKEN * n
            F_ += FLOPS_PER_PAIR * nnz_allowed(n, wl.w, gcur)
        out.append((B_, F_))
    return out


def kernel_source_hash() -> str:
    """sha256 over the CUDA sources and the C header (each file's name, then its bytes)."""
    import glob
    import hashlib
    files = sorted(glob.glob(os.path.join(ROOT, "paper_2310_07109_gb300", "csrc", "*.cu")) +
                   glob.glob(os.path.join(ROOT, "paper_2310_07109_gb300", "csrc", "*.cuh")))
    files.append(os.path.join(ROOT, "include", "sparsecoder.h"))
    h = hashlib.sha256()
    for f in files:
        h.update(os.path.basename(f).encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def host_link_bytes(lens, n_layers, H, d, mask_bytes):
    """Bytes one sc_stack_forward_host call moves over the host link, from the
    lengths it produced (lens [n_layers + 1][B]): host to device, the Q, K, V
    rows of the tokens entering each layer and the padding mask; device to host,
    those tokens' O rows and scores, pos[l][b][:len] for every l <= n_layers,
    and len itself."""
    lens = np.asarray(lens, dtype=np.int64)
    row_bytes = H * d * 2
    in_rows = int(lens[:n_layers].sum())
    h2d = 3 * row_bytes * in_rows + int(mask_bytes)
    d2h = (row_bytes + 4) * in_rows + 4 * int(lens.sum()) + 4 * lens.size
    return h2d, d2h


def measured_traffic(kernels):
    """DRAM bytes (read + write) of one launch of each kernel, summed, from the ncu
    capture recorded in profiles/traffic.json; None once any kernel source has
    changed since that capture."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None, "no recorded capture"
    if rec.get("source_sha256") != kernel_source_hash():
        return None, "kernels changed since the recorded capture"
    try:
        total = sum(rec["kernels"][k]["dram_read_bytes"] + rec["kernels"][k]["dram_write_bytes"]
                    for k in kernels)
    except KeyError:
        return None, "kernel not in the recorded capture"
    return int(total), "ncu dram__bytes_read.sum + dram__bytes_write.sum, profiles/traffic.json"


# ---------------------------------------------------------------------------
# multi-rank aggregation (replicas: no collective on the data path)
# ---------------------------------------------------------------------------
def max_over_ranks(value: float, device=None) -> float:
    """The slowest rank's time: all-reduce MAX (a no-op without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world: int, units_per_step_per_rank: int, ms_per_step: float) -> float:
    """Units processed by all ranks per second, timed by the slowest rank."""
    return world * units_per_step_per_rank / (ms_per_step * 1e-3)


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class _Nvml:
    """Minimal NVML through ctypes (the library ships with the driver): SM clock,
    its maximum, and the clock event reason bits.  Read-only."""
    SM = 1                      # NVML_CLOCK_SM
    BITS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
            0x40: "hw_thermal_slowdown"}

    def __init__(self, uuid, index):
        import ctypes
        self.c = ctypes
        self.lib = ctypes.CDLL("libnvidia-ml.so.1")
        if self.lib.nvmlInit_v2() != 0:
            raise OSError("nvmlInit failed")
        self.h = ctypes.c_void_p()
        rc = 1
        if uuid:
            rc = self.lib.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(self.h))
        if rc != 0:
            rc = self.lib.nvmlDeviceGetHandleByIndex_v2(index, ctypes.byref(self.h))
        if rc != 0:
            raise OSError("no NVML handle for the device")
        fn = getattr(self.lib, "nvmlDeviceGetCurrentClocksEventReasons", None)
        self.reasons_fn = fn or self.lib.nvmlDeviceGetCurrentClocksThrottleReasons

    def clock(self, max_clock=False):
        v = self.c.c_uint()
        f = self.lib.nvmlDeviceGetMaxClockInfo if max_clock else self.lib.nvmlDeviceGetClockInfo
        return v.value if f(self.h, self.SM, self.c.byref(v)) == 0 else None

    def reasons(self):
        v = self.c.c_ulonglong()
        if self.reasons_fn(self.h, self.c.byref(v)) != 0:
            return []
        return [nm for bit, nm in self.BITS.items() if v.value & bit]

    def close(self):
        self.lib.nvmlShutdown()


class ClockSampler:
    """SM clock and throttle reasons sampled every ~1 ms by a thread while the
    timed region runs (NVML; nvidia-smi at 200 ms when NVML is unavailable).
    ``mark_start()`` / ``mark_end()`` bound the samples that count."""
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.samples = []           # (host time, sm MHz, reasons)
        self.max_mhz = None
        self.t_lo = self.t_hi = None
        self.source = None
        self._stop = threading.Event()
        self.proc = None

    def __enter__(self):
        import torch
        uuid = None
        try:
            u = str(torch.cuda.get_device_properties(self.index).uuid)
            uuid = u if u.startswith("GPU-") else "GPU-" + u
        except Exception:
            pass
        try:
            self.nvml = _Nvml(uuid, self.index)
            self.max_mhz = self.nvml.clock(max_clock=True)
            self.source = "nvml"
            self.thread = threading.Thread(target=self._poll, daemon=True)
        except (OSError, AttributeError):
            self.nvml = None
            try:
                self.proc = subprocess.Popen(
                    ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.QUERY,
                     "--format=csv,noheader,nounits", "-lms", "200"],
                    stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
                self.source = "nvidia-smi"
                self.thread = threading.Thread(target=self._read, daemon=True)
            except OSError:
                self.thread = None
        if self.thread is not None:
            self.thread.start()
        return self

    def _poll(self):
        while not self._stop.is_set():
            self.samples.append((time.perf_counter(), self.nvml.clock(), self.nvml.reasons()))
            time.sleep(0.001)

    def _read(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.strip().split(",")]
            if len(parts) < 9:
                continue
            try:
                sm = float(parts[1])
                self.max_mhz = float(parts[2])
            except ValueError:
                continue
            rs = [nm for nm, v in zip(names, parts[5:9]) if v.lower().startswith("active")]
            self.samples.append((time.perf_counter(), sm, rs))

    def mark_start(self):
        self.t_lo = time.perf_counter()

    def mark_end(self):
        self.t_hi = time.perf_counter()

    def __exit__(self, *exc):
        self._stop.set()
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=2)
        if self.nvml is not None:
            self.nvml.close()

    def summary(self):
        lo = self.t_lo if self.t_lo is not None else -1e30
        hi = self.t_hi if self.t_hi is not None else 1e30
        inside = [(sm, rs) for t, sm, rs in self.samples if lo <= t <= hi and sm is not None]
        reasons = sorted({r for _, rs in inside for r in rs})
        sm = [x for x, _ in inside]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": self.max_mhz,
                "reasons": reasons, "samples": len(sm), "source": self.source}


# ---------------------------------------------------------------------------
# CPU oracle (the reference arm and the cpu_baseline)
# ---------------------------------------------------------------------------
def oracle_sample(wl, inp, b, n_layers, threads):
    """Run the oracle stack on sequence b for the first n_layers layers; returns
    (seconds, kept tokens processed, threads used)."""
    import oracle
    sl = slice(b, b + 1)
    mask = None if inp["pad_mask"] is None else inp["pad_mask"][sl]
    Q, K, V = (np.ascontiguousarray(inp[k][:n_layers, sl]) for k in ("Q", "K", "V"))
    t0 = time.perf_counter()
    res = oracle.stack(Q, K, V, mask, inp["global_pos"], wl.w, inp["alpha"][:n_layers],
                       want_O=True, nthreads=threads, keep_rule=wl.keep_rule)
    dt = time.perf_counter() - t0
    return dt, int(res["len"][:n_layers].sum()), min(threads, wl.H), res


def oracle_check(wl, inp, out, res0, n_seq):
    """The benched run's results against the fp64 oracle on the first ``n_seq``
    sequences (all layers): lengths and kept positions exactly, the largest O
    and score errors.  ``res0``: the oracle's sequence-0 stack, already run."""
    import oracle
    lens = out["len"].cpu().numpy()
    pos = out["pos"].cpu().numpy()
    scores = out["scores"].cpu().numpy()
    kept_equal, o_err, s_err, checked = True, 0.0, 0.0, 0
    for b in range(min(n_seq, wl.B)):
        if b == 0:
            res = res0
        else:
            sl = slice(b, b + 1)
            mask = None if inp["pad_mask"] is None else inp["pad_mask"][sl]
            res = oracle.stack(*(np.ascontiguousarray(inp[k][:, sl]) for k in ("Q", "K", "V")),
                               mask, inp["global_pos"], wl.w, inp["alpha"],
                               keep_rule=wl.keep_rule)
        checked += 1
        for l in range(wl.n_layers + 1):
            n = int(res["len"][l, 0])
            if int(lens[l, b]) != n or not np.array_equal(pos[l, b, :n], res["pos"][l, 0, :n]):
                kept_equal = False
        for l in range(wl.n_layers):
            n = int(min(res["len"][l, 0], lens[l, b]))
            if n == 0:
                continue
            o = out["O"][l, b, :n].float().cpu().numpy().astype(np.float64)
            o_err = max(o_err, float(np.abs(o - res["O"][l, 0, :n]).max()))
            s_err = max(s_err, float(np.abs(scores[l, b, :n] - res["scores"][l, 0, :n]).max()))
    return {"sequences": checked, "layers": wl.n_layers, "kept_lists_equal": kept_equal,
            "o_max_abs": o_err, "score_max_abs": s_err, "o_bar": 2e-2, "score_bar": 1e-5}


def run_reference(args, wl):
    import oracle
    oracle.build()
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    inp = wk.make_inputs(wl, wk.stored_redraws(wl))
    threads = oracle.default_threads()
    layers = wl.n_layers if args.ref_layers <= 0 else max(1, min(wl.n_layers, args.ref_layers))
    for s in range(args.warmup):
        oracle_sample(wl, inp, s % wl.B, layers, threads)
    tot_t, tot_tok, cores = 0.0, 0, 1
    for s in range(args.steps):
        dt, tok, cores, _ = oracle_sample(wl, inp, s % wl.B, layers, threads)
        tot_t += dt
        tot_tok += tok
    value = tot_tok / tot_t
    sample = "one sequence of the workload, first %d layer(s), per step" % layers
    line = {"impl": "reference", "metric": metric_name(wl), "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * tot_t / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": wl.describe(), "sample": sample},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# native arm
# ---------------------------------------------------------------------------
def run_native(args, wl):
    import torch
    import torch.distributed as dist

    from paper_2310_07109_gb300 import binding as sc
    from paper_2310_07109_gb300 import build as sc_build

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    sc_build.build_library()
    sc.load()
    sc.select_rows_kernel(sc.SC_ROWS_SINGLE_PASS if args.rows_kernel == "single-pass"
                          else sc.SC_ROWS_TWO_PASS)

    redraws = wk.stored_redraws(wl)
    inp = wk.make_inputs(wl, redraws)
    host = {k: torch.from_numpy(inp[k].view(np.int16)).view(torch.bfloat16).pin_memory()
            for k in ("Q", "K", "V")}
    dQKV = {k: host[k].to(dev) for k in host}
    # Timed steps rotate over copies of the inputs (and of the outputs), so that
    # what one step touches is no longer in L2 when the same copy comes round
    # again: the copies together touch more than three times the L2 size.
    l2_bytes = torch.cuda.get_device_properties(dev).L2_cache_size
    lay0 = 3 * inp["Q"][0].nbytes + inp["Q"][0].nbytes // 3   # layer 0's Q, K, V read + O written
    n_copies = 1 if args.warm_l2 else max(3, -(-3 * l2_bytes // lay0))
    copies = [dQKV] + [{k: t.clone() for k, t in dQKV.items()} for _ in range(n_copies - 1)]
    mask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).to(dev)
    ws = sc.new_workspace(wl.B, wl.L, wl.H, dev)
    alpha = [float(a) for a in inp["alpha"]]
    gpos = [int(g) for g in inp["global_pos"]]

    outs = [None] * n_copies

    def step(events=None, c=0):
        outs[c] = sc.stack_forward(copies[c]["Q"], copies[c]["K"], copies[c]["V"], mask, gpos,
                                   wl.w, alpha, out=outs[c], workspace=ws, events=events,
                                   keep_rule=wl.keep_rule, plain_launches=args.plain_launches)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(max(3, args.warmup)):
        for c in range(n_copies):
            step(c=c)
    rc = sc.workspace_status(ws)
    if rc != 0:
        raise SystemExit("device status after warm-up: %s" % sc.status_string(rc))

    # one step captured as a CUDA graph (the library's launches, descriptors
    # encoded at capture time), replayed for the timed steps
    graphs = []
    if not args.no_graph:
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            for c in range(n_copies):
                step(c=c)
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=side):
                    step(c=c)
                graphs.append(g)
        torch.cuda.current_stream().wait_stream(side)
        for _ in range(max(3, args.warmup)):
            for g in graphs:
                g.replay()
        torch.cuda.synchronize()
    graph = graphs[0] if graphs else None

    def run_steps(k, rotate=True):
        for s_ in range(k):
            c = s_ % n_copies if rotate else 0
            if graphs:
                graphs[c].replay()
            else:
                step(c=c)

    # ---- timed region: K steps, inputs resident, rotating over the copies
    stream = torch.cuda.current_stream()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device()) as clocks:
        time.sleep(0.01)
        barrier()
        clocks.mark_start()
        t0.record(stream)
        run_steps(args.steps)
        t1.record(stream)
        barrier()
        clocks.mark_end()
    rc = sc.workspace_status(ws)
    if rc != 0:
        raise SystemExit("device status after the timed steps: %s" % sc.status_string(rc))
    ms = max_over_ranks(t0.elapsed_time(t1), dev)
    ms_per_step = ms / args.steps
    # the same steps on one copy only (its inputs stay in L2 between steps)
    barrier()
    t0.record(stream)
    run_steps(args.steps, rotate=False)
    t1.record(stream)
    barrier()
    warm_ms_per_step = max_over_ranks(t0.elapsed_time(t1), dev) / args.steps
    out = outs[0]
    for c in range(1, n_copies):
        if not torch.equal(outs[c]["len"], out["len"]):
            raise SystemExit("copies of the same inputs gave different lengths")
    lens = out["len"].cpu().numpy()
    pos = out["pos"].cpu().numpy()
    kept_per_step = int(lens[:wl.n_layers].sum())
    value = whole_job_rate(world, kept_per_step, ms_per_step)

    # ---- kernels launched per timed step.  A captured step, and an eager call
    # (which the library records into a graph of its own), runs the per-layer
    # kernels in a device-driven loop: prep, [padding gather], rows + cols +
    # gather + advance for each layer that some sequence still runs per layer
    # (more than TAIL_MAX_LEN tokens), then the cluster kernel.  With plain
    # launches: the library's plan.
    eager_launches = sc.stack_launch_count(wl.n_layers, wl.B, wl.L, wl.H, wl.w, gpos,
                                           inp["pad_mask"] is not None)
    looped = sum(1 for l in range(wl.n_layers) if (lens[l] > sc.TAIL_MAX_LEN).any())
    graph_launches = (1 + (1 if inp["pad_mask"] is not None else 0) + 4 * looped + 1
                      if wl.L > sc.TAIL_MAX_LEN else 2)
    launches_per_step = (eager_launches if graph is None and args.plain_launches
                         else graph_launches)

    # ---- per-kernel times on the launching stream (same steps, events between kernels)
    nev = 3 + 3 * wl.n_layers
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(nev)]
    for e in evs:
        e.record(stream)
    torch.cuda.synchronize()
    rows_ms = np.zeros(wl.n_layers)
    cols_ms = np.zeros(wl.n_layers)
    gath_ms = np.zeros(wl.n_layers)
    prep_ms = 0.0
    tail_ms = 0.0
    prof_steps = max(1, min(args.steps, 20))
    for _ in range(prof_steps):
        step(evs)
        torch.cuda.synchronize()
        prep_ms += evs[0].elapsed_time(evs[1])
        for l in range(wl.n_layers):
            rows_ms[l] += evs[1 + 3 * l].elapsed_time(evs[2 + 3 * l])
            cols_ms[l] += evs[2 + 3 * l].elapsed_time(evs[3 + 3 * l])
            gath_ms[l] += evs[3 + 3 * l].elapsed_time(evs[4 + 3 * l])
        tail_ms += evs[1 + 3 * wl.n_layers].elapsed_time(evs[2 + 3 * wl.n_layers])
    rows_ms /= prof_steps
    tail_ms /= prof_steps
    cols_ms /= prof_steps
    gath_ms /= prof_steps
    prep_ms /= prof_steps
    # layer 0's rows and cols kernels as one unit, chained as in an
    # uninstrumented step (no event between them: the cols CTAs of the heads
    # whose rows are done run beside the rows kernel's last CTAs)
    pair_ev = [None] * nev
    pair_ev[1] = torch.cuda.Event(enable_timing=True)
    pair_ev[3] = torch.cuda.Event(enable_timing=True)
    for e in (pair_ev[1], pair_ev[3]):   # torch times only events it has seen recorded
        e.record(stream)
    torch.cuda.synchronize()
    pair_ms = 0.0
    for _ in range(prof_steps):
        step(pair_ev)
        torch.cuda.synchronize()
        pair_ms += pair_ev[1].elapsed_time(pair_ev[3])
    pair_ms /= prof_steps

    peaks, peak_src = load_peaks()
    work = layer_work(wl, inp, pos, lens)
    bw = peaks["hbm_gbs"] * 1e9
    fl = peaks["bf16_tflops"] * 1e12
    # the whole stack: every layer's roofline time over the attention kernels' time
    t_roof = sum(max(Bb / bw, Ff / fl) for Bb, Ff in work)
    t_meas = (float((rows_ms + cols_ms).sum()) + tail_ms) * 1e-3
    # the dominant unit: the per-layer kernel pair of the full-length layer 0
    # (rows + cols, one launch each); when every sequence starts in the cluster
    # kernel, that kernel over all layers
    t_l0 = pair_ms * 1e-3
    if rows_ms[0] + cols_ms[0] > 1e-6:
        unit_bytes, unit_flops, unit_t = work[0][0], work[0][1], t_l0
        unit_kernels = ["sc_rows_kernel", "sc_cols_kernel"]
        unit_desc = ("sc_rows_kernel + sc_cols_kernel of layer 0 (one launch each, chained "
                     "as in the timed step; B=%d sequences of %d tokens)"
                     % (wl.B, int(lens[0].max())))
    else:
        unit_bytes = sum(Bb for Bb, _ in work)
        unit_flops = sum(Ff for _, Ff in work)
        unit_t = tail_ms * 1e-3
        unit_kernels = ["sc_tail_kernel"]
        unit_desc = "sc_tail_kernel (one launch: every layer of every sequence)"
    hbm_bound = unit_bytes / bw >= unit_flops / fl
    traffic, traffic_note = measured_traffic(unit_kernels)
    roofline = {
        "bound": "hbm" if hbm_bound else "tensor",
        "achieved": unit_bytes / unit_t / 1e9 if hbm_bound else unit_flops / unit_t / 1e12,
        "peak": peaks["hbm_gbs"] if hbm_bound else peaks["bf16_tflops"],
        "unit": "GB/s" if hbm_bound else "TFLOP/s",
        "frac": max(unit_bytes / bw, unit_flops / fl) / unit_t,
        "traffic": traffic,
        "peak_source": peak_src,
        "kernel": unit_desc,
        "algorithmic": {"bytes": int(unit_bytes), "flops": int(unit_flops),
                        "per_unit": "6152 B per token-layer; 3072 flop per allowed (query, "
                                    "key) pair (all heads, QK^T and PV)"},
        "launch_ms": unit_t * 1e3,
        "serialised_ms": (float(rows_ms[0] + cols_ms[0]) if unit_kernels[0] == "sc_rows_kernel"
                          else unit_t * 1e3),
        "traffic_note": traffic_note,
        "stack_frac": t_roof / t_meas,
        "stack_scope": "sum over layers of max(F_l/peak_bf16, B_l/peak_hbm) over the measured "
                       "time of sc_rows_kernel + sc_cols_kernel (per-layer layers) and "
                       "sc_tail_kernel",
        "kernel_ms_per_step": {"sc_rows_kernel": float(rows_ms.sum()),
                               "sc_cols_kernel": float(cols_ms.sum()),
                               "sc_gather_kernel": float(gath_ms.sum()),
                               "sc_prep_kernel": prep_ms,
                               "sc_tail_kernel": tail_ms},
        "rows_ms_per_layer": [round(float(x), 5) for x in rows_ms],
        "cols_ms_per_layer": [round(float(x), 5) for x in cols_ms],
    }

    # ---- end to end through the public host-buffer call (sc_stack_forward_host):
    # page-locked Q/K/V in, page-locked results out.  The kernels read each
    # layer's surviving rows over the host link and write back the current slots
    # of every layer, all inside the timed steps.
    hout = sc.new_host_outputs(wl.n_layers, wl.B, wl.L, wl.H)
    hmask = None if inp["pad_mask"] is None else torch.from_numpy(inp["pad_mask"]).pin_memory()
    hws = sc.new_stack_host_workspace(wl.n_layers, wl.B, wl.L, wl.H, dev)

    def host_step():
        sc.stack_forward_host(host["Q"], host["K"], host["V"], hmask, gpos, wl.w, alpha,
                              out=hout, workspace=hws, keep_rule=wl.keep_rule,
                              plain_launches=args.plain_launches)

    for _ in range(max(3, args.warmup)):
        host_step()
    hgraph = None
    if not args.no_graph:
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            host_step()
            hgraph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(hgraph, stream=side):
                host_step()
        torch.cuda.current_stream().wait_stream(side)
        for _ in range(max(3, args.warmup)):
            hgraph.replay()
    torch.cuda.synchronize()
    barrier()
    t0.record(stream)
    for _ in range(args.steps):
        if hgraph is not None:
            hgraph.replay()
        else:
            host_step()
    t1.record(stream)
    barrier()
    e2e_ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, dev)
    rc = sc.workspace_status(hws)
    if rc != 0:
        raise SystemExit("device status after the end-to-end steps: %s" % sc.status_string(rc))
    if not torch.equal(hout["len"], out["len"].cpu()):
        raise SystemExit("the host-buffer call disagrees with the device call on the lengths")
    h2d, d2h = host_link_bytes(lens, wl.n_layers, wl.H, wl.d,
                               0 if hmask is None else hmask.numel())
    e2e = {"value": whole_job_rate(world, kept_per_step, e2e_ms), "unit": UNIT,
           "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
           "ms_per_step": e2e_ms, "call": "sc_stack_forward_host",
           "cuda_graph": hgraph is not None}

    line = {"metric": metric_name(wl), "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": wl.describe(), "n_layers": wl.n_layers, "batch": wl.B,
                       "seq_len": wl.L, "heads": wl.H, "head_dim": wl.d, "window": wl.w,
                       "globals": len(gpos), "parallelism": "replicas" if world > 1 else "single",
                       "cuda_graph": graph is not None, "rows_kernel": args.rows_kernel,
                       "plain_launches": bool(args.plain_launches),
                       "l2": ("timed steps rotate over %d copies of the inputs and outputs "
                              "(%.0f MB touched by layer 0 per copy, L2 %.0f MB)" % (
                                  n_copies, lay0 / 1e6, l2_bytes / 1e6)) if n_copies > 1 else
                             "one copy of the inputs: L2 warm between steps",
                       "warm_l2_ms_per_step": warm_ms_per_step,
                       "inputs": "near-threshold resampled (%d redrawn rows, stored)" % len(
                           redraws),
                       "kept_tokens_per_step": kept_per_step,
                       "input_tokens_per_step": int(lens[0].sum()),
                       "survival": [round(float(x), 4) for x in
                                    lens[:wl.n_layers + 1].sum(axis=1) / max(1, lens[0].sum())]},
            "roofline": roofline,
            "e2e": e2e,
            "gpu_launches": args.steps * launches_per_step,
            "clocks": clocks.summary()}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        dt, tok, cores, res0 = oracle_sample(wl, inp, 0, wl.n_layers, oracle.default_threads())
        line["cpu_baseline"] = {"value": tok / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
                                "sample": "sequence 0 of the workload, all %d layers (%d kept "
                                          "token-layers, %.1f s)" % (wl.n_layers, tok, dt)}
        line["oracle_check"] = oracle_check(wl, inp, out, res0, args.check_sequences)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ---------------------------------------------------------------------------
# the encoder layer around the path (--workload encoder_cfg2)
# ---------------------------------------------------------------------------
def encoder_oracle_sample(wl, X0, weights, b, threads):
    """The oracle on sequence b for layer 0 of the encoder: (seconds, tokens, cores)."""
    import oracle
    from oracle import encoder as enc
    D = wl.H * wl.d
    w = {k: (wk.bf16_bits_to_f64(v) if k.startswith("W") else v.astype(np.float64))
         for k, v in weights[0].items()}
    x = wk.bf16_bits_to_f64(X0[b])
    t0 = time.perf_counter()
    q, k, v = enc.qkv(x, w["W_qkv"], w["b_qkv"])
    n = x.shape[0]
    gset = set(int(g) for g in wk.global_positions(wl))
    isg = np.array([c in gset for c in range(n)])
    O, s, keep = oracle.layer(q.reshape(n, wl.H, wl.d), k.reshape(n, wl.H, wl.d),
                              v.reshape(n, wl.H, wl.d), isg, wl.w, wl.alphas()[0] / n,
                              nthreads=threads)
    kc = np.nonzero(keep)[0]
    enc.output_and_ffn(x[kc], O.reshape(n, D)[kc], w["W_o"], w["b_o"], w["ln1_gamma"],
                       w["ln1_beta"], w["W_1"], w["b_1"], w["W_2"], w["b_2"], w["ln2_gamma"],
                       w["ln2_beta"])
    return time.perf_counter() - t0, n, min(threads, wl.H)


def run_reference_encoder(args, wl):
    import oracle
    oracle.build()
    if int(os.environ.get("RANK", "0")) != 0:
        return
    D = wl.H * wl.d
    X0 = wk.encoder_input(wl)
    wts = [wk.encoder_weights(D, 0, wl.seed)]
    threads = oracle.default_threads()
    for s in range(args.warmup):
        encoder_oracle_sample(wl, X0, wts, s % wl.B, threads)
    tot_t, tot_tok, cores = 0.0, 0, 1
    for s in range(args.steps):
        dt, tok, cores = encoder_oracle_sample(wl, X0, wts, s % wl.B, threads)
        tot_t += dt
        tot_tok += tok
    value = tot_tok / tot_t
    sample = "one sequence of the workload, encoder layer 0, per step"
    print(json.dumps({"impl": "reference", "metric": "kept-tokens/sec per %d-layer pruned encoder "
                      "at L=%d" % (wl.n_layers, wl.L), "value": value, "unit": UNIT,
                      "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
                      "ms_per_step": 1e3 * tot_t / args.steps, "higher_is_better": True,
                      "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                      "config": {"workload": wl.describe(), "sample": sample},
                      "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores,
                                       "kind": "oracle", "sample": sample},
                      "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                              "d2h_bytes_per_step": 0}}), flush=True)


def run_encoder(args, wl):
    import torch
    import torch.distributed as dist

    from paper_2310_07109_gb300 import binding as sc
    from paper_2310_07109_gb300 import build as sc_build

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    sc_build.build_library()
    sc.load()
    D = wl.H * wl.d
    nl = wl.n_layers
    X0 = wk.encoder_input(wl)
    wts = [wk.encoder_weights(D, l, wl.seed) for l in range(nl)]
    W = [{k: (torch.from_numpy(v.view(np.int16)).to(dev).view(torch.bfloat16) if k.startswith("W")
              else torch.from_numpy(v).to(dev)) for k, v in wl_w.items()} for wl_w in wts]
    hostX = torch.from_numpy(X0.view(np.int16)).view(torch.bfloat16).pin_memory()
    X = hostX.to(dev)
    len0 = torch.full((wl.B,), wl.L, dtype=torch.int32, device=dev)
    pos0 = torch.arange(wl.L, dtype=torch.int32, device=dev).repeat(wl.B, 1)
    gpos = [int(g) for g in wk.global_positions(wl)]
    alpha = [float(a) for a in wl.alphas()]
    ws = sc.new_encoder_workspace(wl.B, wl.L, wl.H, dev)
    outs = [{"Y": torch.empty((wl.B, wl.L, D), dtype=torch.bfloat16, device=dev),
             "O": torch.empty((wl.B, wl.L, D), dtype=torch.bfloat16, device=dev),
             "scores": torch.empty((wl.B, wl.L), dtype=torch.float32, device=dev),
             "pos_out": torch.empty((wl.B, wl.L), dtype=torch.int32, device=dev),
             "len_out": torch.empty((wl.B,), dtype=torch.int32, device=dev)} for _ in range(nl)]

    def step():
        x, ln, ps = X, len0, pos0
        for l in range(nl):
            o = outs[l]
            sc.encoder_layer_forward(x, ln, ps, wl.w, gpos, W[l], alpha[l], keep_rule=wl.keep_rule,
                                     out=o, workspace=ws)
            x, ln, ps = o["Y"], o["len_out"], o["pos_out"]

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(max(3, args.warmup)):
        step()
    rc = sc.workspace_status(ws)
    if rc != 0:
        raise SystemExit("device status after warm-up: %s" % sc.status_string(rc))
    graph = None
    if not args.no_graph:
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            step()
            graph = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph, stream=side):
                step()
        torch.cuda.current_stream().wait_stream(side)
        for _ in range(max(3, args.warmup)):
            graph.replay()
        torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device()) as clocks:
        time.sleep(0.01)
        barrier()
        clocks.mark_start()
        t0.record(stream)
        for _ in range(args.steps):
            if graph is not None:
                graph.replay()
            else:
                step()
        t1.record(stream)
        barrier()
        clocks.mark_end()
    rc = sc.workspace_status(ws)
    if rc != 0:
        raise SystemExit("device status after the timed steps: %s" % sc.status_string(rc))
    ms_per_step = max_over_ranks(t0.elapsed_time(t1), dev) / args.steps
    lens = np.stack([np.full(wl.B, wl.L)] + [o["len_out"].cpu().numpy() for o in outs]).astype(np.int64)
    kept_per_step = int(lens[:nl].sum())
    value = whole_job_rate(world, kept_per_step, ms_per_step)
    # algorithmic work: the GEMMs (Q/K/V on the current tokens, the rest on the
    # kept ones) and the attention's QK^T and PV over the allowed pairs
    pos = np.stack([np.tile(np.arange(wl.L), (wl.B, 1))] +
                   [o["pos_out"].cpu().numpy() for o in outs])
    work = layer_work(wl, {"global_pos": np.asarray(gpos)}, pos, lens)
    gemm_flops = sum(2 * D * D * (3 * int(lens[l].sum()) + 9 * int(lens[l + 1].sum()))
                     for l in range(nl))
    flops = gemm_flops + sum(F for _, F in work)
    peaks, peak_src = load_peaks()
    t = ms_per_step * 1e-3
    roofline = {"bound": "tensor", "achieved": flops / t / 1e12, "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s", "frac": flops / t / 1e12 / peaks["bf16_tflops"], "traffic": None,
                "peak_source": peak_src,
                "kernel": "the whole encoder step (GEMMs, attention, layer norms)",
                "algorithmic": {"flops": int(flops), "gemm_flops": int(gemm_flops),
                                "per_unit": "2 D^2 (3 n + 9 n') per layer (projections on the n "
                                            "current tokens, the rest on the n' kept ones) + "
                                            "3072 flop per allowed pair"}}
    # end to end: layer-0 hidden states in from pinned memory, the last layer's out
    hostY = torch.empty(outs[-1]["Y"].shape, dtype=torch.bfloat16, pin_memory=True)
    e2e_steps = max(1, min(args.steps, 5))
    barrier()
    t0.record(stream)
    for _ in range(e2e_steps):
        X.copy_(hostX, non_blocking=True)
        step()
        hostY.copy_(outs[-1]["Y"], non_blocking=True)
    t1.record(stream)
    barrier()
    e2e_ms = max_over_ranks(t0.elapsed_time(t1) / e2e_steps, dev)
    line = {"metric": "kept-tokens/sec per %d-layer pruned encoder at L=%d" % (nl, wl.L),
            "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic inputs, random-init weights",
            "config": {"workload": wl.describe() + "; encoder layers (D=%d, FFN %d)" % (D, 4 * D),
                       "n_layers": nl, "batch": wl.B, "seq_len": wl.L, "cuda_graph": graph is not None,
                       "kept_tokens_per_step": kept_per_step,
                       "survival": [round(float(x), 4) for x in lens.sum(axis=1) / lens[0].sum()]},
            "roofline": roofline,
            "e2e": {"value": whole_job_rate(world, kept_per_step, e2e_ms), "unit": UNIT,
                    "h2d_bytes_per_step": int(hostX.numel() * 2),
                    "d2h_bytes_per_step": int(hostY.numel() * 2), "ms_per_step": e2e_ms},
            "gpu_launches": args.steps * nl * 10, "clocks": clocks.summary()}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        dt, tok, cores = encoder_oracle_sample(wl, X0, wts, 0, oracle.default_threads())
        line["cpu_baseline"] = {"value": tok / dt, "unit": UNIT, "cores": cores, "kind": "oracle",
                                "sample": "sequence 0, layer 0 (%d tokens, %.1f s)" % (tok, dt)}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["native", "reference"], default="native")
    ap.add_argument("--workload", default="cfg4")
    ap.add_argument("--ref-layers", type=int, default=0,
                    help="layers of one sequence per reference step (0: all, as the "
                         "cpu_baseline sample)")
    ap.add_argument("--no-cpu-baseline", action="store_true",
                    help="skip the oracle legs (CPU baseline and the check of the results)")
    ap.add_argument("--warm-l2", action="store_true",
                    help="time one copy of the inputs (L2 warm between steps)")
    ap.add_argument("--check-sequences", type=int, default=2,
                    help="sequences of the timed results checked against the oracle")
    ap.add_argument("--no-graph", action="store_true",
                    help="call the library directly for each timed step instead of replaying "
                         "a captured CUDA graph")
    ap.add_argument("--plain-launches", action="store_true",
                    help="with --no-graph: calls launch every layer's kernels directly "
                         "(SC_STACK_PLAIN_LAUNCHES) instead of through the library's own graph")
    ap.add_argument("--rows-kernel", choices=["two-pass", "single-pass"], default="two-pass",
                    help="design of the per-layer attention for windows up to 256 "
                         "(sc_select_rows_kernel)")
    args = ap.parse_args()
    wl = pick_workload(args.workload)
    encoder = args.workload.startswith("encoder")
    if args.impl == "reference":
        (run_reference_encoder if encoder else run_reference)(args, wl)
    else:
        (run_encoder if encoder else run_native)(args, wl)


if __name__ == "__main__":
    main()
