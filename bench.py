#!/usr/bin/env python3
"""Benchmark of the speculative-cascade verification step on GB300.

Default: one GPU, the largest sweep point (B=512 sequences, gamma=8 drafted
positions, V=256000 bf16 Zipf-shaped logits, T=1) under the plug-in optimal
rule OPT alpha=0.2 (Eq. 10): 4.46 GB of logits per step, far more than the
129 MB L2, so steps run back to back without an L2 flush.  A step is one
sc_verify call (one kernel launch) over the whole batch.  Chow 0.5 and Diff 0.1
are timed on the same logits in the same run and reported under
config.other_rules; --sweep adds every sweep point under the three rules.

Prints ONE JSON line (rank 0).  Keys beyond the base contract:
  roofline      achieved HBM GB/s of the verification kernel (algorithmic bytes
                / CUDA-event time) against the measured copy bandwidth
  cpu_baseline  the fp64 oracle timed on this machine's host cores on a bounded
                sample of the same workload
  e2e           the same metric through the public API with host buffers
                (binding.HostVerifier), the host->device copy of the inputs and
                the device->host read of the outputs inside the timed region
  clocks        nvidia-smi SM clock samples taken while the kernel ran

--impl reference times the oracle (the only other implementation of this
method here) on the host cores, on bounded samples of the same workload.
--gpus N under torchrun: every rank verifies its own full batch (weak scaling,
no collective on the data path); value = all ranks' positions / max time.
--vocab-shards W times the vocabulary-sharded step instead (one batch whose
vocabulary is split over W shards; strong scaling when W = world size).
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verified positions/s"
UNIT = "positions/s"
KERNEL_SRC = os.path.join(ROOT, "paper_2405_19261_gb300", "csrc", "sc_verify.cu")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic.json")
NOMINAL_HBM_GBS = 8000.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=4)
    ap.add_argument("--B", type=int, default=None, help="config 4: batch size (default 512)")
    ap.add_argument("--gamma", type=int, default=None, help="config 4: drafted positions (default 8)")
    ap.add_argument("--rule", default=None)
    ap.add_argument("--alpha", type=float, default=None)
    ap.add_argument("--beta", type=float, default=1.0, help="lossy speculative decoding's beta")
    ap.add_argument("--temperature", type=float, default=None, help="config 4 only; 0 = greedy decoding")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--record-traffic", metavar="NCU_CSV", default=None,
                    help="store the DRAM bytes of an ncu capture of this workload for the current kernel source")
    ap.add_argument("--traffic-from-B", type=int, default=None,
                    help="with --record-traffic: the capture ran B0 sequences of this workload's shape; "
                         "its bytes are scaled by B / B0")
    ap.add_argument("--min-warmup-s", type=float, default=0.5,
                    help="keep warming up (untimed) until this long has passed, for clock samples")
    ap.add_argument("--other-rules", default=None,
                    help="comma-separated rule[:alpha] list timed on the same logits after the headline "
                         "(default for config 4: the other two Table 1 rules of the sweep; 'none' for none)")
    ap.add_argument("--sweep", action="store_true",
                    help="config 4: also time every sweep point (B x gamma) under Chow, Diff and OPT")
    ap.add_argument("--e2e-chunks", type=int, default=4,
                    help="e2e: groups of sequences whose host-to-device copy overlaps the verification of the "
                         "previous group (1: copy everything, then verify)")
    ap.add_argument("--vocab-shards", type=int, default=0, metavar="W",
                    help="time the vocabulary-sharded step (include/sc_shard.h) with W shards instead: W ranks "
                         "emulated on one GPU (on-device exchanges, one CUDA graph per step), or under torchrun "
                         "one shard per GPU (W = world size, NCCL all-gathers)")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def kernel_sha():
    """Hash of the kernel's code: comments and blank lines removed, so that a
    comment edit does not orphan counters recorded for identical code."""
    import re
    with open(KERNEL_SRC, encoding="utf-8") as f:
        src = f.read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    lines = [re.sub(r"//.*$", "", ln).rstrip() for ln in src.splitlines()]
    code = "\n".join(ln for ln in lines if ln.strip())
    return hashlib.sha256(code.encode()).hexdigest()[:16]


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


_NCU_UNITS = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "Tbyte": 1e12}


def record_traffic(csv_path, workload_name, command="", scale=1.0, note=""):
    """Store, for the current kernel source, the DRAM bytes ncu measured for one
    sc_unit_kernel launch (the first one in an `ncu --metrics
    dram__bytes_read.sum,dram__bytes_write.sum --csv --log-file` capture),
    multiplied by `scale` when the capture ran a smaller batch of the same rows
    (every unit reads its own rows, so the bytes grow with the units)."""
    import csv
    with open(csv_path, encoding="utf-8") as f:
        rows = list(csv.DictReader(ln for ln in f if ln.startswith('"')))
    launches = {}
    for r in rows:
        if "sc_unit_kernel" in r.get("Kernel Name", ""):
            unit = _NCU_UNITS[r["Metric Unit"]] if r["Metric Unit"] in _NCU_UNITS else None
            if unit is not None:
                launches.setdefault(r["ID"], {})[r["Metric Name"]] = float(r["Metric Value"].replace(",", "")) * unit
    done = [m for m in launches.values() if "dram__bytes_read.sum" in m and "dram__bytes_write.sum" in m]
    if not done:
        raise SystemExit(f"{csv_path}: no sc_unit_kernel launch with both DRAM byte counts")
    m = done[0]
    d = {}
    if os.path.exists(TRAFFIC_FILE):
        with open(TRAFFIC_FILE) as f:
            d = json.load(f)
    d[workload_name] = {"kernel_sha": kernel_sha(),
                        "dram_bytes_per_launch": int(scale * (m["dram__bytes_read.sum"] + m["dram__bytes_write.sum"])),
                        "dram_bytes_read": int(scale * m["dram__bytes_read.sum"]),
                        "dram_bytes_write": int(scale * m["dram__bytes_write.sum"]),
                        "source": command}
    if note:
        d[workload_name]["scaled"] = note
    with open(TRAFFIC_FILE, "w") as f:
        json.dump(d, f, indent=2)
        f.write("\n")
    return d[workload_name]


def stored_traffic(workload_name):
    """ncu DRAM bytes per launch, if recorded for this exact kernel source."""
    if not os.path.exists(TRAFFIC_FILE):
        return None
    with open(TRAFFIC_FILE) as f:
        d = json.load(f)
    e = d.get(workload_name)
    if not e or e.get("kernel_sha") != kernel_sha():
        return None
    return e.get("dram_bytes_per_launch")


# ------------------------------------------------------------------ clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str, interval_ms: int = 50):
        self.gpu_id = gpu_id
        self.interval_ms = interval_ms
        self.proc = None
        self.samples = []
        self.t0 = None

    def start(self):
        self.tmp = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", self.gpu_id, f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", f"-lms={self.interval_ms}"],
                stdout=self.tmp, stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None
        self.t0 = time.time()

    def stop(self):
        if self.proc is None:
            return
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.tmp.flush()
        self.tmp.seek(0)
        for line in self.tmp.read().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                self.samples.append(dict(sm=float(parts[1]), smax=float(parts[2]),
                                         active=parts[4], hw=parts[5], hwt=parts[6],
                                         swt=parts[7], pcap=parts[8]))
            except ValueError:
                continue
        os.unlink(self.tmp.name)

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        reasons = set()
        for s in self.samples:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("pcap", "sw_power_cap")):
                if s[key].lower().startswith("active"):
                    reasons.add(name)
        return {"sm_mhz": statistics.median(s["sm"] for s in self.samples),
                "sm_max_mhz": max(s["smax"] for s in self.samples),
                "reasons": sorted(reasons), "samples": len(self.samples)}


# ------------------------------------------------------------------ oracle timing

def cpu_model():
    """The host CPU's model name (x86 'model name', else lscpu's 'Model name', else the ISA)."""
    import platform
    import subprocess
    try:
        with open("/proc/cpuinfo") as f:
            for ln in f:
                if ln.lower().startswith("model name"):
                    return ln.split(":", 1)[1].strip()
    except OSError:
        pass
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for ln in out.splitlines():
            if ln.startswith("Model name:"):
                return ln.split(":", 1)[1].strip() + f" ({platform.machine()})"
    except (OSError, subprocess.SubprocessError):
        pass
    return platform.machine()


def oracle_throughput(w, max_seqs=64, min_core_s=0.0, threads=0):
    """Time the fp64 oracle (all host cores, or `threads` of them) on a bounded
    sample of sequences: blocks of up to max_seqs sequences, cycling through the
    workload, until at least min_core_s core-seconds (wall time x threads) have
    been spent."""
    import oracle
    cores = oracle.num_threads(threads)
    n = min(w.B, max(1, min(max_seqs, cores * 4)))
    done, passes, start = 0, 0, 0
    t0 = time.perf_counter()
    while True:
        idx = [(start + i) % w.B for i in range(n)]
        oracle.verify_workload(w.subset(idx), nthreads=cores)
        done += n
        passes += 1
        start = (start + n) % w.B
        dt = time.perf_counter() - t0
        if dt * cores >= min_core_s:
            break
    return dict(value=done * w.gamma / dt, unit=UNIT, cores=cores, kind="oracle",
                sample=f"{passes} block(s) of {n} of the {w.B} sequences ({n * (2 * w.gamma + 1)} rows of "
                       f"V={w.V} each), {dt:.2f} s wall on {cores} threads ({dt * cores:.0f} core-s)"), dt, done


# ------------------------------------------------------------------ multi-rank

def step_spread(ms_steps):
    """Median, 10th and 90th percentile of the per-step device times (this rank's),
    by linear interpolation between order statistics."""
    xs = sorted(ms_steps)

    def pct(q):
        if not xs:
            return None
        h = (len(xs) - 1) * q
        lo = int(h)
        hi = min(lo + 1, len(xs) - 1)
        return xs[lo] + (xs[hi] - xs[lo]) * (h - lo)

    return {"p10": pct(0.1), "median": pct(0.5), "p90": pct(0.9), "n": len(xs)}


def max_over_ranks(value, world, device):
    """The largest of every rank's value (all_reduce MAX); value itself on one rank."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank, world, ms_step):
    """Units all ranks processed per second of the slowest rank's step."""
    return units_per_rank * world / (ms_step / 1e3)


# ------------------------------------------------------------------ main

def workload_desc(args):
    """The workload's description (the key of its traffic record), without drawing it."""
    from paper_2405_19261_gb300.workloads import CONFIG_TEXT, SWEEP_ALPHA
    if args.config != 4:
        return f"cfg{args.config}: {CONFIG_TEXT[args.config]}"
    rule = args.rule or "opt"
    alpha = SWEEP_ALPHA[rule] if args.alpha is None else args.alpha
    T = 1.0 if args.temperature is None else args.temperature
    return (f"cfg4: B={args.B or 512} gamma={args.gamma or 8} V=256000 bf16, zipf sigma=0.7, T={T:g}, "
            f"{rule} a={float(alpha)}" + (f" beta={args.beta:g}" if rule == "lossy" else ""))


def workload_from(args, rank=0):
    """The named workload; rank r > 0 of a multi-GPU run gets its own sequences
    (seed offset 1000 r), so the ranks verify disjoint batches of one shape."""
    from paper_2405_19261_gb300.workloads import CONFIG_TEXT, config
    kw = {}
    if rank > 0:
        kw["seed"] = args.config + 1000 * rank
    if args.rule is not None:
        kw["rule"] = args.rule
    if args.alpha is not None:
        kw["alpha"] = args.alpha
    if args.config == 4:
        kw["B"] = args.B or 512
        kw["gamma"] = args.gamma or 8
        kw["temperature"] = args.temperature
    w = config(args.config, **kw)
    w.beta = args.beta
    desc = workload_desc(args)
    if args.config == 4:
        assert desc == (f"cfg4: B={w.B} gamma={w.gamma} V=256000 bf16, zipf sigma=0.7, T={w.temperature:g}, "
                        f"{w.rule} a={w.alpha}" + (f" beta={w.beta:g}" if w.rule == "lossy" else ""))
    return w, desc


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    w, desc = workload_from(args)
    for _ in range(max(0, args.warmup)):  # untimed: loads the oracle library, warms the caches
        oracle_throughput(w, max_seqs=16)
    times, info = [], None
    for _ in range(args.steps):
        info, dt, n_seq = oracle_throughput(w, max_seqs=16)
        times.append(dt)
    ms = 1e3 * sum(times) / len(times)
    value = n_seq * w.gamma / (ms / 1e3)
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": desc, "B": w.B, "gamma": w.gamma, "V": w.V, "rule": w.rule,
                       "alpha": w.alpha, "temperature": w.temperature,
                       "note": "each step runs the oracle on a bounded sample of the workload's sequences"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": info["cores"], "kind": "oracle",
                             "sample": info["sample"]},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_ours(args):
    import torch
    import torch.distributed as dist

    rank, world, local = dist_env()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    from paper_2405_19261_gb300 import binding

    w, desc = workload_from(args, rank)
    d, t, x, u = binding.to_device(w, dev)
    B, g = w.B, w.gamma
    ws = binding.new_workspace(B, g, dev)
    na = torch.empty(B, dtype=torch.int32, device=dev)
    nt = torch.empty(B, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        binding.sc_verify(d, t, x, u, w.rule, w.alpha, w.temperature, beta=w.beta, num_accepted=na,
                          next_token=nt, workspace=ws, stream=stream)

    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush_buf = torch.empty(int(2 * l2), dtype=torch.uint8, device=dev)
    clean_buf = torch.ones(int(2 * l2) // 4, dtype=torch.float32, device=dev)

    def flush_l2():
        # write a buffer larger than L2, then read another one so that the dirty
        # lines are written back now rather than during the timed step
        flush_buf.fill_(1)
        clean_buf.sum()

    def timed(step_fn, steps, flush):
        """K steps timed with CUDA events on the launching stream: (total ms,
        per-step ms).  Inputs smaller than 3x L2 flush L2 before every step."""
        if flush:
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(steps)]
            # Hold the stream with a spin kernel while the host queues every step, so
            # that no step's interval includes the host's launch latency (a small
            # step is shorter than the Python call that launches it).
            sleep = getattr(torch.cuda, "_sleep", None)
            if sleep is not None:
                sleep(int(2e9 * 200e-6 * steps))  # ~200 us of host time per step at ~2 GHz
            for e0, e1 in evs:
                flush_l2()
                e0.record(stream)
                step_fn()
                e1.record(stream)
            torch.cuda.synchronize(dev)
            ms_steps = [e0.elapsed_time(e1) for e0, e1 in evs]
            return sum(ms_steps), ms_steps
        # an event between consecutive steps: the K intervals tile the timed region
        evs = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
        evs[0].record(stream)
        for i in range(steps):
            step_fn()
            evs[i + 1].record(stream)
        torch.cuda.synchronize(dev)
        return evs[0].elapsed_time(evs[-1]), [a.elapsed_time(b) for a, b in zip(evs[:-1], evs[1:])]

    flush = w.logit_bytes < 3 * l2
    peak, peak_kind = measured_peaks()

    props = torch.cuda.get_device_properties(dev)
    gpu_id = str(getattr(props, "uuid", "")) or str(local)
    if gpu_id and not gpu_id.startswith("GPU-") and len(gpu_id) > 8:
        gpu_id = "GPU-" + gpu_id
    sampler = ClockSampler(gpu_id)
    sampler.start()

    # warm-up: at least W steps and at least --min-warmup-s seconds
    t_w = time.perf_counter()
    nwarm = 0
    while nwarm < max(3, args.warmup) or time.perf_counter() - t_w < args.min_warmup_s:
        step()
        nwarm += 1
        if nwarm % 50 == 0:
            torch.cuda.synchronize(dev)
    torch.cuda.synchronize(dev)

    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    ms_total, ms_steps = timed(step, args.steps, flush)
    if world > 1:
        dist.barrier()

    ms_step = max_over_ranks(ms_total / args.steps, world, dev)
    spread = step_spread(ms_steps)
    mean_accepted = float(na.float().mean().item())  # j* of the last step (the method's own statistic)
    positions = B * g * world
    value = whole_job_rate(B * g, world, ms_step)

    # roofline of the verification kernel (the only kernel in a step)
    alg = w.algorithmic_bytes()
    achieved = alg / (ms_step / 1e3) / 1e9
    traffic = stored_traffic(desc)
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": traffic,
                "peak_kind": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
                "frac_of_nominal_8TBs": achieved / NOMINAL_HBM_GBS,
                "algorithmic_bytes_per_launch": alg}

    def rule_line(wr, ms, na_r):
        a = wr.algorithmic_bytes() / (ms / 1e3) / 1e9
        return {"rule": wr.rule, "alpha": wr.alpha, "B": wr.B, "gamma": wr.gamma, "us_per_step": ms * 1e3,
                "positions_per_s": wr.B * wr.gamma / (ms / 1e3), "achieved_gbs": a, "frac": a / peak,
                "frac_of_nominal_8TBs": a / NOMINAL_HBM_GBS, "mean_accepted": float(na_r.float().mean().item())}

    def time_rule(wr, dd, tt, xx, uu):
        """Warm-up and K timed steps of one workload (its own rule and alpha)."""
        ws_r = binding.new_workspace(wr.B, wr.gamma, dev)
        na_r = torch.empty(wr.B, dtype=torch.int32, device=dev)
        nt_r = torch.empty(wr.B, dtype=torch.int32, device=dev)

        def step_r():
            binding.sc_verify(dd, tt, xx, uu, wr.rule, wr.alpha, wr.temperature, beta=getattr(wr, "beta", 1.0),
                              num_accepted=na_r, next_token=nt_r, workspace=ws_r, stream=stream)

        for _ in range(max(3, args.warmup)):
            step_r()
        torch.cuda.synchronize(dev)
        tot, _ = timed(step_r, args.steps, wr.logit_bytes < 3 * l2)
        return rule_line(wr, tot / args.steps, na_r)

    other = []
    others = args.other_rules
    if others is None:
        others = ",".join(r for r in ("chow", "diff", "opt") if r != w.rule) if args.config == 4 else "none"
    if world == 1 and others != "none":
        from paper_2405_19261_gb300.workloads import SWEEP_ALPHA
        for item in others.split(","):
            rname, _, a = item.partition(":")
            wr = w.with_rule(rname, float(a) if a else SWEEP_ALPHA[rname])
            wr.beta = w.beta
            other.append(time_rule(wr, d, t, x, u))
    sweep = []
    if world == 1 and args.sweep and args.config == 4:
        from paper_2405_19261_gb300.workloads import SWEEP_ALPHA, SWEEP_POINTS, config
        for (Bs, gs) in SWEEP_POINTS:
            if (Bs, gs) == (w.B, w.gamma):
                pts = [rule_line(w, ms_step, na)] + [o for o in other]
                sweep.extend(pts)
                continue
            wp = config(4, B=Bs, gamma=gs)
            dp, tp, xp, up = binding.to_device(wp, dev)
            for rname in ("chow", "diff", "opt"):
                wr = wp.with_rule(rname, SWEEP_ALPHA[rname])
                sweep.append(time_rule(wr, dp, tp, xp, up))
            del dp, tp, xp, up
            torch.cuda.empty_cache()
    sampler.stop()  # the clock samples cover the warm-up and every timed step above
    clocks = sampler.summary()

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        hd = d.cpu().pin_memory()
        ht = t.cpu().pin_memory()
        hx = x.cpu().pin_memory()
        hu = u.cpu().pin_memory()
        chunks = max(1, min(args.e2e_chunks, B))
        hv = binding.HostVerifier(B, g, w.V, hd.dtype, chunks=chunks, device=dev)

        def e2e_step():
            hv(hd, ht, hx, hu, w.rule, w.alpha, w.temperature, beta=w.beta)

        for _ in range(max(3, args.warmup)):
            e2e_step()
        torch.cuda.synchronize(dev)
        if world > 1:
            dist.barrier()
        a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for _ in range(args.steps):
            e2e_step()
        a1.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = max_over_ranks(a0.elapsed_time(a1) / args.steps, world, dev)
        h2d = sum(tn.numel() * tn.element_size() for tn in (hd, ht, hx, hu))
        e2e = {"value": whole_job_rate(B * g, world, e2e_ms), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": 8 * B, "ms_per_step": e2e_ms,
               "api": f"binding.HostVerifier: pinned host inputs, {chunks} groups of sequences, each group's "
                      "copy overlapping the previous group's verification"}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu, _, _ = oracle_throughput(w, min_core_s=20.0)
        one, _, _ = oracle_throughput(w, min_core_s=3.0, threads=1)
        cpu["single_thread"] = {"value": one["value"], "sample": one["sample"]}
        cpu["cpu_model"] = cpu_model()

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
                "config": {"workload": desc, "B": B, "gamma": g, "V": w.V, "logits": w.dtype,
                           "rule": w.rule, "alpha": w.alpha, "temperature": w.temperature,
                           "rows_per_s": w.rows * world / (ms_step / 1e3),
                           "sequences_per_s": B * world / (ms_step / 1e3),
                           "mean_accepted": mean_accepted,
                           "acceptance_rate": mean_accepted / g,
                           "l2": ("L2 flushed before every timed step (2x L2 write, then 2x L2 read of another buffer); "
                                  "the steps are queued behind a spin kernel before the first, so no interval waits on the host"
                                  if flush else
                                  f"inputs {w.logit_bytes / 1e6:.0f} MB > L2 {l2 / 1e6:.0f} MB, back to back"),
                           "parallelism": f"{world} independent replica(s), no collective",
                           "other_rules": other},
                "kernel_sha": kernel_sha(),
                "step_ms": spread, "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": args.steps, "clocks": clocks}
        if sweep:
            line["sweep"] = sweep
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_sharded(args):
    """The vocabulary-sharded step on the default workload: W ranks emulated on
    one GPU (world size 1: every rank's kernels and the on-device exchanges,
    captured as one CUDA graph per step) or one shard per GPU under torchrun
    (NCCL all-gathers between the phases)."""
    import torch
    import torch.distributed as dist

    rank, world, local = dist_env()
    W = args.vocab_shards
    if world > 1:
        if W != world:
            raise SystemExit("--vocab-shards must equal the world size under torchrun")
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    from paper_2405_19261_gb300 import binding, sharded

    w, desc = workload_from(args, 0)  # one batch, split over the shards
    bounds = sharded.shard_bounds(w.V, W)
    d, t, x, u = binding.to_device(w, dev)
    stream = torch.cuda.current_stream(dev)
    if world == 1:
        graph = sharded.EmulatedGraph(d, t, x, u, w.rule, w.alpha, w.temperature, bounds)
        ranks = graph.ranks

        def step():
            graph.replay()
        na = graph.num_accepted
        mode = f"{W} ranks emulated on one GPU: every rank's kernels and on-device exchanges, one CUDA graph per step"
    else:
        lo, hi = bounds[rank], bounds[rank + 1]
        ds, ts = d[:, :, lo:hi].contiguous(), t[:, :, lo:hi].contiguous()
        del d, t
        ranks = [sharded.ShardRank(w.B, w.gamma, bounds, rank, ds.dtype, dev)]
        ex = sharded.DistExchange()

        def step():
            sharded.sharded_step(ranks, [(ds, ts)], x, u, w.rule, w.alpha, w.temperature, ex)
        na = ranks[0].num_accepted
        mode = f"one shard per GPU, {W} GPUs, NCCL all-gathers between the phases"
    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    ms_step = max_over_ranks(e0.elapsed_time(e1) / args.steps, world, dev)
    mean_accepted = float(na.float().mean().item())
    # roofline of the dominant kernel, the pass over the logits (rank 0's shard):
    # its algorithmic bytes are the shard's logits read once
    r0 = ranks[0]
    dd = d[:, :, bounds[0]:bounds[1]] if world == 1 else ds
    tt = t[:, :, bounds[0]:bounds[1]] if world == 1 else ts
    for _ in range(3):
        r0.pass1(dd, tt, x, w.temperature, w.rule)
    p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    p0.record(stream)
    for _ in range(args.steps):
        r0.pass1(dd, tt, x, w.temperature, w.rule)
    p1.record(stream)
    torch.cuda.synchronize(dev)
    ms_pass1 = p0.elapsed_time(p1) / args.steps
    peak, peak_kind = measured_peaks()
    alg1 = w.rows * (bounds[1] - bounds[0]) * w.elt_bytes
    achieved = alg1 / (ms_pass1 / 1e3) / 1e9
    alg = w.algorithmic_bytes()
    launches = (11 if w.rule == "opt" else 8) * (W if world == 1 else 1)  # our kernels per rank and step
    if rank == 0:
        line = {"metric": METRIC, "value": w.B * w.gamma / (ms_step / 1e3), "unit": UNIT, "n_gpus": world,
                "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
                "scaling": "strong", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
                "config": {"workload": desc, "B": w.B, "gamma": w.gamma, "V": w.V, "logits": w.dtype,
                           "rule": w.rule, "alpha": w.alpha, "temperature": w.temperature,
                           "vocab_shards": W, "shard_bounds": bounds, "parallelism": mode,
                           "mean_accepted": mean_accepted,
                           "step_gbs_algorithmic": alg / (ms_step / 1e3) / 1e9,
                           "step_frac_algorithmic": alg / (ms_step / 1e3) / 1e9 / peak,
                           "l2": f"inputs {w.logit_bytes / 1e6:.0f} MB > L2, back to back"},
                "roofline": {"bound": "hbm", "kernel": "shard_pass1_kernel (rank 0's shard)",
                             "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                             "traffic": None, "peak_kind": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
                             "algorithmic_bytes_per_launch": alg1, "us_per_launch": ms_pass1 * 1e3},
                "cpu_baseline": None, "e2e": None, "gpu_launches": launches * args.steps}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    if args.record_traffic:
        w_b = args.B or 512
        desc = workload_desc(args)
        scale, note = 1.0, ""
        if args.traffic_from_B:
            scale = w_b / args.traffic_from_B
            note = (f"captured at B={args.traffic_from_B} (same gamma, V, rule), scaled by {scale:g} "
                    f"to B={w_b}: every unit reads its own rows")
        print(json.dumps(record_traffic(args.record_traffic, desc, " ".join(sys.argv), scale, note)))
        return
    if args.impl == "reference":
        run_reference(args)
    elif args.vocab_shards:
        run_sharded(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
