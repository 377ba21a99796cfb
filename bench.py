"""Benchmark of the Aspis PS detection-and-aggregation step on GB300.

One step = one PS round on one GPU: aspis_check (compare every copy pair of
every file, build G), aspis_detect (maximum cliques), aspis_select (one copy
per file) and aspis_aggregate (coordinate-wise lower median), all on one
stream, over synthetic copies already resident in HBM.

Default workload: K=15 workers, r=3, f=455 files, d=11,173,962 fp32 (a
flattened ResNet-18 gradient), optimal (strong) attack with q=3 colluding
ALIE adversaries: 61.0 GB of copies, larger than L2, so no flush is needed
between rounds.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME]
    python bench.py --impl reference ...    # the CPU oracle on a bounded slice

Prints one JSON line (rank 0).  With N > 1 (torchrun) the default is the
coordinate-sharded round: rank p holds coordinates [c0_p, c1_p) of every copy,
and the one exchange of the round is an all-gather (NCCL) of the f per-file
mismatch words, OR-combined on every rank; the whole workload is fixed, so the
scaling is strong.  --replicas runs N independent full rounds instead (weak
scaling); value is then the per-replica ms/round and rounds_per_s the whole
job's rate.

Besides the step, the line reports the model update that follows it
(aspis_sgd: Eq. 1 with momentum 0.9 on the round's output), timed alone with
L2 flushed before every launch (key "update"), and the clique search on the
K = 100, r = 5 graphs of the appendix's timing experiment (aspis_detect_wide,
weak and optimal attacks, q = 5..45; key "table5", beside the paper's
milliseconds), and the round for copies that are not bit-identical
(aspis_round_tolerant at tau = 1e-4 on copies with per-copy noise of std 1e-6;
key "tolerant"), and every other workload of the evaluation at full size (key
"configs").  None of them is part of the step.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

DEFAULT_CONFIG = "k15_r3_d11m_strong_alie"
# Table 5: clique enumeration time (ms) in the K = 100, r = 5 graph, NetworkX
# on an EC2 i3.16xlarge, per number of adversaries q
TABLE5_MS = {"weak": {5: 9, 15: 7, 25: 5, 35: 5, 45: 5},
             "optimal": {5: 11, 15: 11, 25: 9, 35: 8, 45: 6}}
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0      # GB300 HBM3e, nominal (about 8 TB/s)
CONFIG_ORDER = ["k7_r3_d4096_alie", "k15_r3_d1m_weak_reversed", "k15_r3_d11m_strong_alie",
                "k21_r3_d2m_strong_alie", "k15_r5_d1m_strong_alie"]


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    p.add_argument("--config", default=DEFAULT_CONFIG, choices=sorted(synth.CONFIGS))
    p.add_argument("--mode", type=int, default=0, help="0 = lower median, 1 = mean")
    p.add_argument("--d", type=int, default=0,
                   help="override the gradient length (smaller cases for profiling)")
    p.add_argument("--e2e-steps", type=int, default=5)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu", action="store_true")
    p.add_argument("--no-update", action="store_true",
                   help="skip the separate timing of the model update")
    p.add_argument("--no-table5", action="store_true",
                   help="skip the clique-search timing on the K = 100 graphs")
    p.add_argument("--no-tolerant", action="store_true",
                   help="skip the timing of the tolerant round")
    p.add_argument("--no-configs", action="store_true",
                   help="skip the full-size timing of the other workloads")
    p.add_argument("--config-steps", type=int, default=10)
    p.add_argument("--tolerant-noise", type=float, default=1e-6)
    p.add_argument("--tolerant-tau", type=float, default=1e-4)
    p.add_argument("--sharded", action="store_true",
                   help="the coordinate-sharded round (default when N > 1)")
    p.add_argument("--replicas", action="store_true",
                   help="N independent full rounds instead of one sharded round")
    p.add_argument("--cpu-seconds", type=float, default=12.0,
                   help="target CPU time of the oracle baseline sample")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            pk = json.load(fh)
        return float(pk["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def algorithmic_bytes(w, n_sel):
    f = w.f
    cmp_bytes = f * w.r * w.d * 4                  # every copy read once
    agg_bytes = n_sel * w.d * 4 + w.d * 4          # chosen copies read, d written
    return cmp_bytes, agg_bytes


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while timing."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9 and parts[1].replace(".", "").isdigit():
                    rows.append(parts)
        except Exception:
            pass
        finally:
            if self.path and os.path.exists(self.path):
                os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        sm = [float(r[1]) for r in rows]
        mx = max(float(r[2]) for r in rows)
        load = [s for s, r in zip(sm, rows) if float(r[3] or 0) > 300.0] or sm
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in rows for k in range(4) if r[5 + k].lower() == "active"})
        return {"sm_mhz": statistics.median(load), "sm_max_mhz": mx, "reasons": reasons,
                "samples": len(rows), "power_w_max": max(float(r[3] or 0) for r in rows)}


def profile_traffic(kernel_tag: str, workload: str, units: int, source: str):
    """dram bytes per launch from a committed ncu summary, scaled to `units`,
    or None when the summary is absent or older than the kernel source."""
    pdir = os.path.join(ROOT, "profiles")
    sha = hashlib.sha256(open(source, "rb").read()).hexdigest()[:16]
    pat = re.compile(rf"^bench-traffic: {re.escape(kernel_tag)} workload=(\S+) "
                     r"units=(\d+) dram_bytes=(\d+) source_sha=(\w+)")
    if not os.path.isdir(pdir):
        return None
    for fn in sorted(os.listdir(pdir)):
        if not fn.endswith((".md", ".txt")):
            continue
        for line in open(os.path.join(pdir, fn)):
            m = pat.match(line.strip())
            if m and m.group(4) == sha:
                u, b = int(m.group(2)), int(m.group(3))
                return int(round(b * units / u))
    return None


def json_line(obj):
    print(json.dumps(obj), flush=True)


# --------------------------------------------------------------- CPU oracle


def oracle_sample(w, file_workers, ds, host_slice=None, nthreads=None):
    """Times the oracle on coordinates [0, ds) of all copies; returns
    (seconds, RoundResult)."""
    import oracle
    import numpy as np
    if host_slice is None:
        host_slice = synth.build_copies_np(w, file_workers, 0, ds)
    a = oracle.assign(w.K, w.r)
    assert np.array_equal(a.file_workers, file_workers)
    t0 = time.perf_counter()
    res = oracle.run_round(host_slice, a, ds, 0, nthreads)
    return time.perf_counter() - t0, res


def run_reference(args, w):
    """--impl reference: the oracle as it stands on the host cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle
    cores = os.cpu_count() or 1
    a = oracle.assign(w.K, w.r)
    # size the slice so that warmup + steps fit in about two minutes
    probe = 8192
    t_probe, _ = oracle_sample(w, a.file_workers, probe)
    per_step = max(0.5, 90.0 / max(1, args.steps + args.warmup))
    # the slice is also generated on the host, so it stays at most 128 Ki coordinates
    ds = int(min(w.d, 131072, max(probe, probe * per_step / max(t_probe, 1e-3))))
    host = synth.build_copies_np(w, a.file_workers, 0, ds)
    for _ in range(args.warmup):
        oracle_sample(w, a.file_workers, ds, host)
    times = [oracle_sample(w, a.file_workers, ds, host)[0] for _ in range(args.steps)]
    step_ms = statistics.mean(times) * 1e3          # what one timed step took (the slice)
    ms = step_ms * (w.d / ds)
    sample = (f"coordinates [0, {ds}) of all {w.f}x{w.r} copies per step (check, detect, "
              f"select, lower median); ms/round extrapolated from the slice by d/{ds}")
    json_line({
        "impl": "reference", "metric": metric_name(w), "value": ms, "unit": "ms/round",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": step_ms, "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": config_obj(w, args),
        "value_kind": f"extrapolated: oracle time on coordinates [0, {ds}) x d/{ds}; "
                      f"ms_per_step is the measured time of one such slice",
        "slice_coords": ds,
        "cpu_baseline": {"value": ms, "unit": "ms/round", "cores": cores, "kind": "oracle",
                         "sample": sample, "scaled_from_slice": True, "slice_coords": ds},
        "e2e": {"value": ms, "unit": "ms/round", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    })


def metric_name(w):
    return f"PS detect+aggregate ms/round (K={w.K}, r={w.r}, d={w.d})"


def config_obj(w, args, parallelism="single GPU"):
    return {"workload": w.name, "K": w.K, "r": w.r, "f": w.f, "d": w.d, "ld": w.ld, "q": w.q,
            "attack": w.attack, "distortion": w.distortion,
            "aggregator": "lower_median" if args.mode == 0 else "mean",
            "l2": "inputs larger than L2 (no flush)" if w.f * w.r * w.d * 4 > 200e6
            else "L2 flushed between steps",
            "parallelism": parallelism}


def hbm_entry(kernel, nbytes, ms, peak, peak_kind, traffic=None):
    """Roofline object of an HBM-bound pass: algorithmic bytes / event time."""
    gbs = nbytes / (ms * 1e-3) / 1e9
    return {"bound": "hbm", "kernel": kernel, "achieved": gbs, "peak": peak, "unit": "GB/s",
            "frac": gbs / peak, "peak_kind": peak_kind, "frac_nominal": gbs / NOMINAL_HBM_GBS,
            "nominal_peak": NOMINAL_HBM_GBS, "traffic": traffic, "algorithmic_bytes": nbytes,
            "ms": ms}


# --------------------------------------------------------------- GPU arm


def time_rounds(ap, torch, w, a, copies, buf, stream, steps, warmup, mode, flush=None,
                clock_gpu=None, dist=None):
    """Times `steps` rounds (check, detect, select, aggregate) on `stream`
    with events around every step and every pass.  Returns the per-step pass
    times, the total (max over ranks when `dist` is set) and the clocks."""
    from paper_2108_02416_gb300.shard import max_over_ranks

    def one_round(ev=None):
        if flush is not None:
            flush.zero_()
        if ev:
            ev[0].record(stream)
        ap.aspis_check(copies, w.d, a, buf.file_neq, buf.adj, stream)
        if ev:
            ev[1].record(stream)
        ap.aspis_detect(buf.adj, w.K, buf.det, stream)
        ap.aspis_select(buf.file_neq, buf.det, a, buf.sel, stream)
        if ev:
            ev[2].record(stream)
        ap.aspis_aggregate(copies, w.d, a, buf.sel, buf.det, buf.out, mode, stream)
        if ev:
            ev[3].record(stream)

    stream.wait_stream(torch.cuda.current_stream())   # inputs were made on the default stream
    with torch.cuda.stream(stream):
        for _ in range(max(3, warmup)):
            one_round()
    torch.cuda.synchronize()
    det = buf.detection()
    if det.status != ap.OK:
        raise RuntimeError(f"{w.name}: round status {ap.status_str(det.status)}")
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clk = ClockSampler(clock_gpu) if clock_gpu is not None else None
    if clk:
        clk.__enter__()
    try:
        t_start.record(stream)
        for k in range(steps):
            one_round(evs[k])
        t_end.record(stream)
        torch.cuda.synchronize()
    finally:
        if clk:
            clk.__exit__(None, None, None)
    if dist:
        dist.barrier()
    total_ms = t_start.elapsed_time(t_end)
    if flush is not None:         # small inputs: exclude the L2 flush kernels
        total_ms = sum(e[0].elapsed_time(e[3]) for e in evs)
    total_ms = max_over_ranks(total_ms, copies.device)
    return {"total_ms": total_ms,
            "check_ms": [e[0].elapsed_time(e[1]) for e in evs],
            "detsel_ms": [e[1].elapsed_time(e[2]) for e in evs],
            "agg_ms": [e[2].elapsed_time(e[3]) for e in evs],
            "det": buf.detection(), "clocks": clk.summary() if clk else None}


def config_entry(w, t, steps, peak, peak_kind):
    n_sel = t["det"].n_sel
    cmp_bytes, agg_bytes = algorithmic_bytes(w, n_sel)
    det = t["det"]
    return {"round_ms": t["total_ms"] / steps,
            "compare": hbm_entry("compare (aspis_check)", cmp_bytes, statistics.mean(t["check_ms"]),
                                 peak, peak_kind),
            "median": hbm_entry("aggregate (lower median)", agg_bytes,
                                statistics.mean(t["agg_ms"]), peak, peak_kind),
            "detect_select_ms": statistics.mean(t["detsel_ms"]),
            "n_sel": n_sel, "omega": det.omega, "n_max_cliques": det.n_max_cliques,
            "success": det.success, "steps": steps,
            "l2": "inputs larger than L2 (no flush)" if w.f * w.r * w.d * 4 > 200e6
            else "L2 flushed between steps"}


def time_other_configs(args, ap, torch, dev, stream, peak, peak_kind, skip):
    """Every other workload at full size, one at a time (its copies freed
    before the next is built)."""
    out = {}
    for name in CONFIG_ORDER:
        if name == skip:
            continue
        w = synth.CONFIGS[name]
        a = ap.aspis_assign(w.K, w.r)
        copies = synth.build_copies_torch(w, a.file_workers(), dev)
        buf = ap.RoundBuffers(a, w.d, dev)
        small = w.f * w.r * w.d * 4 <= 200e6
        flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev) if small else None
        t = time_rounds(ap, torch, w, a, copies, buf, stream, args.config_steps, 3, args.mode,
                        flush)
        out[name] = config_entry(w, t, args.config_steps, peak, peak_kind)
        del copies, buf, flush
        torch.cuda.empty_cache()
    return out


def table5_hard(ap, torch, np, dev, stream):
    """The clique search on K = 100 random graphs G(100, p) that have many
    maximal cliques (thousands to hundreds of thousands), both modes, checked
    against the oracle; the oracle's host time is the CPU baseline beside it."""
    import oracle
    out = {}
    for p, seed in ((0.5, 7), (0.7, 7)):
        rows = synth.random_graph(100, p, seed)
        words = np.array([[(m >> (32 * i)) & 0xFFFFFFFF for i in range(4)] for m in rows],
                         dtype=np.uint32)
        t0 = time.perf_counter()
        ref = oracle.max_cliques_wide(words, 100)
        cpu_ms = (time.perf_counter() - t0) * 1e3
        adj = torch.from_numpy(words.view(np.int32)).to(dev)
        res = {"graph": f"G(100, {p}), seed {seed}",
               "cpu_baseline": {"value": cpu_ms, "unit": "ms per enumeration of all maximal "
                                "cliques", "cores": 1, "kind": "oracle",
                                "sample": "the whole graph, once"},
               "oracle": {"omega": ref.omega, "n_max_cliques": ref.n_max,
                          "n_maximal": ref.n_maximal}}
        for key, flags in (("detect", 0), ("enumerate_all", ap.WIDE_ALL_MAXIMAL)):
            det_t = ap.wide_detection_buffer(dev, node_budget=1 << 28, flags=flags)
            with torch.cuda.stream(stream):
                ap.aspis_detect_wide(adj, 100, det_t, stream)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(stream):
                e0.record(stream)
                ap.aspis_detect_wide(adj, 100, det_t, stream)
                e1.record(stream)
            torch.cuda.synchronize()
            one = e0.elapsed_time(e1)
            reps = 10 if one < 20.0 else 2
            with torch.cuda.stream(stream):
                torch.cuda._sleep(2_000_000)
                e0.record(stream)
                for _ in range(reps):
                    ap.aspis_detect_wide(adj, 100, det_t, stream)
                e1.record(stream)
            torch.cuda.synchronize()
            dw = ap.DetectionWide.from_tensor(det_t)
            same = (dw.omega == ref.omega and dw.n_max_cliques == ref.n_max and
                    dw.clique_mask == ref.clique and
                    (flags == 0 or dw.n_maximal == ref.n_maximal))
            res[key] = {"ms": e0.elapsed_time(e1) / reps, "launches": reps,
                        "search_nodes": dw.search_nodes, "status": dw.status,
                        "n_maximal": dw.n_maximal, "matches_oracle": bool(same and dw.status == 0)}
        out[f"p={p}"] = res
    return out


def run_sharded(args, w, ap, torch, dev, world, rank, local, dist):
    """One round of the whole workload split by coordinate range over the
    ranks (strong scaling): local compare, all-gather of the f mismatch words,
    graph / cliques / selection on every rank, local median."""
    from paper_2108_02416_gb300 import shard

    c0, c1 = shard.shard_bounds(w.d, world, rank)
    a = ap.aspis_assign(w.K, w.r)
    copies = synth.build_copies_torch(w, a.file_workers(), dev, c0=c0, c1=c1)
    d_local = c1 - c0
    stream = torch.cuda.Stream(device=dev)
    ops = shard.DeviceOps(a, dev, args.mode, stream)
    stream.wait_stream(torch.cuda.current_stream())

    def one_round():
        with torch.cuda.stream(stream):
            res = shard.sharded_round(copies, d_local, c0, ops, timeout_s=120.0)
        if res.status != shard.OK:
            raise RuntimeError(f"sharded round: {res.status} {res.error}")
        return res

    for _ in range(max(3, args.warmup)):
        res = one_round()
    torch.cuda.synchronize()
    det = ops.buf.detection()
    if det.status != ap.OK:
        raise RuntimeError(f"round status {ap.status_str(det.status)}")
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        e0.record(stream)
        for _ in range(args.steps):
            res = one_round()
        e1.record(stream)
        torch.cuda.synchronize()
    if dist:
        dist.barrier()
    ms = shard.max_over_ranks(e0.elapsed_time(e1) / args.steps, dev)
    clocks = clk.summary()

    # end to end: each rank's slice from pinned host memory, the round, its
    # slice of the output back
    host = torch.empty(copies.shape, dtype=torch.float32, pin_memory=True)
    host.copy_(copies)
    hout = torch.empty(max(d_local, 1), dtype=torch.float32, pin_memory=True)
    steps_e2e = args.e2e_steps

    def e2e_round():
        with torch.cuda.stream(stream):
            copies.copy_(host, non_blocking=True)
            r = one_round()
            if r.out is not None:
                hout[:d_local].copy_(r.out, non_blocking=True)

    e2e_round()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record(stream)
    for _ in range(steps_e2e):
        e2e_round()
    f1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = shard.max_over_ranks(f0.elapsed_time(f1) / steps_e2e, dev)
    if rank != 0:
        return
    peak, peak_kind = peaks()
    cmp_bytes, agg_bytes = algorithmic_bytes(w, det.n_sel)
    json_line({
        "metric": metric_name(w), "value": ms, "unit": "ms/round", "n_gpus": world,
        "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms,
        "higher_is_better": False, "scaling": "strong", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded counter-based generator; paper workload shapes)",
        "config": config_obj(w, args, f"coordinate-sharded x{world}: each GPU compares and "
                                      f"aggregates d/{world} coordinates; NCCL all-gather of "
                                      f"the {w.f} mismatch words"),
        "mode": "sharded", "rounds_per_s": 1000.0 / ms,
        "gbps": (cmp_bytes + agg_bytes) / (ms * 1e-3) / 1e9,
        "roofline": hbm_entry("whole round, all GPUs (compare + median bytes)",
                              cmp_bytes + agg_bytes, ms, peak * world, peak_kind),
        "detection": {"omega": det.omega, "n_max_cliques": det.n_max_cliques,
                      "success": det.success, "n_sel": det.n_sel},
        "clocks": clocks, "gpu_launches": 5 * args.steps,
        "e2e": {"value": e2e_ms, "unit": "ms/round", "steps": steps_e2e,
                "h2d_bytes_per_step": int(host.numel() * 4) * world,
                "d2h_bytes_per_step": int(w.d * 4)},
        "cpu_baseline": None,
    })


def main():
    args = parse()
    w = synth.CONFIGS[args.config]
    if args.d:
        import dataclasses
        w = dataclasses.replace(w, d=args.d, name=f"{w.name}@d={args.d}")
    if args.impl == "reference":
        return run_reference(args, w)

    import numpy as np
    import torch
    import paper_2108_02416_gb300 as ap

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if args.sharded or (world > 1 and not args.replicas):
        run_sharded(args, w, ap, torch, dev, world, rank, local, dist)
        if dist:
            dist.destroy_process_group()
        return

    a = ap.aspis_assign(w.K, w.r)
    fw = a.file_workers()
    copies = synth.build_copies_torch(w, fw, dev)
    buf = ap.RoundBuffers(a, w.d, dev)
    stream = torch.cuda.Stream(device=dev)
    small = w.f * w.r * w.d * 4 <= 200e6
    flush = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev) if small else None

    t = time_rounds(ap, torch, w, a, copies, buf, stream, args.steps, args.warmup, args.mode,
                    flush, clock_gpu=local, dist=dist)
    total_ms, det, clocks = t["total_ms"], t["det"], t["clocks"]
    check_ms, detsel_ms, agg_ms = t["check_ms"], t["detsel_ms"], t["agg_ms"]
    n_sel = det.n_sel
    cmp_bytes, agg_bytes = algorithmic_bytes(w, n_sel)
    peak, peak_kind = peaks()
    ms_round = total_ms / args.steps            # per replica (the slowest one)
    all_gbs = (cmp_bytes + agg_bytes) / (ms_round * 1e-3) / 1e9
    csrc = os.path.join(ROOT, "paper_2108_02416_gb300", "csrc")
    cmp_traffic = profile_traffic("compare_vec_kernel", w.name, w.f * w.r * w.d,
                                  os.path.join(csrc, "check.cu"))
    agg_traffic = profile_traffic("aggregate_kernel", w.name, n_sel * w.d,
                                  os.path.join(csrc, "aggregate.cu"))
    main_entry = config_entry(w, t, args.steps, peak, peak_kind)

    # ---- the model update on the round's output, timed alone: w, v <- Eq. 1
    # with momentum 0.9; 20 bytes per coordinate (read g, w, v; write w, v)
    update = None
    if not args.no_update:
        wp = torch.zeros(w.d, dtype=torch.float32, device=dev)
        vp = torch.zeros(w.d, dtype=torch.float32, device=dev)
        fl = flush if flush is not None else torch.empty(256 * 1024 * 1024, dtype=torch.uint8,
                                                         device=dev)
        uev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
        stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(stream):
            for _ in range(max(3, args.warmup)):
                ap.aspis_sgd(buf.out, wp, vp, 0.01, 0.9, stream)
            for k in range(args.steps):
                fl.zero_()
                uev[k][0].record(stream)
                ap.aspis_sgd(buf.out, wp, vp, 0.01, 0.9, stream)
                uev[k][1].record(stream)
        torch.cuda.synchronize()
        upd_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in uev)
        update = hbm_entry("sgd_vec_kernel (aspis_sgd, momentum 0.9)", 20 * w.d, upd_ms, peak,
                           peak_kind)
        update.update({"launches": args.steps, "l2": "flushed before every launch"})
        if flush is None:
            del fl
        del wp, vp

    # ---- Table 5: the clique search alone on the K = 100, r = 5 attack graphs
    table5 = None
    if not args.no_table5:
        table5 = {"unit": "ms per search (mean of 20 back-to-back launches, device time)",
                  "graph": "K=100, r=5 agreement graph of the attack (synth.attack_graph)",
                  "paper": "NetworkX on EC2 i3.16xlarge (Table 5)", "weak": {}, "optimal": {}}
        det_w = ap.wide_detection_buffer(dev)
        det_a = ap.wide_detection_buffer(dev, flags=ap.WIDE_ALL_MAXIMAL)
        for kind, attack in (("weak", "weak"), ("optimal", "strong")):
            for q, paper_ms in TABLE5_MS[kind].items():
                gw = synth.Workload("table5", K=100, r=5, d=1, q=q, attack=attack, seed=q)
                rows = synth.attack_graph(gw)
                words = np.array([[(m >> (32 * i)) & 0xFFFFFFFF for i in range(4)] for m in rows],
                                 dtype=np.uint32)
                adj = torch.from_numpy(words.view(np.int32)).to(dev)
                res = {"paper_ms": paper_ms}
                for key, det_t in (("detect_ms", det_w), ("enumerate_all_ms", det_a)):
                    with torch.cuda.stream(stream):
                        for _ in range(3):
                            ap.aspis_detect_wide(adj, 100, det_t, stream)
                        e0 = torch.cuda.Event(enable_timing=True)
                        e1 = torch.cuda.Event(enable_timing=True)
                        # hold the stream while the host enqueues all 20 launches, so
                        # the events time the device, not the host's call rate
                        torch.cuda._sleep(4_000_000)
                        e0.record(stream)
                        for _ in range(20):
                            ap.aspis_detect_wide(adj, 100, det_t, stream)
                        e1.record(stream)
                    torch.cuda.synchronize()
                    res[key] = e0.elapsed_time(e1) / 20
                dw = ap.DetectionWide.from_tensor(det_a)
                res.update({"omega": dw.omega, "n_max_cliques": dw.n_max_cliques,
                            "n_maximal": dw.n_maximal, "search_nodes": dw.search_nodes,
                            "status": dw.status,
                            "paper_over_enumerate_all": paper_ms / res["enumerate_all_ms"]})
                table5[kind][str(q)] = res
        table5["hard"] = table5_hard(ap, torch, np, dev, stream)

    # ---- end to end through aspis_round_host from pinned host memory
    e2e = None
    if not args.no_e2e:
        host = torch.empty(copies.shape, dtype=torch.float32, pin_memory=True)
        host.copy_(copies)
        hout = torch.empty(w.d, dtype=torch.float32, pin_memory=True)
        hdet = torch.zeros(ap.DETECTION_BYTES, dtype=torch.uint8, pin_memory=True)
        ap.aspis_round_host(host, copies, w.d, a, buf.file_neq, buf.adj, buf.det, buf.sel,
                            buf.out, hout, hdet, args.mode, stream)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.e2e_steps):
            ap.aspis_round_host(host, copies, w.d, a, buf.file_neq, buf.adj, buf.det, buf.sel,
                                buf.out, hout, hdet, args.mode, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = e0.elapsed_time(e1) / args.e2e_steps
        ok = np.array_equal(hout.numpy().view(np.uint32), buf.out.cpu().numpy().view(np.uint32))
        e2e = {"value": e2e_ms, "unit": "ms/round", "steps": args.e2e_steps,
               "h2d_bytes_per_step": int(host.numel() * 4),
               "d2h_bytes_per_step": int(w.d * 4 + ap.DETECTION_BYTES),
               "output_matches_device_run": bool(ok)}
        del host

    # ---- CPU baseline: the oracle on a bounded slice of the same copies
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        probe = 4096
        hs = copies[:, :, :probe].contiguous().cpu().numpy()
        tp, _ = oracle_sample(w, fw, probe, hs)
        ds = int(min(w.d, 2_000_000, max(probe, probe * args.cpu_seconds / max(tp, 1e-3))))
        hs = copies[:, :, :ds].contiguous().cpu().numpy()
        ts, res = oracle_sample(w, fw, ds, hs)
        cores = os.cpu_count() or 1
        cpu = {"value": ts * 1e3 * (w.d / ds), "unit": "ms/round", "cores": cores,
               "kind": "oracle", "scaled_from_slice": True, "slice_coords": ds,
               "sample": f"coordinates [0, {ds}) of all {w.f}x{w.r} copies (check, detect, "
                         f"select, lower median on the slice, {ts:.1f} s); ms/round "
                         f"extrapolated from the slice by d/{ds}",
               "agrees_with_gpu_on_slice": bool(np.array_equal(
                   res.out.view(np.uint32), buf.out[:ds].cpu().numpy().view(np.uint32))
                   if res.out is not None and args.mode == 0 else None)}
        # the same oracle on one host thread, over a slice an eighth as long
        d1 = max(probe, ds // 8)
        t1, _ = oracle_sample(w, fw, d1, np.ascontiguousarray(hs[:, :, :d1]), nthreads=1)
        cpu["single_thread"] = {"value": t1 * 1e3 * (w.d / d1), "unit": "ms/round", "cores": 1,
                                "slice_coords": d1, "scaled_from_slice": True}
        del hs

    # the remaining measurements build their own inputs
    del copies, flush
    torch.cuda.empty_cache()

    # ---- the round for copies that are not bit-identical, at its own
    # workload: the same files with per-copy noise, tau above the noise
    tolerant = None
    if not args.no_tolerant:
        import dataclasses
        wt = dataclasses.replace(w, name=f"{w.name}+copy_noise={args.tolerant_noise:g}",
                                 copy_noise=args.tolerant_noise)
        copies_t = synth.build_copies_torch(wt, fw, dev)
        tb = ap.TolerantBuffers(a, w.d, dev)
        tau = args.tolerant_tau
        fl = torch.empty(256 * 1024 * 1024, dtype=torch.uint8, device=dev) if small else None

        def tol_round():
            ap.aspis_round_tolerant(copies_t, w.d, a, tau, tb.file_neq, tb.adj, tb.det,
                                    tb.slot_mask, tb.sel, tb.means, tb.out, args.mode, stream)

        tev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(5)]
        stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(stream):
            for _ in range(3):
                tol_round()
            for e in tev:
                if fl is not None:
                    fl.zero_()
                e[0].record(stream)
                tol_round()
                e[1].record(stream)
        torch.cuda.synchronize()
        tdet = tb.detection()
        tol_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in tev)
        masks = tb.slot_mask.cpu().numpy()
        chosen = int(sum(bin(int(m)).count("1") for m in masks))
        kept = int((masks != 0).sum())
        # compare reads every copy; the averaging reads the chosen copies and
        # writes one row per kept file; the median reads those rows, writes d
        tol_bytes = (w.f * w.r + chosen + 2 * kept + 1) * w.d * 4
        tolerant = hbm_entry("aspis_round_tolerant (whole round)", tol_bytes, tol_ms, peak,
                             peak_kind)
        tolerant.update({"tau": tau, "copy_noise": args.tolerant_noise, "copies_averaged": chosen,
                         "files_kept": kept, "steps": len(tev), "status": tdet.status,
                         "omega": tdet.omega, "n_max_cliques": tdet.n_max_cliques,
                         "success": tdet.success, "workload": wt.name})
        del copies_t, tb, fl
        torch.cuda.empty_cache()

    configs = None
    if world == 1 and not args.no_configs and not args.d:
        configs = {w.name: main_entry}
        configs.update(time_other_configs(args, ap, torch, dev, stream, peak, peak_kind, w.name))
        configs = {k: configs[k] for k in CONFIG_ORDER if k in configs}

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return
    launches_per_round = 5    # compare, graph, detect, select, aggregate
    rounds_per_s = world * args.steps / (total_ms * 1e-3)
    line = {
        "metric": metric_name(w), "value": ms_round, "unit": "ms/round", "n_gpus": world,
        "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms_round,
        "higher_is_better": False, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded counter-based generator; paper workload shapes)",
        "config": config_obj(w, args, "single GPU" if world == 1 else
                             f"replicas x{world}: independent full rounds, no collective"),
        "mode": "single" if world == 1 else "replicas",
        "rounds_per_s": rounds_per_s,
        "gbps": all_gbs,
        "roofline": dict(hbm_entry("compare (aspis_check)", cmp_bytes, statistics.mean(check_ms),
                                   peak, peak_kind, cmp_traffic)),
        "roofline_aggregate": hbm_entry("aggregate (lower median)", agg_bytes,
                                        statistics.mean(agg_ms), peak, peak_kind, agg_traffic),
        "passes_ms": {"check": statistics.mean(check_ms),
                      "detect_select": statistics.mean(detsel_ms),
                      "aggregate": statistics.mean(agg_ms)},
        "detection": {"omega": det.omega, "n_max_cliques": det.n_max_cliques,
                      "success": det.success, "n_sel": n_sel},
        "clocks": clocks,
        "gpu_launches": launches_per_round * args.steps,
        "e2e": e2e,
        "cpu_baseline": cpu,
        "update": update,
        "table5": table5,
        "tolerant": tolerant,
        "configs": configs,
    }
    json_line(line)
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
