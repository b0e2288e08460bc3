"""Benchmark: batched DynaComm scheduling on GB300.

One step = the whole scheduling path over one batch of synthetic instances:
profile generation (dc_profile_gen), the forward DP (Eq. 8 / Algorithm 3), the
backward DP (Eq. 9 / Algorithm 4) and the timeline replay f_m of both chosen
decisions, with every input already resident in HBM. The end-to-end figure
("e2e") runs the user-facing path instead: profiles in pinned host memory are
copied in, scheduled and replayed, and the results are copied back, all inside
the timed region.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload vgg16]
    python bench.py --impl reference ...   # the CPU oracle on the host cores

Prints one JSON line (rank 0). Under torchrun each rank solves its own batch of
distinct instances (weak scaling, no collective on the data path).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2101_07968_gb300 import workloads as wl  # noqa: E402

METRIC = "scheduling instances/s and DP cells/s on 1 GB300; % of int-ALU/HBM roofline"
UNIT = "instances/s"
PEAKS_PATH = os.path.join(ROOT, "MEASURED_PEAKS.json")
TRAFFIC_PATH = os.path.join(ROOT, "profiles", "dp_traffic.json")

# Integer-ALU roof: GB300's maximum SM clock, and the instructions one
# transition of the 32-bit passes takes (one add-then-max, half a 3-input min).
MAX_SM_MHZ = 2070
ALU_OPS_PER_TRANSITION = 1.5

# Oracle sample sizes for the CPU baseline (instances per timed pass).
CPU_SAMPLE = {"tiny": 4096, "alexnet": 1_000_000, "vgg16": 1_000_000, "resnet50": 65_536,
              "deepchain": 16}


def transitions(L: int) -> int:
    """Finite (m, n, k) triples of one direction's DP: n = 1 has one candidate
    per row; column n >= 2 has m - n + 1 candidates in row m."""
    return L + (L + 1) * L * (L - 1) // 6


def cells(L: int) -> int:
    return L * (L + 1) // 2


def dp_bytes(L: int) -> int:
    """Algorithmic HBM bytes of one direction per instance: two cost rows and dt
    in; makespan, decision words, nseg and status out."""
    W = (L - 1 + 31) // 32
    return 2 * L * 8 + 8 + 8 + 4 * W + 4 + 4


# ------------------------------------------------------------------ helpers
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100", "-f", self.path],
                stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.2)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return None
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


def load_json(path):
    try:
        with open(path) as f:
            return json.load(f)
    except (OSError, ValueError):
        return None


# the sources each first-pass kernel is built from, by the L it serves
FIRST_PASS_SOURCES = {
    "small_dense_kernel": ("dp_small.cu", "dp_small.cuh", "gen_device.cuh", "common.cuh"),
    "mid_kernel": ("dp_mid.cu", "common.cuh"),
    "deep_kernel": ("dp_deep.cu", "common.cuh"),
}


def dp_source_hash(kernel: str = "small_dense_kernel") -> str:
    """Hash of the code (comments and blank space removed) of the sources a first
    pass is built from, which a traffic record must match to be reported."""
    import hashlib
    import re
    h = hashlib.sha256()
    for name in FIRST_PASS_SOURCES[kernel]:
        with open(os.path.join(ROOT, "paper_2101_07968_gb300", "csrc", name)) as f:
            code = re.sub(r"/\*.*?\*/", "", f.read(), flags=re.S)
        code = re.sub(r"//[^\n]*", "", code)
        h.update("".join(code.split()).encode())
    return h.hexdigest()[:16]


def traffic_record(workload: str, L: int):
    """DRAM bytes of one direction's first pass from profiles/dp_traffic.json, if
    a record for this workload matches the kernel's current sources."""
    data = load_json(TRAFFIC_PATH) or {}
    kernel = first_pass_kernel(L)
    for rec in data.get("records", []):
        if (rec.get("workload") == workload and rec.get("kernel") == kernel
                and rec.get("source_hash") == dp_source_hash(kernel)):
            return rec.get("bytes_per_direction")
    return None


def first_pass_kernel(L: int) -> str:
    """The kernel of a direction's first pass over the batch."""
    if L <= 16:
        return "small_dense_kernel"
    return "mid_kernel" if L <= 256 else "deep_kernel"


def binding_roof(*roofs, **extra):
    """The roof that binds: the one with the larger minimal time at peak, i.e. the
    larger achieved fraction; the others follow under other_roof (one) or
    other_roofs (several)."""
    order = sorted(roofs, key=lambda r: -r["frac"])
    out = dict(order[0], **extra)
    rest = order[1:]
    if len(rest) == 1:
        out["other_roof"] = rest[0]
    elif rest:
        out["other_roofs"] = rest
    return out


# ------------------------------------------------------------ multi-rank
def rank_config(base: dict, rank: int) -> dict:
    """Weak scaling: each rank solves its own `batch` distinct instances; rank r
    takes instance numbers [r*batch, (r+1)*batch) of the seeded stream (the
    generator is counter-based, so the shards together are the world-size batch)."""
    return wl.with_batch(base, base["batch"], inst0=base.get("inst0", 0) + rank * base["batch"])


def max_over_ranks(x: float, device=None) -> float:
    """The slowest rank's value (a single process returns x)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------- reference arm
def oracle_pass(cfg, sample: int, nthreads: int):
    """The oracle, as it stands, over the first `sample` instances of cfg:
    generator, Algorithm 3, Algorithm 4 and f_m of both decisions."""
    import oracle
    c = wl.with_batch(cfg, sample, inst0=cfg.get("inst0", 0))
    prof = oracle.profile_gen(c)
    for d, (a, b) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
        out = oracle.schedule_batch(d, prof[a], prof[b], prof["dt"], nthreads=nthreads)
        oracle.replay_batch(d, prof[a], prof[b], prof["dt"], out["bits"], nthreads=nthreads)


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import oracle
    oracle.build()
    cfg = wl.config(args.workload)
    if args.batch:
        cfg = wl.with_batch(cfg, args.batch)
    cores = os.cpu_count() or 1
    sample = min(cfg["batch"], CPU_SAMPLE[args.workload])
    for _ in range(args.warmup):
        oracle_pass(cfg, sample, cores)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_pass(cfg, sample, cores)
    dt = (time.perf_counter() - t0) / max(args.steps, 1)
    value = sample / dt
    desc = (f"first {sample} of {cfg['batch']} instances of {args.workload} per step: "
            f"generator + Alg. 3 + Alg. 4 + f_m, {cores} threads")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": {"workload": args.workload, "batch": cfg["batch"], "L": cfg["L"],
                       "sample_per_step": sample},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": desc},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------- scaling in L
def run_lsweep(args):
    """Scheduling time against depth L (the analogue of the paper's Fig. 12): for
    each L, the GPU's forward + backward DP over a batch, per instance and
    direction, beside the oracle on one host core over a sample of the same
    instances, which are also checked bit for bit; then the log-log slope."""
    import numpy as np
    import torch

    import oracle
    from paper_2101_07968_gb300 import build as libbuild
    from paper_2101_07968_gb300 import dynacomm as dc

    libbuild.build()
    dc.lib()
    oracle.build()
    dev = torch.device("cuda", torch.cuda.current_device())
    rows = []
    with ClockSampler(dev.index) as clk:
        for L in wl.LSWEEP_LS:
            batch = int(min(1 << 20, max(304, (1 << 36) // transitions(L))))
            cfg = wl.lsweep_config(L, batch)
            prof = dc.profile_gen(cfg, device=dev)
            sch = dc.Scheduler(batch, L, device=dev)
            pairs = ((0, ("fc", "pt")), (1, ("bc", "gt")))
            for d, (c, x) in pairs:  # warm-up
                sch.run(d, prof[c], prof[x], prof["dt"])
            torch.cuda.synchronize()
            reps = 3 if L <= 512 else 1
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(reps):
                for d, (c, x) in pairs:
                    sch.run(d, prof[c], prof[x], prof["dt"])
            e1.record()
            torch.cuda.synchronize()
            gpu_s = e0.elapsed_time(e1) * 1e-3 / reps
            got = {d: {k: v.cpu().numpy() for k, v in sch.run(d, prof[c], prof[x], prof["dt"]).items()}
                   for d, (c, x) in pairs}
            # the oracle (Eq. 8 / Eq. 9 cell by cell) on one core; about L^3 / 3
            # loop iterations per instance and direction
            n_or = int(max(1, min(batch, 2e8 // (L ** 3 // 3 + 1))))
            po = oracle.profile_gen(wl.with_batch(cfg, n_or))
            t0 = time.perf_counter()
            exp = {d: oracle.schedule_batch(d, po[c], po[x], po["dt"], nthreads=1) for d, (c, x) in pairs}
            cpu_s = time.perf_counter() - t0
            W = dc.words(L)
            for d in (0, 1):
                g = got[d]
                bits = g["bits"].view(np.uint32)[:n_or, :W] if W else np.zeros((n_or, 0), np.uint32)
                same = (np.array_equal(g["makespan"][:n_or], exp[d]["makespan"])
                        and np.array_equal(g["nseg"][:n_or], exp[d]["nseg"])
                        and np.array_equal(g["status"][:n_or], exp[d]["status"])
                        and np.array_equal(bits, exp[d]["bits"].reshape(n_or, W)))
                if not same:
                    raise RuntimeError(f"GPU and oracle disagree at L={L} dir={d}")
            rows.append({"L": L, "batch": batch,
                         "gpu_us_per_instance_direction": gpu_s / (2 * batch) * 1e6,
                         "gpu_transitions_per_s": 2 * transitions(L) * batch / gpu_s,
                         "oracle_1core_us_per_instance_direction": cpu_s / (2 * n_or) * 1e6,
                         "oracle_sample": n_or, "parity_checked": n_or})

    def slope(key, lo):
        pts = [(np.log(r["L"]), np.log(r[key])) for r in rows if r["L"] >= lo]
        return float(np.polyfit([p[0] for p in pts], [p[1] for p in pts], 1)[0])

    line = {"mode": "lsweep", "metric": "scheduling time per instance and direction against L",
            "unit": "us", "higher_is_better": False, "data": "synthetic",
            "config": {"workload": "deep-chain draws at depth L (seed 5)",
                       "batch": "min(2^20, max(304, 2^36 / C(L)))"},
            "rows": rows,
            "slope_gpu_L_ge_256": slope("gpu_us_per_instance_direction", 256),
            "slope_oracle_L_ge_128": slope("oracle_1core_us_per_instance_direction", 128),
            "parity": "GPU outputs bit-exact with the oracle on every sampled instance, both directions",
            "clocks": clk.summary()}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------- competing strategies
def run_compare(args):
    """DynaComm's optimum against the paper's competing strategies on one
    workload (the analogue of Figs. 5-6 on synthetic profiles): Sequential (one
    transmission), layer by layer (LBL), the greedy schedulers (Algorithm 1
    forward, Algorithm 2 backward), all on the GPU. Per direction: each
    strategy's makespan over the DP optimum (distribution), the share of
    instances where it is optimal, the running-time reduction against
    Sequential, and each strategy's own throughput."""
    import numpy as np
    import torch

    from paper_2101_07968_gb300 import build as libbuild
    from paper_2101_07968_gb300 import dynacomm as dc

    libbuild.build()
    dc.lib()
    dev = torch.device("cuda", torch.cuda.current_device())
    cfg = wl.config(args.workload)
    if args.batch:
        cfg = wl.with_batch(cfg, args.batch)
    B, L = cfg["batch"], cfg["L"]
    W = dc.words(L)
    prof = dc.profile_gen(cfg, device=dev)
    zeros = torch.zeros((B, max(W, 1)), dtype=torch.int32, device=dev)
    ones = torch.zeros((B, max(W, 1)), dtype=torch.int32, device=dev)
    for l in range(1, L):  # p_l / g_l = 1 for every position: layer by layer
        bit = 1 << ((l - 1) % 32)
        ones[:, (l - 1) // 32] |= bit - (1 << 32) if bit >= 1 << 31 else bit
    sch = dc.Scheduler(B, L, device=dev)

    def timed(fn, reps=5):
        fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            out = fn()
        e1.record()
        torch.cuda.synchronize()
        return out, e0.elapsed_time(e1) / reps * 1e-3

    result, result_mk = {}, {}
    with ClockSampler(dev.index) as clk:
        for d, name, (c, x) in ((0, "forward", ("fc", "pt")), (1, "backward", ("bc", "gt"))):
            a = (prof[c], prof[x], prof["dt"])
            dp, t_dp = timed(lambda: sch.run(d, *a)["makespan"].clone())
            gr, t_gr = timed(lambda: dc.greedy(d, *a)["makespan"])
            sq, t_sq = timed(lambda: dc.eval_timeline(d, *a, zeros[:, :W].contiguous() if W else None))
            lb, t_lb = timed(lambda: dc.eval_timeline(d, *a, ones[:, :W].contiguous() if W else None))
            opt = dp.double()
            result_mk[name] = {"dynacomm": dp, "greedy": gr, "sequential": sq, "lbl": lb}
            rows = {}
            for sname, v, t in (("dynacomm", dp, t_dp), ("greedy", gr, t_gr),
                                ("sequential", sq, t_sq), ("lbl", lb, t_lb)):
                r = (v.double() / opt).cpu().numpy()
                rows[sname] = {
                    "makespan_over_optimum": {"mean": float(r.mean()), "p50": float(np.median(r)),
                                              "p90": float(np.percentile(r, 90)),
                                              "p99": float(np.percentile(r, 99)),
                                              "max": float(r.max())},
                    "optimal_share": float((v == dp).double().mean().item()),
                    "mean_reduction_vs_sequential": float(1.0 - (v.double() / sq.double()).mean().item()),
                    "instances_per_s": B / t}
            result[name] = rows
        # whole iteration (Sec. III-A: the backward pass starts after the forward)
        it = {}
        seq_it = result_mk["forward"]["sequential"] + result_mk["backward"]["sequential"]
        for sname in ("dynacomm", "greedy", "sequential", "lbl"):
            tot = result_mk["forward"][sname] + result_mk["backward"][sname]
            it[sname] = {"mean_us": float(tot.double().mean().item()),
                         "mean_reduction_vs_sequential": float(1.0 - (tot.double() / seq_it.double()).mean().item()),
                         "max_reduction_vs_sequential": float(1.0 - (tot.double() / seq_it.double()).min().item())}
        # idle windows (Sec. IV-C): the forward schedule of the next iteration can
        # run during the last push (dt + gt of layer 1), the backward schedule
        # during the first pull (dt + pt of layer 1); the GPU's latency for one
        # instance, launch included, against them
        lat = {}
        sch1 = dc.Scheduler(1, L, device=dev)
        for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
            a1 = (prof[c][:1], prof[x][:1], prof["dt"][:1])
            ts = []
            for _ in range(25):
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                torch.cuda.synchronize()
                e0.record()
                sch1.run(d, *a1)
                e1.record()
                torch.cuda.synchronize()
                ts.append(e0.elapsed_time(e1) * 1e3)
            lat[d] = float(np.median(ts[5:]))
        win_f = (prof["dt"] + prof["gt"][:, 0]).double()  # hides the forward schedule
        win_b = (prof["dt"] + prof["pt"][:, 0]).double()  # hides the backward schedule
        window = {"single_instance_latency_us": {"forward": lat[0], "backward": lat[1]},
                  "window_fwd_us_p01_p50": [float(torch.quantile(win_f, 0.01)), float(win_f.median())],
                  "window_bwd_us_p01_p50": [float(torch.quantile(win_b, 0.01)), float(win_b.median())],
                  "hidden_share_forward": float((win_f >= lat[0]).double().mean()),
                  "hidden_share_backward": float((win_b >= lat[1]).double().mean()),
                  "batch_amortised_us_per_instance": {
                      "forward": 1e6 / result["forward"]["dynacomm"]["instances_per_s"],
                      "backward": 1e6 / result["backward"]["dynacomm"]["instances_per_s"]}}
    line = {"mode": "compare", "metric": "makespan of each strategy over the DP optimum",
            "data": "synthetic", "config": {"workload": args.workload, "batch": B, "L": L},
            "iteration": it, "idle_window": window,
            "strategies": {"dynacomm": "Algorithms 3/4 (dc_schedule_*)",
                           "greedy": "Algorithm 1 forward / Algorithm 2 backward (dc_greedy_*)",
                           "sequential": "one transmission (dc_eval_timeline_batch, no break)",
                           "lbl": "layer by layer (dc_eval_timeline_batch, every break)"},
            "result": result, "clocks": clk.summary()}
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------- fused generate-and-solve
def run_fused(args):
    """Generate-and-solve in one pass (dc_schedule_generated_batch, L <= 16)
    against the unfused dc_profile_gen + forward DP + backward DP on the same
    workload: the same results bit for bit (checked here), without the profiles'
    round trip through HBM. Reported separately from the step: fusion changes
    the algorithmic byte count."""
    import torch

    from paper_2101_07968_gb300 import build as libbuild
    from paper_2101_07968_gb300 import dynacomm as dc

    libbuild.build()
    dc.lib()
    dev = torch.device("cuda", torch.cuda.current_device())
    cfg = wl.config(args.workload)
    if args.batch:
        cfg = wl.with_batch(cfg, args.batch)
    B, L = cfg["batch"], cfg["L"]
    W = dc.words(L)
    fused = dc.GeneratedScheduler(cfg, device=dev)
    prof = {k: torch.empty((B, L), dtype=torch.int64, device=dev) for k in ("fc", "pt", "bc", "gt")}
    prof["dt"] = torch.empty(B, dtype=torch.int64, device=dev)
    sch = dc.Scheduler(B, L, device=dev)
    keep: list = []
    ccfg = dc.make_cfg(cfg, keep)

    def unfused():
        assert dc.dc_profile_gen(ccfg, prof["fc"], prof["pt"], prof["bc"], prof["gt"], prof["dt"]) == 0
        return [sch.run(d, prof[c], prof[x], prof["dt"])["makespan"]
                for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt")))]

    def timed(fn, reps):
        for _ in range(max(args.warmup, 3)):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / reps

    with ClockSampler(dev.index) as clk:
        ms_f = timed(fused.run, args.steps)
        ms_u = timed(unfused, args.steps)
    fo = fused.run()
    mk = unfused()
    torch.cuda.synchronize()
    same = all(torch.equal(fo["makespan"][d], mk[d]) for d in (0, 1))
    if not same:
        raise RuntimeError("fused and unfused results differ")
    out_b = 2 * (8 + 4 * W + 4 + 4)
    line = {"mode": "fused", "metric": "generate + forward DP + backward DP, instances/s",
            "unit": "instances/s", "higher_is_better": True, "data": "synthetic",
            "config": {"workload": args.workload, "batch": B, "L": L},
            "fused": {"value": B / (ms_f * 1e-3), "ms": ms_f,
                      "algorithmic_bytes_per_instance": out_b},
            "unfused": {"value": B / (ms_u * 1e-3), "ms": ms_u,
                        "algorithmic_bytes_per_instance": (4 * L + 1) * 8 + 2 * (2 * L * 8 + 8) + out_b},
            "speedup": ms_u / ms_f, "bit_exact": same, "clocks": clk.summary()}
    print(json.dumps(line), flush=True)
    return 0


# --------------------------------------------------------------- GPU arm
def run_ours(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2101_07968_gb300 import build as libbuild
    from paper_2101_07968_gb300 import dynacomm as dc

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    libbuild.build()
    dc.lib()
    dev = torch.device("cuda", torch.cuda.current_device())

    base = wl.config(args.workload)
    if args.batch:
        base = wl.with_batch(base, args.batch)
    B, L = base["batch"], base["L"]
    cfg = rank_config(base, rank)  # distinct instances per rank
    W = dc.words(L)

    prof = {k: torch.empty((B, L), dtype=torch.int64, device=dev) for k in ("fc", "pt", "bc", "gt")}
    prof["dt"] = torch.empty(B, dtype=torch.int64, device=dev)
    sched = dc.Scheduler(B, L, device=dev)
    rep = {d: torch.empty(B, dtype=torch.int64, device=dev) for d in (0, 1)}
    keep: list = []
    ccfg = dc.make_cfg(cfg, keep)

    def barrier():
        if world > 1:
            dist.barrier()

    def step(ev=None, kev=None):
        if ev is not None:
            ev[0].record()
        assert dc.dc_profile_gen(ccfg, prof["fc"], prof["pt"], prof["bc"], prof["gt"],
                                 prof["dt"]) == 0
        if ev is not None:
            ev[1].record()
        if kev is not None:  # the library records kev[0..1] around the first pass's launches
            assert dc.dc_time_next_pass(kev[0], kev[1]) == 0
        fo = sched.run(0, prof["fc"], prof["pt"], prof["dt"])
        if ev is not None:
            ev[2].record()
        if kev is not None:
            assert dc.dc_time_next_pass(kev[2], kev[3]) == 0
        bo = sched.run(1, prof["bc"], prof["gt"], prof["dt"])
        if ev is not None:
            ev[3].record()
        assert dc.dc_eval_timeline_batch(B, L, 0, prof["fc"], prof["pt"], prof["dt"],
                                         fo["bits"], rep[0]) == 0
        assert dc.dc_eval_timeline_batch(B, L, 1, prof["bc"], prof["gt"], prof["dt"],
                                         bo["bits"], rep[1]) == 0
        if ev is not None:
            ev[4].record()

    for _ in range(max(args.warmup, 0)):
        step()
    torch.cuda.synchronize()
    # consistency of the path itself: replayed decisions reproduce the DP optimum
    for d in (0, 1):
        ok = torch.equal(rep[d], sched.out[d]["makespan"])
        if not ok:
            raise RuntimeError("timeline replay disagrees with the DP makespan")

    # the same step captured once as a CUDA graph (dynacomm.StepGraph): a replay is
    # one launch per step instead of the step's host-side calls
    sg, graph_error = None, None
    if not args.no_graph:
        try:
            sg = dc.StepGraph(cfg, device=dev)
            for _ in range(max(args.warmup, 1)):
                sg.replay()
            torch.cuda.synchronize()
            for d in (0, 1):  # same config, same results as the eager step
                if not torch.equal(sg.sched.out[d]["makespan"], sched.out[d]["makespan"]):
                    raise RuntimeError("graph replay disagrees with the eager step")
        except Exception as exc:  # reported in the line; the eager timing stands
            sg, graph_error = None, f"{type(exc).__name__}: {exc}"

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(args.steps)]
    # the first pass of each direction, timed by the library on its stream
    kevs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    for kv in kevs:
        for e in kv:
            e.record()  # creates the CUDA event the library will record
    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(dev.index if rank == 0 else -1) if rank == 0 else _Null() as clk:
        barrier()
        torch.cuda.synchronize()
        start.record()
        for s in range(args.steps):
            step(evs[s])
        end.record()
        torch.cuda.synchronize()
        barrier()
        if sg is not None:
            g0.record()
            for s in range(args.steps):
                sg.replay()
            g1.record()
            torch.cuda.synchronize()
            barrier()
    eager_ms = max_over_ranks(start.elapsed_time(end) / max(args.steps, 1), dev)
    seg = np.array([[e[j].elapsed_time(e[j + 1]) for j in range(4)] for e in evs])
    gen_ms, fwd_ms, bwd_ms, eval_ms = seg.mean(axis=0)
    # the first passes timed on their own launches, in K more eager steps (the
    # events the library records between a first pass and its work-list pass
    # stop the latter from being scheduled early, so they stay out of the steps
    # timed above)
    for s in range(args.steps):
        step(None, kevs[s])
    torch.cuda.synchronize()
    kseg = np.array([[k[0].elapsed_time(k[1]), k[2].elapsed_time(k[3])] for k in kevs])
    fwd_k_ms, bwd_k_ms = kseg.mean(axis=0)
    # instances each direction's first pass left to its work-list pass (the same
    # every step: the generator redraws the same batch)
    listed = []
    for d, (c, x) in ((0, ("fc", "pt")), (1, ("bc", "gt"))):
        sched.run(d, prof[c], prof[x], prof["dt"])
        torch.cuda.synchronize()
        listed.append(int(sched.workspace[:4].view(torch.int32).item()))
    graph_ms = (max_over_ranks(g0.elapsed_time(g1) / max(args.steps, 1), dev)
                if sg is not None else None)
    ms = graph_ms if graph_ms is not None else eager_ms
    del sg

    # ---- ALU roof: the DP's transition op mix, register-only, all SMs
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    roof_threads, roof_blocks, roof_iters = 512, sms * 4, 20_000
    sink = torch.empty(roof_blocks * roof_threads, dtype=torch.int32, device=dev)
    roof = {}
    for variant in (0, 1):
        assert dc.dc_roof_int_probe(variant, roof_blocks, roof_threads, 400, sink) == 0
        r0, r1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        r0.record()
        assert dc.dc_roof_int_probe(variant, roof_blocks, roof_threads, roof_iters, sink) == 0
        r1.record()
        torch.cuda.synchronize()
        roof[variant] = roof_blocks * roof_threads * roof_iters * 8 / (r0.elapsed_time(r1) * 1e-3)

    # ---- end to end through the public API with host buffers
    e2e = None if args.no_e2e else run_e2e(dc, torch, prof, sched, B, L, W, dev, args,
                                           barrier, world)

    # ---- CPU baseline: the oracle on this host's cores (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        cores = os.cpu_count() or 1
        sample = min(B, CPU_SAMPLE[args.workload])
        t0 = time.perf_counter()
        oracle_pass(base, sample, cores)
        cpu_s = time.perf_counter() - t0
        cpu = {"value": sample / cpu_s, "unit": UNIT, "cores": cores, "kind": "oracle",
               "sample": f"first {sample} of {B} instances of {args.workload}: generator + "
                         f"Alg. 3 + Alg. 4 + f_m, {cores} threads, {cpu_s:.1f} s"}

    if rank != 0:
        return 0
    total = B * world
    value = total / (ms * 1e-3)
    trans = 2 * transitions(L) * B
    dp_s = (fwd_ms + bwd_ms) * 1e-3
    # the dominant kernel: the first pass of both directions, timed on its own
    # launches; its work is the instances it solved (the listed ones are left
    # to the work-list pass)
    first_s = (fwd_k_ms + bwd_k_ms) * 1e-3
    first_trans = transitions(L) * (2 * B - listed[0] - listed[1])
    achieved = first_trans / first_s / 1e9
    # ALU roof from unit counts: 4 x 16 integer-ALU lanes per SM per clock, the
    # 32-bit passes spend 1.5 ALU instructions per transition
    peak = sms * 64 * MAX_SM_MHZ * 1e6 / ALU_OPS_PER_TRANSITION / 1e9
    traffic = traffic_record(args.workload, L)
    hbm_peak = (load_json(PEAKS_PATH) or {}).get("hbm_gbs", 6800.0)
    dp_gbs = dp_bytes(L) * (2 * B - listed[0] - listed[1]) / first_s / 1e9
    # kernels of this library per step: the generator; per direction the first
    # pass (split into several launches for long deep-chain batches) and the
    # pass over its work list; the two timeline replays
    launches_per_step = 1 + 2 * dc.dc_schedule_kernel_launches(B, L) + 2
    # both roofs of the DP pass; the one it comes closer to (the larger minimal
    # time at peak) binds and is reported, the other rides along
    alu_roof = {"bound": "alu", "achieved": achieved, "peak": peak, "unit": "Gtransitions/s",
                "frac": achieved / peak,
                "peak_source": f"{sms} SMs x 64 integer-ALU lanes x {MAX_SM_MHZ} MHz / "
                               f"{ALU_OPS_PER_TRANSITION} ALU instructions per transition",
                "peak_probe": roof[0] / 1e9,
                "peak_probe_source": "register-only loop of the 32-bit passes' op mix, "
                                     "all SMs, measured in this run",
                "peak_u64_probe": roof[1] / 1e9}
    hbm_roof = {"bound": "hbm", "achieved": dp_gbs, "peak": hbm_peak, "unit": "GB/s",
                "frac": dp_gbs / hbm_peak,
                "bytes_per_instance_direction": dp_bytes(L),
                "peak_source": "MEASURED_PEAKS.json hbm_gbs (copy, burst)"}
    # the whole library call per direction (counter reset, first pass, work-list
    # pass), against the same roofs
    call_gtps = trans / dp_s / 1e9
    call_gbs = 2 * dp_bytes(L) * B / dp_s / 1e9
    dp_call = {"ms_forward": fwd_ms, "ms_backward": bwd_ms,
               "alu_frac": call_gtps / peak, "hbm_frac": call_gbs / hbm_peak,
               "note": "the whole dc_schedule_* call per direction: counter reset, "
                       "first pass and work-list pass, all instances"}
    roofline = binding_roof(alu_roof, hbm_roof,
                            kernel=("first DP pass, forward + backward "
                                    f"({first_pass_kernel(L)}), timed on its own launches"),
                            kernel_ms={"forward": fwd_k_ms, "backward": bwd_k_ms},
                            listed_to_work_list={"forward": listed[0], "backward": listed[1]},
                            traffic=traffic, dp_call=dp_call)
    if traffic is None:
        roofline["traffic_note"] = ("no DRAM record in profiles/dp_traffic.json matches this "
                                    "workload and the current sources of its first-pass kernel")
    clocks = clk.summary() if rank == 0 else None
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "config": {"workload": args.workload, "batch_per_gpu": B, "L": L,
                   "global_batch": total,
                   "l2": f"inputs larger than L2: {B * (4 * L + 1) * 8 / 1e6:.0f} MB of "
                         "profiles written and re-read every step",
                   "parallelism": f"independent instances, {world} GPU(s), no collective"},
        "dp_cells_per_s": 2 * cells(L) * B * world / (ms * 1e-3),
        "dp_transitions_per_s": trans * world / (ms * 1e-3),
        "breakdown_ms": {"profile_gen": gen_ms, "dp_forward": fwd_ms, "dp_backward": bwd_ms,
                         "eval_timeline_fwd_bwd": eval_ms},
        "roofline": roofline,
        "e2e": e2e,
        "cpu_baseline": cpu,
        "gpu_launches": launches_per_step * args.steps,
        "timing": ("the step replayed from a CUDA graph (dynacomm.StepGraph), K replays"
                   if graph_ms is not None else
                   "eager launches" + (f" (graph capture failed: {graph_error})"
                                       if graph_error else "")),
        "eager": {"value": total / (eager_ms * 1e-3), "ms_per_step": eager_ms,
                  "note": "the same K steps as separate library calls; breakdown_ms is "
                          "measured on these"},
        "clocks": clocks,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


class _Null:
    def __enter__(self):
        return self

    def __exit__(self, *exc):
        return False

    def summary(self):
        return None


def run_e2e(dc, torch, prof, sched, B, L, W, dev, args, barrier, world):
    """Profiles in pinned host memory -> H2D -> forward + backward DP -> f_m of
    both -> D2H of makespans, decisions, segment counts and replays, every step,
    through dynacomm.HostPipeline (chunked: copies overlap the solves)."""
    # the pipeline's default pieces: one per 65,536 instances, 1 to 8 (ResNet-50:
    # 4 pieces measured twice as fast as 8)
    pipe = dc.HostPipeline(B, L, chunks=args.e2e_chunks or None, device=dev)
    host_in = {k: v.cpu().pin_memory() for k, v in prof.items()}
    # the gradient push of a layer moves its parameter tensor, so gt equals pt
    # (every workload here): the caller passes the one host buffer for both
    shared_xfer = bool(torch.equal(prof["pt"], prof["gt"]))
    if shared_xfer:
        host_in["gt"] = host_in["pt"]
    host_out = pipe.host_buffers()
    h2d, d2h = pipe.bytes_per_run(host_in)
    for _ in range(max(args.warmup, 1)):
        pipe.run(host_in, host_out)
    torch.cuda.synchronize()
    for d in (0, 1):  # the pipelined results equal the device-resident path's
        if not torch.equal(host_out[(d, "makespan")], sched.out[d]["makespan"].cpu()):
            raise RuntimeError("host pipeline disagrees with the device path")
    steps = max(1, min(args.steps, 10))
    barrier()
    # one event per step boundary on the caller's stream (each run ends by joining
    # its streams into it), so that the spread of the steps is visible too
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    ev[0].record()
    for s in range(steps):
        pipe.run(host_in, host_out)
        ev[s + 1].record()
    torch.cuda.synchronize()
    barrier()
    per_step = [ev[s].elapsed_time(ev[s + 1]) for s in range(steps)]
    ms = max_over_ranks(ev[0].elapsed_time(ev[steps]) / steps, dev)
    return {"value": B * world / (ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms, "steps": steps,
            "ms_step_min_max": [min(per_step), max(per_step)],
            "path": f"pinned host profiles -> dynacomm.HostPipeline ({pipe.chunks} "
                    f"piece{'s' if pipe.chunks != 1 else ''}, "
                    "copies overlapped with dc_schedule_forward/backward_batch and "
                    "dc_eval_timeline_batch) -> pinned host results",
            "inputs": "fc, pt, bc, dt; gt is the pt host buffer (equal transfer costs), "
                      "copied once" if shared_xfer else "fc, pt, bc, gt, dt"}


def main(argv=None):
    p = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=10)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", choices=list(wl.CONFIG_NAMES), default="vgg16")
    p.add_argument("--batch", type=int, default=0,
                   help="instances per GPU (default: the workload's batch); for profiling "
                        "small cases")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-graph", action="store_true",
                   help="time eager library calls only (no CUDA-graph replay of the step)")
    p.add_argument("--e2e-chunks", type=int, default=0,
                   help="host pipeline pieces for the e2e leg (0: one per 65,536 instances, 1 to 8)")
    p.add_argument("--lsweep", action="store_true",
                   help="scheduling time against depth L (GPU and one oracle core), one JSON line")
    p.add_argument("--compare", action="store_true",
                   help="DynaComm against Sequential, LBL and the greedy schedulers, one JSON line")
    p.add_argument("--fused", action="store_true",
                   help="generate-and-solve in one pass against the unfused path (L <= 16)")
    args = p.parse_args(argv)
    if args.fused:
        return run_fused(args)
    if args.lsweep:
        return run_lsweep(args)
    if args.compare:
        return run_compare(args)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
