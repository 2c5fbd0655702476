#!/usr/bin/env python
"""Benchmark of one SCOOT suggestion round on GB300.

A step is one pass of the whole scoring path over a resident candidate
pool: known-constraint pruning (Eq. 2) -> random-forest POF (Eq. 3) -> GP
posterior + acquisition (Section 4.3, Eq. 6 / Eq. 7, fused) -> top-q
(Section 4.7).  The default workload is the 8-parameter, 2-objective EHVI
configuration: d=8, n=64 observations, N=2^18 candidates, S=64 base
samples, 100 trees of depth <= 10, q=4.

Prints one JSON line.  `value` is candidates/s with the pool resident in HBM
(CUDA events on the launching stream, L2 flushed between steps); `e2e` is the
same metric through the C ABI from pinned host buffers (state preparation,
host->device copies and the read-back of the picks inside the timed
region); `roofline` is the dominant kernel's algorithmic work per launch
over its measured launch time; `cpu_baseline` is the fp64 oracle timed on a
bounded sample of the same workload on the host.

`--impl reference` times the oracle itself (the only reference this path
has: the paper ships no code) on bounded samples of the same workload.
Under torchrun (--gpus N > 1) each rank scores its own pool of N candidates
(weak scaling) and the ranks' top-q lists are all-gathered and merged.
"""
from __future__ import annotations

import argparse
import math
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "candidate configs scored/sec (prune+RF+GP+acq+top-q) and % FP32/HBM roofline"
UNIT = "candidates/s"
DEFAULT_WORKLOAD = "d12-fantasy"   # the largest workload (N = 2^22, q = 16 sequential picks)
SUBRUN_WORKLOADS = ("d10-ei", "d10-ehvi3")  # the N = 2^20 workloads, measured beside the headline
FLUSH_BYTES = 256 << 20   # > 129 MB of L2
FP32_LANES_PER_SM = 128

# DRAM bytes per launch from ncu (dram__bytes_read.sum + dram__bytes_write.sum),
# keyed by (kernel, workload), valid only while the kernel's sources are
# unchanged (sha256 prefix of their contents when the counters were taken).
KERNEL_FILES = {"prune": ["prune_rf.cu"], "rf": ["prune_rf.cu"],
                "score": ["score.cu", "posterior_tc.cu", "device_common.cuh"],
                "posterior": ["posterior_tc.cu", "device_common.cuh"], "fant_pass": ["fantasy.cu", "device_common.cuh"],
                "topq": ["topq.cu", "device_common.cuh"], "pareto": ["pareto.cu"]}
TRAFFIC = {
    # d12-fantasy: captured on a 2^20 pool of the same workload, scaled to the 2^22 launch by its
    # live candidates (x 4.0025; fant_pass and the posterior) or its pool size (x 4; prune, forest)
    ("fant_pass", "d12-fantasy"): {"bytes": 3561900000, "sha": "3e1f5ef592e904d1"},
    ("posterior", "d12-fantasy"): {"bytes": 3442600000, "sha": "fef1b84575f65e56"},
    ("rf", "d12-fantasy"): {"bytes": 227260000, "sha": "df8284c4f1f3b084"},
    ("prune", "d12-fantasy"): {"bytes": 100700000, "sha": "df8284c4f1f3b084"},
    ("score", "d10-ehvi3"): {"bytes": 44739000, "sha": "6b2aeb7ebc645ff4"},
}


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=DEFAULT_WORKLOAD)
    p.add_argument("--pool", type=int, default=None,
                   help="pool size instead of the workload's own (smaller cases for profiling)")
    p.add_argument("--kernel", choices=["matern52", "matern32"], default="matern52",
                   help="covariance (matern32 with --warp is the paper's own kernel)")
    p.add_argument("--warp", action="store_true", help="Kumaraswamy input warping of ordinal features")
    p.add_argument("--acq", choices=["default", "mace", "ehvi-exact"], default="default",
                   help="mace: UCB/PI/EI and a random subset of their Pareto front (one objective); "
                        "ehvi-exact: EHVI as the exact expectation (several objectives)")
    p.add_argument("--cpu-seconds", type=float, default=15.0, help="budget of the cpu_baseline sample")
    p.add_argument("--warmup-seconds", type=float, default=1.0, help="minimum warm-up time under load")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-extra", action="store_true",
                   help="skip the probes and the N = 2^20 workloads measured beside the headline")
    p.add_argument("--gp-prep", choices=["auto", "host", "device"], default="auto",
                   help="where the end-to-end step builds the GP state (fp64 factorisation); auto: the "
                        "device from 100 observations (measured faster there), the host below")
    p.add_argument("--stage", choices=["round", "rf-train", "gp-mle"], default="round",
                   help="rf-train: the training of the workload's feasibility forest; gp-mle: its GP "
                        "hyperparameter fit (32 starts x 100 Adam steps); instead of a round")
    return p.parse_args()


def workload_config(w, extra=None, acq=None, pool=None):
    acq = acq or w.acq
    pool = w.n_cand if pool is None else int(pool)
    desc = (f"{w.name}: d={w.d}, n={w.n_obs}, N={pool}, M={w.n_obj} {acq.upper()}"
            + (f" S={w.n_mc}" if w.acq == "ehvi" else "")
            + f", RF {w.n_trees} trees depth<={w.max_depth}, q={w.q}")
    cfg = {"workload": desc, "pool": pool, "observations": w.n_obs, "objectives": w.n_obj,
           "acquisition": acq, "trees": w.n_trees, "q": w.q,
           "l2": "flushed between steps (256 MiB write)", "inputs": "seeded synthetic pool, resident in HBM"}
    if extra:
        cfg.update(extra)
    return cfg


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "sm_max_mhz": 2070.0}, "fallback"


def referenced_columns(inst):
    cols = set()
    for c in inst.clauses:
        cols.update(int(c["guard_param"][g]) for g in range(int(c["n_guard"])))
        cols.update(int(c["term_param"][t]) for t in range(int(c["n_term"])))
    return len(cols)


def work_model(inst, n_boxes, acq_kind=None, n_grid=None):
    """Algorithmic work per candidate of each stage (bytes or flops)."""
    w = inst.workload
    acq_kind = acq_kind or w.acq
    d, n = inst.d, inst.n_obs
    m_eff = inst.n_obj if acq_kind in ("ehvi", "ehvi-exact") else 1
    post = m_eff * (n * (3 * d + 12) + 2 * n + n * (n + 1) + 2 * n)
    # EI ~30 flops; MACE adds PI (~15) and UCB (2); exact EHVI: ~12 flops per psi at each grid
    # coordinate and 2M per box
    if acq_kind == "ehvi-exact":
        acq = 12 * int(sum(n_grid)) + 2 * inst.n_obj * n_boxes
    else:
        acq = {"ei": 30, "mace": 47}.get(acq_kind, w.n_mc * n_boxes * 4 * inst.n_obj)
    return {
        "prune": ("hbm", 4 * referenced_columns(inst) + 1),
        "rf": ("hbm", 4 * d + 1 + 1 + 4),
        "score": ("alu", post + acq),
        "topq": ("hbm", 4 + 1),
        "pareto": ("hbm", 12 + 1),
    }


def fantasy_pass_bytes(inst, q, n_live):
    """Algorithmic DRAM bytes of each of the q passes of a fantasy round over
    n_live candidates: pass 0 reads the moments; pass j >= 1 also applies the
    downdate of pick j-1, reading the candidate's n rows of V per objective,
    its d configuration words and the j-1 earlier downdate factors, and
    writing the variance and (if a later downdate needs it) the new factor."""
    M, n, d = inst.n_obj, inst.n_obs, inst.d
    out = []
    for j in range(q):
        b = M * 8
        if j > 0:
            b += M * 4 * n + 4 * d + M * 4 * (j - 1) + M * 4 + (M * 4 if j - 1 < q - 2 else 0)
        out.append(b * n_live)
    return out


def posterior_flops(inst, n_obj=None):
    """Flops per candidate of the GP posterior (covariance row, mean,
    triangular product, variance), all objectives."""
    d, n = inst.d, inst.n_obs
    m = inst.n_obj if n_obj is None else n_obj
    return m * (n * (3 * d + 12) + 2 * n + n * (n + 1) + 2 * n)


def posterior_tensor_flops(inst, n_obj=None):
    """bf16 flops per candidate that the tensor-core posterior issues: per
    objective, k-block kb of 32 columns of L^{-1} reaches rows 32 kb .. n_pad - 1,
    and each of its 32 columns takes six part products (2 flops each)."""
    n_pad = 64 * ((inst.n_obs + 63) // 64)
    m = inst.n_obj if n_obj is None else n_obj
    return m * 6 * 2 * 32 * sum(n_pad - 32 * kb for kb in range(n_pad // 32))


def forest_visits(inst, idx):
    """Mean node visits (root to leaf, leaf included, summed over the trees)
    of the forest walk for the pool candidates idx, by a vectorised walk of
    the host copy of the trees: the work of one candidate in the forest kernel."""
    import numpy as np
    nodes, offs = inst.nodes, inst.tree_offset
    words = inst.cand[:, idx]
    x = np.empty(words.shape, np.float32)
    for c in range(inst.d):
        if int(inst.space[c]["kind"]) == 3:
            x[c] = words[c].view(np.float32)
        else:
            x[c] = words[c].view(np.int32).astype(np.float32)
    cols = np.arange(len(idx))
    total = 0
    for t in range(len(offs) - 1):
        base = int(offs[t])
        node = np.zeros(len(idx), np.int64)
        active = np.ones(len(idx), bool)
        while active.any():
            total += int(active.sum())
            rec = nodes[base + node]
            leaf = (rec["flags"] & 1).astype(bool)
            active &= ~leaf
            go = x[rec["feat"].astype(np.int64), cols] <= rec["val"]
            node = np.where(active, rec["left"].astype(np.int64) + np.where(go, 0, 1), node)
    return total / max(1, len(idx))


def measure_probes(S, ctx, device, stream, sms):
    """Measured peaks: FFMA and FFMA2 chains (TFLOP/s) and dependent node
    gathers from shared memory (visits/s), best of five timed launches."""
    import torch
    blocks = sms * 8
    sink = torch.zeros(blocks, device=device)

    def timed(fn):
        for _ in range(2):
            fn()
        best = float("inf")
        for _ in range(5):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fn()
            e1.record(stream)
            e1.synchronize()
            best = min(best, e0.elapsed_time(e1) / 1e3)
        return best
    iters, steps, n_nodes = 8192, 4096, 4095
    out = {}
    for packed, key in ((0, "ffma_tflops"), (1, "ffma2_tflops")):
        t = timed(lambda: S.scoot_probe_fma(ctx, packed, blocks, iters, sink, stream))
        out[key] = 2 * 16 * 256 * blocks * iters / t / 1e12
    t = timed(lambda: S.scoot_probe_gather(ctx, n_nodes, blocks, steps, sink, stream))
    out["smem_gather_visits_per_s"] = 256 * blocks * steps / t
    out["how"] = (f"{blocks} blocks x 256 threads; 16 independent FMA chains x {iters} steps per thread "
                  f"(scalar / packed pairs); {steps} dependent 8-byte node loads per thread from a "
                  f"{n_nodes}-node tree in shared memory; best of 5 launches, CUDA events")
    return out


def sub_run(name, steps=20, warmup=5):
    """The round of another workload, measured by this script in a child
    process (no CPU baseline, no end-to-end leg): its value, stage times and
    stage roofline fractions."""
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--workload", name, "--steps", str(steps),
           "--warmup", str(warmup), "--no-cpu-baseline", "--no-e2e", "--no-extra"]
    p = subprocess.run(cmd, capture_output=True, text=True, timeout=900)
    if p.returncode != 0:
        return {"error": p.stderr.strip().splitlines()[-1] if p.stderr.strip() else f"exit {p.returncode}"}
    line = json.loads(p.stdout.strip().splitlines()[-1])
    return {"workload": line["config"]["workload"], "value": line["value"], "unit": line["unit"],
            "ms_per_step": line["ms_per_step"], "stages_ms": line["stages_ms"],
            "stage_roofline_frac": line["stage_roofline_frac"], "clocks": line["clocks"],
            "stage_bounds": {"prune": "hbm", "rf": "hbm (effective bytes)", "score": "alu (FP32 peak)",
                             "topq": "hbm"}}


def sources_sha(stage):
    h = hashlib.sha256()
    for f in KERNEL_FILES[stage]:
        with open(os.path.join(ROOT, "paper_2408_04323_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


class ClockSampler:
    QUERY = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
             "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
             "clocks_event_reasons.sw_power_cap,utilization.gpu")

    def __init__(self):
        self.proc = None
        idx = os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[0].strip() or "0"
        self.gpu = idx if idx.isdigit() else "0"

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-i", self.gpu, "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        rows = []
        for line in out.splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 8:
                continue
            try:
                rows.append((float(f[0]), float(f[1]), f[3:7], float(f[7]) if f[7] not in ("", "[N/A]") else 0.0))
            except ValueError:
                continue
        loaded = [r for r in rows if r[3] > 0] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in loaded for i, v in enumerate(r[2]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in loaded) if loaded else None,
                "sm_max_mhz": max(r[1] for r in loaded) if loaded else None,
                "reasons": reasons, "samples": len(loaded)}


def _oracle_code(name, seed, n_sample, mace_kappa=None, acq=None, kernel=0, warp=False, start_at=None):
    """Python source that times the oracle's round on n_sample candidates of
    the workload (same round state) and prints {"seconds": t}: prune, forest,
    posterior, acquisition and top-q; for the fantasy workload the q
    sequential picks with refits; with mace_kappa the MACE round."""
    from workloads import WORKLOADS
    w = WORKLOADS[name]
    gp_opts = "kernel=%d, warp=%s" % (kernel, "warp_params(%r, %d)" % (name, seed) if warp else "None")
    if w.fantasy:
        select = ("feas = oracle.prune_mask(inst.space, inst.clauses, inst.cand, inst.n_cand)\n"
                  "v = oracle.rf_votes(inst.nodes, inst.tree_offset, inst.space, inst.cand, inst.n_cand)\n"
                  "w = inst.workload\n"
                  "feas &= oracle.pof_feasible(v, inst.n_trees, w.leaf_scale, w.delta_num, w.delta_den)\n"
                  "oracle.fantasy_picks(inst, w.q, feas, kernel=%d)\n" % kernel)
    elif mace_kappa is None:
        select = ("r = oracle.score_round(inst, %s, %s)\n" % (repr(acq) if acq else "inst.workload.acq", gp_opts) +
                  "oracle.select_topq(r['acq'], r['feasible'], inst.workload.q)\n")
    else:
        select = ("r = oracle.score_round(inst, 'ei', %s)\n" % gp_opts +
                  "A = oracle.mace_acquisitions(r['mu'][:, 0], r['var'][:, 0], float(inst.y_obs[0].max()), "
                  "1e-4, %r)\n"
                  "A[:, ~r['feasible']] = -np.inf\n"
                  "oracle.mace_select(A, r['feasible'], inst.workload.q, 0)\n" % float(mace_kappa))
    return ("import sys, time, json; sys.path.insert(0, %r)\n"
            "import numpy as np, oracle\n"
            "from workloads import make_instance, warp_params\n"
            "inst = make_instance(%r, %d, n_cand=%d)\n"
            "time.sleep(max(0.0, %r - time.time()))\n"
            "t = time.perf_counter()\n" % (ROOT, name, seed, n_sample, float(start_at or 0.0))
            + select
            + "print(json.dumps({'seconds': time.perf_counter() - t}))\n")


def _one_thread_env():
    return dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")


def cpu_oracle_sample(name, seed, n_sample, mace_kappa=None, acq=None, kernel=0, warp=False, wall=False):
    """Seconds of the oracle's round on n_sample candidates, one thread, in a
    fresh process (with wall: also the process's whole wall time)."""
    code = _oracle_code(name, seed, n_sample, mace_kappa, acq, kernel, warp)
    t0 = time.perf_counter()
    p = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=_one_thread_env(),
                       timeout=900)
    if p.returncode != 0:
        raise RuntimeError(p.stderr[-2000:])
    secs = json.loads(p.stdout.strip().splitlines()[-1])["seconds"]
    return (secs, time.perf_counter() - t0) if wall else secs


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_oracle_all_cores(name, seed, n_sample, procs, startup_s, **opts):
    """The oracle's round on n_sample candidates in each of `procs`
    one-thread processes at once (every core busy): the processes start
    their timers together, after their set-up; returns the slowest one's
    seconds (the throughput is procs * n_sample / seconds)."""
    code = _oracle_code(name, seed, n_sample, start_at=time.time() + 2.0 * startup_s + 2.0, **opts)
    ps = [subprocess.Popen([sys.executable, "-c", code], stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True,
                           env=_one_thread_env()) for _ in range(procs)]
    secs = []
    for p in ps:
        out, err = p.communicate(timeout=1800)
        if p.returncode != 0:
            raise RuntimeError(err[-2000:])
        secs.append(json.loads(out.strip().splitlines()[-1])["seconds"])
    return max(secs)


def calibrate_sample(name, seed, budget_s, mace_kappa=None, acq=None, kernel=0, warp=False):
    """Largest sample whose oracle round fits the budget (scaled from two
    probes), and the set-up seconds of one oracle process."""
    opts = dict(mace_kappa=mace_kappa, acq=acq, kernel=kernel, warp=warp)
    t1, w1 = cpu_oracle_sample(name, seed, 32, wall=True, **opts)
    t2 = cpu_oracle_sample(name, seed, 96, **opts)
    per = max((t2 - t1) / 64, 1e-6)
    fixed = max(t1 - 32 * per, 0.0)
    return max(16, int((budget_s - fixed) / per)), max(w1 - t1, 0.0)


def cpu_baseline_line(name, seed, budget_s, unit, **opts):
    """cpu_baseline: the oracle on a bounded sample of the workload, on one
    core and on every core of the host (one process per core)."""
    sample, startup = calibrate_sample(name, seed, budget_s, **opts)
    t1 = cpu_oracle_sample(name, seed, sample, **opts)
    procs = host_cores()
    tn = cpu_oracle_all_cores(name, seed, sample, procs, startup, **opts)
    from workloads import WORKLOADS
    what = ("prune, forest, then the q sequential EHVI picks with a GP refit per pick"
            if WORKLOADS[name].fantasy else "all five steps")
    return {"value": procs * sample / tn, "unit": unit, "cores": procs, "kind": "oracle",
            "value_one_core": sample / t1,
            "sample": f"{sample} candidates of the {name} pool (same round state) per process, {what}; "
                      f"fp64 numpy, one thread per process, {procs} processes at once (one core: "
                      f"{sample / t1:.4g} {unit})"}


def run_reference(args):
    """The reference arm: the oracle itself (the paper ships no code), each
    step a bounded sample of the workload on every host core (one one-thread
    process per core, timers started together)."""
    from workloads import WORKLOADS, seeds
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    w = WORKLOADS[args.workload]
    seed = seeds(w.name)[0]
    kappa = None
    if args.acq == "mace":
        from paper_2408_04323_gb300.pipeline import mace_beta
        kappa = mace_beta(w.n_obs)
    acq = "ehvi-exact" if args.acq == "ehvi-exact" else None
    kern = 1 if args.kernel == "matern32" else 0
    opts = dict(mace_kappa=kappa, acq=acq, kernel=kern, warp=args.warp)
    procs = host_cores()
    per_step = max(0.05, 100.0 / max(1, args.steps + args.warmup))
    sample, startup = calibrate_sample(w.name, seed, per_step, **opts)
    for _ in range(args.warmup):
        cpu_oracle_all_cores(w.name, seed, sample, procs, startup, **opts)
    times = [cpu_oracle_all_cores(w.name, seed, sample, procs, startup, **opts) for _ in range(args.steps)]
    ms = 1e3 * statistics.mean(times)
    value = procs * sample / (ms / 1e3)
    what = ("prune, forest, then the q sequential EHVI picks with a GP refit per pick" if w.fantasy
            else "all five steps")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(w, {"reference": "fp64 CPU oracle (the paper ships no code)",
                                          "sample_per_step": procs * sample, "kernel": args.kernel,
                                          "warp": bool(args.warp)},
                                      acq=None if args.acq == "default" else args.acq),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": procs, "kind": "oracle",
                             "sample": f"{sample} candidates of the {w.name} pool per process and step, {what}; "
                                       f"{procs} one-thread processes at once"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


RF_METRIC = "CART trees trained/sec (Algorithm 1's feasibility forest, exact split search)"
RF_UNIT = "trees/s"


def rf_train_inputs(name):
    """Observations, crash labels and T bootstrap samples of n draws of a workload."""
    import numpy as np
    from workloads import Stream, make_instance, seeds
    seed = seeds(name)[0]
    inst = make_instance(name, seed, n_cand=4)
    w = inst.workload
    n = w.n_obs
    labels = (inst.label_obs > 0.5).astype(np.uint8)
    boot = Stream(seed, "bootstrap").integers(0, n - 1, w.n_trees * n).reshape(w.n_trees, n).astype(np.int32)
    return inst, labels, boot


def rf_train_config(w, extra=None):
    cfg = {"workload": f"{w.name} forest: {w.n_trees} CART trees on bootstraps of n={w.n_obs} observations, "
                       f"d={w.d}, depth<={w.max_depth}",
           "trees": w.n_trees, "observations": w.n_obs, "max_depth": w.max_depth,
           "l2": "flushed between steps (256 MiB write)", "inputs": "seeded synthetic observations, resident in HBM"}
    cfg.update(extra or {})
    return cfg


def rf_oracle_seconds(name, trees):
    """The oracle's CART on the first `trees` bootstraps, in a fresh one-thread process."""
    code = ("import sys, time, json; sys.path.insert(0, %r)\n"
            "import numpy as np, oracle, bench\n"
            "inst, labels, boot = bench.rf_train_inputs(%r)\n"
            "w = inst.workload\n"
            "feats = oracle.decode(inst.space, inst.x_obs, w.n_obs).astype(np.float32)\n"
            "t = time.perf_counter()\n"
            "oracle.train_forest(feats, labels, boot[:%d], w.max_depth, w.leaf_scale)\n"
            "print(json.dumps({'seconds': time.perf_counter() - t}))\n" % (ROOT, name, trees))
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    p = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=900)
    if p.returncode != 0:
        raise RuntimeError(p.stderr[-2000:])
    return json.loads(p.stdout.strip().splitlines()[-1])["seconds"]


def rf_oracle_sample(name, budget_s, n_trees):
    t1 = rf_oracle_seconds(name, 1)
    k = int(min(n_trees, max(1, budget_s / max(t1, 1e-3))))
    return k, (rf_oracle_seconds(name, k) if k > 1 else t1)


def rf_list_entries(S, nodes, counts, feats, labels, boot, max_depth):
    """List entries the presorted split search touches on the trained trees:
    every node that searches (depth < max_depth, not pure) scans its m'
    samples in each of the d sorted lists, and every split node moves them
    into its children's lists."""
    import numpy as np
    recs = nodes.view(S.NODE_DTYPE)
    d = feats.shape[1]
    total = 0
    for t in range(len(counts)):
        tree = recs[t, :int(counts[t])]
        node = np.zeros(boot.shape[1], np.int64)
        depth = np.zeros(len(tree), np.int64)
        for k in range(len(tree)):
            sel = boot[t][node == k]
            mk, pk = len(sel), int(labels[sel].sum())
            if depth[k] < max_depth and 0 < pk < mk:
                total += d * mk
            if not (tree["flags"][k] & 1):
                total += d * mk
                left = int(tree["left"][k])
                depth[left] = depth[left + 1] = depth[k] + 1
                here = node == k
                go = feats[boot[t], int(tree["feat"][k])] <= tree["val"][k]
                node[here & go] = left
                node[here & ~go] = left + 1
    return total


def run_rf_train(args):
    import numpy as np
    import torch
    import paper_2408_04323_gb300 as pkg
    pkg.build()
    from paper_2408_04323_gb300 import scoot as S
    from workloads import CONTINUOUS, WORKLOADS
    if int(os.environ.get("WORLD_SIZE", "1")) > 1:
        raise SystemExit("--stage rf-train runs on one GPU")
    w = WORKLOADS[args.workload]
    inst, labels_np, boot_np = rf_train_inputs(w.name)
    n, T, d = w.n_obs, w.n_trees, w.d
    device = torch.device("cuda", 0)
    ctx = S.Context(0)
    h_obs = torch.from_numpy(np.ascontiguousarray(inst.x_obs[:, :n]).view(np.int32)).pin_memory()
    h_lab = torch.from_numpy(labels_np).pin_memory()
    h_boot = torch.from_numpy(boot_np).pin_memory()
    obs, lab, boot = h_obs.to(device), h_lab.to(device), h_boot.to(device)
    nodes = torch.zeros((T, 2 * n - 1), dtype=torch.int64, device=device)
    counts = torch.zeros(T, dtype=torch.int32, device=device)
    h_nodes = torch.empty(nodes.shape, dtype=torch.int64, pin_memory=True)
    h_counts = torch.empty(counts.shape, dtype=torch.int32, pin_memory=True)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=device)
    stream = torch.cuda.current_stream(device)

    work = torch.empty(S.scoot_rf_train_work_bytes(n, d), dtype=torch.uint8, device=device)

    def train(o=obs, la=lab, b=boot):
        S.scoot_rf_train(ctx, inst.space, o, n, la, b, w.max_depth, w.leaf_scale, nodes, counts, work, stream)

    sampler = ClockSampler()
    sampler.start()
    t_end = time.perf_counter() + args.warmup_seconds
    k = 0
    while k < max(3, args.warmup) or time.perf_counter() < t_end:
        flush.fill_(k & 0xFF)
        train()
        k += 1
    torch.cuda.synchronize(device)
    ctx.check(stream)
    tev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    for kk in range(args.steps):
        flush.fill_(kk & 0xFF)
        tev[kk][0].record(stream)
        train()
        tev[kk][1].record(stream)
    torch.cuda.synchronize(device)
    clocks = sampler.stop()
    ctx.check(stream)
    ms = statistics.mean(e[0].elapsed_time(e[1]) for e in tev)

    # end to end: inputs from pinned host memory, trees read back
    e2e = None
    if not args.no_e2e:
        d_obs, d_lab, d_boot = torch.empty_like(obs), torch.empty_like(lab), torch.empty_like(boot)
        times = []
        for kk in range(args.warmup + args.steps):
            flush.fill_(kk & 0xFF)
            torch.cuda.synchronize(device)
            t0 = time.perf_counter()
            d_obs.copy_(h_obs, non_blocking=True)
            d_lab.copy_(h_lab, non_blocking=True)
            d_boot.copy_(h_boot, non_blocking=True)
            train(d_obs, d_lab, d_boot)
            h_nodes.copy_(nodes, non_blocking=True)
            h_counts.copy_(counts, non_blocking=True)
            torch.cuda.synchronize(device)
            if kk >= args.warmup:
                times.append(time.perf_counter() - t0)
        e2e_s = statistics.mean(times)
        e2e = {"value": T / e2e_s, "unit": RF_UNIT,
               "h2d_bytes_per_step": int(h_obs.numel() * 4 + h_lab.numel() + h_boot.numel() * 4),
               "d2h_bytes_per_step": int(h_nodes.numel() * 8 + h_counts.numel() * 4), "ms_per_step": 1e3 * e2e_s}

    # roofline: one list entry per FP32/INT32 lane per clock
    peaks, peak_src = measured_peaks()
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    lane_peak = sms * FP32_LANES_PER_SM * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12  # Tops/s
    h_nodes.copy_(nodes)
    h_counts.copy_(counts)
    feats = np.stack([inst.x_obs[j, :n].view(np.float32) if int(inst.space[j]["kind"]) == CONTINUOUS
                      else inst.x_obs[j, :n].view(np.int32).astype(np.float32) for j in range(d)], axis=1)
    entries = rf_list_entries(S, h_nodes.numpy(), h_counts.numpy(), feats, labels_np, boot_np, w.max_depth)
    achieved = entries / (ms / 1e3) / 1e12
    roof = {"bound": "alu", "achieved": achieved, "peak": lane_peak, "unit": "Tentries/s",
            "frac": achieved / lane_peak, "traffic": None, "kernel": "rf_train",
            "peak_source": f"{peak_src} SM clock; one sorted-list entry per lane per clock = SMs x 128 x max SM "
                           "clock (the kernel is bound by the latency of its breadth-first node sequence)",
            "work_per_unit": entries / T, "units_per_launch": T}
    cpu = None
    if not args.no_cpu_baseline:
        k_, secs = rf_oracle_sample(w.name, args.cpu_seconds, T)
        cpu = {"value": k_ / secs, "unit": RF_UNIT, "cores": 1, "kind": "oracle",
               "sample": f"the first {k_} of the {T} trees, pure-Python breadth-first CART, one thread"}
    line = {"metric": RF_METRIC, "value": T / (ms / 1e3), "unit": RF_UNIT, "n_gpus": 1, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int32", "data": "synthetic",
            "config": rf_train_config(w, {"nodes": int(h_counts.sum()),
                                          "launch": "feature ranks, then one block per tree"}),
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": 2 * args.steps, "clocks": clocks}
    print(json.dumps(line), flush=True)
    ctx.close()


def run_rf_reference(args):
    from workloads import WORKLOADS
    if int(os.environ.get("RANK", "0")) != 0:
        return
    w = WORKLOADS[args.workload]
    per_step = max(0.5, 120.0 / max(1, args.steps + args.warmup))
    k, _ = rf_oracle_sample(w.name, per_step, w.n_trees)
    for _ in range(args.warmup):
        rf_oracle_seconds(w.name, k)
    times = [rf_oracle_seconds(w.name, k) for _ in range(args.steps)]
    ms = 1e3 * statistics.mean(times)
    value = k / (ms / 1e3)
    line = {"impl": "reference", "metric": RF_METRIC, "value": value, "unit": RF_UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": rf_train_config(w, {"reference": "CPU oracle (the paper ships no code)",
                                          "trees_per_step": k}),
            "cpu_baseline": {"value": value, "unit": RF_UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"the first {k} of the {w.n_trees} trees per step"},
            "e2e": {"value": value, "unit": RF_UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


MLE_METRIC = "GP log-marginal-likelihood evaluations with gradient/sec (hyperparameter MLE, projected Adam)"
MLE_UNIT = "evaluations/s"
MLE_STARTS, MLE_STEPS, MLE_LR = 32, 100, 0.05
FP64_NOMINAL_TFLOPS = 1.25  # GB300 FP64, nominal


def mle_inputs(name):
    """Observations of a workload and MLE_STARTS starts around its hyperparameters."""
    import numpy as np
    from workloads import Stream, make_instance, seeds
    inst = make_instance(name, seeds(name)[0], n_cand=4)
    M, P = inst.n_obj, inst.d + 2
    base = np.stack([np.concatenate([np.log(inst.lengthscale[m].astype(np.float64)),
                                     [0.0, math.log(max(float(inst.noise_var[m]), 1e-4))]]) for m in range(M)])
    lo, hi = np.full(P, -4.0), np.full(P, 3.0)
    lo[-1] = math.log(1e-4)
    theta0 = np.clip(base[None] + Stream(1, "mle-starts").normal(MLE_STARTS * M * P).reshape(MLE_STARTS, M, P) * 0.5,
                     lo, hi)
    return inst, theta0, lo, hi


def mle_flops(n, d):
    """fp64 flops of one evaluation: the elimination with L^-1 (n^3/3 multiply-adds), K^-1 (n^3/6), the
    two triangular products (n^2), and per pair of observations K's entry and the gradient's (6 d flops
    and two exponentials, counted as 30 flops each)."""
    return 2 * (n ** 3 / 3 + n ** 3 / 6 + n * n) + n * (n + 1) / 2 * (6 * d + 60)


def mle_oracle_seconds(name, evals):
    code = ("import sys, time, json; sys.path.insert(0, %r)\n"
            "import numpy as np, oracle, bench\n"
            "inst, theta0, lo, hi = bench.mle_inputs(%r)\n"
            "n = inst.n_obs\n"
            "t = time.perf_counter()\n"
            "for k in range(%d):\n"
            "    s, m = divmod(k, inst.n_obj)\n"
            "    oracle.log_marginal_likelihood(inst.space, inst.x_obs[:, :n], inst.y_obs[m], theta0[s %% len(theta0), m])\n"
            "print(json.dumps({'seconds': time.perf_counter() - t}))\n" % (ROOT, name, evals))
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    p = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=900)
    if p.returncode != 0:
        raise RuntimeError(p.stderr[-2000:])
    return json.loads(p.stdout.strip().splitlines()[-1])["seconds"]


def mle_config(inst, extra=None):
    w = inst.workload
    cfg = {"workload": f"{w.name} GP fit: n={w.n_obs} observations, d={w.d}, M={w.n_obj} objectives, "
                       f"{MLE_STARTS} starts x {MLE_STEPS} projected Adam steps (all parameters free)",
           "observations": w.n_obs, "objectives": w.n_obj, "starts": MLE_STARTS, "steps": MLE_STEPS,
           "inputs": "seeded synthetic observations, resident in HBM"}
    cfg.update(extra or {})
    return cfg


def run_gp_mle(args):
    import numpy as np
    import torch
    import paper_2408_04323_gb300 as pkg
    pkg.build()
    from paper_2408_04323_gb300 import scoot as S
    if int(os.environ.get("WORLD_SIZE", "1")) > 1:
        raise SystemExit("--stage gp-mle runs on one GPU")
    inst, theta0, lo, hi = mle_inputs(args.workload)
    n, d, M, P = inst.n_obs, inst.d, inst.n_obj, inst.d + 2
    device = torch.device("cuda", 0)
    ctx = S.Context(0)
    h_obs = torch.from_numpy(np.ascontiguousarray(inst.x_obs[:, :n]).view(np.int32)).pin_memory()
    h_y = torch.from_numpy(np.ascontiguousarray(inst.y_obs, np.float32)).pin_memory()
    h_t0 = torch.from_numpy(theta0).pin_memory()
    obs, y, t0 = h_obs.to(device), h_y.to(device), h_t0.to(device)
    th = torch.zeros_like(t0)
    lml = torch.zeros((MLE_STARTS, M), dtype=torch.float64, device=device)
    h_th = torch.empty(th.shape, dtype=torch.float64, pin_memory=True)
    h_lml = torch.empty(lml.shape, dtype=torch.float64, pin_memory=True)
    work = torch.empty(S.scoot_gp_mle_work_bytes(n, d, M, MLE_STARTS), dtype=torch.uint8, device=device)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=device)
    stream = torch.cuda.current_stream(device)
    free = (1 << P) - 1

    def fit(o=obs, yy=y, t=t0):
        S.scoot_gp_mle(ctx, inst.space, o, n, yy, t, lo, hi, free, MLE_STEPS, MLE_LR, th, lml, work=work,
                       stream=stream)

    sampler = ClockSampler()
    sampler.start()
    for k in range(max(3, args.warmup)):
        flush.fill_(k & 0xFF)
        fit()
    torch.cuda.synchronize(device)
    ctx.check(stream)
    steps = max(1, min(args.steps, 20))
    tev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(steps)]
    for kk in range(steps):
        flush.fill_(kk & 0xFF)
        tev[kk][0].record(stream)
        fit()
        tev[kk][1].record(stream)
    torch.cuda.synchronize(device)
    clocks = sampler.stop()
    ctx.check(stream)
    ms = statistics.mean(e[0].elapsed_time(e[1]) for e in tev)
    evals = MLE_STARTS * M * (MLE_STEPS + 1)
    e2e = None
    if not args.no_e2e:
        d_obs, d_y, d_t0 = torch.empty_like(obs), torch.empty_like(y), torch.empty_like(t0)
        times = []
        for kk in range(steps + 2):
            torch.cuda.synchronize(device)
            t_0 = time.perf_counter()
            d_obs.copy_(h_obs, non_blocking=True)
            d_y.copy_(h_y, non_blocking=True)
            d_t0.copy_(h_t0, non_blocking=True)
            fit(d_obs, d_y, d_t0)
            h_th.copy_(th, non_blocking=True)
            h_lml.copy_(lml, non_blocking=True)
            torch.cuda.synchronize(device)
            if kk >= 2:
                times.append(time.perf_counter() - t_0)
        e2e_s = statistics.mean(times)
        e2e = {"value": evals / e2e_s, "unit": MLE_UNIT,
               "h2d_bytes_per_step": int(h_obs.numel() * 4 + h_y.numel() * 4 + h_t0.numel() * 8),
               "d2h_bytes_per_step": int(h_th.numel() * 8 + h_lml.numel() * 8), "ms_per_step": 1e3 * e2e_s}
    achieved = mle_flops(n, d) * evals / (ms / 1e3) / 1e12
    roof = {"bound": "alu", "achieved": achieved, "peak": FP64_NOMINAL_TFLOPS, "unit": "TFLOP/s (fp64)",
            "frac": achieved / FP64_NOMINAL_TFLOPS, "traffic": None, "kernel": "gp_mle",
            "peak_source": "nominal GB300 FP64 rate (no measured fp64 peak on this pool)",
            "work_per_unit": mle_flops(n, d), "units_per_launch": evals}
    cpu = None
    if not args.no_cpu_baseline:
        one = mle_oracle_seconds(args.workload, 2) / 2
        k = max(2, int(args.cpu_seconds / max(one, 1e-4)))
        secs = mle_oracle_seconds(args.workload, k)
        cpu = {"value": k / secs, "unit": MLE_UNIT, "cores": 1, "kind": "oracle",
               "sample": f"{k} evaluations (likelihood and gradient) at the starts, numpy fp64, one thread"}
    line = {"metric": MLE_METRIC, "value": evals / (ms / 1e3), "unit": MLE_UNIT, "n_gpus": 1, "steps": steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": mle_config(inst, {"launch": "features, then one block per (start, objective) for the whole fit",
                                        "l2": "flushed between steps (256 MiB write)"}),
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": 2 * steps, "clocks": clocks}
    print(json.dumps(line), flush=True)
    ctx.close()


def run_mle_reference(args):
    if int(os.environ.get("RANK", "0")) != 0:
        return
    inst, theta0, lo, hi = mle_inputs(args.workload)
    one = mle_oracle_seconds(args.workload, 2) / 2
    per_step = max(0.5, 120.0 / max(1, args.steps + args.warmup))
    k = max(2, int(per_step / max(one, 1e-4)))
    for _ in range(args.warmup):
        mle_oracle_seconds(args.workload, k)
    times = [mle_oracle_seconds(args.workload, k) for _ in range(args.steps)]
    ms = 1e3 * statistics.mean(times)
    value = k / (ms / 1e3)
    line = {"impl": "reference", "metric": MLE_METRIC, "value": value, "unit": MLE_UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": mle_config(inst, {"reference": "CPU oracle (the paper ships no code)", "evaluations_per_step": k}),
            "cpu_baseline": {"value": value, "unit": MLE_UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"{k} evaluations per step"},
            "e2e": {"value": value, "unit": MLE_UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.stage == "rf-train":
        (run_rf_reference if args.impl == "reference" else run_rf_train)(args)
        return
    if args.stage == "gp-mle":
        (run_mle_reference if args.impl == "reference" else run_gp_mle)(args)
        return
    if args.impl == "reference":
        run_reference(args)
        return
    import numpy as np
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(device)

    import paper_2408_04323_gb300 as pkg
    pkg.build()
    from paper_2408_04323_gb300 import scoot as S
    from paper_2408_04323_gb300.pipeline import RoundInputs, ScoringRound, State
    from paper_2408_04323_gb300.shard import gather_mace_front, gather_topq, sharded_fantasy_picks
    from workloads import WORKLOADS, Stream, draw_configs, make_instance, seeds, warp_params

    w = WORKLOADS[args.workload]
    acq_kind = w.acq if args.acq == "default" else args.acq
    if acq_kind == "mace" and (w.n_obj != 1 or w.fantasy):
        raise SystemExit("--acq mace needs a one-objective workload")
    if acq_kind == "ehvi-exact" and (w.n_obj < 2 or w.fantasy):
        raise SystemExit("--acq ehvi-exact needs a multi-objective workload without fantasies")
    seed = seeds(w.name)[0]
    inst = make_instance(w.name, seed, n_cand=args.pool)
    cand_np = inst.cand
    if rank > 0:  # each rank scores a pool of its own; the round state is shared
        cand_np = draw_configs(w, Stream(seed, f"pool-rank{rank}"), inst.n_cand, inst.ld)
    N = inst.n_cand
    inp = RoundInputs(inst.space, inst.clauses, inst.nodes, inst.tree_offset, w.leaf_scale, w.delta_num,
                      w.delta_den, inst.x_obs, inst.y_obs, inst.lengthscale, inst.signal_var,
                      inst.noise_var, inst.ref, inst.eps, acq_kind, w.q, fantasy=w.fantasy,
                      kernel=S.MATERN32 if args.kernel == "matern32" else S.MATERN52,
                      warp=warp_params(w, seed) if args.warp else None)
    if args.warp and w.fantasy:
        raise SystemExit("--warp: fantasy picks take unwarped GP states")
    ctx = S.Context(device.index)
    gp_dev = (args.gp_prep == "device" or (args.gp_prep == "auto" and w.n_obs >= 100)) and not inp.fantasy
    rnd = ScoringRound(ctx, inp, N, device, gp_on_device=gp_dev)
    cand = torch.from_numpy(cand_np.view(np.int32)).to(device)
    stream = torch.cuda.current_stream(device)

    def exchange():
        """The ranks' only exchange after a step: their top-q lists, or for
        MACE their fronts (the fantasy round exchanges once per pick inside
        the step instead)."""
        if inp.fantasy:
            return
        if inp.acq == "mace":
            f = int(rnd.top_count[1].item())
            if f > rnd.front_cap:
                raise SystemExit(f"a front of {f} candidates exceeds the exchange's {rnd.front_cap}")
            gather_mace_front(rnd.acq3, rnd.front, f, rank * N, w.q, rnd.seed)
        else:
            gather_topq(rnd.top_idx, rnd.top_val, rnd.top_count, w.q)
    flush = torch.empty(FLUSH_BYTES, dtype=torch.uint8, device=device)
    st = rnd.state

    def step(evs=None, stream=stream):
        sp = S.scoot_prune
        if evs:
            evs[0].record(stream)
        sp(ctx, inp.space, inp.clauses, cand, N, rnd.mask, rnd.n_known, stream)
        if evs:
            evs[1].record(stream)
        S.scoot_rf_predict(ctx, st.forest_layout, st.forest, inp.space, cand, N, inp.delta_num,
                           inp.delta_den, rnd.votes, rnd.mask, rnd.n_feasible, stream)
        if evs:
            evs[2].record(stream)
        if inp.fantasy:
            if dist:  # the ranks' pools are shards of one pool of world x N candidates
                sharded_fantasy_picks(S, ctx, st.gp_layout, st.gp_state, st.fant_state, st.fant_box_cap, cand, N,
                                      st.eps, inp.q, rnd.work, rnd.top_idx, rnd.top_val, rnd.top_count,
                                      index_offset=rank * N, mask=rnd.mask, stream=stream)
            else:
                S.scoot_suggest_fantasy(ctx, st.gp_layout, st.gp_state, st.fant_state, st.fant_box_cap, cand, N,
                                        st.eps, inp.q, rnd.work, rnd.top_idx, rnd.top_val, rnd.top_count,
                                        mask=rnd.mask, stream=stream)
            if evs:
                evs[3].record(stream)
                evs[4].record(stream)
            return
        if inp.acq == "ei":
            S.scoot_score_ei(ctx, st.gp_layout, st.gp_state, cand, N, inp.xi, rnd.acq, rnd.mask, stream)
        elif inp.acq == "mace":
            S.scoot_score_mace(ctx, st.gp_layout, st.gp_state, cand, N, inp.xi, rnd.kappa, rnd.acq3, rnd.mask,
                               stream)
        elif inp.acq == "ehvi-exact":
            S.scoot_score_ehvi_exact(ctx, st.gp_layout, st.gp_state, cand, N, st.grid, st.n_grid, st.corner,
                                     rnd.acq, rnd.mask, stream)
        else:
            S.scoot_score_ehvi(ctx, st.gp_layout, st.gp_state, cand, N, st.box_lo, st.box_hi, st.eps,
                               rnd.acq, rnd.mask, stream)
        if evs:
            evs[3].record(stream)
        if inp.acq == "mace":
            S.scoot_select_pareto(ctx, rnd.acq3, N, inp.q, rnd.seed, rnd.top_idx, rnd.top_count, rnd.mask,
                                  rnd.front, stream)
        else:
            S.scoot_select_topq(ctx, rnd.acq, N, inp.q, rnd.top_idx, rnd.top_val, rnd.top_count, rnd.mask,
                                stream)
        if evs:
            evs[4].record(stream)

    sampler = ClockSampler()
    sampler.start()
    # warm-up: at least W steps and at least one second of load
    t_end = time.perf_counter() + args.warmup_seconds
    k = 0
    while k < max(3, args.warmup) or time.perf_counter() < t_end:
        flush.fill_(k & 0xFF)
        step()
        k += 1
        if k % 50 == 0:
            torch.cuda.synchronize(device)
    torch.cuda.synchronize(device)
    ctx.check(stream)
    n_feasible = int(rnd.n_feasible.item())
    if dist:
        dist.barrier()
    torch.cuda.synchronize(device)
    # Per-stage times from eagerly launched steps (diagnostic; they feed the roofline).
    n_diag = min(args.steps, 50)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(5)] for _ in range(n_diag)]
    phases = []  # the fantasy call's launches, timed by the library with events on the stream
    if inp.fantasy:
        S.scoot_ctx_set_timing(ctx, True)
    for kk in range(n_diag):
        flush.fill_(kk & 0xFF)
        step(evs[kk])
        if inp.fantasy:
            phases.append(S.scoot_ctx_phase_times(ctx))
    if inp.fantasy:
        S.scoot_ctx_set_timing(ctx, False)
    torch.cuda.synchronize(device)
    stage_names = ["prune", "rf", "score", "pareto" if inp.acq == "mace" else "topq"]
    stage_ms = {s: statistics.mean(e[i].elapsed_time(e[i + 1]) for e in evs) for i, s in enumerate(stage_names)}
    eager_ms = statistics.mean(e[0].elapsed_time(e[4]) for e in evs)

    # The step as one CUDA graph (its launches and memsets replayed without
    # host gaps).
    graph = None
    try:
        if dist and inp.fantasy:
            raise RuntimeError("the sharded fantasy round exchanges records between its launches")
        cap = torch.cuda.Stream(device)
        cap.wait_stream(stream)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=cap, capture_error_mode="thread_local"):
            step(stream=cap)
        torch.cuda.synchronize(device)
        for _ in range(3):
            graph.replay()
        torch.cuda.synchronize(device)
    except Exception as e:  # capture refused: time eager launches instead
        graph = None
        print(f"# CUDA graph capture unavailable ({e}); timing eager launches", file=sys.stderr)
        torch.cuda.synchronize(device)

    # The timed K steps.
    if dist:
        dist.barrier()
    torch.cuda.synchronize(device)
    tev = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(args.steps)]
    for kk in range(args.steps):
        flush.fill_(kk & 0xFF)
        tev[kk][0].record(stream)
        if graph is not None:
            graph.replay()
        else:
            step()
        tev[kk][1].record(stream)
        if dist:
            exchange()
    torch.cuda.synchronize(device)
    if dist:
        dist.barrier()
    clocks = sampler.stop()
    ctx.check(stream)
    step_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in tev)
    if dist:
        t = torch.tensor([step_ms], device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        step_ms = float(t.item())
    value = world * N / (step_ms / 1e3)

    # roofline of the dominant kernel
    peaks, peak_src = measured_peaks()
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    fp32_peak = sms * FP32_LANES_PER_SM * 2 * peaks.get("sm_max_mhz", 2070.0) * 1e6 / 1e12  # TFLOP/s
    hbm = peaks["hbm_gbs"]
    work = work_model(inst, st.n_boxes, inp.acq, getattr(st, "n_grid", None))
    n_known = int(rnd.n_known.item())

    def hbm_roof(bytes_per_launch, launch_ms, name):
        a = bytes_per_launch / (launch_ms / 1e3) / 1e9
        return {"bound": "hbm", "achieved": a, "peak": hbm, "unit": "GB/s", "frac": a / hbm, "kernel": name,
                "work_per_launch": bytes_per_launch, "launch_ms": launch_ms}

    def alu_roof(flops_per_launch, launch_ms, name):
        a = flops_per_launch / (launch_ms / 1e3) / 1e12
        return {"bound": "alu", "achieved": a, "peak": fp32_peak, "unit": "TFLOP/s", "frac": a / fp32_peak,
                "kernel": name, "work_per_launch": flops_per_launch, "launch_ms": launch_ms}

    def tensor_roof(bf16_flops, launch_ms):
        bf16 = peaks.get("bf16_tflops") if peaks else None
        a = bf16_flops / (launch_ms / 1e3) / 1e12
        return {"bf16_flops_per_launch": bf16_flops, "achieved_tflops": a, "peak_tflops": bf16,
                "frac": a / bf16 if bf16 else None,
                "peak_source": "measured (MEASURED_PEAKS.json bf16_tflops, burst)" if bf16 else None,
                "note": "the work above counts the fp32-equivalent product once; the tensor cores run six bf16 "
                        "part products of it"}
    kernels = {}
    for s_ in ("prune", "rf"):
        k_, pc = work[s_]
        kernels[s_] = hbm_roof(pc * N, stage_ms[s_], s_)
    if inp.fantasy:
        def mean_of(kind):
            v = [sum(ms for k, ms in ph if k == kind) for ph in phases]
            c = [sum(1 for k, _ in ph if k == kind) for ph in phases]
            return statistics.mean(v), max(1, c[0])
        post_ms, _ = mean_of("posterior")
        pass_ms, n_pass = mean_of("fant_pass")
        pick_ms, n_pick = mean_of("fant_pick")
        init_ms, _ = mean_of("fant_init")
        kernels["posterior"] = alu_roof(posterior_flops(inst) * n_feasible, post_ms, "posterior (whitened rows)")
        if 64 * ((inst.n_obs + 63) // 64) <= 256:  # the L^{-1} k product runs on the tensor cores
            kernels["posterior"]["tensor"] = tensor_roof(posterior_tensor_flops(inst) * n_feasible, post_ms)
        pb = fantasy_pass_bytes(inst, inp.q, n_feasible)[:n_pass]
        kernels["fant_pass"] = hbm_roof(statistics.mean(pb), pass_ms / n_pass, "fant_pass")
        kernels["fant_pass"]["launches_per_step"] = n_pass
        kernel_ms = {"prune": stage_ms["prune"], "rf": stage_ms["rf"], "posterior": post_ms,
                     "fant_pass": pass_ms, "fant_pick": pick_ms + init_ms}
    else:
        k_, pc = work["score"]
        kernels["score"] = alu_roof(pc * n_feasible, stage_ms["score"], "score")
        if inp.acq in ("ei", "mace") and 64 * ((inst.n_obs + 63) // 64) <= 256:
            # posterior and acquisition in the tensor-core kernel (objective 0)
            kernels["score"]["tensor"] = tensor_roof(posterior_tensor_flops(inst, 1) * n_feasible, stage_ms["score"])
        last = "pareto" if inp.acq == "mace" else "topq"
        kernels[last] = hbm_roof(work[last][1] * N, stage_ms[last], last)
        kernel_ms = {k: stage_ms[k] for k in stage_names}
    dom = max((k for k in kernels), key=lambda k: kernel_ms[k] if k in kernel_ms else 0.0)
    tag = w.name if inp.acq == w.acq and args.pool in (None, w.n_cand) else None
    for k, v in kernels.items():  # DRAM bytes per launch from ncu, while the kernel's sources are unchanged
        tr = TRAFFIC.get((k, tag))
        v["traffic"] = tr["bytes"] if tr and tr["sha"] == sources_sha(k) else None
    roof = dict(kernels[dom])
    roof["peak_source"] = (f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if roof["bound"] == "hbm" else
                           "FP32 = SMs x 128 lanes x 2 x max SM clock (nominal; measured FFMA peaks in probes)")
    stage_roofs = {k: round(v["frac"], 4) for k, v in kernels.items()}
    probes = None
    if not args.no_extra and rank == 0:
        probes = measure_probes(S, ctx, device, stream, sms)
        for k, v in kernels.items():
            if v["bound"] == "alu":
                v["frac_of_measured_ffma2"] = v["achieved"] / max(probes["ffma_tflops"], probes["ffma2_tflops"])
        # the forest's true bound: node visits against the shared-memory gather peak
        st_ = Stream(seed, "visit-sample")
        mask_k = torch.empty(N, dtype=torch.uint8, device=device)
        S.scoot_prune(ctx, inp.space, inp.clauses, cand, N, mask_k, None, stream)
        known = np.nonzero(mask_k.cpu().numpy())[0]
        samp = known[(st_.u64(4096) % np.uint64(max(1, len(known)))).astype(np.int64)] if len(known) else known
        visits = forest_visits(inst, samp) * n_known
        rate = visits / (stage_ms["rf"] / 1e3)
        kernels["rf"].update({"node_visits_per_launch": visits, "node_visits_per_s": rate,
                              "frac_of_smem_gather_peak": rate / probes["smem_gather_visits_per_s"]})
        if inp.fantasy:
            kernels["fant_pass"]["ehvi_flops_per_launch"] = n_feasible * inp.eps.shape[0] * st.n_boxes * 4 * inst.n_obj
        roof = dict(kernels[dom], peak_source=roof["peak_source"])

    # end to end through the C ABI from pinned host buffers
    e2e = None
    if not args.no_e2e:
        host_pool = torch.from_numpy(cand_np.view(np.int32)).pin_memory()
        cand_e2e = torch.empty_like(cand)
        h2d = host_pool.numel() * 4
        copy_stream = torch.cuda.Stream(device)
        pinned_picks = (torch.empty(rnd.top_idx.shape, dtype=rnd.top_idx.dtype, pin_memory=True),
                        torch.empty(rnd.top_val.shape, dtype=rnd.top_val.dtype, pin_memory=True),
                        torch.empty(rnd.top_count.shape, dtype=rnd.top_count.dtype, pin_memory=True))
        times = []
        for kk in range(args.warmup + args.steps):
            flush.fill_(kk & 0xFF)
            torch.cuda.synchronize(device)
            t0 = time.perf_counter()
            # the pool's upload overlaps the host preparation of the round state
            copy_stream.wait_stream(stream)
            with torch.cuda.stream(copy_stream):
                (cand if graph is not None else cand_e2e).copy_(host_pool, non_blocking=True)
            # host preparation through the C ABI + one upload (into the captured
            # step's state buffer when the step is replayed as a graph)
            state = State(inp, device, into=st if graph is not None else None, gp_on_device=gp_dev, ctx=ctx)
            stream.wait_stream(copy_stream)
            if graph is not None:
                graph.replay()
                for dst, src in zip(pinned_picks, (rnd.top_idx, rnd.top_val, rnd.top_count)):
                    dst.copy_(src, non_blocking=True)
                picks = pinned_picks
                if dist:
                    exchange()
                torch.cuda.synchronize(device)
                if kk >= args.warmup:
                    times.append(time.perf_counter() - t0)
                continue
            S.scoot_prune(ctx, inp.space, inp.clauses, cand_e2e, N, rnd.mask, None, stream)
            S.scoot_rf_predict(ctx, state.forest_layout, state.forest, inp.space, cand_e2e, N, inp.delta_num,
                               inp.delta_den, rnd.votes, rnd.mask, None, stream)
            if inp.fantasy and dist:
                sharded_fantasy_picks(S, ctx, state.gp_layout, state.gp_state, state.fant_state, state.fant_box_cap,
                                      cand_e2e, N, state.eps, inp.q, rnd.work, rnd.top_idx, rnd.top_val,
                                      rnd.top_count, index_offset=rank * N, mask=rnd.mask, stream=stream)
            elif inp.fantasy:
                S.scoot_suggest_fantasy(ctx, state.gp_layout, state.gp_state, state.fant_state, state.fant_box_cap,
                                        cand_e2e, N, state.eps, inp.q, rnd.work, rnd.top_idx, rnd.top_val,
                                        rnd.top_count, mask=rnd.mask, stream=stream)
            elif inp.acq == "ei":
                S.scoot_score_ei(ctx, state.gp_layout, state.gp_state, cand_e2e, N, inp.xi, rnd.acq, rnd.mask, stream)
            elif inp.acq == "mace":
                S.scoot_score_mace(ctx, state.gp_layout, state.gp_state, cand_e2e, N, inp.xi, rnd.kappa, rnd.acq3,
                                   rnd.mask, stream)
                S.scoot_select_pareto(ctx, rnd.acq3, N, inp.q, rnd.seed, rnd.top_idx, rnd.top_count, rnd.mask,
                                      rnd.front, stream)
            elif inp.acq == "ehvi-exact":
                S.scoot_score_ehvi_exact(ctx, state.gp_layout, state.gp_state, cand_e2e, N, state.grid, state.n_grid,
                                         state.corner, rnd.acq, rnd.mask, stream)
            else:
                S.scoot_score_ehvi(ctx, state.gp_layout, state.gp_state, cand_e2e, N, state.box_lo, state.box_hi,
                                   state.eps, rnd.acq, rnd.mask, stream)
            if not inp.fantasy and inp.acq != "mace":
                S.scoot_select_topq(ctx, rnd.acq, N, inp.q, rnd.top_idx, rnd.top_val, rnd.top_count, rnd.mask,
                                    stream)
            for dst, src in zip(pinned_picks, (rnd.top_idx, rnd.top_val, rnd.top_count)):
                dst.copy_(src, non_blocking=True)
            picks = pinned_picks
            if dist:
                exchange()
            torch.cuda.synchronize(device)
            if kk >= args.warmup:
                times.append(time.perf_counter() - t0)
        state_bytes = state.upload_bytes  # the one upload: GP state (or its inputs), forest, boxes
        e2e_s = statistics.mean(times)
        if dist:
            t = torch.tensor([e2e_s], device=device)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            e2e_s = float(t.item())
        e2e = {"value": world * N / e2e_s, "unit": UNIT, "h2d_bytes_per_step": int(h2d + state_bytes),
               "d2h_bytes_per_step": int(sum(p.numel() * p.element_size() for p in picks)),
               "ms_per_step": 1e3 * e2e_s}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        kappa = rnd.kappa if inp.acq == "mace" else None
        acq = "ehvi-exact" if inp.acq == "ehvi-exact" else None
        cpu = cpu_baseline_line(w.name, seed, args.cpu_seconds, UNIT, mace_kappa=kappa, acq=acq, kernel=inp.kernel,
                                warp=args.warp)
    extra = None
    if rank == 0 and world == 1 and not args.no_extra:
        extra = {name: sub_run(name) for name in SUBRUN_WORKLOADS if name != w.name}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "f32", "data": "synthetic",
                "config": workload_config(w, {"feasible": n_feasible, "boxes": st.n_boxes,
                                              "front": st.front_size, "parallelism": f"pool shards x{world}",
                                              "launch": "CUDA graph of the step" if graph is not None
                                              else "eager launches",
                                              "eager_ms_per_step": round(eager_ms, 5),
                                              "kernel": args.kernel, "warp": bool(args.warp),
                                              "e2e_gp_state": "built on the device" if gp_dev else
                                              "built on the host"}, acq=inp.acq, pool=N),
                "roofline": roof, "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": args.steps * rnd.kernels_per_round(),
                "clocks": clocks, "stages_ms": {k: round(v, 5) for k, v in stage_ms.items()},
                "kernels_ms": {k: round(v, 5) for k, v in kernel_ms.items()},
                "stage_roofline_frac": stage_roofs, "kernels": kernels, "peaks_measured_here": probes,
                "at_2_20": extra}
        print(json.dumps(line), flush=True)
    ctx.close()
    if dist:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
