#!/usr/bin/env python3
"""Benchmark of the SubZero+ weight path on GB300: ZO steps/s and weight-pass HBM GB/s.

Default workload: the LLaMA-7B-shaped parameter set (224 bf16 matrices, 6.48 G
parameters, r = 32, q = 4 queries, central differences -> 2q + 1 = 9 weight
passes per step, subspace refresh every 25 steps).  One "step" is Alg. 3's
iteration for every matrix: the 2q perturbation passes (+Z0, -2Z0, +Z0+Z1, ...,
-2Z_{q-1}, a loss evaluation after each), the subspace-Adam update fused with the
last restore, and (when t mod F == 0) the batched QR refresh.  The losses
the forward passes would produce are synthetic (2.0 + 0.01 N(0,1)); the weights
are N(0, 0.02^2) bf16.  25.9 GB of weights per pass is far larger than the
129 MB L2, so every pass streams from HBM.

  python bench.py [--gpus N --steps K --warmup W] [--impl reference] [--workload NAME]

Prints ONE JSON line (rank 0).  For N > 1 launch with torch.distributed.run:
each rank runs its own layer partition (matrix indices rank*n .. rank*n+n-1 of an
N-times larger set) with no data-path collective; NCCL is used only for the
barrier and the max over ranks of the timed region.
"""

import argparse
import hashlib
import re
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "ZO weight-pass HBM GB/s (% of peak) and ZO steps/s at 7B shape, 1 GB300"
FALLBACK_HBM_GBS = 6800.0

# dram__bytes_read.sum + dram__bytes_write.sum per launch of the weight-pass kernel,
# from the ncu capture summarised under profiles/, keyed by the sha256 of the kernel
# source it was taken on (reported as null once the source differs).
L2_BYTES = 129e6          # GB300 L2 capacity
TRAFFIC_BY_SOURCE = {
    # code hash of the kernel that runs (comments ignored) -> dram read + write bytes of one
    # launch, from an ncu capture on a small case of the same workload, scaled by weights
    # profiles/wpass_tc_r32_llama7b_2layers.md: 1.5779 GB on the 2-layer subset, x16.0
    ("a733f29ccdac1cbd", "llama7b_bf16_r32"): 25.25e9,
    # profiles/wpass_pair_r128_llama7b_2layers.md: 1.6392 GB on the 2-layer subset, x16.0
    ("45f2d025ab358fe7", "llama7b_bf16_r128_q99"): 26.23e9,
    # profiles/wpass_tmem_r64_dense32b_1layer.md: 1.9271 GB on the 1-layer subset, x64.0
    ("5d6c6cd8669a0a74", "dense32b_bf16_r64"): 123.33e9,
}
# thread instructions per weight of the full-space SPSA kernel (ncu), keyed by source hash
INSTR_PER_WEIGHT_BY_SOURCE = {
    # profiles/mezo_kernel_llama7b_2layers.md: 751.9 M warp instructions x 32 / 404.75 M weights
    "a1a0ede2c35a3971": 59.4,
}


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=25)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="llama7b_bf16_r32")
    p.add_argument("--scheme", choices=["central", "forward"], default="central")
    p.add_argument("--method", choices=["subzero", "mezo", "linear"], default="subzero",
                   help="subzero: the SubZero+ step (default); mezo: the full-space SPSA "
                        "baseline of Eq. (1), 3 passes per step; linear: the linear layers of "
                        "one layer evaluated at the perturbed weights without a weight pass "
                        "(zo_linear_perturbed), --tokens rows of activations")
    p.add_argument("--tokens", type=int, default=4096,
                   help="--method linear: activation rows T per linear layer")
    p.add_argument("--layers", type=int, default=0,
                   help="use only the first N layers of the workload (shape-preserving subset, "
                        "for profiling captures); 0 = all")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--single-sm", action="store_true",
                   help="r = 128: run the single-SM weight-pass kernel instead of the SM-pair one "
                        "(ZO_OPTION_PAIR_MMA = 0; the two give the same bits)")
    p.add_argument("--no-secondary", action="store_true",
                   help="skip the second measurement on the 32B-shaped set (default workload only)")
    p.add_argument("--oracle-sample", action="store_true",
                   help="internal: print one timing of the oracle's bounded sample as JSON and exit "
                        "(run in a single-thread subprocess for cpu_baseline.single_thread)")
    return p.parse_args()


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def _code_hash(names):
    """sha256 (16 hex) of CUDA sources with comments and blank space removed, so that a
    comment edit keeps the hash of the code the ncu counters were taken on."""
    h = hashlib.sha256()
    for name in names:
        path = os.path.join(ROOT, "paper_2608_15665_gb300", "csrc", name)
        if not os.path.exists(path):
            continue
        text = open(path, encoding="utf-8").read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()[:16]


def kernel_source_hash(r=32):
    """Code hash of the tensor-core weight-pass kernel that runs at rank r (r <= 32:
    zo_wpass_tc.cu, r = 64: zo_wpass_tmem.cu, r = 128: zo_wpass_pair.cu) and the headers
    it includes."""
    kernel = "zo_wpass_tc.cu" if r <= 32 else "zo_wpass_tmem.cu" if r == 64 else "zo_wpass_pair.cu"
    headers = ("zo_tc_common.cuh", "zo_sm100.cuh", "zo_device.cuh")
    if r == 128:
        headers += ("zo_cluster.cuh",)
    return _code_hash((kernel,) + headers)


def subset(wl, layers):
    """The first `layers` layers of a workload (its matrices repeat per layer)."""
    if not layers:
        return wl
    from paper_2608_15665_gb300 import workloads
    per_layer = {"opt1.3b_bf16_r16": 6, "llama7b_bf16_r32": 7, "dense32b_bf16_r64": 7,
                 "llama7b_bf16_r128_q99": 7, "llama13b_bf16_r128_q99": 7,
                 "lora_opt13b_f32_r4": 4, "single256_f32_r8": 1}[wl.name]
    k = min(len(wl.shapes), layers * per_layer)
    return workloads.scaled(wl, name=f"{wl.name}[{layers} layers]", shapes=wl.shapes[:k],
                            zero_init=[i for i in wl.zero_init if i < k])


def mezo_source_hash():
    return _code_hash(("zo_mezo.cu", "zo_device.cuh"))


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples every 200 ms while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(prefix="zo_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for nm, v in zip(names, parts[5:9]):
                    if v.lower().startswith("active"):
                        reasons.add(nm)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------- oracle timing
def oracle_sample(wl):
    """The bounded sample both oracle legs time: 1024 rows of matrix 0 and, where the set
    has one, 1024 rows of matrix 4 (the first wide projection of a LLaMA-shaped layer)."""
    return ((0, 1024), (4, 1024)) if wl.n_mats > 4 else ((0, 1024),)


def oracle_sample_step_seconds(wl, scheme, sample=((0, 1024),), seed_shift=0):
    """Time the fp64 oracle, as it stands, on a bounded sample of one step: for each
    (matrix, n_rows) in ``sample``, the refresh of that matrix (Alg. 1 on its full m x r
    and n x r panels) and every weight pass of the step (perturbations, estimator,
    Adam, fused update) on n_rows of its rows (rows of W update independently).
    Returns (step_seconds, refresh_seconds, sample_text, cores) extrapolated to the
    workload: passes by weight count, refresh by panel rows m + n; cores = process CPU
    time / wall time over the timed work (the threads the oracle actually kept busy)."""
    import numpy as np
    import torch
    from oracle import subzero
    from paper_2608_15665_gb300 import workloads
    t_pass = t_ref = 0.0
    el_sample = uv_sample = 0
    used = []                                      # (matrix, rows actually sampled)
    cpu_s = wall_s = 0.0
    seed = wl.seed + seed_shift
    for i, n_rows in sample:
        m, n = wl.shapes[i]
        rows = np.arange(min(n_rows, m))
        W0 = workloads.init_weight(wl, i, "cpu")[: rows.size].to(torch.float64).numpy()
        st = subzero.MatrixState(W0, wl.dtype, wl.r)
        st.m = m                                   # the panels keep the matrix's full shape
        t0, c0 = time.perf_counter(), time.process_time()
        subzero.refresh(st, seed, i, 0, reset_moments=True)
        t_ref += time.perf_counter() - t0
        cpu_s += time.process_time() - c0
        losses = workloads.loss_table(wl, scheme, steps=1)[0]
        passes, restore = subzero.pass_plan(scheme, wl.q)
        t0, c0 = time.perf_counter(), time.process_time()
        for terms in passes:
            C = subzero.perturb_coeff(seed, i, 0, wl.r, terms, wl.eps)
            st.W = subzero.apply_pass(st.W, wl.dtype, st.U, st.V, C, rows=rows)
        rho = subzero.rho_from_losses(losses, scheme, wl.eps, wl.q)
        G = subzero.grad_G(seed, i, 0, wl.r, rho)
        st.M, st.Vm, D, _, _ = subzero.adam(st.M, st.Vm, G, wl.beta1, wl.beta2, wl.eps_adam, 1)
        C = subzero.step_coeff(D, wl.lr, wl.eps, restore, seed, i, 0, wl.r)
        st.W = subzero.apply_pass(st.W, wl.dtype, st.U, st.V, C, rows=rows)
        t_pass += time.perf_counter() - t0
        cpu_s += time.process_time() - c0
        el_sample += rows.size * n
        uv_sample += m + n
        used.append((i, rows.size))
    step_s = t_pass * wl.params / el_sample
    refresh_s = t_ref * sum(m + n for m, n in wl.shapes) / uv_sample
    text = ("fp64 oracle, one step: all weight passes + estimator + Adam on "
            + ", ".join(f"{r} rows of matrix {i} {wl.shapes[i][0]}x{wl.shapes[i][1]}" for i, r in used)
            + f" ({el_sample} of {wl.params} weights) and the refresh of those matrices; "
            f"EXTRAPOLATED to the whole set by weight count (refresh by m+n, amortized over "
            f"F={wl.F})")
    cores = round(cpu_s / (t_pass + t_ref), 1) if t_pass + t_ref > 0 else 1.0
    return step_s, refresh_s, text, cores, t_pass + t_ref


def oracle_single_thread(wl_name, scheme):
    """The same oracle sample timed in a fresh interpreter pinned to one BLAS / OpenMP
    thread (a spawned process: nothing CUDA is inherited).  Returns its JSON or None."""
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "NUMEXPR_NUM_THREADS",
              "VECLIB_MAXIMUM_THREADS"):
        env[k] = "1"
    for k in ("RANK", "LOCAL_RANK", "WORLD_SIZE"):
        env.pop(k, None)
    try:
        res = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-sample",
                              "--workload", wl_name, "--scheme", scheme],
                             capture_output=True, text=True, env=env, timeout=600)
        return json.loads(res.stdout.strip().splitlines()[-1]) if res.returncode == 0 else None
    except Exception:
        return None


def run_oracle_sample(args):
    from paper_2608_15665_gb300 import workloads
    wl = workloads.get(args.workload)
    step_s, refresh_s, text, cores, _ = oracle_sample_step_seconds(wl, args.scheme,
                                                                   sample=oracle_sample(wl))
    print(json.dumps({"value": 1.0 / (step_s + refresh_s / wl.F), "cores": cores}), flush=True)


def cpu_baseline(wl, scheme):
    step_s, refresh_s, text, cores, _ = oracle_sample_step_seconds(wl, scheme,
                                                                   sample=oracle_sample(wl))
    per_step = step_s + refresh_s / wl.F
    one = oracle_single_thread(wl.name, scheme)
    return {"value": 1.0 / per_step, "unit": "ZO steps/s", "cores": cores,
            "host_cores": os.cpu_count(), "kind": "oracle", "sample": text, "extrapolated": True,
            "single_thread": ({"value": one["value"], "unit": "ZO steps/s", "cores": one["cores"],
                               "threads": "1 BLAS / OpenMP thread"} if one else None)}


def max_over_ranks(x, world, device):
    """The largest x over the ranks (one all_reduce MAX on the process group); x itself on
    one rank.  The job takes as long as its slowest rank."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_steps_per_second(ms_per_step, world):
    """Whole-job ZO steps/s of a layer-partitioned run: every rank steps its own partition
    (weak scaling), so the job completes `world` partitions' steps per ms_per_step."""
    return world * 1e3 / ms_per_step


def amortise_refresh(window_ms, K, t0, F, refresh_ms):
    """ms per step of a window of K steps t0 .. t0 + K - 1 with the refreshes it held (steps
    t with t mod F == 0) replaced by refresh_ms / F per step."""
    n_ref = sum(1 for t in range(t0, t0 + K) if t % F == 0)
    return (window_ms - n_ref * refresh_ms) / K + refresh_ms / F


# --------------------------------------------------------------------------- reference arm
def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2608_15665_gb300 import workloads
    wl = workloads.get(args.workload)
    times, cores, sample_s = [], [], []
    for s in range(args.warmup + args.steps):
        step_s, refresh_s, text, c, spent = oracle_sample_step_seconds(
            wl, args.scheme, sample=oracle_sample(wl), seed_shift=s)
        if s >= args.warmup:
            times.append(step_s + refresh_s / wl.F)
            cores.append(c)
            sample_s.append(spent)
    per_step = sum(times) / len(times)
    value = 1.0 / per_step
    passes = 2 * wl.q + 1 if args.scheme == "central" else wl.q + 1
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "ZO steps/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": per_step * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.name, "matrices": wl.n_mats, "params": wl.params, "r": wl.r,
                   "q": wl.q, "scheme": args.scheme, "passes_per_step": passes,
                   "refresh_every": wl.F},
        "cpu_baseline": {"value": value, "unit": "ZO steps/s", "cores": max(cores),
                         "host_cores": os.cpu_count(), "kind": "oracle", "sample": text,
                         "extrapolated": True},
        "e2e": {"value": value, "unit": "ZO steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        # ms_per_step is the whole set's step, extrapolated from the timed sample; the time
        # this run actually spent per step is the sample's
        "extrapolation": {"sample_seconds_per_step": sum(sample_s) / len(sample_s),
                          "weights_sampled_of": [sum(min(r, wl.shapes[i][0]) * wl.shapes[i][1]
                                                     for i, r in oracle_sample(wl)), wl.params]},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------- our arm
def run_ours(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl")

    from paper_2608_15665_gb300 import build
    build.build()
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300 import workloads
    from paper_2608_15665_gb300.schedule import SubZeroPlus, step_plan

    wl0 = wl = subset(workloads.get(args.workload), args.layers)
    part = workloads.partition(wl, rank, world)
    weights = [workloads.init_weight(wl, i, dev, part["matrix_index_base"])
               for i in range(wl.n_mats)]
    z = SubZeroPlus(weights, wl.r, wl.q, part["seed"],
                    matrix_index_base=part["matrix_index_base"])
    if args.single_sm:
        zb.zo_set_option(z.ctx, zb.ZO_OPTION_PAIR_MMA, 0)
    calls, (rq, rc) = step_plan(args.scheme, wl.q)
    passes = len(calls) + 1
    K, W = args.steps, args.warmup
    table = workloads.loss_table(wl, args.scheme, steps=W + 2 * K + 1)
    table_dev = torch.from_numpy(table).to(dev)

    if args.method == "mezo":
        passes = 3

    def do_step_mezo(t, losses, gamma=None):
        # Eq. (1): evaluate at W + eps Z and W - eps Z, then restore fused with the SGD
        # update, W += (eps - lr rho) Z; rho from the step's first loss pair
        lp, lm = (float(losses[0]), float(losses[1])) if not torch.is_tensor(losses) \
            else (float(table[t][0]), float(table[t][1]))
        rho = (lp - lm) / (2.0 * wl.eps)
        z.mezo_perturb(t, wl.eps)
        z.mezo_perturb(t, -2.0 * wl.eps)
        z.mezo_perturb(t, wl.eps - wl.lr * rho)

    def do_step(t, losses, gamma=None):
        if args.method == "mezo":
            return do_step_mezo(t, losses, gamma)
        if t % wl.F == 0:
            z.refresh(t // wl.F, reset_moments=(t == 0))
        for (qa, ca), second in calls:
            qb, cb = second if second is not None else (-1, 0.0)
            z.perturb(t, qa, ca, qb, cb, wl.eps)
        z.step(t, t + 1, losses, args.scheme, wl.eps, wl.lr, wl.beta1, wl.beta2, wl.eps_adam,
               rq, rc, gamma_out=gamma)

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    def max_ranks(x):
        return max_over_ranks(x, world, dev)

    for t in range(W):
        do_step(t, table_dev[t])
    barrier()
    z.sync()

    # ---- device-timed region: inputs resident in HBM ---------------------------------
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_TIMING, 1)
    launches0 = zb.zo_kernel_launches(z.ctx)
    clocks = ClockSampler(local)
    clocks.start()
    barrier()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record()
    for t in range(W, W + K):
        do_step(t, table_dev[t])
    ev1.record()
    barrier()
    clk = clocks.stop()
    elapsed_ms = max_ranks(ev0.elapsed_time(ev1))
    wpass_ms, wpass_n = zb.zo_get_timing(z.ctx)
    launches = zb.zo_kernel_launches(z.ctx) - launches0
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_TIMING, 0)
    path = zb.zo_wpass_path(z.ctx)
    z.sync()

    # ---- one subspace refresh (Alg. 1 for every matrix), timed on its own ----------
    barrier()
    r0, r1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    r0.record()
    z.refresh((W + K) // wl.F)
    r1.record()
    barrier()
    refresh_ms = max_ranks(r0.elapsed_time(r1))
    z.sync()

    # Both timed windows are reported with the refresh amortised: a window of K steps holds
    # floor-or-ceil(K / F) refreshes depending on where it starts, so the refreshes it
    # happened to contain are replaced by refresh_ms / F per step (Alg. 3 refreshes every F
    # steps).  The raw window figures stay in "window".
    def amortised_ms(window_ms, t0):
        if args.method == "mezo":                 # no subspace, no refresh
            return window_ms / K
        return amortise_refresh(window_ms, K, t0, wl.F, refresh_ms)

    # ---- end to end through the public API with host buffers -------------------------
    e2e = None
    if not args.no_e2e:
        host_losses = torch.from_numpy(table[W + K:W + 2 * K + 1].copy()).pin_memory()
        gamma = torch.zeros(wl.n_mats, dtype=torch.float32, device=dev)
        gamma_host = torch.zeros(wl.n_mats, dtype=torch.float32).pin_memory()
        # one untimed step through the host path first (first use of the pinned buffers)
        do_step(W + K, host_losses[0].numpy(), gamma)
        gamma_host.copy_(gamma)
        e_clocks = ClockSampler(local)
        e_clocks.start()
        barrier()
        t0 = time.perf_counter()
        for k, t in enumerate(range(W + K + 1, W + 2 * K + 1)):
            do_step(t, host_losses[k + 1].numpy(), gamma)
            gamma_host.copy_(gamma)            # the step's result back on the host (syncs)
        barrier()
        e2e_s = max_ranks(time.perf_counter() - t0)
        e_clk = e_clocks.stop()
        e2e_ms = amortised_ms(e2e_s * 1e3, W + K + 1)
        e2e = {"value": job_steps_per_second(e2e_ms, world), "unit": "ZO steps/s",
               "h2d_bytes_per_step": int(table.shape[1] * 4),
               "d2h_bytes_per_step": int(wl.n_mats * 4),
               "ms_per_step": e2e_ms,
               "window": {"value": world * K / e2e_s, "ms_per_step": e2e_s * 1e3 / K},
               "clocks": e_clk}
    z.sync()

    step_ms = amortised_ms(elapsed_ms, W)
    value = job_steps_per_second(step_ms, world)
    bytes_pass = wl.bytes_per_pass()
    peak, peak_kind = measured_peaks()
    avg_launch_s = (wpass_ms / wpass_n) / 1e3 if wpass_n else float("nan")
    achieved = bytes_pass / avg_launch_s / 1e9
    src = kernel_source_hash(64 if (wl.r == 128 and args.single_sm) else wl.r)
    l2_resident = bytes_pass / 2 < L2_BYTES
    line = {
        "metric": METRIC, "value": value, "unit": "ZO steps/s", "n_gpus": world, "steps": K,
        "warmup": W, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": wl0.name, "matrices": wl.n_mats, "params": wl.params,
                   "weights": "bf16 N(0,0.02^2)" if wl.dtype == "bf16" else "f32 N(0,0.02^2)",
                   "r": wl.r, "q": wl.q, "scheme": args.scheme, "passes_per_step": passes,
                   "refresh_every": wl.F, "refreshes_in_timed_region":
                       sum(1 for t in range(W, W + K) if t % wl.F == 0),
                   "l2": ("inputs larger than L2 (%.1f GB of weights per pass)" % (bytes_pass / 2e9)
                          if not l2_resident else
                          "weights fit in L2 (%.1f MB per pass): latency-bound" % (bytes_pass / 2e6)),
                   "parallelism": f"layer partition x{world}" if world > 1 else "single GPU"},
        "weight_pass_gbs": passes * bytes_pass * K / (elapsed_ms / 1e3) / 1e9,
        "refresh_ms": refresh_ms,
        "window": {"value": world * K / (elapsed_ms / 1e3), "ms_per_step": elapsed_ms / K,
                   "refreshes": sum(1 for t in range(W, W + K) if t % wl.F == 0)
                   if args.method != "mezo" else 0,
                   "note": "value and ms_per_step replace the refreshes this window held by "
                           "refresh_ms / F per step"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": peak_kind,
                     "traffic": TRAFFIC_BY_SOURCE.get((src, wl.name)),
                     "kernel": {1: "wpass_fma",
                                2: ("wpass_tmem" if args.single_sm else "wpass_pair") if wl.r == 128
                                else "wpass_tmem" if wl.r == 64 else "wpass_tc",
                                3: "wpass_narrow"}.get(path, "?"),
                     "algorithmic_bytes_per_launch": bytes_pass,
                     "avg_launch_ms": avg_launch_s * 1e3, "launches_timed": wpass_n},
        "clocks": clk,
        "gpu_launches": int(launches),
    }
    if l2_resident:
        # the whole set stays in the 129 MB L2 between passes: no HBM fraction, the pass
        # is reported as its latency
        line["roofline"] = {"bound": "latency", "achieved": None, "peak": None, "unit": "GB/s",
                            "frac": None, "traffic": None,
                            "kernel": line["roofline"]["kernel"],
                            "us_per_pass": avg_launch_s * 1e6, "launches_timed": wpass_n}
    if args.method == "mezo":
        # bound by instruction issue: peak = SMs x 128 lanes x max SM clock (thread
        # instructions per second); achieved = instructions per weight (ncu count of the
        # kernel, profiles/mezo_kernel_llama7b_2layers.md) x weights / launch time
        line["metric"] = "MeZO full-space SPSA (Eq. (1)) steps/s at 7B shape, 1 GB300"
        ipw = INSTR_PER_WEIGHT_BY_SOURCE.get(mezo_source_hash())
        issue_peak = 152 * 128 * 2.07e9 / 1e12
        ach = ipw * wl.params / avg_launch_s / 1e12 if ipw else None
        line["roofline"] = {"bound": "alu", "achieved": ach, "peak": issue_peak,
                            "unit": "T thread-instructions/s", "frac": ach / issue_peak if ach else None,
                            "peak_kind": "derived: 152 SMs x 128 lanes x 2.07 GHz",
                            "instructions_per_weight": ipw, "kernel": "mezo_kernel",
                            "weight_gbs": achieved, "weight_gbs_frac_of_hbm": achieved / peak,
                            "avg_launch_ms": avg_launch_s * 1e3, "launches_timed": wpass_n}
        line["config"]["method"] = "mezo"
        line["config"].pop("r"); line["config"].pop("q")
    if e2e:
        line["e2e"] = e2e
    z.close()
    if (world == 1 and args.method == "subzero" and args.workload == "llama7b_bf16_r32"
            and not args.layers and not args.no_secondary):
        # the second shape the weight pass is held to: the 32B-shaped set (r = 64, q = 8); the
        # paper's default scale on the 7B shapes (r = 128, K = 99 queries); the linear layers
        # of one 7B layer evaluated at the perturbed weights without a weight pass (r = 32 and
        # r = 128)
        del weights, z
        torch.cuda.empty_cache()
        # (the short linear measurements first: the long weight-pass ones run under the
        # power cap and leave the clocks lowered for a while; each records its own clocks)
        sec = {}
        sec["perturbed_linear_llama7b_4096tok"] = secondary_linear(dev, local)
        sec["perturbed_linear_llama7b_4096tok_r128"] = secondary_linear(dev, local,
                                                                        "llama7b_bf16_r128_q99")
        sec["dense32b_bf16_r64"] = secondary_weight_pass(dev, local, peak, "dense32b_bf16_r64", 2)
        sec["mezo_llama7b_bf16"] = secondary_mezo(dev, local, peak)
        sec["llama7b_bf16_r128_q99"] = secondary_weight_pass(dev, local, peak,
                                                             "llama7b_bf16_r128_q99", 1)
        line["secondary"] = sec
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl0, args.scheme)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


def secondary_weight_pass(dev, local, peak, name, K):
    """A short measurement of the weight pass on a second workload -- the 32B-shaped set
    (448 bf16 matrices, 31.2 G parameters, r = 64, q = 8: 17 passes per step, refresh every
    5), or the 7B set at the paper's default scale (r = 128, q = 99: 199 passes per step,
    refresh every 50; the SM-pair kernel): one warm-up step (with its refresh), then K
    timed steps with the weight-pass launches timed by CUDA events, and one refresh timed
    on its own."""
    import torch
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300 import workloads
    from paper_2608_15665_gb300.schedule import SubZeroPlus, step_plan
    wl = workloads.get(name)
    weights = [workloads.init_weight(wl, i, dev) for i in range(wl.n_mats)]
    z = SubZeroPlus(weights, wl.r, wl.q, wl.seed)
    calls, (rq, rc) = step_plan("central", wl.q)
    table = torch.from_numpy(workloads.loss_table(wl, "central", steps=1 + K)).to(dev)

    def do_step(t):
        if t % wl.F == 0:
            z.refresh(t // wl.F, reset_moments=(t == 0))
        for (qa, ca), second in calls:
            qb, cb = second if second is not None else (-1, 0.0)
            z.perturb(t, qa, ca, qb, cb, wl.eps)
        z.step(t, t + 1, table[t], "central", wl.eps, wl.lr, wl.beta1, wl.beta2, wl.eps_adam, rq, rc)

    do_step(0)
    z.sync()
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_TIMING, 1)
    clocks = ClockSampler(local)
    clocks.start()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for t in range(1, 1 + K):
        do_step(t)
    e1.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    window_ms = e0.elapsed_time(e1)
    wpass_ms, wpass_n = zb.zo_get_timing(z.ctx)
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_TIMING, 0)
    path = zb.zo_wpass_path(z.ctx)
    r0, r1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    r0.record()
    z.refresh(1)
    r1.record()
    torch.cuda.synchronize()
    refresh_ms = r0.elapsed_time(r1)
    z.sync()
    z.close()
    del weights, z
    torch.cuda.empty_cache()
    avg_s = (wpass_ms / wpass_n) / 1e3
    achieved = wl.bytes_per_pass() / avg_s / 1e9
    step_ms = window_ms / K + refresh_ms / wl.F
    return {"workload": wl.name, "matrices": wl.n_mats, "params": wl.params, "r": wl.r, "q": wl.q,
            "passes_per_step": 2 * wl.q + 1, "refresh_every": wl.F, "steps_timed": K,
            "kernel": {2: "wpass_pair" if wl.r == 128 else "wpass_tmem" if wl.r == 64
                       else "wpass_tc", 1: "wpass_fma"}.get(path, "?"),
            "avg_launch_ms": avg_s * 1e3, "launches_timed": wpass_n,
            "algorithmic_bytes_per_launch": wl.bytes_per_pass(),
            "achieved_gbs": achieved, "peak_gbs": peak, "frac": achieved / peak,
            "traffic": TRAFFIC_BY_SOURCE.get((kernel_source_hash(wl.r), wl.name)),
            "zo_steps_s": 1e3 / step_ms, "ms_per_step": step_ms, "refresh_ms": refresh_ms,
            "clocks": clk}


def secondary_mezo(dev, local, peak, K=3):
    """MeZO's full-space SPSA step (Eq. (1)) on the LLaMA-7B set: three zo_mezo_perturb
    passes per step (+eps, -2 eps, then +eps fused with the SGD update from the step's loss
    pair); one warm-up step, then K timed steps with the passes timed by CUDA events.
    Roofline: bound by instruction issue (thread instructions per weight from the ncu
    count of the kernel, against 152 SMs x 128 lanes x 2.07 GHz)."""
    import torch
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300 import workloads
    from paper_2608_15665_gb300.schedule import SubZeroPlus
    wl = workloads.get("llama7b_bf16_r32")
    weights = [workloads.init_weight(wl, i, dev) for i in range(wl.n_mats)]
    z = SubZeroPlus(weights, wl.r, wl.q, wl.seed)
    table = workloads.loss_table(wl, "central", steps=1 + K)

    def do_step(t):
        rho = (float(table[t][0]) - float(table[t][1])) / (2.0 * wl.eps)
        z.mezo_perturb(t, wl.eps)
        z.mezo_perturb(t, -2.0 * wl.eps)
        z.mezo_perturb(t, wl.eps - wl.lr * rho)

    do_step(0)
    z.sync()
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_TIMING, 1)
    clocks = ClockSampler(local)
    clocks.start()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for t in range(1, 1 + K):
        do_step(t)
    e1.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    window_ms = e0.elapsed_time(e1)
    pass_ms, n = zb.zo_get_timing(z.ctx)
    zb.zo_set_option(z.ctx, zb.ZO_OPTION_TIMING, 0)
    z.sync()
    z.close()
    del weights, z
    torch.cuda.empty_cache()
    avg_s = (pass_ms / n) / 1e3
    ipw = INSTR_PER_WEIGHT_BY_SOURCE.get(mezo_source_hash())
    issue_peak = 152 * 128 * 2.07e9 / 1e12
    ach = ipw * wl.params / avg_s / 1e12 if ipw else None
    return {"workload": wl.name, "params": wl.params, "passes_per_step": 3, "steps_timed": K,
            "kernel": "mezo_kernel", "avg_launch_ms": avg_s * 1e3, "launches_timed": n,
            "mezo_steps_s": 1e3 * K / window_ms, "ms_per_step": window_ms / K,
            "roofline": {"bound": "alu", "achieved": ach, "peak": issue_peak,
                         "unit": "T thread-instructions/s",
                         "frac": ach / issue_peak if ach else None,
                         "instructions_per_weight": ipw},
            "weight_gbs": wl.bytes_per_pass() / avg_s / 1e9,
            "weight_gbs_frac_of_hbm": wl.bytes_per_pass() / avg_s / 1e9 / peak, "clocks": clk}


def linear_measure(dev, wl, T, K, W, compare=True, e2e=True):
    """The linear layers of `wl` (one layer's matrices) at the perturbed weights,
    Y_i = X_i (W_i + U_i C V_i^T)^T with no weight pass (the forward route of one loss
    evaluation: C_i and P_i once, then S = X P^T and X W^T + S U^T per layer), on
    X_i: T x n_i bf16 activations, N(0, 1), resident.  A step is one zo_linear_prepare and
    the layer's zo_linear_perturbed calls; W untimed warm-up steps, K timed ones (CUDA
    events).  With compare: the same route on single-CTA tiles, the same GEMMs without the
    perturbation (torch, i.e. cuBLAS) and the weight-pass route (one zo_perturb pass over
    the layer, then those GEMMs).  With e2e: the route with the activations copied from
    pinned host memory every step and one output row read back."""
    import torch
    from paper_2608_15665_gb300 import binding as zb
    from paper_2608_15665_gb300 import workloads
    from paper_2608_15665_gb300.schedule import SubZeroPlus

    weights = [workloads.init_weight(wl, i, dev) for i in range(wl.n_mats)]
    z = SubZeroPlus(weights, wl.r, wl.q, wl.seed)
    z.init_subspace(0)
    g = torch.Generator(device=dev).manual_seed(wl.seed)
    X = {n: torch.randn(T, n, generator=g, device=dev).to(torch.bfloat16)
         for n in sorted({n for _, n in wl.shapes})}
    Y = [torch.empty(T, m, dtype=torch.bfloat16, device=dev) for m, _ in wl.shapes]
    out = {"flops": sum(2.0 * T * (m * n + wl.r * (m + n)) for m, n in wl.shapes)}

    def fused(t):
        zb.zo_linear_prepare(z.ctx, t, 0, 1.0, -1, 0.0, wl.eps)
        for i, (m, n) in enumerate(wl.shapes):
            zb.zo_linear_perturbed(z.ctx, i, X[n], Y[i])

    def plain():
        for i, (m, n) in enumerate(wl.shapes):
            torch.matmul(X[n], z.weights[i].t(), out=Y[i])

    def timed(fn, K):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record()
        for k in range(K):
            fn(k)
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / K

    for k in range(W):
        fused(k)
        plain()
    z.sync()
    launches0 = zb.zo_kernel_launches(z.ctx)
    clocks = ClockSampler(dev.index or 0)
    clocks.start()
    out["fused_ms"] = timed(fused, K)
    out["clocks"] = clocks.stop()
    out["launches"] = zb.zo_kernel_launches(z.ctx) - launches0
    z.sync()
    names = {1: "128x256", 2: "256x256", 3: "256x224", 4: "256x256 pair", 5: "256x240 pair",
             6: "256x224 pair", 7: "256x192 pair", 8: "256x128 pair"}
    out["tiling"] = []
    for i, (m, n) in enumerate(wl.shapes):
        zb.zo_linear_perturbed(z.ctx, i, X[n], Y[i])
        out["tiling"].append(names[zb.zo_linear_tiling(z.ctx)])
    if compare:
        if wl.r <= 32:
            # the same route with the single-CTA 128 x 256 and 256 x 224 tiles throughout
            # (r <= 32 only)
            zb.zo_set_option(z.ctx, zb.ZO_OPTION_LINEAR_TILE, 1)
            out["fused128_ms"] = timed(fused, K)
            zb.zo_set_option(z.ctx, zb.ZO_OPTION_LINEAR_TILE, 3)
            out["fused224_ms"] = timed(fused, K)
            zb.zo_set_option(z.ctx, zb.ZO_OPTION_LINEAR_TILE, 0)
            z.sync()
        out["plain_ms"] = timed(lambda k: plain(), K)
        out["wpass_ms"] = timed(lambda k: (z.perturb(k, 0, 1.0, -1, 0.0, wl.eps), plain()), K)
        z.sync()
    if e2e:
        host = {n: x.cpu().pin_memory() for n, x in X.items()}
        out_row = torch.empty(wl.shapes[-1][0], dtype=torch.bfloat16).pin_memory()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for k in range(K):
            for n, h in host.items():
                X[n].copy_(h, non_blocking=True)
            fused(k)
            out_row.copy_(Y[-1][0])
        torch.cuda.synchronize()
        out["e2e_s"] = (time.perf_counter() - t0) / K
        out["h2d"] = sum(h.numel() * 2 for h in host.values())
        out["d2h"] = int(out_row.numel() * 2)
    z.close()
    del weights, X, Y, z
    torch.cuda.empty_cache()
    return out


def linear_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            mp = json.load(f)
        # the layer's GEMMs run back to back for tens of ms: the sustained figure
        peak = float(mp.get("bf16_tflops_sustained") or 0.0) or None
        if peak:
            return peak, "measured (cuBLAS bf16, sustained)"
    except Exception:
        pass
    return 1700.0, "fallback (sustained)"


def secondary_linear(dev, local, name="llama7b_bf16_r32"):
    """The perturbed-linear route (zo_linear_perturbed, no weight pass) on one LLaMA-7B
    layer's seven matrices at 4096 tokens (r = 32, or the paper's r = 128): 10 timed steps
    after 2 warm-up ones, with the weight-pass route and the plain cuBLAS GEMMs timed
    beside it."""
    from paper_2608_15665_gb300 import workloads
    wl = subset(workloads.get(name), 1)
    T = 4096
    m = linear_measure(dev, wl, T, K=10, W=2, compare=True, e2e=False)
    peak, peak_kind = linear_peak()
    achieved = m["flops"] / (m["fused_ms"] / 1e3) / 1e12
    return {"workload": wl.name, "tokens": T, "r": wl.r, "tiles": m["tiling"],
            "ms_per_step": m["fused_ms"], "tflops": achieved, "peak_tflops": peak,
            "frac": achieved / peak, "peak_kind": peak_kind,
            "kernel": "linear_pair_kernel" if any("pair" in t for t in m["tiling"])
            else "linear_kernel",
            "weight_pass_route_ms": m["wpass_ms"], "plain_gemm_ms": m["plain_ms"],
            "single_cta_256x224_ms": m.get("fused224_ms"), "clocks": m["clocks"]}


def run_linear(args):
    """bench.py --method linear: the linear layers of the first `--layers` (default 1)
    layers of the workload at the perturbed weights (linear_measure), --tokens rows of
    activations.  value = TFLOP/s of the exact-arithmetic work 2 T (m n + r (m + n)) per
    layer; roofline against the measured bf16 tensor peak."""
    import torch
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    from paper_2608_15665_gb300 import build
    build.build()
    from paper_2608_15665_gb300 import workloads

    wl = subset(workloads.get(args.workload), args.layers or 1)
    T = args.tokens
    K, W = args.steps, args.warmup
    m = linear_measure(dev, wl, T, K, W)
    peak, peak_kind = linear_peak()
    flops = m["flops"]
    achieved = flops / (m["fused_ms"] / 1e3) / 1e12
    line = {
        "metric": "perturbed linear forward TFLOP/s (zo_linear_perturbed, LLaMA-7B layer shapes, 1 GB300)",
        "value": achieved, "unit": "TFLOP/s", "n_gpus": 1, "steps": K, "warmup": W,
        "ms_per_step": m["fused_ms"], "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": wl.name, "matrices": wl.n_mats, "tokens": T, "r": wl.r,
                   "method": "linear", "tiles": m["tiling"],
                   "l2": "inputs larger than L2 (%.0f MB of weights)" % (sum(mm * n for mm, n in wl.shapes) * 2 / 1e6),
                   "parallelism": "single GPU"},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "peak_kind": peak_kind, "traffic": None,
                     "kernel": "linear_pair_kernel" if any("pair" in t for t in m["tiling"])
                     else "linear_kernel", "algorithmic_flops_per_step": flops},
        "tile128_ms": m.get("fused128_ms"),
        "tile224_single_cta_ms": m.get("fused224_ms"),
        "plain_gemm_ms": m["plain_ms"],
        "weight_pass_route_ms": m["wpass_ms"],
        "e2e": {"value": flops / m["e2e_s"] / 1e12, "unit": "TFLOP/s",
                "h2d_bytes_per_step": int(m["h2d"]), "d2h_bytes_per_step": m["d2h"]},
        "clocks": m["clocks"],
        "gpu_launches": int(m["launches"]),
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.oracle_sample:
        run_oracle_sample(args)
    elif args.impl == "reference":
        run_reference(args)
    elif args.method == "linear":
        run_linear(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
