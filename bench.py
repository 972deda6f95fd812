"""Throughput of the MCA trial loop on one GB300 (trials/s), per the bench contract.

Workload (default): the 784-16384-10 tanh / softmax-CE net on N = 60000 synthetic MNIST-shaped
samples, K = 64 speculative candidates per batch, 1M-trial job, Philox seed 0. One step = one
mca_run call of T trials continuing the same trajectory; warm-up + timed steps together cover the
job's 1M trials (T = ceil(1e6 / (warmup + steps))). The cached hidden fields (3.9 GB) are far
larger than L2, so no L2 flush is needed between steps.

--impl reference times the CPU oracle (incremental mode, fp64 numpy) on the same workload, a
bounded number of trials per step, on the host cores.

Multi-GPU: the trial loop is sequential (each trial depends on the previous decision), so N GPUs run
N independent replicas (proposal seed = rank); value = all ranks' trials / max time ("weak").
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "MC mutation trials/sec (full-batch loss evals); fraction of HBM/TC roofline"

# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of the trial-loop kernel per trial,
# from one ncu capture (one pass, one launch: the first timed step, trials 200k..240k) of
# `python bench.py --steps 20 --warmup 5 --no-e2e --no-cpu`, summarised in profiles/. It is only
# valid for the kernel source and the workload it was measured on; anything else reports null.
LOOP_TRAFFIC = {"source_sha1": "2502508233974700a08bab261aa72e3018dd27bb",
                "workload": "mlp784-16384-10_ce_n60000", "bytes_per_trial": 374000.0}
LOOP_SOURCES = ("paper_2607_08406_gb300/csrc/mca_mlp2.cu", "paper_2607_08406_gb300/csrc/mca_device.cuh")


def loop_source_sha1() -> str:
    import hashlib
    h = hashlib.sha1()
    for rel in LOOP_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()
UNIT = "trials/s"
JOB_TRIALS = 1_000_000
DEEP_TRIALS_PER_STEP = 4000


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms while running."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax = float(f[2])
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm)}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def make_workload(args, rank):
    from paper_2607_08406_gb300 import workloads as W
    kw = {}
    if args.workload == "char_transformer":
        if args.N:
            kw["batch"] = args.N
        wl = W.char_transformer(**kw)
    else:
        if args.N:
            kw["N"] = args.N
        if args.H:
            kw["H"] = args.H
        wl = W.make(args.workload, **kw)
    wl.seed = args.seed + rank
    if args.K:
        wl.K = args.K
    if args.beta != float("inf") or args.layer_stretch:
        import dataclasses
        wl.domain = dataclasses.replace(wl.domain, beta=args.beta, layer_stretch=args.layer_stretch)
    return wl


def is_tfm(wl) -> bool:
    return hasattr(wl, "spec")


def acceptance(wl) -> str:
    return ("greedy (Eq. 6)" if wl.domain.beta == float("inf")
            else f"Metropolis (Eq. 7), beta = {wl.domain.beta:g}")


def proposals(wl) -> str:
    return ("uniform over all parameters" if not wl.domain.layer_stretch
            else f"current-layer schedule, {wl.domain.layer_stretch} trials per layer")


def host_arrays(wl):
    """The arrays a job uploads: (X, y, init) for an MLP, (tokens, init) for the Transformer."""
    return (wl.tokens, wl.init) if is_tfm(wl) else (wl.X, wl.y, wl.init)


def create_handle(mca, wl, arrays, **kw):
    if is_tfm(wl):
        tokens, init = arrays
        return mca.mca_create_transformer(wl.spec, wl.domain, tokens, init, K=wl.K, **kw)
    X, y, init = arrays
    return mca.mca_create(wl.layers, wl.loss, wl.domain, X, y, init, K=wl.K, **kw)


def cpu_oracle_rate(wl, n_trials, warm=0):
    """A function running oracle trials t0 .. t0+n: the incremental mode (after an untimed cache
    build) for the MLPs, the full-recompute loop for the Transformer."""
    from oracle import mca_oracle as O
    if is_tfm(wl):
        from oracle import mca_tfm as T
        flat = np.array(wl.init, dtype=np.float32)
        state = {"S": float(T.tfm_seq_losses(wl.spec, flat.astype(np.float64), wl.tokens).sum())}

        def tfm_trials(t0, n):
            for t in range(t0, t0 + n):
                idx, old, new, valid = T.tfm_propose(wl.seed, t, flat, wl.domain)
                if not valid:
                    continue
                flat[idx] = np.float32(new)
                S_new = float(T.tfm_seq_losses(wl.spec, flat.astype(np.float64), wl.tokens).sum())
                theta = float(O.metropolis_threshold(wl.seed, t, wl.domain.beta,
                                                     wl.tokens.shape[0] * wl.spec.ctx))
                if S_new - state["S"] <= theta:
                    state["S"] = S_new
                else:
                    flat[idx] = np.float32(old)
        return tfm_trials
    XT = np.ascontiguousarray(wl.X.astype(np.float64).T)
    params = O.Params(wl.layers, wl.init)
    cache = O._Cache(params, XT, wl.y, wl.loss)
    S = float(cache.ell.sum())

    def trials(t0, n):
        nonlocal S
        for t in range(t0, t0 + n):
            p = O.propose(wl.seed, t, params, wl.domain)
            if not p.valid:
                continue
            dS, updates, ell_new = O._candidate(params, cache, XT, wl.y, wl.loss, p)
            theta = O._threshold(wl.seed, t, wl.domain, XT.shape[1])
            if O._decide(dS, wl.domain.strict, theta):
                O.apply_proposal(params, p)
                for m, upd in updates:
                    if upd[0] == "row":
                        cache.Z[m][upd[1]] = upd[2]
                    else:
                        cache.Z[m] = upd[1]
                cache.ell = ell_new
                S += dS
    return trials


def cpu_sample_trials(wl) -> int:
    """Trials of the bounded CPU sample: about 10-30 s of the oracle on the machine's host cores."""
    if is_tfm(wl):
        return 40
    if len(wl.layers) > 2:
        return 100
    return 20000 if wl.N * wl.layers[0].n_out < 10 ** 8 else 4000


def threads_used(cpu_s: float, wall_s: float) -> int:
    """Threads the sample kept busy on average: process CPU time over wall time, rounded (the
    oracle's numpy calls are single-threaded except its BLAS products)."""
    return max(1, int(round(cpu_s / wall_s))) if wall_s > 0 else 1


def job_totals(local_ms: float, local_units: float, device=None):
    """Whole-job aggregate over the ranks of an initialised process group: the slowest rank's time
    (MAX) and the units every rank processed (SUM). A single process returns its own figures."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return local_ms, local_units
    mx = torch.tensor([local_ms], dtype=torch.float64, device=device)
    sm = torch.tensor([local_units], dtype=torch.float64, device=device)
    dist.all_reduce(mx, op=dist.ReduceOp.MAX)
    dist.all_reduce(sm, op=dist.ReduceOp.SUM)
    return float(mx.item()), float(sm.item())


def run_reference(args):
    rank, local_rank, world = dist_env()
    if rank != 0:
        return 0
    wl = make_workload(args, 0)
    per_step = args.ref_trials
    trials = cpu_oracle_rate(wl, per_step)
    tau = 0
    for _ in range(args.warmup):
        trials(tau, per_step)
        tau += per_step
    t0, c0 = time.perf_counter(), time.process_time()
    for _ in range(args.steps):
        trials(tau, per_step)
        tau += per_step
    dt, dc = time.perf_counter() - t0, time.process_time() - c0
    rate = per_step * args.steps / dt
    cores = threads_used(dc, dt)
    mode = "full-recompute" if is_tfm(wl) else "incremental"
    sample = (f"oracle {mode} mode (fp64 numpy), trials {per_step * args.warmup}.."
              f"{tau} of {wl.name}, after an untimed forward pass")
    line = {"impl": "reference", "metric": METRIC, "value": rate, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": wl.name, "K": wl.K, "trials_per_step": per_step,
                       "acceptance": acceptance(wl), "proposals": proposals(wl)},
            "cpu_baseline": {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": sample, "cpu_s_per_wall_s": dc / dt,
                             "host_cores": len(os.sched_getaffinity(0))},
            "e2e": {"value": rate, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args):
    import torch
    import torch.distributed as dist
    rank, local_rank, world = dist_env()
    torch.cuda.set_device(local_rank)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))

    def barrier():
        if world > 1:
            dist.barrier()

    from paper_2607_08406_gb300 import mca
    from paper_2607_08406_gb300.build import build
    build()
    wl = make_workload(args, rank)
    K, W_ = args.steps, args.warmup
    # single-hidden-layer nets: the 1M-trial job spread over the steps; deep nets and the
    # Transformer (thousands of trials/s): a bounded sample of the job, 4000 trials per step
    deep_wl = is_tfm(wl) or len(wl.layers) > 2
    T = args.trials_per_step or (DEEP_TRIALS_PER_STEP if deep_wl else math.ceil(JOB_TRIALS / (K + W_)))
    stream = torch.cuda.current_stream()

    dev_arrays = [torch.from_numpy(a).cuda() for a in host_arrays(wl)]
    extra = {} if is_tfm(wl) else {"grid": args.grid}
    h = create_handle(mca, wl, dev_arrays, resync_period=args.resync, stream=stream.cuda_stream,
                      fixed_K=args.fixed_K, **extra)
    # one full forward pass (the resync step), timed on its own
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    mca.mca_resync(h)
    ev1.record(stream)
    torch.cuda.synchronize()
    resync_ms = ev0.elapsed_time(ev1)

    for _ in range(W_):
        mca.mca_run(h, T, wl.seed)
    st0 = mca.mca_get_stats(h)
    barrier()
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(K + 1)]
    with ClockSampler(local_rank) as clk:
        evs[0].record(stream)
        for k in range(K):
            mca.mca_run(h, T, wl.seed)
            evs[k + 1].record(stream)
        torch.cuda.synchronize()
    barrier()
    st1 = mca.mca_get_stats(h)
    step_ms = [evs[k].elapsed_time(evs[k + 1]) for k in range(K)]
    total_ms, trials_timed = job_totals(sum(step_ms), float(st1["trials"] - st0["trials"]),
                                        device="cuda")
    value = trials_timed / (total_ms / 1e3)
    launches = st1["launches"] - st0["launches"]
    # dominant kernel: single hidden layer -- the trial loop (one launch per step when no resync
    # falls in the step), HBM-bound; deep nets -- the candidate chains (SIMT fp32 FMA), whose
    # FLOPs are divided by the whole step time (a lower bound: the step also holds the decide and
    # commit kernels and one host round trip per batch)
    deep = is_tfm(wl) or len(wl.layers) > 2
    peak, peak_kind = load_peaks()
    traffic = None
    if deep:
        # FLOPs of the evaluated candidates' recomputation (counted by the library, 2 per fp32
        # multiply-add) over the evaluation kernel's own time (CUDA events around its launches)
        flops_timed = st1["alg_flops"] - st0["alg_flops"]
        eval_s = (st1["phase_ns"][0] - st0["phase_ns"][0]) / 1e9
        achieved = flops_timed / eval_s / 1e12 if eval_s > 0 else 0.0
        if st1["tensor_cores"]:         # the library reports which kernels the handle runs
            # the evaluation kernel runs for seconds inside each step: the sustained bf16 figure
            pk = os.path.join(ROOT, "MEASURED_PEAKS.json")
            if os.path.exists(pk):
                bf16, bf16_kind = float(json.load(open(pk))["bf16_tflops_sustained"]), "measured"
            else:
                bf16, bf16_kind = 1700.0, "fallback"
            peak = bf16 * 0.5 / 3.0
            peak_kind = (f"{bf16_kind} bf16 sustained x 1/2 (nominal tf32 : bf16 dense rate) / 3 "
                         "(3xTF32: three tf32 MMAs per fp32 product)")
            roofline = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                        "frac": achieved / peak, "traffic": None,
                        "kernel": "tfm_tc_kernel" if is_tfm(wl) else "deep_chain_tc_kernel",
                        "peak_kind": peak_kind,
                        "flops": "2 x fp32 multiply-adds of the evaluated chains (not x3), over "
                                 "the evaluation kernel's event-timed duration"}
        else:
            sms = torch.cuda.get_device_properties(local_rank).multi_processor_count
            sm_max = float(json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))["sm_max_mhz"]) \
                if os.path.exists(os.path.join(ROOT, "MEASURED_PEAKS.json")) else 2070.0
            peak = sms * 128 * 2 * sm_max * 1e6 / 1e12        # fp32 FMA lanes x 2 FLOP x clock
            peak_kind = f"derived: {sms} SMs x 128 fp32 lanes x 2 FLOP x {sm_max:.0f} MHz"
            roofline = {"bound": "alu", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                        "frac": achieved / peak, "traffic": None,
                        "kernel": "tfm_seq_kernel" if is_tfm(wl) else "deep_chain_kernel",
                        "peak_kind": peak_kind,
                        "flops": "FLOPs of the evaluated candidates' recomputation, counted by "
                                 "the library, over the evaluation kernel's event-timed duration"}
    else:
        bytes_timed = st1["alg_bytes"] - st0["alg_bytes"]
        achieved = bytes_timed / K / (total_ms / K / 1e3) / 1e9
        if (LOOP_TRAFFIC["source_sha1"] == loop_source_sha1() and
                LOOP_TRAFFIC["workload"] == wl.name and LOOP_TRAFFIC["bytes_per_trial"]):
            traffic = LOOP_TRAFFIC["bytes_per_trial"] * (st1["trials"] - st0["trials"]) / K
        roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                    "frac": achieved / peak, "traffic": traffic, "kernel": "mlp2_window_loop",
                    "peak_kind": peak_kind,
                    "bytes": "compulsory DRAM bytes of the distinct candidates evaluated, "
                             "counted by the kernel (per launch)"}
    loss_end = mca.mca_loss(h)
    h.close()

    # end to end through the public API from pinned host memory: one step = the whole job
    # (create from host arrays -> JOB_TRIALS trials -> parameters back to host)
    e2e = None
    if not args.no_e2e:
        pinned = [torch.from_numpy(a).pin_memory() for a in host_arrays(wl)]
        out = torch.empty(wl.n_params, dtype=torch.float32).pin_memory()
        e2e_trials = args.e2e_trials or (T * K if deep_wl else JOB_TRIALS)

        def job():
            hh = create_handle(mca, wl, pinned, resync_period=args.resync,
                               stream=stream.cuda_stream, fixed_K=args.fixed_K, **extra)
            mca.mca_run(hh, e2e_trials, wl.seed)
            mca.mca_get_params(hh, wl.n_params, out)
            lv = mca.mca_loss(hh)
            hh.close()
            return lv
        job()
        barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            job()
        torch.cuda.synchronize()
        dt, e2e_units = job_totals(time.perf_counter() - t0, float(e2e_trials * args.e2e_steps),
                                   device="cuda")
        e2e = {"value": e2e_units / dt, "unit": UNIT,
               "h2d_bytes_per_step": int(sum(a.nbytes for a in host_arrays(wl))),
               "d2h_bytes_per_step": int(out.numel() * 4 + 8),
               "step": f"create from pinned host arrays + {e2e_trials} trials + params to host"}

    cpu = None
    if rank == 0 and not args.no_cpu:
        n_cpu = args.cpu_trials or cpu_sample_trials(wl)
        trials = cpu_oracle_rate(wl, n_cpu)
        t0, c0 = time.perf_counter(), time.process_time()
        trials(0, n_cpu)
        dt, dc = time.perf_counter() - t0, time.process_time() - c0
        mode = "full-recompute" if is_tfm(wl) else "incremental"
        cpu = {"value": n_cpu / dt, "unit": UNIT, "cores": threads_used(dc, dt),
               "kind": "oracle",
               "sample": f"first {n_cpu} trials of {wl.name}, oracle {mode} mode "
                         f"(fp64 numpy), after an untimed forward pass",
               "cpu_s_per_wall_s": dc / dt, "host_cores": len(os.sched_getaffinity(0))}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": W_, "ms_per_step": total_ms / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": wl.name,
                       "N": int(wl.tokens.shape[0] * wl.spec.ctx) if is_tfm(wl) else wl.N,
                       "hidden": wl.spec.d_model if is_tfm(wl) else wl.layers[0].n_out,
                       "layers": wl.spec.n_layer if is_tfm(wl) else len(wl.layers),
                       "K": wl.K, "trials_per_step": T,
                       "trial_range": [W_ * T, (W_ + K) * T], "seed": args.seed,
                       "resync_period": args.resync, "resync_ms": resync_ms,
                       "l2": (f"no flush: the cached hidden fields "
                              f"({wl.layers[0].n_out * wl.N * 4 / 1e9:.2f} GB) exceed L2"
                              if not deep else "no flush: a step's candidates recompute from "
                              "cached fields / residual streams that exceed L2 or are rewritten"),
                       "parallelism": f"replicas x{world}" if world > 1 else "1 GPU",
                       "acceptance": acceptance(wl), "proposals": proposals(wl),
                       "accepts_timed": st1["accepts"] - st0["accepts"],
                       "batches_timed": st1["batches"] - st0["batches"],
                       "phase_ms": {nm: (st1["phase_ns"][q] - st0["phase_ns"][q]) / 1e6
                                    for q, nm in enumerate(
                                        ["eval_kernel", "decide_commit_kernels"] if deep else
                                        ["setup_and_commit", "evaluate", "wait_decide",
                                         "wait_cta", "add_shares", "unused", "slot_wait"])},
                       "slots_reprepared": 0 if deep else st1["phase_ns"][7] - st0["phase_ns"][7],
                       "candidates_timed": st1["candidates"] - st0["candidates"],
                       "loss_end": loss_end},
            "roofline": roofline,
            "cpu_baseline": cpu,
            "e2e": e2e,
            "clocks": clk.summary(),
            "gpu_launches": launches,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="mlp_wide")
    ap.add_argument("--N", type=int, default=0)
    ap.add_argument("--H", type=int, default=0)
    ap.add_argument("--K", type=int, default=0)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--trials-per-step", dest="trials_per_step", type=int, default=0)
    ap.add_argument("--resync", type=int, default=0)
    ap.add_argument("--grid", type=int, default=0)
    ap.add_argument("--fixed-K", dest="fixed_K", action="store_true")
    ap.add_argument("--cpu-trials", dest="cpu_trials", type=int, default=0,
                    help="trials of the CPU oracle sample (0: sized per workload)")
    ap.add_argument("--ref-trials", dest="ref_trials", type=int, default=200)
    ap.add_argument("--e2e-steps", dest="e2e_steps", type=int, default=1)
    ap.add_argument("--e2e-trials", dest="e2e_trials", type=int, default=0)
    ap.add_argument("--no-e2e", dest="no_e2e", action="store_true")
    ap.add_argument("--no-cpu", dest="no_cpu", action="store_true")
    ap.add_argument("--beta", type=float, default=float("inf"),
                    help="Metropolis selection intensity (Eq. 7); inf: the greedy rule")
    ap.add_argument("--layer-stretch", dest="layer_stretch", type=int, default=0,
                    help="current-layer schedule: trials per randomly chosen layer (MLPs)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
