"""Benchmark of the SLORR regularizer hot path (forward value + weight gradient
over a whole weight set, Listing 1 / Alg. 2) on GB300.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload vit_l16]
                  [--variant hoyer|nuclear] [--compute fp16|bf16|fp32] [--impl ours|reference]
                  [--iters T] [--op fwd_bwd|descent] [--eta ETA] [--flags F]

A step is one slorr_reg_forward_backward call over the whole weight set
(norm, cast, T = 6 Polar Express steps of three grouped GEMMs, dot, combine).
The default workload is the ViT-L/16-shaped set (96 matrices, 302 M weights,
1.21 GB of fp32 weights: larger than the 129 MB L2, so no flush is needed).

Printed: one JSON line.  value = algorithmic TFLOP/s of the whole job, using
the paper's count T * sum_i (4 P_i^2 Q_i + 2 P_i^3) (Sec. 3 "Computational
cost"); e2e = the same through the C ABI's host-buffer call (slorr_pipeline_forward_backward):
the weights and grads copied from page-locked host memory and the grads and
loss copied back inside the timed region, group by group, overlapped with the
kernels of the other groups;
roofline = the tensor-core GEMM kernel measured live with CUDA events around
each of its launches on the call's stream, in a second timed pass of the same
number of steps (events between kernels would serialise the programmatic
dependent launches of the first); cpu_baseline = the fp64 oracle on a bounded
sample of the same workload on this host's cores.

With --gpus N > 1 (launched by torchrun) the matrices are partitioned across
the ranks as in App. F (slorr_partition: longest-processing-time split by
FLOPs; each rank regularizes its subset with grad_scale = N, which the data-
parallel gradient average turns back into lambda): the whole set is done once
per step by all ranks together (strong scaling, no collective on the data
path), and the step time is the max over ranks.  --mode replicas instead has
every rank regularize its own full copy (weak scaling).  --impl reference times the oracle instead.
--op descent times slorr_reg_descent_step instead (the in-place regularizer-only
step W -= eta lambda G of Alg. 1's last line; e2e then copies W in and out).
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
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import workloads  # noqa: E402

METRIC = "regularizer fwd+bwd ms/step & TFLOP/s (% GB300 dense peak) per weight set"
# nominal dense tf32 over bf16 tensor rate on GB300 (1.1 and 2.25 PFLOP/s): the
# tf32 peak is the measured bf16 peak times this ratio
TF32_RATIO = 1.1 / 2.25
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
PROFILE_FILE = os.path.join(ROOT, "profiles", "tc_pair_vit_l16.txt")
# the default tensor-core GEMM (the CTA-pair kernel) and the headers it is built from
TC_SOURCES = [os.path.join(ROOT, "paper_2607_08754_gb300", "csrc", f)
              for f in ("kernels_tc_pair.cu", "tc_common.cuh", "ptx.cuh")]


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--mode", default="partition", choices=["partition", "replicas"],
                    help="N > 1: partition the matrices across ranks (App. F) or run full replicas")
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default="vit_l16", choices=list(workloads.WEIGHT_SETS))
    ap.add_argument("--matrices", type=int, default=0,
                    help="only the first N matrices of the workload (a smaller case of the same shapes, "
                         "for profiling); 0: all")
    ap.add_argument("--variant", default="hoyer", choices=["hoyer", "nuclear"])
    ap.add_argument("--compute", default="fp16", choices=["fp16", "bf16", "fp32", "bf16_split"])
    ap.add_argument("--dtype", default="f32", choices=["f32", "bf16"], help="storage of the weights and grads")
    ap.add_argument("--iters", type=int, default=6)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--flags", type=int, default=0, help="slorr_options.flags (tuning / debug)")
    ap.add_argument("--op", default="fwd_bwd", choices=["fwd_bwd", "descent"],
                    help="fwd_bwd: value + gradient accumulated into .grad (Alg. 2); descent: the in-place "
                         "regularizer-only step W -= eta lambda G (Alg. 1, last line)")
    ap.add_argument("--eta", type=float, default=1e-4, help="step size of --op descent")
    ap.add_argument("--e2e-groups", type=int, default=0,
                    help="groups of the host-buffer pipeline timed as e2e (slorr_pipeline_forward_backward); "
                         "0: about 64 MiB of weights per group, at most 16")
    return ap.parse_args()


def peaks():
    try:
        with open(PEAKS_FILE) as f:
            d = json.load(f)
        return {"hbm": float(d["hbm_gbs"]), "bf16": float(d["bf16_tflops"]),
                "bf16_sustained": float(d["bf16_tflops_sustained"]), "source": "measured"}
    except Exception:
        return {"hbm": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def blas_info() -> dict:
    """numpy's BLAS library and its thread limit, as threadpoolctl or numpy reports them."""
    try:
        from threadpoolctl import threadpool_info
        libs = [d for d in threadpool_info() if d.get("user_api") == "blas"]
        if libs:
            return {"library": libs[0].get("internal_api"), "threads": libs[0].get("num_threads")}
    except Exception:
        pass
    try:
        cfg = np.show_config(mode="dicts")
        blas = cfg.get("Build Dependencies", {}).get("blas", {})
        return {"library": blas.get("name"), "threads": None}
    except Exception:
        return {"library": None, "threads": None}


def oracle_sample(name: str, variant: str, iters: int, budget_s: float, max_steps: int = 1):
    """Times the fp64 oracle on the leading matrices of the weight set until
    about `budget_s` seconds of work; returns (flops, seconds, description)."""
    import oracle
    co = oracle.pe_coefficients(T=iters)
    shapes = workloads.shapes(name)
    flops = 0
    t_total = 0.0
    used = []
    for i, (m, n) in enumerate(shapes):
        W = workloads.generate_one(name, i).astype(np.float64)
        t0 = time.perf_counter()
        oracle.reg_forward_backward([W], variant, co, 1.0)
        t_total += time.perf_counter() - t0
        flops += oracle.pe_flops(m, n, iters)
        used.append(f"{m}x{n}")
        if t_total >= budget_s:
            break
    desc = f"first {len(used)} of {len(shapes)} matrices of {name} ({', '.join(used[:4])}" + \
           (", ..." if len(used) > 4 else "") + f"), fp64 numpy oracle, T={iters}"
    return flops, t_total, desc


def gpu_local_cpus(gpu_index: int):
    """The host CPUs next to the GPU (its PCI device's local_cpulist in sysfs),
    or None.  Page-locked buffers allocated from a thread on them land in the
    GPU's own NUMA node, so host<->device copies do not cross the CPU-CPU link."""
    try:
        out = subprocess.run(["nvidia-smi", f"--id={gpu_index}", "--query-gpu=pci.bus_id",
                              "--format=csv,noheader"], capture_output=True, text=True, timeout=20).stdout.strip()
        dom, rest = out.split(":", 1)
        bus = f"{int(dom, 16):04x}:{rest.lower()}"
        with open(f"/sys/bus/pci/devices/{bus}/local_cpulist") as f:
            text = f.read().strip()
        cpus = set()
        for part in text.split(","):
            if "-" in part:
                a, b = part.split("-")
                cpus.update(range(int(a), int(b) + 1))
            elif part:
                cpus.add(int(part))
        cpus &= os.sched_getaffinity(0)
        return cpus or None
    except Exception:
        return None


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            import tempfile
            fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.out.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            for name, v in zip(names, r[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(name)
        loaded = sorted(sm)[len(sm) // 2:] if sm else []

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        pw = [v for v in (num(r[3]) for r in rows) if v is not None]
        return {"sm_mhz": statistics.median(loaded) if loaded else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons), "samples": len(rows),
                "power_w_median": statistics.median(pw) if pw else None, "power_w_max": max(pw) if pw else None}


def code_only(text: str) -> str:
    """C/CUDA source without its comments, whitespace runs collapsed: what
    the compiler sees, so that a comment edit keeps a capture current."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def tc_source_hash() -> str:
    """sha256 over the code (comments stripped) of the tensor-core kernel's
    source files, in order."""
    h = hashlib.sha256()
    for f in TC_SOURCES:
        h.update(code_only(open(f, encoding="utf-8").read()).encode())
    return h.hexdigest()


def tc_traffic(workload: str, matrices: int, per_phase: bool, compute: str = "fp16"):
    """dram bytes per launch of the tensor-core GEMM from the committed ncu
    summary, or None when the kernel source changed since it was taken, or when
    this run's weight set, matrix count, launch mode or operand mode is not the
    one captured."""
    try:
        src = tc_source_hash()
        vals = {}
        with open(PROFILE_FILE) as f:
            for line in f:
                if ":" in line and not line.startswith("#"):
                    k, v = line.split(":", 1)
                    vals[k.strip()] = v.strip()
        if vals.get("source_sha256") != src:
            return None
        if (vals.get("workload") != workload or int(vals.get("matrices", -1)) != matrices
                or vals.get("launch_mode") != ("per-phase" if per_phase else "dataflow")
                or vals.get("compute") != compute):
            return None
        return float(vals["dram_bytes_per_launch_scaled"])
    except Exception:
        return None


def run_reference(args, rank, world):
    """--impl reference: the fp64 oracle on this host's cores (rank 0 only)."""
    if rank != 0:
        return
    shapes = workloads.shapes(args.workload)
    total_flops = sum(__import__("oracle").pe_flops(m, n, args.iters) for m, n in shapes)
    budget = max(2.0, 120.0 / max(1, args.steps + args.warmup))
    for _ in range(args.warmup):
        oracle_sample(args.workload, args.variant, args.iters, budget * 0.25)
    times = []
    flops_done = 0
    desc = ""
    for _ in range(args.steps):
        f, t, desc = oracle_sample(args.workload, args.variant, args.iters, budget)
        flops_done += f
        times.append(t)
    secs = sum(times)
    tflops = flops_done / secs / 1e12
    ms_full = total_flops / (flops_done / secs) * 1e3
    line = {"metric": METRIC, "value": tflops, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_full, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": f"{args.workload} {args.variant}, T={args.iters}", "matrices": len(shapes)},
            "cpu_baseline": {"value": tflops, "unit": "TFLOP/s", "cores": cpu_cores(), "kind": "oracle",
                             "sample": f"each step: {desc}; ms_per_step extrapolated to the whole set by FLOPs",
                             "blas": blas_info()},
            "e2e": {"value": tflops, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", str(args.gpus)))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return

    import torch
    import torch.distributed as dist

    import __graft_entry__
    __graft_entry__.build() if rank == 0 else None
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        dist.barrier()
    from paper_2607_08754_gb300 import slorr

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    name = args.workload
    set_shapes = workloads.shapes(name)
    if args.matrices > 0:
        set_shapes = set_shapes[: args.matrices]
    partition = args.mode == "partition" and world > 1
    # App. F: this rank's matrices, gradients scaled by the world size
    own = slorr.slorr_partition(set_shapes, world, rank) if partition else list(range(len(set_shapes)))
    assert own, "a rank without matrices: more ranks than matrices"
    shapes = [set_shapes[i] for i in own]
    grad_scale = float(world) if partition else 1.0
    reg = slorr.Regularizer(shapes, variant=args.variant, compute=args.compute, dtype=args.dtype, iters=args.iters,
                            lam=1.0, grad_scale=grad_scale, flags=args.flags)
    tdt = torch.float32 if args.dtype == "f32" else torch.bfloat16
    W_host = [torch.from_numpy(workloads.generate_one(name, i)).to(tdt) for i in own]
    W = [w.to(dev) for w in W_host]
    G = [torch.zeros_like(w) for w in W]
    loss = torch.zeros(1, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    flops_set = slorr.slorr_flops(set_shapes, args.iters)
    flops_step = slorr.slorr_flops(shapes, args.iters)   # this rank's share
    # whole-job FLOPs per step: the set once (partition) or once per rank (replicas)
    flops_job = flops_set if partition else world * flops_set
    flops_exec_t = torch.tensor([slorr.slorr_executed_flops(reg.handle)], dtype=torch.float64, device=dev)
    if world > 1:
        dist.all_reduce(flops_exec_t)   # every rank's padded MMA work (symmetric tiles skipped)
    flops_exec = flops_exec_t.item()

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    descent = args.op == "descent"

    def step(w, g):
        if descent:
            reg.descent_step(w, args.eta, loss=loss)
        else:
            reg(w, g, loss=loss)

    # warm-up
    for _ in range(max(args.warmup, 3)):
        step(W, G)
    barrier()
    assert reg.status() == 0, "device status word reports an error after warm-up"

    # timed region (device-resident inputs).  Per-kernel events would serialise
    # the programmatic dependent launches, so the step time is taken without
    # them and the per-kernel split below in a second timed pass of the same
    # number of steps.
    clocks = ClockSampler(local)
    clocks.start()
    barrier()
    # one event between calls (a call starts with a memset, so this costs no
    # overlap): per-call times for the percentiles
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    evs[0].record(stream)
    for k in range(args.steps):
        step(W, G)
        evs[k + 1].record(stream)
    barrier()
    clk = clocks.stop()
    ms_total = evs[0].elapsed_time(evs[-1])
    per_call = sorted(evs[k].elapsed_time(evs[k + 1]) for k in range(args.steps))
    assert reg.status() == 0, "device status word reports an error in the timed region"
    # per-kernel CUDA events on the call's stream (roofline of the GEMM kernel)
    slorr.slorr_set_timing(reg.handle, True)
    slorr.slorr_read_timing(reg.handle)
    barrier()
    for _ in range(args.steps):
        step(W, G)
    barrier()
    kt = slorr.slorr_read_timing(reg.handle)
    slorr.slorr_set_timing(reg.handle, False)
    ms = torch.tensor([ms_total], dtype=torch.float64, device=dev)
    if world > 1:
        dist.all_reduce(ms, op=dist.ReduceOp.MAX)
    ms_step = ms.item() / args.steps
    value = flops_job / (ms_step * 1e-3) / 1e12
    assert reg.status() == 0, "device status word reports an error in the timed region"

    # e2e: pinned host buffers, copies inside the timed region.  The buffers
    # are allocated, and the copies issued, from the GPU's local CPUs.
    all_cpus = os.sched_getaffinity(0)
    local_cpus = gpu_local_cpus(local)
    if local_cpus:
        os.sched_setaffinity(0, local_cpus)
    Wp = [w.pin_memory() for w in W_host]
    Gp = [torch.zeros_like(w).pin_memory() for w in W_host]
    Lp = torch.zeros(1, dtype=torch.float32).pin_memory()
    Wd = [torch.empty_like(w) for w in W]
    Gd = [torch.empty_like(w) for w in W]
    wbytes = sum(w.numel() * w.element_size() for w in Wp)
    gbytes = 0 if descent else sum(g.numel() * g.element_size() for g in Gp)
    h2d = wbytes + gbytes
    d2h = (wbytes if descent else gbytes) + 4

    pipe = None if descent else slorr.Pipeline(shapes, groups=args.e2e_groups or None, variant=args.variant,
                                               compute=args.compute, dtype=args.dtype, iters=args.iters, lam=1.0,
                                               grad_scale=grad_scale, flags=args.flags)

    def e2e_step():
        if pipe is not None:
            # the public host-buffer call: W and .grad copied in from page-locked
            # host memory, .grad and the loss copied back, per group of matrices,
            # overlapped with the kernels of the other groups
            pipe(Wp, Gp, Wd, Gd, Lp)
            return
        # descent: W in, the updated W and the loss out
        for d, h in zip(Wd, Wp):
            d.copy_(h, non_blocking=True)
        step(Wd, Gd)
        for d, h in zip(Wp, Wd):
            d.copy_(h, non_blocking=True)
        Lp.copy_(loss, non_blocking=True)

    e2e_step()
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.e2e_steps):
        e2e_step()
    e1.record(stream)
    barrier()
    ems = torch.tensor([e0.elapsed_time(e1)], dtype=torch.float64, device=dev)
    if world > 1:
        dist.all_reduce(ems, op=dist.ReduceOp.MAX)
    e2e_ms = ems.item() / args.e2e_steps
    os.sched_setaffinity(0, all_cpus)
    if pipe is not None:
        assert pipe.status() == 0, "device status word reports an error in the e2e region"
    e2e_val = flops_job / (e2e_ms * 1e-3) / 1e12

    if rank == 0:
        pk = peaks()
        gemm_ms = sum(kt[k][0] for k in ("gram", "poly", "update", "gemm"))
        gemm_launches = sum(kt[k][1] for k in ("gram", "poly", "update", "gemm"))
        launches = sum(v[1] for v in kt.values())  # the same launches as the headline timed region
        per_launch_ms = gemm_ms / max(gemm_launches, 1)
        # bf16 hi/lo mode: three bf16 products per product, counted
        split = args.compute == "bf16_split"
        flops_gemm = 3 * flops_step if split else flops_step
        flops_per_launch = flops_gemm * args.steps / max(gemm_launches, 1)
        achieved = flops_per_launch / (per_launch_ms * 1e-3) / 1e12
        peak = pk["bf16"]  # fp16 and bf16 share the dense tensor rate (nominal ratio 1)
        # CUDA-core GEMM (fp32 mode, or the 16-bit check path): bound by FP32
        # instruction issue.  128 FP32 lanes per SM at the maximum SM clock; the
        # compensated (Dot2) multiply-add of fp32 mode takes 10 FP32 operations
        # (product, its FMA error, two-sum, two error adds), the plain one 1.
        simt = bool(args.flags & slorr.FLAG_SIMT_GEMM)
        tf32 = args.compute == "fp32" and not simt
        ops_per_mac = 10 if args.compute == "fp32" else 1
        sm_max = (clk or {}).get("sm_max_mhz") or 2070.0
        nsm = torch.cuda.get_device_properties(dev).multi_processor_count
        alu_peak = nsm * 128 * sm_max * 1e6 * 2 / ops_per_mac / 1e12
        alu_source = ("derived: %d SMs x 128 FP32 lanes x %.0f MHz x 2 FLOP per multiply-add / %d FP32 "
                      "operations per multiply-add" % (nsm, sm_max, ops_per_mac))
        wbytes_dev = sum(w.numel() * w.element_size() for w in W)
        l2_note = ("inputs larger than L2: %s weights %.3f GB (129 MB L2), no flush" % (args.dtype, wbytes_dev / 1e9)
                   if wbytes_dev > 129e6 else
                   "inputs smaller than L2: %s weights %.1f MB, L2-warm timing" % (args.dtype, wbytes_dev / 1e6))
        mem_ms = sum(kt[k][0] for k in ("sumsq", "cast", "normcast", "dot", "combine")) / args.steps
        # memory passes against the measured HBM copy bandwidth: algorithmic bytes per call
        # (sumsq: W; cast: W + the padded iterate; normcast, both in one pass: W + the
        # padded iterate; dot: W + X_T; combine: W + X_T + grad read and written, or W
        # read and written in place for --op descent); passes that did not run are left out
        wsz = 4 if args.dtype == "f32" else 2
        xsz = 4 if args.compute == "fp32" else 2
        elems = sum(m * n for m, n in shapes)
        xelems = sum(((max(m, n) + 127) // 128 * 128) * ((min(m, n) + 127) // 128 * 128) for m, n in shapes)
        comb = (2 * wsz + xsz) if descent else (3 * wsz + xsz)
        mem_bytes = {"sumsq": wsz * elems, "cast": wsz * elems + xsz * xelems,
                     "normcast": wsz * elems + (2 if split else 1) * xsz * xelems, "dot": (wsz + xsz) * elems,
                     "combine": comb * elems}
        memory_roofline = {}
        for k, b in mem_bytes.items():
            if kt[k][1] == 0:
                continue
            t = kt[k][0] / args.steps * 1e-3
            gbs = b / t / 1e9
            memory_roofline[k] = {"bytes": b, "ms": kt[k][0] / args.steps, "achieved_gbs": gbs,
                                  "frac": gbs / pk["hbm"]}
        kernel_breakdown = {k: {"ms_per_step": v[0] / args.steps, "launches_per_step": v[1] / args.steps}
                            for k, v in kt.items()}
        line = {
            "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "strong" if partition else "weak",
            "vs_baseline": None,
            "dtype": {"fp16": "f16", "bf16": "bf16", "bf16_split": "bf16 hi/lo"}.get(args.compute,
                                                                                     "tf32x3" if tf32 else "f32"),
            "data": "synthetic",
            "config": {"workload": f"{name}{' (first %d matrices)' % len(set_shapes) if args.matrices else ''} "
                                   f"{args.variant}{' descent step' if descent else ''}: "
                                   f"{len(set_shapes)} matrices, T={args.iters}, "
                                   f"{args.compute} operands / fp32 accumulate, {args.dtype} weights and grads",
                       "matrices": len(set_shapes), "iters": args.iters, "variant": args.variant, "op": args.op,
                       "gflop_per_step": flops_job / 1e9,
                       "parallelism": (f"layer partition over {world} ranks (App. F), grad_scale {world}; "
                                       f"rank 0 holds {len(shapes)} matrices" if partition else
                                       f"{world} full replicas" if world > 1 else "one GPU"),
                       "l2": l2_note},
            "pct_of_dense_peak": value / world / pk["bf16"],
            "step_ms": {"mean": ms_step, "p10": per_call[len(per_call) // 10],
                        "p50": per_call[len(per_call) // 2], "p90": per_call[(9 * len(per_call)) // 10]},
            "executed": {"gflop_per_step": flops_exec / 1e9,
                         "tflops": flops_exec / (ms_step * 1e-3) / 1e12,
                         "note": "MMA FLOPs the kernels execute: padding included, strictly-lower "
                                 "symmetric tiles skipped"},
            "roofline": ({"bound": "tensor", "achieved": 3 * achieved, "peak": peak * TF32_RATIO, "unit": "TFLOP/s",
                          "frac": 3 * achieved / (peak * TF32_RATIO), "traffic": None,
                          "frac_of_sustained": 3 * achieved / (pk["bf16_sustained"] * TF32_RATIO),
                          "kernel": "tf32_gemm_kernel (Gram/Poly/Update launches: three tf32 products per fp32 "
                                    "product, counted in achieved)",
                          "peak_source": pk["source"] + " bf16 burst x %.4f (nominal dense tf32 / bf16: "
                                                        "1.1 / 2.25 PFLOP/s)" % TF32_RATIO}
                         if tf32 else
                         {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                          "frac": achieved / peak, "traffic": tc_traffic(args.workload, len(shapes), not kt["gemm"][1], args.compute),
                          "frac_of_sustained": achieved / pk["bf16_sustained"],
                          "kernel": "tc_pair_kernel (" + ("one dataflow launch per call: every Gram, Poly and "
                                                          "Update of the T steps" if kt["gemm"][1] else
                                                          "Gram/Poly/Update launches") +
                                    ("; bf16 hi/lo: three bf16 products per product, counted in "
                                     "achieved" if split else "") + ")",
                          "peak_source": pk["source"] + " bf16 burst (fp16 dense rate equal)"}
                         if not simt else
                         {"bound": "alu", "achieved": achieved, "peak": alu_peak, "unit": "TFLOP/s",
                          "frac": achieved / alu_peak, "traffic": None,
                          "kernel": "simt_gemm_kernel (Gram/Poly/Update launches, compensated fp32 sums)"
                                    if args.compute == "fp32" else "simt_gemm_kernel (Gram/Poly/Update launches)",
                          "peak_source": alu_source}),
            "memory_phases_ms_per_step": mem_ms,
            "memory_roofline": memory_roofline,
            "kernels": kernel_breakdown,
            "gpu_launches": launches,
            "e2e": {"value": e2e_val, "unit": "TFLOP/s", "ms_per_step": e2e_ms, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h,
                    "call": "slorr_reg_descent_step with torch copies" if descent else
                            f"slorr_pipeline_forward_backward, {pipe.groups} groups",
                    "host_buffers": ("page-locked, allocated on the GPU's %d local CPUs" % len(local_cpus))
                                    if local_cpus else "page-locked (GPU-local CPUs unknown)"},
            "clocks": clk,
        }
        if not args.no_cpu_baseline and world == 1:
            f, t, desc = oracle_sample(name, args.variant, args.iters, args.cpu_seconds)
            line["cpu_baseline"] = {"value": f / t / 1e12, "unit": "TFLOP/s", "cores": cpu_cores(),
                                    "kind": "oracle", "sample": desc, "blas": blas_info(),
                                    "ms_per_step_est": flops_step / (f / t) * 1e3}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
