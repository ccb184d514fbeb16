"""Benchmark of the GMC layer-boundary compression step on GB300.

python bench.py [--gpus N] [--steps K] [--warmup W] [--workload qwen] [--impl gmc|reference]

One step = one gmc_compress call over one batch of the workload (every stage
of the hot path: message slice, head weights, cosine Gram, client matrix,
selection, assignment, transport, compaction).  Default workload: the
Qwen2.5-VL-7B-shaped boundary (N=1296 on 36x36, T=64, H=28/Hkv=4, d=128,
D=3584, K=257, bf16), synthetic seeded tensors.  Inputs are resident in HBM;
L2 is flushed (a 512 MiB write) before every timed step.  Under torchrun every
rank compresses its own boundaries (independent replicas, weak scaling).

--workload longdoc runs the long-prefix document path instead (N=15876 on
126x126, T=128, K=4096, bounded appearance bank of rank 128 with at most 4096
clients, b=512) through gmc_compress_long.

--impl reference times the fp64 CPU oracle on the host cores on the same
workload (one boundary per step); rank 0 only.
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

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="timed steps (default 400 for gmc: about 0.3 s, several clock samples; 5 for the oracle)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default="qwen")
    ap.add_argument("--impl", default="gmc", choices=["gmc", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--oracle-sample", default=None, help=argparse.SUPPRESS)
    ap.add_argument("--oracle-n", type=int, default=1, help=argparse.SUPPRESS)
    return ap.parse_args()


METRIC = "compressed boundaries/sec (us/boundary) at Qwen2.5-VL-7B shape; % HBM / TC roofline"
UNIT = "boundaries/s"


def long_prefix_cfg(wl):
    """(rademacher map, max_clients, batch_b) of a long-prefix workload, else None."""
    from paper_2608_02134_gb300 import workloads
    cfg = workloads.LONG_PREFIX.get(wl.name)
    if cfg is None:
        return None
    return workloads.rademacher(wl.D, cfg["rank"]), cfg["max_clients"], cfg["batch_b"]


def oracle_step(wl, k: int):
    """One oracle boundary of the workload (image k % B)."""
    import numpy as np
    from oracle import gmc_oracle as O
    f = lambda a: np.asarray(a, dtype=np.float64)
    im = wl.image(k % wl.B)
    lp = long_prefix_cfg(wl)
    p = O.params(batch_b=lp[2]) if lp else O.params()
    long_prefix = {"R": f(lp[0]), "max_clients": lp[1]} if lp else None
    O.compress(f(im.hidden), f(im.keys), f(im.values), f(im.queries), im.pos, f(wl.probe()),
               wl.gh, wl.gw, wl.K, p, long_prefix=long_prefix)


def workload_config(wl) -> dict:
    return {"workload": f"{wl.name}: B={wl.B} N={wl.N} ({wl.gh}x{wl.gw}) T={'ragged' if wl.ragged else wl.T_max} "
                        f"H={wl.H} Hkv={wl.Hkv} d={wl.d} D={wl.D} K={wl.K} {wl.dtype}",
            "boundaries_per_step": wl.B, "l2": "flushed before every timed step (512 MiB write)"}


# ---------------------------------------------------------------------------
# oracle timing (runs in a child process with a fixed BLAS thread count)
# ---------------------------------------------------------------------------
def oracle_sample(name: str, n: int, min_seconds: float = 10.0) -> dict:
    """Oracle boundaries of the workload until min_seconds of CPU work (at most n)."""
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make(name)
    t = 0.0
    k = 0
    while k < n and (k == 0 or t < min_seconds):
        t0 = time.perf_counter()
        oracle_step(wl, k)
        t += time.perf_counter() - t0
        k += 1
    return {"seconds": t, "boundaries": k}


def run_oracle_child(name: str, n: int, cores: int) -> dict:
    env = dict(os.environ)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[v] = str(cores)
    r = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-sample", name,
                        "--oracle-n", str(n)], capture_output=True, text=True, env=env, timeout=1800)
    if r.returncode != 0:
        raise RuntimeError(r.stderr[-2000:])
    return json.loads(r.stdout.strip().splitlines()[-1])


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.th = threading.Thread(target=self._read, daemon=True)
            self.th.start()
        except (FileNotFoundError, OSError):
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
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.th.join(timeout=2)

    def summary(self) -> dict:
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# roofline bookkeeping (algorithmic work per stage, per call)
# ---------------------------------------------------------------------------
# sparse solver rounds run as whole-GPU kernels after the dense first one
# (sparse_gpu_rounds(N) in the library's kernels.cuh)
def wide_rounds(N: int) -> int:
    return 8 if N > 2048 else 4


def stage_work(wl) -> dict:
    """Algorithmic bytes / flops each stage must move or compute for one call."""
    B, N, H, Hkv, d, D, K = wl.B, wl.N, wl.H, wl.Hkv, wl.d, wl.D, wl.K
    es = 2 if wl.dtype == "bf16" else 4
    Tm = sum(wl.T) / B
    lp = long_prefix_cfg(wl)
    MV = min(N, lp[1]) if lp else N
    M = H * Tm + MV + 256
    w = {}
    if lp:  # long prefixes: bounded bank, wide solver, N x K support cosines
        r = lp[0].shape[0]
        w["project"] = ("hbm", B * (N * D * es + N * r * 4.0 + 2 * 2 * N * 3 * r + MV * 3 * r * 2))
        w["app_cos"] = ("hbm", B * (MV * N * 4.0 + (MV + N) * 3 * r * 2))
        w["support_cos"] = ("tensor", B * 2.0 * N * K * D)
        w["select"] = ("hbm", B * -(-K // lp[2]) * (M * N * 4.0))
        w["clients"] = ("hbm", B * (M * N * 4 + H * Tm * N * 4 + MV * N * 4.0))
        w["assign"] = ("hbm", B * (N * K * 4.0))
        w["message"] = ("hbm", B * (H * Tm * N * 4 + 2 * (N + Tm) * Hkv * d * es + Tm * H * d * es))
        w["transport"] = ("hbm", B * ((N + Tm) * D * es + (K + Tm) * D * es
                                      + 2 * (K + Tm) * 2 * Hkv * d * es + 2 * 3 * (K + Tm) * 4 + 3 * N * 4))
        w["heads"] = ("hbm", B * (H * Tm * N * 4))
        w["probe"] = ("hbm", B * N * Hkv * d * es)
        w["rownorm"] = ("hbm", B * N * D * es)
        return w
    # the cosine Gram: the method needs the symmetric half, 2 * N(N+1)/2 * D
    # flops (the kernel issues the 128 x 128 tiles on and above the diagonal)
    w["gram"] = ("tensor", B * 1.0 * N * (N + 1) * D)
    w["message"] = ("hbm", B * (H * Tm * N * 4 + 2 * (N + Tm) * Hkv * d * es + Tm * H * d * es))
    w["clients"] = ("hbm", B * (M * N * 4 + H * Tm * N * 4 + N * N * 4))
    # selection: one read of the M x N clients per round.  Stage "rounds_gpu"
    # runs the dense first round and the next wide_rounds(N) sparse rounds as
    # whole-GPU kernels; stage "select" (the cluster kernel) runs the rest.
    rounds = -(-K // 16)
    wide = min(rounds, 1 + wide_rounds(N))
    w["rounds_gpu"] = ("hbm", B * wide * (M * N * 4.0))
    w["select"] = ("hbm", B * max(1, rounds - wide) * (M * N * 4.0))
    w["transport"] = ("hbm", B * ((N + Tm) * D * es + (K + Tm) * D * es
                                  + 2 * (K + Tm) * 2 * Hkv * d * es + 2 * 3 * (K + Tm) * 4 + 3 * N * 4))
    w["heads"] = ("hbm", B * (H * Tm * N * 4))
    w["assign"] = ("hbm", B * (N * K * 4.0))
    w["probe"] = ("hbm", B * N * Hkv * d * es)
    w["rownorm"] = ("hbm", B * N * D * es)
    return w


# DRAM bytes per launch from an ncu capture (profiles/dram_traffic_qwen.txt); a
# line counts only while the sha256 of its kernel's source files is unchanged.
def recorded_traffic(stage: str):
    import hashlib
    path = os.path.join(ROOT, "profiles", "dram_traffic_qwen.txt")
    try:
        lines = open(path).read().splitlines()
    except OSError:
        return None
    for ln in lines:
        f = dict(kv.split("=", 1) for kv in ln.split() if "=" in kv)
        if f.get("stage") != stage:
            continue
        h = hashlib.sha256()
        for src in f.get("files", "").split(","):
            try:
                h.update(open(os.path.join(ROOT, "paper_2608_02134_gb300", "csrc", src), "rb").read())
            except OSError:
                return None
        if h.hexdigest()[:16] != f.get("sha"):
            return None
        return int(f["dram_bytes"])
    return None


def peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained"), "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


# ---------------------------------------------------------------------------
def run_gmc(args):
    import torch
    import torch.distributed as dist

    from paper_2608_02134_gb300 import gmc, workloads

    from paper_2608_02134_gb300 import replicas

    rank, world, local = replicas.rank_info()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)

    def barrier():
        if world > 1:
            dist.barrier()

    wl = workloads.make(args.workload)
    dt = gmc.GMC_BF16 if wl.dtype == "bf16" else gmc.GMC_F32
    arr = wl.abi_arrays()
    host = {}
    for k, v in arr.items():
        if k == "text_offsets":
            continue
        t = torch.from_numpy(v)
        if v.dtype.name == "uint16":
            t = t.view(torch.int16).view(torch.bfloat16)
        host[k] = t.pin_memory()
    inp = {k: v.to(dev) for k, v in host.items()}
    lpc = long_prefix_cfg(wl)
    lp, params = None, None
    if lpc:
        rmap = torch.from_numpy(lpc[0]).to(torch.bfloat16).to(dev)
        lp = gmc.long_prefix(rmap, lpc[1])
        params = gmc.default_params(batch_b=lpc[2])
    comp = gmc.Compressor(wl.B, wl.gh, wl.gw, wl.T_max, wl.H, wl.Hkv, wl.d, wl.D, wl.K, dt,
                          text_lengths=wl.T if wl.ragged else None, device=dev, params=params,
                          long_prefix=lp)
    flush = torch.empty(512 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step():
        comp.run(inp["hidden"], inp["keys"], inp["queries"], inp["pos_ids"], inp["vo_probe"])

    for _ in range(max(args.warmup, 3)):
        step()
    torch.cuda.synchronize(dev)
    st = comp.status()
    if st != 0:
        raise RuntimeError(f"device status {st:#x} after warm-up")

    # ---- timed region: device-resident inputs --------------------------------
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    launches0 = gmc.launch_count()
    barrier()
    torch.cuda.synchronize(dev)
    with ClockSampler(dev.index or 0) as clk:
        for a, b in evs:
            flush.zero_()
            a.record(stream)
            step()
            b.record(stream)
        torch.cuda.synchronize(dev)
    barrier()
    launches = gmc.launch_count() - launches0
    ms = replicas.max_over_ranks(sum(a.elapsed_time(b) for a, b in evs) / args.steps, dev)
    value = replicas.job_rate(world, wl.B, ms)

    # ---- per-stage profile (separate pass, events on the same stream) --------
    gmc.profile_enable(True)
    prof = {}
    nprof = min(args.steps, 20)
    for _ in range(nprof):
        flush.zero_()
        step()
        for k, v in gmc.profile_read().items():
            prof[k] = prof.get(k, 0.0) + v / nprof
    gmc.profile_enable(False)

    # ---- end to end through pinned host memory --------------------------------
    out_host = {"idx": torch.empty(comp.out_idx.shape, dtype=comp.out_idx.dtype).pin_memory(),
                "hidden": torch.empty(comp.out_hidden.shape, dtype=comp.out_hidden.dtype).pin_memory(),
                "kv": torch.empty(comp.out_kv.shape, dtype=comp.out_kv.dtype).pin_memory(),
                "pos": torch.empty(comp.out_pos.shape, dtype=comp.out_pos.dtype).pin_memory()}
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    d2h = sum(v.numel() * v.element_size() for v in out_host.values())
    e2e_steps = min(args.steps, 20)
    eev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(e2e_steps)]
    def e2e_step():
        if lp is None:
            # gmc_compress_host: the library enqueues the copies, the hidden states'
            # beside the probe, the message slice and the heads
            comp.run_host(host, inp, out_host)
        else:
            for k in inp:
                inp[k].copy_(host[k], non_blocking=True)
            step()
            out_host["idx"].copy_(comp.out_idx, non_blocking=True)
            out_host["hidden"].copy_(comp.out_hidden, non_blocking=True)
            out_host["kv"].copy_(comp.out_kv, non_blocking=True)
            out_host["pos"].copy_(comp.out_pos, non_blocking=True)

    for _ in range(args.warmup):
        e2e_step()
    barrier()
    torch.cuda.synchronize(dev)
    for a, b in eev:
        flush.zero_()
        a.record(stream)
        e2e_step()
        b.record(stream)
    torch.cuda.synchronize(dev)
    barrier()
    e2e_ms = replicas.max_over_ranks(sum(a.elapsed_time(b) for a, b in eev) / e2e_steps, dev)

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    # ---- roofline of the dominant stage ----------------------------------------
    pk = peaks()
    work = stage_work(wl)
    dom = max(prof, key=prof.get) if prof else None

    def roofline(stage):
        bound, amount = work[stage]
        sec = prof[stage] / 1e3
        if bound == "tensor":
            ach, peak, unit = amount / sec / 1e12, pk["bf16_tflops"], "TFLOP/s"
        else:
            ach, peak, unit = amount / sec / 1e9, pk["hbm_gbs"], "GB/s"
        return {"kernel": stage, "bound": bound, "achieved": round(ach, 3), "peak": peak,
                "unit": unit, "frac": round(ach / peak, 5), "peak_source": pk["source"],
                "traffic": recorded_traffic(stage) if wl.name == "qwen" else None,
                "algorithmic": amount, "ms": round(prof[stage], 5)}

    roof = roofline(dom) if dom else None
    stage_roofs = {k: {f: v for f, v in roofline(k).items() if f in ("bound", "achieved", "unit", "frac", "traffic")}
                   for k in prof if k in work}

    cpu = None
    if not args.no_cpu_baseline:
        cores = os.cpu_count() or 1
        try:
            o = run_oracle_child(args.workload, 64, cores)
            cpu = {"value": round(o["boundaries"] / o["seconds"], 6), "unit": UNIT, "cores": cores,
                   "kind": "oracle",
                   "sample": f"{o['boundaries']} boundaries of the {args.workload} workload (about 10 s "
                             f"of CPU work: {o['seconds']:.2f} s), fp64 numpy oracle, one boundary "
                             f"at a time; its matrix products use up to {cores} BLAS threads, the "
                             f"rest runs on one core"}
        except Exception as e:  # keep the GPU line even if the host run fails
            cpu = {"value": None, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": f"failed: {e}"}

    line = {
        "metric": METRIC, "value": round(value, 3), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": max(args.warmup, 3), "ms_per_step": round(ms, 5),
        "us_per_boundary": round(ms * 1000.0 / wl.B, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if wl.dtype == "bf16" else "f32", "data": "synthetic",
        "config": workload_config(wl) | {"parallelism": f"replicas x{world}"},
        "e2e": {"value": round(replicas.job_rate(world, wl.B, e2e_ms), 3), "unit": UNIT,
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": round(e2e_ms, 5)},
        "gpu_launches": int(launches),
        "roofline": roof,
        "stage_roofline": stage_roofs,
        "stages_ms": {k: round(v, 5) for k, v in prof.items()},
        "clocks": clk.summary(),
        "cpu_baseline": cpu,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import numpy as np  # noqa: F401  (thread count fixed by the environment set in main)
    from paper_2608_02134_gb300 import workloads
    wl = workloads.make(args.workload)
    times = []
    for k in range(max(args.warmup, 0) + args.steps):
        t0 = time.perf_counter()
        oracle_step(wl, k)
        if k >= args.warmup:
            times.append(time.perf_counter() - t0)
    sec = sum(times) / len(times)
    value = 1.0 / sec
    cores = int(os.environ.get("OPENBLAS_NUM_THREADS", os.cpu_count() or 1))
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(sec * 1e3, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(wl) | {"parallelism": "host cores",
                                         "boundaries_per_step": 1},
        "cpu_baseline": {"value": round(value, 6), "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"one boundary of the {args.workload} workload per step; "
                                   f"matrix products on up to {cores} BLAS threads, the rest on "
                                   f"one core"},
        "e2e": {"value": round(value, 6), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.steps is None:
        args.steps = 5 if args.impl == "reference" else 400
    if args.oracle_sample:
        print(json.dumps(oracle_sample(args.oracle_sample, args.oracle_n)))
        return
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gmc(args)


if __name__ == "__main__":
    if "--impl" in sys.argv and "reference" in sys.argv:
        n = str(os.cpu_count() or 1)
        for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
            os.environ.setdefault(v, n)
    main()
