"""Benchmark of libfav on one GB300 (or N independent replicas under torchrun).

Headline workload: fp16 MHA causal prefill, B=1, H=32, Nq=Nkv=2048, D=128 -- one step is one
fav_forward call over it (load Q, stream K/V, S = QK^T, causal mask, online softmax,
O += PV, normalise, LSE).  value = attention TFLOP/s (algorithmic FLOPs of the unmasked
pairs: 4 * B * H * D * pairs) over the device time of the timed steps, summed over ranks.
The same JSON line also reports the other workloads of the measurement plan (GQA bf16
prefill with outliers; fp16 GQA and bf16 MQA decode with the split-KV combine, in KV GB/s).

Timing: W warm-up steps, then K timed steps, each bracketed by CUDA events on the launching
stream; L2 is flushed before every timed step by reading a 1 GiB buffer (outside the
events; a read leaves no dirty lines whose write-back would compete with the timed kernel).  e2e = the same metric through the host-buffer C-ABI call fav_forward_host
(pinned host inputs copied in, O and LSE copied out, every step).  cpu_baseline = the fp64
oracle on the host cores on a bounded sample of the workload (rank 0, N=1 only).
--impl reference times that oracle as the reference arm.
"""
import argparse
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

import numpy as np  # noqa: E402

from paper_2608_18656_gb300 import inputs as I  # noqa: E402

HEADLINE = 1          # index of the headline workload in inputs.WORKLOADS
METRIC = "attention TFLOP/s (prefill) and KV GB/s (decode) on 1 GB300, % of roofline"
EXTRA = [0, 2, 3, 4]  # reported alongside (0: the exact fp32 path, timed without a roofline claim)
VARLEN = 0            # index in inputs.VARLEN_WORKLOADS of the packed-batch workload (extra)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="fav", choices=["fav", "reference"])
    ap.add_argument("--no-extra", action="store_true", help="headline workload only")
    ap.add_argument("--extra", default=None,
                    help="comma-separated indices of the extra workloads to time (default: all;"
                         " an empty string: none of them, the packed batch still runs)")
    ap.add_argument("--no-varlen", action="store_true", help="skip the packed-batch workload")
    ap.add_argument("--no-cpu", action="store_true", help="skip the oracle cpu_baseline")
    ap.add_argument("--no-nonflash", action="store_true",
                    help="skip the non-fused comparison (materialised scores) on the headline")
    return ap.parse_args()


# ---------------------------------------------------------------- distributed plumbing
class Dist:
    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        self.device = "cuda"

    def init(self, backend):
        """One process group over the replicas (nccl on GPUs; gloo reduces on the CPU)."""
        if self.world > 1:
            import torch.distributed as dist
            dist.init_process_group(backend)
            self.pg = dist
            self.device = "cpu" if backend == "gloo" else "cuda"

    def barrier(self):
        if self.pg:
            self.pg.barrier()

    def max(self, x):
        if not self.pg:
            return x
        import torch
        t = torch.tensor([x], dtype=torch.float64, device=self.device)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


def job_rate(units_per_rank, seconds_max, world):
    """Whole-job throughput: every rank processes the same units (replicas, weak scaling),
    and the job takes as long as its slowest rank."""
    return units_per_rank * world / seconds_max


# ---------------------------------------------------------------- clocks during timing
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.out = None

    def start(self):
        try:
            self.out = tempfile.TemporaryFile(mode="w+")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except (OSError, ValueError):
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.seek(0)
        rows = [r.split(",") for r in self.out.read().strip().splitlines() if r.strip()]
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 8:
                continue
            try:
                sm.append(float(r[0]))
                smax.append(float(r[1]))
                power.append(float(r[2]))
            except ValueError:
                continue
            for n, val in zip(names, r[4:8]):
                if val.lower().startswith("active"):
                    reasons.add(n)
        busy = [s for s, p in zip(sm, power) if p > 200.0] or sm
        return {"sm_mhz": statistics.median(busy) if busy else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm),
                "power_w_max": max(power) if power else None}


# ---------------------------------------------------------------- helpers
def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        p = json.load(open(path))
        return {"hbm_gbs": p["hbm_gbs"], "tflops": p["bf16_tflops"],
                "tflops_sustained": p.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "tflops": 1900.0, "tflops_sustained": 1700.0,
            "source": "fallback"}


def device_tensors(w, x):
    import torch
    out = []
    for n in ("q", "k", "v"):
        bits = x[n + "_bits"]
        if w.dtype == I.BF16:
            out.append(torch.from_numpy(bits.view(np.int16)).cuda().view(torch.bfloat16))
        else:
            out.append(torch.from_numpy(bits).cuda())
    return out


def kv_bytes(w):
    """Algorithmic decode bytes: K + V + Q + O (I/O dtype) + LSE (fp32), each once."""
    return w.io_bytes


def launches_per_call(fav, w):
    """libfav kernel launches per call: decode 1, plus the split merge (fav_combine_kernel)
    with several splits; prefill 1, plus 2 for bf16 (the V conversion to fp16 and its
    per-head scales)."""
    path = fav.last_path()
    if path == fav.PATH_DECODE:
        return 2 if fav.last_decode_splits() > 1 else 1
    if path == fav.PATH_PREFILL and w.dtype == I.BF16:
        return 3
    return 1


def time_device(fn, steps, warmup, stream, dist):
    """Per-step CUDA-event times (ms) of `fn`, L2 flushed before each timed step.

    The flush READS a 1 GiB buffer (eight times the L2): it evicts the previous step's data and
    leaves only clean lines behind.  (A write-based flush would leave ~126 MB of dirty lines
    whose write-back then competes with the timed kernel's own HBM traffic.)  Its ~150 us of
    device time also keeps the GPU behind the host, so that the host's enqueue time of the
    step never shows up as idle time between the events.
    """
    import torch
    flush = torch.ones(1024 * 1024 * 1024, dtype=torch.uint8, device="cuda")
    sink = torch.empty((), dtype=torch.uint8, device="cuda")
    # Untimed ramp: keep the GPU busy for >= 0.2 s so that its clocks have left their idle
    # state before the warm-up steps proper (a short timed run otherwise starts at idle clocks).
    t_ramp = time.perf_counter()
    while time.perf_counter() - t_ramp < 0.2:
        for _ in range(20):
            fn()
        torch.cuda.synchronize()
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    dist.barrier()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    t0 = time.perf_counter()
    with torch.cuda.stream(stream):
        for s, e in ev:
            torch.amax(flush, dim=0, out=sink)
            s.record(stream)
            fn()
            e.record(stream)
    torch.cuda.synchronize()
    wall = time.perf_counter() - t0
    dist.barrier()
    torch.cuda.synchronize()
    return [s.elapsed_time(e) for s, e in ev], wall


def time_e2e(fav, w, x, steps, warmup):
    """End-to-end: fav_forward_host on pinned host buffers (copies in and out every step)."""
    import torch
    pin = {}
    for n in ("q", "k", "v"):
        a = x[n + "_bits"]
        t = torch.from_numpy(a.view(np.int16) if a.dtype == np.uint16 else a).pin_memory()
        pin[n] = t
    o = torch.empty_like(pin["q"]).pin_memory()
    lse = torch.empty((w.B, w.Hq, w.Nq), dtype=torch.float32).pin_memory()
    stream = torch.cuda.current_stream()

    def call():
        fav.forward_host(pin["q"].data_ptr(), pin["k"].data_ptr(), pin["v"].data_ptr(),
                         o.data_ptr(), lse.data_ptr(), w.B, w.Hq, w.Hkv, w.Nq, w.Nkv, w.D,
                         w.scale, w.causal, w.dtype, stream.cuda_stream)
    for _ in range(warmup):
        call()
    times = []
    for _ in range(steps):
        t0 = time.perf_counter()
        call()
        times.append(time.perf_counter() - t0)
    h2d = sum(pin[n].numel() * pin[n].element_size() for n in ("q", "k", "v"))
    d2h = o.numel() * o.element_size() + lse.numel() * 4
    return statistics.mean(times), h2d, d2h


def oracle_sample(w, budget_rows):
    """Seeded sample of query rows of workload w for the CPU oracle, and its FLOPs."""
    total = w.B * w.Hq * w.Nq
    rng = np.random.Generator(np.random.PCG64(w.seed))
    rows = np.sort(rng.choice(total, size=min(budget_rows, total), replace=False))
    i = rows % w.Nq
    nvis = (w.Nkv - w.Nq + i + 1) if w.causal else np.full_like(i, w.Nkv)
    return rows, float(4 * w.D * nvis.sum())


def run_oracle(w, x, rows):
    import oracle
    t0 = time.perf_counter()
    oracle.attention_rows(x["q"], x["k"], x["v"], rows, w.scale, w.causal)
    return time.perf_counter() - t0, oracle.default_threads()


# ---------------------------------------------------------------- arms
def reference_arm(args, dist):
    """The fp64 oracle as the reference arm (rank 0 only)."""
    if dist.rank != 0:
        return
    w = I.WORKLOADS[HEADLINE]
    x = I.make_inputs(w)
    rows, flops = oracle_sample(w, w.B * w.Hq * w.Nq)
    for _ in range(args.warmup):
        run_oracle(w, x, rows)
    times = []
    cores = 1
    for _ in range(args.steps):
        t, cores = run_oracle(w, x, rows)
        times.append(t)
    ms = statistics.mean(times) * 1e3
    value = flops / (ms * 1e-3) / 1e12
    sample = "%d of %d query rows of %s (seeded), fp64" % (len(rows), w.B * w.Hq * w.Nq, w.name)
    line = {"impl": "reference", "metric": METRIC, "value": value,
            "unit": "TFLOP/s", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "Hq": w.Hq, "Hkv": w.Hkv, "Nq": w.Nq,
                       "Nkv": w.Nkv, "D": w.D, "causal": w.causal},
            "cpu_baseline": {"value": value, "unit": "TFLOP/s", "cores": cores,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def fav_arm(args, dist):
    import torch
    import paper_2608_18656_gb300 as fav
    torch.cuda.set_device(dist.local)
    dist.init("nccl")
    pk = peaks()
    stream = torch.cuda.current_stream()
    sampler = ClockSampler(torch.cuda.current_device()) if dist.rank == 0 else None

    def bench_workload(w, steps, warmup):
        x = I.make_inputs(w)
        q, k, v = device_tensors(w, x)
        o = torch.empty_like(q)
        lse = torch.empty((w.B, w.Hq, w.Nq), dtype=torch.float32, device="cuda")

        def step():
            fav.forward(q, k, v, causal=w.causal, scale=w.scale, out=o, lse_out=lse,
                        stream=stream)
        step()
        torch.cuda.synchronize()
        if fav.device_status() != 0:
            raise RuntimeError("device wait timed out in %s" % w.name)
        nl = launches_per_call(fav, w)
        path = fav.PATH_NAMES[fav.last_path()]
        times, wall = time_device(step, steps, warmup, stream, dist)
        ms = dist.max(statistics.mean(times))
        return x, ms, times, nl, path

    if sampler:
        sampler.start()
    w = I.WORKLOADS[HEADLINE]
    x, ms, times, nl, path = bench_workload(w, args.steps, args.warmup)
    extras = []
    if not args.no_extra:
        chosen = EXTRA if args.extra is None else [int(i) for i in args.extra.split(",") if i]
        for idx in chosen:
            we = I.WORKLOADS[idx]
            _, mse, te, nle, pe = bench_workload(we, args.steps, args.warmup)
            if we.Nq == 1:
                gbs = job_rate(kv_bytes(we), mse * 1e-3, dist.world) / 1e9
                extras.append({"workload": we.name, "value": gbs, "unit": "GB/s",
                               "ms_per_step": mse, "path": pe, "kernel_launches_per_step": nle,
                               "roofline": {"bound": "hbm", "achieved": gbs / dist.world,
                                            "peak": pk["hbm_gbs"], "unit": "GB/s",
                                            "frac": gbs / dist.world / pk["hbm_gbs"],
                                            "frac_of_nominal_7900": gbs / dist.world / 7900.0,
                                            "traffic": traffic_of(we)}})
            elif we.dtype == I.F32:
                tf = job_rate(we.flops, mse * 1e-3, dist.world) / 1e12
                extras.append({"workload": we.name, "value": tf, "unit": "TFLOP/s",
                               "us_per_step": mse * 1e3, "ms_per_step": mse, "path": pe,
                               "kernel_launches_per_step": nle, "roofline": None,
                               "note": "exact fp32 CUDA-core path on 8.4 MFLOP: launch-latency "
                                       "bound, reported without a roofline claim"})
            else:
                tf = job_rate(we.flops, mse * 1e-3, dist.world) / 1e12
                extras.append({"workload": we.name, "value": tf, "unit": "TFLOP/s",
                               "ms_per_step": mse, "path": pe, "kernel_launches_per_step": nle,
                               "roofline": {"bound": "tensor", "achieved": tf / dist.world,
                                            "peak": pk["tflops"], "unit": "TFLOP/s",
                                            "frac": tf / dist.world / pk["tflops"],
                                            "traffic": traffic_of(we)}})
    if not args.no_extra and not args.no_varlen:
        extras.append(bench_varlen(fav, I.VARLEN_WORKLOADS[VARLEN], args, stream, dist, pk))
    nonflash = None
    if not args.no_nonflash:
        nonflash = bench_nonflash(fav, w, x, args, stream, dist, ms)
    clocks = sampler.stop() if sampler else None

    value = job_rate(w.flops, ms * 1e-3, dist.world) / 1e12
    achieved = w.flops / (statistics.mean(times) * 1e-3) / 1e12
    e2e = None
    if True:
        e2e_s, h2d, d2h = time_e2e(fav, w, x, max(3, min(args.steps, 20)), 2)
        e2e_s = dist.max(e2e_s)
        e2e = {"value": job_rate(w.flops, e2e_s, dist.world) / 1e12, "unit": "TFLOP/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}
    cpu = None
    if dist.rank == 0 and dist.world == 1 and not args.no_cpu:
        rows, flops = oracle_sample(w, w.B * w.Hq * w.Nq)
        t, cores = run_oracle(w, x, rows)
        cpu = {"value": flops / t / 1e12, "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
               "sample": "%d of %d query rows of %s, fp64, %.2f s"
                         % (len(rows), w.B * w.Hq * w.Nq, w.name, t)}
    traffic = traffic_of(w)
    line = {
        "metric": METRIC,
        "value": value, "unit": "TFLOP/s", "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": I.DTYPE_NAMES[w.dtype],
        "data": "synthetic (seeded N(0,1) Q/K, U(-1,1) V)",
        "config": {"workload": w.name, "B": w.B, "Hq": w.Hq, "Hkv": w.Hkv, "Nq": w.Nq,
                   "Nkv": w.Nkv, "D": w.D, "causal": w.causal, "path": path,
                   "l2": "flushed before every timed step (1 GiB read, outside the events)",
                   "parallelism": "replicas" if dist.world > 1 else "single GPU"},
        "roofline": {"bound": "tensor", "achieved": achieved, "peak": pk["tflops"],
                     "unit": "TFLOP/s", "frac": achieved / pk["tflops"], "traffic": traffic,
                     "peak_source": pk["source"] + " bf16 dense burst (fp16 taken equal)"},
        "e2e": e2e,
        "gpu_launches": nl * args.steps,
        "clocks": clocks,
        "cpu_baseline": cpu,
        "extra": extras,
        "nonflash": nonflash,
    }
    if dist.rank == 0:
        print(json.dumps(line), flush=True)
    dist.close()


def bench_nonflash(fav, w, x, args, stream, dist, fused_ms):
    """The headline workload through fav_forward_nonflash (two cuBLAS GEMMs around this
    library's masked softmax, the N x N scores in HBM): the non-fused comparison point."""
    import torch
    q, k, v = device_tensors(w, x)
    o = torch.empty_like(q)
    lse = torch.empty((w.B, w.Hq, w.Nq), dtype=torch.float32, device="cuda")
    ws = torch.empty(fav.nonflash_workspace_size(w.B, w.Hq, w.Nq, w.Nkv), dtype=torch.uint8,
                     device="cuda")

    def step():
        fav.forward_nonflash(q, k, v, causal=w.causal, scale=w.scale, out=o, lse_out=lse,
                             workspace=ws, stream=stream)
    try:
        step()
        torch.cuda.synchronize()
    except fav.FavError as e:
        return {"unavailable": str(e)}
    steps = max(3, min(args.steps, 20))
    times, _ = time_device(step, steps, max(3, args.warmup), stream, dist)
    ms = dist.max(statistics.mean(times))
    return {"workload": w.name, "value": job_rate(w.flops, ms * 1e-3, dist.world) / 1e12,
            "unit": "TFLOP/s", "ms_per_step": ms, "steps": steps,
            "fused_speedup": ms / fused_ms,
            "scores_bytes": fav.nonflash_workspace_size(w.B, w.Hq, w.Nq, w.Nkv),
            "kernels": "cuBLAS S = scale Q K^T (fp32 out), fav_nonflash_softmax_kernel, "
                       "cuBLAS O = P V"}


def bench_varlen(fav, w, args, stream, dist, pk):
    """The packed batch of short prompts through fav_prefill_varlen (one call per step: the
    host builds the unit list and copies it to the device, then one launch of the prefill
    kernel)."""
    import torch
    x = I.make_varlen_inputs(w)
    dev = {n: torch.from_numpy(x[n + "_bits"]).cuda() for n in ("q", "k", "v")}
    cu = x["cu_seqlens"]
    o = torch.empty_like(dev["q"])
    lse = torch.empty((w.Hq, int(cu[-1])), dtype=torch.float32, device="cuda")

    def step():
        fav.prefill_varlen(dev["q"], dev["k"], dev["v"], cu, cu, causal=w.causal, scale=w.scale,
                           out=o, lse_out=lse, stream=stream)
    step()
    torch.cuda.synchronize()
    if fav.device_status() != 0:
        raise RuntimeError("device wait timed out in %s" % w.name)
    times, _ = time_device(step, args.steps, args.warmup, stream, dist)
    ms = dist.max(statistics.mean(times))
    tf = job_rate(w.flops, ms * 1e-3, dist.world) / 1e12
    return {"workload": w.name, "value": tf, "unit": "TFLOP/s", "ms_per_step": ms,
            "path": "prefill (packed batch)", "kernel_launches_per_step": 1,
            "sequences": w.n_seq, "tokens": int(cu[-1]),
            "roofline": {"bound": "tensor", "achieved": tf / dist.world, "peak": pk["tflops"],
                         "unit": "TFLOP/s", "frac": tf / dist.world / pk["tflops"],
                         "traffic": traffic_of(w)}}


# Sources each workload's dominant kernel is compiled from (for the traffic record's hash).
KERNEL_SOURCES = {
    "prefill_d128": ("fav_prefill.cu", "fav_device.cuh", "fav_tc.cuh"),
    "prefill_d64": ("fav_prefill_pair.cu", "fav_device.cuh", "fav_tc.cuh"),
    "decode": ("fav_decode.cu", "fav_device.cuh"),
}


def kernel_family(w):
    if getattr(w, "Nq", 0) == 1:
        return "decode"
    return "prefill_d128" if w.D == 128 else "prefill_d64"


def kernel_hash(family="prefill_d128"):
    """Hash of the code (comments and whitespace removed) of the sources a workload's dominant
    kernel is compiled from: a traffic figure recorded under profiles/ is used only while that
    code is unchanged."""
    import hashlib
    import re
    h = hashlib.sha256()
    src = os.path.join(ROOT, "paper_2608_18656_gb300", "csrc")
    for f in KERNEL_SOURCES[family]:
        text = open(os.path.join(src, f)).read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)      # block comments
        text = re.sub(r"//[^\n]*", " ", text)                    # line comments
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()[:16]


def traffic_of(w):
    """DRAM bytes (read + write) of one launch of the workload's dominant kernel, from the ncu
    record in profiles/traffic.json, or None if there is none for the current kernel code."""
    tpath = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(tpath):
        return None
    tr = json.load(open(tpath)).get(w.name)
    if tr and tr.get("kernel_source_hash") == kernel_hash(kernel_family(w)):
        return tr.get("dram_bytes_per_launch")
    return None


def main():
    args = parse()
    dist = Dist()
    if args.impl == "reference":
        reference_arm(args, dist)
        return
    fav_arm(args, dist)


if __name__ == "__main__":
    main()
