"""Throughput of the Gram-Space codebook hot path on GB300.

Headline workload: large-batch fused project + similarity + argmax, bipolar
codebook M = 256, D = 8192, 65,536 queries (codeword + N(0,1) noise), fp32
queries resident in HBM (2 GiB, larger than the 129 MB L2, so no flush is
needed between steps).  One step = one gs_project_similarity call over the
whole batch (argmax + maxval written).  The basis build is initialisation
(paper Sec. 3.3) and is timed separately.

Prints ONE JSON line (rank 0).  `value` is queries/s over all ranks; `e2e`
repeats the measurement through the same API with the queries in pinned host
memory, copied in and the results copied out inside the timed region.
`--impl reference` times the float64 CPU oracle instead (the reference arm).

Multi-GPU: every rank runs its own copy of the workload (independent query
batches, no collective on the data path): weak scaling.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "project+similarity queries/s"
# fp32 FMA peak of the binding kernel (bound "alu"): 152 SMs x 128 fp32 lanes x 2 flop at the
# 2,070 MHz maximum SM clock
FP32_PEAK_TFLOPS = round(152 * 128 * 2 * 2.07e9 / 1e12, 1)
# GB300's nominal HBM3e bandwidth, reported beside the measured copy rate
NOMINAL_HBM_GBS = 8000.0
# rows per staging slot of the end-to-end leg (8192 x 8192 fp32 = 256 MiB a slot)
E2E_CHUNK = 8192
WORKLOAD = "large-batch fused project+similarity+argmax, bipolar M=256, D=8192, 65536 queries (sigma=1)"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--path", default="auto", choices=["auto", "simt", "tensor"])
    p.add_argument("--no-rows", action="store_true", help="skip the per-row side measurements")
    p.add_argument("--no-cpu", action="store_true", help="skip the cpu_baseline leg")
    p.add_argument("--rows", type=int, default=0,
                   help="profiling only: use the first ROWS queries instead of all 65,536")
    p.add_argument("--rows-only", action="store_true",
                   help="profiling only: run just the per-row side measurements and print them")
    return p.parse_args()


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "src": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "src": "fallback"}


def kernel_source_sha(kernel_file, kernel_name):
    """sha256 of one kernel's device source: from its __global__ declaration to the
    file's host-side section marker (edits elsewhere in the file leave it unchanged)."""
    src = open(os.path.join(ROOT, "paper_2608_01528_gb300", "csrc", kernel_file)).read()
    start = src.index(f"\n    {kernel_name}(")
    start = src.rindex("__global__", 0, start)
    end = src.index("// ----------------------------------------------------------------- host side", start)
    return hashlib.sha256(src[start:end].encode()).hexdigest()


def traffic_record(kernel_file, key):
    """DRAM traffic per launch from a committed ncu summary, valid only while the
    kernel's source is unchanged (sha256 of that source recorded next to the number)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)[key]
        h = kernel_source_sha(kernel_file, key.split("/")[0])
        return rec["bytes_per_launch"] if rec.get("source_sha256") == h else None
    except Exception:
        return None


def _cpulist(text):
    cpus = set()
    for part in text.strip().split(","):
        if not part:
            continue
        a, _, b = part.partition("-")
        cpus.update(range(int(a), int(b or a) + 1))
    return cpus


class NearGpuHost:
    """Runs the calling thread on the CPUs attached to the GPU while host buffers are pinned, so
    the pinned pages land on the GPU's NUMA node (pages pinned on the far socket of a two-socket
    node cross the socket link on every host <-> device copy); the affinity is restored after."""

    def __init__(self, index):
        self.index = index
        self.saved = None
        self.node = None
        self.cpus = 0

    def __enter__(self):
        import torch
        try:
            p = torch.cuda.get_device_properties(self.index)
            bus = "%04x:%02x:%02x.0" % (p.pci_domain_id, p.pci_bus_id, p.pci_device_id)
            base = os.path.join("/sys/bus/pci/devices", bus)
            with open(os.path.join(base, "numa_node")) as f:
                self.node = int(f.read())
            with open(os.path.join(base, "local_cpulist")) as f:
                local = _cpulist(f.read())
            self.saved = os.sched_getaffinity(0)
            near = local & self.saved
            if near:
                os.sched_setaffinity(0, near)
                self.cpus = len(near)
        except Exception:  # best effort: no sysfs entry, no affinity API, no device properties
            pass
        return self

    def __exit__(self, *a):
        if self.saved:
            os.sched_setaffinity(0, self.saved)


class ClockSampler:
    """nvidia-smi clock / throttle samples while the timed region runs."""

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.file = None

    def __enter__(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=self.file, stderr=subprocess.DEVNULL)
            time.sleep(0.1)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if getattr(self, "_summary", None) is not None:
            return self._summary
        if self.proc is None or self.file is None:
            return None
        self.file.seek(0)
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.file.read().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        os.unlink(self.file.name)
        self.file = None
        if not sm:
            return None
        self._summary = {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                         "samples": len(sm),
                         "window": "every 50 ms over the timed steps and 0.4 s / 0.3 s of the same step "
                                   "just before / after them"}
        return self._summary


def cpu_baseline(seconds=10.0):
    """The float64 oracle on the host cores, on a bounded sample of the workload."""
    import numpy as np
    import synth
    from oracle import oracle as O
    C = synth.large_codebook()
    Q, R, cn = O.build_basis(C)
    w = synth.large(rows=(0, 256))
    t0 = time.perf_counter()
    O.project_similarity(w["X"], Q, R, cn)
    t1 = time.perf_counter() - t0
    n = int(max(256, min(65536, 256 * seconds / max(t1, 1e-3))) // 256 * 256)
    w = synth.large(rows=(0, n))
    t0 = time.perf_counter()
    out = O.project_similarity(w["X"], Q, R, cn)
    dt = time.perf_counter() - t0
    assert np.array_equal(out["argmax"], w["labels"])
    return {"value": n / dt, "unit": "queries/s", "cores": O.num_threads(), "kind": "oracle",
            "sample": f"first {n} of 65536 queries (float64 oracle: project + similarity + argmax)",
            "seconds": round(dt, 3)}


def max_over_ranks(ms, pg, device):
    """The slowest rank's time (every rank's timed region must end before the job's does);
    `pg` is torch.distributed (any backend) or None for one process."""
    if pg is None:
        return float(ms)
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def job_throughput(units_per_rank, world, steps, ms):
    """Whole-job units per second: every rank processes its own `units_per_rank` per step."""
    return units_per_rank * world * steps / (ms / 1e3)


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    import numpy as np
    import synth
    from oracle import oracle as O
    C = synth.large_codebook()
    Q, R, cn = O.build_basis(C)
    n = 1024
    w = synth.large(rows=(0, n))
    for _ in range(args.warmup):
        O.project_similarity(w["X"][:256], Q, R, cn)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        out = O.project_similarity(w["X"], Q, R, cn)
        times.append(time.perf_counter() - t0)
    assert np.array_equal(out["argmax"], w["labels"])
    dt = sum(times)
    v = n * args.steps / dt
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "queries/s", "n_gpus": 0,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "sample_rows_per_step": n},
            "cpu_baseline": {"value": v, "unit": "queries/s", "cores": O.num_threads(), "kind": "oracle",
                             "sample": f"first {n} of 65536 queries per step"},
            "e2e": {"value": v, "unit": "queries/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
        return
    ws, rank, local = dist_env()
    if args.rows_only:
        import torch
        from paper_2608_01528_gb300 import gramspace as gs
        torch.cuda.set_device(local)
        print(json.dumps({"rows": side_rows(gs, torch.device("cuda", local))}), flush=True)
        return
    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu:
        # the oracle leg runs before CUDA is touched (no forked workers after GPU init)
        cpu = cpu_baseline()

    import numpy as np
    import torch
    import synth
    from paper_2608_01528_gb300 import gramspace as gs

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist

    w = synth.large(rows=(0, args.rows)) if args.rows else synth.large()
    N, D = w["X"].shape
    M = w["C"].shape[0]
    with NearGpuHost(local) as host:
        Xh = torch.from_numpy(w["X"]).pin_memory()
        amh = torch.empty(N, dtype=torch.int32).pin_memory()
        mvh = torch.empty(N, dtype=torch.float32).pin_memory()
    X = Xh.to(dev)
    C = torch.from_numpy(w["C"]).to(dev)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    basis = gs.build_basis(C)
    torch.cuda.synchronize()
    build_ms = 1e3 * (time.perf_counter() - t0)
    r = basis.r
    am = torch.empty(N, dtype=torch.int32, device=dev)
    mv = torch.empty(N, dtype=torch.float32, device=dev)
    outs = {"argmax": am, "maxval": mv}
    stream = torch.cuda.current_stream()

    def step():
        gs.project_similarity(basis, X, path=args.path, out=outs)

    for _ in range(max(3, args.warmup)):
        step()
    gs.stream_status()
    ok = bool(np.array_equal(am.cpu().numpy(), w["labels"]))

    def barrier():
        if pg is not None:
            pg.barrier()
        torch.cuda.synchronize()

    def load(seconds):
        # untimed steps around the timed ones: the timed region itself lasts milliseconds,
        # nvidia-smi samples every 50 ms, so the samples are taken with the GPU under this
        # same load just before, during and just after it
        t_end = time.perf_counter() + seconds
        while time.perf_counter() < t_end:
            for _ in range(16):
                step()
            torch.cuda.synchronize()

    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        load(0.4)
        barrier()
        e0.record(stream)
        for _ in range(args.steps):
            step()
        e1.record(stream)
        barrier()
        load(0.3)
    ms = max_over_ranks(e0.elapsed_time(e1), pg, dev)
    gs.stream_status()
    per_step_ms = ms / args.steps
    value = job_throughput(N, ws, args.steps, ms)

    # end to end through the host-memory entry point: pinned host queries in, argmax /
    # maxval out, streamed through the basis' two staging slots (chunk i copied in while
    # chunk i - 1 is scored); the staging is reserved once, before the timed region
    houts = {"argmax": amh, "maxval": mvh}
    gs.reserve_staging(basis, min(N, E2E_CHUNK))

    def step_e2e():
        gs.project_similarity_host(basis, Xh, path=args.path, out=houts)

    for _ in range(2):
        step_e2e()
    barrier()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ke = max(3, args.steps // 4)
    f0.record(stream)
    for _ in range(ke):
        step_e2e()
    f1.record(stream)
    barrier()
    ms_e2e = max_over_ranks(f0.elapsed_time(f1), pg, dev)
    e2e = {"value": job_throughput(N, ws, ke, ms_e2e), "unit": "queries/s",
           "h2d_bytes_per_step": N * D * 4, "d2h_bytes_per_step": N * 8,
           "call": "gs_project_similarity_host", "chunk_rows": min(N, E2E_CHUNK),
           "host_numa_node": host.node, "host_cpus_near_gpu": host.cpus}
    ok = ok and bool(np.array_equal(amh.numpy(), w["labels"]))

    # roofline of the dominant (only, on the tensor-core path) kernel of the step
    peaks = load_peaks()
    alg_bytes = N * D * 4 + N * 8 + r * D * 2 + M * r * 4
    achieved = alg_bytes / (per_step_ms / 1e3) / 1e9
    tc = args.path == "tensor" or (args.path == "auto" and basis.r <= 256)
    kernel = "k_ps_tc" if tc else "k_gemm (simt)"
    roof = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": round(achieved / peaks["hbm_gbs"], 4), "peak_src": peaks["src"],
            "traffic": traffic_record("gs_tc.cu", "k_ps_tc/large") if tc else None, "kernel": kernel,
            "algorithmic_bytes_per_launch": alg_bytes,
            "frac_of_nominal": round(achieved / NOMINAL_HBM_GBS, 4), "nominal_peak": NOMINAL_HBM_GBS}

    rows = None
    if not args.no_rows and rank == 0:
        rows = side_rows(gs, dev)

    if rank == 0:
        if args.rows:
            WL = WORKLOAD.replace("65536 queries", f"first {N} of 65536 queries (profiling subset)")
        else:
            WL = WORKLOAD
        line = {"metric": METRIC, "value": value, "unit": "queries/s", "n_gpus": ws, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": per_step_ms, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": "f16xf16->f32 (proj), f32 (scores)",
                "data": "synthetic",
                "config": {"workload": WL, "N": N, "D": D, "M": M, "r": r, "path": args.path,
                           "l2": "inputs (2 GiB) larger than L2; no flush", "parallelism": f"replicas x{ws}"},
                "hbm_gbs": round(achieved, 1), "codebook_bytes_ratio": {
                    "coefficient_D_over_r": D / r, "total_MD_over_rD_plus_Mr": (M * D) / (r * D + M * r)},
                "roofline": roof, "e2e": e2e, "gpu_launches": args.steps * (1 if tc else 3),
                "build_ms": round(build_ms, 2), "argmax_matches_labels": ok}
        if cpu is not None:
            line["cpu_baseline"] = cpu
        clocks = clk.summary()
        if clocks is not None:
            line["clocks"] = clocks
        if rows:
            line["rows"] = rows
        print(json.dumps(line), flush=True)
    if pg is not None:
        pg.destroy_process_group()


def side_rows(gs, dev):
    """One timed measurement per other hot-path row (inputs resident in HBM), each
    with its roofline: algorithmic bytes or flops per launch over the measured time,
    against MEASURED_PEAKS.json (HBM copy GB/s; bf16 dense TFLOP/s, which fp16 matches)."""
    import torch
    import synth
    peaks = load_peaks()
    out = {}

    def timeit(fn, reps=10):
        for _ in range(3):
            fn()
        s = torch.cuda.current_stream()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(s)
        for _ in range(reps):
            fn()
        b.record(s)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / reps

    def roof(ms, nbytes, flops, bound):
        sec = ms / 1e3
        d = {"ms": round(ms, 4), "gbs": round(nbytes / sec / 1e9, 1), "tflops": round(flops / sec / 1e12, 1),
             "bound": bound}
        d["frac"] = round(d["gbs"] / peaks["hbm_gbs"] if bound == "hbm" else d["tflops"] / peaks["bf16_tflops"], 4)
        return d

    # basis build (init-time, not rooflined) on the rank-deficient binary codebook
    C4, _ = synth.rankdef_codebook()
    C4d = torch.from_numpy(C4).to(dev)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    b4 = gs.build_basis(C4d)
    torch.cuda.synchronize()
    out["build_rankdef"] = {"ms": round(1e3 * (time.perf_counter() - t0), 2), "r": b4.r}
    r4 = (b4.r + 3) // 4 * 4  # 16-byte rows, as the tensor-core path needs
    # project + similarity with r = 922 > 256 (two tensor-core GEMMs), 16,384 queries
    X4 = torch.from_numpy(synth.rankdef()["X"]).to(dev)
    am = torch.empty(X4.shape[0], dtype=torch.int32, device=dev)
    mv = torch.empty(X4.shape[0], device=dev)
    ms = timeit(lambda: gs.project_similarity(b4, X4, out={"argmax": am, "maxval": mv}))
    N4, D4 = X4.shape
    out["project_similarity_rankdef"] = roof(ms, N4 * D4 * 4, 2 * N4 * D4 * b4.r + 2 * N4 * b4.r * b4.M, "tensor")
    del X4
    # reconstruct 16,384 x 922 -> 16,384 x 10,000
    T = torch.randn(16384, r4, device=dev)[:, :b4.r]
    Xh = torch.empty(16384, 10000, device=dev)
    ms = timeit(lambda: gs.reconstruct(b4, T, out=Xh))
    out["reconstruct_rankdef"] = roof(ms, 16384 * (b4.r + 10000) * 4, 2 * 16384 * b4.r * 10000, "tensor")
    # prob-vectorize + attention on the attention workload (64 x 1024 tokens, r = 512)
    a = synth.attention()
    b5 = gs.build_basis(torch.from_numpy(a["C"]).to(dev))
    Pq = torch.from_numpy(a["Pq"]).to(dev)
    Vq = torch.empty(Pq.shape[0], b5.r, dtype=torch.bfloat16, device=dev)
    ms = timeit(lambda: gs.prob_vectorize(b5, Pq, out=Vq))
    out["probvec_attention"] = roof(ms, Pq.numel() * 4 + Vq.numel() * 2, 2 * Pq.shape[0] * b5.M * b5.r, "hbm")
    # queries and keys from independent probabilities (64 MiB each), scores 256 MiB
    Vk = gs.prob_vectorize(b5, torch.from_numpy(a["Pk"]).to(dev), dtype=torch.bfloat16)
    Vq3, Vk3 = Vq.reshape(64, 1024, -1), Vk.reshape(64, 1024, -1)
    A = torch.empty(64, 1024, 1024, device=dev)
    ms = timeit(lambda: gs.attention_scores(Vq3, Vk3, 1 / 64.0, out=A))
    out["attention"] = roof(ms, (Vq3.numel() + Vk3.numel()) * 2 + A.numel() * 4, 2 * 64 * 1024 * 1024 * b5.r, "hbm")
    # reconstruct + bind at the transition into component-wise operators: 8,192 coefficient rows
    # of the attention basis (r = 512, D = 4096), per-row partners, blocks of 256
    Nb, Lb = 8192, 256
    Tb = torch.from_numpy(synth.attention_probs(12, 1, Nb, b5.M, 1)).to(dev) @ b5.R
    Yb = torch.randn(Nb, b5.D, device=dev)
    Zb = torch.empty(Nb, b5.D, device=dev)
    Xb = torch.empty(Nb, b5.D, device=dev)
    ms_fused = timeit(lambda: gs.reconstruct_bind(b5, Tb, Yb, Lb, out=Zb))
    # one partner row for every row: the basis rows are bound once, one reconstruction GEMM
    ms_fused_one = timeit(lambda: gs.reconstruct_bind(b5, Tb, Yb[:1], Lb, out=Zb))
    ms_rec = timeit(lambda: gs.reconstruct(b5, Tb, out=Xb))
    # binding through block spectra (the default): X, Y read and Z written once, 12 D bytes a row
    ms_bind = timeit(lambda: gs.bind(Xb, Yb, Lb, out=Zb))
    bind_bytes = 3 * Nb * b5.D * 4
    # one partner row for every row (its block spectra computed once per CTA): 8 D bytes a row
    ms_bcast = timeit(lambda: gs.bind(Xb, Yb[:1], Lb, out=Zb))
    # the direct sum for comparison: 2 L flops per output on the fp32 lanes
    ms_direct = timeit(lambda: gs.bind(Xb, Yb, Lb, method="direct", out=Zb))
    direct_tflops = 2 * Nb * b5.D * Lb / (ms_direct / 1e3) / 1e12
    # the fused call (k_rbind_tc: the reconstructed rows stay on chip): T read, Y read, Z written
    fused_bytes = Tb.numel() * 4 + Yb.numel() * 4 + Zb.numel() * 4
    out["reconstruct_bind"] = {"ms": round(ms_fused, 4), "rows": Nb, "D": b5.D, "r": b5.r, "L": Lb,
                               "gbs": round(fused_bytes / (ms_fused / 1e3) / 1e9, 1), "bound": "hbm",
                               "frac": round(fused_bytes / (ms_fused / 1e3) / 1e9 / peaks["hbm_gbs"], 4),
                               "reconstruct_ms": round(ms_rec, 4), "bind_ms": round(ms_bind, 4),
                               "bind_gbs": round(bind_bytes / (ms_bind / 1e3) / 1e9, 1),
                               "bind_frac": round(bind_bytes / (ms_bind / 1e3) / 1e9 / peaks["hbm_gbs"], 4),
                               "bind_one_partner_ms": round(ms_bcast, 4),
                               "one_partner_ms": round(ms_fused_one, 4),
                               "one_partner_gbs": round((Tb.numel() * 4 + Zb.numel() * 4) / (ms_fused_one / 1e3) / 1e9, 1),
                               "bind_direct_ms": round(ms_direct, 4), "bind_direct_tflops": round(direct_tflops, 1),
                               "bind_direct_alu_frac": round(direct_tflops / FP32_PEAK_TFLOPS, 4)}
    del b4, b5, Xb, Yb, Zb
    out["lookup_sweep"] = lookup_sweep(gs, dev)
    out["grouped_attributes"] = grouped_attributes(gs, dev)
    return out


def call_latency(fn, reps=50):
    """Single-call latency in us: events around one call issued to an idle stream, median of
    `reps` calls (host issue time included, as in a lookup)."""
    import torch
    for _ in range(5):
        fn()
    torch.cuda.synchronize()
    s = torch.cuda.current_stream()
    ts = []
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(s)
        fn()
        b.record(s)
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b) * 1e3)
    return round(statistics.median(ts), 1)


def grouped_attributes(gs, dev):
    """The four attribute codebooks (M = 5, 6, 10, 9, D = 1024; 512 queries each): one grouped
    handle scoring all 2,048 queries against all 30 entries plus the per-group argmax (two
    launches), against four handles called one after another.  Launch-bound sizes: latency
    only, no roofline."""
    import numpy as np
    import torch
    import synth
    cases = synth.multiattr()
    C = torch.from_numpy(np.concatenate([a["C"] for a in cases])).to(dev)
    off = np.cumsum([0] + [a["C"].shape[0] for a in cases]).tolist()
    X = torch.from_numpy(np.concatenate([a["X"] for a in cases])).to(dev)
    bg = gs.build_basis_grouped(C, off)
    S = torch.empty(X.shape[0], C.shape[0], device=dev)
    gam = torch.empty(X.shape[0], len(cases), dtype=torch.int32, device=dev)
    t_grouped = call_latency(lambda: (gs.project_similarity(bg, X, want_S=True, want_argmax=False,
                                                            want_maxval=False, out={"S": S}),
                                      gs.group_argmax(S, off, want_maxval=False, out={"argmax": gam})))
    bs = [gs.build_basis(C[off[g]:off[g + 1]].contiguous()) for g in range(len(cases))]
    Xs = [X[off_n:off_n + a["X"].shape[0]] for off_n, a in zip(np.cumsum([0] + [a["X"].shape[0] for a in cases]),
                                                                  cases)]
    ams = [torch.empty(x.shape[0], dtype=torch.int32, device=dev) for x in Xs]

    def separate():
        for b, x, am in zip(bs, Xs, ams):
            gs.project_similarity(b, x, want_maxval=False, out={"argmax": am})

    t_sep = call_latency(separate)
    agree = all(torch.equal(ams[g], gam[n0:n0 + Xs[g].shape[0], g])
                for g, n0 in enumerate(np.cumsum([0] + [x.shape[0] for x in Xs])[:-1]))
    return {"queries": int(X.shape[0]), "groups": len(cases), "unit": "us per batch",
            "grouped_one_handle": t_grouped, "four_handles": t_sep, "argmax_agree": bool(agree)}


def lookup_sweep(gs, dev, reps=50):
    """Similarity-lookup latency across the original dimension D (M = 40, 1,024 lookups per
    batch): uncompressed X Cᵀ + argmax (torch.matmul, fp32: the paper's "original"), the
    compressed lookup on Gram-loc queries (gs_similarity_coeffs: S = Y Rᵀ, no D-dimensional
    work), and projection + compressed scoring from the D-dimensional queries
    (gs_project_similarity).  Single-call latency: events around one call issued to an idle
    stream, median of `reps` calls (host issue time included, as in a lookup)."""
    import torch
    import synth

    def latency(fn):
        return call_latency(fn, reps)

    res = {"M": 40, "lookups_per_batch": 1024, "unit": "us per batch", "D": [], "original_xct": [],
           "compressed_coeffs": [], "project_then_compressed": [], "argmax_agree": True}
    for D in synth.SWEEP_D:
        w = synth.sweep(D)
        C = torch.from_numpy(w["C"]).to(dev)
        X = torch.from_numpy(w["X"]).to(dev)
        b = gs.build_basis(C)
        Y = gs.project_similarity(b, X, want_Y=True, want_argmax=False, want_maxval=False)["Y"]
        am = torch.empty(X.shape[0], dtype=torch.int32, device=dev)
        mv = torch.empty(X.shape[0], device=dev)
        CT = C.t().contiguous()
        t_orig = latency(lambda: torch.matmul(X, CT).argmax(dim=1))
        t_comp = latency(lambda: gs.similarity_coeffs(b, Y, out={"argmax": am, "maxval": mv}))
        t_proj = latency(lambda: gs.project_similarity(b, X, out={"argmax": am, "maxval": mv}))
        gs.similarity_coeffs(b, Y, out={"argmax": am, "maxval": mv})
        agree = bool(torch.equal(am.long(), torch.matmul(X, CT).argmax(dim=1)))
        res["D"].append(D)
        res["original_xct"].append(t_orig)
        res["compressed_coeffs"].append(t_comp)
        res["project_then_compressed"].append(t_proj)
        res["argmax_agree"] = res["argmax_agree"] and agree
        del b
    return res


if __name__ == "__main__":
    main()
