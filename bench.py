"""Benchmark of the W4A4 OBS linear layer set on GB300.

One step = the online hot path of every layer of one DiT block (default: the
PixArt-alpha block at 1024 px, M = 8192 tokens, hidden 1152, b = 64, fp16):
for each of QKV, attention-out, FFN-up and FFN-down, clq_rotate_quant_act
then clq_w4a4_linear (or clq_fused_linear with --fused).  Weight preparation
is offline and untimed.  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl clq|reference]

--impl reference times the CPU oracle on the host cores (bounded row sample
per step) as the reference arm.  Under torchrun every rank runs its own batch
(independent tokens; no collective on the data path): weak scaling.
"""
import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = ("W4A4 linear effective TOPS & us/layer; % INT8 tensor peak; "
          "rotate-quant HBM GB/s")
L2_BYTES = 129 * 1024 * 1024


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=300)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--impl", default="clq", choices=["clq", "reference"])
    p.add_argument("--workload", default="pixart_1024")
    p.add_argument("--fused", action="store_true")
    p.add_argument("--codes", default="auto", choices=list(CODES),
                   help="layouts of the 4-bit weight and activation codes (auto: the "
                        "layer's default, E4M3; packed_w: packed-nibble weights with "
                        "E4M3 activations; packed_a: the reverse; packed: both packed)")
    p.add_argument("--sweep", action="store_true",
                   help="time the 100-cell M x (K, N) x b grid, one JSON line per cell")
    p.add_argument("--bits", action="store_true",
                   help="time the workload at W4A4, W4A8 and W8A8 (separate "
                        "kernels), one JSON line per bit setting")
    p.add_argument("--clip", action="store_true",
                   help="run the per-layer clip search on each layer of the "
                        "workload (offline cost and chosen percentile)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-graph", action="store_true",
                   help="launch the timed steps one call at a time instead of "
                        "replaying one CUDA graph of them")
    p.add_argument("--layer", default=None,
                   help="time only this layer of the workload (profiling)")
    p.add_argument("--tokens", type=int, default=None,
                   help="override the token count M (profiling)")
    p.add_argument("--settle", type=float, default=1.0,
                   help="seconds of untimed steps before timing")
    return p.parse_args()


def layer_ops(cfg, M=None):
    M = cfg["M"] if M is None else M
    return [2.0 * M * N * K for (_, K, N) in cfg["layers"]]


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, 1900.0, "fallback"


# Source files each kernel is built from (globs under csrc/): a recorded ncu
# figure stays valid while these files are unchanged.
KERNEL_SOURCES = {
    "w4a4_gemm": ("w4a4_gemm.cu", "gemm_*.cuh", "clq_device.cuh", "clq_kernels.h"),
    "rotate_quant": ("rotate_quant*.cu", "rq_*.cuh", "clq_device.cuh", "clq_kernels.h"),
    "fused_linear": ("fused_linear.cu", "gemm_*.cuh", "rq_*.cuh", "clq_device.cuh",
                     "clq_kernels.h"),
}


# --codes: (weight layout, activation layout); None = the layer's default.
# Layout numbers: 0 packed INT4 nibbles, 1 E4M3, 3 E2M3 (clq.CLQ_CODES_*).
CODES = {"auto": (None, None), "e4m3": (1, None), "e2m3": (3, None),
         "packed_w": (0, 1), "packed_a": (1, 0), "packed": (0, 0)}


def rq_algorithmic_bytes(M, K):
    """HBM bytes one rotate-quant launch must move, whatever code layout it
    writes: the 16-bit input (2 B an element), the packed INT4 codes (0.5 B an
    element) and one fp32 scale a row: M (2.5 K + 4).  The roofline fraction
    of the kernel is taken on these bytes."""
    return M * (2.5 * K + 4)


def rq_layout_bytes(M, K, code_bytes):
    """Bytes the launch actually moves with `code_bytes` bytes a code (1 for
    the E4M3 layout, 0.75 for E2M3, 0.5 packed, 2 for split 8-bit planes)."""
    return M * ((2.0 + code_bytes) * K + 4)


LAYOUT_NAMES = {0: "int4 packed nibbles", 1: "e4m3", 2: "e4m3 split planes", 3: "e2m3"}


def weight_memory(layers):
    """Resident device bytes of the prepared layers' weight codes, per weight
    and against fp16 (2 B a weight), and of the whole packages (codes, fp32
    scales, swap vectors, biases)."""
    nw = sum(N * K for (_, K, N, _) in layers)
    codes = sum(lay.We.numel() for (_, _, _, lay) in layers)
    total = sum(lay.resident_bytes() for (_, _, _, lay) in layers)
    return {"weight_layout": LAYOUT_NAMES[layers[0][3].w_codes],
            "activation_layout": LAYOUT_NAMES[layers[0][3].act_codes],
            "code_bytes_per_weight": round(codes / nw, 4),
            "fp16_over_codes": round(2.0 * nw / codes, 3),
            "package_bytes": total, "fp16_over_package": round(2.0 * nw / total, 3)}


def gemm_intake_bound(M, shapes, sms, sm_mhz, bytes_per_clk):
    """The GEMM's structural ceiling on this part: TMA fills each SM's shared
    memory with at most `bytes_per_clk` operand bytes per clock (measured in
    the same run by clq_peak_operand_stream, counted in shared-memory bytes,
    which are 128 per row and K step for E4M3 and E2M3 alike), and each 128 x w
    output tile brings (128 + w) K operand bytes in and sends 2 x 128 w output
    bytes out through the same engine.  Tiles are those the launcher picks
    (w = 192 when it covers N in whole tiles with no more rounds, else 256),
    dealt round-robin, so a layer takes ceil(tiles / SMs) tile-times.  Returns
    TFLOP/s over the layer set."""
    rate = bytes_per_clk * sm_mhz * 1e6
    mt = (M + 127) // 128
    t_total, ops = 0.0, 0.0
    for (K, N) in shapes:
        def rounds(w):
            return (mt * ((N + w - 1) // w) + sms - 1) // sms
        w = 192 if rounds(192) * (16 + 192 / 8) < rounds(256) * (16 + 256 / 8) else 256
        t_total += rounds(w) * ((128 + w) * K + 2 * 128 * w) / rate
        ops += 2.0 * M * N * K
    return ops / t_total / 1e12


def job_throughput(local_ms, ops_per_step, steps, world, device=None):
    """Whole-job rate of a weak-scaling run: every rank processes its own
    batch, so the job takes the slowest rank's time; returns (that time in
    ms, all ranks' operations / that time in TOPS).  With world > 1 it needs
    an initialised process group (nccl on GPUs, gloo in the CPU tests)."""
    import torch
    import torch.distributed as dist
    ms = float(local_ms)
    if world > 1:
        t = torch.tensor([ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return ms, ops_per_step * steps * world / (ms * 1e-3) / 1e12


def kernel_source_sha(kernel):
    import glob
    csrc = os.path.join(ROOT, "paper_2509_24416_gb300", "csrc")
    files = sorted({f for pat in KERNEL_SOURCES[kernel]
                    for f in glob.glob(os.path.join(csrc, pat))})
    h = hashlib.sha256()
    for path in files:
        with open(path, "rb") as f:
            h.update(os.path.basename(path).encode() + f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel, workload):
    """DRAM bytes per launch from a committed ncu summary, if it was taken
    on the kernel's current sources; else None."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
    except (OSError, ValueError):
        return None
    e = d.get(kernel, {}).get(workload)
    if not e or e.get("source_sha") != kernel_source_sha(kernel):
        return None
    return e.get("bytes_per_launch")


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,"
         "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid):
        self.uuid = uuid
        self.proc = None

    def start(self):
        cmd = ["nvidia-smi", "--query-gpu=" + self.Q, "--format=csv,noheader,nounits",
               "-lms", "50"]
        if self.uuid:
            cmd += ["-i", self.uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        self.proc.terminate()
        out, _ = self.proc.communicate(timeout=10)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": max(mx),
                "samples": len(sm), "reasons": sorted(reasons)}


# ------------------------------------------------------------- CPU oracle --
def _oracle_sample_worker(args):
    """Runs in a fresh (spawned) single-threaded process."""
    workload, rows, reps = args
    import oracle
    from paper_2509_24416_gb300 import synth
    cfg = synth.WORKLOADS[workload]
    prepared = []
    for li in range(len(cfg["layers"])):
        d = synth.layer_inputs(cfg, li, M=rows)
        perm = oracle.build_permutation(oracle.outlier_scores(d["calib"]))
        Wq, s_w, _, _ = oracle.prepare_weights(d["W32"], perm, cfg["b"])
        prepared.append((d["X32"], perm, Wq, s_w, d["bias32"]))
    times = []
    for _ in range(reps):
        t0 = time.perf_counter()
        for (x, perm, Wq, s_w, bias) in prepared:
            Xq, s_x, _, _ = oracle.rotate_quant_act(x, perm, cfg["b"])
            oracle.w4a4_linear(Xq, s_x, Wq, s_w, cfg["b"], bias)
        times.append(time.perf_counter() - t0)
    return times


def run_oracle(workload, rows, reps):
    import multiprocessing as mp
    env = {"OMP_NUM_THREADS": "1", "OPENBLAS_NUM_THREADS": "1",
           "MKL_NUM_THREADS": "1"}
    old = {k: os.environ.get(k) for k in env}
    os.environ.update(env)
    try:
        ctx = mp.get_context("spawn")
        with ctx.Pool(1) as pool:
            return pool.apply(_oracle_sample_worker, ((workload, rows, reps),))
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def _oracle_slice_worker(workload, rows, w, nworkers, barrier, out):
    """One process of the all-core oracle run: token rows [w rows, (w + 1) rows)
    of a batch of rows * nworkers tokens, prepared untimed, then timed once
    after every worker has reached the barrier."""
    import oracle
    from paper_2509_24416_gb300 import synth
    cfg = synth.WORKLOADS[workload]
    prepared = []
    for li in range(len(cfg["layers"])):
        d = synth.layer_inputs(cfg, li, M=rows * nworkers)
        perm = oracle.build_permutation(oracle.outlier_scores(d["calib"]))
        Wq, s_w, _, _ = oracle.prepare_weights(d["W32"], perm, cfg["b"])
        prepared.append((d["X32"][w * rows:(w + 1) * rows], perm, Wq, s_w, d["bias32"]))
    barrier.wait()
    t0 = time.perf_counter()
    for (x, perm, Wq, s_w, bias) in prepared:
        Xq, s_x, _, _ = oracle.rotate_quant_act(x, perm, cfg["b"])
        oracle.w4a4_linear(Xq, s_x, Wq, s_w, cfg["b"], bias)
    out.put((w, t0, time.perf_counter()))


def run_oracle_all_cores(workload, rows, nworkers):
    """The oracle on `nworkers` single-threaded spawned processes at once,
    each on its own slice of `rows` tokens; returns the wall time from the
    first start to the last end (perf_counter is system-wide monotonic)."""
    import multiprocessing as mp
    env = {"OMP_NUM_THREADS": "1", "OPENBLAS_NUM_THREADS": "1",
           "MKL_NUM_THREADS": "1"}
    old = {k: os.environ.get(k) for k in env}
    os.environ.update(env)
    try:
        ctx = mp.get_context("spawn")
        barrier = ctx.Barrier(nworkers)
        out = ctx.Queue()
        procs = [ctx.Process(target=_oracle_slice_worker,
                             args=(workload, rows, w, nworkers, barrier, out))
                 for w in range(nworkers)]
        for p in procs:
            p.start()
        res = [out.get() for _ in procs]
        for p in procs:
            p.join()
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    return max(r[2] for r in res) - min(r[1] for r in res)


def cpu_baseline(workload, budget_s=20.0):
    """The oracle as it stands on the host cores: one core (a spawned
    single-threaded process, best of 2) and every core (`os.cpu_count()`
    single-threaded processes on disjoint token slices, one pass)."""
    from paper_2509_24416_gb300 import synth
    cfg = synth.WORKLOADS[workload]
    probe_rows = 16
    t = run_oracle(workload, probe_rows, 1)[0]
    rows = int(max(16, min(cfg["M"], probe_rows * budget_s / max(t, 1e-3) / 2)))
    times = run_oracle(workload, rows, 2)
    sec1 = min(times)
    one = sum(layer_ops(cfg, rows)) / sec1 / 1e12
    ncores = os.cpu_count() or 1
    rows_w = int(max(1, min(cfg["M"] // ncores, rows)))
    sec_n = run_oracle_all_cores(workload, rows_w, ncores)
    alln = sum(layer_ops(cfg, rows_w * ncores)) / sec_n / 1e12
    return {"value": alln, "unit": "TOPS", "cores": ncores, "nproc": ncores,
            "kind": "oracle",
            "sample": "%d tokens per core (%d in all) of %d per layer, all %d layers, "
                      "rotate-quant + int64 GEMM + fp64 epilogue, numpy, %d single-threaded "
                      "processes at once, one pass" % (rows_w, rows_w * ncores, cfg["M"],
                                                       len(cfg["layers"]), ncores),
            "single_core": {"value": one, "unit": "TOPS", "cores": 1,
                            "sample": "%d of %d tokens per layer, best of 2" % (rows, cfg["M"])}}


def reference_arm(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2509_24416_gb300 import synth
    cfg = synth.WORKLOADS[args.workload]
    n = args.steps + args.warmup
    t = run_oracle(args.workload, 16, 1)[0]
    per_step_budget = 150.0 / max(n, 1)
    rows = int(max(1, min(cfg["M"], 16 * per_step_budget / max(t, 1e-3))))
    times = run_oracle(args.workload, rows, n)[args.warmup:]
    sec = float(np.sum(times))
    ops = sum(layer_ops(cfg, rows)) * args.steps
    value = ops / sec / 1e12
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "TOPS",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * sec / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64/int64",
        "data": "synthetic",
        "config": dict(config_dict(cfg, args), path="oracle (numpy, one host core)",
                       launch="host", l2="n/a (host)"),
        "cpu_baseline": {"value": value, "unit": "TOPS", "cores": 1,
                         "kind": "oracle",
                         "sample": "%d of %d tokens per layer per step" % (rows, cfg["M"])},
        "e2e": {"value": value, "unit": "TOPS", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def config_dict(cfg, args):
    return {"workload": args.workload + ("" if args.layer is None else ":" + args.layer),
            "tokens": cfg["M"], "b": cfg["b"],
            "layers": ["%s %dx%d" % (n, K, N) for (n, K, N) in cfg["layers"]],
            "io_dtype": cfg["dtype"], "path": "fused" if args.fused else "separate",
            "launch": "eager" if getattr(args, "no_graph", False) else "one cuda graph of the K steps",
            "l2": "inputs rotated over sets totalling > 2x L2 (129 MB)",
            **({} if getattr(args, "codes", "auto") == "auto" else {"codes": args.codes})}


# ------------------------------------------------------------------ sweep ---
SWEEP_M = (256, 1024, 4096, 16384, 65536)
SWEEP_KN = ((1152, 1152), (1152, 4608), (4608, 1152), (3072, 12288), (12288, 3072))
SWEEP_B = (32, 64, 128, 256)


def run_sweep(args):
    """The 100-cell grid: M x (K, N) x b, each valid cell timed as
    rotate-quant alone, rotate-quant + GEMM, the fused kernel and fp16 cuBLAS
    (torch.addmm, independent of b), with inputs of the 256-token case's
    distribution (N(0, 1), 8 channels x 40) generated on the device from a
    fixed seed and rotated over sets larger than L2.  One JSON line per cell."""
    import torch
    from paper_2509_24416_gb300 import clq
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    clq.load()
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    gen = torch.Generator(device=dev)

    def timed(fn, est_us, graph=True):
        """us per call of fn(k, stream_ptr), `reps` calls back to back, replayed
        from one CUDA graph (no host launch work between them) or, with
        graph=False, launched eagerly."""
        reps = int(min(50, max(5, 200000.0 / max(est_us, 1.0))))
        for k in range(3):
            fn(k, sp)
        torch.cuda.synchronize()
        g = None
        if graph:
            cs = torch.cuda.Stream(device=dev)
            cs.wait_stream(stream)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=cs):
                for k in range(reps):
                    fn(k, cs.cuda_stream)
            torch.cuda.synchronize()
            g.replay()
            torch.cuda.synchronize()
        a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        if g is not None:
            g.replay()
        else:
            for k in range(reps):
                fn(k, sp)
        z.record(stream)
        torch.cuda.synchronize()
        return 1e3 * a.elapsed_time(z) / reps

    for (K, N) in SWEEP_KN:
        gen.manual_seed(1)
        W = (torch.randn(N, K, device=dev, generator=gen) * 0.02).half()
        bias = (torch.randn(N, device=dev, generator=gen) * 0.01).half()
        # outlier scores without ties (a calibration mean never ties exactly):
        # U(0, 1) for ordinary channels, 40 for the 8 outlier channels
        cg = torch.Generator().manual_seed(3)
        scores = torch.rand(K, generator=cg)
        scores[torch.randperm(K, generator=cg)[:8]] = 40.0
        perm = clq.build_permutation(scores).to(dev)
        prepared = {b: clq.PreparedLinear.from_weight(W, perm, b, bias=bias)
                    for b in SWEEP_B if K % b == 0}
        for M in SWEEP_M:
            xbytes = M * K * 2
            nsets = max(2, math.ceil(2 * L2_BYTES / xbytes) + 1)
            gen.manual_seed(0)
            outl = (scores > 2).to(dev)
            xs = []
            for _ in range(nsets):
                x = torch.randn(M, K, device=dev, generator=gen)
                x[:, outl] *= 40.0
                xs.append(x.half())
                del x
            Y = torch.empty((M, N), dtype=torch.float16, device=dev)
            xq = torch.empty((M, K), dtype=torch.uint8, device=dev)  # widest 4-bit layout
            s_x = torch.empty(M, dtype=torch.float32, device=dev)
            ws = clq.fused_workspace(M, K, dev)
            ops = 2.0 * M * N * K
            # cuBLAS in its faster launch mode (graph capture or eager)
            cub = lambda k, s_ptr: torch.addmm(bias, xs[k % nsets], W.t(), out=Y)  # noqa: E731
            cub_us = min(timed(cub, ops / 1.5e6), timed(cub, ops / 1.5e6, graph=False))
            for b in SWEEP_B:
                cell = {"M": M, "K": K, "N": N, "b": b}
                if K % b:
                    cell.update({"valid": False, "reason": "K % b != 0"})
                    print(json.dumps(cell), flush=True)
                    continue
                lay = prepared[b]

                def rq(k, s_ptr):
                    st = clq.clq_rotate_quant_act(xs[k % nsets].data_ptr(), clq.CLQ_F16, M, K, K,
                                                  perm.data_ptr(), b, lay.act_codes,
                                                  xq.data_ptr(), s_x.data_ptr(), None, s_ptr)
                    if st:
                        raise clq.ClqError(st, "clq_rotate_quant_act")

                def sep(k, s_ptr):
                    rq(k, s_ptr)
                    st = clq.clq_w4a4_linear(xq.data_ptr(), lay.act_codes, s_x.data_ptr(),
                                             lay.We.data_ptr(), lay.w_codes,
                                             lay.s_w.data_ptr(), lay.bias.data_ptr(), M, N, K, b,
                                             clq.CLQ_F16, Y.data_ptr(), None, s_ptr)
                    if st:
                        raise clq.ClqError(st, "clq_w4a4_linear")

                def fused(k, s_ptr):
                    st = clq.clq_fused_linear(xs[k % nsets].data_ptr(), clq.CLQ_F16, M, K, K,
                                              perm.data_ptr(), b, lay.We.data_ptr(),
                                              lay.w_codes, lay.s_w.data_ptr(),
                                              lay.bias.data_ptr(), N, Y.data_ptr(),
                                              ws.data_ptr(), ws.numel(), s_ptr)
                    if st:
                        raise clq.ClqError(st, "clq_fused_linear")

                rq_us = timed(rq, xbytes / 3e6)
                sep_us = timed(sep, ops / 2.5e6 + rq_us)
                fu_us = timed(fused, ops / 2.5e6 + rq_us)
                cell.update({
                    "valid": True,
                    "rotate_quant_us": round(rq_us, 2),
                    "rotate_quant_GBps": round(rq_algorithmic_bytes(M, K) / (rq_us * 1e-6) / 1e9,
                                               1),
                    "separate_us": round(sep_us, 2),
                    "separate_TOPS": round(ops / (sep_us * 1e-6) / 1e12, 1),
                    "fused_us": round(fu_us, 2),
                    "fused_TOPS": round(ops / (fu_us * 1e-6) / 1e12, 1),
                    "fp16_cublas_us": round(cub_us, 2),
                    "fp16_cublas_TOPS": round(ops / (cub_us * 1e-6) / 1e12, 1),
                    "speedup_separate_vs_cublas": round(cub_us / sep_us, 3),
                    "speedup_fused_vs_cublas": round(cub_us / fu_us, 3),
                })
                print(json.dumps(cell), flush=True)
            del xs, Y, xq, s_x, ws
            torch.cuda.empty_cache()
    status = clq.device_status()
    if status != 0:
        raise RuntimeError("device status %s" % clq.STATUS.get(status, status))


BIT_SETTINGS = (("w4a4", 4, 4, False), ("w4a8", 8, 4, False), ("w8a8", 8, 8, False),
                ("w4a4_asym", 4, 4, True), ("w4a8_asym", 8, 4, True),
                ("w8a8_asym", 8, 8, True))
ERR_ROWS = 512  # token rows per layer for the output-error figure


def run_bits(args):
    """The workload's layers at the paper's three bit settings (Sec. 4.1),
    with symmetric and with asymmetric (Eq. 1, zero-point epilogue)
    activation codes, rotate-quant + GEMM as separate kernels on synthetic
    inputs rotated over sets larger than L2: per layer the rotate-quant and
    GEMM durations (CUDA events around each kernel, after warm-up), per
    setting the whole step (events around the step only), and the output's
    relative Frobenius error against the fp64 product X W^T + bias on the
    first ERR_ROWS tokens of each layer.  One JSON line per setting."""
    import torch
    from paper_2509_24416_gb300 import clq, synth
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    clq.load()
    cfg = dict(synth.WORKLOADS[args.workload])
    if args.tokens is not None:
        cfg["M"] = int(args.tokens)
    M, b = cfg["M"], cfg["b"]
    td = {"f16": torch.float16, "bf16": torch.bfloat16}[cfg["dtype"]]
    stream = torch.cuda.current_stream()
    data = []
    for li in range(len(cfg["layers"])):
        d = synth.layer_inputs(cfg, li)
        calib = torch.from_numpy(d["calib"]).to(td).to(dev)
        perm = clq.build_permutation(clq.outlier_scores(calib)).to(dev)
        data.append((d, perm))
    set_bytes = sum(d["X"].numel() * 2 for d, _ in data)
    nsets = max(2, math.ceil(2 * L2_BYTES / set_bytes) + 1)
    xsets = [[d["X"].to(dev) for d, _ in data] for _ in range(nsets)]
    base_tops = None
    refs = []
    for d, _ in data:
        x64 = d["X32"][:ERR_ROWS].astype("float64")
        refs.append(x64 @ d["W32"].astype("float64").T + d["bias32"].astype("float64")[None, :])
    for name, a_bits, w_bits, asym in BIT_SETTINGS:
        # asymmetric 4-bit codes reach -8, which only the E4M3 layout holds
        w4 = clq.CLQ_CODES_E4M3 if asym and w_bits == 4 else None
        lays = [clq.PreparedLinear.from_weight(d["W"].to(dev), perm, b, bias=d["bias"].to(dev),
                                               a_bits=a_bits, w_bits=w_bits, w_codes=w4)
                for d, perm in data]
        wsums = [clq.weight_code_sums(lay.We, d["K"]) for lay, (d, _) in zip(lays, data)]
        x_codes = lays[0].act_codes
        w_codes = lays[0].w_codes
        xq = [torch.empty((M, clq.codes_width(x_codes, d["K"])), dtype=torch.uint8, device=dev)
              for d, _ in data]
        sx = [torch.empty(M, dtype=torch.float32, device=dev) for _ in data]
        los = [torch.empty(M, dtype=torch.float32, device=dev) for _ in data]
        ys = [torch.empty((M, d["N"]), dtype=td, device=dev) for d, _ in data]

        sp = stream.cuda_stream
        dt = clq._dt(xsets[0][0])

        def step(k, ev=None):
            xs = xsets[k % nsets]
            for i, lay in enumerate(lays):
                K, N = data[i][0]["K"], data[i][0]["N"]
                if ev is not None:
                    ev[3 * i].record(stream)
                if asym:
                    st = clq.clq_rotate_quant_act_asym(xs[i].data_ptr(), dt, M, K, K,
                                                       lay.perm.data_ptr(), b, x_codes,
                                                       xq[i].data_ptr(), sx[i].data_ptr(),
                                                       los[i].data_ptr(), None, sp)
                else:
                    st = clq.clq_rotate_quant_act(xs[i].data_ptr(), dt, M, K, K,
                                                  lay.perm.data_ptr(), b, x_codes,
                                                  xq[i].data_ptr(), sx[i].data_ptr(), None, sp)
                if st:
                    raise clq.ClqError(st, "rotate-quant")
                if ev is not None:
                    ev[3 * i + 1].record(stream)
                if asym:
                    st = clq.clq_linear_asym(xq[i].data_ptr(), x_codes, sx[i].data_ptr(),
                                             los[i].data_ptr(), lay.We.data_ptr(), w_codes,
                                             lay.s_w.data_ptr(), wsums[i].data_ptr(),
                                             lay.bias.data_ptr(), M, N, K, b, dt,
                                             ys[i].data_ptr(), None, sp)
                else:
                    st = clq.clq_linear(xq[i].data_ptr(), x_codes, sx[i].data_ptr(),
                                        lay.We.data_ptr(), w_codes, lay.s_w.data_ptr(),
                                        lay.bias.data_ptr(), M, N, K, b, dt, ys[i].data_ptr(),
                                        None, sp)
                if st:
                    raise clq.ClqError(st, "product")
                if ev is not None:
                    ev[3 * i + 2].record(stream)

        for k in range(max(3, args.warmup)):
            step(k)
        torch.cuda.synchronize()
        a0, z0 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        for k in range(args.steps):
            step(k)
        z0.record(stream)
        torch.cuda.synchronize()
        step_ms = a0.elapsed_time(z0) / args.steps
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3 * len(lays))]
               for _ in range(args.steps)]
        for k in range(args.steps):
            step(k, evs[k])
        torch.cuda.synchronize()
        ops = sum(2.0 * M * d["N"] * d["K"] for d, _ in data)
        per_layer = []
        for i, (d, _) in enumerate(data):
            rq = sum(e[3 * i].elapsed_time(e[3 * i + 1]) for e in evs) / args.steps
            gm = sum(e[3 * i + 1].elapsed_time(e[3 * i + 2]) for e in evs) / args.steps
            K, N = d["K"], d["N"]
            # algorithmic bytes at this activation width: 16-bit input, packed
            # codes (bits / 8 B a code), the per-row scale (and minimum)
            rq_bytes = M * (2.0 * K + (a_bits / 8.0) * K + (8 if asym else 4))
            y = ys[i][:ERR_ROWS].double().cpu().numpy()
            err = float(((y - refs[i]) ** 2).sum() ** 0.5 / (refs[i] ** 2).sum() ** 0.5)
            per_layer.append({
                "layer": d["name"], "K": K, "N": N, "rel_err": round(err, 5),
                "rotate_quant_us": round(rq * 1e3, 2),
                "rotate_quant_GBps": round(rq_bytes / (rq * 1e-3) / 1e9, 1),
                "gemm_us": round(gm * 1e3, 2),
                "gemm_TOPS": round(2.0 * M * N * K / (gm * 1e-3) / 1e12, 1)})
        tops = ops / (step_ms * 1e-3) / 1e12
        base_tops = tops if base_tops is None else base_tops
        print(json.dumps({
            "bits": name, "workload": args.workload, "tokens_per_layer": M, "b": b,
            "value": round(tops, 1), "unit": "TOPS", "ms_per_step": round(step_ms, 4),
            "vs_w4a4": round(tops / base_tops, 3), "steps": args.steps,
            "activations": "asymmetric" if asym else "symmetric",
            "layers": per_layer}), flush=True)
        del lays, xq, sx, ys, los, wsums
        torch.cuda.empty_cache()
    status = clq.device_status()
    if status != 0:
        raise RuntimeError("device status %s" % clq.STATUS.get(status, status))


def run_clip(args):
    """The per-layer clip search (Sec. 3.4, Eq. 3 with the layer as its own
    target) on every layer of the workload: calibration tokens = the first
    --tokens rows (default 1024) of the layer's synthetic input, Yref the
    fp32 product X W^T + bias (torch), the default 11-point grid over
    [0, 0.01].  Reports the wall time of the call (it synchronizes), the
    chosen percentile and the error against the unclipped point.  One JSON
    line per layer."""
    import torch
    from paper_2509_24416_gb300 import clq, synth
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    clq.load()
    cfg = dict(synth.WORKLOADS[args.workload])
    M = int(args.tokens) if args.tokens is not None else 1024
    cfg["M"] = M
    for li in range(len(cfg["layers"])):
        d = synth.layer_inputs(cfg, li)
        calib = torch.from_numpy(d["calib"]).to(d["X"].dtype).to(dev)
        perm = clq.build_permutation(clq.outlier_scores(calib)).to(dev)
        X, W, bias = d["X"].to(dev), d["W"].to(dev), d["bias"].to(dev)
        yref = torch.addmm(bias.float(), X.float(), W.float().t())
        clq.clip_search(W, perm, d["b"], X, yref, bias)  # warm-up
        times = []
        for _ in range(max(1, args.steps)):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            clip, errors, best = clq.clip_search(W, perm, d["b"], X, yref, bias)
            times.append(time.perf_counter() - t0)
        ms = 1e3 * sorted(times)[len(times) // 2]
        G = len(clq.CLIP_GRID)
        ops = G * 2.0 * M * d["N"] * d["K"]
        print(json.dumps({
            "layer": d["name"], "K": d["K"], "N": d["N"], "calib_tokens": M,
            "grid_points": G, "ms": round(ms, 3),
            "inner_products_TOPS": round(ops / (ms * 1e-3) / 1e12, 2),
            "best_p": clq.CLIP_GRID[best],
            "err_unclipped": float(errors[0]), "err_best": float(errors[best]),
            "err_ratio": round(float(errors[best] / errors[0]), 4),
            "errors": [float(e) for e in errors]}), flush=True)
    status = clq.device_status()
    if status != 0:
        raise RuntimeError("device status %s" % clq.STATUS.get(status, status))


# --------------------------------------------------------------- GPU arm ---
def main():
    args = parse()
    if args.impl == "reference":
        reference_arm(args)
        return
    if args.sweep:
        run_sweep(args)
        return
    if args.bits:
        run_bits(args)
        return
    if args.clip:
        run_clip(args)
        return
    import torch
    import torch.distributed as dist
    import ctypes
    from paper_2509_24416_gb300 import clq, synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    clq.load()
    cfg = dict(synth.WORKLOADS[args.workload])
    if args.layer is not None:
        cfg["layers"] = tuple(l for l in cfg["layers"] if l[0] == args.layer)
        if not cfg["layers"]:
            raise SystemExit("no layer %r in %s" % (args.layer, args.workload))
    if args.tokens is not None:
        cfg["M"] = int(args.tokens)
    td = {"f16": torch.float16, "bf16": torch.bfloat16}[cfg["dtype"]]
    b = cfg["b"]
    M = cfg["M"]

    # ---- offline: calibration, swap vectors, prepared weights (untimed) ----
    layers, xs_host, w_dense = [], [], []
    all_names = [l[0] for l in synth.WORKLOADS[args.workload]["layers"]]
    for lname, _, _ in cfg["layers"]:
        li = all_names.index(lname)
        d = synth.layer_inputs(dict(synth.WORKLOADS[args.workload], M=cfg["M"]), li,
                               batch=rank)  # each rank its own token batch
        calib = torch.from_numpy(d["calib"]).to(td).to(dev)
        perm = clq.build_permutation(clq.outlier_scores(calib)).to(dev)
        lay = clq.PreparedLinear.from_weight(d["W"].to(dev), perm, b,
                                             bias=d["bias"].to(dev), w_codes=CODES[args.codes][0],
                                             a_codes=CODES[args.codes][1])
        layers.append((d["name"], d["K"], d["N"], lay))
        xs_host.append(d["X"])
        w_dense.append((d["W"].to(dev), d["bias"].to(dev)))  # fp16 cuBLAS comparator
    set_bytes = sum(x.numel() * 2 for x in xs_host)
    nsets = max(2, math.ceil(2 * L2_BYTES / set_bytes) + 1)
    xsets = [[x.to(dev) for x in xs_host] for _ in range(nsets)]
    xq = [torch.empty((M, clq.codes_width(lay.act_codes, K)), dtype=torch.uint8, device=dev)
          for (_, K, _, lay) in layers]
    sx = [torch.empty(M, dtype=torch.float32, device=dev) for _ in layers]
    ys = [torch.empty((M, N), dtype=td, device=dev) for (_, _, N, _) in layers]
    wss = [clq.fused_workspace(M, K, dev) for (_, K, _, _) in layers]
    stream = torch.cuda.current_stream()
    sp = stream.cuda_stream
    nlay = len(layers)

    def step(si, ev=None, fused=None, s_ptr=None, sets=None):
        fused = args.fused if fused is None else fused
        sp_ = sp if s_ptr is None else s_ptr
        xs = (xsets if sets is None else sets)[si % nsets]
        for i, (_, K, N, lay) in enumerate(layers):
            if ev is not None:
                ev[4 * i].record(stream)
                if fused:  # one kernel: its time is the "gemm" interval
                    ev[4 * i + 1].record(stream)
                    ev[4 * i + 2].record(stream)
            if fused:
                st = clq.clq_fused_linear(xs[i].data_ptr(), clq._dt(xs[i]), M, K, K,
                                          lay.perm.data_ptr(), b, lay.We.data_ptr(),
                                          lay.w_codes, lay.s_w.data_ptr(),
                                          lay.bias.data_ptr(), N, ys[i].data_ptr(),
                                          wss[i].data_ptr(), wss[i].numel(), sp_)
                if st:
                    raise clq.ClqError(st, "clq_fused_linear")
            else:
                st = clq.clq_rotate_quant_act(xs[i].data_ptr(), clq._dt(xs[i]), M, K, K,
                                              lay.perm.data_ptr(), b, lay.act_codes,
                                              xq[i].data_ptr(), sx[i].data_ptr(), None, sp_)
                if st:
                    raise clq.ClqError(st, "clq_rotate_quant_act")
                if ev is not None:
                    ev[4 * i + 1].record(stream)
                    ev[4 * i + 2].record(stream)
                st = clq.clq_w4a4_linear(xq[i].data_ptr(), lay.act_codes,
                                         sx[i].data_ptr(), lay.We.data_ptr(),
                                         lay.w_codes,
                                         lay.s_w.data_ptr(), lay.bias.data_ptr(), M, N, K, b,
                                         clq._dt(ys[i]), ys[i].data_ptr(), None, sp_)
                if st:
                    raise clq.ClqError(st, "clq_w4a4_linear")
            if ev is not None:
                ev[4 * i + 3].record(stream)

    # warm-up, then a clock settle of ~1 s of untimed steps
    for i in range(max(3, args.warmup)):
        step(i)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    n_settle = 0
    while time.perf_counter() - t0 < args.settle:
        step(n_settle)
        n_settle += 1
        if n_settle % 50 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()
    # The K timed steps captured once as one CUDA graph and replayed once in
    # the timed region: the same kernels with the same arguments in the same
    # order, launched without per-call host work, consecutive kernels still
    # overlapping through programmatic dependent launch (also across steps).
    graph = None
    if not args.no_graph:
        cs = torch.cuda.Stream(device=dev)
        cs.wait_stream(stream)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=cs):
            for k in range(args.steps):
                step(k, s_ptr=cs.cuda_stream)
        torch.cuda.synchronize()
        graph.replay()  # one untimed replay
        torch.cuda.synchronize()
    if world > 1:
        dist.barrier()

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        uuid = None
    sampler = ClockSampler(uuid)
    sampler.start()
    time.sleep(0.3)
    # Timed region 1: K steps, events only around the whole region (the
    # reported value).  Timed region 2: the same K steps with events around
    # every kernel (per-kernel durations for the rooflines); event records
    # between kernels serialize the stream, so region 2 is not used for value.
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_start.record(stream)
    if graph is not None:
        graph.replay()
    else:
        for k in range(args.steps):
            step(k)
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    total_ms = t_start.elapsed_time(t_end)
    # Steady state: the same K steps repeated until at least 200 ms have run
    # (at least 3 repeats), events around each repeat; the median per-step
    # time of the repeats is reported beside the value.
    reps = max(3, int(math.ceil(200.0 / max(total_ms, 1e-3))))
    rep_ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(reps)]
    torch.cuda.synchronize()
    for a_ev, z_ev in rep_ev:
        a_ev.record(stream)
        if graph is not None:
            graph.replay()
        else:
            for k in range(args.steps):
                step(k)
        z_ev.record(stream)
    torch.cuda.synchronize()
    rep_ms = [a_ev.elapsed_time(z_ev) for a_ev, z_ev in rep_ev]
    steady = {"repeats": reps, "steps_per_repeat": args.steps,
              "region_ms": round(float(np.sum(rep_ms)), 2),
              "ms_per_step_median": round(float(np.median(rep_ms)) / args.steps, 5),
              "ms_per_step_min": round(float(np.min(rep_ms)) / args.steps, 5),
              "ms_per_step_max": round(float(np.max(rep_ms)) / args.steps, 5)}
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4 * nlay)]
           for _ in range(args.steps)]
    torch.cuda.synchronize()
    for k in range(args.steps):
        step(k, evs[k])
    torch.cuda.synchronize()
    clocks = sampler.stop()

    # ---- context (not part of value): the other path, fp16 cuBLAS on the
    # same layer shapes and rotated inputs, measured peak rates ----
    def time_steps(fn, n, graph=None):
        """ms per call of fn(k, s_ptr) over n calls, launched the way the
        value is (one CUDA graph of the n calls, or eager with --no-graph)."""
        graph = not args.no_graph if graph is None else graph
        for k in range(3):
            fn(k, None)
        torch.cuda.synchronize()
        g = None
        if graph:
            cs = torch.cuda.Stream(device=dev)
            cs.wait_stream(stream)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=cs):
                for k in range(n):
                    fn(k, cs.cuda_stream)
            torch.cuda.synchronize()
            g.replay()
            torch.cuda.synchronize()
        a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        if g is not None:
            g.replay()
        else:
            for k in range(n):
                fn(k, None)
        z.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(z) / n

    other_ms = time_steps(lambda k, s_ptr: step(k, fused=not args.fused, s_ptr=s_ptr),
                          args.steps)
    # The video workload's second token set (the same tokens in temporal
    # order, a pure row permutation): the same layers, the same launch.
    temporal_ms = None
    tcfg = cfg.get("temporal")
    if tcfg is not None and args.layer is None and args.tokens is None:
        tsets = [[synth.temporal_reorder(x, **tcfg).to(dev) for x in xs_host]
                 for _ in range(nsets)]
        temporal_ms = time_steps(lambda k, s_ptr: step(k, s_ptr=s_ptr, sets=tsets), args.steps)
        del tsets

    # Each kernel of the separate path alone, K launches back to back per
    # layer (events around the K launches only): its duration with
    # programmatic dependent launch overlapping its neighbours, as inside the
    # step, without the event records between kernels of region 2.
    rq_b2b, gm_b2b, rq_floor_b2b = None, None, None
    if not args.fused:
        def rq_only(i):
            _, K, N, lay = layers[i]

            def f(k, s_ptr):
                x = xsets[k % nsets][i]
                st = clq.clq_rotate_quant_act(x.data_ptr(), clq._dt(x), M, K, K,
                                              lay.perm.data_ptr(), b, lay.act_codes,
                                              xq[i].data_ptr(), sx[i].data_ptr(), None,
                                              sp if s_ptr is None else s_ptr)
                if st:
                    raise clq.ClqError(st, "clq_rotate_quant_act")
            return f

        def gm_only(i):
            _, K, N, lay = layers[i]

            def f(k, s_ptr):
                st = clq.clq_w4a4_linear(xq[i].data_ptr(), lay.act_codes,
                                         sx[i].data_ptr(), lay.We.data_ptr(),
                                         lay.w_codes, lay.s_w.data_ptr(),
                                         lay.bias.data_ptr(), M, N, K, b,
                                         clq._dt(ys[i]), ys[i].data_ptr(), None,
                                         sp if s_ptr is None else s_ptr)
                if st:
                    raise clq.ClqError(st, "clq_w4a4_linear")
            return f

        rq_b2b = [time_steps(rq_only(i), args.steps) for i in range(nlay)]
        gm_b2b = [time_steps(gm_only(i), args.steps) for i in range(nlay)]

        # The rotate-quant loop's memory side alone on the same inputs and
        # launch (clq_peak_rq_stream: its tiles, copy ring and stores, no
        # arithmetic): the floor its back-to-back time is measured against.
        if all(K % 64 == 0 for (_, K, _, _) in layers):
            fq = torch.empty((M, max(K for (_, K, _, _) in layers)), dtype=torch.uint8,
                             device=dev)
            fs = torch.empty(M, dtype=torch.float32, device=dev)

            def floor_only(i):
                _, K, _, _ = layers[i]
                ops = ctypes.c_int64(0)

                def f(k, s_ptr):
                    x = xsets[k % nsets][i]
                    st = clq.clq_peak_rq_stream(x.data_ptr(), M, K, fq.data_ptr(), fs.data_ptr(),
                                                ctypes.byref(ops), sp if s_ptr is None else s_ptr)
                    if st:
                        raise clq.ClqError(st, "clq_peak_rq_stream")
                return f

            rq_floor_b2b = [time_steps(floor_only(i), args.steps) for i in range(nlay)]
            del fq, fs

    def cublas_step(si, s_ptr=None):
        xs = xsets[si % nsets]
        for i, (w, bias) in enumerate(w_dense):
            torch.addmm(bias, xs[i], w.t(), out=ys[i])

    # cuBLAS gets its faster launch mode (measured: graph capture slows its
    # kernels here)
    cublas_ms = min(time_steps(cublas_step, args.steps, graph=False),
                    time_steps(cublas_step, args.steps, graph=True))
    measured = clq.measure_peaks()
    status = clq.device_status()
    if status != 0:
        raise RuntimeError("device status %s" % clq.STATUS.get(status, status))

    rq_ms = np.zeros(nlay)
    gm_ms = np.zeros(nlay)
    for e in evs:
        for i in range(nlay):
            rq_ms[i] += e[4 * i].elapsed_time(e[4 * i + 1])
            gm_ms[i] += e[4 * i + 2].elapsed_time(e[4 * i + 3])
    ops_step = sum(layer_ops(cfg))
    total_ms, value = job_throughput(total_ms, ops_step, args.steps, world, dev)
    hbm_peak, bf16_peak, peak_src = peaks()
    fp8_peak = 2.0 * bf16_peak  # E4M3 dense rate = 2x bf16 (nominal ratio)
    K_list = [K for (_, K, _, _) in layers]
    N_list = [N for (_, _, N, _) in layers]
    per_layer = []
    gemm_flops = sum(layer_ops(cfg))
    for i, (name, K, N, _) in enumerate(layers):
        rq_us = 1e3 * rq_ms[i] / args.steps
        gm_us = 1e3 * gm_ms[i] / args.steps
        rq_bytes = rq_algorithmic_bytes(M, K)
        per_layer.append({
            "layer": name, "K": K, "N": N,
            "us": round(rq_us + gm_us, 2),
            "rotate_quant_us": round(rq_us, 2),
            "rotate_quant_GBps": round(rq_bytes / (rq_us * 1e-6) / 1e9, 1) if rq_us > 0 else None,
            "gemm_us": round(gm_us, 2),
            "gemm_TOPS": round(2.0 * M * N * K / (gm_us * 1e-6) / 1e12, 1),
        })
        if rq_b2b is not None:
            per_layer[-1]["rotate_quant_us_back_to_back"] = round(1e3 * rq_b2b[i], 2)
            per_layer[-1]["gemm_us_back_to_back"] = round(1e3 * gm_b2b[i], 2)
        if rq_floor_b2b is not None:
            per_layer[-1]["rotate_quant_copy_floor_us_back_to_back"] = round(
                1e3 * rq_floor_b2b[i], 2)
    gm_total_s = gm_ms.sum() * 1e-3 / args.steps
    rq_total_s = rq_ms.sum() * 1e-3 / args.steps
    gemm_kernel = "fused_linear" if args.fused else "w4a4_gemm"
    achieved = gemm_flops / gm_total_s / 1e12
    rq_bytes_all = sum(rq_algorithmic_bytes(M, K) for K in K_list)
    rq_layout_all = sum(rq_layout_bytes(M, K, clq.codes_width(lay.act_codes, K) / K)
                        for (_, K, _, lay) in layers)
    roofline = {"kernel": gemm_kernel, "bound": "tensor", "achieved": round(achieved, 1),
                "peak": fp8_peak, "unit": "TFLOP/s", "frac": round(achieved / fp8_peak, 4),
                "frac_of_measured_tcgen05_e4m3": round(achieved / measured["tcgen05_e4m3_tflops"], 4),
                "frac_of_int8_mma_sync": round(achieved / measured["mma_sync_s8_tops"], 4),
                "traffic": recorded_traffic(gemm_kernel, args.workload),
                "peak_note": "E4M3 kind::f8f6f4 dense = 2 x bf16 %s (%s)" % (bf16_peak, peak_src)}
    if rq_b2b is not None:
        ach_b2b = gemm_flops / (sum(gm_b2b) * 1e-3) / 1e12
        roofline["achieved_back_to_back"] = round(ach_b2b, 1)
        roofline["frac_back_to_back"] = round(ach_b2b / fp8_peak, 4)
    lay_codes = "e2m3" if layers[0][3].w_codes == clq.CLQ_CODES_E2M3 else "e4m3"
    mainloop = measured.get("mainloop_%s_tflops" % lay_codes)
    if mainloop:
        roofline["mainloop_tflops"] = mainloop
        roofline["frac_of_mainloop"] = round(achieved / mainloop, 4)
        roofline["mainloop_note"] = ("clq_peak_operand_stream: the GEMM's TMA + MMA loop on "
                                     "128 x 256 tiles of L2-resident %s codes, no epilogue, "
                                     "this run" % lay_codes)
    if not args.fused:
        sm_mhz = (clocks or {}).get("sm_mhz") or 2070.0
        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        fill = measured["operand_stream_%s_smem_gbs" % lay_codes] * 1e9 / sms / (sm_mhz * 1e6)
        bound = gemm_intake_bound(M, list(zip(K_list, N_list)), sms, sm_mhz, fill)
        roofline["intake_bound"] = {
            "tflops": round(bound, 1), "frac": round(achieved / bound, 4),
            "bytes_per_clk_per_sm": round(fill, 2),
            "model": "TMA fill of shared memory per SM measured in this run "
                     "(clq_peak_operand_stream, no MMA) at the median SM clock, output "
                     "writes through the same engine, the launcher's tiles"}
    rq_roof = None
    if not args.fused:
        rq_ach = rq_bytes_all / rq_total_s / 1e9
        rq_roof = {"kernel": "rotate_quant", "bound": "hbm", "achieved": round(rq_ach, 1),
                   "peak": hbm_peak, "unit": "GB/s", "frac": round(rq_ach / hbm_peak, 4),
                   "frac_of_8TBps": round(rq_ach / 8000.0, 4),
                   "algorithmic_bytes_per_step": int(rq_bytes_all),
                   "bytes_note": "2.5 B/element + 4 B/row (16-bit input, packed INT4 codes, "
                                 "fp32 scale)",
                   "layout_bytes_per_step": int(rq_layout_all),
                   "layout_GBps": round(rq_layout_all / rq_total_s / 1e9, 1),
                   "traffic": recorded_traffic("rotate_quant", args.workload)}
        if rq_b2b is not None:
            rq_b2b_ach = rq_bytes_all / (sum(rq_b2b) * 1e-3) / 1e9
            rq_roof["achieved_back_to_back"] = round(rq_b2b_ach, 1)
            rq_roof["frac_back_to_back"] = round(rq_b2b_ach / hbm_peak, 4)
        if rq_b2b is not None and rq_floor_b2b is not None:
            floor_gbps = rq_bytes_all / (sum(rq_floor_b2b) * 1e-3) / 1e9
            rq_roof["copy_floor"] = {
                "GBps": round(floor_gbps, 1), "frac_of_peak": round(floor_gbps / hbm_peak, 4),
                "kernel_frac_of_floor": round(rq_b2b_ach / floor_gbps, 4),
                "note": "clq_peak_rq_stream: the loop's tiles, copy ring and stores without "
                        "its gather and arithmetic, back to back on the same inputs"}

    # ---- end to end through the public API with host buffers ----
    e2e = None
    if not args.no_e2e:
        xh = [x.pin_memory() for x in xs_host]
        yh = [torch.empty((M, N), dtype=td).pin_memory() for N in N_list]
        h2d = sum(x.numel() * 2 for x in xh)
        d2h = sum(y.numel() * 2 for y in yh)
        reps = max(3, min(args.steps, 30))
        pipe = clq.HostPipeline([(lay, M, K, N) for (_, K, N, lay) in layers], td, dev,
                                fused=args.fused)
        for _ in range(2):
            pipe.run(xh, yh)
        pipe.join(stream)
        torch.cuda.synchronize()
        a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for r in range(reps):
            pipe.run(xh, yh, after=a if r == 0 else None)
        pipe.join(stream)
        z.record(stream)
        torch.cuda.synchronize()
        e2e_s = a.elapsed_time(z) * 1e-3 / reps
        e2e = {"value": ops_step * world / e2e_s / 1e12, "unit": "TOPS",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "path": "public API (clq.HostPipeline over PreparedLinear): input copies, "
                       "kernels and output copies on three streams",
               "ms_per_step": round(e2e_s * 1e3, 3)}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args.workload)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "TOPS",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(total_ms / args.steps, 4), "higher_is_better": True,
            "steady_state": dict(steady, value_median=round(
                ops_step * world / (steady["ms_per_step_median"] * 1e-3) / 1e12, 2)),
            "scaling": "weak", "vs_baseline": None,
            "dtype": "int4 codes on %s tcgen05 operands, f32 accumulate" % (
                "e2m3" if layers[0][3].act_codes == clq.CLQ_CODES_E2M3 else "e4m3"),
            "weights": weight_memory(layers),
            "data": "synthetic (seeded Philox, DiT-shaped; no model weights)",
            "config": config_dict(cfg, args), "roofline": roofline,
            "roofline_rotate_quant": rq_roof, "per_layer": per_layer,
            "cpu_baseline": cpu, "e2e": e2e,
            "comparators": {
                "fp16_cublas_tops": round(ops_step * world / (cublas_ms * 1e-3) / 1e12, 1),
                "speedup_vs_fp16_cublas": round(cublas_ms / (total_ms / args.steps), 3),
                ("separate" if args.fused else "fused") + "_tops":
                    round(ops_step * world / (other_ms * 1e-3) / 1e12, 1),
                "fused_over_separate_time": round(
                    (total_ms / args.steps) / other_ms if args.fused
                    else other_ms / (total_ms / args.steps), 3),
                **({} if temporal_ms is None else {
                    "temporal_token_set_tops":
                        round(ops_step * world / (temporal_ms * 1e-3) / 1e12, 1),
                    "temporal_over_spatial_time":
                        round(temporal_ms / (total_ms / args.steps), 3)})},
            "measured_peaks": measured,
            "gpu_launches": (1 if args.fused else 2) * nlay * args.steps,
            "clocks": clocks,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
