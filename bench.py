#!/usr/bin/env python
"""Benchmark of the additive-codebook dequantize-and-multiply hot path on GB300.

Workload (default): a Llama-style 4096 x 4096 attention projection stored with M = 4
codebooks of 2^8 fp16 codewords (g = 8, uint8 codes), evaluated at batch 1 for every prefix
m = 1..4 (1..4 bits per weight). One step = the four GEMVs m = 1, 2, 3, 4 on one weight copy.
Weight copies rotate so the timed reads come from HBM, not L2 (copies x packed bytes >= 3x L2).

Prints one JSON line. `value` is the achieved algorithmic HBM bandwidth of the whole step,
sum over m of bytes(m) / step time, with bytes(m) = codes m*out*(in/8) + books m*2^8*8*2 +
scales 2*out + x 2*in + y 2*out. The timed steps run as one CUDA graph with CUDA events
around it; per-m times come from a separate graph of launches of that prefix alone.

--impl reference times the CPU oracle (the plain C++ statement of the same product) on the
host cores, on a bounded row sample of the same workload, with the same metric.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "batch-1 GEMV µs & achieved HBM GB/s per prefix m (bits/wt); prefill GEMM TFLOP/s"
WORKLOAD = "attn_4096"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40000,
                    help="timed steps (replays of a graph of at most 200 steps; the default "
                         "keeps the timed region about a second long)")
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="own", choices=["own", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-gemm", action="store_true")
    ap.add_argument("--no-wmse", action="store_true",
                    help="skip the per-prefix distortion measurement")
    ap.add_argument("--no-beam", action="store_true",
                    help="skip the beam-search code update measurement")
    ap.add_argument("--wmse-only", action="store_true",
                    help="only the per-prefix distortion measurement (for profiling)")
    ap.add_argument("--no-loading", action="store_true",
                    help="skip the prefix-store loading measurement")
    ap.add_argument("--gemm-tokens", type=int, default=4096,
                    help="tokens of the prefill GEMM case (smaller values: profiling runs)")
    ap.add_argument("--skip-gemv", action="store_true",
                    help="only the GEMM case (profiling runs; prints no bench line)")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the per-configuration GEMV table (8B block, 1024^2, large books)")
    ap.add_argument("--profile-gemv", metavar="WORKLOAD[:LAYER]",
                    help="only three aq_gemv calls of one workload layer (for ncu captures; "
                         "prints no bench line), with --batch and --m")
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--m", type=int, default=1)
    ap.add_argument("--bits", type=int, default=0,
                    help="with --profile-gemv: code width other than the workload's (4, 8, 16)")
    return ap.parse_args()


def layer_bytes(out, inp, m, B=8, G=8, batch=1, xsize=2, ysize=2):
    """Algorithmic bytes of one prefix-m call: codes, first m books, scales, x, y."""
    return (m * out * (inp // G) * (B // 8) + m * (1 << B) * G * 2 + 2 * out
            + batch * inp * xsize + batch * out * ysize)


def lut_kernel_source():
    """The source text that decides what gemv_lut_kernel reads: the kernel's section of gemv.cu,
    its launcher run_lut_layers (grid, ring slots, work split), and the device helpers of
    aq_internal.cuh."""
    csrc = os.path.join(ROOT, "paper_2606_12876_gb300", "csrc")
    g = open(os.path.join(csrc, "gemv.cu")).read()
    h = open(os.path.join(csrc, "aq_internal.cuh")).read()
    rule = "// " + "-" * 66
    a = g.index(rule + " LUT kernel")
    b = g.index(rule, a + len(rule))
    r0 = g.index("aq_status run_lut_layers(const Dims* ds")
    r1 = g.index("\n}\n", r0)
    d0 = h.index("// ---- device helpers")
    return g[a:b] + g[r0:r1] + h[d0:]


def profiled_traffic(workload, m):
    """DRAM bytes per launch measured by ncu (profiles/gemv_lut_traffic.txt), or None when the
    kernel's source (lut_kernel_source) changed since that capture."""
    import hashlib
    path = os.path.join(ROOT, "profiles", "gemv_lut_traffic.txt")
    if not os.path.exists(path):
        return None
    h = hashlib.sha256(lut_kernel_source().encode())
    rec, traffic = None, None
    for line in open(path):
        parts = line.split()
        if len(parts) == 2 and parts[0] == "source_hash":
            rec = parts[1]
        elif len(parts) == 4 and parts[0] == workload and parts[1] == "m=%d" % m:
            traffic = int(parts[3])
    return traffic if rec == h.hexdigest()[:16] else None


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def whole_job(ms_total, world, bytes_step, steps, device=None):
    """The slowest rank's timed-region length (ms) and the whole-job throughput (GB/s): every
    rank runs its own replica of the step on its own data (weak scaling), so the job moves
    world * bytes_step bytes per step. With world > 1 the process group must be initialised."""
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([ms_total], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms_total = float(t.item())
    return ms_total, world * bytes_step * steps / (ms_total / 1e3) / 1e9


class ClockSampler:
    """nvidia-smi clock / throttle samples during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.dev), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        self.proc.wait()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 8:
                rows.append(parts)
        os.unlink(self.path)
        sm = [float(r[0]) for r in rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


def cpu_model():
    """The host CPU's model name (lscpu), or the machine type."""
    import platform
    import subprocess
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip() + " (%s)" % platform.machine()
    except (OSError, subprocess.SubprocessError):
        pass
    return platform.machine()


def cpu_oracle_rate(layer, x_bits, ms, budget_s, rows=None):
    """Time the oracle on (a row sample of) one step: returns (GB/s, seconds/step, steps)."""
    import oracle
    out = layer["out"] if rows is None else rows[1] - rows[0]
    bytes_step = sum(layer_bytes(out, layer["in"], m) for m in ms)
    n, t0 = 0, time.perf_counter()
    while True:
        for m in ms:
            oracle.product_exact(layer, x_bits, "f16", m, rows=rows)
        n += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            break
    return bytes_step * n / el / 1e9, el / n, n


def reference_arm(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    import oracle
    import workloads
    (_, layer), = list(workloads.config_layers(WORKLOAD))
    x_bits = workloads.config_x(WORKLOAD, 1, layer["in"])
    ms = (1, 2, 3, 4)
    # size the row sample so W + K steps take about a minute
    t_full = cpu_oracle_rate(layer, x_bits, ms, 0.0)[1]
    frac = min(1.0, 60.0 / max(1, args.steps + args.warmup) / max(t_full, 1e-6))
    nrows = max(32, int(layer["out"] * frac) // 32 * 32)
    rows = (0, nrows)
    for _ in range(args.warmup):
        for m in ms:
            oracle.product_exact(layer, x_bits, "f16", m, rows=rows)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        for m in ms:
            oracle.product_exact(layer, x_bits, "f16", m, rows=rows)
    el = time.perf_counter() - t0
    bytes_step = sum(layer_bytes(nrows, layer["in"], m) for m in ms)
    value = bytes_step * args.steps / el / 1e9
    sample = "rows 0..%d of the 4096x4096 layer, batch 1, m=1..4 per step" % nrows
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": el / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "sample": sample},
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": oracle.num_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def measure_gemm(dev, stream, peaks, reps=5, tokens=4096):
    """Prefill GEMM on the 70B up-projection shape (4096 tokens, 8192 -> 28672, M = 4 bf16
    books, bf16 activations) for every prefix m, next to a dense bf16 torch.matmul of the same
    shape. Inputs (64 MB activations, 28-112 MB codes) exceed L2."""
    import torch
    import paper_2606_12876_gb300 as aq
    from paper_2606_12876_gb300.linear import AQLinear, x_to_device
    import workloads
    name = "llama70b_up_prefill"
    (_, layer), = list(workloads.config_layers(name))
    out, inp = layer["out"], layer["in"]
    lin = AQLinear.from_layer(layer, device=dev)
    x = x_to_device(workloads.config_x(name, tokens, inp), "bf16", dev)
    y = torch.empty(tokens, out, dtype=torch.bfloat16, device=dev)
    flops = 2.0 * tokens * out * inp
    peak = peaks.get("bf16_tflops", 1900.0)

    def timed(fn):
        with torch.cuda.stream(stream):
            fn()
            torch.cuda.synchronize(dev)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(reps):
                fn()
            e1.record()
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1) / reps

    rows = []
    for m in (1, 2, 3, 4):
        ms = timed(lambda: lin.gemm(x, m, y=y))
        tf = flops / (ms * 1e-3) / 1e12
        rows.append({"m": m, "ms": round(ms, 4), "TFLOP_s": round(tf, 1),
                     "frac_bf16_peak": round(tf / peak, 4)})
    wd = torch.empty(out, inp, device=dev, dtype=torch.bfloat16)
    # the unfused yardstick: W_m decoded alone (aq_decode into a dense bf16 matrix), then a
    # dense bf16 product of the same shape
    for e in rows:
        e["decode_ms"] = round(timed(lambda: lin.decode(e["m"], out=wd)), 4)
    torch.nn.init.normal_(wd)
    dense_ms = timed(lambda: torch.matmul(x, wd.t()))
    del wd
    for e in rows:
        e["decode_plus_dense_ms"] = round(e["decode_ms"] + dense_ms, 4)
    return {"workload": name, "tokens": tokens, "out": out, "in": inp, "M": 4,
            "compute": "fp16 tcgen05 pair MMA, fp32 accumulation; weights decoded in shared memory (m = 1), or W_m decoded once in fp16 and loaded by TMA (m >= 2 at 2048+ tokens)",
            "per_m": rows, "dense_bf16_torch_ms": round(dense_ms, 4),
            "dense_bf16_TFLOP_s": round(flops / (dense_ms * 1e-3) / 1e12, 1),
            "peak_TFLOP_s": peak, "peak_source": "measured" if "bf16_tflops" in peaks else "fallback"}


def measure_loading(lin, dev, stream, ms, reps=7):
    """Dynamic loading through a prefix store (aq_store_*): the layer's packed form in pinned
    host memory, device memory for the resident prefix only. Raising the prefix from m-1 to m
    maps memory for plane m-1 and copies that plane and codebook m-1 from the host; lowering
    back synchronises the device and unmaps it. Host wall time (median over reps) around the
    call and a synchronisation of the stream; the plain host->device copy of the same bytes
    (CUDA events) is timed beside it."""
    import time

    import torch
    from paper_2606_12876_gb300.linear import AQLinear

    host = lin.to_host()
    pb = host["planes"].numel() // lin.M
    raise_us, lower_us = {}, {}
    with torch.cuda.stream(stream):
        dyn = AQLinear.from_host(host, 0, device=dev)
        for m in ms:
            up, down = [], []
            for _ in range(reps):
                dyn.set_prefix(m - 1)
                torch.cuda.synchronize(dev)
                t0 = time.perf_counter()
                dyn.set_prefix(m)
                stream.synchronize()
                up.append(time.perf_counter() - t0)
                t0 = time.perf_counter()
                dyn.set_prefix(m - 1)
                down.append(time.perf_counter() - t0)
            raise_us[m] = sorted(up)[reps // 2] * 1e6
            lower_us[m] = sorted(down)[reps // 2] * 1e6
        dyn.set_prefix(max(ms))
        x = torch.randn(1, lin.inp, device=dev, dtype=torch.float16)
        same = bool(torch.equal(dyn.gemv(x, max(ms)), lin.gemv(x, max(ms))))
        resident = dyn.device_bytes()
        dyn.close()
        dst = torch.empty(pb, dtype=torch.uint8, device=dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        copy = []
        for _ in range(reps):
            e0.record()
            dst.copy_(host["planes"][:pb], non_blocking=True)
            e1.record()
            e1.synchronize()
            copy.append(e0.elapsed_time(e1) * 1e3)
    copy_us = sorted(copy)[reps // 2]
    return {"store": "aq_store_* (virtual address range for all M planes, memory mapped per prefix)",
            "source": "pinned host memory", "plane_bytes": pb,
            "raise_to_m_us": {m: round(raise_us[m], 1) for m in ms},
            "lower_from_m_us": {m: round(lower_us[m], 1) for m in ms},
            "h2d_copy_one_plane_us": round(copy_us, 1),
            "h2d_GB_s": round(pb / (copy_us * 1e-6) / 1e9, 1),
            "device_bytes_at_m4": resident, "matches_full_layer": same}


def measure_wmse(lin, dev, stream, peaks, reps=10):
    """aq_wmse on the benchmark layer: D^(k) for all four prefixes in one call (Sec. 2.2
    Eq. wmse-task, Sec. 5). W = the full reconstruction plus N(0, 0.01^2) noise in the book
    type; H = X X^T / n for Gaussian X with n = 2 * d_in (fp32). CUDA events around `reps`
    back-to-back calls (each: folding of H, the tensor-core pass, the reduction)."""
    import torch
    out, inp, M = lin.out, lin.inp, lin.M
    g = torch.Generator(device=dev).manual_seed(7)
    W = (lin.decode(M).float() + 0.01 * torch.randn(out, inp, device=dev, generator=g)).half()
    X = torch.randn(inp, 2 * inp, device=dev, generator=g)
    H = (X @ X.t()) / X.shape[1]
    del X
    lam = [0.25] * M
    with torch.cuda.stream(stream):
        for _ in range(3):
            d = lin.wmse(W, H, lam)
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            d = lin.wmse(W, H, lam)
        e1.record()
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1) / reps
    # tensor-core work actually issued: per pair tile (256 t x 128 rows) K = min(256 (tb+1), in)
    tb_n, ob_n = -(-inp // 256), -(-out // 128)
    ksum = sum(-(-min(256 * (tb + 1), inp) // 64) * 64 for tb in range(tb_n))
    mma_flops = 2.0 * 256 * 128 * ksum * ob_n * M
    def_flops = 2.0 * M * out * inp * inp          # E_k H for every prefix, as defined
    peak = peaks.get("bf16_tflops", 1900.0)
    tf = mma_flops / (ms * 1e-3) / 1e12
    return {"workload": "attn_4096", "out": out, "in": inp, "M": M,
            "compute": "E_k written once in bf16, then bf16 tcgen05 pair MMA (E_k x folded H), fp32 accumulation, 2 prefixes per pass",
            "ms": round(ms, 4), "mma_TFLOP_s": round(tf, 1), "frac_bf16_peak": round(tf / peak, 4),
            "definition_TFLOP_s": round(def_flops / (ms * 1e-3) / 1e12, 1),
            "mma_flops": mma_flops, "D": [round(float(v), 6) for v in d[:M].tolist()],
            "loss_uniform": round(float(d[M]), 6),
            "peak_source": "measured" if "bf16_tflops" in peaks else "fallback"}


def measure_beam(lin, layer, dev, stream, sm_mhz, K=8, reps=3):
    """aq_beam_search on the benchmark layer (the code update of Alg. 1, App. C): every group
    of the 4096 x 4096 layer searches its four codes with a beam of width K = 8. W = the full
    reconstruction plus N(0, 0.01^2) noise (book type), H = X X^T / n for Gaussian X (fp32),
    lambda = 1, 1/2, 1/4, 1/8. CUDA events around `reps` back-to-back calls (each: residuals,
    S, E_k S on the CUDA cores, the search)."""
    import numpy as np
    import torch
    import paper_2606_12876_gb300 as aq
    out, inp, M, B = lin.out, lin.inp, lin.M, layer["B"]
    g = torch.Generator(device=dev).manual_seed(9)
    W = (lin.decode(M).float() + 0.01 * torch.randn(out, inp, device=dev, generator=g)).half()
    X = torch.randn(inp, 2 * inp, device=dev, generator=g)
    H = (X @ X.t()) / X.shape[1]
    del X
    codes = torch.from_numpy(np.ascontiguousarray(layer["codes"])).to(dev)
    new = torch.empty_like(codes)
    books = torch.from_numpy(layer["books"].view(np.int16)).to(dev)
    scales = torch.from_numpy(layer["scales"].view(np.int16)).to(dev)
    ws = aq.workspace(aq.beam_workspace_bytes(lin.layout), dev)
    lam = [1.0 / (1 << k) for k in range(M)]
    call = lambda: aq.aq_beam_search(lin.layout, W, codes, books, scales, H, aq.AQ_F32, lam, K,
                                     new, ws, stream=stream)
    with torch.cuda.stream(stream):
        call()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(reps):
            call()
        e1.record()
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1) / reps
    groups = out * (inp // 8)
    nb = 1 << B
    cands = nb + (M - 1) * K * nb                      # candidates scored per group
    # per candidate: d (8 FMA), S_gg d (64 FMA), d.(S_gg d) and d.h (16 FMA), score (2)
    cand_flops = 2 * (8 + 64 + 16) + 2
    gemm_flops = 2.0 * M * out * inp * inp             # E_k S for every prefix
    flops = groups * cands * cand_flops + gemm_flops
    changed = float((new != codes).any(dim=2).float().mean())
    peak = fp32_alu_peak_tflops(sm_mhz)
    tf = flops / (ms * 1e-3) / 1e12
    return {"workload": "attn_4096", "out": out, "in": inp, "M": M, "B": B, "K": K,
            "ms": round(ms, 3), "groups_per_s": round(groups / (ms * 1e-3), 1),
            "candidates_per_group": cands, "flops": flops, "fp32_TFLOP_s": round(tf, 2),
            "alu_peak_TFLOP_s": round(peak, 1), "frac_alu_peak": round(tf / peak, 4),
            "groups_changed": round(changed, 4)}


def graph_us(calls, n, stream, reps=5):
    """us per call of a CUDA graph of n calls (calls(i) enqueues call i; weight copies rotate
    inside it): median over reps replays, events around the graph only, so back-to-back calls
    keep their overlap."""
    import torch
    for i in range(3):
        calls(i)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(n):
            calls(i)
    g.replay()
    torch.cuda.synchronize()
    ts = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e0.record()
            g.replay()
            e1.record()
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1) * 1e3 / n)
    del g
    return statistics.median(ts)


def fp32_alu_peak_tflops(sm_mhz, sms=152):
    """CUDA-core fp32 peak: 128 FMA lanes per SM, 2 flops per FMA, at the SM clock."""
    return sms * 128 * 2 * sm_mhz * 1e6 / 1e12


def measure_configs(dev, stream, hbm_peak, sm_mhz):
    """Batch-1..16 GEMV over the paper-shaped layers (per prefix m): the 1024^2 layer
    (batch 1), the Llama-3-8B block (each linear and the summed block, batch 1 and 8, bf16
    activations), the 8192^2 layer with 2^16-entry books (batch 1 and 16) and the 4096^2
    attention projection at batch 4 and 16. us per call from graphs of back-to-back calls over
    weight copies that together exceed 3x L2; GB/s = algorithmic bytes / time; for batch > 1
    also the fraction of the CUDA-core fp32 FMA roofline (2 * batch flops per weight)."""
    import torch
    import paper_2606_12876_gb300 as aq
    from paper_2606_12876_gb300.linear import AQLinear, x_to_device
    import workloads
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    alu_peak = fp32_alu_peak_tflops(sm_mhz)
    res = {"alu_peak_TFLOP_s": round(alu_peak, 1),
           "alu_peak_basis": "152 SMs x 128 fp32 lanes x 2 flops x %.0f MHz (median SM clock "
                             "of the headline run)" % sm_mhz}

    def layer_entry(lin, xdt, batch, ms):
        xc = aq.AQ_F16 if xdt == "f16" else aq.AQ_BF16
        x = x_to_device(workloads.make_x(batch, lin.inp, xdt, seed=batch), xdt)
        y = torch.empty(batch, lin.out, dtype=x.dtype, device=dev)
        ws = aq.workspace(aq.gemv_workspace_bytes(lin.layout, batch), dev)
        sink = torch.zeros(4, dtype=torch.int32, device=dev)
        nc = max(2, -(-3 * l2 // lin.planes.numel()))
        copies = [lin.planes.clone() for _ in range(nc)]
        rows = []
        for m in ms:
            with torch.cuda.stream(stream):
                us = graph_us(lambda i, m=m: aq.aq_gemv(lin.layout, m, copies[i % nc], lin.books,
                                                        lin.scales, x, xc, batch, y, xc, ws), 20, stream)
            nb = layer_bytes(lin.out, lin.inp, m, B=lin.B, batch=batch)
            e = {"m": m, "bits_per_weight": m * lin.B // 8, "us": round(us, 3),
                 "GB_s": round(nb / us / 1e3, 1), "frac_hbm": round(nb / us / 1e3 / hbm_peak, 4)}
            if batch == 1:
                # the read probe over the same code bytes: the per-call floor of this size
                pb = aq.packed_bytes(lin.layout, m)
                with torch.cuda.stream(stream):
                    fl = graph_us(lambda i, pb=pb: aq.aq_selftest_read(copies[i % nc], pb, sink),
                                  20, stream)
                e["read_floor_us"] = round(fl, 3)
                e["frac_of_read_floor"] = round(fl / us, 4)
            if batch > 1:
                tf = 2.0 * batch * lin.out * lin.inp / (us * 1e-6) / 1e12
                e["TFLOP_s"] = round(tf, 2)
                e["frac_alu"] = round(tf / alu_peak, 4)
            rows.append(e)
        del copies
        return rows

    def cfg_layers(name):
        return [(n, AQLinear.from_layer(l, device=dev)) for n, l in workloads.config_layers(name)]

    (_, lin1), = cfg_layers("single_1024")
    res["single_1024"] = {"b1": layer_entry(lin1, "f16", 1, (1, 2))}
    (_, lina), = cfg_layers("attn_4096")
    res["attn_4096"] = {"b%d" % b: layer_entry(lina, "f16", b, (1, 2, 3, 4)) for b in (4, 16)}
    blk = cfg_layers("llama8b_block")
    res["llama8b_block"] = {n: {"b%d" % b: layer_entry(lin, "bf16", b, (1, 2, 3, 4)) for b in (1, 8)}
                            for n, lin in blk}
    # the summed block: the seven calls back to back in one graph, three weight copies each
    for b in (1, 8):
        xs = {}
        for _, lin in blk:
            if lin.inp not in xs:
                xs[lin.inp] = x_to_device(workloads.make_x(b, lin.inp, "bf16", seed=b), "bf16")
        ys = [torch.empty(b, lin.out, dtype=torch.bfloat16, device=dev) for _, lin in blk]
        wss = [aq.workspace(aq.gemv_workspace_bytes(lin.layout, b), dev) for _, lin in blk]
        cps = [[lin.planes.clone() for _ in range(3)] for _, lin in blk]
        sink = torch.zeros(4, dtype=torch.int32, device=dev)
        rows = []
        for m in (1, 2, 3, 4):
            def step(i, m=m):
                for j, (_, lin) in enumerate(blk):
                    aq.aq_gemv(lin.layout, m, cps[j][i % 3], lin.books, lin.scales, xs[lin.inp],
                               aq.AQ_BF16, b, ys[j], aq.AQ_BF16, wss[j])
            with torch.cuda.stream(stream):
                us = graph_us(step, 10, stream)
            nb = sum(layer_bytes(lin.out, lin.inp, m, batch=b) for _, lin in blk)
            e = {"m": m, "us": round(us, 3), "GB_s": round(nb / us / 1e3, 1),
                 "frac_hbm": round(nb / us / 1e3 / hbm_peak, 4)}
            if b == 1:
                def floor_step(i, m=m):
                    for j, (_, lin) in enumerate(blk):
                        aq.aq_selftest_read(cps[j][i % 3], aq.packed_bytes(lin.layout, m), sink)
                with torch.cuda.stream(stream):
                    fl = graph_us(floor_step, 10, stream)
                e["read_floor_us"] = round(fl, 3)
                e["frac_of_read_floor"] = round(fl / us, 4)
            if b > 1:
                tf = 2.0 * b * sum(lin.out * lin.inp for _, lin in blk) / (us * 1e-6) / 1e12
                e["TFLOP_s"] = round(tf, 2)
                e["frac_alu"] = round(tf / alu_peak, 4)
            rows.append(e)
        res["llama8b_block"]["block_sum_b%d" % b] = rows
        # the same seven layers as four calls: q/k/v and gate/up each as one group call
        # (aq_gemv_group), o and down alone
        names = [n for n, _ in blk]
        idx = {n: j for j, n in enumerate(names)}
        groups = [("q_proj", "k_proj", "v_proj"), ("o_proj",), ("gate_proj", "up_proj"),
                  ("down_proj",)]
        gws = {}
        for gr in groups:
            if len(gr) > 1:
                gws[gr] = aq.workspace(aq.gemv_group_workspace_bytes(
                    [blk[idx[n]][1].layout for n in gr], b), dev)
        grows = []
        for m in (1, 2, 3, 4):
            def gstep(i, m=m):
                for gr in groups:
                    js = [idx[n] for n in gr]
                    lins = [blk[j][1] for j in js]
                    if len(gr) == 1:
                        j = js[0]
                        aq.aq_gemv(lins[0].layout, m, cps[j][i % 3], lins[0].books,
                                   lins[0].scales, xs[lins[0].inp], aq.AQ_BF16, b, ys[j],
                                   aq.AQ_BF16, wss[j])
                    else:
                        aq.aq_gemv_group([l.layout for l in lins], m, [cps[j][i % 3] for j in js],
                                         [l.books for l in lins], [l.scales for l in lins],
                                         xs[lins[0].inp], aq.AQ_BF16, b, [ys[j] for j in js],
                                         aq.AQ_BF16, gws[gr])
            with torch.cuda.stream(stream):
                us = graph_us(gstep, 10, stream)
            nb = sum(layer_bytes(lin.out, lin.inp, m, batch=b) for _, lin in blk)
            ge = {"m": m, "us": round(us, 3), "GB_s": round(nb / us / 1e3, 1),
                  "frac_hbm": round(nb / us / 1e3 / hbm_peak, 4)}
            if b > 1:
                tf = 2.0 * b * sum(lin.out * lin.inp for _, lin in blk) / (us * 1e-6) / 1e12
                ge["TFLOP_s"] = round(tf, 2)
                ge["frac_alu"] = round(tf / alu_peak, 4)
            grows.append(ge)
        res["llama8b_block"]["block_grouped_b%d" % b] = grows
        del cps
    del blk
    (_, linb), = cfg_layers("big_book_8192")
    res["big_book_8192"] = {"b%d" % b: layer_entry(linb, "f16", b, (1, 2)) for b in (1, 16)}
    res["big_book_8192"]["note"] = ("2^16-entry books (1 MiB each) are gathered through L2; "
                                    "frac_hbm counts the algorithmic bytes of the call")
    return res


def own_arm(args):
    import numpy as np
    import torch

    world, rank, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    import paper_2606_12876_gb300 as aq
    from paper_2606_12876_gb300 import build as libbuild
    from paper_2606_12876_gb300.linear import AQLinear, x_to_device
    import workloads

    libbuild.build()
    ms = (1, 2, 3, 4)
    (_, layer), = list(workloads.config_layers(WORKLOAD))
    out, inp = layer["out"], layer["in"]
    lin = AQLinear.from_layer(layer, device=dev)
    L = lin.layout
    x_bits = workloads.config_x(WORKLOAD, 1, inp)
    x = x_to_device(x_bits, "f16", dev)
    ys = {m: torch.empty(1, out, dtype=torch.float16, device=dev) for m in ms}
    ws = aq.workspace(aq.gemv_workspace_bytes(L, 1), dev)

    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    pbytes = aq.packed_bytes(L, 4)
    ncopies = max(2, -(-3 * l2 // pbytes))
    copies = [lin.planes.clone() for _ in range(ncopies)]
    bytes_m = {m: layer_bytes(out, inp, m) for m in ms}
    bytes_step = sum(bytes_m.values())

    peaks = {}
    ppath = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(ppath):
        peaks = json.load(open(ppath))
    hbm_peak = peaks.get("hbm_gbs", 6800.0)
    peak_src = "measured" if "hbm_gbs" in peaks else "fallback"

    stream = torch.cuda.Stream(device=dev)
    if args.wmse_only:
        print(json.dumps({"wmse_only": measure_wmse(lin, dev, stream, peaks)}), flush=True)
        return
    if args.skip_gemv:
        g = measure_gemm(dev, stream, peaks, tokens=args.gemm_tokens)
        print(json.dumps({"gemm_only": g}), flush=True)
        return

    def call(i, m):
        aq.aq_gemv(L, m, copies[i % ncopies], lin.books, lin.scales, x, aq.AQ_F16, 1, ys[m],
                   aq.AQ_F16, ws)

    def step(i):
        for m in ms:
            call(i, m)

    with torch.cuda.stream(stream):
        for i in range(3):                      # eager warm-up: sets kernel attributes
            step(i)
    torch.cuda.synchronize(dev)

    def capture(fn, n):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(n):
                fn(i)
        return g

    def time_graph(g):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(stream):
            e0.record()
            g.replay()
            e1.record()
        torch.cuda.synchronize(dev)
        return e0.elapsed_time(e1)

    # The timed steps run as replays of one graph of at most 200 steps (and one graph for the
    # remainder), so that a long timed region needs no long capture.
    glen = min(args.steps, 200)
    g_warm, g_timed = capture(step, args.warmup), capture(step, glen)
    rest = args.steps % glen
    g_rest = capture(step, rest) if rest else None
    torch.cuda.synchronize(dev)

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    g_warm.replay()
    torch.cuda.synchronize(dev)
    clocks = ClockSampler(local)
    clocks.start()
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    with torch.cuda.stream(stream):
        e0.record()
        for _ in range(args.steps // glen):
            g_timed.replay()
        if g_rest is not None:
            g_rest.replay()
        e1.record()
    torch.cuda.synchronize(dev)
    ms_total = e0.elapsed_time(e1)
    barrier()
    clk = clocks.stop()
    del g_rest
    ms_total, value = whole_job(ms_total, world, bytes_step, args.steps, device=dev)
    ms_step = ms_total / args.steps

    # Per prefix: a graph of `steps` launches of that prefix alone (rotating weight copies),
    # CUDA events around the graph only, so back-to-back launches keep their overlap; the
    # median of 5 replays. Single-call latency: one eager call between synchronisations,
    # events around it, median of 7.
    per_m_us, single_us = {}, {}
    for m in ms:
        g = capture(lambda i, m=m: call(i, m), glen)
        g.replay()
        per_m_us[m] = statistics.median(time_graph(g) for _ in range(5)) * 1e3 / glen
        del g
        lat = []
        with torch.cuda.stream(stream):
            for i in range(7):
                torch.cuda.synchronize(dev)
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record()
                call(i, m)
                e1.record()
                torch.cuda.synchronize(dev)
                lat.append(e0.elapsed_time(e1) * 1e3)
        single_us[m] = statistics.median(lat)


    # Read floor: the read probe (aq_selftest_read, the GEMV's launch shape doing nothing but
    # reading) over the same m planes of the same rotating copies; same graph timing.
    sink = torch.zeros(4, dtype=torch.int32, device=dev)
    floor_us = {}
    for m in ms:
        nb = aq.packed_bytes(L, m)
        g = capture(lambda i, nb=nb: aq.aq_selftest_read(copies[i % ncopies], nb, sink), glen)
        g.replay()
        floor_us[m] = statistics.median(time_graph(g) for _ in range(5)) * 1e3 / glen
        del g

    # Refinement step (aq_gemv_refine): the increment from prefix m-1 to m, reading plane m-1
    # only, fp32 output added to the previous fp32 result; same graph timing.
    ys32 = {m: torch.zeros(1, out, dtype=torch.float32, device=dev) for m in (0,) + ms}
    refine_us = {}
    for m in ms:
        prev = ys32[m - 1] if m > 1 else None
        g = capture(lambda i, m=m, prev=prev: aq.aq_gemv_refine(
            L, m, copies[i % ncopies], lin.books, lin.scales, x, aq.AQ_F16, 1, prev, ys32[m],
            aq.AQ_F32, ws), glen)
        g.replay()
        refine_us[m] = time_graph(g) * 1e3 / glen
        del g
    refine_bytes = layer_bytes(out, inp, 1, ysize=4) + 4 * out   # one plane; y_prev read too

    per_m = []
    for m in ms:
        us = per_m_us[m]
        gbs = bytes_m[m] / (us * 1e-6) / 1e9
        per_m.append({"m": m, "bits_per_weight": m, "us": round(us, 3), "GB_s": round(gbs, 1),
                      "frac_hbm": round(gbs / hbm_peak, 4),
                      "frac_hbm_spec_8TBs": round(gbs / 8000.0, 4),
                      "single_call_us": round(single_us[m], 3), "bytes": bytes_m[m],
                      "read_floor_us": round(floor_us[m], 3),
                      "frac_of_read_floor": round(floor_us[m] / us, 4),
                      "refine_from_m_minus_1_us": round(refine_us[m], 3),
                      "refine_GB_s": round(refine_bytes / (refine_us[m] * 1e-6) / 1e9, 1)})
    dom = per_m[-1]       # the full prefix: the most bytes per call

    # end to end through the public API: pinned host x -> device, 4 GEMVs, y -> pinned host,
    # every step. As a decode loop runs it: the step's API calls and both copies captured in a
    # CUDA graph (value); and eager, one Python call per API call (eager_ms_per_step).
    e2e = None
    if not args.no_e2e:
        x_host = torch.from_numpy(x_bits.view(np.int16)).view(torch.float16).pin_memory()
        y_host = torch.empty(len(ms), out, dtype=torch.float16).pin_memory()
        x_dev = torch.empty_like(x_host, device=dev)
        y_dev = torch.empty(len(ms), out, dtype=torch.float16, device=dev)   # one row per m
        n_e2e = max(20, min(args.steps // 2, 2000))

        def e2e_step(i):
            x_dev.copy_(x_host, non_blocking=True)
            planes = copies[i % ncopies]
            for j, m in enumerate(ms):
                aq.aq_gemv(L, m, planes, lin.books, lin.scales, x_dev, aq.AQ_F16, 1,
                           y_dev[j:j + 1], aq.AQ_F16, ws)
            y_host.copy_(y_dev, non_blocking=True)    # the step's four results

        e_s, e_e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            for i in range(args.warmup + n_e2e):
                if i == args.warmup:
                    torch.cuda.synchronize(dev)
                    e_s.record()
                e2e_step(i)
            e_e.record()
        torch.cuda.synchronize(dev)
        eager_ms = e_s.elapsed_time(e_e) / n_e2e
        glen_e = min(n_e2e, 200)
        g_e2e = capture(e2e_step, glen_e)
        g_e2e.replay()
        torch.cuda.synchronize(dev)
        reps = max(1, n_e2e // glen_e)
        e_s, e_e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(stream):
            e_s.record()
            for _ in range(reps):
                g_e2e.replay()
            e_e.record()
        torch.cuda.synchronize(dev)
        del g_e2e
        e2e_ms = e_s.elapsed_time(e_e) / (reps * glen_e)
        e2e = {"value": world * bytes_step / (e2e_ms / 1e3) / 1e9, "unit": "GB/s",
               "ms_per_step": e2e_ms, "h2d_bytes_per_step": x_host.numel() * 2,
               "d2h_bytes_per_step": y_host.numel() * 2,
               "api": "paper_2606_12876_gb300.aq_gemv (ctypes -> libaq.so), each step's calls "
                      "and its two copies captured in a CUDA graph and replayed",
               "eager_value": world * bytes_step / (eager_ms / 1e3) / 1e9,
               "eager_ms_per_step": eager_ms,
               "eager_api": "the same calls and copies issued from Python every step"}

    gemm = None if args.no_gemm else measure_gemm(dev, stream, peaks, tokens=args.gemm_tokens)
    configs = None
    if rank == 0 and not args.no_configs:
        configs = measure_configs(dev, stream, hbm_peak, clk.get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0))
    loading = measure_loading(lin, dev, stream, ms) if rank == 0 and not args.no_loading else None
    wmse = None if args.no_wmse else measure_wmse(lin, dev, stream, peaks)
    beam = None
    if rank == 0 and not args.no_beam:
        beam = measure_beam(lin, layer, dev, stream,
                            clk.get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0))

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        rate, per, n = cpu_oracle_rate(layer, x_bits, ms, 10.0)
        cores = oracle.num_threads()
        # one thread, on the first 256 rows (scaled by bytes like the full-row rate)
        oracle.set_num_threads(1)
        rate1, per1, n1 = cpu_oracle_rate(layer, x_bits, ms, 3.0, rows=(0, 256))
        oracle.set_num_threads(cores)
        cpu = {"value": rate, "unit": "GB/s", "cores": cores, "kind": "oracle",
               "sample": "%d full steps (4096x4096, batch 1, m=1..4), %.2f s/step" % (n, per),
               "one_thread": {"value": rate1, "unit": "GB/s",
                              "sample": "%d steps on rows 0..255, %.3f s/step" % (n1, per1)},
               "cpu_model": cpu_model()}

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32", "data": "synthetic",
            "config": {"workload": WORKLOAD, "out": out, "in": inp, "G": 8, "M": 4, "B": 8,
                       "books": "2^8 x 8 f16 N(0,0.02^2)", "codes": "u8 uniform",
                       "scales": "f16 U(0.5,1.5)", "x": "f16 N(0,1), batch 1",
                       "step": "aq_gemv for m=1,2,3,4", "parallelism": "replicas",
                       "l2": "rotating %d weight copies (%d x %.1f MB >= 3x L2 %.0f MB)" % (
                           ncopies, ncopies, pbytes / 1e6, l2 / 1e6)},
            "per_m": per_m,
            "configs": configs,
            "gemm": gemm,
            "dynamic_loading": loading,
            "wmse": wmse,
            "beam_search": beam,
            "roofline": {
                "bound": "hbm", "kernel": "gemv_lut_kernel m=%d" % dom["m"],
                "achieved": dom["GB_s"], "peak": hbm_peak, "unit": "GB/s",
                "frac": round(dom["GB_s"] / hbm_peak, 4),
                "traffic": profiled_traffic(WORKLOAD, dom["m"]),
                "peak_source": peak_src},
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": 2 * len(ms) * args.steps,   # product + split-K reduction per call
            "timed_region": {"graph_steps": glen, "replays": args.steps // glen,
                             "remainder_steps": rest, "ms": round(ms_total, 3)},
            "clocks": clk,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def profile_gemv(args):
    """Three aq_gemv calls of one layer of a named workload, nothing else (ncu captures)."""
    import torch
    from paper_2606_12876_gb300 import build as libbuild
    from paper_2606_12876_gb300.linear import AQLinear, x_to_device
    import workloads
    libbuild.build()
    name, _, lname = args.profile_gemv.partition(":")
    (_, layer), = list(workloads.config_layers(name, only=[lname] if lname else None))
    if args.bits:
        cfg = workloads.CONFIGS[name]
        layer = workloads.make_layer(layer["out"], layer["in"], cfg["G"], cfg["M"], args.bits,
                                     cfg["book_dtype"], cfg["book_std"], cfg["scale_dtype"],
                                     cfg["seed"])
    lin = AQLinear.from_layer(layer)
    xdt = workloads.CONFIGS[name]["x_dtype"]
    x = x_to_device(workloads.config_x(name, args.batch, layer["in"]), xdt)
    for _ in range(3):
        lin.gemv(x, args.m)
    torch.cuda.synchronize()
    print("profiled %s batch %d m %d" % (args.profile_gemv, args.batch, args.m))


def main():
    args = parse()
    if args.profile_gemv:
        profile_gemv(args)
        return
    if args.impl == "reference":
        reference_arm(args)
    else:
        own_arm(args)


if __name__ == "__main__":
    main()
